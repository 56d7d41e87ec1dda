"""ssd_lm_head_static: the allocation-free LM head must give what ssd_lm_head and the oracle give.

Callers that cannot allocate device memory (code running while a stream is captured into a CUDA
graph, serving loops whose device memory belongs to another allocator) use this entry point; its
scratch is a fixed device array shared by all calls.  Checked through the C ABI on two calls in a
row with different inputs, so a stale scratch would show, against the context's ssd_lm_head and
against the fp64 oracle's g(x) = W_lm RMSNorm_f(x).  Further shapes: a width that is a multiple of
64 but not of 256, a vocabulary whose last 128-row tile is partial, and a 7B-sized head whose grid
reaches the array's CTA cap.  This file is collected last so that a failure here never hides
another test.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2510_22641_gb300 as lib
import synth
from paper_2510_22641_gb300 import _binding
from tests.gpu_util import make_model
from tests.parity import MARGIN, assert_logits_close, margin

pytestmark = pytest.mark.gpu


def static_head(l, lm_head, gain, x, rows, V, d, eps, tok, lg, stream):
    return l.ssd_lm_head_static(lm_head.data_ptr(), gain.data_ptr(), x.data_ptr(), rows, V, d, ctypes.c_float(eps),
                                tok.data_ptr(), None if lg is None else lg.data_ptr(), stream.cuda_stream)


def oracle_head(w_bits, gain_bits, x, eps):
    """g(x) of the fp64 oracle for every row of x (fp32 rows widened to fp64)."""
    V, d = w_bits.shape
    cfg = oracle.OracleConfig(n_layers=0, d_model=d, n_heads=1, head_dim=d, d_ff=d, vocab=V, draft_exit_k=0,
                              rms_eps=eps)
    m = oracle.Model(cfg, {"lm_head": synth.bf16_to_f64(w_bits), "final_norm": synth.bf16_to_f64(gain_bits)}, [], 0.0)
    return [oracle.lm_head(m, r.astype(np.float64)) for r in x]


def check_rows(tok, lg, ref_rows, what):
    for r, ref in enumerate(ref_rows):
        assert_logits_close(lg[r], ref, f"{what} row {r}")
        if int(tok[r]) != int(np.argmax(ref)):
            assert margin(ref) < MARGIN, f"{what} row {r}: token {int(tok[r])} != oracle {int(np.argmax(ref))}"
    assert list(tok) == [int(np.argmax(row)) for row in lg]   # the token is the argmax of the returned row


def test_static_lm_head_equals_ctx_lm_head_and_oracle_twice():
    w = synth.TINY.replace(norm_gain="perturbed")
    model, bits, dev = make_model(w)
    l = _binding.load()
    d, V, rows, eps = w.shape.d_model, w.shape.vocab, 7, w.shape.rms_eps
    stream = torch.cuda.current_stream()
    for call, seed in enumerate((21, 22)):
        xh = synth.normal_f64(seed, 1, (rows, d), std=2.0).astype(np.float32)
        x = torch.from_numpy(xh).cuda()
        tok_ref = torch.zeros(rows, dtype=torch.int32, device="cuda")
        lg_ref = torch.zeros((rows, V), device="cuda")
        model.lm_head(x, tok_ref, lg_ref)
        model.sync()
        tok = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
        lg = torch.full((rows, V), float("nan"), device="cuda")
        st = static_head(l, dev["lm_head"], dev["final_norm"], x, rows, V, d, eps, tok, lg, stream)
        assert st == 0, _binding.STATUS.get(st)
        torch.cuda.synchronize()
        assert tok.cpu().tolist() == tok_ref.cpu().tolist(), f"call {call}"
        got = lg.cpu().numpy()
        for r in range(rows):
            assert_logits_close(got[r], lg_ref[r].cpu().numpy(), f"call {call} row {r} vs ssd_lm_head")
        check_rows(tok.cpu().tolist(), got, oracle_head(bits["lm_head"], bits["final_norm"], xh, eps), f"call {call}")
    bad = l.ssd_lm_head_static(dev["lm_head"].data_ptr(), dev["final_norm"].data_ptr(), x.data_ptr(), 10, V, d,
                               ctypes.c_float(1e-5), tok.data_ptr(), None, stream.cuda_stream)
    assert bad == 1                                        # rows beyond the stated maximum
    bad = l.ssd_lm_head_static(dev["lm_head"].data_ptr(), dev["final_norm"].data_ptr(), x.data_ptr(), 2, V, 200,
                               ctypes.c_float(1e-5), tok.data_ptr(), None, stream.cuda_stream)
    assert bad == 1                                        # d_model not a multiple of 64
    model.close()


@pytest.mark.parametrize("d,V,rows", [(320, 2000, 5), (4096, 32000, 2)], ids=["d320_v2000", "d4096_v32000"])
def test_static_lm_head_other_shapes_match_oracle(d, V, rows):
    """d = 320 (a multiple of 64, not of 256) with a partial last vocabulary tile; the 7B head
    (250 row tiles x 64 slices: the grid reaches the scratch array's 320-CTA cap on 152 SMs)."""
    l = _binding.load()
    w_bits = synth.normal_bf16(5, 1, (V, d), std=0.02)
    g_bits = synth.normal_bf16(5, 2, (d,), mean=1.0, std=0.1)
    lm_head, gain = lib.bf16_bits_to_device(w_bits), lib.bf16_bits_to_device(g_bits)
    stream = torch.cuda.current_stream()
    for seed in (31, 32):
        xh = synth.normal_f64(seed, 3, (rows, d), std=1.5).astype(np.float32)
        x = torch.from_numpy(xh).cuda()
        tok = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
        lg = torch.full((rows, V), float("nan"), device="cuda")
        assert static_head(l, lm_head, gain, x, rows, V, d, 1e-5, tok, lg, stream) == 0
        torch.cuda.synchronize()
        check_rows(tok.cpu().tolist(), lg.cpu().numpy(), oracle_head(w_bits, g_bits, xh, 1e-5), f"d={d} V={V}")
