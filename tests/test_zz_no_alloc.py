"""ssd_lm_head_static: the allocation-free LM head must give what ssd_lm_head gives.

Callers that cannot allocate device memory (inside a CUDA-graph capture, under
a fixed memory budget owned by another allocator) use this entry point; its
scratch is a fixed device array shared by all calls.  Checked through the C ABI
on two calls in a row with different inputs, so a stale scratch would show.
This file is collected last so that a failure here never hides another test.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth
from paper_2510_22641_gb300 import _binding
from tests.gpu_util import make_model
from tests.parity import assert_logits_close

pytestmark = pytest.mark.gpu


def test_static_lm_head_equals_ctx_lm_head_twice():
    w = synth.TINY.replace(norm_gain="perturbed")
    model, _, dev = make_model(w)
    lib = _binding.load()
    d, V, rows = w.shape.d_model, w.shape.vocab, 7
    stream = torch.cuda.current_stream()
    for call, seed in enumerate((21, 22)):
        x = torch.from_numpy(synth.normal_f64(seed, 1, (rows, d), std=2.0).astype(np.float32)).cuda()
        tok_ref = torch.zeros(rows, dtype=torch.int32, device="cuda")
        lg_ref = torch.zeros((rows, V), device="cuda")
        model.lm_head(x, tok_ref, lg_ref)
        model.sync()
        tok = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
        lg = torch.full((rows, V), float("nan"), device="cuda")
        st = lib.ssd_lm_head_static(dev["lm_head"].data_ptr(), dev["final_norm"].data_ptr(), x.data_ptr(), rows,
                                    V, d, ctypes.c_float(w.shape.rms_eps), tok.data_ptr(), lg.data_ptr(),
                                    stream.cuda_stream)
        assert st == 0, _binding.STATUS.get(st)
        torch.cuda.synchronize()
        assert tok.cpu().tolist() == tok_ref.cpu().tolist(), f"call {call}"
        for r in range(rows):
            assert_logits_close(lg[r].cpu().numpy(), lg_ref[r].cpu().numpy(), f"call {call} row {r}")
    bad = lib.ssd_lm_head_static(dev["lm_head"].data_ptr(), dev["final_norm"].data_ptr(), x.data_ptr(), 10, V, d,
                                 ctypes.c_float(1e-5), tok.data_ptr(), None, stream.cuda_stream)
    assert bad == 1                                        # rows beyond the stated maximum
    model.close()
