"""Encoder-decoder (BLIP-2 FlanT5-shaped) CUDA path vs the fp64 encoder-decoder oracle, through the C ABI.

Tiny workload: 2 encoder + 4 decoder layers, d=256, 4 heads x 64, V=2048.  The encoder runs through
the tensor-core prefill GEMM (one 128-row tile for the default 48 encoder rows); a long case (130
encoder rows, 150 new tokens) spans two row tiles (the second holds 2 rows), three 64-key attention
chunks on both the encoder and the decoder side, and relative offsets beyond max_distance / 2 in
both bucket schemes.  The row prefill (the decode kernels in 8-row chunks) is checked against the
tensor-core one and the oracle, and a model with max_enc = 64 runs the cross-attention folded into
the cross-q projection's epilogue (the fixture's max_enc = 160 keeps the separate kernel).  The
FlanT5-xl-shaped case (24 + 24 layers, d=2048, V=32128) compares the oracle's prefill and first SSD
steps with the GPU's and checks SSD == greedy over all 30 tokens.
"""
import numpy as np
import pytest
import torch

import paper_2510_22641_gb300 as lib
import synth
from oracle import t5_oracle as T
from tests.gpu_util import make_t5_model, t5_device_inputs
from tests.parity import assert_logits_close, common_prefix, steps_before

pytestmark = pytest.mark.gpu

GAMMA_MAX = 8


def tiny(**kw):
    return synth.T5_TINY.replace(norm_gain="perturbed", **kw)


def oracle_model(w, bits):
    return T.model_from_bits(w, bits, synth.bf16_to_f64)


def oracle_run(w, bits, gamma, **kw):
    m = oracle_model(w, bits)
    q, prompt = synth.make_t5_inputs(w)
    z = synth.bf16_to_f64(q)
    if gamma == 0:
        return T.greedy_generate(m, z, prompt, w.max_new)
    return T.ssd_generate(m, z, prompt, w.max_new, gamma, **kw)


def gpu_decode(model, w, gamma, capture=True):
    _, _, v, p = t5_device_inputs(w)
    logits = torch.full((w.max_new, w.shape.vocab), float("nan"), device="cuda") if capture else None
    model.set_logits_capture(logits)
    out = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.prefill(v, p)
    if gamma > 0:
        model.decode(w.max_new, gamma, out, n)
    else:
        model.greedy_decode(w.max_new, out, n)
    model.sync()
    return out[: int(n.item())].cpu().tolist(), (logits.cpu().numpy() if capture else None), model.stats()


def check(toks, logits, stats, ref, gamma):
    agree = common_prefix(toks, ref.tokens, ref.logits)
    for t in range(min(agree + 1, len(ref.tokens))):
        assert_logits_close(logits[t], ref.logits[t], f"logits of token {t}")
    if gamma > 0 and agree == len(ref.tokens):
        assert stats["steps"] == len(ref.accept_lengths)
        assert stats["accepted"] == sum(ref.accept_lengths)
        assert stats["kv_len"] == ref.kv_len
        assert stats["accept_hist"][: gamma + 1] == np.bincount(ref.accept_lengths, minlength=gamma + 1).tolist()
    return agree


def set_s(model, w):
    model.resid_scale.copy_(torch.tensor(w.dec_scale(), device="cuda"))
    model.in_scale.copy_(torch.tensor([w.in_scale()], device="cuda"))


@pytest.fixture(scope="module")
def tiny_bits():
    return synth.make_t5_weights(tiny())


@pytest.fixture(scope="module")
def tiny_model(tiny_bits):
    w = tiny()
    model, _, dev = make_t5_model(w, tiny_bits, gamma_max=GAMMA_MAX, max_seq=200, max_enc=160)
    yield model
    model.close()


def test_t5_greedy_matches_oracle(tiny_model, tiny_bits):
    w = tiny(s=1.0)
    set_s(tiny_model, w)
    toks, logits, st = gpu_decode(tiny_model, w, 0)
    ref = oracle_run(w, tiny_bits, 0)
    assert check(toks, logits, st, ref, 0) >= 8
    assert st["kv_len"] == w.max_new  # decoder positions 0 .. max_new - 1


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.3, 4), (1.0, 4), (0.3, 1), (0.05, 8), (0.3, 3)])
def test_t5_ssd_matches_oracle_and_gpu_greedy(tiny_model, tiny_bits, s, gamma):
    w = tiny(s=s)
    set_s(tiny_model, w)
    toks, logits, st = gpu_decode(tiny_model, w, gamma)
    check(toks, logits, st, oracle_run(w, tiny_bits, gamma), gamma)
    gtoks, glogits, _ = gpu_decode(tiny_model, w, 0)
    assert toks == gtoks  # batch invariance: the verify rows reproduce greedy decoding bitwise
    np.testing.assert_array_equal(logits, glogits)
    assert st["steps"] + st["accepted"] + 1 == w.max_new


def test_t5_tensor_core_prefill_matches_row_prefill(tiny_model, tiny_bits):
    """The encoder through the tcgen05 prefill GEMM and through the decode kernels in 8-row chunks
    give the same greedy stream within the oracle's tolerance; both match the oracle."""
    w = tiny(s=0.3, n_query=100, n_prompt=30, max_new=40)
    set_s(tiny_model, w)
    toks, logits, st = gpu_decode(tiny_model, w, 0)
    rows_model, _, _ = make_t5_model(w, tiny_bits, gamma_max=GAMMA_MAX, max_seq=200, max_enc=160,
                                     options=lib.SSD_OPT_PREFILL_ROWS)
    try:
        set_s(rows_model, w)
        rtoks, rlogits, _ = gpu_decode(rows_model, w, 0)
    finally:
        rows_model.close()
    ref = oracle_run(w, tiny_bits, 0)
    agree = check(toks, logits, st, ref, 0)
    assert agree >= 16
    ragree = common_prefix(rtoks, ref.tokens, ref.logits)
    assert ragree >= 16
    for t in range(min(agree + 1, ragree + 1, w.max_new)):
        assert_logits_close(logits[t], rlogits[t], f"tensor-core vs row prefill, logits of token {t}")


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.3, 3)])
def test_t5_folded_cross_attention(tiny_model, tiny_bits, s, gamma):
    """With max_enc <= 128 the cross-attention runs in the cross-q projection's epilogue: greedy and
    SSD against the oracle, SSD == greedy bitwise, logits within tolerance of the separate
    cross-attention kernel's (the fixture's max_enc = 160 keeps that path)."""
    w = tiny(s=s)
    fold, _, _ = make_t5_model(w, tiny_bits, gamma_max=GAMMA_MAX, max_seq=200, max_enc=64)
    try:
        set_s(fold, w)
        gtoks, glogits, gst = gpu_decode(fold, w, 0)
        toks, logits, st = gpu_decode(fold, w, gamma)
    finally:
        fold.close()
    assert check(gtoks, glogits, gst, oracle_run(w, tiny_bits, 0), 0) >= 8
    check(toks, logits, st, oracle_run(w, tiny_bits, gamma), gamma)
    assert toks == gtoks
    np.testing.assert_array_equal(logits, glogits)
    set_s(tiny_model, w)
    ktoks, klogits, _ = gpu_decode(tiny_model, w, 0)
    n = common_prefix(gtoks, ktoks, klogits)
    for t in range(min(n + 1, w.max_new)):
        assert_logits_close(glogits[t], klogits[t], f"folded vs separate cross-attention, logits of token {t}")


def test_t5_long_encoder_and_decoder(tiny_model, tiny_bits):
    """130 encoder rows and 150 new tokens: several key chunks on both sides, far relative buckets."""
    w = tiny(s=0.3, n_query=100, n_prompt=30, max_new=150)
    set_s(tiny_model, w)
    toks, logits, st = gpu_decode(tiny_model, w, 4)
    ref = oracle_run(w, tiny_bits, 4)
    agree = check(toks, logits, st, ref, 4)
    assert agree >= 16
    gtoks, _, _ = gpu_decode(tiny_model, w, 0, capture=False)
    assert toks == gtoks


def test_t5_step_api_matches_oracle_steps(tiny_model, tiny_bits):
    """ssd_draft / ssd_verify one step at a time: emitted counts equal the oracle's a + 1."""
    w = tiny(s=0.3)
    set_s(tiny_model, w)
    tiny_model.set_logits_capture(None)
    ref = oracle_run(w, tiny_bits, 4, max_steps=4)
    _, _, v, p = t5_device_inputs(w)
    first = torch.zeros(1, dtype=torch.int32, device="cuda")
    ne = torch.zeros(1, dtype=torch.int32, device="cuda")
    em = torch.zeros(GAMMA_MAX + 1, dtype=torch.int32, device="cuda")
    dt = torch.zeros(GAMMA_MAX, dtype=torch.int32, device="cuda")
    tiny_model.prefill(v, p, first)
    tiny_model.sync()
    assert int(first.item()) == ref.tokens[0]
    got = [ref.tokens[0]]
    for step, a in enumerate(ref.accept_lengths):
        tiny_model.draft(4, dt)
        tiny_model.verify(4, ne, em)
        tiny_model.sync()
        n = int(ne.item())
        got += em[:n].cpu().tolist()
        if got != ref.tokens[: len(got)]:
            break  # a near-tie excused below
        assert n == a + 1
        assert dt[:4].cpu().tolist()[:a] == ref.draft_tokens[step][:a]
    common_prefix(got, ref.tokens[: len(got)], ref.logits)


def test_t5_host_buffer_generate_equals_device_path(tiny_model, tiny_bits):
    w = tiny(s=0.3)
    set_s(tiny_model, w)
    tiny_model.set_logits_capture(None)
    q, prompt = synth.make_t5_inputs(w)
    toks, st = tiny_model.generate(q, prompt, w.max_new, 4)
    dtoks, _, dst = gpu_decode(tiny_model, w, 4, capture=False)
    assert toks == dtoks and st["accepted"] == dst["accepted"]
    gtoks, _ = tiny_model.greedy_generate(q, prompt, w.max_new)
    assert gtoks == toks


def test_t5_encoder_rows_over_capacity_are_rejected(tiny_model):
    w = tiny(n_query=150, n_prompt=20)
    _, _, v, p = t5_device_inputs(w)
    with pytest.raises(lib.SSDError) as e:
        tiny_model.prefill(v, p)
    assert e.value.status == 4  # SSD_ERR_CAPACITY


def test_t5_draft_exit_at_last_layer_accepts_everything(tiny_bits):
    w = tiny(in_kind=synth.IN_IDENTITY, draft_exit_k=synth.T5_TINY.shape.n_dec)
    bits = {k: v for k, v in tiny_bits.items() if not k.startswith("in_")}
    model, _, _ = make_t5_model(w, bits, gamma_max=4)
    try:
        toks, _, st = gpu_decode(model, w, 4, capture=False)
        ref = oracle_run(w, bits, 4)
        common_prefix(toks, ref.tokens, ref.logits)
        assert st["accepted"] == st["drafted"]  # every drafted token accepted (g_eff < 4 in the last step)
        assert st["accept_hist"][4] >= st["steps"] - 1
    finally:
        model.close()


# --------------------------------------------------------------------------- FlanT5-xl shape

XL = synth.FLANT5XL


@pytest.fixture(scope="module")
def xl():
    bits = synth.make_t5_weights(XL)
    model, _, _ = make_t5_model(XL, bits, gamma_max=GAMMA_MAX, max_seq=XL.max_new + GAMMA_MAX + 2,
                                max_enc=XL.enc_len)
    yield model, bits
    model.close()


@pytest.mark.parametrize("s", [0.05, 0.2, 1.0])
def test_xl_ssd_equals_greedy_all_tokens(xl, s):
    model, _ = xl
    w = XL.replace(s=s)
    set_s(model, w)
    toks, _, st = gpu_decode(model, w, w.gamma, capture=False)
    gtoks, _, gst = gpu_decode(model, w, 0, capture=False)
    assert toks == gtoks and len(toks) == w.max_new
    assert st["steps"] + st["accepted"] + 1 == w.max_new
    assert st["kv_len"] == gst["kv_len"] == w.max_new


def test_xl_sampled_prefix_matches_oracle(xl):
    model, bits = xl
    set_s(model, XL)
    toks, logits, st = gpu_decode(model, XL, XL.gamma)
    model.set_logits_capture(None)
    ref = oracle_run(XL, bits, XL.gamma, max_steps=2)
    n_ref = len(ref.tokens)
    agree = common_prefix(toks[:n_ref], ref.tokens, ref.logits)
    for t in range(min(agree + 1, n_ref)):
        assert_logits_close(logits[t], ref.logits[t], f"FlanT5-xl logits of token {t}")
    k = steps_before(ref.accept_lengths, agree)
    assert k >= 1 or agree < 2
