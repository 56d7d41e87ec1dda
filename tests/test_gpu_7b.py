"""Full-size parity on the LLaVA-1.5-7B-shaped workload, in the launch configuration bench.py times.

The fp64 oracle cannot decode all 128 tokens at this size within a test, so:
  * sampled outputs: the oracle's prefill and first SSD steps (tokens, full-model
    logits of every emitted token, accept lengths, cache length) are compared
    with the GPU's;
  * properties that hold at any size are checked on all 128 tokens: the GPU's
    SSD stream equals its greedy stream bitwise for every s, and the per-step
    counts add up.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_22641_gb300 as lib
import synth
from tests.gpu_util import device_weights
from tests.parity import assert_draft_logits, assert_logits_close, common_prefix, steps_before

pytestmark = pytest.mark.gpu

W = synth.LLAVA7B


@pytest.fixture(scope="module")
def big():
    bits = synth.make_weights(W)
    dev = device_weights(bits)
    rs = torch.tensor(W.resid_scale(), device="cuda")
    ins = torch.tensor([W.in_scale()], device="cuda")
    cfg = lib.config_dict(W.shape, W.draft_exit_k, W.in_kind, W.in_hidden, lib.SSD_MAX_GAMMA,
                          W.prompt_len + W.max_new + lib.SSD_MAX_GAMMA + 1)
    model = lib.SSDModel(cfg, dev, rs, ins)
    vis, prompt = synth.make_inputs(W)
    v = lib.bf16_bits_to_device(vis)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    yield model, bits, vis, prompt, v, p
    model.close()


def decode(model, v, p, gamma, logits=None):
    model.set_logits_capture(logits)
    out = torch.zeros(W.max_new, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.prefill(v, p)
    if gamma:
        model.decode(W.max_new, gamma, out, n)
    else:
        model.greedy_decode(W.max_new, out, n)
    model.sync()
    return out[: int(n.item())].cpu().tolist(), model.stats()


def set_s(model, s):
    w = W.replace(s=s)
    model.resid_scale.copy_(torch.tensor(w.resid_scale(), device="cuda"))
    model.in_scale.copy_(torch.tensor([w.in_scale()], device="cuda"))


@pytest.mark.parametrize("s", synth.LLAVA7B_S_VALUES)
def test_ssd_equals_greedy_all_tokens(big, s):
    model, _, _, _, v, p = big
    set_s(model, s)
    toks, st = decode(model, v, p, W.gamma)
    gtoks, gst = decode(model, v, p, 0)
    assert toks == gtoks and len(toks) == W.max_new
    assert st["steps"] + st["accepted"] + 1 == W.max_new
    assert st["kv_len"] == gst["kv_len"] == W.prompt_len + W.max_new - 1
    assert sum(st["accept_hist"]) == st["steps"]
    set_s(model, W.s)


@pytest.mark.parametrize("s", [0.05, 0.2])
def test_sampled_prefix_matches_oracle(big, s):
    """The first 8 SSD steps against the fp64 oracle: tokens, the full-model logits of every emitted
    token, the drafting stage's logits g(I(x_k)), and the per-step accept lengths and draft counts
    (bit-exact).  s = 0.05 accepts most drafts, so verification rows with accepted drafts are
    exercised; s = 0.2 is the headline setting."""
    model, bits, vis, prompt, v, p = big
    set_s(model, s)
    steps = 8
    logits = torch.zeros((W.max_new, W.shape.vocab), device="cuda")
    dlog = torch.zeros((steps, lib.SSD_MAX_GAMMA, W.shape.vocab), device="cuda")
    model.set_draft_logits_capture(dlog)
    toks, st = decode(model, v, p, W.gamma, logits)
    acc, dr = model.step_log()
    model.set_logits_capture(None)
    model.set_draft_logits_capture(None)
    w = W.replace(s=s)
    m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    ref = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, W.max_new, W.gamma, max_steps=steps,
                              keep_draft_logits=True)
    assert len(ref.accept_lengths) == steps
    n_ref = len(ref.tokens)
    agree = common_prefix(toks[:n_ref], ref.tokens, ref.logits)
    lg = logits.cpu().numpy()
    for t in range(min(agree + 1, n_ref)):
        assert_logits_close(lg[t], ref.logits[t], f"7B logits of token {t}")
    k = steps_before(ref.accept_lengths, agree)
    assert acc[:k] == ref.accept_lengths[:k]
    assert dr[:k] == [len(d) for d in ref.draft_tokens[:k]]
    rows = assert_draft_logits(dlog.cpu().numpy(), ref, k)
    # the compared prefix may end early only at an oracle near-tie (common_prefix checks the
    # margin); with these seeds the first 8 steps agree at both settings
    assert k == steps and agree == n_ref, (k, agree, n_ref)
    assert rows >= steps
    if s == 0.05:
        assert sum(ref.accept_lengths) >= steps  # verification rows with accepted drafts occur
    set_s(model, W.s)
