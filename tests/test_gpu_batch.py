"""Batched requests (the serving form of Algorithm 1) on the GPU against the fp64 oracle.

B requests with ragged prompts decode in lockstep through ssd_prefill_batch / ssd_decode_batch.
Every request must match the oracle run on it alone (tokens up to an excused near-tie, full-model
and draft logits at the stated tolerance, per-step accept lengths and kv_len bit-exact); the
oracle's lockstep batch loop is pinned on the CPU to give each request exactly that run.
Verification rows beyond 16 (4 requests at gamma >= 4, 16 requests at gamma = 6) go through the
medium-M tensor-core kernel; fewer rows through the weight-streaming GEMV.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import batch_device_inputs, make_model
from tests.parity import assert_draft_logits, assert_logits_close, assert_step_log, common_prefix

pytestmark = pytest.mark.gpu

GAMMA_MAX = 7


def tiny_batch(batch=4, **kw) -> synth.BatchWorkload:
    base = synth.TINY.replace(norm_gain="perturbed", **kw)
    return synth.TINY_B4.replace(base=base, batch=batch)


@pytest.fixture(scope="module")
def tiny_bits():
    return synth.make_weights(synth.TINY.replace(norm_gain="perturbed"))


@pytest.fixture(scope="module")
def model4(tiny_bits):
    bw = tiny_batch(gamma=GAMMA_MAX)
    model, _, dev = make_model(bw.base, tiny_bits, gamma_max=GAMMA_MAX, max_seq=bw.max_seq(), max_batch=4)
    yield model
    model.close()


def set_scale(model, w):
    model.resid_scale.copy_(torch.tensor(w.resid_scale(), device="cuda"))
    model.in_scale.copy_(torch.tensor([w.in_scale()], device="cuda"))


def oracle_runs(bw, bits, gamma, greedy=False):
    m = oracle.model_from_bits(bw.base, bits, synth.bf16_to_f64)
    out = []
    for vis, prompt in synth.make_batch_inputs(bw):
        v = synth.bf16_to_f64(vis)
        if greedy:
            out.append(oracle.greedy_generate(m, v, prompt, bw.base.max_new))
        else:
            out.append(oracle.ssd_generate(m, v, prompt, bw.base.max_new, gamma, keep_draft_logits=True))
    return out


def gpu_batch(model, bw, gamma, capture=True):
    """prefill + decode of the whole batch; per request: tokens, logits, draft logits, stats, step log."""
    B, V, T = bw.batch, bw.base.shape.vocab, bw.base.max_new
    _, dv, nv, dp, npr = batch_device_inputs(bw)
    logits = torch.full((B, T, V), float("nan"), device="cuda") if capture else None
    dlog = (torch.full((B, T, model.cfg["gamma_max"], V), float("nan"), device="cuda")
            if capture and gamma > 0 else None)
    model.set_logits_capture(logits)
    model.set_draft_logits_capture(dlog)
    first = torch.zeros(B, dtype=torch.int32, device="cuda")
    out = torch.zeros(B, T, dtype=torch.int32, device="cuda")
    n = torch.zeros(B, dtype=torch.int32, device="cuda")
    model.prefill_batch(dv, nv, dp, npr, first)
    if gamma > 0:
        model.decode_batch(T, gamma, out, n)
    else:
        model.greedy_decode_batch(T, out, n)
    model.sync()
    res = []
    for b in range(B):
        st = model.batch_stats(b)
        st["accepted_log"], st["drafted_log"] = model.batch_step_log(b)
        res.append({"tokens": out[b, : int(n[b])].cpu().tolist(), "first": int(first[b]),
                    "logits": logits[b].cpu().numpy() if capture else None,
                    "draft_logits": dlog[b].cpu().numpy() if dlog is not None else None, "stats": st})
    model.set_logits_capture(None)
    model.set_draft_logits_capture(None)
    return res


def check_request(r, ref, gamma):
    assert r["first"] == ref.tokens[0]
    agree = common_prefix(r["tokens"], ref.tokens, ref.logits)
    if r["logits"] is not None:
        for t in range(min(agree + 1, len(ref.tokens))):
            assert_logits_close(r["logits"][t], ref.logits[t], f"logits of token {t}")
    st = r["stats"]
    if gamma > 0:
        k = assert_step_log(st["accepted_log"], st["drafted_log"], ref, agree)
        if agree == len(ref.tokens):
            assert st["steps"] == len(ref.accept_lengths)
            assert st["accepted"] == sum(ref.accept_lengths)
            assert st["kv_len"] == ref.kv_len
        if r["draft_logits"] is not None:
            assert assert_draft_logits(r["draft_logits"], ref, k) >= sum(1 for d in ref.draft_tokens[:k] if d)
    elif agree == len(ref.tokens):
        assert st["kv_len"] == ref.kv_len
    return agree


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.2, 4), (1.0, 2), (0.05, 7), (0.2, 1)])
def test_batch_ssd_matches_oracle_per_request(model4, tiny_bits, s, gamma):
    """4 ragged requests; gamma = 4 and 7 verify 20 and 32 rows (medium-M kernel), gamma <= 2 at
    most 12 (GEMV)."""
    bw = tiny_batch(s=s)
    set_scale(model4, bw.base)
    got = gpu_batch(model4, bw, gamma)
    refs = oracle_runs(bw, tiny_bits, gamma)
    for b, (r, ref) in enumerate(zip(got, refs)):
        check_request(r, ref, gamma)


def test_batch_greedy_matches_oracle_per_request(model4, tiny_bits):
    bw = tiny_batch(s=0.2)
    set_scale(model4, bw.base)
    got = gpu_batch(model4, bw, 0)
    for r, ref in zip(got, oracle_runs(bw, tiny_bits, 0, greedy=True)):
        assert check_request(r, ref, 0) >= 8


@pytest.mark.parametrize("gamma", [2, 5])
def test_batch_ssd_equals_batch_greedy(model4, gamma):
    """Each request's SSD tokens equal its greedy tokens (the GPU's verification rows, batched and
    through either projection kernel, reproduce greedy decoding up to near-ties)."""
    bw = tiny_batch(s=0.2)
    set_scale(model4, bw.base)
    ssd = gpu_batch(model4, bw, gamma)
    gr = gpu_batch(model4, bw, 0)
    for a, g in zip(ssd, gr):
        n = 0
        while n < len(a["tokens"]) and a["tokens"][n] == g["tokens"][n]:
            n += 1
        if n < len(g["tokens"]):
            top = np.sort(g["logits"][n])
            assert top[-1] - top[-2] < 1e-2, f"SSD parts from greedy at token {n} (margin {top[-1] - top[-2]})"


def test_batch_of_16_verifies_112_rows(tiny_bits):
    """16 requests at gamma = 6: every verification projection carries 112 rows (7 chunks of the
    medium-M kernel) and every drafting projection 16 rows."""
    bw = tiny_batch(batch=16, s=0.05, gamma=6)
    model, _, _ = make_model(bw.base, tiny_bits, gamma_max=6, max_seq=bw.max_seq(), max_batch=16)
    try:
        set_scale(model, bw.base)
        got = gpu_batch(model, bw, 6)
        refs = oracle_runs(bw, tiny_bits, 6)
        for r, ref in zip(got, refs):
            check_request(r, ref, 6)
    finally:
        model.close()


def test_batch_request_finishing_early_on_eos(model4, tiny_bits):
    """A request that emits eos stops (its tokens end there) while the others go on."""
    bw0 = tiny_batch(s=0.05)
    refs = oracle_runs(bw0, tiny_bits, 4)
    eos = refs[0].tokens[3]
    bw = bw0.replace(base=bw0.base.replace(eos_id=eos))
    model, _, _ = make_model(bw.base, tiny_bits, gamma_max=GAMMA_MAX, max_seq=bw.max_seq(), max_batch=4)
    try:
        set_scale(model, bw.base)
        got = gpu_batch(model, bw, 4)
        refs = oracle_runs(bw, tiny_bits, 4)
        assert len(refs[0].tokens) <= 4
        for r, ref in zip(got, refs):
            check_request(r, ref, 4)
    finally:
        model.close()


def test_batch_host_buffers_and_call_order(model4, tiny_bits):
    """ssd_generate_batch (host buffers) equals the device-buffer calls; a batched decode needs a
    batched prefill; a single-request prefill in between invalidates the batch."""
    import paper_2510_22641_gb300 as lib
    bw = tiny_batch(s=0.2)
    set_scale(model4, bw.base)
    ins = synth.make_batch_inputs(bw)
    vis = np.concatenate([v for v, _ in ins])
    prompt = np.concatenate([p for _, p in ins])
    host = model4.generate_batch(vis, [v.shape[0] for v, _ in ins], prompt, [len(p) for _, p in ins],
                                 bw.base.max_new, 3)
    dev = gpu_batch(model4, bw, 3, capture=False)
    assert host == [r["tokens"] for r in dev]
    v0 = lib.bf16_bits_to_device(ins[0][0])
    p0 = torch.from_numpy(ins[0][1].astype(np.int32)).cuda()
    model4.prefill(v0, p0)
    with pytest.raises(lib.SSDError) as e:
        model4.decode_batch(8, 3)
    assert e.value.status == 5  # SSD_ERR_STATE
    with pytest.raises(lib.SSDError) as e:
        model4.prefill_batch(None, [0] * 5, p0, [3] * 5)
    assert e.value.status == 1  # more requests than max_batch
