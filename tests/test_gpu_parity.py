"""CUDA path vs the fp64 oracle on the tiny workload and its edge cases (through the C ABI).

Sizes here finish in seconds in the oracle yet span several 128x64 weight
units per matrix, several 64-key attention chunks, a ragged prefill chunk and
a vocabulary tail.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2510_22641_gb300 as lib
import synth
from tests.gpu_util import device_inputs, make_model
from tests.parity import assert_draft_logits, assert_logits_close, assert_step_log, common_prefix, steps_before

pytestmark = pytest.mark.gpu


def run_oracle(w, bits, gamma=None, greedy=False):
    m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    if greedy:
        return oracle.greedy_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, max_seq=w.max_seq())
    return oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, gamma or w.gamma,
                               keep_draft_logits=True)


def gpu_decode(model, w, gamma, capture=True):
    """prefill + decode through the device-buffer entry points; returns tokens, logits, stats (with
    capture, stats["draft_logits"] holds the drafting stage's logits [step][j][vocab])."""
    _, _, v, p = device_inputs(w)
    logits = torch.full((w.max_new, w.shape.vocab), float("nan"), device="cuda") if capture else None
    dlog = (torch.full((w.max_new, model.cfg["gamma_max"], w.shape.vocab), float("nan"), device="cuda")
            if capture and gamma > 0 else None)
    model.set_logits_capture(logits)
    model.set_draft_logits_capture(dlog)
    out = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.prefill(v, p)
    if gamma > 0:
        model.decode(w.max_new, gamma, out, n)
    else:
        model.greedy_decode(w.max_new, out, n)
    model.sync()
    toks = out[: int(n.item())].cpu().tolist()
    stats = model.stats()
    stats["accepted_log"], stats["drafted_log"] = model.step_log()
    if dlog is not None:
        stats["draft_logits"] = dlog.cpu().numpy()
    model.set_draft_logits_capture(None)
    return toks, (logits.cpu().numpy() if capture else None), stats


def check_against_oracle(toks, logits, stats, ref, gamma):
    """Tokens up to an excused near-tie, full-model logits of every agreeing token, and for SSD the
    per-step accept lengths and draft counts (bit-exact), the counters, and the draft logits."""
    agree = common_prefix(toks, ref.tokens, ref.logits)
    for t in range(min(agree + 1, len(ref.tokens))):
        assert_logits_close(logits[t], ref.logits[t], f"logits of token {t}")
    if gamma > 0:
        k = assert_step_log(stats["accepted_log"], stats["drafted_log"], ref, agree)
        if agree == len(ref.tokens):
            assert stats["steps"] == len(ref.accept_lengths)
            assert stats["accepted"] == sum(ref.accept_lengths)
            assert stats["kv_len"] == ref.kv_len
            assert stats["accept_hist"][: gamma + 1] == np.bincount(ref.accept_lengths, minlength=gamma + 1).tolist()
        assert k <= stats["steps"]
        if "draft_logits" in stats and ref.draft_logits:
            # at least the first draft row of every compared step that drafted anything
            assert assert_draft_logits(stats["draft_logits"], ref, k) >= sum(1 for d in ref.draft_tokens[:k] if d)
    return agree


def assert_accept_sequence(model, ref, toks):
    """The device's per-step record against the oracle's, over the steps before the streams part
    (toks may be a prefix of the oracle's stream)."""
    acc, dr = model.step_log()
    assert_step_log(acc, dr, ref, common_prefix(toks, ref.tokens[: len(toks)], ref.logits))


@pytest.fixture(scope="module")
def tiny_bits():
    return synth.make_weights(synth.TINY.replace(norm_gain="perturbed"))


@pytest.fixture(scope="module")
def tiny_model(tiny_bits):
    w = synth.TINY.replace(norm_gain="perturbed", gamma=8)
    model, _, dev = make_model(w, tiny_bits, gamma_max=8, max_seq=w.max_seq())
    yield model, dev
    model.close()


def set_scale(model, w):
    model.resid_scale.copy_(torch.tensor(w.resid_scale(), device="cuda"))
    model.in_scale.copy_(torch.tensor([w.in_scale()], device="cuda"))


def test_greedy_matches_oracle(tiny_model, tiny_bits):
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=1.0)
    set_scale(model, w)
    toks, logits, _ = gpu_decode(model, w, 0)
    ref = run_oracle(w, tiny_bits, greedy=True)
    assert check_against_oracle(toks, logits, {}, ref, 0) >= 8


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.2, 4), (1.0, 4), (0.2, 1), (0.05, 8), (0.2, 3)])
def test_ssd_matches_oracle_and_gpu_greedy(tiny_model, tiny_bits, s, gamma):
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=s)
    set_scale(model, w)
    toks, logits, stats = gpu_decode(model, w, gamma)
    ref = run_oracle(w, tiny_bits, gamma)
    check_against_oracle(toks, logits, stats, ref, gamma)
    # batch invariance: the verify pass (gamma+1 rows) reproduces greedy decoding bitwise
    gtoks, glogits, _ = gpu_decode(model, w, 0)
    assert toks == gtoks
    np.testing.assert_array_equal(logits, glogits)
    assert stats["emitted"] == w.max_new
    assert sum(a * c for a, c in enumerate(stats["accept_hist"])) == stats["accepted"]
    assert stats["steps"] + stats["accepted"] + 1 == w.max_new


@pytest.fixture(scope="module")
def tiny_model_host_loop(tiny_bits):
    """The same context driven from the host, one plain graph per step (SSD_OPT_HOST_LOOP)."""
    w = synth.TINY.replace(norm_gain="perturbed", gamma=8)
    model, _, dev = make_model(w, tiny_bits, gamma_max=8, max_seq=w.max_seq(), options=lib.SSD_OPT_HOST_LOOP)
    yield model, dev
    model.close()


@pytest.mark.parametrize("host", [False, True], ids=["device_loop", "host_loop"])
@pytest.mark.parametrize("s,cap,n_max", [(0.05, 8, 120), (0.2, 6, 90), (1.0, 8, 40)])
def test_dynamic_draft_length_matches_oracle(request, tiny_bits, s, cap, n_max, host):
    """Sec. "Choice of d": each step drafts min(d(kv_len + 2), cap) tokens; tokens, logits, steps,
    accept lengths and kv_len match the oracle's dynamic run, and the tokens equal greedy decoding."""
    model, _ = request.getfixturevalue("tiny_model_host_loop" if host else "tiny_model")
    w = synth.TINY.replace(norm_gain="perturbed", s=s)
    set_scale(model, w)
    _, _, v, p = device_inputs(w)
    logits = torch.full((w.max_new, w.shape.vocab), float("nan"), device="cuda")
    dlog = torch.full((w.max_new, 8, w.shape.vocab), float("nan"), device="cuda")
    model.set_logits_capture(logits)
    model.set_draft_logits_capture(dlog)
    out = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.prefill(v, p)
    model.decode_dynamic(w.max_new, 5, n_max, cap, out, n)
    model.sync()
    toks, stats = out[: int(n.item())].cpu().tolist(), model.stats()
    stats["accepted_log"], stats["drafted_log"] = model.step_log()
    stats["draft_logits"] = dlog.cpu().numpy()
    model.set_draft_logits_capture(None)
    m = oracle.model_from_bits(w, tiny_bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    ref = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, cap, dynamic=(5, n_max),
                              keep_draft_logits=True)
    _, dec = model.launch_counts()
    check_against_oracle(toks, logits.cpu().numpy(), stats, ref, cap)
    assert stats["drafted"] == sum(len(d) for d in ref.draft_tokens)
    gtoks, _, _ = gpu_decode(model, w, 0, capture=False)
    assert toks == gtoks
    # launches: setup, loop test at entry, copy-out; per step the branch for gamma_t plus its
    # selection (and, in the device loop, the loop test)
    L, k = w.shape.n_layers, w.draft_exit_k
    body = lambda g: g * (1 + 5 * k + 2 + 1) + (1 + 5 * L + 1 + 1)
    p_, expect = w.prompt_len, 0
    for kv in ref.kv_lens:
        g_t = min(oracle.draft_length(p_ + 2, 5, n_max), cap)
        expect += body(g_t) + (0 if host else 2)
        p_ = kv
    assert dec == expect + (2 if host else 3)


@pytest.fixture(scope="module")
def tiny_model_g15(tiny_bits):
    """gamma_max = 15 (d0 + 10 for d0 = 5): verification passes of up to 16 rows."""
    w = synth.TINY.replace(norm_gain="perturbed", gamma=15)
    model, _, dev = make_model(w, tiny_bits, gamma_max=15, max_seq=w.max_seq())
    yield model, dev
    model.close()


@pytest.mark.parametrize("s,n_max", [(0.05, 32), (0.2, 200)])
def test_dynamic_draft_length_over_generated_tokens(tiny_model_g15, tiny_bits, s, n_max):
    """d(t) with t = the index of the next new token and N the generation length, capped at 15:
    tokens, logits, draft logits, per-step accept lengths and draft counts match the oracle's run
    under the same reading; the steps draft up to 15 tokens (16-row verification passes)."""
    model, _ = tiny_model_g15
    w = synth.TINY.replace(norm_gain="perturbed", s=s)
    set_scale(model, w)
    _, _, v, p = device_inputs(w)
    logits = torch.full((w.max_new, w.shape.vocab), float("nan"), device="cuda")
    dlog = torch.full((w.max_new, 15, w.shape.vocab), float("nan"), device="cuda")
    model.set_logits_capture(logits)
    model.set_draft_logits_capture(dlog)
    out = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.prefill(v, p)
    model.decode_dynamic(w.max_new, 5, n_max, 15, out, n, t_from=lib.SSD_DLEN_GENERATED)
    model.sync()
    toks, stats = out[: int(n.item())].cpu().tolist(), model.stats()
    stats["accepted_log"], stats["drafted_log"] = model.step_log()
    stats["draft_logits"] = dlog.cpu().numpy()
    model.set_draft_logits_capture(None)
    m = oracle.model_from_bits(w, tiny_bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    ref = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, 15, dynamic=(5, n_max, "generated"),
                              keep_draft_logits=True)
    check_against_oracle(toks, logits.cpu().numpy(), stats, ref, 15)
    assert stats["drafted"] == sum(len(d) for d in ref.draft_tokens)
    assert max(len(d) for d in ref.draft_tokens) >= 7


def test_kv_cache_after_rollback_equals_greedy_cache(tiny_model):
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=0.2)
    set_scale(model, w)
    gpu_decode(model, w, 4, capture=False)
    k1, v1, n1 = model.kv()
    k1, v1 = k1[:, :, :n1].clone(), v1[:, :, :n1].clone()
    gpu_decode(model, w, 0, capture=False)
    k2, v2, n2 = model.kv()
    assert n1 == n2 == w.prompt_len + w.max_new - 1
    assert torch.equal(k1.view(torch.int32), k2[:, :, :n2].view(torch.int32))
    assert torch.equal(v1.view(torch.int32), v2[:, :, :n2].view(torch.int32))


def test_prefill_kv_matches_oracle(tiny_bits):
    w = synth.TINY.replace(norm_gain="perturbed", max_new=1)
    model, _, _ = make_model(w, tiny_bits)
    gpu_decode(model, w, 0, capture=False)
    k, v, n = model.kv()
    m = oracle.model_from_bits(w, tiny_bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    cache = oracle.KVCache(m.cfg, w.max_seq())
    oracle.prefill(m, cache, synth.bf16_to_f64(vis), prompt)
    P = w.prompt_len
    assert n == P
    for got, ref in ((k, cache.k), (v, cache.v)):
        g = got[:, :, :P].float().cpu().numpy()
        r = ref[:, :, :P]
        # fp32 cache; the remaining difference is fp32 arithmetic on bf16 weights vs fp64
        rms = float(np.sqrt(np.mean(r * r)))
        np.testing.assert_allclose(g, r, rtol=1e-3, atol=1e-3 * rms)
    model.close()


def test_draft_exit_at_L_identity_accepts_everything(tiny_bits):
    w = synth.TINY.replace(norm_gain="perturbed", draft_exit_k=4, in_kind=synth.IN_IDENTITY, gamma=4, max_new=20)
    model, _, _ = make_model(w, tiny_bits)
    toks, logits, stats = gpu_decode(model, w, 4)
    assert stats["accept_hist"][:5] == [0, 0, 0, 1, 3]
    ref = run_oracle(w, tiny_bits, 4)
    check_against_oracle(toks, logits, stats, ref, 4)
    model.close()


def test_standalone_draft_and_verify_steps(tiny_model, tiny_bits):
    """ssd_draft / ssd_verify per step == the oracle's drafts, accepts and emitted tokens."""
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=0.05, max_new=1000)
    set_scale(model, w)
    gamma = 4
    ref = run_oracle(w.replace(max_new=26), tiny_bits, gamma)
    _, _, v, p = device_inputs(w)
    model.set_logits_capture(None)
    first = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.prefill(v, p, first)
    d = torch.zeros(gamma, dtype=torch.int32, device="cuda")
    ne = torch.zeros(1, dtype=torch.int32, device="cuda")
    em = torch.zeros(gamma + 1, dtype=torch.int32, device="cuda")
    toks = [int(first.item())]
    for step in range(4):
        model.draft(gamma, d)
        model.verify(gamma, ne, em)
        model.sync()
        n = int(ne.item())
        if toks + em[:n].cpu().tolist() != ref.tokens[: len(toks) + n]:
            break  # streams parted (allowed only at a low-margin position, checked below)
        if d.cpu().tolist()[: ref.accept_lengths[step]] != ref.draft_tokens[step][: ref.accept_lengths[step]]:
            raise AssertionError("accepted drafts differ from the oracle's")
        assert n == ref.accept_lengths[step] + 1
        toks += em[:n].cpu().tolist()
    common_prefix(toks, ref.tokens[: len(toks)], ref.logits)
    assert len(toks) > 4
    assert_accept_sequence(model, ref, toks)


@pytest.mark.parametrize("case", ["ragged_prefill", "vocab_tail", "no_visual", "head128", "head128_short",
                                  "narrow_in", "max_new_1", "max_new_2"])
def test_edge_shapes(case):
    base = synth.TINY.replace(norm_gain="perturbed", s=0.2)
    w = {
        "ragged_prefill": base.replace(n_vis=29, n_prompt=14),                 # P = 43, chunks of 8 + 3
        "vocab_tail": base.replace(shape=synth.ModelShape(4, 256, 4, 64, 1024, 2000)),
        "no_visual": base.replace(n_vis=0, n_prompt=21),
        "head128": base.replace(shape=synth.ModelShape(3, 256, 2, 128, 512, 1024), draft_exit_k=1),
        # 5 prompt rows: the first decode steps see at most one 32-key chunk (CTA 0 finishes the
        # head alone), later ones several (the split-KV merge), within one SSD step too
        "head128_short": base.replace(shape=synth.ModelShape(3, 256, 2, 128, 512, 1024), draft_exit_k=1,
                                      n_vis=0, n_prompt=5),
        "narrow_in": base.replace(in_hidden=192),
        "max_new_1": base.replace(max_new=1),
        "max_new_2": base.replace(max_new=2),
    }[case]
    bits = synth.make_weights(w)
    model, _, _ = make_model(w, bits)
    toks, logits, stats = gpu_decode(model, w, w.gamma)
    ref = run_oracle(w, bits, w.gamma)
    check_against_oracle(toks, logits, stats, ref, w.gamma)
    gtoks, _, _ = gpu_decode(model, w, 0)
    assert toks == gtoks
    model.close()


def test_eos_stops_like_oracle(tiny_bits):
    w0 = synth.TINY.replace(norm_gain="perturbed", s=0.2)
    ref0 = run_oracle(w0, tiny_bits, greedy=True)
    eos = ref0.tokens[6]
    w = w0.replace(eos_id=eos)
    model, _, _ = make_model(w, tiny_bits)
    toks, logits, stats = gpu_decode(model, w, w.gamma)
    ref = run_oracle(w, tiny_bits, w.gamma)
    assert ref.tokens[-1] == eos and len(ref.tokens) < w.max_new
    check_against_oracle(toks, logits, stats, ref, w.gamma)
    model.close()


def test_host_buffer_generate_equals_device_decode(tiny_model):
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=0.2)
    set_scale(model, w)
    toks, _, st = gpu_decode(model, w, 4, capture=False)
    vis, prompt = synth.make_inputs(w)
    htoks, hst = model.generate(vis, prompt, w.max_new, 4)
    assert htoks == toks and hst["accepted"] == st["accepted"]
    gt, _ = model.greedy_generate(vis, prompt, w.max_new)
    assert gt == toks


def test_abi_errors_on_gpu(tiny_bits):
    w = synth.TINY.replace(norm_gain="perturbed")
    model, _, _ = make_model(w, tiny_bits)
    with pytest.raises(lib.SSDError) as e:
        model.verify(4)                                   # no prefill / draft
    assert e.value.status == 5
    with pytest.raises(lib.SSDError) as e:
        model.decode(w.max_new, 4)                        # decode before prefill
    assert e.value.status == 5
    _, _, v, p = device_inputs(w)
    model.prefill(v, p)
    with pytest.raises(lib.SSDError) as e:
        model.decode(w.max_seq(), 4)                      # capacity
    assert e.value.status == 4
    with pytest.raises(lib.SSDError) as e:
        model.draft(9)                                    # gamma > gamma_max
    assert e.value.status == 1
    model.draft(2)
    with pytest.raises(lib.SSDError) as e:
        model.verify(3)                                   # gamma differs from the draft's
    assert e.value.status == 5
    bad = p.clone()
    bad[3] = w.shape.vocab + 5                            # token id out of range -> device error word
    model.prefill(v, bad)
    with pytest.raises(lib.SSDError) as e:
        model.sync()
    assert e.value.status == 7
    model.prefill(v, p)                                   # the context stays usable
    model.decode(w.max_new, 4)
    model.sync()
    model.close()


def test_launch_counts(tiny_model):
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=0.2)
    set_scale(model, w)
    _, _, st = gpu_decode(model, w, 4, capture=False)
    pre, dec = model.launch_counts()
    L, k = w.shape.n_layers, w.draft_exit_k
    body = 4 * (1 + 5 * k + 2 + 1) + (1 + 5 * L + 1 + 1)
    # + decode setup, loop begin and copy-out
    assert dec == 3 + st["steps"] * body
    # prefill: begin + input rows, per layer 4 activation splits + 4 tensor-core GEMMs + the attention's
    # operand split + attention, head + finish
    assert pre == 2 + 10 * L + 2


@pytest.mark.parametrize("rows", [1, 5, 9])
def test_lm_head_op_matches_oracle(tiny_model, tiny_bits, rows):
    """ssd_lm_head: logits of W_lm RMSNorm_f(x) within tolerance, argmax exact away from ties."""
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed")
    m = oracle.model_from_bits(w, tiny_bits, synth.bf16_to_f64)
    x = synth.normal_f64(11, rows, (rows, w.shape.d_model), std=3.0)
    xt = torch.from_numpy(x.astype(np.float32)).cuda()
    tok = torch.zeros(rows, dtype=torch.int32, device="cuda")
    lg = torch.zeros((rows, w.shape.vocab), device="cuda")
    model.lm_head(xt, tok, lg)
    model.sync()
    for r in range(rows):
        ref = oracle.lm_head(m, x[r].astype(np.float32).astype(np.float64))
        assert_logits_close(lg[r].cpu().numpy(), ref, f"lm_head row {r}")
        if int(tok[r]) != int(np.argmax(ref)):
            from tests.parity import margin
            assert margin(ref) < 1e-2
    # argmax of the returned logits is the returned token (lowest index on ties)
    assert tok.cpu().tolist() == lg.argmax(dim=1).cpu().int().tolist()


@pytest.mark.parametrize("case", ["tiny", "ragged"])
def test_tensor_core_prefill_matches_row_prefill_and_oracle(case):
    """The tcgen05 prefill (hi/lo bf16 split, fp32 accumulation) against the row-chunked decode-kernel prefill."""
    w = synth.TINY.replace(norm_gain="perturbed", max_new=2)
    if case == "ragged":
        w = w.replace(n_vis=131, n_prompt=14)              # P = 145: a partial 128-row tile and 64-query block
    bits = synth.make_weights(w)
    caches = []
    for options in (lib.SSD_OPT_PREFILL_ROWS, 0):
        model, _, _ = make_model(w, bits, options=options)
        toks, _, _ = gpu_decode(model, w, 0, capture=False)
        k, v, n = model.kv()
        P = w.prompt_len
        caches.append((k[:, :, :P].clone(), v[:, :, :P].clone(), toks))
        model.close()
    (k1, v1, t1), (k2, v2, t2) = caches
    for a, b in ((k1, k2), (v1, v2)):
        rms = float(a.pow(2).mean().sqrt())
        torch.testing.assert_close(b, a, rtol=1e-4, atol=1e-4 * rms)
    m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    cache = oracle.KVCache(m.cfg, w.max_seq())
    ref_logits = oracle.prefill(m, cache, synth.bf16_to_f64(vis), prompt)
    rms = float(np.sqrt(np.mean(cache.k[:, :, :w.prompt_len] ** 2)))
    np.testing.assert_allclose(k2.cpu().numpy(), cache.k[:, :, :w.prompt_len], rtol=1e-3, atol=1e-3 * rms)
    if t2[0] != int(np.argmax(ref_logits)):
        from tests.parity import margin
        assert margin(ref_logits) < 1e-2


def test_profile_projection_bytes_and_state_recovery(tiny_model):
    """The single-kernel timing entry point reports each kernel's algorithmic bytes, raises no
    device error, and a prefill afterwards restores the decode exactly."""
    model, _ = tiny_model
    w = synth.TINY.replace(norm_gain="perturbed", s=0.2)
    set_scale(model, w)
    before, _, _ = gpu_decode(model, w, 4, capture=False)
    sh = w.shape
    d, qd, ff, V = sh.d_model, sh.n_heads * sh.head_dim, sh.d_ff, sh.vocab
    kv = w.prompt_len
    for rows in (1, 5):
        expect = {
            "qkv": 3 * qd * d * 2 + rows * d * 4 + d * 2 + rows * (qd * 4 + 2 * qd * 2),
            "o": d * qd * 2 + rows * qd * 4 + 2 * rows * d * 4,
            "gateup": 2 * ff * d * 2 + rows * d * 4 + d * 2 + rows * ff * 4,
            "down": d * ff * 2 + rows * ff * 4 + 2 * rows * d * 4,
            "head": V * d * 2 + rows * d * 4 + d * 2 + rows * 4,
            "attn": 2 * (kv + rows) * qd * 4 + 2 * rows * qd * 4,
        }
        if rows == 1:
            h = w.in_hidden
            expect["in1"] = h * d * 2 + d * 4 + d * 2 + h * 4
            expect["in2"] = d * h * 2 + h * 4 + 2 * d * 4
        for name, b in expect.items():
            model.prefill(*device_inputs(w)[2:])
            assert model.profile_projection(name, layer=sh.n_layers - 1, rows=rows, reps=2) == b, (name, rows)
            model.sync()
    with pytest.raises(RuntimeError):  # beyond the GEMV's 16 rows in a ctx without batched verification
        model.profile_projection("in1", rows=17)
    after, _, _ = gpu_decode(model, w, 4, capture=False)
    assert after == before


# --------------------------------------------------------------------------- IN_BLOCK imitation (one decoder block)

@pytest.fixture(scope="module")
def block_bits():
    return synth.make_weights(synth.TINY_BLOCK.replace(norm_gain="perturbed"))


@pytest.fixture(scope="module")
def block_model(block_bits):
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", gamma=8)
    model, _, dev = make_model(w, block_bits, gamma_max=8, max_seq=w.max_seq())
    yield model
    model.close()


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.2, 4), (1.0, 3)])
def test_in_block_imitation_matches_oracle(block_model, block_bits, s, gamma):
    """The imitation module as one decoder block with its own KV cache: tokens, logits, steps, accept
    lengths and kv_len match the oracle; the block's cache rows (prompt rows from the prefill, drafted
    rows, and row gamma from the verification) match the oracle's; SSD equals GPU greedy decoding."""
    model = block_model
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", s=s)
    set_scale(model, w)
    toks, logits, stats = gpu_decode(model, w, gamma)
    m = oracle.model_from_bits(w, block_bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    ref = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, gamma, keep_cache=True,
                              keep_draft_logits=True)
    agree = check_against_oracle(toks, logits, stats, ref, gamma)
    K, V, n = model.kv()
    L = w.shape.n_layers
    upto = min(n, w.prompt_len + agree - 1)
    np.testing.assert_allclose(K[L, :, :upto].cpu().numpy(), ref.cache.k[L, :, :upto], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(V[L, :, :upto].cpu().numpy(), ref.cache.v[L, :, :upto], rtol=2e-3, atol=2e-4)
    gtoks, glogits, _ = gpu_decode(model, w, 0)
    assert toks == gtoks
    np.testing.assert_array_equal(logits, glogits)


def test_in_block_with_dynamic_draft_length_matches_oracle(block_model, block_bits):
    """IN_BLOCK and the dynamic draft length d(t) together: tokens, steps, accept lengths, kv_len."""
    model = block_model
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", s=0.05)
    set_scale(model, w)
    _, _, v, p = device_inputs(w)
    out = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    n = torch.zeros(1, dtype=torch.int32, device="cuda")
    model.set_logits_capture(None)
    model.prefill(v, p)
    model.decode_dynamic(w.max_new, 5, 120, 8, out, n)
    model.sync()
    toks, stats = out[: int(n.item())].cpu().tolist(), model.stats()
    m = oracle.model_from_bits(w, block_bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    ref = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, 8, dynamic=(5, 120))
    assert_accept_sequence(model, ref, toks)
    agree = common_prefix(toks, ref.tokens, ref.logits)
    if agree == len(ref.tokens):
        assert stats["steps"] == len(ref.accept_lengths)
        assert stats["accepted"] == sum(ref.accept_lengths)
        assert stats["kv_len"] == ref.kv_len


def test_in_block_draft_exit_at_last_layer(block_bits):
    """k = L: the block's prompt rows come from the final x_L rows (after the last layer), and the
    verification pass has no deep layers; tokens and stats match the oracle."""
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", s=0.2, draft_exit_k=4, gamma=4)
    model, _, _ = make_model(w, block_bits, gamma_max=4, max_seq=w.max_seq())
    try:
        toks, logits, stats = gpu_decode(model, w, 4)
        m = oracle.model_from_bits(w, block_bits, synth.bf16_to_f64)
        vis, prompt = synth.make_inputs(w)
        ref = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, 4, keep_draft_logits=True)
        check_against_oracle(toks, logits, stats, ref, 4)
    finally:
        model.close()
