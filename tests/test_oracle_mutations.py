"""Planted mistakes in the oracle (on the CPU) must be caught by its pins.

Each case monkeypatches one oracle building block with a plausible bug (a
wrong sign, a dropped term, an off-by-one, a transposed operand, a skipped
cache write, a shared cache, a missing norm) and checks that the independent
torch forward or an Algorithm 1 property disagrees.
"""
import numpy as np
import pytest

import oracle
import oracle.ssd_oracle as so
import synth
from tests.test_oracle import build, mlp2_draft_path_error, tiny, torch_logits_all_rows


def _rope_wrong_sign(v, pos, theta):
    half = v.shape[-1] // 2
    ang = so.rope_angles(pos, v.shape[-1], theta)
    c, s = np.cos(ang), np.sin(ang)
    a, b = v[..., :half], v[..., half:]
    return np.concatenate([a * c + b * s, -a * s + b * c], axis=-1)


def _rms_no_gain(x, gain, eps):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def _silu_wrong(x):
    return x / (1.0 + np.exp(x))


def _head_no_norm(m, x):
    return m.w["lm_head"] @ x


MUTATIONS = {
    "rope_sign": ("rope", _rope_wrong_sign),
    "rmsnorm_gain_dropped": ("rms_norm", _rms_no_gain),
    "silu_sign": ("silu", _silu_wrong),
    "final_norm_dropped": ("lm_head", _head_no_norm),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_torch_forward_catches(monkeypatch, name):
    attr, fn = MUTATIONS[name]
    w = tiny(s=1.0)
    m, vis, prompt = build(w)
    ref = torch_logits_all_rows(m, vis, prompt)[-1]
    monkeypatch.setattr(so, attr, fn)
    got = so.prefill(m, so.KVCache(m.cfg, w.max_seq()), vis, prompt)
    assert not np.allclose(got, ref, rtol=1e-6, atol=1e-6)


def test_decode_position_off_by_one_is_caught(monkeypatch):
    w = tiny(s=1.0)
    m, vis, prompt = build(w)
    orig = so.layer_row
    monkeypatch.setattr(so, "layer_row", lambda m_, l, x, pos, c: orig(m_, l, x, pos + (pos > 40), c))
    r = so.greedy_generate(m, vis, prompt, max_new=4)
    ref = torch_logits_all_rows(m, vis, list(prompt) + r.tokens[:-1])
    assert not np.allclose(r.logits[1], ref[w.prompt_len], rtol=1e-6, atol=1e-6)


def test_accept_rule_off_by_one_is_caught(monkeypatch):
    """Accepting one draft too many breaks SSD == greedy."""
    w = tiny(s=0.2)
    m, vis, prompt = build(w)
    g = so.greedy_generate(m, vis, prompt, w.max_new)
    orig_argmax = so.argmax_lowest
    calls = {"n": 0}

    def lying_argmax(v):            # every 7th verify decision returns a wrong token
        calls["n"] += 1
        t = orig_argmax(v)
        return (t + 1) % len(v) if calls["n"] % 7 == 0 else t
    monkeypatch.setattr(so, "argmax_lowest", lying_argmax)
    r = so.ssd_generate(m, vis, prompt, w.max_new, w.gamma)
    assert r.tokens != g.tokens


# --------------------------------------------------------------------------- newer features

def test_in_block_catch_up_row_skipped_is_caught(monkeypatch):
    """Dropping the verification pass's catch-up (the block's cache row of d_gamma's x_k) leaves stale
    block rows that the no-cache torch forward of the block exposes."""
    from tests.test_oracle import torch_block_rows
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", s=1.0, gamma=4)
    m, vis, prompt = build(w)
    monkeypatch.setattr(so, "block_kv", lambda *a, **k: None)
    r = so.ssd_generate(m, vis, prompt, w.max_new, w.gamma, keep_cache=True)
    _, K, _, _ = torch_block_rows(m, vis, list(prompt) + r.tokens[:-1])
    n, L = r.kv_len, m.cfg.n_layers
    assert not np.allclose(r.cache.k[L, :, :n], K.transpose(1, 0, 2)[:, :n], rtol=1e-6, atol=1e-6)


def test_batch_sharing_one_cache_is_caught(monkeypatch):
    """Requests that share one KV cache (a missing per-request cache) no longer reproduce their runs alone."""
    w = tiny(s=0.3, max_new=12)
    m, _, _ = build(w)
    bw = synth.TINY_B4.replace(base=w)
    reqs = [(synth.bf16_to_f64(v), p) for v, p in synth.make_batch_inputs(bw)]
    alone = [so.ssd_generate(m, v, p, w.max_new, w.gamma) for v, p in reqs]
    shared = so.KVCache(m.cfg, bw.max_seq())
    monkeypatch.setattr(so, "KVCache", lambda cfg, max_seq: shared)
    br = so.ssd_generate_batch(m, reqs, w.max_new, w.gamma)
    assert any(b.logits[-1].tolist() != a.logits[-1].tolist() for a, b in zip(alone, br.results))


def test_encoder_decoder_cross_cache_from_unnormed_output_is_caught(monkeypatch):
    """Cross-attention K/V taken from the encoder's residual stream instead of its normed output fails
    the torch forward."""
    from oracle import t5_oracle as T
    from tests.test_t5_oracle import build as t5_build, tiny as t5_tiny, torch_forward
    m, z, prompt = t5_build(t5_tiny())
    toks = [5, 9, 2, 6, 5, 3]
    ref = torch_forward(m, z, prompt, toks)
    orig = T.rms_norm

    def skip_final_norm(x, gain, eps):       # the encoder's final norm is its last rms_norm call on [P][d]
        if x.ndim == 2 and gain is m.w["enc_final"]:
            return x
        return orig(x, gain, eps)
    monkeypatch.setattr(T, "rms_norm", skip_final_norm)
    cache = T.DecCache(m, T.encode(m, z, prompt), len(toks) + 1)
    got = [T.lm_head(m, T.dec_forward_row(m, m.w["embed"][y].copy(), pos, cache, range(m.cfg.n_dec)))
           for pos, y in enumerate([m.cfg.start_token] + toks)]
    assert not np.allclose(np.stack(got), ref, rtol=1e-6, atol=1e-6)


def _imitation_no_residual(m, x, *rest):
    n = so.rms_norm(x, m.w["in_norm"], m.cfg.rms_eps)
    return m.s_in * (m.w["in_w2"] @ so.silu(m.w["in_w1"] @ n))


def test_draft_path_mistake_passes_ssd_equals_greedy_but_not_the_draft_pin(monkeypatch):
    """An imitation network without its residual still gives SSD == greedy (the verification corrects
    every draft), so only the draft-path pin can catch it."""
    w = tiny(s=0.05, gamma=4, max_new=14)
    m, vis, prompt = build(w)
    g = so.greedy_generate(m, vis, prompt, w.max_new)
    err, _ = mlp2_draft_path_error(m, vis, prompt, w.max_new, w.gamma)
    assert err < 1e-9
    monkeypatch.setattr(so, "imitation", _imitation_no_residual)
    assert so.ssd_generate(m, vis, prompt, w.max_new, w.gamma).tokens == g.tokens
    err, _ = mlp2_draft_path_error(m, vis, prompt, w.max_new, w.gamma)
    assert err > 1e-3
