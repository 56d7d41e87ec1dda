"""Planted mistakes in the oracle (on the CPU) must be caught by its pins.

Each case monkeypatches one oracle building block with a plausible bug (a
wrong sign, a dropped term, an off-by-one, a transposed operand) and checks
that the independent torch forward or an Algorithm 1 property disagrees.
"""
import numpy as np
import pytest

import oracle
import oracle.ssd_oracle as so
import synth
from tests.test_oracle import build, tiny, torch_logits_all_rows


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
