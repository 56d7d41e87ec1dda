"""Pins of the encoder-decoder (FlanT5-shaped) fp64 oracle against things other than itself (CPU only).

* closed forms: the relative-position buckets' boundaries are the geometric thresholds
  exact * (max_distance / exact) ** (j / (n - exact)), rounded up, written out below by hand;
* library routines: torch's rms_norm, gelu (tanh form), scaled_dot_product_attention with scale 1
  and an additive bias mask, and a bucket lookup by torch.bucketize over those thresholds (not the
  oracle's logarithm), assembled into an independent no-cache forward of encoder and decoder;
* Algorithm 1's defining properties on the decoder: SSD output == greedy output (bitwise here),
  accepted length <= gamma per step, k = L with the identity imitation network accepts every draft,
  gamma = 1 degenerates correctly;
* planted mistakes (a dropped bias, a 1/sqrt(d) factor, the erf GELU, un-normed encoder output,
  bidirectional buckets in the decoder) must fail the torch comparison.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import t5_oracle as T

# Bucket thresholds for 32 buckets, max_distance 128, derived by hand:
# bidirectional: 16 buckets a side, 8 exact, then 8 log buckets with ratio 16 ** (1/8) = sqrt(2):
#   ceil(8 * sqrt(2) ** j), j = 0..7 -> 8, 12, 16, 23, 32, 46, 64, 91
# past-only: 32 buckets, 16 exact, then 16 log buckets with ratio 8 ** (1/16):
#   ceil(16 * 8 ** (j / 16)), j = 0..15
BIDIR_LOG_START = [8, 12, 16, 23, 32, 46, 64, 91]
CAUSAL_LOG_START = [16, 19, 21, 24, 27, 31, 35, 40, 46, 52, 59, 67, 77, 87, 99, 113]


def test_relative_bucket_thresholds_closed_form():
    for j, d in enumerate(BIDIR_LOG_START):
        assert d == math.ceil(8 * 2 ** (j / 2) - 1e-9)
    for j, d in enumerate(CAUSAL_LOG_START):
        assert d == math.ceil(16 * 8 ** (j / 16) - 1e-9)


def _bucket_by_table(delta: int, bidirectional: bool) -> int:
    if bidirectional:
        base, dist, exact, starts = (16 if delta > 0 else 0), abs(delta), 8, BIDIR_LOG_START
    else:
        base, dist, exact, starts = 0, max(-delta, 0), 16, CAUSAL_LOG_START
    if dist < exact:
        return base + dist
    return base + exact + max(j for j, s in enumerate(starts) if dist >= s)


@pytest.mark.parametrize("bidirectional", [True, False])
def test_relative_bucket_matches_threshold_table(bidirectional):
    for delta in range(-400, 401):
        assert T.rel_bucket(delta, bidirectional, 32, 128) == _bucket_by_table(delta, bidirectional), delta


def test_relative_bucket_special_values():
    assert T.rel_bucket(0, True, 32, 128) == 0
    assert T.rel_bucket(3, True, 32, 128) == 19          # later key: upper half
    assert T.rel_bucket(-3, True, 32, 128) == 3
    assert T.rel_bucket(10 ** 6, True, 32, 128) == 31    # far future shares the last bucket
    assert T.rel_bucket(-(10 ** 6), False, 32, 128) == 31
    assert T.rel_bucket(5, False, 32, 128) == 0          # decoder: later keys share bucket 0 (masked)


# --------------------------------------------------------------------------- independent torch forward

def build(w: synth.T5Workload):
    bits = synth.make_t5_weights(w)
    m = T.model_from_bits(w, bits, synth.bf16_to_f64)
    q, prompt = synth.make_t5_inputs(w)
    return m, synth.bf16_to_f64(q), prompt


def tiny(**kw):
    return synth.T5_TINY.replace(norm_gain="perturbed", **kw)


def _torch_bias(table: torch.Tensor, n_q: int, n_k: int, bidirectional: bool) -> torch.Tensor:
    """[H][n_q][n_k] bias with buckets from torch.bucketize over the threshold tables."""
    delta = torch.arange(n_k)[None, :] - torch.arange(n_q)[:, None]
    if bidirectional:
        dist, base, exact, starts = delta.abs(), (delta > 0).long() * 16, 8, BIDIR_LOG_START
    else:
        dist, base, exact, starts = (-delta).clamp(min=0), torch.zeros_like(delta), 16, CAUSAL_LOG_START
    far = exact + torch.bucketize(dist, torch.tensor(starts), right=True) - 1
    bucket = base + torch.where(dist < exact, dist, far)
    return table[bucket].permute(2, 0, 1)


def torch_forward(m: T.T5Model, z: np.ndarray, prompt, dec_tokens, n_dec: int | None = None):
    """Logits of every decoder row for decoder inputs [start; dec_tokens] (no cache); with n_dec, the
    hidden rows after decoder layers 0..n_dec-1 instead."""
    c, W = m.cfg, m.w
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    H, Dh, d = c.n_heads, c.head_dim, c.d_model

    def heads(Y):
        return Y.view(Y.shape[0], H, Dh).transpose(0, 1)[None]

    def mlp(lw, X):
        U = F.rms_norm(X, (d,), lw["ffn_norm"], c.eps)
        return (F.gelu(U @ lw["wi0"].T, approximate="tanh") * (U @ lw["wi1"].T)) @ lw["wff"].T

    X = torch.cat([t(z), t(W["embed"])[torch.as_tensor(np.asarray(prompt, dtype=np.int64))]], 0)
    P = X.shape[0]
    eb = _torch_bias(t(W["enc_rel"]), P, P, True)[None]
    for l in range(c.n_enc):
        lw = {k: t(v) for k, v in W["enc"][l].items()}
        N = F.rms_norm(X, (d,), lw["attn_norm"], c.eps)
        O = F.scaled_dot_product_attention(heads(N @ lw["wq"].T), heads(N @ lw["wk"].T), heads(N @ lw["wv"].T),
                                           attn_mask=eb, scale=1.0)[0]
        X = X + O.transpose(0, 1).reshape(P, H * Dh) @ lw["wo"].T
        X = X + mlp(lw, X)
    E = F.rms_norm(X, (d,), t(W["enc_final"]), c.eps)

    ids = torch.as_tensor([c.start_token] + list(dec_tokens), dtype=torch.int64)
    Y = t(W["embed"])[ids]
    S = Y.shape[0]
    causal = torch.triu(torch.full((S, S), float("-inf"), dtype=torch.float64), 1)
    db = (_torch_bias(t(W["dec_rel"]), S, S, False) + causal)[None]
    for l in range(c.n_dec if n_dec is None else n_dec):
        lw = {k: t(v) for k, v in W["dec"][l].items()}
        s = m.s[l]
        N = F.rms_norm(Y, (d,), lw["self_norm"], c.eps)
        O = F.scaled_dot_product_attention(heads(N @ lw["wq"].T), heads(N @ lw["wk"].T), heads(N @ lw["wv"].T),
                                           attn_mask=db, scale=1.0)[0]
        Y = Y + s * (O.transpose(0, 1).reshape(S, H * Dh) @ lw["wo"].T)
        N = F.rms_norm(Y, (d,), lw["cross_norm"], c.eps)
        O = F.scaled_dot_product_attention(heads(N @ lw["cq"].T), heads(E @ lw["ck"].T), heads(E @ lw["cv"].T),
                                           scale=1.0)[0]
        Y = Y + s * (O.transpose(0, 1).reshape(S, H * Dh) @ lw["co"].T)
        Y = Y + s * mlp(lw, Y)
    if n_dec is not None:
        return Y
    Yn = F.rms_norm(Y, (d,), t(W["dec_final"]), c.eps)
    return (Yn @ t(W["lm_head"]).T).numpy()


@pytest.fixture(scope="module")
def tiny_model():
    return build(tiny())


def test_greedy_logits_match_torch_no_cache_forward(tiny_model):
    m, z, prompt = tiny_model
    r = T.greedy_generate(m, z, prompt, 12)
    ref = torch_forward(m, z, prompt, r.tokens[:-1])
    np.testing.assert_allclose(np.stack(r.logits), ref, rtol=1e-9, atol=1e-9)
    assert r.tokens == [int(np.argmax(row)) for row in ref]


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.3, 3)])
def test_draft_tokens_match_torch_no_cache_forward(s, gamma):
    """Every drafted token of every SSD step is the argmax of g(I(x_k)) for x_k from a no-cache torch
    forward through decoder layers 0..k-1 of the sequence at that step (the emitted tokens, then the
    step's own drafts), the MLP2 imitation and the head: the draft path's cache rows, positions and
    rollback, which SSD == greedy cannot see.  Rows whose top two logits are within 1e-9 are skipped."""
    w = tiny(s=s, max_new=16)
    m, z, prompt = build(w)
    c = m.cfg
    assert 0 < c.draft_exit_k < c.n_dec
    r = T.ssd_generate(m, z, prompt, w.max_new, gamma)
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    p, checked = 1, 0
    for step, drafts in enumerate(r.draft_tokens):
        Y = torch_forward(m, z, prompt, r.tokens[:p] + list(drafts[:-1]), n_dec=c.draft_exit_k)
        for j, d in enumerate(drafts):
            x = Y[p + j]
            n = F.rms_norm(x, (c.d_model,), t(m.w["in_norm"]), c.eps)
            xi = x + m.s_in * (t(m.w["in_w2"]) @ F.silu(t(m.w["in_w1"]) @ n))
            o = (t(m.w["lm_head"]) @ F.rms_norm(xi, (c.d_model,), t(m.w["dec_final"]), c.eps)).numpy()
            top = np.sort(o)[-2:]
            if top[1] - top[0] > 1e-9:
                assert d == int(np.argmax(o)), (step, j)
                checked += 1
        p = r.kv_lens[step]
    assert checked >= 8


def test_encoder_is_bidirectional_and_decoder_causal(tiny_model):
    """Changing the last prompt id changes every encoder row (no mask); changing a later decoder
    input leaves the earlier decoder rows' logits unchanged."""
    m, z, prompt = tiny_model
    e0 = T.encode(m, z, prompt)
    p2 = np.array(prompt).copy()
    p2[-1] = (p2[-1] + 1) % m.cfg.vocab
    e1 = T.encode(m, z, p2)
    assert np.all(np.abs(e0 - e1).max(axis=1) > 0)
    a = torch_forward(m, z, prompt, [5, 6, 7])
    b = torch_forward(m, z, prompt, [5, 6, 8])
    np.testing.assert_array_equal(a[:3], b[:3])
    assert not np.array_equal(a[3], b[3])


# --------------------------------------------------------------------------- Algorithm 1 properties

@pytest.mark.parametrize("s", [0.05, 0.3, 1.0])
@pytest.mark.parametrize("gamma", [1, 2, 4, 6])
def test_ssd_equals_greedy(s, gamma):
    w = tiny(s=s, gamma=gamma)
    m, z, prompt = build(w)
    g = T.greedy_generate(m, z, prompt, w.max_new)
    r = T.ssd_generate(m, z, prompt, w.max_new, gamma)
    assert r.tokens == g.tokens
    for a, b in zip(r.logits, g.logits):
        np.testing.assert_array_equal(a, b)
    assert all(0 <= a <= gamma for a in r.accept_lengths)
    assert r.kv_len == g.kv_len == len(r.tokens)
    steps = np.cumsum([a + 1 for a in r.accept_lengths])
    assert list(1 + steps) == r.kv_lens


def test_ssd_without_draft_row_reuse_equals_greedy():
    w = tiny(s=0.3)
    m, z, prompt = build(w)
    assert T.ssd_generate(m, z, prompt, w.max_new, 4, reuse_draft_rows=False).tokens == \
        T.greedy_generate(m, z, prompt, w.max_new).tokens


def test_draft_exit_at_last_layer_accepts_everything():
    w = tiny(in_kind=synth.IN_IDENTITY, draft_exit_k=synth.T5_TINY.shape.n_dec)
    m, z, prompt = build(w)
    r = T.ssd_generate(m, z, prompt, w.max_new, 4)
    assert r.accept_lengths[:-1] == [4] * (len(r.accept_lengths) - 1)
    assert r.tokens == T.greedy_generate(m, z, prompt, w.max_new).tokens


def test_acceptance_knob_orders_accept_length():
    mean = []
    for s in (0.02, 1.0):
        w = tiny(s=s)
        m, z, prompt = build(w)
        mean.append(np.mean(T.ssd_generate(m, z, prompt, w.max_new, 4).accept_lengths))
    assert mean[0] > mean[1]


# --------------------------------------------------------------------------- planted mistakes

def _no_rel_bias(m, table, n_q, n_k, bidirectional, q0=0):
    return np.zeros((m.cfg.n_heads, n_q, n_k))


def _gelu_erf(x):
    return 0.5 * x * (1.0 + np.vectorize(math.erf)(x / math.sqrt(2.0)))


def _bucket_bidir_everywhere(delta, bidirectional, n, maxd, _orig=T.rel_bucket):
    return _orig(delta, True, n, maxd)


def _scaled_softmax(x, _orig=T.softmax):
    return _orig(x / 8.0)


def _encode_unnormed(m, z, prompt, _orig=T.encode):
    e = _orig(m, z, prompt)
    return e * 1.5


MUTATIONS = {
    "encoder_rel_bias_dropped": ("bias_table", _no_rel_bias),
    "gelu_erf_form": ("gelu_tanh", _gelu_erf),
    "decoder_bidirectional_buckets": ("rel_bucket", _bucket_bidir_everywhere),
    "attention_scaled_by_rsqrt_dh": ("softmax", _scaled_softmax),
    "encoder_output_scale": ("encode", _encode_unnormed),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_torch_forward_catches(monkeypatch, name, tiny_model):
    attr, fn = MUTATIONS[name]
    m, z, prompt = tiny_model
    toks = [3, 1, 4, 1, 5, 9, 2, 6, 5, 3, 5, 8, 9, 7, 9, 3, 2, 3, 8, 4]
    ref = torch_forward(m, z, prompt, toks)
    monkeypatch.setattr(T, attr, fn)
    cache = T.DecCache(m, T.encode(m, z, prompt), len(toks) + 1)
    got = []
    for pos, y in enumerate([m.cfg.start_token] + toks):
        got.append(T.lm_head(m, T.dec_forward_row(m, m.w["embed"][y].copy(), pos, cache, range(m.cfg.n_dec))))
    assert not np.allclose(np.stack(got), ref, rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("s,cap,n_max", [(0.05, 8, 60), (0.3, 6, 200)])
def test_ssd_dynamic_draft_length_equals_greedy(s, cap, n_max):
    """Sec. "Choice of d" on the decoder: each step drafts min(d(kv_len + 2), cap, remaining - 1) tokens
    and the output is still greedy decoding."""
    w = tiny(s=s, max_new=40)
    m, z, prompt = build(w)
    r = T.ssd_generate(m, z, prompt, w.max_new, cap, dynamic=(5, n_max))
    assert r.tokens == T.greedy_generate(m, z, prompt, w.max_new).tokens
    p, n = 1, 1
    for step, a in enumerate(r.accept_lengths):
        g = min(cap, 5 + int(np.floor(10.0 / (1.0 + np.exp(-0.01 * ((p + 2) - n_max / 2.0))))), w.max_new - n - 1)
        assert len(r.draft_tokens[step]) == g and 0 <= a <= g
        p += a + 1
        n += a + 1


def test_draft_pin_catches_an_imitation_without_residual(monkeypatch):
    """Planted on the CPU: SSD == greedy still holds with a broken imitation network (verification
    corrects every draft), the draft-token pin does not."""
    def no_residual(m, x):
        n = T.rms_norm(x, m.w["in_norm"], m.cfg.eps)
        return m.s_in * (m.w["in_w2"] @ T.silu(m.w["in_w1"] @ n))
    w = tiny(s=0.05, max_new=16)
    m, z, prompt = build(w)
    g = T.greedy_generate(m, z, prompt, w.max_new)
    monkeypatch.setattr(T, "imitation", no_residual)
    assert T.ssd_generate(m, z, prompt, w.max_new, 4).tokens == g.tokens
    with pytest.raises(AssertionError):
        test_draft_tokens_match_torch_no_cache_forward(0.05, 4)
