"""Pins of the fp64 oracle against things other than itself (CPU only).

* library routines: torch's rms_norm, scaled_dot_product_attention and silu,
  and complex multiplication for the rotary embedding, assembled into an
  independent no-cache forward of the whole decoder;
* closed forms: one-key attention, RoPE at position 0, norm preservation,
  relative-position property, RMSNorm output scale;
* Algorithm 1's defining properties: SSD output == greedy output (bitwise
  here), accepted length <= gamma + 1 per step, k = L with the identity
  imitation network accepts every draft, gamma = 1 degenerates correctly,
  and the cache after rollback equals the greedy cache;
* brute force: the cached decode equals recomputing the whole sequence.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import synth


# --------------------------------------------------------------------------- fixtures

def build(w, bits=None):
    bits = bits or synth.make_weights(w)
    m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(w)
    return m, synth.bf16_to_f64(vis), prompt


@pytest.fixture(scope="module")
def tiny_bits():
    return synth.make_weights(synth.TINY.replace(norm_gain="perturbed"))


def tiny(s=1.0, **kw):
    return synth.TINY.replace(norm_gain="perturbed", s=s, **kw)


# --------------------------------------------------------------------------- independent torch forward

def torch_logits_all_rows(m: oracle.Model, vis: np.ndarray, tokens) -> np.ndarray:
    """No-cache forward of rows [z; embed(tokens)] built from torch library routines (fp64)."""
    c, W = m.cfg, m.w
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    H, Dh = c.n_heads, c.head_dim
    X = torch.cat([t(vis), t(W["embed"])[torch.as_tensor(np.asarray(tokens, dtype=np.int64))]], 0)
    P = X.shape[0]
    half = Dh // 2
    inv = c.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / Dh)
    rot = torch.polar(torch.ones(P, half, dtype=torch.float64), torch.arange(P, dtype=torch.float64)[:, None] * inv)

    def rope_c(Z):                               # Z [P][H][Dh]; pair (i, i+half) as a complex number
        z = torch.complex(Z[..., :half], Z[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], -1)

    for l in range(c.n_layers):
        lw = {k: t(v) for k, v in W["layers"][l].items()}
        N = F.rms_norm(X, (c.d_model,), lw["attn_norm"], c.rms_eps)
        Q = rope_c((N @ lw["wq"].T).view(P, H, Dh)).transpose(0, 1)
        K = rope_c((N @ lw["wk"].T).view(P, H, Dh)).transpose(0, 1)
        V = (N @ lw["wv"].T).view(P, H, Dh).transpose(0, 1)
        O = F.scaled_dot_product_attention(Q[None], K[None], V[None], is_causal=True)[0]
        X = X + m.s[l] * (O.transpose(0, 1).reshape(P, H * Dh) @ lw["wo"].T)
        U = F.rms_norm(X, (c.d_model,), lw["ffn_norm"], c.rms_eps)
        X = X + m.s[l] * ((F.silu(U @ lw["w_gate"].T) * (U @ lw["w_up"].T)) @ lw["w_down"].T)
    Xn = F.rms_norm(X, (c.d_model,), t(W["final_norm"]), c.rms_eps)
    return (Xn @ t(W["lm_head"]).T).numpy()


def test_prefill_matches_torch_library_forward(tiny_bits):
    w = tiny()
    m, vis, prompt = build(w, tiny_bits)
    ref = torch_logits_all_rows(m, vis, prompt)
    cache = oracle.KVCache(m.cfg, w.max_seq())
    got = oracle.prefill(m, cache, vis, prompt)
    np.testing.assert_allclose(got, ref[-1], rtol=1e-10, atol=1e-10)


@pytest.mark.parametrize("s", [0.2, 1.0])
def test_cached_greedy_decode_matches_no_cache_recompute(tiny_bits, s):
    """Brute force: every decode step's logits == recomputing the whole sequence from scratch."""
    w = tiny(s=s)
    m, vis, prompt = build(w, tiny_bits)
    r = oracle.greedy_generate(m, vis, prompt, max_new=8)
    ref = torch_logits_all_rows(m, vis, list(prompt) + r.tokens[:-1])
    P = w.prompt_len
    for t in range(8):
        np.testing.assert_allclose(r.logits[t], ref[P - 1 + t], rtol=1e-9, atol=1e-9)
        assert r.tokens[t] == int(np.argmax(ref[P - 1 + t]))


def test_imitation_network_matches_torch(tiny_bits):
    w = tiny(s=0.7)
    m, _, _ = build(w, tiny_bits)
    x = synth.normal_f64(3, 3, (w.shape.d_model,))
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    n = F.rms_norm(t(x), (w.shape.d_model,), t(m.w["in_norm"]), w.shape.rms_eps)
    ref = t(x) + m.s_in * (t(m.w["in_w2"]) @ F.silu(t(m.w["in_w1"]) @ n))
    np.testing.assert_allclose(oracle.imitation(m, x), ref.numpy(), rtol=1e-12, atol=1e-12)


def torch_xk_rows(m: oracle.Model, vis: np.ndarray, tokens, k: int) -> torch.Tensor:
    """No-cache torch forward of rows [z; embed(tokens)] through layers 0..k-1: x_k of every row."""
    c, W = m.cfg, m.w
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    H, Dh, half = c.n_heads, c.head_dim, c.head_dim // 2
    X = torch.cat([t(vis), t(W["embed"])[torch.as_tensor(np.asarray(tokens, dtype=np.int64))]], 0)
    P = X.shape[0]
    inv = c.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / Dh)
    rot = torch.polar(torch.ones(P, half, dtype=torch.float64), torch.arange(P, dtype=torch.float64)[:, None] * inv)

    def rope_c(Z):
        z = torch.complex(Z[..., :half], Z[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], -1)

    for l in range(k):
        lw = {n: t(v) for n, v in W["layers"][l].items()}
        N = F.rms_norm(X, (c.d_model,), lw["attn_norm"], c.rms_eps)
        Q = rope_c((N @ lw["wq"].T).view(P, H, Dh)).transpose(0, 1)
        K = rope_c((N @ lw["wk"].T).view(P, H, Dh)).transpose(0, 1)
        V = (N @ lw["wv"].T).view(P, H, Dh).transpose(0, 1)
        O = F.scaled_dot_product_attention(Q[None], K[None], V[None], is_causal=True)[0]
        X = X + m.s[l] * (O.transpose(0, 1).reshape(P, H * Dh) @ lw["wo"].T)
        U = F.rms_norm(X, (c.d_model,), lw["ffn_norm"], c.rms_eps)
        X = X + m.s[l] * ((F.silu(U @ lw["w_gate"].T) * (U @ lw["w_up"].T)) @ lw["w_down"].T)
    return X


def mlp2_draft_path_error(m: oracle.Model, vis: np.ndarray, prompt, max_new: int, gamma: int) -> tuple[float, int]:
    """Runs ssd_generate and compares every draft row g(I(x_k)) of every step with a no-cache torch
    forward of the sequence as it stands at that step (the emitted tokens, then the step's own
    drafts) through layers 0..k-1, the MLP2 imitation and the head.  Returns the largest absolute
    difference relative to the row's scale, and the number of rows compared."""
    c = m.cfg
    r = oracle.ssd_generate(m, vis, prompt, max_new, gamma, keep_draft_logits=True)
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    n_vis, emitted, worst, rows = vis.shape[0], 1, 0.0, 0
    for step, (drafts, dlog) in enumerate(zip(r.draft_tokens, r.draft_logits)):
        seq = list(prompt) + r.tokens[:emitted] + list(drafts[:-1])
        X = torch_xk_rows(m, vis, seq, c.draft_exit_k)
        row0 = n_vis + len(prompt) + emitted - 1          # the last emitted token's row
        for j in range(len(drafts)):
            x = X[row0 + j]
            n = F.rms_norm(x, (c.d_model,), t(m.w["in_norm"]), c.rms_eps)
            xi = x + m.s_in * (t(m.w["in_w2"]) @ F.silu(t(m.w["in_w1"]) @ n))
            ref = (t(m.w["lm_head"]) @ F.rms_norm(xi, (c.d_model,), t(m.w["final_norm"]), c.rms_eps)).numpy()
            worst = max(worst, float(np.max(np.abs(dlog[j] - ref)) / max(1.0, float(np.max(np.abs(ref))))))
            assert drafts[j] == int(np.argmax(dlog[j]))
            rows += 1
        emitted += r.accept_lengths[step] + 1
    return worst, rows


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.2, 3)])
def test_mlp2_draft_logits_match_torch_no_cache_forward(tiny_bits, s, gamma):
    """Every draft row of every SSD step, g(I(x_k)) with the MLP2 imitation at k < L, equals a no-cache
    torch forward of the sequence at that step: the cached shallow layers, the row and position each
    draft reads, and the rollback of rejected drafts' cache rows all show up in it.  (SSD == greedy
    cannot see a wrong draft: drafts only change how many tokens a step accepts.)"""
    w = tiny(s=s, gamma=gamma, max_new=14)
    m, vis, prompt = build(w, tiny_bits)
    assert m.cfg.draft_exit_k < m.cfg.n_layers
    err, rows = mlp2_draft_path_error(m, vis, prompt, w.max_new, gamma)
    assert rows >= 12 and err < 1e-9, (err, rows)


# --------------------------------------------------------------------------- closed forms

def test_rope_position_zero_is_identity_and_norm_preserving():
    v = synth.normal_f64(1, 1, (4, 64))
    np.testing.assert_array_equal(oracle.rope(v, 0, 10000.0), v)
    r = oracle.rope(v, 37, 10000.0)
    np.testing.assert_allclose(np.linalg.norm(r, axis=-1), np.linalg.norm(v, axis=-1), rtol=1e-13)


def test_rope_relative_position_property():
    q = synth.normal_f64(1, 2, (1, 64))
    k = synth.normal_f64(1, 3, (1, 64))
    d = lambda m_, n_: float(np.sum(oracle.rope(q, m_, 1e4) * oracle.rope(k, n_, 1e4)))
    assert d(10, 3) == pytest.approx(d(107, 100), rel=1e-10)
    assert d(5, 5) == pytest.approx(float(np.sum(q * k)), rel=1e-10)


def test_rope_hand_values():
    # head_dim 4: angles pos * 10000^0 and pos * 10000^-0.5 = pos / 100.
    v = np.array([[1.0, 2.0, 3.0, 4.0]])
    got = oracle.rope(v, 2, 10000.0)[0]
    a0, a1 = 2.0, 0.02
    want = [1 * math.cos(a0) - 3 * math.sin(a0), 2 * math.cos(a1) - 4 * math.sin(a1),
            1 * math.sin(a0) + 3 * math.cos(a0), 2 * math.sin(a1) + 4 * math.cos(a1)]
    np.testing.assert_allclose(got, want, rtol=1e-14)


def test_rms_norm_scale_and_invariance():
    x = synth.normal_f64(2, 1, (3, 256), std=5.0)
    y = oracle.rms_norm(x, np.ones(256), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=-1)), 1.0, rtol=1e-13)
    np.testing.assert_allclose(oracle.rms_norm(7.0 * x, np.ones(256), 0.0), y, rtol=1e-12)


def test_silu_closed_form():
    assert oracle.silu(np.array(0.0)) == 0.0
    assert oracle.silu(np.array(1.0)) == pytest.approx(1.0 / (1.0 + math.exp(-1.0)), rel=1e-15)
    assert oracle.silu(np.array(-40.0)) == pytest.approx(-40.0 * math.exp(-40.0), rel=1e-9)


def _one_layer_model(d=8, H=2, Dh=4, ff=8, V=16):
    cfg = oracle.OracleConfig(n_layers=1, d_model=d, n_heads=H, head_dim=Dh, d_ff=ff, vocab=V,
                              draft_exit_k=1)
    g = lambda st, shp: synth.normal_f64(9, st, shp, std=0.5)
    lw = {"wq": g(1, (H * Dh, d)), "wk": g(2, (H * Dh, d)), "wv": g(3, (H * Dh, d)),
          "wo": g(4, (d, H * Dh)), "w_gate": g(5, (ff, d)), "w_up": g(6, (ff, d)),
          "w_down": g(7, (d, ff)), "attn_norm": np.ones(d), "ffn_norm": np.ones(d)}
    W = {"embed": g(8, (V, d)), "lm_head": g(10, (V, d)), "final_norm": np.ones(d), "layers": [lw]}
    return oracle.Model(cfg, W, [1.0], 0.0), lw


def test_attention_with_one_key_returns_its_value():
    m, lw = _one_layer_model()
    cache = oracle.KVCache(m.cfg, 4)
    x = synth.normal_f64(4, 4, (8,))
    out = oracle.layer_row(m, 0, x, 0, cache)
    n = oracle.rms_norm(x, np.ones(8), m.cfg.rms_eps)
    h = x + lw["wo"] @ (lw["wv"] @ n)                 # softmax over one key == 1
    u = oracle.rms_norm(h, np.ones(8), m.cfg.rms_eps)
    want = h + lw["w_down"] @ (oracle.silu(lw["w_gate"] @ u) * (lw["w_up"] @ u))
    np.testing.assert_allclose(out, want, rtol=1e-13, atol=1e-13)


def test_causal_mask_ignores_future_cache_rows():
    m, _ = _one_layer_model()
    x = synth.normal_f64(5, 5, (8,))
    c1, c2 = oracle.KVCache(m.cfg, 8), oracle.KVCache(m.cfg, 8)
    c2.k[:, :, 3:] = 1e3                              # garbage beyond the row's position
    c2.v[:, :, 3:] = -1e3
    for p in range(3):
        c1.k[:, :, p] = c2.k[:, :, p] = synth.normal_f64(6, p, (2, 4))
        c1.v[:, :, p] = c2.v[:, :, p] = synth.normal_f64(7, p, (2, 4))
    np.testing.assert_array_equal(oracle.layer_row(m, 0, x, 3, c1), oracle.layer_row(m, 0, x, 3, c2))


def test_argmax_matches_full_sort_and_ties_go_low():
    v = synth.normal_f64(8, 8, (2048,))
    assert oracle.argmax_lowest(v) == int(np.argsort(-v, kind="stable")[0])
    t = np.zeros(10)
    t[[3, 7]] = 2.0
    assert oracle.argmax_lowest(t) == 3


def test_imitation_identity_cases(tiny_bits):
    x = synth.normal_f64(3, 4, (256,))
    m0, _, _ = build(tiny(s=0.0), tiny_bits)
    np.testing.assert_array_equal(oracle.imitation(m0, x), x)          # s_in = 0
    mi, _, _ = build(tiny(in_kind=synth.IN_IDENTITY), tiny_bits)
    np.testing.assert_array_equal(oracle.imitation(mi, x), x)          # draft w/o imitation


# --------------------------------------------------------------------------- Algorithm 1 properties

@pytest.mark.parametrize("s,gamma,k", [(0.05, 4, 2), (0.2, 4, 2), (1.0, 4, 2), (0.2, 3, 1), (0.05, 8, 3)])
def test_ssd_equals_greedy(tiny_bits, s, gamma, k):
    w = tiny(s=s, gamma=gamma, draft_exit_k=k)
    m, vis, prompt = build(w, tiny_bits)
    g = oracle.greedy_generate(m, vis, prompt, w.max_new, max_seq=w.max_seq(), keep_cache=True)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, gamma, keep_cache=True)
    assert r.tokens == g.tokens
    assert all(np.array_equal(a, b) for a, b in zip(r.logits, g.logits))
    assert len(r.tokens) == w.max_new
    # per step: 1 <= a + 1 <= gamma + 1 and the counts add up to the tokens after the first
    assert all(0 <= a <= gamma for a in r.accept_lengths)
    assert sum(a + 1 for a in r.accept_lengths) == w.max_new - 1
    assert r.kv_lens[-1] == r.kv_len == w.prompt_len + w.max_new - 1 == g.kv_len
    assert np.all(np.diff([w.prompt_len] + r.kv_lens) == np.array(r.accept_lengths) + 1)
    # rollback by length: the valid cache equals the greedy run's cache bitwise
    n = r.kv_len
    np.testing.assert_array_equal(r.cache.k[:, :, :n], g.cache.k[:, :, :n])
    np.testing.assert_array_equal(r.cache.v[:, :, :n], g.cache.v[:, :, :n])


def test_draft_exit_at_L_with_identity_accepts_everything(tiny_bits):
    w = tiny(s=1.0, draft_exit_k=4, in_kind=synth.IN_IDENTITY, gamma=4, max_new=20)
    m, vis, prompt = build(w, tiny_bits)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, w.gamma)
    assert r.accept_lengths == [4, 4, 4, 3]       # gamma_eff = min(gamma, remaining - 1)
    assert r.tokens == oracle.greedy_generate(m, vis, prompt, w.max_new).tokens


def test_gamma_one_degenerates(tiny_bits):
    w = tiny(s=0.2, gamma=1)
    m, vis, prompt = build(w, tiny_bits)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, 1)
    assert set(r.accept_lengths) <= {0, 1}
    assert r.tokens == oracle.greedy_generate(m, vis, prompt, w.max_new).tokens


def test_reuse_of_draft_rows_equals_recompute(tiny_bits):
    """Shared-KV reuse of the shallow rows (option B) == recomputing them (option A), bitwise."""
    w = tiny(s=0.2)
    m, vis, prompt = build(w, tiny_bits)
    a = oracle.ssd_generate(m, vis, prompt, w.max_new, w.gamma, reuse_draft_rows=True, keep_cache=True)
    b = oracle.ssd_generate(m, vis, prompt, w.max_new, w.gamma, reuse_draft_rows=False, keep_cache=True)
    assert a.tokens == b.tokens and a.accept_lengths == b.accept_lengths
    np.testing.assert_array_equal(a.cache.k[:, :, :a.kv_len], b.cache.k[:, :, :a.kv_len])


def test_eos_stops_generation(tiny_bits):
    w = tiny(s=0.2)
    m, vis, prompt = build(w, tiny_bits)
    g = oracle.greedy_generate(m, vis, prompt, w.max_new)
    eos = g.tokens[5]
    first = g.tokens.index(eos)
    m.cfg.eos_id = eos
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, w.gamma)
    ge = oracle.greedy_generate(m, vis, prompt, w.max_new)
    assert r.tokens == ge.tokens == g.tokens[:first + 1]


def test_draft_mismatch_is_replaced_by_full_model_token(tiny_bits):
    """Every step emits the accepted drafts then f_a; f_a differs from the rejected draft."""
    w = tiny(s=0.2)
    m, vis, prompt = build(w, tiny_bits)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, w.gamma)
    pos = 1
    for a, drafts in zip(r.accept_lengths, r.draft_tokens):
        emitted = r.tokens[pos:pos + a + 1]
        assert emitted[:a] == drafts[:a]
        if a < len(drafts):
            assert emitted[a] != drafts[a]
        pos += a + 1


def test_prefill_rows_equal_sequential_decode(tiny_bits):
    """Prefill's causal sequence pass == feeding the same rows one at a time through the cache."""
    w = tiny(s=1.0)
    m, vis, prompt = build(w, tiny_bits)
    c1 = oracle.KVCache(m.cfg, 64)
    o1 = oracle.prefill(m, c1, vis, prompt)
    c2 = oracle.KVCache(m.cfg, 64)
    rows = list(vis) + [oracle.embed(m, t) for t in prompt]
    for p, x in enumerate(rows):
        x = oracle.forward_row(m, x, p, c2, range(m.cfg.n_layers))
    np.testing.assert_allclose(oracle.lm_head(m, x), o1, rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(c2.k[:, :, :len(rows)], c1.k[:, :, :len(rows)], rtol=1e-10, atol=1e-12)


# --------------------------------------------------------------------------- dynamic draft length d(t)

def test_draft_length_closed_form_pins():
    """Sec. "Choice of d": d(t) = d0 + floor(10 sigmoid(0.01 (t - N/2))).  Pinned by the sigmoid's
    inverse: 10 sigmoid(z) = k exactly at z = ln(k / (10 - k)), so d steps from d0 + k - 1 to d0 + k
    between t = floor and ceil of N/2 + 100 ln(k / (10 - k))."""
    for d0, n_max in [(5, 1000), (5, 4096), (3, 777)]:
        assert oracle.draft_length(n_max // 2, d0, n_max) == d0 + 5 if n_max % 2 == 0 else True
        for k in range(1, 10):
            tk = n_max / 2 + 100.0 * math.log(k / (10 - k))
            lo, hi = math.floor(tk), math.ceil(tk)
            if lo == hi or lo < 0:
                continue
            assert oracle.draft_length(lo, d0, n_max) == d0 + k - 1, (d0, n_max, k)
            assert oracle.draft_length(hi, d0, n_max) == d0 + k, (d0, n_max, k)
        ds = [oracle.draft_length(t, d0, n_max) for t in range(0, 4 * n_max)]
        assert all(b >= a for a, b in zip(ds, ds[1:]))          # non-decreasing in t
        assert min(ds) >= d0 and max(ds) <= d0 + 10
    assert oracle.draft_length(0, 5, 4096) == 5                  # sigmoid(-20.48) * 10 < 1
    assert oracle.draft_length(10**6, 5, 4096) == 15             # sigmoid rounds to 1 in fp64


@pytest.mark.parametrize("s,cap,n_max", [(0.05, 8, 120), (0.2, 6, 90), (1.0, 8, 40)])
def test_ssd_dynamic_draft_length_equals_greedy(tiny_bits, s, cap, n_max):
    w = tiny(s=s, gamma=cap)
    m, vis, prompt = build(w, tiny_bits)
    g = oracle.greedy_generate(m, vis, prompt, w.max_new)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, cap, dynamic=(5, n_max))
    assert r.tokens == g.tokens
    # per step: gamma_t = min(d(kv_len + 2), cap, remaining - 1) drafts, 0 <= a <= gamma_t
    p, n = w.prompt_len, 1
    for drafts, a, kv in zip(r.draft_tokens, r.accept_lengths, r.kv_lens):
        g_t = min(oracle.draft_length(p + 2, 5, n_max), cap, w.max_new - n - 1)
        assert len(drafts) == g_t and 0 <= a <= g_t
        p, n = kv, n + a + 1
    assert p == r.kv_len == g.kv_len


@pytest.mark.parametrize("s,n_max", [(0.05, 32), (0.2, 200)])
def test_ssd_dynamic_draft_length_over_generated_tokens(tiny_bits, s, n_max):
    """The other reading of t: the index of the next new token.  Per step the schedule follows the
    count of emitted tokens (not the cache length), so the first step drafts d(2) whatever the
    prompt's length; with N = 200 over 32 tokens the drafts grow with t; SSD still equals greedy."""
    cap = 15
    w = tiny(s=s, gamma=cap)
    m, vis, prompt = build(w, tiny_bits)
    g = oracle.greedy_generate(m, vis, prompt, w.max_new)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, cap, dynamic=(5, n_max, "generated"))
    assert r.tokens == g.tokens
    n = 1
    for drafts, a in zip(r.draft_tokens, r.accept_lengths):
        t = n + 1                                                 # the next new token's index
        g_t = min(oracle.draft_length(t, 5, n_max), cap, w.max_new - n - 1)
        assert len(drafts) == g_t and 0 <= a <= g_t
        n += a + 1
    assert len(r.draft_tokens[0]) == min(oracle.draft_length(2, 5, n_max), cap)
    if n_max == 200:  # d(t) = 5 + floor(10 sigmoid(0.01 (t - 100))): 7 at t = 2, 8 from t = 16 on
        assert oracle.draft_length(2, 5, 200) == 7 and oracle.draft_length(16, 5, 200) == 8
        assert len(r.draft_tokens[0]) == 7


# --------------------------------------------------------------------------- IN_BLOCK imitation (one decoder block)

def torch_block_rows(m: oracle.Model, vis: np.ndarray, tokens):
    """No-cache torch forward of rows [z; embed(tokens)] through layers 0..k-1 (x_k of every row),
    then the imitation block applied causally over those rows: returns (X_k, block K, block V,
    block output) in fp64."""
    c, W = m.cfg, m.w
    t = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    H, Dh, half = c.n_heads, c.head_dim, c.head_dim // 2
    X = torch.cat([t(vis), t(W["embed"])[torch.as_tensor(np.asarray(tokens, dtype=np.int64))]], 0)
    P = X.shape[0]
    inv = c.rope_theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / Dh)
    rot = torch.polar(torch.ones(P, half, dtype=torch.float64), torch.arange(P, dtype=torch.float64)[:, None] * inv)

    def rope_c(Z):
        z = torch.complex(Z[..., :half], Z[..., half:]) * rot[:, None, :]
        return torch.cat([z.real, z.imag], -1)

    def block(X, lw, s):
        N = F.rms_norm(X, (c.d_model,), lw["attn_norm"], c.rms_eps)
        Q = rope_c((N @ lw["wq"].T).view(P, H, Dh))
        K = rope_c((N @ lw["wk"].T).view(P, H, Dh))
        V = (N @ lw["wv"].T).view(P, H, Dh)
        O = F.scaled_dot_product_attention(Q.transpose(0, 1)[None], K.transpose(0, 1)[None], V.transpose(0, 1)[None],
                                           is_causal=True)[0]
        Y = X + s * (O.transpose(0, 1).reshape(P, H * Dh) @ lw["wo"].T)
        U = F.rms_norm(Y, (c.d_model,), lw["ffn_norm"], c.rms_eps)
        return Y + s * ((F.silu(U @ lw["w_gate"].T) * (U @ lw["w_up"].T)) @ lw["w_down"].T), K, V

    for l in range(c.draft_exit_k):
        X, _, _ = block(X, {k: t(v) for k, v in W["layers"][l].items()}, m.s[l])
    out, K, V = block(X, {k: t(v) for k, v in W["in_block"].items()}, m.s_in)
    return X.numpy(), K.numpy(), V.numpy(), out.numpy()


def test_in_block_first_draft_matches_torch_no_cache_forward():
    """The first draft token's logits g(I(x_k)) with I one decoder block over its own cache (filled by
    the prefill for the prompt rows) equal a no-cache torch forward of the whole sequence."""
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", s=0.2, max_new=3)
    m, vis, prompt = build(w)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, 2, keep_draft_logits=True)
    y = r.tokens[0]
    _, _, _, out = torch_block_rows(m, vis, list(prompt) + [y])
    ref = m.w["lm_head"] @ oracle.rms_norm(out[-1], m.w["final_norm"], m.cfg.rms_eps)
    np.testing.assert_allclose(r.draft_logits[0][0], ref, rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("s,gamma,k", [(0.05, 4, 2), (0.2, 4, 2), (1.0, 3, 1), (0.05, 6, 4)])
def test_in_block_ssd_equals_greedy_and_block_cache_matches(s, gamma, k):
    """SSD with the block imitation equals greedy decoding; afterwards the block's cache rows at
    every position below kv_len hold the block K/V of that token's x_k (no-cache torch forward):
    prompt rows from the prefill, drafted rows from the drafts, row gamma from the verification."""
    w = synth.TINY_BLOCK.replace(norm_gain="perturbed", s=s, gamma=gamma, draft_exit_k=k)
    m, vis, prompt = build(w)
    g = oracle.greedy_generate(m, vis, prompt, w.max_new)
    r = oracle.ssd_generate(m, vis, prompt, w.max_new, gamma, keep_cache=True)
    assert r.tokens == g.tokens
    _, K, V, _ = torch_block_rows(m, vis, list(prompt) + r.tokens[:-1])
    n = r.kv_len
    L = m.cfg.n_layers
    np.testing.assert_allclose(r.cache.k[L, :, :n], K.transpose(1, 0, 2)[:, :n], rtol=1e-9, atol=1e-9)
    np.testing.assert_allclose(r.cache.v[L, :, :n], V.transpose(1, 0, 2)[:, :n], rtol=1e-9, atol=1e-9)


# --------------------------------------------------------------------------- batch of ragged requests

def test_batch_prompt_lengths_are_ragged_and_in_range():
    for bw in (synth.LLAVA13B_B16, synth.TINY_B4):
        n = bw.prompt_lengths()
        assert len(n) == bw.batch and n.min() >= bw.prompt_min and n.max() <= bw.prompt_max
        assert len(set(n.tolist())) > 1
    ins = synth.make_batch_inputs(synth.TINY_B4)
    assert [len(p) for _, p in ins] == synth.TINY_B4.prompt_lengths().tolist()
    assert not np.array_equal(ins[0][0], ins[1][0])      # every request has its own visual rows


@pytest.mark.parametrize("s,gamma", [(0.05, 4), (0.3, 6), (1.0, 2)])
def test_batch_ssd_equals_each_request_alone_and_greedy(tiny_bits, s, gamma):
    """Lockstep batching changes no request's result: tokens, logits, accept lengths and kv_len equal
    ssd_generate on the request alone and its greedy decoding; positions start at the request's own P;
    the batch runs as many steps as its slowest request, each request's rows summing its gamma_eff + 1."""
    bw = synth.TINY_B4.replace(base=tiny(s=s, gamma=gamma, max_new=20))
    m, _, _ = build(bw.base, tiny_bits)
    reqs = [(synth.bf16_to_f64(v), p) for v, p in synth.make_batch_inputs(bw)]
    br = oracle.ssd_generate_batch(m, reqs, bw.base.max_new, gamma)
    assert len(br.results) == bw.batch
    for b, ((vis, prompt), r) in enumerate(zip(reqs, br.results)):
        alone = oracle.ssd_generate(m, vis, prompt, bw.base.max_new, gamma)
        greedy = oracle.greedy_generate(m, vis, prompt, bw.base.max_new)
        assert r.tokens == alone.tokens == greedy.tokens
        assert r.accept_lengths == alone.accept_lengths and r.kv_lens == alone.kv_lens
        for a, g in zip(r.logits, greedy.logits):
            np.testing.assert_array_equal(a, g)
        P = vis.shape[0] + len(prompt)
        assert r.kv_lens[0] == P + r.accept_lengths[0] + 1 and r.kv_len == P + bw.base.max_new - 1
        assert sum(1 for act in br.active if b in act) == len(r.accept_lengths)
    assert len(br.active) == max(len(r.accept_lengths) for r in br.results)
    # rows per batched step: each active request's drafted tokens + 1
    for t, act in enumerate(br.active):
        drafted = sum(len(br.results[b].draft_tokens[sum(1 for u in br.active[:t] if b in u)]) for b in act)
        assert br.rows[t] == drafted + len(act)
