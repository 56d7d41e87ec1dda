"""Randomized pins of both oracles over small random shapes (CPU only; hypothesis).

For random layer counts, widths, head layouts, vocabularies, draft exits, gammas and acceptance
scales, with random fp64 weights:
* the decoder-only oracle's prefill and cached decode rows equal the independent torch no-cache
  forward, and SSD (with and without draft-row reuse) equals greedy decoding bitwise;
* the encoder-decoder oracle's cached decode rows equal its independent torch forward, and SSD equals
  greedy decoding bitwise.
A shape-specific indexing mistake (a head stride, a cache slot, a position offset) that the fixed
tiny workloads happen to hide fails one of these.
"""
import numpy as np
import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import given, settings, strategies as st  # noqa: E402

import oracle  # noqa: E402
from oracle import t5_oracle as T  # noqa: E402
from tests.test_oracle import torch_logits_all_rows  # noqa: E402
from tests.test_t5_oracle import torch_forward  # noqa: E402


def _gain(rng, n):
    return rng.normal(1.0, 0.1, n)


@st.composite
def llama_case(draw):
    L = draw(st.integers(1, 3))
    H = draw(st.sampled_from([1, 2, 3]))
    Dh = draw(st.sampled_from([4, 8, 16]))
    d = H * Dh * draw(st.sampled_from([1, 2]))
    return dict(L=L, H=H, Dh=Dh, d=d, ff=draw(st.sampled_from([8, 24, 40])), V=draw(st.sampled_from([16, 37, 64])),
                k=draw(st.integers(1, L)), in_kind=draw(st.sampled_from([oracle.IN_IDENTITY, oracle.IN_MLP2])),
                gamma=draw(st.integers(1, 5)), s=draw(st.sampled_from([0.05, 0.3, 1.0])),
                n_vis=draw(st.integers(0, 5)), n_prompt=draw(st.integers(1, 6)), seed=draw(st.integers(0, 2 ** 20)))


def llama_model(c):
    rng = np.random.default_rng(c["seed"])
    d, q, ff, V = c["d"], c["H"] * c["Dh"], c["ff"], c["V"]
    std = 0.5 / np.sqrt(d)
    layers = [{"wq": rng.normal(0, std, (q, d)), "wk": rng.normal(0, std, (q, d)), "wv": rng.normal(0, std, (q, d)),
               "wo": rng.normal(0, std, (d, q)), "w_gate": rng.normal(0, std, (ff, d)),
               "w_up": rng.normal(0, std, (ff, d)), "w_down": rng.normal(0, 0.5 / np.sqrt(ff), (d, ff)),
               "attn_norm": _gain(rng, d), "ffn_norm": _gain(rng, d)} for _ in range(c["L"])]
    w = {"embed": rng.normal(0, 1, (V, d)), "lm_head": rng.normal(0, std, (V, d)), "final_norm": _gain(rng, d),
         "layers": layers, "in_norm": _gain(rng, d), "in_w1": rng.normal(0, std, (d, d)),
         "in_w2": rng.normal(0, std, (d, d))}
    cfg = oracle.OracleConfig(n_layers=c["L"], d_model=d, n_heads=c["H"], head_dim=c["Dh"], d_ff=ff, vocab=V,
                              draft_exit_k=c["k"], in_kind=c["in_kind"])
    scale = np.ones(c["L"])
    scale[c["k"]:] = c["s"]
    m = oracle.Model(cfg, w, scale, c["s"])
    vis = rng.normal(0, 1, (c["n_vis"], d))
    prompt = rng.integers(0, V, c["n_prompt"])
    return m, vis, prompt


@settings(max_examples=25, deadline=None)
@given(llama_case())
def test_decoder_oracle_random_shapes(c):
    m, vis, prompt = llama_model(c)
    max_new = 8
    g = oracle.greedy_generate(m, vis, prompt, max_new)
    ref = torch_logits_all_rows(m, vis, list(prompt) + g.tokens[:-1])
    P = vis.shape[0] + len(prompt)
    np.testing.assert_allclose(np.stack(g.logits), ref[P - 1:], rtol=1e-9, atol=1e-9)
    for reuse in (True, False):
        r = oracle.ssd_generate(m, vis, prompt, max_new, c["gamma"], reuse_draft_rows=reuse)
        assert r.tokens == g.tokens
        for a, b in zip(r.logits, g.logits):
            np.testing.assert_array_equal(a, b)
        assert all(0 <= a <= c["gamma"] for a in r.accept_lengths)
        assert r.kv_len == g.kv_len


@st.composite
def t5_case(draw):
    H = draw(st.sampled_from([1, 2]))
    Dh = draw(st.sampled_from([4, 8]))
    n_dec = draw(st.integers(1, 3))
    return dict(n_enc=draw(st.integers(1, 2)), n_dec=n_dec, H=H, Dh=Dh, d=H * Dh * draw(st.sampled_from([1, 2])),
                ff=draw(st.sampled_from([8, 24])), V=draw(st.sampled_from([16, 41])), k=draw(st.integers(1, n_dec)),
                in_kind=draw(st.sampled_from([T.IN_IDENTITY, T.IN_MLP2])), gamma=draw(st.integers(1, 4)),
                s=draw(st.sampled_from([0.05, 0.3, 1.0])), buckets=draw(st.sampled_from([8, 32])),
                maxd=draw(st.sampled_from([20, 128])), n_q=draw(st.integers(1, 6)), n_p=draw(st.integers(0, 5)),
                seed=draw(st.integers(0, 2 ** 20)))


def t5_model(c):
    rng = np.random.default_rng(c["seed"])
    d, q, ff, V, H = c["d"], c["H"] * c["Dh"], c["ff"], c["V"], c["H"]
    std = 0.5 / np.sqrt(d)

    def lin(o, i, s=std):
        return rng.normal(0, s, (o, i))

    enc = [{"attn_norm": _gain(rng, d), "wq": lin(q, d), "wk": lin(q, d), "wv": lin(q, d), "wo": lin(d, q),
            "ffn_norm": _gain(rng, d), "wi0": lin(ff, d), "wi1": lin(ff, d), "wff": lin(d, ff)} for _ in range(c["n_enc"])]
    dec = [{"self_norm": _gain(rng, d), "wq": lin(q, d), "wk": lin(q, d), "wv": lin(q, d), "wo": lin(d, q),
            "cross_norm": _gain(rng, d), "cq": lin(q, d), "ck": lin(q, d), "cv": lin(q, d), "co": lin(d, q),
            "ffn_norm": _gain(rng, d), "wi0": lin(ff, d), "wi1": lin(ff, d), "wff": lin(d, ff)} for _ in range(c["n_dec"])]
    w = {"embed": rng.normal(0, 1, (V, d)), "lm_head": lin(V, d), "enc_final": _gain(rng, d),
         "dec_final": _gain(rng, d), "enc_rel": rng.normal(0, 0.5, (c["buckets"], H)),
         "dec_rel": rng.normal(0, 0.5, (c["buckets"], H)), "enc": enc, "dec": dec,
         "in_norm": _gain(rng, d), "in_w1": lin(d, d), "in_w2": lin(d, d)}
    cfg = T.T5Config(n_enc=c["n_enc"], n_dec=c["n_dec"], d_model=d, n_heads=H, head_dim=c["Dh"], d_ff=ff, vocab=V,
                     draft_exit_k=c["k"], in_kind=c["in_kind"], rel_buckets=c["buckets"], rel_max_distance=c["maxd"])
    scale = np.ones(c["n_dec"])
    scale[c["k"]:] = c["s"]
    m = T.T5Model(cfg, w, scale, c["s"])
    return m, rng.normal(0, 1, (c["n_q"], d)), rng.integers(0, V, c["n_p"])


@settings(max_examples=25, deadline=None)
@given(t5_case())
def test_encoder_decoder_oracle_random_shapes(c):
    m, z, prompt = t5_model(c)
    # the torch forward buckets by the 32-bucket / 128-distance threshold tables only
    max_new = 8
    g = T.greedy_generate(m, z, prompt, max_new)
    if c["buckets"] == 32 and c["maxd"] == 128:
        ref = torch_forward(m, z, prompt, g.tokens[:-1])
        np.testing.assert_allclose(np.stack(g.logits), ref, rtol=1e-9, atol=1e-9)
    r = T.ssd_generate(m, z, prompt, max_new, c["gamma"])
    assert r.tokens == g.tokens
    for a, b in zip(r.logits, g.logits):
        np.testing.assert_array_equal(a, b)
    assert all(0 <= a <= c["gamma"] for a in r.accept_lengths)
    assert r.kv_len == g.kv_len
