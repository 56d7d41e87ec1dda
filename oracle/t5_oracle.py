"""Plain fp64 CPU oracle for greedy self-speculative decoding on an encoder-decoder VLM
(the BLIP-2 + FlanT5-xl setting of Sec. "Experiments"; FastVLM, arXiv 2510.22641).

TEST INFRASTRUCTURE ONLY.  Only ``tests/`` and the ``cpu_baseline`` leg of ``bench.py --encdec``
may import or run this module.  It shares no code with any CUDA path; its inputs come from
``synth`` (seeded generators).

What it computes:

* Sec. "SSD Setup for VLMs": the encoder output z = E(I, T0) feeds the decoder; only the
  decoder decodes autoregressively.  In the BLIP-2 setting the language model is itself an
  encoder-decoder: the query embeddings z (from the image-grounded query generator) and the
  prompt's token embeddings form the input rows of its encoder; its decoder generates.
* The language model has the T5 v1.1 form of FlanT5: pre-norm blocks with RMSNorm
  (eps 1e-6, gain only), no biases, attention logits without the 1/sqrt(head_dim) factor plus
  a learned relative-position bias (bucketed key-minus-query offsets; bidirectional buckets in
  the encoder, past-only buckets in the decoder's self-attention; one bias table per stack,
  used by every layer of that stack), a gated-GELU MLP wo (gelu(wi0 u) * wi1 u) with the tanh
  form of GELU, cross-attention from every decoder layer to the encoder's normed output
  (no bias, no mask), final norms on both stacks and an untied LM head.
* Algorithm 1 on the decoder: the draft is decoder layers 0..k-1 plus the imitation network
  (x + s_in W2 SiLU(W1 RMSNorm(x)), Sec. "Methodology") and the shared LM head; the
  verification runs the whole decoder over the gamma+1 rows; acceptance, bonus token and
  rollback by length as in the decoder-only oracle.  The decoder starts from its start token
  (id 0) at position 0; its first output is the first new token.
* The acceptance knob: s_l scales both residual writes (self-attention + cross-attention count
  as the attention part, and the MLP) of decoder layers k..L-1, s_in the imitation network's.

Decode rows go one at a time through the same function, so SSD and greedy decoding agree
bitwise here.
"""
from __future__ import annotations

import dataclasses
import math
import time

import numpy as np

from .ssd_oracle import draft_length

IN_IDENTITY = 0
IN_MLP2 = 1


@dataclasses.dataclass(frozen=True)
class T5Config:
    n_enc: int
    n_dec: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    draft_exit_k: int
    in_kind: int = IN_MLP2
    eps: float = 1e-6
    rel_buckets: int = 32
    rel_max_distance: int = 128
    start_token: int = 0
    eos_id: int = -1


class T5Model:
    """fp64 weights ([out][in] layouts) and scales.

    enc[l] = {attn_norm, wq, wk, wv, wo, ffn_norm, wi0, wi1, wff}
    dec[l] = {self_norm, wq, wk, wv, wo, cross_norm, cq, ck, cv, co, ffn_norm, wi0, wi1, wff}
    enc_rel [buckets][H], dec_rel [buckets][H], enc_final, dec_final [d], embed [V][d],
    lm_head [V][d], in_norm / in_w1 / in_w2 (IN_MLP2).
    """

    def __init__(self, cfg: T5Config, w: dict, dec_scale, in_scale: float):
        if cfg.rel_buckets < 4 or cfg.rel_buckets % 2 or cfg.rel_max_distance <= cfg.rel_buckets // 2:
            raise ValueError("rel_buckets must be even and >= 4, rel_max_distance > rel_buckets / 2")
        self.cfg = cfg
        self.w = w
        self.s = [float(v) for v in dec_scale]
        self.s_in = float(in_scale)


# --------------------------------------------------------------------------- building blocks

def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * gain


def gelu_tanh(x: np.ndarray) -> np.ndarray:
    """0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def softmax(x: np.ndarray) -> np.ndarray:
    e = np.exp(x - np.max(x, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def argmax_lowest(v: np.ndarray) -> int:
    return int(np.flatnonzero(v == np.max(v))[0])


def rel_bucket(delta: int, bidirectional: bool, n_buckets: int, max_distance: int) -> int:
    """Bucket of the key-minus-query offset ``delta``.

    Bidirectional: half the buckets for keys before the query (and the query itself), half for
    keys after it.  Past-only: every bucket is for keys at or before the query (later keys share
    bucket 0; the decoder masks them anyway).  Within a half, offsets below n/2 get one bucket
    each and larger offsets share logarithmically spaced buckets up to max_distance, beyond which
    they share the last one.  The logarithmic index is evaluated in fp64 and floored after adding
    1e-9: at exact powers (offset 16 of the bidirectional half, for one) the exact index is an integer
    that fp64 rounding could otherwise put one bucket short, and the guard makes the decision
    independent of the platform's log.
    """
    n = n_buckets
    base = 0
    if bidirectional:
        n //= 2
        if delta > 0:
            base = n
        dist = abs(delta)
    else:
        dist = max(-delta, 0)
    exact = n // 2
    if dist < exact:
        return base + dist
    far = exact + int(math.log(dist / exact) / math.log(max_distance / exact) * (n - exact) + 1e-9)
    return base + min(far, n - 1)


def bias_table(m: T5Model, table: np.ndarray, n_q: int, n_k: int, bidirectional: bool, q0: int = 0) -> np.ndarray:
    """[H][n_q][n_k] additive logits bias for queries at positions q0 .. q0+n_q-1 and keys 0 .. n_k-1."""
    c = m.cfg
    b = np.empty((c.n_heads, n_q, n_k))
    for i in range(n_q):
        for j in range(n_k):
            b[:, i, j] = table[rel_bucket(j - (q0 + i), bidirectional, c.rel_buckets, c.rel_max_distance)]
    return b


def ffn(m: T5Model, lw: dict, x: np.ndarray) -> np.ndarray:
    """wo (gelu(wi0 u) * wi1 u) with u = RMSNorm(x); x is one row [d] or rows [n][d]."""
    u = rms_norm(x, lw["ffn_norm"], m.cfg.eps)
    return (gelu_tanh(u @ lw["wi0"].T) * (u @ lw["wi1"].T)) @ lw["wff"].T


# --------------------------------------------------------------------------- encoder

def encode(m: T5Model, z: np.ndarray, prompt) -> np.ndarray:
    """Encoder over the rows [z; embed(prompt)]: bidirectional self-attention with the encoder's
    relative-position bias; returns the normed output [P][d]."""
    c, w = m.cfg, m.w
    H, Dh = c.n_heads, c.head_dim
    X = np.concatenate([z, w["embed"][np.asarray(prompt, dtype=np.int64)]], axis=0)
    P = X.shape[0]
    bias = bias_table(m, w["enc_rel"], P, P, True)
    for l in range(c.n_enc):
        lw = w["enc"][l]
        N = rms_norm(X, lw["attn_norm"], c.eps)
        Q = (N @ lw["wq"].T).reshape(P, H, Dh).transpose(1, 0, 2)
        K = (N @ lw["wk"].T).reshape(P, H, Dh).transpose(1, 0, 2)
        V = (N @ lw["wv"].T).reshape(P, H, Dh).transpose(1, 0, 2)
        S = np.matmul(Q, K.transpose(0, 2, 1)) + bias          # no 1/sqrt(Dh)
        O = np.matmul(softmax(S), V).transpose(1, 0, 2).reshape(P, H * Dh)
        X = X + O @ lw["wo"].T
        X = X + ffn(m, lw, X)
    return rms_norm(X, w["enc_final"], c.eps)


class DecCache:
    """Decoder self-attention K/V [n_dec][H][S_max][Dh] and cross-attention K/V [n_dec][H][P][Dh]."""

    def __init__(self, m: T5Model, enc: np.ndarray, max_seq: int):
        c, w = m.cfg, m.w
        H, Dh, P = c.n_heads, c.head_dim, enc.shape[0]
        self.k = np.zeros((c.n_dec, H, max_seq, Dh))
        self.v = np.zeros((c.n_dec, H, max_seq, Dh))
        self.ck = np.stack([(enc @ w["dec"][l]["ck"].T).reshape(P, H, Dh).transpose(1, 0, 2) for l in range(c.n_dec)])
        self.cv = np.stack([(enc @ w["dec"][l]["cv"].T).reshape(P, H, Dh).transpose(1, 0, 2) for l in range(c.n_dec)])


def dec_layer_row(m: T5Model, l: int, x: np.ndarray, pos: int, cache: DecCache) -> np.ndarray:
    """Decoder layer l on one row at position ``pos``: self-attention over positions 0..pos
    (writes K/V[l][:, pos]) with the decoder's past-only bias, cross-attention, gated-GELU MLP."""
    c, w = m.cfg, m.w
    lw, s = w["dec"][l], m.s[l]
    H, Dh = c.n_heads, c.head_dim
    n = rms_norm(x, lw["self_norm"], c.eps)
    q = (lw["wq"] @ n).reshape(H, Dh)
    cache.k[l, :, pos] = (lw["wk"] @ n).reshape(H, Dh)
    cache.v[l, :, pos] = (lw["wv"] @ n).reshape(H, Dh)
    bias = np.stack([w["dec_rel"][rel_bucket(j - pos, False, c.rel_buckets, c.rel_max_distance)]
                     for j in range(pos + 1)], axis=1)                  # [H][pos+1]
    sc = np.einsum("hd,hjd->hj", q, cache.k[l, :, :pos + 1]) + bias
    o = np.einsum("hj,hjd->hd", softmax(sc), cache.v[l, :, :pos + 1]).reshape(H * Dh)
    x = x + s * (lw["wo"] @ o)
    n = rms_norm(x, lw["cross_norm"], c.eps)
    q = (lw["cq"] @ n).reshape(H, Dh)
    sc = np.einsum("hd,hjd->hj", q, cache.ck[l])
    o = np.einsum("hj,hjd->hd", softmax(sc), cache.cv[l]).reshape(H * Dh)
    x = x + s * (lw["co"] @ o)
    return x + s * ffn(m, lw, x)


def dec_forward_row(m: T5Model, x: np.ndarray, pos: int, cache: DecCache, layers) -> np.ndarray:
    for l in layers:
        x = dec_layer_row(m, l, x, pos, cache)
    return x


def lm_head(m: T5Model, x: np.ndarray) -> np.ndarray:
    return m.w["lm_head"] @ rms_norm(x, m.w["dec_final"], m.cfg.eps)


def imitation(m: T5Model, x: np.ndarray) -> np.ndarray:
    if m.cfg.in_kind == IN_IDENTITY:
        return x
    n = rms_norm(x, m.w["in_norm"], m.cfg.eps)
    return x + m.s_in * (m.w["in_w2"] @ silu(m.w["in_w1"] @ n))


# --------------------------------------------------------------------------- decoding loops

@dataclasses.dataclass
class T5Result:
    tokens: list
    logits: list
    kv_len: int
    accept_lengths: list = dataclasses.field(default_factory=list)
    kv_lens: list = dataclasses.field(default_factory=list)
    draft_tokens: list = dataclasses.field(default_factory=list)
    prefill_s: float = 0.0                                  # wall time of the encoder + first decoder step
    step_s: list = dataclasses.field(default_factory=list)  # wall time per SSD step


def _first(m: T5Model, z, prompt, max_seq: int):
    enc = encode(m, z, prompt)
    cache = DecCache(m, enc, max_seq)
    x = dec_forward_row(m, m.w["embed"][m.cfg.start_token].copy(), 0, cache, range(m.cfg.n_dec))
    o = lm_head(m, x)
    return cache, o


def greedy_generate(m: T5Model, z: np.ndarray, prompt, max_new: int) -> T5Result:
    """Plain greedy decoding with the whole decoder (the definition SSD must reproduce)."""
    c = m.cfg
    cache, o = _first(m, z, prompt, max_new + 1)
    y = argmax_lowest(o)
    res = T5Result(tokens=[y], logits=[o], kv_len=1)
    while len(res.tokens) < max_new and not (c.eos_id >= 0 and y == c.eos_id):
        p = res.kv_len
        x = dec_forward_row(m, m.w["embed"][y].copy(), p, cache, range(c.n_dec))
        o = lm_head(m, x)
        y = argmax_lowest(o)
        res.tokens.append(y)
        res.logits.append(o)
        res.kv_len = p + 1
    return res


def ssd_generate(m: T5Model, z: np.ndarray, prompt, max_new: int, gamma: int,
                 reuse_draft_rows: bool = True, max_steps: int | None = None,
                 dynamic: tuple[int, int] | None = None) -> T5Result:
    """Algorithm 1 on the decoder (see the module docstring); kv_len counts decoder positions.
    max_steps: stop after that many draft + verify steps (a sampled prefix of a long run).
    dynamic = (d0, N): each step drafts min(d(t), gamma, remaining - 1) tokens with t = kv_len + 2
    (Sec. "Choice of d", the decoder-only oracle's draft_length); gamma is then the cap."""
    c = m.cfg
    k, L = c.draft_exit_k, c.n_dec
    t0 = time.perf_counter()
    cache, o = _first(m, z, prompt, max_new + gamma + 1)
    y = argmax_lowest(o)
    res = T5Result(tokens=[y], logits=[o], kv_len=1, prefill_s=time.perf_counter() - t0)
    p, done = 1, (c.eos_id >= 0 and y == c.eos_id)
    while len(res.tokens) < max_new and not done and (max_steps is None or len(res.accept_lengths) < max_steps):
        t0 = time.perf_counter()
        g_step = gamma if dynamic is None else min(gamma, draft_length(p + 2, dynamic[0], dynamic[1]))
        g_eff = min(g_step, max_new - len(res.tokens) - 1)
        toks, xk = [y], []
        for j in range(g_eff):                                   # drafting stage
            x = dec_forward_row(m, m.w["embed"][toks[j]].copy(), p + j, cache, range(k))
            xk.append(x)
            toks.append(argmax_lowest(lm_head(m, imitation(m, x))))
        f, flog = [], []
        for i in range(g_eff + 1):                               # verification stage
            x = xk[i] if (reuse_draft_rows and i < g_eff) else \
                dec_forward_row(m, m.w["embed"][toks[i]].copy(), p + i, cache, range(k))
            of = lm_head(m, dec_forward_row(m, x, p + i, cache, range(k, L)))
            flog.append(of)
            f.append(argmax_lowest(of))
        a = 0                                                    # acceptance
        while a < g_eff and toks[a + 1] == f[a]:
            a += 1
        emitted = toks[1:a + 1] + [f[a]]
        if c.eos_id >= 0 and c.eos_id in emitted:
            emitted = emitted[:emitted.index(c.eos_id) + 1]
            done = True
        res.tokens += emitted
        res.logits += flog[:len(emitted)]
        res.accept_lengths.append(a)
        res.draft_tokens.append(toks[1:])
        p += a + 1
        y = f[a]
        res.kv_lens.append(p)
        res.step_s.append(time.perf_counter() - t0)
    res.kv_len = p
    return res


def model_from_bits(w, bits: dict, to_f64) -> T5Model:
    """Widen a synth T5 workload's bf16 bit arrays to fp64."""
    sh = w.shape
    cfg = T5Config(n_enc=sh.n_enc, n_dec=sh.n_dec, d_model=sh.d_model, n_heads=sh.n_heads, head_dim=sh.head_dim,
                   d_ff=sh.d_ff, vocab=sh.vocab, draft_exit_k=w.draft_exit_k, in_kind=w.in_kind, eos_id=w.eos_id)
    f = {k: to_f64(bits[k]) for k in ("embed", "lm_head", "enc_final", "dec_final", "enc_rel", "dec_rel")}
    f["enc"] = [{n: to_f64(a) for n, a in lw.items()} for lw in bits["enc"]]
    f["dec"] = [{n: to_f64(a) for n, a in lw.items()} for lw in bits["dec"]]
    for n in ("in_norm", "in_w1", "in_w2"):
        if n in bits:
            f[n] = to_f64(bits[n])
    return T5Model(cfg, f, w.dec_scale().astype(np.float64), w.in_scale())
