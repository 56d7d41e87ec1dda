"""Plain fp64 CPU oracle for greedy self-speculative decoding (FastVLM, arXiv 2510.22641).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import or run
this module.  It shares no code with the CUDA library and never reads anything
the CUDA path produced: its inputs come from ``synth`` (seeded generators).

What it computes, in the paper's notation (n = draft exit layer, written k
here; d = draft tokens per step, written gamma):

* Decoder (Sec. "SSD Setup for VLMs"): embeddings x_0, then L layers
  x_{l+1} = x_l + f_l(x_l), then the LM head o = g(x_L) and the greedy token
  argmax softmax(o) = argmax o.  f_l is a pre-norm LLaMA block (RMSNorm,
  multi-head attention with rotary positions, SwiGLU MLP); each sub-block's
  residual write is scaled by s_l (the synthetic acceptance knob).
  g(x) = W_lm RMSNorm_f(x), shared by the draft and the full model.
* Encoder output z (Sec. "SSD Setup for VLMs"): given; its rows are the first
  decoder input rows, followed by the prompt token embeddings.
* Imitation network I (Sec. "Methodology", "Deep Representation Imitation";
  Sec. "Experiments", Training: two fully connected layers and one layer norm):
  I(x) = x + s_in W2 SiLU(W1 RMSNorm_in(x)), hidden width = model width by
  default.  IN_IDENTITY gives "Draft w/o Im" (Table 1).  IN_BLOCK reads the
  module as one decoder block of the model's shape (the NAS space of Sec.
  "Choice of n" holds such blocks): x + f_I(x) with its own weights, residual
  scale s_in and its own KV cache.  Its cache rows hold, for every position
  below kv_len, the block's K/V of that token's x_k: the prefill fills them for
  the prompt rows, each drafting step for its row, and the verification pass
  for row gamma (whose x_k only the verification computes).
* Algorithm 1 (greedy SSD with imitation): draft gamma tokens with
  argmax g(I(x_k)), verify them with the full model in one pass over the
  gamma+1 rows, accept the longest matching prefix, append the full model's
  token at the first mismatch (or the bonus token if all match).
* KV cache (Sec. "Methodology", "KV cache"): one cache shared by the draft and
  the full model; rows of rejected positions are simply overwritten later
  (rollback by length).

Readings where the paper is silent or garbled:
gamma drafts per step (the printed draft loop runs one index too far); the
bonus token is taken after the verify loop; the loop stops after max_new
tokens or after an eos; in the last steps gamma_eff = min(gamma, remaining-1);
argmax ties go to the lowest index; rotate-half RoPE with theta = 10000;
RMSNorm eps = 1e-5.

Dynamic draft length (Sec. "Choice of d"): d(t) = d(0) + floor(10 / (1 + exp(-0.01
(t - N/2)))), evaluated in fp64, where the t-th token is generated from t - 1
tokens of context (so t = kv_len + 2 at a step whose last emitted token y sits at
position kv_len) and N is the longest sequence the model is run with; each step
drafts min(d(t), gamma_cap, remaining - 1) tokens.

Batches of requests (the serving form): ssd_generate_batch runs Algorithm 1 on
independent requests with ragged prompts in lockstep; each request keeps its own
cache, positions and accept lengths, so batching changes no request's result.

Decode rows are always processed one at a time by the same function, so a
row's result does not depend on how many rows a step holds: SSD and greedy
decoding agree bitwise here, not only up to rounding.
"""
from __future__ import annotations

import dataclasses
import time

import numpy as np

IN_IDENTITY = 0
IN_MLP2 = 1
IN_BLOCK = 2


# --------------------------------------------------------------------------- building blocks

def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * gain."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * gain


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def rope_angles(pos: int, head_dim: int, theta: float) -> np.ndarray:
    """Rotation angles pos * theta^(-2i/head_dim), i = 0..head_dim/2-1."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    return pos * theta ** (-2.0 * i / head_dim)


def rope(v: np.ndarray, pos: int, theta: float) -> np.ndarray:
    """Rotary position embedding of one row v[n_heads][head_dim], rotate-half pairing (i, i + half)."""
    half = v.shape[-1] // 2
    ang = rope_angles(pos, v.shape[-1], theta)
    c, s = np.cos(ang), np.sin(ang)
    a, b = v[..., :half], v[..., half:]
    return np.concatenate([a * c - b * s, a * s + b * c], axis=-1)


def softmax(x: np.ndarray) -> np.ndarray:
    e = np.exp(x - np.max(x, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def argmax_lowest(v: np.ndarray) -> int:
    """Greedy token: index of the largest logit, lowest index on ties (np.argmax's rule)."""
    return int(np.argmax(v))


# --------------------------------------------------------------------------- model

@dataclasses.dataclass
class OracleConfig:
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    draft_exit_k: int
    in_kind: int = IN_MLP2
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0
    eos_id: int = -1


class Model:
    """fp64 weights of the decoder, the imitation network and the shared LM head.

    ``weights`` holds fp64 arrays in nn.Linear layout [out][in]:
    embed [V][d], lm_head [V][d], final_norm [d], layers[l] = {wq, wk, wv, wo,
    w_gate, w_up, w_down, attn_norm, ffn_norm}, in_norm/in_w1/in_w2 for IN_MLP2,
    in_block = {the same keys as a layer} for IN_BLOCK.
    ``resid_scale`` = s_l per layer, ``in_scale`` = s_in.
    """

    def __init__(self, cfg: OracleConfig, weights: dict, resid_scale, in_scale: float):
        self.cfg = cfg
        self.w = weights
        self.s = [float(v) for v in resid_scale]
        self.s_in = float(in_scale)


class KVCache:
    """One cache for the draft and the full model: K, V [L][n_heads][S_max][head_dim]
    (slot L: the IN_BLOCK imitation block)."""

    def __init__(self, cfg: OracleConfig, max_seq: int):
        shp = (cfg.n_layers + (1 if cfg.in_kind == IN_BLOCK else 0), cfg.n_heads, max_seq, cfg.head_dim)
        self.k = np.zeros(shp)
        self.v = np.zeros(shp)


def embed(m: Model, token: int) -> np.ndarray:
    return m.w["embed"][token].copy()


def block_row(m: Model, lw: dict, s: float, slot: int, x: np.ndarray, pos: int, cache: KVCache) -> np.ndarray:
    """x + f(x) for one pre-norm block (weights lw, residual scale s) and one row at position
    ``pos``; writes K/V[slot][:, pos] and attends over K/V[slot][:, 0..pos]."""
    c = m.cfg
    H, Dh = c.n_heads, c.head_dim
    n = rms_norm(x, lw["attn_norm"], c.rms_eps)
    q = rope((lw["wq"] @ n).reshape(H, Dh), pos, c.rope_theta)
    k = rope((lw["wk"] @ n).reshape(H, Dh), pos, c.rope_theta)
    v = (lw["wv"] @ n).reshape(H, Dh)
    cache.k[slot, :, pos] = k
    cache.v[slot, :, pos] = v
    keys, vals = cache.k[slot, :, :pos + 1], cache.v[slot, :, :pos + 1]      # causal: keys 0..pos
    scores = np.einsum("hd,hjd->hj", q, keys) / np.sqrt(Dh)
    o = np.einsum("hj,hjd->hd", softmax(scores), vals).reshape(H * Dh)
    h = x + s * (lw["wo"] @ o)
    u = rms_norm(h, lw["ffn_norm"], c.rms_eps)
    return h + s * (lw["w_down"] @ (silu(lw["w_gate"] @ u) * (lw["w_up"] @ u)))


def layer_row(m: Model, l: int, x: np.ndarray, pos: int, cache: KVCache) -> np.ndarray:
    """x_{l+1} = x_l + f_l(x_l) for one row at position ``pos``; writes K/V[l][:, pos]."""
    return block_row(m, m.w["layers"][l], m.s[l], l, x, pos, cache)


def block_kv(m: Model, x: np.ndarray, pos: int, cache: KVCache) -> None:
    """The IN_BLOCK block's K/V of x (a row's x_k) at ``pos``, without the rest of the block."""
    c, lw, slot = m.cfg, m.w["in_block"], m.cfg.n_layers
    n = rms_norm(x, lw["attn_norm"], c.rms_eps)
    cache.k[slot, :, pos] = rope((lw["wk"] @ n).reshape(c.n_heads, c.head_dim), pos, c.rope_theta)
    cache.v[slot, :, pos] = (lw["wv"] @ n).reshape(c.n_heads, c.head_dim)


def forward_row(m: Model, x: np.ndarray, pos: int, cache: KVCache, layers) -> np.ndarray:
    for l in layers:
        x = layer_row(m, l, x, pos, cache)
    return x


def lm_head(m: Model, x: np.ndarray) -> np.ndarray:
    """o = g(x) = W_lm RMSNorm_f(x)."""
    return m.w["lm_head"] @ rms_norm(x, m.w["final_norm"], m.cfg.rms_eps)


def imitation(m: Model, x: np.ndarray, pos: int | None = None, cache: KVCache | None = None) -> np.ndarray:
    """x_I = I(x_k): identity, x + s_in W2 SiLU(W1 RMSNorm_in(x)), or (IN_BLOCK) the imitation
    block at position ``pos`` over its own cache slot."""
    if m.cfg.in_kind == IN_IDENTITY:
        return x
    if m.cfg.in_kind == IN_BLOCK:
        return block_row(m, m.w["in_block"], m.s_in, m.cfg.n_layers, x, pos, cache)
    n = rms_norm(x, m.w["in_norm"], m.cfg.rms_eps)
    return x + m.s_in * (m.w["in_w2"] @ silu(m.w["in_w1"] @ n))


def prefill(m: Model, cache: KVCache, vis: np.ndarray, prompt) -> np.ndarray:
    """Forward the rows [z ; embed(prompt)] at positions 0..P-1 through all layers.

    Writes K/V[:, :, 0:P] and returns the logits of the last row (which give the
    first new token).  Processes the whole sequence per layer with matrix
    products and a causal mask (row i sees keys 0..i).
    """
    c = m.cfg
    H, Dh, P = c.n_heads, c.head_dim, vis.shape[0] + len(prompt)
    X = np.concatenate([vis, m.w["embed"][np.asarray(prompt, dtype=np.int64)]], axis=0)
    causal = np.tril(np.ones((P, P), dtype=bool))

    def block_kv_rows(X):                                        # the imitation block's K/V of every x_k row
        lw = m.w["in_block"]
        N = rms_norm(X, lw["attn_norm"], c.rms_eps)
        K = (N @ lw["wk"].T).reshape(P, H, Dh)
        for p in range(P):
            K[p] = rope(K[p], p, c.rope_theta)
        cache.k[c.n_layers, :, :P] = K.transpose(1, 0, 2)
        cache.v[c.n_layers, :, :P] = (N @ lw["wv"].T).reshape(P, H, Dh).transpose(1, 0, 2)

    for l in range(c.n_layers):
        if l == c.draft_exit_k and c.in_kind == IN_BLOCK:
            block_kv_rows(X)
        lw = m.w["layers"][l]
        N = rms_norm(X, lw["attn_norm"], c.rms_eps)
        Q = (N @ lw["wq"].T).reshape(P, H, Dh)
        K = (N @ lw["wk"].T).reshape(P, H, Dh)
        V = (N @ lw["wv"].T).reshape(P, H, Dh)
        for p in range(P):
            Q[p] = rope(Q[p], p, c.rope_theta)
            K[p] = rope(K[p], p, c.rope_theta)
        cache.k[l, :, :P] = K.transpose(1, 0, 2)
        cache.v[l, :, :P] = V.transpose(1, 0, 2)
        S = np.matmul(Q.transpose(1, 0, 2), K.transpose(1, 2, 0)) / np.sqrt(Dh)     # [H][i][j]
        S = np.where(causal[None], S, -np.inf)
        O = np.matmul(softmax(S), V.transpose(1, 0, 2)).transpose(1, 0, 2).reshape(P, H * Dh)
        Hh = X + m.s[l] * (O @ lw["wo"].T)
        U = rms_norm(Hh, lw["ffn_norm"], c.rms_eps)
        X = Hh + m.s[l] * ((silu(U @ lw["w_gate"].T) * (U @ lw["w_up"].T)) @ lw["w_down"].T)
    if c.draft_exit_k == c.n_layers and c.in_kind == IN_BLOCK:
        block_kv_rows(X)
    return lm_head(m, X[-1])


# --------------------------------------------------------------------------- decoding loops

@dataclasses.dataclass
class Result:
    tokens: list            # emitted new tokens y^{t+1} ... (first one from the prefill)
    logits: list            # full-model logits that produced each emitted token
    kv_len: int             # valid cache length at the end (positions 0..kv_len-1)
    accept_lengths: list = dataclasses.field(default_factory=list)   # a per SSD step
    kv_lens: list = dataclasses.field(default_factory=list)          # kv_len after each step
    draft_tokens: list = dataclasses.field(default_factory=list)     # per step: d_1..d_gamma_eff
    draft_logits: list = dataclasses.field(default_factory=list)     # per step: g(I(x_k)) rows
    cache: KVCache | None = None
    prefill_s: float = 0.0                                            # wall time of the prefill
    step_s: list = dataclasses.field(default_factory=list)            # wall time per decode step


def _truncate_eos(tokens: list, eos_id: int) -> tuple[list, bool]:
    if eos_id >= 0 and eos_id in tokens:
        return tokens[:tokens.index(eos_id) + 1], True
    return tokens, False


def draft_length(t: int, d0: int, n_max: int) -> int:
    """Sec. "Choice of d", the equation for d(t): d0 + floor(10 * sigmoid(0.01 (t - N/2))) in fp64.

    The sigmoid is written as 1 / (1 + exp(-z)); for t far above N/2 it rounds to 1 and d reaches
    d0 + 10, the paper's stated upper end {5, ..., 15} for d0 = 5.
    """
    z = -0.01 * (float(t) - float(n_max) / 2.0)
    return d0 + int(np.floor(10.0 / (1.0 + np.exp(z))))


def greedy_generate(m: Model, vis: np.ndarray, prompt, max_new: int, max_seq: int | None = None,
                    keep_cache: bool = False) -> Result:
    """Plain autoregressive greedy decoding of the full model (the speedup baseline)."""
    P = vis.shape[0] + len(prompt)
    cache = KVCache(m.cfg, max_seq or (P + max_new + 1))
    o = prefill(m, cache, vis, prompt)
    y = argmax_lowest(o)
    tokens, logits, pos = [y], [o], P
    while len(tokens) < max_new and not (m.cfg.eos_id >= 0 and y == m.cfg.eos_id):
        x = forward_row(m, embed(m, y), pos, cache, range(m.cfg.n_layers))
        o = lm_head(m, x)
        y = argmax_lowest(o)
        tokens.append(y)
        logits.append(o)
        pos += 1
    return Result(tokens=tokens, logits=logits, kv_len=pos, cache=cache if keep_cache else None)


class _SSDRun:
    """One request under Algorithm 1: the prefill at construction, then one draft + verify + accept
    step per call to step() (see ssd_generate)."""

    def __init__(self, m: Model, vis: np.ndarray, prompt, max_new: int, gamma: int, max_seq: int | None,
                 reuse_draft_rows: bool, keep_draft_logits: bool, dynamic: tuple | None):
        c = m.cfg
        self.m, self.max_new, self.gamma = m, max_new, gamma
        self.reuse, self.keep_dlog, self.dynamic = reuse_draft_rows, keep_draft_logits, dynamic
        P = vis.shape[0] + len(prompt)
        self.cache = KVCache(c, max_seq or (P + max_new + gamma + 1))
        t0 = time.perf_counter()
        o = prefill(m, self.cache, vis, prompt)
        self.y = argmax_lowest(o)
        self.res = Result(tokens=[self.y], logits=[o], kv_len=P, prefill_s=time.perf_counter() - t0)
        self.p, self.done = P, (c.eos_id >= 0 and self.y == c.eos_id)

    @property
    def finished(self) -> bool:
        return self.done or len(self.res.tokens) >= self.max_new

    def gamma_eff(self) -> int:
        """Drafts of the next step: min(gamma or d(t), remaining - 1)."""
        remaining = self.max_new - len(self.res.tokens)
        g_step = self.gamma
        if self.dynamic is not None:
            d0, n_max = self.dynamic[0], self.dynamic[1]
            over = self.dynamic[2] if len(self.dynamic) > 2 else "context"
            # t: the index of the token this step's verification will emit first, counted over the
            # whole context (a token at position q is the (q + 1)-th; the next one sits at p + 1) or
            # over the generated tokens (the next new token is number len(tokens) + 1)
            t = self.p + 2 if over == "context" else len(self.res.tokens) + 1
            g_step = min(self.gamma, draft_length(t, d0, n_max))
        return min(g_step, remaining - 1)

    def step(self) -> None:
        m, c, res = self.m, self.m.cfg, self.res
        k, L, p, cache = c.draft_exit_k, c.n_layers, self.p, self.cache
        t0 = time.perf_counter()
        g_eff = self.gamma_eff()
        toks, xk, dlog = [self.y], [], []
        for j in range(g_eff):                                   # drafting stage
            x = forward_row(m, embed(m, toks[j]), p + j, cache, range(k))
            xk.append(x)
            od = lm_head(m, imitation(m, x, p + j, cache))
            dlog.append(od)
            toks.append(argmax_lowest(od))
        f, flog = [], []
        for i in range(g_eff + 1):                               # verification stage
            if self.reuse and i < g_eff:
                x = xk[i]
            else:
                x = forward_row(m, embed(m, toks[i]), p + i, cache, range(k))
                if c.in_kind == IN_BLOCK:                        # the block's K/V of this row's x_k
                    block_kv(m, x, p + i, cache)
            x = forward_row(m, x, p + i, cache, range(k, L))
            of = lm_head(m, x)
            flog.append(of)
            f.append(argmax_lowest(of))
        a = 0                                                    # acceptance
        while a < g_eff and toks[a + 1] == f[a]:
            a += 1
        emitted = toks[1:a + 1] + [f[a]]
        emitted, self.done = _truncate_eos(emitted, c.eos_id)
        res.tokens += emitted
        res.logits += flog[:len(emitted)]
        res.accept_lengths.append(a)
        res.draft_tokens.append(toks[1:])
        if self.keep_dlog:
            res.draft_logits.append(dlog)
        self.p = p + a + 1
        self.y = f[a]
        res.kv_lens.append(self.p)
        res.kv_len = self.p
        res.step_s.append(time.perf_counter() - t0)


def ssd_generate(m: Model, vis: np.ndarray, prompt, max_new: int, gamma: int,
                 max_seq: int | None = None, reuse_draft_rows: bool = True,
                 keep_cache: bool = False, keep_draft_logits: bool = False,
                 max_steps: int | None = None, dynamic: tuple | None = None) -> Result:
    """Algorithm 1 (greedy self-speculative decoding with the imitation network).

    Per step, with y the last emitted token at position p = kv_len:
      drafting:  t_0 = y; for j < gamma_eff: x_k = layers 0..k-1 of t_j at p+j,
                 d_{j+1} = argmax g(I(x_k)), t_{j+1} = d_{j+1}
      verifying: for i = 0..gamma_eff: f_i = argmax g(x_L) of row t_i at p+i
                 (shallow layers reused from the draft when reuse_draft_rows)
      accepting: a = largest i <= gamma_eff with d_1..d_i = f_0..f_{i-1};
                 emit d_1..d_a and f_a; kv_len = p + a + 1; y = f_a.
    max_steps (timing samples only) stops after that many steps.
    dynamic = (d0, N) or (d0, N, "generated"): each step drafts min(d(t), gamma, remaining - 1)
    tokens (Sec. "Choice of d"); gamma is then the cap.  t = kv_len + 2 counts the whole context;
    with "generated", t = tokens emitted so far + 1 counts the new tokens only.
    """
    run = _SSDRun(m, vis, prompt, max_new, gamma, max_seq, reuse_draft_rows, keep_draft_logits, dynamic)
    while not run.finished and (max_steps is None or len(run.res.step_s) < max_steps):
        run.step()
    if keep_cache:
        run.res.cache = run.cache
    return run.res


@dataclasses.dataclass
class BatchResult:
    results: list    # per request: Result
    active: list     # per batched step: indices of the requests that stepped
    rows: list       # per batched step: verification rows, the sum of gamma_eff + 1 over the active requests


def ssd_generate_batch(m: Model, requests, max_new: int, gamma: int, max_seq: int | None = None) -> BatchResult:
    """Algorithm 1 on a batch of independent requests in lockstep (the serving form of the method).

    requests: list of (vis, prompt) with prompts of different lengths (ragged).  Each request has its
    own cache, kv_len and accept lengths; in every batched step each unfinished request drafts
    gamma_eff = min(gamma, remaining - 1) tokens at its own positions, the verification covers the
    rows of all active requests at once, and each request accepts and rolls back on its own.  A
    finished request (max_new tokens out, or eos) takes no further rows.  Every request's tokens,
    logits and accept lengths are those of ssd_generate on it alone.
    """
    runs = [_SSDRun(m, vis, prompt, max_new, gamma, max_seq, True, False, None) for vis, prompt in requests]
    out = BatchResult(results=[r.res for r in runs], active=[], rows=[])
    while not all(r.finished for r in runs):
        act = [b for b, r in enumerate(runs) if not r.finished]
        out.rows.append(sum(runs[b].gamma_eff() + 1 for b in act))
        out.active.append(act)
        for b in act:
            runs[b].step()
    return out


# --------------------------------------------------------------------------- construction helpers

def config_from_workload(w) -> OracleConfig:
    sh = w.shape
    return OracleConfig(n_layers=sh.n_layers, d_model=sh.d_model, n_heads=sh.n_heads,
                        head_dim=sh.head_dim, d_ff=sh.d_ff, vocab=sh.vocab,
                        draft_exit_k=w.draft_exit_k, in_kind=w.in_kind, rms_eps=sh.rms_eps,
                        rope_theta=sh.rope_theta, eos_id=w.eos_id)


def model_from_bits(w, bits: dict, to_f64) -> Model:
    """Widen the generator's bf16 bit arrays to fp64 with ``to_f64`` and build a Model."""
    f = {"embed": to_f64(bits["embed"]), "lm_head": to_f64(bits["lm_head"]),
         "final_norm": to_f64(bits["final_norm"]),
         "layers": [{n: to_f64(a) for n, a in lw.items()} for lw in bits["layers"]]}
    for n in ("in_norm", "in_w1", "in_w2"):
        if n in bits:
            f[n] = to_f64(bits[n])
    if "in_block" in bits:
        f["in_block"] = {n: to_f64(a) for n, a in bits["in_block"].items()}
    return Model(config_from_workload(w), f, w.resid_scale().astype(np.float64), w.in_scale())
