"""Seeded synthetic workloads shared by the oracle and the CUDA path.

This module only makes numbers: model shapes, counter-based random weights and
inputs.  It contains none of the decoding method's arithmetic, so both sides
(the fp64 oracle under ``oracle/`` and the CUDA library) can consume the same
arrays without sharing any computation.

All weights are produced as bf16 bit patterns (``numpy.uint16``): the CUDA path
stores them as bf16 and the oracle widens the same bits to fp64 exactly.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gen.c")
_SO = os.path.join(_HERE, "_gen.so")
_lock = threading.Lock()
_lib = None


def build_generator(force: bool = False) -> str:
    """Compile ``gen.c`` into ``_gen.so`` with gcc (OpenMP, no FP contraction)."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                               _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def _gen():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build_generator())
            u64, i64, dbl, vp = ctypes.c_uint64, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p
            lib.synth_normal_bf16.argtypes = [u64, u64, dbl, dbl, i64, vp]
            lib.synth_normal_f64.argtypes = [u64, u64, dbl, dbl, i64, vp]
            lib.synth_uniform_i32.argtypes = [u64, u64, i64, i64, i64, vp]
            lib.synth_raw_u64.argtypes = [u64, u64, i64, vp]
            lib.synth_bf16_to_f64.argtypes = [vp, i64, vp]
            for f in (lib.synth_normal_bf16, lib.synth_normal_f64, lib.synth_uniform_i32,
                      lib.synth_raw_u64, lib.synth_bf16_to_f64):
                f.restype = None
            _lib = lib
    return _lib


# --------------------------------------------------------------------------- primitives

def normal_bf16(seed: int, stream: int, shape, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    """bf16 bits of mean + std * N(0,1), element i drawn from counter i of (seed, stream)."""
    out = np.empty(shape, dtype=np.uint16)
    _gen().synth_normal_bf16(seed, stream, mean, std, out.size, out.ctypes.data)
    return out


def normal_f64(seed: int, stream: int, shape, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.float64)
    _gen().synth_normal_f64(seed, stream, mean, std, out.size, out.ctypes.data)
    return out


def uniform_i32(seed: int, stream: int, shape, lo: int, hi: int) -> np.ndarray:
    out = np.empty(shape, dtype=np.int32)
    _gen().synth_uniform_i32(seed, stream, lo, hi, out.size, out.ctypes.data)
    return out


def raw_u64(seed: int, stream: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint64)
    _gen().synth_raw_u64(seed, stream, n, out.ctypes.data)
    return out


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp64 (multi-threaded)."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(bits.shape, dtype=np.float64)
    _gen().synth_bf16_to_f64(bits.ctypes.data, bits.size, out.ctypes.data)
    return out


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 bits (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


# --------------------------------------------------------------------------- shapes

IN_IDENTITY = 0   # draft without imitation: g(x_k) directly
IN_MLP2 = 1       # x + s_in * W2 SiLU(W1 RMSNorm(x)): two FC layers and one norm
IN_BLOCK = 2      # one decoder block of the model's shape, with its own KV cache
IN_BLOCK_LAYER = 0xFFFF   # stream index of the block's weights (no decoder layer uses it)


@dataclasses.dataclass(frozen=True)
class ModelShape:
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0

    @property
    def qdim(self) -> int:
        return self.n_heads * self.head_dim

    def layer_bytes_bf16(self) -> int:
        d, q, f = self.d_model, self.qdim, self.d_ff
        return 2 * (3 * q * d + d * q + 3 * f * d) + 2 * 2 * d


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic self-speculative decoding workload (bs1)."""
    name: str
    shape: ModelShape
    draft_exit_k: int          # draft = decoder layers 0..k-1 + imitation network
    in_kind: int
    in_hidden: int
    gamma: int                 # draft tokens per step
    n_vis: int                 # synthetic visual embeddings (encoder output z)
    n_prompt: int
    max_new: int
    s: float = 1.0             # deep-layer residual-write scale (acceptance knob)
    weight_std: float = 0.02
    vis_std: float = 1.0
    norm_gain: str = "ones"    # "ones" or "perturbed" (N(1, 0.1))
    eos_id: int = -1
    weight_seed: int = 0
    input_seed: int = 0

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def prompt_len(self) -> int:
        return self.n_vis + self.n_prompt

    def max_seq(self) -> int:
        return self.prompt_len + self.max_new + self.gamma + 1

    def resid_scale(self) -> np.ndarray:
        """s_l: 1 for the draft layers, s for the deep layers k..L-1 (fp32)."""
        sc = np.ones(self.shape.n_layers, dtype=np.float32)
        sc[self.draft_exit_k:] = np.float32(self.s)
        return sc

    def in_scale(self) -> float:
        return float(np.float32(self.s))


TINY_SHAPE = ModelShape(n_layers=4, d_model=256, n_heads=4, head_dim=64, d_ff=1024, vocab=2048)
LLAVA7B_SHAPE = ModelShape(n_layers=32, d_model=4096, n_heads=32, head_dim=128, d_ff=11008, vocab=32000)
LLAVA13B_SHAPE = ModelShape(n_layers=40, d_model=5120, n_heads=40, head_dim=128, d_ff=13824, vocab=32000)

# Tiny parity workload: 4 layers, d=256, draft = layers 0-1 + imitation module, gamma=4.
TINY = Workload(name="tiny_L4_d256", shape=TINY_SHAPE, draft_exit_k=2, in_kind=IN_MLP2,
                in_hidden=1024, gamma=4, n_vis=32, n_prompt=16, max_new=32, s=1.0)

# The same tiny model with the imitation module read literally as one decoder block of the model's
# shape (its own attention over its own KV cache, SwiGLU MLP, two RMSNorms).
TINY_BLOCK = TINY.replace(name="tiny_L4_d256_inblock", in_kind=IN_BLOCK)

# LLaVA-1.5-7B-shaped decoder: 576 visual rows (24x24 grid) + 64 prompt ids, k=8, gamma=5.
LLAVA7B = Workload(name="llava15_7b_shape", shape=LLAVA7B_SHAPE, draft_exit_k=8, in_kind=IN_MLP2,
                   in_hidden=4096, gamma=5, n_vis=576, n_prompt=64, max_new=128, s=0.2)

LLAVA7B_S_VALUES = (0.05, 0.2, 1.0)

# LLaVA-1.5-13B-shaped decoder: 576 visual rows + up to 256 prompt ids, k=10, gamma=6, 256 new tokens.
LLAVA13B = Workload(name="llava15_13b_shape", shape=LLAVA13B_SHAPE, draft_exit_k=10, in_kind=IN_MLP2,
                    in_hidden=5120, gamma=6, n_vis=576, n_prompt=256, max_new=256, s=0.2)


@dataclasses.dataclass(frozen=True)
class BatchWorkload:
    """A batch of independent requests on one model (the serving form of the method): every request
    has the base workload's visual rows and a prompt of length U[prompt_min, prompt_max] (ragged)."""
    base: Workload
    batch: int
    prompt_min: int
    prompt_max: int

    def replace(self, **kw) -> "BatchWorkload":
        return dataclasses.replace(self, **kw)

    def prompt_lengths(self, seed: int | None = None) -> np.ndarray:
        seed = self.base.input_seed if seed is None else seed
        return uniform_i32(seed, stream_id("prompt_len"), (self.batch,), self.prompt_min, self.prompt_max + 1)

    def max_seq(self) -> int:
        b = self.base
        return b.n_vis + self.prompt_max + b.max_new + b.gamma + 1


# 16 requests on the 13B shape, prompts U[32, 256] after the 576 visual rows, s = 0.2.
LLAVA13B_B16 = BatchWorkload(base=LLAVA13B, batch=16, prompt_min=32, prompt_max=256)
# Its tiny stand-in for parity: 4 requests on the tiny model, prompts U[4, 24].
TINY_B4 = BatchWorkload(base=TINY, batch=4, prompt_min=4, prompt_max=24)


# --------------------------------------------------------------------------- weights and inputs

_KIND = {
    "embed": 1, "lm_head": 2, "final_norm": 3,
    "wq": 10, "wk": 11, "wv": 12, "wo": 13, "w_gate": 14, "w_up": 15, "w_down": 16,
    "attn_norm": 17, "ffn_norm": 18,
    "in_norm": 20, "in_w1": 21, "in_w2": 22,
    "vis": 40, "prompt": 41, "prompt_len": 42,
}


def stream_id(kind: str, layer: int = 0) -> int:
    return (_KIND[kind] << 16) | layer


def layer_shapes(shape: ModelShape) -> dict:
    d, q, f = shape.d_model, shape.qdim, shape.d_ff
    return {"wq": (q, d), "wk": (q, d), "wv": (q, d), "wo": (d, q),
            "w_gate": (f, d), "w_up": (f, d), "w_down": (d, f),
            "attn_norm": (d,), "ffn_norm": (d,)}


def _gain(w: Workload, kind: str, layer: int, n: int) -> np.ndarray:
    if w.norm_gain == "ones":
        return np.full(n, 0x3F80, dtype=np.uint16)
    return normal_bf16(w.weight_seed, stream_id(kind, layer), (n,), mean=1.0, std=0.1)


def make_layer_weights(w: Workload, l: int) -> dict:
    """Decoder layer l's weights (l = IN_BLOCK_LAYER: the imitation block's) as bf16 bit arrays."""
    lw = {}
    for name, shp in layer_shapes(w.shape).items():
        if name.endswith("norm"):
            lw[name] = _gain(w, name, l, shp[0])
        else:
            lw[name] = normal_bf16(w.weight_seed, stream_id(name, l), shp, std=w.weight_std)
    return lw


def make_weights(w: Workload, with_layers: bool = True) -> dict:
    """All weights of the workload as bf16 bit arrays, nn.Linear layout [out][in].

    Returns {"embed", "lm_head", "final_norm", "layers": [ {wq, ...}, ... ],
             "in_norm", "in_w1", "in_w2"} (IN_MLP2) or "in_block": {wq, ...} (IN_BLOCK);
    no IN entries for IN_IDENTITY.  with_layers=False leaves "layers" empty (large models build
    them one at a time with make_layer_weights).
    """
    sh = w.shape
    d, V = sh.d_model, sh.vocab
    std = w.weight_std
    out = {
        "embed": normal_bf16(w.weight_seed, stream_id("embed"), (V, d), std=std),
        "lm_head": normal_bf16(w.weight_seed, stream_id("lm_head"), (V, d), std=std),
        "final_norm": _gain(w, "final_norm", 0, d),
        "layers": [],
    }
    if with_layers:
        for l in range(sh.n_layers):
            out["layers"].append(make_layer_weights(w, l))
    if w.in_kind == IN_BLOCK:
        out["in_block"] = make_layer_weights(w, IN_BLOCK_LAYER)
    if w.in_kind == IN_MLP2:
        out["in_norm"] = _gain(w, "in_norm", 0, d)
        out["in_w1"] = normal_bf16(w.weight_seed, stream_id("in_w1"), (w.in_hidden, d), std=std)
        out["in_w2"] = normal_bf16(w.weight_seed, stream_id("in_w2"), (d, w.in_hidden), std=std)
    return out


def make_inputs(w: Workload, seed: int | None = None) -> tuple[np.ndarray, np.ndarray]:
    """Synthetic encoder output z (bf16 bits [n_vis][d], N(0, vis_std)) and prompt ids U[0, V)."""
    seed = w.input_seed if seed is None else seed
    vis = normal_bf16(seed, stream_id("vis"), (w.n_vis, w.shape.d_model), std=w.vis_std)
    prompt = uniform_i32(seed, stream_id("prompt"), (w.n_prompt,), 0, w.shape.vocab)
    return vis, prompt


# --------------------------------------------------------------------------- encoder-decoder (FlanT5-shaped)

@dataclasses.dataclass(frozen=True)
class T5Shape:
    """T5 v1.1 shape: pre-norm blocks, gated-GELU MLP, relative-position bias, untied LM head."""
    n_enc: int
    n_dec: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    rel_buckets: int = 32
    rel_max_distance: int = 128

    @property
    def qdim(self) -> int:
        return self.n_heads * self.head_dim

    def dec_layer_bytes_bf16(self) -> int:
        """Weights one decode row streams per decoder layer (self q/k/v/o, cross q/o, MLP, 3 norms);
        the cross-attention K/V projections run once per request, over the encoder output."""
        d, q, f = self.d_model, self.qdim, self.d_ff
        return 2 * (4 * q * d + 2 * q * d + 3 * f * d) + 2 * 3 * d


@dataclasses.dataclass(frozen=True)
class T5Workload:
    """One synthetic encoder-decoder self-speculative decoding workload (bs1).

    The encoder reads n_query synthetic query embeddings (the image-grounded queries, N(0, vis_std))
    followed by n_prompt prompt ids; the decoder starts from token 0 and drafts with decoder layers
    0..k-1 plus the imitation network.
    """
    name: str
    shape: T5Shape
    draft_exit_k: int
    in_kind: int
    in_hidden: int
    gamma: int
    n_query: int
    n_prompt: int
    max_new: int
    s: float = 1.0
    weight_std: float = 0.02
    embed_std: float = 1.0
    rel_std: float = 0.5
    vis_std: float = 1.0
    norm_gain: str = "ones"
    eos_id: int = -1
    weight_seed: int = 0
    input_seed: int = 0

    def replace(self, **kw) -> "T5Workload":
        return dataclasses.replace(self, **kw)

    @property
    def enc_len(self) -> int:
        return self.n_query + self.n_prompt

    def max_dec(self) -> int:
        return self.max_new + self.gamma + 1

    def dec_scale(self) -> np.ndarray:
        """s_l of the decoder: 1 for layers 0..k-1, s for k..L-1 (fp32)."""
        sc = np.ones(self.shape.n_dec, dtype=np.float32)
        sc[self.draft_exit_k:] = np.float32(self.s)
        return sc

    def in_scale(self) -> float:
        return float(np.float32(self.s))


T5_TINY_SHAPE = T5Shape(n_enc=2, n_dec=4, d_model=256, n_heads=4, head_dim=64, d_ff=512, vocab=2048)
FLANT5XL_SHAPE = T5Shape(n_enc=24, n_dec=24, d_model=2048, n_heads=32, head_dim=64, d_ff=5120, vocab=32128)

# Tiny encoder-decoder parity workload: 2 encoder + 4 decoder layers, draft = decoder layers 0-1 + imitation.
T5_TINY = T5Workload(name="t5_tiny_e2_d4_d256", shape=T5_TINY_SHAPE, draft_exit_k=2, in_kind=IN_MLP2,
                     in_hidden=512, gamma=4, n_query=32, n_prompt=16, max_new=24, s=1.0)

# BLIP-2 FlanT5-xl-shaped language model: 32 queries + 16 prompt ids, draft = decoder layers 0-5, gamma=4.
FLANT5XL = T5Workload(name="blip2_flant5xl_shape", shape=FLANT5XL_SHAPE, draft_exit_k=6, in_kind=IN_MLP2,
                      in_hidden=2048, gamma=4, n_query=32, n_prompt=16, max_new=30, s=0.2)

_T5_KIND = {
    "t5_embed": 60, "t5_lm_head": 61, "enc_final": 62, "dec_final": 63, "enc_rel": 64, "dec_rel": 65,
    "attn_norm": 66, "self_norm": 67, "cross_norm": 68, "ffn_norm": 69,
    "wq": 70, "wk": 71, "wv": 72, "wo": 73, "cq": 74, "ck": 75, "cv": 76, "co": 77,
    "wi0": 78, "wi1": 79, "wff": 80, "in_norm": 81, "in_w1": 82, "in_w2": 83,
    "query": 84, "t5_prompt": 85,
}
_T5_DEC = 0x100   # stream-layer offset of decoder layers


def t5_stream_id(kind: str, layer: int = 0) -> int:
    return (_T5_KIND[kind] << 16) | layer


def t5_layer_shapes(shape: T5Shape, decoder: bool) -> dict:
    d, q, f = shape.d_model, shape.qdim, shape.d_ff
    out = {"wq": (q, d), "wk": (q, d), "wv": (q, d), "wo": (d, q)}
    if decoder:
        out.update({"cq": (q, d), "ck": (q, d), "cv": (q, d), "co": (d, q),
                    "self_norm": (d,), "cross_norm": (d,)})
    else:
        out["attn_norm"] = (d,)
    out.update({"wi0": (f, d), "wi1": (f, d), "wff": (d, f), "ffn_norm": (d,)})
    return out


def make_t5_weights(w: T5Workload) -> dict:
    """All weights as bf16 bit arrays ([out][in] layouts).

    {"embed" [V][d], "lm_head" [V][d], "enc_final", "dec_final" [d], "enc_rel", "dec_rel" [buckets][H],
     "enc": [{wq, wk, wv, wo, attn_norm, wi0, wi1, wff, ffn_norm}], "dec": [{... + cq, ck, cv, co,
     self_norm, cross_norm}], "in_norm", "in_w1", "in_w2" (IN_MLP2)}.
    Query projections (wq, cq) are drawn with std weight_std / sqrt(head_dim): T5 computes attention
    logits without a 1/sqrt(head_dim) factor and folds it into the query projection's scale instead.
    """
    sh = w.shape
    d, V, std = sh.d_model, sh.vocab, w.weight_std
    sd = w.weight_seed

    def gain(kind, layer, n):
        if w.norm_gain == "ones":
            return np.full(n, 0x3F80, dtype=np.uint16)
        return normal_bf16(sd, t5_stream_id(kind, layer), (n,), mean=1.0, std=0.1)

    def block(layer, decoder):
        lw = {}
        for name, shp in t5_layer_shapes(sh, decoder).items():
            if name.endswith("norm"):
                lw[name] = gain(name, layer, shp[0])
            else:
                s = std / np.sqrt(sh.head_dim) if name in ("wq", "cq") else std
                lw[name] = normal_bf16(sd, t5_stream_id(name, layer), shp, std=s)
        return lw

    out = {
        "embed": normal_bf16(sd, t5_stream_id("t5_embed"), (V, d), std=w.embed_std),
        "lm_head": normal_bf16(sd, t5_stream_id("t5_lm_head"), (V, d), std=std),
        "enc_final": gain("enc_final", 0, d),
        "dec_final": gain("dec_final", 0, d),
        "enc_rel": normal_bf16(sd, t5_stream_id("enc_rel"), (sh.rel_buckets, sh.n_heads), std=w.rel_std),
        "dec_rel": normal_bf16(sd, t5_stream_id("dec_rel"), (sh.rel_buckets, sh.n_heads), std=w.rel_std),
        "enc": [block(l, False) for l in range(sh.n_enc)],
        "dec": [block(_T5_DEC + l, True) for l in range(sh.n_dec)],
    }
    if w.in_kind == IN_MLP2:
        out["in_norm"] = gain("in_norm", 0, d)
        out["in_w1"] = normal_bf16(sd, t5_stream_id("in_w1"), (w.in_hidden, d), std=std)
        out["in_w2"] = normal_bf16(sd, t5_stream_id("in_w2"), (d, w.in_hidden), std=std)
    elif w.in_kind != IN_IDENTITY:
        raise ValueError("encoder-decoder workloads take IN_IDENTITY or IN_MLP2")
    return out


def make_t5_inputs(w: T5Workload, seed: int | None = None) -> tuple[np.ndarray, np.ndarray]:
    """Synthetic query embeddings (bf16 bits [n_query][d], N(0, vis_std)) and prompt ids U[0, V)."""
    seed = w.input_seed if seed is None else seed
    q = normal_bf16(seed, t5_stream_id("query"), (w.n_query, w.shape.d_model), std=w.vis_std)
    prompt = uniform_i32(seed, t5_stream_id("t5_prompt"), (w.n_prompt,), 0, w.shape.vocab)
    return q, prompt


def make_batch_inputs(bw: BatchWorkload, seed: int | None = None) -> list:
    """Per request b: synthetic encoder output (bf16 bits [n_vis][d], N(0, vis_std)) and prompt ids
    U[0, V) of the request's ragged length; request b draws from streams of its own (layer field b + 1)."""
    seed = bw.base.input_seed if seed is None else seed
    w = bw.base
    out = []
    for b, n in enumerate(bw.prompt_lengths(seed)):
        vis = normal_bf16(seed, stream_id("vis", b + 1), (w.n_vis, w.shape.d_model), std=w.vis_std)
        prompt = uniform_i32(seed, stream_id("prompt", b + 1), (int(n),), 0, w.shape.vocab)
        out.append((vis, prompt))
    return out
