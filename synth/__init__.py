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


# --------------------------------------------------------------------------- weights and inputs

_KIND = {
    "embed": 1, "lm_head": 2, "final_norm": 3,
    "wq": 10, "wk": 11, "wv": 12, "wo": 13, "w_gate": 14, "w_up": 15, "w_down": 16,
    "attn_norm": 17, "ffn_norm": 18,
    "in_norm": 20, "in_w1": 21, "in_w2": 22,
    "vis": 40, "prompt": 41,
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


def make_weights(w: Workload) -> dict:
    """All weights of the workload as bf16 bit arrays, nn.Linear layout [out][in].

    Returns {"embed", "lm_head", "final_norm", "layers": [ {wq, ...}, ... ],
             "in_norm", "in_w1", "in_w2"} (IN_MLP2) or "in_block": {wq, ...} (IN_BLOCK);
    no IN entries for IN_IDENTITY.
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
    def block(l: int) -> dict:
        lw = {}
        for name, shp in layer_shapes(sh).items():
            if name.endswith("norm"):
                lw[name] = _gain(w, name, l, shp[0])
            else:
                lw[name] = normal_bf16(w.weight_seed, stream_id(name, l), shp, std=std)
        return lw

    for l in range(sh.n_layers):
        out["layers"].append(block(l))
    if w.in_kind == IN_BLOCK:
        out["in_block"] = block(IN_BLOCK_LAYER)
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
