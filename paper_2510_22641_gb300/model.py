"""Python face of the SSD library: owns torch device copies of the weights and
forwards every call to the C ABI (include/ssd.h).  No computation happens here.
"""
from __future__ import annotations

import ctypes

import numpy as np
import torch

from . import _binding as B


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def bf16_bits_to_device(bits: np.ndarray, device="cuda") -> torch.Tensor:
    """Upload bf16 bit patterns (numpy uint16) as a torch.bfloat16 device tensor."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


_ENCDEC_RENAME = {"wq": "wq", "wk": "wk", "wv": "wv", "wo": "wo", "wi0": "w_gate", "wi1": "w_up", "wff": "w_down",
                  "ffn_norm": "ffn_norm"}


def encdec_device_weights(bits: dict, device="cuda") -> dict:
    """Upload an encoder-decoder model given as bf16 bit arrays in T5 naming -- {"embed", "lm_head",
    "enc_final", "dec_final", "enc_rel", "dec_rel", "enc": [{wq, wk, wv, wo, attn_norm, wi0, wi1, wff,
    ffn_norm}], "dec": [{... + self_norm, cq, ck, cv, co, cross_norm}], optional "in_norm", "in_w1",
    "in_w2"} -- into the weights dict SSDModel takes for SSD_ARCH_T5."""
    up = lambda a: bf16_bits_to_device(a, device)

    def stack(lw, norm):
        d = {_ENCDEC_RENAME[n]: up(a) for n, a in lw.items() if n in _ENCDEC_RENAME}
        d["attn_norm"] = up(lw[norm])
        return d

    out = {"embed": up(bits["embed"]), "lm_head": up(bits["lm_head"]), "final_norm": up(bits["dec_final"]),
           "layers": [stack(lw, "self_norm") for lw in bits["dec"]],
           "encdec": {"cross": [{n: up(lw[n]) for n in ("cq", "ck", "cv", "co", "cross_norm")} for lw in bits["dec"]],
                      "enc": [stack(lw, "attn_norm") for lw in bits["enc"]], "enc_final": up(bits["enc_final"]),
                      "enc_rel": up(bits["enc_rel"]), "dec_rel": up(bits["dec_rel"])}}
    for k in ("in_norm", "in_w1", "in_w2"):
        if k in bits:
            out[k] = up(bits[k])
    return out


class _DeviceArray:
    """Minimal __cuda_array_interface__ holder to view library-owned memory from torch."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr, "data": (ptr, False),
                                         "version": 3, "strides": None}


def _device_view(ptr: int, shape) -> torch.Tensor:
    return torch.as_tensor(_DeviceArray(ptr, shape, "<f4"), device="cuda")


class SSDModel:
    """One library context (ssd_ctx) over borrowed device weights.

    weights: dict with bf16 device tensors "embed", "lm_head", "final_norm",
    "layers" (list of dicts wq, wk, wv, wo, w_gate, w_up, w_down, attn_norm,
    ffn_norm) and, for the MLP2 imitation network, "in_norm", "in_w1", "in_w2"; for the block
    imitation network "in_block" (a dict like a layer's).
    resid_scale: fp32 device tensor [n_layers]; in_scale: fp32 device tensor [1].
    Encoder-decoder model (cfg["arch"] == SSD_ARCH_T5): "layers" and "final_norm" are the decoder's
    (w_gate / w_up / w_down = wi_0 / wi_1 / wo of its gated-GELU MLP), and weights["encdec"] holds
    "cross" (list of dicts cq, ck, cv, co, cross_norm per decoder layer), "enc" (list of dicts like a
    layer's), "enc_final", "enc_rel", "dec_rel".
    """

    def __init__(self, cfg: dict, weights: dict, resid_scale: torch.Tensor, in_scale: torch.Tensor,
                 stream: torch.cuda.Stream | None = None):
        self.lib = B.load()
        self.cfg = dict(cfg)
        self.weights = weights            # keep the borrowed tensors alive
        self.resid_scale = resid_scale
        self.in_scale = in_scale
        c = B.SSDConfig(**{k: self.cfg.get(k, 0) for k, _ in B.SSDConfig._fields_})
        L = cfg["n_layers"]
        arrs = {}
        for name in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down", "attn_norm", "ffn_norm"):
            arrs[name] = (ctypes.c_void_p * L)(*[weights["layers"][l][name].data_ptr() for l in range(L)])
        if "in_block" in weights:
            names = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down", "attn_norm", "ffn_norm")
            arrs["in_block"] = (ctypes.c_void_p * 9)(*[weights["in_block"][n].data_ptr() for n in names])
        encdec = None
        if self.cfg.get("arch", 0) == B.SSD_ARCH_T5:
            ed = weights["encdec"]
            E = cfg["n_enc_layers"]
            for n in ("cq", "ck", "cv", "co", "cross_norm"):
                arrs["x_" + n] = (ctypes.c_void_p * L)(*[ed["cross"][l][n].data_ptr() for l in range(L)])
            enc_names = {"enc_wq": "wq", "enc_wk": "wk", "enc_wv": "wv", "enc_wo": "wo", "enc_wi0": "w_gate",
                         "enc_wi1": "w_up", "enc_wff": "w_down", "enc_attn_norm": "attn_norm",
                         "enc_ffn_norm": "ffn_norm"}
            for cn, n in enc_names.items():
                arrs["x_" + cn] = (ctypes.c_void_p * E)(*[ed["enc"][e][n].data_ptr() for e in range(E)])
            encdec = B.SSDEncDecWeights(enc_final=_ptr(ed["enc_final"]), enc_rel=_ptr(ed["enc_rel"]),
                                        dec_rel=_ptr(ed["dec_rel"]),
                                        **{n: ctypes.cast(arrs["x_" + n], B._PP) for n in B.ENCDEC_ARRAYS})
            self._encdec = encdec
        self._arrs = arrs
        w = B.SSDWeights(embed=_ptr(weights["embed"]), lm_head=_ptr(weights["lm_head"]),
                         final_norm=_ptr(weights["final_norm"]),
                         in_norm=_ptr(weights.get("in_norm")), in_w1=_ptr(weights.get("in_w1")),
                         in_w2=_ptr(weights.get("in_w2")), resid_scale=_ptr(resid_scale),
                         in_scale=_ptr(in_scale),
                         encdec=ctypes.pointer(encdec) if encdec is not None else None,
                         **{k: ctypes.cast(v, B._PP) for k, v in arrs.items() if not k.startswith("x_")})
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        ctx = ctypes.c_void_p()
        self._check(self.lib.ssd_create(ctypes.byref(c), ctypes.byref(w), self.stream.cuda_stream,
                                        ctypes.byref(ctx)), None)
        self.ctx = ctx

    # ------------------------------------------------------------------ plumbing
    def _check(self, status: int, ctx) -> None:
        if status != 0:
            msg = self.lib.ssd_last_error(ctx).decode() if ctx else B.STATUS.get(status, "")
            raise B.SSDError(status, msg)

    def _call(self, name: str, *args) -> None:
        self._check(getattr(self.lib, name)(self.ctx, *args), self.ctx)

    def close(self) -> None:
        if getattr(self, "ctx", None):
            self.lib.ssd_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------------ device-buffer calls (async)
    def prefill(self, vis: torch.Tensor | None, prompt: torch.Tensor, first_tok: torch.Tensor | None = None):
        n_vis = 0 if vis is None else vis.shape[0]
        self._call("ssd_prefill", _ptr(vis), n_vis, _ptr(prompt), prompt.shape[0], _ptr(first_tok))

    def draft(self, gamma: int, draft_tok: torch.Tensor | None = None):
        self._call("ssd_draft", gamma, _ptr(draft_tok))

    def verify(self, gamma: int, n_emitted: torch.Tensor | None = None, emitted: torch.Tensor | None = None):
        self._call("ssd_verify", gamma, _ptr(n_emitted), _ptr(emitted))

    def decode(self, max_new: int, gamma: int, out_tok: torch.Tensor | None = None,
               n_out: torch.Tensor | None = None):
        self._call("ssd_decode", max_new, gamma, _ptr(out_tok), _ptr(n_out))

    def decode_dynamic(self, max_new: int, d0: int, n_max: int, gamma_cap: int, out_tok: torch.Tensor | None = None,
                       n_out: torch.Tensor | None = None, t_from: int = B.SSD_DLEN_CONTEXT):
        """SSD with the dynamic draft length d(t) (Sec. "Choice of d"), capped at gamma_cap; t counted
        over the whole context (SSD_DLEN_CONTEXT) or over the generated tokens (SSD_DLEN_GENERATED)."""
        self._call("ssd_decode_dynamic", max_new, d0, n_max, t_from, gamma_cap, _ptr(out_tok), _ptr(n_out))

    def greedy_decode(self, max_new: int, out_tok: torch.Tensor | None = None, n_out: torch.Tensor | None = None):
        self._call("ssd_greedy_decode", max_new, _ptr(out_tok), _ptr(n_out))

    # ------------------------------------------------------------------ host-buffer calls (sync)
    def _generate(self, name, vis: np.ndarray | torch.Tensor | None, prompt, max_new: int, *extra):
        vis_p, n_vis = None, 0
        if vis is not None:
            n_vis = vis.shape[0]
            vis_p = vis.data_ptr() if isinstance(vis, torch.Tensor) else vis.ctypes.data
        prompt_arr = prompt if isinstance(prompt, torch.Tensor) else np.ascontiguousarray(prompt, dtype=np.int32)
        pp = prompt_arr.data_ptr() if isinstance(prompt_arr, torch.Tensor) else prompt_arr.ctypes.data
        out = np.zeros(max_new, dtype=np.int32)
        n = ctypes.c_int(0)
        st = B.SSDStats()
        self._call(name, vis_p, n_vis, pp, len(prompt_arr), max_new, *extra, out.ctypes.data, ctypes.byref(n),
                   ctypes.byref(st))
        return out[:n.value].tolist(), st.as_dict()

    def generate(self, vis, prompt, max_new: int, gamma: int):
        """ssd_generate: host inputs in, host tokens + stats out."""
        return self._generate("ssd_generate", vis, prompt, max_new, gamma)

    def greedy_generate(self, vis, prompt, max_new: int):
        return self._generate("ssd_greedy_generate", vis, prompt, max_new)

    # ------------------------------------------------------------------ inspection
    def sync(self):
        self._call("ssd_sync")

    def stats(self) -> dict:
        st = B.SSDStats()
        self._call("ssd_get_stats", ctypes.byref(st))
        return st.as_dict()

    def set_logits_capture(self, buf: torch.Tensor | None):
        """buf: device fp32 [max_rows][vocab], or [batch][max_rows][vocab] for batched requests."""
        self._call("ssd_set_logits_capture", _ptr(buf), 0 if buf is None else buf.shape[-2])

    def set_draft_logits_capture(self, buf: torch.Tensor | None):
        """buf: device fp32 [max_steps][gamma_max][vocab] (draft j of step s writes buf[s][j]), or
        [batch][max_steps][gamma_max][vocab] for batched requests."""
        self._call("ssd_set_draft_logits_capture", _ptr(buf), 0 if buf is None else buf.shape[-3])

    def step_log(self, cap: int = 4096) -> tuple[list, list]:
        """(accepted a, drafted gamma_eff) of every step since the last prefill."""
        acc = np.zeros(cap, dtype=np.int32)
        dr = np.zeros(cap, dtype=np.int32)
        n = ctypes.c_int(0)
        self._call("ssd_get_step_log", acc.ctypes.data, dr.ctypes.data, cap, ctypes.byref(n))
        m = min(n.value, cap)
        return acc[:m].tolist(), dr[:m].tolist()

    def kv(self):
        """(K, V, kv_len): zero-copy torch views [L][H][max_seq][Dh] (fp32) of the library's cache
        ([L + 1] with the block imitation network, whose rows are slot L; [L][max_batch][H][max_seq][Dh]
        for a ctx with max_batch > 1)."""
        k, v, n = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_int()
        self._call("ssd_get_kv", ctypes.byref(k), ctypes.byref(v), ctypes.byref(n))
        c = self.cfg
        slots = c["n_layers"] + (1 if c["in_kind"] == B.SSD_IN_BLOCK else 0)
        shape = (slots, c["n_heads"], c["max_seq"], c["head_dim"])
        if c.get("max_batch", 1) > 1:
            shape = (slots, c["max_batch"], c["n_heads"], c["max_seq"], c["head_dim"])
        return _device_view(k.value, shape), _device_view(v.value, shape), n.value

    def lm_head(self, x: torch.Tensor, tok: torch.Tensor, logits: torch.Tensor | None = None):
        """ssd_lm_head: argmax of W_lm RMSNorm_f(x) per row (x fp32 [rows][d_model] on the device)."""
        self._call("ssd_lm_head", x.data_ptr(), x.shape[0], tok.data_ptr(), _ptr(logits))

    PROJECTIONS = {"qkv": 0, "o": 1, "gateup": 2, "down": 3, "head": 4, "in1": 5, "in2": 6, "attn": 7}

    def profile_projection(self, which: str, layer: int = 0, rows: int = 1, reps: int = 1) -> int:
        """Enqueue reps launches of one projection kernel; returns algorithmic bytes per launch."""
        b = ctypes.c_int64()
        self._call("ssd_profile_projection", self.PROJECTIONS[which], layer, rows, reps, ctypes.byref(b))
        return b.value

    # ------------------------------------------------------------------ batched requests
    def prefill_batch(self, vis: torch.Tensor | None, n_vis, prompt: torch.Tensor, n_prompt,
                      first_tok: torch.Tensor | None = None):
        """ssd_prefill_batch: vis bf16 [sum n_vis][d] and prompt int32 [sum n_prompt] on the device, the
        requests' rows concatenated in order; n_vis / n_prompt: per-request counts (host)."""
        nv = np.ascontiguousarray(n_vis, dtype=np.int32)
        npr = np.ascontiguousarray(n_prompt, dtype=np.int32)
        self._call("ssd_prefill_batch", len(nv), _ptr(vis), nv.ctypes.data, _ptr(prompt), npr.ctypes.data,
                   _ptr(first_tok))

    def decode_batch(self, max_new: int, gamma: int, out_tok: torch.Tensor | None = None,
                     n_out: torch.Tensor | None = None):
        """ssd_decode_batch: out_tok int32 [B][max_new], n_out int32 [B] on the device."""
        self._call("ssd_decode_batch", max_new, gamma, _ptr(out_tok), _ptr(n_out))

    def greedy_decode_batch(self, max_new: int, out_tok: torch.Tensor | None = None,
                            n_out: torch.Tensor | None = None):
        self._call("ssd_greedy_decode_batch", max_new, _ptr(out_tok), _ptr(n_out))

    def generate_batch(self, vis: np.ndarray | None, n_vis, prompt: np.ndarray, n_prompt, max_new: int,
                       gamma: int) -> list:
        """ssd_generate_batch with host buffers (vis: bf16 bit patterns [sum n_vis][d], prompt int32);
        gamma = 0 decodes greedily.  Returns each request's tokens."""
        nv = np.ascontiguousarray(n_vis, dtype=np.int32)
        npr = np.ascontiguousarray(n_prompt, dtype=np.int32)
        pr = np.ascontiguousarray(prompt, dtype=np.int32)
        vp = None if vis is None else np.ascontiguousarray(vis)
        out = np.zeros((len(nv), max_new), dtype=np.int32)
        n = np.zeros(len(nv), dtype=np.int32)
        self._call("ssd_generate_batch", len(nv), None if vp is None else vp.ctypes.data, nv.ctypes.data,
                   pr.ctypes.data, npr.ctypes.data, max_new, gamma, out.ctypes.data, n.ctypes.data)
        return [out[b, :n[b]].tolist() for b in range(len(nv))]

    def batch_stats(self, b: int) -> dict:
        st = B.SSDStats()
        self._call("ssd_get_batch_stats", b, ctypes.byref(st))
        return st.as_dict()

    def batch_step_log(self, b: int, cap: int = 4096) -> tuple[list, list]:
        acc = np.zeros(cap, dtype=np.int32)
        dr = np.zeros(cap, dtype=np.int32)
        n = ctypes.c_int(0)
        self._call("ssd_get_batch_step_log", b, acc.ctypes.data, dr.ctypes.data, cap, ctypes.byref(n))
        m = min(n.value, cap)
        return acc[:m].tolist(), dr[:m].tolist()

    def probe_bounded_wait(self, limit_ns: int):
        """ssd_probe_bounded_wait: one device wait runs out after limit_ns; the next sync reports it."""
        self._call("ssd_probe_bounded_wait", limit_ns)

    def launch_counts(self) -> tuple[int, int]:
        a, b = ctypes.c_int64(), ctypes.c_int64()
        self._call("ssd_last_launch_count", ctypes.byref(a), ctypes.byref(b))
        return a.value, b.value
