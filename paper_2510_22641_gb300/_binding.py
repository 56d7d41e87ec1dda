"""ctypes binding of libssd.so: argument marshalling only.

Every computation happens in the CUDA library; this module converts Python
and torch objects to the C ABI of include/ssd.h.  There is no fallback: if the
library is missing or fails to load, loading raises.
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libssd.so")

SSD_MAX_GAMMA = 15
SSD_MAX_ROWS = 16
SSD_IN_IDENTITY = 0
SSD_IN_MLP2 = 1
SSD_IN_BLOCK = 2
SSD_ARCH_LLAMA = 0
SSD_ARCH_T5 = 1
SSD_OPT_HOST_LOOP = 1
SSD_OPT_PREFILL_ROWS = 2
SSD_DLEN_CONTEXT = 0
SSD_DLEN_GENERATED = 1
SSD_FAULT_NONE = 0
SSD_FAULT_ALLOC = 1
SSD_FAULT_LAUNCH = 2

STATUS = {0: "SSD_OK", 1: "SSD_ERR_INVALID_ARG", 2: "SSD_ERR_OOM", 3: "SSD_ERR_CUDA", 4: "SSD_ERR_CAPACITY",
          5: "SSD_ERR_STATE", 6: "SSD_ERR_TIMEOUT", 7: "SSD_ERR_DEVICE", 8: "SSD_ERR_UNSUPPORTED"}

EXPORTED = ("ssd_create", "ssd_destroy", "ssd_prefill", "ssd_draft", "ssd_verify", "ssd_decode", "ssd_decode_dynamic",
            "ssd_draft_length", "ssd_rel_bucket",
            "ssd_greedy_decode", "ssd_generate", "ssd_greedy_generate", "ssd_sync", "ssd_get_stats",
            "ssd_set_logits_capture", "ssd_set_draft_logits_capture", "ssd_get_step_log", "ssd_get_kv",
            "ssd_last_launch_count", "ssd_prefill_batch", "ssd_decode_batch", "ssd_greedy_decode_batch",
            "ssd_generate_batch", "ssd_get_batch_stats", "ssd_get_batch_step_log", "ssd_lm_head",
            "ssd_lm_head_static", "ssd_profile_projection", "ssd_set_fault_injection", "ssd_probe_bounded_wait",
            "ssd_status_string", "ssd_last_error")


class SSDConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("d_ff", ctypes.c_int), ("vocab", ctypes.c_int),
                ("draft_exit_k", ctypes.c_int), ("in_kind", ctypes.c_int), ("in_hidden", ctypes.c_int),
                ("gamma_max", ctypes.c_int), ("max_seq", ctypes.c_int), ("rms_eps", ctypes.c_float),
                ("rope_theta", ctypes.c_float), ("eos_id", ctypes.c_int), ("arch", ctypes.c_int),
                ("n_enc_layers", ctypes.c_int), ("max_enc", ctypes.c_int), ("rel_buckets", ctypes.c_int),
                ("rel_max_distance", ctypes.c_int), ("start_token", ctypes.c_int), ("options", ctypes.c_int),
                ("max_batch", ctypes.c_int)]


_PP = ctypes.POINTER(ctypes.c_void_p)

ENCDEC_ARRAYS = ("cq", "ck", "cv", "co", "cross_norm", "enc_wq", "enc_wk", "enc_wv", "enc_wo", "enc_wi0", "enc_wi1",
                 "enc_wff", "enc_attn_norm", "enc_ffn_norm")


class SSDEncDecWeights(ctypes.Structure):
    _fields_ = [(n, _PP) for n in ENCDEC_ARRAYS] + [("enc_final", ctypes.c_void_p), ("enc_rel", ctypes.c_void_p),
                                                    ("dec_rel", ctypes.c_void_p)]


class SSDWeights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("lm_head", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("wq", _PP), ("wk", _PP), ("wv", _PP), ("wo", _PP), ("w_gate", _PP), ("w_up", _PP),
                ("w_down", _PP), ("attn_norm", _PP), ("ffn_norm", _PP),
                ("in_norm", ctypes.c_void_p), ("in_w1", ctypes.c_void_p), ("in_w2", ctypes.c_void_p),
                ("resid_scale", ctypes.c_void_p), ("in_scale", ctypes.c_void_p), ("in_block", _PP),
                ("encdec", ctypes.POINTER(SSDEncDecWeights))]


class SSDStats(ctypes.Structure):
    _fields_ = [("steps", ctypes.c_int64), ("drafted", ctypes.c_int64), ("accepted", ctypes.c_int64),
                ("emitted", ctypes.c_int64), ("accept_hist", ctypes.c_int64 * (SSD_MAX_GAMMA + 1)),
                ("kv_len", ctypes.c_int64)]

    def as_dict(self) -> dict:
        return {"steps": self.steps, "drafted": self.drafted, "accepted": self.accepted, "emitted": self.emitted,
                "accept_hist": list(self.accept_hist), "kv_len": self.kv_len}


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libssd.so (raises OSError if it is missing: there is no CPU fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise OSError(f"{path} not found: build it with paper_2510_22641_gb300.build.build()")
    lib = ctypes.CDLL(path)
    i32, vp, pi32 = ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p
    sig = {
        "ssd_create": [ctypes.POINTER(SSDConfig), ctypes.POINTER(SSDWeights), vp, ctypes.POINTER(vp)],
        "ssd_destroy": [vp],
        "ssd_prefill": [vp, vp, i32, pi32, i32, pi32],
        "ssd_draft": [vp, i32, pi32],
        "ssd_verify": [vp, i32, pi32, pi32],
        "ssd_decode": [vp, i32, i32, pi32, pi32],
        "ssd_decode_dynamic": [vp, i32, i32, i32, i32, i32, pi32, pi32],
        "ssd_greedy_decode": [vp, i32, pi32, pi32],
        "ssd_generate": [vp, vp, i32, vp, i32, i32, i32, vp, ctypes.POINTER(i32), ctypes.POINTER(SSDStats)],
        "ssd_greedy_generate": [vp, vp, i32, vp, i32, i32, vp, ctypes.POINTER(i32), ctypes.POINTER(SSDStats)],
        "ssd_sync": [vp],
        "ssd_get_stats": [vp, ctypes.POINTER(SSDStats)],
        "ssd_set_logits_capture": [vp, vp, i32],
        "ssd_set_draft_logits_capture": [vp, vp, i32],
        "ssd_get_step_log": [vp, vp, vp, i32, ctypes.POINTER(i32)],
        "ssd_get_kv": [vp, ctypes.POINTER(vp), ctypes.POINTER(vp), ctypes.POINTER(i32)],
        "ssd_last_launch_count": [vp, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)],
        "ssd_profile_projection": [vp, i32, i32, i32, i32, ctypes.POINTER(ctypes.c_int64)],
        "ssd_prefill_batch": [vp, i32, vp, vp, vp, vp, pi32],
        "ssd_decode_batch": [vp, i32, i32, pi32, pi32],
        "ssd_greedy_decode_batch": [vp, i32, pi32, pi32],
        "ssd_generate_batch": [vp, i32, vp, vp, vp, vp, i32, i32, vp, vp],
        "ssd_get_batch_stats": [vp, i32, ctypes.POINTER(SSDStats)],
        "ssd_get_batch_step_log": [vp, i32, vp, vp, i32, ctypes.POINTER(i32)],
        "ssd_lm_head": [vp, vp, i32, vp, vp],
        "ssd_probe_bounded_wait": [vp, ctypes.c_int64],
        "ssd_lm_head_static": [vp, vp, vp, i32, i32, i32, ctypes.c_float, vp, vp, vp],
    }
    for name, args in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = ctypes.c_int
    lib.ssd_set_fault_injection.argtypes = [ctypes.c_int, ctypes.c_int]
    lib.ssd_set_fault_injection.restype = None
    lib.ssd_draft_length.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int]
    lib.ssd_draft_length.restype = ctypes.c_int
    lib.ssd_rel_bucket.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int]
    lib.ssd_rel_bucket.restype = ctypes.c_int
    lib.ssd_status_string.argtypes = [ctypes.c_int]
    lib.ssd_status_string.restype = ctypes.c_char_p
    lib.ssd_last_error.argtypes = [vp]
    lib.ssd_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


class SSDError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status
