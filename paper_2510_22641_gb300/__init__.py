"""GB300 (sm_103a) library for greedy self-speculative decoding (FastVLM, arXiv 2510.22641).

The compute lives in libssd.so (hand-written CUDA, C ABI in include/ssd.h);
this package only builds it and marshals arguments.
"""
from . import _binding
from ._binding import (SSD_ARCH_LLAMA, SSD_ARCH_T5, SSD_DLEN_CONTEXT, SSD_DLEN_GENERATED, SSD_FAULT_ALLOC, SSD_FAULT_LAUNCH, SSD_FAULT_NONE, SSD_IN_IDENTITY,
                       SSD_IN_MLP2, SSD_MAX_GAMMA, SSD_OPT_HOST_LOOP, SSD_OPT_PREFILL_ROWS, SSDError, load)
from .build import build

__all__ = ["build", "load", "SSDError", "SSD_ARCH_LLAMA", "SSD_ARCH_T5", "SSD_IN_IDENTITY", "SSD_IN_MLP2",
           "SSD_MAX_GAMMA", "SSD_OPT_HOST_LOOP", "SSD_OPT_PREFILL_ROWS", "SSD_DLEN_CONTEXT", "SSD_DLEN_GENERATED",
           "SSD_FAULT_NONE", "SSD_FAULT_ALLOC",
           "SSD_FAULT_LAUNCH", "SSDModel", "bf16_bits_to_device", "encdec_device_weights", "config_dict",
           "t5_config_dict", "set_fault_injection"]


def set_fault_injection(kind: int, countdown: int) -> None:
    """ssd_set_fault_injection: the countdown-th allocation or launch after this call fails once on
    the host (tests of the error paths; no GPU fault)."""
    load().ssd_set_fault_injection(kind, countdown)


def __getattr__(name):
    # torch is only needed for the model wrapper; the ABI loader works without it.
    if name in ("SSDModel", "bf16_bits_to_device", "encdec_device_weights"):
        from . import model
        return getattr(model, name)
    raise AttributeError(name)


def config_dict(shape, draft_exit_k: int, in_kind: int, in_hidden: int, gamma_max: int, max_seq: int,
                eos_id: int = -1, options: int = 0, max_batch: int = 1) -> dict:
    """ssd_config fields from a model shape (anything with n_layers, d_model, ... attributes)."""
    return {"n_layers": shape.n_layers, "d_model": shape.d_model, "n_heads": shape.n_heads,
            "head_dim": shape.head_dim, "d_ff": shape.d_ff, "vocab": shape.vocab, "draft_exit_k": draft_exit_k,
            "in_kind": in_kind, "in_hidden": in_hidden, "gamma_max": gamma_max, "max_seq": max_seq,
            "rms_eps": shape.rms_eps, "rope_theta": shape.rope_theta, "eos_id": eos_id, "arch": SSD_ARCH_LLAMA,
            "n_enc_layers": 0, "max_enc": 0, "rel_buckets": 0, "rel_max_distance": 0, "start_token": 0,
            "options": options, "max_batch": max_batch}


def t5_config_dict(shape, draft_exit_k: int, in_kind: int, in_hidden: int, gamma_max: int, max_seq: int,
                   max_enc: int, eos_id: int = -1, start_token: int = 0, eps: float = 1e-6, options: int = 0) -> dict:
    """ssd_config fields of the encoder-decoder (T5 v1.1) model from a shape with n_enc, n_dec, d_model,
    n_heads, head_dim, d_ff, vocab, rel_buckets, rel_max_distance attributes."""
    return {"n_layers": shape.n_dec, "d_model": shape.d_model, "n_heads": shape.n_heads,
            "head_dim": shape.head_dim, "d_ff": shape.d_ff, "vocab": shape.vocab, "draft_exit_k": draft_exit_k,
            "in_kind": in_kind, "in_hidden": in_hidden, "gamma_max": gamma_max, "max_seq": max_seq,
            "rms_eps": eps, "rope_theta": 0.0, "eos_id": eos_id, "arch": SSD_ARCH_T5, "n_enc_layers": shape.n_enc,
            "max_enc": max_enc, "rel_buckets": shape.rel_buckets, "rel_max_distance": shape.rel_max_distance,
            "start_token": start_token, "options": options}
