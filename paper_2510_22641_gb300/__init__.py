"""GB300 (sm_103a) library for greedy self-speculative decoding (FastVLM, arXiv 2510.22641).

The compute lives in libssd.so (hand-written CUDA, C ABI in include/ssd.h);
this package only builds it and marshals arguments.
"""
from . import _binding
from ._binding import SSD_IN_IDENTITY, SSD_IN_MLP2, SSD_MAX_GAMMA, SSDError, load
from .build import build

__all__ = ["build", "load", "SSDError", "SSD_IN_IDENTITY", "SSD_IN_MLP2", "SSD_MAX_GAMMA", "SSDModel",
           "bf16_bits_to_device", "config_dict"]


def __getattr__(name):
    # torch is only needed for the model wrapper; the ABI loader works without it.
    if name in ("SSDModel", "bf16_bits_to_device"):
        from . import model
        return getattr(model, name)
    raise AttributeError(name)


def config_dict(shape, draft_exit_k: int, in_kind: int, in_hidden: int, gamma_max: int, max_seq: int,
                eos_id: int = -1) -> dict:
    """ssd_config fields from a model shape (anything with n_layers, d_model, ... attributes)."""
    return {"n_layers": shape.n_layers, "d_model": shape.d_model, "n_heads": shape.n_heads,
            "head_dim": shape.head_dim, "d_ff": shape.d_ff, "vocab": shape.vocab, "draft_exit_k": draft_exit_k,
            "in_kind": in_kind, "in_hidden": in_hidden, "gamma_max": gamma_max, "max_seq": max_seq,
            "rms_eps": shape.rms_eps, "rope_theta": shape.rope_theta, "eos_id": eos_id}
