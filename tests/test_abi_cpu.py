"""The C-ABI library builds, loads without a GPU and exports every symbol include/ssd.h declares."""
import ctypes
import os
import re

import pytest

import paper_2510_22641_gb300 as lib
from paper_2510_22641_gb300 import _binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def so():
    path = lib.build()
    return ctypes.CDLL(path), path


def declared():
    txt = open(os.path.join(ROOT, "include", "ssd.h")).read()
    return sorted(set(re.findall(r"^SSD_API [^(]*?\b(ssd_\w+)\(", txt, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared()
    for required in ("ssd_create", "ssd_prefill", "ssd_draft", "ssd_verify", "ssd_generate", "ssd_destroy"):
        assert required in names
    assert sorted(_binding.EXPORTED) == names


def test_every_declared_symbol_is_exported(so):
    dll, path = so
    out = os.popen(f"nm -D --defined-only {path}").read()
    exported = set(re.findall(r" T (ssd_\w+)", out))
    assert set(declared()) <= exported
    for n in declared():
        assert getattr(dll, n)


def test_status_strings_without_gpu(so):
    l = _binding.load()
    assert l.ssd_status_string(0) == b"ok"
    assert l.ssd_status_string(4) == b"KV cache capacity exceeded"
    assert l.ssd_last_error(None) == b"null context"
    assert l.ssd_destroy(None) == 0


def test_create_rejects_bad_arguments_before_touching_the_device(so):
    l = _binding.load()
    ctx = ctypes.c_void_p()
    assert l.ssd_create(None, None, None, ctypes.byref(ctx)) == 1
    cfg = _binding.SSDConfig(n_layers=1, d_model=100, n_heads=1, head_dim=64, d_ff=128, vocab=10,
                             draft_exit_k=1, in_kind=0, in_hidden=0, gamma_max=2, max_seq=16, rms_eps=1e-5,
                             rope_theta=1e4, eos_id=-1)
    w = _binding.SSDWeights()
    assert l.ssd_create(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == 1  # d_model % 64
    assert not ctx.value


def test_draft_length_matches_the_oracle(so):
    """The library's d(t) table (Sec. "Choice of d") equals the oracle's, point by point."""
    import oracle
    l = _binding.load()
    for d0, n_max in [(5, 777), (5, 1000), (5, 4096), (3, 120)]:
        for t in range(0, 2 * n_max + 50):
            assert l.ssd_draft_length(t, d0, n_max) == oracle.draft_length(t, d0, n_max), (t, d0, n_max)
