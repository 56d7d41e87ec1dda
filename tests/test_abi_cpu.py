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


def test_rel_bucket_matches_the_oracle(so):
    """The library's relative-position buckets (encoder-decoder bias tables) equal the oracle's."""
    from oracle import t5_oracle
    l = _binding.load()
    for n, maxd in [(32, 128), (16, 64), (8, 20), (64, 256)]:
        for bidir in (True, False):
            for delta in range(-700, 701):
                assert l.ssd_rel_bucket(delta, int(bidir), n, maxd) == t5_oracle.rel_bucket(delta, bidir, n, maxd), \
                    (delta, bidir, n, maxd)
    assert l.ssd_rel_bucket(0, 1, 7, 128) == -1 and l.ssd_rel_bucket(0, 1, 32, 16) == -1


def _c_layout(tmp_path, structs):
    """offsetof / sizeof of header structs, from a C program compiled against include/ssd.h."""
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "ssd.h"', "int main(void) {"]
    for cname, fields in structs.items():
        lines.append(f'  printf("{cname} size %zu\\n", sizeof({cname}));')
        for f in fields:
            lines.append(f'  printf("{cname} {f} %zu\\n", offsetof({cname}, {f}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    assert os.system(f"gcc -I{os.path.join(ROOT, 'include')} {src} -o {exe}") == 0
    out = {}
    for line in os.popen(str(exe)).read().splitlines():
        a, b, v = line.split()
        out[(a, b)] = int(v)
    return out


def test_ctypes_structs_match_the_header(tmp_path):
    pairs = {"ssd_config": _binding.SSDConfig, "ssd_weights": _binding.SSDWeights,
             "ssd_encdec_weights": _binding.SSDEncDecWeights, "ssd_stats": _binding.SSDStats}
    c = _c_layout(tmp_path, {n: [f for f, _ in t._fields_] for n, t in pairs.items()})
    for n, t in pairs.items():
        assert c[(n, "size")] == ctypes.sizeof(t), n
        for f, _ in t._fields_:
            assert c[(n, f)] == getattr(t, f).offset, (n, f)


def test_create_rejects_bad_encoder_decoder_arguments_before_touching_the_device(so):
    l = _binding.load()
    ctx = ctypes.c_void_p()
    base = dict(n_layers=1, d_model=128, n_heads=1, head_dim=128, d_ff=128, vocab=64, draft_exit_k=1, in_kind=0,
                in_hidden=0, gamma_max=2, max_seq=16, rms_eps=1e-6, rope_theta=0.0, eos_id=-1, n_enc_layers=1,
                max_enc=8, rel_buckets=32, rel_max_distance=128, start_token=0)
    dummy = ctypes.c_void_p(16)   # never dereferenced: every check below runs before any device call
    arr = (ctypes.c_void_p * 1)(16)
    pp = ctypes.cast(arr, _binding._PP)
    w = _binding.SSDWeights(embed=dummy, lm_head=dummy, final_norm=dummy, wq=pp, wk=pp, wv=pp, wo=pp, w_gate=pp,
                            w_up=pp, w_down=pp, attn_norm=pp, ffn_norm=pp, resid_scale=dummy)
    for bad in ({"arch": 7}, {"arch": 1}, {"arch": 1, "rel_buckets": 31}, {"arch": 1, "max_enc": 0},
                {"arch": 1, "start_token": 64}, {"arch": 1, "in_kind": 2}):
        cfg = _binding.SSDConfig(**{**base, **bad})
        assert l.ssd_create(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == 1, bad
        assert not ctx.value
