"""Comparison rules between the CUDA path and the fp64 oracle.

Tolerances (stated for a bf16-weight, fp32-activation path against fp64):
  logits:  |gpu - ref| <= 3e-2 + 2e-2 * |ref|   (3e-2 absolute / 2e-2 relative)
  tokens:  identical, except that once the oracle's top-1/top-2 logit margin
           at a position is below 1e-2 the two streams may part from there on;
  accept lengths and KV lengths: bit-exact over the steps before the streams part.
"""
from __future__ import annotations

import numpy as np

LOGIT_ATOL = 3e-2
LOGIT_RTOL = 2e-2
MARGIN = 1e-2


def margin(logits: np.ndarray) -> float:
    top2 = np.partition(np.asarray(logits, dtype=np.float64), -2)[-2:]
    return float(top2[1] - top2[0])


def common_prefix(gpu_tokens, ref_tokens, ref_logits) -> int:
    """Length of the prefix that must agree; asserts the first disagreement is excused."""
    n = min(len(gpu_tokens), len(ref_tokens))
    for t in range(n):
        if gpu_tokens[t] != ref_tokens[t]:
            m = margin(ref_logits[t])
            assert m < MARGIN, (f"token {t}: gpu {gpu_tokens[t]} != oracle {ref_tokens[t]} "
                                f"with oracle margin {m:.4g} >= {MARGIN}")
            return t
    assert len(gpu_tokens) == len(ref_tokens), (len(gpu_tokens), len(ref_tokens))
    return n


def assert_logits_close(gpu: np.ndarray, ref: np.ndarray, what: str = "logits") -> float:
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(gpu - ref)
    bound = LOGIT_ATOL + LOGIT_RTOL * np.abs(ref)
    bad = err > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} outside 3e-2 + 2e-2|ref|; "
                           f"max err {err.max():.4g}")
    return float(err.max())


def steps_before(accept_lengths, n_tokens_agreeing: int) -> int:
    """Number of SSD steps whose emitted tokens all lie in the agreeing prefix (first token is the prefill's)."""
    pos, k = 1, 0
    for a in accept_lengths:
        if pos + a + 1 > n_tokens_agreeing:
            break
        pos += a + 1
        k += 1
    return k
