"""Comparison rules between the CUDA path and the fp64 oracle.

Tolerances (stated for a bf16-weight, fp32-activation path against fp64):
  logits:  |gpu - ref| <= 3e-2 + 2e-2 * |ref|   (3e-2 absolute / 2e-2 relative)
  tokens:  identical, except that once the oracle's top-1/top-2 logit margin
           at a position is below 1e-2 the two streams may part from there on;
  accept lengths and KV lengths: bit-exact over the steps before the streams part;
  draft logits g(I(x_k)): the same logit tolerance for every draft row of those steps up to the
           first draft whose token differs, which must sit at an oracle draft margin below 1e-2.
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


def assert_step_log(accepted, drafted, ref, n_tokens_agreeing: int) -> int:
    """The device's per-step (a, gamma_eff) record equals the oracle's accept lengths and draft
    counts over every step before the streams part (all steps when they never part)."""
    k = steps_before(ref.accept_lengths, n_tokens_agreeing)
    if n_tokens_agreeing == len(ref.tokens):
        k = len(ref.accept_lengths)
        assert len(accepted) == k, (len(accepted), k)
    assert list(accepted[:k]) == list(ref.accept_lengths[:k]), (accepted[:k], ref.accept_lengths[:k])
    assert list(drafted[:k]) == [len(d) for d in ref.draft_tokens[:k]]
    return k


def assert_draft_logits(draft_logits: np.ndarray, ref, n_steps: int) -> int:
    """draft_logits[s][j]: the GPU's g(I(x_k)) of draft j in step s.  For the first n_steps steps,
    every draft row the oracle computed is compared at the logit tolerance until the first draft
    token that differs (argmax of the GPU row vs the oracle's d_{j+1}); that one must be a near-tie
    of the oracle's draft logits, after which the step's later drafts see other inputs.  Returns
    the number of rows compared."""
    rows = 0
    for s in range(n_steps):
        for j, ref_row in enumerate(ref.draft_logits[s]):
            assert_logits_close(draft_logits[s][j], ref_row, f"draft logits of step {s} row {j}")
            rows += 1
            if int(np.argmax(draft_logits[s][j])) != ref.draft_tokens[s][j]:
                m = margin(ref_row)
                assert m < MARGIN, f"draft {j} of step {s} differs at oracle margin {m:.4g}"
                break
    return rows
