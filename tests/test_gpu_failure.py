"""Failure paths, made without a GPU fault: an allocation that fails (injected on the host), a kernel
launch that fails (injected on the host), and a bounded device wait that runs out.  After each, the
library reports the documented status and keeps working."""
import numpy as np
import pytest

import oracle
import paper_2510_22641_gb300 as lib
import synth
from tests.gpu_util import device_inputs, make_model

pytestmark = pytest.mark.gpu

W = synth.TINY.replace(s=0.2, max_new=16)


@pytest.fixture(scope="module")
def bits():
    return synth.make_weights(W)


@pytest.fixture(scope="module")
def ref_tokens(bits):
    m = oracle.model_from_bits(W, bits, synth.bf16_to_f64)
    vis, prompt = synth.make_inputs(W)
    r = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, W.max_new, W.gamma)
    return r.tokens


def generate(model, n_prompt=None):
    vis, prompt = synth.make_inputs(W)
    if n_prompt is not None:
        prompt = prompt[:n_prompt]
    toks, _ = model.generate(vis, prompt, W.max_new, W.gamma)
    return toks


def test_injected_allocation_failure_reports_oom(bits, ref_tokens):
    lib.set_fault_injection(lib.SSD_FAULT_ALLOC, 6)
    try:
        with pytest.raises(lib.SSDError) as e:
            make_model(W, bits)
        assert e.value.status == 2  # SSD_ERR_OOM
    finally:
        lib.set_fault_injection(lib.SSD_FAULT_NONE, 0)
    model, _, _ = make_model(W, bits)  # the injected fault fired once; a new ctx is whole
    try:
        assert generate(model) == ref_tokens
    finally:
        model.close()


def test_injected_launch_failure_reports_cuda_error_and_ctx_recovers(bits, ref_tokens):
    model, _, _ = make_model(W, bits)
    try:
        assert generate(model) == ref_tokens
        # a prefill of a new prompt length captures a new graph: its 12th launch fails
        lib.set_fault_injection(lib.SSD_FAULT_LAUNCH, 12)
        try:
            with pytest.raises(lib.SSDError) as e:
                generate(model, n_prompt=W.n_prompt - 3)
            assert e.value.status == 3  # SSD_ERR_CUDA
        finally:
            lib.set_fault_injection(lib.SSD_FAULT_NONE, 0)
        assert generate(model) == ref_tokens
        short = generate(model, n_prompt=W.n_prompt - 3)
        assert len(short) == W.max_new
    finally:
        model.close()


def test_bounded_wait_runs_out_and_reports_timeout(bits, ref_tokens):
    model, _, _ = make_model(W, bits)
    try:
        model.probe_bounded_wait(50_000)  # 50 us
        with pytest.raises(lib.SSDError) as e:
            model.sync()
        assert e.value.status == 6  # SSD_ERR_TIMEOUT
        with pytest.raises(lib.SSDError) as e:  # no decode without a prefill after the timeout
            model.decode(W.max_new, W.gamma)
        assert e.value.status == 5
        assert generate(model) == ref_tokens  # the prefill clears the error word
        model.sync()
    finally:
        model.close()
