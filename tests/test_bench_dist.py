"""The multi-rank (replica) path of bench.py on CPU: world_size 2 over gloo.

Each rank reports its own elapsed time; the job's time is the slowest rank's
and the value counts the tokens of every rank (weak scaling)."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = 1000.0 + 500.0 * rank                      # rank 1 is slower
    m = bench.reduce_max(ms, dist, device="cpu")
    out[rank] = (m, bench.whole_job_tokens_per_s(world, steps=4, tokens_per_step=128, max_ms=m))
    dist.destroy_process_group()


def test_replicas_take_the_slowest_rank_and_count_all_tokens():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 1500.0
    assert res[0][1] == pytest.approx(2 * 4 * 128 / 1.5)


def test_single_process_needs_no_process_group():
    assert bench.reduce_max(12.5) == 12.5
    assert bench.whole_job_tokens_per_s(1, 10, 128, 2000.0) == pytest.approx(640.0)


def test_encoder_decoder_oracle_sample_on_the_tiny_model():
    """bench.py --encdec's CPU leg: the encoder-decoder oracle timed over a bounded number of steps."""
    import synth
    w = synth.T5_TINY.replace(s=0.3)
    bits = synth.make_t5_weights(w)
    q, prompt = synth.make_t5_inputs(w)
    r = bench.oracle_sample_encdec(w, bits, q, prompt, max_steps=3)
    assert r["n_steps"] == 3 and r["prefill_s"] > 0 and r["step_s"] > 0
    assert 1.0 <= r["tokens_per_step"] <= w.gamma + 1
    assert r["decode_tok_s"] == pytest.approx(r["tokens_per_step"] / r["step_s"])


def test_decoder_oracle_sample_on_the_tiny_model():
    """bench.py's cpu_baseline / --impl reference leg: prefill plus bounded SSD steps of the oracle."""
    import synth
    w = synth.TINY.replace(s=0.3)
    bits = synth.make_weights(w)
    vis, prompt = synth.make_inputs(w)
    r = bench.oracle_sample(w, bits, vis, prompt, max_steps=3, warm_steps=1)
    assert r["n_steps"] == 3 and r["prefill_s"] > 0 and r["step_s"] > 0
    assert 1.0 <= r["tokens_per_step"] <= w.gamma + 1
    request_s = r["prefill_s"] + (w.max_new - 1) / r["tokens_per_step"] * r["step_s"]
    assert r["value"] == pytest.approx(w.max_new / request_s)
