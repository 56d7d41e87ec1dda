"""Prefill lengths around the tile edges of the prefill kernels, against the fp64 oracle.

The prefill GEMM has 128-row tiles and the tensor-core attention 128-query blocks of 64-key steps,
so lengths 1, 63..65, 127..129 and 200 hit an empty-but-one tile, partial key blocks, exact block
ends and a ragged second query block, for head_dim 64 and 128.  A prompt of a single id with no
visual rows is the smallest input.  Checked per length: every layer's K/V rows and the first
token's logits.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_22641_gb300 as lib
import synth
from tests.gpu_util import make_model
from tests.parity import assert_logits_close

pytestmark = pytest.mark.gpu

LENGTHS = [(0, 1), (32, 31), (32, 32), (33, 32), (64, 63), (64, 64), (65, 64), (100, 100)]


@pytest.mark.parametrize("head_dim", [64, 128])
def test_prefill_lengths_match_oracle(head_dim):
    shape = synth.ModelShape(2, 256, 256 // head_dim, head_dim, 512, 2048)
    w0 = synth.TINY.replace(shape=shape, draft_exit_k=1, norm_gain="perturbed", max_new=1)
    bits = synth.make_weights(w0)
    model, _, _ = make_model(w0, bits, gamma_max=4, max_seq=256)
    m = oracle.model_from_bits(w0, bits, synth.bf16_to_f64)
    logits = torch.full((1, shape.vocab), float("nan"), device="cuda")
    try:
        model.set_logits_capture(logits)
        for n_vis, n_prompt in LENGTHS:
            w = w0.replace(n_vis=n_vis, n_prompt=n_prompt)
            vis, prompt = synth.make_inputs(w)
            v = lib.bf16_bits_to_device(vis) if n_vis > 0 else None
            p = torch.from_numpy(prompt.astype(np.int32)).cuda()
            model.prefill(v, p)
            model.sync()
            k, vv, n = model.kv()
            P = n_vis + n_prompt
            assert n == P
            cache = oracle.KVCache(m.cfg, 256)
            ref = oracle.prefill(m, cache, synth.bf16_to_f64(vis).reshape(n_vis, shape.d_model), prompt)
            for got, r in ((k, cache.k), (vv, cache.v)):
                g = got[:, :, :P].float().cpu().numpy()
                r = r[:, :, :P]
                rms = float(np.sqrt(np.mean(r * r)))
                np.testing.assert_allclose(g, r, rtol=1e-3, atol=1e-3 * rms, err_msg=f"P = {P}")
            assert_logits_close(logits[0].cpu().numpy(), np.asarray(ref).reshape(-1, shape.vocab)[-1],
                                f"first token logits, P = {P}")
    finally:
        model.set_logits_capture(None)
        model.close()
