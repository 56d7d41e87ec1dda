"""Prefill at the LLaVA-1.5-13B layer shape (2 layers, 777 prompt rows) against the fp64 oracle.

At this size the prefill GEMMs run their 256-column tiles (q/k/v: 7 row tiles x 60 wide tiles;
gate/up: 7 x 108), which the tiny workloads never reach, and 777 rows leave a ragged last row tile
of 9 rows; the tensor-core attention runs 7 query blocks of 13 key blocks at most.  Checked: both
layers' K/V cache rows and the first token's logits and token.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_22641_gb300 as lib
import synth
from tests.gpu_util import device_weights
from tests.parity import assert_logits_close

pytestmark = pytest.mark.gpu


def test_wide_tile_prefill_matches_oracle():
    base = synth.LLAVA13B_B16.base
    w = base.replace(shape=synth.ModelShape(2, 5120, 40, 128, 13824, 32000), draft_exit_k=1, n_prompt=201,
                     max_new=1)
    bits = synth.make_weights(w)
    dev = device_weights(bits)
    cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, 4, w.prompt_len + 8)
    model = lib.SSDModel(cfg, dev, torch.tensor(w.resid_scale(), device="cuda"),
                         torch.tensor([w.in_scale()], device="cuda"))
    try:
        vis, prompt = synth.make_inputs(w)
        v = lib.bf16_bits_to_device(vis)
        p = torch.from_numpy(prompt.astype(np.int32)).cuda()
        logits = torch.full((1, w.shape.vocab), float("nan"), device="cuda")
        model.set_logits_capture(logits)
        first = torch.zeros(1, dtype=torch.int32, device="cuda")
        model.prefill(v, p, first)
        model.sync()
        k, vv, n = model.kv()
        P = w.prompt_len
        assert n == P == 777
        m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
        cache = oracle.KVCache(m.cfg, P + 8)
        ref_logits = oracle.prefill(m, cache, synth.bf16_to_f64(vis), prompt)
        for got, ref in ((k, cache.k), (vv, cache.v)):
            g = got[:, :, :P].float().cpu().numpy()
            r = ref[:, :, :P]
            rms = float(np.sqrt(np.mean(r * r)))
            np.testing.assert_allclose(g, r, rtol=1e-3, atol=1e-3 * rms)
        ref_row = np.asarray(ref_logits).reshape(-1, w.shape.vocab)[-1]
        assert_logits_close(logits[0].cpu().numpy(), ref_row, "first token logits")
        top = np.sort(ref_row)
        if top[-1] - top[-2] >= 1e-2:
            assert int(first.item()) == int(np.argmax(ref_row))
    finally:
        model.set_logits_capture(None)
        model.close()
