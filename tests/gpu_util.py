"""Builds a library context for a synthetic workload (device weights from synth)."""
from __future__ import annotations

import numpy as np
import torch

import paper_2510_22641_gb300 as lib
import synth


def device_weights(bits: dict) -> dict:
    up = lib.bf16_bits_to_device
    out = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm")}
    out["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
    if "in_block" in bits:
        out["in_block"] = {n: up(a) for n, a in bits["in_block"].items()}
    for k in ("in_norm", "in_w1", "in_w2"):
        if k in bits:
            out[k] = up(bits[k])
    return out


def make_model(w: synth.Workload, bits: dict | None = None, dev: dict | None = None, gamma_max: int | None = None,
               max_seq: int | None = None, options: int = 0, max_batch: int = 1):
    bits = bits if bits is not None else synth.make_weights(w)
    dev = dev if dev is not None else device_weights(bits)
    cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, gamma_max or max(w.gamma, 1),
                          max_seq or w.max_seq(), w.eos_id, options=options, max_batch=max_batch)
    rs = torch.tensor(w.resid_scale(), dtype=torch.float32, device="cuda")
    ins = torch.tensor([w.in_scale()], dtype=torch.float32, device="cuda")
    return lib.SSDModel(cfg, dev, rs, ins), bits, dev


def device_inputs(w: synth.Workload, seed: int | None = None):
    vis, prompt = synth.make_inputs(w, seed)
    v = lib.bf16_bits_to_device(vis) if w.n_vis > 0 else None
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    return vis, prompt, v, p


def batch_device_inputs(bw: synth.BatchWorkload, seed: int | None = None):
    """The batch's per-request inputs (host) and their concatenated device copies with the counts."""
    ins = synth.make_batch_inputs(bw, seed)
    nv = [v.shape[0] for v, _ in ins]
    npr = [len(p) for _, p in ins]
    vis = np.concatenate([v for v, _ in ins]) if sum(nv) else None
    dv = lib.bf16_bits_to_device(vis) if vis is not None else None
    dp = torch.from_numpy(np.concatenate([p for _, p in ins]).astype(np.int32)).cuda()
    return ins, dv, nv, dp, npr


def t5_device_weights(bits: dict) -> dict:
    """Device copies of a synth encoder-decoder workload in the layout lib.SSDModel takes."""
    return lib.encdec_device_weights(bits)


def make_t5_model(w: synth.T5Workload, bits: dict | None = None, dev: dict | None = None,
                  gamma_max: int | None = None, max_seq: int | None = None, max_enc: int | None = None,
                  options: int = 0):
    bits = bits if bits is not None else synth.make_t5_weights(w)
    dev = dev if dev is not None else t5_device_weights(bits)
    cfg = lib.t5_config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, gamma_max or max(w.gamma, 1),
                             max_seq or (w.max_dec() + 1), max_enc or w.enc_len, w.eos_id, options=options)
    rs = torch.tensor(w.dec_scale(), dtype=torch.float32, device="cuda")
    ins = torch.tensor([w.in_scale()], dtype=torch.float32, device="cuda")
    return lib.SSDModel(cfg, dev, rs, ins), bits, dev


def t5_device_inputs(w: synth.T5Workload, seed: int | None = None):
    q, prompt = synth.make_t5_inputs(w, seed)
    v = lib.bf16_bits_to_device(q) if w.n_query > 0 else None
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    return q, prompt, v, p
