"""Driver for ncu captures: runs one decode phase of a 7B-shaped model inside a
cudaProfilerStart/Stop window (use `ncu --profile-from-start off`).

  python -m paper_2510_22641_gb300.profile_run --layers 32 --phase greedy --tokens 8
  python -m paper_2510_22641_gb300.profile_run --layers 2 --phase greedy --tokens 1
  python -m paper_2510_22641_gb300.profile_run --layers 1 --phase proj --proj gateup --rows 1

--layers keeps the 7B layer shape (d=4096, ff=11008, 32x128 heads, V=32000)
but fewer layers, so full metric sets can be captured with a few GB on the
device; every weight matrix is still larger or comparable to what one kernel
streams at full size.

  python -m paper_2510_22641_gb300.profile_run --encdec --layers 24 --phase greedy --tokens 2

--encdec runs the BLIP-2 FlanT5-xl-shaped encoder-decoder instead (d=2048, 32x64 heads,
gated-GELU 5120, V=32128; --layers encoder and decoder layers each, 24 at full size).
"""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--phase", choices=["greedy", "ssd", "prefill", "proj"], default="greedy")
    ap.add_argument("--proj", default="gateup", help="--phase proj: qkv, o, gateup, down, head, in1, in2 or attn")
    ap.add_argument("--rows", type=int, default=1, help="--phase proj: activation rows")
    ap.add_argument("--tokens", type=int, default=8)
    ap.add_argument("--s", type=float, default=0.2)
    ap.add_argument("--encdec", action="store_true", help="the FlanT5-xl-shaped encoder-decoder model")
    args = ap.parse_args()

    import torch

    import paper_2510_22641_gb300 as lib
    import synth

    if args.encdec:
        encdec(args, lib, synth, torch)
        return

    base = synth.LLAVA7B
    shape = synth.ModelShape(args.layers, 4096, 32, 128, 11008, 32000)
    w = base.replace(shape=shape, draft_exit_k=min(base.draft_exit_k, args.layers), s=args.s)
    lib.build()
    bits = synth.make_weights(w)
    up = lib.bf16_bits_to_device
    dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm", "in_norm", "in_w1", "in_w2")}
    dev["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
    cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                          w.prompt_len + w.max_new + lib.SSD_MAX_GAMMA + 1)
    model = lib.SSDModel(cfg, dev, torch.tensor(w.resid_scale(), device="cuda"),
                         torch.tensor([w.in_scale()], device="cuda"))
    vis, prompt = synth.make_inputs(w)
    v = up(vis)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()

    def run():
        model.prefill(v, p)
        if args.phase == "greedy":
            model.greedy_decode(1 + args.tokens)
        elif args.phase == "ssd":
            model.decode(1 + args.tokens, w.gamma)

    if args.phase == "proj":  # isolated launches of one projection kernel (attention: over the prompt's cache)
        model.prefill(v, p)
        model.profile_projection(args.proj, 0, args.rows, 3)
        model.prefill(v, p)
        model.sync()
        torch.cuda.profiler.start()
        model.profile_projection(args.proj, 0, args.rows, 3)
        model.sync()
        torch.cuda.profiler.stop()
        print("profile_run done", args.proj, args.rows)
        model.close()
        return
    run()                       # builds the graphs, warms up
    model.sync()
    if args.phase != "prefill":
        model.prefill(v, p)
        model.sync()
        torch.cuda.profiler.start()
        if args.phase == "greedy":
            model.greedy_decode(1 + args.tokens)
        else:
            model.decode(1 + args.tokens, w.gamma)
        model.sync()
        torch.cuda.profiler.stop()
    else:
        torch.cuda.profiler.start()
        model.prefill(v, p)
        model.sync()
        torch.cuda.profiler.stop()
    print("profile_run done", model.stats())
    model.close()


def encdec(args, lib, synth, torch) -> None:
    """Prefill (encoder + cross K/V + first decoder step) and one decode phase of the FlanT5-xl shape."""
    base = synth.FLANT5XL
    shape = synth.T5Shape(args.layers, args.layers, 2048, 32, 64, 5120, 32128)
    w = base.replace(shape=shape, draft_exit_k=min(base.draft_exit_k, args.layers), s=args.s)
    lib.build()
    bits = synth.make_t5_weights(w)
    up = lib.bf16_bits_to_device
    dev = lib.encdec_device_weights(bits)
    cfg = lib.t5_config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                             w.max_new + lib.SSD_MAX_GAMMA + 2, w.enc_len)
    model = lib.SSDModel(cfg, dev, torch.tensor(w.dec_scale(), device="cuda"),
                         torch.tensor([w.in_scale()], device="cuda"))
    q, prompt = synth.make_t5_inputs(w)
    v = up(q)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    n = 1 + args.tokens
    model.prefill(v, p)
    model.greedy_decode(n) if args.phase == "greedy" else model.decode(n, w.gamma)
    if args.phase != "prefill":
        model.prefill(v, p)
    model.sync()
    torch.cuda.profiler.start()
    if args.phase == "greedy":
        model.greedy_decode(n)
    elif args.phase == "ssd":
        model.decode(n, w.gamma)
    else:
        model.prefill(v, p)
    model.sync()
    torch.cuda.profiler.stop()
    print("profile_run done", model.stats())
    model.close()


if __name__ == "__main__":
    main()
