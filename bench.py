"""Benchmark of greedy self-speculative decoding on the LLaVA-1.5-7B-shaped workload.

One step = one request through the whole hot path with inputs resident in HBM:
prefill of 576 synthetic visual rows + 64 prompt ids, then 128 new tokens by
self-speculative decoding (draft = layers 0..7 + imitation network, gamma = 5,
full-model verification, on-device accept/rollback), batch 1.

Printed as one JSON line (rank 0):
  value          new tokens / second over whole requests (prefill included)
  e2e            the same through ssd_generate with pinned host buffers
                 (host->device inputs and device->host tokens inside the timing)
  roofline       the dominant kernel (weight-streaming GEMV, gate/up, 1 row)
                 timed alone with CUDA events, against the measured HBM copy peak
  per_s          decode tokens/s of SSD and of greedy decoding (same kernels), and of SSD with the
                 dynamic draft length d(t) (d0 = 5, capped at gamma_max = 15; t over the context with
                 N = the context's max_seq, and t over the generated tokens with N = max_new)
                 and their ratio for s in {0.05, 0.2, 1.0}
  cpu_baseline   the fp64 oracle on the host cores over a bounded sample

--impl reference times that oracle itself (rank 0 only).
Multi-GPU (torchrun): independent replicas, one request stream per GPU.

--profile PHASE opens a profiler window around one phase for ncu (no JSON line).
Other workloads, one JSON line each: --sweep (k x gamma x s on the 7B shape), --in-block (the
imitation module as one decoder block), --encdec (the BLIP-2 FlanT5-xl-shaped encoder-decoder:
decode tokens/s per s, per-kernel table, encoder prefill, and its oracle on the host cores).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "tokens/s and speedup vs full-model greedy decode (7B shape, bs1); HBM GB/s"

# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of one gate/up GEMV
# launch from an ncu capture, valid only for the kernel sources it was taken on.
GEMV_TRAFFIC = {"gemv_sources_sha256_prefix": "0126cd8e90bde7c5", "bytes": 182_910_208}
UNIT = "tokens/s"
S_VALUES = synth.LLAVA7B_S_VALUES


def workload_config(w: synth.Workload) -> dict:
    sh = w.shape
    return {"workload": f"{w.name}: L={sh.n_layers} d={sh.d_model} H={sh.n_heads}x{sh.head_dim} "
                        f"ff={sh.d_ff} V={sh.vocab}, {w.n_vis} visual + {w.n_prompt} prompt, "
                        f"{w.max_new} new tokens, k={w.draft_exit_k}, gamma={w.gamma}, s={w.s}, bs1",
            "batch": 1, "prompt_rows": w.prompt_len, "max_new": w.max_new, "draft_exit_k": w.draft_exit_k,
            "gamma": w.gamma, "s": w.s, "weights": "bf16 N(0,0.02) random-init, seed 0",
            "inputs": "visual N(0,1) bf16 + prompt ids U[0,V), seeded",
            "l2": "no flush needed: each step streams 13.5 GB of weights (>> 129 MB L2) dozens of times"}


def algorithmic_bytes(w: synth.Workload) -> dict:
    """Bytes the method must move (bf16 weights; KV per position per layer = 2*H*Dh*2)."""
    sh = w.shape
    layer = 2 * (4 * sh.d_model * sh.qdim + 3 * sh.d_model * sh.d_ff)
    head = 2 * sh.vocab * sh.d_model
    imit = 2 * 2 * sh.d_model * w.in_hidden if w.in_kind == synth.IN_MLP2 else 0
    kv_pos = 2 * sh.n_heads * sh.head_dim * 2
    return {"layer": layer, "head": head, "imit": imit, "kv_pos_layer": kv_pos, "kv_pos_layer_f32": 2 * kv_pos,
            "draft_token": w.draft_exit_k * layer + imit + head,
            "verify": sh.n_layers * layer + head, "greedy_token": sh.n_layers * layer + head}


def measured_peak(key: str, fallback: float = 6800.0) -> float:
    """A roofline denominator from MEASURED_PEAKS.json (the machine's measured copy / GEMM peaks)."""
    try:
        return float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))[key])
    except (OSError, KeyError, ValueError):
        return fallback


KERNEL_ROWS = (("qkv", "ssd_wstream_kernel<M, QKV> (q/k/v + RoPE + KV write)"),
               ("o", "ssd_wstream_kernel<M, RESID> (o_proj)"),
               ("gateup", "ssd_wstream_kernel<M, GATE_SILU> (gate/up)"),
               ("down", "ssd_wstream_kernel<M, RESID> (down)"),
               ("attn", "ssd_splitkv_attn_kernel<M, 128> (split-KV, cache after prefill)"),
               ("head", "ssd_wstream_kernel<M, ARGMAX> (LM head)"),
               ("in1", "ssd_wstream_kernel<1, SILU> (imitation FC1)"),
               ("in2", "ssd_wstream_kernel<1, RESID> (imitation FC2)"))


ENCDEC_KERNEL_ROWS = (("qkv", "ssd_wstream_kernel<M, QKV> (self q/k/v + KV write, no RoPE)"),
                      ("o", "ssd_wstream_kernel<M, RESID> (self o; cross q / cross o have this shape)"),
                      ("gateup", "ssd_wstream_kernel<M, GATE_SILU> (wi_0/wi_1, gated GELU)"),
                      ("down", "ssd_wstream_kernel<M, RESID> (wo of the MLP)"),
                      ("attn", "ssd_splitkv_attn_kernel<M, 64, EXT> (self-attention, relative-position bias)"),
                      ("head", "ssd_wstream_kernel<M, ARGMAX> (LM head)"),
                      ("in1", "ssd_wstream_kernel<1, SILU> (imitation FC1)"),
                      ("in2", "ssd_wstream_kernel<1, RESID> (imitation FC2)"))


def kernel_table(model, w, v, p, stream, hbm_peak, reps=50, rows_table=KERNEL_ROWS, layer_sum=True):
    """Every decode kernel timed alone (CUDA events, `reps` back-to-back launches) at the draft's
    1 row and the verification's gamma + 1 rows, against the HBM copy peak.  `layer_m*` sums one
    decoder layer's kernels (bytes / time), the fraction a layer would reach with no launch gaps."""
    import torch
    rows_out, layer = [], {}
    for rows in (1, w.gamma + 1):
        for name, label in rows_table:
            if name in ("in1", "in2") and rows != 1:
                continue
            model.prefill(v, p)
            model.profile_projection(name, layer=0, rows=rows, reps=3)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            a.record(stream)
            nbytes = model.profile_projection(name, layer=0, rows=rows, reps=reps)
            b.record(stream)
            torch.cuda.synchronize()
            us = a.elapsed_time(b) / reps * 1e3
            gbs = nbytes / us / 1e3
            rows_out.append({"kernel": label.replace("<M,", f"<{rows},"), "rows": rows, "bytes": nbytes,
                             "us": round(us, 2), "gbs": round(gbs, 1), "frac": round(gbs / hbm_peak, 3)})
            if layer_sum and name in ("qkv", "o", "gateup", "down", "attn"):
                lb, lt = layer.get(rows, (0, 0.0))
                layer[rows] = (lb + nbytes, lt + us)
    summary = {f"layer_m{r}": {"us": round(t, 1), "gbs": round(b_ / t / 1e3, 1), "frac": round(b_ / t / 1e3 / hbm_peak, 3)}
               for r, (b_, t) in layer.items()}
    return {"peak_gbs": hbm_peak, "launches": rows_out, **summary}


def gemv_traffic_bytes():
    """Measured bytes per launch if the GEMV's sources (gemv.cuh, tcgen05.cuh, common.cuh) are the
    captured version, else None."""
    import hashlib
    h = hashlib.sha256()
    try:
        for name in ("gemv.cuh", "tcgen05.cuh", "common.cuh"):
            h.update(open(os.path.join(ROOT, "paper_2510_22641_gb300", "csrc", name), "rb").read())
    except OSError:
        return None
    return GEMV_TRAFFIC["bytes"] if h.hexdigest().startswith(GEMV_TRAFFIC["gemv_sources_sha256_prefix"]) else None


def prefill_flops(w: synth.Workload) -> float:
    """Tensor-core work of one prefill: 2 flops per weight per row, times 2 for the bf16 hi/lo activation parts."""
    sh = w.shape
    params = 4 * sh.d_model * sh.qdim + 3 * sh.d_model * sh.d_ff
    return 2.0 * 2.0 * w.prompt_len * params * sh.n_layers


def reduce_max(value: float, dist=None, device=None) -> float:
    """Max over ranks (the slowest rank defines the whole job's time)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_tokens_per_s(world: int, steps: int, tokens_per_step: int, max_ms: float) -> float:
    """Weak scaling: every rank generates `steps` requests; the job lasts as long as the slowest rank."""
    return world * steps * tokens_per_step / (max_ms / 1e3)


# --------------------------------------------------------------------------- clocks

CLOCK_Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
           "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
           "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    def __init__(self, gpu: int):
        self.p = None
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={CLOCK_Q}", "--format=csv,noheader,nounits",
                                       "-i", str(gpu), "-lms", "200"], stdout=subprocess.PIPE,
                                      stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.p = None

    def stop(self) -> dict | None:
        if self.p is None:
            return None
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
            out, _ = self.p.communicate()
        sm, smax, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = max(smax, float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------------- oracle legs (CPU)

def oracle_sample(w: synth.Workload, bits, vis, prompt, max_steps: int, warm_steps: int = 0) -> dict:
    """Time the fp64 oracle on this workload: its prefill and `max_steps` SSD steps."""
    import oracle
    t0 = time.perf_counter()
    m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    t_conv = time.perf_counter() - t0
    r = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, w.gamma,
                            max_steps=warm_steps + max_steps)
    steps = r.step_s[warm_steps:]
    acc = r.accept_lengths[warm_steps:]
    toks_per_step = (sum(acc) + len(acc)) / max(len(acc), 1)
    step_mean = sum(steps) / max(len(steps), 1)
    request_s = r.prefill_s + (w.max_new - 1) / toks_per_step * step_mean
    return {"value": w.max_new / request_s, "prefill_s": r.prefill_s, "step_s": step_mean,
            "tokens_per_step": toks_per_step, "n_steps": len(steps), "convert_s": t_conv,
            "cores": os.cpu_count()}


def oracle_sample_encdec(w: synth.T5Workload, bits, query, prompt, max_steps: int) -> dict:
    """Time the fp64 encoder-decoder oracle: its encoder + first decoder step and `max_steps` SSD steps."""
    from oracle import t5_oracle
    m = t5_oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    r = t5_oracle.ssd_generate(m, synth.bf16_to_f64(query), prompt, w.max_new, w.gamma, max_steps=max_steps)
    acc = r.accept_lengths
    toks_per_step = (sum(acc) + len(acc)) / max(len(acc), 1)
    step_mean = sum(r.step_s) / max(len(r.step_s), 1)
    return {"decode_tok_s": toks_per_step / step_mean if step_mean > 0 else None, "prefill_s": r.prefill_s,
            "step_s": step_mean, "tokens_per_step": toks_per_step, "n_steps": len(r.step_s),
            "cores": os.cpu_count()}


def run_reference(args) -> None:
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = synth.LLAVA7B.replace(s=args.s)
    bits = synth.make_weights(w)
    vis, prompt = synth.make_inputs(w)
    r = oracle_sample(w, bits, vis, prompt, max_steps=args.steps, warm_steps=args.warmup)
    sample = (f"fp64 numpy oracle: one prefill ({w.prompt_len} rows) + {args.warmup} warm-up and "
              f"{r['n_steps']} timed SSD steps; tokens/s = {w.max_new} / (prefill + {w.max_new - 1} tokens "
              f"at the sampled tokens per step and step time)")
    line = {"impl": "reference", "metric": METRIC, "value": r["value"], "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["step_s"] * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(w),
            "cpu_baseline": {"value": r["value"], "unit": UNIT, "cores": r["cores"], "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": r["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "prefill_s": r["prefill_s"], "tokens_per_step": r["tokens_per_step"]}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- GPU arm

def run_in_block(args) -> None:
    """The LLaVA-1.5-7B-shaped workload (k = 8, gamma = 5, 128 new tokens) with the imitation module
    read as one decoder block with its own KV cache (IN_BLOCK): decode tokens/s of SSD and greedy,
    speedup, accept length and the drafting stage's HBM GB/s, per s.  One JSON line."""
    import torch

    import paper_2510_22641_gb300 as lib
    lib.build()
    w = synth.LLAVA7B.replace(in_kind=synth.IN_BLOCK)
    bits = synth.make_weights(w)
    up = lib.bf16_bits_to_device
    dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm")}
    dev["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
    dev["in_block"] = {n: up(a) for n, a in bits["in_block"].items()}
    vis, prompt = synth.make_inputs(w)
    v = up(vis)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    stream = torch.cuda.current_stream()
    rs = torch.tensor(w.resid_scale(), device="cuda")
    ins = torch.tensor([w.in_scale()], device="cuda")
    cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                          w.prompt_len + w.max_new + lib.SSD_MAX_GAMMA + 1)
    model = lib.SSDModel(cfg, dev, rs, ins)
    ab = algorithmic_bytes(w)
    draft_bytes = w.draft_exit_k * ab["layer"] + ab["layer"] + ab["head"]   # shallow layers + the block + g

    def timed(fn):
        model.prefill(v, p)
        fn()
        model.prefill(v, p)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b)

    rows = []
    for s_val in S_VALUES:
        ws = w.replace(s=s_val)
        rs.copy_(torch.tensor(ws.resid_scale(), device="cuda"))
        ins.copy_(torch.tensor([ws.in_scale()], device="cuda"))
        g_ms = timed(lambda: model.greedy_decode(w.max_new))
        s_ms = timed(lambda: model.decode(w.max_new, w.gamma))
        st = model.stats()
        model.prefill(v, p)
        model.draft(w.gamma)
        model.verify(w.gamma)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        model.draft(w.gamma)
        b.record(stream)
        torch.cuda.synchronize()
        d_ms = a.elapsed_time(b)
        rows.append({"s": s_val, "ssd_decode_tok_s": (w.max_new - 1) / (s_ms / 1e3),
                     "greedy_decode_tok_s": (w.max_new - 1) / (g_ms / 1e3), "speedup": g_ms / s_ms,
                     "mean_accept": st["accepted"] / max(st["steps"], 1), "draft_ms": d_ms,
                     "draft_gbs": w.gamma * draft_bytes / (d_ms / 1e3) / 1e9})
    model.close()
    print(json.dumps({"workload": workload_config(w)["workload"] + ", imitation = one decoder block (IN_BLOCK)",
                      "per_s": rows}), flush=True)


def run_encdec(args) -> None:
    """The BLIP-2 FlanT5-xl-shaped encoder-decoder workload (24 + 24 layers, d = 2048, 32 x 64 heads,
    gated-GELU 5120, V = 32128; 32 query embeddings + 16 prompt ids; draft = decoder layers 0-5 + the
    imitation network; gamma = 4; 30 new tokens): decode tokens/s of SSD and of greedy decoding with
    the same kernels, speedup, accept length, the drafting stage's and the greedy decoder's HBM GB/s
    (of measured), and the encoder prefill time, per s.  One JSON line."""
    import torch

    import paper_2510_22641_gb300 as lib
    lib.build()
    w = synth.FLANT5XL
    sh = w.shape
    bits = synth.make_t5_weights(w)
    up = lib.bf16_bits_to_device
    dev = lib.encdec_device_weights(bits)
    q, prompt = synth.make_t5_inputs(w)
    v = up(q)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    stream = torch.cuda.current_stream()
    rs = torch.tensor(w.dec_scale(), device="cuda")
    ins = torch.tensor([w.in_scale()], device="cuda")
    cfg = lib.t5_config_dict(sh, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                             w.max_new + lib.SSD_MAX_GAMMA + 2, w.enc_len, w.eos_id)
    model = lib.SSDModel(cfg, dev, rs, ins)
    # algorithmic bytes per decode row: a decoder layer's weights (self q/k/v/o, cross q/o, MLP, norms)
    # plus the cross-attention K/V it reads (fp32); the imitation network; the LM head
    layer = sh.dec_layer_bytes_bf16() + 2 * sh.n_heads * w.enc_len * sh.head_dim * 4
    in_bytes = 2 * 2 * w.in_hidden * sh.d_model + 2 * sh.d_model
    head = 2 * sh.vocab * sh.d_model + 2 * sh.d_model
    draft_bytes = w.draft_exit_k * layer + in_bytes + head
    greedy_bytes = sh.n_dec * layer + head
    try:
        peak = float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))["hbm_gbs"])
    except (OSError, KeyError, ValueError):
        peak = None

    def ev_ms(fn):
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b)

    def timed(fn):
        model.prefill(v, p)
        fn()
        model.prefill(v, p)
        return ev_ms(fn)

    model.prefill(v, p)
    prefill_ms = min(ev_ms(lambda: model.prefill(v, p)) for _ in range(3))
    kernels = kernel_table(model, w, v, p, stream, peak or 6800.0, rows_table=ENCDEC_KERNEL_ROWS, layer_sum=False)
    rows = []
    for s_val in S_VALUES:
        ws = w.replace(s=s_val)
        rs.copy_(torch.tensor(ws.dec_scale(), device="cuda"))
        ins.copy_(torch.tensor([ws.in_scale()], device="cuda"))
        g_ms = min(timed(lambda: model.greedy_decode(w.max_new)) for _ in range(3))
        s_ms = min(timed(lambda: model.decode(w.max_new, w.gamma)) for _ in range(3))
        st = model.stats()
        model.prefill(v, p)
        model.draft(w.gamma)
        model.verify(w.gamma)
        d_ms = ev_ms(lambda: model.draft(w.gamma))
        g_gbs = (w.max_new - 1) * greedy_bytes / (g_ms / 1e3) / 1e9
        d_gbs = w.gamma * draft_bytes / (d_ms / 1e3) / 1e9
        rows.append({"s": s_val, "ssd_decode_tok_s": (w.max_new - 1) / (s_ms / 1e3),
                     "greedy_decode_tok_s": (w.max_new - 1) / (g_ms / 1e3), "speedup": g_ms / s_ms,
                     "mean_accept": st["accepted"] / max(st["steps"], 1), "steps": st["steps"],
                     "draft_ms": d_ms, "draft_gbs": d_gbs, "greedy_gbs": g_gbs,
                     "draft_frac": d_gbs / peak if peak else None, "greedy_frac": g_gbs / peak if peak else None})
    model.close()
    cpu = None
    if not args.no_cpu_baseline:
        r = oracle_sample_encdec(w, bits, q, prompt, max_steps=args.cpu_steps)
        cpu = {"value": r["decode_tok_s"], "unit": UNIT, "cores": r["cores"], "kind": "oracle",
               "sample": f"fp64 numpy encoder-decoder oracle at s = {w.s}: encoder + first decoder step "
                         f"({r['prefill_s']:.1f} s) and {r['n_steps']} SSD steps ({r['step_s']:.2f} s each, "
                         f"{r['tokens_per_step']:.2f} tokens/step); value = decode tokens/s"}
    print(json.dumps({"workload": f"{w.name}: {sh.n_enc}+{sh.n_dec} layers, d={sh.d_model}, {sh.n_heads}x"
                                  f"{sh.head_dim} heads, gated-GELU {sh.d_ff}, V={sh.vocab}; {w.n_query} queries + "
                                  f"{w.n_prompt} prompt ids; k={w.draft_exit_k}, gamma={w.gamma}, "
                                  f"{w.max_new} new tokens; bs1",
                      "prefill_ms": prefill_ms, "peak_hbm_gbs": peak, "bytes_per_token":
                          {"draft": draft_bytes, "greedy": greedy_bytes}, "per_s": rows, "kernels": kernels,
                      "cpu_baseline": cpu}),
          flush=True)


BATCH_KERNEL_ROWS = (("qkv", "ssd_wstream_mid_kernel<QKV> (q/k/v + RoPE + KV write)"),
                     ("o", "ssd_wstream_mid_kernel<RESID> (o_proj)"),
                     ("gateup", "ssd_wstream_mid_kernel<GATE_SILU> (gate/up)"),
                     ("down", "ssd_wstream_mid_kernel<RESID> (down)"),
                     ("head", "ssd_wstream_mid_kernel<ARGMAX> (LM head)"))


def batch_algorithmic_bytes(w: synth.Workload, prompts, accept_logs, gamma: int) -> dict:
    """Bytes a batched decode must move: per step the drafting stage's weights gamma times, the
    verification pass's weights once, and the K/V of every active request read once per drafting
    row and once per verification pass (positions up to the row; fp32 K and V)."""
    ab = algorithmic_bytes(w)
    sh = w.shape
    L, k = sh.n_layers, w.draft_exit_k
    steps = max(len(a) for a in accept_logs)
    weights = kv = 0
    kv_len = list(prompts)
    for s in range(steps):
        weights += gamma * ab["draft_token"] + ab["verify"] if gamma > 0 else ab["greedy_token"]
        for b, acc in enumerate(accept_logs):
            if s >= len(acc):
                continue
            if gamma > 0:
                kv += sum(k * (kv_len[b] + j + 1) for j in range(gamma)) * ab["kv_pos_layer_f32"]
                kv += L * (kv_len[b] + gamma + 1) * ab["kv_pos_layer_f32"]
            else:
                kv += L * (kv_len[b] + 1) * ab["kv_pos_layer_f32"]
            kv_len[b] += acc[s] + 1
    return {"weights": weights, "kv": kv, "total": weights + kv, "steps": steps}


def run_batch16(args) -> None:
    """Batched requests (BASELINE configs[4]): 16 requests on the LLaVA-1.5-13B shape (40 layers,
    d = 5120, 40 x 128 heads, SwiGLU 13824, V = 32000), each with 576 visual rows and a prompt of
    U[32, 256] ids, k = 10, gamma = 6, s = 0.2, 256 new tokens per request, decoded in lockstep
    (ragged positions and accept lengths): batched SSD and batched greedy decode tokens/s over all
    requests, the speedup, accept lengths, the decode's HBM bytes per second, the verification
    projections at 112 rows through the medium-M tensor-core kernel timed alone, and the fp64
    oracle's rate on the host cores.  One JSON line."""
    import torch

    import paper_2510_22641_gb300 as lib
    lib.build()
    bw = synth.LLAVA13B_B16.replace(base=synth.LLAVA13B.replace(s=args.s))
    w = bw.base
    up = lib.bf16_bits_to_device
    bits = synth.make_weights(w, with_layers=False)
    dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm", "in_norm", "in_w1", "in_w2")}
    dev["layers"] = []
    for l in range(w.shape.n_layers):   # one layer at a time: 634 MB of bf16 each
        dev["layers"].append({n: up(a) for n, a in synth.make_layer_weights(w, l).items()})
    ins = synth.make_batch_inputs(bw)
    nv = [v.shape[0] for v, _ in ins]
    npr = [len(p) for _, p in ins]
    prompts = [a + b for a, b in zip(nv, npr)]
    dv = up(np.concatenate([v for v, _ in ins]))
    dp = torch.from_numpy(np.concatenate([p for _, p in ins]).astype(np.int32)).cuda()
    rs = torch.tensor(w.resid_scale(), device="cuda")
    ins_t = torch.tensor([w.in_scale()], device="cuda")
    cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, w.gamma, bw.max_seq(),
                          options=lib.SSD_OPT_HOST_LOOP if args.host_loop else 0, max_batch=bw.batch)
    model = lib.SSDModel(cfg, dev, rs, ins_t)
    B, T = bw.batch, w.max_new
    out = torch.zeros(B, T, dtype=torch.int32, device="cuda")
    n_out = torch.zeros(B, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    hbm_peak = measured_peak("hbm_gbs")

    def run(gamma):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        torch.cuda.synchronize()
        ev[0].record(stream)
        model.prefill_batch(dv, nv, dp, npr)
        ev[1].record(stream)
        if gamma > 0:
            model.decode_batch(T, gamma, out, n_out)
        else:
            model.greedy_decode_batch(T, out, n_out)
        ev[2].record(stream)
        torch.cuda.synchronize()
        model.sync()
        assert all(int(x) == T for x in n_out.cpu()), n_out
        return ev[0].elapsed_time(ev[1]), ev[1].elapsed_time(ev[2])

    def set_s(s_val):
        ws = w.replace(s=s_val)
        rs.copy_(torch.tensor(ws.resid_scale(), device="cuda"))
        ins_t.copy_(torch.tensor([ws.in_scale()], device="cuda"))

    run(w.gamma)   # warm-up: builds the graphs
    run(0)
    clocks = ClockSampler(torch.cuda.current_device())
    rows = []
    greedy_ms = run(0)[1]
    greedy_tokens = B * (T - 1)
    gb = batch_algorithmic_bytes(w, prompts, [[0] * (T - 1)] * B, 0)
    for s_val in (args.s, 0.05, 1.0):
        set_s(s_val)
        pre_ms, dec_ms = run(w.gamma)
        logs = [model.batch_step_log(b)[0] for b in range(B)]
        ab = batch_algorithmic_bytes(w, prompts, logs, w.gamma)
        acc = [a for lg in logs for a in lg]
        rows.append({"s": s_val, "ssd_decode_tok_s": B * (T - 1) / (dec_ms / 1e3),
                     "speedup": greedy_ms / dec_ms, "mean_accept": sum(acc) / max(len(acc), 1),
                     "batch_steps": ab["steps"], "decode_ms": dec_ms, "prefill_ms": pre_ms,
                     "decode_hbm_gbs": ab["total"] / (dec_ms / 1e3) / 1e9,
                     "decode_hbm_frac": ab["total"] / (dec_ms / 1e3) / 1e9 / hbm_peak,
                     "weight_gb": ab["weights"] / 1e9, "kv_gb": ab["kv"] / 1e9})
    set_s(args.s)
    clk = clocks.stop()
    head = rows[0]

    # the verification projections at B * (gamma + 1) rows, each kernel timed alone
    vrows = B * (w.gamma + 1)
    kernels = []
    flops_total = 0.0
    for name, label in BATCH_KERNEL_ROWS:
        model.profile_projection(name, layer=w.draft_exit_k, rows=vrows, reps=3)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = 20
        torch.cuda.synchronize()
        a.record(stream)
        nbytes = model.profile_projection(name, layer=w.draft_exit_k, rows=vrows, reps=reps)
        b.record(stream)
        torch.cuda.synchronize()
        us = a.elapsed_time(b) / reps * 1e3
        sh = w.shape
        n_out_rows = {"qkv": 3 * sh.qdim, "o": sh.d_model, "gateup": 2 * sh.d_ff, "down": sh.d_model,
                      "head": sh.vocab}[name]
        k_in = {"qkv": sh.d_model, "o": sh.qdim, "gateup": sh.d_model, "down": sh.d_ff, "head": sh.d_model}[name]
        flops = 2.0 * vrows * n_out_rows * k_in * 2   # bf16 hi + lo parts
        kernels.append({"kernel": label + " + split", "rows": vrows, "bytes": nbytes, "us": round(us, 2),
                        "gbs": round(nbytes / us / 1e3, 1), "frac": round(nbytes / us / 1e3 / hbm_peak, 3),
                        "tflops_issued": round(flops / us / 1e6, 1)})
    cpu = None
    if not args.no_cpu_baseline:
        cpu = oracle_batch_sample(w, ins[0], max_steps=1)
    model.close()
    line = {"metric": "batched decode tokens/s (16 requests, 13B shape) and speedup vs batched greedy",
            "value": head["ssd_decode_tok_s"], "unit": UNIT, "n_gpus": 1, "higher_is_better": True,
            "dtype": "bf16 weights, fp32 activations / KV / accumulation", "data": "synthetic",
            "config": {"workload": f"{w.name} x {B} requests: L={w.shape.n_layers} d={w.shape.d_model} "
                                   f"H={w.shape.n_heads}x{w.shape.head_dim} ff={w.shape.d_ff} V={w.shape.vocab}, "
                                   f"576 visual + prompts U[{bw.prompt_min},{bw.prompt_max}] "
                                   f"({min(npr)}..{max(npr)}), {T} new tokens each, k={w.draft_exit_k}, "
                                   f"gamma={w.gamma}, s={args.s}", "batch": B, "prompt_rows": prompts},
            "greedy_decode_tok_s": greedy_tokens / (greedy_ms / 1e3),
            "greedy_decode_hbm_frac": gb["total"] / (greedy_ms / 1e3) / 1e9 / hbm_peak,
            "per_s": rows, "verify_kernels": kernels, "clocks": clk,
            "cpu_baseline": cpu}
    print(json.dumps(line), flush=True)


def oracle_batch_sample(w: synth.Workload, request, max_steps: int) -> dict:
    """The fp64 oracle on one request of the batch (it decodes requests one after another, so the
    batch's oracle rate is one request's): its prefill and `max_steps` SSD steps, weights widened
    from bf16 to fp64 (about 8 bytes per parameter of host memory)."""
    import oracle
    bits = synth.make_weights(w)
    vis, prompt = request
    m = oracle.model_from_bits(w, bits, synth.bf16_to_f64)
    del bits
    r = oracle.ssd_generate(m, synth.bf16_to_f64(vis), prompt, w.max_new, w.gamma, max_steps=max_steps)
    acc = r.accept_lengths
    tps = (sum(acc) + len(acc)) / max(len(acc), 1)
    step = sum(r.step_s) / max(len(r.step_s), 1)
    return {"value": tps / step if step > 0 else None, "unit": "decode tokens/s", "cores": os.cpu_count(),
            "kind": "oracle", "prefill_s": r.prefill_s, "step_s": step,
            "sample": f"fp64 numpy oracle, request 0 of the batch ({vis.shape[0] + len(prompt)} prompt rows): "
                      f"its prefill and {len(acc)} SSD step(s); the oracle runs requests one at a time"}


def run_sweep(args) -> None:
    """Sweep k x gamma x s on the 7B shape (256 new tokens): accept length, tokens/s, speedup
    over greedy, draft and verify HBM GB/s.  One JSON line per point."""
    import torch

    import paper_2510_22641_gb300 as lib
    lib.build()
    base = synth.LLAVA7B.replace(max_new=256)
    bits = synth.make_weights(base)
    up = lib.bf16_bits_to_device
    dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm", "in_norm", "in_w1", "in_w2")}
    dev["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
    vis, prompt = synth.make_inputs(base)
    v = up(vis)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    stream = torch.cuda.current_stream()
    rs = torch.tensor(base.resid_scale(), device="cuda")
    ins = torch.tensor([base.in_scale()], device="cuda")

    def ev():
        e = torch.cuda.Event(enable_timing=True)
        e.record(stream)
        return e

    greedy_tok_s = {}
    for k in (4, 8, 12, 16):
        w0 = base.replace(draft_exit_k=k)
        cfg = lib.config_dict(w0.shape, k, w0.in_kind, w0.in_hidden, lib.SSD_MAX_GAMMA,
                              w0.prompt_len + w0.max_new + lib.SSD_MAX_GAMMA + 1)
        model = lib.SSDModel(cfg, dev, rs, ins)
        ab = algorithmic_bytes(w0)
        for s_val in S_VALUES:
            w = w0.replace(s=s_val)
            rs.copy_(torch.tensor(w.resid_scale(), device="cuda"))
            ins.copy_(torch.tensor([w.in_scale()], device="cuda"))
            if s_val not in greedy_tok_s:
                model.prefill(v, p)
                model.greedy_decode(w.max_new)
                model.prefill(v, p)
                a = ev()
                model.greedy_decode(w.max_new)
                b = ev()
                torch.cuda.synchronize()
                greedy_tok_s[s_val] = (w.max_new - 1) / (a.elapsed_time(b) / 1e3)
            for gamma in (2, 3, 4, 5, 6, 8):
                model.prefill(v, p)
                model.decode(w.max_new, gamma)          # warm-up and graph build
                model.prefill(v, p)
                a = ev()
                model.decode(w.max_new, gamma)
                b = ev()
                torch.cuda.synchronize()
                st = model.stats()
                dec_ms = a.elapsed_time(b)
                # draft / verify stages timed separately over a few steps
                model.prefill(v, p)
                model.draft(gamma)
                model.verify(gamma)
                d_ms, v_ms, n = 0.0, 0.0, 6
                for _ in range(n):
                    e0 = ev()
                    model.draft(gamma)
                    e1 = ev()
                    model.verify(gamma)
                    e2 = ev()
                    torch.cuda.synchronize()
                    d_ms += e0.elapsed_time(e1)
                    v_ms += e1.elapsed_time(e2)
                S = w.prompt_len + w.max_new // 2
                draft_bytes = gamma * (ab["draft_token"] + ab["kv_pos_layer"] * k * S)
                verify_bytes = ab["verify"] + ab["kv_pos_layer"] * w.shape.n_layers * S
                tok_s = (w.max_new - 1) / (dec_ms / 1e3)
                print(json.dumps({"k": k, "gamma": gamma, "s": s_val, "steps": st["steps"],
                                  "mean_accept": st["accepted"] / max(st["steps"], 1),
                                  "tokens_per_step": (w.max_new - 1) / max(st["steps"], 1),
                                  "ssd_tok_s": tok_s, "greedy_tok_s": greedy_tok_s[s_val],
                                  "speedup": tok_s / greedy_tok_s[s_val],
                                  "draft_ms": d_ms / n, "verify_ms": v_ms / n,
                                  "draft_gbs": draft_bytes / (d_ms / n / 1e3) / 1e9,
                                  "verify_gbs": verify_bytes / (v_ms / n / 1e3) / 1e9}), flush=True)
        model.close()


def run_profile(args) -> None:
    """A profiler window around one phase (run under `ncu --profile-from-start off`): the 7B layer
    shape with --layers layers (fewer layers keep a capture to a few GB on the device while every
    weight matrix keeps its full size), with --encdec the FlanT5-xl layer shape, or with --batch16
    the 13B layer shape and 16 batched ragged requests (proj at --rows up to 112 then runs the
    medium-M kernel).  Decode phases
    run the host-driven loop (SSD_OPT_HOST_LOOP), since profilers do not see kernels inside
    conditional graph nodes.  Phases: greedy / ssd (--tokens new tokens), prefill, proj (reps
    launches of one kernel alone: --proj qkv, o, gateup, down, head, in1, in2 or attn at --rows)."""
    import torch

    import paper_2510_22641_gb300 as lib

    lib.build()
    up = lib.bf16_bits_to_device
    if args.encdec:
        base = synth.FLANT5XL
        shape = synth.T5Shape(args.layers, args.layers, 2048, 32, 64, 5120, 32128)
        w = base.replace(shape=shape, draft_exit_k=min(base.draft_exit_k, args.layers), s=args.s)
        bits = synth.make_t5_weights(w)
        dev = lib.encdec_device_weights(bits)
        cfg = lib.t5_config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                                 w.max_new + lib.SSD_MAX_GAMMA + 2, w.enc_len, options=lib.SSD_OPT_HOST_LOOP)
        rs = torch.tensor(w.dec_scale(), device="cuda")
        vis, prompt = synth.make_t5_inputs(w)
    elif args.batch16:   # the 13B layer shape, 16 ragged requests (batched calls)
        bw = synth.LLAVA13B_B16
        shape = synth.ModelShape(args.layers, 5120, 40, 128, 13824, 32000)
        w = bw.base.replace(shape=shape, draft_exit_k=min(bw.base.draft_exit_k, args.layers), s=args.s)
        bw = bw.replace(base=w)
        bits = synth.make_weights(w)
        dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm", "in_norm", "in_w1", "in_w2")}
        dev["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
        cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, w.gamma, bw.max_seq(),
                              options=lib.SSD_OPT_HOST_LOOP, max_batch=bw.batch)
        rs = torch.tensor(w.resid_scale(), device="cuda")
        ins = synth.make_batch_inputs(bw)
        vis = np.concatenate([v for v, _ in ins])
        prompt = np.concatenate([p for _, p in ins])
        counts = ([v.shape[0] for v, _ in ins], [len(p) for _, p in ins])
    else:
        base = synth.LLAVA7B
        shape = synth.ModelShape(args.layers, 4096, 32, 128, 11008, 32000)
        w = base.replace(shape=shape, draft_exit_k=min(base.draft_exit_k, args.layers), s=args.s)
        bits = synth.make_weights(w)
        dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm", "in_norm", "in_w1", "in_w2")}
        dev["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
        cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                              w.prompt_len + w.max_new + lib.SSD_MAX_GAMMA + 1, options=lib.SSD_OPT_HOST_LOOP)
        rs = torch.tensor(w.resid_scale(), device="cuda")
        vis, prompt = synth.make_inputs(w)
    model = lib.SSDModel(cfg, dev, rs, torch.tensor([w.in_scale()], device="cuda"))
    v = up(vis)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    n = 1 + args.tokens

    def prefill():
        if args.batch16:
            model.prefill_batch(v, counts[0], p, counts[1])
        else:
            model.prefill(v, p)

    def phase():
        if args.profile == "greedy":
            (model.greedy_decode_batch if args.batch16 else model.greedy_decode)(n)
        elif args.profile == "ssd":
            (model.decode_batch if args.batch16 else model.decode)(n, w.gamma)
        elif args.profile == "proj":
            model.profile_projection(args.proj, 0, args.rows, 3)
        else:
            prefill()

    prefill()
    phase()                     # builds the graphs, warms up
    prefill()
    model.sync()
    torch.cuda.profiler.start()
    phase()
    model.sync()
    torch.cuda.profiler.stop()
    print("profile done", args.profile, model.stats(), flush=True)
    model.close()


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--s", type=float, default=0.2, help="deep-layer residual scale of the headline run")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-steps", type=int, default=3, help="oracle SSD steps in the CPU sample")
    ap.add_argument("--sweep", action="store_true", help="k x gamma x s sweep (one JSON line per point)")
    ap.add_argument("--in-block", action="store_true",
                    help="the 7B workload with the imitation module as one decoder block (one JSON line)")
    ap.add_argument("--encdec", action="store_true",
                    help="the BLIP-2 FlanT5-xl-shaped encoder-decoder workload (one JSON line)")
    ap.add_argument("--batch16", action="store_true",
                    help="16 batched ragged requests on the 13B shape (one JSON line)")
    ap.add_argument("--profile", choices=["greedy", "ssd", "prefill", "proj"],
                    help="a profiler window around one phase instead of the bench (see run_profile)")
    ap.add_argument("--layers", type=int, default=32, help="--profile: layers of the model")
    ap.add_argument("--tokens", type=int, default=4, help="--profile greedy/ssd: new tokens")
    ap.add_argument("--proj", default="gateup", help="--profile proj: the kernel")
    ap.add_argument("--rows", type=int, default=1, help="--profile proj: activation rows")
    ap.add_argument("--host-loop", action="store_true",
                    help="drive the decode loop from the host (same kernels and results; lets ncu list them)")
    args = ap.parse_args()
    if args.profile:
        run_profile(args)
        return
    if args.encdec:
        run_encdec(args)
        return
    if args.batch16:
        run_batch16(args)
        return
    if args.sweep:
        run_sweep(args)
        return
    if args.in_block:
        run_in_block(args)
        return
    if args.impl == "reference":
        run_reference(args)
        return
    assert args.warmup >= 3, "at least 3 warm-up steps"

    import torch
    import torch.distributed as dist

    import paper_2510_22641_gb300 as lib

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    lib.build()
    dev_id = torch.cuda.current_device()

    w = synth.LLAVA7B.replace(s=args.s)
    bits = synth.make_weights(w)
    up = lib.bf16_bits_to_device
    dev = {k: up(bits[k]) for k in ("embed", "lm_head", "final_norm", "in_norm", "in_w1", "in_w2")}
    dev["layers"] = [{n: up(a) for n, a in lw.items()} for lw in bits["layers"]]
    rs = torch.tensor(w.resid_scale(), device="cuda")
    ins = torch.tensor([w.in_scale()], device="cuda")
    cfg = lib.config_dict(w.shape, w.draft_exit_k, w.in_kind, w.in_hidden, lib.SSD_MAX_GAMMA,
                          w.prompt_len + w.max_new + lib.SSD_MAX_GAMMA + 1,
                          options=lib.SSD_OPT_HOST_LOOP if args.host_loop else 0)
    model = lib.SSDModel(cfg, dev, rs, ins)
    vis, prompt = synth.make_inputs(w, seed=rank)
    v = up(vis)
    p = torch.from_numpy(prompt.astype(np.int32)).cuda()
    out = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    n_out = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()

    dyn_n = w.prompt_len + w.max_new + lib.SSD_MAX_GAMMA + 1   # N of d(t): the longest sequence of this context

    def request(gamma: int, ev=None):
        model.prefill(v, p)
        if ev is not None:
            ev.record(stream)
        if gamma == -1:   # dynamic draft length d(t), d0 = 5, capped at gamma_max; t over the context
            model.decode_dynamic(w.max_new, 5, dyn_n, lib.SSD_MAX_GAMMA, out, n_out)
        elif gamma == -2:  # the same with t over the generated tokens and N = max_new
            model.decode_dynamic(w.max_new, 5, w.max_new, lib.SSD_MAX_GAMMA, out, n_out, t_from=lib.SSD_DLEN_GENERATED)
        elif gamma > 0:
            model.decode(w.max_new, gamma, out, n_out)
        else:
            model.greedy_decode(w.max_new, out, n_out)

    for _ in range(args.warmup):
        request(w.gamma)
    model.greedy_decode(w.max_new, out, n_out)   # builds the greedy graph outside the timed region
    model.sync()

    # ---------------- timed region: K requests
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(2 * args.steps + 1)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(dev_id)
    time.sleep(0.3)
    evs[0].record(stream)
    for i in range(args.steps):
        request(w.gamma, evs[2 * i + 1])
        evs[2 * i + 2].record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    total_ms = evs[0].elapsed_time(evs[-1])
    prefill_ms = [evs[2 * i].elapsed_time(evs[2 * i + 1]) for i in range(args.steps)]
    decode_ms = [evs[2 * i + 1].elapsed_time(evs[2 * i + 2]) for i in range(args.steps)]
    model.sync()
    assert int(n_out.item()) == w.max_new
    st = model.stats()
    pre_l, dec_l = model.launch_counts()
    total_ms = reduce_max(total_ms, dist if world > 1 else None, device="cuda")
    value = whole_job_tokens_per_s(world, args.steps, w.max_new, total_ms)

    # ---------------- end to end through ssd_generate with pinned host buffers
    vis_h = torch.from_numpy(vis.view(np.int16)).pin_memory()
    prompt_h = torch.from_numpy(prompt.astype(np.int32)).pin_memory()
    model.generate(vis_h, prompt_h, w.max_new, w.gamma)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        toks, _ = model.generate(vis_h, prompt_h, w.max_new, w.gamma)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    e2e = {"value": args.steps * w.max_new / (e2e_ms / 1e3), "unit": UNIT,
           "h2d_bytes_per_step": int(vis.nbytes + 4 * prompt.size), "d2h_bytes_per_step": 4 * w.max_new}

    # ---------------- speedup over greedy decoding per acceptance knob s (decode only)
    per_s = []
    for s in S_VALUES:
        ws = w.replace(s=s)
        rs.copy_(torch.tensor(ws.resid_scale(), device="cuda"))
        ins.copy_(torch.tensor([ws.in_scale()], device="cuda"))
        row = {"s": s}
        for name, gamma in (("ssd", w.gamma), ("greedy", 0), ("ssd_dynamic", -1), ("ssd_dynamic_gen", -2)):
            ts = []
            for _ in range(2):
                a, b, c = (torch.cuda.Event(enable_timing=True) for _ in range(3))
                a.record(stream)
                request(gamma, b)
                c.record(stream)
                torch.cuda.synchronize()
                ts.append(b.elapsed_time(c))
            row[f"{name}_decode_tok_s"] = (w.max_new - 1) / (min(ts) / 1e3)
            if name == "ssd":
                sst = model.stats()
                row["mean_accept"] = sst["accepted"] / max(sst["steps"], 1)
                row["steps"] = sst["steps"]
            if name.startswith("ssd_dynamic"):
                sst = model.stats()
                acc, dr = model.step_log()
                tag = name[len("ssd_"):]
                row[f"{tag}_mean_accept"] = sst["accepted"] / max(sst["steps"], 1)
                row[f"{tag}_mean_gamma"] = sst["drafted"] / max(sst["steps"], 1)
                row[f"{tag}_gamma_first_max"] = [dr[0], max(dr)] if dr else None   # the schedule grows with t
        row["speedup"] = row["ssd_decode_tok_s"] / row["greedy_decode_tok_s"]
        row["dynamic_speedup"] = row["ssd_dynamic_decode_tok_s"] / row["greedy_decode_tok_s"]
        row["dynamic_gen_speedup"] = row["ssd_dynamic_gen_decode_tok_s"] / row["greedy_decode_tok_s"]
        per_s.append(row)
    rs.copy_(torch.tensor(w.resid_scale(), device="cuda"))
    ins.copy_(torch.tensor([w.in_scale()], device="cuda"))

    # ---------------- dominant kernel alone: gate/up GEMV, 1 row (the draft's largest projection)
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except OSError:
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    peak_src = "measured" if "hbm_gbs" in peaks else "fallback"
    reps = 200
    model.profile_projection("gateup", layer=0, rows=1, reps=10)
    k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    k0.record(stream)
    nbytes = model.profile_projection("gateup", layer=0, rows=1, reps=reps)
    k1.record(stream)
    torch.cuda.synchronize()
    kern_ms = k0.elapsed_time(k1) / reps
    achieved = nbytes / (kern_ms / 1e3) / 1e9
    roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                "frac": achieved / hbm_peak, "traffic": gemv_traffic_bytes(),
                "kernel": "ssd_wstream_kernel<1, GATE_SILU> (layer gate/up, 2x11008x4096 bf16, 1 row)",
                "bytes_per_launch": nbytes, "launch_us": kern_ms * 1e3,
                "peak_source": f"{peak_src} HBM copy (burst)"}
    kernels = kernel_table(model, w, v, p, stream, hbm_peak)
    model.prefill(v, p)   # the profiling launches clobbered the decode state
    model.sync()

    # decode-phase bandwidth from algorithmic bytes
    ab = algorithmic_bytes(w)
    steps_per_req = st["steps"]
    kv_read = ab["kv_pos_layer"] * (w.prompt_len + w.max_new / 2) * (
        steps_per_req * (w.gamma * w.draft_exit_k + w.shape.n_layers))
    dec_bytes = steps_per_req * (w.gamma * ab["draft_token"] + ab["verify"]) + kv_read
    dec_ms = statistics.median(decode_ms)

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {**workload_config(w), "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       "arithmetic": "fp32 FMA on bf16 weights, fp32 activations and KV cache"},
            "e2e": e2e, "gpu_launches": int(args.steps * (pre_l + dec_l)),
            "roofline": roofline, "kernels": kernels, "clocks": clk,
            "prefill_ms": statistics.median(prefill_ms), "decode_ms": dec_ms,
            "prefill_roofline": {"bound": "tensor", "kernel": "ssd_prefill_tc_kernel (all prefill projections) + prefill attention",
                                 "achieved": prefill_flops(w) / (statistics.median(prefill_ms) / 1e3) / 1e12,
                                 "peak": float(peaks.get("bf16_tflops", 1900.0)), "unit": "TFLOP/s",
                                 "frac": prefill_flops(w) / (statistics.median(prefill_ms) / 1e3) / 1e12
                                 / float(peaks.get("bf16_tflops", 1900.0)),
                                 "note": "whole-prefill time incl. attention and activation splits; "
                                         "flops counted as issued (bf16 hi + lo parts)"},
            "decode_tokens_per_s": (w.max_new - 1) / (dec_ms / 1e3),
            "decode_hbm_gbs": dec_bytes / (dec_ms / 1e3) / 1e9,
            "decode_hbm_frac": dec_bytes / (dec_ms / 1e3) / 1e9 / hbm_peak,
            "ssd_steps": st["steps"], "accepted": st["accepted"], "drafted": st["drafted"],
            "accept_hist": st["accept_hist"][: w.gamma + 1], "per_s": per_s}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        r = oracle_sample(w, bits, vis, prompt, max_steps=args.cpu_steps)
        line["cpu_baseline"] = {"value": r["value"], "unit": UNIT, "cores": r["cores"], "kind": "oracle",
                                "sample": (f"fp64 numpy oracle on this workload: prefill ({w.prompt_len} rows, "
                                           f"{r['prefill_s']:.1f} s) + {r['n_steps']} SSD steps "
                                           f"({r['step_s']:.2f} s each, {r['tokens_per_step']:.2f} tokens/step), "
                                           f"scaled to {w.max_new} tokens per request")}
    if rank == 0:
        print(json.dumps(line), flush=True)
    model.close()
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
