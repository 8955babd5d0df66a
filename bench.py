#!/usr/bin/env python
"""Benchmark: greedy generation (prefill + KV-cached decode) of a synthetic
Llama-family decoder through the C ABI on one GB300 per process.

One step = one generate pass over the workload: prefill of B x S prompt
tokens, then n_new decode steps (one new token per sequence each).
`value` = B * n_new / step time (generated tokens per second, the paper's
generate throughput measure; Sec. Results, Measures); the prefill and decode
phases are also reported separately.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle on the host cores

Under torchrun every rank runs an independent replica (no collective on the
data path); rank 0 prints one JSON line with the max-over-ranks time.
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

import synth_inputs as si  # noqa: E402

METRIC = "decode & prefill tokens/s on 1 GB300; % of HBM / BF16 tensor roofline"
DEFAULT_WORKLOAD = "0.5b_b1_s512_n128"


def model_bytes(m):
    L, D, H, G, d, F, V = (m[k] for k in ("L", "D", "H", "G", "d", "F", "V"))
    lin = L * ((H + 2 * G) * d * D + D * H * d + 2 * F * D + D * F)
    return lin, V * D


def decode_bytes_per_step(m, B, T_list):
    """Algorithmic HBM bytes of one decode step: every weight once (bf16),
    norms/biases, KV read of all cached tokens + the new token, KV write,
    fp32 logits write."""
    lin, head = model_bytes(m)
    L, D, G, d, V = m["L"], m["D"], m["G"], m["d"], m["V"]
    small = (2 * L + 1) * D * 4 + (L * (m["H"] + 2 * G) * d * 4 if m["bias"] else 0)
    kv_tok = L * 2 * G * d * 2
    kv_read = sum((t + 1) for t in T_list) * kv_tok
    kv_write = B * kv_tok
    return 2 * (lin + head) + small + kv_read + kv_write + B * V * 4


def prefill_flops(m, B, S):
    lin, head = model_bytes(m)
    attn = m["L"] * B * 4 * m["H"] * m["d"] * S * (S + 1) / 2
    return 2 * B * S * lin + attn + 2 * B * head


def read_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", 0)) or None, "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms."""

    def __init__(self, index):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits", "-lms",
                                       "200", "-i", str(index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                      text=True)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        out, _ = self.p.communicate(timeout=10)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def oracle_generate_timed(wl, budget_s=20.0):
    """Time the CPU oracle on a bounded sample of the workload's generate
    pass; returns (generated tokens/s, sample description)."""
    import torch
    from oracle import decoder as od
    m = si.MODEL_SHAPES[wl["model"]]
    B = wl.get("B", 1)
    S = wl.get("S", 512)
    w = si.make_weights(m, device="cpu")
    o = od.Oracle(od.DecoderConfig.from_dict(m), si.weights_as_f32_numpy(w), keep_f64=m["L"] * m["D"] < 100000)
    del w
    torch.set_num_threads(1)
    ids = si.make_ids(B, S, m["V"])
    cache = o.new_contiguous_cache(B, S + wl["n_new"] + 16)
    t0 = time.perf_counter()
    lg = o.prefill(ids, cache, last_only=True)[:, -1]
    t_pre = time.perf_counter() - t0
    tok = od.argmax_lowest(lg)
    lens = np.full(B, S)
    n = 0
    t1 = time.perf_counter()
    while n < wl["n_new"] and time.perf_counter() - t0 < budget_s:
        tok = od.argmax_lowest(o.decode_step(tok, cache, lens))
        lens = lens + 1
        n += 1
    t_dec = time.perf_counter() - t1
    per_step = t_dec / max(n, 1)
    # generate time for the full workload = prefill + n_new decode steps (decode
    # steps past the sample extrapolated at the sampled per-step time)
    t_full = t_pre + per_step * wl["n_new"]
    sample = (f"prefill B={B} S={S} timed in full ({t_pre:.2f}s) + {n} of {wl['n_new']} decode steps "
              f"({per_step * 1e3:.1f} ms/step), remainder extrapolated")
    return B * wl["n_new"] / t_full, sample, n


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


def run_reference(args, rank, world):
    if rank != 0:
        return
    wl = si.WORKLOADS[args.workload]
    vals = []
    sample = ""
    for _ in range(args.steps):
        v, sample, _ = oracle_generate_timed(wl, budget_s=15.0)
        vals.append(v)
    v = statistics.median(vals)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.workload},
        "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(si.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return

    import torch
    from paper_2608_19889_gb300 import build
    build.build()
    import paper_2608_19889_gb300 as ax

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    wl = si.WORKLOADS[args.workload]
    m = si.MODEL_SHAPES[wl["model"]]
    if wl["layout"] != "contiguous":
        raise SystemExit("paged workloads are benchmarked by a later revision")
    B, S, n_new = wl["B"], wl["S"], wl["n_new"]
    max_ctx = (S + n_new + 15) // 16 * 16
    w = si.make_weights(m, device="cuda")
    cfg = ax.make_config(m, max_batch=B, max_context=max_ctx, max_prefill_tokens=B * S)
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        model = ax.axon_model_create(cfg, w, stream=st)
    del w
    torch.cuda.empty_cache()

    ids = torch.from_numpy(si.make_ids(B, S, m["V"])).cuda()
    tok = torch.empty(B, dtype=torch.int32, device="cuda")
    ctx = torch.empty(B, dtype=torch.int32, device="cuda")
    logits = torch.empty(B, m["V"], device="cuda")
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]

    def one_step(events=None):
        if events:
            events[0].record(st)
        ax.axon_prefill(model, ids, logits_mode=ax.AXON_LOGITS_LAST, logits=logits, next_tokens=tok, stream=st)
        if events:
            events[1].record(st)
        ctx.fill_(S)  # positions restart at the prompt length (torch fill on the same stream)
        for _ in range(n_new):
            ax.axon_decode_step(model, tok, ctx, logits=logits, next_tokens=tok, stream=st)
        if events:
            events[2].record(st)

    with torch.cuda.stream(st):
        for _ in range(args.warmup):
            one_step()
    torch.cuda.synchronize()
    rc, bits = ax.axon_check_device(model, stream=st)
    if rc != 0:
        raise SystemExit(f"device check failed after warm-up: {rc} bits={bits}")

    clocks = ClockSampler(local)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    with torch.cuda.stream(st):
        for k in range(args.steps):
            one_step(ev[k])
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    if dist:
        dist.barrier()
    clk = clocks.stop()
    t_pre = [e[0].elapsed_time(e[1]) for e in ev]
    t_dec = [e[1].elapsed_time(e[2]) for e in ev]
    t_step = [e[0].elapsed_time(e[2]) for e in ev]
    ms = float(np.mean(t_step))
    if dist:
        t = torch.tensor([ms], device="cuda")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())

    # ---- end to end through the public API with host buffers: pinned ids in,
    # generated tokens out, copies inside the timed region.
    ids_h = torch.from_numpy(si.make_ids(B, S, m["V"])).pin_memory()
    out_h = torch.empty(n_new, B, dtype=torch.int32).pin_memory()
    hist = torch.empty(n_new, B, dtype=torch.int32, device="cuda")
    ids_d = torch.empty_like(ids)
    e2e_ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    e2e_ms = []
    with torch.cuda.stream(st):
        for k in range(args.steps):
            e2e_ev[0].record(st)
            ids_d.copy_(ids_h, non_blocking=True)
            ax.axon_prefill(model, ids_d, logits_mode=ax.AXON_LOGITS_LAST, logits=None, next_tokens=tok, stream=st)
            ctx.fill_(S)
            for t in range(n_new):
                ax.axon_decode_step(model, tok, ctx, logits=None, next_tokens=tok, stream=st)
                hist[t].copy_(tok)
            out_h.copy_(hist, non_blocking=True)
            e2e_ev[1].record(st)
            e2e_ev[1].synchronize()
            e2e_ms.append(e2e_ev[0].elapsed_time(e2e_ev[1]))
    e2e_val = B * n_new / (float(np.mean(e2e_ms)) / 1e3)

    hbm, tf_burst, tf_sus, peak_kind = read_peaks()
    T_list = [S + i for i in range(n_new)]
    dec_bytes = sum(decode_bytes_per_step(m, B, [T] * B) for T in T_list)
    dec_ms = float(np.mean(t_dec))
    dec_gbs = dec_bytes / (dec_ms / 1e3) / 1e9
    pre_flops = prefill_flops(m, B, S)
    pre_ms = float(np.mean(t_pre))
    pre_tflops = pre_flops / (pre_ms / 1e3) / 1e12
    # embed + 5 per layer + LM head + finaliser, for the prefill and each decode step
    launches_per_step = (5 * m["L"] + 3) * (1 + n_new)

    # ---- per-kernel timing (CUDA events around each launch, no graph) of one
    # prefill and of decode steps at the start, middle and end of the run.
    with torch.cuda.stream(st):
        prof_pre = ax.axon_profile_prefill(model, ids, next_tokens=tok, stream=st)
        prof_dec = {}
        for T in (S, S + n_new // 2, S + n_new - 1):
            ctx.fill_(T)
            for e in ax.axon_profile_decode_step(model, tok, ctx, next_tokens=tok, stream=st):
                a = prof_dec.setdefault(e["name"], dict(launches=0, total_ms=0.0, bytes=0.0, flops=0.0))
                for k in ("launches", "total_ms", "bytes", "flops"):
                    a[k] += e[k]
    torch.cuda.synchronize()
    # whole-run weight of each kernel kind: prefill once + n_new decode steps
    kinds = []
    for e in prof_pre:
        kinds.append((e["total_ms"], e["name"], e["launches"], e["total_ms"], e["bytes"], e["flops"]))
    for name, e in prof_dec.items():
        kinds.append((e["total_ms"] / 3 * n_new, name, e["launches"], e["total_ms"], e["bytes"], e["flops"]))
    kinds.sort(reverse=True)
    _, top_name, top_n, top_ms, top_bytes, top_flops = kinds[0]
    per_launch_ms = top_ms / top_n
    if top_name.startswith("prefill") and top_flops > 0 and top_bytes / top_flops < 0.05:
        ach = top_flops / top_n / (per_launch_ms / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": ach, "peak": tf_burst, "unit": "TFLOP/s", "frac": ach / tf_burst}
    else:
        ach = top_bytes / top_n / (per_launch_ms / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm}
    roof.update({"kernel": top_name, "launch_ms": per_launch_ms, "per_launch_units": (top_bytes if roof["bound"] == "hbm" else top_flops) / top_n,
                 "peak_kind": peak_kind, "traffic": None})
    kernel_table = {k[1]: {"share_of_run": k[0] / sum(x[0] for x in kinds), "launch_ms": k[3] / k[2]} for k in kinds}

    out = {
        "metric": METRIC,
        "value": world * B * n_new / (ms / 1e3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded random-init weights N(0,0.02), uniform random ids)",
        "config": {"workload": args.workload, "B": B, "S": S, "n_new": n_new, "layers": m["L"],
                   "hidden": m["D"], "vocab": m["V"], "kv": "contiguous",
                   "l2": "inputs larger than L2 (weights " + f"{2 * sum(model_bytes(m)) / 1e9:.2f} GB > 129 MB)"},
        "prefill_tok_s": world * B * S / (pre_ms / 1e3),
        "decode_tok_s": world * B * n_new / (dec_ms / 1e3),
        "prefill_ms": pre_ms,
        "decode_ms": dec_ms,
        "roofline": roof,
        "roofline_decode_step": {"bound": "hbm", "achieved": dec_gbs, "peak": hbm, "unit": "GB/s",
                                 "frac": dec_gbs / hbm, "peak_kind": peak_kind,
                                 "what": "all decode bytes (weights + KV + logits) / timed decode phase"},
        "roofline_prefill_phase": {"bound": "tensor", "achieved": pre_tflops, "peak": tf_burst, "unit": "TFLOP/s",
                                   "frac": pre_tflops / tf_burst, "peak_kind": peak_kind,
                                   "what": "prefill FLOPs / timed prefill phase"},
        "kernels": kernel_table,
        "e2e": {"value": world * e2e_val, "unit": "tokens/s", "h2d_bytes_per_step": B * S * 4,
                "d2h_bytes_per_step": B * n_new * 4},
        "gpu_launches": args.steps * launches_per_step,
        "clocks": clk,
        "wall_s": wall,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, sample, _ = oracle_generate_timed(wl, budget_s=15.0)
        out["cpu_baseline"] = {"value": v, "unit": "tokens/s", "cores": cores(), "kind": "oracle", "sample": sample}
    ax.axon_free(model)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
