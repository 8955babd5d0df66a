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
DEFAULT_WORKLOAD = "32b_b16_s2048_n256"


def moe_layers(m):
    """Layers with a mixture-of-experts MLP."""
    return max(0, m["L"] - m.get("first_dense", 0)) if m.get("n_experts", 0) else 0


def expected_active_experts(m, tokens):
    """Distinct experts that `tokens` tokens route to when each picks top_k
    of E uniformly: E (1 - (1 - k/E)^tokens). The algorithmic expert bytes
    of a decode step; the routing itself is decided on the device."""
    E, k = m["n_experts"], m["top_k"]
    return E * (1.0 - (1.0 - k / E) ** tokens)


def model_bytes(m, active_experts=None):
    """(linear weight elements, LM head elements). Mixture-of-experts layers
    count the router, the shared experts and `active_experts` routed experts
    (all E when None)."""
    L, D, H, G, d, F, V = (m[k] for k in ("L", "D", "H", "G", "d", "F", "V"))
    attn = (H + 2 * G) * d * D + D * H * d
    Lm = moe_layers(m)
    lin = L * attn + (L - Lm) * 3 * F * D
    if Lm:
        E, Fe = m["n_experts"], m["moe_F"]
        act = E if active_experts is None else active_experts
        lin += Lm * (E * D + 3 * m.get("n_shared", 0) * Fe * D + act * 3 * Fe * D)
    return lin, V * D


def linear_flops_per_token(m):
    """2 x the weight elements one token multiplies: attention projections,
    dense MLPs, and in MoE layers the router, the shared experts and top_k
    routed experts."""
    L, D, H, G, d, F = (m[k] for k in ("L", "D", "H", "G", "d", "F"))
    Lm = moe_layers(m)
    per = L * ((H + 2 * G) * d * D + D * H * d) + (L - Lm) * 3 * F * D
    if Lm:
        per += Lm * (m["n_experts"] * D + 3 * (m.get("n_shared", 0) + m["top_k"]) * m["moe_F"] * D)
    return 2 * per


def keys_seen(pos, window):
    """Keys a query at position pos attends to: pos + 1, or at most the
    sliding window."""
    return pos + 1 if not window else min(pos + 1, window)


def keys_seen_by_run(past, n, window):
    """Sum of keys_seen over positions past .. past + n - 1."""
    if not window:
        return n * past + n * (n + 1) / 2
    return sum(keys_seen(p, window) for p in range(past, past + n))


def decode_bytes_per_step(m, B, T_list):
    """Algorithmic HBM bytes of one decode step: every weight once (bf16),
    norms/biases, KV read of the keys each new token sees (all cached tokens
    + itself, or its sliding window), KV write, fp32 logits write."""
    lin, head = model_bytes(m, expected_active_experts(m, B) if moe_layers(m) else None)
    L, D, G, d, V = m["L"], m["D"], m["G"], m["d"], m["V"]
    small = (2 * L + 1) * D * 4 + (L * (m["H"] + 2 * G) * d * 4 if m["bias"] else 0)
    small += moe_layers(m) * m.get("n_experts", 0) * D * 2  # fp32 routers counted in bf16 above
    kv_tok = L * 2 * G * d * 2
    kv_read = sum(keys_seen(int(t), m.get("window", 0)) for t in T_list) * kv_tok
    kv_write = B * kv_tok
    return 2 * (lin + head) + small + kv_read + kv_write + B * V * 4


def prefill_flops(m, B, S):
    _, head = model_bytes(m)
    attn = m["L"] * B * 4 * m["H"] * m["d"] * keys_seen_by_run(0, S, m.get("window", 0))
    return B * S * linear_flops_per_token(m) + attn + 2 * B * head


def tensor_peak(burst, sustained, phase_ms):
    """Tensor-core peak for a kernel timed inside a phase of phase_ms: the
    burst figure for short phases, the power-capped sustained one for phases
    of 100 ms and more. fp16 and bf16 share one dense rate (nominal ratio 1),
    so the measured bf16 peak serves both."""
    if sustained and phase_ms >= 100.0:
        return sustained, "sustained"
    return burst, "burst"


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


def default_precision(workload):
    """Operand type the workload runs in by default: fp16 operands at the
    8B/32B widths, where bf16 operand rounding alone exceeds the 5e-2 logit
    tolerance; bf16 below."""
    return "fp16" if si.MODEL_SHAPES[si.WORKLOADS[workload]["model"]]["D"] >= 4096 else "bf16"


def _timed(fn):
    t0 = time.perf_counter()
    r = fn()
    return time.perf_counter() - t0, r


def oracle_full_model_timed(wl, budget_s=15.0):
    """Small models: the whole oracle on the workload's generate pass --
    prefill in full, then decode steps until the budget, the remaining steps
    extrapolated at the sampled per-step time. Returns (generated tokens/s,
    sample description)."""
    from oracle import decoder as od
    m = si.MODEL_SHAPES[wl["model"]]
    B, S = wl["B"], wl["S"]
    w = si.make_weights(m, device="cpu")
    o = od.Oracle(od.DecoderConfig.from_dict(m), si.weights_as_f32_numpy(w), keep_f64=True)
    del w
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
    per_step = (time.perf_counter() - t1) / max(n, 1)
    t_full = t_pre + per_step * wl["n_new"]
    sample = (f"whole model: prefill B={B} S={S} timed in full ({t_pre:.2f}s) + {n} of {wl['n_new']} decode "
              f"steps ({per_step * 1e3:.1f} ms/step), remaining steps extrapolated")
    return B * wl["n_new"] / t_full, sample


def oracle_one_layer_timed(wl, n_dec=2):
    """Large models: the oracle on one full-width layer plus the embedding,
    final norm and LM head, extrapolated by the layer count. The layer part
    is the difference between an L=1 and an L=0 run on the same float64
    weights (each a real oracle call), so
        t(model) = t(L=0) + L * (t(L=1) - t(L=0)).
    Contiguous workloads: prefill of one sequence at the workload's prompt
    length S (prefill sequences are independent: B of them take B times as
    long), then n_dec decode steps of the workload's whole batch B over a
    cache holding S tokens per sequence. Paged workloads: n_dec decode steps
    of the whole batch over a paged cache at the workload's context lengths,
    its K/V set to a constant (timing only: the oracle's cost does not depend
    on the values). Returns (generated tokens/s, sample description)."""
    from oracle import decoder as od
    m = si.MODEL_SHAPES[wl["model"]]
    V = m["V"]
    # the layer timed is a typical one: with a mixture of experts, the first
    # layer after the leading dense ones (which the base run includes)
    base = m.get("first_dense", 0) if m.get("n_experts", 0) else 0
    L = m["L"] - base
    m1 = dict(m, L=base + 1)
    w = si.make_weights(m1, device="cpu")
    W = si.weights_as_f32_numpy(w)
    del w
    o1 = od.Oracle(od.DecoderConfig.from_dict(m1), W, keep_f64=True)
    del W
    # the base layers only, on the same float64 arrays (no copy)
    o0 = od.Oracle(od.DecoderConfig.from_dict(dict(m, L=base)), o1.W, keep_f64=False)
    B, n_new = wl["B"], wl["n_new"]
    tok = si.make_ids(1, B, V, seed=7)[0]

    def decode_time(o, cache, lens):
        t0 = time.perf_counter()
        ln = np.asarray(lens, dtype=np.int64).copy()
        for _ in range(n_dec):
            o.decode_step(tok, cache, ln)
            ln = ln + 1
        return (time.perf_counter() - t0) / n_dec

    if wl["layout"] == "paged":
        lo, hi = wl["ctx"]
        lens = si.make_context_lens(B, lo, hi)
        max_ctx = (hi + n_new + 15) // 16 * 16
        caps = lens + n_new
        num_blocks = int(sum(-(-int(c) // 16) for c in caps)) + 64
        bt = si.make_block_table(caps, 16, max_ctx // 16, num_blocks)
        c1 = o1.new_paged_cache(num_blocks, 16, bt)
        for li in range(len(c1.K)):
            c1.K[li].fill(0.01)
            c1.V[li].fill(0.01)
        c0 = o0.new_paged_cache(num_blocks, 16, bt)
        d1 = decode_time(o1, c1, lens)
        d0 = decode_time(o0, c0, lens)
        per_step = d0 + L * max(d1 - d0, 0.0)
        sample = (f"one full-width layer + embedding/norm/LM head{" + " + str(base) + " leading dense layer(s)" if base else ""}, extrapolated by {L} layers: {n_dec} decode steps of "
                  f"B={B} over a paged cache at contexts {lo}..{hi} (K/V contents constant, timing only): "
                  f"{d1:.2f}s/step with the layer, {d0:.2f}s/step without")
        return B * n_new / (n_new * per_step), sample
    S = wl["S"]
    ids = si.make_ids(1, S, V)
    c1 = o1.new_contiguous_cache(1, S)
    p1, _ = _timed(lambda: o1.prefill(ids, c1, last_only=True))
    p0, _ = _timed(lambda: o0.prefill(ids, o0.new_contiguous_cache(1, S), last_only=True))
    cB = o1.new_contiguous_cache(B, S + n_dec)
    for li in range(len(cB.K)):
        cB.K[li][:, :S] = c1.K[li][0]
        cB.V[li][:, :S] = c1.V[li][0]
    del c1
    lens = np.full(B, S)
    d1 = decode_time(o1, cB, lens)
    d0 = decode_time(o0, o0.new_contiguous_cache(B, S + n_dec), lens)
    t_pre = B * (p0 + L * max(p1 - p0, 0.0))
    per_step = d0 + L * max(d1 - d0, 0.0)
    t_full = t_pre + n_new * per_step
    sample = (f"one full-width layer + embedding/norm/LM head{' + ' + str(base) + ' leading dense layer(s)' if base else ''}, "
              f"extrapolated by {L} layers: prefill of 1 x {S} tokens "
              f"({p1:.2f}s with the layer, {p0:.2f}s without; x B={B}) + {n_dec} decode steps of B={B} at context "
              f"{S} ({d1:.3f}s/step with the layer, {d0:.3f}s/step without); generate = prefill + {n_new} steps")
    return B * n_new / t_full, sample


def oracle_generate_timed(wl):
    """The CPU oracle on a bounded sample of the workload (about 10-30 s of
    host work): the whole model for the small configs, one layer extrapolated
    for the 8B/32B ones. Returns (generated tokens/s, sample, extrapolated)."""
    m = si.MODEL_SHAPES[wl["model"]]
    if wl["layout"] == "contiguous" and m["L"] * m["D"] * m["D"] < 5e7:
        v, s = oracle_full_model_timed(wl)
        return v, s, False
    v, s = oracle_one_layer_timed(wl)
    return v, s, True


def kernel_source_sha():
    """sha256 over the CUDA sources; a DRAM-traffic record taken from an ncu
    capture is only valid for the sources it was taken on."""
    import hashlib
    d = os.path.join(os.path.dirname(os.path.abspath(__file__)), "paper_2608_19889_gb300", "csrc")
    h = hashlib.sha256()
    for f in sorted(os.listdir(d)):
        if f.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(d, f), "rb") as fh:
                h.update(f.encode() + b"\0" + fh.read())
    return h.hexdigest()


def recorded_traffic(workload, precision, kind):
    """DRAM bytes per launch of profiler kind `kind` from the committed ncu
    summary profiles/dram_<workload>_<precision>.md (lines `traffic <kind>:
    <bytes>` after a `source_sha256:` line), or None when there is none or
    the CUDA sources changed since it was captured."""
    p = os.path.join(os.path.dirname(os.path.abspath(__file__)), "profiles", f"dram_{workload}_{precision}.md")
    if not os.path.exists(p):
        return None
    sha, rec = None, {}
    with open(p) as fh:
        for line in fh:
            line = line.strip().strip("`")
            if line.startswith("source_sha256:"):
                sha = line.split(":", 1)[1].strip()
            elif line.startswith("traffic ") and ":" in line:
                k, v = line[len("traffic "):].split(":", 1)
                try:
                    rec[k.strip()] = float(v)
                except ValueError:
                    pass
    if sha != kernel_source_sha():
        return None
    return rec.get(kind)


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


def max_over_ranks(ms, dist, device):
    """The slowest rank's time: every replica's timed region is bracketed by
    barriers, and the job is done when the last replica is."""
    if dist is None:
        return float(ms)
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank, world, ms):
    """Units all replicas processed (each rank runs the full workload on its
    own GPU, weak scaling) per second of the slowest rank."""
    return world * units_per_rank / (ms / 1e3)


def run_reference(args, rank, world):
    """The oracle as it stands on the host cores, on this arm's workload:
    one bounded sample (the same one as the GPU arm's cpu_baseline), timed
    once; its throughput stands for each of the --steps steps."""
    if rank != 0:
        return
    wl = si.WORKLOADS[args.workload]
    import torch
    torch.set_num_threads(max(1, cores()))
    v, sample, extrap = oracle_generate_timed(wl)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": args.workload},
        "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores(), "kind": "oracle",
                         "sample": sample + "; timed once", "extrapolated": extrap},
        "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


class GenerateRun:
    """Contiguous-cache workload: one step = prefill B x S + n_new decode steps."""

    def __init__(self, ax, torch, model, m, wl, st):
        self.ax, self.torch, self.model, self.m, self.st = ax, torch, model, m, st
        self.B, self.S, self.n_new = wl["B"], wl["S"], wl["n_new"]
        B = self.B
        self.ids = torch.from_numpy(si.make_ids(B, self.S, m["V"])).cuda()
        self.tok = torch.empty(B, dtype=torch.int32, device="cuda")
        self.ctx = torch.empty(B, dtype=torch.int32, device="cuda")
        self.logits = torch.empty(B, m["V"], device="cuda")
        self.bt = None
        self.kind = "contiguous"

    def step(self, ev=None):
        ax, st = self.ax, self.st
        if ev:
            ev[0].record(st)
        ax.axon_prefill(self.model, self.ids, logits_mode=ax.AXON_LOGITS_LAST, logits=self.logits,
                        next_tokens=self.tok, stream=st)
        if ev:
            ev[1].record(st)
        self.ctx.fill_(self.S)  # positions restart at the prompt length (torch fill on the same stream)
        for _ in range(self.n_new):
            ax.axon_decode_step(self.model, self.tok, self.ctx, logits=self.logits, next_tokens=self.tok, stream=st)
        if ev:
            ev[2].record(st)

    def e2e_step(self, ids_h, out_h, hist, ids_d):
        ax, st = self.ax, self.st
        ids_d.copy_(ids_h, non_blocking=True)
        ax.axon_prefill(self.model, ids_d, logits_mode=ax.AXON_LOGITS_LAST, logits=None, next_tokens=self.tok,
                        stream=st)
        self.ctx.fill_(self.S)
        for t in range(self.n_new):
            ax.axon_decode_step(self.model, self.tok, self.ctx, logits=None, next_tokens=self.tok, stream=st)
            hist[t].copy_(self.tok)
        out_h.copy_(hist, non_blocking=True)

    def host_inputs(self):
        return self.torch.from_numpy(si.make_ids(self.B, self.S, self.m["V"])).pin_memory(), self.ids

    def decode_positions(self):
        return [[self.S + i] * self.B for i in range(self.n_new)]

    def generated_per_step(self):
        return self.B * self.n_new

    def profile_positions(self):
        return [[self.S] * self.B, [self.S + self.n_new // 2] * self.B, [self.S + self.n_new - 1] * self.B]


PAGED_PREFILL_TOKENS = 16384  # rows per variable-length prefill call of the paged set-up


def varlen_prefill_flops(m, calls):
    """Algorithmic FLOPs of variable-length prefill calls; calls = list of
    [(past, chunk)] per call: every new token through every linear, causal
    attention of token past + i over past + i + 1 keys, the LM head on each
    chunk's last token."""
    _, head = model_bytes(m)
    total = 0.0
    for chunks in calls:
        T = sum(n for _, n in chunks)
        keys = sum(keys_seen_by_run(past, n, m.get("window", 0)) for past, n in chunks)
        total += T * linear_flops_per_token(m) + m["L"] * 4 * m["H"] * m["d"] * keys + 2 * len(chunks) * head
    return total


def plan_chunks(lens, budget):
    """Chunked prefill schedule: sequences in order, cut into calls of at
    most `budget` tokens; a sequence may continue in the next call. Returns
    per call (first sequence, [(past, chunk) per sequence])."""
    calls, cur, first, left = [], [], 0, budget
    b, done = 0, 0
    while b < len(lens):
        n = min(int(lens[b]) - done, left)
        if not cur:
            first = b
        cur.append((done, n))
        done += n
        left -= n
        if done == int(lens[b]):
            b, done = b + 1, 0
        if left == 0 or b == len(lens):
            calls.append((first, cur))
            cur, left = [], budget
    return calls


class PagedDecodeRun:
    """Paged-cache workload: sequences with context lengths drawn from [lo, hi]
    are prefilled into a shuffled block pool by chunked variable-length
    prefill calls of PAGED_PREFILL_TOKENS tokens (set-up, timed separately);
    one step = n_new decode steps of the whole batch."""

    def __init__(self, ax, torch, model, m, wl, st, lens, bt_np):
        self.ax, self.torch, self.model, self.m, self.st = ax, torch, model, m, st
        self.B, self.n_new = wl["B"], wl["n_new"]
        self.lens = torch.from_numpy(lens.astype(np.int32)).cuda()
        self.lens_np = lens
        self.bt = torch.from_numpy(bt_np).cuda()
        self.tok = torch.empty(self.B, dtype=torch.int32, device="cuda")
        self.first_tok = torch.empty(self.B, dtype=torch.int32, device="cuda")
        self.ctx = torch.zeros(self.B, dtype=torch.int32, device="cuda")
        self.logits = torch.empty(self.B, m["V"], device="cuda")
        self.kind = "paged"
        # chunked varlen prefill: each call covers consecutive sequences
        # [first, first + n) -- block-table rows and context lengths are
        # contiguous views -- with a piece of each
        seqs = [si.make_ids(1, int(lens[b]), m["V"], seed=100 + b)[0] for b in range(self.B)]
        self.calls = plan_chunks(lens, PAGED_PREFILL_TOKENS)
        staged = []
        for first, chunks in self.calls:
            ids = np.concatenate([seqs[first + i][p:p + n] for i, (p, n) in enumerate(chunks)]).astype(np.int32)
            cu = np.concatenate([[0], np.cumsum([n for _, n in chunks])]).astype(np.int32)
            staged.append((first, len(chunks), max(n for _, n in chunks), torch.from_numpy(ids).cuda(),
                           torch.from_numpy(cu).cuda()))
        nxt = torch.empty(self.B, dtype=torch.int32, device="cuda")
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        torch.cuda.synchronize()
        with torch.cuda.stream(st):
            ev[0].record(st)
            for first, n, mx, ids, cu in staged:
                ax.axon_prefill_varlen(model, ids, cu, self.ctx[first:first + n], mx,
                                       block_table=self.bt[first:first + n], next_tokens=nxt[:n], stream=st)
                # a sequence continued by the next call gets its token there
                self.first_tok[first:first + n].copy_(nxt[:n])
            ev[1].record(st)
        torch.cuda.synchronize()
        assert np.array_equal(self.ctx.cpu().numpy(), lens), "chunked prefill left wrong context lengths"
        self.prefill_ms = ev[0].elapsed_time(ev[1])
        self.prefill_tokens = int(lens.sum())
        self.prefill_flops = varlen_prefill_flops(m, [c for _, c in self.calls])

    def step(self, ev=None):
        ax, st = self.ax, self.st
        self.ctx.copy_(self.lens)
        self.tok.copy_(self.first_tok)
        if ev:
            ev[0].record(st)
            ev[1].record(st)
        for _ in range(self.n_new):
            ax.axon_decode_step(self.model, self.tok, self.ctx, block_table=self.bt, logits=self.logits,
                                next_tokens=self.tok, stream=st)
        if ev:
            ev[2].record(st)

    def e2e_step(self, tok_h, out_h, hist, tok_d):
        ax, st = self.ax, self.st
        tok_d.copy_(tok_h, non_blocking=True)
        self.ctx.copy_(self.lens)
        for t in range(self.n_new):
            ax.axon_decode_step(self.model, tok_d, self.ctx, block_table=self.bt, logits=None, next_tokens=tok_d,
                                stream=st)
            hist[t].copy_(tok_d)
        out_h.copy_(hist, non_blocking=True)

    def host_inputs(self):
        return self.first_tok.cpu().pin_memory(), self.tok

    def decode_positions(self):
        return [list(self.lens_np + i) for i in range(self.n_new)]

    def generated_per_step(self):
        return self.B * self.n_new

    def profile_positions(self):
        return [list(self.lens_np), list(self.lens_np + self.n_new // 2), list(self.lens_np + self.n_new - 1)]


def build_model(ax, torch, wl, m, st, layers=None, vocab=None, precision=0):
    m = dict(m)
    if layers is not None:
        m["L"] = layers
    if vocab is not None:
        m["V"] = vocab
    w = si.make_weights(m, device="cuda")
    lens = bt_np = None
    if wl["layout"] == "paged":
        B, (lo, hi) = wl["B"], wl["ctx"]
        lens = si.make_context_lens(B, lo, hi)
        max_ctx = (hi + wl["n_new"] + 15) // 16 * 16
        caps = lens + wl["n_new"]
        num_blocks = int(sum(-(-int(c) // 16) for c in caps)) + 64
        bt_np = si.make_block_table(caps, 16, max_ctx // 16, num_blocks)
        cfg = ax.make_config(m, max_batch=B, max_context=max_ctx, kv_layout=ax.AXON_KV_PAGED,
                             kv_num_blocks=num_blocks, max_prefill_tokens=PAGED_PREFILL_TOKENS,
                             precision=precision)
    else:
        B, S = wl["B"], wl["S"]
        max_ctx = (S + wl["n_new"] + 15) // 16 * 16
        cfg = ax.make_config(m, max_batch=B, max_context=max_ctx, max_prefill_tokens=B * S, precision=precision)
    with torch.cuda.stream(st):
        model = ax.axon_model_create(cfg, w, stream=st)
    del w
    torch.cuda.empty_cache()
    return model, m, lens, bt_np


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(si.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--precision", default="auto", choices=["auto", "bf16", "fp16"],
                    help="operand type on the tensor cores; fp16 converts the bf16 checkpoint to fp16 weights and splits "
                         "normalized activations into two fp16 terms (same weight bytes, same tensor rate); "
                         "auto: fp16 at the 8B/32B widths, bf16 below")
    ap.add_argument("--case", action="store_true",
                    help="profiling case: build the workload's model, run one prefill and --case-steps decode "
                         "steps, print nothing but a status line (for ncu)")
    ap.add_argument("--case-layers", type=int, default=None)
    ap.add_argument("--case-vocab", type=int, default=None)
    ap.add_argument("--case-steps", type=int, default=2)
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.precision == "auto":
        args.precision = default_precision(args.workload)
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
    st = torch.cuda.Stream()
    prec = ax.AXON_FP16 if args.precision == "fp16" else ax.AXON_BF16
    model, m, lens, bt_np = build_model(ax, torch, wl, si.MODEL_SHAPES[wl["model"]], st,
                                        layers=args.case_layers if args.case else None,
                                        vocab=args.case_vocab if args.case else None, precision=prec)
    if wl["layout"] == "paged":
        run = PagedDecodeRun(ax, torch, model, m, wl, st, lens, bt_np)
    else:
        run = GenerateRun(ax, torch, model, m, wl, st)
    B, n_new = run.B, run.n_new

    if args.case:
        with torch.cuda.stream(st):
            if run.kind == "contiguous":
                ax.axon_prefill(model, run.ids, next_tokens=run.tok, stream=st)
                run.ctx.fill_(run.S)
            else:
                run.ctx.copy_(run.lens)
                run.tok.copy_(run.first_tok)
            for _ in range(args.case_steps):
                ax.axon_decode_step(model, run.tok, run.ctx, block_table=run.bt, next_tokens=run.tok, stream=st)
        torch.cuda.synchronize()
        print("case ok", ax.axon_check_device(model, stream=st), flush=True)
        ax.axon_free(model)
        return

    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    with torch.cuda.stream(st):
        for _ in range(args.warmup):
            run.step()
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
            run.step(ev[k])
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    if dist:
        dist.barrier()
    clk = clocks.stop()
    t_pre = [e[0].elapsed_time(e[1]) for e in ev]
    t_dec = [e[1].elapsed_time(e[2]) for e in ev]
    t_step = [e[0].elapsed_time(e[2]) for e in ev]
    ms = max_over_ranks(np.mean(t_step), dist, "cuda")

    # ---- end to end through the public API with host buffers: inputs copied in
    # from pinned memory, generated tokens copied out, inside the timed region.
    in_h, in_d_like = run.host_inputs()
    in_d = torch.empty_like(in_d_like)
    out_h = torch.empty(n_new, B, dtype=torch.int32).pin_memory()
    hist = torch.empty(n_new, B, dtype=torch.int32, device="cuda")
    e2e_ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    e2e_ms = []
    e2e_steps = max(1, min(args.steps, 3))
    with torch.cuda.stream(st):
        run.e2e_step(in_h, out_h, hist, in_d)  # untimed: records this pointer set's decode graph
        torch.cuda.synchronize()
        for k in range(e2e_steps):
            e2e_ev[0].record(st)
            run.e2e_step(in_h, out_h, hist, in_d)
            e2e_ev[1].record(st)
            e2e_ev[1].synchronize()
            e2e_ms.append(e2e_ev[0].elapsed_time(e2e_ev[1]))
    e2e_val = whole_job_rate(run.generated_per_step(), world, max_over_ranks(np.mean(e2e_ms), dist, "cuda"))

    hbm, tf_burst, tf_sus, peak_kind = read_peaks()
    dec_bytes = sum(decode_bytes_per_step(m, B, T) for T in run.decode_positions())
    dec_ms = max_over_ranks(np.mean(t_dec), dist, "cuda")
    dec_gbs = dec_bytes / (dec_ms / 1e3) / 1e9

    # ---- per-kernel timing (CUDA events around each launch, no graph) of
    # decode steps at the start, middle and end of the run (and one prefill).
    prof_pre = []
    prof_dec = {}
    with torch.cuda.stream(st):
        if run.kind == "contiguous":
            prof_pre = ax.axon_profile_prefill(model, run.ids, next_tokens=run.tok, stream=st)
        positions = run.profile_positions()
        for pos in positions:
            run.ctx.copy_(torch.tensor(pos, dtype=torch.int32))
            for e in ax.axon_profile_decode_step(model, run.tok, run.ctx, block_table=run.bt, next_tokens=run.tok,
                                                 stream=st):
                a = prof_dec.setdefault(e["name"], dict(launches=0, total_ms=0.0, bytes=0.0, flops=0.0))
                for k in ("launches", "total_ms", "bytes", "flops"):
                    a[k] += e[k]
    torch.cuda.synchronize()
    # Kernel launches per timed step, counted by the profiler on the same
    # code path: one prefill (contiguous runs) + n_new decode steps.
    dec_launches = sum(e["launches"] for e in prof_dec.values()) / len(positions)
    launches_per_step = sum(e["launches"] for e in prof_pre) + n_new * dec_launches
    kinds = []  # (weight over the run, name, launches, ms, bytes, flops)
    for e in prof_pre:
        kinds.append((e["total_ms"], e["name"], e["launches"], e["total_ms"], e["bytes"], e["flops"]))
    for name, e in prof_dec.items():
        kinds.append((e["total_ms"] / 3 * n_new, name, e["launches"], e["total_ms"], e["bytes"], e["flops"]))
    kinds.sort(reverse=True)
    _, top_name, top_n, top_ms, top_bytes, top_flops = kinds[0]
    prof_pre_ms = sum(e["total_ms"] for e in prof_pre)
    per_launch_ms = top_ms / top_n
    if top_name.startswith("prefill") and top_flops > 0 and top_bytes / top_flops < 0.05:
        ach = top_flops / top_n / (per_launch_ms / 1e3) / 1e12
        tf, tf_kind = tensor_peak(tf_burst, tf_sus, prof_pre_ms)
        roof = {"bound": "tensor", "achieved": ach, "peak": tf, "unit": "TFLOP/s", "frac": ach / tf,
                "peak_which": tf_kind}
    else:
        ach = top_bytes / top_n / (per_launch_ms / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm}
    roof.update({"kernel": top_name, "launch_ms": per_launch_ms,
                 "per_launch_units": (top_bytes if roof["bound"] == "hbm" else top_flops) / top_n,
                 "peak_kind": peak_kind,
                 "traffic": recorded_traffic(args.workload, args.precision, top_name)})
    total_w = sum(x[0] for x in kinds)
    kernel_table = {k[1]: {"share_of_run": k[0] / total_w, "launch_ms": k[3] / k[2]} for k in kinds}

    config = {"workload": args.workload, "B": B, "n_new": n_new, "layers": m["L"], "hidden": m["D"],
              "vocab": m["V"], "kv": run.kind,
              "l2": "inputs larger than L2 (weights " + f"{2 * sum(model_bytes(m)) / 1e9:.2f} GB > 129 MB)"}
    out = {
        "metric": METRIC,
        "value": whole_job_rate(run.generated_per_step(), world, ms),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": args.precision,
        "data": "synthetic (seeded random-init weights N(0,0.02), uniform random ids)",
        "config": config,
        "decode_tok_s": whole_job_rate(B * n_new, world, dec_ms),
        "decode_ms": dec_ms,
        "roofline": roof,
        "roofline_decode_step": {"bound": "hbm", "achieved": dec_gbs, "peak": hbm, "unit": "GB/s",
                                 "frac": dec_gbs / hbm, "peak_kind": peak_kind,
                                 "what": "all decode bytes (weights + KV + logits) / timed decode phase"},
        "kernels": kernel_table,
        "e2e": {"value": e2e_val, "unit": "tokens/s", "steps": e2e_steps,
                "h2d_bytes_per_step": int(in_h.numel()) * 4, "d2h_bytes_per_step": B * n_new * 4},
        "gpu_launches": int(round(args.steps * launches_per_step)),
        "clocks": clk,
        "wall_s": wall,
    }
    if run.kind == "contiguous":
        S = run.S
        config["S"] = S
        pre_ms = max_over_ranks(np.mean(t_pre), dist, "cuda")
        pre_tflops = prefill_flops(m, B, S) / (pre_ms / 1e3) / 1e12
        out["prefill_tok_s"] = whole_job_rate(B * S, world, pre_ms)
        out["prefill_ms"] = pre_ms
        tf, tf_kind = tensor_peak(tf_burst, tf_sus, pre_ms)
        out["roofline_prefill_phase"] = {"bound": "tensor", "achieved": pre_tflops, "peak": tf,
                                         "unit": "TFLOP/s", "frac": pre_tflops / tf, "peak_kind": peak_kind,
                                         "peak_which": tf_kind, "what": "prefill FLOPs / timed prefill phase"}
    else:
        config["context_lens"] = f"uniform in {wl['ctx']}, mean {float(np.mean(run.lens_np)):.0f}"
        vl_tflops = run.prefill_flops / (run.prefill_ms / 1e3) / 1e12
        tf, tf_kind = tensor_peak(tf_burst, tf_sus, run.prefill_ms)
        out["setup_prefill"] = {"tokens": run.prefill_tokens, "ms": run.prefill_ms, "calls": len(run.calls),
                                "tok_s": run.prefill_tokens / (run.prefill_ms / 1e3),
                                "roofline": {"bound": "tensor", "achieved": vl_tflops, "peak": tf,
                                             "unit": "TFLOP/s", "frac": vl_tflops / tf,
                                             "peak_kind": peak_kind, "peak_which": tf_kind},
                                "what": f"chunked variable-length paged prefill of the contexts, "
                                        f"{PAGED_PREFILL_TOKENS}-token calls, ids already on the device "
                                        f"(not in value)"}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        torch.set_num_threads(max(1, cores()))
        v, sample, extrap = oracle_generate_timed(wl)
        out["cpu_baseline"] = {"value": v, "unit": "tokens/s", "cores": cores(), "kind": "oracle", "sample": sample,
                               "extrapolated": extrap}
    ax.axon_free(model)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
