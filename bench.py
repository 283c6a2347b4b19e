#!/usr/bin/env python3
"""Benchmark of one speculative step's KV-cache attention (BudgetDraft, Algorithm 2) on GB300.

A step = KV-budget selection + gamma drafter decode passes over the sparse view + the
verifier's (gamma+1)-query block pass, for every layer of the workload, through the C ABI.
Default workload: Llama-3-8B-shaped layer, batch 8, 16K context, B = 512 (4 sink, 128
recent), gamma = 5, window 32, selection with the carried window LSE.

Prints ONE JSON line.  value = algorithmic HBM bytes of all ranks' steps / max-over-ranks
time (GB/s); us_per_step and the per-kernel breakdown come from CUDA events on the
launching stream inside the timed region.  The step is captured in a CUDA graph; inputs
(K+V 537 MB at the default workload) exceed the 129 MB L2, so L2 is not flushed.

  python bench.py [--config l8b_16k_b8] [--budget 512] [--sel-mode carry|self]
                  [--steps K] [--warmup W] [--gpus N] [--impl reference]
"""

import os
import sys

if "OMP_NUM_THREADS" not in os.environ:   # host-side numpy here may use every core (the oracle's
                                          # worker processes run one BLAS thread each: OraclePool)
    _n = str(len(os.sched_getaffinity(0)))
    for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ.setdefault(_v, _n)

import argparse
import ctypes
import dataclasses
import json
import math
import statistics
import subprocess
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np
import torch

from paper_2606_00144_gb300 import workload as W

METRIC = "spec-step attention µs & HBM GB/s (% of ~8 TB/s) at 16K ctx, B=512, γ=5"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


# ----------------------------------------------------------------------------- bytes the method must read

def step_bytes(wl, budget, n_recent, sel_mode, n_sink=None):
    """Algorithmic HBM bytes of one step on one layer, by phase."""
    row = wl.head_dim * 2
    units = wl.batch * wl.h_kv
    t = wl.t_ctx
    sink = wl.n_sink if n_sink is None else n_sink
    if budget >= t:
        sel = 0
    else:
        sel = (t - sink - n_recent) * row * units               # middle keys, once
        if sel_mode == "self":
            sel += t * row * units                               # window LSE over the prefix
    draft = (min(budget, t) + wl.gamma) * 2 * row * units       # sparse view once + drafted rows
    verify = (t + wl.gamma + 1) * 2 * row * units
    return dict(select=sel, draft=draft, verify=verify, total=sel + draft + verify)


def view_rereads(wl):
    """Bytes of a step's sparse views read again by draft passes 2..gamma over all layers:
    counted for a stack, whose per-pass views together are far above L2."""
    view = min(wl.budget, wl.t_ctx) * 2 * wl.head_dim * 2 * wl.batch * wl.h_kv * wl.layers
    return (wl.gamma - 1) * view


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device):
        self.proc = None
        self.lines = []
        try:
            uuid = str(torch.cuda.get_device_properties(device).uuid)
            self.sel = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            self.sel = str(device)

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.sel, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        for ln in out.strip().splitlines():
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(self.NAMES, parts[3:7]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        loaded = sorted(sm)[len(sm) // 2:] or sm                # samples under load (upper half)
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- distributed helpers

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(x, world):
    """The largest x over the ranks (the slowest rank's time)."""
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(bytes_per_step_per_rank, steps, world, ms_max):
    """Whole-job GB/s: every rank runs its own replica of the step (weak scaling), so the
    job moves world x the per-rank bytes in the slowest rank's time."""
    return bytes_per_step_per_rank * steps * world / (ms_max / 1e3) / 1e9


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ----------------------------------------------------------------------------- events inside graphs

def timing_event():
    try:
        return torch.cuda.Event(enable_timing=True, external=True), None
    except TypeError:       # older torch: record through the driver with the external flag
        ev = torch.cuda.Event(enable_timing=True)
        ev.record()
        return ev, ctypes.CDLL("libcuda.so.1")


def record(ev_pair):
    ev, drv = ev_pair
    if drv is None:
        ev.record()
    else:
        drv.cuEventRecordWithFlags(ctypes.c_void_p(ev.cuda_event),
                                   ctypes.c_void_p(torch.cuda.current_stream().cuda_stream), ctypes.c_uint(1))


# ----------------------------------------------------------------------------- the GPU arm

class Step:
    """All layers of one workload: inputs, carried window LSE, one SpecStep per layer.

    `share`: another Step whose inputs and carried LSE this one reuses (a policy variant on
    the same data)."""

    def __init__(self, wl, budget, n_recent, sel_mode, device, share=None, n_sink=None, chunk=1, seq_lens=None):
        import paper_2606_00144_gb300 as bd
        self.wl, self.budget, self.n_recent, self.sel_mode = wl, budget, n_recent, sel_mode
        self.n_sink = wl.n_sink if n_sink is None else n_sink
        self.steps = [bd.SpecStep(wl.batch, wl.h_q, wl.h_kv, wl.head_dim, wl.t_ctx, wl.t_cap, budget, self.n_sink,
                                  n_recent, wl.window, wl.gamma, chunk, device, seq_lens)
                      for _ in range(wl.layers)]
        if share is not None:
            self.layers, self.lse = share.layers, share.lse
            return
        self.layers = [W.make_layer(wl, l, device) for l in range(wl.layers)]
        self.lse = []
        for st, inp in zip(self.steps, self.layers):
            # carried state: the window rows' LSE as the verify kernel leaves it
            self.lse.append(st.window_lse(inp.k_cache, inp.q_win) if sel_mode == "carry" else None)
        torch.cuda.synchronize()

    def launches_per_step(self):
        # selection: top-B only (B >= T), else score + top-B (+ the window-LSE pass in self mode)
        if self.budget >= self.wl.t_ctx:
            sel = 1
        else:
            sel = 2 + (1 if self.sel_mode == "self" else 0)
        return self.wl.layers * (sel + self.wl.gamma + 1)

    def run(self, marks=None, select=True):
        """One step; marks = [select, draft, verify, end] timing events (or None).  With
        select=False the sparse views of the last selection are reused (selection amortised
        over steps, as Algorithm 2 sparsifies once at prefill)."""
        L = range(self.wl.layers)
        if marks:
            record(marks[0])
        if select:
            # the window queries and LSE are this step's inputs, written before the kernel
            # that precedes the selection (the previous step's verify)
            for l in L:
                self.steps[l].select(self.layers[l].k_cache, self.layers[l].q_win, self.lse[l], window_ready=True)
        if marks:
            record(marks[1])
        for j in range(self.wl.gamma):
            for l in L:
                inp = self.layers[l]
                # the selection of layer l was not written by the kernel just before this one,
                # except for the first pass of a one-layer step (right after its top-B)
                ready = j > 0 or self.wl.layers > 1 or not select
                self.steps[l].draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache, view_ready=ready)
        if marks:
            record(marks[2])
        for l in L:
            inp = self.layers[l]
            self.steps[l].verify(inp.q_verify, inp.k_cache, inp.v_cache)
        if marks:
            record(marks[3])


def capture(fn, n):
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            for i in range(n):
                fn(i)
    torch.cuda.current_stream().wait_stream(s)
    return g


def timed_replays(graphs, world):
    barrier(world)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    # the GPU idles for about a millisecond ahead of the start event, so that the host's launch
    # of the first graph (and its one-time upload to the device) completes before the timed
    # region opens: the events then bracket the steps' kernels alone
    torch.cuda._sleep(1 << 21)
    t0.record()
    for g in graphs:
        g.replay()
    t1.record()
    torch.cuda.synchronize()
    barrier(world)
    return t0.elapsed_time(t1)


def graph_len(k, limit):
    """Steps per captured graph: the largest divisor of k not above limit, so that the
    timed region is a whole number of replays of one graph."""
    for s in range(max(1, min(k, limit)), 0, -1):
        if k % s == 0:
            return s
    return 1


def gpu_arm(args):
    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    wl = resolve_workload(args)
    n_recent = wl.n_recent
    budget = wl.budget
    step = Step(wl, budget, n_recent, args.sel_mode, "cuda")
    per = step_bytes(wl, budget, n_recent, args.sel_mode)
    layer_bytes = {k: v * wl.layers for k, v in per.items()}

    # eager warm-up (first calls set kernel attributes), then capture
    step.run()
    torch.cuda.synchronize()
    S = graph_len(args.steps, args.graph_steps)
    g_main = capture(lambda i: step.run(), S)
    marks = [[timing_event() for _ in range(4)] for _ in range(S)]
    g_marked = capture(lambda i: step.run(marks[i]), S)
    g_warm = capture(lambda i: step.run(), 1)
    for _ in range(args.warmup):
        g_warm.replay()
    torch.cuda.synchronize()

    # timed region: K steps, kernels only (programmatic dependent launch between them)
    sampler = ClockSampler(local)
    sampler.start()
    ms = timed_replays([g_main] * (args.steps // S), world)
    clocks = sampler.stop()
    ms = max_over_ranks(ms, world)
    # per-phase durations: the same K steps with event nodes between the phases (which
    # also stop the dependent-launch overlap at those boundaries); the last replay's marks
    timed_replays([g_marked] * (args.steps // S), world)
    ph = {"select": [], "draft": [], "verify": []}
    for i in range(S):
        e = [m[0] for m in marks[i]]
        ph["select"].append(e[0].elapsed_time(e[1]))
        ph["draft"].append(e[1].elapsed_time(e[2]))
        ph["verify"].append(e[2].elapsed_time(e[3]))
    phase_us = {k: 1000.0 * statistics.fmean(v) for k, v in ph.items()}

    ms_per_step = ms / args.steps
    us = 1000.0 * ms_per_step
    value = job_throughput(layer_bytes["total"], args.steps, world, ms)
    peak, peak_src = measured_hbm_peak()
    verify_launch_bytes = per["verify"]
    verify_us = phase_us["verify"] / wl.layers
    achieved = verify_launch_bytes / (verify_us * 1e-6) / 1e9
    line = {
        "metric": METRIC,
        "value": round(value, 1),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 5),
        "us_per_step": round(us, 2),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "accum": "f32",
        "data": "synthetic (seeded N(0,1) Q/K/V with planted heavy-hitter keys; see workload.py)",
        "config": {
            "workload": wl.name, "layers": wl.layers, "batch": wl.batch, "h_q": wl.h_q, "h_kv": wl.h_kv,
            "head_dim": wl.head_dim, "t_ctx": wl.t_ctx, "budget": budget, "n_sink": wl.n_sink,
            "n_recent": n_recent, "window": wl.window, "gamma": wl.gamma, "sel_mode": args.sel_mode,
            "parallelism": f"replicas x{world}", "graph_steps": S,
            "l2": "not flushed: K+V inputs (%.0f MB per layer) exceed the 129 MB L2"
                  % ((wl.t_cap * 2 * wl.head_dim * 2 * wl.batch * wl.h_kv) / 1e6),
        },
        "pct_of_8tbs": round(100.0 * value / world / NOMINAL_HBM_GBS, 1),
        "pct_of_measured_hbm": round(100.0 * value / world / peak, 1),
        "tokens_verified_per_s": round(wl.batch * (wl.gamma + 1) * world / (ms_per_step / 1e3), 1),
        "algorithmic_bytes_per_step": layer_bytes,
        "breakdown_us": {k: round(v, 2) for k, v in phase_us.items()},
        "roofline": {
            "kernel": "verify_kernel (bd_verify_attn)",
            "bound": "hbm",
            "achieved": round(achieved, 1),
            "peak": peak,
            "peak_source": peak_src,
            "unit": "GB/s",
            "frac": round(achieved / peak, 3),
            "bytes_per_launch": verify_launch_bytes,
            "traffic": profiled_traffic("verify_kernel", wl.name, ("bd_verify.cu", "bd_attn_warp.cuh", "bd_common.cuh")),
            "traffic_source": "profiles/verify_kernel_%s.md (ncu dram__bytes_read.sum + dram__bytes_write.sum)" % wl.name,
        },
        "gpu_launches": step.launches_per_step() * args.steps,
        "clocks": clocks,
    }
    # the oracle's processes start here (spawned: they import while the GPU lines below run)
    pool = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        pool = OraclePool(min(len(os.sched_getaffinity(0)), wl.batch * wl.h_kv * wl.layers))
    try:
        if not args.no_e2e:
            line["e2e"] = e2e_measure(step, args, world, layer_bytes["total"])
        if world == 1 and not args.no_extras:
            line["extras"] = extras(step, args)
            line["extras"]["configs"] = config_table(step, args, us, peak)
        if pool is not None:
            line["cpu_baseline"] = cpu_baseline(wl, budget, n_recent, args.sel_mode, args.cpu_seconds, pool)
            for name, row in line.get("extras", {}).get("configs", {}).items():
                cw = W.WORKLOADS[name]
                secs, n_unit, _ = oracle_step(pool, cw, cw.budget, cw.n_recent, "carry", layers=[0])
                row["cpu_oracle"] = {"us_per_step": round(1e6 * secs, 1), "cores": pool.n,
                                     "GB/s": round(row["bytes_per_step"] / secs / 1e9, 4),
                                     "ratio_gpu_vs_oracle": round(1e6 * secs / row["us_per_step"], 1),
                                     "sample": "one pass over every unit of layer 0" +
                                               (f", extrapolated x{cw.layers} to all layers" if cw.layers > 1 else "")}
    finally:
        if pool is not None:
            pool.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def time_per_step(fn, n_steps, graph_steps):
    """µs per call of fn, captured graph_steps calls per CUDA graph (CUDA events)."""
    S = graph_len(n_steps, graph_steps)
    fn()
    torch.cuda.synchronize()
    g = capture(lambda i: fn(), S)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    ms = timed_replays([g] * (n_steps // S), 1)
    return 1000.0 * ms / n_steps


VOCAB = 128256        # Llama-3 vocabulary (the logits rows the acceptance reads)


def extras(step, args):
    """Measurements of the steps beside the headline path (not part of `value`):
    selection amortised over steps, the greedy acceptance, and the paper's chunk policy."""
    import paper_2606_00144_gb300 as bd
    wl = step.wl
    n = args.extra_steps
    gs = args.graph_steps
    out = {}

    # drafts + verify only: the sparse views of one selection reused (Algorithm 2 sparsifies at prefill)
    per = step_bytes(wl, step.budget, step.n_recent, step.sel_mode)
    us = time_per_step(lambda: step.run(select=False), n, gs)
    b = (per["draft"] + per["verify"]) * wl.layers
    out["amortized_step"] = {"us_per_step": round(us, 2), "GB/s": round(b / (us * 1e-6) / 1e9, 1),
                             "bytes_per_step": b, "launches_per_step": wl.layers * (wl.gamma + 1)}

    # greedy acceptance (Eq. accept, Algorithm 2): arg max of every drafter pass and of the
    # verify block over a Llama-3 vocabulary, then the prefix test; synthetic bf16 logits
    gen = torch.Generator(device="cuda").manual_seed(wl.seed + 77)
    dl = torch.randn(wl.gamma, wl.batch, VOCAB, device="cuda", generator=gen).to(torch.bfloat16)
    vl = torch.randn(wl.batch, wl.gamma + 1, VOCAB, device="cuda", generator=gen).to(torch.bfloat16)
    d_ids = torch.empty(wl.gamma, wl.batch, dtype=torch.int32, device="cuda")
    v_ids = torch.empty(wl.batch, wl.gamma + 1, dtype=torch.int32, device="cuda")
    n_acc = torch.empty(wl.batch, dtype=torch.int32, device="cuda")
    emit = torch.empty(wl.batch, wl.gamma + 1, dtype=torch.int32, device="cuda")

    def accept():
        for j in range(wl.gamma):
            bd.bd_argmax(dl[j], d_ids[j])
        bd.bd_argmax(vl.view(-1, VOCAB), v_ids.view(-1))
        bd.bd_accept(d_ids, v_ids, n_acc, emit)

    def step_with_accept():
        # the step in its dependency order: each drafter pass is followed by its token choice
        L = range(wl.layers)
        for l in L:
            step.steps[l].select(step.layers[l].k_cache, step.layers[l].q_win, step.lse[l])
        for j in range(wl.gamma):
            for l in L:
                inp = step.layers[l]
                step.steps[l].draft(j, inp.q_draft[j], inp.k_cache, inp.v_cache, view_ready=j > 0 or wl.layers > 1)
            bd.bd_argmax(dl[j], d_ids[j])
        for l in L:
            inp = step.layers[l]
            step.steps[l].verify(inp.q_verify, inp.k_cache, inp.v_cache)
        bd.bd_argmax(vl.view(-1, VOCAB), v_ids.view(-1))
        bd.bd_accept(d_ids, v_ids, n_acc, emit)

    us_acc = time_per_step(accept, n, gs)
    us_full = time_per_step(step_with_accept, n, gs)
    lb = (dl.numel() + vl.numel()) * 2
    out["accept"] = {"vocab": VOCAB, "us_per_step": round(us_acc, 2), "logits_bytes": lb,
                     "GB/s": round(lb / (us_acc * 1e-6) / 1e9, 1), "launches_per_step": wl.gamma + 2,
                     "step_with_accept_us": round(us_full, 2)}

    # self mode: the window LSE computed in the call instead of carried (same inputs)
    if step.budget < wl.t_ctx and step.sel_mode == "carry":
        v = Step(wl, step.budget, step.n_recent, "self", "cuda", share=step)
        v.lse = [None] * wl.layers
        us = time_per_step(v.run, n, gs)
        pb = step_bytes(wl, step.budget, step.n_recent, "self")["total"] * wl.layers
        out["self_mode"] = {"us_per_step": round(us, 2), "GB/s": round(pb / (us * 1e-6) / 1e9, 1),
                            "bytes_per_step": pb, "launches_per_step": v.launches_per_step()}
        del v

    # token-level budget sweep with a recent window of B/4 (B >= T keeps the whole context)
    rows = []
    for bb in (256, 512, 1024, 2048, wl.t_ctx):
        rec = min(bb // 4, wl.t_ctx)
        v = Step(wl, bb, rec, step.sel_mode, "cuda", share=step)
        us = time_per_step(v.run, n, gs)
        pb = step_bytes(wl, bb, rec, step.sel_mode)["total"] * wl.layers
        rows.append({"budget": bb, "n_recent": rec, "us_per_step": round(us, 2),
                     "GB/s": round(pb / (us * 1e-6) / 1e9, 1), "bytes_per_step": pb})
        del v
    out["budget_sweep"] = rows

    # the paper's chunk policy (Sec. 3.4, s = 8): same sink/recent/budget, and the pure
    # top-floor(B/s)-chunks form with no sink or recent window over a budget sweep
    if step.budget < wl.t_ctx:
        rows = []
        cases = [(step.budget, wl.n_sink, step.n_recent)] + [(bb, 0, 0) for bb in (256, 512, 1024, 2048)]
        for bb, sink, rec in cases:
            v = Step(wl, bb, rec, step.sel_mode, "cuda", share=step, n_sink=sink, chunk=8)
            us = time_per_step(v.run, n, gs)
            pb = step_bytes(wl, bb, rec, step.sel_mode, n_sink=sink)["total"] * wl.layers
            rows.append({"budget": bb, "n_sink": sink, "n_recent": rec, "chunk": 8, "us_per_step": round(us, 2),
                         "GB/s": round(pb / (us * 1e-6) / 1e9, 1)})
            del v
        out["chunk_policy"] = rows
        # a ragged batch: per-sequence context lengths spread over the lower quarter of T (the
        # same cache, window and carried LSE; the timing does not depend on their values)
        lens = [wl.t_ctx - (wl.t_ctx // 4) * i // max(1, wl.batch - 1) for i in range(wl.batch)]
        lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
        v = Step(wl, step.budget, step.n_recent, step.sel_mode, "cuda", share=step, seq_lens=lens_d)
        us = time_per_step(v.run, n, gs)
        row, units_per_seq = wl.head_dim * 2, wl.h_kv
        rb = sum(((t - wl.n_sink - step.n_recent) + (min(step.budget, t) + wl.gamma) * 2 + (t + wl.gamma + 1) * 2)
                 * row * units_per_seq for t in lens) * wl.layers
        out["ragged_lengths"] = {"seq_lens": lens, "us_per_step": round(us, 2), "GB/s": round(rb / (us * 1e-6) / 1e9, 1),
                                 "bytes_per_step": rb}
        del v
        if step.sel_mode == "carry":   # the same batch with the window LSE computed in the call
            v = Step(wl, step.budget, step.n_recent, "self", "cuda", share=step, seq_lens=lens_d)
            v.lse = [None] * wl.layers
            out["ragged_lengths"]["self_mode_us_per_step"] = round(time_per_step(v.run, n, gs), 2)
            del v
    out["note"] = "each timed over %d graphed steps outside the headline timed region" % n
    return out


CONFIGS = ("tiny_1k", "l8b_4k", "l8b_8k_b4", "l8b_16k_b8", "l8b_32L_16k_b16")


def config_table(head, args, head_us, peak):
    """Every evaluation workload at its own budget, carry mode, graphed steps: µs per step,
    tokens verified per second (batch x (gamma + 1) per step), algorithmic bytes and their
    rate against 8 TB/s and the measured HBM peak.  The headline workload's row is the
    headline measurement itself."""
    rows = {}
    for name in CONFIGS:
        wl = W.WORKLOADS[name]
        if name == head.wl.name and head.budget == wl.budget and head.sel_mode == "carry":
            us, n = head_us, args.steps
        else:
            st = Step(wl, wl.budget, wl.n_recent, "carry", "cuda")
            n = args.extra_steps if wl.layers == 1 else max(20, args.extra_steps // 25)
            us = time_per_step(st.run, n, args.graph_steps if wl.layers == 1 else 5)
            del st
            torch.cuda.empty_cache()
        b = step_bytes(wl, wl.budget, wl.n_recent, "carry")["total"] * wl.layers
        gbs = b / (us * 1e-6) / 1e9
        rows[name] = {"layers": wl.layers, "batch": wl.batch, "t_ctx": wl.t_ctx, "budget": wl.budget,
                      "n_sink": wl.n_sink, "n_recent": wl.n_recent, "gamma": wl.gamma, "steps_timed": n,
                      "us_per_step": round(us, 2),
                      "tokens_verified_per_s": round(wl.batch * (wl.gamma + 1) / (us * 1e-6), 1),
                      "bytes_per_step": b, "GB/s": round(gbs, 1), "pct_of_8tbs": round(100 * gbs / NOMINAL_HBM_GBS, 1),
                      "frac_of_measured_hbm": round(gbs / peak, 3)}
        if wl.layers > 1:
            # a stack's per-pass sparse views are read again by each of the gamma passes:
            # the bytes with the views counted gamma times
            bg = b + view_rereads(wl)
            gbg = bg / (us * 1e-6) / 1e9
            rows[name].update({"bytes_per_step_views_x_gamma": bg, "GB/s_views_x_gamma": round(gbg, 1),
                               "frac_of_measured_hbm_views_x_gamma": round(gbg / peak, 3)})
    return rows


def e2e_measure(step, args, world, bytes_per_step):
    """The same steps driven from pinned host buffers through HostStepIO (the package's
    host-buffer API): every step copies its inputs host->device and its results back,
    packed, on a side stream overlapping the neighbouring steps' kernels."""
    import paper_2606_00144_gb300 as bd
    wl = step.wl
    g1 = wl.gamma + 1
    layers = [(st, inp.k_cache, inp.v_cache, step.lse[l] is not None)
              for l, (st, inp) in enumerate(zip(step.steps, step.layers))]
    io = bd.HostStepIO(layers)
    for slot in range(2):
        h = io.host_inputs(slot)
        for l, inp in enumerate(step.layers):
            h[f"q_win{l}"].copy_(inp.q_win)
            h[f"q_draft{l}"].copy_(inp.q_draft)
            h[f"q_verify{l}"].copy_(inp.q_verify)
            h[f"k_rows{l}"].copy_(inp.k_cache[:, :, wl.t_ctx: wl.t_ctx + g1])
            h[f"v_rows{l}"].copy_(inp.v_cache[:, :, wl.t_ctx: wl.t_ctx + g1])
            if step.lse[l] is not None:
                h[f"lse{l}"].copy_(step.lse[l])
    torch.cuda.synchronize()
    S = graph_len(args.steps, args.graph_steps)
    io.run(2)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            io.run(S)
    torch.cuda.current_stream().wait_stream(s)
    g.replay()
    torch.cuda.synchronize()
    ms = timed_replays([g] * (args.steps // S), world)
    ms = max_over_ranks(ms, world)
    value = job_throughput(bytes_per_step, args.steps, world, ms)
    return {"value": round(value, 1), "unit": "GB/s", "us_per_step": round(1000.0 * ms / args.steps, 2),
            "h2d_bytes_per_step": io.bytes_in, "d2h_bytes_per_step": io.bytes_out,
            "api": "paper_2606_00144_gb300.HostStepIO (packed pinned-host transfers on two side streams, "
                   "double-buffered) around SpecStep through the C ABI, one CUDA graph"}


def code_lines(text):
    """The source without whole-line comments and blank lines: what the kernel is built from
    (a comment edit leaves the profiled counters valid)."""
    return "\n".join(ln.strip() for ln in text.splitlines() if ln.strip() and not ln.strip().startswith("//"))


def profiled_traffic(kernel, workload, sources):
    """dram bytes read + written per launch from the committed ncu summary, or None when
    the summary is missing or was taken on other kernel sources than the ones built now."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    h = hashlib.sha256()
    for f in sources:
        with open(os.path.join(ROOT, "paper_2606_00144_gb300", "csrc", f)) as fh:
            h.update(code_lines(fh.read()).encode())
    fields = dict(ln.split(":", 1) for ln in text.splitlines() if ln.startswith(("source_sha256:", "traffic_bytes")))
    if fields.get("source_sha256", "").split()[0:1] != [h.hexdigest()[:16]]:
        return None
    try:
        return int(fields["traffic_bytes_per_launch"].strip())
    except (KeyError, ValueError):
        return None


def measured_hbm_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs, copy)"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ----------------------------------------------------------------------------- oracle timing

def unit_bytes(wl, budget, n_recent, sel_mode, n_sink=None):
    """Algorithmic bytes of one (sequence, KV head) unit's step."""
    units = wl.batch * wl.h_kv
    return step_bytes(wl, budget, n_recent, sel_mode, n_sink)["total"] / units


def _draw_sequence(wl, layer, b):
    """Sequence b of `layer` drawn on the host by the workload recipe, as fp64 arrays."""
    one = dataclasses.replace(wl, batch=1)
    inp = W.make_layer(one, layer, "cpu", first_seq=b)
    f = lambda t: t.to(torch.float64).numpy()
    return tuple(map(f, (inp.k_cache, inp.v_cache, inp.q_win, inp.q_draft, inp.q_verify)))


def _oracle_worker(rank, tasks, results, barrier):
    """One host core (single-threaded BLAS): per task, draws its (layer, sequence, KV head)
    units' inputs and the carried window LSE (not timed), then for every pass waits for the
    other workers and runs the oracle's whole step on each of its units: the selection, the
    gamma draft passes over the oracle's own view, the verify block."""
    import oracle
    while True:
        task = tasks.get()
        if task is None:
            return
        wl, budget, n_recent, sel_mode, units, passes = task
        g = wl.group
        data, seq = [], {}
        for (l, b, kv) in units:
            if (l, b) not in seq:
                seq.clear()
                seq[(l, b)] = _draw_sequence(wl, l, b)
            K, V, QW, QD, QV = seq[(l, b)]
            hs = slice(kv * g, (kv + 1) * g)
            u = dict(K=K[:, kv:kv + 1].copy(), V=V[:, kv:kv + 1].copy(), QW=QW[:, hs].copy(),
                     QD=QD[:, :, hs].copy(), QV=QV[:, hs].copy())
            u["lse"] = oracle.window_lse(u["QW"], u["K"], wl.t_ctx) if sel_mode == "carry" else None
            data.append(u)
        seq.clear()
        out = []
        for _ in range(passes):
            barrier.wait()
            t0 = time.monotonic()
            for u in data:
                oracle.spec_step(u["K"], u["V"], u["QW"], u["QD"], u["QV"], wl.t_ctx, budget, wl.n_sink, n_recent,
                                 lse_win=u["lse"])
            out.append((t0, time.monotonic(), len(data)))
        results.put((rank, out))


class OraclePool:
    """The fp64 oracle on the host cores: one spawned process per core of
    os.sched_getaffinity(0), each with single-threaded BLAS, over independent
    (layer, sequence, KV head) units.  A pass runs every unit of the sample once, all
    workers starting together; its time is the span from the first start to the last end."""

    def __init__(self, n_workers=None):
        import multiprocessing as mp
        self.n = max(1, n_workers or len(os.sched_getaffinity(0)))
        ctx = mp.get_context("spawn")
        self.barrier = ctx.Barrier(self.n)
        self.tasks = [ctx.Queue() for _ in range(self.n)]
        self.results = ctx.Queue()
        saved = {v: os.environ.get(v) for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
        os.environ.update({v: "1" for v in saved})            # the children inherit one BLAS thread each
        try:
            self.procs = [ctx.Process(target=_oracle_worker, args=(i, self.tasks[i], self.results, self.barrier),
                                      daemon=True) for i in range(self.n)]
            for p in self.procs:
                p.start()
        finally:
            for v, x in saved.items():
                if x is None:
                    os.environ.pop(v, None)
                else:
                    os.environ[v] = x

    def run(self, wl, budget, n_recent, sel_mode, units, passes):
        """Runs `passes` passes over `units` [(layer, b, kv)]; returns [(seconds, unit_steps)] per pass."""
        per = (len(units) + self.n - 1) // self.n
        for i in range(self.n):
            self.tasks[i].put((wl, budget, n_recent, sel_mode, units[i * per:(i + 1) * per], passes))
        res = [self.results.get(timeout=3600) for _ in range(self.n)]
        spans = []
        for p in range(passes):
            starts = [r[1][p][0] for r in res]
            ends = [r[1][p][1] for r in res]
            spans.append((max(ends) - min(starts), sum(r[1][p][2] for r in res)))
        return spans

    def close(self):
        for q in self.tasks:
            q.put(None)
        for p in self.procs:
            p.join(timeout=30)


def layer_units(wl, layers=None):
    layers = range(wl.layers) if layers is None else layers
    return [(l, b, kv) for l in layers for b in range(wl.batch) for kv in range(wl.h_kv)]


def oracle_step(pool, wl, budget, n_recent, sel_mode, layers=None, passes=1):
    """The oracle's time for one whole step of the workload (every unit of the given layers,
    scaled to all layers when only a sample of them ran)."""
    units = layer_units(wl, layers)
    spans = pool.run(wl, budget, n_recent, sel_mode, units, passes)
    secs = sum(s for s, _ in spans) / len(spans)
    scale = wl.layers / (len(units) / (wl.batch * wl.h_kv))
    return secs * scale, len(units) * len(spans), secs


def cpu_baseline(wl, budget, n_recent, sel_mode, budget_s=12.0, pool=None):
    own = pool is None
    pool = pool or OraclePool(min(len(os.sched_getaffinity(0)), wl.batch * wl.h_kv))
    try:
        # one pass to size the sample, then enough whole-layer passes for about budget_s of CPU work
        s1, _, _ = oracle_step(pool, wl, budget, n_recent, sel_mode, layers=[0])
        passes = max(1, min(50, int(budget_s / max(s1 * pool.n, 1e-3))))
        secs, n_unit, _ = oracle_step(pool, wl, budget, n_recent, sel_mode, layers=[0], passes=passes)
    finally:
        if own:
            pool.close()
    step_b = step_bytes(wl, budget, n_recent, sel_mode)["total"]
    return {"value": round(step_b / secs / 1e9, 4), "unit": "GB/s", "cores": pool.n, "kind": "oracle",
            "us_per_step": round(1e6 * secs, 1),
            "sample": f"{passes} whole steps of one layer ({wl.batch * wl.h_kv} (sequence, KV head) units, each the "
                      f"selection with {'the carried' if sel_mode == 'carry' else 'its own'} window LSE, "
                      f"{wl.gamma} draft passes and the verify block), the "
                      f"units spread over {pool.n} single-threaded processes; numpy fp64"}


def reference_arm(args):
    world, rank, local = dist_env()
    if rank != 0:
        return
    wl = resolve_workload(args)
    units = layer_units(wl, [0])
    pool = OraclePool(min(len(os.sched_getaffinity(0)), len(units)))
    try:
        spans = pool.run(wl, wl.budget, wl.n_recent, args.sel_mode, units, args.warmup + args.steps)
    finally:
        pool.close()
    secs = sum(s for s, _ in spans[args.warmup:])
    step_b = step_bytes(wl, wl.budget, wl.n_recent, args.sel_mode)["total"]
    value = step_b * args.steps / secs / 1e9
    sample = (f"each step = one whole step of one layer of the workload ({len(units)} (sequence, KV head) units: "
              f"selection with the carried window LSE, {wl.gamma} draft passes, the verify block) on "
              f"{pool.n} single-threaded processes; fp64 numpy oracle")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * secs / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (same recipe as the GPU arm, drawn on the host)",
        "config": {"workload": wl.name, "layers": wl.layers, "batch": wl.batch, "h_q": wl.h_q, "h_kv": wl.h_kv,
                   "head_dim": wl.head_dim, "t_ctx": wl.t_ctx, "budget": wl.budget, "n_sink": wl.n_sink,
                   "n_recent": wl.n_recent, "window": wl.window, "gamma": wl.gamma, "sel_mode": args.sel_mode},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": pool.n, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    if wl.layers > 1:
        line["note"] = f"one layer of {wl.layers} per step"
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- CLI

def resolve_workload(args):
    wl = W.WORKLOADS[args.config]
    if args.budget is not None and args.budget != wl.budget:
        wl = wl.with_budget(args.budget)
    return wl


def parse():
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=4000)
    p.add_argument("--warmup", type=int, default=50)
    p.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    p.add_argument("--config", default="l8b_16k_b8", choices=sorted(W.WORKLOADS))
    p.add_argument("--budget", type=int, default=None)
    p.add_argument("--sel-mode", choices=["carry", "self"], default="carry")
    p.add_argument("--graph-steps", type=int, default=100, help="steps captured per CUDA graph")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-extras", action="store_true", help="skip the amortised / acceptance / chunk-policy lines")
    p.add_argument("--extra-steps", type=int, default=500)
    a = p.parse_args()
    if a.warmup < 3:
        p.error("--warmup must be >= 3")
    return a


def main():
    args = parse()
    if args.impl == "reference":
        reference_arm(args)
    else:
        gpu_arm(args)


if __name__ == "__main__":
    main()
