#!/usr/bin/env python3
"""Benchmark of the Gefen optimizer step on the Llama-3-style ~1.5B set.

A step is one Gefen iteration (Algorithm 1) over all 182 tensors (1,479,100,416
fp32 parameters, bf16 gradients, u8 codes), with the workload's cadence: every
10th step also histograms the normalised momentum (4096 cells, 16 per level)
and refits the 256-level codebook by the exact DP (Algorithm 3); the next step
decodes with the old codebook and encodes with the new one.  Blocks are
inferred once from the first gradient (Algorithm 2) and the first codebook is
learned from it.

`--workload flat:N:P` runs one flat tensor of N parameters with blocks of P
(given, not inferred): the small case the kernel profiles are taken on.

Prints one JSON line.  `value` is whole-job parameters updated per second over
the timed steps (refit steps included); `e2e` is the same metric through the
public call with the gradient copied in from pinned host memory and the step's
status word read back every step (and, as a second figure, all updated
parameters copied back too).  `--impl reference` times the CPU oracle instead, on a bounded
sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

WORKLOAD = "llama-1.5b"  # the default; --workload selects another
METRIC = "Gefen step throughput (Gparams/s)"
UNIT = "Gparams/s"
REFIT_EVERY = 10
BINS = 4096          # Algorithm 3: 16k cells with k = 256
MICRO_BINS = 65536   # the refit micro-benchmark
MICRO_N = 1_499_987_968  # 1.5e9 values rounded to whole blocks of 4096
K = 256
HP = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0)  # Appendix I, Llama
SEED = 0
PROFILE = os.path.join(ROOT, "profiles", "step_stream4k_llama1p5b.md")
DOMINANT = "k_step_stream<4096> (blocks of p <= 4096, p % 16 == 0, p > 1)"


def dominant(p: int) -> bool:
    """Tensors served by the streamed 4096-element tile kernel, the one that
    carries most of the step's bytes on this workload."""
    return p > 1 and p % 16 == 0 and p <= 4096


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def step_kernel_source_hash() -> str:
    h = hashlib.sha256()
    for f in ("step.cu", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2606_13894_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(n_elems: int):
    """DRAM bytes of one launch of the dominant kernel: the committed ncu
    summary's bytes per element times the elements one launch processes here;
    None when the summary is missing or the kernel source changed since."""
    try:
        txt = open(PROFILE).read()
    except OSError:
        return None
    m = re.search(r"source_hash:\s*([0-9a-f]+)", txt)
    t = re.search(r"dram_bytes_per_element:\s*([0-9.eE+]+)", txt)
    if not m or not t or m.group(1) != step_kernel_source_hash():
        return None
    return float(t.group(1)) * n_elems


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.p = None
        self.path = os.path.join("/tmp", f"gefen_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.p = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "50"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        try:
            os.remove(self.path)
        except OSError:
            pass
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def job_time_ms(elapsed_ms: float, world: int, device) -> float:
    """The job's time over the timed steps: the slowest rank's (every rank
    starts after the same barrier), agreed by all ranks."""
    if world == 1:
        return elapsed_ms
    import torch.distributed as dist
    t = torch.tensor([elapsed_ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.barrier()
    return float(t.item())


def whole_job_value(params_per_rank: int, world: int, steps: int, job_ms: float) -> float:
    """Parameters all replicas updated per second (each rank steps its own
    copy of the workload: weak scaling), in Gparams/s."""
    return world * params_per_rank * steps / (job_ms * 1e-3) / 1e9


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def launches_per_call(periods, flags_hist: bool) -> int:
    """Kernels one gefen_step call launches for these periods (mirrors the
    library's path classes; fewer than 300 tensors per class)."""
    if not periods:
        return 0
    cls = set()
    big = 0
    for p in periods:
        if p == 1:
            cls.add("p1")
        elif p % 16 == 0 and p <= 4096:
            cls.add("s4k")
        elif p % 16 == 0 and p <= 8192:
            cls.add("s8k")
        elif p % 16 == 0 and p <= 16384:
            cls.add("t16v4")
        elif p <= 2048:
            cls.add("gen")
        else:
            big |= 1 if p % 16 == 0 else 2
    n = len(cls) + 3 * bin(big).count("1")
    return n + (1 if flags_hist else 0)


def workload_specs(synth, name: str):
    """Tensor specs of a workload, and its periods when they are given rather
    than inferred (flat:N:P)."""
    if name.startswith("flat:"):
        _, n, p = name.split(":")
        n, p = int(float(n)), int(p)
        if n % p:
            raise SystemExit(f"flat workload: {n} is not a multiple of {p}")
        return synth.flat_set(n, p), [p]
    return synth.CONFIGS[name](), None


def period_summary(specs, periods):
    """Inferred period -> (tensors, params) over the workload."""
    out = {}
    for s, p in zip(specs, periods):
        t, n = out.get(str(p), (0, 0))
        out[str(p)] = (t + 1, n + s.numel)
    return out


# ----------------------------------------------------------------- GPU arm
def run_gpu(args, world, rank, local):
    from paper_2606_13894_gb300 import gefen as G
    from paper_2606_13894_gb300 import synth

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    G.load()
    specs, given_periods = workload_specs(synth, args.workload)
    offs, total = synth.pack_offsets(specs)
    nparams = synth.total_params(specs)
    stream = torch.cuda.current_stream()

    theta = synth.init_params(specs, SEED + rank, device=dev)
    gpool = [synth.draw_grads(specs, SEED + rank, step=s, device=dev) for s in (1, 2)]
    torch.cuda.synchronize()

    # Algorithm 2 on the first gradient of every tensor
    t0 = time.perf_counter()
    periods = list(given_periods) if given_periods else []
    iws = None
    for s, o in zip(specs, offs) if not given_periods else []:
        need = G.gefen_infer_workspace_size(s.numel)
        if iws is None or iws.numel() < need:
            iws = G.workspace(need, dev)
        p, _ = G.gefen_infer_blocks(gpool[0][o:o + s.numel], HP["eps"], workspace_buf=iws, want_scores=False)
        periods.append(p)
    infer_s = time.perf_counter() - t0
    del iws
    entries, boff = [], 0
    for s, o, p in zip(specs, offs, periods):
        entries.append((o, s.numel, p, boff))
        boff += s.numel // p
    nblocks = boff
    table = G.tensor_table(entries)
    # a step is two calls: the tensors of the dominant kernel, then the rest,
    # so CUDA events time that kernel's launch on its own
    ent_a = [e for e in entries if dominant(e[2])]
    ent_b = [e for e in entries if not dominant(e[2])]
    table_a, table_b = G.tensor_table(ent_a), G.tensor_table(ent_b)
    n_a = sum(e[1] for e in ent_a)
    blocks_a = sum(e[1] // e[2] for e in ent_a)
    codes = torch.empty(total, dtype=torch.uint8, device=dev)
    v = torch.zeros(nblocks, dtype=torch.float32, device=dev)
    sc = torch.zeros(nblocks, dtype=torch.float32, device=dev)
    hist = torch.zeros(BINS, dtype=torch.int64, device=dev)
    cb = torch.empty(K, dtype=torch.float32, device=dev)
    cb_new = torch.empty(K, dtype=torch.float32, device=dev)

    # Algorithm 3 on the first gradient: histogram of g / block absmax, DP
    ws = G.workspace(G.gefen_step_workspace_size(table, G.GEFEN_HIST), dev)
    ws_b = G.workspace(G.gefen_step_workspace_size(table_b, G.GEFEN_HIST), dev)
    rws = G.workspace(G.gefen_refit_workspace_size(BINS, K), dev)
    t0 = time.perf_counter()
    G.gefen_step(table, theta, gpool[0], codes, v, sc, cb, cb, step=1, flags=G.GEFEN_HIST_GRAD_ONLY,
                 hist=hist, workspace_buf=ws, **HP)
    G.gefen_refit_codebook(bins=BINS, k=K, codebook_out=cb, hist_in=hist, workspace_buf=rws)
    G.gefen_refit_status(rws)
    init_codebook_s = time.perf_counter() - t0
    zc = int(torch.argmin(cb.abs()).item())
    codes.fill_(zc)

    step_events = []   # (start, end) of plain steps
    dom_events = []    # (start, end) of the dominant kernel's call in plain steps
    refit_events = []  # (step start, step end, dp end)
    state = {"t": 0, "switch": False}

    def one_step(timed: bool):
        state["t"] += 1
        t = state["t"]
        g = gpool[t % 2]
        refit = (t % REFIT_EVERY == 0)
        enc = cb_new if state["switch"] else cb
        e0 = torch.cuda.Event(enable_timing=True) if timed else None
        e1 = torch.cuda.Event(enable_timing=True) if timed else None
        e2 = torch.cuda.Event(enable_timing=True) if timed and refit else None
        ea = torch.cuda.Event(enable_timing=True) if timed and not refit else None
        if timed:
            e0.record(stream)
        flags = G.GEFEN_HIST if refit else 0
        if refit:
            hist.zero_()
        G.gefen_step(table_a, theta, g, codes, v, sc, cb, enc, step=t, flags=flags, hist=hist if refit else None,
                     workspace_buf=ws, **HP)
        if ea is not None:
            ea.record(stream)
            dom_events.append((e0, ea))
        G.gefen_step(table_b, theta, g, codes, v, sc, cb, enc, step=t, flags=flags, hist=hist if refit else None,
                     workspace_buf=ws_b, **HP)
        if timed:
            e1.record(stream)
        if state["switch"]:
            cb.copy_(cb_new)
            state["switch"] = False
        if refit:
            G.gefen_refit_codebook(bins=BINS, k=K, codebook_out=cb_new, hist_in=hist, workspace_buf=rws)
            state["switch"] = True
            if timed:
                e2.record(stream)
                refit_events.append((e0, e1, e2))
        elif timed:
            step_events.append((e0, e1))

    warm = max(3, args.warmup)
    for _ in range(warm):
        one_step(False)
    torch.cuda.synchronize()

    group = None
    if world > 1:
        import torch.distributed as dist
        group = dist.group.WORLD
        dist.barrier()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    clocks.start()
    time.sleep(0.15)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        one_step(True)
    ev1.record(stream)
    torch.cuda.synchronize()
    time.sleep(0.05)
    ck = clocks.stop()
    G.gefen_step_status(ws)  # raises if a bounded device wait gave up
    G.gefen_step_status(ws_b)
    elapsed_ms = job_time_ms(ev0.elapsed_time(ev1), world, dev)

    plain_ms = [a.elapsed_time(b) for a, b in step_events]
    refit_step_ms = [a.elapsed_time(b) for a, b, _ in refit_events]
    dp_ms = [b.elapsed_time(c) for _, b, c in refit_events]
    avg_step_ms = statistics.mean(plain_ms) if plain_ms else float("nan")

    alg_bytes = 12 * nparams + 16 * nblocks + 8 * K
    hbm, peak_kind = peaks()
    # the dominant kernel alone: 12 bytes per parameter and 16 per block
    dom_ms = statistics.mean([a.elapsed_time(b) for a, b in dom_events]) if dom_events else float("nan")
    alg_bytes_a = 12 * n_a + 16 * blocks_a
    achieved = alg_bytes_a / (dom_ms * 1e-3) / 1e9
    traffic = profiled_traffic(n_a)

    # e2e: gradient in from pinned host memory, parameters back, every step
    e2e = None
    if rank == 0 or world > 1:
        e2e = run_e2e(G, table, theta, codes, v, sc, cb, ws, gpool, nparams, stream, args, state, one_step_ctx=(
            hist, cb_new, rws))

    per_a = [e[2] for e in ent_a]
    per_b = [e[2] for e in ent_b]
    n_launch_plain = launches_per_call(per_a, False) + launches_per_call(per_b, False)
    # refit steps: one histogram per call, then the DP: prefix, levels 1..K-1 and the last, backtrack
    n_launch_refit = launches_per_call(per_a, True) + launches_per_call(per_b, True) + 1 + (K - 1) + 1
    nref = len(refit_events)
    launches = (args.steps - nref) * n_launch_plain + nref * n_launch_refit

    res = {
        "metric": METRIC, "value": whole_job_value(nparams, world, args.steps, elapsed_ms), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": warm, "ms_per_step": elapsed_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded; shapes and gradient-scale structure of the Llama-3-1.5B run)",
        "config": {"workload": f"{args.workload} shaped set: {len(specs)} tensors, {nparams} fp32 params, "
                               f"{nblocks} inferred blocks; 256-level codebook; refit every {REFIT_EVERY} "
                               f"steps with {BINS} cells",
                   "params": nparams, "tensors": len(specs), "blocks": nblocks, "refit_every": REFIT_EVERY,
                   "bins": BINS, "levels": K, "hparams": HP,
                   "l2": "inputs larger than L2: 17.7 GB of step traffic per step, no flush needed",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "traffic": traffic,
                     "kernel": DOMINANT, "peak_kind": peak_kind,
                     "alg_bytes_per_launch": alg_bytes_a, "params_per_launch": n_a, "blocks_per_launch": blocks_a,
                     "avg_launch_ms": dom_ms,
                     "whole_step": {"alg_bytes": alg_bytes, "avg_ms": avg_step_ms,
                                    "achieved_gbs": alg_bytes / (avg_step_ms * 1e-3) / 1e9}},
        "step_only": {"value": nparams / (avg_step_ms * 1e-3) / 1e9 if plain_ms else None, "unit": UNIT,
                      "ms": avg_step_ms},
        "refit": {"dp_ms": statistics.mean(dp_ms) if dp_ms else None,
                  "hist_step_ms": statistics.mean(refit_step_ms) if refit_step_ms else None,
                  "count": nref},
        "init": {"infer_blocks_s": infer_s, "first_codebook_s": init_codebook_s},
        "periods": period_summary(specs, periods),
        "e2e": e2e, "gpu_launches": launches, "clocks": ck,
    }
    if rank == 0 and not args.no_microbench:
        res["refit_microbench"] = refit_microbench(G, synth, dev, args.micro_values, args.micro_bins)
    if rank == 0 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline(args)
    return res


def refit_microbench(G, synth, dev, n=MICRO_N, bins=MICRO_BINS):
    """Histogram of n normalised values (default 1.5e9) into `bins` cells
    (default 65536), then the exact DP to 256 levels; CUDA-event times of each
    part (after one untimed run)."""
    x = synth.refit_values(n, SEED + 7, device=dev)
    hist = torch.zeros(bins, dtype=torch.int64, device=dev)
    cb = torch.empty(K, dtype=torch.float32, device=dev)
    ws = G.workspace(G.gefen_refit_workspace_size(bins, K), dev)
    G.gefen_refit_codebook(bins=bins, k=K, codebook_out=cb, x=x, hist_out=hist, workspace_buf=ws)
    torch.cuda.synchronize()
    e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    e[0].record()
    G.gefen_refit_codebook(bins=bins, k=K, codebook_out=cb, x=x, hist_out=hist, workspace_buf=ws)
    e[1].record()
    G.gefen_refit_codebook(bins=bins, k=K, codebook_out=cb, hist_in=hist, workspace_buf=ws)
    e[2].record()
    torch.cuda.synchronize()
    ke = G.gefen_refit_status(ws)
    hist_dp_ms, dp_ms = e[0].elapsed_time(e[1]), e[1].elapsed_time(e[2])
    del x
    torch.cuda.empty_cache()
    return {"values": n, "bins": bins, "levels": K, "k_eff": ke,
            "nonempty_cells": int((hist > 0).sum().item()),
            "hist_ms": hist_dp_ms - dp_ms, "dp_ms": dp_ms, "total_ms": hist_dp_ms,
            "hist_gbs": 4 * n / ((hist_dp_ms - dp_ms) * 1e-3) / 1e9}


def run_e2e(G, table, theta, codes, v, sc, cb, ws, gpool, nparams, stream, args, state, one_step_ctx):
    """Same step through the public API with host buffers: every step copies
    its bf16 gradient in from pinned memory, runs gefen_step and reads the
    step's result back (its 4-byte status word, gefen_step_status, which
    waits for the step).  A second figure also copies all updated fp32
    parameters back to pinned memory every step."""
    hist, cb_new, rws = one_step_ctx
    n = gpool[0].numel()
    g_host = torch.empty(n, dtype=torch.bfloat16, pin_memory=True)
    th_host = torch.empty(theta.numel(), dtype=torch.float32, pin_memory=True)
    g_host.copy_(gpool[1])
    gdev = torch.empty_like(gpool[0])
    steps = max(3, min(args.steps, 10))

    def e2e_step(readback_params: bool):
        state["t"] += 1
        gdev.copy_(g_host, non_blocking=True)
        G.gefen_step(table, theta, gdev, codes, v, sc, cb, cb, step=state["t"], workspace_buf=ws, **HP)
        if readback_params:
            th_host.copy_(theta, non_blocking=True)
        G.gefen_step_status(ws)

    if state["switch"]:
        cb.copy_(cb_new)
        state["switch"] = False
    out = {}
    for key, rb in (("status", False), ("params", True)):
        for _ in range(2):
            e2e_step(rb)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(steps):
            e2e_step(rb)
        torch.cuda.synchronize()
        out[key] = time.perf_counter() - t0
    return {"value": nparams * steps / out["status"] / 1e9, "unit": UNIT, "steps": steps,
            "h2d_bytes_per_step": 2 * n, "d2h_bytes_per_step": 4,
            "result_read": "the step's status word (gefen_step_status), every step",
            "with_params_readback": {"value": nparams * steps / out["params"] / 1e9, "unit": UNIT,
                                     "h2d_bytes_per_step": 2 * n, "d2h_bytes_per_step": 4 * theta.numel() + 4}}


# ------------------------------------------------------------ CPU oracle arm
def oracle_sample_data(max_params: int, workload: str):
    """Whole tensors of the workload (first tensors first, the first one, the
    embedding, left out) up to about `max_params` parameters, with their
    row-length periods (a flat workload: a prefix of whole blocks): host
    arrays the oracle steps in place."""
    from paper_2606_13894_gb300 import synth

    specs, given = workload_specs(synth, workload)
    if given:
        pg = given[0]
        specs = synth.flat_set(max(pg, min(specs[0].numel, max_params) // pg * pg), pg)
    else:
        specs = specs[1:]
    rng = np.random.default_rng(SEED)
    cb = np.concatenate([[-1.0], np.sort(np.clip(rng.standard_t(4, K - 2) * 0.1, -0.99, 0.99)),
                         [1.0]]).astype(np.float32)
    out, done = [], 0
    for s in specs:
        if done >= max_params:
            break
        n = s.numel
        g = synth.draw_grads([s], SEED, step=1, device="cpu")[:n]
        bits = g.view(torch.int16).numpy().view(np.uint16).copy()
        th = synth.init_params([s], SEED, device="cpu")[:n].numpy().copy()
        p = given[0] if given else (s.cols if len(s.shape) > 1 else n)
        out.append(dict(name=s.name, theta=th, bits=bits, p=p,
                        codes=np.full(n, int(np.argmin(np.abs(cb))), np.uint8),
                        v=np.zeros(n // p, np.float32), s=np.zeros(n // p, np.float32)))
        done += n
    return out, cb, done


def oracle_steps(data, cb, t):
    import oracle
    t0 = time.perf_counter()
    for d in data:
        oracle.step(d["theta"], d["bits"], d["codes"], d["v"], d["s"], cb, cb, period=d["p"], t=t, **HP)
    return time.perf_counter() - t0


def cpu_baseline(args):
    import oracle
    data, cb, done = oracle_sample_data(args.cpu_params, args.workload)
    secs, t = 0.0, 0
    while secs < args.cpu_budget or t == 0:
        t += 1
        secs += oracle_steps(data, cb, t)
    return {"value": done * t / secs / 1e9, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{t} oracle steps (single thread, double precision) over {len(data)} whole tensors "
                      f"of the {args.workload} set ({done} params: {data[0]['name']} .. {data[-1]['name']}), "
                      f"{secs:.1f} s",
            "threads_available": os.cpu_count(), "oracle_threads": oracle.num_threads()}


def run_reference(args, world, rank):
    if rank != 0:
        return None
    warm = max(3, args.warmup)
    data, cb, done = oracle_sample_data(int(args.ref_params), args.workload)
    t = 0
    for _ in range(warm):
        t += 1
        oracle_steps(data, cb, t)
    secs = 0.0
    for _ in range(args.steps):
        t += 1
        secs += oracle_steps(data, cb, t)
    val = done * args.steps / secs / 1e9
    return {"impl": "reference", "metric": METRIC, "value": val, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": warm, "ms_per_step": secs * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": {"workload": f"{args.workload} shaped set, bounded sample: {len(data)} whole tensors "
                                   f"({done} params) per step, oracle step"},
            "cpu_baseline": {"value": val, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{done} params per step ({len(data)} tensors of the {args.workload} set)"},
            "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gefen", choices=["gefen", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--cpu-params", type=int, default=20_000_000, help="params in the cpu_baseline sample")
    ap.add_argument("--ref-params", type=float, default=20e6, help="oracle params per reference step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-microbench", action="store_true", help="skip the 65536-cell refit measurement")
    ap.add_argument("--microbench-only", action="store_true",
                    help="run only the refit micro-benchmark and print its figures (one GPU)")
    ap.add_argument("--micro-values", type=int, default=MICRO_N, help="refit micro-benchmark values (multiple of 4096)")
    ap.add_argument("--micro-bins", type=int, default=MICRO_BINS, help="refit micro-benchmark histogram cells")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="llama-1.5b (default), gpt2-125m, tiny, or flat:N:P (one tensor, blocks of P)")
    args = ap.parse_args()
    if args.microbench_only:
        from paper_2606_13894_gb300 import gefen as G
        from paper_2606_13894_gb300 import synth
        G.load()
        dev = torch.device("cuda", 0)
        print(json.dumps({"refit_microbench": refit_microbench(G, synth, dev, args.micro_values, args.micro_bins)}),
              flush=True)
        return
    world, rank, local = dist_env()
    if args.impl == "reference":
        res = run_reference(args, world, rank)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    res = run_gpu(args, world, rank, local)
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
