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

Under torchrun with N ranks the model is block-sharded over the ranks
(paper_2606_13894_gb300/shard.py): each rank steps its own blocks, and a refit
sums the ranks' histograms with one all-reduce before every rank runs the same
DP.  The model is fixed, so N ranks scale it strongly.

Prints one JSON line.  `value` is whole-job parameters updated per second over
the timed steps (refit steps included); `e2e` is the same metric through the
public call with the gradient copied in from pinned host memory and the step's
status word read back every step (and, as a second figure, all updated
parameters copied back too).  On one GPU the line also carries the same job
with 65536-cell refits, the GPT-2-125M-shaped set and a flat sweep.
`--impl reference` times the CPU oracle instead, on a bounded sample of the
same workload.
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
DOMINANT = "k_step_stream<4096, shape 512-multiple> (blocks of p <= 4096, p % 512 == 0)"


def dominant(p: int) -> bool:
    """Tensors served by the streamed 4096-element tile kernel's launch for
    blocks of whole warps' slices, the one that carries most of the step's
    bytes on this workload."""
    return p % 512 == 0 and p <= 4096


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def step_kernel_source_hash() -> str:
    h = hashlib.sha256()
    for f in ("step.cu", "step_kernels.cuh", "step_s4k.cu", "common.cuh"):
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


def whole_job_value(params_total: int, steps: int, job_ms: float) -> float:
    """Parameters of the model updated per second, in Gparams/s: the ranks
    share one model (each steps its own blocks), so this is the model's
    parameter count over the slowest rank's time per step."""
    return params_total * steps / (job_ms * 1e-3) / 1e9


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


SHAPE_SPLIT_ELEMS = 1 << 28  # the library's kShapeSplitElems


def launches_per_call(entries, flags_hist: bool) -> int:
    """Kernels one gefen_step call launches for these (period, numel) pairs
    (mirrors the library's path classes; fewer than 300 tensors per class)."""
    if not entries:
        return 0
    classes = set()
    big = 0
    streamed = {}  # streamed class -> [elements, block shapes]
    for p, n in entries:
        if p == 1:
            classes.add("p1")
        elif p % 16 == 0 and p <= 8192:
            shape = "w" if p % 512 == 0 else ("s" if p <= 256 and (p & (p - 1)) == 0 else "a")
            acc = streamed.setdefault("s4k" if p <= 4096 else "s8k", [0, set()])
            acc[0] += n
            acc[1].add(shape)
        elif p % 16 == 0 and p <= 16384:
            classes.add("t16v4")
        elif p <= 2048:
            classes.add("gen")
        else:
            big |= 1 if p % 16 == 0 else 2
    # a streamed class launches once per block shape, or once in all when it
    # has under SHAPE_SPLIT_ELEMS elements
    n_streamed = sum(1 if tot < SHAPE_SPLIT_ELEMS else len(shapes) for tot, shapes in streamed.values())
    n = len(classes) + n_streamed + 3 * bin(big).count("1")
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
def infer_periods(G, specs, grads, dev):
    """Algorithm 2 on the first gradient of every tensor (arena `grads`)."""
    from paper_2606_13894_gb300 import synth
    offs, _ = synth.pack_offsets(specs)
    periods, iws = [], None
    for s, o in zip(specs, offs):
        need = G.gefen_infer_workspace_size(s.numel)
        if iws is None or iws.numel() < need:
            iws = G.workspace(need, dev)
        p, _ = G.gefen_infer_blocks(grads[o:o + s.numel], HP["eps"], workspace_buf=iws, want_scores=False)
        periods.append(p)
    return periods


def make_shard(G, synth, dev, specs, periods, rank, world, group, bins, refit_every, split):
    """This rank's shard of the workload (block-aligned; the whole model on
    one rank) with its parameters and a pool of two gradients (steps 1, 2)."""
    from paper_2606_13894_gb300 import shard
    sh = shard.RankShard([(s.numel, p) for s, p in zip(specs, periods)], rank, world, dev, levels=K, bins=bins,
                         refit_every=refit_every, group=group, split=split)
    offs, _ = synth.pack_offsets(specs)
    if world == 1:  # the rank's arena is the model's arena
        synth.init_params(specs, SEED, device=dev, out=sh.theta)
        gpool = [synth.draw_grads(specs, SEED, step=s, device=dev) for s in (1, 2)]
    else:
        th = synth.init_params(specs, SEED, device=dev)
        sh.gather(lambda i: th[offs[i]:offs[i] + specs[i].numel], torch.float32, out=sh.theta)
        del th
        gpool = []
        for s in (1, 2):
            g = synth.draw_grads(specs, SEED, step=s, device=dev)
            gpool.append(sh.gather(lambda i: g[offs[i]:offs[i] + specs[i].numel], torch.bfloat16))
            del g
    torch.cuda.synchronize()
    return sh, gpool


class Cadence:
    """The workload's steps on one rank's shard (refit every REFIT_EVERY
    steps), with CUDA events on the launching stream: plain steps, the first
    call of a plain step (the dominant kernel's tensors, when the step is
    split), refit steps (step, then DP)."""

    def __init__(self, sh, gpool, stream, hp, dominant_first: bool):
        self.sh, self.gpool, self.stream, self.hp = sh, gpool, stream, hp
        self.dominant_first = dominant_first
        self.plain, self.dom, self.refit = [], [], []

    def _ev(self):
        e = torch.cuda.Event(enable_timing=True)
        e.record(self.stream)
        return e

    def step(self, timed: bool, g=None) -> bool:
        sh = self.sh
        if g is None:
            g = self.gpool[(sh.t + 1) % 2]
        e0 = self._ev() if timed else None
        ea = []

        def after(i):
            if timed and i == 0 and self.dominant_first:
                ea.append(self._ev())

        refit = sh.step_local(g, self.hp, after_call=after)
        e1 = self._ev() if timed else None
        if refit:
            sh.refit_codebook()
            if timed:
                self.refit.append((e0, e1, self._ev()))
        elif timed:
            self.plain.append((e0, e1))
            if ea:
                self.dom.append((e0, ea[0]))
        return refit

    def reset_events(self):
        self.plain, self.dom, self.refit = [], [], []

    def mean_ms(self, which: str, part: int = 0):
        ev = getattr(self, which)
        if not ev:
            return None
        if which == "refit":
            return statistics.mean(e[part].elapsed_time(e[part + 1]) for e in ev)
        return statistics.mean(a.elapsed_time(b) for a, b in ev)


def timed_steps(cad: Cadence, steps: int, warm: int, stream, world: int, dev, clocks=None):
    """warm untimed steps, then `steps` timed ones bracketed by a barrier and
    synchronisation; returns the job time (slowest rank) in ms."""
    for _ in range(warm):
        cad.step(False)
    torch.cuda.synchronize()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    cad.reset_events()
    if clocks is not None:
        clocks.start()
        time.sleep(0.15)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(steps):
        cad.step(True)
    ev1.record(stream)
    torch.cuda.synchronize()
    ck = None
    if clocks is not None:
        time.sleep(0.05)
        ck = clocks.stop()
    return job_time_ms(ev0.elapsed_time(ev1), world, dev), ck


def run_gpu(args, world, rank, local):
    from paper_2606_13894_gb300 import gefen as G
    from paper_2606_13894_gb300 import synth

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    G.load()
    group = None
    if world > 1:
        import torch.distributed as dist
        group = dist.group.WORLD
    specs, given_periods = workload_specs(synth, args.workload)
    nparams = synth.total_params(specs)
    stream = torch.cuda.current_stream()

    # Algorithm 2 on the first gradient of every tensor: every rank infers
    # the same blocks from the same gradient
    t0 = time.perf_counter()
    if given_periods:
        periods = given_periods * len(specs)
    else:
        g1 = synth.draw_grads(specs, SEED, step=1, device=dev)
        periods = infer_periods(G, specs, g1, dev)
        del g1
    infer_s = time.perf_counter() - t0
    # a step is two calls on each rank: the tensors of the dominant kernel,
    # then the rest, so CUDA events time that kernel's launch on its own
    sh, gpool = make_shard(G, synth, dev, specs, periods, rank, world, group, BINS, REFIT_EVERY, dominant)
    dom_first = bool(sh.call_entries) and all(dominant(e[2]) for e in sh.call_entries[0])
    n_rank, blocks_rank = sh.numel, sum(pc.nblocks for pc in sh.pieces)
    n_a = sum(e[1] for e in sh.call_entries[0]) if dom_first else 0
    blocks_a = sum(e[1] // e[2] for e in sh.call_entries[0]) if dom_first else 0
    nblocks = sum(s.numel // p for s, p in zip(specs, periods))

    # Algorithm 3 on the first gradient: histogram of g / block absmax (summed
    # over the ranks), then the exact DP
    t0 = time.perf_counter()
    sh.init_codebook(gpool[0], HP)
    G.gefen_refit_status(sh.rws)
    init_codebook_s = time.perf_counter() - t0

    cad = Cadence(sh, gpool, stream, HP, dom_first)
    warm = max(3, args.warmup)
    elapsed_ms, ck = timed_steps(cad, args.steps, warm, stream, world, dev, clocks=Clocks(local))
    G.gefen_step_status(sh.ws)  # raises if a bounded device wait gave up
    G.gefen_refit_status(sh.rws)

    avg_step_ms = cad.mean_ms("plain")
    dom_ms = cad.mean_ms("dom")
    hbm, peak_kind = peaks()
    alg_bytes = 12 * n_rank + 16 * blocks_rank + 8 * K
    alg_bytes_a = 12 * n_a + 16 * blocks_a
    achieved = alg_bytes_a / (dom_ms * 1e-3) / 1e9 if dom_ms else None
    traffic = profiled_traffic(n_a) if dom_first else None

    e2e = run_e2e(G, cad, args, stream)

    per = [[(e[2], e[1]) for e in ce] for ce in sh.call_entries]
    n_launch_plain = sum(launches_per_call(x, False) for x in per)
    # refit steps: the step's calls with their histograms, then the DP's four
    # launches (prefix, first level, the cooperative levels launch, backtrack)
    n_launch_refit = sum(launches_per_call(x, True) for x in per) + 4
    nref = len(cad.refit)
    launches = (args.steps - nref) * n_launch_plain + nref * n_launch_refit

    whole_step_ms = avg_step_ms
    res = {
        "metric": METRIC, "value": whole_job_value(nparams, args.steps, elapsed_ms), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": warm, "ms_per_step": elapsed_ms / args.steps,
        "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "f32",
        "data": f"synthetic (seeded; shapes and gradient-scale structure of the {args.workload} set)",
        "config": {"workload": f"{args.workload} shaped set: {len(specs)} tensors, {nparams} fp32 params, "
                               f"{nblocks} inferred blocks; 256-level codebook; refit every {REFIT_EVERY} "
                               f"steps with {BINS} cells (16 per level: Algorithm 3's 16k cells read as 16 k); "
                               f"the same job with 65536-cell refits is under refit_65536",
                   "params": nparams, "tensors": len(specs), "blocks": nblocks, "refit_every": REFIT_EVERY,
                   "bins": BINS, "levels": K, "hparams": HP,
                   "l2": (f"inputs larger than L2: {alg_bytes / 1e9:.2f} GB of step traffic per step against a "
                          f"129 MB L2, no flush needed" if alg_bytes > 4 * 129e6 else
                          f"{alg_bytes / 1e9:.3f} GB of step traffic per step against a 129 MB L2: timings "
                          f"of this workload include L2 reuse between steps"),
                   "parallelism": ("single GPU" if world == 1 else
                                   f"block-sharded over {world} ranks ({n_rank} params on rank {rank}); "
                                   f"one histogram all-reduce per refit")},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm if achieved else None, "traffic": traffic,
                     "kernel": DOMINANT, "peak_kind": peak_kind,
                     "alg_bytes_per_launch": alg_bytes_a, "params_per_launch": n_a, "blocks_per_launch": blocks_a,
                     "avg_launch_ms": dom_ms,
                     "whole_step": {"alg_bytes": alg_bytes, "avg_ms": whole_step_ms,
                                    "achieved_gbs": alg_bytes / (whole_step_ms * 1e-3) / 1e9,
                                    "frac": alg_bytes / (whole_step_ms * 1e-3) / 1e9 / hbm}},
        "step_only": {"value": nparams / (avg_step_ms * 1e-3) / 1e9 if avg_step_ms else None,
                      "unit": UNIT, "ms": avg_step_ms},
        "refit": {"dp_ms": cad.mean_ms("refit", 1), "hist_step_ms": cad.mean_ms("refit", 0), "count": nref},
        "init": {"infer_blocks_s": infer_s, "first_codebook_s": init_codebook_s},
        "periods": period_summary(specs, periods),
        "e2e": e2e, "gpu_launches": launches, "clocks": ck,
    }
    if world == 1 and not args.no_extras:
        res["refit_65536"] = cadence_65536(G, cad, args, stream, dev, nparams)
    del cad, sh, gpool
    torch.cuda.empty_cache()
    if rank == 0 and not args.no_microbench:
        res["refit_microbench"] = refit_microbench(G, synth, dev, args.micro_values, args.micro_bins)
    if world == 1 and not args.no_extras:
        res["gpt2_125m"] = gpt2_figures(G, synth, dev, args, stream, hbm)
        res["flat_sweep"] = flat_sweep(G, synth, dev, stream, hbm)
        res["gefen_muon"] = muon_figures(G, dev)
    if rank == 0 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline(args)
    return res


def cadence_65536(G, cad, args, stream, dev, nparams):
    """The same job with refits from 65536-cell histograms (the other reading
    of Algorithm 3's histogram size for this set: 65536 cells rather than 16
    per level): the x of every tensor is staged and counted by the 65536-cell
    histogram kernel, then the 65536 x 256 DP."""
    sh = cad.sh
    sh.set_refit_bins(65536)
    cad.reset_events()
    ms, _ = timed_steps(cad, args.steps, 3, stream, 1, dev)
    G.gefen_refit_status(sh.rws)
    out = {"value": whole_job_value(nparams, args.steps, ms), "unit": UNIT, "ms_per_step": ms / args.steps,
           "steps": args.steps, "refit_every": REFIT_EVERY, "bins": 65536,
           "dp_ms": cad.mean_ms("refit", 1), "hist_step_ms": cad.mean_ms("refit", 0), "count": len(cad.refit)}
    sh.set_refit_bins(BINS)
    return out


GPT2_HP = dict(lr=6e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1)  # Appendix I, GPT-2


def gpt2_figures(G, synth, dev, args, stream, hbm):
    """The GPT-2-125M-shaped set (blocks inferred from its first gradient):
    the whole job with the same refit cadence, and a plain step's throughput
    and algorithmic bytes per second."""
    specs = synth.gpt2_125m_set()
    n = synth.total_params(specs)
    g1 = synth.draw_grads(specs, SEED, step=1, device=dev)
    periods = infer_periods(G, specs, g1, dev)
    del g1
    sh, gpool = make_shard(G, synth, dev, specs, periods, 0, 1, None, BINS, REFIT_EVERY, None)
    sh.init_codebook(gpool[0], GPT2_HP)
    cad = Cadence(sh, gpool, stream, GPT2_HP, False)
    steps = max(args.steps, 20)
    ms, _ = timed_steps(cad, steps, 3, stream, 1, dev)
    G.gefen_step_status(sh.ws)
    step_ms = cad.mean_ms("plain")
    nb = sum(s.numel // p for s, p in zip(specs, periods))
    alg = 12 * n + 16 * nb + 8 * K
    out = {"params": n, "blocks": nb, "hparams": GPT2_HP,
           "whole_job": {"value": whole_job_value(n, steps, ms), "unit": UNIT, "ms_per_step": ms / steps,
                         "steps": steps, "refit_every": REFIT_EVERY, "bins": BINS},
           "step": {"value": n / (step_ms * 1e-3) / 1e9, "unit": UNIT, "ms": step_ms,
                    "alg_bytes": alg, "achieved_gbs": alg / (step_ms * 1e-3) / 1e9,
                    "frac": alg / (step_ms * 1e-3) / 1e9 / hbm},
           "periods": period_summary(specs, periods),
           "l2": "1.5 GB of step traffic per step against a 129 MB L2: no flush needed"}
    del cad, sh, gpool
    torch.cuda.empty_cache()
    return out


def flat_sweep(G, synth, dev, stream, hbm, sizes=(1 << 28, 1 << 31)):
    """One flat tensor of N fp32 parameters with given blocks of p: a plain
    step's time and algorithmic GB/s (12 B per parameter and 16 per block)."""
    out = {}
    for n in sizes:
        for p in (1, 64, 4096, 1 << 20, n):
            specs = synth.flat_set(n, p)
            sh, gpool = make_shard(G, synth, dev, specs, [p], 0, 1, None, BINS, 0, None)
            sh.init_codebook(gpool[0], HP)
            cad = Cadence(sh, gpool, stream, HP, False)
            timed_steps(cad, 5, 3, stream, 1, dev)
            G.gefen_step_status(sh.ws)
            ms = cad.mean_ms("plain")
            alg = 12 * n + 16 * (n // p)
            out[f"2^{n.bit_length() - 1}/{'n' if p == n else p}"] = {
                "ms": ms, "gparams": n / (ms * 1e-3) / 1e9, "achieved_gbs": alg / (ms * 1e-3) / 1e9,
                "frac": alg / (ms * 1e-3) / 1e9 / hbm}
            del cad, sh, gpool
            torch.cuda.empty_cache()
    return out


def refit_microbench(G, synth, dev, n=MICRO_N, bins=MICRO_BINS):
    """Histogram of n normalised values (default 1.5e9) into `bins` cells
    (default 65536), then the exact DP to 256 levels; CUDA-event times of each
    part (after one untimed run): the median of three runs of the whole refit
    from the values and of three from the histogram (the DP alone)."""
    x = synth.refit_values(n, SEED + 7, device=dev)
    hist = torch.zeros(bins, dtype=torch.int64, device=dev)
    cb = torch.empty(K, dtype=torch.float32, device=dev)
    ws = G.workspace(G.gefen_refit_workspace_size(bins, K), dev)
    G.gefen_refit_codebook(bins=bins, k=K, codebook_out=cb, x=x, hist_out=hist, workspace_buf=ws)
    torch.cuda.synchronize()
    whole, dp = [], []
    for _ in range(3):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        e[0].record()
        G.gefen_refit_codebook(bins=bins, k=K, codebook_out=cb, x=x, hist_out=hist, workspace_buf=ws)
        e[1].record()
        G.gefen_refit_codebook(bins=bins, k=K, codebook_out=cb, hist_in=hist, workspace_buf=ws)
        e[2].record()
        torch.cuda.synchronize()
        whole.append(e[0].elapsed_time(e[1]))
        dp.append(e[1].elapsed_time(e[2]))
    ke = G.gefen_refit_status(ws)
    hist_dp_ms, dp_ms = sorted(whole)[1], sorted(dp)[1]
    del x
    torch.cuda.empty_cache()
    return {"values": n, "bins": bins, "levels": K, "k_eff": ke,
            "nonempty_cells": int((hist > 0).sum().item()),
            "hist_ms": hist_dp_ms - dp_ms, "dp_ms": dp_ms, "total_ms": hist_dp_ms,
            "hist_gbs": 4 * n / ((hist_dp_ms - dp_ms) * 1e-3) / 1e9}


def muon_figures(G, dev, shapes=((2048, 8192), (8192, 2048), (2048, 2048)), warm=3, reps=5, steps_ns=5):
    """Gefen-Muon (bf16 products on the tensor cores): CUDA-event time of one
    gefen_muon_step per shape (period = cols, 5 Newton-Schulz steps) and the
    Newton-Schulz flops over that whole step time, against the measured bf16
    peak."""
    out = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        peak, kind = float(pk["bf16_tflops"]), "measured"
    except Exception:
        peak, kind = 1900.0, "fallback"
    for rows, cols in shapes:
        n = rows * cols
        g = torch.Generator(device=dev).manual_seed(rows + cols)
        th = torch.randn(n, device=dev, generator=g) * 0.02
        gr = (torch.randn(n, device=dev, generator=g) * 1e-3).to(torch.bfloat16)
        codes = torch.full((n,), 128, dtype=torch.uint8, device=dev)
        sc = torch.zeros(n // cols, device=dev)
        cb = torch.linspace(-1, 1, K, device=dev)
        ws = None
        for _ in range(warm):
            ws = G.gefen_muon_step(rows, cols, cols, th, gr, codes, sc, cb, cb, lr=1e-3, ns_steps=steps_ns,
                                   flags=G.GEFEN_MUON_BF16_GEMM, workspace_buf=ws)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            ws = G.gefen_muon_step(rows, cols, cols, th, gr, codes, sc, cb, cb, lr=1e-3, ns_steps=steps_ns,
                                   flags=G.GEFEN_MUON_BF16_GEMM, workspace_buf=ws)
        e1.record()
        torch.cuda.synchronize()
        G.gefen_step_status(ws)
        ms = e0.elapsed_time(e1) / reps
        sm, lg = min(rows, cols), max(rows, cols)
        flops = steps_ns * (2 * 2 * sm * sm * lg + 2 * sm ** 3)  # X X^T, A A, B X per step
        tf = flops / (ms * 1e-3) / 1e12
        out[f"{rows}x{cols}"] = {"ms": ms, "ns_tflops": tf, "frac": tf / peak}
        del th, gr, codes, sc, ws
        torch.cuda.empty_cache()
    return {"shapes": out, "peak_tflops": peak, "peak_kind": kind,
            "note": "Newton-Schulz flops (2 s^2 n + 2 s^3 + 2 s^2 n per step) over the whole step time "
                    "(element-wise kernels included), bf16 products with fp32 accumulation"}


def run_e2e(G, cad, args, stream):
    """The same job through the public API with host buffers: every step
    copies its bf16 gradient in from pinned memory and runs the step (refit
    steps included, with the timed region's cadence and step count), and the
    step's result is read back: its 4-byte status word (gefen_step_status,
    which waits for the step).  The copies run on their own stream into two
    device buffers, as a data loader's would: step i + 1's gradient is copied
    while step i computes, and step i + 2's copy waits until step i has read
    its buffer.  Every copy of the timed steps, the first two included, is in
    the timed region.  A second figure also copies the rank's updated fp32
    parameters back to pinned memory every step (on the step's stream, so the
    next step waits for it)."""
    sh = cad.sh
    n = sh.numel_arena
    g_host = torch.empty(n, dtype=torch.bfloat16, pin_memory=True)
    th_host = torch.empty(n, dtype=torch.float32, pin_memory=True)
    g_host.copy_(cad.gpool[1])
    gdev = [torch.empty_like(cad.gpool[0]) for _ in range(2)]
    cstream = torch.cuda.Stream(device=gdev[0].device)
    steps = args.steps

    def run(count: int, readback_params: bool):
        copied = [torch.cuda.Event() for _ in range(2)]
        freed = [torch.cuda.Event() for _ in range(2)]

        def copy_in(i):
            b = i % 2
            if i >= 2:
                cstream.wait_event(freed[b])  # step i - 2 has read buffer b
            with torch.cuda.stream(cstream):
                gdev[b].copy_(g_host, non_blocking=True)
            copied[b].record(cstream)

        for i in range(min(2, count)):
            copy_in(i)
        for i in range(count):
            b = i % 2
            stream.wait_event(copied[b])
            cad.step(False, g=gdev[b])
            freed[b].record(stream)
            if i + 2 < count:
                copy_in(i + 2)
            if readback_params:
                th_host.copy_(sh.theta, non_blocking=True)
            G.gefen_step_status(sh.ws)

    out = {}
    for key, rb in (("status", False), ("params", True)):
        run(2, rb)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        run(steps, rb)
        torch.cuda.synchronize()
        out[key] = time.perf_counter() - t0
    nparams = sum(pc.numel for pc in sh.pieces)
    return {"value": nparams * steps / out["status"] / 1e9, "unit": UNIT, "steps": steps,
            "refit_every": sh.refit_every,
            "h2d_bytes_per_step": 2 * n, "d2h_bytes_per_step": 4,
            "result_read": "the step's status word (gefen_step_status), every step",
            "copies": "gradient copies on their own stream, one step ahead of the step that reads them",
            "with_params_readback": {"value": nparams * steps / out["params"] / 1e9, "unit": UNIT,
                                     "h2d_bytes_per_step": 2 * n, "d2h_bytes_per_step": 4 * n + 4}}


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


def host_cpu():
    """Host CPU model name (lscpu) and logical core count."""
    name = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                name = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    return {"model": name, "nproc": os.cpu_count()}


def cpu_baseline(args):
    """The oracle's step on the host: single-threaded and with its loop over
    blocks on every core (the figure reported as `value`)."""
    import oracle
    data, cb, done = oracle_sample_data(args.cpu_params, args.workload)
    runs = {}
    ncores = os.cpu_count() or 1
    t = 0
    for threads in (1, ncores):
        oracle.set_num_threads(threads)
        secs, steps = 0.0, 0
        while secs < args.cpu_budget / 2 or steps == 0:
            t += 1
            steps += 1
            secs += oracle_steps(data, cb, t)
        runs[threads] = (done * steps / secs / 1e9, steps, secs)
    oracle.set_num_threads(ncores)
    val, steps, secs = runs[ncores]
    return {"value": val, "unit": UNIT, "cores": ncores, "kind": "oracle",
            "sample": f"{steps} oracle steps (double precision, its loop over blocks on {ncores} threads) over "
                      f"{len(data)} whole tensors of the {args.workload} set ({done} params: {data[0]['name']} .. "
                      f"{data[-1]['name']}), {secs:.1f} s",
            "single_thread": {"value": runs[1][0], "unit": UNIT, "cores": 1, "steps": runs[1][1],
                              "seconds": runs[1][2]},
            "host": host_cpu()}


def run_reference(args, world, rank):
    if rank != 0:
        return None
    import oracle
    ncores = os.cpu_count() or 1
    oracle.set_num_threads(ncores)
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
            "cpu_baseline": {"value": val, "unit": UNIT, "cores": ncores, "kind": "oracle",
                             "sample": f"{done} params per step ({len(data)} tensors of the {args.workload} set), "
                                       f"the oracle's loop over blocks on {ncores} threads",
                             "host": host_cpu()},
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
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the 65536-cell cadence, GPT-2-125M and flat-sweep figures")
    ap.add_argument("--microbench-only", action="store_true",
                    help="run only the refit micro-benchmark and print its figures (one GPU)")
    ap.add_argument("--micro-values", type=int, default=MICRO_N, help="refit micro-benchmark values (multiple of 4096)")
    ap.add_argument("--muon-only", default=None, metavar="ROWSxCOLS",
                    help="time only gefen_muon_step (bf16 products) on one matrix shape and print its figures")
    ap.add_argument("--micro-bins", type=int, default=MICRO_BINS, help="refit micro-benchmark histogram cells")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="llama-1.5b (default), gpt2-125m, tiny, or flat:N:P (one tensor, blocks of P)")
    args = ap.parse_args()
    if args.muon_only:
        from paper_2606_13894_gb300 import gefen as G
        G.load()
        r, c = (int(v) for v in args.muon_only.lower().split("x"))
        print(json.dumps({"gefen_muon": muon_figures(G, torch.device("cuda", 0), shapes=((r, c),))}), flush=True)
        return
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
