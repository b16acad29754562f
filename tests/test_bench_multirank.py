"""The bench's multi-rank path on CPU: the job time is the slowest rank's, the
value is the model's parameters per second over that time (the ranks share
one block-sharded model), and under torchrun only rank 0 prints the reference
arm's line."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = [120.0, 80.0][rank]
        job = bench.job_time_ms(local_ms, world, torch.device("cpu"))
        q.put((rank, job, bench.whole_job_value(1000, 10, job)))
    finally:
        dist.destroy_process_group()


def test_job_time_is_the_slowest_rank_and_value_counts_all_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    for _, job, value in got:
        assert job == 120.0
        # a 1000-parameter model, 10 steps in 0.12 s
        assert value == pytest.approx(1000 * 10 / 0.12 / 1e9)


def test_single_rank_needs_no_process_group():
    assert bench.job_time_ms(42.0, 1, torch.device("cpu")) == 42.0


def test_reference_arm_under_torchrun_prints_one_line_from_rank_0():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3", "--ref-params", "2e5",
           "--workload", "flat:262144:2048"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_launch_count_follows_the_librarys_launch_plan():
    # The bench's gpu_launches claim mirrors gefen_step's plan: one launch
    # per class of blocks; the streamed classes (p % 16 == 0, p <= 8192) once
    # per block shape (multiples of 512; powers of two 16..256; any other),
    # or once in all for a class of under 2^28 elements; three launches for
    # big blocks (partial, finalise, apply); one more for a histogram step.
    big = 1 << 28
    # the Llama-shaped dominant call: blocks of 2048 and 512 share a shape
    assert bench.launches_per_call([(2048, 934_805_504), (512, 8192)], False) == 1
    # its second call: p = 1, 8192 tiles, blocks of 64 to 256, big blocks
    second = [(1, 63_488), (8192, 335_544_320), (64, 75_499_520), (128, 8_392_704), (256, 6144),
              (131072, 118_489_088), (262144, 6_291_456)]
    assert bench.launches_per_call(second, False) == 1 + 1 + 1 + 3
    assert bench.launches_per_call(second, True) == 7
    # a large class of mixed shapes: one launch per shape
    assert bench.launches_per_call([(2048, big), (64, big), (48, big)], False) == 3
    # a small class of mixed shapes (the GPT-2-shaped set): one launch in all
    assert bench.launches_per_call([(64, 75_108_096), (128, 46_857_216), (192, 2_361_600)], False) == 1
    # other classes: 16K tiles, the generic tile, unaligned big blocks
    assert bench.launches_per_call([(12288, 24576), (24, 4608), (30001, 60002)], False) == 1 + 1 + 3
    assert bench.launches_per_call([], True) == 0
