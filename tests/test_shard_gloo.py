"""The sharded step's one exchange, on CPU ranks (gloo, world size 2): each
rank steps only the blocks shard.partition gives it, the ranks' histograms are
summed by shard.all_reduce_histogram (the product's collective), and every
rank runs the exact DP on the sum.  The all-reduced histograms and the
codebooks equal the single-rank run's bit for bit, and every rank's block
state (parameters, codes, v, scale) equals the same blocks of the single-rank
run.  The CUDA step cannot run here, so the oracle computes each rank's step:
it is the checker of the partition and the exchange, not their product."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2606_13894_gb300 import shard

TENSORS = [(64 * 48, 64), (3 * 501, 3), (1000, 1), (256 * 40, 256), (4096, 4096), (50 * 30, 30)]
K, BINS = 16, 512
HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


def _data(seed=0):
    rng = np.random.default_rng(seed)
    theta = [rng.normal(0, 0.02, n).astype(np.float32) for n, _ in TENSORS]
    grads = []
    for _ in range(4):
        gs = []
        for n, p in TENSORS:
            sig = np.repeat(10 ** rng.uniform(-4, -2, n // p), p)
            g = torch.from_numpy((rng.normal(0, 1, n) * sig).astype(np.float32)).to(torch.bfloat16)
            gs.append(g.view(torch.int16).numpy().view(np.uint16).copy())
        grads.append(gs)
    return theta, grads


def _run(pieces, reduce):
    """The workload cadence over `pieces` with the oracle as the step: first
    codebook from the first gradient, a plain step, a refit step, then a step
    that decodes with the old codebook and encodes with the new one."""
    theta, grads = _data()
    st = []
    for pc in pieces:
        a, e = pc.first_element, pc.first_element + pc.numel
        st.append(dict(pc=pc, theta=theta[pc.tensor][a:e].copy(), codes=np.zeros(pc.numel, np.uint8),
                       v=np.zeros(pc.nblocks, np.float32), s=np.zeros(pc.nblocks, np.float32)))

    def g_of(d, t):
        pc = d["pc"]
        return grads[t][pc.tensor][pc.first_element:pc.first_element + pc.numel].copy()

    def do_step(gi, t, dec, enc, mode):
        hist = np.zeros(BINS, np.uint64)
        for d in st:
            oracle.step(d["theta"], g_of(d, gi), d["codes"], d["v"], d["s"], dec, enc, period=d["pc"].period, t=t,
                        hist=hist, hist_mode=mode, **HP)
        return hist

    hists, cbs = [], []
    zeros = np.zeros(K, np.float32)
    h = reduce(do_step(0, 1, zeros, zeros, 2))  # the first gradient's g / block absmax
    cb = oracle.dp(h, K)["codebook"]
    hists.append(h)
    cbs.append(cb)
    z = int(np.argmin(np.abs(cb.astype(np.float64))))
    for d in st:
        d["codes"][:] = z
    do_step(1, 1, cb, cb, 0)
    h = reduce(do_step(2, 2, cb, cb, 1))  # refit step: x = m / s'
    cb_new = oracle.dp(h, K)["codebook"]
    hists.append(h)
    cbs.append(cb_new)
    do_step(3, 3, cb, cb_new, 0)
    return hists, cbs, [(d["pc"], d["theta"], d["codes"], d["v"], d["s"]) for d in st]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        def reduce(h):
            t = torch.from_numpy(h.astype(np.int64))
            return shard.all_reduce_histogram(t).numpy().astype(np.uint64)
        q.put((rank, _run(shard.partition(TENSORS, world)[rank], reduce)))
    except Exception as e:  # report instead of leaving the parent waiting
        q.put((rank, repr(e)))
        raise
    finally:
        dist.destroy_process_group()


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_sharded_refit_and_block_state_equal_the_single_rank_run():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in ps:
        p.start()
    got = dict(q.get(timeout=300) for _ in range(world))
    for r in range(world):
        assert not isinstance(got[r], str), got[r]
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    ref_h, ref_cb, ref_st = _run(shard.partition(TENSORS, 1)[0], lambda h: h)
    # the ranks split the model: both own blocks
    assert all(len(got[r][2]) > 0 for r in range(world))
    for r in range(world):
        hists, cbs, st = got[r]
        for a, b in zip(hists, ref_h):
            np.testing.assert_array_equal(a, b)
        for a, b in zip(cbs, ref_cb):
            np.testing.assert_array_equal(a, b)
        for pc, th, cd, v, s in st:
            whole = next(x for x in ref_st if x[0].tensor == pc.tensor)
            a, e = pc.first_element, pc.first_element + pc.numel
            np.testing.assert_array_equal(th, whole[1][a:e])
            np.testing.assert_array_equal(cd, whole[2][a:e])
            np.testing.assert_array_equal(v, whole[3][pc.first_block:pc.first_block + pc.nblocks])
            np.testing.assert_array_equal(s, whole[4][pc.first_block:pc.first_block + pc.nblocks])
    # the histograms the ranks summed are each only part of the whole
    assert int(ref_h[1].sum()) > 0
