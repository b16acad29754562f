"""Full-size parity in the launch configuration bench.py times.

The workloads are the bench's: every tensor of the Llama-3-style 1.5B set and
of the GPT-2-125M set with blocks inferred on the GPU from the first gradient
(Algorithm 2) and the first codebook learned from it (Algorithm 3), stepped as
the bench steps them (the tensors of the 4096-element tile kernel in one call,
the rest in a second); and flat tensors up to 2^31 elements.  The step is local
to a block, so a sample of whole blocks (two per tensor, both ends of every
tensor's range among them) is recomputed by the oracle from those blocks'
pre-step state and compared with the tolerances of the other step tests."""
import numpy as np
import pytest
import torch

import bench
import gpu_util as U
import oracle
from paper_2606_13894_gb300 import gefen as G
from paper_2606_13894_gb300 import synth

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

HP = bench.HP  # the workload's hyper-parameters (lr 1e-4, betas 0.9 / 0.999, eps 1e-8)


class Sample:
    """Sampled whole blocks of an arena, packed as a compact host arena the
    oracle and the comparison helpers take (entries (offset, p, p, block))."""

    def __init__(self, picks, device):
        # picks: (first element, period, global block index)
        self.picks = picks
        self.entries, off = [], 0
        for j, (e0, p, bi) in enumerate(picks):
            self.entries.append((off, p, p, j))
            off += p
        self.N, self.NB = off, len(picks)
        self.eidx = torch.cat([torch.arange(e0, e0 + p, device=device) for e0, p, _ in picks])
        self.bidx = torch.tensor([bi for _, _, bi in picks], device=device)

    def gather(self, theta, codes, v, s):
        return (theta[self.eidx].cpu().numpy().copy(), codes[self.eidx].cpu().numpy().copy(),
                v[self.bidx].cpu().numpy().copy(), s[self.bidx].cpu().numpy().copy())

    def gbits(self, g):
        return U.bits(g[self.eidx])


def pick_blocks(entries, rng, per_tensor=2):
    picks = []
    for (o, n, p, b) in entries:
        nb = n // p
        sel = {0, nb - 1} if per_tensor >= 2 else {0}
        while len(sel) < min(per_tensor, nb):
            sel.add(int(rng.integers(nb)))
        for j in sorted(sel):
            picks.append((o + j * p, p, b + j))
    return picks


def compare(sample, pre, gbits, post, cb_dec, cb_enc, t, hp):
    th, cd, v, s, _ = U.oracle_step(sample, pre, gbits, cb_dec, cb_enc, t, hp)
    te = U.theta_err(post[0], th, hp["lr"])
    ve = U.rel_err(post[2], v)
    M = U.summand_scale(sample, pre, gbits, cb_dec, hp["beta1"])
    sok, se = U.scale_ok(post[3], s, M)
    ok, flips = U.code_flips_ok(sample, pre, gbits, cb_dec, cb_enc, post[1], cd, hp, M)
    assert te <= U.THETA_TOL, f"step {t}: theta error {te}"
    assert ve <= U.STATE_TOL, f"step {t}: v error {ve}"
    assert sok, f"step {t}: s error {se}"
    assert ok, f"step {t}: {flips} code flips beyond the margin rule"
    return dict(t=t, theta=te, v=ve, s=se, flips=flips)


def run_workload(specs, periods=None, steps=3, seed=0, per_tensor=2):
    """Bench-style set-up and steps; returns the per-step comparison report."""
    dev = torch.device("cuda")
    offs, total = synth.pack_offsets(specs)
    theta = synth.init_params(specs, seed, device=dev)
    grads = [synth.draw_grads(specs, seed, step=s, device=dev) for s in (1, 2)]
    if periods is None:
        periods, iws = [], None
        for s, o in zip(specs, offs):
            need = G.gefen_infer_workspace_size(s.numel)
            if iws is None or iws.numel() < need:
                iws = G.workspace(need, dev)
            p, _ = G.gefen_infer_blocks(grads[0][o:o + s.numel], HP["eps"], workspace_buf=iws, want_scores=False)
            periods.append(p)
        del iws
    entries, boff = [], 0
    for s, o, p in zip(specs, offs, periods):
        entries.append((o, s.numel, p, boff))
        boff += s.numel // p
    table = G.tensor_table(entries)
    ent_a = [e for e in entries if bench.dominant(e[2])]
    ent_b = [e for e in entries if not bench.dominant(e[2])]
    tables = [G.tensor_table(x) for x in (ent_a, ent_b) if x]
    codes = torch.empty(total, dtype=torch.uint8, device=dev)
    v = torch.zeros(boff, dtype=torch.float32, device=dev)
    sc = torch.zeros(boff, dtype=torch.float32, device=dev)
    K, B = bench.K, bench.BINS
    hist = torch.zeros(B, dtype=torch.int64, device=dev)
    cb = torch.empty(K, dtype=torch.float32, device=dev)
    G.gefen_step(table, theta, grads[0], codes, v, sc, cb, cb, step=1, flags=G.GEFEN_HIST_GRAD_ONLY, hist=hist,
                 **HP)
    G.gefen_refit_codebook(bins=B, k=K, codebook_out=cb, hist_in=hist)
    codes.fill_(int(torch.argmin(cb.abs()).item()))
    cb_h = cb.cpu().numpy()
    # a second codebook for the last step: decode with cb, encode with cb_new
    cb_new = torch.empty(K, dtype=torch.float32, device=dev)
    hist.zero_()
    G.gefen_step(table, theta, grads[1], codes, v, sc, cb, cb, step=1, flags=G.GEFEN_HIST_GRAD_ONLY, hist=hist,
                 **HP)
    G.gefen_refit_codebook(bins=B, k=K, codebook_out=cb_new, hist_in=hist)
    cbn_h = cb_new.cpu().numpy()

    rng = np.random.default_rng(seed + 7)
    sample = Sample(pick_blocks(entries, rng, per_tensor), dev)
    report = []
    for t in range(1, steps + 1):
        g = grads[t % 2]
        enc, enc_h = (cb_new, cbn_h) if t == steps else (cb, cb_h)
        pre = sample.gather(theta, codes, v, sc)
        gb = sample.gbits(g)
        for tb in tables:
            G.gefen_step(tb, theta, g, codes, v, sc, cb, enc, step=t, **HP)
        torch.cuda.synchronize()
        post = sample.gather(theta, codes, v, sc)
        report.append(compare(sample, pre, gb, post, cb_h, enc_h, t, HP))
    return report, periods


def test_llama_1p5b_set_sampled_parity():
    report, periods = run_workload(synth.llama_1p5b_set())
    assert len(report) == 3
    # the GPU-inferred blocks the steps ran with are the oracle's, tensor by tensor
    assert periods == U.oracle_model_periods("llama-1.5b", 0)[0]


def test_gpt2_125m_set_sampled_parity():
    report, periods = run_workload(synth.gpt2_125m_set())
    assert len(report) == 3
    assert periods == U.oracle_model_periods("gpt2-125m", 0)[0]


@pytest.mark.parametrize("log2n,p", [(20, 1), (20, 64), (20, 4096), (20, 1 << 20), (24, 4096), (26, 1 << 26),
                                     (28, 1), (28, 64), (31, 4096), (31, 1 << 20)])
def test_flat_sweep_sampled_parity(log2n, p):
    n = 1 << log2n
    per = min(n // p, 256 if p <= 4096 else 2)  # blocks sampled (small blocks: many)
    report, _ = run_workload(synth.flat_set(n, p), periods=[p], steps=2, per_tensor=per)
    assert len(report) == 2


def test_refit_microbench_histogram_full_size():
    """The 1.5e9-value refit input (Student-t mixture, 65536 cells): the GPU
    histogram equals the oracle's, cell for cell, and sums to N."""
    n, bins = bench.MICRO_N, bench.MICRO_BINS
    x = synth.refit_values(n, seed=bench.SEED, device="cuda")
    ho = torch.zeros(bins, dtype=torch.int64, device="cuda")
    cbo = torch.empty(4, dtype=torch.float32, device="cuda")
    G.gefen_refit_codebook(bins=bins, k=4, codebook_out=cbo, x=x, hist_out=ho)
    got = ho.cpu().numpy().astype(np.uint64)
    xh = x.cpu().numpy()
    del x
    ref = oracle.histogram(xh, bins)
    assert int(ref.sum()) == n
    np.testing.assert_array_equal(got, ref)
