"""GPU parity of gefen_step (Algorithm 1) against the oracle, step by step:
each step starts the oracle from the GPU's own pre-step state, so every step
is compared on identical inputs.  One case per kernel path of the step."""
import numpy as np
import pytest
import torch

import gpu_util as U
import oracle
from paper_2606_13894_gb300 import gefen as G

pytestmark = pytest.mark.gpu

PATH_CASES = {
    # blocks of one: the first tensor four at a time (three left for the
    # scalar form), the others at block offsets that are not multiples of four
    "p1": [(999, 1), (4096, 1), (1000, 1)],
    "stream4k": [(64 * 300, 64), (2048 * 7, 2048), (4096 * 3, 4096), (16 * 999, 16), (768 * 5, 768), (48 * 401, 48)],
    "stream8k": [(8192 * 3, 8192), (6144 * 5, 6144), (4112 * 4, 4112)],
    "tile16_v4": [(16384 * 3, 16384), (12288 * 2, 12288)],
    "generic": [(3 * 1000, 3), (7 * 333, 7), (100 * 50, 100), (2047 * 3, 2047), (2 * 4001, 2)],
    "big_aligned": [(65536 * 2, 65536), (20000 * 3, 20000), (1 << 20, 1 << 20)],
    "big_unaligned": [(30001 * 2, 30001), (8193 * 3, 8193)],
    "mixed": [(1000, 1), (64 * 40, 64), (3 * 77, 3), (40000, 40000), (16384, 16384), (0, 4), (8192, 8192)],
}
# several tiles per persistent CTA, so the shared-memory stage ring wraps
RING_CASES = [(64 * 100_000, 64), (8192 * 1500, 8192), (2048 * 4000, 2048)]


def _run(cases, steps=3, k=256, hist_mode=0, bins=4096, seed=0, switch=False, zero_blocks=0.0, hp=None):
    hp = dict(U.HP, **(hp or {}))
    rng = np.random.default_rng(seed + 100)
    A = U.Arena(cases, seed=seed)
    cb = U.codebook(k, rng)
    cb_new = U.codebook(k, rng) if switch else cb
    A.init_codes(cb)
    d_cb, d_new = torch.from_numpy(cb).cuda(), torch.from_numpy(cb_new).cuda()
    ws = None
    report = []
    for t in range(1, steps + 1):
        gb = A.draw_grad(zero_blocks=zero_blocks)
        gbits = U.bits(gb)
        pre = A.host()
        enc = d_new if (switch and t == steps) else d_cb
        cbe = cb_new if (switch and t == steps) else cb
        flags = {0: 0, 1: G.GEFEN_HIST, 2: G.GEFEN_HIST_GRAD_ONLY}[hist_mode]
        hist = torch.zeros(bins, dtype=torch.int64, device="cuda") if hist_mode else None
        ws = G.gefen_step(A.table, A.theta, gb, A.codes, A.v, A.s, d_cb, enc, step=t, flags=flags,
                          hist=hist, workspace_buf=ws, **hp)
        G.gefen_step_status(ws)
        th, cd, v, s, h = U.oracle_step(A, pre, gbits, cb, cbe, t, hp, hist_mode=hist_mode, bins=bins)
        got = A.host()
        if hist_mode == 2:
            # only the histogram is written; the state is untouched
            for a, b in zip(got, pre):
                np.testing.assert_array_equal(a, b)
            np.testing.assert_array_equal(hist.cpu().numpy().astype(np.uint64), h)
            report.append(dict(t=t, hist_total=int(h.sum())))
            continue
        te = U.theta_err(got[0], th, hp["lr"])
        ve = U.rel_err(got[2], v)
        M = U.summand_scale(A, pre, gbits, cb, hp["beta1"])
        sok, se = U.scale_ok(got[3], s, M)
        ok, flips = U.code_flips_ok(A, pre, gbits, cb, cbe, got[1], cd, hp, M)
        assert te <= U.THETA_TOL, f"step {t}: theta error {te}"
        assert ve <= U.STATE_TOL, f"step {t}: v error {ve}"
        assert sok, f"step {t}: s error {se} (relative to the summand scale)"
        assert ok, f"step {t}: {flips} code flips beyond the margin rule"
        if hist_mode == 1:
            hg = hist.cpu().numpy().astype(np.int64)
            assert hg.sum() == int(h.sum())
            # cells may differ only by values within 1e-6 of a cell edge, or
            # whose m is within fp32 error of 0 (the sign itself is ambiguous)
            x_all, amb_sign = [], 0
            for (o, n, p, b) in A.entries:
                if n == 0:
                    continue
                m, smax = oracle.step_momentum(gbits[o:o + n].copy(), pre[1][o:o + n].copy(),
                                               pre[3][b:b + n // p].copy(), cb, period=p, beta1=hp["beta1"])
                sm = np.repeat(smax, p)
                mb = np.repeat(M[b:b + n // p], p)
                x_all.append((m / np.where(sm > 0, sm, 1))[sm > 0])
                amb_sign += int(np.count_nonzero(np.abs(m) <= U.MARGIN * mb))
            amb = (U.ambiguous_bins(np.concatenate(x_all), bins) if x_all else 0) + amb_sign
            assert np.abs(hg - h.astype(np.int64)).sum() <= 2 * amb
        report.append(dict(t=t, theta=te, v=ve, s=se, flips=flips))
    return report


@pytest.mark.parametrize("path", list(PATH_CASES))
def test_step_parity_per_path(path):
    _run(PATH_CASES[path], steps=3)


@pytest.mark.parametrize("path", ["stream4k", "stream8k", "generic", "big_aligned", "big_unaligned", "p1"])
def test_step_histogram_of_normalised_momentum(path):
    _run(PATH_CASES[path], steps=2, hist_mode=1, bins=4096)


@pytest.mark.parametrize("path", ["stream4k", "mixed", "big_unaligned"])
def test_step_histogram_65536_cells(path):
    _run(PATH_CASES[path], steps=2, hist_mode=1, bins=65536)


@pytest.mark.parametrize("path", list(PATH_CASES))
def test_grad_only_histogram_is_bit_exact(path):
    _run(PATH_CASES[path], steps=1, hist_mode=2, bins=4096)
    _run(PATH_CASES[path], steps=1, hist_mode=2, bins=65536, seed=1)


def test_codebook_switch_decodes_old_encodes_new():
    _run(PATH_CASES["mixed"], steps=3, switch=True)


def test_zero_blocks_and_16_level_codebook():
    _run(PATH_CASES["mixed"] + [(64 * 50, 64)], steps=3, k=16, zero_blocks=0.3)


def test_hyperparameter_variants():
    _run(PATH_CASES["stream4k"], steps=2, hp=dict(beta1=0.0, beta2=0.95, weight_decay=0.1, lr=6e-4))
    _run(PATH_CASES["generic"], steps=2, hp=dict(beta1=0.5, beta2=0.0, weight_decay=0.0, lr=1e-2))


def test_step_leaves_untouched_padding_alone():
    """Elements between tensors (arena padding) are never written."""
    A = U.Arena([(100, 4), (64 * 3, 64)], seed=3)
    cb = U.codebook(256, np.random.default_rng(0))
    A.init_codes(cb)
    A.theta[100:128] = 7.0
    A.codes[100:128] = 9
    gb = A.draw_grad()
    d = torch.from_numpy(cb).cuda()
    G.gefen_step(A.table, A.theta, gb, A.codes, A.v, A.s, d, d, step=1, **U.HP)
    torch.cuda.synchronize()
    assert torch.all(A.theta[100:128] == 7.0) and torch.all(A.codes[100:128] == 9)


def test_stream_ring_wraps_over_many_tiles():
    """Large enough that every persistent CTA streams many tiles through its
    three shared-memory stages (16-level codebook keeps the oracle quick)."""
    _run(RING_CASES, steps=2, k=16)


def test_stream_ring_histogram_and_grad_only():
    _run(RING_CASES[:1], steps=1, k=16, hist_mode=1, bins=4096)
    _run(RING_CASES, steps=1, k=16, hist_mode=2, bins=65536)
