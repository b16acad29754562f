"""Pins for the oracle's exact histogram DP (Algorithm 3, Appendix D) against
brute force, exact rational arithmetic, the centroid condition and the
Lloyd-Max bound the paper claims (Appendix C.1)."""
import itertools
from fractions import Fraction

import numpy as np
import pytest

import oracle


def _centers(B):
    return (2 * np.arange(B) + 1 - B) / B


def _rand_hist(rng, B, nonempty, total=10_000, ends=True):
    h = np.zeros(B, np.uint64)
    idx = rng.choice(np.arange(1, B - 1), size=nonempty - (2 if ends else 0), replace=False)
    if ends:
        idx = np.concatenate([idx, [0, B - 1]])
    w = rng.dirichlet(np.ones(idx.size) * 0.7)
    h[idx] = np.maximum(1, np.round(w * total)).astype(np.uint64)
    return h


def _exact_cost(counts, centers, labels, k):
    """Exact (Fraction) quantisation error of a labelling, centres -1/+1 for the
    first/last level and the weighted mean otherwise."""
    tot = Fraction(0)
    for j in range(k):
        sel = [i for i, lab in enumerate(labels) if lab == j]
        if not sel:
            return None
        c = [Fraction(int(counts[i])) for i in sel]
        m = [Fraction(centers[i]) for i in sel]
        if j == 0:
            a = Fraction(-1)
        elif j == k - 1:
            a = Fraction(1)
        else:
            a = sum(ci * mi for ci, mi in zip(c, m)) / sum(c)
        tot += sum(ci * (mi - a) ** 2 for ci, mi in zip(c, m))
    return tot


@pytest.mark.parametrize("seed,B,b,k", [(0, 64, 9, 3), (1, 32, 10, 4), (2, 128, 11, 5),
                                        (3, 16, 8, 2), (4, 256, 12, 3)])
def test_dp_equals_exact_bruteforce_over_contiguous_partitions(seed, B, b, k):
    rng = np.random.default_rng(seed)
    h = _rand_hist(rng, B, b)
    nz = np.flatnonzero(h)
    centers = [Fraction(int(2 * i + 1 - B), B) for i in nz]
    counts = h[nz]
    best, best_starts = None, None
    for cuts in itertools.combinations(range(1, b), k - 1):
        labels = np.zeros(b, int)
        for j, c in enumerate(cuts):
            labels[c:] = j + 1
        cost = _exact_cost(counts, centers, labels, k)
        if best is None or cost < best:
            best, best_starts = cost, (0,) + cuts
    r = oracle.dp(h, k)
    assert r["k_eff"] == k
    got = tuple(int(np.searchsorted(nz, c)) for c in r["cell_start"][:k])
    exact_got = _exact_cost(counts, centers, np.searchsorted(got, np.arange(b), side="right") - 1, k)
    # the oracle's partition is optimal in exact arithmetic (to double rounding)
    assert float(abs(exact_got - best)) <= 1e-12 * float(best) + 1e-300
    # the reported cost is the optimum in units of 1/B^2
    assert r["cost"] == pytest.approx(float(best) * B * B, rel=1e-12)
    if got != best_starts:  # only an exact tie may select another partition
        assert exact_got == best


def test_dp_contiguity_against_all_labelings():
    """b = 12 nonempty bins, k = 3 levels: all 3^12 labelings (with every level
    used) reach no lower error than the DP's contiguous optimum (Appendix D,
    optimal substructure)."""
    rng = np.random.default_rng(7)
    B = 64
    h = _rand_hist(rng, B, 12)
    nz = np.flatnonzero(h)
    c = h[nz].astype(np.float64)
    m = _centers(B)[nz]
    k = 3
    labels = np.array(list(itertools.product(range(k), repeat=12)), dtype=np.int8)
    cost = np.zeros(labels.shape[0])
    valid = np.ones(labels.shape[0], bool)
    for j in range(k):
        mask = (labels == j)
        s0 = mask @ c
        s1 = mask @ (c * m)
        s2 = mask @ (c * m * m)
        valid &= s0 > 0
        if j == 0:
            a = -1.0
            cj = s2 - 2 * a * s1 + a * a * s0
        elif j == k - 1:
            a = 1.0
            cj = s2 - 2 * a * s1 + a * a * s0
        else:
            with np.errstate(invalid="ignore", divide="ignore"):
                cj = s2 - np.where(s0 > 0, s1 * s1 / np.where(s0 > 0, s0, 1), 0)
        cost += cj
    brute = cost[valid].min() * B * B
    r = oracle.dp(h, k)
    assert r["cost"] == pytest.approx(brute, rel=1e-9)


@pytest.mark.parametrize("seed,B,nonempty,k", [(10, 4096, 900, 64), (11, 1024, 1024, 256),
                                               (12, 512, 300, 16)])
def test_centroid_condition_and_sorted_endpoints(seed, B, nonempty, k):
    rng = np.random.default_rng(seed)
    h = _rand_hist(rng, B, nonempty, total=10**6)
    r = oracle.dp(h, k)
    cb, cs = r["codebook"], r["cell_start"]
    assert cb[0] == -1.0 and cb[-1] == 1.0
    assert np.all(np.diff(cb.astype(np.float64)) > 0)
    centers = _centers(B)
    bounds = list(cs[:k]) + [B]
    assert cs[0] == np.flatnonzero(h)[0]
    for j in range(1, k - 1):
        lo, hi = bounds[j], bounds[j + 1]
        w = h[lo:hi].astype(np.float64)
        assert w.sum() > 0 and h[lo] > 0
        mean = (w * centers[lo:hi]).sum() / w.sum()
        assert abs(float(cb[j]) - mean) <= 2.0 ** -23 * max(abs(mean), 2.0 ** -20)
    # the reported cost is the sum of the cells' canonical costs
    nz = np.flatnonzero(h)
    ranks = [int(np.searchsorted(nz, x)) + 1 for x in cs[:k]] + [nz.size + 1]
    tot = 0.0
    for j in range(k):
        kind = 1 if j == 0 else (2 if j == k - 1 else 0)
        tot += oracle.dp_cell_cost(h, ranks[j], ranks[j + 1] - 1, kind)
    assert tot == pytest.approx(r["cost"], rel=1e-12)


def _lloyd_cost(h, k, init):
    """Lloyd-Max with the endpoints held at -1 and +1 (Sec. 5.1.1)."""
    B = h.size
    nz = np.flatnonzero(h)
    c = h[nz].astype(np.float64)
    m = _centers(B)[nz]
    if init == "linear":
        lv = np.linspace(-1, 1, k)
    else:
        cdf = np.cumsum(c) / c.sum()
        lv = np.interp(np.linspace(0, 1, k), cdf, m)
        lv[0], lv[-1] = -1.0, 1.0
    for _ in range(200):
        lab = np.argmin(np.abs(m[:, None] - lv[None, :]), axis=1)
        new = lv.copy()
        for j in range(1, k - 1):
            sel = lab == j
            if sel.any():
                new[j] = (c[sel] * m[sel]).sum() / c[sel].sum()
        new = np.sort(new)
        if np.allclose(new, lv, rtol=0, atol=1e-15):
            break
        lv = new
    lab = np.argmin(np.abs(m[:, None] - lv[None, :]), axis=1)
    return float((c * (m - lv[lab]) ** 2).sum() * B * B)


@pytest.mark.parametrize("init", ["linear", "quantile"])
def test_dp_never_worse_than_lloyd_max(init):
    """Appendix C.1: the exact DP reaches the lowest quantisation error.  Block
    absmax normalisation puts values at both -1 and +1, so both end cells are
    populated (the recurrence gives every level at least one bin)."""
    rng = np.random.default_rng(20)
    B = 1024
    x = rng.standard_t(4, 200_000)
    x = x / np.abs(x).max()
    x[:2] = (-1.0, 1.0)
    h = oracle.histogram(x.astype(np.float32), B)
    for k in (4, 16, 64):
        r = oracle.dp(h, k)
        assert r["cost"] <= _lloyd_cost(h, k, init) * (1 + 1e-12)


def test_symmetric_histogram_gives_symmetric_codebook():
    B = 256
    rng = np.random.default_rng(21)
    half = rng.integers(0, 50, B // 2).astype(np.uint64)
    half[0] = 5
    h = np.concatenate([half, half[::-1]])
    r = oracle.dp(h, 9)  # odd k: the middle level sits at 0 when unique
    cb = r["codebook"].astype(np.float64)
    np.testing.assert_allclose(cb, -cb[::-1], atol=1e-7)


def test_canonical_costs_match_exact_rationals():
    """Each cell cost is the exact value rounded at most twice (interior) or
    once (fixed centre)."""
    rng = np.random.default_rng(22)
    B = 65536
    h = _rand_hist(rng, B, 200, total=10**9)
    nz = np.flatnonzero(h)
    u = [2 * int(i) + 1 - B for i in nz]
    for _ in range(60):
        l, r = sorted(rng.integers(1, nz.size + 1, 2))
        cs = [int(h[nz[i - 1]]) for i in range(l, r + 1)]
        us = u[l - 1:r]
        s0 = sum(cs)
        s1 = sum(c * x for c, x in zip(cs, us))
        s2 = sum(c * x * x for c, x in zip(cs, us))
        exact_int = Fraction(s0 * s2 - s1 * s1, s0)
        got = oracle.dp_cell_cost(h, l, r, 0)
        assert abs(Fraction(got) - exact_int) <= abs(exact_int) * Fraction(2 ** -52)
        first = s2 + 2 * B * s1 + B * B * s0
        last = s2 - 2 * B * s1 + B * B * s0
        assert oracle.dp_cell_cost(h, l, r, 1) == float(first)
        assert oracle.dp_cell_cost(h, l, r, 2) == float(last)


def test_degenerate_histograms():
    B = 64
    h = np.zeros(B, np.uint64)
    r = oracle.dp(h, 8)
    assert r["k_eff"] == 0 and r["codebook"][0] == -1 and np.all(r["codebook"][1:] == 1)
    h[10] = 3
    r = oracle.dp(h, 8)
    assert r["k_eff"] == 1 and r["cell_start"][0] == 10
    h[[3, 40, 50]] = 1
    r = oracle.dp(h, 8)  # b = 4 < k: every bin its own level, padded with +1
    assert r["k_eff"] == 4
    c = _centers(B)
    np.testing.assert_allclose(r["codebook"][:4], [-1, c[10], c[40], 1], rtol=1e-7)
    assert np.all(r["codebook"][4:] == 1) and np.all(r["cell_start"][4:] == -1)
    assert list(r["cell_start"][:4]) == [3, 10, 40, 50]


def test_dp_entries_reproduce_table_rows():
    rng = np.random.default_rng(23)
    B = 512
    h = _rand_hist(rng, B, 200, total=10**6)
    k = 12
    r = oracle.dp(h, k, tables=True)
    D, A = r["D"], r["A"]
    b = D.shape[1] - 1
    for lev in (2, 5, 11):
        rs = np.arange(lev, b + 1)
        val, arg = oracle.dp_entries(h, lev, D[lev - 1], rs)
        np.testing.assert_array_equal(val, D[lev, lev:])
        np.testing.assert_array_equal(arg, A[lev, lev:])
    val, arg = oracle.dp_entries(h, k, D[k - 1], np.array([b]), last=True)
    assert val[0] == D[k, b] == r["cost"]


def _exact_interior(cs, us):
    s0 = sum(cs)
    s1 = sum(c * x for c, x in zip(cs, us))
    s2 = sum(c * x * x for c, x in zip(cs, us))
    return Fraction(s0 * s2 - s1 * s1, s0)


@pytest.mark.parametrize("seed", range(4))
def test_interior_cost_satisfies_the_quadrangle_inequality(seed):
    """Appendix D's interior cost (squared error of a run of cells about its
    weighted mean), in exact rationals: for a <= b <= c <= d,
    cost(a..c) + cost(b..d) <= cost(a..d) + cost(b..c).  The CUDA DP's
    anchored bracketing rests on this inequality; it also makes the exact
    smallest minimiser of each DP row non-decreasing in r, checked here on
    exact rational D rows."""
    rng = np.random.default_rng(100 + seed)
    B = 4096
    h = _rand_hist(rng, B, 40, total=10**7)
    nz = np.flatnonzero(h)
    cs = [int(h[i]) for i in nz]
    us = [2 * int(i) + 1 - B for i in nz]
    b = len(cs)
    w = {}

    def cost(l, r):  # 1-based ranks, l <= r
        if (l, r) not in w:
            w[(l, r)] = _exact_interior(cs[l - 1:r], us[l - 1:r])
        return w[(l, r)]

    for _ in range(400):
        a, bb, c, d = sorted(rng.integers(1, b + 1, 4))
        assert cost(a, c) + cost(bb, d) <= cost(a, d) + cost(bb, c)
    # exact D rows for levels 2..4 (first level at -1) and their smallest minimisers
    first = [None] + [sum(Fraction(cs[j]) * Fraction(us[j] + B) ** 2 for j in range(r)) for r in range(1, b + 1)]
    prev = first
    for kk in range(2, 5):
        row, arg = [None] * (b + 1), [0] * (b + 1)
        for r in range(kk, b + 1):
            vals = [(prev[l - 1] + cost(l, r), l) for l in range(kk, r + 1)]
            best = min(v for v, _ in vals)
            row[r] = best
            arg[r] = min(l for v, l in vals if v == best)
        assert all(arg[r] <= arg[r + 1] for r in range(kk, b))
        prev = row
