"""Pins for the oracle's histogram (Algorithm 3's binning over [-1, 1]) and
its automatic block partitioning (Algorithm 2, Sec. 5.1 partition score)."""
import json
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- histogram
@pytest.mark.parametrize("B", [16, 4096, 65536])
def test_bin_edges_by_hand(B):
    """Cell i is [-1 + 2i/B, -1 + 2(i+1)/B); +1 belongs to the last cell."""
    assert oracle.bin_index(-1.0, B) == 0
    assert oracle.bin_index(1.0, B) == B - 1
    assert oracle.bin_index(0.0, B) == B // 2
    assert oracle.bin_index(float("nan"), B) == -1
    assert oracle.bin_index(-7.0, B) == 0 and oracle.bin_index(3.0, B) == B - 1
    for i in (0, 1, 2, B // 4, B // 2 - 1, B // 2 + 1, B - 2, B - 1):
        edge = np.float32(-1.0 + 2.0 * i / B)
        assert oracle.bin_index(float(edge), B) == i
        mid = np.float32(-1.0 + (2.0 * i + 1.0) / B)
        assert oracle.bin_index(float(mid), B) == i
        if i > 0:
            below = np.nextafter(edge, np.float32(-2.0), dtype=np.float32)
            if np.float32(below + np.float32(1.0)) != np.float32(edge + np.float32(1.0)):
                assert oracle.bin_index(float(below), B) == i - 1


@pytest.mark.parametrize("B", [4096, 1000, 16385, 65535])
def test_histogram_matches_numpy_away_from_edges(B):
    # odd B: the cell edges are not fp32 values, so only values clear of them
    # have a cell that does not depend on rounding
    rng = np.random.default_rng(B)
    x = np.clip(rng.standard_t(4, 300_000) / 12, -1, 1).astype(np.float32)
    t = (x.astype(np.float64) + 1) * B / 2
    # clear of cell edges by more than the two fp32 roundings of the cell
    # definition can move t (each at most 2^-24 relative: together < B 2^-23)
    keep = np.abs(t - np.round(t)) > max(1e-3, B * 2.0 ** -21)
    x = x[keep]
    h = oracle.histogram(x, B)
    ref, _ = np.histogram(x.astype(np.float64), bins=B, range=(-1.0, 1.0))
    np.testing.assert_array_equal(h, ref.astype(np.uint64))
    assert int(h.sum()) == x.size


# ---------------------------------------------------------- block inference
def _bits(g: np.ndarray):
    return torch.from_numpy(g.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("rows,cols,stripe", [(48, 768, 64), (24, 512, 128), (16, 960, 40)])
def test_planted_stripe_periods_are_recovered(rows, cols, stripe):
    """Gradient scales that alternate between two levels every `stripe`
    columns make every stripe boundary a jump of log g^2 while every block of
    two stripes has the same mean: S(stripe) is the unique peak (Sec. 5.1)."""
    rng = np.random.default_rng(rows * cols + stripe)
    sig = np.where((np.arange(cols) // stripe) % 2 == 0, 1e-2, 1e-3)[None, :]
    g = rng.normal(0, 1, (rows, cols)) * sig
    p, divs, S = oracle.infer_blocks(_bits(g.reshape(-1)))
    assert p == stripe, (p, dict(zip(divs.tolist(), np.round(S, 3).tolist())))


@pytest.mark.parametrize("rows,cols", [(64, 256), (96, 1024), (40, 384)])
def test_planted_row_periods_are_recovered(rows, cols):
    """One log-uniform scale per row (the Tiny and Llama-FFN structure): the
    row length is the peak (rows differ, halves of a row do not)."""
    rng = np.random.default_rng(rows * cols)
    sig = 10 ** rng.uniform(-3, -1, rows)[:, None]
    g = rng.normal(0, 1, (rows, cols)) * sig
    p, divs, S = oracle.infer_blocks(_bits(g.reshape(-1)))
    assert p == cols, (p, dict(zip(divs.tolist(), np.round(S, 3).tolist())))


def test_iid_and_prime_sizes_fall_back_to_one():
    rng = np.random.default_rng(3)
    assert oracle.infer_blocks(_bits(rng.normal(0, 1e-3, 7919)))[0] == 1  # prime n
    assert oracle.infer_blocks(_bits(np.array([0.5])))[0] == 1
    p, divs, S = oracle.infer_blocks(_bits(rng.normal(0, 1e-3, 2)))
    assert p == 1 and list(divs) == [1, 2] and np.isnan(S[-1])


def test_scores_match_direct_definition():
    rng = np.random.default_rng(4)
    n = 2 * 2 * 3 * 5 * 7 * 4  # 1680, 40 divisors
    g = rng.normal(0, 1e-3, n) * np.repeat(10 ** rng.uniform(-4, -2, n // 30), 30)
    bits = _bits(g)
    gd = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    z = np.log(gd * gd + 1e-8)
    p, divs, S = oracle.infer_blocks(bits, eps=1e-8)
    assert list(divs) == [d for d in range(1, n + 1) if n % d == 0]
    for d, s in zip(divs, S):
        mu = z.reshape(-1, d).mean(axis=1)
        ref = np.abs(np.diff(mu)).mean() if mu.size > 1 else np.nan
        if np.isnan(ref):
            assert np.isnan(s)
        else:
            assert s == pytest.approx(ref, rel=1e-12)
    # selection rule: strict local maxima among 1 < p < n, then the largest
    cand = [(S[i], divs[i]) for i in range(1, len(divs) - 1) if S[i] > S[i - 1] and S[i] > S[i + 1]]
    assert p == (max(cand, key=lambda t: (t[0], -t[1]))[1] if cand else 1)


def _max_tau(lo, hi):
    """max number of divisors over [lo, hi] by a segmented sieve (independent
    of the oracle's trial division)."""
    n = hi - lo + 1
    cnt = np.zeros(n, dtype=np.uint16)
    r = int(np.sqrt(hi)) + 1
    for d in range(1, r + 1):
        start = max(-(-lo // d) * d, d * d)
        if start > hi:
            continue
        cnt[start - lo::d] += 2
    sq = np.arange(int(np.ceil(np.sqrt(lo))), int(np.sqrt(hi)) + 1, dtype=np.int64) ** 2
    cnt[sq - lo] -= 1
    i = int(np.argmax(cnt))
    return int(cnt[i]), lo + i


def test_divisor_count_maximum_printed_in_paper_small_interval():
    """Sec. 5.1 prints max tau(n) over [0.9e6, 1.1e6] = 256."""
    fx = json.load(open(os.path.join(GOLDEN, "divisor_count_maxima.json")))
    case = fx["cases"][0]
    tau, arg = _max_tau(*case["interval"])
    assert tau == case["max_tau"]
    assert oracle.divisors(arg).size == tau


@pytest.mark.slow
def test_divisor_count_maximum_printed_in_paper_large_interval():
    """Sec. 5.1 prints max tau(n) over [0.9e9, 1.1e9] = 1344."""
    fx = json.load(open(os.path.join(GOLDEN, "divisor_count_maxima.json")))
    case = fx["cases"][1]
    lo, hi = case["interval"]
    best, arg = 0, 0
    step = 20_000_000
    for a in range(lo, hi + 1, step):
        t, x = _max_tau(a, min(hi, a + step - 1))
        if t > best:
            best, arg = t, x
    assert best == case["max_tau"]
    assert oracle.divisors(arg).size == best


def test_largest_proper_divisor_is_never_selected():
    """Two halves with very different scales make S(n/2) the largest score,
    but its right neighbour S(n) is undefined (one block), so n/2 is not a
    strict local maximum over the sorted divisors (Algorithm 2)."""
    rng = np.random.default_rng(5)
    n = 4096
    g = rng.normal(0, 1, n) * np.where(np.arange(n) < n // 2, 1e-4, 1e-1)
    p, divs, S = oracle.infer_blocks(_bits(g))
    interior = S[1:-1]
    assert divs[1 + int(np.nanargmax(interior))] == n // 2  # n/2 scores highest
    assert p != n // 2


def test_nearest_level_ties_go_to_the_lower_index():
    cb = np.array([-1.0, -0.5, 0.0, 0.5, 1.0], np.float32)
    assert oracle.nearest_level(0.25, cb) == 2
    assert oracle.nearest_level(-0.75, cb) == 0
    assert oracle.nearest_level(0.2500001, cb) == 3
    sym = np.array([-1.0, -0.25, 0.25, 1.0], np.float32)
    assert oracle.nearest_level(0.0, sym) == 1
