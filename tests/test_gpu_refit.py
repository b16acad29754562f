"""GPU parity of gefen_refit_codebook (Algorithm 3, Appendix D): histograms
and DP results bit-exact against the oracle on the same input; at the full
65536-cell / 256-level size, sampled DP entries are recomputed by the oracle's
full scan from the GPU's own previous-level row."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_13894_gb300 import gefen as G
from paper_2606_13894_gb300 import synth

pytestmark = pytest.mark.gpu


def _refit_from_hist(h, k):
    bins = h.size
    hd = torch.from_numpy(h.astype(np.int64)).cuda()
    cbo = torch.empty(k, dtype=torch.float32, device="cuda")
    cs = torch.empty(k, dtype=torch.int32, device="cuda")
    cost = torch.empty(1, dtype=torch.float64, device="cuda")
    ws = G.gefen_refit_codebook(bins=bins, k=k, codebook_out=cbo, hist_in=hd, cell_start_out=cs, cost_out=cost)
    ke = G.gefen_refit_status(ws)
    return cbo.cpu().numpy(), cs.cpu().numpy(), float(cost.cpu()[0]), ke, ws


# 16385 and 65535: cell counts that are not powers of two (the clamped cell
# form); 65536 and 65535: the kernel whose end cells and shoulders leave the
# central shared-memory counters
@pytest.mark.parametrize("bins", [16, 4096, 65536, 1000, 16385, 65535])
@pytest.mark.parametrize("n", [0, 1, 7, 100_003, 3_000_001])
def test_histogram_bit_exact(bins, n):
    rng = np.random.default_rng(n + bins)
    x = np.clip(rng.standard_t(4, n) / 8, -1.2, 1.2).astype(np.float32)
    if n > 20:
        x[:6] = [-1.0, 1.0, 0.0, np.nan, -0.0, np.float32(-1.0 + 2.0 / bins)]
        # outside [-1, 1] (clamped to the end cells) and next to a cell edge
        x[6:14] = [np.inf, -np.inf, 1e30, -1e30, 1.5, -3.0, np.nextafter(np.float32(1), np.float32(0)),
                   np.nextafter(np.float32(-1), np.float32(0))]
    xd = torch.from_numpy(x).cuda()
    ho = torch.zeros(bins, dtype=torch.int64, device="cuda")
    cbo = torch.empty(4, dtype=torch.float32, device="cuda")
    G.gefen_refit_codebook(bins=bins, k=4, codebook_out=cbo, x=xd, hist_out=ho)
    ref = oracle.histogram(x, bins)
    np.testing.assert_array_equal(ho.cpu().numpy().astype(np.uint64), ref)


@pytest.mark.parametrize("bins", [4096, 65536])
@pytest.mark.parametrize("offset", [0, 4])
def test_histogram_one_cell(bins, offset):
    # every value in one cell (x = 0 and its neighbours within the cell), a
    # start past the array's first element, counts far above 2^16 per CTA
    # (about four 32768-value units per CTA, most of them added 512 at a time)
    n = 20_000_003
    x = np.zeros(n + offset, np.float32)
    x[offset + 1::7] = np.float32(0.25 / bins)
    x[offset + 2::11] = -0.0
    xd = torch.from_numpy(x).cuda()[offset:]
    ho = torch.zeros(bins, dtype=torch.int64, device="cuda")
    cbo = torch.empty(4, dtype=torch.float32, device="cuda")
    G.gefen_refit_codebook(bins=bins, k=4, codebook_out=cbo, x=xd, hist_out=ho)
    ref = oracle.histogram(x[offset:], bins)
    assert ref.max() == n
    np.testing.assert_array_equal(ho.cpu().numpy().astype(np.uint64), ref)


@pytest.mark.parametrize("bins", [65536, 40000])
def test_histogram_runs_of_one_cell(bins):
    # runs of 512 to 4096 equal values (a warp round whose values share one
    # cell is counted by one atomic) between random values, NaN runs, and a
    # start that is not a multiple of four values
    rng = np.random.default_rng(bins)
    parts = []
    for _ in range(3000):
        m = int(rng.integers(1, 9)) * 512
        kind = rng.integers(3)
        if kind == 0:
            parts.append(np.full(m, rng.uniform(-1, 1), np.float32))
        elif kind == 1:
            parts.append(rng.uniform(-1, 1, int(rng.integers(1, 700))).astype(np.float32))
        else:
            parts.append(np.full(m, np.nan, np.float32))
    x = np.concatenate([np.zeros(3, np.float32)] + parts)
    xd = torch.from_numpy(x).cuda()[4:]  # 16-byte aligned start past the first values
    ho = torch.zeros(bins, dtype=torch.int64, device="cuda")
    cbo = torch.empty(4, dtype=torch.float32, device="cuda")
    G.gefen_refit_codebook(bins=bins, k=4, codebook_out=cbo, x=xd, hist_out=ho)
    np.testing.assert_array_equal(ho.cpu().numpy().astype(np.uint64), oracle.histogram(x[4:], bins))


def test_histogram_input_must_be_16_byte_aligned():
    # rejected on the host before any launch
    xd = torch.zeros(1027, dtype=torch.float32, device="cuda")[3:]
    ho = torch.zeros(4096, dtype=torch.int64, device="cuda")
    cbo = torch.empty(4, dtype=torch.float32, device="cuda")
    with pytest.raises(G.GefenError):
        G.gefen_refit_codebook(bins=4096, k=4, codebook_out=cbo, x=xd, hist_out=ho)


def _t_hist(B, n, seed):
    x = synth.refit_values(n, seed, device="cpu", block=4096).numpy()
    return oracle.histogram(x, B)


@pytest.fixture
def anchor_stride(request):
    """Forces the DP's anchor stride for one test (0: every end position
    searched over its whole range; s: an anchor every s positions, the other
    positions bracketed by their two anchors), then restores the default."""
    G.gefen_refit_debug(request.param, 0, 0)
    yield request.param
    G.gefen_refit_debug(-1, 0, 0)


@pytest.mark.parametrize("anchor_stride", [0, 2, 7, 32], indirect=True)
@pytest.mark.parametrize("B,k,kind", [(64, 3, "rand"), (512, 16, "rand"), (4096, 256, "t"), (1024, 256, "rand"),
                                      (4096, 16, "t"), (300, 2, "rand"), (65536, 4, "rand"), (2000, 100, "t")])
def test_dp_bit_exact_with_full_tables(B, k, kind, anchor_stride):
    rng = np.random.default_rng(B * 7 + k)
    if kind == "t":
        h = _t_hist(B, 4096 * 256, seed=k)
    else:
        h = np.zeros(B, np.uint64)
        nz = min(B, max(k + 3, B // 3))
        idx = rng.choice(B, nz, replace=False)
        h[idx] = rng.integers(1, 10_000, nz).astype(np.uint64)
    r = oracle.dp(h, k, tables=True)
    cb, cs, cost, ke, ws = _refit_from_hist(h, k)
    assert ke == r["k_eff"]
    np.testing.assert_array_equal(cb, r["codebook"])
    np.testing.assert_array_equal(cs, r["cell_start"])
    assert cost == r["cost"]
    D, A = G.gefen_refit_tables(ws, B, k)
    b = r["D"].shape[1] - 1
    Dg = D.cpu().numpy()[: ke + 1, : b + 1]
    Ag = A.cpu().numpy()[: ke + 1, : b + 1]
    # the last level defines only D[k_eff][b]
    np.testing.assert_array_equal(Dg[:ke], r["D"][:ke])
    np.testing.assert_array_equal(Ag[:ke], r["A"][:ke])
    assert Dg[ke, b] == r["D"][ke, b] and Ag[ke, b] == r["A"][ke, b]


@pytest.mark.parametrize("b", [0, 1, 2, 5])
def test_dp_degenerate_histograms(b):
    B, k = 128, 8
    h = np.zeros(B, np.uint64)
    h[np.linspace(3, 120, b).astype(int)] = 5
    r = oracle.dp(h, k)
    cb, cs, cost, ke, _ = _refit_from_hist(h, k)
    assert ke == r["k_eff"]
    np.testing.assert_array_equal(cb, r["codebook"])
    np.testing.assert_array_equal(cs, r["cell_start"])
    assert cost == r["cost"]


def test_dp_rejects_moment_overflow_on_device():
    B, k = 65536, 4
    h = np.zeros(B, np.uint64)
    h[[0, 5, B - 1]] = np.uint64(1) << np.uint64(40)  # N (B-1)^2 >= 2^64
    hd = torch.from_numpy(h.astype(np.int64)).cuda()
    cbo = torch.full((k,), 7.0, device="cuda")
    ws = G.gefen_refit_codebook(bins=B, k=k, codebook_out=cbo, hist_in=hd)
    with pytest.raises(G.GefenError):
        G.gefen_refit_status(ws)
    assert torch.all(cbo == 7.0)  # outputs untouched


def test_dp_full_size_anchored_equals_unanchored():
    """65536 cells, 256 levels: the anchored search (the automatic choice at
    this size) and the search of every position over its whole range give the
    same D and argmin tables bit for bit."""
    B, k = 65536, 256
    x = synth.refit_values(4096 * 1024, seed=5, device="cuda")
    out = []
    for stride in (-1, 0):
        G.gefen_refit_debug(stride, 0, 0)
        try:
            cbo = torch.empty(k, dtype=torch.float32, device="cuda")
            ws = G.gefen_refit_codebook(bins=B, k=k, codebook_out=cbo, x=x)
            G.gefen_refit_status(ws)
            D, A = G.gefen_refit_tables(ws, B, k)
            out.append((D.cpu().numpy(), A.cpu().numpy(), cbo.cpu().numpy()))
        finally:
            G.gefen_refit_debug(-1, 0, 0)
    np.testing.assert_array_equal(out[0][0], out[1][0])
    np.testing.assert_array_equal(out[0][1], out[1][1])
    np.testing.assert_array_equal(out[0][2], out[1][2])


def test_dp_full_size_sampled_entries_and_properties():
    """65536 cells, 256 levels, Student-t mixture values (the refit
    micro-benchmark's distribution): every sampled D[r][k'] and its argmin
    equal the oracle's full scan over the GPU's own row k'-1, and the codebook
    satisfies the centroid condition and the cost identity."""
    B, k = 65536, 256
    x = synth.refit_values(4096 * 2048, seed=3, device="cuda")
    hd = torch.zeros(B, dtype=torch.int64, device="cuda")
    cbo = torch.empty(k, dtype=torch.float32, device="cuda")
    cs = torch.empty(k, dtype=torch.int32, device="cuda")
    cost = torch.empty(1, dtype=torch.float64, device="cuda")
    ws = G.gefen_refit_codebook(bins=B, k=k, codebook_out=cbo, x=x, hist_out=hd, cell_start_out=cs,
                                cost_out=cost)
    ke = G.gefen_refit_status(ws)
    h = hd.cpu().numpy().astype(np.uint64)
    np.testing.assert_array_equal(h, oracle.histogram(x.cpu().numpy(), B))
    D, A = G.gefen_refit_tables(ws, B, k)
    D, A = D.cpu().numpy(), A.cpu().numpy()
    b = int(np.count_nonzero(h))
    assert ke == min(k, b)
    rng = np.random.default_rng(0)
    for lev in (2, 3, 17, 128, 200, ke - 1):
        rs = np.unique(rng.integers(lev, b + 1, 24))
        val, arg = oracle.dp_entries(h, lev, D[lev - 1, : b + 1], rs)
        np.testing.assert_array_equal(D[lev, rs], val)
        np.testing.assert_array_equal(A[lev, rs], arg)
    val, arg = oracle.dp_entries(h, ke, D[ke - 1, : b + 1], np.array([b]), last=True)
    assert D[ke, b] == val[0] and A[ke, b] == arg[0] and float(cost.cpu()[0]) == val[0]
    # centroid condition and the cost as the sum of the cells' canonical costs
    cb = cbo.cpu().numpy().astype(np.float64)
    starts = cs.cpu().numpy()
    nz = np.flatnonzero(h)
    ranks = [int(np.searchsorted(nz, s)) + 1 for s in starts[:ke]] + [b + 1]
    centers = (2 * np.arange(B) + 1 - B) / B
    tot = 0.0
    for j in range(ke):
        lo, hi = starts[j], (starts[j + 1] if j + 1 < ke else B)
        if 0 < j < ke - 1:
            w = h[lo:hi].astype(np.float64)
            mean = (w * centers[lo:hi]).sum() / w.sum()
            assert abs(cb[j] - mean) <= 2.0 ** -23 * max(abs(mean), 2.0 ** -20)
        kind = 1 if j == 0 else (2 if j == ke - 1 else 0)
        tot += oracle.dp_cell_cost(h, ranks[j], ranks[j + 1] - 1, kind)
    assert tot == pytest.approx(float(cost.cpu()[0]), rel=1e-12)
    assert cb[0] == -1 and cb[ke - 1] == 1 and np.all(np.diff(cb[:ke]) > 0)
