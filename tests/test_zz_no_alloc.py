"""gefen_refit_codebook_static: the refit for callers that cannot allocate
device memory (their memory is reserved up front by a framework or serving
runtime, or they must not synchronise the device as cudaFree does).  It uses
the library's own device array as scratch.  Checked here against the
workspace entry point, bit for bit (the tolerance of the other refit tests),
on two calls in a row whose data and sizes differ, so the second call cannot
lean on what the first left in the shared array.  This file is collected last."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_13894_gb300 import gefen as G
from paper_2606_13894_gb300 import synth

pytestmark = pytest.mark.gpu


def _refit(static, *, bins, k, x=None, hist_in=None):
    cb = torch.empty(k, dtype=torch.float32, device="cuda")
    cs = torch.empty(k, dtype=torch.int32, device="cuda")
    cost = torch.empty(1, dtype=torch.float64, device="cuda")
    ho = torch.zeros(bins, dtype=torch.int64, device="cuda") if x is not None else None
    if static:
        G.gefen_refit_codebook_static(bins=bins, k=k, codebook_out=cb, x=x, hist_in=hist_in, hist_out=ho,
                                      cell_start_out=cs, cost_out=cost)
    else:
        G.gefen_refit_codebook(bins=bins, k=k, codebook_out=cb, x=x, hist_in=hist_in, hist_out=ho,
                               cell_start_out=cs, cost_out=cost)
    torch.cuda.synchronize()
    out = dict(cb=cb.cpu().numpy(), cs=cs.cpu().numpy(), cost=float(cost.cpu()[0]))
    if ho is not None:
        out["hist"] = ho.cpu().numpy()
    return out


def _same(a, b):
    np.testing.assert_array_equal(a["cb"], b["cb"])
    np.testing.assert_array_equal(a["cs"], b["cs"])
    assert a["cost"] == b["cost"]
    if "hist" in a:
        np.testing.assert_array_equal(a["hist"], b["hist"])


def test_static_refit_matches_workspace_refit_on_two_calls_in_a_row():
    # call 1: values, the largest accepted size (4096 cells, 256 levels)
    x1 = synth.refit_values(4096 * 512, seed=11, device="cuda")
    got1 = _refit(True, bins=4096, k=256, x=x1)
    # call 2, right after: a different histogram with fewer cells and levels
    rng = np.random.default_rng(12)
    h = np.zeros(1000, np.int64)
    h[rng.choice(1000, 700, replace=False)] = rng.integers(1, 5000, 700)
    h2 = torch.from_numpy(h).cuda()
    got2 = _refit(True, bins=1000, k=16, hist_in=h2)
    _same(got1, _refit(False, bins=4096, k=256, x=x1))
    _same(got2, _refit(False, bins=1000, k=16, hist_in=h2))
    assert got1["cb"][0] == -1.0 and got1["cb"][-1] == 1.0


def test_static_refit_allocates_nothing():
    # init first (module, array and kernels loaded), then no call changes the
    # device's free memory, outputs being allocated beforehand
    G.gefen_refit_static_init()
    x = synth.refit_values(4096 * 256, seed=13, device="cuda")
    cb = torch.empty(256, dtype=torch.float32, device="cuda")
    ho = torch.zeros(4096, dtype=torch.int64, device="cuda")
    G.gefen_refit_codebook_static(bins=4096, k=256, codebook_out=cb, x=x, hist_out=ho)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(2):
        ho.zero_()
        G.gefen_refit_codebook_static(bins=4096, k=256, codebook_out=cb, x=x, hist_out=ho)
    assert G.gefen_refit_static_status() == 256
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0


def test_static_refit_reports_moment_overflow():
    # N (B-1)^2 >= 2^64: the device-side check fails, the outputs stay as
    # they were and the static status call reports it
    B, k = 4096, 4
    h = np.zeros(B, np.int64)
    h[[0, 7, B - 1]] = 1 << 40
    hd = torch.from_numpy(h).cuda()
    cb = torch.full((k,), 7.0, device="cuda")
    G.gefen_refit_codebook_static(bins=B, k=k, codebook_out=cb, hist_in=hd)
    with pytest.raises(G.GefenError) as e:
        G.gefen_refit_static_status()
    assert e.value.status == G.GEFEN_EDEVICE
    assert torch.all(cb == 7.0)
    # and a valid histogram afterwards is refit normally
    h2 = torch.from_numpy(np.arange(1, B + 1, dtype=np.int64)).cuda()
    G.gefen_refit_codebook_static(bins=B, k=k, codebook_out=cb, hist_in=h2)
    assert G.gefen_refit_static_status() == k


def test_static_refit_rejects_sizes_beyond_its_array():
    cb = torch.empty(256, dtype=torch.float32, device="cuda")
    h = torch.ones(8192, dtype=torch.int64, device="cuda")
    with pytest.raises(G.GefenError, match="bins <= 4096"):
        G.gefen_refit_codebook_static(bins=8192, k=256, codebook_out=cb, hist_in=h)
    # the C entry point itself refuses as well
    st = G.load().gefen_refit_codebook_static(None, 0, ctypes.c_void_p(h.data_ptr()), 8192, 256,
                                              ctypes.c_void_p(cb.data_ptr()), None, None, None, None)
    assert st == G.GEFEN_EUNSUPPORTED
