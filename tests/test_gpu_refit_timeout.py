"""The DP's level barriers wait a bounded time: a barrier that can never be
met (the test hook asks for one arrival more than the grid has) gives up
without any fault, the refit's status reports GEFEN_ETIMEOUT to the host, the
outputs are left untouched, and the context stays usable for the next refit."""
import numpy as np
import pytest
import torch

from paper_2606_13894_gb300 import gefen as G

pytestmark = pytest.mark.gpu

SHORT_SPIN = 1 << 22  # cycles: a few milliseconds at the SM clock


def _hist(B, seed):
    rng = np.random.default_rng(seed)
    h = rng.integers(1, 1000, B).astype(np.int64)
    return torch.from_numpy(h).cuda()


@pytest.mark.parametrize("stride", [0, 8])
def test_barrier_wait_runs_out_and_reaches_the_host(stride):
    B, k = 1024, 16
    h = _hist(B, 1)
    cb = torch.full((k,), 7.0, device="cuda")
    cs = torch.full((k,), -7, dtype=torch.int32, device="cuda")
    G.gefen_refit_debug(stride, 1, SHORT_SPIN)
    try:
        ws = G.gefen_refit_codebook(bins=B, k=k, codebook_out=cb, hist_in=h, cell_start_out=cs)
        with pytest.raises(G.GefenError) as e:
            G.gefen_refit_status(ws)
        assert e.value.status == G.GEFEN_ETIMEOUT
    finally:
        G.gefen_refit_debug(-1, 0, 0)
    torch.cuda.synchronize()
    assert torch.all(cb == 7.0) and torch.all(cs == -7)  # outputs untouched
    # the same workspace and context work again
    ws = G.gefen_refit_codebook(bins=B, k=k, codebook_out=cb, hist_in=h, cell_start_out=cs, workspace_buf=ws)
    assert G.gefen_refit_status(ws) == k
    c = cb.cpu().numpy()
    assert c[0] == -1.0 and c[-1] == 1.0 and np.all(np.diff(c) > 0)


def test_static_refit_reports_a_timeout():
    B, k = 512, 8
    h = _hist(B, 2)
    cb = torch.full((k,), 7.0, device="cuda")
    G.gefen_refit_debug(-1, 1, SHORT_SPIN)
    try:
        G.gefen_refit_codebook_static(bins=B, k=k, codebook_out=cb, hist_in=h)
        with pytest.raises(G.GefenError) as e:
            G.gefen_refit_static_status()
        assert e.value.status == G.GEFEN_ETIMEOUT
    finally:
        G.gefen_refit_debug(-1, 0, 0)
    assert torch.all(cb == 7.0)
    G.gefen_refit_codebook_static(bins=B, k=k, codebook_out=cb, hist_in=h)
    assert G.gefen_refit_static_status() == k
