"""GPU parity of gefen_muon_step (Gefen-Muon) against the oracle
(oracle/muon.py), step by step from the GPU's own pre-step state.  Codes and
scales follow the step tests' rules; the orthogonalised update X is held to
2e-4 of max|X| with fp32 products (five Newton-Schulz rounds of fp32 GEMMs)
and to 6e-2 with bf16 products (bf16 storage between the rounds, as in
Muon's own), so theta to lr sqrt(max(1, rows/cols)) times that plus 1e-5 of
max(|theta|, lr)."""
import math

import numpy as np
import pytest
import torch

import gpu_util as U
from oracle import muon as M
from paper_2606_13894_gb300 import gefen as G

pytestmark = pytest.mark.gpu


class _One:
    def __init__(self, n, p):
        self.entries, self.NB = [(0, n, p, 0)], n // p


@pytest.mark.parametrize("rows,cols,period", [(64, 256, 256), (256, 64, 64), (128, 128, 32), (33, 100, 100),
                                              (512, 96, 48)])
@pytest.mark.parametrize("bf16", [False, True])
def test_muon_step_parity(rows, cols, period, bf16):
    rng = np.random.default_rng(rows * 7 + cols)
    n = rows * cols
    hp = dict(lr=2e-2, momentum=0.9, weight_decay=0.1, eps=1e-7, nesterov=True)
    cb = U.codebook(256, rng)
    theta = torch.from_numpy(rng.normal(0, 0.02, n).astype(np.float32)).cuda()
    codes = torch.full((n,), U.zero_code(cb), dtype=torch.uint8, device="cuda")
    s = torch.zeros(n // period, dtype=torch.float32, device="cuda")
    d_cb = torch.from_numpy(cb).cuda()
    flags = G.GEFEN_MUON_BF16_GEMM if bf16 else 0
    tolx = 6e-2 if bf16 else 2e-4
    ws = None
    V = _One(n, period)
    adj = hp["lr"] * math.sqrt(max(1.0, rows / cols))
    for t in range(1, 4):
        sig = np.repeat(10 ** rng.uniform(-4, -2, rows), cols)
        gb = torch.from_numpy((rng.normal(size=n) * sig).astype(np.float32)).to(torch.bfloat16).cuda()
        gbits = U.bits(gb)
        pre = (theta.cpu().numpy().copy(), codes.cpu().numpy().copy(), np.zeros(1, np.float32),
               s.cpu().numpy().copy())
        ws = G.gefen_muon_step(rows, cols, period, theta, gb, codes, s, d_cb, d_cb, flags=flags,
                               workspace_buf=ws, **hp)
        torch.cuda.synchronize()
        th, cd, ss = pre[0].copy(), pre[1].copy(), pre[3].copy()
        X = M.muon_step(th, gbits, cd, ss, cb, cb, rows=rows, cols=cols, period=period, **hp)
        got = theta.cpu().numpy()
        tol = adj * tolx * np.abs(X).max() + 1e-5 * np.maximum(np.abs(th.astype(np.float64)), hp["lr"])
        err = np.abs(got.astype(np.float64) - th.astype(np.float64))
        assert np.all(err <= tol), f"step {t}: theta off by {float((err / tol).max()):.3g} x tolerance"
        Mb = U.summand_scale(V, pre, gbits, cb, hp["momentum"])
        assert U.scale_ok(s.cpu().numpy(), ss, Mb)[0], t
        ohp = dict(beta1=hp["momentum"])
        ok, flips = U.code_flips_ok(V, pre, gbits, cb, cb, codes.cpu().numpy(), cd, ohp, Mb)
        assert ok, (t, flips)


def test_muon_step_parity_2048x8192_bf16():
    """The shape the Newton-Schulz timings are quoted on (bf16 products on the
    tensor cores), one step against the oracle."""
    rows, cols, period = 2048, 8192, 8192
    rng = np.random.default_rng(2048)
    n = rows * cols
    hp = dict(lr=2e-2, momentum=0.95, weight_decay=0.1, eps=1e-7, nesterov=True)
    cb = U.codebook(256, rng)
    theta = torch.from_numpy(rng.normal(0, 0.02, n).astype(np.float32)).cuda()
    codes = torch.full((n,), U.zero_code(cb), dtype=torch.uint8, device="cuda")
    s = torch.zeros(n // period, dtype=torch.float32, device="cuda")
    d_cb = torch.from_numpy(cb).cuda()
    sig = np.repeat(10 ** rng.uniform(-4, -2, rows), cols)
    gb = torch.from_numpy((rng.normal(size=n) * sig).astype(np.float32)).to(torch.bfloat16).cuda()
    gbits = U.bits(gb)
    th, cd, ss = theta.cpu().numpy().copy(), codes.cpu().numpy().copy(), s.cpu().numpy().copy()
    ws = G.gefen_muon_step(rows, cols, period, theta, gb, codes, s, d_cb, d_cb, flags=G.GEFEN_MUON_BF16_GEMM, **hp)
    G.gefen_step_status(ws)
    X = M.muon_step(th, gbits, cd, ss, cb, cb, rows=rows, cols=cols, period=period, **hp)
    adj = hp["lr"] * math.sqrt(max(1.0, rows / cols))
    got = theta.cpu().numpy().astype(np.float64)
    tol = adj * 6e-2 * np.abs(X).max() + 1e-5 * np.maximum(np.abs(th.astype(np.float64)), hp["lr"])
    err = np.abs(got - th.astype(np.float64))
    assert np.all(err <= tol), f"theta off by {float((err / tol).max()):.3g} x tolerance"
