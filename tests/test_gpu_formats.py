"""GPU parity of the storage formats (GEFEN_CODES_4BIT: k <= 16, two codes
per byte; GEFEN_PARAMS_BF16: bf16 parameters) on every path that stores them
(p = 1, the streamed tiles, big blocks applied as streamed tiles), step by
step against the oracle from the GPU's own pre-step state.  The oracle works
on unpacked codes and fp32 parameters: codes are unpacked and bf16 values
widened (exactly) before it runs.  A bf16 parameter must be a correct
rounding of a value within the step tolerance of the oracle's: within half a
bf16 unit in the last place plus 1e-5 of max(|theta|, lr)."""
import numpy as np
import pytest
import torch

import gpu_util as U
from paper_2606_13894_gb300 import gefen as G

pytestmark = pytest.mark.gpu

CASES = {
    "p1": [(1000, 1), (4096, 1), (33, 1)],
    # large enough that the flip budget (1e-5 of the entries) is a few flips
    "stream4k": [(64 * 1200, 64), (2048 * 28, 2048), (4096 * 12, 4096), (32 * 3996, 32), (128 * 308, 128)],
    "stream8k": [(8192 * 3, 8192), (6144 * 5, 6144)],
    "big": [(65536 * 2, 65536), (1 << 20, 1 << 20)],
    "mixed": [(1000, 1), (64 * 40, 64), (40960, 40960), (8192, 8192), (0, 4)],
}


def pack4(c):
    c = c.astype(np.uint8)
    if c.size % 2:
        c = np.concatenate([c, np.zeros(1, np.uint8)])
    return (c[0::2] | (c[1::2] << 4)).astype(np.uint8)


def unpack4(b, n):
    out = np.empty(2 * b.size, np.uint8)
    out[0::2] = b & 0xF
    out[1::2] = b >> 4
    return out[:n]


def bf16_ulp(x):
    a = np.abs(x.astype(np.float64))
    e = np.floor(np.log2(np.maximum(a, 1e-38)))
    return np.exp2(e - 7)


def _run(cases, fmt_flags, k, steps=3, hist_step=True, seed=0):
    hp = dict(U.HP)
    rng = np.random.default_rng(seed + 100)
    A = U.Arena(cases, seed=seed)
    cb = U.codebook(k, rng)
    c4 = bool(fmt_flags & G.GEFEN_CODES_4BIT)
    b16 = bool(fmt_flags & G.GEFEN_PARAMS_BF16)
    zc = U.zero_code(cb)
    codes_host = np.full(A.N, zc, np.uint8)
    codes = torch.from_numpy(pack4(codes_host) if c4 else codes_host).cuda()
    if c4:
        codes = torch.cat([codes, torch.zeros(16, dtype=torch.uint8, device="cuda")])
    theta = A.theta.to(torch.bfloat16) if b16 else A.theta
    d_cb = torch.from_numpy(cb).cuda()
    ws = None
    for t in range(1, steps + 1):
        gb = A.draw_grad()
        gbits = U.bits(gb)
        th_pre = theta.float().cpu().numpy().copy()
        cd_pre = unpack4(codes.cpu().numpy(), A.N) if c4 else codes.cpu().numpy().copy()
        pre = (th_pre, cd_pre, A.v.cpu().numpy().copy(), A.s.cpu().numpy().copy())
        hist_mode = 1 if (hist_step and t == steps) else 0
        hist = torch.zeros(4096, dtype=torch.int64, device="cuda") if hist_mode else None
        flags = fmt_flags | (G.GEFEN_HIST if hist_mode else 0)
        ws = G.gefen_step(A.table, theta, gb, codes, A.v, A.s, d_cb, d_cb, step=t, flags=flags, hist=hist,
                          workspace_buf=ws, **hp)
        G.gefen_step_status(ws)
        th, cd, v, s, h = U.oracle_step(A, pre, gbits, cb, cb, t, hp, hist_mode=hist_mode, bins=4096)
        got_th = theta.float().cpu().numpy()
        got_cd = unpack4(codes.cpu().numpy(), A.N) if c4 else codes.cpu().numpy()
        live = np.concatenate([np.arange(o, o + n) for (o, n, _, _) in A.entries if n]) if A.entries else None
        if b16:
            ref = th[live].astype(np.float64)
            tol = 0.5 * bf16_ulp(ref) * (1 + 2 ** -10) + U.THETA_TOL * np.maximum(np.abs(ref), hp["lr"])
            bad = np.abs(got_th[live].astype(np.float64) - ref) > tol
            assert not bad.any(), f"step {t}: {int(bad.sum())} bf16 parameters off"
        else:
            assert U.theta_err(got_th, th, hp["lr"]) <= U.THETA_TOL, t
        assert U.rel_err(A.v.cpu().numpy(), v) <= U.STATE_TOL, t
        M = U.summand_scale(A, pre, gbits, cb, hp["beta1"])
        assert U.scale_ok(A.s.cpu().numpy(), s, M)[0], t
        ok, flips = U.code_flips_ok(A, pre, gbits, cb, cb, got_cd, cd, hp, M)
        assert ok, (t, flips)
        if hist_mode:
            hg = hist.cpu().numpy().astype(np.int64)
            assert hg.sum() == int(h.sum())
    if c4:  # arena padding between tensors keeps its nibbles
        untouched = np.ones(A.N, bool)
        for (o, n, _, _) in A.entries:
            untouched[o:o + n] = False
        assert np.all(unpack4(codes.cpu().numpy(), A.N)[untouched] == zc)


@pytest.mark.parametrize("path", list(CASES))
@pytest.mark.parametrize("fmt", ["c4", "bf16", "c4_bf16"])
def test_format_parity(path, fmt):
    flags = {"c4": G.GEFEN_CODES_4BIT, "bf16": G.GEFEN_PARAMS_BF16,
             "c4_bf16": G.GEFEN_CODES_4BIT | G.GEFEN_PARAMS_BF16}[fmt]
    k = 256 if fmt == "bf16" else 16
    _run(CASES[path], flags, k)
