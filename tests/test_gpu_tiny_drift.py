"""The Tiny configuration (4 tensors, blocks = rows, 256-level codebook from
the first gradient's 4096-cell histogram, bit-exact on both sides).

Step parity: 20 steps, each compared with the oracle started from the GPU's
own pre-step state, within the step tolerances.

Drift: the CUDA step and the oracle then run free from the same start for 100
steps on the same seeded gradients.  After one step the parameters agree
within 1e-5 of max(|theta|, lr); later a code decision within rounding of a
midpoint may go either way, after which that element's momentum differs by a
codebook level and its block's scale and codes follow their own path, so the
two trajectories separate.  The curve is printed (run with -s)."""
import numpy as np
import pytest
import torch

import gpu_util as U
import oracle
from paper_2606_13894_gb300 import gefen as G
from paper_2606_13894_gb300 import synth

pytestmark = pytest.mark.gpu

HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
BINS, K, SEED = 4096, 256, 0


def _setup():
    specs = synth.tiny_set()
    offs, total = synth.pack_offsets(specs)
    entries, boff = [], 0
    for s, o in zip(specs, offs):
        entries.append((o, s.numel, s.period, boff))
        boff += s.numel // s.period
    theta = synth.init_params(specs, SEED, device="cuda")
    return specs, entries, total, boff, theta


def _grad(specs, t):
    return synth.draw_grads(specs, SEED, step=t, device="cuda")


def test_tiny_free_running_drift():
    specs, entries, total, nb, theta = _setup()
    table = G.tensor_table(entries)
    codes = torch.zeros(total, dtype=torch.uint8, device="cuda")
    v = torch.zeros(nb, dtype=torch.float32, device="cuda")
    s = torch.zeros(nb, dtype=torch.float32, device="cuda")
    # first codebook from the first gradient (Algorithm 3), on both sides
    g1 = _grad(specs, 1)
    hist = torch.zeros(BINS, dtype=torch.int64, device="cuda")
    cb = torch.empty(K, dtype=torch.float32, device="cuda")
    G.gefen_step(table, theta, g1, codes, v, s, cb, cb, step=1, flags=G.GEFEN_HIST_GRAD_ONLY, hist=hist, **HP)
    G.gefen_refit_codebook(bins=BINS, k=K, codebook_out=cb, hist_in=hist)
    gb1 = U.bits(g1)
    h_ref = np.zeros(BINS, np.uint64)
    for (o, n, p, b) in entries:
        oracle.step(np.zeros(n, np.float32), gb1[o:o + n].copy(), np.zeros(n, np.uint8), np.zeros(n // p, np.float32),
                    np.zeros(n // p, np.float32), np.zeros(K, np.float32), np.zeros(K, np.float32), period=p, t=1,
                    hist=h_ref, hist_mode=2, **HP)
    np.testing.assert_array_equal(hist.cpu().numpy().astype(np.uint64), h_ref)
    cb_ref = oracle.dp(h_ref, K)["codebook"].astype(np.float32)
    np.testing.assert_array_equal(cb.cpu().numpy(), cb_ref)
    zc = U.zero_code(cb_ref)
    codes.fill_(zc)

    th_o = theta.cpu().numpy().copy()
    cd_o = np.full(total, zc, np.uint8)
    v_o = np.zeros(nb, np.float32)
    s_o = np.zeros(nb, np.float32)
    drift = []
    for t in range(1, 101):
        g = _grad(specs, t)
        G.gefen_step(table, theta, g, codes, v, s, cb, cb, step=t, **HP)
        gb = U.bits(g)
        for (o, n, p, b) in entries:
            sl, bl = slice(o, o + n), slice(b, b + n // p)
            tv, cv, vv, sv = th_o[sl].copy(), cd_o[sl].copy(), v_o[bl].copy(), s_o[bl].copy()
            oracle.step(tv, gb[sl].copy(), cv, vv, sv, cb_ref, cb_ref, period=p, t=t, **HP)
            th_o[sl], cd_o[sl], v_o[bl], s_o[bl] = tv, cv, vv, sv
        th_g = theta.cpu().numpy()
        live = np.concatenate([np.arange(o, o + n) for (o, n, _, _) in entries])
        err = U.theta_err(th_g[live], th_o[live], HP["lr"])
        flips = int(np.count_nonzero(codes.cpu().numpy()[live] != cd_o[live]))
        mean_err = float(np.mean(np.abs(th_g[live].astype(np.float64) - th_o[live]) /
                                 np.maximum(np.abs(th_o[live].astype(np.float64)), HP["lr"])))
        drift.append((t, err, mean_err, flips))
        if t == 1:
            assert err <= U.THETA_TOL, f"after one step: {err}"
    print("\nTiny drift (step, max and mean |dtheta| / max(|theta|, lr), codes differing of %d):" % live.size)
    for t, e, me, f in drift:
        if t in (1, 2, 3, 5, 10, 20, 50, 100):
            print(f"  {t:4d}  {e:.3e}  {me:.3e}  {f}")
    # the trajectories separate through individual codes, not as a whole
    assert drift[-1][2] <= 1e-2


def test_tiny_20_steps_step_parity():
    specs, entries, total, nb, theta = _setup()
    table = G.tensor_table(entries)
    codes = torch.zeros(total, dtype=torch.uint8, device="cuda")
    v = torch.zeros(nb, dtype=torch.float32, device="cuda")
    s = torch.zeros(nb, dtype=torch.float32, device="cuda")
    g1 = _grad(specs, 1)
    hist = torch.zeros(BINS, dtype=torch.int64, device="cuda")
    cb = torch.empty(K, dtype=torch.float32, device="cuda")
    G.gefen_step(table, theta, g1, codes, v, s, cb, cb, step=1, flags=G.GEFEN_HIST_GRAD_ONLY, hist=hist, **HP)
    G.gefen_refit_codebook(bins=BINS, k=K, codebook_out=cb, hist_in=hist)
    cb_h = cb.cpu().numpy()
    codes.fill_(U.zero_code(cb_h))

    class Arena:  # the layout the comparison helpers take
        pass
    A = Arena()
    A.entries, A.NB = entries, nb
    for t in range(1, 21):
        g = _grad(specs, t)
        gb = U.bits(g)
        pre = (theta.cpu().numpy().copy(), codes.cpu().numpy().copy(), v.cpu().numpy().copy(), s.cpu().numpy().copy())
        G.gefen_step(table, theta, g, codes, v, s, cb, cb, step=t, **HP)
        got = (theta.cpu().numpy(), codes.cpu().numpy(), v.cpu().numpy(), s.cpu().numpy())
        th, cd, vv, ss, _ = U.oracle_step(A, pre, gb, cb_h, cb_h, t, HP)
        assert U.theta_err(got[0], th, HP["lr"]) <= U.THETA_TOL, t
        assert U.rel_err(got[2], vv) <= U.STATE_TOL, t
        M = U.summand_scale(A, pre, gb, cb_h, HP["beta1"])
        assert U.scale_ok(got[3], ss, M)[0], t
        ok, flips = U.code_flips_ok(A, pre, gb, cb_h, cb_h, got[1], cd, HP, M)
        assert ok, (t, flips)
