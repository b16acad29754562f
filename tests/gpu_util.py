"""Helpers shared by the GPU parity tests: arenas of tensors, a step-local
comparison of the CUDA step with the oracle, and the tolerances of the
acceptance bar (codes exact except sub-1e-6 decision margins, parameters and
block state within 1e-5).

The CUDA step computes m = beta1*dec*s + (1-beta1)*g in fp32.  When the two
summands nearly cancel, no fp32 evaluation is accurate relative to m itself,
only relative to the summands.  So the scale s' = max|m| of a block is checked
against M_b, the largest |beta1*dec*s| + |(1-beta1)*g| in the block, and a code
decision counts as ambiguous when moving m by 1e-6 * M_b (or x by 1e-6
relative) can change it."""
import math

import numpy as np
import torch

import oracle
from paper_2606_13894_gb300 import gefen as G

HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
THETA_TOL = 1e-5
STATE_TOL = 1e-5
MARGIN = 1e-6
FLIP_FRAC = 1e-5


def codebook(k, rng, kind="t"):
    """Sorted codebook with the forced -1/+1 endpoints."""
    if kind == "uniform":
        cb = np.linspace(-1.0, 1.0, k)
    else:
        inner = np.sort(np.clip(rng.standard_t(4, k - 2) * 0.15, -0.98, 0.98))
        inner = np.unique(inner)
        while inner.size < k - 2:
            inner = np.unique(np.concatenate([inner, rng.uniform(-0.9, 0.9, k - 2 - inner.size)]))
        cb = np.concatenate([[-1.0], inner, [1.0]])
    return cb.astype(np.float32)


def zero_code(cb):
    return int(np.argmin(np.abs(cb.astype(np.float64))))


class Arena:
    """Tensors packed at 64-element offsets, blocks numbered consecutively."""

    def __init__(self, cases, seed=0, device="cuda"):
        self.rng = np.random.default_rng(seed)
        self.entries, off, boff = [], 0, 0
        for n, p in cases:
            self.entries.append((off, n, p, boff))
            off += (n + 63) // 64 * 64
            boff += n // p
        self.N = max(off, 16)
        self.NB = max(boff, 1)
        self.table = G.tensor_table(self.entries)
        self.device = device
        th = np.zeros(self.N, np.float32)
        for (o, n, p, b) in self.entries:
            th[o:o + n] = self.rng.normal(0, 0.02, n)
        self.theta = torch.from_numpy(th).to(device)
        self.codes = torch.zeros(self.N, dtype=torch.uint8, device=device)
        self.v = torch.zeros(self.NB, dtype=torch.float32, device=device)
        self.s = torch.zeros(self.NB, dtype=torch.float32, device=device)
        # per-block gradient scale, log-uniform over [1e-4, 1e-2]
        self.sig = np.zeros(self.N, np.float32)
        for (o, n, p, b) in self.entries:
            self.sig[o:o + n] = np.repeat(10 ** self.rng.uniform(-4, -2, n // p), p)

    def init_codes(self, cb):
        zc = zero_code(cb)
        self.codes.fill_(zc)

    def draw_grad(self, zero_blocks=0.0):
        g = self.rng.normal(0, 1, self.N).astype(np.float32) * self.sig
        if zero_blocks:
            for (o, n, p, b) in self.entries:
                nb = n // p
                z = self.rng.random(nb) < zero_blocks
                g[o:o + n].reshape(nb, p)[z] = 0.0
        gb = torch.from_numpy(g).to(torch.bfloat16)
        return gb.to(self.device)

    def host(self):
        return (self.theta.cpu().numpy().copy(), self.codes.cpu().numpy().copy(),
                self.v.cpu().numpy().copy(), self.s.cpu().numpy().copy())


def bits(gb: torch.Tensor):
    return gb.detach().cpu().view(torch.int16).numpy().view(np.uint16).copy()


def oracle_step(arena, pre, gbits, cb_dec, cb_enc, t, hp, hist_mode=0, bins=0):
    th, cd, v, s = (a.copy() for a in pre)
    hist = np.zeros(bins, np.uint64) if hist_mode else None
    for (o, n, p, b) in arena.entries:
        sl, bl = slice(o, o + n), slice(b, b + n // p)
        tv, cv, vv, sv = th[sl].copy(), cd[sl].copy(), v[bl].copy(), s[bl].copy()
        oracle.step(tv, gbits[sl].copy(), cv, vv, sv, cb_dec, cb_enc, period=p, t=t,
                    hist=hist, hist_mode=hist_mode, **hp)
        th[sl], cd[sl], v[bl], s[bl] = tv, cv, vv, sv
    return th, cd, v, s, hist


def summand_scale(arena, pre, gbits, cb_dec, beta1):
    """M_b per block: max_i beta1*|dec(c_i)|*s_b + (1-beta1)*|g_i| (double)."""
    _, cd, _, s = pre
    g = torch.from_numpy(gbits.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    M = np.zeros(arena.NB)
    for (o, n, p, b) in arena.entries:
        if n == 0:
            continue
        nb = n // p
        a = beta1 * np.abs(cb_dec.astype(np.float64)[cd[o:o + n]]) * np.repeat(s[b:b + nb].astype(np.float64), p)
        t = a + (1 - beta1) * np.abs(g[o:o + n])
        M[b:b + nb] = t.reshape(nb, p).max(axis=1)
    return M


def scale_ok(got_s, ref_s, M):
    """|s_gpu - s_ref| <= 1e-5 * max(M_b, |s_ref|) for every block."""
    d = np.abs(got_s.astype(np.float64) - ref_s.astype(np.float64))
    tol = STATE_TOL * np.maximum(M, np.abs(ref_s.astype(np.float64)))
    return bool(np.all(d <= tol)), float(np.max(d / np.maximum(tol / STATE_TOL, 1e-300))) if d.size else 0.0


def code_flips_ok(arena, pre, gbits, cb_dec, cb_enc, got, ref, hp, M=None):
    """Codes equal except ambiguous decisions (see the module note), and such
    flips touch at most 1e-5 of the entries (at least one allowed)."""
    bad = np.flatnonzero(got != ref)
    if bad.size == 0:
        return True, 0
    if M is None:
        M = summand_scale(arena, pre, gbits, cb_dec, hp["beta1"])
    _, cd, _, s = pre
    cbe = cb_enc.astype(np.float64)
    for i in bad:
        for (o, n, p, b) in arena.entries:
            if o <= i < o + n:
                blk = b + (i - o) // p
                lo = o + (i - o) // p * p
                m, smax = oracle.step_momentum(gbits[lo:lo + p].copy(), cd[lo:lo + p].copy(),
                                               s[blk:blk + 1].copy(), cb_dec, period=p, beta1=hp["beta1"])
                mi, sp = m[i - lo], smax[0]
                delta = MARGIN * M[blk]
                if abs(mi) <= delta:
                    break  # the sign of m itself is within fp32 error
                x = mi / sp
                dist = np.sort(np.abs(x - cbe))
                slack = MARGIN * max(abs(x), 2.0 ** -20) + 2.0 * delta / sp
                if dist[1] - dist[0] > slack:
                    return False, bad.size
                break
    total = sum(n for (_, n, _, _) in arena.entries)
    return bad.size <= max(1, math.ceil(FLIP_FRAC * total)), bad.size


def theta_err(got, ref, lr):
    den = np.maximum(np.abs(ref.astype(np.float64)), lr)
    return float(np.max(np.abs(got.astype(np.float64) - ref.astype(np.float64)) / den)) if got.size else 0.0


def rel_err(got, ref):
    g, r = got.astype(np.float64), ref.astype(np.float64)
    den = np.maximum(np.abs(r), 1e-30)
    return float(np.max(np.abs(g - r) / den)) if g.size else 0.0


def ambiguous_bins(x64, bins):
    """Number of values whose histogram cell changes within +-1e-6 relative."""
    def cell(x):
        t = (x.astype(np.float32) + np.float32(1.0)).astype(np.float32) * np.float32(0.5 * bins)
        return np.clip(np.floor(t), 0, bins - 1)
    return int(np.count_nonzero(cell(x64 * (1 - MARGIN)) != cell(x64 * (1 + MARGIN))))


_ORACLE_PERIODS = {}


def oracle_model_periods(name: str, seed: int, grads_host=None):
    """The oracle's periods (Algorithm 2) for every tensor of a model-shaped
    set, from its first gradient as the bench draws it (seed, step 1); cached
    per (set, seed) for the test session.  Returns (periods, scores)."""
    from paper_2606_13894_gb300 import synth
    key = (name, seed)
    if key not in _ORACLE_PERIODS:
        specs = synth.CONFIGS[name]()
        offs, _ = synth.pack_offsets(specs)
        if grads_host is None:
            grads_host = bits(synth.draw_grads(specs, seed, step=1, device="cuda"))
        periods, scores = [], []
        for s, o in zip(specs, offs):
            p, _, sc = oracle.infer_blocks(grads_host[o:o + s.numel])
            periods.append(p)
            scores.append(sc)
        _ORACLE_PERIODS[key] = (periods, scores)
    return _ORACLE_PERIODS[key]
