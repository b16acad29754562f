"""Pins for the oracle's optimizer step (Algorithm 1), checked against things
other than the oracle itself: torch's AdamW, the closed form of the first step,
and invariants the paper states for the quantizer (Sec. 5.1.1)."""
import numpy as np
import pytest
import torch

import oracle

HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


def _bf16(x: np.ndarray):
    t = torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    bits = t.view(torch.int16).numpy().view(np.uint16).copy()
    return bits, t.to(torch.float64).numpy()


def _uniform_codebook(k=256):
    return np.linspace(-1.0, 1.0, k).astype(np.float32)


def _zero_code(cb):
    return int(np.argmin(np.abs(cb.astype(np.float64))))


def test_unquantized_p1_matches_torch_adamw():
    """With p = 1 and m kept exactly, the step is textbook AdamW (Sec. 3)."""
    rng = np.random.default_rng(0)
    n = 257
    theta = rng.normal(0, 0.02, n)
    th_t = torch.tensor(theta.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([th_t], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]),
                            eps=HP["eps"], weight_decay=HP["weight_decay"])
    m = np.zeros(n)
    v = np.zeros(n)
    for t in range(1, 11):
        g = rng.normal(0, 1e-3, n) * rng.lognormal(0, 1, n)
        oracle.step_unquantized(theta, g, m, v, period=1, t=t, **HP)
        th_t.grad = torch.tensor(g)
        opt.step()
        np.testing.assert_allclose(theta, th_t.detach().numpy(), rtol=1e-12, atol=1e-15)


def test_first_step_closed_form_any_period():
    """At t = 1 the decoded momentum is 0 (scale 0), so m_1 = (1-beta1) g and
    the update is theta - lr*(g / (rms_b(g) + eps) + wd*theta) for every block."""
    rng = np.random.default_rng(1)
    for p in (1, 4, 16, 96):
        n = p * 7
        theta = rng.normal(0, 0.02, n).astype(np.float32)
        bits, g = _bf16(rng.normal(0, 1e-3, n))
        cb = _uniform_codebook(256)
        codes = np.full(n, _zero_code(cb), np.uint8)
        v = np.zeros(n // p, np.float32)
        s = np.zeros(n // p, np.float32)
        th0 = theta.astype(np.float64)
        oracle.step(theta, bits, codes, v, s, cb, cb, period=p, t=1, **HP)
        rms = np.sqrt((g.reshape(-1, p) ** 2).mean(axis=1))
        expect = th0 - HP["lr"] * (g / (np.repeat(rms, p) + HP["eps"]) + HP["weight_decay"] * th0)
        np.testing.assert_allclose(theta, expect.astype(np.float32), rtol=2e-7, atol=1e-12)
        np.testing.assert_allclose(v, ((1 - HP["beta2"]) * rms ** 2).astype(np.float32), rtol=1e-6)
        np.testing.assert_allclose(s, (np.abs(g).reshape(-1, p).max(1) * (1 - HP["beta1"])).astype(np.float32),
                                   rtol=1e-6)


def test_quantized_p1_is_adamw_up_to_fp32_state():
    """With p = 1 every block's own element has |x| = 1, and the forced +-1
    levels store m exactly (up to fp32): the step must track AdamW."""
    rng = np.random.default_rng(2)
    n = 300
    theta = rng.normal(0, 0.02, n).astype(np.float32)
    th_t = torch.tensor(theta.astype(np.float64), requires_grad=True)
    opt = torch.optim.AdamW([th_t], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]),
                            eps=HP["eps"], weight_decay=HP["weight_decay"])
    cb = _uniform_codebook(256)
    codes = np.full(n, _zero_code(cb), np.uint8)
    v = np.zeros(n, np.float32)
    s = np.zeros(n, np.float32)
    for t in range(1, 11):
        bits, g = _bf16(rng.normal(0, 1e-3, n))
        oracle.step(theta, bits, codes, v, s, cb, cb, period=1, t=t, **HP)
        th_t.grad = torch.tensor(g)
        opt.step()
        assert set(np.unique(codes)) <= {0, 255, _zero_code(cb)}
        np.testing.assert_allclose(theta, th_t.detach().numpy(), rtol=2e-6, atol=2e-9)


def _run_blocks(seed, p, nblk, k, steps=3):
    rng = np.random.default_rng(seed)
    n = p * nblk
    theta = rng.normal(0, 0.02, n).astype(np.float32)
    cb = np.sort(np.concatenate([[-1.0, 1.0], rng.uniform(-0.9, 0.9, k - 2)])).astype(np.float32)
    codes = np.full(n, _zero_code(cb), np.uint8)
    v = np.zeros(nblk, np.float32)
    s = np.zeros(nblk, np.float32)
    sig = np.repeat(10 ** rng.uniform(-4, -2, nblk), p)
    for t in range(1, steps + 1):
        bits, g = _bf16(rng.normal(0, 1, n) * sig)
        prev = (codes.copy(), s.copy())
        oracle.step(theta, bits, codes, v, s, cb, cb, period=p, t=t, **HP)
    return dict(theta=theta, codes=codes, v=v, s=s, cb=cb, bits=bits, prev=prev, p=p, n=n)


@pytest.mark.parametrize("p,k", [(16, 256), (33, 16), (128, 256)])
def test_codes_are_nearest_levels_and_absmax_is_kept(p, k):
    """Every stored code is the nearest level to m/s' (brute force over the
    codebook), and each block's largest |m| maps to -1 or +1: the forced
    endpoints keep the absmax (no contraction, Sec. 5.1.1)."""
    r = _run_blocks(3, p, 20, k)
    m, smax = oracle.step_momentum(r["bits"], r["prev"][0], r["prev"][1], r["cb"],
                                   period=p, beta1=HP["beta1"])
    cb = r["cb"].astype(np.float64)
    x = m / np.repeat(smax, p)
    brute = np.argmin(np.abs(x[:, None] - cb[None, :]), axis=1)
    np.testing.assert_array_equal(r["codes"], brute)
    xb = x.reshape(-1, p)
    cb_blocks = r["codes"].reshape(-1, p)
    top = np.argmax(np.abs(xb), axis=1)
    ends = cb_blocks[np.arange(xb.shape[0]), top]
    assert np.all((ends == 0) | (ends == k - 1))
    # decoded momentum is within half the local level gap of m
    dec = cb[r["codes"]] * np.repeat(r["s"].astype(np.float64), p)
    gaps = np.diff(cb).max() * 0.5 * np.repeat(r["s"].astype(np.float64), p)
    assert np.all(np.abs(dec - m) <= gaps * (1 + 1e-6) + 1e-30)
    assert np.all(r["v"] >= 0)
    np.testing.assert_allclose(r["s"], smax.astype(np.float32), rtol=0)


def test_zero_block_stores_zero_code_and_skips_histogram():
    """A block whose momentum is all zero keeps s = 0, stores the level nearest
    0 everywhere, and adds nothing to the refit histogram ("each nonzero
    block", Algorithm 3)."""
    p, n = 8, 32
    theta = np.zeros(n, np.float32)
    bits = np.zeros(n, np.uint16)
    g = np.zeros(n, np.float32)
    g[8:16] = np.linspace(-1e-3, 1e-3, 8)
    bits, _ = _bf16(g)
    cb = np.array([-1.0, -0.25, 0.125, 1.0], np.float32)
    codes = np.full(n, 2, np.uint8)
    v = np.zeros(4, np.float32)
    s = np.zeros(4, np.float32)
    hist = np.zeros(64, np.uint64)
    oracle.step(theta, bits, codes, v, s, cb, cb, period=p, t=1, hist=hist, hist_mode=1, **HP)
    assert s[0] == 0 and s[2] == 0 and s[3] == 0 and s[1] > 0
    assert np.all(codes[:8] == 2) and np.all(codes[16:] == 2)
    assert int(hist.sum()) == 8


def test_beta1_zero_uses_gradient_exactly():
    """With beta1 = 0 the momentum is the gradient itself: the update equals
    the block-shared-v update computed directly from g (t = 3)."""
    rng = np.random.default_rng(4)
    p, nb = 64, 5
    n = p * nb
    hp = dict(HP, beta1=0.0)
    cb = _uniform_codebook(256)
    theta = rng.normal(0, 0.02, n).astype(np.float32)
    codes = np.full(n, _zero_code(cb), np.uint8)
    v = np.zeros(nb, np.float32)
    s = np.zeros(nb, np.float32)
    vref = np.zeros(nb)
    for t in (1, 2, 3):
        bits, g = _bf16(rng.normal(0, 1e-3, n))
        th0 = theta.astype(np.float64)
        oracle.step(theta, bits, codes, v, s, cb, cb, period=p, t=t, **hp)
        vref = hp["beta2"] * vref.astype(np.float32).astype(np.float64) + (1 - hp["beta2"]) * (g.reshape(nb, p) ** 2).mean(1)
        vhat = vref / (1 - hp["beta2"] ** t)
        expect = th0 - hp["lr"] * (g / (np.repeat(np.sqrt(vhat), p) + hp["eps"]) + hp["weight_decay"] * th0)
        np.testing.assert_allclose(theta, expect, rtol=2e-7, atol=1e-12)


def test_grad_only_histogram_counts_every_nonzero_block_entry():
    """The init histogram holds exactly p entries per nonzero block, and each
    block contributes a value of magnitude 1 (its absmax) at a +-1 cell."""
    rng = np.random.default_rng(5)
    p, nb = 12, 9
    g = rng.normal(0, 1e-3, p * nb).astype(np.float32)
    g[24:36] = 0  # one zero block
    bits, _ = _bf16(g)
    n = g.size
    hist = np.zeros(4096, np.uint64)
    theta = np.zeros(n, np.float32)
    codes = np.zeros(n, np.uint8)
    v = np.zeros(nb, np.float32)
    s = np.zeros(nb, np.float32)
    cb = _uniform_codebook(16)
    oracle.step(theta, bits, codes, v, s, cb, cb, period=p, t=1, hist=hist, hist_mode=2, **HP)
    assert int(hist.sum()) == p * (nb - 1)
    assert int(hist[0] + hist[-1]) >= nb - 1
    assert np.all(theta == 0) and np.all(v == 0)
