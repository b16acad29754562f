"""Gefen-Muon CPU oracle -- TEST INFRASTRUCTURE ONLY.

Gefen-Muon (the paper's appendix "Gefen-Muon") keeps Muon's momentum buffer
in Gefen's form -- codes of a learned codebook and a per-block absmax scale
(Algorithm 1, Quantize) -- and leaves Muon's orthogonalisation unchanged.
Muon's step (Jordan et al.'s optimizer, in the form of PyTorch's
torch.optim.Muon, which the paper uses for the orthogonalisation):

    buf  <- lerp(buf, g, 1 - mu)              (= mu * buf + (1 - mu) * g)
    U    <- lerp(g, buf, mu) with Nesterov, else buf
    X    <- U / max(||U||_F, eps), on the transpose when rows > cols
    X    <- a X + (b A + c A A) X,  A = X X^T   (ns_steps times)
    theta <- theta (1 - lr wd) - lr sqrt(max(1, rows/cols)) X

Here buf is decoded from the codes (Algorithm 1's m_{t-1}) and re-encoded
after the step.  Plain numpy in double precision; matrix products use
numpy's matmul.  Only tests/ may import this module.
"""
from __future__ import annotations

import numpy as np

NS_COEFFICIENTS = (3.4445, -4.7750, 2.0315)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def newton_schulz(U: np.ndarray, steps: int = 5, coefficients=NS_COEFFICIENTS, eps: float = 1e-7) -> np.ndarray:
    """Muon's quintic Newton-Schulz iteration on a 2-D matrix (double)."""
    a, b, c = coefficients
    X = np.array(U, dtype=np.float64)
    transposed = X.shape[0] > X.shape[1]
    if transposed:
        X = X.T
    X = X / max(np.linalg.norm(X), eps)
    for _ in range(steps):
        A = X @ X.T
        B = b * A + c * (A @ A)
        X = a * X + B @ X
    return X.T if transposed else X


def nearest_codes(x: np.ndarray, codebook: np.ndarray) -> np.ndarray:
    """Index of the nearest level (ties to the lower index) of each x."""
    cb = codebook.astype(np.float64)
    mids = 0.5 * (cb[:-1] + cb[1:])
    return np.searchsorted(mids, x, side="left").astype(np.uint8)


def muon_step(theta, grad_bits, codes, s, cb_dec, cb_enc, *, rows, cols, period, lr, momentum,
              weight_decay, nesterov=True, ns_steps=5, ns_coefficients=NS_COEFFICIENTS, eps=1e-7):
    """One Gefen-Muon step on one rows x cols matrix (row-major), in place on
    theta (f32), codes (u8, unpacked) and s (f32 per block of `period`).
    Returns the orthogonalised update X (double, rows x cols)."""
    n = rows * cols
    p = period
    nb = n // p
    g = bf16_to_f64(grad_bits)
    sb = np.repeat(s.astype(np.float64), p)
    m = momentum * cb_dec.astype(np.float64)[codes] * sb + (1.0 - momentum) * g
    s_new = np.abs(m).reshape(nb, p).max(axis=1)
    zero = int(nearest_codes(np.zeros(1), cb_enc)[0])
    snr = np.repeat(s_new, p)
    x = np.divide(m, snr, out=np.zeros_like(m), where=snr > 0)
    c = nearest_codes(x, cb_enc)
    c[snr == 0] = zero
    U = g + momentum * (m - g) if nesterov else m
    X = newton_schulz(U.reshape(rows, cols), ns_steps, ns_coefficients, eps)
    adj = lr * np.sqrt(max(1.0, rows / cols))
    th = theta.astype(np.float64) * (1.0 - lr * weight_decay) - adj * X.reshape(-1)
    theta[:] = th.astype(np.float32)
    codes[:] = c
    s[:] = s_new.astype(np.float32)
    return X
