"""Gefen CPU oracle -- TEST INFRASTRUCTURE ONLY.

A plain, slow restatement of the Gefen paper's hot path (arXiv 2606.13894):
Algorithm 1 (the optimizer step), Algorithm 2 (automatic block partitioning),
Algorithm 3 with Appendix D (histogram + exact DP codebook).  The arithmetic
lives in ``gefen_oracle.c`` (double precision, no fused multiply-add); this
module only builds it with gcc and marshals numpy arrays through ctypes.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never links it, and
the two share no code.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gefen_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-ffp-contract=off", "-fPIC", "-shared", "-std=gnu11"]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when the compiler offers it)."""
    with _lock:
        if (not force and os.path.exists(_LIB_PATH)
                and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
            return _LIB_PATH
        os.makedirs(_BUILD, exist_ok=True)
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", *CFLAGS, "-fopenmp", "-o", tmp, _SRC, "-lm"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:  # no OpenMP runtime: build single-threaded
            cmd = ["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"]
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError("oracle build failed:\n" + r.stderr)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    P = ctypes.c_void_p
    i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
    lib.oracle_num_threads.restype = ctypes.c_int
    lib.oracle_set_num_threads.argtypes = [ctypes.c_int32]
    lib.oracle_set_num_threads.restype = None
    lib.oracle_bin.argtypes = [ctypes.c_float, i32]
    lib.oracle_bin.restype = i64
    lib.oracle_histogram.argtypes = [P, i64, i32, P]
    lib.oracle_histogram.restype = None
    lib.oracle_nearest_level.argtypes = [f64, P, i32]
    lib.oracle_nearest_level.restype = i32
    lib.oracle_step.argtypes = [i64, i64, P, P, P, P, P, P, P, i32, f64, f64,
                                f64, f64, f64, i64, P, i32, i32]
    lib.oracle_step.restype = ctypes.c_int
    lib.oracle_step_momentum.argtypes = [i64, i64, P, P, P, P, f64, P, P]
    lib.oracle_step_momentum.restype = ctypes.c_int
    lib.oracle_step_unquantized.argtypes = [i64, i64, P, P, P, P, f64, f64, f64,
                                            f64, f64, i64]
    lib.oracle_step_unquantized.restype = ctypes.c_int
    lib.oracle_dp.argtypes = [P, i32, i32, P, P, P, P, P]
    lib.oracle_dp.restype = i32
    lib.oracle_dp_cell_cost.argtypes = [P, i32, i64, i64, i32]
    lib.oracle_dp_cell_cost.restype = f64
    lib.oracle_dp_entries.argtypes = [P, i32, i32, i32, P, P, i64, P, P]
    lib.oracle_dp_entries.restype = ctypes.c_int
    lib.oracle_divisors.argtypes = [i64, P, i64]
    lib.oracle_divisors.restype = i64
    lib.oracle_infer_blocks.argtypes = [P, i64, f64, P, P, P, i64]
    lib.oracle_infer_blocks.restype = i64
    _lib = lib
    return lib


def _ptr(a: np.ndarray):
    assert a.flags.c_contiguous, "oracle arrays must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


def set_num_threads(n: int) -> None:
    """Threads of the oracle's parallel loops (results do not depend on it)."""
    _load().oracle_set_num_threads(int(n))


def num_threads() -> int:
    """Threads the oracle's OpenMP loops use (1 without OpenMP)."""
    return int(_load().oracle_num_threads())


def bin_index(x: float, bins: int) -> int:
    """Histogram cell of one fp32 value (-1 for NaN)."""
    return int(_load().oracle_bin(ctypes.c_float(x), bins))


def histogram(x: np.ndarray, bins: int, hist: np.ndarray | None = None) -> np.ndarray:
    """Counts of fp32 values in ``bins`` uniform cells over [-1, 1] (uint64)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    if hist is None:
        hist = np.zeros(bins, dtype=np.uint64)
    _load().oracle_histogram(_ptr(x), x.size, bins, _ptr(hist))
    return hist


def nearest_level(x: float, codebook: np.ndarray) -> int:
    cb = np.ascontiguousarray(codebook, dtype=np.float32)
    return int(_load().oracle_nearest_level(float(x), _ptr(cb), cb.size))


def step(theta, grad_bits, codes, v, s, cb_dec, cb_enc, *, period, lr, beta1,
         beta2, eps, weight_decay, t, hist=None, hist_mode=0):
    """One Gefen step (Algorithm 1) on one flattened tensor, in place.

    theta f32[n], grad_bits uint16[n] (bf16 bit patterns), codes uint8[n],
    v/s f32[n/period], cb_dec/cb_enc f32[k].  hist_mode 1 adds x = m/s' of
    every nonzero block to ``hist``; 2 histograms g/max|g| and updates nothing.
    """
    n = theta.size
    for a, dt in ((theta, np.float32), (grad_bits, np.uint16), (codes, np.uint8),
                  (v, np.float32), (s, np.float32)):
        assert a.dtype == dt and a.flags.c_contiguous
    cbd = np.ascontiguousarray(cb_dec, dtype=np.float32)
    cbe = np.ascontiguousarray(cb_enc, dtype=np.float32)
    hp = _ptr(hist) if hist is not None else None
    bins = hist.size if hist is not None else 0
    rc = _load().oracle_step(n, period, _ptr(theta), _ptr(grad_bits), _ptr(codes),
                             _ptr(v), _ptr(s), _ptr(cbd), _ptr(cbe), cbd.size,
                             lr, beta1, beta2, eps, weight_decay, t, hp, bins,
                             hist_mode)
    if rc != 0:
        raise ValueError("oracle_step: bad arguments")


def step_momentum(grad_bits, codes, s, cb_dec, *, period, beta1):
    """Unquantised momenta m (double) and per-block max|m| of one step."""
    n = grad_bits.size
    m = np.empty(n, dtype=np.float64)
    smax = np.empty(n // period, dtype=np.float64)
    cbd = np.ascontiguousarray(cb_dec, dtype=np.float32)
    rc = _load().oracle_step_momentum(n, period, _ptr(grad_bits), _ptr(codes),
                                      _ptr(s), _ptr(cbd), beta1, _ptr(m), _ptr(smax))
    if rc != 0:
        raise ValueError("oracle_step_momentum: bad arguments")
    return m, smax


def step_unquantized(theta, g, m, v, *, period, lr, beta1, beta2, eps,
                     weight_decay, t):
    """Gefen step with m kept in double (no codebook); p=1 is AdamW."""
    for a in (theta, g, m, v):
        assert a.dtype == np.float64 and a.flags.c_contiguous
    rc = _load().oracle_step_unquantized(theta.size, period, _ptr(theta), _ptr(g),
                                         _ptr(m), _ptr(v), lr, beta1, beta2, eps,
                                         weight_decay, t)
    if rc != 0:
        raise ValueError("oracle_step_unquantized: bad arguments")


def dp(hist: np.ndarray, k: int, *, tables: bool = False):
    """Exact histogram DP codebook (Algorithm 3, Appendix D).

    Returns dict(codebook f32[k], cell_start int32[k] (first bin of each level,
    -1 for padding), cost (units of 1/B^2), k_eff) and, with ``tables``, the
    full D table and argmin table, shape (k_eff+1, b+1).
    """
    hist = np.ascontiguousarray(hist, dtype=np.uint64)
    B = hist.size
    cb = np.empty(k, dtype=np.float32)
    cs = np.empty(k, dtype=np.int32)
    cost = np.zeros(1, dtype=np.float64)
    b = int(np.count_nonzero(hist))
    D = A = None
    if tables:
        ke = min(k, b)
        D = np.empty((ke + 1) * (b + 1), dtype=np.float64)
        A = np.empty((ke + 1) * (b + 1), dtype=np.int32)
    ke = _load().oracle_dp(_ptr(hist), B, k, _ptr(cb), _ptr(cs), _ptr(cost),
                           _ptr(D) if tables else None, _ptr(A) if tables else None)
    if ke < 0:
        raise ValueError("oracle_dp: bad arguments")
    out = dict(codebook=cb, cell_start=cs, cost=float(cost[0]), k_eff=int(ke))
    if tables:
        out["D"] = D.reshape(ke + 1, b + 1)
        out["A"] = A.reshape(ke + 1, b + 1)
    return out


def dp_cell_cost(hist: np.ndarray, l: int, r: int, kind: int = 0) -> float:
    """Canonical cost of nonempty-bin run [l..r] (1-based); kind 0 interior,
    1 first level (centre -1), 2 last level (centre +1)."""
    hist = np.ascontiguousarray(hist, dtype=np.uint64)
    return float(_load().oracle_dp_cell_cost(_ptr(hist), hist.size, l, r, kind))


def dp_entries(hist, level, dprev, rs, *, last=False):
    """Full-scan D[r][level] and argmin for the given r, from a supplied
    previous-level row ``dprev`` (length b+1)."""
    hist = np.ascontiguousarray(hist, dtype=np.uint64)
    dprev = np.ascontiguousarray(dprev, dtype=np.float64)
    rs = np.ascontiguousarray(rs, dtype=np.int64)
    val = np.empty(rs.size, dtype=np.float64)
    arg = np.empty(rs.size, dtype=np.int32)
    _load().oracle_dp_entries(_ptr(hist), hist.size, level, int(last), _ptr(dprev),
                              _ptr(rs), rs.size, _ptr(val), _ptr(arg))
    return val, arg


def divisors(n: int) -> np.ndarray:
    lib = _load()
    cnt = lib.oracle_divisors(n, None, 0)
    out = np.empty(cnt, dtype=np.int64)
    lib.oracle_divisors(n, _ptr(out), cnt)
    return out


def infer_blocks(grad_bits: np.ndarray, eps: float = 1e-8):
    """Automatic Block Partitioning (Algorithm 2) of one flattened bf16 gradient.

    Returns (period, divisors int64[tau], scores f64[tau]).
    """
    g = np.ascontiguousarray(grad_bits, dtype=np.uint16)
    n = g.size
    divs = divisors(n)
    scores = np.empty(divs.size, dtype=np.float64)
    period = np.zeros(1, dtype=np.int64)
    nd = _load().oracle_infer_blocks(_ptr(g), n, eps, _ptr(period), _ptr(divs),
                                     _ptr(scores), divs.size)
    if nd < 0:
        raise ValueError("oracle_infer_blocks: bad arguments")
    return int(period[0]), divs, scores
