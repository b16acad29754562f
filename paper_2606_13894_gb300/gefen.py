"""ctypes binding of libgefen.so (declared in include/gefen.h).

Argument marshalling only: every function here passes device pointers, sizes
and the current CUDA stream to the entry point of the same name, and raises on
a non-OK status.  Workspaces the caller does not provide are allocated as torch
uint8 tensors (the library itself never allocates).  There is no fallback: if
the library cannot be built or loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Iterable, Optional, Sequence

import torch

from . import build as _build

GEFEN_OK, GEFEN_EINVAL, GEFEN_ECUDA, GEFEN_ENOMEM, GEFEN_ETIMEOUT, GEFEN_EUNSUPPORTED, GEFEN_EDEVICE = range(7)
GEFEN_HIST = 1
GEFEN_HIST_GRAD_ONLY = 2
GEFEN_CODES_4BIT = 4
GEFEN_PARAMS_BF16 = 8
GEFEN_MAX_BINS = 65536
GEFEN_MAX_LEVELS = 256
WS_ALIGN = 256


class GefenError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn}: {msg} (status {status})")
        self.status = status


class gefen_tensor_t(ctypes.Structure):
    _fields_ = [("offset", ctypes.c_int64), ("numel", ctypes.c_int64),
                ("period", ctypes.c_int64), ("block_offset", ctypes.c_int64)]


class gefen_hparams_t(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_double), ("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
                ("eps", ctypes.c_double), ("weight_decay", ctypes.c_double),
                ("step", ctypes.c_int64), ("flags", ctypes.c_uint32)]


EXPORTS = ("gefen_status_string", "gefen_sync_status", "gefen_step_workspace_size", "gefen_step",
           "gefen_step_status",
           "gefen_refit_workspace_size", "gefen_refit_codebook", "gefen_refit_status",
           "gefen_refit_tables", "gefen_infer_workspace_size", "gefen_infer_blocks",
           "gefen_refit_codebook_static", "gefen_refit_static_init", "gefen_refit_static_status",
           "gefen_refit_debug", "gefen_muon_workspace_size", "gefen_muon_step", "gefen_gemm_bf16",
           "gefen_gemm_bf16_sym")

GEFEN_MUON_BF16_GEMM = 1


class gefen_muon_hparams_t(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_double), ("momentum", ctypes.c_double), ("weight_decay", ctypes.c_double),
                ("eps", ctypes.c_double), ("nesterov", ctypes.c_int32), ("ns_steps", ctypes.c_int32),
                ("ns_a", ctypes.c_double), ("ns_b", ctypes.c_double), ("ns_c", ctypes.c_double),
                ("flags", ctypes.c_uint32)]

_lib = None
_lock = threading.Lock()


def lib_path() -> str:
    return _build.LIB


def load(build_if_needed: bool = True):
    """Open libgefen.so (building it first when missing or stale)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if build_if_needed and not _build.up_to_date():
            _build.build()
        if not os.path.exists(_build.LIB):
            raise RuntimeError(f"libgefen.so is not built ({_build.LIB}); run __graft_entry__.build()")
        L = ctypes.CDLL(_build.LIB)
        P, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        L.gefen_status_string.argtypes = [ctypes.c_int]
        L.gefen_status_string.restype = ctypes.c_char_p
        L.gefen_sync_status.argtypes = [P]
        L.gefen_sync_status.restype = ctypes.c_int
        L.gefen_step_workspace_size.argtypes = [P, i32, ctypes.c_uint32]
        L.gefen_step_workspace_size.restype = sz
        L.gefen_step.argtypes = [P, i32, P, P, P, P, P, P, P, i32, gefen_hparams_t, P, i32, P, sz, P]
        L.gefen_step.restype = ctypes.c_int
        L.gefen_step_status.argtypes = [P, P]
        L.gefen_step_status.restype = ctypes.c_int
        L.gefen_refit_workspace_size.argtypes = [i32, i32]
        L.gefen_refit_workspace_size.restype = sz
        L.gefen_refit_codebook.argtypes = [P, i64, P, i32, i32, P, P, P, P, P, sz, P]
        L.gefen_refit_codebook.restype = ctypes.c_int
        L.gefen_refit_codebook_static.argtypes = [P, i64, P, i32, i32, P, P, P, P, P]
        L.gefen_refit_codebook_static.restype = ctypes.c_int
        L.gefen_refit_static_init.argtypes = []
        L.gefen_refit_static_init.restype = ctypes.c_int
        L.gefen_refit_static_status.argtypes = [ctypes.POINTER(i32), P]
        L.gefen_refit_static_status.restype = ctypes.c_int
        L.gefen_refit_debug.argtypes = [i32, ctypes.c_uint32, i64]
        L.gefen_refit_debug.restype = ctypes.c_int
        L.gefen_refit_status.argtypes = [P, ctypes.POINTER(i32), P]
        L.gefen_refit_status.restype = ctypes.c_int
        L.gefen_refit_tables.argtypes = [P, i32, i32, P, P, P]
        L.gefen_refit_tables.restype = ctypes.c_int
        L.gefen_infer_workspace_size.argtypes = [i64]
        L.gefen_infer_workspace_size.restype = sz
        L.gefen_infer_blocks.argtypes = [P, i64, ctypes.c_double, ctypes.POINTER(i64),
                                         ctypes.POINTER(ctypes.c_double), i64, ctypes.POINTER(i64),
                                         P, sz, P]
        L.gefen_infer_blocks.restype = ctypes.c_int
        L.gefen_muon_workspace_size.argtypes = [i64, i64, i64, ctypes.c_uint32]
        L.gefen_muon_workspace_size.restype = sz
        L.gefen_muon_step.argtypes = [i64, i64, i64, P, P, P, P, P, P, i32, gefen_muon_hparams_t, P, sz, P]
        L.gefen_muon_step.restype = ctypes.c_int
        f32 = ctypes.c_float
        L.gefen_gemm_bf16.argtypes = [i32, i32, i32, f32, P, i32, P, i32, f32, P, i32, P, i32, P, i32, P, sz, P]
        L.gefen_gemm_bf16.restype = ctypes.c_int
        L.gefen_gemm_bf16_sym.argtypes = [i32, i32, f32, P, i32, f32, P, i32, P, i32, P, sz, P]
        L.gefen_gemm_bf16_sym.restype = ctypes.c_int
        _lib = L
        return L


def _check(fn: str, status: int):
    if status != GEFEN_OK:
        msg = load().gefen_status_string(status).decode()
        raise GefenError(fn, status, msg)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def tensor_table(entries: Iterable[Sequence[int]]):
    """ctypes array of gefen_tensor_t from (offset, numel, period, block_offset)."""
    entries = list(entries)
    arr = (gefen_tensor_t * max(1, len(entries)))()
    for i, (o, n, p, b) in enumerate(entries):
        arr[i] = gefen_tensor_t(int(o), int(n), int(p), int(b))
    return arr, len(entries)


def workspace(nbytes: int, device=None) -> torch.Tensor:
    """A zero-filled device buffer of at least nbytes, 256-byte aligned (torch
    allocation)."""
    if device is None:
        device = torch.device("cuda", torch.cuda.current_device())
    buf = torch.zeros(max(1, int(nbytes)) + WS_ALIGN, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % WS_ALIGN
    return buf[off:off + max(1, int(nbytes))]


def gefen_status_string(status: int) -> str:
    return load().gefen_status_string(status).decode()


def gefen_sync_status(stream=None):
    _check("gefen_sync_status", load().gefen_sync_status(_stream(stream)))


def gefen_step_workspace_size(table, flags: int = 0) -> int:
    arr, n = table
    return int(load().gefen_step_workspace_size(arr, n, flags))


def gefen_step(table, params, grads, codes, v, scale, codebook_dec, codebook_enc, *, lr, beta1, beta2,
               eps, weight_decay, step, flags=0, hist=None, workspace_buf=None, stream=None):
    """One Gefen step (Algorithm 1) over every tensor of `table` (see tensor_table).

    grads may be a bf16 tensor or its int16/uint16 bit view.  Returns the
    workspace used (reuse it on the next call to avoid reallocation)."""
    arr, n = table
    need = gefen_step_workspace_size(table, flags)
    if workspace_buf is None or workspace_buf.numel() < need:
        workspace_buf = workspace(need, params.device if params is not None else grads.device)
    hp = gefen_hparams_t(float(lr), float(beta1), float(beta2), float(eps), float(weight_decay),
                         int(step), int(flags))
    k = codebook_enc.numel() if codebook_enc is not None else 2
    bins = hist.numel() if hist is not None else 0
    st = load().gefen_step(arr, n, _ptr(params), _ptr(grads), _ptr(codes), _ptr(v), _ptr(scale),
                           _ptr(codebook_dec), _ptr(codebook_enc), k, hp, _ptr(hist), bins,
                           _ptr(workspace_buf), workspace_buf.numel(), _stream(stream))
    _check("gefen_step", st)
    return workspace_buf


def gefen_step_status(workspace_buf, stream=None):
    """Raises GefenError(GEFEN_ETIMEOUT) if a step using this workspace gave up
    a bounded wait (its outputs are then invalid); waits for the stream."""
    _check("gefen_step_status", load().gefen_step_status(_ptr(workspace_buf), _stream(stream)))


def gefen_refit_workspace_size(bins: int, k: int) -> int:
    return int(load().gefen_refit_workspace_size(bins, k))


def gefen_refit_codebook(*, bins: int, k: int, codebook_out, x=None, hist_in=None, hist_out=None,
                         cell_start_out=None, cost_out=None, workspace_buf=None, stream=None):
    """Exact DP codebook (Algorithm 3) from fp32 values x or a u64 histogram.
    Returns the workspace (its DP tables stay valid until the next refit)."""
    need = gefen_refit_workspace_size(bins, k)
    dev = codebook_out.device
    if workspace_buf is None or workspace_buf.numel() < need:
        workspace_buf = workspace(need, dev)
    n = x.numel() if x is not None else 0
    xp = _ptr(x)
    if x is not None and n == 0:  # an empty input still selects the x path
        xp = _ptr(workspace_buf)
    st = load().gefen_refit_codebook(xp, n, _ptr(hist_in), bins, k, _ptr(codebook_out), _ptr(hist_out),
                                     _ptr(cell_start_out), _ptr(cost_out), _ptr(workspace_buf),
                                     workspace_buf.numel(), _stream(stream))
    _check("gefen_refit_codebook", st)
    return workspace_buf


STATIC_MAX_BINS = 4096
STATIC_MAX_LEVELS = 256


def gefen_refit_codebook_static(*, bins: int, k: int, codebook_out, x=None, hist_in=None, hist_out=None,
                                cell_start_out=None, cost_out=None, stream=None):
    """gefen_refit_codebook without a workspace: the library's own device
    array serves as scratch (bins <= 4096, k <= 256).  Nothing is allocated."""
    if bins > STATIC_MAX_BINS or k > STATIC_MAX_LEVELS:
        raise GefenError("gefen_refit_codebook_static",
                         GEFEN_EUNSUPPORTED,
                         f"bins <= {STATIC_MAX_BINS} and k <= {STATIC_MAX_LEVELS} (got bins={bins}, k={k})")
    n = x.numel() if x is not None else 0
    xp = _ptr(x)
    if x is not None and n == 0:  # an empty input still selects the x path
        xp = _ptr(codebook_out)
    st = load().gefen_refit_codebook_static(xp, n, _ptr(hist_in), bins, k, _ptr(codebook_out), _ptr(hist_out),
                                            _ptr(cell_start_out), _ptr(cost_out), _stream(stream))
    _check("gefen_refit_codebook_static", st)


def gefen_refit_static_init():
    """Loads the static refit's module, array and kernels on the current device."""
    _check("gefen_refit_static_init", load().gefen_refit_static_init())


def gefen_refit_static_status(stream=None) -> int:
    """Status of the last static refit on the current device (waits for the
    stream); raises on a device-side failure; returns k_eff."""
    ke = ctypes.c_int32(0)
    _check("gefen_refit_static_status", load().gefen_refit_static_status(ctypes.byref(ke), _stream(stream)))
    return int(ke.value)


def gefen_refit_debug(anchor_stride: int = -1, barrier_extra: int = 0, barrier_spin_cycles: int = 0):
    """Test hook of the refit (see gefen.h); (-1, 0, 0) restores the defaults."""
    _check("gefen_refit_debug", load().gefen_refit_debug(int(anchor_stride), int(barrier_extra),
                                                         int(barrier_spin_cycles)))


def gefen_refit_status(workspace_buf, stream=None) -> int:
    """Waits for the stream; raises on a device-side check failure; returns k_eff."""
    ke = ctypes.c_int32(0)
    st = load().gefen_refit_status(_ptr(workspace_buf), ctypes.byref(ke), _stream(stream))
    _check("gefen_refit_status", st)
    return int(ke.value)


def gefen_refit_tables(workspace_buf, bins: int, k: int, stream=None):
    """(D, A) DP tables of the last refit, shape (k+1, bins+1), on the device."""
    D = torch.empty((k + 1, bins + 1), dtype=torch.float64, device=workspace_buf.device)
    A = torch.empty((k + 1, bins + 1), dtype=torch.int32, device=workspace_buf.device)
    st = load().gefen_refit_tables(_ptr(workspace_buf), bins, k, _ptr(D), _ptr(A), _stream(stream))
    _check("gefen_refit_tables", st)
    return D, A


def gefen_infer_workspace_size(numel: int) -> int:
    return int(load().gefen_infer_workspace_size(numel))


def gefen_infer_blocks(grad, eps: float = 1e-8, *, workspace_buf=None, want_scores: bool = True, stream=None):
    """Automatic Block Partitioning (Algorithm 2) of one gradient tensor.
    Returns (period, scores as a list ordered by ascending divisor)."""
    n = grad.numel()
    need = gefen_infer_workspace_size(n)
    if workspace_buf is None or workspace_buf.numel() < need:
        workspace_buf = workspace(need, grad.device)
    period = ctypes.c_int64(0)
    nd = ctypes.c_int64(0)
    cap = 8192 if want_scores else 0
    scores = (ctypes.c_double * max(1, cap))()
    st = load().gefen_infer_blocks(_ptr(grad), n, float(eps), ctypes.byref(period),
                                   scores if want_scores else None, cap, ctypes.byref(nd),
                                   _ptr(workspace_buf), workspace_buf.numel(), _stream(stream))
    _check("gefen_infer_blocks", st)
    return int(period.value), [scores[i] for i in range(min(cap, nd.value))]


MUON_NS = (3.4445, -4.7750, 2.0315)


def gefen_muon_workspace_size(rows: int, cols: int, period: int, flags: int = 0) -> int:
    return int(load().gefen_muon_workspace_size(rows, cols, period, flags))


def gefen_muon_step(rows, cols, period, params, grads, codes, scale, codebook_dec, codebook_enc, *, lr,
                    momentum=0.95, weight_decay=0.1, eps=1e-7, nesterov=True, ns_steps=5, ns=MUON_NS,
                    flags=0, workspace_buf=None, stream=None):
    """One Gefen-Muon step on a rows x cols matrix (see gefen.h).  Returns the
    workspace used."""
    need = gefen_muon_workspace_size(rows, cols, period, flags)
    if workspace_buf is None or workspace_buf.numel() < need:
        workspace_buf = workspace(need, params.device)
    hp = gefen_muon_hparams_t(float(lr), float(momentum), float(weight_decay), float(eps), int(bool(nesterov)),
                              int(ns_steps), float(ns[0]), float(ns[1]), float(ns[2]), int(flags))
    st = load().gefen_muon_step(rows, cols, period, _ptr(params), _ptr(grads), _ptr(codes), _ptr(scale),
                                _ptr(codebook_dec), _ptr(codebook_enc), codebook_enc.numel(), hp,
                                _ptr(workspace_buf), workspace_buf.numel(), _stream(stream))
    _check("gefen_muon_step", st)
    return workspace_buf


def gefen_gemm_bf16(A, B, *, alpha=1.0, beta=0.0, D=None, C=None, CT=None, workspace_buf=None, stream=None):
    """C = alpha A B^T + beta D (bf16 row-major tensors; CT gets C transposed).
    Allocates C when neither C nor CT is given.  Returns (C, CT, workspace)."""
    M, K = A.shape
    N = B.shape[0]
    if C is None and CT is None:
        C = torch.empty((M, N), dtype=torch.bfloat16, device=A.device)
    if workspace_buf is None:
        workspace_buf = workspace(256, A.device)
    st = load().gefen_gemm_bf16(M, N, K, float(alpha), _ptr(A), A.stride(0), _ptr(B), B.stride(0), float(beta),
                                _ptr(D), D.stride(0) if D is not None else 0, _ptr(C),
                                C.stride(0) if C is not None else 0, _ptr(CT),
                                CT.stride(0) if CT is not None else 0, _ptr(workspace_buf), workspace_buf.numel(),
                                _stream(stream))
    _check("gefen_gemm_bf16", st)
    return C, CT, workspace_buf


def gefen_gemm_bf16_sym(A, *, alpha=1.0, beta=0.0, D=None, C=None, workspace_buf=None, stream=None):
    """C = alpha A A^T + beta D (bf16 row-major; D symmetric), symmetric bit
    for bit.  Allocates C when not given.  Returns (C, workspace)."""
    N, K = A.shape
    if C is None:
        C = torch.empty((N, N), dtype=torch.bfloat16, device=A.device)
    if workspace_buf is None:
        workspace_buf = workspace(256, A.device)
    st = load().gefen_gemm_bf16_sym(N, K, float(alpha), _ptr(A), A.stride(0), float(beta), _ptr(D),
                                    D.stride(0) if D is not None else 0, _ptr(C), C.stride(0),
                                    _ptr(workspace_buf), workspace_buf.numel(), _stream(stream))
    _check("gefen_gemm_bf16_sym", st)
    return C, workspace_buf
