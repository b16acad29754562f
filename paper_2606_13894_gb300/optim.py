"""A torch.optim-compatible Gefen optimizer (AdamW's signature) on libgefen.

Each parameter group's parameters are moved into one flat fp32 arena on first
use (the parameters become views of it, so the model sees every update); their
gradients are gathered into a bf16 arena before each step.  The first step
infers every tensor's blocks from its gradient (Algorithm 2, unless periods
are given) and learns the first codebook from that gradient (Algorithm 3 on
the histogram of g / block absmax); from then on each step is one gefen_step
call over the whole group (Algorithm 1).  With refit_every = N > 0, every N-th
step also histograms the normalised momentum and refits the codebook; the next
step decodes with the old codebook and encodes with the new one.

All arithmetic of the step runs in the library's CUDA kernels; this module
only lays out memory and sequences calls.  CUDA fp32 or bf16 parameters are
required (bf16 ones are kept in bf16, the update computed in fp32); with at
most 16 levels the codes are stored two per byte.  There is no CPU path.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence

import torch

from . import gefen as G

ALIGN = 64  # elements between tensors in an arena (16 is the library's minimum)


class _Arena:
    """The packed state of one parameter group."""

    def __init__(self, params: List[torch.nn.Parameter], levels: int, bins: int, four_bit: bool):
        dev = params[0].device
        dtype = params[0].dtype
        self.params = params
        self.four_bit = four_bit
        self.flags = (G.GEFEN_CODES_4BIT if four_bit else 0) | (G.GEFEN_PARAMS_BF16 if dtype == torch.bfloat16 else 0)
        self.offsets, o = [], 0
        for p in params:
            self.offsets.append(o)
            o += (p.numel() + ALIGN - 1) // ALIGN * ALIGN
        self.total = max(o, ALIGN)
        self.theta = torch.zeros(self.total, dtype=dtype, device=dev)
        with torch.no_grad():
            for p, off in zip(params, self.offsets):
                self.theta[off:off + p.numel()].copy_(p.detach().reshape(-1))
                p.data = self.theta[off:off + p.numel()].view_as(p)
        self.grads = torch.zeros(self.total, dtype=torch.bfloat16, device=dev)
        self.gviews = [self.grads[off:off + p.numel()].view_as(p) for p, off in zip(params, self.offsets)]
        self.codes = torch.zeros(self.total // 2 if four_bit else self.total, dtype=torch.uint8, device=dev)
        self.levels, self.bins = levels, bins
        self.cb = torch.empty(levels, dtype=torch.float32, device=dev)
        self.cb_new = torch.empty(levels, dtype=torch.float32, device=dev)
        self.hist = torch.zeros(bins, dtype=torch.int64, device=dev)
        self.periods: Optional[List[int]] = None
        self.v = self.s = None
        self.table = None
        self.entries: List[tuple] = []
        self.t = 0
        self.switch = False  # the next step encodes with cb_new
        self.ws = self.rws = None
        self._sub = {}

    def set_periods(self, periods: Sequence[int]):
        self.periods = [int(p) for p in periods]
        self.entries, b = [], 0
        for p, off, per in zip(self.params, self.offsets, self.periods):
            if per < 1 or p.numel() % per:
                raise ValueError(f"period {per} does not divide a tensor of {p.numel()} elements")
            self.entries.append((off, p.numel(), per, b))
            b += p.numel() // per
        dev = self.theta.device
        self.v = torch.zeros(max(b, 1), dtype=torch.float32, device=dev)
        self.s = torch.zeros(max(b, 1), dtype=torch.float32, device=dev)
        self.table = G.tensor_table(self.entries)
        self._sub = {}

    def table_for(self, present: Sequence[bool]):
        """The tensor table of the parameters that have a gradient this step."""
        if all(present):
            return self.table
        key = tuple(present)
        if key not in self._sub:
            self._sub[key] = G.tensor_table([e for e, ok in zip(self.entries, present) if ok])
        return self._sub[key]


class Gefen(torch.optim.Optimizer):
    """Gefen (Algorithm 1) with AdamW's arguments.

    levels: codebook size k (256: 8-bit codes).  bins: histogram cells of the
    codebook refit (default 16 per level).  refit_every: refit the codebook
    every N steps (0: learn it once, from the first gradient).  periods:
    optional block size of every parameter, all groups in order (default:
    inferred from the first gradient, Algorithm 2).  four_bit: store the codes
    two per byte (default: when levels <= 16).  The compact formats (four-bit
    codes, bf16 parameters) cover blocks of 1, of p <= 8192 with p % 32 == 0
    (p % 16 == 0 for bf16 alone) and of multiples of 4096; the library
    reports any other block size as unsupported (give periods= then).
    Parameters without a gradient at a step are left untouched, as in AdamW.
    """

    def __init__(self, params, lr: float = 1e-3, betas=(0.9, 0.999), eps: float = 1e-8,
                 weight_decay: float = 1e-2, *, levels: int = 256, bins: Optional[int] = None,
                 refit_every: int = 0, periods: Optional[Sequence[int]] = None,
                 four_bit: Optional[bool] = None):
        if not 0.0 <= lr or not 0.0 <= eps or not 0.0 <= weight_decay:
            raise ValueError("lr, eps and weight_decay must be non-negative")
        if not (0.0 <= betas[0] < 1.0 and 0.0 <= betas[1] < 1.0):
            raise ValueError("betas must lie in [0, 1)")
        if not 2 <= levels <= G.GEFEN_MAX_LEVELS:
            raise ValueError(f"levels must lie in [2, {G.GEFEN_MAX_LEVELS}]")
        defaults = dict(lr=lr, betas=tuple(betas), eps=eps, weight_decay=weight_decay)
        super().__init__(params, defaults)
        self.levels = int(levels)
        self.bins = int(bins) if bins else 16 * self.levels
        if not self.levels <= self.bins <= G.GEFEN_MAX_BINS:
            raise ValueError(f"bins must lie in [levels, {G.GEFEN_MAX_BINS}]")
        self.refit_every = int(refit_every)
        self.four_bit = (self.levels <= 16) if four_bit is None else bool(four_bit)
        if self.four_bit and self.levels > 16:
            raise ValueError("four-bit codes hold at most 16 levels")
        self._given_periods = list(periods) if periods is not None else None
        for group in self.param_groups:
            for p in group["params"]:
                if not p.is_cuda or p.dtype not in (torch.float32, torch.bfloat16):
                    raise ValueError("Gefen needs CUDA fp32 or bf16 parameters (the library has no CPU path)")
            if len({p.dtype for p in group["params"]}) > 1:
                raise ValueError("the parameters of one group must share a dtype")
        G.load()  # fails loudly when the CUDA library is missing
        self._arenas: List[Optional[_Arena]] = [None] * len(self.param_groups)
        self._pending: Optional[list] = None

    # ------------------------------------------------------------ set-up
    def _first_step(self, gi: int, group, present):
        params = list(group["params"])
        A = _Arena(params, self.levels, self.bins, self.four_bit)
        self._arenas[gi] = A
        if self._pending is not None and self._pending[gi] is not None:
            self._restore(A, self._pending[gi])
            return
        if not all(present):
            raise RuntimeError("the first step needs a gradient for every parameter (it infers their blocks)")
        self._gather(A, present)
        beta1, beta2 = group["betas"]
        if self._given_periods is not None:
            # the periods list follows the parameters of all groups in order
            start = sum(len(g["params"]) for g in self.param_groups[:gi])
            periods = self._given_periods[start:start + len(params)]
        else:
            periods, iws = [], None
            for p, gv in zip(params, A.gviews):
                need = G.gefen_infer_workspace_size(p.numel())
                if iws is None or iws.numel() < need:
                    iws = G.workspace(need, p.device)
                per, _ = G.gefen_infer_blocks(gv.reshape(-1), group["eps"], workspace_buf=iws, want_scores=False)
                periods.append(per)
        A.set_periods(periods)
        # first codebook: histogram of g / block absmax, then the exact DP
        A.ws = G.gefen_step(A.table, A.theta, A.grads, A.codes, A.v, A.s, A.cb, A.cb, lr=group["lr"],
                            beta1=beta1, beta2=beta2, eps=group["eps"], weight_decay=group["weight_decay"],
                            step=1, flags=G.GEFEN_HIST_GRAD_ONLY, hist=A.hist, workspace_buf=A.ws)
        A.rws = G.gefen_refit_codebook(bins=self.bins, k=self.levels, codebook_out=A.cb, hist_in=A.hist,
                                       workspace_buf=A.rws)
        zc = int(torch.argmin(A.cb.abs()).item())  # the level nearest 0, lower index on ties
        A.codes.fill_(zc | (zc << 4) if A.four_bit else zc)

    def _gather(self, A: _Arena, present):
        src = [p.grad for p, ok in zip(A.params, present) if ok]
        dst = [g for g, ok in zip(A.gviews, present) if ok]
        if any(g.is_sparse for g in src):
            raise RuntimeError("Gefen does not take sparse gradients")
        torch._foreach_copy_(dst, src)

    # --------------------------------------------------------------- step
    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        for gi, group in enumerate(self.param_groups):
            present = [p.grad is not None for p in group["params"]]
            if not any(present):
                continue
            if self._arenas[gi] is None:
                self._first_step(gi, group, present)
            A = self._arenas[gi]
            self._gather(A, present)
            A.t += 1
            beta1, beta2 = group["betas"]
            refit = self.refit_every > 0 and A.t % self.refit_every == 0
            enc = A.cb_new if A.switch else A.cb
            if refit:
                A.hist.zero_()
            A.ws = G.gefen_step(A.table_for(present), A.theta, A.grads, A.codes, A.v, A.s, A.cb, enc,
                                lr=group["lr"], beta1=beta1, beta2=beta2, eps=group["eps"],
                                weight_decay=group["weight_decay"], step=A.t,
                                flags=A.flags | (G.GEFEN_HIST if refit else 0), hist=A.hist if refit else None,
                                workspace_buf=A.ws)
            if A.switch:
                A.cb.copy_(A.cb_new)
                A.switch = False
            if refit:
                A.rws = G.gefen_refit_codebook(bins=self.bins, k=self.levels, codebook_out=A.cb_new,
                                               hist_in=A.hist, workspace_buf=A.rws)
                A.switch = True
        return loss

    def check(self):
        """Waits for the device and raises if a step or refit gave up a
        bounded wait (GEFEN_ETIMEOUT) or failed a device-side check."""
        for A in self._arenas:
            if A is not None and A.ws is not None:
                G.gefen_step_status(A.ws)
            if A is not None and A.rws is not None:
                G.gefen_refit_status(A.rws)

    # --------------------------------------------------- checkpointing
    def state_dict(self):
        sd = super().state_dict()
        groups = []
        for A in self._arenas:
            if A is None:
                groups.append(None)
                continue
            groups.append(dict(t=A.t, periods=list(A.periods), switch=A.switch,
                               codes=A.codes.clone(), v=A.v.clone(), s=A.s.clone(),
                               cb=A.cb.clone(), cb_new=A.cb_new.clone()))
        sd["gefen"] = dict(levels=self.levels, bins=self.bins, refit_every=self.refit_every, groups=groups)
        return sd

    def load_state_dict(self, state_dict):
        state_dict = dict(state_dict)
        gst = state_dict.pop("gefen", None)
        super().load_state_dict(state_dict)
        if gst is None:
            return
        if gst["levels"] != self.levels or gst["bins"] != self.bins:
            raise ValueError("checkpoint was written with another codebook size or histogram")
        self._pending = list(gst["groups"])
        for gi, A in enumerate(self._arenas):
            if A is not None and self._pending[gi] is not None:
                self._restore(A, self._pending[gi])

    @staticmethod
    def _restore(A: _Arena, st: Dict):
        A.set_periods(st["periods"])
        A.t = int(st["t"])
        A.switch = bool(st["switch"])
        for name in ("codes", "v", "s", "cb", "cb_new"):
            src = st[name]
            dst = getattr(A, name)
            if src.numel() != dst.numel():
                raise ValueError(f"checkpoint {name} has {src.numel()} entries, expected {dst.numel()}")
            dst.copy_(src.to(dst.device))


class GefenMuon(torch.optim.Optimizer):
    """Gefen-Muon (the paper's appendix "Gefen-Muon") with Muon's arguments:
    Muon's momentum buffer kept as Gefen codes and per-block scales, Muon's
    orthogonalisation (gefen_muon_step).  Like Muon it is for matrices: a
    parameter of more than two dimensions is viewed as (dim 0, the rest); a
    vector is refused.  Blocks are inferred per matrix from its first
    gradient (Algorithm 2) unless periods are given; the codebook is learned
    once from the first gradients (Algorithm 3).  bf16_products runs the
    Newton-Schulz products on bf16 tensor cores, as Muon does.
    """

    def __init__(self, params, lr: float = 1e-3, weight_decay: float = 0.1, momentum: float = 0.95,
                 nesterov: bool = True, ns_coefficients=G.MUON_NS, eps: float = 1e-7, ns_steps: int = 5, *,
                 levels: int = 256, bins: Optional[int] = None, periods: Optional[Sequence[int]] = None,
                 bf16_products: bool = True):
        if not 0.0 <= momentum < 1.0:
            raise ValueError("momentum must lie in [0, 1)")
        defaults = dict(lr=lr, weight_decay=weight_decay, momentum=momentum, nesterov=nesterov,
                        ns_coefficients=tuple(ns_coefficients), eps=eps, ns_steps=ns_steps)
        super().__init__(params, defaults)
        self.levels = int(levels)
        self.bins = int(bins) if bins else 16 * self.levels
        self.flags = G.GEFEN_MUON_BF16_GEMM if bf16_products else 0
        self._given_periods = list(periods) if periods is not None else None
        for group in self.param_groups:
            for p in group["params"]:
                if not p.is_cuda or p.dtype != torch.float32 or p.dim() < 2 or not p.is_contiguous():
                    raise ValueError("GefenMuon needs contiguous CUDA fp32 matrices (the library has no CPU path)")
        G.load()
        self._setup = [None] * len(self.param_groups)
        self._ws = None

    @staticmethod
    def _shape(p):
        return p.shape[0], p.numel() // p.shape[0]

    def _first_step(self, gi, group):
        params = [p for p in group["params"]]
        if any(p.grad is None for p in params):
            raise RuntimeError("the first step needs a gradient for every parameter (it learns the codebook)")
        dev = params[0].device
        offs, o = [], 0
        for p in params:
            offs.append(o)
            o += (p.numel() + 63) // 64 * 64
        garena = torch.zeros(max(o, 64), dtype=torch.bfloat16, device=dev)
        for p, off in zip(params, offs):
            garena[off:off + p.numel()].copy_(p.grad.reshape(-1))
        if self._given_periods is not None:
            start = sum(len(g["params"]) for g in self.param_groups[:gi])
            periods = self._given_periods[start:start + len(params)]
        else:
            periods, iws = [], None
            for p, off in zip(params, offs):
                need = G.gefen_infer_workspace_size(p.numel())
                if iws is None or iws.numel() < need:
                    iws = G.workspace(need, dev)
                per, _ = G.gefen_infer_blocks(garena[off:off + p.numel()], 1e-8, workspace_buf=iws,
                                              want_scores=False)
                periods.append(per)
        entries, b = [], 0
        for p, off, per in zip(params, offs, periods):
            entries.append((off, p.numel(), per, b))
            b += p.numel() // per
        table = G.tensor_table(entries)
        hist = torch.zeros(self.bins, dtype=torch.int64, device=dev)
        cb = torch.empty(self.levels, dtype=torch.float32, device=dev)
        dummy = torch.zeros(max(b, 1), dtype=torch.float32, device=dev)
        G.gefen_step(table, None, garena, None, dummy, dummy, cb, cb, lr=0.0, beta1=0.0, beta2=0.0, eps=1.0,
                     weight_decay=0.0, step=1, flags=G.GEFEN_HIST_GRAD_ONLY, hist=hist)
        G.gefen_refit_codebook(bins=self.bins, k=self.levels, codebook_out=cb, hist_in=hist)
        zc = int(torch.argmin(cb.abs()).item())
        states = []
        for p, per in zip(params, periods):
            states.append(dict(period=int(per), codes=torch.full((p.numel(),), zc, dtype=torch.uint8, device=dev),
                               scale=torch.zeros(p.numel() // per, dtype=torch.float32, device=dev)))
        self._setup[gi] = dict(cb=cb, states=states)

    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        for gi, group in enumerate(self.param_groups):
            if self._setup[gi] is None:
                if all(p.grad is None for p in group["params"]):
                    continue
                self._first_step(gi, group)
            S = self._setup[gi]
            for p, st in zip(group["params"], S["states"]):
                if p.grad is None:
                    continue
                rows, cols = self._shape(p)
                g = p.grad.reshape(-1).to(torch.bfloat16).contiguous()
                self._ws = G.gefen_muon_step(rows, cols, st["period"], p.data, g, st["codes"], st["scale"],
                                             S["cb"], S["cb"], lr=group["lr"], momentum=group["momentum"],
                                             weight_decay=group["weight_decay"], eps=group["eps"],
                                             nesterov=group["nesterov"], ns_steps=group["ns_steps"],
                                             ns=group["ns_coefficients"], flags=self.flags, workspace_buf=self._ws)
        return loss
