"""Block-aligned sharding of Gefen's state over the ranks of a process group.

The paper runs Gefen under DDP, FSDP and ZeRO-3 (appendix on
distributability).  Blocks are independent in the step (Algorithm 1): a
block's v, scale, codes and parameters depend only on that block.  So each
rank owns whole blocks -- their parameters, codes, v and scale -- and steps
them with no exchange (the framework delivers each rank the gradient of the
blocks it owns, e.g. by a reduce-scatter).  A codebook refit (Algorithm 3)
needs the histogram of the whole model: each rank counts its own blocks, one
all-reduce (sum) of the u64 histogram gives every rank the same counts, and
every rank runs the same exact DP on them, which yields the same codebook bit
for bit, so nothing else is exchanged.

`partition` cuts the model's blocks into contiguous ranges of about equal
size, only at block boundaries; `RankShard` lays out one rank's part as a
tensor table of the C ABI and steps it.  All arithmetic runs in libgefen's
CUDA kernels; this module only lays out memory and sequences calls.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Callable, List, Optional, Sequence, Tuple

import torch

from . import gefen as G

ALIGN = 64  # elements between pieces in a rank's arena (16 is the library's minimum)


@dataclass(frozen=True)
class Piece:
    """Blocks [first_block, first_block + nblocks) of tensor `tensor`, whose
    blocks hold `period` elements each."""
    tensor: int
    first_block: int
    nblocks: int
    period: int

    @property
    def numel(self) -> int:
        return self.nblocks * self.period

    @property
    def first_element(self) -> int:
        return self.first_block * self.period


def partition(tensors: Sequence[Tuple[int, int]], world: int) -> List[List[Piece]]:
    """Splits tensors given as (numel, period), in order, into `world`
    contiguous ranges of the concatenated elements, each cut moved to the
    block boundary nearest to an equal share.  Returns each rank's pieces
    (possibly none); every block belongs to exactly one rank."""
    if world < 1:
        raise ValueError("world must be >= 1")
    starts, total = [], 0
    for n, p in tensors:
        if p < 1 or n < 0 or n % p:
            raise ValueError(f"period {p} does not divide a tensor of {n} elements")
        starts.append(total)
        total += n
    # cut points in global element coordinates, each on a block boundary
    cuts = [0]
    ti = 0
    for r in range(1, world):
        c = total * r // world
        while ti < len(tensors) and starts[ti] + tensors[ti][0] <= c:
            ti += 1
        if ti == len(tensors):
            b = total
        else:
            n, p = tensors[ti]
            b = starts[ti] + min(n, (c - starts[ti] + p // 2) // p * p)
        cuts.append(max(b, cuts[-1]))
    cuts.append(total)
    out: List[List[Piece]] = []
    for r in range(world):
        lo, hi = cuts[r], cuts[r + 1]
        pieces = []
        for i, (n, p) in enumerate(tensors):
            a, e = max(lo, starts[i]), min(hi, starts[i] + n)
            if a < e:
                pieces.append(Piece(i, (a - starts[i]) // p, (e - a) // p, p))
        out.append(pieces)
    return out


def local_entries(pieces: Sequence[Piece]):
    """Tensor-table entries (offset, numel, period, block_offset) of a rank's
    arena holding its pieces in order, and the arena's element and block
    counts."""
    entries, off, boff = [], 0, 0
    for pc in pieces:
        entries.append((off, pc.numel, pc.period, boff))
        off += (pc.numel + ALIGN - 1) // ALIGN * ALIGN
        boff += pc.nblocks
    return entries, max(off, ALIGN), max(boff, 1)


def all_reduce_histogram(hist: torch.Tensor, group=None) -> torch.Tensor:
    """Sums the u64 cell counts (held in an int64 tensor) of every rank in
    place: the one exchange a refit needs."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(hist, op=dist.ReduceOp.SUM, group=group)
    return hist


class RankShard:
    """One rank's part of the model: its pieces' parameters (fp32), codes, v
    and scale in a local arena, stepped by gefen_step over a local tensor
    table.  `reduce` sums a histogram over the ranks (default: an all-reduce
    on `group`).

    Steps follow the workload cadence: with refit_every = N > 0, every N-th
    step also counts x = m / s' of the rank's blocks into the histogram, the
    histogram is summed over the ranks and the exact DP refits the codebook
    (identically on every rank); the next step decodes with the old codebook
    and encodes with the new one."""

    def __init__(self, tensors: Sequence[Tuple[int, int]], rank: int, world: int, device, *,
                 levels: int = 256, bins: int = 4096, refit_every: int = 10, group=None,
                 reduce: Optional[Callable[[torch.Tensor], torch.Tensor]] = None,
                 split: Optional[Callable[[int], bool]] = None):
        self.pieces = partition(tensors, world)[rank]
        self.entries, self.numel_arena, self.nblocks = local_entries(self.pieces)
        self.table = G.tensor_table(self.entries)
        # a step makes one gefen_step call per table: with `split`, the pieces
        # whose period it accepts, then the rest (the same step, in two calls)
        if split is None:
            self.call_entries = [self.entries]
        else:
            self.call_entries = [x for x in ([e for e in self.entries if split(e[2])],
                                             [e for e in self.entries if not split(e[2])]) if x]
        self.tables = [G.tensor_table(x) for x in self.call_entries] or [self.table]
        self.device = torch.device(device)
        self.levels, self.bins, self.refit_every = levels, bins, refit_every
        self.reduce = reduce if reduce is not None else (lambda h: all_reduce_histogram(h, group))
        dev = self.device
        self.theta = torch.zeros(self.numel_arena, dtype=torch.float32, device=dev)
        self.codes = torch.zeros(self.numel_arena, dtype=torch.uint8, device=dev)
        self.v = torch.zeros(self.nblocks, dtype=torch.float32, device=dev)
        self.scale = torch.zeros(self.nblocks, dtype=torch.float32, device=dev)
        self.cb = torch.empty(levels, dtype=torch.float32, device=dev)
        self.cb_new = torch.empty(levels, dtype=torch.float32, device=dev)
        self.ws = G.workspace(max(G.gefen_step_workspace_size(t, G.GEFEN_HIST) for t in [self.table] + self.tables),
                              dev)
        self.set_refit_bins(bins)
        self.t = 0
        self.switch = False

    def set_refit_bins(self, bins: int):
        """Histogram cells of the following refits (and their DP workspace)."""
        self.bins = bins
        self.hist = torch.zeros(bins, dtype=torch.int64, device=self.device)
        self.rws = G.workspace(G.gefen_refit_workspace_size(bins, self.levels), self.device)

    @property
    def numel(self) -> int:
        return sum(pc.numel for pc in self.pieces)

    def views(self, arena: torch.Tensor):
        """Views of each piece inside a tensor laid out like this rank's arena."""
        return [arena[o:o + n] for (o, n, _, _) in self.entries]

    def gather(self, per_tensor_flat: Callable[[int], torch.Tensor], dtype, out: Optional[torch.Tensor] = None):
        """This rank's arena of a model-wide quantity: per_tensor_flat(i) is
        tensor i flattened; each piece's part is copied to its place."""
        if out is None:
            out = torch.zeros(self.numel_arena, dtype=dtype, device=self.device)
        for pc, (o, n, _, _) in zip(self.pieces, self.entries):
            out[o:o + n].copy_(per_tensor_flat(pc.tensor)[pc.first_element:pc.first_element + n])
        return out

    def init_codebook(self, grads: torch.Tensor, hp):
        """Algorithm 3 on the first gradient: every rank counts g / block
        absmax of its blocks, the counts are summed, every rank runs the DP
        (the new codebook then serves both decoding and encoding); codes start
        at the level nearest 0."""
        self.count_first_gradient(grads, hp)
        self.refit_codebook(first=True)

    def count_first_gradient(self, grads: torch.Tensor, hp):
        self.hist.zero_()
        G.gefen_step(self.table, self.theta, grads, self.codes, self.v, self.scale, self.cb, self.cb, step=1,
                     flags=G.GEFEN_HIST_GRAD_ONLY, hist=self.hist, workspace_buf=self.ws, **hp)

    def step(self, grads: torch.Tensor, hp, stream=None) -> bool:
        """One step of this rank's blocks (and, on a refit step, the summed
        histogram and the DP); returns whether it was a refit step."""
        refit = self.step_local(grads, hp, stream)
        if refit:
            self.refit_codebook(stream=stream)
        return refit

    def step_local(self, grads: torch.Tensor, hp, stream=None,
                   after_call: Optional[Callable[[int], None]] = None) -> bool:
        """The step of this rank's blocks alone; on a refit step it also
        counts the rank's x = m / s' into self.hist (zeroed first).
        after_call(i) runs after the i-th gefen_step call is enqueued."""
        self.t += 1
        refit = self.refit_every > 0 and self.t % self.refit_every == 0
        enc = self.cb_new if self.switch else self.cb
        if refit:
            self.hist.zero_()
        for i, tb in enumerate(self.tables):
            G.gefen_step(tb, self.theta, grads, self.codes, self.v, self.scale, self.cb, enc, step=self.t,
                         flags=G.GEFEN_HIST if refit else 0, hist=self.hist if refit else None,
                         workspace_buf=self.ws, stream=stream, **hp)
            if after_call is not None:
                after_call(i)
        if self.switch:
            self.cb.copy_(self.cb_new)
            self.switch = False
        return refit

    def refit_codebook(self, *, reduce: bool = True, first: bool = False, stream=None):
        """Sums self.hist over the ranks (unless reduce=False: the caller has
        summed it) and runs the exact DP.  The first codebook replaces cb at
        once and resets the codes; a periodic one is used for encoding from
        the next step on."""
        if reduce:
            self.reduce(self.hist)
        out = self.cb if first else self.cb_new
        G.gefen_refit_codebook(bins=self.bins, k=self.levels, codebook_out=out, hist_in=self.hist,
                               workspace_buf=self.rws, stream=stream)
        if first:
            self.codes.fill_(int(torch.argmin(self.cb.abs()).item()))
        else:
            self.switch = True
