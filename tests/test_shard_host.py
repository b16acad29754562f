"""Block-aligned partition of the model over ranks (paper_2606_13894_gb300/
shard.py): every block belongs to exactly one rank, cuts fall only on block
boundaries, and each rank's share is within one block of an equal share."""
import numpy as np
import pytest

from paper_2606_13894_gb300 import shard
from paper_2606_13894_gb300 import synth


def _check(tensors, world):
    parts = shard.partition(tensors, world)
    assert len(parts) == world
    total = sum(n for n, _ in tensors)
    seen = {i: [] for i in range(len(tensors))}
    prev_end = (0, 0)  # ranks hold consecutive ranges in model order
    for pieces in parts:
        for pc in pieces:
            n, p = tensors[pc.tensor]
            assert pc.period == p and pc.nblocks >= 1
            assert 0 <= pc.first_block and (pc.first_block + pc.nblocks) * p <= n
            seen[pc.tensor].append((pc.first_block, pc.first_block + pc.nblocks))
            assert (pc.tensor, pc.first_block) >= prev_end
            prev_end = (pc.tensor, pc.first_block + pc.nblocks)
    for i, (n, p) in enumerate(tensors):
        rs = sorted(seen[i])
        if n == 0:
            assert rs == []
            continue
        # the pieces of a tensor tile its blocks exactly once
        assert rs[0][0] == 0 and rs[-1][1] == n // p
        assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
    # balance: each rank's share is within a block of the equal share
    biggest = max((p for n, p in tensors if n), default=0)
    for pieces in parts:
        got = sum(pc.numel for pc in pieces)
        assert abs(got - total / world) <= biggest
    return parts


@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
def test_random_tables(world):
    rng = np.random.default_rng(world)
    for _ in range(50):
        tensors = []
        for _ in range(int(rng.integers(1, 12))):
            p = int(rng.choice([1, 3, 16, 64, 100, 4096]))
            tensors.append((p * int(rng.integers(0, 300)), p))
        _check(tensors, world)


def test_model_shaped_set_and_a_single_huge_block():
    specs = synth.gpt2_125m_set()
    tensors = [(s.numel, s.cols if len(s.shape) > 1 else s.numel) for s in specs]
    parts = _check(tensors, 8)
    assert all(parts)
    # one tensor that is one block cannot be cut: one rank takes it whole
    parts = shard.partition([(1 << 20, 1 << 20)], 4)
    assert sum(len(p) for p in parts) == 1 and sum(pc.numel for p in parts for pc in p) == 1 << 20


def test_local_entries_align_pieces():
    pieces = [shard.Piece(0, 2, 3, 7), shard.Piece(1, 0, 5, 64)]
    entries, n, nb = shard.local_entries(pieces)
    assert entries == [(0, 21, 7, 0), (64, 320, 64, 3)]
    assert n == 384 and nb == 8
