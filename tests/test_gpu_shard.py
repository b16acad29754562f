"""The sharded step (paper_2606_13894_gb300/shard.py) on one GPU: the model's
blocks split over two ranks' arenas, each stepped by its own gefen_step calls,
the two histograms summed as the all-reduce sums them, and the DP run by both.
Against the unsharded run of the same model: histograms, codebooks and every
block's parameters, codes, v and scale equal bit for bit (a block's step reads
only that block), over the workload cadence -- first codebook, refit every
second step, the codebook switch after it."""
import pytest
import torch

from paper_2606_13894_gb300 import shard

pytestmark = pytest.mark.gpu

# one tensor per kernel class: blocks of 1, of 100 (generic), of 64, 384 and
# 4096 (streamed 4096 tiles), 8192 (8192 tiles), 2^17 (big blocks)
TENSORS = [(1000 * 64, 1), (100 * 300, 100), (64 * 2000, 64), (384 * 500, 384), (4096 * 64, 4096),
           (8192 * 16, 8192), (1 << 19, 1 << 17)]
HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


def _global(seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    theta = [torch.randn(n, device="cuda", generator=g) * 0.02 for n, _ in TENSORS]
    grads = []
    for _ in range(6):
        gs = []
        for n, p in TENSORS:
            sig = torch.pow(10.0, torch.empty(n // p, device="cuda").uniform_(-4, -2, generator=g))
            gs.append((torch.randn(n, device="cuda", generator=g) * sig.repeat_interleave(p)).to(torch.bfloat16))
        grads.append(gs)
    return theta, grads


def _fill(sh, per_tensor, dtype):
    out = torch.zeros(sh.numel_arena, dtype=dtype, device="cuda")
    for pc, (o, n, _, _) in zip(sh.pieces, sh.entries):
        out[o:o + n] = per_tensor[pc.tensor][pc.first_element:pc.first_element + n]
    return out


def test_two_shards_equal_the_unsharded_run():
    theta, grads = _global(3)
    whole = shard.RankShard(TENSORS, 0, 1, "cuda", levels=256, bins=4096, refit_every=2, reduce=lambda h: h)
    ranks = [shard.RankShard(TENSORS, r, 2, "cuda", levels=256, bins=4096, refit_every=2) for r in range(2)]
    assert all(r.pieces for r in ranks)
    assert sum(r.numel for r in ranks) == whole.numel
    for sh in [whole] + ranks:
        sh.theta.copy_(_fill(sh, theta, torch.float32))

    def summed():
        h = ranks[0].hist + ranks[1].hist
        for r in ranks:
            r.hist.copy_(h)
        for r in ranks:
            r.refit_codebook(reduce=False, first=first)

    whole.init_codebook(_fill(whole, grads[0], torch.bfloat16), HP)
    for r in ranks:
        r.count_first_gradient(_fill(r, grads[0], torch.bfloat16), HP)
    first = True
    summed()
    first = False
    for r in ranks:
        assert torch.equal(r.hist, whole.hist) and torch.equal(r.cb, whole.cb)
    refits = 0
    for t in range(1, 6):
        refit = whole.step(_fill(whole, grads[t], torch.bfloat16), HP)
        got = [r.step_local(_fill(r, grads[t], torch.bfloat16), HP) for r in ranks]
        assert got == [refit, refit]
        if refit:
            refits += 1
            summed()
            for r in ranks:
                assert torch.equal(r.hist, whole.hist) and torch.equal(r.cb_new, whole.cb_new)
    assert refits == 2
    torch.cuda.synchronize()
    for r in ranks:
        for pc, (o, n, _, bo) in zip(r.pieces, r.entries):
            wo, _, _, wbo = whole.entries[pc.tensor]
            a = wo + pc.first_element
            b = wbo + pc.first_block
            assert torch.equal(r.theta[o:o + n], whole.theta[a:a + n]), pc
            assert torch.equal(r.codes[o:o + n], whole.codes[a:a + n]), pc
            assert torch.equal(r.v[bo:bo + pc.nblocks], whole.v[b:b + pc.nblocks]), pc
            assert torch.equal(r.scale[bo:bo + pc.nblocks], whole.scale[b:b + pc.nblocks]), pc
