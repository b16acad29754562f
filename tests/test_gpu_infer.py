"""GPU parity of gefen_infer_blocks (Algorithm 2): identical periods, and
scores within 1e-9 relative plus 1e-11 absolute of the oracle's direct sums on
the same bf16 input.  The absolute term covers the oracle's own sequential
double sums (about p * 1e-16 * |z| per block mean) and the GPU's fixed-point z
(2^-48); both matter only where adjacent block means nearly cancel."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_13894_gb300 import gefen as G
from paper_2606_13894_gb300 import synth

pytestmark = pytest.mark.gpu

SCORE_TOL = 1e-9
SCORE_ATOL = 1e-11


def _check(g: torch.Tensor, eps=1e-8):
    bits = g.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    p_ref, divs, s_ref = oracle.infer_blocks(bits, eps)
    p, s = G.gefen_infer_blocks(g.contiguous().cuda(), eps)
    assert p == p_ref
    s = np.array(s)
    assert s.size == s_ref.size
    fin = np.isfinite(s_ref)
    np.testing.assert_array_equal(np.isfinite(s), fin)
    np.testing.assert_allclose(s[fin], s_ref[fin], rtol=SCORE_TOL, atol=SCORE_ATOL)
    return p


def _bf16(a):
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16)


@pytest.mark.parametrize("rows,cols,stripe", [(48, 768, 64), (24, 512, 128), (16, 960, 40)])
def test_planted_stripes(rows, cols, stripe):
    rng = np.random.default_rng(rows + cols)
    sig = np.where((np.arange(cols) // stripe) % 2 == 0, 1e-2, 1e-3)[None, :]
    assert _check(_bf16((rng.normal(0, 1, (rows, cols)) * sig).reshape(-1))) == stripe


@pytest.mark.parametrize("n", [1, 2, 7919, 4096, 1680, 100_000, 999_983 * 2])
def test_sizes(n):
    rng = np.random.default_rng(n)
    _check(_bf16(rng.normal(0, 1e-3, n) * np.repeat(10 ** rng.uniform(-4, -2, n), 1)))


def test_zero_gradients_and_eps():
    g = np.zeros(3072, np.float32)
    g[::7] = 1e-3
    _check(_bf16(g), eps=1e-8)
    _check(_bf16(g), eps=1e-3)


@pytest.mark.parametrize("name", ["gpt2-125m", "llama-1.5b"])
def test_model_shaped_tensors(name):
    """Each distinct tensor shape of the model-shaped sets (first gradient):
    identical periods; the largest tensor is compared on a prefix of rows."""
    specs = synth.CONFIGS[name]()
    seen = set()
    for i, s in enumerate(specs):
        key = (s.shape, s.structure)
        if key in seen:
            continue
        seen.add(key)
        if s.numel > 40_000_000:
            s = synth.TensorSpec(s.name, (s.shape[0] // 64, s.shape[1]), s.structure)
        g = synth.draw_grads([s], seed=i, step=1, device="cuda")[: s.numel]
        _check(g)
