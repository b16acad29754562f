"""Algorithm 2 at full size on the model-shaped sets: every tensor of the
Llama-3-style 1.5B set (the 128256 x 2048 tied embedding, 262,668,288
elements, included) and of the GPT-2-125M set, on the first gradient as the
bench draws it.  For every tensor the GPU's period equals the oracle's, and
every divisor's score is within the tolerance of the other inference tests
(the partition-score equation of Sec. 5.1)."""
import numpy as np
import pytest

import bench
import gpu_util as U
from paper_2606_13894_gb300 import gefen as G
from paper_2606_13894_gb300 import synth
from test_gpu_infer import SCORE_ATOL, SCORE_TOL

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

LARGEST = {"llama-1.5b": 128256 * 2048, "gpt2-125m": 50257 * 768}


@pytest.mark.parametrize("name", ["gpt2-125m", "llama-1.5b"])
def test_full_size_periods_and_scores_equal_oracle(name):
    specs = synth.CONFIGS[name]()
    offs, _ = synth.pack_offsets(specs)
    assert max(s.numel for s in specs) == LARGEST[name]
    g = synth.draw_grads(specs, bench.SEED, step=1, device="cuda")
    ref_p, ref_s = U.oracle_model_periods(name, bench.SEED, grads_host=U.bits(g))
    iws = None
    for s, o, pr, sr in zip(specs, offs, ref_p, ref_s):
        need = G.gefen_infer_workspace_size(s.numel)
        if iws is None or iws.numel() < need:
            iws = G.workspace(need, g.device)
        p, sc = G.gefen_infer_blocks(g[o:o + s.numel], bench.HP["eps"], workspace_buf=iws)
        sc = np.array(sc)
        assert p == pr, f"{s.name} ({s.numel} elements): period {p}, oracle {pr}"
        assert sc.size == sr.size
        fin = np.isfinite(sr)
        np.testing.assert_array_equal(np.isfinite(sc), fin)
        np.testing.assert_allclose(sc[fin], sr[fin], rtol=SCORE_TOL, atol=SCORE_ATOL, err_msg=s.name)
