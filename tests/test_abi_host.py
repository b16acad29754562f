"""Host-side checks of the C ABI: the library builds and loads, exports every
function include/gefen.h declares, and rejects bad arguments on the host
(before any device work), so none of these calls needs a GPU.

The calls pass fake device pointers and rely on the host-side validation
returning first.  They run only in a process that sees no CUDA device
(tests/test_abi_host_isolated.py starts one), so that a validation regression
ends in the library's device check instead of a launch on a bogus address."""
import ctypes
import os
import re

import pytest

from paper_2606_13894_gb300 import gefen as G

pytestmark = pytest.mark.skipif(os.environ.get("CUDA_VISIBLE_DEVICES") != "",
                                reason="runs in a child process with no visible CUDA device")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gefen.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gefen_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported():
    lib = G.load()
    names = _declared()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(G.EXPORTS)


def test_status_strings():
    assert G.gefen_status_string(0) == "ok"
    assert "invalid" in G.gefen_status_string(1)
    assert G.gefen_status_string(99) == "unknown status"


def _table(entries):
    return G.tensor_table(entries)


def test_step_workspace_sizes_follow_the_plan():
    # small blocks need only the 256-byte status header; big blocks need
    # per-chunk partials as well
    assert G.gefen_step_workspace_size(_table([(0, 4096, 64, 0)])) == 256
    big = G.gefen_step_workspace_size(_table([(0, 1 << 20, 1 << 20, 0)]))
    assert big > 0
    hist = G.gefen_step_workspace_size(_table([(0, 4096, 64, 0)]), G.GEFEN_HIST)
    assert hist >= 4096 * 4
    # invalid tables report 0
    assert G.gefen_step_workspace_size(_table([(0, 100, 7, 0)])) == 0
    assert G.gefen_step_workspace_size(_table([(8, 64, 64, 0)])) == 0


def test_refit_and_infer_workspace_sizes():
    assert G.gefen_refit_workspace_size(4096, 256) > 257 * 4097 * 12
    assert G.gefen_refit_workspace_size(0, 256) == 0
    assert G.gefen_refit_workspace_size(65537, 256) == 0
    assert G.gefen_refit_workspace_size(4096, 1) == 0
    assert G.gefen_infer_workspace_size(1000) > 1001 * 16
    assert G.gefen_infer_workspace_size(0) == 0


def _hp(**kw):
    d = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0, step=1, flags=0)
    d.update(kw)
    return G.gefen_hparams_t(d["lr"], d["beta1"], d["beta2"], d["eps"], d["weight_decay"], d["step"], d["flags"])


FAKE = ctypes.c_void_p(1 << 20)  # 16-byte aligned, never dereferenced on these paths


def _step(table, hp=None, k=256, params=FAKE, grads=FAKE, ws=None, ws_bytes=0, hist=None, bins=0):
    arr, n = table
    return G.load().gefen_step(arr, n, params, grads, FAKE, FAKE, FAKE, FAKE, FAKE, k, hp or _hp(),
                               hist, bins, ws, ws_bytes, None)


@pytest.mark.parametrize("entries", [
    [(0, 100, 7, 0)],                 # period does not divide numel
    [(8, 64, 64, 0)],                 # offset not a multiple of 16
    [(0, 64, 0, 0)],                  # period 0
    [(0, 64, 16, 0), (32, 64, 16, 8)],  # overlapping element ranges
    [(0, 64, 16, 0), (64, 64, 16, 2)],  # overlapping block ranges
    [(-16, 64, 16, 0)],               # negative offset
])
def test_step_rejects_bad_tables(entries):
    assert _step(_table(entries)) == G.GEFEN_EINVAL


def test_step_rejects_bad_scalars_and_pointers():
    t = _table([(0, 64, 16, 0)])
    assert _step(t, k=1) == G.GEFEN_EINVAL
    assert _step(t, k=257) == G.GEFEN_EINVAL
    assert _step(t, hp=_hp(step=0)) == G.GEFEN_EINVAL
    assert _step(t, hp=_hp(beta1=1.0)) == G.GEFEN_EINVAL
    assert _step(t, hp=_hp(beta2=-0.1)) == G.GEFEN_EINVAL
    assert _step(t, hp=_hp(eps=float("nan"))) == G.GEFEN_EINVAL
    assert _step(t, hp=_hp(flags=3)) == G.GEFEN_EINVAL
    assert _step(t, hp=_hp(flags=16)) == G.GEFEN_EINVAL
    assert _step(t, params=None) == G.GEFEN_EINVAL
    assert _step(t, params=ctypes.c_void_p((1 << 20) + 4)) == G.GEFEN_EINVAL  # misaligned
    assert _step(t, hp=_hp(flags=G.GEFEN_HIST)) == G.GEFEN_EINVAL             # hist missing
    assert _step(t, hp=_hp(flags=G.GEFEN_HIST), hist=FAKE, bins=70000) == G.GEFEN_EINVAL
    big = _table([(0, 1 << 20, 1 << 20, 0)])
    assert _step(big) == G.GEFEN_ENOMEM  # scratch needed but none given
    assert _step(t) == G.GEFEN_ENOMEM    # the status header is always needed
    assert _step(t, ws=ctypes.c_void_p((1 << 20) + 64), ws_bytes=4096) == G.GEFEN_EINVAL  # misaligned


def test_refit_and_infer_reject_bad_arguments():
    L = G.load()
    P = FAKE
    assert L.gefen_refit_codebook(None, 0, None, 4096, 256, P, None, None, None, P, 1 << 30, None) == G.GEFEN_EINVAL
    assert L.gefen_refit_codebook(P, 10, None, 4096, 1, P, None, None, None, P, 1 << 30, None) == G.GEFEN_EINVAL
    assert L.gefen_refit_codebook(P, 10, None, 0, 256, P, None, None, None, P, 1 << 30, None) == G.GEFEN_EINVAL
    assert L.gefen_refit_codebook(P, 10, None, 4096, 256, P, None, None, None, P, 16, None) == G.GEFEN_ENOMEM
    per = ctypes.c_int64(0)
    assert L.gefen_infer_blocks(P, 0, 1e-8, ctypes.byref(per), None, 0, None, P, 1 << 30, None) == G.GEFEN_EINVAL
    assert L.gefen_infer_blocks(P, 64, 0.0, ctypes.byref(per), None, 0, None, P, 1 << 30, None) == G.GEFEN_EINVAL
    assert L.gefen_infer_blocks(P, 64, 1e-8, None, None, 0, None, P, 1 << 30, None) == G.GEFEN_EINVAL
    assert L.gefen_infer_blocks(P, 64, 1e-8, ctypes.byref(per), None, 0, None, P, 8, None) == G.GEFEN_ENOMEM


def test_storage_format_checks():
    t = _table([(0, 64 * 4, 64, 0)])
    ws = ctypes.c_void_p(1 << 21)
    # two codes per byte: at most 16 levels, offsets on 32 elements
    assert _step(t, hp=_hp(flags=G.GEFEN_CODES_4BIT), k=256, ws=ws, ws_bytes=1 << 20) == G.GEFEN_EINVAL
    assert _step(_table([(16, 64 * 4, 64, 0)]), hp=_hp(flags=G.GEFEN_CODES_4BIT), k=16, ws=ws,
                 ws_bytes=1 << 20) == G.GEFEN_EINVAL
    # a shape outside the kernels that store these formats
    for f in (G.GEFEN_CODES_4BIT, G.GEFEN_PARAMS_BF16):
        assert _step(_table([(0, 3 * 100, 3, 0)]), hp=_hp(flags=f), k=16, ws=ws, ws_bytes=1 << 20) == \
            G.GEFEN_EUNSUPPORTED
    # 4-bit codes need p % 32 == 0 on the streamed tiles
    assert _step(_table([(0, 48 * 10, 48, 0)]), hp=_hp(flags=G.GEFEN_CODES_4BIT), k=16, ws=ws,
                 ws_bytes=1 << 20) == G.GEFEN_EUNSUPPORTED
    # histograms above the in-kernel cells
    assert _step(t, hp=_hp(flags=G.GEFEN_PARAMS_BF16 | G.GEFEN_HIST), k=16, ws=ws, ws_bytes=1 << 30,
                 hist=FAKE, bins=8192) == G.GEFEN_EUNSUPPORTED


def test_muon_rejects_bad_arguments():
    L = G.load()
    hp = G.gefen_muon_hparams_t(1e-3, 0.95, 0.1, 1e-7, 1, 5, 3.4445, -4.775, 2.0315, 0)
    P = FAKE
    big = 1 << 30
    assert L.gefen_muon_step(0, 8, 1, P, P, P, P, P, P, 16, hp, P, big, None) == G.GEFEN_EINVAL
    assert L.gefen_muon_step(4, 8, 3, P, P, P, P, P, P, 16, hp, P, big, None) == G.GEFEN_EINVAL  # 3 does not divide 32
    assert L.gefen_muon_step(4, 8, 8, P, P, P, P, P, P, 1, hp, P, big, None) == G.GEFEN_EINVAL
    bad = G.gefen_muon_hparams_t(1e-3, 1.0, 0.1, 1e-7, 1, 5, 3.4445, -4.775, 2.0315, 0)
    assert L.gefen_muon_step(4, 8, 8, P, P, P, P, P, P, 16, bad, P, big, None) == G.GEFEN_EINVAL
    badf = G.gefen_muon_hparams_t(1e-3, 0.9, 0.1, 1e-7, 1, 5, 3.4445, -4.775, 2.0315, 4)
    assert L.gefen_muon_step(4, 8, 8, P, P, P, P, P, P, 16, badf, P, big, None) == G.GEFEN_EINVAL
    assert L.gefen_muon_step(4, 8, 8, P, P, P, P, P, P, 16, hp, P, 64, None) == G.GEFEN_ENOMEM
    assert G.gefen_muon_workspace_size(4, 8, 3) == 0
    assert G.gefen_muon_workspace_size(64, 256, 64) > 2 * 64 * 256 * 4
