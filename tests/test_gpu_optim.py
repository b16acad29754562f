"""The torch.optim wrapper (paper_2606_13894_gb300.optim.Gefen): each of its
steps equals the oracle's step from the wrapper's own pre-step state (right
hyper-parameters, step count, codebook switch after a refit), a checkpoint
resumes bit for bit, and it trains a small regression."""
import numpy as np
import pytest
import torch

import gpu_util as U
from paper_2606_13894_gb300.optim import Gefen

pytestmark = pytest.mark.gpu


def _model(seed=0):
    torch.manual_seed(seed)
    return torch.nn.Sequential(torch.nn.Linear(64, 256), torch.nn.ReLU(), torch.nn.Linear(256, 32)).cuda()


def _batch(i):
    g = torch.Generator(device="cuda").manual_seed(1000 + i)
    x = torch.randn(128, 64, device="cuda", generator=g)
    y = torch.randn(128, 32, device="cuda", generator=g)
    return x, y


def _backward(model, i):
    x, y = _batch(i)
    model.zero_grad(set_to_none=True)
    loss = torch.nn.functional.mse_loss(model(x), y)
    loss.backward()
    return loss


class _View:
    """The comparison helpers' arena interface over the wrapper's arena."""

    def __init__(self, A):
        self.entries, self.NB = A.entries, A.v.numel()


def test_each_wrapper_step_matches_the_oracle():
    model = _model()
    hp = dict(lr=3e-3, betas=(0.9, 0.99), eps=1e-8, weight_decay=0.05)
    opt = Gefen(model.parameters(), **hp, refit_every=3)
    ohp = dict(lr=hp["lr"], beta1=hp["betas"][0], beta2=hp["betas"][1], eps=hp["eps"], weight_decay=hp["weight_decay"])
    for i in range(8):
        _backward(model, i)
        A = opt._arenas[0]
        if A is None:  # the first step sets up blocks and the first codebook
            opt.step()
            A = opt._arenas[0]
            assert A.t == 1 and all(p.data.data_ptr() >= A.theta.data_ptr() for p in model.parameters())
            continue
        pre = (A.theta.cpu().numpy().copy(), A.codes.cpu().numpy().copy(), A.v.cpu().numpy().copy(),
               A.s.cpu().numpy().copy())
        dec = A.cb.cpu().numpy().copy()
        enc = (A.cb_new if A.switch else A.cb).cpu().numpy().copy()
        opt.step()
        gbits = U.bits(A.grads)
        got = (A.theta.cpu().numpy(), A.codes.cpu().numpy(), A.v.cpu().numpy(), A.s.cpu().numpy())
        V = _View(A)
        th, cd, vv, ss, _ = U.oracle_step(V, pre, gbits, dec, enc, A.t, ohp)
        assert U.theta_err(got[0], th, ohp["lr"]) <= U.THETA_TOL, i
        assert U.rel_err(got[2], vv) <= U.STATE_TOL, i
        M = U.summand_scale(V, pre, gbits, dec, ohp["beta1"])
        assert U.scale_ok(got[3], ss, M)[0], i
        assert U.code_flips_ok(V, pre, gbits, dec, enc, got[1], cd, ohp, M)[0], i
    opt.check()


def test_checkpoint_resumes_bit_for_bit():
    m1 = _model(1)
    o1 = Gefen(m1.parameters(), lr=2e-3, refit_every=2)
    for i in range(5):
        _backward(m1, i)
        o1.step()
    sd_m, sd_o = m1.state_dict(), o1.state_dict()
    m2 = _model(2)
    m2.load_state_dict(sd_m)
    o2 = Gefen(m2.parameters(), lr=2e-3, refit_every=2)
    o2.load_state_dict(sd_o)
    for i in range(5, 9):
        _backward(m1, i)
        o1.step()
        _backward(m2, i)
        o2.step()
    for a, b in zip(m1.parameters(), m2.parameters()):
        assert torch.equal(a, b)


def test_trains_a_regression():
    torch.manual_seed(3)
    w_true = torch.randn(64, 8, device="cuda")
    model = torch.nn.Linear(64, 8, bias=False).cuda()
    opt = Gefen(model.parameters(), lr=3e-2, weight_decay=0.0, refit_every=10)
    losses = []
    for i in range(60):
        g = torch.Generator(device="cuda").manual_seed(i)
        x = torch.randn(256, 64, device="cuda", generator=g)
        model.zero_grad(set_to_none=True)
        loss = torch.nn.functional.mse_loss(model(x), x @ w_true)
        loss.backward()
        opt.step()
        losses.append(float(loss.detach()))
    assert losses[-1] < 0.1 * losses[0]


def test_parameters_without_grad_are_untouched():
    model = _model(4)
    opt = Gefen(model.parameters(), lr=1e-2)
    _backward(model, 0)
    opt.step()
    frozen = model[2].weight.detach().clone()
    model[2].weight.requires_grad_(False)
    x, y = _batch(1)
    model.zero_grad(set_to_none=True)
    torch.nn.functional.mse_loss(model(x), y).backward()
    assert model[2].weight.grad is None
    opt.step()
    assert torch.equal(model[2].weight, frozen)


@pytest.mark.parametrize("dtype,levels", [(torch.float32, 16), (torch.bfloat16, 256), (torch.bfloat16, 16)])
def test_wrapper_storage_formats_match_the_oracle(dtype, levels):
    """Four-bit codes (levels <= 16) and bf16 parameters through the wrapper,
    each step against the oracle (codes unpacked, bf16 widened)."""
    import test_gpu_formats as F
    model = _model(5).to(dtype)
    hp = dict(lr=3e-3, betas=(0.9, 0.99), eps=1e-8, weight_decay=0.05)
    opt = Gefen(model.parameters(), **hp, levels=levels, refit_every=3)
    ohp = dict(lr=hp["lr"], beta1=hp["betas"][0], beta2=hp["betas"][1], eps=hp["eps"], weight_decay=hp["weight_decay"])
    c4 = levels <= 16
    for i in range(6):
        x, y = _batch(i)
        model.zero_grad(set_to_none=True)
        torch.nn.functional.mse_loss(model(x.to(dtype)).float(), y).backward()
        A = opt._arenas[0]
        if A is None:
            opt.step()
            continue
        n = A.total
        pre = (A.theta.float().cpu().numpy().copy(),
               F.unpack4(A.codes.cpu().numpy(), n) if c4 else A.codes.cpu().numpy().copy(),
               A.v.cpu().numpy().copy(), A.s.cpu().numpy().copy())
        dec = A.cb.cpu().numpy().copy()
        enc = (A.cb_new if A.switch else A.cb).cpu().numpy().copy()
        opt.step()
        gbits = U.bits(A.grads)
        V = _View(A)
        th, cd, vv, ss, _ = U.oracle_step(V, pre, gbits, dec, enc, A.t, ohp)
        got_th = A.theta.float().cpu().numpy()
        live = np.concatenate([np.arange(o, o + m) for (o, m, _, _) in A.entries])
        if dtype == torch.bfloat16:
            ref = th[live].astype(np.float64)
            tol = 0.5 * F.bf16_ulp(ref) * (1 + 2 ** -10) + U.THETA_TOL * np.maximum(np.abs(ref), ohp["lr"])
            assert not (np.abs(got_th[live] - ref) > tol).any(), i
        else:
            assert U.theta_err(got_th, th, ohp["lr"]) <= U.THETA_TOL, i
        assert U.rel_err(A.v.cpu().numpy(), vv) <= U.STATE_TOL, i
        got_cd = F.unpack4(A.codes.cpu().numpy(), n) if c4 else A.codes.cpu().numpy()
        M = U.summand_scale(V, pre, gbits, dec, ohp["beta1"])
        assert U.code_flips_ok(V, pre, gbits, dec, enc, got_cd, cd, ohp, M)[0], i
    opt.check()


@pytest.mark.parametrize("bf16_products", [False, True])
def test_gefen_muon_wrapper_steps_match_the_oracle(bf16_products):
    """GefenMuon on the matrices of a small MLP: every step against the
    Gefen-Muon oracle from the wrapper's own pre-step state."""
    import math
    from oracle import muon as OM
    from paper_2606_13894_gb300.optim import GefenMuon
    torch.manual_seed(6)
    model = torch.nn.Sequential(torch.nn.Linear(64, 256, bias=False), torch.nn.ReLU(),
                                torch.nn.Linear(256, 32, bias=False)).cuda()
    hp = dict(lr=2e-2, weight_decay=0.1, momentum=0.9)
    opt = GefenMuon(model.parameters(), **hp, bf16_products=bf16_products)
    tolx = 6e-2 if bf16_products else 2e-4
    for i in range(5):
        _backward(model, i)
        if opt._setup[0] is None:
            opt.step()
            continue
        S = opt._setup[0]
        cb = S["cb"].cpu().numpy()
        pres = []
        for p, st in zip(model.parameters(), S["states"]):
            pres.append((p.detach().reshape(-1).cpu().numpy().copy(), st["codes"].cpu().numpy().copy(),
                         st["scale"].cpu().numpy().copy(), U.bits(p.grad.reshape(-1).to(torch.bfloat16))))
        opt.step()
        for (th0, cd0, s0, gbits), p, st in zip(pres, model.parameters(), S["states"]):
            rows, cols = p.shape[0], p.numel() // p.shape[0]
            th, cd, ss = th0.copy(), cd0.copy(), s0.copy()
            X = OM.muon_step(th, gbits, cd, ss, cb, cb, rows=rows, cols=cols, period=st["period"], **hp)
            adj = hp["lr"] * math.sqrt(max(1.0, rows / cols))
            tol = adj * tolx * np.abs(X).max() + 1e-5 * np.maximum(np.abs(th.astype(np.float64)), hp["lr"])
            got = p.detach().reshape(-1).cpu().numpy().astype(np.float64)
            assert np.all(np.abs(got - th) <= tol), i
            V = _View(type("A", (), {"entries": [(0, p.numel(), st["period"], 0)], "v": st["scale"]})())
            pre = (th0, cd0, np.zeros(1, np.float32), s0)
            Mb = U.summand_scale(V, pre, gbits, cb, hp["momentum"])
            assert U.scale_ok(st["scale"].cpu().numpy(), ss, Mb)[0], i
            assert U.code_flips_ok(V, pre, gbits, cb, cb, st["codes"].cpu().numpy(), cd,
                                   dict(beta1=hp["momentum"]), Mb)[0], i
