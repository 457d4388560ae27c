"""The trainer's global gradient-norm clip applied inside the step (skew_step_scaled).

The paper's training setup (Sec. 4) and App. A Table 9 clip the global gradient norm
at 1.0 before the optimizer step. skew_step_scaled takes that step's factor gamma as a
device scalar and steps on gamma * G. These tests compare it with the oracle (whose
gscale forms gamma * G in fp64) on every tier and path, and check that gamma = 1
reproduces skew_step bit for bit.
"""
import numpy as np
import pytest
import torch

from paper_2607_19058_gb300 import skewadam as S
from paper_2607_19058_gb300 import workloads as WL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_19058_gb300 import _build
    _build.build()
    import oracle
    oracle.build()


def _harness(*a, **k):
    import parity
    return parity.Harness(*a, **k)


def _mixed_workload():
    """Every path a gradient takes: whole-row tiles with and without momentum (4096 and
    1024 wide), strip tiles of factored matrices, the router's and a vector's exact
    second moment (flat tiles), and a momentum-free vector-shaped matrix."""
    B, E, R = WL.TIER_BACKBONE, WL.TIER_EXPERT, WL.TIER_ROUTER
    specs = [WL.Spec("e300x4096", (300, 4096), E, expert=0), WL.Spec("b257x4096", (257, 4096), B),
             WL.Spec("e700x1024", (700, 1024), E, expert=1), WL.Spec("e300x1000", (300, 1000), E, expert=2),
             WL.Spec("b100x136", (100, 136), B), WL.Spec("router", (4096, 127), R),
             WL.Spec("norm", (4096,), B), WL.Spec("e1x4096", (1, 4096), E, expert=3)]
    return WL.Workload("gscale", specs, WL.HP(), "normal", steps=4)


def test_grad_scale_toy():
    """The toy set (strip and flat tiles, zero-gradient experts) with gamma = 0.37."""
    h = _harness(WL.toy())
    for t in range(1, 5):
        h.step(t, seed=5, gscale=0.37)
    h.close()


@pytest.mark.parametrize("gammas", [(0.37, 0.37, 0.37, 0.37), (1.0, 0.25, 0.8, 0.5)])
def test_grad_scale_every_path(gammas):
    """gamma constant, and gamma changing from step to step as a norm clip does."""
    h = _harness(_mixed_workload())
    assert h.opt.info(0).rowpath == 1 and h.opt.info(1).rowpath == 1 and h.opt.info(1).momentum == 1
    for t, g in enumerate(gammas, start=1):
        h.step(t, seed=3 * t, gscale=g)
    h.close()


def test_grad_scale_with_clamp_fallback():
    """eps = 1e-8 (App. A): the clamp binds, so the row-path tensors take phase B."""
    h = _harness(_mixed_workload(), hp_override=dict(eps=1e-8, lr=3e-4, weight_decay=0.05))
    for t in range(1, 4):
        h.step(t, seed=77, gscale=0.6)
    h.close()


def test_grad_scale_one_is_skew_step():
    """A pointer to 1.0f gives skew_step's step bit for bit (weights and state)."""
    wl = _mixed_workload()
    dev = torch.device("cuda")
    W = [WL.init_weight(wl, k, dev) for k in range(len(wl.specs))]
    Wb = [w.clone() for w in W]
    G = [torch.zeros_like(w) for w in W]
    hp = S.hparams(0.9, 0.999, 1e-30, 1.0, 0.1, S.POLICY_TIERED)
    a = S.SkewAdam([(W[k], G[k], s.tier) for k, s in enumerate(wl.specs)], hp)
    b = S.SkewAdam([(Wb[k], G[k], s.tier) for k, s in enumerate(wl.specs)], hp)
    one = torch.ones(1, dtype=torch.float32, device=dev)
    for t in (1, 2, 3):
        for k in range(len(wl.specs)):
            G[k].copy_(WL.grad(wl, k, t, dev))
        a.step(t, 1e-3, 11)
        b.step(t, 1e-3, 11, grad_scale=one)
        torch.cuda.synchronize()
        for k in range(len(wl.specs)):
            assert torch.equal(W[k].view(torch.int16), Wb[k].view(torch.int16)), (t, wl.specs[k].name)
        assert torch.equal(a.state, b.state), t
    a.sync_status()
    b.sync_status()
    a.close()
    b.close()


def test_grad_scale_is_not_a_learning_rate():
    """At t = 1 a router's update is sign(g) whatever gamma, so its weights do not change
    with gamma; scaling the learning rate by gamma instead changes them (Algorithm 1,
    full second moment)."""
    R = WL.TIER_ROUTER
    wl = WL.Workload("r", [WL.Spec("router", (4096, 128), R)], WL.HP(), "normal", steps=1)
    dev = torch.device("cuda")
    w0 = WL.init_weight(wl, 0, dev)
    g = WL.grad(wl, 0, 1, dev)
    hp = S.hparams(0.9, 0.999, 1e-30, 1.0, 0.0, S.POLICY_TIERED)
    out = {}
    for key, gam, lr in (("one", None, 1e-3), ("gamma", 0.37, 1e-3), ("lr", None, 0.37e-3)):
        w = w0.clone()
        o = S.SkewAdam([(w, g, R, S.F_NO_DECAY)], hp)
        gs = None if gam is None else torch.tensor([gam], dtype=torch.float32, device=dev)
        o.step(1, lr, 4, grad_scale=gs)
        o.sync_status()
        out[key] = w.view(torch.int16).clone()
        o.close()
    n = out["one"].numel()
    d_gamma = (out["one"].int() - out["gamma"].int()).abs()
    d_lr = (out["one"].int() - out["lr"].int()).abs()
    # U = sign(g) up to the rounding of the stored fp32 v: at most a few dithered weights
    # one bf16 ulp apart (the printed tolerance's 1e-4 share)
    assert int((d_gamma > 0).sum()) <= 1e-4 * n and int(d_gamma.max()) <= 1
    # a learning rate scaled by gamma shrinks every update instead
    assert int((d_lr > 0).sum()) > 0.5 * n


def test_grad_scale_fp32_tensors():
    """fp32 router and LayerNorm vectors (the paper's precision, App. A) beside bf16 matrices,
    with gamma changing from step to step."""
    h = _harness(WL.toy_fp32())
    for t, g in ((1, 0.37), (2, 0.9), (3, 1.0), (4, 0.5)):
        h.step(t, seed=13 * t, gscale=g)
    h.close()


def test_grad_scale_adafactor_comparator():
    """The Adafactor comparator's annealed beta2_t with gamma: every increment (1 - beta2_t)
    gamma^2 g^2, on the strip path (toy) and the whole-row path."""
    for wl in (WL.toy(), _mixed_workload()):
        h = _harness(wl, hp_override=dict(policy=WL.POLICY_ADAFACTOR))
        for t, g in ((1, 0.6), (2, 0.37), (3, 1.0)):
            h.step(t, seed=17 * t, gscale=g)
        h.close()
