"""GPU parity on numerically extreme inputs (the Sec. 3 dithered write-back and Algorithm 1
at the edges of fp32 / bf16):
  * bf16-subnormal weights whose update is zero, so x stays subnormal and is rounded by
    the dither on its subnormal bit pattern (no flush to zero on either side);
  * gradients of about 1e-20, whose squares and moving-average increments lie among the
    fp32 subnormals;
  * x pushed just past the largest finite bf16 value, so that the dithered rounding
    carries to +-Inf, as stochastic rounding does.
"""
import numpy as np
import pytest
import torch

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


def _paths_workload(name):
    """A tensor on each path: whole-row tiles (4096 wide), strip tiles, the router's and a
    backbone vector's exact second moment (flat tiles), a momentum row-path matrix."""
    B, E, R = WL.TIER_BACKBONE, WL.TIER_EXPERT, WL.TIER_ROUTER
    specs = [WL.Spec("e200x4096", (200, 4096), E, expert=0), WL.Spec("e100x136", (100, 136), E, expert=1),
             WL.Spec("router", (512, 64), R), WL.Spec("norm", (4096,), B), WL.Spec("b64x4096", (64, 4096), B)]
    return WL.Workload(name, specs, WL.HP(), "normal", steps=2)


def _bits_to_bf16(bits: np.ndarray, like: torch.Tensor) -> torch.Tensor:
    return torch.from_numpy(bits.astype(np.uint16).view(np.int16)).to(like.device).view(torch.bfloat16).view(like.shape)


def test_subnormal_weights_keep_their_dithered_rounding():
    """Weights among the bf16 subnormals, gradient zero on every other row (update 0 there,
    x = w (1 - lr*lambda) stays subnormal) and N(0, 1e-3^2) on the rest."""
    h = _harness(_paths_workload("subnormal"))
    rng = np.random.default_rng(5)
    for k, w in enumerate(h.W):
        n = w.numel()
        mant = rng.integers(1, 0x80, n)                      # exponent field 0, mantissa != 0
        sign = rng.integers(0, 2, n) << 15
        w.copy_(_bits_to_bf16(sign | mant, w))
    for t in (1, 2):
        for k, g in enumerate(h.G):
            gg = WL.grad(h.wl, k, t, g.device).float()
            if gg.dim() == 2:
                gg[::2] = 0
            else:
                gg[::2] = 0
            g.copy_(gg.to(torch.bfloat16))
        h.step(t, seed=t, grads_loaded=True)
    # the weights of the zero-gradient rows are still subnormal after the steps
    w0 = h.W[0].view(torch.int16)[::2].int() & 0x7FFF
    assert int((w0 < 0x80).sum()) > 0.9 * w0.numel()
    h.close()


def test_gradients_in_the_fp32_subnormal_range():
    """G ~ N(0, (1e-20)^2): g^2 ~ 1e-40 and (1 - beta2) g^2 ~ 1e-43 are fp32 subnormals;
    at eps = 1e-30 the clamp binds (row-path tensors take phase B)."""
    h = _harness(_paths_workload("tiny_grads"))
    for t in (1, 2):
        for k, g in enumerate(h.G):
            g.copy_((WL.grad(h.wl, k, t, g.device).float() * 1e-17).to(torch.bfloat16))
        h.step(t, seed=9 + t, grads_loaded=True)
    h.close()


def test_dithered_rounding_carries_to_infinity():
    """Router weights at +-(largest bf16), gradients pushing them outward and a learning
    rate (6e35) that moves x a fraction of a bf16 ulp past the largest finite value: the
    dither carries part of them to +-Inf, the same elements on both sides."""
    R = WL.TIER_ROUTER
    wl = WL.Workload("carry", [WL.Spec("router", (256, 128), R)], WL.HP(lr=6e35), "normal", steps=1)
    h = _harness(wl)
    w = h.W[0]
    n = w.numel()
    sign = (np.arange(n) % 2).astype(np.int64) << 15
    w.copy_(_bits_to_bf16(sign | 0x7F7F, w))
    gg = torch.rand(n, device=w.device) * 1e-3 + 1e-4
    gg = torch.where(torch.from_numpy(sign != 0).to(w.device), gg, -gg)   # outward: U opposite to the weight's sign
    h.G[0].copy_(gg.view(w.shape).to(torch.bfloat16))
    h.step(1, seed=21, grads_loaded=True)
    bits = h.W[0].view(torch.int16).int() & 0xFFFF
    n_inf = int(((bits == 0x7F80) | (bits == 0xFF80)).sum())
    assert 0.1 * n < n_inf < 0.9 * n, n_inf
    h.close()
