"""Non-finite gradients: the GPU follows the oracle (the paper's step in fp64).

One NaN / +Inf / -Inf gradient element in a row-path expert matrix, a strip-path
backbone matrix with momentum, a backbone vector and the router. The factored
second moment of such a matrix becomes NaN or Inf in a row and a column, mean(R)
with it; max(V_hat, eps) then selects eps wherever V_hat is NaN (the clamp of
Algorithm 1, C's fmax), the sum of U^2 is NaN and the clip factor 1/max(1, NaN / d)
is 1. Checked over two steps (the second with finite gradients, the non-finite
state carried over):
  * every weight that is NaN or +-Inf on either side is the same bf16 on both;
  * the finite weights differ in at most 1e-4 of the elements, by one ulp;
  * state: NaN / Inf in the same places, finite entries within 1e-5 relative (the
    momentum relative to the magnitude of its terms, as in the parity harness);
  * RMS and clip factor agree (NaN with NaN).
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


def _nonfinite_bf16(b):
    return (b & 0x7F80) == 0x7F80


def _check_state(gpu, ora, where, scale=None):
    """Non-finite entries equal; finite ones within 1e-5 of the oracle, relative to the
    value or (momentum, which cancels) to `scale`, the magnitude of its terms."""
    gpu = gpu.astype(np.float64)
    ora = ora.astype(np.float64)
    nf = ~np.isfinite(ora) | ~np.isfinite(gpu)
    assert np.array_equal(gpu[nf], ora[nf], equal_nan=True), f"{where}: non-finite state differs"
    fin = ~nf
    if fin.any():
        den = np.maximum(np.abs(ora[fin]) if scale is None else np.maximum(np.abs(ora[fin]), scale[fin]), 1e-300)
        err = np.abs(gpu[fin] - ora[fin]) / den
        err[ora[fin] == 0] = np.abs(gpu[fin][ora[fin] == 0])
        assert err.max() <= 1e-5, f"{where}: state rel err {err.max():.3g}"


INJECT = [  # (tensor, flat index, value)
    (0, 3 * 4096 + 5, float("nan")),
    (1, 7 * 1000 + 11, float("inf")),
    (2, 100, float("-inf")),
    (3, 0, float("nan")),
]


def test_nonfinite_gradients_follow_the_oracle():
    import oracle as O
    import parity
    E, B, R = WL.TIER_EXPERT, WL.TIER_BACKBONE, WL.TIER_ROUTER
    specs = [WL.Spec("e256x4096", (256, 4096), E, expert=0), WL.Spec("b300x1000", (300, 1000), B),
             WL.Spec("v4096", (4096,), B), WL.Spec("router64x8", (64, 8), R)]
    wl = WL.Workload("nonfinite", specs, WL.HP(), "normal", steps=2)
    h = parity.Harness(wl)
    assert h.opt.info(0).rowpath == 1 and h.opt.info(1).rowpath == 0
    for t in (1, 2):
        h.load_grads(t)
        if t == 1:
            for k, idx, val in INJECT:
                h.G[k].view(-1)[idx] = val
        torch.cuda.synchronize()
        pre = {}
        for k in range(len(specs)):  # teacher forcing from the GPU's pre-step state
            st = h.ostate[k][0]
            gs = h._gpu_state(k)[0]
            for key in ("M", "v", "R", "C"):
                if getattr(st, key) is not None:
                    getattr(st, key)[:] = gs[key]
            pre[k] = (parity.bits16(h.W[k]), parity.bits16(h.G[k]), None if st.M is None else st.M.copy())
        h.opt.step(t, h.lr, 99)
        h.opt.sync_status()
        for k in range(len(specs)):
            w0, g, m_prev = pre[k]
            st = h.ostate[k][0]
            o = O.tensor_step(w0, g, st, k, h.ohp, t, h.lr, 99)
            where = f"{specs[k].name} step {t}"
            gw = parity.bits16(h.W[k])
            nf = _nonfinite_bf16(gw) | _nonfinite_bf16(w0)
            assert np.array_equal(gw[nf], w0[nf]), f"{where}: non-finite weights differ"
            diff = np.nonzero(gw != w0)[0]
            assert diff.size <= 1e-4 * gw.size + 1, f"{where}: {diff.size} weights differ"
            step = np.abs(gw[diff].astype(np.int32) - w0[diff].astype(np.int32))
            assert (step <= 1).all(), f"{where}: weights more than one ulp apart"
            gs = h._gpu_state(k)[0]
            for key in ("M", "v", "R", "C"):
                if getattr(st, key) is not None:
                    scale = None
                    if key == "M":  # the terms of M = b1 M_prev + (1 - b1) g
                        gd = (g.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
                        b1 = float(np.float32(h.hpd["beta1"]))
                        with np.errstate(invalid="ignore", over="ignore"):
                            scale = b1 * np.abs(m_prev.astype(np.float64)) + (1 - b1) * np.abs(gd)
                    _check_state(gs[key], getattr(st, key), f"{where} {key}", scale)
            sc = h.opt.scalars(k)
            for key in ("rms", "kappa"):
                a, b = sc[key], o[key]
                assert (np.isnan(a) and np.isnan(b)) or a == b or abs(a - b) <= 1e-6 * abs(b), \
                    f"{where}: {key} {a!r} vs oracle {b!r}"
            if t == 1 and k == 0:
                assert np.isnan(o["rms"]) and o["kappa"] == 1.0  # the NaN element makes sum(U^2) NaN
    h.close()
