"""P8: brute force on tiny inputs.

An independent numpy fp64 restatement of Algorithm 1 (Sec. 3) that materialises
the full reconstructed second-moment matrix Vhat = R C^T / Rbar and the update U
as dense arrays, written without looking at the oracle's loops. The oracle must
agree: fp32 state and pre-rounding values to within one fp32 rounding, the
per-tensor scalars (Rbar, sum U^2, RMS, kappa) to 1e-12 relative, dithers and
bf16 outputs bit for bit (where x agrees bit for bit).
"""
import numpy as np
import pytest

import oracle as O

F32 = np.float32


def _f(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def _bf16(x):
    b = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    return ((b + 0x7FFF + ((b >> 16) & 1)) >> 16).astype(np.uint16)


def _philox(ctr, key):
    M0, M1, W0, W1 = 0xD2511F53, 0xCD9E8D57, 0x9E3779B9, 0xBB67AE85
    c0, c1, c2, c3 = ctr
    k0, k1 = key
    for r in range(10):
        p0, p1 = M0 * c0, M1 * c2
        c0, c1, c2, c3 = ((p1 >> 32) ^ c1 ^ k0) & 0xFFFFFFFF, p1 & 0xFFFFFFFF, ((p0 >> 32) ^ c3 ^ k1) & 0xFFFFFFFF, p0 & 0xFFFFFFFF
        k0, k1 = (k0 + W0) & 0xFFFFFFFF, (k1 + W1) & 0xFFFFFFFF
    return (c0, c1, c2, c3)


def _dither(seed, t, tid, numel):
    out = np.empty(numel, np.uint32)
    for e in range(numel):
        o = _philox(((e >> 3) & 0xFFFFFFFF, e >> 35, tid, t & 0xFFFFFFFF), (seed & 0xFFFFFFFF, seed >> 32))
        out[e] = (o[(e & 7) >> 1] >> (16 * (e & 1))) & 0xFFFF
    return out


class Brute:
    """Dense fp64 SkewAdam for one tensor; state stored as fp32 like the paper's memory model."""

    def __init__(self, shape, kind, momentum, decay):
        self.n, self.m = shape[0], (shape[1] if len(shape) == 2 else 1)
        self.kind, self.mom, self.decay = kind, momentum, decay
        z = lambda *s: np.zeros(s, F32)
        self.M = z(self.n, self.m) if momentum else None
        self.v = z(self.n, self.m) if kind == O.KIND_FULL else None
        self.R = z(self.n) if kind == O.KIND_FACTORED else None
        self.C = z(self.m) if kind == O.KIND_FACTORED else None

    def step(self, w_bits, g_bits, t, lr, seed, tid, b1, b2, eps, d, lam, gscale=1.0):
        G = gscale * _f(g_bits).astype(np.float64).reshape(self.n, self.m)
        Wt = _f(w_bits).astype(np.float64).reshape(self.n, self.m)
        G2 = G * G
        rbar = 0.0
        if self.kind == O.KIND_FULL:
            self.v = (b2 * self.v.astype(np.float64) + (1 - b2) * G2).astype(F32)
            V = self.v.astype(np.float64)
        else:
            self.R = (b2 * self.R.astype(np.float64) + (1 - b2) * G2.mean(axis=1)).astype(F32)
            self.C = (b2 * self.C.astype(np.float64) + (1 - b2) * G2.mean(axis=0)).astype(F32)
            rbar = float(self.R.astype(np.float64).mean())
            V = np.outer(self.R.astype(np.float64), self.C.astype(np.float64))
            V = V / rbar if rbar > 0 else np.zeros_like(V)
        D = np.sqrt(np.maximum(V, eps))
        bc1 = 1 - b1 ** t
        s2 = np.sqrt(1 - b2 ** t)
        if self.mom:
            self.M = (b1 * self.M.astype(np.float64) + (1 - b1) * G).astype(F32)
            U = (s2 / bc1) * self.M.astype(np.float64) / D
        else:
            U = s2 * G / D
        rms = np.sqrt((U * U).sum() / U.size)
        kappa = 1.0 / max(1.0, rms / d)
        lam_t = lam if self.decay else 0.0
        x = (Wt * (1 - lr * lam_t) - lr * kappa * U).astype(F32).reshape(-1)
        r = _dither(seed, t, tid, x.size)
        b = x.view(np.uint32).astype(np.uint64)
        out = ((b + r) >> 16).astype(np.uint16)
        nan = np.isnan(x)
        out[nan] = (0x7FC0 | ((b[nan] >> 16) & 0x8000)).astype(np.uint16)
        return out, x, r.astype(np.uint16), dict(rbar=rbar, sumu2=float((U * U).sum()), rms=float(rms), kappa=kappa)


CASES = [((3, 5), O.TIER_EXPERT, O.POLICY_TIERED), ((7, 1), O.TIER_EXPERT, O.POLICY_TIERED),
         ((1, 7), O.TIER_BACKBONE, O.POLICY_TIERED), ((2, 2), O.TIER_BACKBONE, O.POLICY_TIERED),
         ((9,), O.TIER_BACKBONE, O.POLICY_TIERED), ((5, 3), O.TIER_ROUTER, O.POLICY_TIERED),
         ((4, 6), O.TIER_ROUTER, O.POLICY_UNIFORM), ((6, 4), O.TIER_EXPERT, O.POLICY_EXPERT_MOMENTUM),
         ((11, 13), O.TIER_EXPERT, O.POLICY_TIERED)]


def _ulps(a, b):
    a = np.asarray(a, F32).view(np.int32).astype(np.int64)
    b = np.asarray(b, F32).view(np.int32).astype(np.int64)
    return np.abs(a - b)


@pytest.mark.parametrize("shape,tier,policy", CASES)
@pytest.mark.parametrize("eps,lr,lam,gscale", [(1e-30, 1e-3, 0.1, 1.0), (1e-8, 3e-4, 0.05, 1.0),
                                               (1e-30, 1e-3, 0.1, 0.37)])
def test_oracle_matches_brute_force(shape, tier, policy, eps, lr, lam, gscale):
    """`gscale` is the trainer's global gradient-norm clip factor of the step (Sec. 4 training
    setup, App. A Table 9): the brute force forms gscale * G and steps on it."""
    rng = np.random.default_rng(hash((shape, tier, policy, eps)) & 0xFFFF)
    b1, b2 = float(F32(0.9)), float(F32(0.999))
    eps32, lr32, lam32, d32 = float(F32(eps)), float(F32(lr)), float(F32(lam)), float(F32(0.5))
    gs32 = float(F32(gscale))
    hp = O.hparams(0.9, 0.999, eps, 0.5, lam, gscale=gscale)
    st = O.TensorState(shape, tier, policy)
    br = Brute(shape, st.kind, st.momentum, st.decay)
    numel = int(np.prod(shape))
    w = _bf16(rng.normal(0, 0.02, numel).astype(F32))
    wb = w.copy()
    seed, tid = 0xA5A5_1234_5678_9ABC, 5
    for t in range(1, 6):
        scale = [1e-3, 0.0, 1e-1, 1e-5, 1e-3][t - 1]
        g = _bf16(rng.normal(0, 1, numel).astype(F32) * F32(scale))
        if t == 5:
            g[: max(1, numel // 3)] = 0
        o = O.tensor_step(w, g, st, tid, hp, t, lr32, seed, want_x=True)
        bw, bx, brr, bs = br.step(wb, g, t, lr32, seed, tid, b1, b2, eps32, d32, lam32, gs32)
        for k in ("M", "v", "R", "C"):
            a, b = getattr(st, k), getattr(br, k)
            if a is not None:
                assert _ulps(a, b.reshape(-1)).max() <= 1, (k, t)
        for k in ("rbar", "sumu2", "rms", "kappa"):
            assert abs(o[k] - bs[k]) <= 1e-12 * max(abs(bs[k]), 1e-300), (k, t, o[k], bs[k])
        assert np.array_equal(o["r"], brr)
        assert _ulps(o["x"], bx).max() <= 1
        same = o["x"].view(np.uint32) == bx.view(np.uint32)
        assert np.array_equal(w[same], bw[same])
        # continue both from the oracle's weights so that the runs stay in lock-step
        wb = w.copy()
        for k in ("M", "v", "R", "C"):
            if getattr(st, k) is not None:
                setattr(br, k, getattr(st, k).reshape(getattr(br, k).shape).copy())
