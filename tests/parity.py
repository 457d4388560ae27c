"""Parity harness: libskewadam (CUDA, through the C ABI) against the CPU oracle.

Per step and per checked tensor, with teacher forcing: the oracle starts from
the GPU's pre-step weights and state, takes the same gradient, and the two
post-step results are compared with the acceptance bars of the method:
  * fp32 state (R, C, v, M): max relative error <= 1e-5. R, C and v are sums
    of non-negative terms; the momentum M = b1 M + (1-b1) g is a difference
    when the terms have opposite signs, and the relative error of a cancelling
    sum evaluated in fp32 (the precision the paper computes the step in,
    Sec. 3) has no bound, so M's error is measured against the magnitude of
    its terms, b1 |M_prev| + (1-b1) |g|, which for a sum without cancellation
    is its value;
  * bf16 weights: identical except for at most 1e-4 of the checked elements,
    and every differing element must be the dithered rounding, with the same
    16-bit draw r, of a value within 1e-6 of the oracle's pre-rounding x,
    relative to the magnitude of x's terms S = |w (1 - lr*lambda)| + |lr*kappa*U|.
    Where x does not cancel (S ~ |x|) this is "x within 1e-6 relative of a
    dither threshold, the outputs one bf16 ulp apart"; where the update nearly
    cancels the weight, fp32 evaluation (the paper's precision) can only place
    x to within ~1e-7 S, which may span several ulps of the small x. A wrong
    draw r or a wrong update is not admitted by the bound;
  * per-tensor RMS(U) and clip factor: relative error <= 1e-6.
Every step also counts the elements that pass only through the widened readings:
weights whose x lies within 1e-6 S but not within 1e-6 |x| of the dither's set
(w_widened), and momenta within 1e-5 of their terms' scale but not of their value
(m_widened); the full-size subsets assert these stay within the 1e-4 share.
Tensors are independent, so checking a subset of a large parameter set is
exact parity for that subset while the GPU runs the whole set. A stacked
(E, n, m) tensor is checked as E matrices, each against its own oracle run
whose dither index starts at the matrix's flat offset e*n*m.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

import oracle as O
from paper_2607_19058_gb300 import skewadam as S
from paper_2607_19058_gb300 import workloads as WL

STATE_RTOL = 1e-5
W_MISMATCH_FRAC = 1e-4
X_RTOL = 1e-6
SCALAR_RTOL = 1e-6
# fp32 spaces its subnormals 2^-149 apart, so a state value below the normal range cannot
# be evaluated in fp32 to 1e-5 relative: state is also accepted within a few such steps
STATE_ATOL = 4.0 * 2.0 ** -149


def fma_f32(a: np.ndarray, b: np.ndarray, c: np.ndarray) -> np.ndarray:
    """fp32 fused multiply-add, correctly rounded (what fmaf / FFMA compute), emulated
    exactly for results in fp32's normal range: a*b is exact in fp64, TwoSum gives
    a*b + c = s + e exactly (s = fl64(a*b + c), |e| <= half an fp64 ulp of s), and
    rounding s to fp32 equals rounding s + e unless s is itself an fp32 rounding midpoint,
    where the sign of e decides."""
    a = np.asarray(a, np.float32).astype(np.float64)
    b = np.asarray(b, np.float32).astype(np.float64)
    c = np.asarray(c, np.float32).astype(np.float64)
    p = a * b
    s = p + c
    bp = s - p
    e = (p - (s - bp)) + (c - bp)
    r = s.astype(np.float32)
    # an fp32 midpoint in fp64: the 29 significand bits below fp32's are 1000...0
    mid = (s.view(np.uint64) & np.uint64((1 << 29) - 1)) == np.uint64(1 << 28)
    fix = np.nonzero(mid & (e != 0))[0]
    if fix.size:
        t = r[fix]
        below = t.astype(np.float64) < s[fix]
        lo = np.where(below, t, np.nextafter(t, np.float32(-np.inf)))
        hi = np.where(below, np.nextafter(t, np.float32(np.inf)), t)
        r[fix] = np.where(e[fix] > 0, hi, lo)
    return r


def bits16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16).reshape(-1).copy()


def host_copy(t: torch.Tensor) -> np.ndarray:
    """Host copy of a weight / gradient tensor as the oracle takes it: bf16 bit patterns, or
    fp32 values for a tensor kept in fp32."""
    if t.dtype == torch.float32:
        return t.detach().contiguous().cpu().numpy().reshape(-1).copy()
    return bits16(t)


def as_f64(a: np.ndarray) -> np.ndarray:
    """bf16 bit patterns or fp32 values as float64."""
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def f32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().reshape(-1).copy()


@dataclasses.dataclass
class Report:
    elements: int = 0
    w_mismatch: int = 0
    worst_state_rel: float = 0.0
    worst_scalar_rel: float = 0.0
    worst_thresh: float = 0.0
    clipped: int = 0
    tensors: int = 0
    w_widened: int = 0     # weights passing only because S > |x| (reading R18)
    m_widened: int = 0     # momenta passing only because their terms' scale > |M| (reading R17)
    m_unexplained: int = 0  # of those, momenta that are not fma(b1, M_prev, fl(c1 g)) in fp32
    s_floor: int = 0       # state values passing only through the subnormal floor (reading R24)

    def merge(self, o: "Report"):
        self.elements += o.elements
        self.w_mismatch += o.w_mismatch
        self.w_widened += o.w_widened
        self.m_widened += o.m_widened
        self.m_unexplained += o.m_unexplained
        self.s_floor += o.s_floor
        self.worst_state_rel = max(self.worst_state_rel, o.worst_state_rel)
        self.worst_scalar_rel = max(self.worst_scalar_rel, o.worst_scalar_rel)
        self.worst_thresh = max(self.worst_thresh, o.worst_thresh)
        self.clipped += o.clipped
        self.tensors += o.tensors


def rel_err(a: np.ndarray, b: np.ndarray) -> float:
    """Max error of fp32 state `a` against the oracle's `b`, relative to max(|b|, the floor
    below which fp32 state is judged in absolute terms): an element passes at STATE_RTOL
    when it is within STATE_RTOL * |b| or within STATE_ATOL of b."""
    a = a.astype(np.float64)
    b = b.astype(np.float64)
    if not (np.isfinite(a).all() and np.isfinite(b).all()):
        return 0.0 if np.array_equal(a, b, equal_nan=True) else float("inf")
    if a.size == 0:
        return 0.0
    den = np.maximum(np.abs(b), STATE_ATOL / STATE_RTOL)
    return float((np.abs(a - b) / den).max())


def floor_only(a: np.ndarray, b: np.ndarray) -> int:
    """Elements of `a` within STATE_ATOL of `b` but not within STATE_RTOL * |b| (state in
    fp32's subnormal range)."""
    a = a.astype(np.float64)
    b = b.astype(np.float64)
    fin = np.isfinite(a) & np.isfinite(b)
    d = np.abs(a - b)[fin]
    return int(np.count_nonzero((d > STATE_RTOL * np.abs(b[fin])) & (d <= STATE_ATOL)))


def rel_err_terms(a: np.ndarray, b: np.ndarray, scale: np.ndarray) -> float:
    """Relative error of `a` against `b`, measured against max(|b|, scale of the terms)."""
    a = a.astype(np.float64)
    b = b.astype(np.float64)
    if not (np.isfinite(a).all() and np.isfinite(b).all()):
        return 0.0 if np.array_equal(a, b, equal_nan=True) else float("inf")
    den = np.maximum(np.abs(b), scale)
    d = np.abs(a - b)
    zero = den == 0
    if np.any(d[zero] != 0):
        return float("inf")
    return float((d[~zero] / den[~zero]).max()) if (~zero).any() else 0.0


def widened_terms(a: np.ndarray, b: np.ndarray, scale: np.ndarray, rtol: float) -> np.ndarray:
    """Indices of the elements of `a` within rtol of `b` measured against the terms' scale
    but not against |b|."""
    a = a.astype(np.float64)
    b = b.astype(np.float64)
    d = np.abs(a - b)
    ok = np.isfinite(a) & np.isfinite(b)
    return np.nonzero(ok & (d > rtol * np.abs(b)) & (d <= rtol * np.maximum(np.abs(b), scale)))[0]


def check_momentum(gpu_m: np.ndarray, ora_m: np.ndarray, m_prev: np.ndarray, g: np.ndarray, b1: float,
                   gscale: float = 1.0):
    """Momentum M = b1 M_prev + (1 - b1) gamma g (Algorithm 1) from the GPU against the
    oracle's fp64 value. Returns (error relative to max(|M|, the terms' scale), the count of
    elements passing only because their terms' scale exceeds |M| (reading R17), and how many
    of those are not, bit for bit, fp32's fma(b1, M_prev, fl(c1 g)) with c1 = fl(1 - b1) gamma:
    a momentum that cancels far below its terms is accepted only as that fp32 evaluation)."""
    gd = gscale * as_f64(g)
    scale = b1 * np.abs(m_prev.astype(np.float64)) + (1 - b1) * np.abs(gd)
    err = rel_err_terms(gpu_m, ora_m, scale)
    wid = widened_terms(gpu_m, ora_m, scale, STATE_RTOL)
    if wid.size == 0:
        return err, 0, 0
    c1 = np.float32(np.float32(1.0 - b1) * np.float32(gscale))
    want = fma_f32(np.full(wid.size, np.float32(b1)), m_prev[wid], c1 * as_f64(g[wid]).astype(np.float32))
    unexplained = int(np.count_nonzero(want.view(np.uint32) != np.asarray(gpu_m, np.float32)[wid].view(np.uint32)))
    return err, int(wid.size), unexplained


def _bits_to_f64(b32: np.ndarray) -> np.ndarray:
    return np.asarray(b32, np.uint32).view(np.float32).astype(np.float64)


def compare_weights_f32(gpu_w: np.ndarray, x: np.ndarray, w_pre: np.ndarray, wdf: float, where: str,
                        upd_terms=None) -> (int, float):
    """fp32 tensors (no dither): the GPU's weight is its fp32 evaluation of x; every element
    must lie within X_RTOL * S of the oracle's x, S = |w (1 - lr lambda)| + the magnitude of
    the update's terms, and non-finite values must match exactly."""
    g64, x64 = gpu_w.astype(np.float64), x.astype(np.float64)
    fin = np.isfinite(x64)
    inf = np.isinf(x64)
    assert np.array_equal(np.isnan(g64), np.isnan(x64)) and np.array_equal(g64[inf], x64[inf]), \
        f"{where}: non-finite fp32 weights differ"
    diff = (gpu_w.view(np.uint32) != x.view(np.uint32)) & fin
    nbad = int(diff.sum())
    worst, widened = 0.0, 0
    if nbad:
        t1 = w_pre[diff].astype(np.float64) * wdf
        upd = np.abs(t1 - x64[diff])
        if upd_terms is not None:
            upd = np.maximum(upd, upd_terms(np.nonzero(diff)[0]))
        S = np.abs(t1) + upd
        dist = np.abs(g64[diff] - x64[diff])
        rel = dist / np.maximum(S, 1e-300)
        worst = float(rel.max())
        assert worst <= X_RTOL, f"{where}: fp32 weight {worst:.3e} S from the oracle's x"
        widened = int(np.count_nonzero(dist > X_RTOL * np.abs(x64[diff])))
    return 0, worst, widened


def compare_weights(gpu_w: np.ndarray, ora_w: np.ndarray, x: np.ndarray, r: np.ndarray, w_pre: np.ndarray,
                    wdf: float, where: str, upd_terms=None) -> (int, float):
    """Counts differing weights and returns the worst distance (in units of S) of x from the
    set of values whose dithered rounding with the same r gives the GPU's bf16.

    `upd_terms(idx)`, when given, returns the magnitude of the update's own terms at
    those elements (momentum tensors: the update is proportional to M, itself a
    possibly cancelling sum); otherwise the update's magnitude |w(1-lr*lambda) - x| is used.
    """
    diff = gpu_w != ora_w
    nbad = int(diff.sum())
    worst, widened = 0.0, 0
    if nbad:
        g = gpu_w[diff].astype(np.int64)
        rr = r[diff].astype(np.int64)
        xo = x[diff].astype(np.float64)
        sign = (g & 0x8000) << 16
        lo_mag = np.maximum((g & 0x7FFF) * 65536 - rr, 0)
        hi_mag = (g & 0x7FFF) * 65536 - rr + 65535
        assert np.all(hi_mag >= 0), f"{where}: impossible dithered output"
        xa = _bits_to_f64((sign | lo_mag).astype(np.uint32))
        xb = _bits_to_f64((sign | hi_mag).astype(np.uint32))
        lo, hi = np.minimum(xa, xb), np.maximum(xa, xb)
        dist = np.where(xo < lo, lo - xo, np.where(xo > hi, xo - hi, 0.0))
        t1 = (w_pre[diff].astype(np.uint32) << 16).view(np.float32).astype(np.float64) * wdf
        upd = np.abs(t1 - xo)
        if upd_terms is not None:
            upd = np.maximum(upd, upd_terms(np.nonzero(diff)[0]))
        S = np.abs(t1) + upd
        rel = dist / np.maximum(S, 1e-300)
        worst = float(rel.max())
        k = int(np.argmax(rel))
        assert worst <= X_RTOL, (f"{where}: GPU bf16 {g[k]:#06x} is not a dithered rounding of any value within "
                                 f"{X_RTOL:g}*S of x={xo[k]!r} (S={S[k]:.3e}, distance {worst:.3e} S)")
        widened = int(np.count_nonzero(dist > X_RTOL * np.abs(xo)))
    return nbad, worst, widened


class Harness:
    """GPU handle over a whole workload, oracle copies of the `check` tensors."""

    def __init__(self, wl: WL.Workload, check: Optional[Sequence[int]] = None, device="cuda",
                 grad_device: Optional[str] = None, hp_override: Optional[dict] = None,
                 misalign: Sequence[int] = (), matrices: Optional[Dict[int, Sequence[int]]] = None,
                 max_widened_frac: Optional[float] = None):
        """`matrices[k]`, when given, limits the check of stacked tensor k to those matrices.
        `step(..., gscale=g)` steps on g * G (the trainer's global-norm clip factor), passed
        to the GPU as a device scalar and to the oracle as its gscale."""
        self.wl = wl
        hpd = dataclasses.asdict(wl.hp)
        if hp_override:
            hpd.update(hp_override)
        self.hpd = hpd
        self.dev = torch.device(device)
        self.gdev = grad_device or device
        self.W, self.G = [], []
        for k in range(len(wl.specs)):
            w0 = WL.init_weight(wl, k, self.gdev).to(self.dev)
            if k in misalign:   # contiguous views whose data pointers are only 2-byte aligned
                shape = w0.shape
                bw = torch.empty(w0.numel() + 1, dtype=torch.bfloat16, device=self.dev)
                bg = torch.zeros(w0.numel() + 1, dtype=torch.bfloat16, device=self.dev)
                w = bw[1:].view(shape)
                w.copy_(w0)
                self.W.append(w)
                self.G.append(bg[1:].view(shape))
            else:
                self.W.append(w0)
                self.G.append(torch.zeros_like(w0))
        params = [(self.W[k], self.G[k], s.tier, S.F_NO_DECAY if s.no_decay else 0) for k, s in enumerate(wl.specs)]
        self.hp = S.hparams(hpd["beta1"], hpd["beta2"], hpd["eps"], hpd["clip_d"], hpd["weight_decay"], hpd["policy"])
        self.opt = S.SkewAdam(params, self.hp)
        self.check = list(range(len(wl.specs))) if check is None else list(check)
        self.ostate = {k: {e: O.TensorState(self._mat_shape(k), wl.specs[k].tier, hpd["policy"], wl.specs[k].no_decay)
                           for e in (matrices or {}).get(k, range(self._stack(k)))} for k in self.check}
        self.ohp = O.hparams(hpd["beta1"], hpd["beta2"], hpd["eps"], hpd["clip_d"], hpd["weight_decay"],
                             annealed=hpd["policy"] == WL.POLICY_ADAFACTOR)
        self.lr = hpd["lr"]
        self.max_widened_frac = max_widened_frac

    def load_grads(self, t: int):
        for k in range(len(self.wl.specs)):
            self.G[k].copy_(WL.grad(self.wl, k, t, self.gdev).to(self.dev))

    def _stack(self, k: int) -> int:
        return self.wl.specs[k].shape[0] if len(self.wl.specs[k].shape) == 3 else 1

    def _mat_shape(self, k: int):
        shp = self.wl.specs[k].shape
        return tuple(shp[1:]) if len(shp) == 3 else tuple(shp)

    def _gpu_state(self, k: int) -> List[Dict[str, Optional[np.ndarray]]]:
        """Per matrix of tensor k (one entry unless it is a stack): its M, v, R, C."""
        v = {key: (None if a is None else f32(a)) for key, a in self.opt.state_views(k).items()}
        E = self._stack(k)
        out = []
        for e in range(E):
            d = {}
            for key, a in v.items():
                ln = None if a is None else a.size // E
                d[key] = None if a is None else a[e * ln:(e + 1) * ln]
            out.append(d)
        return out

    def step(self, t: int, seed: int = 1234, grads_loaded: bool = False, gscale: Optional[float] = None) -> Report:
        if not grads_loaded:
            self.load_grads(t)
        self.gscale = 1.0 if gscale is None else float(np.float32(gscale))
        self.ohp.gscale = self.gscale
        torch.cuda.synchronize()
        pre = {}
        for k in self.check:   # teacher forcing: the oracle starts from the GPU's pre-step values
            gs = self._gpu_state(k)
            wb, gb = host_copy(self.W[k]), host_copy(self.G[k])
            nm = wb.size // self._stack(k)
            pre[k] = {}
            for e, st in self.ostate[k].items():
                for key in ("M", "v", "R", "C"):
                    if getattr(st, key) is not None:
                        getattr(st, key)[:] = gs[e][key]
                pre[k][e] = (wb[e * nm:(e + 1) * nm].copy(), gb[e * nm:(e + 1) * nm].copy(),
                             None if st.M is None else st.M.copy())
        if gscale is None:
            self.opt.step(t, self.lr, seed)
        else:
            self.opt.step(t, self.lr, seed, grad_scale=torch.tensor([gscale], dtype=torch.float32, device=self.dev))
        self.opt.sync_status()
        rep = Report()
        for k in self.check:
            gws, gss = host_copy(self.W[k]), self._gpu_state(k)
            for e, st in self.ostate[k].items():
                rep.merge(self._check_matrix(k, e, st, pre[k][e], gws, gss[e], t, seed))
        assert rep.w_mismatch <= W_MISMATCH_FRAC * rep.elements, \
            f"{self.wl.name} step {t}: {rep.w_mismatch} of {rep.elements} weights differ"
        print(f"parity {self.wl.name} step {t}: {rep.elements} weights, {rep.w_mismatch} one-ulp dither "
              f"mismatches; passing only through a reading: {rep.w_widened} weights (R18), {rep.m_widened} "
              f"momenta (R17; {rep.m_unexplained} of them not fp32's fma(b1, M_prev, fl(c1 g))), "
              f"{rep.s_floor} state values (R24)")
        if self.max_widened_frac is not None:
            assert rep.w_widened <= self.max_widened_frac * rep.elements, \
                f"{self.wl.name} step {t}: {rep.w_widened} weights pass only through reading R18"
            assert rep.m_unexplained == 0, \
                f"{self.wl.name} step {t}: {rep.m_unexplained} momenta pass only through reading R17 and are " \
                f"not the fp32 evaluation of their update"
        return rep

    def _check_matrix(self, k, e, st, pre, gws, gs, t, seed) -> Report:
        """Matrix e of tensor k (e = 0 unless it is a stack) against one oracle step."""
        w0, g, m_prev = pre
        wpre = w0.copy()
        nm = w0.size
        o = O.tensor_step(w0, g, st, k, self.ohp, t, self.lr, seed, want_x=True, idx0=e * nm)
        where = f"{self.wl.name}/{self.wl.specs[k].name}" + (f"[{e}]" if self._stack(k) > 1 else "") + f" step {t}"
        gw = gws[e * nm:(e + 1) * nm]
        lam = float(np.float32(self.hpd["weight_decay"])) if st.decay else 0.0
        wdf = 1.0 - float(np.float32(self.lr)) * lam
        terms = self._momentum_update_terms(st, o, g, m_prev, t) if st.momentum else None
        if gw.dtype == np.float32:
            nbad, worst, wwid = compare_weights_f32(gw, o["x"], wpre, wdf, where, terms)
        else:
            nbad, worst, wwid = compare_weights(gw, w0, o["x"], o["r"], wpre, wdf, where, terms)
        worst_state, mwid, munex, sfloor = 0.0, 0, 0, 0
        for key in ("M", "v", "R", "C"):
            if getattr(st, key) is not None:
                if key == "M":
                    err, mwid, munex = check_momentum(gs[key], st.M, m_prev, g, float(np.float32(self.hpd["beta1"])),
                                                      self.gscale)
                else:
                    err = rel_err(gs[key], getattr(st, key))
                    sfloor += floor_only(gs[key], getattr(st, key))
                assert err <= STATE_RTOL, f"{where}: state {key} rel err {err:.3g}"
                worst_state = max(worst_state, err)
        sc = self.opt.scalars(k, matrix=e)
        se = 0.0
        for key in ("rms", "kappa"):
            err = abs(sc[key] - o[key]) / max(abs(o[key]), 1e-300)
            if o[key] == 0.0:
                err = abs(sc[key])
            assert err <= SCALAR_RTOL, f"{where}: {key} {sc[key]!r} vs oracle {o[key]!r}"
            se = max(se, err)
        return Report(elements=gw.size, w_mismatch=nbad, worst_state_rel=worst_state, worst_scalar_rel=se,
                      worst_thresh=worst, clipped=int(o["kappa"] < 1.0), tensors=1, w_widened=wwid, m_widened=mwid,
                      m_unexplained=munex, s_floor=sfloor)

    def _momentum_update_terms(self, st, o, g, m_prev, t):
        """lr*kappa*coef/D * (b1|M_prev| + (1-b1)|g|) from the oracle's post-step state."""
        f = lambda key: float(np.float32(self.hpd[key]))
        b1, b2, eps, lr = f("beta1"), f("beta2"), f("eps"), f("lr")
        coef = np.sqrt(1 - b2 ** t) / (1 - b1 ** t)

        def fn(idx):
            if st.kind == O.KIND_FULL:
                vhat = st.v[idx].astype(np.float64)
            else:
                i, j = idx // st.m, idx % st.m
                vhat = (st.R[i].astype(np.float64) * st.C[j].astype(np.float64) / o["rbar"]
                        if o["rbar"] > 0 else np.zeros(idx.size))
            inv = 1.0 / np.sqrt(np.maximum(vhat, eps))
            gd = self.gscale * as_f64(g[idx])
            mterms = b1 * np.abs(m_prev[idx].astype(np.float64)) + (1 - b1) * np.abs(gd)
            return lr * o["kappa"] * coef * inv * mterms
        return fn

    def close(self):
        self.opt.close()
