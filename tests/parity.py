"""Parity harness: libskewadam (CUDA, through the C ABI) against the CPU oracle.

Per step and per checked tensor, with teacher forcing: the oracle starts from
the GPU's pre-step weights and state, takes the same gradient, and the two
post-step results are compared with the acceptance bars of the method:
  * fp32 state (R, C, v, M): max relative error <= 1e-5;
  * bf16 weights: identical except for at most 1e-4 of the checked elements,
    each differing by exactly one bf16 ulp and only where the oracle's fp32
    value x lies within 8 fp32 ulps of its dither threshold, i.e.
    |low16(bits(x)) + r - 2^16| <= 8 (which also shows the dither bits agree);
  * per-tensor RMS(U) and clip factor: relative error <= 1e-6.
Tensors are independent, so checking a subset of a large parameter set is
exact parity for that subset while the GPU runs the whole set.
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
THRESH_ULPS = 8
SCALAR_RTOL = 1e-6


def bits16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16).reshape(-1).copy()


def f32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().reshape(-1).copy()


@dataclasses.dataclass
class Report:
    elements: int = 0
    w_mismatch: int = 0
    worst_state_rel: float = 0.0
    worst_scalar_rel: float = 0.0
    worst_thresh: int = 0
    clipped: int = 0
    tensors: int = 0

    def merge(self, o: "Report"):
        self.elements += o.elements
        self.w_mismatch += o.w_mismatch
        self.worst_state_rel = max(self.worst_state_rel, o.worst_state_rel)
        self.worst_scalar_rel = max(self.worst_scalar_rel, o.worst_scalar_rel)
        self.worst_thresh = max(self.worst_thresh, o.worst_thresh)
        self.clipped += o.clipped
        self.tensors += o.tensors


def rel_err(a: np.ndarray, b: np.ndarray) -> float:
    """Max relative error of fp32 state `a` against the oracle's `b` (exact zeros must match)."""
    a = a.astype(np.float64)
    b = b.astype(np.float64)
    if not (np.isfinite(a).all() and np.isfinite(b).all()):
        return 0.0 if np.array_equal(a, b, equal_nan=True) else float("inf")
    if a.size == 0:
        return 0.0
    d = np.abs(a - b)
    zero = b == 0
    if np.any(d[zero] != 0):
        return float("inf")
    return float((d[~zero] / np.abs(b[~zero])).max()) if (~zero).any() else 0.0


def compare_weights(gpu_w: np.ndarray, ora_w: np.ndarray, x: np.ndarray, r: np.ndarray, where: str) -> (int, int):
    diff = gpu_w != ora_w
    nbad = int(diff.sum())
    worst = 0
    if nbad:
        gw = gpu_w[diff].astype(np.int64)
        ow = ora_w[diff].astype(np.int64)
        same_sign = (gw & 0x8000) == (ow & 0x8000)
        one_ulp = np.abs(gw - ow) == 1
        assert np.all(same_sign & one_ulp), f"{where}: weight differs by more than one bf16 ulp"
        low = x[diff].view(np.uint32).astype(np.int64) & 0xFFFF
        dist = np.abs(low + r[diff].astype(np.int64) - 65536)
        worst = int(dist.max())
        assert worst <= THRESH_ULPS, f"{where}: mismatch {worst} fp32 ulps from the dither threshold"
    return nbad, worst


class Harness:
    """GPU handle over a whole workload, oracle copies of the `check` tensors."""

    def __init__(self, wl: WL.Workload, check: Optional[Sequence[int]] = None, device="cuda",
                 grad_device: Optional[str] = None, hp_override: Optional[dict] = None,
                 misalign: Sequence[int] = ()):
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
        self.ostate = {k: O.TensorState(wl.specs[k].shape, wl.specs[k].tier, hpd["policy"], wl.specs[k].no_decay)
                       for k in self.check}
        self.ohp = O.hparams(hpd["beta1"], hpd["beta2"], hpd["eps"], hpd["clip_d"], hpd["weight_decay"])
        self.lr = hpd["lr"]

    def load_grads(self, t: int):
        for k in range(len(self.wl.specs)):
            self.G[k].copy_(WL.grad(self.wl, k, t, self.gdev).to(self.dev))

    def _gpu_state(self, k: int) -> Dict[str, Optional[np.ndarray]]:
        v = self.opt.state_views(k)
        return {key: (None if a is None else f32(a)) for key, a in v.items()}

    def step(self, t: int, seed: int = 1234, grads_loaded: bool = False) -> Report:
        if not grads_loaded:
            self.load_grads(t)
        torch.cuda.synchronize()
        pre = {}
        for k in self.check:   # teacher forcing: the oracle starts from the GPU's pre-step values
            st = self.ostate[k]
            gs = self._gpu_state(k)
            for key in ("M", "v", "R", "C"):
                if getattr(st, key) is not None:
                    getattr(st, key)[:] = gs[key]
            pre[k] = (bits16(self.W[k]), bits16(self.G[k]))
        self.opt.step(t, self.lr, seed)
        self.opt.sync_status()
        rep = Report()
        for k in self.check:
            w0, g = pre[k]
            st = self.ostate[k]
            o = O.tensor_step(w0, g, st, k, self.ohp, t, self.lr, seed, want_x=True)
            where = f"{self.wl.name}/{self.wl.specs[k].name} step {t}"
            gw = bits16(self.W[k])
            nbad, worst = compare_weights(gw, w0, o["x"], o["r"], where)
            gs = self._gpu_state(k)
            worst_state = 0.0
            for key in ("M", "v", "R", "C"):
                if getattr(st, key) is not None:
                    e = rel_err(gs[key], getattr(st, key))
                    assert e <= STATE_RTOL, f"{where}: state {key} rel err {e:.3g}"
                    worst_state = max(worst_state, e)
            sc = self.opt.scalars(k)
            se = 0.0
            for key in ("rms", "kappa"):
                e = abs(sc[key] - o[key]) / max(abs(o[key]), 1e-300)
                if o[key] == 0.0:
                    e = abs(sc[key])
                assert e <= SCALAR_RTOL, f"{where}: {key} {sc[key]!r} vs oracle {o[key]!r}"
                se = max(se, e)
            r = Report(elements=gw.size, w_mismatch=nbad, worst_state_rel=worst_state, worst_scalar_rel=se,
                       worst_thresh=worst, clipped=int(o["kappa"] < 1.0), tensors=1)
            rep.merge(r)
        assert rep.w_mismatch <= W_MISMATCH_FRAC * rep.elements, \
            f"{self.wl.name} step {t}: {rep.w_mismatch} of {rep.elements} weights differ"
        return rep

    def close(self):
        self.opt.close()
