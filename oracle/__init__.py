"""SkewAdam CPU oracle: ctypes front end to ``skew_oracle.c``.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this package. It
shares no code with the CUDA library in ``paper_2607_19058_gb300``; the two
meet only through the seeded inputs the tests feed to both.

Every function here marshals numpy arrays into the C oracle; the arithmetic
(paper Sec. 3: Eq. 1, Algorithm 1, update clipping, dithered rounding, Eq. 2)
lives in ``skew_oracle.c``.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "skew_oracle.c")
LIB = os.path.join(HERE, "libskew_oracle.so")

KIND_FULL, KIND_FACTORED = 0, 1
TIER_BACKBONE, TIER_EXPERT, TIER_ROUTER = 0, 1, 2
POLICY_TIERED, POLICY_EXPERT_MOMENTUM, POLICY_FACTORED_ROUTER, POLICY_UNIFORM, POLICY_ADAFACTOR = 0, 1, 2, 3, 4

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no FP contraction, so x86 and Arm agree)."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-o", tmp, SRC, "-lm"]
        )
        os.replace(tmp, LIB)
    return LIB


class _Tensor(C.Structure):
    _fields_ = [
        ("w", C.c_void_p), ("g", C.c_void_p), ("M", C.c_void_p), ("v", C.c_void_p),
        ("R", C.c_void_p), ("C", C.c_void_p), ("n", C.c_int64), ("m", C.c_int64),
        ("kind", C.c_int32), ("momentum", C.c_int32), ("decay", C.c_int32), ("tid", C.c_uint32),
        ("idx0", C.c_uint64), ("wf", C.c_void_p), ("gf", C.c_void_p),
    ]


class _HParams(C.Structure):
    _fields_ = [("beta1", C.c_double), ("beta2", C.c_double), ("eps", C.c_double),
                ("clip_d", C.c_double), ("weight_decay", C.c_double), ("annealed", C.c_int32),
                ("gscale", C.c_double)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            L.so_philox4x32_10.argtypes = [C.POINTER(C.c_uint32)] * 3
            L.so_philox4x32_10.restype = None
            L.so_dither16.argtypes = [C.c_uint64, C.c_int64, C.c_uint32, C.c_uint64]
            L.so_dither16.restype = C.c_uint16
            L.so_sr_bf16.argtypes = [C.c_float, C.c_uint16]
            L.so_sr_bf16.restype = C.c_uint16
            L.so_resolve.argtypes = [C.c_int, C.c_int, C.c_int, C.c_int] + [C.POINTER(C.c_int)] * 3
            L.so_resolve.restype = C.c_int
            L.so_state_bytes.argtypes = [C.c_int, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32]
            L.so_state_bytes.restype = C.c_int64
            L.so_tensor_step.argtypes = [C.POINTER(_Tensor), C.POINTER(_HParams), C.c_int64, C.c_double,
                                         C.c_uint64, C.c_void_p, C.c_void_p, C.c_void_p]
            L.so_tensor_step.restype = C.c_int
            L.so_dither16_array.argtypes = [C.c_uint64, C.c_int64, C.c_uint32, C.c_uint64, C.c_int64, C.c_void_p]
            L.so_dither16_array.restype = None
            L.so_sr_bf16_array.argtypes = [C.c_void_p, C.c_void_p, C.c_int64, C.c_void_p]
            L.so_sr_bf16_array.restype = None
            _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data


def philox4x32_10(ctr, key):
    """Philox-4x32-10 block: 4 counter words, 2 key words -> 4 output words."""
    c = (C.c_uint32 * 4)(*[int(x) & 0xFFFFFFFF for x in ctr])
    k = (C.c_uint32 * 2)(*[int(x) & 0xFFFFFFFF for x in key])
    o = (C.c_uint32 * 4)()
    lib().so_philox4x32_10(c, k, o)
    return [int(x) for x in o]


def dither16(seed: int, step: int, tid: int, idx0: int, count: int) -> np.ndarray:
    """16-bit dithers of elements idx0 .. idx0+count-1 of tensor `tid`."""
    out = np.empty(count, dtype=np.uint16)
    lib().so_dither16_array(seed & (2**64 - 1), step, tid, idx0, count, _ptr(out))
    return out


def sr_bf16(x: np.ndarray, r: np.ndarray) -> np.ndarray:
    """Dithered rounding of fp32 values `x` with 16-bit draws `r` -> bf16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    r = np.ascontiguousarray(r, dtype=np.uint16)
    assert x.shape == r.shape
    out = np.empty(x.shape, dtype=np.uint16)
    lib().so_sr_bf16_array(_ptr(x), _ptr(r), x.size, _ptr(out))
    return out


def resolve(ndim: int, tier: int, policy: int = POLICY_TIERED, no_decay: bool = False):
    """Tier policy -> (kind, momentum, decay)."""
    k, mo, d = C.c_int(), C.c_int(), C.c_int()
    rc = lib().so_resolve(ndim, tier, policy, int(no_decay), C.byref(k), C.byref(mo), C.byref(d))
    if rc != 0:
        raise ValueError(f"bad tensor description ndim={ndim} tier={tier} policy={policy}")
    return k.value, mo.value, d.value


def state_bytes(specs, policy: int = POLICY_TIERED) -> int:
    """Closed-form state bytes (Eq. 2 + full v of vectors) for (shape, tier) specs."""
    nd = np.array([len(s) for s, _ in specs], dtype=np.int32)
    n = np.array([s[0] for s, _ in specs], dtype=np.int64)
    m = np.array([s[1] if len(s) == 2 else 1 for s, _ in specs], dtype=np.int64)
    t = np.array([tier for _, tier in specs], dtype=np.int32)
    v = lib().so_state_bytes(len(specs), _ptr(nd), _ptr(n), _ptr(m), _ptr(t), policy)
    if v < 0:
        raise ValueError("bad spec")
    return int(v)


class TensorState:
    """fp32 state of one tensor as the oracle keeps it (zero-initialised)."""

    def __init__(self, shape, tier, policy=POLICY_TIERED, no_decay=False):
        self.shape = tuple(shape)
        self.n = int(shape[0])
        self.m = int(shape[1]) if len(shape) == 2 else 1
        self.kind, self.momentum, self.decay = resolve(len(shape), tier, policy, no_decay)
        numel = self.n * self.m
        self.M = np.zeros(numel, np.float32) if self.momentum else None
        self.v = np.zeros(numel, np.float32) if self.kind == KIND_FULL else None
        self.R = np.zeros(self.n, np.float32) if self.kind == KIND_FACTORED else None
        self.C = np.zeros(self.m, np.float32) if self.kind == KIND_FACTORED else None

    def nbytes(self) -> int:
        return sum(a.nbytes for a in (self.M, self.v, self.R, self.C) if a is not None)


def hparams(beta1, beta2, eps, clip_d, weight_decay, annealed: bool = False, gscale: float = 1.0):
    """The fp32 hyper-parameters widened to double (both sides use the fp32 values).
    `annealed`: the Adafactor comparator's decay 1 - t^-0.8 without bias correction.
    `gscale`: the trainer's global gradient-norm clip factor of the step (an fp32 value):
    the step sees gscale * G."""
    f = lambda x: float(np.float32(x))
    return _HParams(f(beta1), f(beta2), f(eps), f(clip_d), f(weight_decay), int(annealed), f(gscale))


def tensor_step(w_bits: np.ndarray, g_bits: np.ndarray, st: TensorState, tid: int, hp, step: int,
                lr: float, seed: int, want_x: bool = False, idx0: int = 0):
    """One oracle step of one tensor; `w_bits` and the state update in place. Weights and
    gradient are both bf16 bit patterns (uint16) or both fp32 (an fp32 tensor: the new
    weight is x, no dither).

    Returns a dict with Rbar, sum of U^2, RMS and kappa, plus the fp32 pre-rounding
    values `x` and the dithers `r` (0 for an fp32 tensor) when `want_x`.
    """
    f32 = w_bits.dtype == np.float32
    assert (w_bits.dtype, g_bits.dtype) in ((np.uint16, np.uint16), (np.float32, np.float32))
    assert w_bits.flags.c_contiguous and g_bits.flags.c_contiguous
    numel = st.n * st.m
    assert w_bits.size == numel and g_bits.size == numel
    T = _Tensor(None if f32 else _ptr(w_bits), None if f32 else _ptr(g_bits), _ptr(st.M), _ptr(st.v), _ptr(st.R),
                _ptr(st.C), st.n, st.m, st.kind, st.momentum, st.decay, tid, idx0,
                _ptr(w_bits) if f32 else None, _ptr(g_bits) if f32 else None)
    x = np.empty(numel, np.float32) if want_x else None
    r = np.empty(numel, np.uint16) if want_x else None
    stats = np.zeros(4, np.float64)
    rc = lib().so_tensor_step(C.byref(T), C.byref(hp), step, float(np.float32(lr)), seed & (2**64 - 1),
                              _ptr(x), _ptr(r), _ptr(stats))
    if rc != 0:
        raise RuntimeError("oracle step failed")
    out = {"rbar": stats[0], "sumu2": stats[1], "rms": stats[2], "kappa": stats[3]}
    if want_x:
        out["x"] = x
        out["r"] = r
    return out
