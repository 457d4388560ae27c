"""ctypes binding of libskewadam (include/skewadam.h).

Argument marshalling only: every step of the optimizer runs in the library's
CUDA kernels. PyTorch provides device memory (state and workspace buffers are
``torch.empty`` allocations) and the current CUDA stream. The functions keep the
C names; ``SkewAdam`` bundles create / bind / step for torch tensors.

If the library has not been built this module raises on first use; there is no
CPU fallback.
"""
from __future__ import annotations

import ctypes as C
import os
import threading
from typing import Iterable, List, Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libskewadam.so")

SKEW_OK, SKEW_EINVAL, SKEW_ENOMEM, SKEW_ECUDA, SKEW_ETIMEOUT, SKEW_ESTATE, SKEW_ETOOBIG = 0, -1, -2, -3, -4, -5, -6
NOALLOC_SCRATCH_BYTES = 16 * 1024 * 1024
TIER_BACKBONE, TIER_EXPERT, TIER_ROUTER = 0, 1, 2
POLICY_TIERED, POLICY_EXPERT_MOMENTUM, POLICY_FACTORED_ROUTER, POLICY_UNIFORM, POLICY_ADAFACTOR = 0, 1, 2, 3, 4
F_NO_DECAY = 1
F_FP32 = 2
KIND_FULL, KIND_FACTORED = 0, 1

EXPORTS = ["skew_create", "skew_destroy", "skew_state_bytes", "skew_workspace_bytes", "skew_bind", "skew_step",
           "skew_sync_status", "skew_tensor_scalars", "skew_matrix_scalars", "skew_tensor_info", "skew_num_tensors", "skew_last_error",
           "skew_profile_begin", "skew_profile_end", "skew_kernel_name", "skew_step_tensor_noalloc",
           "skew_launches_per_step", "skew_selftest_wait_timeout", "skew_noalloc_sync_status", "skew_step_scaled",
           "skew_noalloc_selftest_wait_timeout"]


class SkewError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"libskewadam error {code}: {msg}")
        self.code = code


class ParamDesc(C.Structure):
    _fields_ = [("weight", C.c_void_p), ("grad", C.c_void_p), ("shape", C.c_int64 * 2), ("ndim", C.c_int32),
                ("tier", C.c_int32), ("flags", C.c_uint32), ("stack", C.c_uint32)]


class HParams(C.Structure):
    _fields_ = [("beta1", C.c_float), ("beta2", C.c_float), ("eps", C.c_float), ("clip_d", C.c_float),
                ("weight_decay", C.c_float), ("policy", C.c_int32)]


class TensorInfo(C.Structure):
    _fields_ = [("kind", C.c_int32), ("momentum", C.c_int32), ("decay", C.c_int32), ("vectorized", C.c_int32),
                ("rows", C.c_int64), ("cols", C.c_int64), ("numel", C.c_int64), ("m_offset", C.c_int64),
                ("v_offset", C.c_int64), ("r_offset", C.c_int64), ("c_offset", C.c_int64), ("rowpath", C.c_int32),
                ("stack", C.c_int32)]


_lock = threading.Lock()
_lib = None


def load(path: Optional[str] = None) -> C.CDLL:
    """Loads libskewadam.so (built by ``__graft_entry__.build()``); raises if absent."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build it with __graft_entry__.build() "
                               "(no CPU fallback exists)")
        L = C.CDLL(p)
        vp, i32, i64, u64, sz = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64, C.c_size_t
        L.skew_create.argtypes = [C.POINTER(ParamDesc), i32, C.POINTER(HParams), C.POINTER(vp)]
        L.skew_create.restype = C.c_int
        L.skew_destroy.argtypes = [vp]
        L.skew_destroy.restype = C.c_int
        L.skew_state_bytes.argtypes = [vp]
        L.skew_state_bytes.restype = sz
        L.skew_workspace_bytes.argtypes = [vp]
        L.skew_workspace_bytes.restype = sz
        L.skew_bind.argtypes = [vp, vp, sz, vp, sz, vp]
        L.skew_bind.restype = C.c_int
        L.skew_step.argtypes = [vp, i64, C.c_float, u64, vp]
        L.skew_step.restype = C.c_int
        L.skew_step_scaled.argtypes = [vp, i64, C.c_float, u64, vp, vp]
        L.skew_step_scaled.restype = C.c_int
        L.skew_sync_status.argtypes = [vp, vp]
        L.skew_sync_status.restype = C.c_int
        L.skew_selftest_wait_timeout.argtypes = [vp, vp]
        L.skew_selftest_wait_timeout.restype = C.c_int
        L.skew_tensor_scalars.argtypes = [vp, i32, C.POINTER(C.c_double), vp]
        L.skew_tensor_scalars.restype = C.c_int
        L.skew_matrix_scalars.argtypes = [vp, i32, i32, C.POINTER(C.c_double), vp]
        L.skew_matrix_scalars.restype = C.c_int
        L.skew_tensor_info.argtypes = [vp, i32, C.POINTER(TensorInfo)]
        L.skew_tensor_info.restype = C.c_int
        L.skew_launches_per_step.argtypes = [vp]
        L.skew_launches_per_step.restype = i64
        L.skew_num_tensors.argtypes = [vp]
        L.skew_num_tensors.restype = i32
        L.skew_last_error.argtypes = [vp]
        L.skew_last_error.restype = C.c_char_p
        L.skew_profile_begin.argtypes = [vp, i32]
        L.skew_profile_begin.restype = C.c_int
        L.skew_profile_end.argtypes = [vp, C.POINTER(C.c_double), i64, C.POINTER(i32), C.POINTER(i32)]
        L.skew_profile_end.restype = C.c_int
        L.skew_kernel_name.argtypes = [i32]
        L.skew_kernel_name.restype = C.c_char_p
        L.skew_step_tensor_noalloc.argtypes = [vp, vp, i32, i64, i64, i32, C.c_uint32, C.POINTER(HParams), vp, sz,
                                               C.c_uint32, i64, C.c_float, u64, vp]
        L.skew_step_tensor_noalloc.restype = C.c_int
        L.skew_noalloc_sync_status.argtypes = [vp]
        L.skew_noalloc_sync_status.restype = C.c_int
        L.skew_noalloc_selftest_wait_timeout.argtypes = [vp]
        L.skew_noalloc_selftest_wait_timeout.restype = C.c_int
        if path is None:
            _lib = L
        return L


def _check(rc: int, h=None):
    if rc != SKEW_OK:
        msg = load().skew_last_error(h)
        raise SkewError(rc, msg.decode() if msg else "")


# --------------------------------------------------------------------------
# C entry points, same names
# --------------------------------------------------------------------------
def skew_create(params: Sequence[ParamDesc], hp: HParams) -> C.c_void_p:
    arr = (ParamDesc * max(1, len(params)))(*params)
    h = C.c_void_p()
    _check(load().skew_create(arr, len(params), C.byref(hp), C.byref(h)))
    return h


def skew_destroy(h) -> None:
    load().skew_destroy(h)


def skew_state_bytes(h) -> int:
    return int(load().skew_state_bytes(h))


def skew_workspace_bytes(h) -> int:
    return int(load().skew_workspace_bytes(h))


def skew_bind(h, state_ptr: int, state_bytes: int, ws_ptr: int, ws_bytes: int, stream: int) -> None:
    _check(load().skew_bind(h, state_ptr, state_bytes, ws_ptr, ws_bytes, stream), h)


def skew_step(h, step: int, lr: float, seed: int, stream: int) -> None:
    _check(load().skew_step(h, step, lr, seed & (2**64 - 1), stream), h)


def skew_step_scaled(h, step: int, lr: float, seed: int, grad_scale_ptr: int, stream: int) -> None:
    """skew_step on gamma * G, gamma read by the kernels from the device pointer (0: gamma = 1)."""
    _check(load().skew_step_scaled(h, step, lr, seed & (2**64 - 1), grad_scale_ptr or None, stream), h)


def skew_sync_status(h, stream: int) -> None:
    _check(load().skew_sync_status(h, stream), h)


def skew_selftest_wait_timeout(h, stream: int) -> None:
    _check(load().skew_selftest_wait_timeout(h, stream), h)


def skew_tensor_scalars(h, tid: int, stream: int):
    out = (C.c_double * 4)()
    _check(load().skew_tensor_scalars(h, tid, out, stream), h)
    return {"rbar": out[0], "sumu2": out[1], "rms": out[2], "kappa": out[3]}


def skew_matrix_scalars(h, tid: int, e: int, stream: int):
    out = (C.c_double * 4)()
    _check(load().skew_matrix_scalars(h, tid, e, out, stream), h)
    return {"rbar": out[0], "sumu2": out[1], "rms": out[2], "kappa": out[3]}


def skew_tensor_info(h, tid: int) -> TensorInfo:
    info = TensorInfo()
    _check(load().skew_tensor_info(h, tid, C.byref(info)), h)
    return info


def skew_launches_per_step(h) -> int:
    return int(load().skew_launches_per_step(h))


def skew_num_tensors(h) -> int:
    return int(load().skew_num_tensors(h))


def skew_last_error(h=None) -> str:
    m = load().skew_last_error(h)
    return m.decode() if m else ""


def skew_profile_begin(h, max_steps: int) -> None:
    _check(load().skew_profile_begin(h, max_steps), h)


def skew_profile_end(h, cap: int = 1 << 16):
    """-> (kernel names, list of per-step lists of per-kernel milliseconds)."""
    buf = (C.c_double * cap)()
    ns, nk = C.c_int32(), C.c_int32()
    _check(load().skew_profile_end(h, buf, cap, C.byref(ns), C.byref(nk)), h)
    names = [skew_kernel_name(k) for k in range(nk.value)]
    rows = [[buf[s * nk.value + k] for k in range(nk.value)] for s in range(ns.value) if (s + 1) * nk.value <= cap]
    return names, rows


def skew_kernel_name(k: int) -> str:
    m = load().skew_kernel_name(k)
    return m.decode() if m else ""


def skew_step_tensor_noalloc(weight_ptr: int, grad_ptr: int, ndim: int, rows: int, cols: int, tier: int, flags: int,
                             hp: HParams, state_ptr: int, state_bytes: int, tensor_id: int, step: int, lr: float,
                             seed: int, stream: int) -> None:
    """One tensor's step with the library's fixed scratch array (no allocation of any kind)."""
    rc = load().skew_step_tensor_noalloc(weight_ptr, grad_ptr, ndim, rows, cols, tier, flags, C.byref(hp), state_ptr,
                                         state_bytes, tensor_id, step, lr, seed & (2**64 - 1), stream)
    if rc != SKEW_OK:
        why = {SKEW_EINVAL: "invalid argument or state size", SKEW_ECUDA: "CUDA error",
               SKEW_ETOOBIG: f"tensor needs more than the {NOALLOC_SCRATCH_BYTES} bytes of fixed scratch"}
        raise SkewError(rc, why.get(rc, "error"))


def skew_noalloc_sync_status(stream: int) -> None:
    """Synchronises `stream`; raises SkewError(SKEW_ETIMEOUT) once if a bounded device wait of a
    no-alloc call gave up since the last read (the status word is then cleared)."""
    rc = load().skew_noalloc_sync_status(stream)
    if rc != SKEW_OK:
        why = {SKEW_ETIMEOUT: "a bounded device wait of a no-alloc step gave up", SKEW_ECUDA: "CUDA error"}
        raise SkewError(rc, why.get(rc, "error"))


def skew_noalloc_selftest_wait_timeout(stream: int) -> None:
    """Makes one bounded device wait run out against the no-alloc status word."""
    rc = load().skew_noalloc_selftest_wait_timeout(stream)
    if rc != SKEW_OK:
        raise SkewError(rc, "CUDA error")


def hparams(beta1=0.9, beta2=0.999, eps=1e-8, clip_d=1.0, weight_decay=0.05, policy=POLICY_TIERED) -> HParams:
    return HParams(beta1, beta2, eps, clip_d, weight_decay, policy)


# --------------------------------------------------------------------------
# torch convenience wrapper
# --------------------------------------------------------------------------
class SkewAdam:
    """SkewAdam over a list of (weight, grad, tier[, flags]) CUDA tensors, bf16 or fp32
    (an fp32 pair, as the paper keeps the norms and the router, is stepped in fp32
    with no dithered cast; F_FP32 is set for it).

    A 3-D tensor (E, n, m) is a stack of E matrices (e.g. an MoE layer's experts
    kept in one array), each stepped with its own second-moment factors and clip
    factor. The optimizer state is one device buffer of exactly ``state_bytes``
    bytes (the paper's closed form); the workspace holds scratch and tables.
    """

    def __init__(self, params: Iterable, hp: HParams, stream=None):
        import torch
        self.torch = torch
        self.params = []
        descs: List[ParamDesc] = []
        for p in params:
            w, g, tier = p[0], p[1], p[2]
            flags = p[3] if len(p) > 3 else 0
            if w.dtype != g.dtype or w.dtype not in (torch.bfloat16, torch.float32):
                raise TypeError("weights and gradients must both be bf16 or both fp32")
            if w.dtype == torch.float32:
                flags |= F_FP32
            if not (w.is_cuda and g.is_cuda and w.is_contiguous() and g.is_contiguous()):
                raise ValueError("weights and gradients must be contiguous CUDA tensors")
            if w.shape != g.shape or w.dim() not in (1, 2, 3):
                raise ValueError("weight / grad shapes must match and be 1-D, 2-D or 3-D")
            if w.dim() == 3:
                shape, stack = (int(w.shape[1]), int(w.shape[2])), int(w.shape[0])
            else:
                shape, stack = (int(w.shape[0]), int(w.shape[1]) if w.dim() == 2 else 0), 0
            descs.append(ParamDesc(w.data_ptr(), g.data_ptr(), (C.c_int64 * 2)(*shape), w.dim(), tier, flags, stack))
            self.params.append((w, g))
        self.hp = hp
        self.h = skew_create(descs, hp)
        dev = self.params[0][0].device if self.params else torch.device("cuda")
        self.state = torch.empty(max(1, skew_state_bytes(self.h)), dtype=torch.uint8, device=dev)
        self.workspace = torch.empty(max(1, skew_workspace_bytes(self.h)), dtype=torch.uint8, device=dev)
        skew_bind(self.h, self.state.data_ptr(), skew_state_bytes(self.h), self.workspace.data_ptr(),
                  skew_workspace_bytes(self.h), self._stream(stream))

    def _stream(self, stream) -> int:
        if stream is None:
            return self.torch.cuda.current_stream().cuda_stream
        return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)

    @property
    def state_bytes(self) -> int:
        return skew_state_bytes(self.h)

    @property
    def workspace_bytes(self) -> int:
        return skew_workspace_bytes(self.h)

    def step(self, step: int, lr: float, seed: int, stream=None, grad_scale=None) -> None:
        """One step. `grad_scale`: optional one-element fp32 device tensor gamma (the trainer's
        global gradient-norm clip factor); the step then sees gamma * G."""
        if grad_scale is None:
            skew_step(self.h, step, lr, seed, self._stream(stream))
            return
        if not (grad_scale.is_cuda and grad_scale.dtype == self.torch.float32 and grad_scale.numel() == 1):
            raise ValueError("grad_scale must be a one-element float32 CUDA tensor")
        skew_step_scaled(self.h, step, lr, seed, grad_scale.data_ptr(), self._stream(stream))

    def sync_status(self, stream=None) -> None:
        skew_sync_status(self.h, self._stream(stream))

    def scalars(self, tid: int, stream=None, matrix: int = 0):
        """mean(R), sum of U^2, RMS and clip factor of tensor `tid` (of its matrix
        `matrix` when it is a stack)."""
        return skew_matrix_scalars(self.h, tid, matrix, self._stream(stream))

    def info(self, tid: int) -> TensorInfo:
        return skew_tensor_info(self.h, tid)

    def state_views(self, tid: int):
        """fp32 views (M, v, R, C; None when absent) into the state buffer."""
        f = self.state[: self.state_bytes].view(self.torch.float32)
        i = self.info(tid)
        out = {}
        E = max(1, i.stack)  # a stack's arrays hold its matrices' in order
        for key, off, cnt in (("M", i.m_offset, i.numel), ("v", i.v_offset, i.numel), ("R", i.r_offset, E * i.rows),
                              ("C", i.c_offset, E * i.cols)):
            out[key] = None if off < 0 else f[off: off + cnt]
        return out

    def close(self):
        if getattr(self, "h", None):
            skew_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
