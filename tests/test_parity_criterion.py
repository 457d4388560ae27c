"""The GPU-vs-oracle weight criterion itself (CPU): legitimate dither-threshold
flips and cancellation are accepted; a wrong draw or a wrong update is not."""
import numpy as np
import pytest

import oracle as O
import parity as P


def _case(n=4096, seed=0):
    rng = np.random.default_rng(seed)
    w = rng.normal(0, 0.02, n).astype(np.float32)
    w_bits = ((w.view(np.uint32) + 0x8000) >> 16).astype(np.uint16)
    wf = (w_bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    upd = rng.normal(0, 1e-3, n)
    x = (wf - upd).astype(np.float32)
    r = O.dither16(7, 1, 0, 0, n)
    return w_bits, x, r, O.sr_bf16(x, r)


def test_identical_passes():
    w, x, r, out = _case()
    assert P.compare_weights(out.copy(), out, x, r, w, 1.0, "t") == (0, 0.0)


def test_threshold_flip_passes():
    w, x, r, out = _case()
    low = x.view(np.uint32) & 0xFFFF
    k = int(np.argmin(np.abs(low.astype(np.int64) + r - 65536)))   # the element closest to its threshold
    g = out.copy()
    up = int(low[k]) + int(r[k]) >= 65536
    g[k] = out[k] - 1 if up else out[k] + 1
    n, worst = P.compare_weights(g, out, x, r, w, 1.0, "t")
    assert n == 1 and worst <= P.X_RTOL


def test_wrong_draw_fails():
    w, x, r, out = _case()
    r2 = r.copy()
    r2[::97] ^= 0x8000                                     # planted: wrong dither bits
    g = O.sr_bf16(x, r2)
    with pytest.raises(AssertionError):
        P.compare_weights(g, out, x, r, w, 1.0, "t")


def test_wrong_update_fails():
    w, x, r, out = _case()
    x2 = (x.astype(np.float64) * (1 + 1e-4)).astype(np.float32)   # planted: update off by 1e-4 relative
    g = O.sr_bf16(x2, r)
    with pytest.raises(AssertionError):
        P.compare_weights(g, out, x, r, w, 1.0, "t")


def test_two_ulp_far_from_threshold_fails():
    w, x, r, out = _case()
    low = x.view(np.uint32) & 0xFFFF
    k = int(np.argmax(np.abs(low.astype(np.int64) + r - 65536)))
    g = out.copy()
    g[k] = out[k] + 2
    with pytest.raises(AssertionError):
        P.compare_weights(g, out, x, r, w, 1.0, "t")
