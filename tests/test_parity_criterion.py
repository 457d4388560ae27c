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
    assert P.compare_weights(out.copy(), out, x, r, w, 1.0, "t") == (0, 0.0, 0)


def test_threshold_flip_passes():
    w, x, r, out = _case()
    low = x.view(np.uint32) & 0xFFFF
    k = int(np.argmin(np.abs(low.astype(np.int64) + r - 65536)))   # the element closest to its threshold
    g = out.copy()
    up = int(low[k]) + int(r[k]) >= 65536
    g[k] = out[k] - 1 if up else out[k] + 1
    n, worst, widened = P.compare_weights(g, out, x, r, w, 1.0, "t")
    assert n == 1 and worst <= P.X_RTOL and widened == 0      # within 1e-6 |x| of the threshold


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


def test_cancelling_element_counts_as_widened():
    """An element whose update nearly cancels its weight (x ~ 1e-4 S): a GPU value a few
    ulps of x away passes within 1e-6 S but not within 1e-6 |x|, and is counted."""
    w, x, r, out = _case()
    k = 5
    wf = float((w[k].astype(np.uint32) << 16).view(np.float32))
    xk = np.float32(wf * 1e-4)                        # the update cancels all but 1e-4 of w
    x = x.copy()
    x[k] = xk
    out = O.sr_bf16(x, r)
    g = out.copy()
    g[k] = out[k] + 1   # one bf16 ulp of x: ~4e-3 |x|, ~2e-7 S
    n, worst, widened = P.compare_weights(g, out, x, r, w, 1.0, "t")
    assert n == 1 and worst <= P.X_RTOL and widened == 1


def _round_f32_exact(v):
    """Round-to-nearest-even of a Fraction to fp32 (normal range), by integer arithmetic."""
    from fractions import Fraction
    if v == 0:
        return np.float32(0.0)
    sign = -1 if v < 0 else 1
    v = abs(v)
    e = v.numerator.bit_length() - v.denominator.bit_length()
    while Fraction(2) ** e > v:
        e -= 1
    while Fraction(2) ** (e + 1) <= v:
        e += 1
    scale = Fraction(2) ** (23 - e)
    q = v * scale
    n = q.numerator // q.denominator
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    return np.float32(sign * float(Fraction(n) / scale))


def test_fma_f32_emulation_is_exact():
    """The harness's fp32 FMA (used to explain momenta that pass only through reading R17)
    equals exact rational arithmetic rounded to fp32: on near-cancelling random inputs and
    on inputs whose exact sum lies just off an fp32 rounding midpoint that fp64 rounds onto."""
    from fractions import Fraction
    rng = np.random.default_rng(12)
    n = 3000
    a = rng.normal(0, 1, n).astype(np.float32)
    b = rng.normal(0, 1, n).astype(np.float32)
    c = (-(a.astype(np.float64) * b) * (1 + rng.normal(0, 1e-6, n))).astype(np.float32)
    # midpoint cases: c = x, a*b = (half an fp32 ulp of x) * (1 - 2^-40): the exact sum is just
    # below the midpoint between x and its upper neighbour, and fp64 rounds it onto the midpoint
    x = rng.uniform(1, 2, 200).astype(np.float32) * np.float32(2.0) ** rng.integers(-20, 20, 200).astype(np.float32)
    x = np.where(rng.integers(0, 2, 200) == 1, x, -x).astype(np.float32)
    half = (np.nextafter(np.abs(x), np.float32(np.inf)).astype(np.float64) - np.abs(x).astype(np.float64)) / 2
    am = (np.sign(x) * half * (1 + 2.0 ** -20)).astype(np.float32)
    bm = np.full(200, 1 - 2.0 ** -20, np.float32)
    a, b, c = np.concatenate([a, am]), np.concatenate([b, bm]), np.concatenate([c, x])
    got = P.fma_f32(a, b, c)
    want = np.array([_round_f32_exact(Fraction(float(p)) * Fraction(float(q)) + Fraction(float(r)))
                     for p, q, r in zip(a, b, c)], np.float32)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    # the midpoint cases do take the correction (plain fp32(fl64(.)) would be wrong there)
    s = am.astype(np.float64) * bm + x
    assert np.count_nonzero(s.astype(np.float32).view(np.uint32) != want[n:].view(np.uint32)) > 0


def test_state_in_the_fp32_subnormal_range_needs_an_absolute_floor():
    """Reading R24: for gradients ~1e-20, g^2 ~ 1e-40 and (1 - beta2) * mean(g^2) ~ 1e-43
    are fp32 subnormals, spaced 2^-149 apart. Evaluated in fp32 in the kernels' order
    (each square rounded, an fp32 sum, the mean, the scale by 1 - beta2, the moving
    average), a row's R differs from the fp64 value rounded once by more than 1e-5
    relative on some rows, yet by at most a few subnormal steps on every row; the same
    holds for the elementwise v = fma(beta2, 0, (1 - beta2) g^2)."""
    rng = np.random.default_rng(13)
    rows, m = 2000, 4096
    g = (rng.normal(0, 1, (rows, m)) * 1e-20).astype(np.float32)
    b2 = np.float32(0.999)
    c2 = np.float32(1.0 - float(b2))
    exact = (float(c2) * (g.astype(np.float64) ** 2).mean(axis=1)).astype(np.float32)
    sq = g * g                                                    # fp32 subnormal squares
    mean = np.float32(sq.sum(axis=1, dtype=np.float32) * np.float32(1.0 / m))
    f32 = P.fma_f32(np.full(rows, b2), np.zeros(rows, np.float32), c2 * mean)
    d = np.abs(f32.astype(np.float64) - exact.astype(np.float64))
    assert float(exact.max()) < 2.0 ** -126                            # all subnormal
    assert np.count_nonzero(d > P.STATE_RTOL * np.abs(exact.astype(np.float64))) > 0
    assert float(d.max()) <= P.STATE_ATOL
    ge = g[0]
    v_exact = (float(c2) * ge.astype(np.float64) ** 2).astype(np.float32)
    v_f32 = P.fma_f32(np.full(m, b2), np.zeros(m, np.float32), c2 * (ge * ge))
    dv = np.abs(v_f32.astype(np.float64) - v_exact.astype(np.float64))
    assert np.count_nonzero(dv > P.STATE_RTOL * np.abs(v_exact.astype(np.float64))) > 0
    assert float(dv.max()) <= P.STATE_ATOL


def test_cancelling_momenta_are_explained_bit_for_bit():
    """Reading R17's momenta (cancelling far below their terms) pass only as fp32's
    fma(b1, M_prev, fl(c1 g)): the fp32 evaluation is accepted and counted as explained, a
    value one fp32 ulp away from it (still within the terms-relative bar) is counted as
    unexplained, and gamma scales c1 as the kernels do."""
    rng = np.random.default_rng(31)
    n = 20000
    b1 = float(np.float32(0.9))
    gb = (rng.normal(0, 1e-3, n).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    gv = P.as_f64(gb)
    for gam in (1.0, 0.37):
        c1 = np.float32(np.float32(1.0 - b1) * np.float32(gam))
        # M_prev close to -(1 - b1) gamma g / b1, so that M cancels to a few fp32 ulps of the terms
        m_prev = (-(1 - b1) * gam * gv / b1 * (1 + rng.normal(0, 1e-7, n))).astype(np.float32)
        gpu = P.fma_f32(np.full(n, np.float32(b1)), m_prev, c1 * gv.astype(np.float32))
        ora = b1 * m_prev.astype(np.float64) + (1 - b1) * gam * gv
        err, wid, unex = P.check_momentum(gpu, ora, m_prev, gb, b1, gam)
        assert err <= P.STATE_RTOL and wid > 100 and unex == 0, (gam, err, wid, unex)
        # plant a one-ulp error on a widened element
        scale = b1 * np.abs(m_prev.astype(np.float64)) + (1 - b1) * np.abs(gam * gv)
        k = int(P.widened_terms(gpu, ora, scale, P.STATE_RTOL)[0])
        bad = gpu.copy()
        bad[k] = np.nextafter(bad[k], np.float32(np.inf))
        err2, wid2, unex2 = P.check_momentum(bad, ora, m_prev, gb, b1, gam)
        assert err2 <= P.STATE_RTOL and unex2 == 1, (gam, err2, wid2, unex2)
    # the unscaled c1 is wrong for gamma != 1
    err, wid, unex = P.check_momentum(gpu, ora, m_prev, gb, b1, 1.0)
    assert unex > 0 or err > P.STATE_RTOL


def test_state_floor_counts():
    a = np.array([1e-43, 1.0, 0.0], np.float32)
    b = np.array([1.0089348943138683e-43, 1.0, 0.0], np.float32)
    assert P.floor_only(a, b) == (1 if a[0] != b[0] else 0)
    assert P.rel_err(a, b) <= P.STATE_RTOL
    assert P.rel_err(np.array([1e-40], np.float32), np.array([1.1e-40], np.float32)) > P.STATE_RTOL
