"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test names the passage it follows. None of them re-types the oracle's own
formula: they check closed forms, exact identities, the paper's printed numbers
and independent implementations (a second, separately written Philox and the
one that ships with triton).
"""
import math
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest

import oracle as O
from paper_2607_19058_gb300 import workloads as WL

F32 = np.float32
B1, B2 = float(F32(0.9)), float(F32(0.999))


def _bf16(x):
    """fp32 -> bf16 bits by round-to-nearest-even (test-side conversion)."""
    b = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return b.astype(np.uint16)


def _f(bits):
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def _hp(eps=1e-30, d=1.0, wd=0.1):
    return O.hparams(0.9, 0.999, eps, d, wd)


# --------------------------------------------------------------------------
# P1: closed-form state bytes vs Table 5, Table 3, Fig. 1, Sec. 3 "Memory model"
# --------------------------------------------------------------------------
def _specs(wl):
    return [(s.shape, s.tier) for s in wl.specs]


def test_state_bytes_table5_total():
    """Table 5 / Table 1: SkewAdam state 1.29 GB (GiB) on the App. B shapes."""
    wl = WL.appb()
    assert wl.numel == 6_784_327_680                        # App. B: 6,784.3M
    S = O.state_bytes(_specs(wl), O.POLICY_TIERED)
    assert S == 1_380_800_000
    assert round(S / 2**30, 2) == 1.29


def test_state_bytes_table5_components():
    """Table 5 rows: 1,302.2 / 0.5 / 0.2 / 12.0 / 2.0 MB (MiB)."""
    wl = WL.appb()
    bb = [s for s in wl.specs if s.tier == WL.TIER_BACKBONE]
    ex = [s for s in wl.specs if s.tier == WL.TIER_EXPERT]
    rt = [s for s in wl.specs if s.tier == WL.TIER_ROUTER]
    mib = lambda b: b / 2**20
    n_bb = sum(s.numel for s in bb)
    assert round(n_bb / 1e6, 1) == 341.4
    assert round(mib(4 * n_bb), 1) == 1302.2
    bb_mats = [s for s in bb if len(s.shape) == 2]
    bb_vecs = [s for s in bb if len(s.shape) == 1]
    assert round(mib(4 * sum(s.shape[0] + s.shape[1] for s in bb_mats)), 1) == 0.5
    assert round(sum(s.numel for s in bb_vecs) / 1e6, 2) == 0.04
    assert round(mib(4 * sum(s.numel for s in bb_vecs)), 1) == 0.2
    assert round(mib(4 * sum(s.shape[0] + s.shape[1] for s in ex)), 1) == 12.0
    assert round(mib(4 * sum(s.numel for s in rt)), 1) == 2.0
    # the oracle's per-tier sums add up to the same components
    parts = [O.state_bytes([(s.shape, s.tier)]) for s in wl.specs]
    assert sum(parts) == O.state_bytes(_specs(wl))


def test_state_bytes_adamw_and_fig1():
    """Table 5 last row (AdamW 8N = 50.55 GB) and Fig. 1's per-tier figures."""
    wl = WL.appb()
    assert round(8 * wl.numel / 2**30, 2) == 50.55
    tiers = {t: sum(s.numel for s in wl.specs if s.tier == t) for t in (0, 1, 2)}
    assert round(tiers[0] / 1e6) == 341 and round(tiers[1] / 1e6) == 6442 and round(tiers[2] / 1e6, 1) == 0.5
    assert round(100 * tiers[1] / wl.numel, 1) == 95.0
    assert round(4 * tiers[0] / 2**30, 2) == 1.27                      # m: 1.27 GB
    ex_rc = 4 * sum(s.shape[0] + s.shape[1] for s in wl.specs if s.tier == 1)
    assert round(ex_rc / 1e6, 1) == 12.6                               # experts V 12.6 MB
    assert round(4 * tiers[2] / 1e6, 1) == 2.1                          # router V 2.1 MB


def test_state_bytes_table3_variants():
    """Table 3: +expert momentum 25.29 GB, factored router 1.28 GB, uniform 25.29 GB."""
    sp = _specs(WL.appb())
    em = O.state_bytes(sp, O.POLICY_EXPERT_MOMENTUM)
    fr = O.state_bytes(sp, O.POLICY_FACTORED_ROUTER)
    un = O.state_bytes(sp, O.POLICY_UNIFORM)
    assert em == 27_150_603_776 and round(em / 2**30, 2) == 25.29
    assert fr == 1_378_719_744 and round(fr / 2**30, 2) == 1.28
    assert round(un / 2**30, 2) == 25.29


def test_state_bytes_adafactor():
    """Sec. 5 / Table 4: uniform Adafactor carries about 12 MB (0.01 GB): R and C of every
    matrix (the router's too) and the vectors' full v, no momentum. Hand sum over the App. B
    shapes: 384 experts, embedding, positions, 2 x attention, dense FFN, router, 10 vectors."""
    ad = O.state_bytes(_specs(WL.appb()), O.POLICY_ADAFACTOR)
    want = 4 * (384 * (4096 + 4096) + (50304 + 4096) + (256 + 4096) + 2 * (2 * 8192 + 2 * 5120)
                + 3 * 8192 + (4096 + 128) + 10 * 4096)
    assert ad == want == 13_309_952
    assert round(ad / 1e9, 2) == 0.01 and 12 <= ad / 2**20 < 13


def test_adafactor_annealed_decay_closed_forms():
    """Adafactor comparator (Sec. 5 footnote: decay 1 - t^-0.8; App. A: no momentum; no bias
    correction). beta2_1 = 0, so at t = 1 a vector's v is g^2 and U = sign(g). A zero gradient
    at t = 1 and g at t = 2 give v = (1 - beta2_2) g^2 with 1 - beta2_2 ~ 2^-0.8: U = g / sqrt(v),
    RMS = 1/sqrt(1 - beta2_2) ~ 2^0.4 > 1, and the clip turns the update into sign(g)."""
    rng = np.random.default_rng(12)
    n = 512
    g = _bf16(rng.normal(0, 1e-3, n).astype(np.float32))
    g[g == 0] = _bf16(np.float32(1e-3))
    w = _bf16(rng.normal(0, 0.02, n).astype(np.float32))
    lr = float(F32(1e-3))
    hp = O.hparams(0.9, 0.999, 1e-30, 1.0, 0.0, annealed=True)
    gd = _f(g).astype(np.float64)
    st = O.TensorState((n,), O.TIER_BACKBONE, O.POLICY_ADAFACTOR)
    assert st.momentum == 0 and st.kind == O.KIND_FULL
    w1 = w.copy()
    o = O.tensor_step(w1, g, st, 0, hp, 1, lr, 3, want_x=True)
    assert np.array_equal(st.v, (gd * gd).astype(np.float32))
    assert abs(o["rms"] - 1.0) < 1e-7 and o["kappa"] == 1.0
    want = (_f(w).astype(np.float64) - lr * np.sign(gd)).astype(np.float32)
    assert np.max(np.abs(o["x"].astype(np.float64) - want)) <= 4e-7 * lr + np.spacing(want).max()
    # t = 1 with a zero gradient, t = 2 with g
    st = O.TensorState((n,), O.TIER_BACKBONE, O.POLICY_ADAFACTOR)
    w2 = w.copy()
    O.tensor_step(w2, np.zeros_like(g), st, 0, hp, 1, lr, 3)
    w2_pre = w2.copy()
    o = O.tensor_step(w2, g, st, 0, hp, 2, lr, 3, want_x=True)
    c2 = 1.0 - float(np.float32(1.0 - 2.0 ** -0.8))
    assert abs(c2 - 2.0 ** -0.8) < 1e-7
    assert np.array_equal(st.v, (c2 * gd * gd).astype(np.float32))
    assert abs(o["rms"] - 1.0 / np.sqrt(c2)) < 2e-7 * o["rms"]
    assert abs(o["kappa"] - np.sqrt(c2)) < 2e-7
    want = (_f(w2_pre).astype(np.float64) - lr * np.sign(gd)).astype(np.float32)
    assert np.max(np.abs(o["x"].astype(np.float64) - want)) <= 4e-7 * lr + np.spacing(want).max()


def test_state_bytes_other_shape_sets():
    """Hand-summed closed form for the toy, slice, literal and ablation sets."""
    assert O.state_bytes(_specs(WL.toy())) == 356_096
    assert O.state_bytes(_specs(WL.slice_())) == 278_593_536
    assert O.state_bytes(_specs(WL.literal())) == 2_687_972_352
    ab = WL.ablation()
    assert O.state_bytes(_specs(ab), ab.hp.policy) == 27_166_250_308


def test_tier_policy():
    """Sec. 3 'The tiers' + Algorithm 1: (kind, momentum, decay) per tier."""
    FULL, FACT = O.KIND_FULL, O.KIND_FACTORED
    assert O.resolve(2, O.TIER_BACKBONE) == (FACT, 1, 1)
    assert O.resolve(1, O.TIER_BACKBONE) == (FULL, 1, 1)
    assert O.resolve(2, O.TIER_EXPERT) == (FACT, 0, 1)
    assert O.resolve(2, O.TIER_ROUTER) == (FULL, 0, 0)
    assert O.resolve(2, O.TIER_EXPERT, O.POLICY_EXPERT_MOMENTUM) == (FACT, 1, 1)
    assert O.resolve(2, O.TIER_ROUTER, O.POLICY_FACTORED_ROUTER) == (FACT, 0, 0)
    assert O.resolve(2, O.TIER_ROUTER, O.POLICY_UNIFORM) == (FACT, 1, 0)
    assert O.resolve(2, O.TIER_EXPERT, no_decay=True) == (FACT, 0, 0)
    # the Adafactor comparator (Sec. 5, App. A): every matrix factored, no momentum anywhere
    AD = O.POLICY_ADAFACTOR
    assert O.resolve(2, O.TIER_BACKBONE, AD) == (FACT, 0, 1)
    assert O.resolve(1, O.TIER_BACKBONE, AD) == (FULL, 0, 1)
    assert O.resolve(2, O.TIER_EXPERT, AD) == (FACT, 0, 1)
    assert O.resolve(2, O.TIER_ROUTER, AD) == (FACT, 0, 0)
    with pytest.raises(ValueError):
        O.resolve(3, O.TIER_EXPERT)
    with pytest.raises(ValueError):
        O.resolve(2, O.TIER_EXPERT, 5)


# --------------------------------------------------------------------------
# Philox / dither: independent implementations and determinism
# --------------------------------------------------------------------------
def _philox_py(ctr, key):
    """Philox-4x32-10, written separately from the oracle from SC'11's description."""
    M = (0xD2511F53, 0xCD9E8D57)
    W = (0x9E3779B9, 0xBB67AE85)
    x = list(ctr)
    k = list(key)
    for r in range(10):
        a = M[0] * x[0]
        b = M[1] * x[2]
        x = [((b >> 32) ^ x[1] ^ k[0]) & 0xFFFFFFFF, b & 0xFFFFFFFF,
             ((a >> 32) ^ x[3] ^ k[1]) & 0xFFFFFFFF, a & 0xFFFFFFFF]
        k = [(k[0] + W[0]) & 0xFFFFFFFF, (k[1] + W[1]) & 0xFFFFFFFF]
    return x


def test_philox_matches_python_restatement():
    rng = np.random.default_rng(1)
    for _ in range(200):
        ctr = [int(v) for v in rng.integers(0, 2**32, 4)]
        key = [int(v) for v in rng.integers(0, 2**32, 2)]
        assert O.philox4x32_10(ctr, key) == _philox_py(ctr, key)
    assert O.philox4x32_10([0] * 4, [0] * 2) == _philox_py([0] * 4, [0] * 2)


def test_philox_matches_triton():
    """Cross-check against triton's Philox-4x32 (CPU interpreter, in a subprocess)."""
    pytest.importorskip("triton")
    code = textwrap.dedent("""
        import os, sys, json
        os.environ["TRITON_INTERPRET"] = "1"
        import torch, triton, triton.language as tl
        @triton.jit
        def k(c_ptr, o_ptr, seed, N: tl.constexpr):
            i = tl.arange(0, N)
            c0 = tl.load(c_ptr + i * 4 + 0); c1 = tl.load(c_ptr + i * 4 + 1)
            c2 = tl.load(c_ptr + i * 4 + 2); c3 = tl.load(c_ptr + i * 4 + 3)
            a, b, c, d = tl.philox(seed, c0, c1, c2, c3, 10)
            tl.store(o_ptr + i * 4 + 0, a); tl.store(o_ptr + i * 4 + 1, b)
            tl.store(o_ptr + i * 4 + 2, c); tl.store(o_ptr + i * 4 + 3, d)
        ctr = json.loads(sys.argv[1]); seed = int(sys.argv[2])
        c = torch.tensor(ctr, dtype=torch.int64).to(torch.int32)
        o = torch.zeros_like(c)
        k[(1,)](c, o, seed, len(ctr) // 4)
        print(json.dumps([x & 0xFFFFFFFF for x in o.tolist()]))
    """)
    rng = np.random.default_rng(7)
    ctr = [int(v) for v in rng.integers(0, 2**32, 4 * 16)]
    ctr = [v - 2**32 if v >= 2**31 else v for v in ctr]
    seed = 0x0123456789ABCDEF
    env = dict(os.environ, TRITON_INTERPRET="1")
    out = subprocess.run([sys.executable, "-c", code, str(ctr), str(seed)], capture_output=True,
                         text=True, env=env, timeout=300)
    if out.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + out.stderr[-300:])
    import json
    got = json.loads(out.stdout.strip().splitlines()[-1])
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for q in range(16):
        c = [x & 0xFFFFFFFF for x in ctr[4 * q:4 * q + 4]]
        assert got[4 * q:4 * q + 4] == O.philox4x32_10(c, key)


def test_dither_counter_layout():
    """The dither of element idx is half (idx&1) of word (idx&7)>>1 of the block idx>>3."""
    seed, step, tid = 0xDEADBEEFCAFEF00D, 123456, 77
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for idx in [0, 1, 7, 8, 15, 2**31 + 5, 2**35 + 3, 6_442_450_943]:
        blk = idx >> 3
        o = _philox_py([blk & 0xFFFFFFFF, blk >> 32, tid, step & 0xFFFFFFFF], key)
        k = idx & 7
        want = (o[k >> 1] >> (16 * (k & 1))) & 0xFFFF
        assert int(O.dither16(seed, step, tid, idx, 1)[0]) == want


def test_dither_golden():
    """Frozen dither bits (written once by tests/golden/make_goldens.py from the oracle)."""
    path = os.path.join(os.path.dirname(__file__), "golden", "dither16.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    assert len(rows) >= 16
    for seed, step, tid, idx0, *vals in rows:
        got = O.dither16(int(seed, 0), int(step), int(tid), int(idx0), len(vals))
        assert [int(v, 16) for v in vals] == [int(x) for x in got]


def test_dither_index_of_a_stacked_matrix():
    """Matrix e of a stacked (E, n, m) tensor draws the dithers of its flat position
    e*n*m + k in the stack (Sec. 3 dithered write-back, the index running over the
    whole array). An elementwise tier with no clip makes the two halves of a (2n, m)
    tensor independent, so stepping them as two stacked matrices must reproduce the
    whole tensor's step bit for bit; n*m = 222 starts the second half inside a block."""
    rng = np.random.default_rng(21)
    n, m = 6, 37
    g = _bf16(rng.normal(0, 1e-3, (2 * n, m)).astype(np.float32)).reshape(-1)
    w = _bf16(rng.normal(0, 0.02, (2 * n, m)).astype(np.float32)).reshape(-1)
    hp, lr = _hp(d=1e30), float(F32(1e-3))
    whole = w.copy()
    O.tensor_step(whole, g, O.TensorState((2 * n, m), O.TIER_ROUTER), 3, hp, 1, lr, 5)
    for idx0, want_equal in ((lambda e: e * n * m, True), (lambda e: 0, False)):
        halves = []
        for e in range(2):
            we = w[e * n * m:(e + 1) * n * m].copy()
            O.tensor_step(we, g[e * n * m:(e + 1) * n * m].copy(), O.TensorState((n, m), O.TIER_ROUTER), 3, hp, 1,
                          lr, 5, idx0=idx0(e))
            halves.append(we)
        assert np.array_equal(np.concatenate(halves), whole) == want_equal


def test_dither_uniform_chi2():
    """The 16-bit draws are uniform: chi-square over 256 bins of the top byte and the low byte."""
    r = O.dither16(42, 7, 3, 0, 1 << 20).astype(np.int64)
    for vals in (r >> 8, r & 0xFF):
        cnt = np.bincount(vals, minlength=256)
        exp = r.size / 256
        chi2 = float(((cnt - exp) ** 2 / exp).sum())
        assert 150 < chi2 < 380   # 255 dof: mean 255, sd 22.6


# --------------------------------------------------------------------------
# P5: the dithered rounding is unbiased (Sec. 3)
# --------------------------------------------------------------------------
def test_sr_exact_expectation_over_all_draws():
    """Averaging SR(x, r) over every r in [0, 2^16) returns x exactly (finite x)."""
    rng = np.random.default_rng(3)
    xs = np.concatenate([rng.normal(0, 1, 64), rng.normal(0, 1e-30, 8), -rng.uniform(1, 2, 8),
                         [1e-40, -3e-42, 0.0, -0.0, 3.0e38]]).astype(np.float32)
    r = np.arange(65536, dtype=np.uint16)
    for x in xs:
        out = O.sr_bf16(np.full(65536, x, np.float32), r)
        vals = _f(out).astype(np.float64)
        assert math.fsum(vals) / 65536 == float(x), x


def test_sr_round_up_probability_and_specials():
    rng = np.random.default_rng(4)
    xs = rng.normal(0, 1, 32).astype(np.float32)
    for x in xs:
        b = int(np.float32(x).view(np.uint32))
        low = b & 0xFFFF
        r = np.arange(65536, dtype=np.uint16)
        out = O.sr_bf16(np.full(65536, x, np.float32), r).astype(np.int64)
        ups = int((out != (b >> 16)).sum())
        assert ups == low                             # P(round up) = low16 / 2^16 exactly
        assert set(np.unique(out)) <= {b >> 16, (b >> 16) + 1}
    one = np.ones(1, np.uint16)
    assert O.sr_bf16(np.array([np.inf], np.float32), one * 65535)[0] == 0x7F80
    assert O.sr_bf16(np.array([-np.inf], np.float32), one * 65535)[0] == 0xFF80
    assert O.sr_bf16(np.array([np.nan], np.float32), one)[0] == 0x7FC0
    assert O.sr_bf16(-np.array([np.nan], np.float32), one)[0] == 0xFFC0
    big = np.array([np.float32(3.4e38)], np.float32)    # above bf16 max: rounds to Inf or max
    outs = set(O.sr_bf16(np.repeat(big, 65536), np.arange(65536, dtype=np.uint16)).tolist())
    assert outs == {0x7F7F, 0x7F80}


def test_sr_mean_over_seeds_converges():
    """The mean of bf16(SR(x)) over many dithers of the real hash tends to x (~ulp/sqrt(K))."""
    K = 1 << 14
    rng = np.random.default_rng(5)
    x = rng.normal(0, 0.02, 64).astype(np.float32)
    acc = np.zeros(64)
    for s in range(K // 64):
        r = O.dither16(1000 + s, 1, 0, 0, 64 * 64).reshape(64, 64)
        acc += _f(O.sr_bf16(np.repeat(x[None], 64, 0), r)).astype(np.float64).sum(0)
    mean = acc / K
    ulp = np.abs(_f(_bf16(x) + 1).astype(np.float64) - _f(_bf16(x)).astype(np.float64))
    assert np.all(np.abs(mean - x) <= 5 * ulp / math.sqrt(K) + 1e-12)


# --------------------------------------------------------------------------
# Algorithm 1 special cases and closed forms
# --------------------------------------------------------------------------
def _run(shape, tier, g, w, steps, policy=O.POLICY_TIERED, hp=None, lr=1e-3, seed=9, want_x=True):
    st = O.TensorState(shape, tier, policy)
    w = w.copy()
    outs = []
    for t, gt in enumerate(g, start=1):
        outs.append(O.tensor_step(w, gt, st, 0, hp or _hp(), t, lr, seed, want_x=want_x))
    return st, w, outs


def test_step1_full_v_gives_sign():
    """Full v at t=1 with tiny eps: U = sign(g) for momentum-free and momentum tiers (Alg. 1)."""
    rng = np.random.default_rng(6)
    shape = (64, 8)
    g = _bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1)
    g[::7] = 0
    w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
    lr = float(F32(1e-3))
    for tier, shp in ((O.TIER_ROUTER, shape), (O.TIER_BACKBONE, (512,))):
        st, _, outs = _run(shp, tier, [g], w, 1)
        o = outs[0]
        frac = np.count_nonzero(_f(g)) / g.size
        assert abs(o["rms"] - math.sqrt(frac)) < 1e-6
        assert o["kappa"] == 1.0
        lam = 0.0 if tier == O.TIER_ROUTER else float(F32(0.1))
        want = (_f(w).astype(np.float64) * (1 - lr * lam) - lr * np.sign(_f(g))).astype(np.float32)
        assert np.max(np.abs(o["x"].astype(np.float64) - want)) <= 4e-7 * lr + np.spacing(want).max()


def test_fp32_tensor_step1_and_bf16_agreement():
    """fp32 norms and router (App. A): the new weight is the fp32 x itself (no dithered cast).
    Step 1 on an fp32 vector gives U = sign(g) (Algorithm 1, full v); on inputs that are
    exactly bf16 values, an fp32 tensor and a bf16 tensor see the same x and state, and the
    bf16 tensor's weight is the dithered rounding of that x."""
    rng = np.random.default_rng(31)
    n = 777
    gb = _bf16(rng.normal(0, 1e-3, n).astype(np.float32))
    gb[::9] = 0
    wb = _bf16(rng.normal(0, 0.02, n).astype(np.float32))
    lr = float(F32(1e-3))
    gf, wf = _f(gb), _f(wb)  # fp32 copies of the same values
    for tier, shape in ((O.TIER_BACKBONE, (n,)), (O.TIER_ROUTER, (7, 111))):
        sf, sb = O.TensorState(shape, tier), O.TensorState(shape, tier)
        w32, w16 = wf.copy(), wb.copy()
        for t in (1, 2):
            of = O.tensor_step(w32, gf, sf, 5, _hp(), t, lr, 8, want_x=True)
            ob = O.tensor_step(w16, gb, sb, 5, _hp(), t, lr, 8, want_x=True)
            assert np.array_equal(w32.view(np.uint32), of["x"].view(np.uint32))   # stored as is
            assert not of["r"].any()
            if t == 1:  # x of step 1 is the bf16 path's x (same inputs, same state)
                assert np.array_equal(of["x"].view(np.uint32), ob["x"].view(np.uint32))
                for key in ("M", "v", "R", "C"):
                    if getattr(sf, key) is not None:
                        assert np.array_equal(getattr(sf, key), getattr(sb, key))
                assert np.array_equal(w16, O.sr_bf16(ob["x"], ob["r"]))
                if tier == O.TIER_BACKBONE:  # Algorithm 1, full v at t = 1: U = sign(g)
                    lam = float(F32(0.1))
                    want = (wf.astype(np.float64) * (1 - lr * lam) - lr * np.sign(gf)).astype(np.float32)
                    assert np.max(np.abs(of["x"].astype(np.float64) - want)) <= 4e-7 * lr + np.spacing(want).max()
            w16 = _bf16(w32)  # keep both paths on the same weights for the next step
            w32 = _f(w16).copy()


def test_clip_closed_form():
    """Zero grad at t=1 then g at t=2 on the full path: RMS = sqrt(1+beta2), update = sign(g)."""
    rng = np.random.default_rng(8)
    shape = (32, 16)
    g2 = _bf16(rng.choice([-1, 1], shape) * rng.uniform(1e-4, 1e-2, shape).astype(np.float32)).reshape(-1)
    g1 = np.zeros_like(g2)
    w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
    lr = float(F32(1e-3))
    st, _, outs = _run(shape, O.TIER_ROUTER, [g1, g2], w, 2)
    assert outs[0]["rms"] == 0.0 and outs[0]["kappa"] == 1.0
    assert abs(outs[1]["rms"] - math.sqrt(1 + B2)) < 1e-6
    assert abs(outs[1]["kappa"] - 1 / math.sqrt(1 + B2)) < 1e-6
    w1 = _f(O.sr_bf16(outs[0]["x"], outs[0]["r"])).astype(np.float64)
    want = w1 - lr * np.sign(_f(g2))
    assert np.allclose(outs[1]["x"], want, rtol=0, atol=2 * lr * 1e-6 + 1e-9)


def test_momentum_step2_closed_form():
    """Backbone vector, g at t=1 then zero: U_2 = sign(g) b1 sqrt(1+b2) / ((1+b1) sqrt(b2))."""
    rng = np.random.default_rng(9)
    g1 = _bf16(rng.choice([-1, 1], 256) * rng.uniform(1e-4, 1e-2, 256).astype(np.float32))
    w = _bf16(rng.normal(0, 0.02, 256).astype(np.float32))
    st, _, outs = _run((256,), O.TIER_BACKBONE, [g1, np.zeros_like(g1)], w, 2, hp=_hp(wd=0.0))
    u2 = B1 * math.sqrt(1 + B2) / ((1 + B1) * math.sqrt(B2))
    assert abs(outs[1]["rms"] - u2) < 1e-6
    assert outs[1]["kappa"] == 1.0   # u2 < 1
    # the state itself: M_2 = b1 (1-b1) g, v_2 = b2 (1-b2) g^2 (fp32-rounded twice)
    gd = _f(g1).astype(np.float64)
    assert np.allclose(st.M, B1 * (1 - B1) * gd, rtol=2e-7, atol=0)
    assert np.allclose(st.v, B2 * (1 - B2) * gd * gd, rtol=2e-7, atol=0)


def test_zero_grad_pure_decay():
    """P4: zero gradients multiply R, C, v by beta2 and M by beta1; U = 0 on momentum-free tiers."""
    rng = np.random.default_rng(10)
    lr = float(F32(1e-3))
    lam = float(F32(0.1))
    for shape, tier in (((48, 40), O.TIER_EXPERT), ((48, 40), O.TIER_BACKBONE), ((40, 8), O.TIER_ROUTER),
                        ((96,), O.TIER_BACKBONE)):
        g = _bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1)
        w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
        st = O.TensorState(shape, tier)
        O.tensor_step(w, g, st, 0, _hp(), 1, lr, 1)
        before = {k: (None if a is None else a.copy()) for k, a in
                  (("M", st.M), ("v", st.v), ("R", st.R), ("C", st.C))}
        wb = w.copy()
        o = O.tensor_step(w, np.zeros_like(g), st, 0, _hp(), 2, lr, 1, want_x=True)
        for k, beta in (("v", B2), ("R", B2), ("C", B2), ("M", B1)):
            if before[k] is not None:
                want = (beta * before[k].astype(np.float64)).astype(np.float32)
                assert np.array_equal(getattr(st, k), want), (shape, tier, k)
        if tier in (O.TIER_EXPERT, O.TIER_ROUTER):
            l = 0.0 if tier == O.TIER_ROUTER else lam
            want_x = (_f(wb).astype(np.float64) * (1 - lr * l)).astype(np.float32)
            assert np.array_equal(o["x"], want_x)
            assert o["sumu2"] == 0.0


def test_zero_grad_expert_at_step1_rbar_zero():
    """An expert that saw no tokens at t=1: R = C = 0, Rbar = 0, U = 0, only decay applies."""
    rng = np.random.default_rng(11)
    shape = (16, 24)
    w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
    st = O.TensorState(shape, O.TIER_EXPERT)
    lr = float(F32(1e-3))
    o = O.tensor_step(w.copy(), np.zeros_like(w), st, 0, _hp(), 1, lr, 1, want_x=True)
    assert o["rbar"] == 0.0 and o["sumu2"] == 0.0 and o["kappa"] == 1.0
    assert not st.R.any() and not st.C.any()
    want = (_f(w).astype(np.float64) * (1 - lr * float(F32(0.1)))).astype(np.float32)
    assert np.array_equal(o["x"], want)


def test_rank1_factored_equals_full():
    """P2 (Sec. 3, Eq. 1): if G*G is rank one at every step, the factored Vhat equals the full v."""
    rng = np.random.default_rng(12)
    n, m = 24, 40
    alpha = 2.0 ** rng.integers(-14, -8, n)
    beta = 2.0 ** rng.integers(-3, 3, m)
    w = _bf16(rng.normal(0, 0.02, (n, m)).astype(np.float32)).reshape(-1)
    gs = []
    for t in range(6):
        c = 2.0 ** rng.integers(-2, 3)
        sign = rng.choice([-1.0, 1.0], (n, m))
        gs.append(_bf16((sign * c * np.outer(alpha, beta)).astype(np.float32)).reshape(-1))
    stf = O.TensorState((n, m), O.TIER_EXPERT)
    stv = O.TensorState((n, m), O.TIER_ROUTER)
    hp = _hp(wd=0.0)
    lr = float(F32(1e-3))
    for t, g in enumerate(gs, start=1):
        wf, wv = w.copy(), w.copy()        # both runs start each step from the same weights
        a = O.tensor_step(wf, g, stf, 0, hp, t, lr, 9, want_x=True)
        b = O.tensor_step(wv, g, stv, 0, hp, t, lr, 9, want_x=True)
        vhat = np.outer(stf.R.astype(np.float64), stf.C.astype(np.float64)) / a["rbar"]
        assert np.allclose(vhat.reshape(-1), stv.v.astype(np.float64), rtol=3e-6, atol=0)
        assert abs(a["sumu2"] - b["sumu2"]) <= 1e-5 * b["sumu2"]
        # |U| differs by the fp32 rounding of R, C, v only: a few fp32 ulps of the update
        du = np.abs(a["x"].astype(np.float64) - b["x"].astype(np.float64))
        assert du.max() <= 4e-6 * lr
        w = wf


def test_nx1_and_1xm_factored_exact():
    """P3: on an n x 1 (or 1 x m) matrix the factored Vhat is the full v (Rbar = C)."""
    rng = np.random.default_rng(13)
    for shape in ((37, 1), (1, 53)):
        w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
        gs = [_bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1) for _ in range(4)]
        stf, _, of = _run(shape, O.TIER_EXPERT, gs, w, 4)
        stv, _, ov = _run(shape, O.TIER_ROUTER, gs, w, 4, hp=_hp())
        vhat = np.outer(stf.R.astype(np.float64), stf.C.astype(np.float64)).reshape(-1) / of[-1]["rbar"]
        assert np.allclose(vhat, stv.v, rtol=3e-7, atol=0)
        # decay differs between tiers (router exempt); U and its RMS do not
        for a, b in zip(of, ov):
            assert abs(a["rms"] - b["rms"]) <= 1e-6 * b["rms"]


# --------------------------------------------------------------------------
# The trainer's global gradient-norm clip (Sec. 4 training setup, App. A Table 9:
# clip 1.0) applied as a per-step scale gamma of the gradient the step sees
# --------------------------------------------------------------------------
def _hp_g(gscale, **kw):
    return O.hparams(0.9, 0.999, kw.get("eps", 1e-30), 1.0, kw.get("wd", 0.1), gscale=gscale)


def test_gscale_power_of_two_equals_halved_gradient():
    """gamma = 0.5 is the same step, bit for bit, as gamma = 1 on a gradient halved
    exactly in bf16 (a power-of-two scale of a normal bf16 value is exact), on every
    tier and over three steps, so every place the gradient enters takes gamma."""
    rng = np.random.default_rng(41)
    for shape, tier in (((33, 17), O.TIER_EXPERT), ((20, 40), O.TIER_BACKBONE), ((16, 8), O.TIER_ROUTER),
                        ((129,), O.TIER_BACKBONE)):
        w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
        gs = [_bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1) for _ in range(3)]
        half = [_bf16(_f(g) * np.float32(0.5)) for g in gs]
        assert all(np.array_equal(_f(h).astype(np.float64), 0.5 * _f(g).astype(np.float64)) for h, g in zip(half, gs))
        sa, sb = O.TensorState(shape, tier), O.TensorState(shape, tier)
        wa, wb = w.copy(), w.copy()
        for t in (1, 2, 3):
            oa = O.tensor_step(wa, gs[t - 1], sa, 3, _hp_g(0.5), t, 1e-3, 17, want_x=True)
            ob = O.tensor_step(wb, half[t - 1], sb, 3, _hp_g(1.0), t, 1e-3, 17, want_x=True)
            assert np.array_equal(oa["x"].view(np.uint32), ob["x"].view(np.uint32)), (shape, t)
            assert np.array_equal(wa, wb)
            for key in ("M", "v", "R", "C"):
                if getattr(sa, key) is not None:
                    assert np.array_equal(getattr(sa, key), getattr(sb, key)), (shape, t, key)


def test_gscale_step1_full_v_leaves_sign_and_is_not_a_learning_rate():
    """Algorithm 1, full v at t = 1: U = sign(g) whatever gamma > 0 (v = (1-b2) gamma^2 g^2),
    so the step's weights do not depend on gamma; scaling the learning rate by gamma
    instead changes them. The clip factor therefore cannot be folded into lr."""
    rng = np.random.default_rng(42)
    shape = (64, 8)
    g = _bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1)
    w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
    lr, gam = float(F32(1e-3)), float(F32(0.37))
    for tier, shp in ((O.TIER_ROUTER, shape), (O.TIER_BACKBONE, (512,))):
        outs = {}
        for key, gscale, lr_k in (("one", 1.0, lr), ("gamma", gam, lr), ("lr", 1.0, lr * gam)):
            st = O.TensorState(shp, tier)
            ww = w.copy()
            outs[key] = (O.tensor_step(ww, g, st, 0, _hp_g(gscale), 1, lr_k, 9, want_x=True), ww, st)
        x1, xg, xl = (outs[k][0]["x"].astype(np.float64) for k in ("one", "gamma", "lr"))
        terms = np.abs(_f(w).astype(np.float64)) + lr          # |w (1 - lr lam)| + lr |U|
        # x unchanged by gamma up to fp32 rounding of the terms (the stored v is rounded)
        assert np.max(np.abs(x1 - xg) / terms) <= 1e-6
        # a learning rate scaled by gamma moves x by (1 - gamma) lr on every nonzero g
        moved = np.abs(x1 - xl) / terms > 1e-3
        assert np.count_nonzero(moved) >= 0.9 * np.count_nonzero(_f(g))
        assert np.allclose(outs["gamma"][2].v, gam * gam * outs["one"][2].v, rtol=2e-7, atol=0)
        if tier == O.TIER_BACKBONE:
            assert np.allclose(outs["gamma"][2].M, gam * outs["one"][2].M, rtol=2e-7, atol=0)


def test_gscale_second_step_is_not_scale_invariant():
    """With a history the EMAs mix steps seen at different scales: a gradient scaled at
    step 2 only (zero at step 1 leaves v = 0, so take g at both steps) changes the step
    on every tier, factored experts included."""
    rng = np.random.default_rng(43)
    shape = (24, 32)
    g1 = _bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1)
    g2 = _bf16(rng.normal(0, 1e-3, shape).astype(np.float32)).reshape(-1)
    w = _bf16(rng.normal(0, 0.02, shape).astype(np.float32)).reshape(-1)
    for tier in (O.TIER_EXPERT, O.TIER_BACKBONE, O.TIER_ROUTER):
        res = []
        for gam2 in (1.0, 0.37):
            st = O.TensorState(shape, tier)
            ww = w.copy()
            O.tensor_step(ww, g1, st, 0, _hp_g(1.0), 1, 1e-3, 9)
            o = O.tensor_step(ww, g2, st, 0, _hp_g(gam2), 2, 1e-3, 9, want_x=True)
            res.append(o["x"])
        assert np.max(np.abs(res[0].astype(np.float64) - res[1].astype(np.float64))) > 1e-6
