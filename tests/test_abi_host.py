"""Host-side checks of the C ABI (no GPU needed: no compute call is made).

The library must load, export every function include/skewadam.h declares, and
its ctypes structs must have the header's layout. skew_create is host-only
planning, so tiering, the closed-form state size, the state layout and the
argument validation are all checked here on the CPU.
"""
import ctypes as C
import os
import re
import subprocess
import tempfile

import numpy as np
import pytest

import oracle as O
from paper_2607_19058_gb300 import _build
from paper_2607_19058_gb300 import skewadam as S
from paper_2607_19058_gb300 import workloads as WL

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "skewadam.h")


@pytest.fixture(scope="module", autouse=True)
def lib():
    _build.build()
    return S.load()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(skew_[a-z_]+)\s*\(", src)))


def test_exports_every_declared_symbol(lib):
    names = _declared()
    assert set(names) == set(S.EXPORTS)
    out = subprocess.run(["nm", "-D", "--defined-only", S.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (skew_\w+)", out))
    for n in names:
        assert n in exported, n
        assert hasattr(lib, n)


def test_struct_layout_matches_header():
    prog = r'''
    #include <stdio.h>
    #include <stddef.h>
    #include "skewadam.h"
    int main(void) {
      printf("%zu %zu %zu %zu %zu %zu %zu %zu %zu\n", sizeof(skew_param_desc_t), sizeof(skew_hparams_t),
             sizeof(skew_tensor_info_t), offsetof(skew_param_desc_t, shape), offsetof(skew_param_desc_t, ndim),
             offsetof(skew_param_desc_t, flags), offsetof(skew_tensor_info_t, m_offset),
             offsetof(skew_param_desc_t, stack), offsetof(skew_tensor_info_t, stack));
      return 0; }
    '''
    with tempfile.TemporaryDirectory() as d:
        src, exe = os.path.join(d, "l.c"), os.path.join(d, "l")
        open(src, "w").write(prog)
        subprocess.check_call(["gcc", "-I", os.path.dirname(HEADER), src, "-o", exe])
        got = [int(x) for x in subprocess.check_output([exe]).split()]
    want = [C.sizeof(S.ParamDesc), C.sizeof(S.HParams), C.sizeof(S.TensorInfo), S.ParamDesc.shape.offset,
            S.ParamDesc.ndim.offset, S.ParamDesc.flags.offset, S.TensorInfo.m_offset.offset,
            S.ParamDesc.stack.offset, S.TensorInfo.stack.offset]
    assert got == want


def _descs(wl, base=0x100000):
    out = []
    for k, s in enumerate(wl.specs):
        shp = tuple(s.shape[1:]) if len(s.shape) == 3 else (s.shape[0], s.shape[1] if len(s.shape) == 2 else 0)
        out.append(S.ParamDesc(base * (k + 1), base * (k + 1) + 64, (C.c_int64 * 2)(*shp), len(s.shape), s.tier,
                               S.F_NO_DECAY if s.no_decay else 0, s.shape[0] if len(s.shape) == 3 else 0))
    return out


@pytest.mark.parametrize("name", ["toy", "slice", "appb", "literal", "skewed", "ablation"])
def test_state_bytes_is_closed_form(name):
    wl = WL.get(name)
    for policy in (wl.hp.policy, S.POLICY_UNIFORM, S.POLICY_FACTORED_ROUTER, S.POLICY_ADAFACTOR):
        h = S.skew_create(_descs(wl), S.hparams(policy=policy))
        want = O.state_bytes([(s.shape, s.tier) for s in wl.specs], policy)
        assert S.skew_state_bytes(h) == want
        S.skew_destroy(h)


def test_appb_headline_state_bytes():
    h = S.skew_create(_descs(WL.appb()), S.hparams())
    assert S.skew_state_bytes(h) == 1_380_800_000
    S.skew_destroy(h)


@pytest.mark.parametrize("name", ["toy", "appb", "ablation"])
def test_stacked_experts_plan_like_separate_matrices(name):
    """Experts kept as (E, n, m) stacks: each matrix keeps its own factors, so the state
    is the closed form of the E separate matrices; a stack's arrays are contiguous."""
    wl, st = WL.get(name), WL.stack_experts(WL.get(name))
    assert any(len(s.shape) == 3 for s in st.specs)
    for policy in (wl.hp.policy, S.POLICY_UNIFORM):
        h = S.skew_create(_descs(st), S.hparams(policy=policy))
        want = O.state_bytes([(s.shape, s.tier) for s in wl.specs], policy)
        assert S.skew_state_bytes(h) == want
        assert S.skew_num_tensors(h) == len(st.specs)
        total = S.skew_state_bytes(h) // 4
        spans = []
        for k, s in enumerate(st.specs):
            i = S.skew_tensor_info(h, k)
            E = s.shape[0] if len(s.shape) == 3 else 1
            assert i.stack == (E if len(s.shape) == 3 else 0)
            assert (i.rows, i.cols) == ((s.shape[-2], s.shape[-1]) if len(s.shape) >= 2 else (s.shape[0], 1))
            assert i.numel == s.numel
            for off, cnt in ((i.m_offset, i.numel), (i.v_offset, i.numel), (i.r_offset, E * i.rows),
                             (i.c_offset, E * i.cols)):
                if off >= 0:
                    spans.append((off, off + cnt))
        spans.sort()
        assert spans[0][0] == 0 and spans[-1][1] == total
        assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
        S.skew_destroy(h)


def test_matrix_scalars_range():
    h = S.skew_create([_one((3, 4, 8)), _one((4, 8))], S.hparams())
    for tid, e in ((0, 3), (0, -1), (1, 1), (2, 0)):
        with pytest.raises(S.SkewError) as err:
            S.skew_matrix_scalars(h, tid, e, 0)
        assert err.value.code == S.SKEW_EINVAL
    with pytest.raises(S.SkewError) as err:   # in range, but nothing is bound yet
        S.skew_matrix_scalars(h, 0, 2, 0)
    assert err.value.code == S.SKEW_ESTATE
    S.skew_destroy(h)


@pytest.mark.parametrize("name", ["toy", "ablation"])
def test_state_layout_tiles_the_buffer(name):
    """Every state array has its own range, they do not overlap and they cover the buffer."""
    wl = WL.get(name)
    h = S.skew_create(_descs(wl), S.hparams(policy=wl.hp.policy))
    total = S.skew_state_bytes(h) // 4
    spans = []
    for k, s in enumerate(wl.specs):
        i = S.skew_tensor_info(h, k)
        kind, mo, dec = O.resolve(len(s.shape), s.tier, wl.hp.policy, s.no_decay)
        assert (i.kind, i.momentum, i.decay) == (kind, mo, dec)
        assert i.numel == s.numel
        for off, cnt in ((i.m_offset, i.numel), (i.v_offset, i.numel), (i.r_offset, i.rows), (i.c_offset, i.cols)):
            if off >= 0:
                spans.append((off, off + cnt))
        assert (i.m_offset >= 0) == bool(mo)
        assert (i.v_offset >= 0) == (kind == O.KIND_FULL)
        assert (i.r_offset >= 0) == (i.c_offset >= 0) == (kind == O.KIND_FACTORED)
    spans.sort()
    assert spans[0][0] == 0 and spans[-1][1] == total
    assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))   # no gap, no overlap
    S.skew_destroy(h)


def _one(shape=(4, 8), tier=S.TIER_EXPERT, **kw):
    d = dict(weight=0x1000, grad=0x2000, ndim=len(shape), tier=tier, flags=0, stack=shape[0] if len(shape) == 3 else 0)
    d.update(kw)
    shp = tuple(shape[-2:]) if len(shape) == 3 else (shape[0], shape[1] if len(shape) == 2 else 0)
    return S.ParamDesc(d["weight"], d["grad"], (C.c_int64 * 2)(*shp), d["ndim"], d["tier"], d["flags"], d["stack"])


@pytest.mark.parametrize("desc,msg", [
    (dict(weight=0), "null"), (dict(grad=0), "null"), (dict(weight=0x1001), "aligned"), (dict(ndim=4), "ndim"),
    (dict(ndim=0), "ndim"), (dict(tier=5), "tier"), (dict(flags=8), "flags"), (dict(stack=1), "stack"),
    (dict(ndim=3, stack=0), "stack"),
])
def test_create_rejects_bad_descriptors(desc, msg):
    with pytest.raises(S.SkewError) as e:
        S.skew_create([_one(**desc)], S.hparams())
    assert e.value.code == S.SKEW_EINVAL and msg in str(e.value)


@pytest.mark.parametrize("shape", [(0, 8), (8, 0), (-1, 4), (2**41, 2)])
def test_create_rejects_bad_extents(shape):
    with pytest.raises(S.SkewError):
        S.skew_create([_one(shape)], S.hparams())


@pytest.mark.parametrize("hp", [dict(beta1=1.0), dict(beta2=-0.1), dict(eps=0.0), dict(eps=float("nan")),
                                dict(clip_d=0.0), dict(weight_decay=-1.0), dict(policy=5), dict(beta1=float("inf"))])
def test_create_rejects_bad_hparams(hp):
    with pytest.raises(S.SkewError) as e:
        S.skew_create([_one()], S.hparams(**hp))
    assert e.value.code == S.SKEW_EINVAL


def test_step_before_bind_and_bad_bind_sizes():
    h = S.skew_create([_one()], S.hparams())
    with pytest.raises(S.SkewError) as e:
        S.skew_step(h, 1, 1e-3, 0, 0)
    assert e.value.code == S.SKEW_ESTATE
    with pytest.raises(S.SkewError) as e:   # the wait self-test too needs a bound handle
        S.skew_selftest_wait_timeout(h, 0)
    assert e.value.code == S.SKEW_ESTATE
    with pytest.raises(S.SkewError) as e:   # wrong sizes are rejected before any CUDA call
        S.skew_bind(h, 0x100000, S.skew_state_bytes(h) + 4, 0x200000, S.skew_workspace_bytes(h), 0)
    assert e.value.code == S.SKEW_EINVAL
    with pytest.raises(S.SkewError) as e:
        S.skew_bind(h, 0x100010, S.skew_state_bytes(h), 0x200000, S.skew_workspace_bytes(h), 0)
    assert e.value.code == S.SKEW_EINVAL and "aligned" in str(e.value)
    with pytest.raises(S.SkewError):
        S.skew_tensor_info(h, 3)
    S.skew_destroy(h)


def test_empty_parameter_list():
    h = S.skew_create([], S.hparams())
    assert S.skew_state_bytes(h) == 0 and S.skew_num_tensors(h) == 0
    S.skew_destroy(h)


def test_64bit_extents_plan():
    """A tensor past 2^31 elements plans fine (64-bit indexing, cf. the 2^31 crash of 8-bit optimizers)."""
    h = S.skew_create([_one((65536, 40000)), _one((3 * 2**30,), tier=S.TIER_BACKBONE)], S.hparams())
    i = S.skew_tensor_info(h, 0)
    assert i.numel == 65536 * 40000 > 2**31
    assert S.skew_state_bytes(h) == 4 * (65536 + 40000) + 4 * 2 * 3 * 2**30
    S.skew_destroy(h)


def test_fp32_tensors_plan():
    """SKEW_F_FP32 (App. A: fp32 norms and router): accepted for any tier, 4-byte alignment
    required, never on the whole-row bf16 path; the state is the same closed form."""
    h = S.skew_create([_one((4096, 4096), flags=S.F_FP32), _one((4096, 4096)), _one((4096,), flags=S.F_FP32,
                                                                                    tier=S.TIER_BACKBONE)],
                      S.hparams())
    assert [S.skew_tensor_info(h, k).rowpath for k in range(3)] == [0, 1, 0]
    assert S.skew_state_bytes(h) == 4 * (2 * (4096 + 4096) + 2 * 4096)
    S.skew_destroy(h)
    with pytest.raises(S.SkewError) as e:
        S.skew_create([_one((8, 8), weight=0x1002, flags=S.F_FP32)], S.hparams())
    assert e.value.code == S.SKEW_EINVAL and "4-byte" in str(e.value)


def _noalloc(**kw):
    """skew_step_tensor_noalloc with fake device pointers: every check below happens on the
    host before any CUDA call; returns the error code (SKEW_OK never: no GPU here)."""
    a = dict(weight=0x100000, grad=0x200000, ndim=2, rows=64, cols=128, tier=S.TIER_EXPERT, flags=0,
             hp=S.hparams(), state=0x300000, tensor_id=0, step=1, lr=1e-3, seed=0, stream=0)
    a.update(kw)
    if "state_bytes" not in a:   # the closed form for an expert matrix under the tiered policy: R and C
        a["state_bytes"] = 4 * (a["rows"] + (a["cols"] if a["ndim"] == 2 else 0))
    try:
        S.skew_step_tensor_noalloc(a["weight"], a["grad"], a["ndim"], a["rows"], a["cols"], a["tier"], a["flags"],
                                   a["hp"], a["state"], a["state_bytes"], a["tensor_id"], a["step"], a["lr"],
                                   a["seed"], a["stream"])
    except S.SkewError as e:
        return e.code
    return S.SKEW_OK


@pytest.mark.parametrize("kw", [dict(weight=0), dict(grad=0), dict(state=0), dict(weight=0x100001),
                                dict(state=0x300002), dict(ndim=3), dict(ndim=0), dict(tier=3), dict(flags=4),
                                dict(step=0), dict(lr=-1.0), dict(lr=float("nan")), dict(rows=0),
                                dict(hp=S.hparams(beta2=1.0)), dict(hp=S.hparams(policy=5)),
                                dict(state_bytes=4 * (64 + 128) + 4)])
def test_noalloc_rejects_bad_arguments_on_the_host(kw):
    assert _noalloc(**kw) == S.SKEW_EINVAL


def test_noalloc_scratch_limit_on_the_host():
    """The fixed scratch holds a 4096-wide matrix of about 65,000 rows (the paper's 50,304 x 4096
    embedding included): smaller ones pass every host check (and then need a GPU: SKEW_ECUDA
    here), larger ones are SKEW_ETOOBIG before any CUDA call."""
    import torch
    mom = S.TIER_BACKBONE  # momentum + factored: state M, R, C
    if not torch.cuda.is_available():  # (with a GPU the fake pointers would reach the kernels)
        fits = _noalloc(rows=50304, cols=4096, tier=mom, state_bytes=4 * (50304 * 4096 + 50304 + 4096))
        assert fits == S.SKEW_ECUDA
    big = _noalloc(rows=80000, cols=4096, tier=mom, state_bytes=4 * (80000 * 4096 + 80000 + 4096))
    assert big == S.SKEW_ETOOBIG
    # without momentum the 256-row tiles halve the partials: about twice the rows fit
    ex = S.TIER_EXPERT
    if not torch.cuda.is_available():
        assert _noalloc(rows=120000, cols=4096, tier=ex, state_bytes=4 * (120000 + 4096)) == S.SKEW_ECUDA
    assert _noalloc(rows=140000, cols=4096, tier=ex, state_bytes=4 * (140000 + 4096)) == S.SKEW_ETOOBIG
    assert _noalloc(rows=1 << 20, cols=8192) == S.SKEW_ETOOBIG


def test_random_plans_tile_the_state():
    """Random parameter lists (vectors, matrices, stacks; every tier; no-decay and fp32
    flags; every policy): the planner's state is the oracle's closed form, each tensor's
    kind / momentum / decay is the oracle's, and its arrays tile the state buffer exactly.
    The row path is chosen exactly for bf16 factored matrices 512 to 4096 wide (powers of
    two) with 16-byte aligned pointers."""
    hyp = pytest.importorskip("hypothesis")
    st = hyp.strategies

    tensor = st.tuples(st.sampled_from([1, 2, 3]), st.integers(1, 3000), st.sampled_from([1, 7, 64, 512, 1000, 1024,
                                                                                            2048, 4096, 5000]),
                       st.integers(1, 3), st.sampled_from([S.TIER_BACKBONE, S.TIER_EXPERT, S.TIER_ROUTER]),
                       st.booleans(), st.booleans(), st.booleans())

    @hyp.settings(max_examples=150, deadline=None, derandomize=True)
    @hyp.given(st.lists(tensor, max_size=10), st.sampled_from([S.POLICY_TIERED, S.POLICY_EXPERT_MOMENTUM,
                                                              S.POLICY_FACTORED_ROUTER, S.POLICY_UNIFORM,
                                                              S.POLICY_ADAFACTOR]))
    def check(tensors, policy):
        descs, specs, meta = [], [], []
        for k, (nd, n, m, e, tier, nodecay, fp32, misalign) in enumerate(tensors):
            base = 0x10000000 * (k + 1)
            w, g = base + (4 if misalign else 0), base + 0x8000000
            flags = (S.F_NO_DECAY if nodecay else 0) | (S.F_FP32 if fp32 else 0)
            shp = (n, m) if nd >= 2 else (n, 0)
            descs.append(S.ParamDesc(w, g, (C.c_int64 * 2)(*shp), nd, tier, flags, e if nd == 3 else 0))
            mats = [((n, m) if nd >= 2 else (n,), tier)] * (e if nd == 3 else 1)
            specs += mats
            meta.append((nd, n, m if nd >= 2 else 1, e if nd == 3 else 1, tier, nodecay, fp32, misalign))
        h = S.skew_create(descs, S.hparams(policy=policy))
        try:
            assert S.skew_state_bytes(h) == O.state_bytes(specs, policy)
            total = S.skew_state_bytes(h) // 4
            spans = []
            for k, (nd, n, m, E, tier, nodecay, fp32, misalign) in enumerate(meta):
                i = S.skew_tensor_info(h, k)
                kind, mo, dec = O.resolve(2 if nd == 3 else nd, tier, policy, nodecay)
                assert (i.kind, i.momentum, i.decay) == (kind, mo, dec)
                assert i.numel == E * n * m and (i.rows, i.cols) == (n, m)
                want_row = kind == O.KIND_FACTORED and not fp32 and not misalign and m in (512, 1024, 2048, 4096)
                assert bool(i.rowpath) == want_row
                for off, cnt in ((i.m_offset, i.numel), (i.v_offset, i.numel), (i.r_offset, E * n),
                                 (i.c_offset, E * m)):
                    if off >= 0:
                        spans.append((off, off + cnt))
            spans.sort()
            if spans:
                assert spans[0][0] == 0 and spans[-1][1] == total
                assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))
            else:
                assert total == 0
        finally:
            S.skew_destroy(h)

    check()
