"""GPU parity: libskewadam through its C ABI against the CPU oracle (teacher forced).

Covers the toy MoE set over its 10 steps (zero-grad experts on odd steps, so
Rbar = 0 at step 1), the paper's own hyper-parameters (eps = 1e-8 clamps at
step 1), ragged / awkward shapes on the vector and scalar paths, misaligned
pointers, and the large shape sets at full size in the launch configuration
the benchmark uses, checking a subset of their tensors.
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


def _harness(*a, **k):
    import parity
    return parity.Harness(*a, **k)


def test_toy_all_steps():
    h = _harness(WL.toy())
    for t in range(1, 11):
        rep = h.step(t)
        assert rep.tensors == len(h.wl.specs)
    h.close()


def test_toy_paper_hyperparameters():
    """eps = 1e-8, lr = 3e-4, lambda = 0.05 (App. A): the eps clamp binds at step 1."""
    h = _harness(WL.toy(), hp_override=dict(eps=1e-8, lr=3e-4, weight_decay=0.05))
    for t in range(1, 4):
        h.step(t, seed=77)
    h.close()


def _edge_workload():
    B, E, R = WL.TIER_BACKBONE, WL.TIER_EXPERT, WL.TIER_ROUTER
    specs = [WL.Spec("e300x1000", (300, 1000), E), WL.Spec("b517x136", (517, 136), B),
             WL.Spec("v100003", (100003,), B), WL.Spec("router4096x127", (4096, 127), R),
             WL.Spec("b1x4096", (1, 4096), B), WL.Spec("e4095x1000", (4095, 1000), E),
             WL.Spec("e3x5", (3, 5), E), WL.Spec("e7x1", (7, 1), E), WL.Spec("b1x7", (1, 7), B),
             WL.Spec("v13", (13,), B), WL.Spec("b2x2", (2, 2), B), WL.Spec("e11x13", (11, 13), E),
             WL.Spec("router8x127", (8, 127), R), WL.Spec("e64x8", (64, 8), E), WL.Spec("e2000x24", (2000, 24), E),
             WL.Spec("nodecay", (129, 256), B, no_decay=True)]
    return WL.Workload("edge", specs, WL.HP(), "normal", steps=4)


def test_edge_shapes():
    h = _harness(_edge_workload())
    for t in range(1, 5):
        h.step(t, seed=t * 1001)
    h.close()


def test_misaligned_pointers_use_scalar_path():
    wl = _edge_workload()
    h = _harness(wl, misalign=(0, 1, 2, 3, 5))
    for k in (0, 1, 2, 3, 5):
        assert h.opt.info(k).vectorized == 0
    assert h.opt.info(4).vectorized == 1
    for t in range(1, 3):
        h.step(t, seed=5)
    h.close()


@pytest.mark.parametrize("policy", [WL.POLICY_EXPERT_MOMENTUM, WL.POLICY_FACTORED_ROUTER, WL.POLICY_UNIFORM])
def test_table3_variants(policy):
    wl = WL.toy()
    wl.hp = WL.HP(policy=policy)
    h = _harness(wl)
    for t in range(1, 4):
        h.step(t)
    h.close()


def test_state_bytes_equal_closed_form_and_layout():
    import oracle as O
    for name in ("toy", "slice", "appb", "ablation"):
        wl = WL.get(name)
        descs = []
        buf = torch.empty(2, dtype=torch.bfloat16, device="cuda")
        import ctypes as C
        for s in wl.specs:
            shp = (s.shape[0], s.shape[1] if len(s.shape) == 2 else 0)
            descs.append(S.ParamDesc(buf.data_ptr(), buf.data_ptr(), (C.c_int64 * 2)(*shp), len(s.shape), s.tier, 0, 0))
        h = S.skew_create(descs, S.hparams(policy=wl.hp.policy))
        assert S.skew_state_bytes(h) == O.state_bytes([(s.shape, s.tier) for s in wl.specs], wl.hp.policy)
        S.skew_destroy(h)


def test_empty_handle_steps():
    h = S.skew_create([], S.hparams())
    assert S.skew_state_bytes(h) == 0
    ws = torch.empty(max(1, S.skew_workspace_bytes(h)), dtype=torch.uint8, device="cuda")
    S.skew_bind(h, 0, 0, ws.data_ptr(), S.skew_workspace_bytes(h), torch.cuda.current_stream().cuda_stream)
    S.skew_step(h, 1, 1e-3, 0, torch.cuda.current_stream().cuda_stream)
    S.skew_sync_status(h, torch.cuda.current_stream().cuda_stream)
    S.skew_destroy(h)


def test_deterministic_and_resumable():
    """Same inputs -> bit-identical weights and state; save/restore mid-run changes nothing."""
    wl = _edge_workload()

    def run(steps, restore_at=None):
        import parity
        h = parity.Harness(wl, check=[])
        snap = None
        for t in range(1, steps + 1):
            h.step(t, seed=99)
            if restore_at == t:
                snap = ([w.clone() for w in h.W], h.opt.state.clone())
        if snap is not None:
            h2 = parity.Harness(wl, check=[])
            for w, s in zip(h2.W, snap[0]):
                w.copy_(s)
            h2.opt.state.copy_(snap[1])
            for t in range(restore_at + 1, steps + 1):
                h2.step(t, seed=99)
            h = h2
        torch.cuda.synchronize()
        return [w.clone() for w in h.W], h.opt.state.clone()

    w1, s1 = run(5)
    w2, s2 = run(5)
    w3, s3 = run(5, restore_at=2)
    for a, b, c in zip(w1, w2, w3):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
        assert torch.equal(a.view(torch.int16), c.view(torch.int16))
    assert torch.equal(s1, s2) and torch.equal(s1, s3)


def _subset(wl, names):
    idx = [k for k, s in enumerate(wl.specs) if s.name in names]
    assert len(idx) == len(names), names
    return idx


def test_slice_full_size_subset():
    wl = WL.slice_()
    chk = _subset(wl, ["attn.q", "attn.k", "norm.attn", "router", "expert0.w0", "expert0.w1", "expert77.w2",
                       "expert127.w1"])
    h = _harness(wl, check=chk, max_widened_frac=1e-4)
    for t in (1, 2, 3):
        h.step(t)
    h.close()


def test_appb_full_size_subset():
    wl = WL.appb()
    chk = _subset(wl, ["embed", "pos", "b0.ln1.weight", "b0.attn.k", "b1.attn.o", "b1.router", "expert3.w1",
                       "expert127.w2", "ln_f.bias"])
    h = _harness(wl, check=chk, max_widened_frac=1e-4)
    for t in (1, 2):
        h.step(t)
    h.close()


def test_skewed_full_size_subset():
    """Zipf loads: 40 zero-grad experts per step, Student-t grads, 100x router spikes at t % 10 == 7."""
    wl = WL.skewed()
    ranks = WL.zipf_ranks(wl.n_experts, wl.seed, 7)
    zero_e = int(np.argmax(ranks.numpy()))          # least loaded at step 7 -> zero grads
    busy_e = int(np.argmin(ranks.numpy()))
    chk = _subset(wl, ["b1.router", "b0.attn.q", f"expert{zero_e}.w0", f"expert{busy_e}.w1", "b0.ln2.bias"])
    h = _harness(wl, check=chk, max_widened_frac=1e-4)
    clipped = 0
    for t in range(1, 8):
        if t in (1, 6, 7):
            rep = h.step(t)
            clipped += rep.clipped
        else:
            h.load_grads(t)
            h.opt.step(t, h.lr, 1234)
    assert clipped >= 1
    h.close()


def test_ablation_awkward_full_size_subset():
    wl = WL.ablation()
    chk = _subset(wl, ["embed", "odd.a", "odd.b", "b1.router", "expert0.w0", "expert5.w2", "b1.ln2.weight"])
    h = _harness(wl, check=chk, max_widened_frac=1e-4)
    for t in (1, 2):
        h.step(t)
    h.close()


def _row_path_workload():
    """Momentum-free matrices of width 4096 / 2048 / 1024 / 512 (the whole-row
    phases A and C): ragged row tiles and chunks, and expert 5 with zero gradients on
    odd steps."""
    E = WL.TIER_EXPERT
    specs = [WL.Spec("e512x4096", (512, 4096), E, expert=0), WL.Spec("e301x4096", (301, 4096), E, expert=1),
             WL.Spec("e1000x2048", (1000, 2048), E, expert=2), WL.Spec("e77x2048", (77, 2048), E, expert=3),
             WL.Spec("e1333x1024", (1333, 1024), E, expert=4), WL.Spec("e2101x512", (2101, 512), E, expert=6),
             WL.Spec("zero_odd", (256, 4096), E, expert=5)]
    return WL.Workload("rowpath", specs, WL.HP(), "toy", steps=4)


def test_row_path_bilinear_sum():
    """eps = 1e-30: no clamp can bind, so sum(U^2) comes from the whole-row partials."""
    h = _harness(_row_path_workload())
    assert all(h.opt.info(k).rowpath == 1 for k in range(len(h.wl.specs)))
    for t in range(1, 5):
        h.step(t, seed=t * 31)
    h.close()


def test_row_path_tiny_matrices():
    """Momentum-free row-path matrices with fewer rows than one chunk (1 to 5 rows; a stack
    of one-row matrices): every tile is one ragged chunk."""
    E = WL.TIER_EXPERT
    specs = [WL.Spec("e1x4096", (1, 4096), E, expert=0), WL.Spec("e2x1024", (2, 1024), E, expert=1),
             WL.Spec("e3x512", (3, 512), E, expert=2), WL.Spec("e5x2048", (5, 2048), E, expert=3),
             WL.Spec("e3x1x1024", (3, 1, 1024), E)]
    h = _harness(WL.Workload("tiny_rows", specs, WL.HP(), "normal", steps=3))
    assert all(h.opt.info(k).rowpath == 1 for k in range(len(specs)))
    for t in range(1, 4):
        h.step(t, seed=11 * t)
    h.close()


def test_row_path_clamp_falls_back_to_phase_b():
    """eps = 1e-8 (App. A): the clamp binds at step 1, so the finalize queues the
    tensors for phase B and sum(U^2) is taken element by element."""
    h = _harness(_row_path_workload(), hp_override=dict(eps=1e-8, lr=3e-4, weight_decay=0.05))
    for t in range(1, 4):
        h.step(t, seed=77)
    h.close()


def _stacked_workload():
    """Stacked (E, n, m) tensors on every path: the row path (m = 1024, 4096), the strip
    path with m % 8 != 0 (each matrix's dither index starts inside a Philox block),
    an elementwise router stack with an odd matrix size, a momentum stack and a stack
    of one, with a plain matrix between them so descriptor ids and matrices differ."""
    B, E, R = WL.TIER_BACKBONE, WL.TIER_EXPERT, WL.TIER_ROUTER
    specs = [WL.Spec("e4x300x1024", (4, 300, 1024), E), WL.Spec("b100x48", (100, 48), B),
             WL.Spec("e3x37x100", (3, 37, 100), E), WL.Spec("r3x33x65", (3, 33, 65), R),
             WL.Spec("b2x64x256", (2, 64, 256), B), WL.Spec("e2x700x4096", (2, 700, 4096), E),
             WL.Spec("e1x128x512", (1, 128, 512), E), WL.Spec("v999", (999,), B)]
    return WL.Workload("stacked", specs, WL.HP(), "normal", steps=3)


def test_stacked_tensors():
    """Every matrix of a stack keeps its own factors and clip factor; a matrix whose
    gradient is zero (mean(R) = 0 at step 1) sits beside live ones."""
    h = _harness(_stacked_workload())
    assert h.opt.info(0).stack == 4 and h.opt.info(0).rowpath == 1 and h.opt.info(2).rowpath == 0
    assert h.opt.info(1).stack == 0
    for t in range(1, 4):
        h.load_grads(t)
        if t == 1:
            h.G[0][2].zero_()
            h.G[2][1].zero_()
        rep = h.step(t, seed=5 + t, grads_loaded=True)
        assert rep.tensors == sum(s.shape[0] if len(s.shape) == 3 else 1 for s in h.wl.specs)
    h.close()


def test_stacked_appb_experts_full_size_subset():
    """App. B with the 128 experts of each weight kept as one (128, 4096, 4096) array,
    in the benchmark's launch configuration; the router and matrices 0, 1, 77 and 127
    of the first stack are checked."""
    wl = WL.stack_experts(WL.appb())
    names = {"b1.router", "experts.w0"}
    check = [k for k, s in enumerate(wl.specs) if s.name in names]
    assert len(check) == 2
    h = _harness(wl, check=check, max_widened_frac=1e-4, matrices={check[1]: (0, 1, 77, 127)})
    h.step(1, seed=3)
    h.close()


def test_adafactor_comparator():
    """The Adafactor comparator (every matrix factored, no momentum, beta2_t = 1 - t^-0.8, no
    bias correction) on the toy set (strip path, exact vectors, zero-gradient experts at t = 1)
    and on the whole-row path, over steps whose decay changes every step."""
    h = _harness(WL.toy(), hp_override=dict(policy=WL.POLICY_ADAFACTOR))
    assert all(h.opt.info(k).momentum == 0 for k in range(len(h.wl.specs)))
    for t in range(1, 5):
        h.step(t, seed=t)
    h.close()
    h = _harness(_row_path_workload(), hp_override=dict(policy=WL.POLICY_ADAFACTOR))
    for t in range(1, 4):
        h.step(t, seed=11 * t)
    h.close()


def test_fp32_router_and_norms():
    """The paper's precision (App. A): router and LayerNorm vectors in fp32, stepped with no
    dithered cast, beside bf16 matrices; over the toy steps and at the paper's hyper-parameters."""
    h = _harness(WL.toy_fp32())
    assert any(w.dtype == torch.float32 for w in h.W)
    for t in range(1, 6):
        h.step(t)
    h.close()
    h = _harness(WL.toy_fp32(), hp_override=dict(eps=1e-8, lr=3e-4, weight_decay=0.05))
    for t in range(1, 4):
        h.step(t, seed=5)
    h.close()


def test_fp32_awkward_shapes_and_policies():
    """fp32 tensors on the strip path (factored, with and without momentum, ragged), flat
    tiles with a ragged tail, a stack, and under the factored-router and Adafactor policies."""
    B, E, R = WL.TIER_BACKBONE, WL.TIER_EXPERT, WL.TIER_ROUTER
    specs = [WL.Spec("r300x127", (300, 127), R, fp32=True), WL.Spec("v1001", (1001,), B, fp32=True),
             WL.Spec("b37x4096", (37, 4096), B, fp32=True), WL.Spec("e77x333", (77, 333), E, fp32=True),
             WL.Spec("s3x21x40", (3, 21, 40), E, fp32=True), WL.Spec("e64x4096", (64, 4096), E)]
    for policy in (WL.POLICY_TIERED, WL.POLICY_FACTORED_ROUTER, WL.POLICY_ADAFACTOR):
        wl = WL.Workload("fp32_edge", specs, WL.HP(policy=policy), "normal", steps=3)
        h = _harness(wl)
        for t in range(1, 4):
            h.step(t, seed=t + policy)
        h.close()


def _momentum_row_workload():
    """Momentum matrices on the whole-row path (the backbone; experts under the momentum
    variants): every width, ragged tiles and chunks, one-row and tiny matrices, a stack."""
    B, E = WL.TIER_BACKBONE, WL.TIER_EXPERT
    specs = [WL.Spec("b300x4096", (300, 4096), B), WL.Spec("b1x4096", (1, 4096), B),
             WL.Spec("b77x2048", (77, 2048), B), WL.Spec("b1333x1024", (1333, 1024), B),
             WL.Spec("b2101x512", (2101, 512), B), WL.Spec("s3x130x4096", (3, 130, 4096), B),
             WL.Spec("e257x4096", (257, 4096), E, expert=0), WL.Spec("v4096", (4096,), B)]
    return WL.Workload("momrow", specs, WL.HP(policy=WL.POLICY_EXPERT_MOMENTUM), "normal", steps=4)


def test_momentum_row_path():
    """The new M is stored in phase A and sum(U^2) comes from Q_j = sum_i M_ij^2 / R_i."""
    h = _harness(_momentum_row_workload())
    assert all(h.opt.info(k).rowpath == 1 and h.opt.info(k).momentum == 1
               for k, s in enumerate(h.wl.specs) if len(s.shape) >= 2)
    for t in range(1, 5):
        h.step(t, seed=7 * t)
    h.close()


def test_momentum_row_path_fallbacks():
    """eps = 1e-8 (the clamp binds at step 1: phase B runs on the stored new M, not a second
    update) and a matrix whose gradient is zero at step 1 (R_i == 0 rows: phase B too)."""
    h = _harness(_momentum_row_workload(), hp_override=dict(eps=1e-8, lr=3e-4, weight_decay=0.05))
    for t in range(1, 4):
        h.step(t, seed=3)
    h.close()
    h = _harness(_momentum_row_workload())
    for t in range(1, 4):
        h.load_grads(t)
        if t == 1:
            h.G[0].zero_()
            h.G[5][1].zero_()
        h.step(t, seed=9, grads_loaded=True)
    h.close()


def _wide_tile_workload():
    """Momentum-free 4096-wide matrices of at least 2048 rows, whose phase-A tiles are 256
    rows (phase C keeps 128): ragged last tiles of 1 row, of 63 whole chunks, and of 63
    chunks and a 2-row chunk, a stack of two such matrices, and a 2047-row matrix (the
    largest that keeps 128-row phase-A tiles) beside them."""
    E = WL.TIER_EXPERT
    specs = [WL.Spec("e2049x4096", (2049, 4096), E, expert=0), WL.Spec("e2300x4096", (2300, 4096), E, expert=1),
             WL.Spec("e2302x4096", (2302, 4096), E, expert=2), WL.Spec("s2x2050x4096", (2, 2050, 4096), E),
             WL.Spec("e2047x4096", (2047, 4096), E, expert=3)]
    return WL.Workload("wide", specs, WL.HP(), "normal", steps=3)


def test_wide_phase_a_tiles_ragged():
    h = _harness(_wide_tile_workload())
    assert all(h.opt.info(k).rowpath == 1 for k in range(len(h.wl.specs)))
    for t in range(1, 4):
        h.step(t, seed=7 * t)
    h.close()


def test_wide_phase_a_tiles_with_grad_scale_and_clamp():
    """The same shapes under the trainer's clip factor, and with eps = 1e-8 (App. A), where
    the clamp binds and the tensors take phase B."""
    h = _harness(_wide_tile_workload())
    for t, g in ((1, 0.37), (2, 1.0), (3, 0.8)):
        h.step(t, seed=3 * t, gscale=g)
    h.close()
    h = _harness(_wide_tile_workload(), hp_override=dict(eps=1e-8, lr=3e-4, weight_decay=0.05))
    for t in (1, 2):
        h.step(t, seed=19 * t)
    h.close()
