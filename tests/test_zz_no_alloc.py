"""skew_step_tensor_noalloc: the one-tensor step that allocates nothing.

It exists for callers that cannot allocate device memory when they step the
optimizer (a framework allocator holding all free memory, plugins handed only
pre-sized buffers, runtimes that forbid allocation after start-up): its
scratch is a fixed array inside the library instead of a caller workspace.

Checked through the C ABI against the regular path (skew_create / skew_bind /
skew_step on a one-tensor handle) on two consecutive steps, for a factored
expert matrix, a momentum backbone matrix, the router's exact second moment
and a backbone vector; and its status word: a bounded device wait that gives
up is reported once by skew_noalloc_sync_status, after which the entry point
keeps stepping in parity. The file is named so that pytest collects it last.
"""
import ctypes as C

import pytest
import torch

from paper_2607_19058_gb300 import skewadam as S
from paper_2607_19058_gb300 import workloads as WL

pytestmark = pytest.mark.gpu

# (8192, 4096) expert: a momentum-free matrix on the whole-row path; (50304, 4096)
# backbone: the paper's embedding, the largest tensor the fixed scratch is sized for;
# (4096, 4096) and (3001, 2048) experts: matrices that skew_step runs in its pipelined
# launch, which the no-alloc entry point must match with the separate launches.
SHAPES = [((300, 1000), S.TIER_EXPERT), ((517, 136), S.TIER_BACKBONE), ((4096, 127), S.TIER_ROUTER),
          ((100003,), S.TIER_BACKBONE), ((8192, 4096), S.TIER_EXPERT), ((50304, 4096), S.TIER_BACKBONE),
          ((4096, 4096), S.TIER_EXPERT), ((3001, 2048), S.TIER_EXPERT)]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_19058_gb300 import _build
    _build.build()


@pytest.mark.parametrize("shape,tier", SHAPES)
def test_noalloc_matches_regular_path_two_steps(shape, tier):
    torch.manual_seed(0)
    dev = torch.device("cuda")
    w0 = (torch.randn(shape, device=dev) * 0.02).to(torch.bfloat16)
    g = torch.empty(shape, dtype=torch.bfloat16, device=dev)
    hp = S.hparams(0.9, 0.999, 1e-30, 1.0, 0.1, S.POLICY_TIERED)
    w_ref, w_na = w0.clone(), w0.clone()
    ref = S.SkewAdam([(w_ref, g, tier)], hp)
    nbytes = ref.state_bytes
    state = torch.zeros(nbytes // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream().cuda_stream
    rows = shape[0]
    cols = shape[1] if len(shape) == 2 else 0
    for t in (1, 2):
        g.copy_((torch.randn(shape, device=dev) * 1e-3).to(torch.bfloat16))
        ref.step(t, 1e-3, 77)
        S.skew_step_tensor_noalloc(w_na.data_ptr(), g.data_ptr(), len(shape), rows, cols, tier, 0, hp,
                                   state.data_ptr(), nbytes, 0, t, 1e-3, 77, stream)
        torch.cuda.synchronize()
        # same kernels on the same inputs: the results agree bit for bit (inside every tolerance)
        assert torch.equal(w_ref.view(torch.int16), w_na.view(torch.int16)), f"weights differ at step {t}"
        assert torch.equal(ref.state[:nbytes].view(torch.float32), state), f"state differs at step {t}"
    ref.close()


def test_noalloc_rejects_oversized_tensor():
    dev = torch.device("cuda")
    w = torch.zeros(8, dtype=torch.bfloat16, device=dev)
    hp = S.hparams()
    rows, cols = 1 << 20, 8192           # needs far more than the fixed scratch; nothing is launched
    nbytes = 4 * (rows + cols)
    with pytest.raises(S.SkewError) as e:
        S.skew_step_tensor_noalloc(w.data_ptr(), w.data_ptr(), 2, rows, cols, S.TIER_EXPERT, 0, hp, w.data_ptr(),
                                   nbytes, 0, 1, 1e-3, 0, torch.cuda.current_stream().cuda_stream)
    assert e.value.code == S.SKEW_ETOOBIG


def test_noalloc_fp32_matches_regular_path():
    """An fp32 tensor (SKEW_F_FP32) through the no-alloc entry point equals skew_step's result."""
    dev = torch.device("cuda")
    for shape, tier in (((300, 127), S.TIER_ROUTER), ((4097,), S.TIER_BACKBONE)):
        torch.manual_seed(1)
        w0 = torch.randn(shape, device=dev) * 0.02
        g = torch.empty(shape, device=dev)
        hp = S.hparams(0.9, 0.999, 1e-30, 1.0, 0.1, S.POLICY_TIERED)
        w_ref, w_na = w0.clone(), w0.clone()
        ref = S.SkewAdam([(w_ref, g, tier)], hp)
        nbytes = ref.state_bytes
        state = torch.zeros(nbytes // 4, dtype=torch.float32, device=dev)
        stream = torch.cuda.current_stream().cuda_stream
        for t in (1, 2):
            g.copy_(torch.randn(shape, device=dev) * 1e-3)
            ref.step(t, 1e-3, 5)
            S.skew_step_tensor_noalloc(w_na.data_ptr(), g.data_ptr(), len(shape), shape[0],
                                       shape[1] if len(shape) == 2 else 0, tier, S.F_FP32, hp, state.data_ptr(),
                                       nbytes, 0, t, 1e-3, 5, stream)
            torch.cuda.synchronize()
            assert torch.equal(w_ref, w_na), f"fp32 weights differ at step {t}"
            assert torch.equal(ref.state[:nbytes].view(torch.float32), state)
        ref.close()


def test_noalloc_reports_a_timed_out_wait_once_then_steps_in_parity():
    """The self-test makes one bounded wait give up against the no-alloc status word (no
    fault: an mbarrier phase that nothing completes). The next skew_noalloc_sync_status
    reports SKEW_ETIMEOUT and clears the word; a read after that is clean, and whole-row
    steps through the entry point keep matching the regular path bit for bit."""
    dev = torch.device("cuda")
    stream = torch.cuda.current_stream().cuda_stream
    S.skew_noalloc_sync_status(stream)            # whatever an earlier test left is cleared
    shape, tier = (8192, 4096), S.TIER_EXPERT
    torch.manual_seed(3)
    w0 = (torch.randn(shape, device=dev) * 0.02).to(torch.bfloat16)
    g = torch.empty(shape, dtype=torch.bfloat16, device=dev)
    hp = S.hparams(0.9, 0.999, 1e-30, 1.0, 0.1, S.POLICY_TIERED)
    w_ref, w_na = w0.clone(), w0.clone()
    ref = S.SkewAdam([(w_ref, g, tier)], hp)
    nbytes = ref.state_bytes
    state = torch.zeros(nbytes // 4, dtype=torch.float32, device=dev)
    S.skew_noalloc_selftest_wait_timeout(stream)
    for t in (1, 2):
        g.copy_((torch.randn(shape, device=dev) * 1e-3).to(torch.bfloat16))
        ref.step(t, 1e-3, 91)
        S.skew_step_tensor_noalloc(w_na.data_ptr(), g.data_ptr(), 2, shape[0], shape[1], tier, 0, hp,
                                   state.data_ptr(), nbytes, 0, t, 1e-3, 91, stream)
        if t == 1:
            with pytest.raises(S.SkewError) as e:
                S.skew_noalloc_sync_status(stream)
            assert e.value.code == S.SKEW_ETIMEOUT
            S.skew_noalloc_sync_status(stream)    # reported once: the word is clear again
        torch.cuda.synchronize()
        assert torch.equal(w_ref.view(torch.int16), w_na.view(torch.int16)), f"weights differ at step {t}"
        assert torch.equal(ref.state[:nbytes].view(torch.float32), state), f"state differs at step {t}"
    S.skew_noalloc_sync_status(stream)
    ref.sync_status()
    ref.close()
