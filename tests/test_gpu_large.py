"""GPU parity on tensors of more than 2^31 elements.

The paper's Sec. 3 footnote names the crash of 8-bit optimizers on tensors past 2^31
elements as the failure tiered state must avoid. Every index of the step is 64-bit;
these tests step two such tensors twice and compare them whole against the oracle:
  * an expert matrix of 524,800 x 4,096 (2,149,580,800 elements) on the whole-row path
    (k_rowsq / k_finalize / k_apply_rows, row tiles and partials past 2^31 elements);
  * a router-tier tensor of 2^31 + 37 elements kept as one vector (exact second moment,
    flat tiles on the scalar path: its length is not a multiple of 8, so the last tile
    is ragged).
Each needs about 9-26 GB of device memory and a few minutes of oracle time.
"""
import pytest
import torch

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


def _free_bytes():
    free, _ = torch.cuda.mem_get_info()
    return free


def test_expert_matrix_past_2_31_elements():
    n, m = 524_800, 4096
    assert n * m > 2**31
    if _free_bytes() < 3 * n * m * 2:
        pytest.skip("needs about 13 GB of free device memory")
    wl = WL.Workload("big_expert", [WL.Spec("e524800x4096", (n, m), WL.TIER_EXPERT, expert=0)], WL.HP(),
                     "normal", steps=2)
    h = _harness(wl)
    assert h.opt.info(0).rowpath == 1
    for t in (1, 2):
        rep = h.step(t, seed=2**33 + t)
        assert rep.elements == n * m
    h.close()


def test_vector_past_2_31_elements():
    numel = 2**31 + 37
    if _free_bytes() < 4 * numel * 2 + 4 * numel:
        pytest.skip("needs about 26 GB of free device memory")
    wl = WL.Workload("big_vector", [WL.Spec("router_flat", (numel,), WL.TIER_ROUTER)], WL.HP(), "normal", steps=2)
    h = _harness(wl)
    for t in (1, 2):
        rep = h.step(t, seed=5 + t)
        assert rep.elements == numel
    h.close()
