"""Failure detection on the GPU without a fault: a bounded device wait that runs out.

skew_selftest_wait_timeout makes one thread wait, as the whole-row kernels wait for a
copied chunk, on an mbarrier phase that nothing completes. The wait gives up after its
poll limit and records the timeout in the handle's status word. skew_sync_status must
then report SKEW_ETIMEOUT and clear the word, and the same context and handle must keep
stepping in parity with the oracle (row-path matrices included, whose kernels use the
same bounded waits).
"""
import time

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


def test_wait_timeout_is_reported_and_context_survives():
    import parity
    E = WL.TIER_EXPERT
    wl = WL.Workload("rows", [WL.Spec("e300x4096", (300, 4096), E, expert=0),
                              WL.Spec("e2x200x1024", (2, 200, 1024), E),
                              WL.Spec("norm", (4096,), WL.TIER_BACKBONE)], WL.HP(), "normal", steps=3)
    h = parity.Harness(wl, device="cuda:0")
    assert h.opt.info(0).rowpath == 1
    h.step(1)
    stream = torch.cuda.current_stream().cuda_stream
    t0 = time.monotonic()
    S.skew_selftest_wait_timeout(h.opt.h, stream)
    with pytest.raises(S.SkewError) as err:
        S.skew_sync_status(h.opt.h, stream)
    assert err.value.code == S.SKEW_ETIMEOUT
    assert time.monotonic() - t0 < 60          # bounded: about two seconds at most
    S.skew_sync_status(h.opt.h, stream)        # the word was cleared
    h.step(2)                                  # the context and the handle still work
    h.step(3)
    h.opt.sync_status()
    h.close()

