"""Failure detection on the GPU, without a fault: every pipeline wait in the
library is bounded, and a wait that gives up raises CURE_DEVERR_TIMEOUT in
the device error word instead of hanging the GPU.  The self-test entry point
runs that same bounded wait on a barrier nothing ever completes; the status
must come back through cure_device_error() and the context must stay usable.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_00531_gb300 import workload as W

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda:0")


@pytest.fixture(scope="module")
def cure():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import cure as c
    torch.cuda.set_device(DEV)
    return c


def test_bounded_wait_reports_a_timeout_and_the_context_stays_usable(cure):
    from paper_2608_00531_gb300 import _lib
    assert cure.cure_device_error() in (0, _lib.DEVERR_TIMEOUT)   # start from a clear word
    assert cure.cure_device_error() == 0
    cure.cure_selftest_wait_timeout(1 << 22)          # about 2 ms of SM clock
    assert cure.cure_device_error() == _lib.DEVERR_TIMEOUT
    assert cure.cure_device_error() == 0              # reading cleared it
    # the context still runs kernels, with correct results
    rng = np.random.default_rng(1)
    x = W.to_bf16(rng.standard_normal((6, 3001)).astype(np.float32))
    ids, vals, margin, logp1 = cure.cure_score_draft(x.to(DEV), 3)
    o_ids, _, o_m, _, _ = oracle.score_draft(W.bf16_to_f64(x), 3)
    assert np.array_equal(ids.cpu().numpy(), o_ids)
    assert np.array_equal(margin.cpu().numpy(), o_m.astype(np.float32))
    assert cure.cure_device_error() == 0
