"""Failure detection on the GPU without a fault: a bounded wait that runs out.

Every wait inside the library's kernels is bounded. This test makes one run out
(an mbarrier that nothing completes, through the library's own bounded wait)
and checks that the kernel gives up after the budget, that the host reads the
TIMEOUT bit from the device status word, and that the context stays usable.
"""
import time

import pytest
import torch

from paper_2608_25332_gb300 import provip as P

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import __graft_entry__
    __graft_entry__.build()
    yield
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, f"device status {rc} {bits}"


def test_bounded_wait_gives_up_and_the_host_reads_it():
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0, "status not clean before the test"
    t0 = time.time()
    P.provip_selftest_wait_timeout(DEV)
    rc, bits = P.provip_device_status(clear=True)  # synchronises
    waited = time.time() - t0
    assert rc == P.ERR_TIMEOUT and bits & P.DEVSTAT_TIMEOUT, (rc, bits)
    assert 1.9 < waited < 30.0, f"the wait gave up after {waited:.2f} s (budget 2 s)"
    # the context is still usable, and the cleared word stays clear
    s = torch.rand(3, 1000, device=DEV)
    idx = P.provip_topk(s, 17)
    ref = torch.sort(torch.topk(s, 17, dim=1).indices, dim=1).values.to(torch.int32)
    assert torch.equal(idx, ref)
    rc, bits = P.provip_device_status(clear=True)
    assert rc == 0 and bits == 0
