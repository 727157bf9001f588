"""Failure detection on the GPU without a fault: the bounded waits of the
kernels give up after their wall-clock limit, record AVITS_ERR_TIMEOUT in the
status word, release the other roles of the CTA through the abort flag, and
leave the context usable.  The wait that times out is on an mbarrier nothing
arrives at (a flag that nothing sets); every wait in it is bounded."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def av():
    import paper_2608_17995_gb300 as av
    av.build()
    av.lib()
    return av


@pytest.mark.parametrize("limit_ns", [200_000, 2_000_000])
def test_bounded_wait_times_out_and_releases_the_other_role(av, limit_ns):
    import torch
    res = torch.full((5,), -1, dtype=torch.int64, device="cuda")
    assert av.avits_device_status() == 0
    av.avits_selftest_bounded_wait(limit_ns, res)
    st = av.avits_device_status()
    r = res.cpu().tolist()
    assert st == 4                      # AVITS_ERR_TIMEOUT, read by the host
    assert r[0] == 0 and r[2] == 0      # neither wait completed
    assert r[4] == 1                    # the timing-out warp raised the abort flag
    assert r[1] >= limit_ns             # it waited at least its limit
    assert r[1] < limit_ns + 50_000_000
    # warp 1 (limit 100x) was released by the abort flag, not by its own timer
    assert r[3] < 50 * limit_ns
    assert av.avits_device_status() == 0   # the word was cleared


def test_context_usable_after_a_timeout(av):
    """A real call right after a timed-out wait runs and is correct."""
    import torch
    import oracle as orc
    from paper_2608_17995_gb300.workloads import random_scores
    res = torch.zeros(5, dtype=torch.int64, device="cuda")
    av.avits_selftest_bounded_wait(100_000, res)
    assert av.avits_device_status() == 4
    A, V = random_scores(3, 2, 1024, ties=True)
    k = 307
    dev = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
    sel = torch.empty(2, k, dtype=torch.int32, device="cuda")
    off = torch.empty(2, 1024, dtype=torch.int32, device="cuda")
    av.avits_fuse_select(dev(A), dev(V), 0.5, k, sel, off)
    assert av.avits_device_status() == 0
    sel_o, _, off_o = orc.topk(orc.fuse(A, V, 0.5), k)
    assert np.array_equal(sel.cpu().numpy(), sel_o)
    assert np.array_equal(off.cpu().numpy(), off_o)
