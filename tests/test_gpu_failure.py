"""Failure detection on the GPU without a fault: a kernel wait that runs out.

mpm_selftest_wait_timeout waits, with the bounded wait of the tensor-core
kernels, on a barrier that nothing completes.  The wait must give up after
its limit, record MPM_ERR_DEVICE_TIMEOUT in the status word and return, and
the context must stay usable: a merge right after it still matches the
oracle.
"""

from __future__ import annotations

import time

import numpy as np
import pytest
import torch

from parity import check_merge_batch, to_f64
from workloads import make_custom

pytestmark = pytest.mark.gpu

MPM_ERR_DEVICE_TIMEOUT = 7


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


def test_wait_that_nothing_completes_times_out_and_reports(mpm):
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    status = mpm.selftest_wait_timeout(20000)  # 20 ms
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert status.cpu().tolist() == [MPM_ERR_DEVICE_TIMEOUT, 99]
    assert 0.02 <= elapsed < 5.0, elapsed


def test_context_usable_after_a_timeout(mpm):
    status = mpm.selftest_wait_timeout(1000)
    batch = make_custom([300, 77, 1, 0], 128, "bf16", seed=5)
    x = batch.tokens.cuda()
    off = torch.from_numpy(batch.offsets).cuda()
    out, out_off, rmap = mpm.merge(x, off)
    torch.cuda.synchronize()
    assert status.cpu().tolist()[0] == MPM_ERR_DEVICE_TIMEOUT
    t = int(out_off[-1])
    rows = batch.rows
    nn, _ = mpm.nearest_neighbors(x, off)
    check_merge_batch(batch.tokens.double().numpy(), batch.offsets, nn.cpu().numpy()[:rows],
                      rmap.cpu().numpy()[:rows], to_f64(out[:t]), out_off.cpu().numpy(), "bf16", "after timeout")


def test_invalid_limits_are_rejected_on_the_host(mpm):
    with pytest.raises(mpm.MPMError):
        mpm.selftest_wait_timeout(0)
    with pytest.raises(mpm.MPMError):
        mpm.selftest_wait_timeout(20_000_000)
