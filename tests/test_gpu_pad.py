"""GPU parity of the padded-batch entry points (mpm_pad_batch / mpm_unpad_batch)
against the oracle's definition: images padded to a common length with a key
mask, as the paper batches merged sequences for dense attention (Section 4).
Bit-exact: both are copies."""

from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from parity import to_f64
from workloads import DTYPES, make_custom

pytestmark = pytest.mark.gpu

DEV = "cuda"
COUNTS = [300, 0, 1, 257, 33, 1024, 2]


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


def _i64(a):
    return torch.from_numpy(np.asarray(a, dtype=np.int64)).to(DEV)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("extra", [0, 5])
def test_pad_matches_oracle_and_roundtrips(mpm, dtype, extra):
    batch = make_custom(COUNTS, 96, dtype, seed=21)
    x = batch.tokens.to(DEV)
    off = _i64(batch.offsets)
    L = int(np.diff(batch.offsets).max()) + extra
    status = torch.zeros(2, dtype=torch.int32, device=DEV)
    out, mask, stats = mpm.pad_batch(x, off, L, device_status=status)
    want, want_mask, want_stats = oracle.pad_batch(batch.tokens.double().numpy(), batch.offsets, L)
    assert np.array_equal(to_f64(out), want)
    assert np.array_equal(mask.cpu().numpy(), want_mask)
    assert tuple(stats.cpu().tolist()) == want_stats
    back = mpm.unpad_batch(out, off, rows=batch.rows, device_status=status)
    assert torch.equal(back, x)
    assert int(status[0]) == 0


def test_pad_cuts_and_reports_long_images(mpm):
    batch = make_custom(COUNTS, 64, "bf16", seed=22)
    x = batch.tokens.to(DEV)
    off = _i64(batch.offsets)
    L = 40
    status = torch.zeros(2, dtype=torch.int32, device=DEV)
    out, mask, _ = mpm.pad_batch(x, off, L, device_status=status)
    want, want_mask, _ = oracle.pad_batch(batch.tokens.double().numpy(), batch.offsets, L)
    assert np.array_equal(to_f64(out), want)
    assert np.array_equal(mask.cpu().numpy(), want_mask)
    assert int(status[0]) == 6  # MPM_ERR_DEVICE_CHECK: an image longer than L
    assert int(status[1]) in [b for b, n in enumerate(COUNTS) if n > L]


def test_pad_merged_output_for_attention(mpm):
    """The use the paper makes of it: pad a merge's packed output to the longest merged image."""
    batch = make_custom([500, 260, 129, 1], 128, "bf16", seed=23)
    x = batch.tokens.to(DEV)
    off = _i64(batch.offsets)
    ws = mpm.new_workspace(x.shape[0], 4, 128, x.dtype, DEV)
    x1, off1, _ = mpm.merge(x, off, workspace=ws)
    o1 = off1.cpu().numpy()
    n1 = np.diff(o1)
    assert n1.max() <= 500 and n1.min() >= 1
    out, mask, stats = mpm.pad_batch(x1, off1, int(n1.max()))
    want, want_mask, want_stats = oracle.pad_batch(to_f64(x1[:o1[-1]]), o1, int(n1.max()))
    assert np.array_equal(to_f64(out), want)
    assert np.array_equal(mask.cpu().numpy(), want_mask)
    assert tuple(stats.cpu().tolist()) == want_stats
    assert out.dtype == DTYPES["bf16"]
