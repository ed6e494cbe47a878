"""mpm_merge_no_alloc, the merge for callers that cannot allocate.

Such a caller (a plug-in inside a framework that owns the whole device
memory pool, or a loop where cudaMalloc's blocking is not allowed) cannot
provide mpm_merge's workspace; the library then uses its own fixed scratch
array.  These tests call that entry point through the C ABI, twice in a row
on different batches and dtypes (so the second call starts from the first
call's leftovers in the shared array), and require each result to be
bitwise equal to mpm_merge's (a merge is deterministic) and to pass the
oracle parity check.  They also check that an error left behind by a call
with bad offsets is reported and does not leak into the next call, that a
repeated call allocates no device memory, and the Python wrapper.  The file
is collected last so that a failure here stops a -x run only after every
other test ran; it also passes on its own in a fresh process.
"""

from __future__ import annotations

import ctypes

import numpy as np
import pytest
import torch

from parity import check_merge_batch, to_f64
from workloads import make_custom

pytestmark = pytest.mark.gpu

DEV = "cuda"
MPM_ERR_WORKSPACE, MPM_ERR_DEVICE_CHECK = 4, 6


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr() if t.numel() else None)


def _inputs(batch):
    return batch.tokens.to(DEV), torch.from_numpy(batch.offsets).to(DEV)


def _outputs(x, off):
    return (torch.empty_like(x), torch.empty(off.numel(), dtype=torch.int64, device=DEV),
            torch.empty(x.shape[0], dtype=torch.int32, device=DEV))


def _no_alloc_call(mpm, x, off, outs=None):
    """One call of the C entry point; outputs are preallocated by the caller."""
    rows, dim = x.shape
    out, out_off, out_map = outs if outs is not None else _outputs(x, off)
    dtype = 1 if x.dtype == torch.bfloat16 else 0
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    code = mpm.library().mpm_merge_no_alloc(_ptr(x), _ptr(off), off.numel() - 1, rows, dim, dtype, _ptr(out),
                                            _ptr(out_off), _ptr(out_map), stream)
    assert code == 0, mpm.mpm.status_string(code)
    return out, out_off, out_map


def _status(mpm) -> int:
    code = ctypes.c_int32(-1)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert mpm.library().mpm_no_alloc_get_device_status(ctypes.byref(code), stream) == 0
    return int(code.value)


def _bitwise_same(ref, got, rows):
    r_out, r_off, r_map = ref
    g_out, g_off, g_map = got
    assert torch.equal(r_off, g_off)
    assert torch.equal(r_map[:rows], g_map[:rows])
    t = int(r_off[-1])
    assert torch.equal(r_out[:t], g_out[:t])


def _oracle_check(mpm, batch, got, what):
    out, out_off, out_map = got
    x, off = _inputs(batch)
    nn, _ = mpm.nearest_neighbors(x, off, with_score=False)
    off_h = out_off.cpu().numpy()
    check_merge_batch(batch.tokens.double().numpy(), batch.offsets, nn.cpu().numpy(), out_map.cpu().numpy(),
                      to_f64(out[:off_h[-1]]), off_h, batch.dtype, what)


def test_no_alloc_matches_merge_twice_in_a_row(mpm):
    first = make_custom([1000, 1, 333, 0, 517], 384, "bf16", seed=31)
    second = make_custom([700, 64, 2], 96, "f32", seed=32)
    inputs = [_inputs(first), _inputs(second)]
    refs = [mpm.merge(x, off) for x, off in inputs]
    got = [_no_alloc_call(mpm, x, off) for x, off in inputs]  # two calls in a row
    torch.cuda.synchronize()
    assert _status(mpm) == 0
    _bitwise_same(refs[0], got[0], first.rows)
    _bitwise_same(refs[1], got[1], second.rows)
    _oracle_check(mpm, first, got[0], "no-alloc bf16")
    _oracle_check(mpm, second, got[1], "no-alloc fp32")


def test_error_left_behind_is_reported_and_cleared(mpm):
    """Non-monotone offsets: the kernels stay in bounds and report MPM_ERR_DEVICE_CHECK
    through the no-alloc status word; the next valid call starts clean."""
    x = torch.randn(150, 64, device=DEV).to(torch.bfloat16)
    bad = torch.tensor([0, 100, 50, 150], dtype=torch.int64, device=DEV)
    _no_alloc_call(mpm, x, bad)
    torch.cuda.synchronize()
    assert _status(mpm) == MPM_ERR_DEVICE_CHECK
    assert _status(mpm) == 0                       # reading the word clears it
    good = torch.tensor([0, 100, 150], dtype=torch.int64, device=DEV)
    _no_alloc_call(mpm, x, bad)                    # leaves an error in the shared array ...
    got = _no_alloc_call(mpm, x, good)             # ... which this call clears before it runs
    torch.cuda.synchronize()
    assert _status(mpm) == 0
    _bitwise_same(mpm.merge(x, good), got, 150)


def test_repeat_call_allocates_nothing(mpm):
    batch = make_custom([900, 450, 3], 256, "bf16", seed=33)
    x, off = _inputs(batch)
    outs = _outputs(x, off)
    _no_alloc_call(mpm, x, off, outs)
    torch.cuda.synchronize()
    torch_before = torch.cuda.memory_allocated()
    free_before, _ = torch.cuda.mem_get_info()
    _no_alloc_call(mpm, x, off, outs)
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info()
    assert torch.cuda.memory_allocated() == torch_before
    assert free_after == free_before
    _bitwise_same(mpm.merge(x, off), outs, batch.rows)


def test_python_wrapper(mpm):
    batch = make_custom([300, 77], 128, "f32", seed=34)
    x, off = _inputs(batch)
    got = mpm.merge_no_alloc(x, off, *_outputs(x, off))
    torch.cuda.synchronize()
    assert mpm.no_alloc_device_status() == 0
    _bitwise_same(mpm.merge(x, off), got, batch.rows)


def test_no_alloc_rejects_sizes_beyond_its_scratch(mpm):
    lib = mpm.library()
    limit = 8 << 20
    fake = ctypes.c_void_p(1 << 20)
    # bf16: about 20 bytes per row.
    assert lib.mpm_merge_workspace_size(400_000, 4, 64, 1) <= limit
    assert lib.mpm_merge_workspace_size(1 << 22, 4, 64, 1) > limit
    assert lib.mpm_merge_no_alloc(fake, fake, 4, 1 << 22, 64, 1, fake, fake, fake, None) == MPM_ERR_WORKSPACE
    # fp32: 20 + 8 * dim bytes per row (the tf32 split copies), so 1,360 rows at dim 768.
    assert lib.mpm_merge_workspace_size(1300, 2, 768, 0) <= limit
    assert lib.mpm_merge_workspace_size(1400, 2, 768, 0) > limit
    assert lib.mpm_merge_no_alloc(fake, fake, 2, 1400, 768, 0, fake, fake, fake, None) == MPM_ERR_WORKSPACE
    assert int(np.floor(limit / (20 + 8 * 192))) > 5000   # the header's 5,400 rows at dim 192
