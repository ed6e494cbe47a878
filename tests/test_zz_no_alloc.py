"""mpm_merge_no_alloc, the merge for callers that cannot allocate.

Such a caller (a plug-in inside a framework that owns the whole device
memory pool, or a loop where cudaMalloc's blocking is not allowed) cannot
provide mpm_merge's workspace; the library then uses its own fixed scratch
array.  This file calls that entry point through the C ABI, twice in a row on
different batches and dtypes (so the second call starts from the first
call's leftovers in the shared array), and checks each result against
mpm_merge's with the tolerance the other parity tests use.  It is collected
last so that a failure here stops a -x run only after every other test ran;
it also passes on its own in a fresh process.
"""

from __future__ import annotations

import ctypes

import pytest
import torch

from parity import TOL, check_rowwise_tolerance, to_f64
from workloads import make_custom

pytestmark = pytest.mark.gpu

DEV = "cuda"


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
    x = batch.tokens.to(DEV)
    off = torch.from_numpy(batch.offsets).to(DEV)
    return x, off


def _no_alloc_call(mpm, x, off):
    """One call of the C entry point; outputs are preallocated by the caller."""
    rows, dim = x.shape
    out = torch.empty_like(x)
    out_off = torch.empty(off.numel(), dtype=torch.int64, device=DEV)
    out_map = torch.empty(rows, dtype=torch.int32, device=DEV)
    dtype = 1 if x.dtype == torch.bfloat16 else 0
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    code = mpm.library().mpm_merge_no_alloc(_ptr(x), _ptr(off), off.numel() - 1, rows, dim, dtype, _ptr(out),
                                            _ptr(out_off), _ptr(out_map), stream)
    assert code == 0, mpm.mpm.status_string(code)
    return out, out_off, out_map


def _same(ref, got, rows, dtype):
    r_out, r_off, r_map = ref
    g_out, g_off, g_map = got
    assert torch.equal(r_off, g_off)
    assert torch.equal(r_map[:rows], g_map[:rows])
    t = int(r_off[-1])
    want, have = to_f64(r_out[:t]), to_f64(g_out[:t])
    check_rowwise_tolerance(have, want, TOL[dtype], "no-alloc merge")


def test_no_alloc_matches_merge_twice_in_a_row(mpm):
    first = make_custom([1000, 1, 333, 0, 517], 384, "bf16", seed=31)
    second = make_custom([700, 64, 2], 96, "f32", seed=32)
    inputs = [_inputs(first), _inputs(second)]
    refs = [mpm.merge(x, off) for x, off in inputs]
    got = [_no_alloc_call(mpm, x, off) for x, off in inputs]  # two calls in a row
    torch.cuda.synchronize()
    _same(refs[0], got[0], first.rows, "bf16")
    _same(refs[1], got[1], second.rows, "f32")


def test_no_alloc_rejects_sizes_beyond_its_scratch(mpm):
    lib = mpm.library()
    limit = 8 << 20
    rows = 1 << 22
    assert lib.mpm_merge_workspace_size(rows, 4, 64, 1) > limit
    fake = ctypes.c_void_p(1 << 20)
    code = lib.mpm_merge_no_alloc(fake, fake, 4, rows, 64, 1, fake, fake, fake, None)
    assert code == 4  # MPM_ERR_WORKSPACE, before any launch
