"""The C-ABI library: builds, loads, exports every declared entry point, and
rejects bad arguments on the host (no GPU needed: validation happens before
any CUDA call)."""

from __future__ import annotations

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mpm.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2604_05718_gb300 import build, mpm

    build.build()
    return mpm.library()


def declared_entry_points() -> list:
    text = open(HEADER).read()
    return re.findall(r"MPM_API\s+[\w\s\*]+?\b(mpm_\w+)\s*\(", text)


def test_header_declares_the_boundary():
    names = declared_entry_points()
    for want in ("mpm_merge", "mpm_compose_maps", "mpm_unmerge_gather", "mpm_nearest_neighbors",
                 "mpm_merge_workspace_size", "mpm_get_device_status", "mpm_status_string"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_entry_points():
        assert hasattr(lib, name), name


def test_only_mpm_symbols_exported(lib):
    import subprocess

    from paper_2604_05718_gb300 import mpm

    out = subprocess.run(["readelf", "-Ws", "--dyn-syms", mpm.LIB_PATH], capture_output=True, text=True).stdout
    exported = set()
    for line in out.splitlines():
        f = line.split()
        if len(f) >= 8 and f[3] == "FUNC" and f[4] == "GLOBAL" and f[6] != "UND":
            exported.add(f[7].split("@")[0])
    assert exported == set(declared_entry_points())


def test_version_and_status_strings(lib):
    assert lib.mpm_abi_version() == 1
    for code in range(9):
        assert lib.mpm_status_string(code)
    assert lib.mpm_status_string(99) == b"unknown status"


def test_workspace_size(lib):
    n = lib.mpm_merge_workspace_size(65536, 64, 768, 1)
    assert n >= 65536 * (4 + 8 + 8) and n % 256 == 0
    assert lib.mpm_merge_workspace_size(-1, 4, 64, 1) == 0
    assert lib.mpm_merge_workspace_size(10, 0, 64, 1) == 0
    assert lib.mpm_merge_workspace_size(10, 4, 64, 7) == 0
    # Grows with rows and batch.
    assert lib.mpm_merge_workspace_size(2000, 4, 64, 1) > lib.mpm_merge_workspace_size(1000, 4, 64, 1)


P = ctypes.c_void_p
FAKE = 1 << 20  # 16-byte aligned stand-in address; never dereferenced on these paths


def merge(lib, tokens=FAKE, offsets=FAKE, batch=2, rows=100, dim=64, dtype=1, out=FAKE * 64,
          out_off=FAKE, out_map=FAKE, ws=FAKE, ws_bytes=1 << 30):
    return lib.mpm_merge(P(tokens), P(offsets), batch, rows, dim, dtype, P(out), P(out_off), P(out_map), P(ws),
                         ws_bytes, None)


def test_merge_argument_validation(lib):
    assert merge(lib, batch=0) == 1                    # no images
    assert merge(lib, rows=-1) == 1
    assert merge(lib, offsets=None) == 1
    assert merge(lib, out_off=None) == 1
    assert merge(lib, dtype=5) == 1
    assert merge(lib, dim=0) == 1
    assert merge(lib, dim=20000) == 2                  # beyond MPM_MAX_DIM
    assert merge(lib, dim=12) == 3                     # 24-byte bf16 rows
    assert merge(lib, dim=6, dtype=0) == 3             # 24-byte fp32 rows
    assert merge(lib, tokens=FAKE + 8) == 3            # misaligned tokens
    assert merge(lib, out=FAKE * 64 + 4) == 3
    assert merge(lib, out=FAKE + 64) == 8              # output overlaps input
    assert merge(lib, ws=None) == 4
    assert merge(lib, ws=FAKE + 16) == 4               # workspace not 256-byte aligned
    assert merge(lib, ws_bytes=16) == 4


def test_nn_compose_gather_validation(lib):
    nn = lib.mpm_nearest_neighbors
    assert nn(P(FAKE), P(FAKE), 1, 10, 64, 1, 0, None, None, P(FAKE), 1 << 20, None) == 1
    assert nn(P(FAKE), P(FAKE), 1, 10, 64, 0, 2, P(FAKE), None, P(FAKE), 1 << 20, None) == 2  # tcgen05 needs bf16
    assert nn(P(FAKE), P(FAKE), 1, 10, 64, 1, 9, P(FAKE), None, P(FAKE), 1 << 20, None) in (1, 5)
    comp = lib.mpm_compose_maps
    assert comp(P(FAKE), None, 10, P(FAKE), P(FAKE), 10, 1, P(FAKE), None, None) == 1
    assert comp(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 0, P(FAKE), None, None) == 1
    assert comp(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, P(FAKE + 8), None, None) == 8  # out aliases map2
    gat = lib.mpm_unmerge_gather
    assert gat(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 64, 1, None, None, None) == 1
    assert gat(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 64, 1, P(FAKE + 128), None, None) == 8
    assert gat(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 60, 1, P(FAKE * 8), None, None) == 3
    cg = lib.mpm_compose_gather
    # (merged, merged_offsets, merged_rows, map1, offsets0, rows0, map2, offsets1, rows1, batch, dim, dtype,
    #  out, out_map, device_status, stream)
    assert cg(P(FAKE), None, 10, P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 64, 1, P(FAKE * 8), None, None,
              None) == 1                                                                   # no merged offsets
    assert cg(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 64, 1, None, None, None,
              None) == 1                                                                   # no output
    assert cg(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 64, 1, P(FAKE + 128), None,
              None, None) == 8                                                             # out overlaps merged
    assert cg(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, P(FAKE * 4), P(FAKE), 10, 1, 64, 1, P(FAKE * 8),
              P(FAKE * 4 + 8), None, None) == 8                                            # out_map overlaps map2
    assert cg(P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, P(FAKE), P(FAKE), 10, 1, 60, 1, P(FAKE * 8), None,
              None, None) == 3                                                             # rows not 16-byte multiples
    pad = lib.mpm_pad_batch
    # (tokens, offsets, batch, rows, dim, dtype, max_len, out, out_mask, out_stats, device_status, stream)
    assert pad(P(FAKE), None, 2, 10, 64, 1, 8, P(FAKE * 8), None, None, None, None) == 1         # no offsets
    assert pad(P(FAKE), P(FAKE), 2, 10, 64, 1, -1, P(FAKE * 8), None, None, None, None) == 1     # negative L
    assert pad(P(FAKE), P(FAKE), 2, 10, 64, 1, 8, None, None, None, None, None) == 1             # no output
    assert pad(P(FAKE), P(FAKE), 2, 10, 64, 1, 8, P(FAKE + 128), None, None, None, None) == 8    # out overlaps tokens
    assert pad(P(FAKE), P(FAKE), 2, 10, 64, 1, 8, P(FAKE * 8 + 4), None, None, None, None) == 3  # unaligned out
    unpad = lib.mpm_unpad_batch
    # (padded, batch, max_len, dim, dtype, offsets, rows, out, device_status, stream)
    assert unpad(P(FAKE), 2, 8, 64, 1, None, 10, P(FAKE * 8), None, None) == 1                   # no offsets
    assert unpad(P(FAKE), 2, 8, 64, 1, P(FAKE), 10, None, None, None) == 1                       # no output
    assert unpad(P(FAKE), 2, 8, 64, 1, P(FAKE), 10, P(FAKE + 128), None, None) == 8              # out overlaps padded
    assert unpad(P(FAKE), 2, 8, 60, 1, P(FAKE), 10, P(FAKE * 8), None, None) == 3                # 120-byte rows
    mc = lib.mpm_merge_chunked
    # (tokens, offsets, batch, rows, dim, dtype, chunk, out_tokens, out_offsets, out_map, workspace, bytes, stream)
    args = (P(FAKE), P(FAKE), 1, 10, 64, 1)
    outs = (P(FAKE * 8), P(FAKE * 16), P(FAKE * 24), P(FAKE * 32), 1 << 24, None)
    assert mc(*args, -1, *outs) == 1     # negative chunk
    assert mc(*args, 100, *outs) == 2    # not a whole number of 256-token tiles
    nnc = lib.mpm_nearest_neighbors_chunked
    # (tokens, offsets, batch, rows, dim, dtype, algo, chunk, out_nn, out_score, workspace, bytes, stream)
    assert nnc(P(FAKE), P(FAKE), 1, 10, 64, 1, 2, 256, P(FAKE * 8), None, P(FAKE * 32), 1 << 24, None) == 2
    assert nnc(P(FAKE), P(FAKE), 1, 10, 64, 1, 4, -256, P(FAKE * 8), None, P(FAKE * 32), 1 << 24, None) == 1
    assert lib.mpm_get_device_status(None, None, None) == 1
    assert lib.mpm_no_alloc_get_device_status(None, None) == 1   # checked before any CUDA call


def test_ordinary_library_has_no_timeline(lib):
    import numpy as np

    out = np.zeros(18, dtype=np.uint64)
    assert lib.mpm_trace_read(out.ctypes.data) == 2   # MPM_ERR_UNSUPPORTED
    assert lib.mpm_trace_reset() == 2
