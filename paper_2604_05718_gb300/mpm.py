"""Python binding of the MPM C ABI (libmpm.so) through ctypes.

Argument marshalling only: tensors are checked for device, dtype and layout,
outputs and workspace are allocated with torch (device memory is torch's
job), and every step of the computation runs in the library's CUDA kernels
on the caller's current torch stream.  There is no CPU fallback: without the
compiled library every call raises.

Names follow the paper (arxiv 2604.05718): ``merge`` is one MPM call
(Algorithm 1), ``compose_maps`` is Eq. 3 and ``unmerge_gather`` is Eq. 4.
"""

from __future__ import annotations

import ctypes
import os

import torch

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmpm.so")
# The same library with the device timeline compiled in (build(trace=True)).
TRACE_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmpm_trace.so")
TRACE_KINDS = ("prep", "affinity", "mutual_scan", "pair_average", "gather", "compose")

MPM_F32, MPM_BF16 = 0, 1
ALGOS = {"auto": 0, "simt": 1, "tcgen05": 2, "tcgen05_sym": 3, "tcgen05_pair": 4}
STATUS_NAMES = {
    0: "MPM_OK", 1: "MPM_ERR_INVALID_ARG", 2: "MPM_ERR_UNSUPPORTED", 3: "MPM_ERR_ALIGNMENT",
    4: "MPM_ERR_WORKSPACE", 5: "MPM_ERR_CUDA", 6: "MPM_ERR_DEVICE_CHECK", 7: "MPM_ERR_DEVICE_TIMEOUT",
    8: "MPM_ERR_ALIASING",
}
EXPORTS = ("mpm_abi_version", "mpm_status_string", "mpm_merge_workspace_size", "mpm_merge", "mpm_merge_timed",
           "mpm_compose_maps", "mpm_unmerge_gather", "mpm_nearest_neighbors", "mpm_get_device_status",
           "mpm_merge_no_alloc", "mpm_no_alloc_get_device_status", "mpm_compose_gather", "mpm_pad_batch",
           "mpm_unpad_batch", "mpm_merge_chunked", "mpm_nearest_neighbors_chunked")

_lib = None


class MPMError(RuntimeError):
    """A non-OK status returned by the C ABI."""

    def __init__(self, fn: str, code: int):
        self.code = code
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(code, code)} ({status_string(code)})")


def _declare(lib: ctypes.CDLL) -> None:
    P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    sigs = {
        "mpm_abi_version": (I32, []),
        "mpm_status_string": (ctypes.c_char_p, [ctypes.c_int]),
        "mpm_merge_workspace_size": (SZ, [I64, I32, I32, ctypes.c_int]),
        "mpm_merge": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, P, P, P, P, SZ, P]),
        "mpm_merge_timed": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, P, P, P, P, SZ, P, P]),
        "mpm_compose_maps": (ctypes.c_int, [P, P, I64, P, P, I64, I32, P, P, P]),
        "mpm_unmerge_gather": (ctypes.c_int, [P, P, I64, P, P, I64, I32, I32, ctypes.c_int, P, P, P]),
        "mpm_nearest_neighbors": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, ctypes.c_int, P, P, P,
                                                 SZ, P]),
        "mpm_get_device_status": (ctypes.c_int, [P, P, P]),
        "mpm_merge_no_alloc": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, P, P, P, P]),
        "mpm_no_alloc_get_device_status": (ctypes.c_int, [P, P]),
        "mpm_compose_gather": (ctypes.c_int, [P, P, I64, P, P, I64, P, P, I64, I32, I32, ctypes.c_int, P, P, P,
                                              P]),
        "mpm_pad_batch": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, I64, P, P, P, P, P]),
        "mpm_merge_chunked": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, I64, P, P, P, P, SZ, P]),
        "mpm_nearest_neighbors_chunked": (ctypes.c_int, [P, P, I32, I64, I32, ctypes.c_int, ctypes.c_int, I64, P, P,
                                                         P, SZ, P]),
        "mpm_unpad_batch": (ctypes.c_int, [P, I32, I64, I32, ctypes.c_int, P, I64, P, P, P]),
        "mpm_selftest_wait_timeout": (ctypes.c_int, [P, ctypes.c_uint32, P]),
        "mpm_trace_read": (ctypes.c_int, [P]),
        "mpm_trace_reset": (ctypes.c_int, []),
    }
    for name, (res, args) in sigs.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args


def library(path: str | None = None) -> ctypes.CDLL:
    """Loads libmpm.so once; raises if it has not been built."""
    global _lib
    if _lib is None:
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"MPM CUDA library missing ({p}); build it with "
                               "paper_2604_05718_gb300.build.build()")
        lib = ctypes.CDLL(p)
        _declare(lib)
        _lib = lib
    return _lib


def status_string(code: int) -> str:
    return library().mpm_status_string(int(code)).decode()


def _check(fn: str, code: int) -> None:
    if code != 0:
        raise MPMError(fn, code)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return MPM_BF16
    if t.dtype == torch.float32:
        return MPM_F32
    raise TypeError(f"tokens must be bfloat16 or float32, got {t.dtype}")


def _cuda(t: torch.Tensor, name: str, dtype=None, ndim=None) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dimensions")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _stream(dev: torch.device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)


def _ptr(t: torch.Tensor | None) -> ctypes.c_void_p:
    return ctypes.c_void_p(t.data_ptr() if t is not None and t.numel() > 0 else None)


def workspace_size(rows: int, batch: int, dim: int, dtype: torch.dtype) -> int:
    code = MPM_BF16 if dtype == torch.bfloat16 else MPM_F32
    n = library().mpm_merge_workspace_size(int(rows), int(batch), int(dim), code)
    if n == 0:
        raise ValueError("invalid sizes for the MPM workspace")
    return int(n)


def new_workspace(rows: int, batch: int, dim: int, dtype: torch.dtype, device) -> torch.Tensor:
    """Device scratch for merge / nearest_neighbors (uint8, 256-byte aligned)."""
    return torch.empty(workspace_size(rows, batch, dim, dtype), dtype=torch.uint8, device=device)


def merge(tokens: torch.Tensor, offsets: torch.Tensor, workspace: torch.Tensor | None = None,
          out_tokens: torch.Tensor | None = None, out_offsets: torch.Tensor | None = None,
          out_map: torch.Tensor | None = None, stage_events: list | None = None, chunk: int = 0):
    """One MPM call on a packed batch (Algorithm 1).

    tokens [rows, D] bf16/fp32 and offsets int64 [B+1] on the same GPU.
    Returns (out_tokens [rows, D], out_offsets int64 [B+1], out_map int32 [rows]);
    the first out_offsets[B] rows of out_tokens are the merged tokens.
    stage_events: optional 8 torch.cuda.Event (timing enabled, already
    recorded once so that they exist) bracketing the four kernels.
    chunk: > 0 restricts every token's nearest-neighbour search to its run of
    `chunk` consecutive tokens (mpm_merge_chunked; a multiple of 256).
    """
    _cuda(tokens, "tokens", ndim=2)
    _cuda(offsets, "offsets", torch.int64, 1)
    dev = tokens.device
    rows, dim = tokens.shape
    batch = offsets.numel() - 1
    if workspace is None:
        workspace = new_workspace(rows, batch, dim, tokens.dtype, dev)
    if out_tokens is None:
        out_tokens = torch.empty_like(tokens)
    if out_offsets is None:
        out_offsets = torch.empty(batch + 1, dtype=torch.int64, device=dev)
    if out_map is None:
        out_map = torch.empty(rows, dtype=torch.int32, device=dev)
    events = None
    if stage_events is not None:
        if len(stage_events) != 8:
            raise ValueError("stage_events needs 8 events")
        events = (ctypes.c_void_p * 8)(*[ctypes.c_void_p(e.cuda_event) for e in stage_events])
    if chunk and stage_events is not None:
        raise ValueError("stage_events are only recorded by the unchunked merge")
    with torch.cuda.device(dev):
        if chunk:
            code = library().mpm_merge_chunked(_ptr(tokens), _ptr(offsets), batch, rows, dim, _dtype_code(tokens),
                                               int(chunk), _ptr(out_tokens), _ptr(out_offsets), _ptr(out_map),
                                               _ptr(workspace), workspace.numel(), _stream(dev))
        else:
            code = library().mpm_merge_timed(_ptr(tokens), _ptr(offsets), batch, rows, dim, _dtype_code(tokens),
                                             _ptr(out_tokens), _ptr(out_offsets), _ptr(out_map), _ptr(workspace),
                                             workspace.numel(), _stream(dev), events)
    _check("mpm_merge", code)
    return out_tokens, out_offsets, out_map


def nearest_neighbors(tokens: torch.Tensor, offsets: torch.Tensor, algo: str = "auto",
                      workspace: torch.Tensor | None = None, with_score: bool = True, chunk: int = 0):
    """b(i) (local index, -1 when alone) and its fp32 cosine, per token (within chunks if chunk > 0)."""
    _cuda(tokens, "tokens", ndim=2)
    _cuda(offsets, "offsets", torch.int64, 1)
    dev = tokens.device
    rows, dim = tokens.shape
    batch = offsets.numel() - 1
    if workspace is None:
        workspace = new_workspace(rows, batch, dim, tokens.dtype, dev)
    nn = torch.empty(rows, dtype=torch.int32, device=dev)
    score = torch.empty(rows, dtype=torch.float32, device=dev) if with_score else None
    with torch.cuda.device(dev):
        if chunk:
            code = library().mpm_nearest_neighbors_chunked(_ptr(tokens), _ptr(offsets), batch, rows, dim,
                                                           _dtype_code(tokens), ALGOS[algo], int(chunk), _ptr(nn),
                                                           _ptr(score), _ptr(workspace), workspace.numel(),
                                                           _stream(dev))
        else:
            code = library().mpm_nearest_neighbors(_ptr(tokens), _ptr(offsets), batch, rows, dim,
                                                   _dtype_code(tokens), ALGOS[algo], _ptr(nn), _ptr(score),
                                                   _ptr(workspace), workspace.numel(), _stream(dev))
    _check("mpm_nearest_neighbors", code)
    return nn, score


def compose_maps(map1: torch.Tensor, offsets0: torch.Tensor, map2: torch.Tensor, offsets1: torch.Tensor,
                 out: torch.Tensor | None = None, device_status: torch.Tensor | None = None) -> torch.Tensor:
    """Eq. 3: r*(p) = r2(r1(p)) per image, local int32 indices."""
    _cuda(map1, "map1", torch.int32, 1)
    _cuda(map2, "map2", torch.int32, 1)
    _cuda(offsets0, "offsets0", torch.int64, 1)
    _cuda(offsets1, "offsets1", torch.int64, 1)
    dev = map1.device
    if out is None:
        out = torch.empty_like(map1)
    with torch.cuda.device(dev):
        code = library().mpm_compose_maps(_ptr(map1), _ptr(offsets0), map1.numel(), _ptr(map2),
                                          _ptr(offsets1), map2.numel(), offsets0.numel() - 1, _ptr(out),
                                          _ptr(device_status), _stream(dev))
    _check("mpm_compose_maps", code)
    return out


def unmerge_gather(merged: torch.Tensor, merged_offsets: torch.Tensor, rmap: torch.Tensor,
                   grid_offsets: torch.Tensor, out: torch.Tensor | None = None,
                   device_status: torch.Tensor | None = None) -> torch.Tensor:
    """Eq. 4: out[p] = merged[r*(p)] per image; out has rmap.numel() rows."""
    _cuda(merged, "merged", ndim=2)
    _cuda(merged_offsets, "merged_offsets", torch.int64, 1)
    _cuda(rmap, "map", torch.int32, 1)
    _cuda(grid_offsets, "grid_offsets", torch.int64, 1)
    dev = merged.device
    if out is None:
        out = torch.empty(rmap.numel(), merged.shape[1], dtype=merged.dtype, device=dev)
    with torch.cuda.device(dev):
        code = library().mpm_unmerge_gather(_ptr(merged), _ptr(merged_offsets), merged.shape[0], _ptr(rmap),
                                            _ptr(grid_offsets), out.shape[0], grid_offsets.numel() - 1,
                                            merged.shape[1], _dtype_code(merged), _ptr(out),
                                            _ptr(device_status), _stream(dev))
    _check("mpm_unmerge_gather", code)
    return out


def compose_gather(merged: torch.Tensor, merged_offsets: torch.Tensor, map1: torch.Tensor,
                   offsets0: torch.Tensor, map2: torch.Tensor, offsets1: torch.Tensor,
                   out: torch.Tensor | None = None, out_map: torch.Tensor | None = None,
                   device_status: torch.Tensor | None = None) -> torch.Tensor:
    """Eq. 3 and Eq. 4 in one pass: out[p] = merged[r2(r1(p))] per image.

    out has map1.numel() rows; out_map, if given, receives the composed map.
    """
    _cuda(merged, "merged", ndim=2)
    _cuda(merged_offsets, "merged_offsets", torch.int64, 1)
    _cuda(map1, "map1", torch.int32, 1)
    _cuda(offsets0, "offsets0", torch.int64, 1)
    _cuda(map2, "map2", torch.int32, 1)
    _cuda(offsets1, "offsets1", torch.int64, 1)
    if out_map is not None:
        _cuda(out_map, "out_map", torch.int32, 1)
        if out_map.numel() < map1.numel():
            raise ValueError("out_map needs map1.numel() entries")
    dev = merged.device
    if out is None:
        out = torch.empty(map1.numel(), merged.shape[1], dtype=merged.dtype, device=dev)
    with torch.cuda.device(dev):
        code = library().mpm_compose_gather(_ptr(merged), _ptr(merged_offsets), merged.shape[0], _ptr(map1),
                                            _ptr(offsets0), out.shape[0], _ptr(map2), _ptr(offsets1),
                                            map2.numel(), offsets0.numel() - 1, merged.shape[1],
                                            _dtype_code(merged), _ptr(out), _ptr(out_map),
                                            _ptr(device_status), _stream(dev))
    _check("mpm_compose_gather", code)
    return out


def pad_batch(tokens: torch.Tensor, offsets: torch.Tensor, max_len: int, out: torch.Tensor | None = None,
              mask: torch.Tensor | None = None, stats: torch.Tensor | None = None,
              device_status: torch.Tensor | None = None):
    """Packed tokens -> ([B, max_len, D] padded, [B, max_len] uint8 key mask, int64 [3] N_b min/max/total).

    Nothing is read back to the host: pass max_len = the largest N_b if the
    caller knows it (e.g. from a host copy of offsets), or any upper bound.
    """
    _cuda(tokens, "tokens", ndim=2)
    _cuda(offsets, "offsets", torch.int64, 1)
    dev = tokens.device
    batch = offsets.numel() - 1
    max_len = int(max_len)
    if out is None:
        out = torch.empty(batch, max_len, tokens.shape[1], dtype=tokens.dtype, device=dev)
    if mask is None:
        mask = torch.empty(batch, max_len, dtype=torch.uint8, device=dev)
    if stats is None:
        stats = torch.empty(3, dtype=torch.int64, device=dev)
    with torch.cuda.device(dev):
        code = library().mpm_pad_batch(_ptr(tokens), _ptr(offsets), batch, tokens.shape[0], tokens.shape[1],
                                       _dtype_code(tokens), max_len, _ptr(out), _ptr(mask), _ptr(stats),
                                       _ptr(device_status), _stream(dev))
    _check("mpm_pad_batch", code)
    return out, mask, stats


def unpad_batch(padded: torch.Tensor, offsets: torch.Tensor, rows: int | None = None,
                out: torch.Tensor | None = None, device_status: torch.Tensor | None = None) -> torch.Tensor:
    """[B, L, D] padded -> packed [rows, D] with out[offsets[b] + t] = padded[b, t]."""
    _cuda(padded, "padded", ndim=3)
    _cuda(offsets, "offsets", torch.int64, 1)
    dev = padded.device
    batch, max_len, dim = padded.shape
    if out is None:
        out = torch.empty(int(rows) if rows is not None else batch * max_len, dim, dtype=padded.dtype, device=dev)
    with torch.cuda.device(dev):
        code = library().mpm_unpad_batch(_ptr(padded), batch, max_len, dim, _dtype_code(padded), _ptr(offsets),
                                         out.shape[0], _ptr(out), _ptr(device_status), _stream(dev))
    _check("mpm_unpad_batch", code)
    return out


def device_status(workspace: torch.Tensor) -> int:
    """First device-side error recorded in a merge workspace (0 = none); clears it."""
    code = ctypes.c_int32(0)
    dev = workspace.device
    with torch.cuda.device(dev):
        _check("mpm_get_device_status",
               library().mpm_get_device_status(_ptr(workspace), ctypes.byref(code), _stream(dev)))
    return int(code.value)


def merge_no_alloc(tokens: torch.Tensor, offsets: torch.Tensor, out_tokens: torch.Tensor,
                   out_offsets: torch.Tensor, out_map: torch.Tensor):
    """merge() for callers that cannot allocate device memory.

    The caller provides every output buffer; the scratch space is a fixed
    array inside the library (see mpm_merge_no_alloc in include/mpm.h for the
    size limit, the first-call set-up and why overlapping calls race).
    """
    _cuda(tokens, "tokens", ndim=2)
    _cuda(offsets, "offsets", torch.int64, 1)
    _cuda(out_tokens, "out_tokens", tokens.dtype, 2)
    _cuda(out_offsets, "out_offsets", torch.int64, 1)
    _cuda(out_map, "out_map", torch.int32, 1)
    dev = tokens.device
    rows, dim = tokens.shape
    with torch.cuda.device(dev):
        code = library().mpm_merge_no_alloc(_ptr(tokens), _ptr(offsets), offsets.numel() - 1, rows, dim,
                                            _dtype_code(tokens), _ptr(out_tokens), _ptr(out_offsets),
                                            _ptr(out_map), _stream(dev))
    _check("mpm_merge_no_alloc", code)
    return out_tokens, out_offsets, out_map


def no_alloc_device_status(device=None) -> int:
    """First device-side error of the last merge_no_alloc call on a device (0 = none); clears it."""
    dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    code = ctypes.c_int32(0)
    with torch.cuda.device(dev):
        _check("mpm_no_alloc_get_device_status",
               library().mpm_no_alloc_get_device_status(ctypes.byref(code), _stream(dev)))
    return int(code.value)


def selftest_wait_timeout(limit_us: int, device=None) -> torch.Tensor:
    """Runs the device timeout self-test (mpm_selftest_wait_timeout): a
    bounded wait on a barrier that nothing completes.  Returns the int32[2]
    device status word it wrote ([MPM_ERR_DEVICE_TIMEOUT, 99] when the wait
    gave up as it should); the caller synchronises before reading it."""
    dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    status = torch.zeros(2, dtype=torch.int32, device=dev)
    with torch.cuda.device(dev):
        code = library().mpm_selftest_wait_timeout(_ptr(status), int(limit_us), _stream(dev))
    _check("mpm_selftest_wait_timeout", code)
    return status


def trace_reset() -> None:
    """Clears the device timeline (libmpm_trace.so only; synchronous)."""
    _check("mpm_trace_reset", library().mpm_trace_reset())


def trace_read() -> dict:
    """Device timeline since the last reset (libmpm_trace.so only;
    synchronous): for each kernel kind that ran, (first block start, first
    block past its wait for the previous kernel, last warp end) in ns of the
    GPU global timer."""
    import numpy as np

    out = np.zeros(3 * len(TRACE_KINDS), dtype=np.uint64)
    _check("mpm_trace_read", library().mpm_trace_read(out.ctypes.data))
    res = {}
    for k, name in enumerate(TRACE_KINDS):
        start, waited, end = (int(v) for v in out[3 * k:3 * k + 3])
        if end != 0:
            res[name] = (start, waited, end)
    return res
