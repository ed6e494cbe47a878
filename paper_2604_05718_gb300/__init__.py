"""GB300 (sm_103a) Mutual Pair Merging: C-ABI CUDA library + thin binding.

The compute path lives in ``libmpm.so`` (CUDA kernels for sm_103a, built by
``paper_2604_05718_gb300.build.build()``); ``paper_2604_05718_gb300.mpm``
marshals torch tensors into its C entry points.
"""

from .mpm import (  # noqa: F401
    MPMError,
    compose_gather,
    compose_maps,
    device_status,
    library,
    merge,
    merge_no_alloc,
    nearest_neighbors,
    new_workspace,
    no_alloc_device_status,
    pad_batch,
    selftest_wait_timeout,
    trace_read,
    trace_reset,
    unmerge_gather,
    unpad_batch,
    workspace_size,
)
