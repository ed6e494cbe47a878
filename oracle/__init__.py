"""fp64 CPU oracle for Mutual Pair Merging.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline legs of ``bench.py``; never by the product path.
"""

from .mpm_oracle import (  # noqa: F401
    NEAR_TIE_GAP,
    NORM_EPS,
    BatchMerge,
    MergeResult,
    Neighbours,
    cluster_average,
    compact_map,
    compose,
    compose_batch,
    cosine_affinity,
    gather,
    gather_batch,
    merge_batch,
    merge_image,
    mutual_partners,
    nearest_neighbours,
    normalise_rows,
    pad_batch,
    round_bf16,
    round_f32,
    unpad_batch,
)
