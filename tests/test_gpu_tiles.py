"""GPU parity of the SM-pair kernel's launch shapes against the fp64 oracle.

The kernel deals its 256 x 256 tiles to the SM pairs round-robin.  Two
shapes depart from the plain tile:
- narrow tiles: a column block holding at most 128 tokens of its image (the
  last block of a ragged image) runs N = 128 MMAs;
- the split last round: with 8 epilogue warps (bf16 rows of more than 512
  features, and fp32), a leftover round of at most half the SM pairs is
  dealt as 256 x 128 halves, and so is every tile of a launch of at most
  that many tiles.
Each case below builds a batch whose tile count puts the launch on one side
of these rules, from images with and without a narrow last block.
"""

from __future__ import annotations

import numpy as np
import pytest
import torch

from parity import check_merge_batch, to_f64
from workloads import make_custom

pytestmark = pytest.mark.gpu

DEV = "cuda"
# Tokens per image -> (tiles, of which narrow): R = ceil(n / 256) block rows,
# R (R + 1) / 2 tiles; the R tiles of the last column block are narrow when
# that block holds at most 128 tokens.
SHAPES = {862: (10, 4), 1024: (10, 0), 300: (3, 2), 200: (1, 0), 100: (1, 1)}


def tiles_of(n: int) -> tuple[int, int]:
    r = -(-n // 256)
    narrow = r if n > 0 and n - 256 * (r - 1) <= 128 else 0
    return r * (r + 1) // 2, narrow


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


@pytest.fixture(scope="module")
def pairs():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.cuda.get_device_properties(0).multi_processor_count // 2


def sizes_for(tiles: int) -> list[int]:
    """Images (alternating 862 and 1024 tokens, then 300, 100 and 200) whose
    tiles add up to exactly `tiles`."""
    out, left, big = [], tiles, [862, 1024]
    while left >= 10:
        out.append(big[len(out) % 2])
        left -= 10
    while left >= 3:
        out.append(300)
        left -= 3
    out += [100, 200][:left] + [100] * max(0, left - 2)
    assert sum(tiles_of(n)[0] for n in out) == tiles
    return out


def check(mpm, sizes, dim, dtype, seed, what):
    batch = make_custom(sizes, dim, dtype, seed=seed)
    x = batch.tokens.to(DEV)
    off = torch.from_numpy(np.asarray(batch.offsets, dtype=np.int64)).to(DEV)
    ws = mpm.new_workspace(x.shape[0], len(sizes), dim, x.dtype, DEV)
    nn, _ = mpm.nearest_neighbors(x, off, workspace=ws)
    out, out_off, rmap = mpm.merge(x, off, workspace=ws)
    assert mpm.device_status(ws) == 0
    torch.cuda.synchronize()
    t, rows = int(out_off[-1]), int(batch.offsets[-1])
    check_merge_batch(batch.tokens.double().numpy(), batch.offsets, nn.cpu().numpy()[:rows],
                      rmap.cpu().numpy()[:rows], to_f64(out[:t]), out_off.cpu().numpy(), dtype, what)


def test_tile_table_matches_the_rule():
    for n, expect in SHAPES.items():
        assert tiles_of(n) == expect, n


@pytest.mark.parametrize("case", ["split_last_round", "full_last_round", "all_split"])
def test_launch_shapes_bf16_8_warps(mpm, pairs, case):
    # D = 640 > 512: the 8-warp epilogue, where the split applies.
    rest = {"split_last_round": pairs // 2 - 3, "full_last_round": pairs // 2 + 5, "all_split": 0}[case]
    tiles = pairs // 2 - 1 if case == "all_split" else 2 * pairs + rest
    sizes = sizes_for(tiles)
    assert any(tiles_of(n)[1] for n in sizes) and any(not tiles_of(n)[1] for n in sizes)
    check(mpm, sizes, 640, "bf16", 71, f"{case}: {tiles} tiles on {pairs} pairs")


def test_narrow_tiles_16_warps(mpm, pairs):
    # D = 256: the 16-warp epilogue (narrow tiles, no split).
    sizes = sizes_for(2 * pairs + pairs // 2 - 3)
    check(mpm, sizes, 256, "bf16", 72, "16 warps")


def test_all_split_fp32(mpm, pairs):
    # fp32 tokens take the three-product tf32 kernel with 8 epilogue warps.
    sizes = sizes_for(pairs // 2 - 1)
    check(mpm, sizes, 128, "f32", 73, "fp32 all split")


def test_split_past_the_listed_items(mpm, pairs):
    # Each pair lists its first 160 items in shared memory and decodes the
    # rest on the fly, the narrow bit included: 161 tiles per pair and a
    # split leftover round of pairs // 2 - 3 tiles, from images of 1 to 5
    # tokens (one narrow tile each), on the 8-warp epilogue.
    n_img = 161 * pairs + pairs // 2 - 3
    rng = np.random.default_rng(74)
    sizes = rng.integers(1, 6, n_img).tolist()
    check(mpm, sizes, 640, "bf16", 74, f"{n_img} one-tile images")
