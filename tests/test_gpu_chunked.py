"""GPU parity of the chunked similarity (mpm_merge_chunked): every token's
nearest neighbour is sought only within its run of `chunk` consecutive tokens,
the bound Section 5 proposes for very large N.  Same bar as the full merge:
decisive rows bit-exact, near ties validated, features exactly the rounded
means."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from parity import check_merge_batch, to_f64
from workloads import make_custom

pytestmark = pytest.mark.gpu

DEV = "cuda"
COUNTS = [1024, 513, 257, 256, 1, 2, 700, 1500]


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


def run(mpm, batch, chunk, algo="auto"):
    x = batch.tokens.to(DEV)
    off = torch.from_numpy(batch.offsets).to(DEV)
    ws = mpm.new_workspace(x.shape[0], batch.batch, x.shape[1], x.dtype, DEV)
    nn, _ = mpm.nearest_neighbors(x, off, algo=algo, workspace=ws, chunk=chunk)
    assert mpm.device_status(ws) == 0
    out, out_off, rmap = mpm.merge(x, off, workspace=ws, chunk=chunk)
    assert mpm.device_status(ws) == 0
    t = int(out_off[-1])
    return nn.cpu().numpy(), rmap.cpu().numpy(), to_f64(out[:t]), out_off.cpu().numpy()


@pytest.mark.parametrize("dim", [128, 768])
@pytest.mark.parametrize("chunk", [256, 512])
def test_chunked_bf16_matches_oracle(mpm, chunk, dim):
    # D = 128 runs the SM-pair kernel with 16 epilogue warps, D = 768 with 8.
    batch = make_custom(COUNTS, dim, "bf16", seed=41)
    nn, rmap, out, out_off = run(mpm, batch, chunk)
    # No neighbour crosses a chunk; a token alone in its chunk has none.
    for b in range(batch.batch):
        n = int(batch.offsets[b + 1] - batch.offsets[b])
        i = np.arange(n)
        j = nn[batch.offsets[b]:batch.offsets[b + 1]]
        assert np.all((j < 0) | (j // chunk == i // chunk))
    check_merge_batch(batch.tokens.double().numpy(), batch.offsets, nn, rmap, out, out_off, "bf16",
                      f"chunked {chunk}", chunk=chunk)


def test_chunked_f32_matches_oracle(mpm):
    batch = make_custom([600, 257, 3], 64, "f32", seed=42)
    nn, rmap, out, out_off = run(mpm, batch, 256)
    check_merge_batch(batch.tokens.double().numpy(), batch.offsets, nn, rmap, out, out_off, "f32",
                      "chunked f32", chunk=256)


def test_chunk_zero_and_whole_image_equal_the_full_merge(mpm):
    batch = make_custom([700, 300, 1], 64, "bf16", seed=43)
    full = run(mpm, batch, 0)
    whole = run(mpm, batch, 768)
    for a, b in zip(full, whole):
        assert np.array_equal(a, b)
