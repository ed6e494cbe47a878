"""Seeded synthetic token batches for MPM tests and benchmarks.

This module only draws inputs.  It holds none of the method's arithmetic and
is the one piece of code that both the fp64 oracle's tests and the GPU path's
tests and benchmark use.

Stand-in for the paper's datasets (ADE20K 512^2 -> 32x32 patches, Cityscapes
768^2 -> 48x48, and the 3136/4096-token high-resolution cases of Section 4),
which are not available here.  Each image is a grid of side s (N = s^2 patch
tokens in raster order).  K Voronoi sites are drawn uniformly in [0, s)^2;
each cell centre (r + 0.5, c + 0.5) belongs to its Euclidean-nearest site
(ties to the lowest site index).  Site means m_k ~ N(0, I_D) are drawn in site
order, then token (r, c) = m_site + sigma * N(0, I_D), drawn in raster order.
Values are drawn in fp64 and stored as fp32, or as bf16 via fp32 (each step
rounds to nearest even).

Random streams (numpy PCG64): for workload seed S and image b,
  default_rng([S, b, 0])  per-image shape parameters (mixed-resolution only)
  default_rng([S, b, 1])  the image's sites, means and token noise
  default_rng([S, b, 2])  the N(0, 0.05^2) noise that stands in for the
                          encoder blocks between the two MPM insertions
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

DTYPES = {"f32": torch.float32, "bf16": torch.bfloat16}


@dataclass(frozen=True)
class WorkloadConfig:
    """One synthetic workload.

    sides: grid sides to draw from (one entry = fixed side).  k_range and
    sigma_range are inclusive integer / uniform ranges; a one-element range
    means a fixed value.
    """

    name: str
    batch: int
    sides: tuple
    dim: int
    dtype: str
    k_range: tuple
    sigma_range: tuple
    insertions: int
    seed: int
    description: str = ""

    @property
    def mixed(self) -> bool:
        return len(self.sides) > 1 or len(self.k_range) > 1 or len(self.sigma_range) > 1


# The five workloads: ViT-T single image (fp32, one insertion), ViT-S, ViT-B,
# ViT-L at 768^2, and a mixed-resolution ragged batch (bf16, two insertions).
CONFIGS = {
    "vit_t_single": WorkloadConfig(
        "vit_t_single", 1, (32,), 192, "f32", (32,), (0.3,), 1, 1001,
        "B=1, 32x32 grid (N=1024), D=192, fp32, K=32, sigma=0.3, one insertion + unmerge"),
    "vit_s": WorkloadConfig(
        "vit_s", 32, (32,), 384, "bf16", (32,), (0.3,), 2, 1002,
        "B=32, 512x512 / patch 16 (N=1024), D=384, bf16, K=32, sigma=0.3, two insertions"),
    "vit_b": WorkloadConfig(
        "vit_b", 64, (32,), 768, "bf16", (64,), (0.3,), 2, 1003,
        "B=64, N=1024, D=768, bf16, K=64, sigma=0.3, two insertions"),
    "vit_l": WorkloadConfig(
        "vit_l", 16, (48,), 1024, "bf16", (96,), (0.25,), 2, 1004,
        "B=16, 768x768 / patch 16 (N=2304), D=1024, bf16, K=96, sigma=0.25, two insertions"),
    "mixed": WorkloadConfig(
        "mixed", 24, (32, 40, 48, 64), 768, "bf16", (16, 128), (0.1, 0.5), 2, 1005,
        "B=24, sides in {32,40,48,64} (1024-4096 tokens), D=768, bf16, K in [16,128], "
        "sigma in [0.1,0.5], two insertions"),
}
CONFIG_ORDER = ["vit_t_single", "vit_s", "vit_b", "vit_l", "mixed"]

STAGE_NOISE_STD = 0.05


def image_shape(cfg: WorkloadConfig, b: int) -> tuple[int, int, float]:
    """(side, K, sigma) of image b."""
    if not cfg.mixed:
        return int(cfg.sides[0]), int(cfg.k_range[0]), float(cfg.sigma_range[0])
    rng = np.random.default_rng([cfg.seed, b, 0])
    side = int(cfg.sides[int(rng.integers(0, len(cfg.sides)))])
    k = int(rng.integers(cfg.k_range[0], cfg.k_range[-1] + 1))
    sigma = float(rng.uniform(cfg.sigma_range[0], cfg.sigma_range[-1]))
    return side, k, sigma


def voronoi_tokens(rng: np.random.Generator, side: int, dim: int, k: int,
                   sigma: float) -> np.ndarray:
    """One image of side*side tokens (fp64, raster order)."""
    sites = rng.uniform(0.0, float(side), size=(k, 2))
    rr, cc = np.meshgrid(np.arange(side) + 0.5, np.arange(side) + 0.5, indexing="ij")
    centres = np.stack([rr.ravel(), cc.ravel()], axis=1)
    d2 = ((centres[:, None, :] - sites[None, :, :]) ** 2).sum(axis=2)
    site = np.argmin(d2, axis=1)
    means = rng.standard_normal((k, dim))
    return means[site] + sigma * rng.standard_normal((side * side, dim))


def to_storage(x: np.ndarray, dtype: str) -> torch.Tensor:
    """fp64 -> fp32 (RNE) -> storage dtype (RNE), as a CPU tensor."""
    t = torch.from_numpy(np.ascontiguousarray(np.asarray(x, dtype=np.float64).astype(np.float32)))
    return t if dtype == "f32" else t.to(DTYPES[dtype])


@dataclass
class Batch:
    """A packed ragged batch: tokens [T, D] (CPU tensor), offsets int64 [B+1]."""

    tokens: torch.Tensor
    offsets: np.ndarray
    dtype: str
    cfg: WorkloadConfig | None = None
    shapes: list = field(default_factory=list)

    @property
    def batch(self) -> int:
        return int(self.offsets.shape[0] - 1)

    @property
    def rows(self) -> int:
        return int(self.offsets[-1])

    @property
    def dim(self) -> int:
        return int(self.tokens.shape[1])


def make_batch(cfg: WorkloadConfig, images: range | list | None = None) -> Batch:
    """Tokens of the given images of a workload (all B images by default)."""
    idx = list(range(cfg.batch)) if images is None else list(images)
    chunks, shapes = [], []
    offsets = [0]
    for b in idx:
        side, k, sigma = image_shape(cfg, b)
        rng = np.random.default_rng([cfg.seed, b, 1])
        x = voronoi_tokens(rng, side, cfg.dim, k, sigma)
        chunks.append(to_storage(x, cfg.dtype))
        shapes.append((side, k, sigma))
        offsets.append(offsets[-1] + side * side)
    tokens = torch.cat(chunks, dim=0) if chunks else torch.zeros(0, cfg.dim, dtype=DTYPES[cfg.dtype])
    return Batch(tokens.contiguous(), np.array(offsets, dtype=np.int64), cfg.dtype, cfg, shapes)


def make_custom(counts: list, dim: int, dtype: str, seed: int, k: int = 8,
                sigma: float = 0.3) -> Batch:
    """A small ragged batch with arbitrary per-image token counts.

    Each image with n tokens is the first n raster tokens of a Voronoi grid of
    side ceil(sqrt(n)), so counts need not be squares (ragged tails).
    """
    chunks, offsets = [], [0]
    for b, n in enumerate(counts):
        side = max(1, int(np.ceil(np.sqrt(max(n, 1)))))
        rng = np.random.default_rng([seed, b, 1])
        x = voronoi_tokens(rng, side, dim, max(1, min(k, side * side)), sigma)[:n]
        chunks.append(to_storage(x, dtype))
        offsets.append(offsets[-1] + n)
    tokens = torch.cat(chunks, dim=0) if chunks else torch.zeros(0, dim, dtype=DTYPES[dtype])
    return Batch(tokens.contiguous(), np.array(offsets, dtype=np.int64), dtype)


def stage_noise(seed: int, counts: list, dim: int, images: list | None = None,
                stage: int = 2) -> torch.Tensor:
    """Packed fp32 N(0, 0.05^2) noise for a stage input with the given counts.

    Image b's block is drawn from default_rng([seed, b, stage]) in row-major
    order; ``images`` gives the image indices b when only some are used.
    """
    idx = list(range(len(counts))) if images is None else list(images)
    blocks = []
    for b, n in zip(idx, counts):
        rng = np.random.default_rng([seed, b, stage])
        blocks.append((STAGE_NOISE_STD * rng.standard_normal((int(n), dim))).astype(np.float32))
    if not blocks:
        return torch.zeros(0, dim, dtype=torch.float32)
    return torch.from_numpy(np.concatenate(blocks, axis=0))


def apply_noise(x: torch.Tensor, noise: torch.Tensor) -> torch.Tensor:
    """The stand-in for the encoder blocks: (fp32(x) + noise) rounded to x's dtype.

    Runs with torch on whichever device x lives on; fp32 addition and the RNE
    cast give bitwise the same result on the CPU and on the GPU.
    """
    return (x.float() + noise.to(x.device)).to(x.dtype)
