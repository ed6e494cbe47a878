"""A ViT encoder with Mutual Pair Merging inserted before chosen blocks.

Layout: the tokens of a batch are kept packed, image after image, each image
as [E special tokens, n_b patch tokens]; ``cu`` (int32 [B+1]) marks the
sequence starts for the varlen attention.  An insertion (Section 3.1):
  1. split the patch tokens of every image from its special tokens,
  2. merge the patch tokens with MPM (one library call for the whole batch),
  3. join the special tokens back in front of each image's merged tokens.
After the last block the patch tokens are unmerged to the full grid through
all insertions' maps (Eq. 3 and Eq. 4) for the dense head.

The attention, projections, MLP and norms are PyTorch operations (cuBLAS /
FlashAttention varlen); only the merge, composition and gather are this
project's kernels.  Weights are random (seeded): no trained checkpoint is
available here, and the timing does not depend on the values.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import torch
import torch.nn.functional as F


@dataclass(frozen=True)
class ViTConfig:
    name: str
    depth: int
    dim: int
    heads: int
    mlp: int
    patch: int
    image: int
    special: int = 1          # E: class token(s), never merged
    classes: int = 150        # dense head outputs per patch (ADE20K has 150 classes)
    insert_at: tuple = (2, 5)  # MPM before these blocks (0-based)

    @property
    def grid(self) -> int:
        return self.image // self.patch

    @property
    def tokens(self) -> int:
        return self.grid * self.grid


VIT_CONFIGS = {
    "vit_t16": ViTConfig("vit_t16", 12, 192, 3, 768, 16, 512),
    "vit_s16": ViTConfig("vit_s16", 12, 384, 6, 1536, 16, 512),
    "vit_b16": ViTConfig("vit_b16", 12, 768, 12, 3072, 16, 512),
    "vit_l16": ViTConfig("vit_l16", 24, 1024, 16, 4096, 16, 512, insert_at=(2, 5)),
}


def synthetic_images(batch: int, image: int, patch: int, seed: int, device, dtype=torch.bfloat16,
                     sites: int = 64, noise: float = 0.05) -> torch.Tensor:
    """[B, 3, H, W] images made of Voronoi regions of constant colour plus noise.

    The regions are drawn on the patch grid (every patch lies in one region),
    so that patches of one region differ only by noise, as flat areas of real
    images do.  Seeded: image b uses generator seed (seed, b).
    """
    g = image // patch
    out = torch.empty(batch, 3, image, image, dtype=dtype, device=device)
    rr, cc = torch.meshgrid(torch.arange(g, dtype=torch.float64) + 0.5,
                            torch.arange(g, dtype=torch.float64) + 0.5, indexing="ij")
    centres = torch.stack([rr.reshape(-1), cc.reshape(-1)], dim=1)
    for b in range(batch):
        gen = torch.Generator().manual_seed(seed * 100003 + b)
        pos = torch.rand(sites, 2, generator=gen, dtype=torch.float64) * g
        colour = torch.rand(sites, 3, generator=gen, dtype=torch.float64)
        site = torch.cdist(centres, pos).argmin(dim=1)
        grid = colour[site].reshape(g, g, 3).permute(2, 0, 1)                  # [3, g, g]
        img = grid.repeat_interleave(patch, dim=1).repeat_interleave(patch, dim=2)
        img = img + noise * torch.randn(3, image, image, generator=gen, dtype=torch.float64)
        out[b] = img.to(device=device, dtype=dtype)
    return out


def varlen_attention(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, cu: torch.Tensor,
                     max_len: int) -> torch.Tensor:
    """Softmax attention within each packed sequence: q, k, v [S, H, Dh] -> [S, H, Dh]."""
    out = torch.ops.aten._flash_attention_forward(q, k, v, cu, cu, max_len, max_len, 0.0, False, False)
    return out[0]


class ViT:
    """Random-init ViT encoder + linear dense head, packed-token forward."""

    def __init__(self, cfg: ViTConfig, device, dtype=torch.bfloat16, seed: int = 0):
        self.cfg, self.device, self.dtype = cfg, torch.device(device), dtype
        g = torch.Generator().manual_seed(seed)
        d, m = cfg.dim, cfg.mlp

        def w(*shape, fan_in):
            return (torch.randn(*shape, generator=g) / math.sqrt(fan_in)).to(self.device, dtype)

        def zeros(*shape):
            return torch.zeros(*shape, device=self.device, dtype=dtype)

        def ones(*shape):
            return torch.ones(*shape, device=self.device, dtype=dtype)

        pp = 3 * cfg.patch * cfg.patch
        self.patch_w, self.patch_b = w(d, pp, fan_in=pp), zeros(d)
        self.special = w(cfg.special, d, fan_in=1) * 0.02
        self.pos = w(cfg.tokens + cfg.special, d, fan_in=1) * 0.02
        self.blocks = []
        for _ in range(cfg.depth):
            self.blocks.append(dict(
                ln1_w=ones(d), ln1_b=zeros(d), qkv_w=w(3 * d, d, fan_in=d), qkv_b=zeros(3 * d),
                proj_w=w(d, d, fan_in=d), proj_b=zeros(d), ln2_w=ones(d), ln2_b=zeros(d),
                fc1_w=w(m, d, fan_in=d), fc1_b=zeros(m), fc2_w=w(d, m, fan_in=m), fc2_b=zeros(d)))
        self.head_ln_w, self.head_ln_b = ones(d), zeros(d)
        self.head_w, self.head_b = w(cfg.classes, d, fan_in=d), zeros(cfg.classes)

    # -- layers ------------------------------------------------------------
    def embed(self, images: torch.Tensor) -> torch.Tensor:
        """[B, 3, H, W] -> packed [B * (E + N), D]: special tokens first in every image."""
        cfg = self.cfg
        b = images.shape[0]
        p = F.unfold(images, kernel_size=cfg.patch, stride=cfg.patch)            # [B, 3*P*P, N]
        x = F.linear(p.transpose(1, 2), self.patch_w, self.patch_b)              # [B, N, D]
        x = torch.cat([self.special.expand(b, -1, -1), x], dim=1) + self.pos     # [B, E+N, D]
        return x.reshape(b * (cfg.special + cfg.tokens), cfg.dim).contiguous()

    def block(self, x: torch.Tensor, p: dict, cu: torch.Tensor, max_len: int) -> torch.Tensor:
        cfg = self.cfg
        s = x.shape[0]
        h = F.layer_norm(x, (cfg.dim,), p["ln1_w"], p["ln1_b"])
        qkv = F.linear(h, p["qkv_w"], p["qkv_b"]).view(s, 3, cfg.heads, cfg.dim // cfg.heads)
        q, k, v = (qkv[:, i].contiguous() for i in range(3))
        a = varlen_attention(q, k, v, cu, max_len).reshape(s, cfg.dim)
        x = x + F.linear(a, p["proj_w"], p["proj_b"])
        h = F.layer_norm(x, (cfg.dim,), p["ln2_w"], p["ln2_b"])
        return x + F.linear(F.gelu(F.linear(h, p["fc1_w"], p["fc1_b"])), p["fc2_w"], p["fc2_b"])

    def head(self, patches: torch.Tensor) -> torch.Tensor:
        h = F.layer_norm(patches, (self.cfg.dim,), self.head_ln_w, self.head_ln_b)
        return F.linear(h, self.head_w, self.head_b)

    # -- special-token split / join ------------------------------------------
    def split(self, x: torch.Tensor, off: torch.Tensor):
        """Packed [E specials, n_b patches] per image -> (specials [B*E, D], patches packed by off)."""
        e = self.cfg.special
        b = off.numel() - 1
        rows = torch.arange(int(x.shape[0]) - e * b, device=x.device)
        img = torch.searchsorted(off[1:], rows, right=True)
        patches = x.index_select(0, rows + e * (img + 1))
        starts = off[:-1] + e * torch.arange(b, device=x.device)
        sp_rows = (starts[:, None] + torch.arange(e, device=x.device)[None, :]).reshape(-1)
        return x.index_select(0, sp_rows), patches

    def join(self, specials: torch.Tensor, patches: torch.Tensor, off: torch.Tensor) -> torch.Tensor:
        """Inverse of split for patches packed by off (patches has exactly off[-1] rows)."""
        e = self.cfg.special
        b = off.numel() - 1
        out = torch.empty(patches.shape[0] + e * b, patches.shape[1], dtype=patches.dtype, device=patches.device)
        rows = torch.arange(patches.shape[0], device=patches.device)
        img = torch.searchsorted(off[1:], rows, right=True)
        out.index_copy_(0, rows + e * (img + 1), patches)
        starts = off[:-1] + e * torch.arange(b, device=patches.device)
        sp_rows = (starts[:, None] + torch.arange(e, device=patches.device)[None, :]).reshape(-1)
        out.index_copy_(0, sp_rows, specials)
        return out

    # -- forward -------------------------------------------------------------
    def forward(self, images: torch.Tensor, mpm=None, workspace=None, insert_at=None, trace=None):
        """Dense logits [B*N, classes] on the patch grid.

        mpm: the MPM package (paper_2604_05718_gb300) to merge with, or None
        for the full model.  insert_at overrides cfg.insert_at.  trace, if a
        list, receives (block, patch tokens, offsets) at every insertion.
        """
        cfg = self.cfg
        b = images.shape[0]
        e, n = cfg.special, cfg.tokens
        x = self.embed(images)
        off = torch.arange(b + 1, device=self.device, dtype=torch.int64) * n   # patch offsets
        counts_host = [n] * b
        maps = []
        points = set(cfg.insert_at if insert_at is None else insert_at) if mpm is not None else set()
        for i, p in enumerate(self.blocks):
            if i in points:
                specials, patches = self.split(x, off)
                if trace is not None:
                    trace.append((i, patches, off))
                merged, off1, m = mpm.merge(patches, off, workspace=workspace)
                off1_host = off1.cpu()                       # the merged length decides the next shapes
                total = int(off1_host[-1])
                counts_host = (off1_host[1:] - off1_host[:-1]).tolist()
                maps.append((m, off))
                off = off1
                x = self.join(specials, merged[:total], off)
            cu = (off + e * torch.arange(b + 1, device=self.device)).to(torch.int32)
            x = self.block(x, p, cu, max(counts_host) + e)
        _, patches = self.split(x, off)
        if len(maps) == 0:
            grid = patches
        elif len(maps) == 1:
            grid = mpm.unmerge_gather(patches, off, maps[0][0], maps[0][1])
        else:
            # Compose all but the last two maps into the first, then gather through the last pair.
            m_first, off0 = maps[0]
            for m_next, off_next in maps[1:-1]:
                m_first = mpm.compose_maps(m_first, off0, m_next, off_next)
            grid = mpm.compose_gather(patches, off, m_first, off0, maps[-1][0], maps[-1][1])
        return self.head(grid)

    def forward_dense_sdpa(self, images: torch.Tensor) -> torch.Tensor:
        """The full model with batched [B, E+N, D] attention (PyTorch SDPA picks its fastest kernel)."""
        cfg = self.cfg
        b = images.shape[0]
        x = self.embed(images).view(b, cfg.special + cfg.tokens, cfg.dim)
        for p in self.blocks:
            h = F.layer_norm(x, (cfg.dim,), p["ln1_w"], p["ln1_b"])
            qkv = F.linear(h, p["qkv_w"], p["qkv_b"]).view(b, -1, 3, cfg.heads, cfg.dim // cfg.heads)
            q, k, v = (qkv[:, :, i].transpose(1, 2) for i in range(3))
            a = F.scaled_dot_product_attention(q, k, v).transpose(1, 2).reshape(b, -1, cfg.dim)
            x = x + F.linear(a, p["proj_w"], p["proj_b"])
            h = F.layer_norm(x, (cfg.dim,), p["ln2_w"], p["ln2_b"])
            x = x + F.linear(F.gelu(F.linear(h, p["fc1_w"], p["fc1_b"])), p["fc2_w"], p["fc2_b"])
        return self.head(x[:, cfg.special:].reshape(-1, cfg.dim))
