"""Frames per second of a ViT encoder + dense head with and without MPM.

Prints one JSON line: the full model and the model with MPM before the
configured blocks, both with the same packed varlen attention kernel, plus
the full model with batched PyTorch SDPA (its fastest kernel for fixed
lengths) for reference, and the token counts after each insertion.
Synthetic images, random-init weights (seeded); the shapes follow the
paper's Seg-*/16 models at 512 x 512 (1024 patch tokens).

    python vit_insertion/bench_vit.py --model vit_b16 --batch 32
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

import paper_2604_05718_gb300 as mpm  # noqa: E402
from paper_2604_05718_gb300 import build  # noqa: E402
from vit_insertion import VIT_CONFIGS, ViT, synthetic_images  # noqa: E402


def timed(fn, steps: int, warmup: int) -> float:
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ts = []
    for _ in range(steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fn()
        e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    return statistics.median(ts)


def main() -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--model", default="vit_b16", choices=sorted(VIT_CONFIGS))
    ap.add_argument("--batch", type=int, default=32)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--seed", type=int, default=0)
    args = ap.parse_args()
    if not torch.cuda.is_available():
        raise RuntimeError("bench_vit.py needs a CUDA device")
    build.build()
    mpm.library()
    dev = torch.device("cuda", 0)
    cfg = VIT_CONFIGS[args.model]
    model = ViT(cfg, dev, seed=args.seed)
    images = synthetic_images(args.batch, cfg.image, cfg.patch, args.seed, dev)
    ws = mpm.new_workspace(args.batch * cfg.tokens, args.batch, cfg.dim, torch.bfloat16, dev)

    with torch.inference_mode():
        trace = []
        model.forward(images, mpm=mpm, workspace=ws, trace=trace)
        merged_out = []
        for _, patches, off in trace:
            _, o, _ = mpm.merge(patches, off, workspace=ws)
            merged_out.append(int(o[-1]))
        ms_full = timed(lambda: model.forward(images), args.steps, args.warmup)
        ms_mpm = timed(lambda: model.forward(images, mpm=mpm, workspace=ws), args.steps, args.warmup)
        ms_sdpa = timed(lambda: model.forward_dense_sdpa(images), args.steps, args.warmup)
    line = {
        "metric": "ViT encoder + dense head frames/s, with and without MPM",
        "model": cfg.name, "depth": cfg.depth, "dim": cfg.dim, "heads": cfg.heads, "image": cfg.image,
        "patch_tokens": cfg.tokens, "special_tokens": cfg.special, "batch": args.batch,
        "insert_before_blocks": list(cfg.insert_at),
        "tokens_into_insertions": [int(off[-1]) for _, _, off in trace],
        "tokens_out_of_insertions": merged_out,
        "fps_full_varlen": args.batch / (ms_full * 1e-3),
        "fps_mpm_varlen": args.batch / (ms_mpm * 1e-3),
        "fps_full_sdpa": args.batch / (ms_sdpa * 1e-3),
        "speedup_vs_full_varlen": ms_full / ms_mpm,
        "speedup_vs_full_sdpa": ms_sdpa / ms_mpm,
        "ms": {"full_varlen": ms_full, "mpm_varlen": ms_mpm, "full_sdpa": ms_sdpa},
        "data": "synthetic Voronoi images, random-init bf16 weights",
        "attention": "aten._flash_attention_forward (varlen) for the packed paths; SDPA (batched) for full_sdpa",
    }
    print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
