"""In-model insertion of MPM: a ViT encoder (random-init weights) on
synthetic images, with MPM before chosen blocks, special tokens passed
through, ragged (varlen) attention on the merged sequences, and the gather
unmerge back to the patch grid for a dense head (Section 3.1 and Section 4,
Tables 1 and 5 in shape).  The model layers are plain PyTorch; every merge,
composition and gather runs in the MPM library's kernels."""

from .model import ViTConfig, VIT_CONFIGS, ViT, synthetic_images  # noqa: F401
