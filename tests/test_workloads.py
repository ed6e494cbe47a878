"""The seeded input generator: determinism, shapes and the workload recipe."""

import numpy as np
import torch

from workloads import (CONFIGS, CONFIG_ORDER, apply_noise, image_shape, make_batch, make_custom,
                       stage_noise)


def test_configs_shapes():
    want = {"vit_t_single": (1, 1024, 192, "f32"), "vit_s": (32, 1024, 384, "bf16"),
            "vit_b": (64, 1024, 768, "bf16"), "vit_l": (16, 2304, 1024, "bf16")}
    for name, (b, n, d, dt) in want.items():
        cfg = CONFIGS[name]
        assert cfg.batch == b and cfg.dim == d and cfg.dtype == dt
        side, k, sigma = image_shape(cfg, 0)
        assert side * side == n
    assert CONFIG_ORDER[0] == "vit_t_single" and len(CONFIG_ORDER) == 5


def test_mixed_shapes_are_drawn_per_image():
    cfg = CONFIGS["mixed"]
    shapes = [image_shape(cfg, b) for b in range(cfg.batch)]
    assert {s for s, _, _ in shapes} <= {32, 40, 48, 64}
    assert all(16 <= k <= 128 and 0.1 <= sg <= 0.5 for _, k, sg in shapes)
    assert len({s for s, _, _ in shapes}) > 1
    assert shapes == [image_shape(cfg, b) for b in range(cfg.batch)]


def test_make_batch_deterministic_and_packed():
    cfg = CONFIGS["vit_s"]
    a = make_batch(cfg, images=range(3))
    b = make_batch(cfg, images=range(3))
    assert torch.equal(a.tokens, b.tokens)
    assert a.tokens.dtype == torch.bfloat16 and a.tokens.shape == (3 * 1024, 384)
    assert a.offsets.tolist() == [0, 1024, 2048, 3072]
    # A subset of images is the same data as in the full batch.
    c = make_batch(cfg, images=[1])
    assert torch.equal(c.tokens, a.tokens[1024:2048])


def test_voronoi_structure():
    """Tokens of one region are much closer to each other than to other regions."""
    batch = make_custom([400], 64, "f32", seed=1, k=4, sigma=0.1)
    x = batch.tokens.double().numpy()
    xt = x / np.linalg.norm(x, axis=1, keepdims=True)
    s = xt @ xt.T
    np.fill_diagonal(s, -1)
    assert np.median(s.max(axis=1)) > 0.95


def test_stage_noise_and_apply():
    n = stage_noise(1003, [5, 0, 7], 16)
    assert n.shape == (12, 16) and n.dtype == torch.float32
    assert 0.02 < float(n.std()) < 0.09
    again = stage_noise(1003, [7], 16, images=[2])
    assert torch.equal(again, n[5:])
    x = torch.randn(12, 16).to(torch.bfloat16)
    y = apply_noise(x, n)
    assert y.dtype == torch.bfloat16
    assert torch.equal(y, (x.float() + n).to(torch.bfloat16))
