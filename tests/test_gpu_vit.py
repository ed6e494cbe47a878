"""In-model insertion harness (vit_insertion/) on the GPU: the packed varlen
attention, the special-token split / join around each insertion, the merges
inside the model against the oracle, and the unmerge back to the grid."""

from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from parity import check_merge_batch

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


def tiny(insert_at=(1, 2)):
    from vit_insertion.model import ViTConfig

    return ViTConfig("tiny", depth=4, dim=64, heads=2, mlp=128, patch=8, image=128, special=2,
                     classes=5, insert_at=insert_at)


def test_varlen_attention_matches_per_sequence_softmax():
    from vit_insertion.model import varlen_attention

    torch.manual_seed(0)
    lens = [17, 1, 64, 40]
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=DEV)
    s = sum(lens)
    q, k, v = (torch.randn(s, 2, 32, device=DEV, dtype=torch.bfloat16) for _ in range(3))
    got = varlen_attention(q, k, v, cu, max(lens)).float()
    for a, b in zip(cu[:-1].tolist(), cu[1:].tolist()):
        qs, ks, vs = (t[a:b].float().transpose(0, 1) for t in (q, k, v))
        want = torch.softmax(qs @ ks.transpose(1, 2) / np.sqrt(32), dim=-1) @ vs
        torch.testing.assert_close(got[a:b], want.transpose(0, 1), rtol=2e-2, atol=2e-2)


def test_split_join_roundtrip_keeps_special_tokens():
    from vit_insertion import ViT, synthetic_images

    cfg = tiny()
    model = ViT(cfg, DEV)
    x = model.embed(synthetic_images(3, cfg.image, cfg.patch, 1, DEV))
    off = torch.arange(4, device=DEV) * cfg.tokens
    specials, patches = model.split(x, off)
    assert torch.equal(specials, model.special.repeat(3, 1) + model.pos[:cfg.special].repeat(3, 1))
    assert torch.equal(model.join(specials, patches, off), x)


def test_no_insertion_equals_full_model(mpm):
    from vit_insertion import ViT, synthetic_images

    cfg = tiny()
    model = ViT(cfg, DEV)
    img = synthetic_images(2, cfg.image, cfg.patch, 2, DEV)
    ws = mpm.new_workspace(2 * cfg.tokens, 2, cfg.dim, torch.bfloat16, DEV)
    with torch.inference_mode():
        full = model.forward(img)
        none = model.forward(img, mpm=mpm, workspace=ws, insert_at=())
    assert torch.equal(full, none)


def test_insertions_merge_patch_tokens_like_the_oracle(mpm):
    from vit_insertion import ViT, synthetic_images

    cfg = tiny()
    model = ViT(cfg, DEV)
    img = synthetic_images(3, cfg.image, cfg.patch, 3, DEV, sites=12)
    ws = mpm.new_workspace(3 * cfg.tokens, 3, cfg.dim, torch.bfloat16, DEV)
    trace = []
    with torch.inference_mode():
        logits = model.forward(img, mpm=mpm, workspace=ws, trace=trace)
    assert logits.shape == (3 * cfg.tokens, cfg.classes)
    assert torch.isfinite(logits.float()).all()
    assert [blk for blk, _, _ in trace] == [1, 2]
    n_in = [int(off[-1]) for _, _, off in trace]
    assert n_in[0] == 3 * cfg.tokens and n_in[1] < n_in[0]      # the first insertion merged some pairs
    for k, (_, patches, off) in enumerate(trace):
        with torch.inference_mode():
            nn, _ = mpm.nearest_neighbors(patches, off, workspace=ws)
            x1, off1, m1 = mpm.merge(patches, off, workspace=ws)
        rows, t = int(off[-1]), int(off1[-1])
        check_merge_batch(patches.double().cpu().numpy(), off.cpu().numpy(), nn.cpu().numpy()[:rows],
                          m1.cpu().numpy()[:rows], x1[:t].double().cpu().numpy(), off1.cpu().numpy(), "bf16",
                          f"vit insertion {k}")


def test_unmerge_restores_the_grid_through_both_insertions(mpm):
    """The head sees one row per patch; a grid row equals the merged token its pixels ended up in."""
    from vit_insertion import ViT, synthetic_images

    cfg = tiny()
    model = ViT(cfg, DEV)
    img = synthetic_images(2, cfg.image, cfg.patch, 4, DEV, sites=10)
    ws = mpm.new_workspace(2 * cfg.tokens, 2, cfg.dim, torch.bfloat16, DEV)
    trace = []
    with torch.inference_mode():
        model.forward(img, mpm=mpm, workspace=ws, trace=trace)
        (_, p1, off0), (_, p2, off1) = trace
        _, o1, m1 = mpm.merge(p1, off0, workspace=ws)
        z, o2, m2 = mpm.merge(p2, off1, workspace=ws)
        grid = mpm.compose_gather(z, o2, m1, off0, m2, off1)
    r1, r2 = m1.cpu().numpy(), m2.cpu().numpy()
    r_star = oracle.compose_batch(r1, off0.cpu().numpy(), r2, off1.cpu().numpy())
    want = oracle.gather_batch(z.float().cpu().numpy(), o2.cpu().numpy(), r_star, off0.cpu().numpy())
    assert np.array_equal(grid.float().cpu().numpy(), want)
