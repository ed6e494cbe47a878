"""GPU parity of the CUDA path (through the C ABI) against the fp64 oracle.

Small and medium cases that span several tiles with ragged tails, the
hand-worked examples, exact ties, zero rows, maximum sizes, and the kernels'
own error reporting on invalid inputs.
"""

from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
from golden_io import load_hand_examples
from parity import ParityStats, check_merge_batch, round_to, to_f64
from workloads import DTYPES, make_custom

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


def run_merge(mpm, tokens: torch.Tensor, offsets: np.ndarray, algo: str = "auto"):
    x = tokens.to(DEV)
    off = torch.from_numpy(np.asarray(offsets, dtype=np.int64)).to(DEV)
    ws = mpm.new_workspace(x.shape[0], len(offsets) - 1, x.shape[1], x.dtype, DEV)
    nn, score = mpm.nearest_neighbors(x, off, algo=algo, workspace=ws)
    assert mpm.device_status(ws) == 0
    out, out_off, rmap = mpm.merge(x, off, workspace=ws)
    assert mpm.device_status(ws) == 0
    torch.cuda.synchronize()
    t = int(out_off[-1])
    rows = int(offsets[-1])
    return {
        "nn": nn.cpu().numpy()[:rows], "score": score.cpu().numpy()[:rows],
        "map": rmap.cpu().numpy()[:rows], "out": to_f64(out[:t]), "out_offsets": out_off.cpu().numpy(),
    }


def merge_parity(mpm, batch, what: str, algo: str = "auto") -> ParityStats:
    g = run_merge(mpm, batch.tokens, batch.offsets, algo)
    x = batch.tokens.double().numpy()
    st = check_merge_batch(x, batch.offsets, g["nn"], g["map"], g["out"], g["out_offsets"], batch.dtype, what)
    return st


RAGGED = [0, 1, 2, 3, 127, 128, 129, 255, 256, 257, 300, 1000]


@pytest.mark.parametrize("algo", ["tcgen05_pair", "tcgen05_sym", "tcgen05"])
@pytest.mark.parametrize("dim", [8, 64, 200, 384, 1024])
def test_bf16_ragged_tcgen05(mpm, dim, algo):
    batch = make_custom(RAGGED, dim, "bf16", seed=dim)
    st = merge_parity(mpm, batch, f"bf16 d={dim} {algo}", algo=algo)
    assert st.images == len(RAGGED)


@pytest.mark.parametrize("dim", [8, 64, 384])
def test_bf16_ragged_simt(mpm, dim):
    batch = make_custom(RAGGED, dim, "bf16", seed=100 + dim)
    g = run_merge(mpm, batch.tokens, batch.offsets, algo="simt")
    x = batch.tokens.double().numpy()
    # The SIMT nearest neighbours obey the same acceptance rule.
    check_merge_batch(x, batch.offsets, g["nn"], g["map"], g["out"], g["out_offsets"], "bf16", "simt-nn")


@pytest.mark.parametrize("dim", [4, 192, 260])
def test_f32_ragged(mpm, dim):
    batch = make_custom(RAGGED, dim, "f32", seed=200 + dim)
    merge_parity(mpm, batch, f"f32 d={dim}")


@pytest.mark.parametrize("dtype,algo", [("bf16", "auto"), ("bf16", "tcgen05_sym"), ("bf16", "tcgen05"),
                                        ("bf16", "simt"), ("f32", "auto"), ("f32", "simt")])
def test_hand_examples_on_gpu(mpm, dtype, algo):
    """Every hand-worked example, packed into one ragged batch, zero-padded to 64 features."""
    exs = load_hand_examples()
    rows = [np.concatenate([e.tokens, np.zeros((e.tokens.shape[0], 64 - e.tokens.shape[1]))], axis=1)
            for e in exs]
    x = np.concatenate(rows, axis=0)
    offsets = np.concatenate([[0], np.cumsum([r.shape[0] for r in rows])]).astype(np.int64)
    t = torch.from_numpy(x.astype(np.float32))
    t = t.to(DTYPES[dtype])
    g = run_merge(mpm, t, offsets, algo)
    for k, e in enumerate(exs):
        a0, a1 = offsets[k], offsets[k + 1]
        assert g["nn"][a0:a1].tolist() == e.b, e.name
        assert g["map"][a0:a1].tolist() == e.r, e.name
        o0, o1 = g["out_offsets"][k], g["out_offsets"][k + 1]
        assert o1 - o0 == e.n_out, e.name
        want = round_to(dtype, oracle.merge_image(t[a0:a1].double().numpy()).x_out)
        np.testing.assert_array_equal(g["out"][o0:o1], want, err_msg=e.name)


@pytest.mark.parametrize("dtype,algo", [("bf16", "tcgen05_pair"), ("bf16", "tcgen05_sym"), ("bf16", "tcgen05"),
                                        ("bf16", "simt"), ("f32", "simt")])
def test_exact_ties_duplicates_and_zero_rows(mpm, dtype, algo):
    rng = np.random.default_rng(5)
    dim = 64
    same = np.tile(rng.standard_normal((1, dim)), (300, 1))                      # all identical
    dup = rng.standard_normal((150, dim))
    dup = np.concatenate([dup, dup[::-1] * 3.0], axis=0)                         # parallel pairs far apart
    zero = rng.standard_normal((200, dim))
    zero[[0, 17, 199]] = 0.0                                                     # zero rows
    onehot = np.eye(dim)[:40]                                                    # all cosines 0
    parts = [same, dup, zero, onehot]
    x = np.concatenate(parts, axis=0)
    offsets = np.concatenate([[0], np.cumsum([p.shape[0] for p in parts])]).astype(np.int64)
    t = torch.from_numpy(x.astype(np.float32)).to(DTYPES[dtype])
    g = run_merge(mpm, t, offsets, algo)
    # Identical tokens: b(0) = 1, b(i >= 1) = 0, one pair.
    assert g["nn"][0] == 1 and np.all(g["nn"][1:300] == 0)
    assert g["out_offsets"][1] == 299
    # Parallel pairs: i pairs with 299 - i.
    nn_dup = g["nn"][300:600]
    assert np.array_equal(nn_dup, 299 - np.arange(300))
    assert g["out_offsets"][2] - g["out_offsets"][1] == 150
    xs = t.double().numpy()
    check_merge_batch(xs, offsets, g["nn"], g["map"], g["out"], g["out_offsets"], dtype, "ties")


@pytest.mark.parametrize("algo", ["tcgen05_pair", "tcgen05_sym", "tcgen05"])
def test_large_dim_and_large_image(mpm, algo):
    batch = make_custom([300, 77], 4096, "bf16", seed=41)
    merge_parity(mpm, batch, "d=4096", algo=algo)
    big = make_custom([6000], 64, "bf16", seed=42, k=60)
    merge_parity(mpm, big, "n=6000", algo=algo)


@pytest.mark.parametrize("algo", ["tcgen05_pair", "simt"])
def test_rows_longer_than_a_prep_stage(mpm, algo):
    # 24 KiB bf16 rows: prep reads them with plain loads instead of staging
    # them through a 16 KiB shared-memory chunk.
    batch = make_custom([70, 33], 12288, "bf16", seed=43)
    merge_parity(mpm, batch, "d=12288", algo=algo)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_maximum_dim(mpm, dtype):
    # D = MPM_MAX_DIM = 16384: 32 KiB bf16 / 64 KiB fp32 rows, every K
    # stage of the default kernels (the fp32 one through its tf32 split).
    batch = make_custom([40, 17, 1], 16384, dtype, seed=45)
    merge_parity(mpm, batch, f"d=16384 {dtype}")


@pytest.mark.parametrize("algo", ["tcgen05_pair", "simt"])
def test_many_tiny_images(mpm, algo):
    # 16,000 images of 0-5 tokens, one tile each: more images than the
    # SM-pair kernel keeps in shared memory (511) and more tiles per pair of
    # SMs than it decodes up front (160).
    rng = np.random.default_rng(44)
    counts = rng.choice([0, 1, 2, 3, 5], size=16000, p=[0.05, 0.2, 0.25, 0.25, 0.25]).tolist()
    batch = make_custom(counts, 16, "bf16", seed=44)
    merge_parity(mpm, batch, "16000 tiny images", algo=algo)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_merge_is_bitwise_deterministic(mpm, dtype):
    # Candidates from many tiles meet in 64-bit atomicMax on packed (score,
    # lowest index) keys, so the order in which the SM pairs finish cannot
    # change a result: three merges (two workspaces, two streams) agree bit
    # for bit.
    batch = make_custom([1024] * 24 + [700, 513, 1, 0], 768 if dtype == "bf16" else 256, dtype, seed=47)
    x = batch.tokens.to(DEV)
    off = torch.from_numpy(batch.offsets).to(DEV)
    runs = []
    side = torch.cuda.Stream()
    for k in range(3):
        ws = mpm.new_workspace(x.shape[0], batch.batch, x.shape[1], x.dtype, DEV)
        stream = side if k == 2 else torch.cuda.current_stream()
        stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(stream):
            out, out_off, rmap = mpm.merge(x, off, workspace=ws)
        torch.cuda.synchronize()
        t = int(out_off[-1])
        runs.append((out[:t].cpu(), out_off.cpu(), rmap[:batch.rows].cpu()))
    for other in runs[1:]:
        assert torch.equal(runs[0][1], other[1])
        assert torch.equal(runs[0][2], other[2])
        assert torch.equal(runs[0][0].view(torch.int16 if dtype == "bf16" else torch.int32),
                           other[0].view(torch.int16 if dtype == "bf16" else torch.int32))


@pytest.mark.parametrize("dim", [384, 768])
def test_tcgen05_and_simt_agree(mpm, dim):
    # D = 384 runs the SM-pair kernel with 16 epilogue warps, D = 768 with 8.
    batch = make_custom([1000, 513, 64, 2300], dim, "bf16", seed=9)
    runs = {algo: run_merge(mpm, batch.tokens, batch.offsets, algo)
            for algo in ("tcgen05", "tcgen05_sym", "tcgen05_pair", "simt")}
    res = [oracle.merge_image(batch.tokens[batch.offsets[k]:batch.offsets[k + 1]].double().numpy())
           for k in range(batch.batch)]
    decisive = np.concatenate([~r.nn.near_tie for r in res])
    for algo in ("tcgen05_sym", "tcgen05_pair", "simt"):
        assert np.array_equal(runs["tcgen05"]["nn"][decisive], runs[algo]["nn"][decisive]), algo
        np.testing.assert_allclose(runs["tcgen05"]["score"], runs[algo]["score"], rtol=0, atol=1e-5)
    # Every tensor-core tiling sees the very same dot products: identical results.
    assert np.array_equal(runs["tcgen05"]["nn"], runs["tcgen05_sym"]["nn"])
    assert np.array_equal(runs["tcgen05"]["nn"], runs["tcgen05_pair"]["nn"])


@pytest.mark.parametrize("algo", ["tcgen05_pair", "tcgen05_sym", "tcgen05"])
def test_scores_are_cosines(mpm, algo):
    batch = make_custom([500, 300], 256, "bf16", seed=3)
    g = run_merge(mpm, batch.tokens, batch.offsets, algo)
    x = batch.tokens.double().numpy()
    for k in range(2):
        a0, a1 = batch.offsets[k], batch.offsets[k + 1]
        res = oracle.merge_image(x[a0:a1])
        np.testing.assert_allclose(g["score"][a0:a1], res.nn.top1, rtol=0, atol=1e-5)


def test_stage_chain_and_nondefault_stream(mpm):
    """merge -> merge -> compose -> gather on a side stream, reusing one workspace."""
    batch = make_custom([700, 2, 333], 128, "bf16", seed=12)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        x0 = batch.tokens.to(DEV, non_blocking=False)
        off0 = torch.from_numpy(batch.offsets).to(DEV)
        ws = mpm.new_workspace(x0.shape[0], 3, 128, x0.dtype, DEV)
        x1, off1, m1 = mpm.merge(x0, off0, workspace=ws)
        x2, off2, m2 = mpm.merge(x1, off1, workspace=ws)
        rs = mpm.compose_maps(m1, off0, m2, off1)
        up = mpm.unmerge_gather(x2, off2, rs, off0)
    s.synchronize()
    x = batch.tokens.double().numpy()
    o1 = oracle.merge_batch(x, batch.offsets)
    s1 = round_to("bf16", o1.x_out)
    assert np.array_equal(off1.cpu().numpy(), o1.out_offsets)
    assert np.array_equal(to_f64(x1[:o1.out_offsets[-1]]), s1)
    o2 = oracle.merge_batch(s1, o1.out_offsets)
    r_star = oracle.compose_batch(o1.r, batch.offsets, o2.r, o1.out_offsets)
    assert np.array_equal(rs.cpu().numpy()[:batch.rows], r_star)
    want = oracle.gather_batch(round_to("bf16", o2.x_out), o2.out_offsets, r_star, batch.offsets)
    assert np.array_equal(to_f64(up[:batch.rows]), want)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_compose_and_gather_kernels_on_oracle_maps(mpm, dtype):
    """Eq. 3 and Eq. 4 kernels fed the oracle's own maps and features."""
    batch = make_custom([400, 0, 1, 257, 90], 96, dtype, seed=77)
    x = batch.tokens.double().numpy()
    o1 = oracle.merge_batch(x, batch.offsets)
    o2 = oracle.merge_batch(round_to(dtype, o1.x_out), o1.out_offsets)
    r_star = oracle.compose_batch(o1.r, batch.offsets, o2.r, o1.out_offsets)
    i32 = lambda a: torch.from_numpy(np.asarray(a, dtype=np.int32)).to(DEV)  # noqa: E731
    i64 = lambda a: torch.from_numpy(np.asarray(a, dtype=np.int64)).to(DEV)  # noqa: E731
    status = torch.zeros(2, dtype=torch.int32, device=DEV)
    got = mpm.compose_maps(i32(o1.r), i64(batch.offsets), i32(o2.r), i64(o1.out_offsets), device_status=status)
    assert np.array_equal(got.cpu().numpy(), r_star)
    z = torch.from_numpy(round_to(dtype, o2.x_out).astype(np.float32)).to(DTYPES[dtype]).to(DEV)
    up = mpm.unmerge_gather(z, i64(o2.out_offsets), i32(r_star), i64(batch.offsets), device_status=status)
    want = oracle.gather_batch(z.double().cpu().numpy(), o2.out_offsets, r_star, batch.offsets)
    assert np.array_equal(to_f64(up), want)
    # Eq. 3 and Eq. 4 fused: the same grid and the same composed map, also in place over map1.
    rmap = torch.full((batch.rows,), -7, dtype=torch.int32, device=DEV)
    fused = mpm.compose_gather(z, i64(o2.out_offsets), i32(o1.r), i64(batch.offsets), i32(o2.r),
                               i64(o1.out_offsets), out_map=rmap, device_status=status)
    assert np.array_equal(to_f64(fused), want)
    assert np.array_equal(rmap.cpu().numpy(), r_star)
    inplace = i32(o1.r)
    fused2 = mpm.compose_gather(z, i64(o2.out_offsets), inplace, i64(batch.offsets), i32(o2.r),
                                i64(o1.out_offsets), out_map=inplace, device_status=status)
    assert np.array_equal(inplace.cpu().numpy(), r_star)
    assert torch.equal(fused2, fused)
    assert int(status[0]) == 0


def test_invalid_offsets_are_reported_not_faulted(mpm):
    """Non-monotone and out-of-range offsets: the kernels clamp, stay in bounds and report."""
    x = torch.randn(150, 64, device=DEV).to(torch.bfloat16)
    for bad in ([0, 100, 50, 150], [0, 100, 300], [5, 60, 150], [0, -7, 150]):
        off = torch.tensor(bad, dtype=torch.int64, device=DEV)
        ws = mpm.new_workspace(150, len(bad) - 1, 64, x.dtype, DEV)
        out, out_off, rmap = mpm.merge(x, off, workspace=ws)
        torch.cuda.synchronize()
        assert mpm.device_status(ws) == 6, bad
        assert int(out_off[-1]) <= 150


def test_bad_maps_are_reported_not_faulted(mpm):
    z = torch.randn(10, 32, device=DEV)
    zoff = torch.tensor([0, 10], dtype=torch.int64, device=DEV)
    goff = torch.tensor([0, 6], dtype=torch.int64, device=DEV)
    rmap = torch.tensor([0, 9, 10, -1, 3, 1 << 30], dtype=torch.int32, device=DEV)
    status = torch.zeros(2, dtype=torch.int32, device=DEV)
    up = mpm.unmerge_gather(z, zoff, rmap, goff, device_status=status)
    torch.cuda.synchronize()
    assert int(status[0]) == 6
    assert torch.equal(up[0], z[0]) and torch.equal(up[1], z[9]) and torch.equal(up[4], z[3])
    assert torch.count_nonzero(up[[2, 3, 5]]) == 0
    status.zero_()
    m2 = torch.arange(10, dtype=torch.int32, device=DEV)
    got = mpm.compose_maps(rmap, goff, m2, zoff, device_status=status)
    torch.cuda.synchronize()
    assert int(status[0]) == 6
    assert got.cpu().tolist() == [0, 9, -1, -1, 3, -1]


def test_empty_rows_capacity(mpm):
    """rows == 0 (every image empty) is legal."""
    x = torch.zeros(0, 64, dtype=torch.bfloat16, device=DEV)
    off = torch.zeros(4, dtype=torch.int64, device=DEV)
    out, out_off, rmap = mpm.merge(x, off)
    torch.cuda.synchronize()
    assert out_off.cpu().tolist() == [0, 0, 0, 0]
