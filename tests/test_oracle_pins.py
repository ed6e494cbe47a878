"""Pins for the fp64 oracle (CPU only).

The oracle is checked against things other than itself: hand-worked examples
(tests/golden), an exact-rational brute force on tiny integer inputs,
special cases with known answers, invariants of the method, a second library
(torch) computing the textbook cosine 1-NN, and the closed forms of Eq. 2-4.
The last test plants plausible mistakes in the oracle and checks that these
pins catch every one of them.
"""

from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle
from oracle import mpm_oracle
from exact_mpm import (exact_maximisers, exact_merge, exact_nearest, exact_row_diagnostics,
                       exact_top_gap_positive)
from golden_io import load_hand_examples
from workloads import make_custom

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


# ---------------------------------------------------------------------------
# Hand-worked examples
# ---------------------------------------------------------------------------
def check_hand_example(ex) -> None:
    res = mpm_oracle.merge_image(ex.tokens)
    assert res.nn.b.tolist() == ex.b, ex.name
    assert res.r.tolist() == ex.r, ex.name
    assert res.n_out == ex.n_out, ex.name
    means = np.stack([ex.tokens[c].mean(axis=0) for c in ex.clusters])
    np.testing.assert_allclose(res.x_out, means, rtol=0, atol=1e-15, err_msg=ex.name)
    if ex.x_out is not None:
        np.testing.assert_allclose(res.x_out, ex.x_out, rtol=0, atol=1e-15, err_msg=ex.name)
    check_hand_diagnostics(ex, res.nn)


def check_hand_diagnostics(ex, nn) -> None:
    """Best / second-best cosine and the near-tie flag against the hand values."""
    if ex.top1 is not None:
        np.testing.assert_allclose(nn.top1, ex.top1, rtol=0, atol=1e-12, err_msg=ex.name + " top1")
    if ex.top2 is not None:
        np.testing.assert_allclose(nn.top2, ex.top2, rtol=0, atol=1e-12, err_msg=ex.name + " top2")
    if ex.near_tie is not None:
        assert nn.near_tie.astype(int).tolist() == ex.near_tie, ex.name + " near_tie"


@pytest.mark.parametrize("ex", load_hand_examples(), ids=lambda e: e.name)
def test_hand_examples(ex):
    check_hand_example(ex)


@pytest.mark.parametrize("pad", [6, 62])
def test_hand_examples_zero_padding(pad):
    """Zero-padding the feature dimension changes neither dots nor norms."""
    for ex in load_hand_examples():
        wide = np.concatenate([ex.tokens, np.zeros((ex.tokens.shape[0], pad))], axis=1)
        res = mpm_oracle.merge_image(wide)
        assert res.nn.b.tolist() == ex.b and res.r.tolist() == ex.r, ex.name


# ---------------------------------------------------------------------------
# Exact-rational brute force on tiny integer inputs
# ---------------------------------------------------------------------------
def _random_int_tokens(rng, n, d, lo=-3, hi=3):
    return rng.integers(lo, hi + 1, size=(n, d))


def check_exact_bruteforce(seed_count: int = 400) -> None:
    rng = np.random.default_rng(20260405)
    strict_images = 0
    for _ in range(seed_count):
        n = int(rng.integers(1, 9))
        d = int(rng.integers(1, 6))
        x = _random_int_tokens(rng, n, d)
        xl = x.tolist()
        b_exact = exact_nearest(xl)
        res = mpm_oracle.merge_image(x.astype(np.float64))
        strict = [exact_top_gap_positive(xl, i) for i in range(n)]
        for i in range(n):
            if strict[i]:
                assert res.nn.b[i] == b_exact[i], (xl, i)
        if all(strict):
            strict_images += 1
            b, pairs, r, x_out = exact_merge(xl)
            assert res.nn.b.tolist() == b
            got_pairs = sorted((int(i), int(j)) for i, j in zip(res.rep_index, res.rep_partner) if j >= 0)
            assert got_pairs == pairs
            assert res.r.tolist() == r
            exact = np.array([[float(v) for v in row] for row in x_out], dtype=np.float64)
            np.testing.assert_array_equal(res.x_out, exact.reshape(res.x_out.shape))
    assert strict_images > seed_count // 4


def test_exact_bruteforce_tiny():
    check_exact_bruteforce()


def test_exact_bruteforce_duplicate_ties():
    """Exact duplicates give bitwise-equal fp64 cosines, so the lowest j wins.

    Every pick must be an exact maximiser, and no lower-indexed duplicate of
    the picked token may exist.
    """
    rng = np.random.default_rng(7)
    checked = 0
    for _ in range(300):
        n = int(rng.integers(3, 9))
        d = int(rng.integers(1, 5))
        base = _random_int_tokens(rng, n, d)
        for _ in range(int(rng.integers(1, 3))):
            i, j = rng.integers(0, n, size=2)
            base[j] = base[i]
        xl = base.tolist()
        res = mpm_oracle.merge_image(base.astype(np.float64))
        for i in range(n):
            j = int(res.nn.b[i])
            assert j in exact_maximisers(xl, i), (xl, i)
            assert not any(xl[k] == xl[j] for k in range(j) if k != i), (xl, i)
            checked += 1
    assert checked > 1000


# ---------------------------------------------------------------------------
# Near-tie diagnostics: the runner-up cosine and the 1e-4 gap rule
# ---------------------------------------------------------------------------
def check_exact_diagnostics(seed_count: int = 300, seed: int = 20261202) -> tuple:
    """top1 / top2 / near_tie against exact arithmetic on tiny integer tokens.

    Small entries give many exact ties (gap 0: near-tie); wide entries give
    gaps of every size.  A row whose exact gap lies within 1e-9 of the 1e-4
    threshold is not judged (fp64 may round either way there).
    Returns (decisive rows, near-tie rows without an exact tie, exact ties).
    """
    rng = np.random.default_rng(seed)
    counts = [0, 0, 0]
    for k in range(seed_count):
        n = int(rng.integers(1, 9))
        d = int(rng.integers(1, 6))
        if k % 3 == 2:
            # Near-parallel tokens (a, u, v) with a in [100, 400] and small
            # integer offsets: cosines near 1 whose differences span 1e-6..1e-2.
            n, d = int(rng.integers(3, 8)), 3
            x = np.concatenate([rng.integers(100, 401, size=(n, 1)),
                                rng.integers(-12, 13, size=(n, 2))], axis=1)
        else:
            hi = 3 if k % 3 == 0 else 60
            x = _random_int_tokens(rng, n, d, -hi, hi)
        xl = x.tolist()
        nn = mpm_oracle.nearest_neighbours(x.astype(np.float64))
        near = nn.near_tie
        for i in range(n):
            top1, top2, tied = exact_row_diagnostics(xl, i)
            if top1 is None:
                assert nn.top1[i] == -np.inf and nn.top2[i] == -np.inf and near[i], (xl, i)
                continue
            assert abs(nn.top1[i] - float(top1)) <= 1e-12, (xl, i)
            if top2 is None:
                assert nn.top2[i] == -np.inf and not near[i], (xl, i)
                counts[0] += 1
                continue
            assert abs(nn.top2[i] - float(top2)) <= 1e-12, (xl, i)
            if tied:
                assert near[i], (xl, i)
                counts[2] += 1
                continue
            gap = float(top1 - top2)
            assert gap > 0, (xl, i)
            if abs(gap - oracle.NEAR_TIE_GAP) <= 1e-9:
                continue
            assert bool(near[i]) == (gap < oracle.NEAR_TIE_GAP), (xl, i, gap)
            counts[0 if gap > oracle.NEAR_TIE_GAP else 1] += 1
    return tuple(counts)


def test_exact_bruteforce_near_tie_diagnostics():
    decisive, near_untied, ties = check_exact_diagnostics()
    assert decisive > 500 and ties > 50 and near_untied > 50, (decisive, near_untied, ties)


def check_near_tie_threshold() -> None:
    """R14: a gap of exactly 1e-4 is near-tie ("exceeds" is strict).

    The affinity rows are written out: row 0 has best 1e-4 and second 0
    (gap == 1e-4 in fp64), row 1 best just above 1e-4 (gap > 1e-4), row 2
    two equal candidates (gap 0).
    """
    above = np.nextafter(1e-4, 1.0)
    s = np.array([[-np.inf, 1e-4, 0.0],
                  [above, -np.inf, 0.0],
                  [0.25, 0.25, -np.inf]])
    nn = mpm_oracle.nearest_neighbours(np.eye(3), affinity=s)
    assert nn.b.tolist() == [1, 0, 0]
    assert nn.top1.tolist() == [1e-4, above, 0.25] and nn.top2.tolist() == [0.0, 0.0, 0.25]
    assert nn.gap[0] == oracle.NEAR_TIE_GAP
    assert nn.near_tie.tolist() == [True, False, True]


def test_near_tie_threshold_is_strict():
    check_near_tie_threshold()


def test_chunked_runner_up_stays_in_the_chunk():
    """Under chunking the runner-up is sought inside the row's chunk only (Section 5 reading).

    Chunks of 2: each row has a single candidate, so top2 is -inf and no row
    is near-tie, although the full image would tie (identical tokens).
    """
    x = np.tile(np.array([[1.0, 2.0, -1.0]]), (5, 1))
    full = mpm_oracle.nearest_neighbours(x)
    assert full.near_tie.all()
    nn = mpm_oracle.nearest_neighbours(x, chunk=2)
    assert nn.b.tolist() == [1, 0, 3, 2, -1]
    np.testing.assert_allclose(nn.top1[:4], 1.0, atol=1e-15)
    assert np.all(nn.top2 == -np.inf) and nn.near_tie.tolist() == [False] * 4 + [True]


# ---------------------------------------------------------------------------
# Special cases
# ---------------------------------------------------------------------------
def test_identical_tokens_give_one_pair():
    for n in (2, 3, 8, 33):
        x = np.tile(np.array([[0.5, -2.0, 1.0, 3.0]]), (n, 1))
        res = mpm_oracle.merge_image(x)
        assert res.nn.b[0] == 1 and np.all(res.nn.b[1:] == 0)
        assert res.n_pairs == 1 and res.n_out == n - 1


def test_duplicate_pairs_far_apart():
    rng = np.random.default_rng(3)
    k, d = 6, 16
    dirs = np.linalg.qr(rng.standard_normal((d, d)))[0][:k]   # orthonormal directions
    x = np.concatenate([dirs, dirs * 2.0], axis=0)            # token i and k+i parallel
    res = mpm_oracle.merge_image(x)
    assert res.n_pairs == k
    assert res.nn.b.tolist() == [k + i for i in range(k)] + list(range(k))
    assert res.r.tolist() == list(range(k)) * 2
    np.testing.assert_allclose(res.x_out, 1.5 * dirs, atol=1e-15)


def test_empty_and_single():
    empty = mpm_oracle.merge_image(np.zeros((0, 4)))
    assert empty.n_out == 0 and empty.r.shape == (0,)
    one = mpm_oracle.merge_image(np.array([[1.0, 2.0]]))
    assert one.nn.b.tolist() == [-1] and one.r.tolist() == [0] and one.n_out == 1


def test_all_zero_tokens():
    res = mpm_oracle.merge_image(np.zeros((5, 3)))
    assert res.nn.b.tolist() == [1, 0, 0, 0, 0]
    assert res.r.tolist() == [0, 0, 1, 2, 3]


# ---------------------------------------------------------------------------
# Invariants
# ---------------------------------------------------------------------------
def check_invariants(x: np.ndarray) -> None:
    res = mpm_oracle.merge_image(x)
    n = x.shape[0]
    b, partner, r = res.nn.b, res.partner, res.r
    # Pairs are mutual and disjoint.
    for i in range(n):
        if partner[i] >= 0:
            j = partner[i]
            assert partner[j] == i and b[i] == j and b[j] == i and j != i
    # Non-mutual tokens are singletons.
    for i in range(n):
        if n > 1 and b[b[i]] != i:
            assert partner[i] == -1
    # Size statement (corrected): N' = N - |P| >= ceil(N/2).
    assert res.n_out == n - res.n_pairs
    assert res.n_out >= math.ceil(n / 2)
    # The map is onto 0..N'-1, representatives get increasing IDs.
    assert sorted(set(r.tolist())) == list(range(res.n_out))
    assert np.array_equal(r[res.rep_index], np.arange(res.n_out))
    assert np.all(np.diff(res.rep_index) > 0)
    for k, j in enumerate(res.rep_partner):
        if j >= 0:
            assert r[j] == k and j > res.rep_index[k]
    # One insertion: the reconstructed grid keeps the per-feature sum (Eq. 2 + Eq. 4).
    up = mpm_oracle.gather(res.x_out, r)
    np.testing.assert_allclose(up.sum(axis=0), x.sum(axis=0), rtol=1e-12, atol=1e-9)
    # Each reconstructed token is its cluster's mean.
    for i in range(n):
        members = np.nonzero(r == r[i])[0]
        np.testing.assert_allclose(up[i], x[members].mean(axis=0), rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("seed", range(4))
def test_invariants_voronoi(seed):
    batch = make_custom([1, 2, 3, 37, 130, 257], 24, "f32", seed=seed)
    x = batch.tokens.double().numpy()
    for b in range(batch.batch):
        check_invariants(x[batch.offsets[b]:batch.offsets[b + 1]])


@pytest.mark.parametrize("seed", range(3))
def test_invariants_gaussian(seed):
    rng = np.random.default_rng(seed)
    for n in (2, 5, 64, 300):
        check_invariants(rng.standard_normal((n, 12)))


def test_composition_equals_sequential_gather():
    """Eq. 3 + Eq. 4: gather(gather(Z, r2), r1) == gather(Z, r2[r1])."""
    batch = make_custom([200, 77], 16, "f32", seed=11)
    x = batch.tokens.double().numpy()
    for b in range(2):
        x0 = x[batch.offsets[b]:batch.offsets[b + 1]]
        m1 = mpm_oracle.merge_image(x0)
        m2 = mpm_oracle.merge_image(m1.x_out + 0.01 * np.sin(np.arange(m1.x_out.size)).reshape(m1.x_out.shape))
        z = np.random.default_rng(b).standard_normal((m2.n_out, 16))
        seq = mpm_oracle.gather(mpm_oracle.gather(z, m2.r), m1.r)
        comp = mpm_oracle.gather(z, mpm_oracle.compose(m1.r, m2.r))
        np.testing.assert_array_equal(seq, comp)


def test_compose_and_gather_hand():
    # Stage 1 merges (0,1) and (4,5) of six tokens; stage 2 merges its outputs (1,2).
    r1 = np.array([0, 0, 1, 2, 3, 3])
    r2 = np.array([0, 1, 1, 2])
    assert mpm_oracle.compose(r1, r2).tolist() == [0, 0, 1, 1, 2, 2]
    z = np.array([[10.0], [20.0], [30.0]])
    assert mpm_oracle.gather(z, [0, 0, 1, 1, 2, 2]).ravel().tolist() == [10, 10, 20, 20, 30, 30]


def test_batch_is_per_image():
    batch = make_custom([0, 1, 50, 2, 99], 8, "f32", seed=5)
    x = batch.tokens.double().numpy()
    bm = mpm_oracle.merge_batch(x, batch.offsets)
    assert bm.out_offsets[0] == 0
    for b in range(batch.batch):
        a0, a1 = batch.offsets[b], batch.offsets[b + 1]
        single = mpm_oracle.merge_image(x[a0:a1])
        o0, o1 = bm.out_offsets[b], bm.out_offsets[b + 1]
        assert o1 - o0 == single.n_out
        np.testing.assert_array_equal(bm.x_out[o0:o1], single.x_out)
        np.testing.assert_array_equal(bm.r[a0:a1], single.r)


def test_batch_compose_gather_roundtrip():
    batch = make_custom([40, 3, 65], 8, "f32", seed=9)
    x = batch.tokens.double().numpy()
    m1 = mpm_oracle.merge_batch(x, batch.offsets)
    m2 = mpm_oracle.merge_batch(m1.x_out[:, ::-1].copy(), m1.out_offsets)
    rs = mpm_oracle.compose_batch(m1.r, batch.offsets, m2.r, m1.out_offsets)
    up = mpm_oracle.gather_batch(m2.x_out, m2.out_offsets, rs, batch.offsets)
    for b in range(batch.batch):
        a0, a1 = batch.offsets[b], batch.offsets[b + 1]
        z = m2.x_out[m2.out_offsets[b]:m2.out_offsets[b + 1]]
        np.testing.assert_array_equal(up[a0:a1], z[m2.r[m1.out_offsets[b]:m1.out_offsets[b + 1]][m1.r[a0:a1]]])


def test_chunked_hand():
    # Four tokens in two chunks of 2: 0 and 2 are the same direction, but only
    # pairs inside a chunk may form, so the pairs are (0, 1) and (2, 3).
    x = np.array([[1.0, 0.0], [0.6, 0.8], [1.0, 0.01], [0.0, 1.0]])
    full = mpm_oracle.merge_image(x)
    assert full.nn.b.tolist() == [2, 3, 0, 1]
    res = mpm_oracle.merge_image(x, chunk=2)
    assert res.nn.b.tolist() == [1, 0, 3, 2]
    assert res.r.tolist() == [0, 0, 1, 1]
    # A token alone in its (last, shorter) chunk has no neighbour.
    res3 = mpm_oracle.merge_image(x[:3], chunk=2)
    assert res3.nn.b.tolist() == [1, 0, -1] and res3.r.tolist() == [0, 0, 1]


@pytest.mark.parametrize("chunk", [3, 4, 7, 64])
def test_chunked_is_per_chunk_merge(chunk):
    """Pairs never cross chunks, so the chunked merge of an image is the merge of
    each chunk on its own, the IDs of later chunks shifted by the earlier chunks' outputs."""
    batch = make_custom([29], 12, "f32", seed=31)
    x = batch.tokens.double().numpy()
    got = mpm_oracle.merge_image(x, chunk=chunk)
    xs, rs, shift = [], [], 0
    for c0 in range(0, x.shape[0], chunk):
        part = mpm_oracle.merge_image(x[c0:c0 + chunk])
        xs.append(part.x_out)
        rs.append(part.r + shift)
        shift += part.n_out
    np.testing.assert_array_equal(got.r, np.concatenate(rs))
    np.testing.assert_array_equal(got.x_out, np.concatenate(xs))


def test_chunked_exact_bruteforce_tiny():
    """Exact rationals, chunk by chunk: every pick is an exact maximiser within its chunk."""
    rng = np.random.default_rng(17)
    checked = 0
    for _ in range(200):
        n = int(rng.integers(2, 10))
        chunk = int(rng.integers(1, 6))
        x = rng.integers(-3, 4, size=(n, 3))
        got = mpm_oracle.merge_image(x.astype(np.float64), chunk=chunk)
        for c0 in range(0, n, chunk):
            part = x[c0:c0 + chunk].tolist()
            if len(part) < 2:
                assert got.nn.b[c0] == -1
                continue
            for i in range(len(part)):
                j = int(got.nn.b[c0 + i])
                assert c0 <= j < c0 + len(part), (part, i, j)
                assert j - c0 in exact_maximisers(part, i), (part, i, j)
                top1, top2, tied = exact_row_diagnostics(part, i)
                assert abs(got.nn.top1[c0 + i] - float(top1)) <= 1e-12, (part, i)
                if top2 is None:
                    assert got.nn.top2[c0 + i] == -np.inf, (part, i)
                else:
                    assert abs(got.nn.top2[c0 + i] - float(top2)) <= 1e-12, (part, i)
                    assert not tied or got.nn.near_tie[c0 + i], (part, i)
                checked += 1
    assert checked > 500


def test_chunk_covering_the_image_is_the_full_merge():
    batch = make_custom([40], 16, "f32", seed=32)
    x = batch.tokens.double().numpy()
    a, b = mpm_oracle.merge_image(x), mpm_oracle.merge_image(x, chunk=64)
    np.testing.assert_array_equal(a.r, b.r)
    np.testing.assert_array_equal(a.x_out, b.x_out)


def test_pad_batch_hand():
    # Three images of 2, 0 and 3 one-feature tokens, padded to L = 3 (values written out by hand).
    x = np.array([[1.0], [2.0], [3.0], [4.0], [5.0]])
    off = np.array([0, 2, 2, 5])
    out, mask, stats = mpm_oracle.pad_batch(x, off, 3)
    assert out[..., 0].tolist() == [[1, 2, 0], [0, 0, 0], [3, 4, 5]]
    assert mask.tolist() == [[1, 1, 0], [0, 0, 0], [1, 1, 1]]
    assert stats == (0, 3, 5)
    # L = 2 cuts the third image to its first two rows.
    out2, mask2, _ = mpm_oracle.pad_batch(x, off, 2)
    assert out2[..., 0].tolist() == [[1, 2], [0, 0], [3, 4]]
    assert mask2.tolist() == [[1, 1], [0, 0], [1, 1]]
    assert mpm_oracle.unpad_batch(out, off)[:, 0].tolist() == [1, 2, 3, 4, 5]


def test_pad_unpad_roundtrip_and_mask_counts():
    batch = make_custom([7, 0, 1, 30, 12], 16, "f32", seed=4)
    x = batch.tokens.double().numpy()
    counts = np.diff(batch.offsets)
    out, mask, stats = mpm_oracle.pad_batch(x, batch.offsets, int(counts.max()))
    np.testing.assert_array_equal(mpm_oracle.unpad_batch(out, batch.offsets), x)
    np.testing.assert_array_equal(mask.sum(axis=1), counts)
    assert stats == (int(counts.min()), int(counts.max()), int(counts.sum()))
    assert np.all(out[mask == 0] == 0)


# ---------------------------------------------------------------------------
# Second library: torch's cosine 1-NN (first-occurrence arg max, documented)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(3))
def test_torch_cosine_nn_crosscheck(seed):
    batch = make_custom([513, 64, 2], 40, "bf16", seed=seed)
    x = batch.tokens.double()
    for b in range(batch.batch):
        xi = x[batch.offsets[b]:batch.offsets[b + 1]]
        xt = torch.nn.functional.normalize(xi, dim=1, eps=1e-12)
        s = xt @ xt.T
        s.fill_diagonal_(-float("inf"))
        want = torch.argmax(s, dim=1).numpy()
        got = mpm_oracle.nearest_neighbours(xi.numpy())
        assert np.array_equal(got.b, want)


# ---------------------------------------------------------------------------
# Storage rounding
# ---------------------------------------------------------------------------
def test_round_bf16_matches_torch_on_fp32_values():
    rng = np.random.default_rng(1)
    v = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        [0.0, -0.0, 1.0, -1.0, 3.0e38, -3.0e38, 1e-40, -1e-42]]).astype(np.float32)
    want = torch.from_numpy(v).to(torch.bfloat16).double().numpy()
    got = mpm_oracle.round_bf16(v.astype(np.float64))
    np.testing.assert_array_equal(got, want)


def test_round_bf16_ties_to_even():
    one = 1.0
    ulp = 2.0 ** -7
    assert mpm_oracle.round_bf16(np.array([one + ulp / 2]))[0] == one           # tie -> even
    assert mpm_oracle.round_bf16(np.array([one + 3 * ulp / 2]))[0] == one + 2 * ulp
    assert mpm_oracle.round_bf16(np.array([one + ulp / 2 + 2.0 ** -40]))[0] == one + ulp
    # Largest bf16 is 255 * 2^120; the halfway point to 2^128 rounds to even (overflow).
    assert mpm_oracle.round_bf16(np.array([np.ldexp(255.49, 120)]))[0] == np.ldexp(255.0, 120)
    assert mpm_oracle.round_bf16(np.array([np.ldexp(255.5, 120)]))[0] == np.inf


# ---------------------------------------------------------------------------
# The pins catch planted mistakes
# ---------------------------------------------------------------------------
def _all_pins_pass() -> bool:
    try:
        for ex in load_hand_examples():
            check_hand_example(ex)
        check_exact_bruteforce(120)
        check_exact_diagnostics(120)
        check_near_tie_threshold()
        test_duplicate_pairs_far_apart()
        rng = np.random.default_rng(0)
        check_invariants(rng.standard_normal((50, 6)))
    except (AssertionError, IndexError, ValueError):
        # A mutated oracle that crashes on a pin is caught as well.
        return False
    return True


def _nn_highest_tie(x, affinity=None, chunk=None):
    nn = _orig_nn(x, affinity)
    n = np.asarray(x).shape[0]
    if n > 1:
        s = mpm_oracle.cosine_affinity(x)
        nn.b = (n - 1 - np.argmax(s[:, ::-1], axis=1)).astype(np.int64)
    return nn


def _nn_no_mask(x, affinity=None, chunk=None):
    xt = mpm_oracle.normalise_rows(x)
    s = xt @ xt.T
    return _orig_nn(x, s)


def _nn_argmin(x, affinity=None, chunk=None):
    n = np.asarray(x).shape[0]
    if n <= 1:
        return _orig_nn(x, affinity)
    s = mpm_oracle.cosine_affinity(x)
    np.fill_diagonal(s, np.inf)
    return _orig_nn(x, -s)


def _nn_unnormalised(x, affinity=None, chunk=None):
    n = np.asarray(x).shape[0]
    if n <= 1:
        return _orig_nn(x, affinity)
    x = np.asarray(x, dtype=np.float64)
    s = x @ x.T
    np.fill_diagonal(s, -np.inf)
    return _orig_nn(x, s)


def _partners_not_mutual(b):
    b = np.asarray(b)
    p = np.full(b.shape[0], -1, dtype=np.int64)
    for i in range(b.shape[0]):
        j = b[i]
        if j >= 0 and p[i] < 0 and p[j] < 0 and j != i:
            p[i], p[j] = j, i
    return p


def _compact_upper_rep(partner):
    r, ri, rp = _orig_compact(partner)
    # Representative = upper member: scan assigns IDs at the upper index.
    n = partner.shape[0]
    rr = np.full(n, -1, dtype=np.int64)
    nid = 0
    for i in range(n):
        p = partner[i]
        if p < 0 or i > p:
            rr[i] = nid
            if p >= 0:
                rr[p] = nid
            nid += 1
    order = [int(np.nonzero(rr == k)[0].min()) for k in range(nid)]
    return rr, np.array(order), np.array([partner[i] for i in order])


def _compact_one_based(partner):
    r, ri, rp = _orig_compact(partner)
    return r + 1, ri, rp


def _average_sum(x, r, n_out):
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros((n_out, x.shape[1]))
    for i in range(x.shape[0]):
        out[r[i]] += x[i]
    return out


def _average_first(x, r, n_out):
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros((n_out, x.shape[1]))
    seen = set()
    for i in range(x.shape[0]):
        if r[i] not in seen:
            out[r[i]] = x[i]
            seen.add(r[i])
    return out


def _affinity_for(x, affinity, chunk):
    return mpm_oracle.cosine_affinity(x, chunk) if affinity is None else affinity


def _nn_top2_drops_ties(x, affinity=None, chunk=None):
    # Runner-up taken among the candidates strictly below the best: an exact
    # tie then looks like a clear win.
    nn = _orig_nn(x, affinity, chunk)
    if nn.b.shape[0] > 2:
        s = _affinity_for(x, affinity, chunk)
        nn.top2 = np.where(s >= nn.top1[:, None], -np.inf, s).max(axis=1)
    return nn


def _nn_top2_row_min(x, affinity=None, chunk=None):
    # Runner-up replaced by the worst candidate.
    nn = _orig_nn(x, affinity, chunk)
    if nn.b.shape[0] > 2:
        s = _affinity_for(x, affinity, chunk)
        nn.top2 = np.where(np.isneginf(s), np.inf, s).min(axis=1)
    return nn


def _nn_top2_keeps_self(x, affinity=None, chunk=None):
    # Runner-up searched over an affinity whose diagonal was never masked.
    nn = _orig_nn(x, affinity, chunk)
    n = nn.b.shape[0]
    if n > 2:
        xt = mpm_oracle.normalise_rows(x)
        s = xt @ xt.T
        s[np.arange(n), nn.b] = -np.inf
        nn.top2 = s.max(axis=1)
    return nn


_orig_nn = mpm_oracle.nearest_neighbours
_orig_compact = mpm_oracle.compact_map
_N = mpm_oracle.Neighbours

MUTATIONS = {
    "tie_to_highest_j": (mpm_oracle, "nearest_neighbours", _nn_highest_tie),
    "no_diagonal_mask": (mpm_oracle, "nearest_neighbours", _nn_no_mask),
    "argmin_instead_of_argmax": (mpm_oracle, "nearest_neighbours", _nn_argmin),
    "dot_not_cosine": (mpm_oracle, "nearest_neighbours", _nn_unnormalised),
    "pairs_not_mutual": (mpm_oracle, "mutual_partners", _partners_not_mutual),
    "upper_index_representative": (mpm_oracle, "compact_map", _compact_upper_rep),
    "one_based_ids": (mpm_oracle, "compact_map", _compact_one_based),
    "sum_not_mean": (mpm_oracle, "cluster_average", _average_sum),
    "keep_first_member": (mpm_oracle, "cluster_average", _average_first),
    # Near-tie diagnostics (Section 3.2's b(i) runner-up and the 1e-4 gap rule).
    "gap_always_zero": (_N, "gap", property(lambda self: np.zeros_like(self.top1))),
    "gap_sign_flipped": (_N, "gap", property(lambda self: self.top2 - self.top1)),
    "near_tie_at_or_above_threshold": (
        _N, "near_tie", property(lambda self: ~(self.gap >= mpm_oracle.NEAR_TIE_GAP))),
    "near_tie_ignores_undefined_gap": (
        _N, "near_tie", property(lambda self: self.gap <= mpm_oracle.NEAR_TIE_GAP)),
    "top2_drops_ties_of_top1": (mpm_oracle, "nearest_neighbours", _nn_top2_drops_ties),
    "top2_is_row_minimum": (mpm_oracle, "nearest_neighbours", _nn_top2_row_min),
    "top2_sees_the_diagonal": (mpm_oracle, "nearest_neighbours", _nn_top2_keeps_self),
}


def test_pins_pass_on_the_oracle():
    assert _all_pins_pass()


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, monkeypatch):
    owner, attr, value = MUTATIONS[name]
    monkeypatch.setattr(owner, attr, value)
    assert not _all_pins_pass(), f"planted mistake {name} went unnoticed"


def test_public_names():
    assert oracle.merge_image is mpm_oracle.merge_image
    assert oracle.NEAR_TIE_GAP == 1e-4
