"""Plain fp64 CPU oracle for Mutual Pair Merging (MPM), arxiv 2604.05718.

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously correct
statement of what the GPU path computes.  Only the test suite, the smoke check
in ``__graft_entry__`` and the ``cpu_baseline`` / ``--impl reference`` legs of
``bench.py`` may import it.  The product path (the C-ABI library and its
Python binding) never calls it, and it shares no code with that path.

Every function follows one step of the paper, cited by section, equation or
algorithm step (Section 3.2 "Mutual Pair Merging", Eq. 1-4, Algorithm 1):

  * ``nearest_neighbours``  - Eq. 1 and Algorithm 1 steps 1-3
  * ``mutual_partners``     - the pair set P (Section 3.2, Algorithm 1 step 4)
  * ``compact_map``         - RepMask and the left-to-right ID scan (steps 5-6)
  * ``cluster_average``     - Eq. 2 (step 7)
  * ``merge_image``         - one MPM call on one image (Algorithm 1)
  * ``compose``             - Eq. 3
  * ``gather``              - Eq. 4
  * ``merge_batch`` / ``compose_batch`` / ``gather_batch`` - the same steps
    applied image by image over a packed ragged batch ("batches are processed
    independently", Section 3.1).
  * ``pad_batch`` / ``unpad_batch`` - the padded batch of Section 4
    (Analyses): images padded to the longest merged sequence, with a key mask.

Readings of points the paper leaves open:
  * zero-norm rows are normalised by max(||x||, 1e-12) (Eq. 1 says only
    "L2-normalize");
  * ties in the arg max go to the lowest index j (the paper only says ties are
    resolved deterministically, Section 3.2);
  * an image with a single token has no neighbour: it is a singleton;
  * cluster IDs are 0-based (Algorithm 1 numbers them from 1);
  * merged rows are ordered by their representative (lower) index, so a pair
    sits where its lower member was;
  * the average is the plain mean of the current cluster, with no size
    tracking across insertions (Eq. 2);
  * merge maps hold per-image local indices.

Precision: all arithmetic is float64; inputs are widened exactly from their
bf16/fp32 storage.  ``round_bf16`` / ``round_f32`` give the value the oracle
would store in the I/O dtype (round to nearest, ties to even).
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np

# Eq. 1 reading: the normalisation floor used for zero-norm tokens.
NORM_EPS = 1e-12
# A row whose best and second-best cosine differ by at most this much is a
# "near-tie" row: its arg max is not decided robustly by finite precision.
NEAR_TIE_GAP = 1e-4


# ---------------------------------------------------------------------------
# Algorithm 1, steps 1-3 (Eq. 1): cosine affinity and nearest neighbour.
# ---------------------------------------------------------------------------
def normalise_rows(x: np.ndarray) -> np.ndarray:
    """Algorithm 1 step 1 / Eq. 1: x_i / max(||x_i||_2, 1e-12), in fp64."""
    x = np.asarray(x, dtype=np.float64)
    n = np.sqrt(np.sum(x * x, axis=1))
    return x / np.maximum(n, NORM_EPS)[:, None]


def cosine_affinity(x: np.ndarray, chunk: int | None = None) -> np.ndarray:
    """Eq. 1: S = X~ X~^T with the diagonal set to -inf (no self match).

    chunk: the chunked similarity that Section 5 proposes for very large N.
    S_ij is kept only when i and j lie in the same run of `chunk`
    consecutive tokens (raster order, the last run may be shorter); every
    other entry is -inf.
    """
    xt = normalise_rows(x)
    s = xt @ xt.T
    np.fill_diagonal(s, -np.inf)
    if chunk:
        run = np.arange(s.shape[0]) // int(chunk)
        s[run[:, None] != run[None, :]] = -np.inf
    return s


@dataclass
class Neighbours:
    """Result of Algorithm 1 step 3 for one image.

    b      int64[N]   b(i) = arg max_{j != i} S_ij (lowest j on ties); -1 if N == 1
    top1   float64[N] max_{j != i} S_ij (-inf if N == 1)
    top2   float64[N] second largest S_ij over j != i (-inf if N <= 2)
    """

    b: np.ndarray
    top1: np.ndarray
    top2: np.ndarray

    @property
    def gap(self) -> np.ndarray:
        """top1 - top2 (NaN for a single token, +inf for two tokens)."""
        with np.errstate(invalid="ignore"):
            return self.top1 - self.top2

    @property
    def near_tie(self) -> np.ndarray:
        """Rows whose top-1/top-2 gap does not exceed NEAR_TIE_GAP."""
        return ~(self.gap > NEAR_TIE_GAP)


def nearest_neighbours(x: np.ndarray, affinity: np.ndarray | None = None,
                       chunk: int | None = None) -> Neighbours:
    """Algorithm 1 step 3: b(i) = arg max_{j != i} S_ij.

    ``np.argmax`` returns the first maximal index, which is the lowest-j tie
    rule.  For N == 1 the candidate set is empty and b(0) = -1; so is it for
    a token alone in its chunk under the chunked similarity.
    """
    n = np.asarray(x).shape[0]
    if n == 0:
        e = np.zeros(0)
        return Neighbours(np.zeros(0, dtype=np.int64), e, e)
    if n == 1:
        return Neighbours(np.array([-1], dtype=np.int64), np.array([-np.inf]), np.array([-np.inf]))
    s = cosine_affinity(x, chunk) if affinity is None else affinity
    b = np.argmax(s, axis=1).astype(np.int64)
    top1 = s[np.arange(n), b]
    b[np.isneginf(top1)] = -1  # no candidate at all
    if n == 2:
        top2 = np.full(n, -np.inf)
    else:
        s2 = s.copy()
        s2[np.arange(n), b] = -np.inf
        top2 = np.max(s2, axis=1)
    return Neighbours(b, top1, top2)


# ---------------------------------------------------------------------------
# Algorithm 1 steps 4-6: mutual pairs, RepMask and compact IDs.
# ---------------------------------------------------------------------------
def mutual_partners(b: np.ndarray) -> np.ndarray:
    """Pair set P of Section 3.2: (i, j) with b(i) = j, b(j) = i, i != j.

    Returns partner[i] = j when i belongs to a mutual pair, else -1.
    """
    b = np.asarray(b, dtype=np.int64)
    n = b.shape[0]
    partner = np.full(n, -1, dtype=np.int64)
    for i in range(n):
        j = b[i]
        if 0 <= j < n and j != i and b[j] == i:
            partner[i] = j
    return partner


def compact_map(partner: np.ndarray) -> tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Algorithm 1 steps 5-6.

    RepMask[i] is true for a singleton and for the lower member of a pair.  A
    left-to-right scan gives each representative the next free 0-based ID;
    the upper member of a pair inherits its representative's ID.

    Returns (r, rep_index, rep_partner):
      r            int64[N]   cluster ID of every input token
      rep_index    int64[N']  input index of cluster k's representative
      rep_partner  int64[N']  the pair's upper member, or -1 for a singleton
    """
    partner = np.asarray(partner, dtype=np.int64)
    n = partner.shape[0]
    r = np.full(n, -1, dtype=np.int64)
    rep_index: list[int] = []
    rep_partner: list[int] = []
    next_id = 0
    for i in range(n):
        p = partner[i]
        is_rep = p < 0 or i < p
        if is_rep:
            r[i] = next_id
            rep_index.append(i)
            rep_partner.append(int(p) if p >= 0 else -1)
            next_id += 1
        else:
            # Upper member: its representative p < i was scanned already.
            r[i] = r[p]
    return r, np.array(rep_index, dtype=np.int64), np.array(rep_partner, dtype=np.int64)


def cluster_average(x: np.ndarray, r: np.ndarray, n_out: int) -> np.ndarray:
    """Eq. 2: x'_k = (1/|C_k|) sum_{i: r(i)=k} x_i, in fp64."""
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros((n_out, x.shape[1]), dtype=np.float64)
    count = np.zeros(n_out, dtype=np.float64)
    for i in range(x.shape[0]):
        out[r[i]] += x[i]
        count[r[i]] += 1.0
    return out / count[:, None]


@dataclass
class MergeResult:
    """One MPM call on one image (Algorithm 1): inputs N x d -> (X', r)."""

    x_out: np.ndarray        # float64 [N', d], exact fp64 averages
    r: np.ndarray            # int64 [N], 0-based cluster IDs
    nn: Neighbours           # b(i) with top-1/top-2 diagnostics
    partner: np.ndarray      # int64 [N], mutual partner or -1
    rep_index: np.ndarray    # int64 [N']
    rep_partner: np.ndarray  # int64 [N']

    @property
    def n_out(self) -> int:
        return int(self.x_out.shape[0])

    @property
    def n_pairs(self) -> int:
        return int(np.sum(self.rep_partner >= 0))


def merge_image(x: np.ndarray, chunk: int | None = None) -> MergeResult:
    """Algorithm 1 on a single image's tokens X (N x d); chunk as in cosine_affinity."""
    x = np.asarray(x, dtype=np.float64)
    nn = nearest_neighbours(x, chunk=chunk)
    partner = mutual_partners(nn.b)
    r, rep_index, rep_partner = compact_map(partner)
    x_out = cluster_average(x, r, int(rep_index.shape[0]))
    return MergeResult(x_out, r, nn, partner, rep_index, rep_partner)


# ---------------------------------------------------------------------------
# Eq. 3 and Eq. 4: map composition and gather reconstruction.
# ---------------------------------------------------------------------------
def compose(r1: np.ndarray, r2: np.ndarray) -> np.ndarray:
    """Eq. 3: r*(i) = r2(r1(i))."""
    r1 = np.asarray(r1, dtype=np.int64)
    r2 = np.asarray(r2, dtype=np.int64)
    return r2[r1]


def gather(z: np.ndarray, r_star: np.ndarray) -> np.ndarray:
    """Eq. 4: Z_up[i] = Z[r*(i)], a pure copy in raster order."""
    return np.asarray(z)[np.asarray(r_star, dtype=np.int64)]


# ---------------------------------------------------------------------------
# Packed ragged batches: images are independent (Section 3.1).
# ---------------------------------------------------------------------------
@dataclass
class BatchMerge:
    """A merged batch: out tokens packed by out_offsets, maps packed by offsets."""

    x_out: np.ndarray        # float64 [T', d]
    out_offsets: np.ndarray  # int64 [B+1]
    r: np.ndarray            # int64 [T], local IDs
    images: list             # list[MergeResult]


def merge_batch(tokens: np.ndarray, offsets: np.ndarray, chunk: int | None = None) -> BatchMerge:
    """Algorithm 1 applied to each image of a packed batch (chunk as in cosine_affinity)."""
    tokens = np.asarray(tokens, dtype=np.float64)
    offsets = np.asarray(offsets, dtype=np.int64)
    b_count = offsets.shape[0] - 1
    outs, maps, images = [], [], []
    out_offsets = np.zeros(b_count + 1, dtype=np.int64)
    for b in range(b_count):
        res = merge_image(tokens[offsets[b]:offsets[b + 1]], chunk)
        images.append(res)
        outs.append(res.x_out)
        maps.append(res.r)
        out_offsets[b + 1] = out_offsets[b] + res.n_out
    d = tokens.shape[1]
    x_out = np.concatenate(outs, axis=0) if outs else np.zeros((0, d))
    r = np.concatenate(maps) if maps else np.zeros(0, dtype=np.int64)
    return BatchMerge(x_out, out_offsets, r, images)


def compose_batch(r1: np.ndarray, offsets0: np.ndarray, r2: np.ndarray,
                  offsets1: np.ndarray) -> np.ndarray:
    """Eq. 3 per image, with local indices into each stage's image."""
    out = np.empty_like(np.asarray(r1, dtype=np.int64))
    for b in range(len(offsets0) - 1):
        a0, a1 = offsets0[b], offsets0[b + 1]
        c0, c1 = offsets1[b], offsets1[b + 1]
        out[a0:a1] = compose(r1[a0:a1], r2[c0:c1])
    return out


def gather_batch(z: np.ndarray, z_offsets: np.ndarray, r_star: np.ndarray,
                 grid_offsets: np.ndarray) -> np.ndarray:
    """Eq. 4 per image: out[g0_b + p] = Z[z0_b + r*(p)]."""
    z = np.asarray(z)
    out = np.empty((int(grid_offsets[-1]), z.shape[1]), dtype=z.dtype)
    for b in range(len(grid_offsets) - 1):
        g0, g1 = grid_offsets[b], grid_offsets[b + 1]
        z0, z1 = z_offsets[b], z_offsets[b + 1]
        out[g0:g1] = gather(z[z0:z1], r_star[g0:g1])
    return out


# ---------------------------------------------------------------------------
# Padded batches for dense-attention consumers (Section 4, Analyses: the
# images of a batch are padded to the longest merged sequence, and the
# padding is masked out of attention).
# ---------------------------------------------------------------------------
def pad_batch(x: np.ndarray, offsets: np.ndarray, max_len: int):
    """Packed [T, d] tokens -> ([B, L, d] padded, [B, L] key mask, (min, max, total) of N_b).

    Row t of image b is copied when t < min(N_b, L); every other row is zero and
    masked out (mask 0).  An image longer than L is cut to its first L rows.
    """
    x = np.asarray(x)
    offsets = np.asarray(offsets, dtype=np.int64)
    batch = len(offsets) - 1
    counts = offsets[1:] - offsets[:-1]
    out = np.zeros((batch, max_len, x.shape[1]), dtype=x.dtype)
    mask = np.zeros((batch, max_len), dtype=np.uint8)
    for b in range(batch):
        n = min(int(counts[b]), max_len)
        out[b, :n] = x[offsets[b]:offsets[b] + n]
        mask[b, :n] = 1
    stats = (int(counts.min()) if batch else 0, int(counts.max()) if batch else 0, int(counts.sum()))
    return out, mask, stats


def unpad_batch(padded: np.ndarray, offsets: np.ndarray) -> np.ndarray:
    """Inverse of pad_batch: packed row offsets[b] + t = padded[b, t] for t < N_b (N_b <= L)."""
    padded = np.asarray(padded)
    offsets = np.asarray(offsets, dtype=np.int64)
    out = np.zeros((int(offsets[-1]), padded.shape[2]), dtype=padded.dtype)
    for b in range(len(offsets) - 1):
        n = int(offsets[b + 1] - offsets[b])
        out[offsets[b]:offsets[b] + n] = padded[b, :n]
    return out


# ---------------------------------------------------------------------------
# Storage rounding: what the oracle would store in the I/O dtype.
# ---------------------------------------------------------------------------
def round_f32(x: np.ndarray) -> np.ndarray:
    """Round fp64 values to fp32 (round to nearest, ties to even)."""
    return np.asarray(x, dtype=np.float64).astype(np.float32)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round fp64 values directly to bfloat16 (RNE), returned as fp64 values.

    bfloat16 keeps 8 significant bits and fp32's exponent range.  For
    |x| in [2^(e-1), 2^e) the spacing of bf16 values is 2^(e-8); below the
    smallest normal (2^-126) the spacing stays 2^-133.  Scaling by a power of
    two is exact in fp64, and ``np.rint`` rounds half to even.
    """
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)
    q = np.ldexp(1.0, np.maximum(e, -125) - 8)
    y = np.rint(x / q) * q
    bf16_max = np.ldexp(255.0, 120)  # (2 - 2^-7) * 2^127
    return np.where(np.abs(y) > bf16_max, np.copysign(np.inf, x), y)
