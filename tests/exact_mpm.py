"""Exact-rational brute force of one MPM call, for pinning the fp64 oracle.

Works on small integer-valued tokens only.  Nothing here is shared with the
oracle: cosines are never formed.  For a fixed row i, the cosine S_ij =
(x_i . x_j) / (|x_i| |x_j|) orders the candidates j like d_ij / |x_j| with
d_ij = x_i . x_j, because |x_i| > 0 is common to the row (a zero row has
S_ij = 0 for every j under the max(|x|, eps) normalisation of Eq. 1).  Two
such ratios are compared exactly with integers: d / sqrt(q) against
e / sqrt(p) by sign first, then by d^2 p against e^2 q.

Definitions followed: Eq. 1 (affinity), Section 3.2 (b(i), the pair set P,
lower index as representative), Algorithm 1 steps 5-7 (left-to-right compact
IDs, cluster means, Eq. 2).
"""

from __future__ import annotations

from fractions import Fraction


def _dot(a, b) -> int:
    return sum(int(u) * int(v) for u, v in zip(a, b))


def _cmp_ratio(d1: int, q1: int, d2: int, q2: int) -> int:
    """Sign of d1/sqrt(q1) - d2/sqrt(q2) with q1, q2 > 0 (exact)."""
    s1 = (d1 > 0) - (d1 < 0)
    s2 = (d2 > 0) - (d2 < 0)
    if s1 != s2:
        return (s1 > s2) - (s1 < s2)
    if s1 == 0:
        return 0
    lhs = d1 * d1 * q2
    rhs = d2 * d2 * q1
    c = (lhs > rhs) - (lhs < rhs)
    return c if s1 > 0 else -c


def exact_nearest(x: list) -> list:
    """b(i) = lowest j != i with maximal exact cosine; -1 when N == 1."""
    n = len(x)
    q = [_dot(v, v) for v in x]
    out = []
    for i in range(n):
        best = -1
        for j in range(n):
            if j == i:
                continue
            if best < 0:
                best = j
                continue
            if q[i] == 0:
                continue  # zero row: every cosine is 0, keep the lowest j
            # A zero candidate has cosine 0: represent it as the ratio 0 / 1.
            dj, qj = (_dot(x[i], x[j]), q[j]) if q[j] else (0, 1)
            db, qb = (_dot(x[i], x[best]), q[best]) if q[best] else (0, 1)
            if _cmp_ratio(dj, qj, db, qb) > 0:
                best = j
        out.append(best)
    return out


def exact_top_gap_positive(x: list, i: int) -> bool:
    """True when row i's best cosine strictly beats every other candidate."""
    n = len(x)
    b = exact_nearest(x)[i]
    if b < 0 or n <= 2:
        return True
    q = [_dot(v, v) for v in x]
    if q[i] == 0:
        return False
    db, qb = (_dot(x[i], x[b]), q[b]) if q[b] else (0, 1)
    for j in range(n):
        if j in (i, b):
            continue
        dj, qj = (_dot(x[i], x[j]), q[j]) if q[j] else (0, 1)
        if _cmp_ratio(dj, qj, db, qb) == 0:
            return False
    return True


def exact_merge(x: list):
    """One MPM call in exact arithmetic.

    Returns (b, pairs, r, x_out) with pairs a sorted list of (i, j), i < j,
    r the 0-based compact IDs and x_out a list of Fraction rows.
    """
    n = len(x)
    b = exact_nearest(x)
    pairs = sorted((i, b[i]) for i in range(n)
                   if b[i] > i and b[b[i]] == i)
    upper = {j: i for i, j in pairs}
    r = [-1] * n
    nid = 0
    for i in range(n):
        if i in upper:
            r[i] = r[upper[i]]
        else:
            r[i] = nid
            nid += 1
    members = [[] for _ in range(nid)]
    for i in range(n):
        members[r[i]].append(i)
    d = len(x[0]) if n else 0
    x_out = [[sum(Fraction(int(x[i][k])) for i in m) / len(m) for k in range(d)]
             for m in members]
    return b, pairs, r, x_out


def exact_maximisers(x: list, i: int) -> set:
    """All j != i attaining row i's maximal exact cosine."""
    n = len(x)
    b = exact_nearest(x)[i]
    if b < 0:
        return set()
    q = [_dot(v, v) for v in x]
    if q[i] == 0:
        return {j for j in range(n) if j != i}
    db, qb = (_dot(x[i], x[b]), q[b]) if q[b] else (0, 1)
    out = set()
    for j in range(n):
        if j == i:
            continue
        dj, qj = (_dot(x[i], x[j]), q[j]) if q[j] else (0, 1)
        if _cmp_ratio(dj, qj, db, qb) == 0:
            out.add(j)
    return out


def _cos_decimal(x: list, i: int, j: int):
    """cos(x_i, x_j) to 50 significant digits; 0 when either token is zero."""
    from decimal import Decimal, localcontext

    qi, qj = _dot(x[i], x[i]), _dot(x[j], x[j])
    if qi == 0 or qj == 0:
        return Decimal(0)
    with localcontext() as ctx:
        ctx.prec = 50
        return Decimal(_dot(x[i], x[j])) / (Decimal(qi) * Decimal(qj)).sqrt()


def exact_row_diagnostics(x: list, i: int):
    """Best and second-best cosine of row i over j != i (Section 3.2's b(i) and runner-up).

    Candidates are ordered by the exact comparator (no rounding decides the
    order); the two values are then evaluated to 50 digits.  Returns
    (top1, top2, tied): top1/top2 are Decimals or None for "no candidate"
    (-inf), and tied is True when the two best candidates have exactly equal
    cosines (gap exactly 0).
    """
    from functools import cmp_to_key

    n = len(x)
    cands = [j for j in range(n) if j != i]
    if not cands:
        return None, None, False
    q = [_dot(v, v) for v in x]

    def ratio(j):
        if q[i] == 0 or q[j] == 0:
            return 0, 1
        return _dot(x[i], x[j]), q[j]

    def cmp(a, b):  # descending by exact cosine
        return -_cmp_ratio(*ratio(a), *ratio(b))

    order = sorted(cands, key=cmp_to_key(cmp))
    top1 = _cos_decimal(x, i, order[0])
    if len(order) == 1:
        return top1, None, False
    tied = cmp(order[0], order[1]) == 0
    return top1, _cos_decimal(x, i, order[1]), tied
