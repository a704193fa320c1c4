"""Pins for the oracle's span codec (Sec. 1 "The code", Sec. 2, Sec. 5).

Checked against: hand-worked midpoint points, the Sierpinski (N = 3) and
diamond (N = 4) binary-digit readings, the exact rational closed form of the
map, exhaustive round trips on tiny streams, the capacity of one double, and
the 2 r^s suffix decay.
"""
import itertools
import math
import os
from fractions import Fraction

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "midpoint_points.txt")


def _golden_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            N, syms, x, y = [t.strip() for t in line.split("|")]
            rows.append((int(N), [int(s) for s in syms.split()], float(x), float(y)))
    return rows


@pytest.mark.parametrize("row", _golden_rows(), ids=lambda r: "N%d-%s" % (r[0], "".join(map(str, r[1]))))
def test_hand_worked_midpoint_points(oracle_mod, row):
    N, syms, x, y = row
    pts = oracle_mod.span_encode(syms, N, 0.5, len(syms))
    assert pts.shape == (1, 2)
    assert pts[0, 0] == x and pts[0, 1] == y


def test_sierpinski_binary_digits(oracle_mod):
    # Sec. 1: for N = 3, r = 1/2 the attractor is the Sierpinski gasket and the
    # point's barycentric coordinates are binary expansions of the symbols:
    # lambda_j = sum_{k: c_k = j} 2^-(m-k+1) + (1/3) 2^-m (anchor at the centroid).
    rng = np.random.default_rng(3)
    V = oracle_mod.vertices(3)
    A = np.vstack([V.T, np.ones(3)])
    for m in [1, 2, 5, 13, 30, 44]:
        for _ in range(50):
            c = rng.integers(0, 3, size=m)
            p = oracle_mod.span_encode(c, 3, 0.5, m)[0]
            lam = np.linalg.solve(A, np.array([p[0], p[1], 1.0]))
            want = np.full(3, 2.0 ** -m / 3.0)
            for k in range(m):
                want[c[k]] += 2.0 ** -(m - k)
            assert np.max(np.abs(lam - want)) < 1e-14


def test_diamond_binary_digits(oracle_mod):
    # N = 4, r = 1/2: u = x + y and v = x - y each walk a binary expansion
    # (u(V) = +1 for symbols 0,1 and -1 for 2,3; v(V) = +1 for 0,3, -1 for 1,2),
    # so the symbols can be read back from the bits of (u + 1 - 2^-m) / 2.
    rng = np.random.default_rng(4)
    for m in [1, 7, 20, 44]:
        c = rng.integers(0, 4, size=m)
        p = oracle_mod.span_encode(c, 4, 0.5, m)[0]
        for coord, plus in ((p[0] + p[1], {0, 1}), (p[0] - p[1], {0, 3})):
            frac = Fraction(coord) + 1 - Fraction(1, 2 ** m)
            frac /= 2
            bits = []
            for _ in range(m):
                frac *= 2
                b = int(frac >= 1)
                bits.append(b)
                frac -= b
            assert frac == 0
            # bit i (most significant first) belongs to symbol c_{m-i}
            assert bits == [int(int(ck) in plus) for ck in c[::-1]]


@pytest.mark.parametrize("N", [3, 5, 16, 256])
def test_closed_form_exact_rational(oracle_mod, N):
    # p_m = r^m p_0 + (1 - r) sum_k r^(m-k) V(c_k), evaluated exactly on the
    # binary64 values of r and V; the oracle's rounded walk stays within
    # (m + 1) 2^-52 of it.
    rng = np.random.default_rng(N)
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    V = oracle_mod.vertices(N)
    R = Fraction(r)
    VF = [(Fraction(V[c, 0]), Fraction(V[c, 1])) for c in range(N)]
    for _ in range(40):
        m = int(rng.integers(1, L + 1))
        c = rng.integers(0, N, size=m)
        p = oracle_mod.span_encode(c, N, r, m)[0]
        ex = ey = Fraction(0)
        for k in range(m):
            w = (1 - R) * R ** (m - 1 - k)
            ex += w * VF[c[k]][0]
            ey += w * VF[c[k]][1]
        tol = (m + 1) * 2.0 ** -52
        assert abs(float(Fraction(p[0]) - ex)) <= tol
        assert abs(float(Fraction(p[1]) - ey)) <= tol


def _all_streams(N, m):
    return np.array(list(itertools.product(range(N), repeat=m)), dtype=np.int32).reshape(-1)


@pytest.mark.parametrize("N,mmax", [(3, 12), (4, 10), (16, 5), (256, 2)])
def test_exhaustive_round_trip(oracle_mod, N, mmax):
    # Sec. 1-2: the code is lossless.  Every stream up to length mmax, each as
    # one span from the anchor.
    r = oracle_mod.packing_ratio(N)
    for m in range(1, mmax + 1):
        s = _all_streams(N, m)
        pts = oracle_mod.span_encode(s, N, r, m)
        d, anchor, bad = oracle_mod.span_decode(pts, s.size, N, r, m)
        assert bad == 0
        assert np.array_equal(d, s)
        # distinct streams -> distinct points (injective)
        assert np.unique(pts, axis=0).shape[0] == N ** m


def test_exhaustive_round_trip_n256_len3(oracle_mod):
    N = 256
    r = oracle_mod.packing_ratio(N)
    s = _all_streams(N, 3)
    pts = oracle_mod.span_encode(s, N, r, 3)
    d, _, bad = oracle_mod.span_decode(pts, s.size, N, r, 3)
    assert bad == 0 and np.array_equal(d, s)


@pytest.mark.parametrize("N", [3, 4, 16, 256])
def test_every_tail_length(oracle_mod, N):
    rng = np.random.default_rng(10 + N)
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    for t in range(0, L):
        n = 7 * L + t
        s = rng.integers(0, N, size=n).astype(np.int32)
        pts = oracle_mod.span_encode(s, N, r, L)
        assert pts.shape[0] == 7 + (t > 0)
        d, _, bad = oracle_mod.span_decode(pts, n, N, r, L)
        assert bad == 0 and np.array_equal(d, s)


def _adversarial(N, L):
    out = []
    for c in range(N):
        out.append(np.full(L, c))                               # constant
        out.append(np.resize([c, (c + 1) % N], L))              # alternating neighbours
        out.append(np.resize([(c + 1) % N, c], L))
        out.append(np.concatenate([[c], np.full(L - 1, (c + 1) % N)]))  # one then the neighbour
    return np.concatenate(out).astype(np.int32)


@pytest.mark.parametrize("N", [3, 4, 5, 8, 16, 64, 256])
def test_adversarial_streams_at_full_span(oracle_mod, N):
    # Streams that push points toward the kissing points (smallest margin).
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    s = _adversarial(N, L)
    pts = oracle_mod.span_encode(s, N, r, L)
    d, _, bad = oracle_mod.span_decode(pts, s.size, N, r, L)
    assert bad == 0 and np.array_equal(d, s)


@pytest.mark.parametrize("N", [3, 4, 16, 256])
def test_capacity_of_one_double(oracle_mod, N):
    # Sec. 1: inversion amplifies rounding by 1/r per step, so one double
    # carries about 44/log2(1/r) symbols.  Round trips hold through the span
    # length and fail on random streams once the span is far beyond it
    # (about 53/log2(1/r), where the 53-bit significand runs out).
    rng = np.random.default_rng(20 + N)
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    for LL in range(1, L + 1):
        s = rng.integers(0, N, size=LL * 3000).astype(np.int32)
        pts = oracle_mod.span_encode(s, N, r, LL)
        d, _, _ = oracle_mod.span_decode(pts, s.size, N, r, LL, tol=1e300)
        assert np.array_equal(d, s), LL
    LL = int(math.ceil(56.0 / math.log2(1.0 / r)))
    s = rng.integers(0, N, size=LL * 3000).astype(np.int32)
    pts = oracle_mod.span_encode(s, N, r, LL)
    d, _, _ = oracle_mod.span_decode(pts, s.size, N, r, LL, tol=1e300)
    assert not np.array_equal(d, s)


@pytest.mark.parametrize("N", [3, 16, 256])
def test_suffix_decay(oracle_mod, N):
    # Sec. 5: two streams sharing an s-symbol suffix have points within 2 r^s.
    rng = np.random.default_rng(30 + N)
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    for s_len in range(0, L + 1):
        a = rng.integers(0, N, size=(500, L)).astype(np.int32)
        b = rng.integers(0, N, size=(500, L)).astype(np.int32)
        if s_len:
            b[:, L - s_len:] = a[:, L - s_len:]
        pa = oracle_mod.span_encode(a.reshape(-1), N, r, L)
        pb = oracle_mod.span_encode(b.reshape(-1), N, r, L)
        dist = np.linalg.norm(pa - pb, axis=1)
        assert dist.max() <= 2 * r ** s_len + 1e-15


def test_anchor_check_flags_a_corrupted_point(oracle_mod):
    N = 256
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(5)
    s = rng.integers(0, N, size=L * 1000).astype(np.int32)
    pts = oracle_mod.span_encode(s, N, r, L)
    _, anchor, bad = oracle_mod.span_decode(pts, s.size, N, r, L)
    assert bad == 0 and anchor.max() < 2.0 ** -10
    bits = pts.view(np.uint64).copy()
    bits[17, 0] ^= np.uint64(1) << np.uint64(40)     # flip a mantissa bit
    _, anchor2, bad2 = oracle_mod.span_decode(bits.view(np.float64), s.size, N, r, L)
    assert bad2 >= 1 and anchor2[17] > 2.0 ** -4


def test_read_and_append_definitions(oracle_mod):
    # Sec. 2: random access decodes only the span holding the position, append
    # re-walks only the tail; both equal the full computation.
    N = 16
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(6)
    s = rng.integers(0, N, size=1000).astype(np.int32)
    pts = oracle_mod.span_encode(s, N, r, L)
    pos = rng.integers(0, s.size, size=300)
    assert np.array_equal(oracle_mod.read(pts, s.size, pos, N, r, L), s[pos])
    extra = rng.integers(0, N, size=37).astype(np.int32)
    p2 = oracle_mod.append(s, extra, N, r, L)
    assert np.array_equal(p2[: s.size // L], pts[: s.size // L])
    d, _, bad = oracle_mod.span_decode(p2, s.size + extra.size, N, r, L)
    assert bad == 0 and np.array_equal(d, np.concatenate([s, extra]))
