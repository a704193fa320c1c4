"""Pins for the oracle's geometry (Sec. 1 "The code", Fig. 1 caption).

The N-gon, the packing ratio r_N and the span length are checked against
facts the paper and plane geometry fix independently of the oracle's code:
closed forms, a brute-force separating-axis search for the largest ratio with
disjoint cells, and the cell-containment meaning of nearest-vertex decoding.
"""
import math

import numpy as np
import pytest

NS = [3, 4, 5, 6, 8, 16, 64, 256]


def test_midpoint_is_the_boundary_for_small_alphabets(oracle_mod):
    # Sec. 1: the midpoint code r = 1/2 is exactly the boundary case for N <= 4.
    assert oracle_mod.packing_ratio(3) == 0.5
    assert oracle_mod.packing_ratio(4) == 0.5
    for N in range(5, 40):
        assert oracle_mod.packing_ratio(N) < 0.5   # must be tightened for N > 4


@pytest.mark.parametrize("N,closed", [
    (5, (3.0 - math.sqrt(5.0)) / 2.0),          # 1 / (1 + golden ratio)
    (6, 1.0 / 3.0),
    (8, 1.0 / (2.0 + math.sqrt(2.0))),
    (12, 1.0 / (3.0 + math.sqrt(3.0))),
])
def test_packing_ratio_closed_forms(oracle_mod, N, closed):
    # Known closed forms of the N-flake (touching-cells) ratio.
    assert oracle_mod.packing_ratio(N) == pytest.approx(closed, rel=4e-16)


def test_area_argument(oracle_mod):
    # Fig. 1 caption: a cell at ratio r has r^2 of the polygon's area, so N
    # disjoint cells need N r^2 <= 1 (N = 4 tiles exactly at r = 1/2).
    for N in range(3, 300):
        r = oracle_mod.packing_ratio(N)
        assert N * r * r <= 1.0 + 1e-15
    assert 4 * oracle_mod.packing_ratio(4) ** 2 == 1.0


def _cell(V, c, r):
    return V[c] + r * (V - V[c])


def _separation(A, B, normals):
    """Largest gap between the projections of convex polygons A and B over
    the candidate axes (> 0 disjoint, 0 touching, < 0 overlapping)."""
    pa = A @ normals.T
    pb = B @ normals.T
    gap = np.maximum(pb.min(0) - pa.max(0), pa.min(0) - pb.max(0))
    return gap.max()


def _normals(V):
    e = np.roll(V, -1, axis=0) - V
    n = np.stack([e[:, 1], -e[:, 0]], axis=1)
    return n / np.linalg.norm(n, axis=1, keepdims=True)


@pytest.mark.parametrize("N", NS)
def test_bruteforce_largest_disjoint_ratio(oracle_mod, N):
    # Independent of the oracle's formula: bisect on r for the largest ratio at
    # which cells 0 and 1 (adjacent, the closest pair) stay disjoint.
    V = oracle_mod.vertices(N)
    nrm = _normals(V)
    lo, hi = 0.01 / N, 0.75
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if _separation(_cell(V, 0, mid), _cell(V, 1, mid), nrm) >= 0.0:
            lo = mid
        else:
            hi = mid
    rN = oracle_mod.packing_ratio(N)
    assert abs(lo - rN) <= 1e-12 * rN, (N, lo, rN)


@pytest.mark.parametrize("N", NS)
def test_cells_disjoint_at_rN_and_overlap_above(oracle_mod, N):
    V = oracle_mod.vertices(N)
    nrm = _normals(V)
    rN = oracle_mod.packing_ratio(N)
    for j in range(1, N // 2 + 1):
        sep = _separation(_cell(V, 0, rN), _cell(V, j, rN), nrm)
        assert sep >= -1e-14, (N, j, sep)          # disjoint interiors (touch allowed)
    over = _separation(_cell(V, 0, rN * (1 + 1e-9)), _cell(V, 1, rN * (1 + 1e-9)), nrm)
    assert over < 0.0


@pytest.mark.parametrize("N", NS)
def test_nearest_vertex_is_cell_containment(oracle_mod, N):
    # Sec. 1: the symbol is the vertex whose cell contains the point.  Random
    # points of random cells must decode (one backward step) to that cell.
    rng = np.random.default_rng(N)
    V = oracle_mod.vertices(N)
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    m = 4000
    c = rng.integers(0, N, size=m)
    w = rng.dirichlet(np.full(N, 0.5), size=m)
    q = w @ V                                     # uniform-ish points of the hull
    p = V[c] + r * (q - V[c])
    for i in range(m):
        sym, _, _ = oracle_mod.span_decode(p[i:i + 1], 1, N, r, L, tol=10.0)
        assert sym[0] == c[i]


def test_vertices_against_high_precision(oracle_mod):
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 40
    for N in NS:
        V = oracle_mod.vertices(N)
        for c in range(N):
            if (4 * c) % N == 0:
                continue
            # the reading evaluates cos/sin at the binary64 angle 2.0*pi*c/N:
            # within 1 ulp of the true cos/sin of that rounded angle ...
            th64 = mpmath.mpf(2.0 * np.pi * c / N)
            ex, ey = float(mpmath.cos(th64)), float(mpmath.sin(th64))
            assert abs(V[c, 0] - ex) <= np.spacing(abs(ex))
            assert abs(V[c, 1] - ey) <= np.spacing(abs(ey))
            # ... and within 1e-15 of the exact regular polygon
            th = 2 * mpmath.pi * c / N
            assert abs(V[c, 0] - float(mpmath.cos(th))) < 1e-15
            assert abs(V[c, 1] - float(mpmath.sin(th))) < 1e-15
        assert tuple(V[0]) == (1.0, 0.0)
        if N % 4 == 0:
            assert tuple(V[N // 4]) == (0.0, 1.0)
            assert tuple(V[N // 2]) == (-1.0, 0.0)


@pytest.mark.parametrize("N,L", [(3, 44), (4, 44), (16, 16), (256, 6), (1024, 5)])
def test_span_length(oracle_mod, N, L):
    # Sec. 1: about 44 / log2(1/r) symbols per double; the span is its floor.
    r = oracle_mod.packing_ratio(N)
    assert oracle_mod.max_span_len(r) == L
    assert L == math.floor(44.0 / math.log2(1.0 / r))
