"""Pins of the oracle's in-place suffix retrieval (Sec. 5) against facts the
paper and the geometry fix: the 2 r^s decay law between points sharing an
s-symbol suffix, recall 1 by construction, exact string matching checked by
brute force on the known input symbols, and the degenerate cases."""
import numpy as np
import pytest

NS = [3, 4, 16, 256]


def _span_ends(sym, n, L, qlen):
    """Brute force on the input symbols: spans whose last qlen symbols, taken
    from the span itself, equal each other -> dict suffix -> span list."""
    out = {}
    for u in range((n + L - 1) // L):
        m = min(L, n - u * L)
        if m >= qlen:
            out.setdefault(tuple(sym[u * L + m - qlen:u * L + m]), []).append(u)
    return out


@pytest.mark.parametrize("N", NS)
def test_decay_law_between_points_sharing_a_suffix(oracle_mod, N):
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(N)
    for s in range(1, L + 1):
        tail = rng.integers(0, N, s)
        a = np.concatenate([rng.integers(0, N, L - s), tail])
        b = np.concatenate([rng.integers(0, N, L - s), tail])
        pa = oracle_mod.span_encode(a, N, r, L)[0]
        pb = oracle_mod.span_encode(b, N, r, L)[0]
        q = oracle_mod.span_encode(tail, N, r, s)[0]     # the suffix alone, from the origin
        # every point of the polygon is within the unit circle, so the
        # prefix contributes at most r^s (to the query) and 2 r^s (to a peer)
        assert np.hypot(*(pa - pb)) <= 2.0 * r ** s * (1 + 1e-12)
        assert np.hypot(*(pa - q)) <= r ** s * (1 + 1e-12)


@pytest.mark.parametrize("N", NS)
def test_matches_equal_brute_force_and_recall_is_one(oracle_mod, N):
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(100 + N)
    n = 400 * L + L // 2 + 1                           # a ragged tail span
    sym = rng.integers(0, min(N, 4), n).astype(np.int32)   # a small alphabet: many true matches
    pts = oracle_mod.span_encode(sym, N, r, L)
    for qlen in sorted({1, 2, max(1, L // 2), L}):
        ends = _span_ends(sym, n, L, qlen)
        for key in list(ends)[:6]:
            match, cand = oracle_mod.suffix_search(pts, n, key, N, r, L)
            assert match.tolist() == sorted(ends[key])            # exact string matches
            assert set(match.tolist()) <= set(cand.tolist())     # recall 1: every match is inside the ball
        miss = tuple(int(N - 1) for _ in range(qlen)) if N > 4 else None
        if miss is not None and miss not in ends:
            match, _ = oracle_mod.suffix_search(pts, n, miss, N, r, L)
            assert match.size == 0


def test_full_span_query_hits_its_point_exactly(oracle_mod):
    N = 256
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(7)
    sym = rng.integers(0, N, 50 * L).astype(np.int32)
    pts = oracle_mod.span_encode(sym, N, r, L)
    u = 17
    q = oracle_mod.span_encode(sym[u * L:(u + 1) * L], N, r, L)[0]
    assert np.array_equal(q, pts[u])                   # same map chain from the origin: equal bits
    match, cand = oracle_mod.suffix_search(pts, sym.size, sym[u * L:(u + 1) * L], N, r, L)
    assert u in match.tolist()


def test_short_tail_span_never_matches_and_bad_queries_raise(oracle_mod):
    N = 16
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    sym = np.zeros(3 * L + 2, np.int32)                 # tail span of 2 symbols
    pts = oracle_mod.span_encode(sym, N, r, L)
    match, cand = oracle_mod.suffix_search(pts, sym.size, np.zeros(3, np.int32), N, r, L)
    assert match.tolist() == [0, 1, 2] and 3 not in cand.tolist()
    match, _ = oracle_mod.suffix_search(pts, sym.size, np.zeros(2, np.int32), N, r, L)
    assert match.tolist() == [0, 1, 2, 3]
    with pytest.raises(ValueError):
        oracle_mod.suffix_search(pts, sym.size, np.zeros(L + 1, np.int32), N, r, L)
    with pytest.raises(ValueError):
        oracle_mod.suffix_search(pts, sym.size, np.zeros(0, np.int32), N, r, L)


def test_radius_is_the_product_form(oracle_mod):
    r = oracle_mod.packing_ratio(256)
    for l in range(1, 7):
        t = 2.0 * r ** l
        assert oracle_mod.suffix_radius2(r, l) == pytest.approx(t * t, rel=1e-14)
