"""Pins for the oracle's lossy truncation (Sec. 4): the B-bit code of a
coordinate, the packed layout, the lossless limit at full precision, the
recency allocation across spans, and where the damage falls inside a span."""
import numpy as np
import pytest


def test_truncation_codes_by_hand(oracle_mod):
    # floor(x 2^(B-1)): -0.3 * 8 = -2.4 -> -3 (value -0.375); 0.3 * 8 = 2.4 -> 2 (0.25)
    c = oracle_mod.truncate_codes(np.array([[-0.3, 0.3], [-0.375, 0.999], [0.0, -1e-300]]), 4)
    assert c.tolist() == [[-3, 2], [-3, 7], [0, -1]]
    v = oracle_mod.truncated_points(c, 4)
    assert v.tolist() == [[-0.375, 0.25], [-0.375, 0.875], [0.0, -0.125]]
    # every truncated value is at most x and within 2^-(B-1) of it
    rng = np.random.default_rng(0)
    x = rng.uniform(-1, 1, size=(1000, 2))
    for b in (2, 9, 24, 40, 53):
        t = oracle_mod.truncated_points(oracle_mod.truncate_codes(x, b), b)
        assert np.all(t <= x) and np.all(x - t < 2.0 ** -(b - 1))
    with pytest.raises(ValueError):
        oracle_mod.truncate_codes(x, 1)


def test_packed_layout_by_hand(oracle_mod):
    # B = 3: fields 001, 110, 011, 100 laid out least significant bit first
    w = oracle_mod.pack_codes(np.array([[1, -2], [3, -4]]), 3)
    assert w.tolist() == [0b100011110001]


@pytest.mark.parametrize("bits", [2, 5, 16, 20, 31, 32, 33, 53])
def test_packed_layout_matches_big_integer(oracle_mod, bits):
    # the same layout written as one big integer: field i at bit i * B
    rng = np.random.default_rng(bits)
    codes = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(37, 2))
    big = 0
    for i, v in enumerate(codes.reshape(-1)):
        big |= (int(v) & ((1 << bits) - 1)) << (i * bits)
    nwords = (codes.size * bits + 31) // 32
    want = [(big >> (32 * j)) & 0xFFFFFFFF for j in range(nwords)]
    assert oracle_mod.pack_codes(codes, bits).tolist() == want


@pytest.mark.parametrize("N", [3, 16, 256, 1024])
def test_full_precision_is_lossless(oracle_mod, N):
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(N)
    sym = rng.integers(0, N, size=600 * L + 3).astype(np.int32)
    adv = np.concatenate([np.full(L, c) for c in range(min(N, 64))] +
                         [np.resize([c, (c + 1) % N], L) for c in range(min(N, 64))]).astype(np.int32)
    for s in (sym, adv):
        pts = oracle_mod.span_encode(s, N, r, L)
        for bits in (48, 53):
            assert np.array_equal(oracle_mod.lossy_decode(pts, s.size, N, r, L, bits, 0), s)


def test_recent_spans_stay_exact(oracle_mod):
    N = 256
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(7)
    n = 400 * L + 2
    sym = rng.integers(0, N, size=n).astype(np.int32)
    pts = oracle_mod.span_encode(sym, N, r, L)
    keep = 50
    got = oracle_mod.lossy_decode(pts, n, N, r, L, 2, keep)
    t = pts.shape[0] - keep
    assert np.array_equal(got[t * L:], sym[t * L:])            # the recent spans: exact
    assert np.mean(got[:t * L] != sym[:t * L]) > 0.5           # two bits per coordinate: mostly lost
    lp = oracle_mod.lossy_points(pts, 2, keep)
    assert np.array_equal(lp[t:], pts[t:]) and np.all(np.abs(lp[:t]) <= 1.0)


def test_damage_falls_on_each_span_start(oracle_mod):
    """Sec. 4: the bits dropped last describe the symbols coded first in this
    map's orientation (the stored point's coarsest bits hold a span's last
    symbol), so truncation damages the start of every span and leaves its end
    exact; the exact tail grows by about one symbol per log2(1/r) bits."""
    N = 256
    r = oracle_mod.packing_ratio(N)
    L = oracle_mod.max_span_len(r)
    rng = np.random.default_rng(11)
    n = 3000 * L
    sym = rng.integers(0, N, size=n).astype(np.int32)
    pts = oracle_mod.span_encode(sym, N, r, L)
    per_symbol = np.log2(1.0 / r)
    prev = None
    for bits in (12, 18, 24, 30, 36, 42):
        wrong = (oracle_mod.lossy_decode(pts, n, N, r, L, bits, 0) != sym).reshape(-1, L)
        rate = wrong.mean(axis=0)                             # error rate by in-span offset
        assert np.all(np.diff(rate) <= 1e-3)                  # damage concentrates at the span start
        exact_tail = np.array([L - (np.max(np.nonzero(w)[0]) + 1) if w.any() else L for w in wrong])
        # about (B - 1) / log2(1/r) trailing symbols survive; at least that many minus two
        assert np.mean(exact_tail >= min(L, int((bits - 1) / per_symbol) - 2)) > 0.99
        if prev is not None:
            assert exact_tail.mean() >= prev
        prev = exact_tail.mean()
