"""Pins for the oracle's probability-weighted maps (Sec. 6 eq. (1),
arithmetic coding): the uniform model's exact bit pattern, the lossless
round trip, and the code length against the model's cross-entropy."""
import numpy as np
import pytest


@pytest.mark.parametrize("k", [1, 2, 4, 8])
def test_uniform_power_of_two_is_plain_binary(oracle_mod, k):
    # p(c) = 1/N with N = 2^k: every step settles exactly k bits (the symbol,
    # most significant bit first); the end adds "01"
    N = 1 << k
    rng = np.random.default_rng(k)
    sym = rng.integers(0, N, size=300)
    words, nb = oracle_mod.ac_encode(sym, N, adaptive=False)
    bits = "".join(format(int(c), "0%db" % k) for c in sym) + "01"
    assert nb == len(bits)
    got = "".join(format(int(w), "032b") for w in words)[:nb]
    assert got == bits


@pytest.mark.parametrize("N", [2, 3, 16, 70, 256, 1024])
@pytest.mark.parametrize("adaptive", [True, False])
def test_round_trip(oracle_mod, N, adaptive):
    rng = np.random.default_rng(N)
    streams = [rng.integers(0, N, size=2000),
               np.minimum(rng.zipf(1.3, size=2000) - 1, N - 1),
               np.full(1500, N - 1), np.zeros(1, np.int64), np.zeros(0, np.int64),
               np.resize(np.arange(N), 3000)]
    for s in streams:
        words, nb = oracle_mod.ac_encode(s, N, adaptive)
        assert np.array_equal(oracle_mod.ac_decode(words, nb, s.size, N, adaptive), s)


@pytest.mark.parametrize("N", [3, 16, 256])
def test_code_length_is_the_model_cross_entropy(oracle_mod, N):
    # Sec. 6: the code length of a string is -sum log2 p(c_k); 32-bit interval
    # arithmetic adds at most the two final bits and a vanishing rounding term
    rng = np.random.default_rng(3 * N)
    for s in (rng.integers(0, N, size=4000), np.minimum(rng.zipf(1.2, size=4000) - 1, N - 1),
              np.full(4000, 1)):
        for adaptive in (True, False):
            _, nb = oracle_mod.ac_encode(s, N, adaptive)
            h = oracle_mod.ac_model_bits(s, N, adaptive)
            assert h - 1e-6 <= nb <= h + 2 + s.size * 2.0 ** -16, (adaptive, nb, h)
    # the uniform code spends log2 N bits per symbol whatever the data
    s = np.full(4000, 0)
    _, nb = oracle_mod.ac_encode(s, N, adaptive=False)
    assert abs(nb - 4000 * np.log2(N)) <= 2
    _, nb_ad = oracle_mod.ac_encode(s, N, adaptive=True)
    assert nb_ad < 0.05 * nb                             # a constant stream costs little adaptively
