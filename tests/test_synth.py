"""The seeded input generators (shared by the oracle side and the CUDA side)."""
import numpy as np
import pytest

import synth


def test_philox_known_answers():
    # Known-answer vectors of Philox4x32-10 (Salmon et al., SC'11; Random123).
    kat = [
        ((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
        ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
        ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
         (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1)),
    ]
    for ctr, key, want in kat:
        got = synth.philox4x32(*ctr, *key)
        assert tuple(int(g) for g in got) == want


def test_irwin_hall_moments():
    z = synth.irwin_hall(np.arange(400000), synth.TID_K, 0).astype(np.float64)
    z /= synth.IRWIN_HALL_STD
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1) < 0.01
    assert np.abs(z).max() < 4.9


def test_kv_elements_match_whole_cache():
    cfg = synth.small_config(synth.CFG1, 101, n_layers=2, batch=2, seq=40, n_heads=3)
    whole = synth.kv_cache(cfg, 0)
    assert whole.dtype == np.float16 and whole.shape == cfg.cache_shape()
    got = synth.kv_elements(cfg, 0, [1, 0], [1, 1], [2, 0], [39, 5])
    assert np.array_equal(got[0], whole[1, 1, 2, 39]) and np.array_equal(got[1], whole[0, 1, 0, 5])


def test_outlier_key_channels():
    cfg = synth.CFG0
    sig = synth.channel_sigma(cfg, 0)
    assert sig.shape == (1, 12, 64)
    assert np.all((sig == 1.0).sum(-1) == 60) and np.all((sig == 8.0).sum(-1) == 4)
    assert np.all(synth.channel_sigma(cfg, 1) == 1.0)
    l3 = synth.channel_sigma(synth.small_config(synth.CFG3, 103, 2, 1, 64), 0)
    assert l3.shape == (2, 8, 128)


def test_bf16_rounding_bits():
    x = np.array([1.0, 1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, -2.5], np.float32)
    b = synth.round_f32_to(x, "bf16")
    assert list(synth.bf16_bits_to_f32(b)) == [1.0, 1.0, 1 + 2.0 ** -6, -2.5]


@pytest.mark.parametrize("N", [3, 4, 16, 256])
def test_symbol_streams(N):
    u = synth.symbols(N, "uniform", 0, np.arange(200000))
    z = synth.symbols(N, "zipf", 0, np.arange(200000))
    assert u.max() < N and z.max() < N
    cu = np.bincount(u, minlength=N)
    assert cu.min() > 0.8 * 200000 / N
    cz = np.bincount(z, minlength=N)
    assert cz[0] == cz.max()                      # symbol 0 most frequent
    w = np.arange(1, N + 1) ** -1.1
    assert abs(cz[0] / 200000 - w[0] / w.sum()) < 0.01


def test_codebooks_shape_and_shrink():
    cb = synth.codebooks(synth.CFG0, 0)
    assert cb.shape == (1, 12, 2, 256, 64) and cb.dtype == np.float32
    s0 = cb[:, :, 0].std()
    s1 = cb[:, :, 1].std()
    assert abs(s1 / s0 - synth.STAGE_SHRINK) < 0.05
