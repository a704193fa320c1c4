"""Pins for the oracle's residual VQ and archive bookkeeping (Sec. 3 "Setup").

Checked against a brute-force numpy search written here, planted structure,
exact special cases, the paper's storage identities, and the
round-to-nearest-even casts.
"""
import numpy as np
import pytest
import torch


def _bruteforce_rvq(x, cb):
    res = np.asarray(x, np.float64).copy()
    idx = []
    for C in np.asarray(cb, np.float64):
        d = ((res[:, None, :] - C[None, :, :]) ** 2).sum(-1)
        j = d.argmin(axis=1)                       # numpy: first minimum = lowest index
        idx.append(j)
        res -= C[j]
    return np.stack(idx, axis=1)


def test_matches_bruteforce(oracle_mod):
    rng = np.random.default_rng(0)
    for D, S in [(8, 1), (16, 3), (64, 4), (128, 2)]:
        x = rng.normal(size=(300, D))
        cb = (rng.normal(size=(S, 256, D)) * 0.8 ** np.arange(S)[:, None, None]).astype(np.float32)
        idx, gap = oracle_mod.rvq_encode(x, cb)
        assert np.array_equal(idx, _bruteforce_rvq(x, cb))
        assert np.all(gap >= 0)


def test_matches_bruteforce_1024_codewords(oracle_mod):
    # Table 2's k = 1024 rows: the same nearest-codeword search over 1024 entries
    rng = np.random.default_rng(5)
    for D, S in [(64, 1), (64, 2)]:
        x = rng.normal(size=(200, D))
        cb = (rng.normal(size=(S, 1024, D)) * 0.8 ** np.arange(S)[:, None, None]).astype(np.float32)
        idx, gap = oracle_mod.rvq_encode(x, cb)
        assert np.array_equal(idx, _bruteforce_rvq(x, cb))
        assert idx.max() >= 768                    # the upper codewords are reachable
    cb = rng.normal(size=(1, 1024, 16)).astype(np.float32)
    cb[0, 1000] = cb[0, 3]                         # a tie across the 256-codeword blocks
    idx, gap = oracle_mod.rvq_encode(cb[0, [3, 1000]].astype(np.float64), cb)
    assert list(idx[:, 0]) == [3, 3] and np.all(gap[:, 0] == 0.0)


def test_storage_identities_k1024():
    # Table 2: one pooled k = 1024 codebook per layer; 12 heads x (K, V) x 2
    # stages of 10-bit symbols per layer and token, five symbols per double.
    import synth
    c = synth.CFG5
    assert c.record_len == 48 and c.pooled and c.N == 1024
    cb = synth.codebooks(synth.small_config(c, 905, n_layers=2, batch=1, seq=40), 0)
    assert cb.shape == (2, 1, 2, 1024, 64)


def test_codeword_equal_to_input(oracle_mod):
    rng = np.random.default_rng(1)
    cb = rng.normal(size=(1, 256, 64)).astype(np.float32)
    pick = rng.integers(0, 256, size=50)
    x = cb[0, pick].astype(np.float64)
    idx, gap = oracle_mod.rvq_encode(x, cb)
    assert np.array_equal(idx[:, 0], pick)
    y = oracle_mod.rvq_decode(idx, cb)
    assert np.array_equal(y, x)                   # single stage: exactly C[idx]


def test_planted_two_stage(oracle_mod):
    rng = np.random.default_rng(2)
    c0 = rng.normal(size=(256, 32)).astype(np.float32)
    c1 = (0.01 * rng.normal(size=(256, 32))).astype(np.float32)
    a = rng.integers(0, 256, size=200)
    b = rng.integers(0, 256, size=200)
    x = c0[a].astype(np.float64) + c1[b].astype(np.float64)
    idx, _ = oracle_mod.rvq_encode(x, np.stack([c0, c1]))
    assert np.array_equal(idx[:, 0], a) and np.array_equal(idx[:, 1], b)
    y = oracle_mod.rvq_decode(idx, np.stack([c0, c1]))
    assert np.array_equal(y, x)


def test_ties_take_the_lowest_index(oracle_mod):
    rng = np.random.default_rng(3)
    cb = rng.normal(size=(1, 256, 16)).astype(np.float32)
    cb[0, 200] = cb[0, 7]
    idx, gap = oracle_mod.rvq_encode(cb[0, [7, 200]].astype(np.float64), cb)
    assert list(idx[:, 0]) == [7, 7]
    assert np.all(gap[:, 0] == 0.0)


def test_reconstruction_is_the_centroid_sum(oracle_mod):
    rng = np.random.default_rng(4)
    cb = rng.normal(size=(4, 256, 64)).astype(np.float32)
    idx = rng.integers(0, 256, size=(100, 4)).astype(np.int32)
    y = oracle_mod.rvq_decode(idx, cb)
    want = sum(cb[s, idx[:, s]].astype(np.float64) for s in range(4))
    assert np.max(np.abs(y - want)) == 0.0


def test_storage_identities():
    # Sec. 3: the fp16 GPT-2 cache is 2 x 12 x 12 x 64 values = 36,864 B/token,
    # and 288 per-head codebooks of 2 stages x 256 x 64 float32 are 36 MB.
    import synth
    c = synth.CFG1
    assert 2 * c.n_layers * c.n_heads * c.dim * 2 == 36864
    assert 2 * c.n_layers * c.n_heads * 2 * 256 * c.dim * 4 == 36 * 2 ** 20
    assert 2 * c.n_layers * c.n_heads == 288


def test_exact_window(oracle_mod):
    # Sec. 3: 4 sinks + 32 recent stay exact; at 1024 tokens 988 are archived.
    pos = oracle_mod.archived_positions(1024)
    assert pos.start == 4 and pos.stop == 992 and len(pos) == 988
    assert len(oracle_mod.archived_positions(32768)) == 32732
    assert len(oracle_mod.archived_positions(36)) == 0


def test_record_order_round_trip(oracle_mod):
    rng = np.random.default_rng(5)
    H, P, SK, SV = 12, 9, 4, 2
    k = rng.integers(0, 256, size=(H, P, SK))
    v = rng.integers(0, 256, size=(H, P, SV))
    s = oracle_mod.records_from_indices(k, v)
    assert s.size == P * oracle_mod.record_len(H, SK, SV) == P * 72
    # position-major; within a record K of head 0..H-1 (stages inner) then V
    assert list(s[:SK]) == list(k[0, 0]) and list(s[SK:2 * SK]) == list(k[1, 0])
    assert list(s[H * SK:H * SK + SV]) == list(v[0, 0])
    k2, v2 = oracle_mod.indices_from_records(s, H, SK, SV)
    assert np.array_equal(k2, k) and np.array_equal(v2, v)


def test_round_to_nearest_even(oracle_mod):
    rng = np.random.default_rng(6)
    x32 = (rng.normal(size=20000) * 10.0 ** rng.integers(-3, 4, size=20000)).astype(np.float32)
    got = oracle_mod.round_to(x32.astype(np.float64), "bf16")
    want = torch.from_numpy(x32).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(got, want)
    # ties to even from float64 (no double rounding through float32)
    assert oracle_mod.round_to(np.array([1 + 2.0 ** -8]), "bf16")[0] == 1.0
    assert oracle_mod.round_to(np.array([1 + 3 * 2.0 ** -8]), "bf16")[0] == 1 + 2.0 ** -6
    assert oracle_mod.round_to(np.array([1 + 2.0 ** -8 + 2.0 ** -40]), "bf16")[0] == 1 + 2.0 ** -7
    x64 = rng.normal(size=20000) * 100
    assert np.array_equal(oracle_mod.round_to(x64, "f16"),
                          torch.from_numpy(x64).to(torch.float16).to(torch.float64).numpy())
    assert oracle_mod.round_to(np.array([1 + 2.0 ** -11]), "f16")[0] == 1.0


def _bruteforce_gap(x, cb):
    """Per stage: (second-best - best squared distance) / ||stage residual||^2,
    from a numpy float64 search that keeps its own residual."""
    res = np.asarray(x, np.float64).copy()
    gaps = []
    for C in np.asarray(cb, np.float64):
        d = ((res[:, None, :] - C[None, :, :]) ** 2).sum(-1)
        part = np.partition(d, 1, axis=1)
        rn = (res * res).sum(1)
        gaps.append((part[:, 1] - part[:, 0]) / rn)
        res -= C[d.argmin(axis=1)]
    return np.stack(gaps, axis=1)


@pytest.mark.parametrize("D,S,K", [(8, 1, 256), (16, 3, 256), (64, 4, 256), (128, 2, 256), (64, 1, 1024),
                                   (64, 2, 1024)])
def test_gap_matches_bruteforce(oracle_mod, D, S, K):
    # the quantity the GPU parity criterion excuses mismatches on: the top-2
    # distance gap of each stage over that stage's residual norm
    rng = np.random.default_rng(10 + D + S + K)
    x = rng.normal(size=(150, D))
    cb = (rng.normal(size=(S, K, D)) * 0.8 ** np.arange(S)[:, None, None]).astype(np.float32)
    idx, gap = oracle_mod.rvq_encode(x, cb)
    want = _bruteforce_gap(x, cb)
    assert np.all(np.isfinite(gap))
    np.testing.assert_allclose(gap, want, rtol=1e-9, atol=1e-12)


def test_gap_is_normalised_by_the_stage_residual(oracle_mod):
    # stage 2 residuals are ~1e-3 of the input, so a gap divided by ||x||^2
    # (instead of the stage residual's norm) would be ~1e-6 of the right value
    rng = np.random.default_rng(11)
    c0 = (10.0 * rng.normal(size=(256, 32))).astype(np.float32)
    c1 = (0.01 * rng.normal(size=(256, 32))).astype(np.float32)
    a = rng.integers(0, 256, size=120)
    x = c0[a].astype(np.float64) + 0.01 * rng.normal(size=(120, 32))
    cb = np.stack([c0, c1])
    idx, gap = oracle_mod.rvq_encode(x, cb)
    want = _bruteforce_gap(x, cb)
    assert np.all(idx[:, 0] == a)
    np.testing.assert_allclose(gap, want, rtol=1e-9, atol=1e-12)
    assert np.median(gap[:, 1]) > 1e-2          # O(1) gaps at the small second stage


def test_gap_when_the_best_codeword_comes_first(oracle_mod):
    # the winner at index 0 leaves the second-best to the later candidates
    # only (the branch that tracks a runner-up below the current best)
    rng = np.random.default_rng(12)
    cb = rng.normal(size=(1, 256, 24)).astype(np.float32)
    x = cb[0, 0].astype(np.float64)[None, :] + 1e-3 * rng.normal(size=(40, 24))
    idx, gap = oracle_mod.rvq_encode(x, cb)
    assert np.all(idx[:, 0] == 0)
    np.testing.assert_allclose(gap, _bruteforce_gap(x, cb), rtol=1e-9, atol=1e-12)
    assert np.all(np.isfinite(gap)) and np.all(gap > 0)
