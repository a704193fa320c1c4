"""GPU parity of the probability-weighted maps (Sec. 6 eq. (1), arithmetic
coding of independent streams) against the oracle: code words and bit counts
bit for bit, lossless decode."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _dt(N):
    return np.uint8 if N <= 256 else np.int16


def _check(oracle_mod, ctx, sym, adaptive):
    words, nbits = ctx.ac_encode(torch.from_numpy(sym).cuda(), adaptive)
    dec = ctx.ac_decode(words, nbits, sym.shape[1], adaptive)
    assert ctx.sync_status() == 0
    wh = words.cpu().numpy().view(np.uint32)
    nb = nbits.cpu().numpy()
    for i, s in enumerate(sym):
        ow, onb = oracle_mod.ac_encode(s.astype(np.int32), ctx.N, adaptive)
        assert nb[i] == onb
        assert np.array_equal(wh[i, :ow.size], ow)
    assert np.array_equal(dec.cpu().numpy(), sym)
    return nb


@pytest.mark.parametrize("N", [3, 16, 70, 256, 300, 1024])
@pytest.mark.parametrize("adaptive", [True, False])
def test_random_and_skewed_streams(fkv, oracle_mod, N, adaptive):
    ctx = fkv.Context(N)
    rng = np.random.default_rng(N + 7 * adaptive)
    n = 3001
    sym = np.stack([rng.integers(0, N, n), np.minimum(rng.zipf(1.3, n) - 1, N - 1),
                    np.full(n, N - 1), np.resize(np.arange(N), n)]).astype(_dt(N))
    nb = _check(oracle_mod, ctx, sym, adaptive)
    if not adaptive:
        assert np.all(np.abs(nb - n * np.log2(N)) <= 2)       # the uniform code: log2 N bits per symbol


@pytest.mark.parametrize("n", [0, 1, 2, 31, 32, 33, 1000])
def test_short_streams(fkv, oracle_mod, n):
    ctx = fkv.Context(256)
    rng = np.random.default_rng(n)
    sym = rng.integers(0, 256, size=(5, n)).astype(np.uint8)
    for adaptive in (True, False):
        if n == 0:
            words, nbits = ctx.ac_encode(torch.from_numpy(sym).cuda(), adaptive)
            assert nbits.cpu().tolist() == [2] * 5
            continue
        _check(oracle_mod, ctx, sym, adaptive)


def test_bad_symbols_and_bits_are_reported(fkv):
    ctx = fkv.Context(10)
    sym = torch.tensor([[1, 2, 12, 3]], dtype=torch.uint8, device="cuda")
    ctx.ac_encode(sym)
    assert ctx.sync_status() == -5
    rng = np.random.default_rng(1)
    words = torch.from_numpy(rng.integers(-2 ** 31, 2 ** 31, size=(3, 64)).astype(np.int32)).cuda()
    nbits = torch.tensor([2048, 100, 5], dtype=torch.int64, device="cuda")
    out = ctx.ac_decode(words, nbits, 5000)                   # garbage bits: decodes, never hangs
    torch.cuda.synchronize()
    assert int(out.max()) < 10
    ctx.sync_status()


def test_archive_streams_full_size(fkv, oracle_mod):
    """The GPT-2 archive's 96 streams of 989 records x 72 symbols (Zipf and
    uniform symbols): every stream round trips; three against the oracle."""
    ctx = fkv.Context(256)
    ns, n = 96, 989 * 72
    for dist in ("zipf", "uniform"):
        sym = synth.gpu_symbols(256, dist, ns, n)
        words, nbits = ctx.ac_encode(sym)
        dec = ctx.ac_decode(words, nbits, n)
        assert ctx.sync_status() == 0
        assert torch.equal(dec, sym)
        sh = sym.cpu().numpy()
        wh = words.cpu().numpy().view(np.uint32)
        nb = nbits.cpu().numpy()
        for i in (0, 50, 95):
            ow, onb = oracle_mod.ac_encode(sh[i].astype(np.int32), 256, True)
            assert nb[i] == onb and np.array_equal(wh[i, :ow.size], ow)
        # the rate approaches the source entropy (plus the add-one model's
        # learning cost, about (N - 1) log2(n) / (2 n) bits per symbol)
        w = np.arange(1, 257, dtype=np.float64) ** -1.1
        p = w / w.sum()
        H = float(-(p * np.log2(p)).sum()) if dist == "zipf" else 8.0
        rate = nb.sum() / (ns * n)
        assert H - 0.02 < rate < H + 0.05, (dist, rate, H)
