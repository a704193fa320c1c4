"""GPU parity of the lossy archive (Sec. 4: truncation of span points to B
bits, recency allocation across spans) against the oracle.

Codes and tail points must equal the oracle's bit for bit, and the decoded
symbols too -- damaged ones included: the GPU decodes a lossy point in the
paper's binary64 arithmetic, exactly as the oracle does."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from paper_2607_07144_gb300._binding import EINVAL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _streams(N, ns, n, seed):
    rng = np.random.default_rng(seed)
    return rng.integers(0, N, size=(ns, n)).astype(np.uint8 if N <= 256 else np.int16)


def _oracle(oracle_mod, ctx, pts_h, n, bits, keep):
    """Per stream: (packed words, tail points, decoded symbols) from the oracle."""
    out = []
    for p in pts_h:
        T = max(0, p.shape[0] - keep)
        words = oracle_mod.pack_codes(oracle_mod.truncate_codes(p[:T], bits), bits)
        sym = oracle_mod.lossy_decode(p, n, ctx.N, ctx.r, ctx.L, bits, keep)
        out.append((words, p[T:], sym))
    return out


CASES = [(3, 2, 0), (3, 33, 5), (16, 5, 3), (16, 24, 0), (256, 2, 0), (256, 12, 40), (256, 24, 7),
         (256, 32, 0), (256, 42, 0), (256, 53, 11), (1024, 16, 9), (1024, 30, 0), (1024, 53, 0)]


@pytest.mark.parametrize("N,bits,keep", CASES)
def test_codes_tail_and_decode_equal_oracle(fkv, oracle_mod, N, bits, keep):
    ctx = fkv.Context(N)
    L = ctx.L
    ns, n = 3, 300 * L + L // 2 + 1
    sym = _streams(N, ns, n, 100 * N + bits)
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    codes, tail = ctx.truncate(pts, n, bits, keep)
    dec = ctx.lossy_decode(codes, tail, n, bits, keep)
    assert ctx.sync_status() == 0
    T, words, ts = ctx.lossy_geometry(n, bits, keep)
    ph = pts.cpu().numpy()
    ch, th, dh = codes.cpu().numpy().view(np.uint32), tail.cpu().numpy(), dec.cpu().numpy()
    for i, (w, t, s) in enumerate(_oracle(oracle_mod, ctx, ph, n, bits, keep)):
        assert np.array_equal(ch[i, :words], w)
        assert np.array_equal(th[i, :ts].view(np.uint64), t.view(np.uint64))
        assert np.array_equal(dh[i].astype(np.int32), s)
    if bits == 53:
        assert np.array_equal(dh, sym)                     # full precision: lossless


@pytest.mark.parametrize("N", [4, 256])
def test_adversarial_and_tiny_budgets(fkv, oracle_mod, N):
    """Spans of one repeated symbol (points next to a vertex) and alternating
    neighbours, at budgets down to 2 bits: the damaged walks leave the unit
    disk by factors of 1/r per step and exercise every branch of the cell test."""
    ctx = fkv.Context(N)
    L = ctx.L
    rows = []
    for c in range(N):
        rows.append(np.full(L, c))
        rows.append(np.resize([c, (c + 1) % N], L))
        rows.append(np.concatenate([[c], np.full(L - 1, (c + N - 1) % N)]))
    sym = np.concatenate(rows).astype(np.uint8)[None, :]
    n = sym.shape[1]
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    for bits in (2, 3, 7, 20, 40):
        codes, tail = ctx.truncate(pts, n, bits, 0)
        dec = ctx.lossy_decode(codes, tail, n, bits, 0).cpu().numpy()
        want = oracle_mod.lossy_decode(pts[0].cpu().numpy(), n, N, ctx.r, L, bits, 0)
        assert np.array_equal(dec[0].astype(np.int32), want), bits


def test_strided_buffers_and_reads(fkv, oracle_mod):
    N, bits, keep = 256, 21, 13
    ctx = fkv.Context(N)
    L = ctx.L
    ns, n = 4, 2000 * L + 5
    sym = _streams(N, ns, n, 5)
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    T, words, ts = ctx.lossy_geometry(n, bits, keep)
    codes = torch.full((ns, words + 9), -1, dtype=torch.int32, device="cuda")
    tail = torch.full((ns, ts + 3, 2), 7.0, dtype=torch.float64, device="cuda")
    ctx.truncate(pts, n, bits, keep, codes=codes[:, :words + 5], tail=tail[:, :ts + 1])
    assert torch.all(codes[:, words + 5:] == -1) and torch.all(tail[:, ts + 1:] == 7.0)
    full = ctx.lossy_decode(codes[:, :words + 5], tail[:, :ts + 1], n, bits, keep)
    ph = pts.cpu().numpy()
    for i in range(ns):
        assert np.array_equal(full[i].cpu().numpy().astype(np.int32),
                              oracle_mod.lossy_decode(ph[i], n, N, ctx.r, L, bits, keep))
    rng = np.random.default_rng(3)
    req = np.stack([rng.integers(0, ns, 30000), rng.integers(0, n, 30000)], axis=1)
    req[:ns, 1] = n - 1
    got = ctx.lossy_read(codes[:, :words + 5], tail[:, :ts + 1], n, bits, keep, torch.from_numpy(req).cuda())
    assert torch.equal(got, full[torch.from_numpy(req[:, 0]).cuda(), torch.from_numpy(req[:, 1]).cuda()])
    bad = torch.tensor([[0, n], [ns, 0], [-1, 3]], dtype=torch.int64, device="cuda")
    out = ctx.lossy_read(codes[:, :words + 5], tail[:, :ts + 1], n, bits, keep, bad).cpu().numpy()
    assert np.all(out == 0xFF) and ctx.sync_status() == -2     # FKV_ERANGE


def test_bad_arguments_are_rejected(fkv):
    ctx = fkv.Context(256)
    lib = fkv.lib()
    pts = torch.zeros((1, 10, 2), dtype=torch.float64, device="cuda")
    codes = torch.zeros((1, 64), dtype=torch.int32, device="cuda")
    tail = torch.zeros((1, 10, 2), dtype=torch.float64, device="cuda")
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    for bits in (1, 54):
        assert lib.fkv_truncate(ctx.handle, P(pts), 1, 60, 10, bits, 0, P(codes), 64, P(tail), 10, None) == EINVAL
    # 10 spans x 2 codes x 24 bits = 15 words: a stride of 14 is short
    assert lib.fkv_truncate(ctx.handle, P(pts), 1, 60, 10, 24, 0, P(codes), 14, P(tail), 10, None) == EINVAL
    assert lib.fkv_lossy_decode(ctx.handle, P(codes), 64, None, 0, 1, 60, 24, 3, P(codes), 60, None) == EINVAL
    assert lib.fkv_truncate(ctx.handle, P(pts), 1, 60, 10, 24, 0, P(codes), 15, None, 0, None) == 0
    assert ctx.sync_status() == 0


def test_gpt2_archive_full_size(fkv, oracle_mod):
    """The GPT-2 archive's 96 streams of 989 records x 72 symbols at 24 bits
    per coordinate, the last 64 records exact: codes of every stream, the
    decode of sampled streams against the oracle, the error profile."""
    N = 256
    ctx = fkv.Context(N)
    L = ctx.L
    ns, n = 96, 989 * 72
    sym = synth.gpu_symbols(N, "uniform", ns, n)
    pts = ctx.span_encode(sym)
    bits, keep = 24, 64 * 72 // L
    codes, tail = ctx.truncate(pts, n, bits, keep)
    dec = ctx.lossy_decode(codes, tail, n, bits, keep)
    assert ctx.sync_status() == 0
    T, words, ts = ctx.lossy_geometry(n, bits, keep)
    ph = pts.cpu().numpy()
    ch = codes.cpu().numpy().view(np.uint32)
    for i in range(ns):
        assert np.array_equal(ch[i, :words], oracle_mod.pack_codes(oracle_mod.truncate_codes(ph[i, :T], bits), bits))
    for i in (0, 47, 95):
        assert np.array_equal(dec[i].cpu().numpy().astype(np.int32),
                              oracle_mod.lossy_decode(ph[i], n, N, ctx.r, L, bits, keep))
    wrong = (dec != sym).cpu().numpy()
    assert not wrong[:, T * L:].any()                      # the recent spans are exact
    rate = wrong[:, :T * L].reshape(ns, T, L).mean(axis=(0, 1))
    assert rate[-1] < 0.01 and rate[0] > 0.9              # each span keeps its end, loses its start
