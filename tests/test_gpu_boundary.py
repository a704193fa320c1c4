"""Spans that drive the decoder to its smallest decision margins (Sec. 1:
the inverse map classifies the cell holding the point; points built by
alternating neighbouring vertices sit closest to the boundary between their
Voronoi sectors, about r^(m-1) (1 - cos(2 pi / N)) (1 - 2 r) away in the
decoder's scaled coordinates).  At every alphabet size, the stored points of
such spans must equal the oracle's bit for bit, and decoding them, whole or
by random access, must return the input exactly."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _adversarial(N, L, seed):
    rng = np.random.default_rng(seed)
    pats = []
    for c in sorted({0, 1, N // 4, N // 3, N // 2, N - 2, N - 1}):
        a, b, z = c % N, (c + 1) % N, (c - 1) % N
        pats += [[a] * L, [a, b] * L, [a, z] * L, [b] + [a] * (L - 1), [a] + [b] * (L - 1),
                 [a, (a + N // 2) % N] * L, [a, a, b, b] * L]
    streams = []
    for p in pats:
        s = np.array(p[:L], np.int64)
        streams.append(s)
    # every cut of the alternating pattern (tails of every length)
    for m in range(1, L + 1):
        streams.append(np.array(([0, 1] * L)[:m], np.int64))
    return streams


@pytest.mark.parametrize("N", [3, 4, 5, 7, 8, 9, 16, 64, 255, 256, 257, 1000, 1024])
def test_boundary_spans_round_trip_bit_exact(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    L = ctx.L
    spans = _adversarial(N, L, N)
    flat = np.concatenate(spans)
    np_t = np.uint8 if ctx.sym_bytes == 1 else np.int16
    so, po = ctx.ragged_offsets([len(s) for s in spans])
    d = torch.from_numpy(flat.astype(np_t)).cuda()
    pts = ctx.span_encode_ragged(d, so, po)
    dec = ctx.span_decode_ragged(pts, po, so)
    assert ctx.sync_status() == 0
    assert np.array_equal(dec.cpu().numpy()[:flat.size].astype(np.int64) & 0xFFFF, flat)
    ph = pts.cpu().numpy()
    pob = po.cpu().numpy()
    for i, s in enumerate(spans):
        want = oracle_mod.span_encode(s.astype(np.int32), N, ctx.r, L)
        assert np.array_equal(ph[pob[i]:pob[i + 1]].view(np.uint64), want.view(np.uint64))
        sym, anchor, bad = oracle_mod.span_decode(want, len(s), N, ctx.r, L)
        assert bad == 0 and np.array_equal(sym, s)
    req = np.array([(i, p) for i, s in enumerate(spans) for p in range(len(s))], np.int64)
    got = ctx.read_ragged(pts, po, so, torch.from_numpy(req).cuda()).cpu().numpy().astype(np.int64) & 0xFFFF
    assert ctx.sync_status() == 0
    assert np.array_equal(got, flat)
