"""GPU parity of the span codec (Sec. 1 "The code", Sec. 2) against the oracle.

Stored points must equal the oracle's bit for bit; decoded symbols, random
reads and appends must equal the input stream and the oracle exactly."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

NS = [3, 4, 5, 16, 64, 256]


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _ctx(fkv, N, L=None):
    return fkv.Context(N, span_len=L)


def _rand_streams(N, ns, n, seed):
    rng = np.random.default_rng(seed)
    return rng.integers(0, N, size=(ns, n)).astype(np.uint8)


def _oracle_points(oracle_mod, sym, N, r, L):
    return np.stack([oracle_mod.span_encode(s, N, r, L) for s in sym])


@pytest.mark.parametrize("N", NS)
def test_vertex_table_equals_oracle(fkv, oracle_mod, N):
    ctx = _ctx(fkv, N)
    assert np.array_equal(ctx.vertices(), oracle_mod.vertices(N))
    assert ctx.r == oracle_mod.packing_ratio(N) and ctx.L == oracle_mod.max_span_len(ctx.r)


@pytest.mark.parametrize("N", NS)
def test_encode_bit_exact_and_decode_round_trip(fkv, oracle_mod, N):
    ctx = _ctx(fkv, N)
    L = ctx.L
    n = 300 * L + (L // 2 + 1 if L > 1 else 0)      # several blocks and a ragged tail
    sym = _rand_streams(N, 5, n, N)
    d_sym = torch.from_numpy(sym).cuda()
    pts = ctx.span_encode(d_sym)
    want = _oracle_points(oracle_mod, sym, N, ctx.r, L)
    got = pts.cpu().numpy()
    assert got.shape == want.shape
    assert np.array_equal(got.view(np.uint64), want.view(np.uint64))
    dec = ctx.span_decode(pts, n)
    assert ctx.sync_status() == 0
    assert np.array_equal(dec.cpu().numpy(), sym)
    o_dec, _, bad = oracle_mod.span_decode(want[0], n, N, ctx.r, L)
    assert bad == 0 and np.array_equal(o_dec, sym[0])


@pytest.mark.parametrize("N", [3, 4, 16, 256])
def test_every_span_length_and_tail(fkv, oracle_mod, N):
    r = oracle_mod.packing_ratio(N)
    for L in range(1, oracle_mod.max_span_len(r) + 1, 3):
        ctx = fkv.Context(N, span_len=L)
        for n in [1, L - 1, L, L + 1, 257 * L + 3]:
            if n <= 0:
                continue
            sym = _rand_streams(N, 2, n, 1000 * N + L + n)
            pts = ctx.span_encode(torch.from_numpy(sym).cuda())
            want = _oracle_points(oracle_mod, sym, N, r, L)
            assert np.array_equal(pts.cpu().numpy().view(np.uint64), want.view(np.uint64)), (L, n)
            assert np.array_equal(ctx.span_decode(pts, n).cpu().numpy(), sym), (L, n)


@pytest.mark.parametrize("N", [3, 4, 5, 8, 16, 64, 256])
def test_adversarial_streams(fkv, oracle_mod, N):
    ctx = _ctx(fkv, N)
    L = ctx.L
    rows = []
    for c in range(N):
        rows.append(np.full(L, c))
        rows.append(np.resize([c, (c + 1) % N], L))
        rows.append(np.concatenate([[c], np.full(L - 1, (c + 1) % N)]))
    sym = np.concatenate(rows).astype(np.uint8)[None, :]
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    want = _oracle_points(oracle_mod, sym, N, ctx.r, L)
    assert np.array_equal(pts.cpu().numpy().view(np.uint64), want.view(np.uint64))
    assert np.array_equal(ctx.span_decode(pts, sym.shape[1]).cpu().numpy(), sym)
    assert ctx.sync_status() == 0


def test_unaligned_and_strided_buffers(fkv, oracle_mod):
    N = 256
    ctx = _ctx(fkv, N)
    L = ctx.L
    n = 1000
    base = torch.from_numpy(_rand_streams(N, 3, n + 40, 7)).cuda()
    for off in [1, 3, 7, 15, 16]:
        view = base[:, off:off + n]                 # misaligned start, row stride n + 40
        pts = ctx.span_encode(view)
        want = _oracle_points(oracle_mod, view.cpu().numpy(), N, ctx.r, L)
        assert np.array_equal(pts.cpu().numpy().view(np.uint64), want.view(np.uint64))
        out = torch.full((3, n + 40), 0xAB, dtype=torch.uint8, device="cuda")
        ctx.span_decode(pts, n, sym=out[:, off:off + n])
        o = out.cpu().numpy()
        assert np.array_equal(o[:, off:off + n], view.cpu().numpy())
        assert np.all(o[:, :off] == 0xAB) and np.all(o[:, off + n:] == 0xAB)   # nothing outside touched


def test_empty_and_degenerate(fkv):
    ctx = _ctx(fkv, 16)
    e = torch.empty((0, 10), dtype=torch.uint8, device="cuda")
    assert ctx.span_encode(e).shape == (0, ctx.n_spans(10), 2)
    z = torch.empty((2, 0), dtype=torch.uint8, device="cuda")
    assert ctx.span_encode(z).numel() == 0
    assert ctx.span_decode(torch.empty((2, 0, 2), dtype=torch.float64, device="cuda"), 0).numel() == 0
    assert ctx.sync_status() == 0


def test_symbol_outside_alphabet_is_reported(fkv):
    ctx = _ctx(fkv, 5)
    sym = torch.tensor([[0, 1, 2, 7, 4, 0, 1]], dtype=torch.uint8, device="cuda")
    pts = ctx.span_encode(sym)
    assert ctx.sync_status() == -5
    assert np.isnan(pts.cpu().numpy()[0, 0, 0])
    assert ctx.sync_status() == 0          # the status word was cleared


def test_corrupt_point_fails_anchor_check(fkv):
    ctx = _ctx(fkv, 256)
    sym = torch.from_numpy(_rand_streams(256, 1, 600, 9)).cuda()
    pts = ctx.span_encode(sym)
    ctx.span_decode(pts, 600)
    assert ctx.sync_status() == 0
    bits = pts.view(torch.int64).clone()
    bits[0, 17, 0] ^= (1 << 40)
    ctx.span_decode(bits.view(torch.float64), 600)
    assert ctx.sync_status() == -5


@pytest.mark.parametrize("N", [3, 4, 16, 256])
def test_random_read_equals_full_decode(fkv, oracle_mod, N):
    ctx = _ctx(fkv, N)
    ns, n = 4, 5000 + 3
    sym = _rand_streams(N, ns, n, 11 + N)
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    rng = np.random.default_rng(N)
    req = np.stack([rng.integers(0, ns, 20000), rng.integers(0, n, 20000)], axis=1)
    req[:ns, 1] = n - 1                                   # last symbol of every stream
    req[ns:2 * ns, 1] = 0
    got = ctx.read(pts, n, torch.from_numpy(req).cuda()).cpu().numpy()
    assert np.array_equal(got, sym[req[:, 0], req[:, 1]])
    p0 = pts[0].cpu().numpy()
    sel = req[:, 0] == 0
    assert np.array_equal(got[sel], oracle_mod.read(p0, n, req[sel, 1], N, ctx.r, ctx.L))
    bad = torch.tensor([[0, n], [ns, 0], [-1, 0]], dtype=torch.int64, device="cuda")
    out = ctx.read(pts, n, bad).cpu().numpy()
    assert np.all(out == 0xFF) and ctx.sync_status() == -2     # FKV_ERANGE


@pytest.mark.parametrize("N", [3, 16, 256])
def test_append_equals_scratch_encode(fkv, oracle_mod, N):
    ctx = _ctx(fkv, N)
    L = ctx.L
    ns = 3
    st = fkv.Streams(ctx, ns, capacity=5)
    rng = np.random.default_rng(N)
    full = np.zeros((ns, 0), np.uint8)
    for m in [1, L - 1, L, 1, 3 * L + 2, 2, 50 * L + 1]:
        if m <= 0:
            continue
        new = rng.integers(0, N, size=(ns, m)).astype(np.uint8)
        st.append(torch.from_numpy(new).cuda())
        full = np.concatenate([full, new], axis=1)
        assert st.length == full.shape[1]
        got = st.export()
        want = _oracle_points(oracle_mod, full, N, ctx.r, L)
        assert np.array_equal(got.view(np.uint64), want.view(np.uint64)), m
    ns_, ln, stride, _ = st.info()
    dec = ctx.span_decode(st.points(), ln)
    assert np.array_equal(dec.cpu().numpy(), full)
    # checkpoint round trip: export -> import is bit-identical
    st2 = fkv.Streams.import_(ctx, ln, got)
    assert np.array_equal(st2.export().view(np.uint64), got.view(np.uint64))
    assert ctx.sync_status() == 0


# ----------------------------------------------------------- full size --
CFG2 = [(3, "uniform"), (4, "zipf"), (16, "uniform"), (16, "zipf"), (256, "uniform"), (256, "zipf"),
        (3, "zipf"), (4, "uniform")]


@pytest.mark.parametrize("N,dist", CFG2)
def test_symbol_codec_stress_full_size(fkv, oracle_mod, N, dist):
    """Four streams of 2^28 seeded symbols: encode, full decode and 2^20
    random reads per stream; points checked bit-exact on sampled spans."""
    ctx = _ctx(fkv, N)
    L = ctx.L
    ns, n = 4, 1 << 28
    sym = synth.gpu_symbols(N, dist, ns, n)
    pts = ctx.span_encode(sym)
    dec = ctx.span_decode(pts, n)
    assert ctx.sync_status() == 0
    assert torch.equal(dec, sym)
    del dec
    spans = pts.shape[1]
    rng = np.random.default_rng(N)
    for s in range(ns):
        pick = np.unique(np.concatenate([rng.integers(0, spans, 2000), [0, spans - 1]]))
        for u in pick[:200]:
            b, e = u * L, min(n, (u + 1) * L)
            host = synth.symbols(N, dist, s, np.arange(b, e))
            assert np.array_equal(host, sym[s, b:e].cpu().numpy())       # generator twin
            want = oracle_mod.span_encode(host.astype(np.int32), N, ctx.r, L)[0]
            got = pts[s, u].cpu().numpy()
            assert np.array_equal(got.view(np.uint64), want.view(np.uint64))
    # 2^20 random reads per stream
    reads = 1 << 20
    req = torch.stack([torch.arange(ns, device="cuda").repeat_interleave(reads),
                       torch.cat([synth.gpu_positions(n, reads, s) for s in range(ns)])], dim=1)
    got = ctx.read(pts, n, req)
    assert torch.equal(got, sym[req[:, 0], req[:, 1]])
    assert ctx.sync_status() == 0
