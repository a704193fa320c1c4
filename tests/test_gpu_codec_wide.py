"""GPU parity of the span codec with uint16 symbols: alphabets 256 < N <= 1024
(the k = 1024 codebooks of Sec. 3, Table 2) against the oracle.

The same bar as the uint8 codec: stored points bit for bit equal to the
oracle's, decoded symbols, random reads, appends and suffix matches exactly
equal to the input stream and the oracle."""
import ctypes

import numpy as np
import pytest
import torch

import synth
from paper_2607_07144_gb300._binding import EINVAL

pytestmark = pytest.mark.gpu

NS = [257, 300, 512, 1000, 1024]


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _rand(N, ns, n, seed):
    rng = np.random.default_rng(seed)
    return rng.integers(0, N, size=(ns, n)).astype(np.int16)


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _oracle_points(oracle_mod, sym, N, r, L):
    return np.stack([oracle_mod.span_encode(s.astype(np.int32), N, r, L) for s in sym])


def _bits(a):
    return np.ascontiguousarray(a).view(np.uint64)


@pytest.mark.parametrize("N", NS)
def test_context_geometry(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    assert ctx.sym_bytes == 2 and ctx.sym_dtype == torch.int16
    assert np.array_equal(ctx.vertices(), oracle_mod.vertices(N))
    assert ctx.r == oracle_mod.packing_ratio(N) and ctx.L == oracle_mod.max_span_len(ctx.r)


def test_table2_k1024_geometry(fkv):
    # Table 2 k = 1024 rows: r_1024 = 0.0030586 and five symbols per double
    ctx = fkv.Context(1024)
    assert abs(ctx.r - 0.0030586) < 5e-8 and ctx.L == 5


@pytest.mark.parametrize("N", NS)
def test_encode_bit_exact_and_decode_round_trip(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    L = ctx.L
    n = 600 * L + L // 2 + 1                  # several 256-span blocks and a ragged tail
    sym = _rand(N, 4, n, N)
    pts = ctx.span_encode(_dev(sym))
    want = _oracle_points(oracle_mod, sym, N, ctx.r, L)
    assert np.array_equal(_bits(pts.cpu().numpy()), _bits(want))
    dec = ctx.span_decode(pts, n)
    assert ctx.sync_status() == 0
    assert dec.dtype == torch.int16 and np.array_equal(dec.cpu().numpy(), sym)
    o_dec, _, bad = oracle_mod.span_decode(want[1], n, N, ctx.r, L)
    assert bad == 0 and np.array_equal(o_dec, sym[1])


@pytest.mark.parametrize("N", [300, 1024])
def test_every_span_length_and_tail(fkv, oracle_mod, N):
    r = oracle_mod.packing_ratio(N)
    for L in range(1, oracle_mod.max_span_len(r) + 1):
        ctx = fkv.Context(N, span_len=L)
        for n in [1, L - 1, L, L + 1, 257 * L + 3]:
            if n <= 0:
                continue
            sym = _rand(N, 2, n, 1000 * N + 10 * L + n)
            pts = ctx.span_encode(_dev(sym))
            want = _oracle_points(oracle_mod, sym, N, r, L)
            assert np.array_equal(_bits(pts.cpu().numpy()), _bits(want)), (L, n)
            assert np.array_equal(ctx.span_decode(pts, n).cpu().numpy(), sym), (L, n)


@pytest.mark.parametrize("N", [257, 512, 1024])
def test_adversarial_streams(fkv, oracle_mod, N):
    """Every symbol repeated, alternating with its neighbour, and one symbol
    followed by its neighbour: points on the cell boundaries' doorstep."""
    ctx = fkv.Context(N)
    L = ctx.L
    rows = []
    for c in range(N):
        rows.append(np.full(L, c))
        rows.append(np.resize([c, (c + 1) % N], L))
        rows.append(np.concatenate([[c], np.full(L - 1, (c + N - 1) % N)]))
    sym = np.concatenate(rows).astype(np.int16)[None, :]
    pts = ctx.span_encode(_dev(sym))
    want = _oracle_points(oracle_mod, sym, N, ctx.r, L)
    assert np.array_equal(_bits(pts.cpu().numpy()), _bits(want))
    assert np.array_equal(ctx.span_decode(pts, sym.shape[1]).cpu().numpy(), sym)
    assert ctx.sync_status() == 0


def test_unaligned_and_strided_buffers(fkv, oracle_mod):
    N = 1024
    ctx = fkv.Context(N)
    n = 1000
    base = _dev(_rand(N, 3, n + 40, 7))
    for off in [1, 3, 7, 8, 15]:                 # element offsets: 2..30 bytes
        view = base[:, off:off + n]
        pts = ctx.span_encode(view)
        want = _oracle_points(oracle_mod, view.cpu().numpy(), N, ctx.r, ctx.L)
        assert np.array_equal(_bits(pts.cpu().numpy()), _bits(want))
        out = torch.full((3, n + 40), 0x5AB, dtype=torch.int16, device="cuda")
        ctx.span_decode(pts, n, sym=out[:, off:off + n])
        o = out.cpu().numpy()
        assert np.array_equal(o[:, off:off + n], view.cpu().numpy())
        assert np.all(o[:, :off] == 0x5AB) and np.all(o[:, off + n:] == 0x5AB)


def test_width_and_alignment_are_checked(fkv):
    ctx = fkv.Context(1024)
    with pytest.raises(ValueError):
        ctx.span_encode(torch.zeros((1, 10), dtype=torch.uint8, device="cuda"))
    raw = torch.zeros(64, dtype=torch.uint8, device="cuda")
    pts = torch.zeros((1, 4, 2), dtype=torch.float64, device="cuda")
    lib = fkv.lib()
    odd = ctypes.c_void_p(raw.data_ptr() + 1)
    rc = lib.fkv_span_encode(ctx.handle, odd, 1, 10, 10, ctypes.c_void_p(pts.data_ptr()), 4, None)
    assert rc == EINVAL
    rc = lib.fkv_span_decode(ctx.handle, ctypes.c_void_p(pts.data_ptr()), 1, 10, 4, odd, 10, None)
    assert rc == EINVAL
    assert fkv.lib().fkv_symbol_bytes(ctx.handle) == 2 and fkv.Context(256).sym_bytes == 1


def test_symbol_outside_alphabet_is_reported(fkv):
    ctx = fkv.Context(1000)
    for bad in [1000, 1023, 1024, 0x7FFF, -1]:   # -1 is 0xFFFF as uint16
        sym = torch.tensor([[0, 1, 2, bad, 4, 0, 1]], dtype=torch.int16, device="cuda")
        pts = ctx.span_encode(sym)
        assert ctx.sync_status() == -5, bad
        assert np.isnan(pts.cpu().numpy()[0, 0, 0])
        assert ctx.sync_status() == 0


@pytest.mark.parametrize("N", [300, 1024])
def test_random_read_equals_full_decode(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    ns, n = 4, 5000 + 3
    sym = _rand(N, ns, n, 11 + N)
    pts = ctx.span_encode(_dev(sym))
    rng = np.random.default_rng(N)
    req = np.stack([rng.integers(0, ns, 20000), rng.integers(0, n, 20000)], axis=1)
    req[:ns, 1] = n - 1
    req[ns:2 * ns, 1] = 0
    got = ctx.read(pts, n, _dev(req)).cpu().numpy()
    assert np.array_equal(got, sym[req[:, 0], req[:, 1]])
    sel = req[:, 0] == 2
    assert np.array_equal(got[sel], oracle_mod.read(pts[2].cpu().numpy(), n, req[sel, 1], N, ctx.r, ctx.L))
    bad = torch.tensor([[0, n], [ns, 0], [-1, 0]], dtype=torch.int64, device="cuda")
    out = ctx.read(pts, n, bad).cpu().numpy()
    assert np.all(out.view(np.uint16) == 0xFFFF) and ctx.sync_status() == -2   # FKV_ERANGE


@pytest.mark.parametrize("N", [257, 1024])
def test_append_equals_scratch_encode(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    L = ctx.L
    ns = 3
    st = fkv.Streams(ctx, ns, capacity=5)
    rng = np.random.default_rng(N)
    full = np.zeros((ns, 0), np.int16)
    for m in [1, L - 1, L, 1, 3 * L + 2, 2, 50 * L + 1, 700 * L + 3]:
        if m <= 0:
            continue
        new = rng.integers(0, N, size=(ns, m)).astype(np.int16)
        st.append(_dev(new))
        full = np.concatenate([full, new], axis=1)
        got = st.export()
        want = _oracle_points(oracle_mod, full, N, ctx.r, L)
        assert np.array_equal(_bits(got), _bits(want)), m
    assert np.array_equal(ctx.span_decode(st.points(), st.length).cpu().numpy(), full)
    assert ctx.sync_status() == 0


@pytest.mark.parametrize("N", [512, 1024])
def test_suffix_search_equals_oracle(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    L = ctx.L
    ns, n = 3, 8000 * L + 2
    # a small alphabet slice so that suffixes repeat often
    sym = (_rand(8, ns, n, N) * (N // 8)).astype(np.int16)
    pts = ctx.span_encode(_dev(sym))
    pth = pts.cpu().numpy()
    for ql in range(1, L + 1):
        q = sym[1, 5 * L - ql:5 * L]              # the suffix of span 4 of stream 1
        m, c0, c1 = ctx.suffix_search(pts, n, q)
        got = sorted(map(tuple, m.cpu().numpy().tolist()))
        want = []
        ocand = 0
        for s in range(ns):
            mm, cc = oracle_mod.suffix_search(pth[s], n, q.astype(np.int32), N, ctx.r, L)
            want += [(s, int(u)) for u in mm]
            ocand += len(cc)
        assert got == sorted(want) and c0 == len(want) and c1 == ocand, ql
        assert (1, 4) in got
    assert ctx.sync_status() == 0


@pytest.mark.parametrize("N,dist", [(1024, "uniform"), (1024, "zipf"), (300, "zipf")])
def test_symbol_codec_stress_full_size(fkv, oracle_mod, N, dist):
    """Two streams of 2^28 seeded uint16 symbols: encode, full decode and 2^20
    random reads per stream; points checked bit-exact on sampled spans."""
    ctx = fkv.Context(N)
    L = ctx.L
    ns, n = 2, 1 << 28
    sym = synth.gpu_symbols(N, dist, ns, n)
    assert sym.dtype == torch.int16
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
            assert np.array_equal(host.astype(np.int16), sym[s, b:e].cpu().numpy())
            want = oracle_mod.span_encode(host.astype(np.int32), N, ctx.r, L)[0]
            assert np.array_equal(_bits(pts[s, u].cpu().numpy()), _bits(want))
    reads = 1 << 20
    req = torch.stack([torch.arange(ns, device="cuda").repeat_interleave(reads),
                       torch.cat([synth.gpu_positions(n, reads, s) for s in range(ns)])], dim=1)
    got = ctx.read(pts, n, req)
    assert torch.equal(got, sym[req[:, 0], req[:, 1]])
    assert ctx.sync_status() == 0
