"""GPU parity of the ragged-batch codec calls (streams of different lengths
in one call, Sec. 2's per-sequence code) against the oracle, stream by
stream: points bit-exact, decoded symbols and random reads exact, and the
range status for requests and offsets outside the batch."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _lengths(L, seed):
    rng = np.random.default_rng(seed)
    # empty streams, one-symbol streams, exact multiples of L, ragged tails and
    # long streams spanning several blocks
    ln = [0, 1, L, L + 1, 2 * L - 1, 0, 3] + list(rng.integers(0, 700 * L, size=9))
    return np.array(ln, np.int64)


@pytest.mark.parametrize("N", [3, 16, 256, 1024])
def test_ragged_encode_decode_read_equal_oracle(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    L = ctx.L
    ln = _lengths(L, N)
    rng = np.random.default_rng(N + 1)
    streams = [rng.integers(0, N, size=int(n)) for n in ln]
    np_t = np.uint8 if ctx.sym_bytes == 1 else np.int16
    flat = np.concatenate(streams).astype(np_t)
    so, po = ctx.ragged_offsets(ln)
    d_sym = torch.from_numpy(flat).cuda()
    pts = ctx.span_encode_ragged(d_sym, so, po)
    assert ctx.sync_status() == 0
    ph = pts.cpu().numpy()
    pob = po.cpu().numpy()
    for i, s in enumerate(streams):
        want = oracle_mod.span_encode(s.astype(np.int32), N, ctx.r, L)
        got = ph[pob[i]:pob[i + 1]]
        assert got.shape == want.shape
        assert np.array_equal(got.view(np.uint64), want.view(np.uint64)), i
    dec = ctx.span_decode_ragged(pts, po, so)
    assert ctx.sync_status() == 0
    assert np.array_equal(dec.cpu().numpy()[:flat.size], flat)
    # random reads, every stream's first and last symbol included
    req = []
    for i, n in enumerate(ln):
        if n:
            req += [(i, 0), (i, n - 1)] + [(i, int(p)) for p in rng.integers(0, n, size=50)]
    req = np.array(req, np.int64)
    got = ctx.read_ragged(pts, po, so, torch.from_numpy(req).cuda()).cpu().numpy()
    assert ctx.sync_status() == 0
    want = np.array([streams[i][p] for i, p in req])
    assert np.array_equal(got.astype(np.int64) & 0xFFFF, want)
    # positions outside a stream (its own length, an empty stream, no stream)
    bad = torch.tensor([[1, 1], [0, 0], [len(ln), 0], [-1, 0], [3, int(ln[3])]], dtype=torch.int64, device="cuda")
    out = ctx.read_ragged(pts, po, so, bad).cpu().numpy().astype(np.int64) & 0xFFFF
    assert np.all(out == (0xFF if ctx.sym_bytes == 1 else 0xFFFF))
    assert ctx.sync_status() == -2                       # FKV_ERANGE


def test_ragged_points_with_slack_and_equal_to_the_equal_length_call(fkv, oracle_mod):
    # point slots may exceed a stream's spans; the extra slots stay untouched,
    # and equal lengths give the equal-length call's points
    ctx = fkv.Context(256)
    L, ns, n = ctx.L, 6, 1000 * ctx.L + 5
    rng = np.random.default_rng(7)
    sym = rng.integers(0, 256, size=(ns, n)).astype(np.uint8)
    d = torch.from_numpy(sym).cuda()
    ref = ctx.span_encode(d)
    spans = ctx.n_spans(n)
    slot = spans + 3
    so = torch.arange(ns + 1, dtype=torch.int64, device="cuda") * n
    po = torch.arange(ns + 1, dtype=torch.int64, device="cuda") * slot
    pts = torch.full((ns * slot, 2), 7.0, dtype=torch.float64, device="cuda")
    ctx.span_encode_ragged(d.reshape(-1), so, po, pts=pts)
    assert ctx.sync_status() == 0
    got = pts.reshape(ns, slot, 2)
    assert torch.equal(got[:, :spans], ref)
    assert torch.all(got[:, spans:] == 7.0)
    dec = ctx.span_decode_ragged(pts, po, so)
    assert torch.equal(dec.reshape(ns, n), d)


def test_ragged_inconsistent_offsets_report_range(fkv):
    ctx = fkv.Context(16)
    L = ctx.L
    sym = torch.zeros(10 * L, dtype=torch.uint8, device="cuda")
    # stream 1 has 5 L symbols but only 2 point slots; stream 2 a negative length
    so = torch.tensor([0, L, 6 * L, 5 * L], dtype=torch.int64, device="cuda")
    po = torch.tensor([0, 1, 3, 4], dtype=torch.int64, device="cuda")
    pts = torch.full((4, 2), 7.0, dtype=torch.float64, device="cuda")
    ctx.span_encode_ragged(sym, so, po, pts=pts)
    assert ctx.sync_status() == -2
    p = pts.cpu().numpy()
    assert np.all(p[1:] == 7.0) and np.all(p[0] != 7.0)        # the consistent stream 0 is encoded
    with pytest.raises(fkv.FkvError) as ei:
        ctx.span_encode_ragged(sym, so, po, pts=pts.view(-1)[1:])          # points not 16-byte aligned
    assert ei.value.code == -1
