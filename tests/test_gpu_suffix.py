"""GPU parity of in-place suffix retrieval (Sec. 5) against the oracle.

Match sets must equal the oracle's exactly (they are exact string matches,
verified by decoding); candidate counts must equal the oracle's (both sides
evaluate the same binary64 distance test); order is free, so sets are
compared sorted."""
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


def _oracle_all(oracle_mod, sym, pts, n, query, N, r, L):
    match, cand = [], 0
    for s in range(sym.shape[0]):
        mm, cc = oracle_mod.suffix_search(pts[s], n, query, N, r, L)
        match += [(s, int(u)) for u in mm]
        cand += cc.size
    return sorted(match), cand


@pytest.mark.parametrize("N", [3, 4, 16, 256])
def test_suffix_search_equals_oracle(fkv, oracle_mod, N):
    ctx = fkv.Context(N)
    L, r = ctx.L, ctx.r
    rng = np.random.default_rng(300 + N)
    ns, n = 3, 700 * L + L // 2 + 1
    sym = rng.integers(0, min(N, 4), (ns, n)).astype(np.uint8)   # small alphabet: many matches
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    host_pts = pts.cpu().numpy()
    queries = []
    for qlen in sorted({1, 2, max(1, L // 2), L}):
        u = int(rng.integers(0, n // L))
        queries.append(sym[1, u * L + L - qlen:u * L + L])      # present
        queries.append(rng.integers(0, N, qlen).astype(np.uint8))
    for q in queries:
        got, count, cand = ctx.suffix_search(pts, n, q)
        want, wcand = _oracle_all(oracle_mod, sym, host_pts, n, q, N, r, L)
        assert count == len(want) and cand == wcand, (q, count, len(want), cand, wcand)
        assert sorted(map(tuple, got.cpu().tolist())) == want
    assert ctx.sync_status() == 0


def test_cap_and_counts(fkv, oracle_mod):
    ctx = fkv.Context(16)
    L = ctx.L
    sym = np.zeros((2, 100 * L), np.uint8)
    pts = ctx.span_encode(torch.from_numpy(sym).cuda())
    got, count, cand = ctx.suffix_search(pts, sym.shape[1], np.zeros(3, np.uint8), cap=37)
    assert count == 200 and cand == 200 and got.shape[0] == 37
    allm = {(s, u) for s in range(2) for u in range(100)}
    assert set(map(tuple, got.cpu().tolist())) <= allm
    assert len(set(map(tuple, got.cpu().tolist()))) == 37


def test_bad_queries_and_empty(fkv):
    ctx = fkv.Context(16)
    L = ctx.L
    pts = ctx.span_encode(torch.zeros((1, 5 * L), dtype=torch.uint8, device="cuda"))
    for q in [np.zeros(0, np.uint8), np.zeros(L + 1, np.uint8), np.array([16], np.uint8)]:
        with pytest.raises(fkv.FkvError):
            ctx.suffix_search(pts, 5 * L, q)
    e = torch.empty((0, 1, 2), dtype=torch.float64, device="cuda")
    _, count, cand = ctx.suffix_search(e, 0, np.zeros(1, np.uint8))
    assert count == 0 and cand == 0


def test_archive_suffix_search(fkv, oracle_mod):
    """Retrieval over a token-record archive: the last span of a record is
    found from its own symbols, across every (sequence, layer) stream."""
    cfg = synth.small_config(synth.CFG1, 601, n_layers=2, batch=2, seq=36 + 300)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    K, V = synth.gpu_kv_cache(cfg, 0), synth.gpu_kv_cache(cfg, 1)
    P, R = cfg.n_archived, ctx.record_len()
    sym = torch.empty((cfg.batch * cfg.n_layers, P * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, cfg.t0, cfg.t1, sym)
    ctx.rvq_encode(1, V, cfg.t0, cfg.t1, sym)
    pts = ctx.span_encode(sym)
    host = sym.cpu().numpy()
    L = ctx.L
    for s, u in [(0, 5), (3, 100), (1, (P * R) // L - 1)]:
        q = host[s, u * L:(u + 1) * L]
        got, count, cand = ctx.suffix_search(pts, P * R, q)
        want, wcand = _oracle_all(oracle_mod, host, pts.cpu().numpy(), P * R, q, 256, ctx.r, L)
        assert (s, u) in want
        assert sorted(map(tuple, got.cpu().tolist())) == want and cand == wcand


def test_symbol_stress_suffix_full_size(fkv, oracle_mod):
    """Four streams of 2^28 seeded symbols (N = 256, span 6): planted span
    queries are found, and every returned match decodes to the query."""
    ctx = fkv.Context(256)
    L = ctx.L
    ns, n = 4, 1 << 28
    sym = synth.gpu_symbols(256, "uniform", ns, n)
    pts = ctx.span_encode(sym)
    spans = pts.shape[1]
    rng = np.random.default_rng(5)
    for qlen in [3, 6]:
        s, u = int(rng.integers(0, ns)), int(rng.integers(0, spans - 1))
        q = sym[s, u * L + L - qlen:u * L + L].cpu().numpy()
        got, count, cand = ctx.suffix_search(pts, n, q, cap=1 << 20)
        pairs = got.cpu().numpy()
        assert count <= 1 << 20 and (s, u) in set(map(tuple, pairs.tolist()))
        # every reported span ends with the query (checked on the host twin of the generator)
        for st, uu in pairs[:2000]:
            tail = synth.symbols(256, "uniform", int(st), np.arange(uu * L + L - qlen, uu * L + L))
            assert np.array_equal(tail, q)
        if qlen == 3:
            # 2^30 / 6 spans, 2^-24 chance each: a few dozen matches expected
            assert 1 <= count < 1000
    assert ctx.sync_status() == 0
