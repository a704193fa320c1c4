"""GPU parity of the archive with 1024-codeword and pooled codebooks (Sec. 3,
Table 2: pooled VQ k = 1024 and pooled RVQ k = 1024 x 2), uint16 symbols.

The bar is the one of the k = 256 archive: every index equal to the oracle's
wherever the oracle's top-2 gap exceeds 1e-4 ||residual||^2, float32 sums
within 1e-3 of the oracle's float64 sums, rounded outputs equal to the
oracle's except across a rounding boundary, stored points bit for bit, and
the full decode, record reads and allocation-free decode all equal to the
gather of the encoded indices."""
import dataclasses

import numpy as np
import pytest
import torch

import synth
from test_gpu_rvq import _check_rounded, compare_rvq

pytestmark = pytest.mark.gpu
TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def make_ctx(fkv, cfg, cbk=None, cbv=None):
    cbk = synth.codebooks(cfg, 0) if cbk is None else cbk
    cbv = synth.codebooks(cfg, 1) if cbv is None else cbv
    return fkv.Context(cfg.N, codebooks=(cbk, cbv), pooled=cfg.pooled, n_heads=cfg.n_heads)


def cb_of(cb, cfg, l, h):
    return cb[l, 0 if cfg.pooled else h]


def encode(fkv, cfg, K, V, ctx):
    P, R = cfg.n_archived, ctx.record_len()
    sym = torch.zeros((cfg.batch * cfg.n_layers, P * R), dtype=ctx.sym_dtype, device="cuda")
    ctx.rvq_encode(0, K, cfg.t0, cfg.t1, sym)
    ctx.rvq_encode(1, V, cfg.t0, cfg.t1, sym)
    assert ctx.sync_status() == 0
    return sym


def indices(oracle_mod, sym, cfg, b, l):
    s = sym.cpu().numpy().astype(np.int32).reshape(cfg.batch, cfg.n_layers, -1)
    return oracle_mod.indices_from_records(s[b, l], cfg.n_heads, cfg.stages_k, cfg.stages_v)


SMALL = [
    synth.small_config(synth.CFG5, 501, n_layers=2, batch=3, seq=36 + 300),
    synth.small_config(synth.CFG6, 502, n_layers=2, batch=2, seq=36 + 300),
    dataclasses.replace(synth.small_config(synth.CFG5, 503, n_layers=2, batch=2, seq=36 + 260), pooled=False),
    dataclasses.replace(synth.small_config(synth.CFG5, 504, n_layers=1, batch=2, seq=36 + 333), dtype="f32"),
    dataclasses.replace(synth.small_config(synth.CFG5, 505, n_layers=1, batch=2, seq=36 + 290), dtype="bf16"),
    # pooled k = 256 on both RVQ kernels (64- and 128-dimensional heads)
    dataclasses.replace(synth.small_config(synth.CFG1, 506, n_layers=2, batch=2, seq=36 + 300), pooled=True),
    dataclasses.replace(synth.small_config(synth.CFG3, 507, n_layers=2, batch=1, seq=36 + 300), pooled=True),
]


@pytest.mark.parametrize("cfg", SMALL, ids=lambda c: "%s-%s-%s" % (c.N, "pooled" if c.pooled else "head", c.dtype))
def test_rvq_and_reconstruction(fkv, oracle_mod, cfg):
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx = make_ctx(fkv, cfg)
    assert ctx.sym_bytes == (2 if cfg.N > 256 else 1)
    sym = encode(fkv, cfg, K, V, ctx)
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    K64 = synth.storage_to_f64(synth.kv_cache(cfg, 0), cfg.dtype)
    V64 = synth.storage_to_f64(synth.kv_cache(cfg, 1), cfg.dtype)
    P = cfg.n_archived
    Kr = torch.zeros_like(K)
    Vr = torch.zeros_like(V)
    ctx.rvq_decode(sym, P, Kr, Vr, t0=cfg.t0)
    assert ctx.sync_status() == 0
    Kh = Kr.float().cpu().numpy().astype(np.float64)
    Vh = Vr.float().cpu().numpy().astype(np.float64)
    hard = near = seen = 0
    hi_used = 0
    for b in range(cfg.batch):
        for l in range(cfg.n_layers):
            ik, iv = indices(oracle_mod, sym, cfg, b, l)
            for h in range(cfg.n_heads):
                for X, cb, gi, Y in ((K64, cbk, ik, Kh), (V64, cbv, iv, Vh)):
                    c = cb_of(cb, cfg, l, h)
                    oi, gap = oracle_mod.rvq_encode(X[l, b, h, cfg.t0:cfg.t1], c)
                    hd, nr, sn = compare_rvq(gi[h], oi, gap)
                    hard, near, seen = hard + hd, near + nr, seen + sn
                    hi_used += int((gi[h] >= 768).sum())
                    y = oracle_mod.rvq_decode(gi[h], c)
                    got = Y[l, b, h, cfg.t0:cfg.t1]
                    if cfg.dtype == "f32":
                        assert np.max(np.abs(got - y)) <= 1e-3
                    else:
                        _check_rounded(got, y, cfg.dtype, oracle_mod.rvq_decode(gi[h], np.abs(c)))
    print("%s: compared %d, near-tie mismatches %d" % (cfg.name, seen, near))
    assert hard == 0
    if cfg.N == 1024:
        assert hi_used > 0                      # codewords of the last 256-block are chosen too
    assert torch.count_nonzero(Kr[:, :, :, :cfg.t0]) == 0 and torch.count_nonzero(Kr[:, :, :, cfg.t1:]) == 0


def test_tie_across_codeword_blocks_takes_lowest_index(fkv):
    """Codeword 1000 (last 256-block) duplicates codeword 3 (first block) and
    codeword 700 duplicates 300: inputs equal to them must take 3 and 300."""
    cfg = dataclasses.replace(synth.small_config(synth.CFG6, 508, n_layers=1, batch=1, seq=36 + 64), dtype="f32")
    cbk = np.array(synth.codebooks(cfg, 0))
    cbv = np.array(synth.codebooks(cfg, 1))
    cbk[0, 0, 0, 1000] = cbk[0, 0, 0, 3]
    cbk[0, 0, 0, 700] = cbk[0, 0, 0, 300]
    ctx = make_ctx(fkv, cfg, cbk, cbv)
    K = torch.zeros(cfg.cache_shape(), dtype=torch.float32, device="cuda")
    pick = np.resize([3, 1000, 300, 700], cfg.seq)
    K[0, 0, :, :] = torch.from_numpy(cbk[0, 0, 0, pick]).cuda()[None]
    V = synth.gpu_kv_cache(cfg, 1)
    sym = encode(fkv, cfg, K, V, ctx)
    s = sym.cpu().numpy().astype(np.int32).reshape(-1, ctx.record_len())
    want = np.where(pick == 1000, 3, np.where(pick == 700, 300, pick))[cfg.t0:cfg.t1]
    for h in range(cfg.n_heads):
        assert np.array_equal(s[:, h], want)


@pytest.mark.parametrize("cfg", SMALL[:3], ids=["pooled-rvq1024x2", "pooled-vq1024", "head-rvq1024x2"])
def test_archive_round_trip(fkv, oracle_mod, cfg):
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx = make_ctx(fkv, cfg)
    sym = encode(fkv, cfg, K, V, ctx)
    pts = ctx.span_encode(sym)
    P, R = cfg.n_archived, ctx.record_len()
    assert ctx.L == 5
    symh = sym.cpu().numpy().astype(np.int32)
    for i in range(symh.shape[0]):
        want = oracle_mod.span_encode(symh[i], 1024, ctx.r, ctx.L)
        assert np.array_equal(pts[i].cpu().numpy().view(np.uint64), want.view(np.uint64))
    Kg, Vg = torch.zeros_like(K), torch.zeros_like(V)
    ctx.rvq_decode(sym, P, Kg, Vg, t0=cfg.t0)
    for dec in (ctx.decode_kv, ctx.decode_kv_static):
        Kr, Vr = torch.zeros_like(K), torch.zeros_like(V)
        dec(pts, P, Kr, Vr, t0=cfg.t0)
        assert ctx.sync_status() == 0
        assert torch.equal(Kr, Kg) and torch.equal(Vr, Vg)
    n_req = 2000
    rng = np.random.default_rng(cfg.cfg_id)
    req = np.stack([rng.integers(0, cfg.batch * cfg.n_layers, n_req), rng.integers(0, P, n_req)], axis=1)
    out = torch.empty((n_req, 2, cfg.n_heads, cfg.dim), dtype=K.dtype, device="cuda")
    ctx.read_kv(pts, P, torch.from_numpy(req).cuda(), out)
    assert ctx.sync_status() == 0
    b, l, t = req[:, 0] // cfg.n_layers, req[:, 0] % cfg.n_layers, req[:, 1] + cfg.t0
    ti = lambda a: torch.from_numpy(a).cuda()
    assert torch.equal(out[:, 0], Kg[ti(l), ti(b), :, ti(t)])
    assert torch.equal(out[:, 1], Vg[ti(l), ti(b), :, ti(t)])


def test_decode_time_append(fkv, oracle_mod):
    """Records appended one position at a time equal the RVQ of the whole
    range, and the appended stream equals the oracle's encode."""
    cfg = synth.small_config(synth.CFG5, 509, n_layers=2, batch=3, seq=36 + 40 + 13)
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx = make_ctx(fkv, cfg)
    R, ns = ctx.record_len(), cfg.batch * cfg.n_layers
    st = fkv.Streams(ctx, ns, capacity=8)
    rec = torch.empty((ns, R), dtype=ctx.sym_dtype, device="cuda")
    for t in range(cfg.t0, cfg.t1):
        ctx.rvq_encode(0, K, t, t + 1, rec)
        ctx.rvq_encode(1, V, t, t + 1, rec)
        st.append(rec)
    whole = encode(fkv, cfg, K, V, ctx).cpu().numpy()
    got = st.export()
    for i in range(ns):
        want = oracle_mod.span_encode(whole[i].astype(np.int32), 1024, ctx.r, ctx.L)
        assert np.array_equal(got[i].view(np.uint64), want.view(np.uint64))
    assert ctx.sync_status() == 0


def test_full_size_pooled_rvq1024x2(fkv, oracle_mod):
    """The whole Table 2 pooled RVQ 1024 x 2 workload (12 layers x 8 sequences
    x 12 heads x 988 archived positions): indices on sampled (sequence, layer)
    streams against the oracle, and the archive round trip."""
    cfg = synth.CFG5
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx = make_ctx(fkv, cfg)
    sym = encode(fkv, cfg, K, V, ctx)
    pts = ctx.span_encode(sym)
    P = cfg.n_archived
    Kg, Vg = torch.zeros_like(K), torch.zeros_like(V)
    ctx.rvq_decode(sym, P, Kg, Vg, t0=cfg.t0)
    Kr, Vr = torch.zeros_like(K), torch.zeros_like(V)
    ctx.decode_kv(pts, P, Kr, Vr, t0=cfg.t0)
    assert ctx.sync_status() == 0
    assert torch.equal(Kr, Kg) and torch.equal(Vr, Vg)
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    hard = seen = 0
    for (b, l) in [(0, 0), (3, 7), (7, 11)]:
        ik, iv = indices(oracle_mod, sym, cfg, b, l)
        hs = [0, 5, 11]
        X = {0: synth.storage_to_f64(synth.kv_elements(cfg, 0, l, b, np.array(hs)[:, None],
                                                       np.arange(cfg.t0, cfg.t1)[None, :]), cfg.dtype),
             1: synth.storage_to_f64(synth.kv_elements(cfg, 1, l, b, np.array(hs)[:, None],
                                                       np.arange(cfg.t0, cfg.t1)[None, :]), cfg.dtype)}
        for j, h in enumerate(hs):
            for kv, cb, gi in ((0, cbk, ik), (1, cbv, iv)):
                oi, gap = oracle_mod.rvq_encode(X[kv][j], cb[l, 0])
                hd, _, sn = compare_rvq(gi[h], oi, gap)
                hard, seen = hard + hd, seen + sn
    assert hard == 0 and seen > 0
