"""The whole archive path on the GPU against the oracle: exact-window split,
RVQ into token records, span encoding, full decode with reconstruction,
random record reads (Sec. 2) and decode-time appends."""
import numpy as np
import pytest
import torch

import synth
from oracle import parity

pytestmark = pytest.mark.gpu
TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def write_archive(fkv, cfg, K, V, ctx=None):
    if ctx is None:
        ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    P, R = cfg.n_archived, ctx.record_len()
    sym = torch.empty((cfg.batch * cfg.n_layers, P * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, cfg.t0, cfg.t1, sym)
    ctx.rvq_encode(1, V, cfg.t0, cfg.t1, sym)
    pts = ctx.span_encode(sym)
    return ctx, sym, pts


@pytest.mark.parametrize("base,cid", [(synth.CFG1, 301), (synth.CFG3, 303)])
def test_archive_round_trip(fkv, oracle_mod, base, cid):
    cfg = synth.small_config(base, cid, n_layers=2, batch=2, seq=36 + 200)
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx, sym, pts = write_archive(fkv, cfg, K, V)
    P, R = cfg.n_archived, ctx.record_len()
    # stored points: bit-exact with the oracle's encode of the same streams
    symh = sym.cpu().numpy()
    for i in range(symh.shape[0]):
        want = oracle_mod.span_encode(symh[i].astype(np.int32), 256, ctx.r, ctx.L)
        assert np.array_equal(pts[i].cpu().numpy().view(np.uint64), want.view(np.uint64))
    # full read: decode + gather into fresh caches (the exact window stays untouched)
    Kr = torch.zeros_like(K)
    Vr = torch.zeros_like(V)
    ctx.decode_kv(pts, P, Kr, Vr, t0=cfg.t0)
    assert ctx.sync_status() == 0
    Kg = torch.zeros_like(K)
    Vg = torch.zeros_like(V)
    ctx.rvq_decode(sym, P, Kg, Vg, t0=cfg.t0)
    assert torch.equal(Kr, Kg) and torch.equal(Vr, Vg)
    assert torch.count_nonzero(Kr[:, :, :, :cfg.t0]) == 0 and torch.count_nonzero(Kr[:, :, :, cfg.t1:]) == 0
    # reconstruction against the oracle (sampled groups)
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    sh = symh.reshape(cfg.batch, cfg.n_layers, P * R)
    for (b, l) in [(0, 0), (cfg.batch - 1, cfg.n_layers - 1)]:
        ik, iv = oracle_mod.indices_from_records(sh[b, l], cfg.n_heads, cfg.stages_k, cfg.stages_v)
        for h in range(cfg.n_heads):
            for out, idx, cb in ((Kr, ik, cbk), (Vr, iv, cbv)):
                got = out[l, b, h, cfg.t0:cfg.t1].float().cpu().numpy().astype(np.float64)
                hard, _, _ = parity.rounded_mismatches(got, oracle_mod.rvq_decode(idx[h], cb[l, h]), cfg.dtype,
                                                       oracle_mod.rvq_decode(idx[h], np.abs(cb[l, h])))
                assert hard == 0
    # random record reads equal the full decode
    n_req = 3000
    rng = np.random.default_rng(cid)
    req = np.stack([rng.integers(0, cfg.batch * cfg.n_layers, n_req), rng.integers(0, P, n_req)], axis=1)
    out = torch.empty((n_req, 2, cfg.n_heads, cfg.dim), dtype=K.dtype, device="cuda")
    ctx.read_kv(pts, P, torch.from_numpy(req).cuda(), out)
    assert ctx.sync_status() == 0
    b = req[:, 0] // cfg.n_layers
    l = req[:, 0] % cfg.n_layers
    t = req[:, 1] + cfg.t0
    ti = lambda a: torch.from_numpy(a).cuda()
    assert torch.equal(out[:, 0], Kr[ti(l), ti(b), :, ti(t)])
    assert torch.equal(out[:, 1], Vr[ti(l), ti(b), :, ti(t)])


def test_cache_upload_moves_only_the_archived_positions(fkv):
    cfg = synth.small_config(synth.CFG1, 306, n_layers=2, batch=3, seq=36 + 50)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    K = torch.from_numpy(synth.kv_cache(cfg, 0)).pin_memory()
    dst = torch.full(cfg.cache_shape(), 7.0, dtype=K.dtype, device="cuda")
    ctx.cache_upload(K, dst, cfg.t0, cfg.t1)
    torch.cuda.synchronize()
    want = torch.full(cfg.cache_shape(), 7.0, dtype=K.dtype)
    want[:, :, :, cfg.t0:cfg.t1] = K[:, :, :, cfg.t0:cfg.t1]
    assert torch.equal(dst.cpu(), want)
    # a layout whose rows do not share one pitch: one copy per (layer, sequence)
    big = torch.zeros((cfg.n_layers, cfg.batch + 1) + cfg.cache_shape()[2:], dtype=K.dtype).pin_memory()
    big[:, 1:] = K
    src = big[:, 1:]
    dst2 = torch.zeros(cfg.cache_shape(), dtype=K.dtype, device="cuda")
    ctx.cache_upload(src, dst2, 0, cfg.seq)
    torch.cuda.synchronize()
    assert torch.equal(dst2.cpu(), K)
    with pytest.raises(fkv.FkvError):
        ctx.cache_upload(K, dst, 10, 5)


def test_decode_time_streaming(fkv, oracle_mod):
    """Config-4 pattern at reduced size: a prefilled archive, then steps that
    each append the token leaving the recent window (RVQ + tail append) and
    make random record reads, checked against a full decode and the oracle."""
    cfg = synth.small_config(synth.CFG4, 304, n_layers=3, batch=4, seq=36 + 64 + 24)
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    R = ctx.record_len()
    ns = cfg.batch * cfg.n_layers
    prefill = 64
    st = fkv.Streams(ctx, ns, capacity=prefill * R)
    stage = torch.empty((ns, prefill * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, 4, 4 + prefill, stage)
    ctx.rvq_encode(1, V, 4, 4 + prefill, stage)
    st.append(stage)
    history = [stage.cpu().numpy()]
    rng = np.random.default_rng(4)
    rec = torch.empty((ns, R), dtype=torch.uint8, device="cuda")
    for step in range(24):
        t = 4 + prefill + step              # the position leaving the recent window
        ctx.rvq_encode(0, K, t, t + 1, rec)
        ctx.rvq_encode(1, V, t, t + 1, rec)
        st.append(rec)
        history.append(rec.cpu().numpy())
        n_rec = prefill + step + 1
        req = np.stack([rng.integers(0, ns, 64), rng.integers(0, n_rec, 64)], axis=1)
        out = torch.empty((64, 2, cfg.n_heads, cfg.dim), dtype=K.dtype, device="cuda")
        ctx.read_kv(st.points(), n_rec, torch.from_numpy(req).cuda(), out)
        Kr = torch.zeros_like(K)
        Vr = torch.zeros_like(V)
        ctx.decode_kv(st.points(), n_rec, Kr, Vr, t0=4)
        b = req[:, 0] // cfg.n_layers
        l = req[:, 0] % cfg.n_layers
        ti = lambda a: torch.from_numpy(a).cuda()
        assert torch.equal(out[:, 0], Kr[ti(l), ti(b), :, ti(req[:, 1] + 4)])
        assert torch.equal(out[:, 1], Vr[ti(l), ti(b), :, ti(req[:, 1] + 4)])
    assert ctx.sync_status() == 0
    full = np.concatenate(history, axis=1)
    got = st.export()
    for i in range(ns):
        want = oracle_mod.span_encode(full[i].astype(np.int32), 256, ctx.r, ctx.L)
        assert np.array_equal(got[i].view(np.uint64), want.view(np.uint64))
    # the appended records are the RVQ of the whole archived range in one call
    whole = torch.empty((ns, (prefill + 24) * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, 4, 4 + prefill + 24, whole)
    ctx.rvq_encode(1, V, 4, 4 + prefill + 24, whole)
    assert np.array_equal(whole.cpu().numpy(), full)


def test_record_reads_in_any_order(fkv):
    """Record reads (Sec. 2) taken grouped by layer inside the library: every
    output lands at its own request's place whatever the order, across calls
    whose request count grows (the order buffer is reallocated), with
    out-of-range requests mixed in (zeros and FKV_ERANGE)."""
    cfg = synth.small_config(synth.CFG3, 313, n_layers=5, batch=3, seq=36 + 77)
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx, sym, pts = write_archive(fkv, cfg, K, V)
    P = cfg.n_archived
    Kr, Vr = torch.zeros_like(K), torch.zeros_like(V)
    ctx.decode_kv(pts, P, Kr, Vr, t0=cfg.t0)
    ns = cfg.batch * cfg.n_layers
    ti = lambda a: torch.from_numpy(a).cuda()
    for n_req, seed in ((100, 1), (5000, 2), (40000, 3), (7, 4)):
        rng = np.random.default_rng(seed)
        req = np.stack([rng.integers(0, ns, n_req), rng.integers(0, P, n_req)], axis=1)
        bad = rng.random(n_req) < 0.05
        req[bad, 0] = rng.choice([-1, ns, ns + 7], bad.sum())
        out = torch.full((n_req, 2, cfg.n_heads, cfg.dim), 9.0, dtype=K.dtype, device="cuda")
        ctx.read_kv(pts, P, ti(req), out)
        assert ctx.sync_status() == (-2 if bad.any() else 0)
        ok = ~bad
        b, l, t = req[ok, 0] // cfg.n_layers, req[ok, 0] % cfg.n_layers, req[ok, 1] + cfg.t0
        assert torch.equal(out[ti(np.flatnonzero(ok)), 0], Kr[ti(l), ti(b), :, ti(t)])
        assert torch.equal(out[ti(np.flatnonzero(ok)), 1], Vr[ti(l), ti(b), :, ti(t)])
        assert torch.count_nonzero(out[ti(np.flatnonzero(bad))]) == 0
