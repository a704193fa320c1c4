"""GPU parity of per-head residual VQ and the codebook gather (Sec. 3 "Setup").

Criterion: every index must equal the oracle's wherever the oracle's top-2
distance gap exceeds 1e-4 * ||residual||^2 (stage s compared only where the
earlier stages agreed); closer ties are counted and reported.  Rebuilt K/V:
float32 sums within 1e-3 of the oracle's float64 sums, and fp16/bf16 outputs
equal to the oracle sum rounded to nearest-even except where the float32
summation error bound straddles a rounding boundary."""
import dataclasses

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu
GAP = 1e-4
TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def compare_rvq(gpu, ora, gap):
    """-> (hard mismatches, near-tie mismatches, compared entries)."""
    from oracle import parity
    return parity.compare_rvq(gpu, ora, gap, GAP)


def host_cache(cfg, kv):
    a = synth.kv_cache(cfg, kv)
    return synth.storage_to_f64(a, cfg.dtype)


def to_device(cfg, a64):
    t = torch.from_numpy(a64).to(TORCH_DT[cfg.dtype])
    return t.cuda()


def run_rvq(fkv, cfg, K, V, cbk, cbv, t0=None, t1=None):
    ctx = fkv.Context(256, codebooks=(cbk, cbv))
    t0 = cfg.t0 if t0 is None else t0
    t1 = cfg.t1 if t1 is None else t1
    R = ctx.record_len()
    sym = torch.zeros((cfg.batch * cfg.n_layers, (t1 - t0) * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, t0, t1, sym)
    ctx.rvq_encode(1, V, t0, t1, sym)
    assert ctx.sync_status() == 0
    return ctx, sym


def gpu_indices(oracle_mod, sym, cfg, P):
    s = sym.cpu().numpy().reshape(cfg.batch, cfg.n_layers, P * cfg.record_len)
    out = {}
    for b in range(cfg.batch):
        for l in range(cfg.n_layers):
            out[b, l] = oracle_mod.indices_from_records(s[b, l], cfg.n_heads, cfg.stages_k, cfg.stages_v)
    return out


def check_config_full(fkv, oracle_mod, cfg):
    K64, V64 = host_cache(cfg, 0), host_cache(cfg, 1)
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    ctx, sym = run_rvq(fkv, cfg, to_device(cfg, K64), to_device(cfg, V64), cbk, cbv)
    P = cfg.n_archived
    gi = gpu_indices(oracle_mod, sym, cfg, P)
    tot_hard = tot_near = tot_seen = 0
    for b in range(cfg.batch):
        for l in range(cfg.n_layers):
            ik, iv = gi[b, l]
            for h in range(cfg.n_heads):
                for kv, X, cb, gidx in ((0, K64, cbk, ik), (1, V64, cbv, iv)):
                    x = X[l, b, h, cfg.t0:cfg.t1]
                    oi, gap = oracle_mod.rvq_encode(x, cb[l, h])
                    hard, near, seen = compare_rvq(gidx[h], oi, gap)
                    tot_hard += hard
                    tot_near += near
                    tot_seen += seen
    print("rvq %s: compared %d, near-tie mismatches %d" % (cfg.name, tot_seen, tot_near))
    assert tot_hard == 0
    return ctx, sym, gi, K64, V64, cbk, cbv


def test_config0_full(fkv, oracle_mod):
    cfg = synth.CFG0
    ctx, sym, gi, K64, V64, cbk, cbv = check_config_full(fkv, oracle_mod, cfg)
    # reconstruction in float32: within 1e-3 of the oracle's float64 sum
    P = cfg.n_archived
    Kr = torch.zeros(cfg.cache_shape(), dtype=torch.float32, device="cuda")
    Vr = torch.zeros(cfg.cache_shape(), dtype=torch.float32, device="cuda")
    ctx.rvq_decode(sym, P, Kr, Vr, t0=cfg.t0)
    assert ctx.sync_status() == 0
    Kr, Vr = Kr.cpu().numpy(), Vr.cpu().numpy()
    ik, iv = gi[0, 0]
    worst = 0.0
    for h in range(cfg.n_heads):
        yk = oracle_mod.rvq_decode(ik[h], cbk[0, h])
        yv = oracle_mod.rvq_decode(iv[h], cbv[0, h])
        worst = max(worst, np.abs(Kr[0, 0, h, cfg.t0:cfg.t1] - yk).max(), np.abs(Vr[0, 0, h, cfg.t0:cfg.t1] - yv).max())
    assert worst <= 1e-3
    assert np.all(Kr[0, 0, :, :cfg.t0] == 0) and np.all(Kr[0, 0, :, cfg.t1:] == 0)   # exact window untouched


def _check_rounded(got, ref64, dtype, absum):
    """got (rounded on the GPU from a float32 sum) must equal the oracle's
    float64 sum rounded to nearest-even, except where the float32 summation
    error bound (4 * 2^-24 * sum |c_s|, plus 1e-6 relative) straddles a
    rounding boundary.  Returns the number of such borderline differences."""
    from oracle import parity
    hard, border, _ = parity.rounded_mismatches(got, ref64, dtype, absum)
    assert hard == 0, hard
    return border


def test_small_gpt2_fp16_full(fkv, oracle_mod):
    cfg = synth.small_config(synth.CFG1, 201, n_layers=2, batch=3, seq=36 + 300)
    ctx, sym, gi, K64, V64, cbk, cbv = check_config_full(fkv, oracle_mod, cfg)
    P = cfg.n_archived
    Kr = torch.zeros(cfg.cache_shape(), dtype=torch.float16, device="cuda")
    Vr = torch.zeros(cfg.cache_shape(), dtype=torch.float16, device="cuda")
    ctx.rvq_decode(sym, P, Kr, Vr, t0=cfg.t0)
    Kr = Kr.cpu().numpy().astype(np.float64)
    Vr = Vr.cpu().numpy().astype(np.float64)
    mid = 0
    for (b, l), (ik, iv) in gi.items():
        for h in range(cfg.n_heads):
            mid += _check_rounded(Kr[l, b, h, cfg.t0:cfg.t1], oracle_mod.rvq_decode(ik[h], cbk[l, h]), "f16",
                                  oracle_mod.rvq_decode(ik[h], np.abs(cbk[l, h])))
            mid += _check_rounded(Vr[l, b, h, cfg.t0:cfg.t1], oracle_mod.rvq_decode(iv[h], cbv[l, h]), "f16",
                                  oracle_mod.rvq_decode(iv[h], np.abs(cbv[l, h])))
    print("fp16 midpoint cases:", mid)


def test_small_llama_bf16_d128(fkv, oracle_mod):
    cfg = synth.small_config(synth.CFG3, 203, n_layers=2, batch=2, seq=36 + 260)
    ctx, sym, gi, K64, V64, cbk, cbv = check_config_full(fkv, oracle_mod, cfg)
    P = cfg.n_archived
    Kr = torch.zeros(cfg.cache_shape(), dtype=torch.bfloat16, device="cuda")
    Vr = torch.zeros(cfg.cache_shape(), dtype=torch.bfloat16, device="cuda")
    ctx.rvq_decode(sym, P, Kr, Vr, t0=cfg.t0)
    Kr = Kr.float().cpu().numpy().astype(np.float64)
    Vr = Vr.float().cpu().numpy().astype(np.float64)
    for (b, l), (ik, iv) in gi.items():
        for h in range(cfg.n_heads):
            _check_rounded(Kr[l, b, h, cfg.t0:cfg.t1], oracle_mod.rvq_decode(ik[h], cbk[l, h]), "bf16",
                           oracle_mod.rvq_decode(ik[h], np.abs(cbk[l, h])))
            _check_rounded(Vr[l, b, h, cfg.t0:cfg.t1], oracle_mod.rvq_decode(iv[h], cbv[l, h]), "bf16",
                           oracle_mod.rvq_decode(iv[h], np.abs(cbv[l, h])))


def _one_group_cfg(dim, dtype, seq):
    return synth.KVConfig(900 + dim, "edge", 1, 1, 1, dim, seq, dtype, 2, 1, 0, 1.0, 0.0)


@pytest.mark.parametrize("dim", [64, 128])
def test_edge_vectors(fkv, oracle_mod, dim):
    """Codeword-equal inputs, duplicate codewords (ties -> lowest index),
    huge, tiny and zero vectors, partial tiles."""
    rng = np.random.default_rng(dim)
    cbk = rng.normal(size=(1, 1, 2, 256, dim)).astype(np.float32)
    cbk[0, 0, 1] *= 0.5
    cbk[0, 0, 0, 200] = cbk[0, 0, 0, 9]                  # duplicate codeword
    cbv = rng.normal(size=(1, 1, 1, 256, dim)).astype(np.float32)
    for n in [1, 6, 16, 127, 129, 300]:
        x = rng.normal(size=(n, dim))
        x[0] = cbk[0, 0, 0, 9]                            # equal to a (duplicated) codeword
        if n > 5:
            x[1] = cbk[0, 0, 0, 77]
            x[2] *= 1e4
            x[3] *= 1e-6
            x[4] = 0.0
            x[5] = cbk[0, 0, 0, 3] + cbk[0, 0, 1, 5]
        cfg = _one_group_cfg(dim, "f32", n)
        X = torch.from_numpy(x.astype(np.float32)).reshape(1, 1, 1, n, dim).cuda()
        ctx, sym = run_rvq(fkv, cfg, X, X, cbk, cbv, t0=0, t1=n)
        idx = sym.cpu().numpy().reshape(n, 3)
        oi, gap = oracle_mod.rvq_encode(x.astype(np.float32).astype(np.float64), cbk[0, 0])
        hard, near, seen = compare_rvq(idx[:, :2].astype(np.int32), oi, gap)
        assert hard == 0, (n, hard)
        assert idx[0, 0] == 9
        if n > 5:
            assert idx[1, 0] == 77 and idx[5, 0] == 3


@pytest.mark.parametrize("dim,dtype,K,pooled", [(64, "f16", 256, False), (64, "f32", 256, False),
                                                (64, "bf16", 1024, True), (128, "bf16", 256, False),
                                                (128, "bf16", 256, True), (128, "f32", 256, False)])
def test_small_batch(fkv, oracle_mod, dim, dtype, K, pooled):
    """At most 16 vectors per codebook group (a decode step's appended
    position: tiles with 1 to 16 live rows of 128): every index equals the
    oracle's outside near ties, for several (batch, positions) shapes, with
    rows far outside and far inside the codebooks' scale, codeword-equal rows
    and zero rows, per-head and pooled codebooks."""
    rng = np.random.default_rng(dim + K + len(dtype))
    L, H = 2, 3
    Hc = 1 if pooled else H
    SK = 2 if K == 1024 else 3                          # 1024-codeword codebooks: two stages at most
    cbk = rng.normal(size=(L, Hc, SK, K, dim)).astype(np.float32)
    cbk[:, :, 1] *= 0.3
    cbk[:, :, SK - 1] *= 1e-3                           # another power-of-two scale
    cbv = rng.normal(size=(L, Hc, 2, K, dim)).astype(np.float32)
    big, small = (1e3, 1e-3) if dtype == "f16" else (1e30, 1e-30)
    ctx = fkv.Context(K, codebooks=(cbk, cbv), pooled=pooled, n_heads=H if pooled else None)
    R = ctx.record_len()
    for batch, npos in [(1, 1), (8, 1), (3, 5), (2, 8), (1, 16)]:
        t0, seq = 3, npos + 7
        x = rng.normal(size=(L, batch, H, seq, dim))
        x[0, 0, 0, t0] *= big
        x[1, 0, 1, t0] *= small
        x[0, 0, 2, t0] = 0.0
        x[1, 0, 0, t0] = cbk[1, 0, 0, 17]
        X = torch.from_numpy(x).to(TORCH_DT[dtype]).cuda()
        x64 = X.double().cpu().numpy()
        sym = torch.zeros((batch * L, npos * R), dtype=ctx.sym_dtype, device="cuda")
        ctx.rvq_encode(0, X, t0, t0 + npos, sym)
        ctx.rvq_encode(1, X, t0, t0 + npos, sym)
        assert ctx.sync_status() == 0
        s = sym.cpu().numpy().astype(np.int32).reshape(batch, L, npos * R)
        assert s.max() < K
        for b in range(batch):
            for l in range(L):
                ik, iv = oracle_mod.indices_from_records(s[b, l], H, SK, 2)
                for h in range(H):
                    for gidx, cb in ((ik, cbk), (iv, cbv)):
                        oi, gap = oracle_mod.rvq_encode(x64[l, b, h, t0:t0 + npos], cb[l, 0 if pooled else h])
                        hard, near, seen = compare_rvq(gidx[h], oi, gap)
                        assert hard == 0, (batch, npos, b, l, h, hard)
        ik, _ = oracle_mod.indices_from_records(s[0, 1], H, SK, 2)
        assert ik[0, 0, 0] == 17                        # the codeword-equal row


@pytest.mark.parametrize("dim,k1024", [(64, False), (64, True), (128, False)])
def test_extreme_magnitudes_and_stage_scale_change(fkv, oracle_mod, dim, k1024):
    """Rows far outside the codebook (1e20, 1e30), far inside it (1e-30,
    subnormal), and a second stage 1e4 times smaller than the first (its
    codebook takes another power-of-two scale, so every row is rescaled and its
    shift chosen again between the stages, from the maximum over both halves
    of a 128-dimensional row), with 256 and 1024 codewords."""
    K = 1024 if k1024 else 256
    rng = np.random.default_rng(11 + k1024 + dim)
    cbk = rng.normal(size=(1, 1, 2, K, dim)).astype(np.float32)
    cbk[0, 0, 1] *= 1e-4
    cbv = rng.normal(size=(1, 1, 1, K, dim)).astype(np.float32)
    n = 400
    x = rng.normal(size=(n, dim))
    x[:50] += cbk[0, 0, 0, rng.integers(0, K, 50)] * 3.0
    x[50:60] *= 1e20
    x[60:70] *= 1e30
    x[70:80] *= 1e-30
    x[80:90] *= 1e-40                                   # float32 subnormals
    x[90:200] = cbk[0, 0, 0, rng.integers(0, K, 110)] + 0.5 * cbk[0, 0, 1, rng.integers(0, K, 110)]
    cfg = dataclasses.replace(_one_group_cfg(dim, "f32", n), N=K)
    X = torch.from_numpy(x.astype(np.float32)).reshape(1, 1, 1, n, dim).cuda()
    ctx = fkv.Context(K, codebooks=(cbk, cbv))
    sym = torch.zeros((1, n * 3), dtype=ctx.sym_dtype, device="cuda")
    ctx.rvq_encode(0, X, 0, n, sym)
    ctx.rvq_encode(1, X, 0, n, sym)
    assert ctx.sync_status() == 0
    idx = sym.cpu().numpy().astype(np.int32).reshape(n, 3)
    assert idx.max() < K
    oi, gap = oracle_mod.rvq_encode(x.astype(np.float32).astype(np.float64), cbk[0, 0])
    hard, near, seen = compare_rvq(idx[:, :2], oi, gap)
    assert hard == 0, hard


def test_strided_cache_view(fkv, oracle_mod):
    """A non-contiguous view (layer dimension interleaved with an unused
    buffer) gives the same symbols as the contiguous copy."""
    cfg = synth.small_config(synth.CFG1, 205, n_layers=2, batch=2, seq=36 + 140)
    K = to_device(cfg, host_cache(cfg, 0))
    V = to_device(cfg, host_cache(cfg, 1))
    big = torch.zeros((cfg.n_layers, 2) + cfg.cache_shape()[1:], dtype=K.dtype, device="cuda")
    big[:, 1] = K
    Ks = big[:, 1]
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    _, s1 = run_rvq(fkv, cfg, K, V, cbk, cbv)
    _, s2 = run_rvq(fkv, cfg, Ks, V, cbk, cbv)
    assert torch.equal(s1, s2)


def _sampled_check(fkv, oracle_mod, cfg, n_sample):
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    ctx, sym = run_rvq(fkv, cfg, K, V, cbk, cbv)
    R, P = cfg.record_len, cfg.n_archived
    rng = np.random.default_rng(cfg.cfg_id)
    l = rng.integers(0, cfg.n_layers, n_sample)
    b = rng.integers(0, cfg.batch, n_sample)
    h = rng.integers(0, cfg.n_heads, n_sample)
    t = rng.integers(cfg.t0, cfg.t1, n_sample)
    symh = sym.view(cfg.batch, cfg.n_layers, P, R)
    hard_total = near_total = 0
    for kv, X, cb, S, off in ((0, K, cbk, cfg.stages_k, 0), (1, V, cbv, cfg.stages_v, cfg.n_heads * cfg.stages_k)):
        xs = synth.storage_to_f64(synth.kv_elements(cfg, kv, l, b, h, t), cfg.dtype)
        dev = X[torch.from_numpy(l).cuda(), torch.from_numpy(b).cuda(), torch.from_numpy(h).cuda(),
                torch.from_numpy(t).cuda()].float().cpu().numpy().astype(np.float64)
        assert np.array_equal(xs, dev)                  # device generator == host twin
        g = np.empty((n_sample, S), np.int32)
        sl = symh[torch.from_numpy(b).cuda(), torch.from_numpy(l).cuda(), torch.from_numpy(t - cfg.t0).cuda()]
        sl = sl.cpu().numpy()
        for i in range(n_sample):
            g[i] = sl[i, off + h[i] * S: off + (h[i] + 1) * S]
        oi = np.empty((n_sample, S), np.int32)
        gap = np.empty((n_sample, S))
        for grp in set(zip(l.tolist(), h.tolist())):
            sel = (l == grp[0]) & (h == grp[1])
            oi[sel], gap[sel] = oracle_mod.rvq_encode(xs[sel], cb[grp[0], grp[1]])
        hard, near, seen = compare_rvq(g, oi, gap)
        hard_total += hard
        near_total += near
    print("%s sampled %d vectors: near-tie mismatches %d" % (cfg.name, n_sample, near_total))
    assert hard_total == 0
    return ctx, sym, K, V


def test_config1_full_size_sampled(fkv, oracle_mod):
    _sampled_check(fkv, oracle_mod, synth.CFG1, 4000)


def test_config3_full_size_sampled(fkv, oracle_mod):
    free, total = torch.cuda.mem_get_info()
    if free < 48e9:
        pytest.skip("needs ~40 GB of device memory")
    ctx, sym, K, V = _sampled_check(fkv, oracle_mod, synth.CFG3, 3000)
    del K, V, sym
    torch.cuda.empty_cache()
