"""Decode-time streaming at full size (Llama-3-8B shape, 64 sequences): a
131072-position archive prefilled through RVQ and appends, then 512 steps that
each archive the position leaving the recent window (RVQ + tail append) and
read 4096 seeded random records per sequence.  Checks: sampled record reads
against an independent symbol read + gather every step, whole streams against
a full decode and the oracle's encode, sampled RVQ indices against the oracle."""
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


def test_config4_full_size_streaming(fkv, oracle_mod):
    free, _ = torch.cuda.mem_get_info()
    if free < 120e9:
        pytest.skip("needs about 60 GB of device memory")
    cfg = synth.CFG4
    P, steps = synth.CFG4_PREFILL, synth.CFG4_STEPS
    Ly, B, H, D = cfg.n_layers, cfg.batch, cfg.n_heads, cfg.dim
    t0 = cfg.t0
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    ctx = fkv.Context(256, codebooks=(cbk, cbv))
    R = ctx.record_len()
    ns = B * Ly
    st = fkv.Streams(ctx, ns, capacity=(P + steps) * R)
    keep = [(0, 0), (37, 21), (63, 31)]                      # (sequence, layer) streams kept on the host
    kept = {k: [] for k in keep}
    C = 4096
    sym = torch.empty((ns, C * R), dtype=torch.uint8, device="cuda")
    for c0 in range(0, P, C):
        Kc = synth.gpu_kv_cache(cfg, 0, t0=t0 + c0, count=C)
        Vc = synth.gpu_kv_cache(cfg, 1, t0=t0 + c0, count=C)
        if c0 == 0:                                           # the range generator equals the host twin
            h = np.array([0, 3, 7])
            xs = synth.kv_elements(cfg, 0, np.array([0, 5, 31]), np.array([0, 9, 63]), h, t0 + np.array([0, 7, C - 1]))
            got = Kc[torch.tensor([0, 5, 31]), torch.tensor([0, 9, 63]), torch.from_numpy(h), torch.tensor([0, 7, C - 1])]
            assert np.array_equal(synth.storage_to_f64(xs, cfg.dtype), got.float().cpu().numpy().astype(np.float64))
        ctx.rvq_encode(0, Kc, 0, C, sym)
        ctx.rvq_encode(1, Vc, 0, C, sym)
        st.append(sym)
        for (b, l) in keep:
            kept[b, l].append(sym[b * Ly + l].cpu().numpy())
        del Kc, Vc
    assert ctx.sync_status() == 0
    rec = torch.empty((ns, R), dtype=torch.uint8, device="cuda")
    n_req = 4096 * B
    out = torch.empty((n_req, 2, H, D), dtype=torch.bfloat16, device="cuda")
    gen = torch.Generator(device="cuda").manual_seed(2607)
    seq_of = torch.arange(B, device="cuda").repeat_interleave(4096)
    one = torch.zeros((ns, R), dtype=torch.uint8, device="cuda")
    K1 = torch.empty((Ly, B, H, 1, D), dtype=torch.bfloat16, device="cuda")
    V1 = torch.empty_like(K1)
    for i in range(steps):
        t = t0 + P + i                                        # the position leaving the recent window
        Kt = synth.gpu_kv_cache(cfg, 0, t0=t, count=1)
        Vt = synth.gpu_kv_cache(cfg, 1, t0=t, count=1)
        ctx.rvq_encode(0, Kt, 0, 1, rec)
        ctx.rvq_encode(1, Vt, 0, 1, rec)
        st.append(rec)
        for (b, l) in keep:
            kept[b, l].append(rec[b * Ly + l].cpu().numpy())
        n_rec = P + i + 1
        layer = torch.randint(0, Ly, (n_req,), generator=gen, device="cuda")
        recno = torch.randint(0, n_rec, (n_req,), generator=gen, device="cuda")
        req = torch.stack([seq_of * Ly + layer, recno], dim=1)
        ctx.read_kv(st.points(), n_rec, req, out)
        # two reads per step against the record's symbols (symbol reads) and the gather
        for q in (int(i * 7919 % n_req), int(i * 104729 % n_req)):
            s_, r_ = int(req[q, 0]), int(req[q, 1])
            pos = torch.tensor([[s_, r_ * R + j] for j in range(R)], dtype=torch.int64, device="cuda")
            one.zero_()
            one[s_] = ctx.read(st.points(), n_rec * R, pos)
            ctx.rvq_decode(one, 1, K1, V1, t0=0)
            b, l = s_ // Ly, s_ % Ly
            assert torch.equal(out[q, 0], K1[l, b, :, 0]) and torch.equal(out[q, 1], V1[l, b, :, 0]), (i, q)
    assert ctx.sync_status() == 0
    n_rec = P + steps
    pts = st.points()
    for (b, l), parts in kept.items():
        want = np.concatenate(parts)
        assert want.size == n_rec * R
        s_ = b * Ly + l
        got = ctx.span_decode(pts[s_:s_ + 1], n_rec * R)
        assert np.array_equal(got[0].cpu().numpy(), want)        # a full decode of the stream
    (b, l) = keep[1]
    want = np.concatenate(kept[b, l]).astype(np.int32)
    opts = oracle_mod.span_encode(want, 256, ctx.r, ctx.L)
    assert np.array_equal(pts[b * Ly + l, :opts.shape[0]].cpu().numpy().view(np.uint64), opts.view(np.uint64))
    # sampled RVQ indices of the kept streams against the oracle
    rng = np.random.default_rng(4)
    hard = seen = 0
    for (b, l), parts in kept.items():
        s_all = np.concatenate(parts).reshape(n_rec, R)
        recs = np.unique(np.concatenate([rng.integers(0, n_rec, 40), [0, P - 1, P, n_rec - 1]]))
        for kv, cb, S, off in ((0, cbk, cfg.stages_k, 0), (1, cbv, cfg.stages_v, H * cfg.stages_k)):
            for h in range(H):
                x = synth.storage_to_f64(synth.kv_elements(cfg, kv, l, b, h, t0 + recs), cfg.dtype)
                oi, gap = oracle_mod.rvq_encode(x.reshape(-1, D), cb[l, h])
                g = s_all[recs][:, off + h * S: off + (h + 1) * S].astype(np.int32)
                diff = (g != oi) & (gap > 1e-4)
                for v in range(g.shape[0]):                      # stage s counts where earlier stages agree
                    for s in range(S):
                        if g[v, s] != oi[v, s]:
                            hard += int(diff[v, s])
                            break
                seen += g.size
    assert hard == 0 and seen > 0
