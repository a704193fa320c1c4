"""The GPT-2-shaped full cache (12 layers x 8 sequences x 12 heads x 1024
positions x 64 dims, fp16; K 4 / V 2 stages) end to end on the GPU against
the oracle, every vector, span and value (Sec. 3 "Setup", Sec. 1):
  * every RVQ index of the 1.14 M key and value vectors, stage by stage,
    under the 1e-4 gap rule (near ties counted and printed);
  * every stored point of the 96 (sequence, layer) streams bit-exact with the
    oracle's encode of the GPU's symbols, and the decoded symbols equal;
  * every rebuilt fp16 K/V value equal to the oracle's float64 sum rounded to
    nearest-even outside the float32 summation error band (borderline cases
    counted and printed)."""
import numpy as np
import pytest
import torch

import synth
from oracle import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def test_gpt2_full_cache_every_vector(fkv, oracle_mod):
    cfg = synth.CFG1
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    ctx = fkv.Context(256, codebooks=(cbk, cbv))
    P, R = cfg.n_archived, ctx.record_len()
    ns = cfg.batch * cfg.n_layers
    sym = torch.empty((ns, P * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, cfg.t0, cfg.t1, sym)
    ctx.rvq_encode(1, V, cfg.t0, cfg.t1, sym)
    pts = ctx.span_encode(sym)
    Kr, Vr = torch.zeros_like(K), torch.zeros_like(V)
    ctx.decode_kv(pts, P, Kr, Vr, t0=cfg.t0)
    dec = ctx.span_decode(pts, P * R)
    assert ctx.sync_status() == 0
    assert torch.equal(dec, sym)

    Kh = K[:, :, :, cfg.t0:cfg.t1].float().cpu().numpy().astype(np.float64)
    Vh = V[:, :, :, cfg.t0:cfg.t1].float().cpu().numpy().astype(np.float64)
    Krh = Kr[:, :, :, cfg.t0:cfg.t1].float().cpu().numpy().astype(np.float64)
    Vrh = Vr[:, :, :, cfg.t0:cfg.t1].float().cpu().numpy().astype(np.float64)
    symh = sym.cpu().numpy()
    ph = pts.cpu().numpy()
    tot = dict(rvq_seen=0, rvq_hard=0, rvq_near=0, spans=0, kv=0, kv_hard=0, kv_border=0)
    for b in range(cfg.batch):
        for l in range(cfg.n_layers):
            i = b * cfg.n_layers + l
            want = oracle_mod.span_encode(symh[i].astype(np.int32), 256, ctx.r, ctx.L)
            assert np.array_equal(ph[i].view(np.uint64), want.view(np.uint64)), (b, l)
            tot["spans"] += want.shape[0]
            gk, gv = oracle_mod.indices_from_records(symh[i], cfg.n_heads, cfg.stages_k, cfg.stages_v)
            for h in range(cfg.n_heads):
                for X, Xr, cb, gi in ((Kh, Krh, cbk, gk), (Vh, Vrh, cbv, gv)):
                    oi, gap = oracle_mod.rvq_encode(X[l, b, h], cb[l, h])
                    hard, near, seen = parity.compare_rvq(gi[h], oi, gap)
                    tot["rvq_hard"] += hard
                    tot["rvq_near"] += near
                    tot["rvq_seen"] += seen
                    hard, border, n = parity.rounded_mismatches(Xr[l, b, h], oracle_mod.rvq_decode(gi[h], cb[l, h]),
                                                                "f16", oracle_mod.rvq_decode(gi[h], np.abs(cb[l, h])))
                    tot["kv_hard"] += hard
                    tot["kv_border"] += border
                    tot["kv"] += n
    print("gpt2 full cache: %d RVQ decisions compared, %d near-tie mismatches; %d spans bit-exact; "
          "%d K/V values, %d rounding-borderline" % (tot["rvq_seen"], tot["rvq_near"], tot["spans"], tot["kv"],
                                                    tot["kv_border"]))
    assert tot["rvq_hard"] == 0 and tot["kv_hard"] == 0
    assert tot["rvq_seen"] >= 2 * ns * cfg.n_heads * P                 # every vector's first stage at least
    assert tot["kv"] == 2 * ns * cfg.n_heads * P * cfg.dim
