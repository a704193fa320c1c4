"""Key and value reconstruction (Sec. 3 "Setup": the sum of the selected
centroids) for pairs of key and value stage counts other than the paper's:
both caches rebuilt in one call equal each rebuilt alone, the archive read
gives the same caches, and every vector matches the oracle's float64 sum."""
import dataclasses

import numpy as np
import pytest
import torch

import synth
from oracle import parity

pytestmark = pytest.mark.gpu
TORCH_DT = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}

# (4, 2) is the paper's; the rest span every slice width of the gather (64,
# 32 and 16 floats) on either side
PAIRS = [(1, 1), (2, 1), (4, 2), (3, 3), (4, 4), (1, 4), (2, 3), (4, 3), (5, 3), (8, 8)]


@pytest.fixture(scope="module")
def fkv():
    import paper_2607_07144_gb300 as m
    m.lib()
    return m


def _case(SK, SV, dt, D, n_arch):
    base = dataclasses.replace(synth.CFG3, stages_k=SK, stages_v=SV, dim=D, dtype=dt)
    return synth.small_config(base, 500 + 10 * SK + SV, n_layers=2, batch=3, seq=36 + n_arch, n_heads=3)


@pytest.mark.parametrize("n_arch", [5, 517])
@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("dt", ["bf16", "f32"])
@pytest.mark.parametrize("SK,SV", PAIRS)
def test_kv_gather_equals_one_sided_and_oracle(fkv, oracle_mod, SK, SV, dt, D, n_arch):
    cfg = _case(SK, SV, dt, D, n_arch)
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    ctx = fkv.Context(256, codebooks=(cbk, cbv))
    P, R = cfg.n_archived, ctx.record_len()
    g = torch.Generator().manual_seed(1000 * SK + 100 * SV + D + n_arch)
    sym = torch.randint(0, 256, (cfg.batch * cfg.n_layers, P * R), generator=g, dtype=torch.uint8).cuda()
    shape = cfg.cache_shape()
    z = lambda: torch.zeros(shape, dtype=TORCH_DT[dt], device="cuda")
    Kf, Vf, Ks, Vs = z(), z(), z(), z()
    ctx.rvq_decode(sym, P, Kf, Vf, t0=cfg.t0)
    ctx.rvq_decode(sym, P, Ks, None, t0=cfg.t0)
    ctx.rvq_decode(sym, P, None, Vs, t0=cfg.t0)
    assert torch.equal(Kf, Ks) and torch.equal(Vf, Vs)
    # the archive read (planar symbols from the span decoder) gives the same caches
    pts = ctx.span_encode(sym)
    Kd, Vd = z(), z()
    ctx.decode_kv(pts, P, Kd, Vd, t0=cfg.t0)
    assert ctx.sync_status() == 0
    assert torch.equal(Kd, Kf) and torch.equal(Vd, Vf)
    for X in (Kf, Vf):
        assert torch.count_nonzero(X[:, :, :, :cfg.t0]) == 0 and torch.count_nonzero(X[:, :, :, cfg.t1:]) == 0
    # every rebuilt vector against the oracle's float64 sum
    sh = sym.cpu().numpy().reshape(cfg.batch, cfg.n_layers, P * R)
    for b in range(cfg.batch):
        for l in range(cfg.n_layers):
            ik, iv = oracle_mod.indices_from_records(sh[b, l], cfg.n_heads, SK, SV)
            for h in range(cfg.n_heads):
                for out, idx, cb, S in ((Kf, ik, cbk, SK), (Vf, iv, cbv, SV)):
                    got = out[l, b, h, cfg.t0:cfg.t1].float().cpu().numpy().astype(np.float64)
                    want = oracle_mod.rvq_decode(idx[h], cb[l, h])
                    if dt == "f32":
                        # float32 sums in stage order: S - 1 roundings, each within 2^-24 of a
                        # partial sum, itself at most the sum of magnitudes
                        bound = (S - 1) * 2.0 ** -24 * oracle_mod.rvq_decode(idx[h], np.abs(cb[l, h]))
                        assert np.all(np.abs(got - want) <= bound)
                    else:
                        hard, _, _ = parity.rounded_mismatches(got, want, dt,
                                                               oracle_mod.rvq_decode(idx[h], np.abs(cb[l, h])))
                        assert hard == 0


def test_kv_gather_into_wider_caches(fkv):
    """Output caches holding more sequences' worth of positions than are
    archived, written at an offset: only [t0, t0 + n_rec) changes."""
    cfg = _case(4, 2, "bf16", 128, 300)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    P, R = cfg.n_archived, ctx.record_len()
    g = torch.Generator().manual_seed(7)
    sym = torch.randint(0, 256, (cfg.batch * cfg.n_layers, P * R), generator=g, dtype=torch.uint8).cuda()
    big = (cfg.n_layers, cfg.batch, cfg.n_heads, cfg.seq + 100, cfg.dim)
    Kb = torch.full(big, 3.0, dtype=torch.bfloat16, device="cuda")
    Vb = torch.full(big, 5.0, dtype=torch.bfloat16, device="cuda")
    ctx.rvq_decode(sym, P, Kb, Vb, t0=50)
    Ks = torch.full(big, 3.0, dtype=torch.bfloat16, device="cuda")
    Vs = torch.full(big, 5.0, dtype=torch.bfloat16, device="cuda")
    ctx.rvq_decode(sym, P, Ks, None, t0=50)
    ctx.rvq_decode(sym, P, None, Vs, t0=50)
    assert torch.equal(Kb, Ks) and torch.equal(Vb, Vs)
    assert torch.all(Kb[:, :, :, :50] == 3.0) and torch.all(Kb[:, :, :, 50 + P:] == 3.0)
    assert torch.all(Vb[:, :, :, :50] == 5.0) and torch.all(Vb[:, :, :, 50 + P:] == 5.0)
