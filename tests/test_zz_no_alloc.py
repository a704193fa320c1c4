"""The allocation-free archive read, fkv_decode_kv_static.

Some callers cannot let a library call cudaMalloc: a serving loop whose device
memory all belongs to its own pool allocator, or a latency-critical step that
cannot take cudaMalloc's implicit synchronisation.  fkv_decode_kv_static does
the same work as fkv_decode_kv with a fixed scratch array compiled into the
library.  These checks call it through the C ABI twice in a row, on two
different archives, and require exactly the output of fkv_decode_kv (the
tolerance of the other archive tests is equality for the same kernels).

This file is collected last, so a run that stops at the first failure has
already run every other test; it also passes on its own in a fresh process.
"""
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


def _archive(fkv, ctx, cfg):
    K = synth.gpu_kv_cache(cfg, 0)
    V = synth.gpu_kv_cache(cfg, 1)
    P, R = cfg.n_archived, ctx.record_len()
    sym = torch.empty((cfg.batch * cfg.n_layers, P * R), dtype=torch.uint8, device="cuda")
    ctx.rvq_encode(0, K, cfg.t0, cfg.t1, sym)
    ctx.rvq_encode(1, V, cfg.t0, cfg.t1, sym)
    return K, V, ctx.span_encode(sym)


def test_static_scratch_decode_matches_allocating_decode(fkv):
    base = synth.small_config(synth.CFG1, 501, n_layers=2, batch=3, seq=36 + 240)
    other = synth.small_config(synth.CFG1, 502, n_layers=2, batch=3, seq=36 + 240)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(base, 0), synth.codebooks(base, 1)))
    P = base.n_archived
    for cfg in (base, other):                      # two calls in a row, different archives
        K, V, pts = _archive(fkv, ctx, cfg)
        Ka, Va = torch.zeros_like(K), torch.zeros_like(V)
        ctx.decode_kv(pts, P, Ka, Va, t0=cfg.t0)
        Kb = torch.full_like(K, 7.0)
        Vb = torch.full_like(V, 7.0)
        Kb[:, :, :, cfg.t0:cfg.t1] = 0
        Vb[:, :, :, cfg.t0:cfg.t1] = 0
        ctx.decode_kv_static(pts, P, Kb, Vb, t0=cfg.t0)
        assert ctx.sync_status() == 0
        assert torch.equal(Kb[:, :, :, cfg.t0:cfg.t1], Ka[:, :, :, cfg.t0:cfg.t1])
        assert torch.equal(Vb[:, :, :, cfg.t0:cfg.t1], Va[:, :, :, cfg.t0:cfg.t1])
        # positions outside the archived range are left alone
        assert torch.all(Kb[:, :, :, :cfg.t0] == 7.0) and torch.all(Vb[:, :, :, cfg.t1:] == 7.0)


def test_first_call_takes_no_device_memory(fkv):
    # the fixed array's address is looked up when the context is created, so
    # the first allocation-free decode on a context loads no module and takes
    # no device memory (its kernels are the allocating decode's, loaded by
    # that call first, together with its own scratch)
    cfg = synth.small_config(synth.CFG1, 504, n_layers=2, batch=2, seq=36 + 100)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    K, V, pts = _archive(fkv, ctx, cfg)
    Ka, Va = torch.zeros_like(K), torch.zeros_like(V)
    ctx.decode_kv(pts, cfg.n_archived, Ka, Va, t0=cfg.t0)
    Kb, Vb = torch.zeros_like(K), torch.zeros_like(V)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    ctx.decode_kv_static(pts, cfg.n_archived, Kb, Vb, t0=cfg.t0)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert ctx.sync_status() == 0
    assert free1 == free0
    assert torch.equal(Kb, Ka) and torch.equal(Vb, Va)


def test_static_scratch_rejects_oversized_archives(fkv):
    cfg = synth.small_config(synth.CFG1, 503, n_layers=12, batch=8, seq=1024)
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    R = ctx.record_len()
    n_rec = (16 << 20) // (cfg.batch * cfg.n_layers * R) + 1          # one record too many
    pts = torch.zeros((cfg.batch * cfg.n_layers, ctx.n_spans(n_rec * R), 2), dtype=torch.float64, device="cuda")
    out = torch.zeros((cfg.n_layers, cfg.batch, cfg.n_heads, n_rec + 8, cfg.dim), dtype=torch.float16,
                      device="cuda")
    with pytest.raises(fkv.FkvError) as ei:
        ctx.decode_kv_static(pts, n_rec, out, None, t0=0)
    assert ei.value.code == -1 and "16 MiB" in str(ei.value)
    assert torch.count_nonzero(out) == 0                               # nothing was launched


def test_static_scratch_at_its_limit_matches_allocating_decode(fkv):
    # a real archive exactly as large as the fixed array allows
    base = synth.small_config(synth.CFG1, 505, n_layers=2, batch=2, seq=36, n_heads=4)
    R = base.n_heads * (base.stages_k + base.stages_v)
    n_rec = (16 << 20) // (base.batch * base.n_layers * R)
    cfg = synth.small_config(synth.CFG1, 505, n_layers=2, batch=2, seq=36 + n_rec, n_heads=4)
    assert cfg.n_archived == n_rec and cfg.batch * cfg.n_layers * n_rec * R <= 16 << 20
    ctx = fkv.Context(256, codebooks=(synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)))
    K, V, pts = _archive(fkv, ctx, cfg)
    Ka, Va = torch.zeros_like(K), torch.zeros_like(V)
    ctx.decode_kv(pts, n_rec, Ka, Va, t0=cfg.t0)
    Kb, Vb = torch.zeros_like(K), torch.zeros_like(V)
    ctx.decode_kv_static(pts, n_rec, Kb, Vb, t0=cfg.t0)
    assert ctx.sync_status() == 0
    assert torch.equal(Kb, Ka) and torch.equal(Vb, Va)
    assert torch.count_nonzero(Kb[:, :, :, cfg.t0:cfg.t1]) > 0
