#!/usr/bin/env python
"""Throughput of the fractal KV-cache archive path on one GB300.

Workload: a GPT-2-shaped full KV cache -- 12 layers x 8 sequences x 12 heads x
1024 positions x 64 dims, fp16, synthetic (seeded Irwin-Hall values with 4
outlier key channels per head), per-head RVQ codebooks with 4 key stages and 2
value stages of 256 codewords, alphabet N = 256 at r = r_256, span length 6.

One step is one pass of the whole archive path over that cache:
  1. exact-window split: positions [4, 992) of every (layer, sequence) leave
     the 4-sink + 32-recent window and are archived;
  2. RVQ assignment of their K and V head vectors into token records;
  3. span encoding of the 96 (sequence, layer) symbol streams (append from empty);
  4. decode-time append: position 992 leaves the window -> RVQ + tail append;
  5. full decode of the archive and reconstruction of K/V at [4, 993);
  6. 4096 random record reads (K and V of all heads of one position).
value = archived KV positions (sequence x layer x position records) per second
over the whole step.  Inputs (302 MB) are larger than L2, so no flush is needed.
`e2e` times the same step through the public API with the caches in pinned host
memory (host -> device copies and the result read-back inside the timed region).

After the timed steps the line also reports, under "kernels", secondary
workloads, each measured on its own (a --no-<name> flag skips it):
  suffix    Sec. 5 retrieval over 4 streams x 2^28 symbols;
  codec     the span codec on the symbol-stress streams (N = 3, 4, 16, 256);
  k1024     Table 2's pooled RVQ 1024 x 2 archive of the same cache;
  lossy     Sec. 4 truncation and lossy decode of this step's streams;
  llama     the Llama-3-8B-shaped archive (--llama-seq sets its cache length);
  weighted  Sec. 6 probability-weighted maps of this step's index streams.

--impl reference times the float64 CPU oracle on a bounded sample of the same
workload (the paper ships no GPU implementation; the oracle is the reference).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "archived KV positions/s (RVQ+span encode) and decoded KV GB/s, % of roofline"
UNIT = "archived KV positions/s"
N_READS = 4096


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# DRAM bytes (read + write) per k_rvq64 launch of this workload, the mean of
# the key launch (197,526,272) and the value launch (171,083,008) in one ncu
# capture (dram__bytes_read.sum + dram__bytes_write.sum) of the current
# kernel; set it to None whenever that kernel changes until it is captured
# again.
RVQ_DRAM_BYTES_PER_LAUNCH = 184304640

# FP64 add/mul peak: GB300's nominal 1.25 TFLOP/s of FP64 FMA is 625 G add or
# mul instructions per second at the 2070 MHz boost clock, 1.99 per clock per SM
# (a dependent-chain probe reached 1.6, the span encoder 1.67)
FP64_OPS_PER_CLK_SM = 1.25e12 / 2 / (152 * 2070e6)


class ClockSampler:
    """nvidia-smi clock/throttle samples during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------ multi-rank --
def rank_workload(rank: int):
    """One rank's replica of the workload: the GPT-2 full cache with its own
    seed (rank 0 runs the base configuration); the archive shards by
    (sequence, layer) stream, so ranks share nothing but the codebooks."""
    base = synth.CFG1
    return synth.dataclasses.replace(base, cfg_id=base.cfg_id + 1000 * rank) if rank else base


def max_over_ranks(values, device):
    """Element-wise maximum of per-rank timings over all ranks (one
    all_reduce; the job's time is its slowest rank's)."""
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


# ---------------------------------------------------------------- GPU arm --
def run_gpu(args, rank, world, local_rank):
    import torch
    import paper_2607_07144_gb300 as fkv

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    base = synth.CFG1
    cfg = rank_workload(rank)
    cbk, cbv = synth.codebooks(base, 0), synth.codebooks(base, 1)     # replicated codebooks
    K = synth.gpu_kv_cache(cfg, 0, device=dev)
    V = synth.gpu_kv_cache(cfg, 1, device=dev)
    ctx = fkv.Context(256, codebooks=(cbk, cbv))
    R = ctx.record_len()
    ns = cfg.batch * cfg.n_layers
    t0, t1 = cfg.t0, cfg.t1                      # archived range [4, 992)
    P = t1 - t0
    n_rec = P + 1                                # + the appended position 992
    sym = torch.empty((ns, P * R), dtype=torch.uint8, device=dev)
    rec = torch.empty((ns, R), dtype=torch.uint8, device=dev)
    st = fkv.Streams(ctx, ns, capacity=n_rec * R)
    Kr = torch.zeros_like(K)
    Vr = torch.zeros_like(V)
    g = torch.Generator().manual_seed(7 + rank)
    req = torch.stack([torch.randint(0, ns, (N_READS,), generator=g),
                       torch.randint(0, n_rec, (N_READS,), generator=g)], dim=1).to(dev)
    out = torch.empty((N_READS, 2, cfg.n_heads, cfg.dim), dtype=K.dtype, device=dev)
    stream = torch.cuda.current_stream()
    names = ["rvq_k", "rvq_v", "span_encode", "append_rvq", "append", "decode_kv", "read_kv"]
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)]

    def step(record=False, K=K, V=V, st=st, out=out):
        e = iter(ev) if record else None
        rec_ = (lambda: next(e).record(stream)) if record else (lambda: None)
        rec_()
        ctx.rvq_encode(0, K, t0, t1, sym)
        rec_()
        ctx.rvq_encode(1, V, t0, t1, sym)
        rec_()
        st.reset()
        st.append(sym)
        rec_()
        ctx.rvq_encode(0, K, t1, t1 + 1, rec)
        ctx.rvq_encode(1, V, t1, t1 + 1, rec)
        rec_()
        st.append(rec)
        rec_()
        ctx.decode_kv(st.points(), n_rec, Kr, Vr, t0=t0)
        rec_()
        ctx.read_kv(st.points(), n_rec, req, out)
        rec_()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if ctx.sync_status() != 0:
        raise RuntimeError("device status error during warm-up")

    # per-phase durations (CUDA events on the launching stream), averaged
    phase = np.zeros(len(names))
    for _ in range(max(1, min(args.steps, 5))):
        step(record=True)
        torch.cuda.synchronize()
        phase += np.array([ev[i].elapsed_time(ev[i + 1]) for i in range(len(names))])
    phase /= max(1, min(args.steps, 5))

    # timed region: K steps, barrier + sync on both sides
    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(args.steps):
        step()
    stop.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    ms = start.elapsed_time(stop) / args.steps
    clk = clocks.stop()
    ok = ctx.sync_status() == 0

    # end-to-end through the public API with host buffers: every step copies
    # its K/V caches in from pinned host memory and reads its result (the
    # archive points and the random-read records) back; steps are pipelined
    # over three streams (copy in, compute, copy out) with double-buffered
    # device inputs and archives, as a serving loop would run them
    e2e = None
    if not args.no_e2e:
        Kh = K.cpu().pin_memory()
        Vh = V.cpu().pin_memory()
        n_sp = ctx.n_spans(n_rec * R)
        Kd, Vd = [K, torch.empty_like(K)], [V, torch.empty_like(V)]
        sts = [st, fkv.Streams(ctx, ns, capacity=n_rec * R)]
        outs = [out, torch.empty_like(out)]
        ptsh = [torch.empty((ns, n_sp, 2), dtype=torch.float64).pin_memory() for _ in range(2)]
        outh = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(2)]
        s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
        free = [None, None]      # compute is done with buffer b's inputs
        read = [None, None]      # buffer b's results are back on the host

        def step_e2e(i, after=None):
            b = i % 2
            with torch.cuda.stream(s_in):
                if after is not None:
                    s_in.wait_event(after)
                if free[b] is not None:
                    s_in.wait_event(free[b])
                # only the positions that leave the exact window travel
                ctx.cache_upload(Kh, Kd[b], t0, t1 + 1, stream=s_in)
                ctx.cache_upload(Vh, Vd[b], t0, t1 + 1, stream=s_in)
                ev_in = torch.cuda.Event()
                ev_in.record(s_in)
            stream.wait_event(ev_in)
            if read[b] is not None:
                stream.wait_event(read[b])
            step(K=Kd[b], V=Vd[b], st=sts[b], out=outs[b])
            done = torch.cuda.Event()
            done.record(stream)
            free[b] = done
            with torch.cuda.stream(s_out):
                s_out.wait_event(done)
                ptsh[b].copy_(sts[b].points()[:, :n_sp], non_blocking=True)
                outh[b].copy_(outs[b], non_blocking=True)
                back = torch.cuda.Event()
                back.record(s_out)
                read[b] = back
        for i in range(2):
            step_e2e(i)
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        s2, t2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record(stream)
        for i in range(args.steps):
            step_e2e(i, after=s2 if i < 2 else None)
        for b in range(2):
            stream.wait_event(read[b])
        t2.record(stream)
        torch.cuda.synchronize()
        e2e_ms = s2.elapsed_time(t2) / args.steps
        h2d = Kh[:, :, :, t0:t1 + 1].numel() * Kh.element_size() * 2
        d2h = ptsh[0].numel() * 8 + outh[0].numel() * outh[0].element_size()
        e2e = {"ms": e2e_ms, "h2d": h2d, "d2h": d2h}

    # Sec. 5 in-place suffix retrieval, measured on its own workload: four
    # streams of 2^28 seeded uniform symbols (N = 256, span 6; 2.86 GB of
    # stored points, far above L2), one 6-symbol query planted from a span
    suffix = None
    if not args.no_suffix:
        sctx = fkv.Context(256)
        s_sym = synth.gpu_symbols(256, "uniform", 4, 1 << 28, device=dev)
        s_pts = sctx.span_encode(s_sym)
        q = s_sym[2, 6 * 1000:6 * 1001].cpu().numpy()
        del s_sym
        match = torch.empty((1 << 16, 2), dtype=torch.int64, device=dev)
        counts = torch.empty(2, dtype=torch.int64, device=dev)
        for _ in range(3):
            sctx.suffix_search(s_pts, 1 << 28, q, match=match, counts=counts)
        reps = 10
        ss, se = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ss.record(stream)
        for _ in range(reps):
            fkv._binding.lib().fkv_suffix_search(
                sctx.handle, fkv._binding._ptr(s_pts), 4, 1 << 28, s_pts.shape[1], q.ctypes.data_as(
                    fkv._binding.ctypes.c_void_p), q.size, fkv._binding._ptr(match), match.shape[0],
                fkv._binding._ptr(counts), fkv._binding._stream(stream))
        se.record(stream)
        torch.cuda.synchronize()
        c = counts.cpu().tolist()
        suffix = {"ms": ss.elapsed_time(se) / reps, "bytes": s_pts.numel() * 8, "matches": c[0], "candidates": c[1],
                  "workload": "4 streams x 2^28 uniform symbols, N=256, span 6, one 6-symbol query"}
        del s_pts, sctx

    # The span codec on the symbol-stress workload: per alphabet N in
    # {3, 4, 16, 256} (spans 44, 44, 16, 6), four streams of 2^28 seeded
    # uniform symbols encoded to points, decoded whole, and 2^20 seeded random
    # positions per stream read back; every result checked against the input
    codec = None
    if not args.no_codec:
        codec = {}
        c_n = 1 << 28
        for c_N in (3, 4, 16, 256):
            cc = fkv.Context(c_N)
            c_sym = synth.gpu_symbols(c_N, "uniform", 4, c_n, device=dev)
            c_pts = cc.span_encode(c_sym)
            c_dec = torch.empty_like(c_sym)
            c_req = torch.cat([torch.stack([torch.full((1 << 20,), s_, dtype=torch.int64, device=dev),
                                          synth.gpu_positions(c_n, 1 << 20, s_, device=dev)], 1) for s_ in range(4)])
            c_out = torch.empty(c_req.shape[0], dtype=c_sym.dtype, device=dev)
            ops = (lambda: cc.span_encode(c_sym, c_pts), lambda: cc.span_decode(c_pts, c_n, c_dec),
                   lambda: cc.read(c_pts, c_n, c_req, c_out))
            for op in ops:
                op()
            reps = 3
            ms_ = []
            for op in ops:
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for _ in range(reps):
                    op()
                e1.record(stream)
                torch.cuda.synchronize()
                ms_.append(e0.elapsed_time(e1) / reps)
            exact = bool(torch.equal(c_dec, c_sym)) and bool(torch.equal(c_out, c_sym[c_req[:, 0], c_req[:, 1]]))
            codec[c_N] = {"L": cc.L, "spans": c_pts.shape[1], "encode_ms": ms_[0], "decode_ms": ms_[1],
                        "read_ms": ms_[2], "reads": c_req.shape[0], "exact": exact, "ok": cc.sync_status() == 0}
            del c_sym, c_pts, c_dec, c_req, c_out, cc

    # Sec. 4 lossy archive of this step's streams: spans older than the last
    # 64 records truncated to 24 bits per coordinate (6 B instead of 16 B per
    # span), the recent ones exact; truncation and the full lossy decode
    lossy = None
    if not args.no_lossy:
        bits, keep = 24, 64 * R // ctx.L
        step()
        torch.cuda.synchronize()
        lp = st.points()
        n_sym = n_rec * R
        T, words, ts = ctx.lossy_geometry(n_sym, bits, keep)
        codes = torch.empty((ns, words), dtype=torch.int32, device=dev)
        tail = torch.empty((ns, ts, 2), dtype=torch.float64, device=dev)
        lsym = torch.empty((ns, n_sym), dtype=torch.uint8, device=dev)
        evl = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        reps = 10
        for _ in range(2):
            ctx.truncate(lp, n_sym, bits, keep, codes=codes, tail=tail)
            ctx.lossy_decode(codes, tail, n_sym, bits, keep, sym=lsym)
        torch.cuda.synchronize()
        evl[0].record(stream)
        for _ in range(reps):                      # back to back: device time, not launch gaps
            ctx.truncate(lp, n_sym, bits, keep, codes=codes, tail=tail)
        evl[1].record(stream)
        for _ in range(reps):
            ctx.lossy_decode(codes, tail, n_sym, bits, keep, sym=lsym)
        evl[2].record(stream)
        torch.cuda.synchronize()
        acc = np.array([evl[0].elapsed_time(evl[1]), evl[1].elapsed_time(evl[2])]) / reps
        exact = ctx.span_decode(lp, n_sym)
        err = (lsym[:, :T * ctx.L] != exact[:, :T * ctx.L]).float().mean().item()
        lossy = {"truncate": acc[0], "decode": acc[1], "bits": bits, "keep": keep, "T": T, "spans": T + ts,
                 "symbols": ns * n_sym, "code_bytes": ns * words * 4, "tail_bytes": ns * ts * 16,
                 "point_bytes": ns * (T + ts) * 16, "sym_err_truncated": err, "ok": ctx.sync_status() == 0}
        del codes, tail, lsym, exact

    # Sec. 6 probability-weighted maps: this step's 96 archived index streams
    # arithmetic-coded with the adaptive add-one model (one warp per stream;
    # decoding is sequential within a stream), encode and decode
    weighted = None
    if not args.no_weighted:
        words, nbits = ctx.ac_encode(sym)
        wsym = torch.empty_like(sym)
        ctx.ac_decode(words, nbits, sym.shape[1], sym=wsym)
        torch.cuda.synchronize()
        evw = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        reps = 3
        evw[0].record(stream)
        for _ in range(reps):
            ctx.ac_encode(sym, words=words, nbits=nbits)
        evw[1].record(stream)
        for _ in range(reps):
            ctx.ac_decode(words, nbits, sym.shape[1], sym=wsym)
        evw[2].record(stream)
        torch.cuda.synchronize()
        weighted = {"encode": evw[0].elapsed_time(evw[1]) / reps, "decode": evw[1].elapsed_time(evw[2]) / reps,
                    "symbols": sym.numel(), "bits": int(nbits.sum().item()), "exact": bool(torch.equal(wsym, sym)),
                    "ok": ctx.sync_status() == 0}
        del words, nbits, wsym

    # Llama-3-8B-shaped archive (32 layers x batch 4 x 8 KV heads x 32768
    # positions x 128 dims, bf16, K 4 / V 2 stages): the same write and read
    # path as the step above, on 128-dimensional heads
    llama = None
    if not args.no_llama:
        c3 = synth.CFG3 if args.llama_seq == synth.CFG3.seq else synth.small_config(
            synth.CFG3, synth.CFG3.cfg_id, n_layers=synth.CFG3.n_layers, batch=synth.CFG3.batch, seq=args.llama_seq)
        lctx = fkv.Context(256, codebooks=(synth.codebooks(c3, 0), synth.codebooks(c3, 1)))
        K3 = synth.gpu_kv_cache(c3, 0, device=dev)
        V3 = synth.gpu_kv_cache(c3, 1, device=dev)
        R3, P3, ns3 = lctx.record_len(), c3.n_archived, c3.batch * c3.n_layers
        sym3 = torch.empty((ns3, P3 * R3), dtype=torch.uint8, device=dev)
        pts3 = torch.empty((ns3, lctx.n_spans(P3 * R3), 2), dtype=torch.float64, device=dev)
        K3r, V3r = torch.zeros_like(K3), torch.zeros_like(V3)
        g3 = torch.Generator().manual_seed(9)
        req3 = torch.stack([torch.randint(0, ns3, (N_READS,), generator=g3),
                            torch.randint(0, P3, (N_READS,), generator=g3)], dim=1).to(dev)
        out3 = torch.empty((N_READS, 2, c3.n_heads, c3.dim), dtype=K3.dtype, device=dev)
        ev3 = [torch.cuda.Event(enable_timing=True) for _ in range(6)]

        def step3(record=False):
            r_ = (lambda i: ev3[i].record(stream)) if record else (lambda i: None)
            r_(0)
            lctx.rvq_encode(0, K3, c3.t0, c3.t1, sym3)
            r_(1)
            lctx.rvq_encode(1, V3, c3.t0, c3.t1, sym3)
            r_(2)
            lctx.span_encode(sym3, pts3)
            r_(3)
            lctx.decode_kv(pts3, P3, K3r, V3r, t0=c3.t0)
            r_(4)
            lctx.read_kv(pts3, P3, req3, out3)
            r_(5)
        step3()
        acc = np.zeros(5)
        reps = 3
        for _ in range(reps):
            step3(record=True)
            torch.cuda.synchronize()
            acc += np.array([ev3[i].elapsed_time(ev3[i + 1]) for i in range(5)])
        acc /= reps
        llama = {"phase": acc.tolist(), "records": ns3 * P3, "nvec": ns3 * P3 * c3.n_heads,
                 "stages": (c3.stages_k, c3.stages_v), "R": R3, "L": lctx.L, "spans": ns3 * lctx.n_spans(P3 * R3),
                 "out_bytes": 2 * ns3 * P3 * c3.n_heads * c3.dim * 2, "ok": lctx.sync_status() == 0}
        del K3, V3, K3r, V3r, sym3, pts3, out3, lctx

    # Table 2's pooled RVQ 1024 x 2 archive on the same GPT-2 shape: one
    # 1024-codeword codebook per layer and stage shared by the 12 heads,
    # uint16 symbols (N = 1024, r_1024, span 5); archive write and full read
    k1024 = None
    if not args.no_k1024:
        c5 = synth.CFG5
        kctx = fkv.Context(c5.N, codebooks=(synth.codebooks(c5, 0), synth.codebooks(c5, 1)), pooled=True,
                           n_heads=c5.n_heads)
        K5 = synth.gpu_kv_cache(c5, 0, device=dev)
        V5 = synth.gpu_kv_cache(c5, 1, device=dev)
        R5, P5 = kctx.record_len(), c5.n_archived
        sym5 = torch.empty((ns, P5 * R5), dtype=kctx.sym_dtype, device=dev)
        pts5 = torch.empty((ns, kctx.n_spans(P5 * R5), 2), dtype=torch.float64, device=dev)
        K5r, V5r = torch.zeros_like(K5), torch.zeros_like(V5)
        ev5 = [torch.cuda.Event(enable_timing=True) for _ in range(5)]

        def step5(record=False):
            if record:
                ev5[0].record(stream)
            kctx.rvq_encode(0, K5, c5.t0, c5.t1, sym5)
            if record:
                ev5[1].record(stream)
            kctx.rvq_encode(1, V5, c5.t0, c5.t1, sym5)
            if record:
                ev5[2].record(stream)
            kctx.span_encode(sym5, pts5)
            if record:
                ev5[3].record(stream)
            kctx.decode_kv(pts5, P5, K5r, V5r, t0=c5.t0)
            if record:
                ev5[4].record(stream)
        for _ in range(3):
            step5()
        reps = 5
        acc = np.zeros(4)
        for _ in range(reps):
            step5(record=True)
            torch.cuda.synchronize()
            acc += np.array([ev5[i].elapsed_time(ev5[i + 1]) for i in range(4)])
        acc /= reps
        k1024 = {"rvq_k": acc[0], "rvq_v": acc[1], "span_encode": acc[2], "decode_kv": acc[3],
                 "nvec": ns * c5.n_heads * P5, "stages": (c5.stages_k, c5.stages_v), "R": R5, "P": P5, "L": kctx.L,
                 "ok": kctx.sync_status() == 0,
                 "out_bytes": 2 * K5.numel() // c5.seq * P5 * K5.element_size()}
        del K5, V5, K5r, V5r, sym5, pts5, kctx

    units = ns * n_rec
    return dict(cfg=cfg, ms=ms, phase=dict(zip(names, phase.tolist())), clocks=clk, ok=ok, e2e=e2e, units=units,
                R=R, ns=ns, P=P, n_rec=n_rec, spans=ctx.n_spans(n_rec * R), L=ctx.L, suffix=suffix, codec=codec, k1024=k1024,
                lossy=lossy, weighted=weighted, llama=llama)


def roofline(res, peaks, launches_traffic=None):
    cfg = res["cfg"]
    ph = res["phase"]
    D, H = cfg.dim, cfg.n_heads
    nvec = cfg.batch * cfg.n_layers * H * res["P"]
    flops_k = nvec * cfg.stages_k * 2 * D * 256
    flops_v = nvec * cfg.stages_v * 2 * D * 256
    rvq_ms = ph["rvq_k"] + ph["rvq_v"]
    rvq_tf = (flops_k + flops_v) / (rvq_ms * 1e-3) / 1e12
    symbols = res["ns"] * res["P"] * res["R"]
    spans = res["ns"] * res["P"] * res["R"] // res["L"]
    enc_bytes = symbols + spans * 16
    out_bytes = res["ns"] * res["n_rec"] * 2 * H * D * cfg.elem_bytes
    dec_bytes = res["ns"] * res["n_rec"] * res["R"] * 1 + res["spans"] * res["ns"] * 16 + out_bytes
    sm_mhz = res["clocks"].get("sm_mhz") or 1900.0
    fp64_peak = FP64_OPS_PER_CLK_SM * 152 * sm_mhz * 1e6
    kernels = {
        "rvq (tcgen05)": {"bound": "tensor", "achieved_tflops": rvq_tf, "ms": rvq_ms,
                          "frac": rvq_tf / peaks["bf16_tflops"]},
        "span_encode": {"bound": "fp64", "ms": ph["span_encode"],
                        "achieved_gbs": enc_bytes / (ph["span_encode"] * 1e-3) / 1e9,
                        "frac_hbm": enc_bytes / (ph["span_encode"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                        "frac_fp64": symbols * 6 / (ph["span_encode"] * 1e-3) / fp64_peak},
        "decode_kv (decode + gather)": {"bound": "hbm", "ms": ph["decode_kv"],
                                        "achieved_gbs": dec_bytes / (ph["decode_kv"] * 1e-3) / 1e9,
                                        "frac": dec_bytes / (ph["decode_kv"] * 1e-3) / 1e9 / peaks["hbm_gbs"]},
    }
    dominant = {
        "bound": "tensor", "achieved": rvq_tf, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
        "frac": rvq_tf / peaks["bf16_tflops"], "traffic": launches_traffic,
        "kernel": "k_rvq64 (RVQ assignment), algorithmic 2*64*256 flop per vector-stage, %s peak (fp16 dense = bf16 rate)"
                  % ("of measured" if peaks["source"] == "measured" else "of fallback"),
    }
    return dominant, kernels, dec_bytes, out_bytes


# ----------------------------------------------------------- CPU oracle ---
def oracle_sample(budget_s, cfg=synth.CFG1, max_streams=None):
    """The float64 oracle on whole (sequence, layer) streams of the workload
    until `budget_s` seconds of work: RVQ, serialisation, span encode, append,
    decode, reconstruction and random reads."""
    import oracle
    oracle.build()
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    r = oracle.packing_ratio(256)
    L = oracle.max_span_len(r)
    H = cfg.n_heads
    P = cfg.n_archived
    streams = [(b, l) for b in range(cfg.batch) for l in range(cfg.n_layers)]
    done = 0
    t_work = 0.0
    rng = np.random.default_rng(1)
    for (b, l) in streams:
        if max_streams is not None and done >= max_streams:
            break
        pos = np.arange(cfg.t0, cfg.t1 + 1)                      # archived + appended position
        hh, tt = np.meshgrid(np.arange(H), pos, indexing="ij")
        Kx = synth.storage_to_f64(synth.kv_elements(cfg, 0, l, b, hh, tt), cfg.dtype)
        Vx = synth.storage_to_f64(synth.kv_elements(cfg, 1, l, b, hh, tt), cfg.dtype)
        t_start = time.perf_counter()
        ik = np.stack([oracle.rvq_encode(Kx[h], cbk[l, h])[0] for h in range(H)])
        iv = np.stack([oracle.rvq_encode(Vx[h], cbv[l, h])[0] for h in range(H)])
        stream = oracle.records_from_indices(ik[:, :P], iv[:, :P])
        pts = oracle.span_encode(stream, 256, r, L)
        tail = oracle.records_from_indices(ik[:, P:], iv[:, P:])
        pts = oracle.append(stream, tail, 256, r, L)
        full = np.concatenate([stream, tail])
        dec, _, bad = oracle.span_decode(pts, full.size, 256, r, L)
        k2, v2 = oracle.indices_from_records(dec, H, cfg.stages_k, cfg.stages_v)
        for h in range(H):
            oracle.round_to(oracle.rvq_decode(k2[h], cbk[l, h]), cfg.dtype)
            oracle.round_to(oracle.rvq_decode(v2[h], cbv[l, h]), cfg.dtype)
        reads = rng.integers(0, full.size, N_READS // len(streams) + 1)
        oracle.read(pts, full.size, reads, 256, r, L)
        t_work += time.perf_counter() - t_start
        done += 1
        if t_work >= budget_s:
            break
    records = done * (P + 1)
    return records / t_work, done, t_work, oracle.threads()


def cpu_desc():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True).stdout
        for ln in out.splitlines():
            if ln.startswith("Model name"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    return "unknown"


# ---------------------------------------------------------------- main ----
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="fkv", choices=["fkv", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-suffix", action="store_true")
    ap.add_argument("--no-k1024", action="store_true")
    ap.add_argument("--no-lossy", action="store_true")
    ap.add_argument("--no-codec", action="store_true")
    ap.add_argument("--no-weighted", action="store_true")
    ap.add_argument("--no-llama", action="store_true")
    ap.add_argument("--llama-seq", type=int, default=synth.CFG3.seq,
                    help="positions of the Llama-shaped cache (a shorter one for profiling captures)")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--no-cpu", action="store_true")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        per_step = max(1.0, 150.0 / (args.steps + args.warmup))
        for _ in range(args.warmup):
            oracle_sample(per_step / 4, max_streams=1)
        vals = []
        tot_rec = tot_t = 0.0
        cores = 1
        for _ in range(args.steps):
            v, done, t, cores = oracle_sample(per_step)
            vals.append(v)
            tot_rec += v * t
            tot_t += t
        value = tot_rec / tot_t
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot_t / args.steps * 1e3,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic",
                "config": {"workload": "gpt2-shaped full KV cache: 12 layers x batch 8 x 12 heads x 1024 tok x 64, fp16; "
                                       "K 4 / V 2 RVQ stages x 256; N=256, r=r_256, L=6; bounded sample of whole "
                                       "(sequence, layer) streams per step", "sample": "whole streams"},
                "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                                 "sample": "whole (sequence, layer) streams, %.0f s of oracle work per step" % per_step,
                                 "cpu": cpu_desc()},
                "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import torch
    if world > 1:
        torch.distributed.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    res = run_gpu(args, rank, world, local_rank)
    ms = res["ms"]
    if world > 1:
        ms, e2e_ms = max_over_ranks([ms, res["e2e"]["ms"] if res["e2e"] else 0.0], "cuda")
        if res["e2e"]:
            res["e2e"]["ms"] = e2e_ms
    if rank != 0:
        torch.distributed.destroy_process_group()
        return
    peaks = load_peaks()
    dominant, kernels, dec_bytes, out_bytes = roofline(res, peaks, RVQ_DRAM_BYTES_PER_LAUNCH)
    if res["suffix"]:
        sx = res["suffix"]
        gbs = sx["bytes"] / (sx["ms"] * 1e-3) / 1e9
        kernels["suffix_search (Sec. 5)"] = {"bound": "hbm", "ms": sx["ms"], "achieved_gbs": gbs,
                                             "frac": gbs / peaks["hbm_gbs"], "matches": sx["matches"],
                                             "candidates": sx["candidates"], "workload": sx["workload"]}
    if res["codec"]:
        fp64_peak = FP64_OPS_PER_CLK_SM * 152 * (res["clocks"].get("sm_mhz") or 1900.0) * 1e6
        per_n = {}
        for N, cx in res["codec"].items():
            syms = 4 * (1 << 28)
            nbytes = syms + 4 * cx["spans"] * 16          # 1 B per symbol + one 16 B point per span
            per_n["N=%d" % N] = {
                "L": cx["L"],
                "encode_ms": cx["encode_ms"], "encode_symbols_per_s": syms / (cx["encode_ms"] * 1e-3),
                "encode_frac_hbm": nbytes / (cx["encode_ms"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                "encode_frac_fp64": syms * 6 / (cx["encode_ms"] * 1e-3) / fp64_peak,
                "decode_ms": cx["decode_ms"], "decode_symbols_per_s": syms / (cx["decode_ms"] * 1e-3),
                "decode_frac_hbm": nbytes / (cx["decode_ms"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                "read_ms": cx["read_ms"], "reads_per_s": cx["reads"] / (cx["read_ms"] * 1e-3),
                "exact": cx["exact"], "status_ok": cx["ok"]}
        kernels["span codec, symbol stress"] = {
            "workload": "4 streams x 2^28 seeded uniform symbols per N; full encode, full decode, 2^20 seeded "
                        "random reads per stream; all decoded and read symbols checked equal to the input",
            "encode_bound": "fp64", "decode_bound": "integer ALU", "read_bound": "latency", "per_N": per_n}
    if res["k1024"]:
        kx = res["k1024"]
        rvq_ms = kx["rvq_k"] + kx["rvq_v"]
        flops = kx["nvec"] * sum(kx["stages"]) * 2 * 64 * 1024
        tf = flops / (rvq_ms * 1e-3) / 1e12
        dec_b = res["ns"] * kx["P"] * kx["R"] * 2 + res["ns"] * (-(-kx["P"] * kx["R"] // kx["L"])) * 16 + kx["out_bytes"]
        kernels["pooled RVQ 1024 x 2 archive (Table 2)"] = {
            "workload": "gpt2-shaped full KV cache (12 layers x batch 8 x 12 heads x 1024 tok x 64, fp16), one "
                        "1024-codeword codebook per layer and stage shared by all heads, K 2 / V 2 stages; "
                        "uint16 symbols, N=1024, r=r_1024, L=5",
            "rvq_ms": rvq_ms, "bound": "tensor", "achieved_tflops": tf, "frac": tf / peaks["bf16_tflops"],
            "span_encode_ms": kx["span_encode"], "decode_kv_ms": kx["decode_kv"],
            "decode_kv_gbs": dec_b / (kx["decode_kv"] * 1e-3) / 1e9,
            "decode_kv_frac": dec_b / (kx["decode_kv"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "archived_positions_per_s": res["ns"] * kx["P"] / ((rvq_ms + kx["span_encode"]) * 1e-3),
            "status_ok": kx["ok"]}
    if res["lossy"]:
        lx = res["lossy"]
        tb = lx["point_bytes"] + lx["code_bytes"]             # points read, codes written
        kernels["lossy archive (Sec. 4)"] = {
            "workload": "this step's 96 streams x 989 records x 72 symbols (N=256, span 6); spans older than the "
                        "last %d truncated to %d bits per coordinate" % (lx["keep"], lx["bits"]),
            "truncate_ms": lx["truncate"], "truncate_bound": "hbm",
            "truncate_gbs": tb / (lx["truncate"] * 1e-3) / 1e9,
            "truncate_frac": tb / (lx["truncate"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "decode_ms": lx["decode"], "decode_bound": "fp64 (binary64 walk with IEEE division, as the paper)",
            "decode_symbols_per_s": lx["symbols"] / (lx["decode"] * 1e-3),
            "archive_bytes": lx["code_bytes"] + lx["tail_bytes"], "exact_archive_bytes": lx["point_bytes"],
            "symbol_error_rate_truncated_spans": lx["sym_err_truncated"], "status_ok": lx["ok"]}
    if res["llama"]:
        lx = res["llama"]
        ph3 = lx["phase"]
        rvq3 = ph3[0] + ph3[1]
        tf3 = lx["nvec"] * sum(lx["stages"]) * 2 * 128 * 256 / (rvq3 * 1e-3) / 1e12
        sym3 = lx["records"] * lx["R"]
        dec3 = sym3 + lx["spans"] * 16 + lx["out_bytes"]
        kernels["llama3-8b-shaped archive (config 3)"] = {
            "workload": "32 layers x batch 4 x 8 KV heads x %d tok x 128 dims, bf16; 4+32 exact window; K 4 / V 2 "
                        "RVQ stages x 256; N=256, r=r_256, L=6" % args.llama_seq,
            "records_per_s": lx["records"] / (sum(ph3) * 1e-3), "step_ms": sum(ph3),
            "rvq_ms": rvq3, "rvq_tflops": tf3, "rvq_frac": tf3 / peaks["bf16_tflops"],
            "rvq_kernel": "k_rvq128 (persistent, two tile slots, codebook streamed in 64-dim K blocks)",
            "span_encode_ms": ph3[2], "span_encode_frac_fp64": sym3 * 6 / (ph3[2] * 1e-3) /
            (FP64_OPS_PER_CLK_SM * 152 * (res["clocks"].get("sm_mhz") or 1900.0) * 1e6),
            "decode_kv_ms": ph3[3], "decode_kv_gbs": dec3 / (ph3[3] * 1e-3) / 1e9,
            "decode_kv_frac": dec3 / (ph3[3] * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "read_kv_ms_4096": ph3[4], "status_ok": lx["ok"]}
    if res["weighted"]:
        wx = res["weighted"]
        kernels["probability-weighted maps (Sec. 6)"] = {
            "workload": "this step's 96 archived RVQ index streams (989 records x 72 symbols, N=256), adaptive "
                        "add-one model, one warp per stream",
            "encode_ms": wx["encode"], "decode_ms": wx["decode"], "bound": "latency (sequential within a stream)",
            "encode_symbols_per_s": wx["symbols"] / (wx["encode"] * 1e-3),
            "decode_symbols_per_s": wx["symbols"] / (wx["decode"] * 1e-3),
            "bits_per_symbol": wx["bits"] / wx["symbols"], "uniform_bits_per_symbol": 8.0,
            "lossless": wx["exact"], "status_ok": wx["ok"]}
    units = res["units"] * world
    value = units / (ms * 1e-3)
    cpu = None
    if world == 1 and not args.no_cpu:
        v, done, t, cores = oracle_sample(args.cpu_budget)
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": "%d whole (sequence, layer) streams of the workload (%d records), %.1f s" %
                         (done, done * res["n_rec"], t), "cpu": cpu_desc()}
    e2e = None
    if res["e2e"]:
        e2e = {"value": units / (res["e2e"]["ms"] * 1e-3), "unit": UNIT,
               "h2d_bytes_per_step": res["e2e"]["h2d"], "d2h_bytes_per_step": res["e2e"]["d2h"],
               "ms_per_step": res["e2e"]["ms"]}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "fp16 in / fp16-split tensor / f64 codec", "data": "synthetic",
        "config": {"workload": "gpt2-shaped full KV cache: 12 layers x batch 8 x 12 heads x 1024 tok x 64 dims, "
                               "fp16; 4+32 exact window; K 4 / V 2 RVQ stages x 256; N=256, r=r_256, L=6",
                   "records_per_step": res["units"], "global_batch": 8 * world, "seq_len": 1024,
                   "l2": "inputs (302 MB) larger than L2; no flush", "parallelism": "replicas (weak)"},
        "decoded_kv_gbs": out_bytes / (res["phase"]["decode_kv"] * 1e-3) / 1e9,
        "write_positions_per_s": res["units"] / ((res["phase"]["rvq_k"] + res["phase"]["rvq_v"]
                                                 + res["phase"]["span_encode"]) * 1e-3),
        "phase_ms": res["phase"],
        "roofline": dominant,
        "kernels": kernels,
        "cpu_baseline": cpu,
        "e2e": e2e,
        # per step: k_rvq64 x4 (K and V archive, K and V of the appended
        # position), k_span_encode x2 (archive, tail append),
        # k_span_decode_planar, k_gather x2, k_read_kv (as the ncu launch list shows)
        "gpu_launches": 10 * args.steps,
        "clocks": res["clocks"],
        "status_ok": res["ok"],
    }
    print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
