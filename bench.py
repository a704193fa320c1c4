#!/usr/bin/env python
"""Throughput of the fractal KV-cache archive path on one GB300.

Headline workload: a Llama-3-8B-shaped KV cache -- 32 layers x 4 sequences x
8 KV heads x 32768 positions x 128 dims, bf16, synthetic (seeded Irwin-Hall
values with log-normal channel scales and 3 outlier key channels per head),
per-head RVQ codebooks with 4 key stages and 2 value stages of 256 codewords,
alphabet N = 256 at r = r_256, span length 6.  It is the largest of the
single-GPU configurations (17.2 GB of K/V).

One step is one pass of the whole archive path over that cache:
  1. exact-window split: positions [4, 32736) of every (layer, sequence)
     leave the 4-sink + 32-recent window and are archived;
  2. RVQ assignment of their K and V head vectors into token records;
  3. span encoding of the 128 (sequence, layer) symbol streams (append from
     empty into library-owned streams);
  4. decode-time append: position 32736 leaves the window -> RVQ + tail append;
  5. full decode of the archive and reconstruction of K/V at [4, 32737);
  6. 4096 random record reads (K and V of all heads of one position).
value = archived KV records (sequence x layer x position) per second over the
whole step.  Inputs (17.2 GB) are far larger than L2, so no flush is needed.
`e2e` times the same step through the public API with the caches in pinned
host memory: every step copies the archived positions in (fkv_cache_upload)
and reads its results (archive points, record reads) back.

The line also carries, each measured on its own after the timed region:
  parity   the headline step's outputs for the oracle's sample streams against
           the oracle (RVQ indices under the 1e-4 gap rule, stored points bit
           for bit, rebuilt K/V under the rounding rule), with near-tie counts;
  fp64     binary64 add/mul throughput measured by independent chains (the
           span encoder's roofline denominator), next to the nominal figure;
and under "kernels" the secondary workloads (a --no-<name> flag skips one):
  gpt2     the GPT-2-shaped full cache (12 layers x 8 x 12 heads x 1024 x 64,
           fp16, K 4 / V 2 stages), the same step on 64-dimensional heads;
  stream   decode-time streaming: 64 Llama-shaped sequences with 131072
           archived positions each; per step one appended position per
           sequence and 4096 random record reads per sequence;
  suffix   Sec. 5 retrieval over 4 streams x 2^28 symbols;
  codec    the span codec on the symbol-stress streams (N = 3, 4, 16, 256);
  k1024    Table 2's pooled RVQ 1024 x 2 archive of the GPT-2 cache;
  lossy    Sec. 4 truncation and lossy decode of the GPT-2 step's streams;
  weighted Sec. 6 probability-weighted maps of the GPT-2 step's index streams.

--impl reference times the float64 CPU oracle on a bounded sample of the same
workload (the paper ships no GPU implementation; the oracle is the reference).
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import threading
import time
import types

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "archived KV positions/s (RVQ+span encode) and decoded KV GB/s, % of roofline"
UNIT = "archived KV positions/s"
N_READS = 4096
HEADLINE = synth.CFG3
WORKLOAD = ("llama3-8b-shaped KV cache: 32 layers x batch 4 x 8 KV heads x 32768 tok x 128 dims, bf16; 4+32 exact "
            "window; K 4 / V 2 RVQ stages x 256 per head; N=256, r=r_256, L=6")


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per RVQ launch of
# the headline workload, from ncu captures of the current k_rvq128 on the same
# cache cut to 4096 and to 8192 archived positions (the full cache is too large
# for a multi-metric capture): key launch 1,340,126,208 and 2,458,886,400 B,
# value launch 1,209,800,960 and 2,317,281,024 B.  Traffic is a fixed part (the
# codebooks) plus a part that grows with the positions, so the two lengths fix
# a line, extrapolated to the headline length; the figure is the mean of the
# key and value launches.  Set it to None when k_rvq128 changes until it is
# captured again.
RVQ_TRAFFIC_CAPTURES = ((4096, 8192), ((1340126208, 2458886400), (1209800960, 2317281024)))


def _rvq_traffic_full(positions=None, captures=RVQ_TRAFFIC_CAPTURES):
    (p1, p2), launches = captures
    p = HEADLINE.n_archived if positions is None else positions
    full = [b1 + (b2 - b1) * (p - p1) / (p2 - p1) for b1, b2 in launches]
    return sum(full) / len(full)


RVQ_DRAM_BYTES_PER_LAUNCH = _rvq_traffic_full()

# GB300's nominal HBM3e bandwidth (the measured copy bandwidth is the roofline's
# denominator; this one is reported beside it).
HBM_NOMINAL_GBS = 7900.0

# Nominal FP64 add/mul rate: GB300's 1.25 TFLOP/s of FP64 FMA is 625 G add or
# mul instructions per second at the 2070 MHz boost clock (1.99 per clock per
# SM); the measured rate (fkv_measure_fp64_rate) is reported beside it.
FP64_NOMINAL_OPS_PER_CLK_SM = 1.25e12 / 2 / (152 * 2070e6)


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
def rank_workload(rank: int, base=HEADLINE):
    """One rank's replica of the workload: the base configuration with its own
    seed (rank 0 runs the base configuration itself); the archive shards by
    (sequence, layer) stream, so ranks share nothing but the codebooks."""
    return dataclasses.replace(base, cfg_id=base.cfg_id + 1000 * rank) if rank else base


def max_over_ranks(values, device):
    """Element-wise maximum of per-rank timings over all ranks (one
    all_reduce; the job's time is its slowest rank's)."""
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


# ------------------------------------------------------- archive step ----
PHASES = ["rvq_k", "rvq_v", "span_encode", "append_rvq", "append", "decode_kv", "read_kv"]


def archive_state(fkv, cfg, cb_cfg, dev, seed=7, K=None, V=None):
    """Buffers and the step closure of one pass of the archive path over the
    cache of `cfg` (codebooks of `cb_cfg`): RVQ of the archived positions,
    span encoding into library-owned streams, the decode-time append of the
    position leaving the window, the full decode with reconstruction, and
    N_READS random record reads."""
    import torch
    g = types.SimpleNamespace(cfg=cfg)
    g.K = synth.gpu_kv_cache(cfg, 0, device=dev) if K is None else K
    g.V = synth.gpu_kv_cache(cfg, 1, device=dev) if V is None else V
    g.ctx = fkv.Context(256, codebooks=(synth.codebooks(cb_cfg, 0), synth.codebooks(cb_cfg, 1)))
    g.R = g.ctx.record_len()
    g.ns = cfg.batch * cfg.n_layers
    g.t0, g.t1 = cfg.t0, cfg.t1
    g.P = g.t1 - g.t0
    g.n_rec = g.P + 1                               # + the appended position t1
    g.sym = torch.empty((g.ns, g.P * g.R), dtype=torch.uint8, device=dev)
    g.rec = torch.empty((g.ns, g.R), dtype=torch.uint8, device=dev)
    g.st = fkv.Streams(g.ctx, g.ns, capacity=g.n_rec * g.R)
    g.Kr = torch.zeros_like(g.K)
    g.Vr = torch.zeros_like(g.V)
    gen = torch.Generator().manual_seed(seed)
    g.req = torch.stack([torch.randint(0, g.ns, (N_READS,), generator=gen),
                         torch.randint(0, g.n_rec, (N_READS,), generator=gen)], dim=1).to(dev)
    g.out = torch.empty((N_READS, 2, cfg.n_heads, cfg.dim), dtype=g.K.dtype, device=dev)
    g.stream = torch.cuda.current_stream()
    g.ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(PHASES) + 1)]
    g.spans = g.ctx.n_spans(g.n_rec * g.R)

    def step(record=False, K=None, V=None, st=None, out=None):
        K = g.K if K is None else K
        V = g.V if V is None else V
        st = g.st if st is None else st
        out = g.out if out is None else out
        e = iter(g.ev) if record else None
        mark = (lambda: next(e).record(g.stream)) if record else (lambda: None)
        mark()
        g.ctx.rvq_encode(0, K, g.t0, g.t1, g.sym)
        mark()
        g.ctx.rvq_encode(1, V, g.t0, g.t1, g.sym)
        mark()
        st.reset()
        st.append(g.sym)
        mark()
        g.ctx.rvq_encode(0, K, g.t1, g.t1 + 1, g.rec)
        g.ctx.rvq_encode(1, V, g.t1, g.t1 + 1, g.rec)
        mark()
        st.append(g.rec)
        mark()
        g.ctx.decode_kv(st.points(), g.n_rec, g.Kr, g.Vr, t0=g.t0)
        mark()
        g.ctx.read_kv(st.points(), g.n_rec, g.req, out)
        mark()
    g.step = step
    return g


def phase_times(g, reps):
    """Mean per-phase durations (CUDA events on the launching stream)."""
    import torch
    acc = np.zeros(len(PHASES))
    for _ in range(reps):
        g.step(record=True)
        torch.cuda.synchronize()
        acc += np.array([g.ev[i].elapsed_time(g.ev[i + 1]) for i in range(len(PHASES))])
    return dict(zip(PHASES, (acc / reps).tolist()))


def archive_rates(cfg, phase, R, P, n_rec, spans, ns, peaks, fp64_ops_per_s):
    """Algorithmic rates of one archive step's kernels (all fixed by the
    method and the workload's shape): RVQ 2*D*256 flop per vector and stage;
    span encode 1 B in per symbol + 16 B per span out and 6 binary64
    operations per symbol; the archive read 1 B per symbol + 16 B per span in
    and the rebuilt K/V out."""
    D, H = cfg.dim, cfg.n_heads
    nvec = cfg.batch * cfg.n_layers * H * P
    flops = nvec * (cfg.stages_k + cfg.stages_v) * 2 * D * 256
    rvq_ms = phase["rvq_k"] + phase["rvq_v"]
    rvq_tf = flops / (rvq_ms * 1e-3) / 1e12
    symbols = ns * P * R
    enc_bytes = symbols + ns * (-(-P * R // 6)) * 16
    out_bytes = ns * n_rec * 2 * H * D * cfg.elem_bytes
    dec_bytes = ns * n_rec * R + ns * spans * 16 + out_bytes
    enc_fp64 = symbols * 6 / (phase["span_encode"] * 1e-3)
    return {
        "rvq": {"bound": "tensor", "ms": rvq_ms, "flops": flops, "achieved_tflops": rvq_tf,
                "frac": rvq_tf / peaks["bf16_tflops"]},
        "span_encode": {"bound": "fp64", "ms": phase["span_encode"],
                        "achieved_gbs": enc_bytes / (phase["span_encode"] * 1e-3) / 1e9,
                        "frac_hbm": enc_bytes / (phase["span_encode"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                        "fp64_ops_per_s": enc_fp64,
                        "frac_fp64_measured": enc_fp64 / fp64_ops_per_s["measured"]
                        if fp64_ops_per_s.get("measured") else None,
                        "frac_fp64_nominal": enc_fp64 / fp64_ops_per_s["nominal"]},
        "decode_kv": {"bound": "hbm", "ms": phase["decode_kv"], "bytes": dec_bytes,
                      "achieved_gbs": dec_bytes / (phase["decode_kv"] * 1e-3) / 1e9,
                      "frac": dec_bytes / (phase["decode_kv"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                      # against GB300's nominal 7.9 TB/s as well as the measured copy
                      "frac_nominal": dec_bytes / (phase["decode_kv"] * 1e-3) / 1e9 / HBM_NOMINAL_GBS},
        "out_bytes": out_bytes,
    }


def roofline(rates, peaks, traffic, kernel_name):
    """The line's roofline object: the dominant kernel (RVQ assignment on the
    tensor cores) against the measured dense bf16 peak (fp16 dense runs at
    the bf16 rate)."""
    r = rates["rvq"]
    return {"bound": "tensor", "achieved": r["achieved_tflops"], "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
            "frac": r["achieved_tflops"] / peaks["bf16_tflops"], "traffic": traffic,
            "kernel": "%s, algorithmic 2*D*256 flop per vector-stage, %s peak (burst)"
                      % (kernel_name, "of measured" if peaks["source"] == "measured" else "of fallback")}


# ---------------------------------------------------------------- GPU arm --
def run_gpu(args, rank, world, local_rank):
    import torch
    import paper_2607_07144_gb300 as fkv

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    base = HEADLINE if args.seq == HEADLINE.seq else synth.small_config(
        HEADLINE, HEADLINE.cfg_id, n_layers=HEADLINE.n_layers, batch=HEADLINE.batch, seq=args.seq)
    cfg = rank_workload(rank, base)
    g = archive_state(fkv, cfg, base, dev, seed=7 + rank)      # codebooks replicated over ranks
    stream = g.stream

    for _ in range(args.warmup):
        g.step()
    torch.cuda.synchronize()
    if g.ctx.sync_status() != 0:
        raise RuntimeError("device status error during warm-up")
    phase = phase_times(g, max(1, min(args.steps, 5)))

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
        g.step()
    stop.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    ms = start.elapsed_time(stop) / args.steps
    clk = clocks.stop()
    ok = g.ctx.sync_status() == 0

    e2e = None if args.no_e2e else run_e2e(fkv, g, args, dev, world)
    g.step()                                           # the outputs the parity check reads
    torch.cuda.synchronize()
    parity_src = None
    if world == 1 and not args.no_cpu:
        parity_src = gpu_sample(g, oracle_streams(cfg))

    fp64 = {"nominal": FP64_NOMINAL_OPS_PER_CLK_SM * 152 * (clk.get("sm_mhz") or 2070.0) * 1e6}
    if not args.no_fp64:
        fp64["measured"] = fkv.measure_fp64_rate()
    res = dict(cfg=cfg, ms=ms, phase=phase, clocks=clk, ok=ok, e2e=e2e, units=g.ns * g.n_rec, R=g.R, ns=g.ns,
               P=g.P, n_rec=g.n_rec, spans=g.spans, fp64=fp64, parity_src=parity_src)
    del g
    torch.cuda.empty_cache()

    res["gpt2"] = None if args.no_gpt2 else run_gpt2(fkv, args, dev, rank)
    torch.cuda.empty_cache()
    res["stream"] = None if args.no_stream else run_stream(fkv, args, dev)
    torch.cuda.empty_cache()
    res["secondary"] = run_secondary(fkv, args, dev, res["gpt2"])
    return res


def run_e2e(fkv, g, args, dev, world):
    """The step through the public API with host buffers: every step copies
    the positions that leave the exact window in from pinned host memory
    (fkv_cache_upload) and reads its results (the archive points and the
    record reads) back; steps are pipelined over three streams (copy in,
    compute, copy out) with double-buffered device inputs and archives, as a
    serving loop runs them.  The rebuilt K/V stays on the device, where
    attention consumes it."""
    import torch
    stream = g.stream
    Kh = g.K.cpu().pin_memory()
    Vh = g.V.cpu().pin_memory()
    Kd, Vd = [g.K, torch.empty_like(g.K)], [g.V, torch.empty_like(g.V)]
    sts = [g.st, fkv.Streams(g.ctx, g.ns, capacity=g.n_rec * g.R)]
    outs = [g.out, torch.empty_like(g.out)]
    ptsh = [torch.empty((g.ns, g.spans, 2), dtype=torch.float64).pin_memory() for _ in range(2)]
    outh = [torch.empty(g.out.shape, dtype=g.out.dtype).pin_memory() for _ in range(2)]
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
            g.ctx.cache_upload(Kh, Kd[b], g.t0, g.t1 + 1, stream=s_in)
            g.ctx.cache_upload(Vh, Vd[b], g.t0, g.t1 + 1, stream=s_in)
            ev_in = torch.cuda.Event()
            ev_in.record(s_in)
        stream.wait_event(ev_in)
        if read[b] is not None:
            stream.wait_event(read[b])
        g.step(K=Kd[b], V=Vd[b], st=sts[b], out=outs[b])
        done = torch.cuda.Event()
        done.record(stream)
        free[b] = done
        with torch.cuda.stream(s_out):
            s_out.wait_event(done)
            ptsh[b].copy_(sts[b].points()[:, :g.spans], non_blocking=True)
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
    h2d = Kh[:, :, :, g.t0:g.t1 + 1].numel() * Kh.element_size() * 2
    d2h = ptsh[0].numel() * 8 + outh[0].numel() * outh[0].element_size()
    ok = g.ctx.sync_status() == 0
    # the host link on its own: one pinned host -> device copy of the key cache
    flat_h, flat_d = Kh.view(-1), Kd[1].view(-1)
    with torch.cuda.stream(stream):
        for _ in range(2):
            flat_d.copy_(flat_h, non_blocking=True)
        torch.cuda.synchronize()
        s2.record(stream)
        flat_d.copy_(flat_h, non_blocking=True)
        t2.record(stream)
    torch.cuda.synchronize()
    link_gbs = flat_h.numel() * flat_h.element_size() / (s2.elapsed_time(t2) * 1e-3) / 1e9
    del Kh, Vh, Kd, Vd, sts, outs, ptsh, outh, flat_h, flat_d
    return {"ms": e2e_ms, "h2d": h2d, "d2h": d2h, "ok": ok, "link_gbs": link_gbs}


def oracle_streams(cfg, count=8):
    """The (sequence, layer) streams the oracle samples, in order: first and
    last, then seeded others."""
    all_ = [(b, l) for b in range(cfg.batch) for l in range(cfg.n_layers)]
    first = [all_[0], all_[-1]]
    rng = np.random.default_rng(2607)
    rest = [all_[i] for i in rng.permutation(len(all_)) if all_[i] not in first]
    return (first + rest)[:count]


def gpu_sample(g, streams):
    """Host copies of the headline step's inputs and outputs for the sampled
    streams: K/V inputs, token records, stored points, rebuilt K/V."""
    cfg = g.cfg
    out = []
    pts = g.st.points()
    for (b, l) in streams:
        i = b * cfg.n_layers + l
        out.append({"b": b, "l": l,
                    "K": g.K[l, b, :, g.t0:g.t1 + 1].cpu(), "V": g.V[l, b, :, g.t0:g.t1 + 1].cpu(),
                    "sym": np.concatenate([g.sym[i].cpu().numpy(), g.rec[i].cpu().numpy()]),
                    "pts": pts[i, :g.spans].cpu().numpy(),
                    "Kr": g.Kr[l, b, :, g.t0:g.t1 + 1].cpu(), "Vr": g.Vr[l, b, :, g.t0:g.t1 + 1].cpu()})
    return out


# ------------------------------------------------------- secondary: GPT-2 --
def run_gpt2(fkv, args, dev, rank):
    """The same archive step on the GPT-2-shaped full cache (64-dimensional
    heads, fp16): its own warm-up and timed loop."""
    import torch
    c1 = rank_workload(rank, synth.CFG1)
    g = archive_state(fkv, c1, synth.CFG1, dev, seed=11 + rank)
    for _ in range(args.warmup):
        g.step()
    phase = phase_times(g, 5)
    reps = max(args.steps, 10)
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(g.stream)
    for _ in range(reps):
        g.step()
    e.record(g.stream)
    torch.cuda.synchronize()
    g.ms = s.elapsed_time(e) / reps
    g.phase = phase
    g.ok = g.ctx.sync_status() == 0
    return g


# ---------------------------------------------- secondary: streaming -----
def run_stream(fkv, args, dev):
    """Decode-time streaming: 64 Llama-shaped sequences (32 layers, 8 KV
    heads, 128 dims), each (sequence, layer) stream prefilled with 131072
    archived records; then per step, for every sequence, the position leaving
    the exact window is RVQ-encoded and appended (2048 records), and 4096
    seeded random records per sequence are read back (262,144 reads of K and
    V of all heads, 4 KB each).  The prefill's archived values do not change
    the cost of an append or a read, so it is written from seeded index
    streams; the RVQ-prefilled archive at full size is checked against a full
    decode in the tests."""
    import torch
    c4 = synth.CFG4
    ctx = fkv.Context(256, codebooks=(synth.codebooks(c4, 0), synth.codebooks(c4, 1)))
    R = ctx.record_len()
    ns = c4.batch * c4.n_layers
    pre = synth.CFG4_PREFILL
    steps_total = min(synth.CFG4_STEPS, args.stream_steps + args.warmup)
    st = fkv.Streams(ctx, ns, capacity=(pre + steps_total) * R)
    sym = synth.gpu_symbols(256, "uniform", ns, pre * R, device=dev, cfg_id=c4.cfg_id)   # 12.9 GB
    st.append(sym)
    del sym
    torch.cuda.synchronize()
    t_new = c4.t0 + pre                                # positions leaving the window, one per step
    Kn = synth.gpu_kv_cache(c4, 0, device=dev, t0=t_new, count=steps_total)
    Vn = synth.gpu_kv_cache(c4, 1, device=dev, t0=t_new, count=steps_total)
    rec = torch.empty((ns, R), dtype=torch.uint8, device=dev)
    gen = torch.Generator().manual_seed(44)
    n_reads = 4096 * c4.batch
    b = torch.randint(0, c4.batch, (n_reads,), generator=gen)
    l = torch.randint(0, c4.n_layers, (n_reads,), generator=gen)
    req = torch.stack([b * c4.n_layers + l, torch.randint(0, pre, (n_reads,), generator=gen)], 1).to(dev)
    out = torch.empty((n_reads, 2, c4.n_heads, c4.dim), dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    acc = np.zeros(3)
    timed = 0
    for i in range(steps_total):
        rec_ = i >= args.warmup
        if rec_:
            ev[0].record(stream)
        ctx.rvq_encode(0, Kn, i, i + 1, rec)
        ctx.rvq_encode(1, Vn, i, i + 1, rec)
        if rec_:
            ev[1].record(stream)
        st.append(rec)
        if rec_:
            ev[2].record(stream)
        ctx.read_kv(st.points(), pre + i + 1, req, out)
        if rec_:
            ev[3].record(stream)
            torch.cuda.synchronize()
            acc += np.array([ev[k].elapsed_time(ev[k + 1]) for k in range(3)])
            timed += 1
    ok = ctx.sync_status() == 0
    acc /= max(timed, 1)
    res = {"steps": timed, "append_rvq_ms": acc[0], "append_ms": acc[1], "read_ms": acc[2],
           "step_us": acc.sum() * 1e3, "reads": n_reads, "appended_records": ns, "ok": ok,
           "read_bytes_in": 8 * 16, "read_bytes_out": 2 * c4.n_heads * c4.dim * 2,
           "archive_bytes": ns * ctx.n_spans((pre + steps_total) * R) * 16}
    del st, Kn, Vn, out, req
    return res


# ------------------------------------------------- secondary workloads ----
def run_secondary(fkv, args, dev, g):
    """The other rows' workloads, each measured on its own; lossy and weighted
    run on the GPT-2 step's streams (g)."""
    import torch
    stream = torch.cuda.current_stream()
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
    if not args.no_lossy and g is not None:
        ctx, st, sym, R, ns, n_rec, step = g.ctx, g.st, g.sym, g.R, g.ns, g.n_rec, g.step
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
    if not args.no_weighted and g is not None:
        ctx, sym = g.ctx, g.sym
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
        ns5 = c5.batch * c5.n_layers
        sym5 = torch.empty((ns5, P5 * R5), dtype=kctx.sym_dtype, device=dev)
        pts5 = torch.empty((ns5, kctx.n_spans(P5 * R5), 2), dtype=torch.float64, device=dev)
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
                 "nvec": ns5 * c5.n_heads * P5, "ns": ns5, "stages": (c5.stages_k, c5.stages_v), "R": R5, "P": P5, "L": kctx.L,
                 "ok": kctx.sync_status() == 0,
                 "out_bytes": 2 * K5.numel() // c5.seq * P5 * K5.element_size()}
        del K5, V5, K5r, V5r, sym5, pts5, kctx

    return dict(suffix=suffix, codec=codec, k1024=k1024, lossy=lossy, weighted=weighted)


# ----------------------------------------------------------- CPU oracle ---
def _host_inputs(cfg, b, l, n_pos):
    """float64 K and V [H, n_pos, D] of stream (b, l) from the seeded
    generator, positions t0 .. t0 + n_pos - 1."""
    H = cfg.n_heads
    pos = np.arange(cfg.t0, cfg.t0 + n_pos)
    hh, tt = np.meshgrid(np.arange(H), pos, indexing="ij")
    return (synth.storage_to_f64(synth.kv_elements(cfg, 0, l, b, hh, tt), cfg.dtype),
            synth.storage_to_f64(synth.kv_elements(cfg, 1, l, b, hh, tt), cfg.dtype))


def _f64(t):
    import torch
    return t.to(torch.float64).numpy()


def oracle_sample(budget_s, cfg=HEADLINE, src=None, max_streams=None, max_records=None):
    """The float64 oracle on (sequence, layer) streams of the workload until
    `budget_s` seconds of work: RVQ, serialisation, span encode, append,
    decode, reconstruction and random reads of each stream, timed.  With
    `src` (host copies of the GPU step's sample streams) the inputs are those
    of the GPU step and, untimed, every GPU output of the stream is compared
    with the oracle's (the parity counts); without it the inputs come from the
    seeded generator, each stream cut to its first `max_records` records.
    Returns (records per second, streams, seconds of work, threads, parity)."""
    import oracle
    from oracle import parity
    oracle.build()
    cbk, cbv = synth.codebooks(cfg, 0), synth.codebooks(cfg, 1)
    r = oracle.packing_ratio(256)
    L = oracle.max_span_len(r)
    H, SK, SV = cfg.n_heads, cfg.stages_k, cfg.stages_v
    items = src if src is not None else [{"b": b, "l": l} for (b, l) in oracle_streams(cfg, cfg.batch * cfg.n_layers)]
    done = records = 0
    t_work = 0.0
    rng = np.random.default_rng(1)
    par = {"rvq_compared": 0, "rvq_hard": 0, "rvq_near_tie": 0, "points_compared": 0, "points_bit_equal": 0,
           "kv_compared": 0, "kv_hard": 0, "kv_rounding_borderline": 0}
    for it in items:
        if max_streams is not None and done >= max_streams:
            break
        b, l = it["b"], it["l"]
        if src is not None:
            Kx, Vx = _f64(it["K"]), _f64(it["V"])
        else:
            Kx, Vx = _host_inputs(cfg, b, l, min(cfg.n_archived + 1, max_records or cfg.n_archived + 1))
        n_pos = Kx.shape[1]
        P = n_pos - 1                                      # archived, then one appended position
        t_start = time.perf_counter()
        ok_ = [oracle.rvq_encode(Kx[h], cbk[l, h]) for h in range(H)]
        ov_ = [oracle.rvq_encode(Vx[h], cbv[l, h]) for h in range(H)]
        ik = np.stack([o[0] for o in ok_])
        iv = np.stack([o[0] for o in ov_])
        stream = oracle.records_from_indices(ik[:, :P], iv[:, :P])
        oracle.span_encode(stream, 256, r, L)
        tail = oracle.records_from_indices(ik[:, P:], iv[:, P:])
        pts = oracle.append(stream, tail, 256, r, L)
        full = np.concatenate([stream, tail])
        dec, _, bad = oracle.span_decode(pts, full.size, 256, r, L)
        k2, v2 = oracle.indices_from_records(dec, H, SK, SV)
        for h in range(H):
            oracle.round_to(oracle.rvq_decode(k2[h], cbk[l, h]), cfg.dtype)
            oracle.round_to(oracle.rvq_decode(v2[h], cbv[l, h]), cfg.dtype)
        reads = rng.integers(0, full.size, N_READS // 32 + 1)
        oracle.read(pts, full.size, reads, 256, r, L)
        t_work += time.perf_counter() - t_start
        done += 1
        records += n_pos
        if src is not None:
            gk, gv = oracle.indices_from_records(it["sym"], H, SK, SV)
            for h in range(H):
                for gi, o in ((gk[h], ok_[h]), (gv[h], ov_[h])):
                    hard, near, seen = parity.compare_rvq(gi, o[0], o[1])
                    par["rvq_hard"] += hard
                    par["rvq_near_tie"] += near
                    par["rvq_compared"] += seen
            want = oracle.span_encode(it["sym"].astype(np.int32), 256, r, L)
            par["points_compared"] += want.shape[0]
            par["points_bit_equal"] += int(np.all(want.view(np.uint64) == it["pts"].view(np.uint64), axis=1).sum())
            for h in range(H):
                for out, gi, cb in ((it["Kr"], gk, cbk), (it["Vr"], gv, cbv)):
                    hard, border, n = parity.rounded_mismatches(
                        _f64(out[h]), oracle.rvq_decode(gi[h], cb[l, h]), cfg.dtype,
                        oracle.rvq_decode(gi[h], np.abs(cb[l, h])))
                    par["kv_hard"] += hard
                    par["kv_rounding_borderline"] += border
                    par["kv_compared"] += n
        if t_work >= budget_s:
            break
    return records / t_work, done, t_work, oracle.threads(), (par if src is not None else None)


def cpu_desc():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True).stdout
        for ln in out.splitlines():
            if ln.startswith("Model name"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    return "unknown"


# -------------------------------------------------------------- report ----
def secondary_report(res, peaks, fp64, sm_mhz):
    kernels = {}
    gx = res.get("gpt2")
    if gx is not None:
        rates = archive_rates(gx.cfg, gx.phase, gx.R, gx.P, gx.n_rec, gx.spans, gx.ns, peaks, fp64)
        kernels["gpt2-shaped archive (64-dim heads)"] = {
            "workload": "gpt2-shaped full KV cache: 12 layers x batch 8 x 12 heads x 1024 tok x 64 dims, fp16; "
                        "4+32 exact window; K 4 / V 2 RVQ stages x 256; N=256, r=r_256, L=6",
            "records_per_s": gx.ns * gx.n_rec / (gx.ms * 1e-3), "ms_per_step": gx.ms, "phase_ms": gx.phase,
            "rvq_kernel": "k_rvq64", "rvq_ms": rates["rvq"]["ms"], "rvq_tflops": rates["rvq"]["achieved_tflops"],
            "rvq_frac": rates["rvq"]["frac"], "span_encode_ms": rates["span_encode"]["ms"],
            "span_encode_frac_fp64_measured": rates["span_encode"]["frac_fp64_measured"],
            "decode_kv_ms": rates["decode_kv"]["ms"], "decode_kv_gbs": rates["decode_kv"]["achieved_gbs"],
            "decode_kv_frac": rates["decode_kv"]["frac"], "status_ok": gx.ok}
    sx = res.get("stream")
    if sx is not None:
        kernels["decode-time streaming (64 sequences)"] = {
            "workload": "64 llama3-8b-shaped sequences (32 layers x 8 KV heads x 128 dims, bf16), 131072 archived "
                        "positions per (sequence, layer) stream (34 GB of points); per step: RVQ + tail append of "
                        "the position leaving the window for every sequence (2048 records), then 4096 seeded "
                        "random record reads per sequence (262,144 reads, K and V of all heads)",
            "us_per_step": sx["step_us"], "append_rvq_us": sx["append_rvq_ms"] * 1e3,
            "append_us": sx["append_ms"] * 1e3, "read_us": sx["read_ms"] * 1e3,
            "reads_per_s": sx["reads"] / (sx["read_ms"] * 1e-3),
            "bytes_per_read": {"points_in": sx["read_bytes_in"], "kv_out": sx["read_bytes_out"]},
            "read_gbs_out": sx["reads"] * sx["read_bytes_out"] / (sx["read_ms"] * 1e-3) / 1e9,
            "timed_steps": sx["steps"], "status_ok": sx["ok"]}
    sec = res.get("secondary") or {}
    if sec.get("suffix"):
        sx = sec["suffix"]
        gbs = sx["bytes"] / (sx["ms"] * 1e-3) / 1e9
        kernels["suffix_search (Sec. 5)"] = {"bound": "hbm", "ms": sx["ms"], "achieved_gbs": gbs,
                                             "frac": gbs / peaks["hbm_gbs"], "matches": sx["matches"],
                                             "candidates": sx["candidates"], "workload": sx["workload"]}
    if sec.get("codec"):
        per_n = {}
        for N, cx in sec["codec"].items():
            syms = 4 * (1 << 28)
            nbytes = syms + 4 * cx["spans"] * 16          # 1 B per symbol + one 16 B point per span
            enc = syms * 6 / (cx["encode_ms"] * 1e-3)
            per_n["N=%d" % N] = {
                "L": cx["L"],
                "encode_ms": cx["encode_ms"], "encode_symbols_per_s": syms / (cx["encode_ms"] * 1e-3),
                "encode_frac_hbm": nbytes / (cx["encode_ms"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                "encode_frac_fp64_measured": enc / fp64["measured"] if fp64.get("measured") else None,
                "encode_frac_fp64_nominal": enc / fp64["nominal"],
                "decode_ms": cx["decode_ms"], "decode_symbols_per_s": syms / (cx["decode_ms"] * 1e-3),
                "decode_frac_hbm": nbytes / (cx["decode_ms"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
                "read_ms": cx["read_ms"], "reads_per_s": cx["reads"] / (cx["read_ms"] * 1e-3),
                "exact": cx["exact"], "status_ok": cx["ok"]}
        kernels["span codec, symbol stress"] = {
            "workload": "4 streams x 2^28 seeded uniform symbols per N; full encode, full decode, 2^20 seeded "
                        "random reads per stream; all decoded and read symbols checked equal to the input",
            "encode_bound": "fp64", "decode_bound": "integer ALU", "read_bound": "latency", "per_N": per_n}
    if sec.get("k1024"):
        kx = sec["k1024"]
        rvq_ms = kx["rvq_k"] + kx["rvq_v"]
        flops = kx["nvec"] * sum(kx["stages"]) * 2 * 64 * 1024
        tf = flops / (rvq_ms * 1e-3) / 1e12
        dec_b = kx["ns"] * kx["P"] * kx["R"] * 2 + kx["ns"] * (-(-kx["P"] * kx["R"] // kx["L"])) * 16 + kx["out_bytes"]
        kernels["pooled RVQ 1024 x 2 archive (Table 2)"] = {
            "workload": "gpt2-shaped full KV cache (12 layers x batch 8 x 12 heads x 1024 tok x 64, fp16), one "
                        "1024-codeword codebook per layer and stage shared by all heads, K 2 / V 2 stages; "
                        "uint16 symbols, N=1024, r=r_1024, L=5",
            "rvq_ms": rvq_ms, "bound": "tensor", "achieved_tflops": tf, "frac": tf / peaks["bf16_tflops"],
            "span_encode_ms": kx["span_encode"], "decode_kv_ms": kx["decode_kv"],
            "decode_kv_gbs": dec_b / (kx["decode_kv"] * 1e-3) / 1e9,
            "decode_kv_frac": dec_b / (kx["decode_kv"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "archived_positions_per_s": kx["ns"] * kx["P"] / ((rvq_ms + kx["span_encode"]) * 1e-3),
            "status_ok": kx["ok"]}
    if sec.get("lossy"):
        lx = sec["lossy"]
        tb = lx["point_bytes"] + lx["code_bytes"]             # points read, codes written
        kernels["lossy archive (Sec. 4)"] = {
            "workload": "the gpt2 step's 96 streams x 989 records x 72 symbols (N=256, span 6); spans older than "
                        "the last %d truncated to %d bits per coordinate" % (lx["keep"], lx["bits"]),
            "truncate_ms": lx["truncate"], "truncate_bound": "hbm",
            "truncate_gbs": tb / (lx["truncate"] * 1e-3) / 1e9,
            "truncate_frac": tb / (lx["truncate"] * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "decode_ms": lx["decode"], "decode_bound": "fp64 (binary64 walk with IEEE division, as the paper)",
            "decode_symbols_per_s": lx["symbols"] / (lx["decode"] * 1e-3),
            "archive_bytes": lx["code_bytes"] + lx["tail_bytes"], "exact_archive_bytes": lx["point_bytes"],
            "symbol_error_rate_truncated_spans": lx["sym_err_truncated"], "status_ok": lx["ok"]}
    if sec.get("weighted"):
        wx = sec["weighted"]
        kernels["probability-weighted maps (Sec. 6)"] = {
            "workload": "the gpt2 step's 96 archived RVQ index streams (989 records x 72 symbols, N=256), adaptive "
                        "add-one model, one warp per stream",
            "encode_ms": wx["encode"], "decode_ms": wx["decode"], "bound": "latency (sequential within a stream)",
            "encode_symbols_per_s": wx["symbols"] / (wx["encode"] * 1e-3),
            "decode_symbols_per_s": wx["symbols"] / (wx["decode"] * 1e-3),
            "bits_per_symbol": wx["bits"] / wx["symbols"], "uniform_bits_per_symbol": 8.0,
            "lossless": wx["exact"], "status_ok": wx["ok"]}
    return kernels


# ---------------------------------------------------------------- main ----
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="fkv", choices=["fkv", "reference"])
    ap.add_argument("--seq", type=int, default=HEADLINE.seq,
                    help="positions of the headline cache (a shorter one for profiling captures)")
    ap.add_argument("--stream-steps", type=int, default=64, help="timed steps of the streaming workload")
    for name in ("e2e", "gpt2", "stream", "suffix", "k1024", "lossy", "codec", "weighted", "fp64", "cpu"):
        ap.add_argument("--no-" + name, action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle work for cpu_baseline")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        max_records = 4096
        per_step = max(1.0, 150.0 / (args.steps + args.warmup))
        for _ in range(args.warmup):
            oracle_sample(per_step / 4, max_streams=1, max_records=max_records)
        tot_rec = tot_t = 0.0
        cores = 1
        for _ in range(args.steps):
            v, done, t, cores, _ = oracle_sample(per_step, max_records=max_records)
            tot_rec += v * t
            tot_t += t
        value = tot_rec / tot_t
        sample = ("(sequence, layer) streams of the workload cut to their first %d archived positions, about "
                  "%.0f s of oracle work per step" % (max_records, per_step))
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot_t / args.steps * 1e3,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic", "config": {"workload": WORKLOAD, "sample": sample},
                "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample,
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
    cfg = res["cfg"]
    sm_mhz = res["clocks"].get("sm_mhz") or 2070.0
    rates = archive_rates(cfg, res["phase"], res["R"], res["P"], res["n_rec"], res["spans"], res["ns"], peaks,
                          res["fp64"])
    traffic = RVQ_DRAM_BYTES_PER_LAUNCH if args.seq == HEADLINE.seq else None
    dominant = roofline(rates, peaks, traffic, "k_rvq128 (RVQ assignment, 128-dim heads)")
    kernels = {"rvq (tcgen05, k_rvq128)": rates["rvq"], "span_encode": rates["span_encode"],
               "decode_kv (decode + gather)": rates["decode_kv"]}
    kernels.update(secondary_report(res, peaks, res["fp64"], sm_mhz))
    units = res["units"] * world
    value = units / (ms * 1e-3)
    cpu = par = None
    if world == 1 and not args.no_cpu:
        v, done, t, cores, par = oracle_sample(args.cpu_budget, cfg, src=res["parity_src"])
        sample = ("%d whole (sequence, layer) streams of the headline step (%d records), %.1f s of oracle work"
                  % (done, sum(x["K"].shape[1] for x in res["parity_src"][:done]), t))
        cpu = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample, "cpu": cpu_desc()}
        par = dict(par, streams=done, sample=sample,
                   rule="RVQ indices equal where the oracle's top-2 gap exceeds 1e-4 of the stage residual's "
                        "squared norm (near ties counted); points bit-equal to the oracle's encode of the GPU's "
                        "symbols; bf16 K/V equal to the oracle's float64 sum rounded to nearest-even outside the "
                        "float32 summation error band (borderline cases counted)")
    e2e = None
    if res["e2e"]:
        e2e = {"value": units / (res["e2e"]["ms"] * 1e-3), "unit": UNIT,
               "h2d_bytes_per_step": res["e2e"]["h2d"], "d2h_bytes_per_step": res["e2e"]["d2h"],
               "ms_per_step": res["e2e"]["ms"], "status_ok": res["e2e"]["ok"],
               # the step's host -> device bytes against the link measured alone
               "h2d_link_gbs": res["e2e"]["link_gbs"],
               "h2d_link_frac": res["e2e"]["h2d"] / (res["e2e"]["ms"] * 1e-3) / 1e9 / res["e2e"]["link_gbs"]}
    fp64 = {"measured_ops_per_s": res["fp64"].get("measured"), "nominal_ops_per_s": res["fp64"]["nominal"],
            "how": "fkv_measure_fp64_rate: independent chains of binary64 multiply and add (no FMA) on every SM; "
                   "nominal = 1.25 TFLOP/s FMA = 625 G add/mul per s at 2070 MHz, scaled to the sampled clock"}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 in / fp16-split tensor / f64 codec", "data": "synthetic",
        "config": {"workload": WORKLOAD if args.seq == HEADLINE.seq else WORKLOAD.replace("32768", str(args.seq)),
                   "records_per_step": res["units"], "global_batch": cfg.batch * world, "seq_len": args.seq,
                   "l2": "inputs (17.2 GB) larger than L2; no flush", "parallelism": "replicas (weak)"},
        "decoded_kv_gbs": rates["out_bytes"] / (res["phase"]["decode_kv"] * 1e-3) / 1e9,
        "write_positions_per_s": res["units"] / ((res["phase"]["rvq_k"] + res["phase"]["rvq_v"]
                                                 + res["phase"]["span_encode"]) * 1e-3),
        "phase_ms": res["phase"],
        "roofline": dominant,
        "kernels": kernels,
        "fp64": fp64,
        "parity": par,
        "cpu_baseline": cpu,
        "e2e": e2e,
        # per step: RVQ x4 (K and V archive, K and V of the appended position),
        # k_span_encode x2 (archive, tail append), k_span_decode_planar,
        # k_gather x2, the record reads' k_order_count, k_order_scan and
        # k_order_scatter, and k_read_kv (as the ncu launch list shows)
        "gpu_launches": 13 * args.steps,
        "clocks": res["clocks"],
        "status_ok": res["ok"],
    }
    print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
