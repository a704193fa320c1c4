"""Host arithmetic of bench.py's roofline object (no GPU).

The algorithmic work per step is fixed by the method, independently of any
kernel: 2*D*256 flop per vector and RVQ stage (Sec. 3 "Setup"), one byte per
symbol plus 16 B per span in and the rebuilt K/V out for the archive read,
six binary64 operations per encoded symbol (Sec. 1).  These tests rebuild
those totals from the workloads' shapes and check the fractions bench.py
reports against them."""
import bench
import synth

PEAKS = {"hbm_gbs": 6698.5, "bf16_tflops": 1950.6, "bf16_tflops_sustained": 1749.7, "source": "measured"}
FP64 = {"measured": 600e9, "nominal": 625e9}


def _rates(cfg, ms_rvq_k, ms_rvq_v, ms_enc, ms_dec):
    P = cfg.n_archived
    R = cfg.record_len
    ns = cfg.batch * cfg.n_layers
    n_rec = P + 1
    spans = -(-n_rec * R // 6)
    phase = {"rvq_k": ms_rvq_k, "rvq_v": ms_rvq_v, "span_encode": ms_enc, "append_rvq": 0.03, "append": 0.008,
             "decode_kv": ms_dec, "read_kv": 0.04}
    return bench.archive_rates(cfg, phase, R, P, n_rec, spans, ns, PEAKS, FP64), (P, R, ns, n_rec, spans)


def test_headline_is_the_largest_single_gpu_config():
    c = bench.HEADLINE
    assert c is synth.CFG3
    assert c.n_layers * c.batch * c.n_heads * c.seq * c.dim * 2 * 2 == 17179869184     # 17.2 GB of K and V
    assert c.n_archived == 32768 - 36 and c.record_len == 48


def test_rvq_flops_match_the_llama_workload():
    cfg = synth.CFG3
    rates, (P, R, ns, n_rec, spans) = _rates(cfg, 33.0, 17.0, 2.4, 5.6)
    # 4 sequences x 32 layers x 8 heads x 32732 archived positions, K 4 + V 2 stages
    nvec = 4 * 32 * 8 * 32732
    flops = nvec * (4 + 2) * 2 * 128 * 256
    assert rates["rvq"]["flops"] == flops and abs(flops - 1.317e13) / 1.317e13 < 0.001
    tf = flops / 50e-3 / 1e12
    assert abs(rates["rvq"]["achieved_tflops"] - tf) < 1e-9 * tf
    dom = bench.roofline(rates, PEAKS, None, "k_rvq128")
    assert abs(dom["frac"] - tf / PEAKS["bf16_tflops"]) < 1e-12
    assert dom["unit"] == "TFLOP/s" and dom["bound"] == "tensor" and dom["traffic"] is None
    assert "of measured" in dom["kernel"]


def test_rvq_traffic_scaling():
    """The per-launch DRAM traffic line through the two captured lengths: it
    returns the captures at their own lengths and, at the headline length,
    stays close to the algorithmic bytes (input + codebook operands +
    indices) of a full-length launch."""
    (p1, p2), launches = bench.RVQ_TRAFFIC_CAPTURES
    assert bench._rvq_traffic_full(p1) == sum(b[0] for b in launches) / 2
    assert bench._rvq_traffic_full(p2) == sum(b[1] for b in launches) / 2
    c = synth.CFG3
    nvec = c.n_layers * c.batch * c.n_heads * c.n_archived
    groups = c.n_layers * c.n_heads
    alg = [nvec * c.dim * 2 + groups * s * 256 * c.dim * 4 + nvec * s for s in (4, 2)]
    assert abs(bench.RVQ_DRAM_BYTES_PER_LAUNCH / (sum(alg) / 2) - 1) < 0.05


def test_decode_bytes_and_fp64_fractions():
    cfg = synth.CFG1
    rates, (P, R, ns, n_rec, spans) = _rates(cfg, 0.445, 0.237, 0.088, 0.160)
    assert (ns, P, R) == (96, 988, 72)
    out_bytes = ns * n_rec * 2 * 12 * 64 * 2                   # fp16 K and V of every archived position
    assert rates["out_bytes"] == out_bytes
    d = rates["decode_kv"]
    assert d["bytes"] == ns * n_rec * R + ns * spans * 16 + out_bytes   # symbols + points in, K/V out
    assert abs(d["achieved_gbs"] - d["bytes"] / 0.160e-3 / 1e9) < 1e-6
    assert abs(d["frac"] - d["achieved_gbs"] / PEAKS["hbm_gbs"]) < 1e-12
    assert abs(d["frac_nominal"] - d["achieved_gbs"] / 7900.0) < 1e-12
    e = rates["span_encode"]
    # six binary64 add/sub/mul per symbol against the measured and nominal rates
    assert abs(e["frac_fp64_measured"] - ns * P * R * 6 / 0.088e-3 / 600e9) < 1e-9
    assert abs(e["frac_fp64_nominal"] - ns * P * R * 6 / 0.088e-3 / 625e9) < 1e-9


def test_fallback_peaks_are_labelled():
    rates, _ = _rates(synth.CFG1, 0.445, 0.237, 0.088, 0.160)
    dom = bench.roofline(rates, dict(PEAKS, source="fallback"), None, "k_rvq64")
    assert "of fallback" in dom["kernel"]


def test_oracle_sample_streams_are_distinct_and_start_at_the_ends():
    cfg = synth.CFG3
    s = bench.oracle_streams(cfg, 8)
    assert s[0] == (0, 0) and s[1] == (cfg.batch - 1, cfg.n_layers - 1)
    assert len(set(s)) == 8 and all(0 <= b < cfg.batch and 0 <= l < cfg.n_layers for b, l in s)


def test_reference_sample_runs_the_oracle_on_a_cut_stream(oracle_mod):
    # the reference arm's unit: a (sequence, layer) stream cut to its first
    # archived positions, every head and both K and V (whole records)
    cfg = synth.small_config(synth.CFG3, 3, n_layers=2, batch=1, seq=36 + 40, n_heads=2)
    v, done, t, cores, par = bench.oracle_sample(0.0, cfg, max_streams=1, max_records=17)
    assert done == 1 and v > 0 and par is None and cores >= 1
