"""Host arithmetic of bench.py's roofline object (no GPU).

The algorithmic work per step of the GPT-2-shaped workload is fixed by the
method, independently of any kernel: 2*D*256 flop per vector and RVQ stage
(Sec. 3 "Setup"), one byte per symbol plus 16 B per span in and the rebuilt
fp16 K/V out for the archive read.  These tests rebuild those totals from the
workload's shape and check the fractions bench.py reports against them."""
import bench
import synth


def fake_result(ms_rvq_k=0.445, ms_rvq_v=0.237, ms_enc=0.088, ms_dec=0.160, sm_mhz=2070.0):
    cfg = synth.CFG1
    P = cfg.n_archived
    R = cfg.record_len
    L = 6
    ns = cfg.batch * cfg.n_layers
    spans = -(-P * R // L)
    phase = {"rvq_k": ms_rvq_k, "rvq_v": ms_rvq_v, "span_encode": ms_enc, "append_rvq": 0.03, "append": 0.008,
             "decode_kv": ms_dec, "read_kv": 0.04}
    return dict(cfg=cfg, ms=sum(phase.values()), phase=phase, clocks={"sm_mhz": sm_mhz}, ok=True, e2e=None,
                units=ns * P, R=R, ns=ns, P=P, n_rec=P, spans=spans, L=L)


PEAKS = {"hbm_gbs": 6698.5, "bf16_tflops": 1950.6, "bf16_tflops_sustained": 1749.7, "source": "measured"}


def test_rvq_flops_match_the_workload():
    res = fake_result()
    dom, kernels, _, _ = bench.roofline(res, PEAKS, 184304640)
    cfg = res["cfg"]
    # 8 sequences x 12 layers x 12 heads x 988 archived positions (T = 1024 minus 4 + 32 exact)
    nvec = 8 * 12 * 12 * (1024 - 36)
    flops = nvec * (4 + 2) * 2 * 64 * 256
    assert abs(flops - 2.24e11) / 2.24e11 < 0.005
    ms = res["phase"]["rvq_k"] + res["phase"]["rvq_v"]
    assert abs(dom["achieved"] - flops / (ms * 1e-3) / 1e12) < 1e-9 * dom["achieved"]
    assert abs(dom["frac"] - dom["achieved"] / PEAKS["bf16_tflops"]) < 1e-12
    assert dom["unit"] == "TFLOP/s" and dom["bound"] == "tensor" and dom["traffic"] == 184304640
    assert "of measured" in dom["kernel"]
    assert kernels["rvq (tcgen05)"]["frac"] == dom["frac"]
    assert cfg.n_archived == 1024 - 36


def test_decode_bytes_and_fp64_fraction():
    res = fake_result()
    _, kernels, dec_bytes, out_bytes = bench.roofline(res, PEAKS)
    ns, P, R = 96, 988, 72
    spans = P * R // 6
    assert out_bytes == ns * P * 2 * 12 * 64 * 2                 # fp16 K and V of every archived position
    assert dec_bytes == ns * P * R + ns * spans * 16 + out_bytes  # symbols + points in, K/V out
    d = kernels["decode_kv (decode + gather)"]
    assert abs(d["achieved_gbs"] - dec_bytes / 0.160e-3 / 1e9) < 1e-6
    assert abs(d["frac"] - d["achieved_gbs"] / PEAKS["hbm_gbs"]) < 1e-12
    e = kernels["span_encode"]
    # six binary64 add/sub/mul per symbol against the nominal 625 G per s at 2070 MHz
    assert abs(e["frac_fp64"] - ns * P * R * 6 / 0.088e-3 / 625e9) < 1e-9


def test_fallback_peaks_are_labelled():
    res = fake_result()
    dom, _, _, _ = bench.roofline(res, dict(PEAKS, source="fallback"))
    assert "of fallback" in dom["kernel"]
