"""Seeded synthetic inputs for the fractal KV-cache archive.

This module is the one thing the oracle side and the CUDA side share: it makes
inputs and holds none of the method's arithmetic (no codec step, no nearest-
codeword search).  Every value is a pure function of (seed, tensor id, flat
element index) through Philox4x32-10, the counter-based generator of Salmon,
Moraes, Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3" (SC'11).
numpy implements it here; ``csrc/synth_gen.cu`` implements the same published
definition for bulk generation on the device (large configurations), so any
sampled element can be regenerated on the host and checked.

Value recipe (stands in for GPT-2 / Llama KV activations, which are not
available): one Philox call per element gives four 32-bit words = eight 16-bit
uniforms; their centred sum z (an Irwin-Hall(8) variate, near-Gaussian, tails
at 4.9 sigma) is an exact integer, and the element is the float32 product
float32(z) * scale[channel] (one IEEE rounding), then rounded to nearest-even
into the storage dtype.  Per-channel scales carry the outlier key channels and
log-normal channel scales of each configuration.
"""
from __future__ import annotations

import dataclasses
import functools
import math
from typing import Tuple

import numpy as np

# Philox4x32 constants (Salmon et al. 2011, Sec. 5 / Random123).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
PHILOX_ROUNDS = 10

BASE_SEED = 2607_07144
IRWIN_HALL_MEAN = 8 * 65535 // 2            # 262140: centre of the sum of 8 u16
IRWIN_HALL_STD = math.sqrt(8 * (65536.0 ** 2 - 1.0) / 12.0)   # 53510.57...

# Tensor ids (third Philox counter word) keep streams disjoint.
TID_K, TID_V, TID_CB_K, TID_CB_V, TID_SYM, TID_POS, TID_AUX = 0, 1, 2, 3, 4, 5, 6

# Residual shrink per RVQ stage for the synthetic codebooks (see codebooks()).
STAGE_SHRINK = 0.85


def philox4x32(c0, c1, c2, c3, k0: int, k1: int):
    """Philox4x32-10 on uint32 arrays (broadcast); returns four uint32 arrays."""
    x0 = np.asarray(c0, np.uint64) & 0xFFFFFFFF
    x1 = np.asarray(c1, np.uint64) & 0xFFFFFFFF
    x2 = np.asarray(c2, np.uint64) & 0xFFFFFFFF
    x3 = np.asarray(c3, np.uint64) & 0xFFFFFFFF
    x0, x1, x2, x3 = np.broadcast_arrays(x0, x1, x2, x3)
    x0, x1, x2, x3 = (a.copy() for a in (x0, x1, x2, x3))
    k0 = np.uint64(k0 & 0xFFFFFFFF)
    k1 = np.uint64(k1 & 0xFFFFFFFF)
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    mask = np.uint64(0xFFFFFFFF)
    s32 = np.uint64(32)
    for rnd in range(PHILOX_ROUNDS):
        p0 = x0 * m0            # exact: both factors < 2**32
        p1 = x2 * m1
        hi0, lo0 = p0 >> s32, p0 & mask
        hi1, lo1 = p1 >> s32, p1 & mask
        x0, x1, x2, x3 = hi1 ^ x1 ^ k0, lo1, hi0 ^ x3 ^ k1, lo0
        if rnd != PHILOX_ROUNDS - 1:
            k0 = (k0 + np.uint64(PHILOX_W0)) & mask
            k1 = (k1 + np.uint64(PHILOX_W1)) & mask
    return (x0.astype(np.uint32), x1.astype(np.uint32),
            x2.astype(np.uint32), x3.astype(np.uint32))


def seed_key(cfg_id: int) -> Tuple[int, int]:
    s = BASE_SEED + int(cfg_id)
    return s & 0xFFFFFFFF, (s >> 32) & 0xFFFFFFFF


def irwin_hall(flat_index, tensor_id: int, cfg_id: int) -> np.ndarray:
    """Centred sum of eight 16-bit uniforms for each flat element index (int32)."""
    e = np.asarray(flat_index, np.uint64)
    k0, k1 = seed_key(cfg_id)
    w = philox4x32(e & np.uint64(0xFFFFFFFF), e >> np.uint64(32), tensor_id, 0, k0, k1)
    z = np.zeros(e.shape, np.int64)
    for word in w:
        ww = word.astype(np.int64)
        z += (ww & 0xFFFF) + (ww >> 16)
    return (z - IRWIN_HALL_MEAN).astype(np.int32)


def uniform_u32(flat_index, tensor_id: int, cfg_id: int, word: int = 0) -> np.ndarray:
    e = np.asarray(flat_index, np.uint64)
    k0, k1 = seed_key(cfg_id)
    return philox4x32(e & np.uint64(0xFFFFFFFF), e >> np.uint64(32), tensor_id, 0, k0, k1)[word]


# --------------------------------------------------------- configurations --
@dataclasses.dataclass(frozen=True)
class KVConfig:
    """One synthetic KV-cache workload (shapes of the paper's GPT-2 study and
    of a Llama-3-8B-shaped cache)."""
    cfg_id: int
    name: str
    n_layers: int
    batch: int
    n_heads: int
    dim: int
    seq: int              # T, positions in the cache
    dtype: str            # 'f32' | 'f16' | 'bf16'
    stages_k: int
    stages_v: int
    outlier_channels: int  # key channels per head scaled up
    outlier_scale: float
    lognormal_sigma: float  # per-channel log-normal scale sigma (0 = none)
    N: int = 256            # symbol alphabet (= codewords per stage)
    pooled: bool = False    # one codebook per layer shared by its heads (Sec. 3, Table 2)

    @property
    def record_len(self) -> int:
        return self.n_heads * (self.stages_k + self.stages_v)

    @property
    def t0(self) -> int:
        return 4

    @property
    def t1(self) -> int:
        return max(4, self.seq - 32)

    @property
    def n_archived(self) -> int:
        return self.t1 - self.t0

    @property
    def elem_bytes(self) -> int:
        return {"f32": 4, "f16": 2, "bf16": 2}[self.dtype]

    def cache_shape(self):
        return (self.n_layers, self.batch, self.n_heads, self.seq, self.dim)


CFG0 = KVConfig(0, "gpt2-1layer-b1-t1024-f32", 1, 1, 12, 64, 1024, "f32", 2, 1, 4, 8.0, 0.0)
CFG1 = KVConfig(1, "gpt2-12layer-b8-t1024-f16", 12, 8, 12, 64, 1024, "f16", 4, 2, 4, 8.0, 0.0)
CFG3 = KVConfig(3, "llama3-8b-32layer-b4-t32768-bf16", 32, 4, 8, 128, 32768, "bf16", 4, 2, 3, 10.0, 0.5)
# Decode-time streaming (Llama-3-8B shape, 64 sequences): 131072 archived
# positions prefilled, then 512 steps that each archive one more position; the
# cache holds all of them plus the 4 + 32 exact window.
CFG4 = KVConfig(4, "llama3-8b-stream-b64-t131072-bf16", 32, 64, 8, 128, 131072 + 512 + 36, "bf16", 4, 2, 3, 10.0,
                0.5)
CFG4_PREFILL, CFG4_STEPS = 131072, 512
# Table 2's pooled rows at k = 1024 on the GPT-2 shape: RVQ 1024 x 2 and VQ 1024.
CFG5 = KVConfig(5, "gpt2-12layer-b8-t1024-f16-pooled-rvq1024x2", 12, 8, 12, 64, 1024, "f16", 2, 2, 4, 8.0, 0.0,
                N=1024, pooled=True)
CFG6 = KVConfig(6, "gpt2-12layer-b8-t1024-f16-pooled-vq1024", 12, 8, 12, 64, 1024, "f16", 1, 1, 4, 8.0, 0.0,
                N=1024, pooled=True)


def small_config(base: KVConfig, cfg_id: int, n_layers: int, batch: int, seq: int,
                 n_heads: int = None) -> KVConfig:
    """A reduced copy of a configuration (same distributions) for fast tests."""
    return dataclasses.replace(base, cfg_id=cfg_id, name=base.name + "-small",
                               n_layers=n_layers, batch=batch, seq=seq,
                               n_heads=n_heads or base.n_heads)


def channel_sigma(cfg: KVConfig, kv: int) -> np.ndarray:
    """Per-(layer, head, channel) standard deviation, float64 [Ly, H, D].
    Keys get `outlier_channels` channels per head scaled by `outlier_scale`
    (chosen per head by the seed); Llama-shaped configs also get a log-normal
    scale per channel for keys and values."""
    rng = np.random.default_rng([BASE_SEED, cfg.cfg_id, 17, kv])
    sig = np.ones((cfg.n_layers, cfg.n_heads, cfg.dim), np.float64)
    if cfg.lognormal_sigma > 0:
        sig *= np.exp(rng.normal(0.0, cfg.lognormal_sigma, size=sig.shape))
    if kv == 0 and cfg.outlier_channels > 0:
        for l in range(cfg.n_layers):
            for h in range(cfg.n_heads):
                ch = rng.choice(cfg.dim, size=cfg.outlier_channels, replace=False)
                sig[l, h, ch] *= cfg.outlier_scale
    return sig


def channel_scale32(cfg: KVConfig, kv: int) -> np.ndarray:
    """float32 multiplier applied to the Irwin-Hall integer, [Ly, H, D]."""
    return (channel_sigma(cfg, kv) / IRWIN_HALL_STD).astype(np.float32)


def round_f32_to(x32: np.ndarray, dtype: str) -> np.ndarray:
    """Nearest-even cast of float32 to the storage dtype; bf16 is returned as
    its uint16 bit pattern, f16 as float16, f32 unchanged."""
    x32 = np.asarray(x32, np.float32)
    if dtype == "f32":
        return x32
    if dtype == "f16":
        return x32.astype(np.float16)
    if dtype == "bf16":
        b = x32.view(np.uint32).astype(np.uint64)
        lsb = (b >> np.uint64(16)) & np.uint64(1)
        r = (b + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
        nan = np.isnan(x32)
        out = r.astype(np.uint16)
        out[nan] = 0x7FC0
        return out
    raise ValueError(dtype)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, np.uint32) << np.uint32(16)).view(np.float32)


def storage_to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return bf16_bits_to_f32(a).astype(np.float64)
    return np.asarray(a).astype(np.float64)


def kv_elements(cfg: KVConfig, kv: int, layer, batch, head, pos) -> np.ndarray:
    """Values (storage dtype; bf16 as uint16 bits) of whole head vectors at the
    given (layer, batch, head, position) index arrays, shape [..., D]."""
    l = np.asarray(layer, np.int64)[..., None]
    b = np.asarray(batch, np.int64)[..., None]
    h = np.asarray(head, np.int64)[..., None]
    t = np.asarray(pos, np.int64)[..., None]
    d = np.arange(cfg.dim, dtype=np.int64)
    flat = ((((l * cfg.batch + b) * cfg.n_heads + h) * cfg.seq + t) * cfg.dim + d)
    z = irwin_hall(flat, TID_K if kv == 0 else TID_V, cfg.cfg_id)
    sc = channel_scale32(cfg, kv)[np.broadcast_to(l, flat.shape), np.broadcast_to(h, flat.shape), d]
    x32 = (z.astype(np.float32) * sc).astype(np.float32)
    return round_f32_to(x32, cfg.dtype)


def kv_cache(cfg: KVConfig, kv: int) -> np.ndarray:
    """The whole cache [Ly, B, H, T, D] in the storage dtype (host; small configs)."""
    Ly, B, H, T, D = cfg.cache_shape()
    l, b, h, t = np.meshgrid(np.arange(Ly), np.arange(B), np.arange(H), np.arange(T), indexing="ij")
    return kv_elements(cfg, kv, l, b, h, t)


@functools.lru_cache(maxsize=8)
def codebooks(cfg: KVConfig, kv: int) -> np.ndarray:
    """Synthetic RVQ codebooks, float32 [Ly, H, S, K, D] per head, or
    [Ly, 1, S, K, D] pooled (memoised, returned read-only); K = cfg.N.

    The paper trains them by k-means on KV from a disjoint span of the same
    text; here stage s draws K codewords from the data's own per-channel
    distribution (a disjoint Philox stream) shrunk by STAGE_SHRINK**s, standing
    in for samples of the stage-s residual.  A pooled codebook serves every
    head of its layer, so codeword j draws from head j mod H's distribution."""
    S = cfg.stages_k if kv == 0 else cfg.stages_v
    Ly, D = cfg.n_layers, cfg.dim
    H = 1 if cfg.pooled else cfg.n_heads
    K = cfg.N
    l, h, s, j, d = np.meshgrid(np.arange(Ly), np.arange(H), np.arange(S), np.arange(K),
                                np.arange(D), indexing="ij")
    flat = ((((l * H + h) * S + s) * K + j) * D + d).astype(np.int64)
    z = irwin_hall(flat, TID_CB_K if kv == 0 else TID_CB_V, cfg.cfg_id)
    hs = j % cfg.n_heads if cfg.pooled else h
    sig = channel_sigma(cfg, kv)[l, hs, d] * (STAGE_SHRINK ** s)
    sc = (sig / IRWIN_HALL_STD).astype(np.float32)
    out = (z.astype(np.float32) * sc).astype(np.float32)
    out.flags.writeable = False
    return out


# ----------------------------------------------------------- symbol streams --
def zipf_thresholds(N: int, s: float = 1.1) -> np.ndarray:
    """uint64 thresholds T_k = floor(CDF_k * 2**32), k = 0..N-2, of Zipf(s) over
    ranks 1..N with symbol 0 the most frequent."""
    w = np.arange(1, N + 1, dtype=np.float64) ** (-s)
    cdf = np.cumsum(w) / w.sum()
    return np.floor(cdf[:-1] * 2.0 ** 32).astype(np.uint64)


def symbols(N: int, dist: str, stream: int, index, cfg_id: int = 2) -> np.ndarray:
    """Symbol at each flat index of a stream: 'uniform' -> floor(w N / 2**32),
    'zipf' -> inverse-CDF of Zipf(1.1).  uint16 (fits any N <= 65536)."""
    e = np.asarray(index, np.uint64) + (np.uint64(stream) << np.uint64(40))
    w = uniform_u32(e, TID_SYM + (0 if dist == "uniform" else 16) + 32 * N, cfg_id).astype(np.uint64)
    if dist == "uniform":
        return ((w * np.uint64(N)) >> np.uint64(32)).astype(np.uint16)
    if dist == "zipf":
        return np.searchsorted(zipf_thresholds(N), w, side="right").astype(np.uint16)
    raise ValueError(dist)


def positions(n: int, count: int, stream: int, cfg_id: int = 2, salt: int = 0) -> np.ndarray:
    """`count` seeded uniform positions in [0, n) (n < 2**32)."""
    e = np.arange(count, dtype=np.uint64) + (np.uint64(stream) << np.uint64(40))
    w = uniform_u32(e, TID_POS + 64 * salt, cfg_id).astype(np.uint64)
    return ((w * np.uint64(n)) >> np.uint64(32)).astype(np.int64)


# ------------------------------------------------- device-side generation --
import ctypes as _ct
import os as _os
import subprocess as _sp
import threading as _th

_SYN_DIR = _os.path.dirname(_os.path.abspath(__file__))
_SYN_SRC = _os.path.join(_SYN_DIR, "csrc", "synth_gen.cu")
_SYN_LIB = _os.path.join(_SYN_DIR, "_build", "libsynth.so")
_syn_lock = _th.Lock()
_syn = None


def build(force: bool = False) -> str:
    """Compile csrc/synth_gen.cu into _build/libsynth.so (nvcc, sm_103a)."""
    _os.makedirs(_os.path.dirname(_SYN_LIB), exist_ok=True)
    if (not force and _os.path.exists(_SYN_LIB)
            and _os.path.getmtime(_SYN_LIB) >= _os.path.getmtime(_SYN_SRC)):
        return _SYN_LIB
    tmp = _SYN_LIB + ".tmp%d" % _os.getpid()
    nvcc = "/usr/local/cuda/bin/nvcc" if _os.path.exists("/usr/local/cuda/bin/nvcc") else "nvcc"
    _sp.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-Xcompiler", "-fPIC", "-shared",
             _SYN_SRC, "-o", tmp], check=True)
    _os.replace(tmp, _SYN_LIB)
    return _SYN_LIB


def _gpu():
    global _syn
    with _syn_lock:
        if _syn is None:
            L = _ct.CDLL(build())
            i64, u32, u64, p = _ct.c_int64, _ct.c_uint32, _ct.c_uint64, _ct.c_void_p
            L.synth_gen_kv.argtypes = [p, _ct.c_int, i64, i64, i64, i64, i64, i64, i64, u32, u32, u32, p, p]
            L.synth_gen_symbols.argtypes = [p, i64, u64, u32, u32, _ct.c_int, p, u32, u32, p]
            L.synth_gen_positions.argtypes = [p, i64, u64, u32, u64, u32, u32, i64, i64, p]
            _syn = L
        return _syn


def gpu_kv_cache(cfg: KVConfig, kv: int, device="cuda", out=None, t0: int = 0, count: int = None):
    """The cache [Ly, B, H, T, D] generated on the device (torch tensor),
    element for element equal to kv_cache()/kv_elements(); with t0/count only
    positions [t0, t0 + count) of it, as [Ly, B, H, count, D] (for caches too
    large to hold whole)."""
    import torch
    tdt = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[cfg.dtype]
    Ly, B, H, T, D = cfg.cache_shape()
    C = T - t0 if count is None else int(count)
    if out is None:
        out = torch.empty((Ly, B, H, C, D), dtype=tdt, device=device)
    scale = torch.from_numpy(channel_scale32(cfg, kv)).to(device)
    k0, k1 = seed_key(cfg.cfg_id)
    rc = _gpu().synth_gen_kv(out.data_ptr(), {"f32": 0, "f16": 1, "bf16": 2}[cfg.dtype], Ly, B, H, T, D, int(t0), C,
                             TID_K if kv == 0 else TID_V, k0, k1, scale.data_ptr(),
                             torch.cuda.current_stream().cuda_stream)
    if rc != 0:
        raise RuntimeError("synth_gen_kv failed (%d)" % rc)
    torch.cuda.current_stream().synchronize()
    return out


def gpu_symbols(N: int, dist: str, n_streams: int, n: int, device="cuda", cfg_id: int = 2, first_stream: int = 0):
    """[n_streams, n] symbol streams on the device, equal to symbols(): uint8
    for N <= 256, else int16 holding the uint16 symbols."""
    import torch
    out = torch.empty((n_streams, n), dtype=torch.uint8 if N <= 256 else torch.int16, device=device)
    thr = torch.from_numpy(zipf_thresholds(N).astype(np.uint32)).to(device)
    k0, k1 = seed_key(cfg_id)
    tid = TID_SYM + (0 if dist == "uniform" else 16) + 32 * N
    for s in range(n_streams):
        rc = _gpu().synth_gen_symbols(out[s].data_ptr(), n, first_stream + s, tid, N, int(dist == "zipf"),
                                      thr.data_ptr(), k0, k1, torch.cuda.current_stream().cuda_stream)
        if rc != 0:
            raise RuntimeError("synth_gen_symbols failed (%d)" % rc)
    return out


def gpu_positions(n: int, count: int, stream: int, device="cuda", cfg_id: int = 2, salt: int = 0):
    """int64 [count] positions on the device, equal to positions()."""
    import torch
    out = torch.empty(count, dtype=torch.int64, device=device)
    k0, k1 = seed_key(cfg_id)
    rc = _gpu().synth_gen_positions(out.data_ptr(), count, stream, TID_POS + 64 * salt, n, k0, k1, 1, 0,
                                    torch.cuda.current_stream().cuda_stream)
    if rc != 0:
        raise RuntimeError("synth_gen_positions failed (%d)" % rc)
    return out
