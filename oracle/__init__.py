"""Float64 CPU oracle of the fractal KV-cache archive -- TEST INFRASTRUCTURE.

This package is the slow, obviously-correct restatement of the paper
(arXiv 2607.07144) that the CUDA library is checked against.  Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it; the library never does, and the two share no code.

The arithmetic lives in ``fkv_oracle.c`` (plain C, binary64, no FMA
contraction); this module compiles it with gcc, marshals numpy arrays to it
and adds the bookkeeping the paper states in words:

* the exact window of Sec. 3 "Setup" (4 sink + 32 recent positions kept),
* the token-record order of the archived index stream (a reading: the paper
  does not state it), and
* the round-to-nearest-even cast of a float64 reconstruction to fp16/bf16/fp32,
* the in-place suffix retrieval of Sec. 5,
* the lossy truncation of Sec. 4 (B-bit codes of the stored points, their
  packed layout, recency allocation across spans), and
* the probability-weighted maps of Sec. 6 eq. (1) (integer arithmetic coding
  with an add-one adaptive or a uniform model).

Pins (tests/test_oracle_*.py): r_N = 1/2 at N = 3, 4 and a brute-force
disjointness bisection for other N; the N = 3 and N = 4 midpoint closed forms
(hand-worked points in tests/golden/) and exact rational evaluation of the
map's closed form; exhaustive round
trips of tiny streams and the 44/log2(1/r) capacity; the 2 r^s suffix decay;
RVQ against brute force and codeword-equal inputs; the storage identities of
Sec. 3; hand-computed lossy codes and layouts with the lossless limit; the
uniform arithmetic code's plain-binary pattern and the code-length bound.
Parity unpinned: the paper's printed byte counts of Table 2, Table 3's lossy
rates and Table 4's bits per character (they need the paper's corpus and
trained codebooks; the functions computing them are pinned as above).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fkv_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

# Sec. 3 "Setup": the first 4 positions (attention sinks) and the most recent
# 32 stay exact; every other position is archived.
SINK_TOKENS = 4
RECENT_TOKENS = 32
CODEWORDS = 256  # k = 256 codewords per stage (Sec. 3, Table 2)


def build(force: bool = False) -> str:
    """Compile fkv_oracle.c into _build/liboracle.so (gcc, no FMA contraction)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
           "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        I = ctypes.c_int
        D = ctypes.c_double
        lib.oracle_vertices.argtypes = [I, P]
        lib.oracle_vertices.restype = None
        lib.oracle_packing_ratio.argtypes = [I]
        lib.oracle_packing_ratio.restype = D
        lib.oracle_max_span_len.argtypes = [D]
        lib.oracle_max_span_len.restype = I
        lib.oracle_span_encode.argtypes = [P, D, I, P, I64, P]
        lib.oracle_span_encode.restype = None
        lib.oracle_span_decode.argtypes = [P, I, D, I, P, I64, P, P, D]
        lib.oracle_span_decode.restype = I64
        lib.oracle_rvq_encode.argtypes = [P, I64, I, P, I, I, P, P]
        lib.oracle_rvq_encode.restype = None
        lib.oracle_rvq_decode.argtypes = [P, I64, I, P, I, I, P]
        lib.oracle_rvq_decode.restype = None
        lib.oracle_ac_encode.argtypes = [P, I64, I, I, P, I64]
        lib.oracle_ac_encode.restype = I64
        lib.oracle_ac_decode.argtypes = [P, I64, I64, I, I, P]
        lib.oracle_ac_decode.restype = I
        lib.oracle_threads.argtypes = []
        lib.oracle_threads.restype = I
        _lib = lib
        return lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def threads() -> int:
    """OpenMP threads the oracle runs on."""
    return int(_load().oracle_threads())


# ---------------------------------------------------------------- geometry --
def vertices(N: int) -> np.ndarray:
    """Sec. 1: the regular N-gon's vertices, [N, 2] float64."""
    V = np.empty((N, 2), np.float64)
    _load().oracle_vertices(int(N), _ptr(V))
    return V


def packing_ratio(N: int) -> float:
    """Sec. 1 / Fig. 1: kissing ratio r_N (N-flake reading)."""
    return float(_load().oracle_packing_ratio(int(N)))


def max_span_len(r: float) -> int:
    """Sec. 1: floor(44 / log2(1/r)) symbols per stored double."""
    return int(_load().oracle_max_span_len(float(r)))


def n_spans(n: int, L: int) -> int:
    return (int(n) + L - 1) // L


# ------------------------------------------------------------ span codec ---
def span_encode(sym, N: int, r: float, L: int) -> np.ndarray:
    """Sec. 1: stored point of every span, [ceil(n/L), 2] float64."""
    s = np.ascontiguousarray(sym, dtype=np.int32).ravel()
    if s.size and (s.min() < 0 or s.max() >= N):
        raise ValueError("symbol outside the alphabet")
    V = vertices(N)
    pts = np.empty((n_spans(s.size, L), 2), np.float64)
    _load().oracle_span_encode(_ptr(V), float(r), int(L), _ptr(s), s.size, _ptr(pts))
    return pts


def span_decode(pts, n: int, N: int, r: float, L: int, tol: float = 2.0 ** -4):
    """Sec. 1 inverse map.  Returns (symbols int32 [n], anchor residual [spans],
    number of spans failing the anchor check)."""
    p = np.ascontiguousarray(pts, dtype=np.float64).reshape(-1, 2)
    if p.shape[0] != n_spans(n, L):
        raise ValueError("point count does not match n and L")
    V = vertices(N)
    sym = np.empty(int(n), np.int32)
    anchor = np.empty(p.shape[0], np.float64)
    bad = _load().oracle_span_decode(_ptr(V), int(N), float(r), int(L), _ptr(p),
                                     int(n), _ptr(sym), _ptr(anchor), float(tol))
    return sym, anchor, int(bad)


def read(pts, n: int, positions, N: int, r: float, L: int) -> np.ndarray:
    """O(1) random access (Sec. 2): the symbol at each position, by decoding
    only the span that holds it.  Defined as equal to the full decode there."""
    p = np.ascontiguousarray(pts, dtype=np.float64).reshape(-1, 2)
    pos = np.asarray(positions, dtype=np.int64).ravel()
    if pos.size and (pos.min() < 0 or pos.max() >= n):
        raise IndexError("position outside the stream")
    out = np.empty(pos.size, np.int32)
    spans = pos // L
    for u in np.unique(spans):
        m = min(L, int(n) - int(u) * L)
        sym, _, _ = span_decode(p[u:u + 1], m, N, r, L)
        sel = spans == u
        out[sel] = sym[pos[sel] - u * L]
    return out


def append(sym_old, sym_new, N: int, r: float, L: int) -> np.ndarray:
    """O(1) amortised append (Sec. 2), defined as the from-scratch encode of
    the extended stream."""
    s = np.concatenate([np.asarray(sym_old, np.int32).ravel(),
                        np.asarray(sym_new, np.int32).ravel()])
    return span_encode(s, N, r, L)


# ------------------------------------------------------------------- RVQ ---
def rvq_encode(x, cb):
    """Sec. 3 "Setup": residual VQ.  x [n, D] (any float dtype, taken exactly
    into float64), cb [S, K, D] float32.  Returns (idx int32 [n, S],
    gap [n, S]) where gap is (second - best) / ||residual||^2 per stage."""
    xx = np.ascontiguousarray(x, dtype=np.float64)
    c = np.ascontiguousarray(cb, dtype=np.float32)
    n, D = xx.shape
    S, K, D2 = c.shape
    if D2 != D or D > 1024:
        raise ValueError("codebook / vector dimension mismatch")
    idx = np.empty((n, S), np.int32)
    gap = np.empty((n, S), np.float64)
    _load().oracle_rvq_encode(_ptr(xx), n, D, _ptr(c), S, K, _ptr(idx), _ptr(gap))
    return idx, gap


def rvq_decode(idx, cb) -> np.ndarray:
    """Sec. 3 "Setup": float64 sum of the selected centroids, [n, D]."""
    i = np.ascontiguousarray(idx, dtype=np.int32)
    c = np.ascontiguousarray(cb, dtype=np.float32)
    n, S = i.shape
    S2, K, D = c.shape
    if S2 < S:
        raise ValueError("more stages than codebooks")
    y = np.empty((n, D), np.float64)
    _load().oracle_rvq_decode(_ptr(i), n, D, _ptr(c), S, K, _ptr(y))
    return y


# --------------------------------------------------------------- rounding --
def round_to(y, dtype: str) -> np.ndarray:
    """Round-to-nearest-even of float64 values to 'f32', 'f16' or 'bf16'.
    Returns float64 holding the rounded values (bf16 has no numpy type)."""
    y = np.asarray(y, np.float64)
    if dtype == "f32":
        return y.astype(np.float32).astype(np.float64)
    if dtype == "f16":
        return y.astype(np.float16).astype(np.float64)
    if dtype == "bf16":
        return _round_binary(y, mant_bits=8, emin=-126, emax=127)
    raise ValueError(dtype)


def _round_binary(y, mant_bits: int, emin: int, emax: int) -> np.ndarray:
    """Round float64 to a binary format with mant_bits significant bits and the
    normal exponent range [emin, emax] (subnormals below), ties to even."""
    out = np.zeros_like(y)
    nz = (y != 0) & np.isfinite(y)
    m, e = np.frexp(y[nz])          # y = m * 2**e, 0.5 <= |m| < 1
    e = np.maximum(e, emin + 1)     # subnormal range keeps a fixed quantum
    q = np.ldexp(np.rint(np.ldexp(y[nz], mant_bits - e)), e - mant_bits)
    big = np.abs(q) >= np.ldexp(1.0, emax + 1)
    q[big] = np.copysign(np.inf, q[big])
    out[nz] = q
    out[~np.isfinite(y)] = y[~np.isfinite(y)]
    return out


# ----------------------------------------------------------- KV archive ---
def archived_positions(T: int):
    """Sec. 3 "Setup": positions [4, T - 32) leave the exact window."""
    return range(SINK_TOKENS, max(SINK_TOKENS, T - RECENT_TOKENS))


def record_len(n_heads: int, stages_k: int, stages_v: int) -> int:
    return n_heads * (stages_k + stages_v)


def records_from_indices(idx_k, idx_v) -> np.ndarray:
    """Token-record order of one (sequence, layer) index stream (a reading;
    the paper does not state it): for each archived position, the key indices
    of head 0..H-1 with each head's stages 0..S_K-1, then the value indices in
    the same order.  idx_k [H, P, S_K], idx_v [H, P, S_V] -> int32 [P * R]."""
    k = np.asarray(idx_k, np.int32)
    v = np.asarray(idx_v, np.int32)
    H, P, SK = k.shape
    _, _, SV = v.shape
    kk = k.transpose(1, 0, 2).reshape(P, H * SK)
    vv = v.transpose(1, 0, 2).reshape(P, H * SV)
    return np.concatenate([kk, vv], axis=1).reshape(-1)


def indices_from_records(stream, n_heads: int, stages_k: int, stages_v: int):
    """Inverse of records_from_indices: -> (idx_k [H, P, S_K], idx_v [H, P, S_V])."""
    R = record_len(n_heads, stages_k, stages_v)
    s = np.asarray(stream, np.int32).reshape(-1, R)
    P = s.shape[0]
    k = s[:, :n_heads * stages_k].reshape(P, n_heads, stages_k).transpose(1, 0, 2)
    v = s[:, n_heads * stages_k:].reshape(P, n_heads, stages_v).transpose(1, 0, 2)
    return np.ascontiguousarray(k), np.ascontiguousarray(v)


# ------------------------------------------------------- suffix retrieval ---
def suffix_radius2(r: float, qlen: int) -> float:
    """Sec. 5: positions sharing an l-symbol suffix have points within 2 r^l of
    each other.  The squared radius (2 r^l)^2 of the retrieval ball, with r^l
    formed by l successive binary64 multiplications."""
    rl = 1.0
    for _ in range(int(qlen)):
        rl = rl * r
    t = 2.0 * rl
    return t * t


def suffix_search(pts, n: int, query, N: int, r: float, L: int):
    """Sec. 5 retrieval on one span-anchored stream, done in place.

    The query (l symbols, 1 <= l <= L) is encoded from the origin by the Sec. 1
    map.  A stored point within the 2 r^l ball is a candidate; a candidate is a
    match when its span's last l symbols equal the query, which the decode
    verifies.  A span-end point carries only its own span's symbols, so a span
    shorter than l is never a candidate.  Returns (matches, candidates): sorted
    int64 arrays of span indices."""
    qs = np.asarray(query, dtype=np.int32).ravel()
    l = qs.size
    if l < 1 or l > L:
        raise ValueError("query length outside [1, L]")
    p = np.ascontiguousarray(pts, dtype=np.float64).reshape(-1, 2)
    spans = p.shape[0]
    if spans != n_spans(n, L):
        raise ValueError("point count does not match n and L")
    q = span_encode(qs, N, r, l)[0]                  # the query's point, one span from the origin
    m = np.minimum(L, int(n) - np.arange(spans, dtype=np.int64) * L)
    dx = p[:, 0] - q[0]
    dy = p[:, 1] - q[1]
    d2 = dx * dx + dy * dy
    cand = np.nonzero((m >= l) & (d2 <= suffix_radius2(r, l)))[0].astype(np.int64)
    sym, _, _ = span_decode(p, n, N, r, L)
    match = [u for u in cand
             if np.array_equal(sym[u * L + m[u] - l:u * L + m[u]], qs)]
    return np.asarray(match, dtype=np.int64), cand


# ------------------------------------------------------ lossy truncation ---
def truncate_codes(pts, bits: int) -> np.ndarray:
    """Sec. 4: truncating a code point to B bits.  Reading: each coordinate
    x of a stored point (|x| < 1) becomes the B-bit two's complement code
    k = floor(x * 2^(B-1)) (one sign bit, B-1 fraction bits), so that
    k * 2^-(B-1) is x with every bit below 2^-(B-1) dropped.  Exact in binary64
    (power-of-two scaling and floor).  Returns int64 [spans, 2]."""
    if not 2 <= bits <= 53:
        raise ValueError("bits outside [2, 53]")
    p = np.ascontiguousarray(pts, dtype=np.float64).reshape(-1, 2)
    return np.floor(np.ldexp(p, bits - 1)).astype(np.int64)


def truncated_points(codes, bits: int) -> np.ndarray:
    """The truncated point k * 2^-(B-1) of each code, float64 [spans, 2] (exact)."""
    return np.ldexp(np.asarray(codes, dtype=np.int64).reshape(-1, 2).astype(np.float64), -(bits - 1))


def pack_codes(codes, bits: int) -> np.ndarray:
    """Packed form of one stream's codes (a reading: the paper keeps B bits per
    point but fixes no format).  Span u's x code occupies bits
    [2uB, 2uB + B) and its y code bits [2uB + B, 2uB + 2B) of a stream of
    uint32 words, bit i of the stream being bit i % 32 of word i // 32, each
    code as a B-bit two's complement field, least significant bit first.
    Returns uint32 [ceil(2 * spans * B / 32)]."""
    c = np.asarray(codes, dtype=np.int64).reshape(-1)            # x0, y0, x1, y1, ...
    field = c & np.int64((1 << bits) - 1)                        # B-bit two's complement
    bitmat = ((field[:, None] >> np.arange(bits, dtype=np.int64)[None, :]) & 1).astype(np.uint8)
    flat = bitmat.reshape(-1)                                    # stream bit i = flat[i]
    nwords = (flat.size + 31) // 32
    flat = np.concatenate([flat, np.zeros(nwords * 32 - flat.size, np.uint8)])
    by = np.packbits(flat, bitorder="little")                    # byte j holds bits 8j .. 8j+7
    return by.view("<u4").astype(np.uint32)


def lossy_points(pts, bits: int, keep_exact: int) -> np.ndarray:
    """Sec. 4, recency allocation across spans: the stream's last keep_exact
    spans keep their exact points, every earlier span its B-bit truncated
    point.  float64 [spans, 2]."""
    p = np.ascontiguousarray(pts, dtype=np.float64).reshape(-1, 2).copy()
    t = max(0, p.shape[0] - int(keep_exact))
    p[:t] = truncated_points(truncate_codes(p[:t], bits), bits)
    return p


def lossy_decode(pts, n: int, N: int, r: float, L: int, bits: int, keep_exact: int) -> np.ndarray:
    """Sec. 4: the symbols a decoder recovers from the lossy archive -- the
    Sec. 1 inverse map (span_decode: nearest vertex, binary64 inverse step) run
    from each span's kept point.  Truncation perturbs the point by less than
    2^-(B-1) per coordinate and the inverse map amplifies that by 1/r per step,
    so a span's last symbols stay exact and its first ones degrade.  int32 [n]."""
    sym, _, _ = span_decode(lossy_points(pts, bits, keep_exact), n, N, r, L)
    return sym


# ------------------------------------------- probability-weighted maps ---
def ac_capacity_words(n: int, N: int) -> int:
    """Words that always hold the code of n symbols: a step emits at most
    log2(T / count) + 1 <= ceil(log2(N + n)) + 1 bits, plus two final bits."""
    per = int(np.ceil(np.log2(N + n))) + 1
    return (int(n) * per + 2 + 31) // 32 + 1


def ac_encode(sym, N: int, adaptive: bool = True):
    """Sec. 6 eq. (1): arithmetic coding of one stream (oracle_ac_encode).
    Returns (uint32 words, number of bits)."""
    s = np.ascontiguousarray(sym, dtype=np.int32).ravel()
    if s.size and (s.min() < 0 or s.max() >= N):
        raise ValueError("symbol outside the alphabet")
    cap = ac_capacity_words(s.size, N)
    out = np.zeros(cap, np.uint32)
    nb = _load().oracle_ac_encode(_ptr(s), s.size, int(N), int(bool(adaptive)), _ptr(out), cap)
    if nb < 0:
        raise RuntimeError("code longer than its bound")
    return out[:(nb + 31) // 32].copy(), int(nb)


def ac_decode(words, nbits: int, n: int, N: int, adaptive: bool = True) -> np.ndarray:
    """The inverse of ac_encode: int32 [n]."""
    w = np.ascontiguousarray(words, dtype=np.uint32)
    sym = np.empty(int(n), np.int32)
    _load().oracle_ac_decode(_ptr(w), int(nbits), int(n), int(N), int(bool(adaptive)), _ptr(sym))
    return sym


def ac_model_bits(sym, N: int, adaptive: bool = True) -> float:
    """Sec. 6: the model's code length -sum_k log2 p(c_k) in bits (float64),
    p from the same add-one counts the coder uses."""
    s = np.asarray(sym, dtype=np.int64).ravel()
    if not adaptive:
        return float(s.size * np.log2(N))
    cnt = np.ones(N, np.float64)
    bits = 0.0
    for k, c in enumerate(s):                      # pure-Python loop: small cases
        bits -= np.log2(cnt[c] / (N + k))
        cnt[c] += 1.0
    return bits

