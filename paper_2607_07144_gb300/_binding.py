"""ctypes binding of libfkv.so (include/fkv.h).  Argument marshalling only:
every step of the archive path runs in the library's CUDA kernels.  PyTorch
supplies device memory and the current CUDA stream."""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libfkv.so")

OK, EINVAL, ERANGE, ENOMEM, ECUDA, ECORRUPT, ETIMEOUT = 0, -1, -2, -3, -4, -5, -6
F32, F16, BF16 = 0, 1, 2
_DTYPE = {torch.float32: F32, torch.float16: F16, torch.bfloat16: BF16}
_ERRNAME = {EINVAL: "EINVAL", ERANGE: "ERANGE", ENOMEM: "ENOMEM", ECUDA: "ECUDA",
            ECORRUPT: "ECORRUPT", ETIMEOUT: "ETIMEOUT"}

_lock = threading.Lock()
_lib = None


class FkvError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("%s (%d): %s" % (_ERRNAME.get(code, "?"), code, msg))
        self.code = code


class _Codebooks(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("n_heads", ctypes.c_int), ("dim", ctypes.c_int),
                ("stages_k", ctypes.c_int), ("stages_v", ctypes.c_int),
                ("k", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("codewords", ctypes.c_int), ("pooled", ctypes.c_int)]


class _Cache(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("dtype", ctypes.c_int), ("batch", ctypes.c_int64),
                ("seq", ctypes.c_int64), ("stride_layer", ctypes.c_int64),
                ("stride_batch", ctypes.c_int64), ("stride_head", ctypes.c_int64),
                ("stride_pos", ctypes.c_int64)]


# name -> (restype, argtypes)
_P, _I, _I64, _D = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_double
SIGNATURES = {
    "fkv_packing_ratio": (_D, [_I]),
    "fkv_max_span_len": (_I, [_D]),
    "fkv_create": (_I, [_I, _D, _I, _P, ctypes.POINTER(_P)]),
    "fkv_destroy": (_I, [_P]),
    "fkv_vertices": (_I, [_P, _P]),
    "fkv_params": (_I, [_P, _P, _P, _P]),
    "fkv_symbol_bytes": (_I, [_P]),
    "fkv_last_error": (ctypes.c_char_p, [_P]),
    "fkv_sync_status": (_I, [_P, _P]),
    "fkv_span_encode": (_I, [_P, _P, _I64, _I64, _I64, _P, _I64, _P]),
    "fkv_span_decode": (_I, [_P, _P, _I64, _I64, _I64, _P, _I64, _P]),
    "fkv_read": (_I, [_P, _P, _I64, _I64, _I64, _P, _I64, _P, _P]),
    "fkv_span_encode_ragged": (_I, [_P, _P, _P, _I64, _P, _P, _P]),
    "fkv_span_decode_ragged": (_I, [_P, _P, _P, _I64, _P, _P, _P]),
    "fkv_read_ragged": (_I, [_P, _P, _P, _P, _I64, _P, _I64, _P, _P]),
    "fkv_suffix_search": (_I, [_P, _P, _I64, _I64, _I64, _P, _I, _P, _I64, _P, _P]),
    "fkv_truncate": (_I, [_P, _P, _I64, _I64, _I64, _I, _I64, _P, _I64, _P, _I64, _P]),
    "fkv_lossy_decode": (_I, [_P, _P, _I64, _P, _I64, _I64, _I64, _I, _I64, _P, _I64, _P]),
    "fkv_lossy_read": (_I, [_P, _P, _I64, _P, _I64, _I64, _I64, _I, _I64, _P, _I64, _P, _P]),
    "fkv_ac_capacity_words": (_I64, [_P, _I64]),
    "fkv_ac_encode": (_I, [_P, _P, _I64, _I64, _I64, _I, _P, _I64, _P, _P]),
    "fkv_ac_decode": (_I, [_P, _P, _I64, _P, _I64, _I64, _I, _P, _I64, _P]),
    "fkv_measure_fp64_rate": (_I, [_P, _P]),
    "fkv_check_bounded_wait": (_I, [_P, _I64, _P, _P]),
    "fkv_record_len": (_I, [_P]),
    "fkv_rvq_encode": (_I, [_P, _I, _P, _I64, _I64, _P, _I64, _I64, _P]),
    "fkv_rvq_decode": (_I, [_P, _P, _I64, _I64, _P, _P, _I64, _P]),
    "fkv_decode_kv": (_I, [_P, _P, _I64, _I64, _P, _P, _I64, _P]),
    "fkv_decode_kv_static": (_I, [_P, _P, _I64, _I64, _P, _P, _I64, _P]),
    "fkv_read_kv": (_I, [_P, _P, _I64, _I64, _I64, _P, _I64, _P, _I, _P]),
    "fkv_cache_upload": (_I, [_P, _P, _P, _I64, _I64, _P]),
    "fkv_streams_create": (_I, [_P, _I64, _I64, ctypes.POINTER(_P)]),
    "fkv_streams_destroy": (_I, [_P]),
    "fkv_streams_reset": (_I, [_P]),
    "fkv_streams_info": (_I, [_P, _P, _P, _P, _P]),
    "fkv_append": (_I, [_P, _P, _P, _I64, _I64, _P]),
    "fkv_streams_export": (_I, [_P, _P, _P, _P]),
    "fkv_streams_import": (_I, [_P, _I64, _I64, _P, ctypes.POINTER(_P)]),
}


def lib():
    """The loaded library.  Raises if it has not been built: there is no
    fallback implementation."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError("libfkv.so is not built (run __graft_entry__.build())")
            L = ctypes.CDLL(LIB_PATH)
            for name, (res, args) in SIGNATURES.items():
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
        return _lib


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t: torch.Tensor):
    return ctypes.c_void_p(t.data_ptr())


def _rows(t: torch.Tensor, unit: int = 1) -> int:
    """Row stride of a [rows, ...] tensor in units of `unit` elements; a
    single row has no meaningful stride, so report its own extent."""
    if t.shape[0] <= 1:
        return max(1, t[0].numel() // unit if t.shape[0] else 1)
    return t.stride(0) // unit


def packing_ratio(N: int) -> float:
    return lib().fkv_packing_ratio(int(N))


def max_span_len(r: float) -> int:
    return lib().fkv_max_span_len(float(r))


def measure_fp64_rate(stream=None) -> float:
    """Binary64 add/mul instructions per second of the current device."""
    v = ctypes.c_double()
    rc = lib().fkv_measure_fp64_rate(ctypes.byref(v), _stream(stream))
    if rc != OK:
        raise FkvError(rc, "fkv_measure_fp64_rate failed")
    return v.value


def cache_view(t: torch.Tensor, host: bool = False) -> _Cache:
    """fkv_cache view of a tensor shaped [n_layers, batch, n_heads, seq, dim]
    (any strides with a contiguous last dimension): a CUDA tensor, or with
    host=True a CPU tensor (pinned for full transfer speed)."""
    if t.dim() != 5 or t.stride(4) != 1 or t.is_cuda == host:
        raise ValueError("cache must be a %s tensor [layers, batch, heads, seq, dim] with contiguous dim"
                         % ("CPU" if host else "CUDA"))
    c = _Cache()
    c.data = t.data_ptr()
    c.dtype = _DTYPE[t.dtype]
    c.batch = t.shape[1]
    c.seq = t.shape[3]
    c.stride_layer, c.stride_batch, c.stride_head, c.stride_pos = t.stride(0), t.stride(1), t.stride(2), t.stride(3)
    return c


class Context:
    """An fkv_ctx: alphabet N, ratio r (default r_N), span length (default
    floor(44/log2(1/r))) and optional codebooks (k, v) as float32 arrays
    [n_layers, n_heads, stages, N, dim] (N = 256 or 1024 codewords per stage),
    or, pooled (one codebook per layer shared by its heads), arrays
    [n_layers, 1, stages, N, dim] with the head count given as n_heads."""

    def __init__(self, N: int, r: float = None, span_len: int = None, codebooks=None, pooled: bool = False,
                 n_heads: int = None):
        L = lib()
        self.N = int(N)
        self.r = float(r) if r is not None else L.fkv_packing_ratio(self.N)
        self.L = int(span_len) if span_len is not None else L.fkv_max_span_len(self.r)
        self._h = ctypes.c_void_p()
        cbp = None
        if codebooks is not None:
            k, v = (np.ascontiguousarray(a, np.float32) for a in codebooks)
            if (k.ndim != 5 or v.ndim != 5 or k.shape[:2] != v.shape[:2] or k.shape[3:] != v.shape[3:]
                    or (pooled and k.shape[1] != 1)):
                raise ValueError("codebooks must be [layers, heads (1 if pooled), stages, codewords, dim]")
            H = int(n_heads) if pooled else k.shape[1]
            if pooled and n_heads is None:
                raise ValueError("pooled codebooks need n_heads")
            self._cb_arrays = (k, v)          # keep alive during create
            cb = _Codebooks(k.shape[0], H, k.shape[4], k.shape[2], v.shape[2],
                            k.ctypes.data, v.ctypes.data, k.shape[3], int(bool(pooled)))
            cbp = ctypes.byref(cb)
            self.n_layers, self.n_heads, self.dim = k.shape[0], H, k.shape[4]
            self.pooled = bool(pooled)
            self.stages_k, self.stages_v = k.shape[2], v.shape[2]
        rc = L.fkv_create(self.N, self.r, self.L, cbp, ctypes.byref(self._h))
        self._cb_arrays = None
        if rc != OK:
            raise FkvError(rc, "fkv_create(N=%d, r=%r, span_len=%d) rejected" % (self.N, self.r, self.L))
        # symbols are uint8 up to N = 256, uint16 above; torch.int16 holds the
        # uint16 symbols bit for bit (every symbol is below 1024)
        self.sym_bytes = L.fkv_symbol_bytes(self._h)
        self.sym_dtype = torch.uint8 if self.sym_bytes == 1 else torch.int16

    # -- plumbing
    def _check(self, rc):
        if rc != OK:
            raise FkvError(rc, lib().fkv_last_error(self._h).decode())

    def _sym(self, t: torch.Tensor) -> torch.Tensor:
        if t.element_size() != self.sym_bytes:
            raise ValueError("symbols of this context are %d-byte integers, got %s" % (self.sym_bytes, t.dtype))
        return t

    def close(self):
        if self._h:
            lib().fkv_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def handle(self):
        return self._h

    # -- ABI calls
    def vertices(self) -> np.ndarray:
        out = np.empty((self.N, 2), np.float64)
        self._check(lib().fkv_vertices(self._h, out.ctypes.data))
        return out

    def record_len(self) -> int:
        return lib().fkv_record_len(self._h)

    def sync_status(self, stream=None) -> int:
        return lib().fkv_sync_status(self._h, _stream(stream))

    def check_bounded_wait(self, limit_ns: int, stream=None) -> list:
        """fkv_check_bounded_wait: the six results, as ints."""
        res = (ctypes.c_int32 * 6)()
        self._check(lib().fkv_check_bounded_wait(self._h, int(limit_ns), res, _stream(stream)))
        return list(res)

    def n_spans(self, n: int) -> int:
        return (int(n) + self.L - 1) // self.L

    def span_encode(self, sym: torch.Tensor, pts: torch.Tensor = None, stream=None) -> torch.Tensor:
        """sym [n_streams, n] (sym_dtype) -> pts float64 [n_streams, spans, 2]."""
        ns, n = self._sym(sym).shape
        if pts is None:
            pts = torch.empty((ns, self.n_spans(n), 2), dtype=torch.float64, device=sym.device)
        self._check(lib().fkv_span_encode(self._h, _ptr(sym), ns, n, _rows(sym), _ptr(pts), _rows(pts, 2),
                                          _stream(stream)))
        return pts

    def span_decode(self, pts: torch.Tensor, n: int, sym: torch.Tensor = None, stream=None) -> torch.Tensor:
        ns = pts.shape[0]
        if sym is None:
            sym = torch.empty((ns, n), dtype=self.sym_dtype, device=pts.device)
        self._sym(sym)
        self._check(lib().fkv_span_decode(self._h, _ptr(pts), ns, n, _rows(pts, 2), _ptr(sym), _rows(sym),
                                          _stream(stream)))
        return sym

    def read(self, pts: torch.Tensor, n: int, req: torch.Tensor, out: torch.Tensor = None, stream=None):
        """req int64 [n_req, 2] = (stream, position) -> symbols [n_req] (sym_dtype)."""
        if out is None:
            out = torch.empty(req.shape[0], dtype=self.sym_dtype, device=pts.device)
        self._sym(out)
        self._check(lib().fkv_read(self._h, _ptr(pts), pts.shape[0], n, _rows(pts, 2), _ptr(req), req.shape[0],
                                   _ptr(out), _stream(stream)))
        return out

    # -- ragged batches (streams of different lengths in one call)
    def ragged_offsets(self, lengths, device="cuda"):
        """Packed offsets for streams of the given lengths: (sym_off, pt_off),
        int64 [n_streams + 1] device tensors (points packed with no slack)."""
        ln = np.asarray(lengths, np.int64).ravel()
        so = np.concatenate([[0], np.cumsum(ln)]).astype(np.int64)
        po = np.concatenate([[0], np.cumsum((ln + self.L - 1) // self.L)]).astype(np.int64)
        return torch.from_numpy(so).to(device), torch.from_numpy(po).to(device)

    def span_encode_ragged(self, sym: torch.Tensor, sym_off: torch.Tensor, pt_off: torch.Tensor,
                           pts: torch.Tensor = None, n_slots: int = None, stream=None) -> torch.Tensor:
        """sym: flat symbols (sym_dtype) of all streams; sym_off, pt_off: int64
        [n_streams + 1] device offsets -> pts float64 [slots, 2] (n_slots, or
        pt_off's last entry read back, a synchronisation, when pts is None)."""
        self._sym(sym)
        ns = sym_off.numel() - 1
        if pts is None:
            slots = int(pt_off[-1].item()) if n_slots is None else int(n_slots)
            pts = torch.empty((max(slots, 1), 2), dtype=torch.float64, device=sym.device)
        self._check(lib().fkv_span_encode_ragged(self._h, _ptr(sym), _ptr(sym_off), ns, _ptr(pts), _ptr(pt_off),
                                                 _stream(stream)))
        return pts

    def span_decode_ragged(self, pts: torch.Tensor, pt_off: torch.Tensor, sym_off: torch.Tensor,
                           sym: torch.Tensor = None, n_sym: int = None, stream=None) -> torch.Tensor:
        ns = sym_off.numel() - 1
        if sym is None:
            n = int(sym_off[-1].item()) if n_sym is None else int(n_sym)
            sym = torch.empty(max(n, 1), dtype=self.sym_dtype, device=pts.device)
        self._sym(sym)
        self._check(lib().fkv_span_decode_ragged(self._h, _ptr(pts), _ptr(pt_off), ns, _ptr(sym), _ptr(sym_off),
                                                 _stream(stream)))
        return sym

    def read_ragged(self, pts: torch.Tensor, pt_off: torch.Tensor, sym_off: torch.Tensor, req: torch.Tensor,
                    out: torch.Tensor = None, stream=None) -> torch.Tensor:
        """req int64 [n_req, 2] = (stream, position within it) -> symbols [n_req]."""
        if out is None:
            out = torch.empty(req.shape[0], dtype=self.sym_dtype, device=pts.device)
        self._sym(out)
        self._check(lib().fkv_read_ragged(self._h, _ptr(pts), _ptr(pt_off), _ptr(sym_off), sym_off.numel() - 1,
                                          _ptr(req), req.shape[0], _ptr(out), _stream(stream)))
        return out

    def suffix_search(self, pts: torch.Tensor, n: int, query, cap: int = 1 << 16, match: torch.Tensor = None,
                      counts: torch.Tensor = None, stream=None):
        """Sec. 5 in-place retrieval: spans whose last len(query) symbols equal
        the query.  Returns (match int64 [min(count, cap), 2] = (stream, span)
        in no particular order, number of matches, number of candidates); reads
        the two counts back (a device synchronisation on `stream`)."""
        q = np.asarray(query).ravel()
        if q.size and (q.min() < 0 or q.max() >= 1 << (8 * self.sym_bytes)):
            raise ValueError("query symbol does not fit the symbol width")
        q = np.ascontiguousarray(q.astype(np.uint8 if self.sym_bytes == 1 else np.uint16))
        if match is None:
            match = torch.empty((max(cap, 1), 2), dtype=torch.int64, device=pts.device)
        if counts is None:
            counts = torch.empty(2, dtype=torch.int64, device=pts.device)
        self._check(lib().fkv_suffix_search(self._h, _ptr(pts), pts.shape[0], n, _rows(pts, 2),
                                            q.ctypes.data_as(ctypes.c_void_p), q.size, _ptr(match), cap,
                                            _ptr(counts), _stream(stream)))
        c = counts.cpu().tolist()
        return match[:min(c[0], cap)], c[0], c[1]

    # -- Sec. 6 probability-weighted maps (arithmetic coding)
    def ac_encode(self, sym: torch.Tensor, adaptive: bool = True, words: torch.Tensor = None,
                  nbits: torch.Tensor = None, stream=None):
        """sym [n_streams, n] -> (words int32 [n_streams, capacity] holding the
        uint32 code words, nbits int64 [n_streams])."""
        ns, n = self._sym(sym).shape
        cap = lib().fkv_ac_capacity_words(self._h, n)
        if words is None:
            words = torch.zeros((ns, cap), dtype=torch.int32, device=sym.device)
        if nbits is None:
            nbits = torch.empty(ns, dtype=torch.int64, device=sym.device)
        self._check(lib().fkv_ac_encode(self._h, _ptr(sym), ns, n, _rows(sym), int(bool(adaptive)), _ptr(words),
                                        _rows(words), _ptr(nbits), _stream(stream)))
        return words, nbits

    def ac_decode(self, words: torch.Tensor, nbits: torch.Tensor, n: int, adaptive: bool = True,
                  sym: torch.Tensor = None, stream=None) -> torch.Tensor:
        ns = words.shape[0]
        if sym is None:
            sym = torch.empty((ns, n), dtype=self.sym_dtype, device=words.device)
        self._sym(sym)
        self._check(lib().fkv_ac_decode(self._h, _ptr(words), _rows(words), _ptr(nbits), ns, n, int(bool(adaptive)),
                                        _ptr(sym), _rows(sym), _stream(stream)))
        return sym

    # -- Sec. 4 lossy archive
    def lossy_geometry(self, n: int, bits: int, keep_exact: int):
        """(truncated spans T, code words per stream, exact tail spans)."""
        S = self.n_spans(n)
        T = max(0, S - int(keep_exact))
        return T, (2 * T * int(bits) + 31) // 32, S - T

    def truncate(self, pts: torch.Tensor, n: int, bits: int, keep_exact: int, codes: torch.Tensor = None,
                 tail: torch.Tensor = None, stream=None):
        """pts float64 [n_streams, spans, 2] -> (codes int32 [n_streams, words]
        holding the uint32 code words, tail float64 [n_streams, S - T, 2])."""
        ns = pts.shape[0]
        T, words, ts = self.lossy_geometry(n, bits, keep_exact)
        if codes is None:
            codes = torch.empty((ns, max(words, 1)), dtype=torch.int32, device=pts.device)
        if tail is None:
            tail = torch.empty((ns, max(ts, 1), 2), dtype=torch.float64, device=pts.device)
        self._check(lib().fkv_truncate(self._h, _ptr(pts), ns, n, _rows(pts, 2), int(bits), int(keep_exact),
                                       _ptr(codes), _rows(codes), _ptr(tail), _rows(tail, 2), _stream(stream)))
        return codes, tail

    def lossy_decode(self, codes: torch.Tensor, tail: torch.Tensor, n: int, bits: int, keep_exact: int,
                     sym: torch.Tensor = None, stream=None) -> torch.Tensor:
        ns = codes.shape[0]
        if sym is None:
            sym = torch.empty((ns, n), dtype=self.sym_dtype, device=codes.device)
        self._sym(sym)
        self._check(lib().fkv_lossy_decode(self._h, _ptr(codes), _rows(codes), _ptr(tail), _rows(tail, 2), ns, n,
                                           int(bits), int(keep_exact), _ptr(sym), _rows(sym), _stream(stream)))
        return sym

    def lossy_read(self, codes: torch.Tensor, tail: torch.Tensor, n: int, bits: int, keep_exact: int,
                   req: torch.Tensor, out: torch.Tensor = None, stream=None) -> torch.Tensor:
        if out is None:
            out = torch.empty(req.shape[0], dtype=self.sym_dtype, device=codes.device)
        self._sym(out)
        self._check(lib().fkv_lossy_read(self._h, _ptr(codes), _rows(codes), _ptr(tail), _rows(tail, 2),
                                         codes.shape[0], n, int(bits), int(keep_exact), _ptr(req), req.shape[0],
                                         _ptr(out), _stream(stream)))
        return out

    def rvq_encode(self, kv: int, x: torch.Tensor, t0: int, t1: int, sym: torch.Tensor, rec0: int = 0, stream=None):
        """x: cache [layers, batch, heads, seq, dim]; sym: [batch*layers, >= (rec0+t1-t0)*R] of sym_dtype."""
        self._sym(sym)
        c = cache_view(x)
        self._check(lib().fkv_rvq_encode(self._h, int(kv), ctypes.byref(c), t0, t1, _ptr(sym), _rows(sym), rec0,
                                         _stream(stream)))
        return sym

    def rvq_decode(self, sym: torch.Tensor, n_rec: int, k_out: torch.Tensor = None, v_out: torch.Tensor = None,
                   t0: int = 0, stream=None):
        self._sym(sym)
        ck = cache_view(k_out) if k_out is not None else None
        cv = cache_view(v_out) if v_out is not None else None
        self._check(lib().fkv_rvq_decode(self._h, _ptr(sym), _rows(sym), n_rec,
                                         ctypes.byref(ck) if ck else None, ctypes.byref(cv) if cv else None,
                                         t0, _stream(stream)))

    def decode_kv(self, pts: torch.Tensor, n_rec: int, k_out: torch.Tensor = None, v_out: torch.Tensor = None,
                  t0: int = 0, stream=None):
        ck = cache_view(k_out) if k_out is not None else None
        cv = cache_view(v_out) if v_out is not None else None
        self._check(lib().fkv_decode_kv(self._h, _ptr(pts), n_rec, _rows(pts, 2),
                                        ctypes.byref(ck) if ck else None, ctypes.byref(cv) if cv else None,
                                        t0, _stream(stream)))

    def decode_kv_static(self, pts: torch.Tensor, n_rec: int, k_out: torch.Tensor = None,
                         v_out: torch.Tensor = None, t0: int = 0, stream=None):
        """decode_kv without any device allocation: the decoded symbols go
        through the library's fixed 16 MiB scratch array (for callers whose
        device memory must all come from their own allocator)."""
        ck = cache_view(k_out) if k_out is not None else None
        cv = cache_view(v_out) if v_out is not None else None
        self._check(lib().fkv_decode_kv_static(self._h, _ptr(pts), n_rec, _rows(pts, 2),
                                               ctypes.byref(ck) if ck else None, ctypes.byref(cv) if cv else None,
                                               t0, _stream(stream)))

    def cache_upload(self, src_host: torch.Tensor, dst: torch.Tensor, t0: int, t1: int, stream=None):
        """Copy positions [t0, t1) of a host cache (CPU tensor, pinned) into a device cache."""
        cs, cd = cache_view(src_host, host=True), cache_view(dst)
        self._check(lib().fkv_cache_upload(self._h, ctypes.byref(cs), ctypes.byref(cd), t0, t1, _stream(stream)))
        return dst

    def read_kv(self, pts: torch.Tensor, n_rec: int, req: torch.Tensor, out: torch.Tensor, stream=None):
        """req int64 [n_req, 2] = (stream, record) -> out [n_req, 2, heads, dim]."""
        self._check(lib().fkv_read_kv(self._h, _ptr(pts), pts.shape[0], n_rec, _rows(pts, 2), _ptr(req),
                                      req.shape[0], _ptr(out), _DTYPE[out.dtype], _stream(stream)))
        return out


class Streams:
    """An fkv_streams set: n_streams library-owned appendable streams."""

    def __init__(self, ctx: Context, n_streams: int, capacity: int = 0, _handle=None):
        self.ctx = ctx
        self._h = ctypes.c_void_p()
        if _handle is not None:
            self._h = _handle
        else:
            ctx._check(lib().fkv_streams_create(ctx.handle, n_streams, capacity, ctypes.byref(self._h)))

    @classmethod
    def import_(cls, ctx: Context, length: int, host_pts: np.ndarray):
        h = ctypes.c_void_p()
        p = np.ascontiguousarray(host_pts, np.float64)
        ctx._check(lib().fkv_streams_import(ctx.handle, p.shape[0], length, p.ctypes.data, ctypes.byref(h)))
        return cls(ctx, p.shape[0], _handle=h)

    def info(self):
        ns, ln, st = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        p = ctypes.c_void_p()
        lib().fkv_streams_info(self._h, ctypes.byref(ns), ctypes.byref(ln), ctypes.byref(st), ctypes.byref(p))
        return ns.value, ln.value, st.value, p.value

    def points(self) -> torch.Tensor:
        """A [n_streams, cap_spans, 2] float64 view of the library-owned point
        buffer (valid until the next growing append)."""
        ns, ln, st, p = self.info()
        return _device_view(p, (ns, st, 2))

    @property
    def length(self) -> int:
        return self.info()[1]

    def reset(self):
        lib().fkv_streams_reset(self._h)

    def append(self, sym: torch.Tensor, stream=None):
        """sym [n_streams, m] of the context's sym_dtype."""
        self.ctx._sym(sym)
        self.ctx._check(lib().fkv_append(self.ctx.handle, self._h, _ptr(sym), sym.shape[1], _rows(sym),
                                         _stream(stream)))

    def export(self, stream=None) -> np.ndarray:
        ns, ln, st, p = self.info()
        out = np.empty((ns, self.ctx.n_spans(ln), 2), np.float64)
        length = ctypes.c_int64()
        self.ctx._check(lib().fkv_streams_export(self._h, ctypes.byref(length), out.ctypes.data, _stream(stream)))
        return out

    def close(self):
        if self._h:
            lib().fkv_streams_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _device_view(ptr: int, shape):
    """Wrap a library-owned float64 device buffer as a torch tensor (no copy)."""
    n = int(np.prod(shape))

    class _Holder:
        __cuda_array_interface__ = {"shape": tuple(shape), "typestr": "<f8", "data": (ptr, False),
                                    "version": 3, "strides": None}
    if n == 0:
        return torch.empty(shape, dtype=torch.float64, device="cuda")
    return torch.as_tensor(_Holder(), device="cuda")
