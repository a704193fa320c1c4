// Span codec kernels: the iterated-map code of Sec. 1 "The code", applied
// span-parallel (one span per thread) for encoding, decoding, random reads
// and tail appends (Sec. 2, Table 1).
//
// Encoding must reproduce the binary64 walk bit for bit, so it runs on the
// FP64 pipe with explicit round-to-nearest intrinsics (no FMA contraction):
// d = p - V(c); t = r * d; p = V(c) + t per coordinate.
//
// Decoding only has to recover the symbols, so it runs in exact 64-bit
// fixed point (Q1.62) on the integer pipes with no division at all (see
// decode_core.cuh).
#include "decode_core.cuh"

namespace {

constexpr int kThreads = 256;   // spans per block
constexpr int kMaxSpan = 44;    // floor(44 / log2(1/r)) with r <= 1/2

// Symbols are uint8 for alphabets N <= 256 and uint16 up to FKV_MAX_N; every
// kernel that touches symbols is instantiated for both.
template <typename Sym>
__host__ __device__ constexpr int stage_bytes() { return kThreads * kMaxSpan * static_cast<int>(sizeof(Sym)) + 32; }
// Block size of the bulk decoders: 256 spans per chunk for uint8 symbols; for
// uint16 (N up to 1024, 104 KB of decoder tables per block) one 1024-thread
// block per SM shares the tables.
template <typename Sym>
__host__ __device__ constexpr int dec_threads() { return sizeof(Sym) == 1 ? 256 : 1024; }
// Shared staging of one decoded chunk: dec_threads spans of L symbols plus
// the 16-byte realignment slack.
template <typename Sym>
__host__ __device__ inline int dec_stage_bytes(int L)
{
    return (dec_threads<Sym>() * L * static_cast<int>(sizeof(Sym)) + 32 + 15) & ~15;
}
template <typename Sym>
__host__ __device__ constexpr int vtab_len() { return sizeof(Sym) == 1 ? 256 : FKV_MAX_N; }

// Copy len bytes from global src into shared buf so that buf[off + i] =
// src[i], off = src mod 16: aligned 16-byte vectors inside the range, single
// bytes at the two ragged ends.  Never touches bytes outside [src, src+len).
__device__ __forceinline__ int stage_in(uint8_t *buf, const uint8_t *src, int len)
{
    const int off = static_cast<int>(reinterpret_cast<uintptr_t>(src) & 15);
    const uint8_t *a = src - off;
    const int total = off + len;
    const int nv = (total + 15) >> 4;
    for (int v = threadIdx.x; v < nv; v += blockDim.x) {
        const int b0 = v << 4;
        if (b0 >= off && b0 + 16 <= total) {
            *reinterpret_cast<uint4 *>(buf + b0) = __ldg(reinterpret_cast<const uint4 *>(a + b0));
        } else {
            const int lo = b0 > off ? b0 : off;
            const int hi = b0 + 16 < total ? b0 + 16 : total;
            for (int q = lo; q < hi; ++q)
                buf[q] = a[q];
        }
    }
    return off;
}

// The mirror of stage_in: dst[i] = buf[off + i], off = dst mod 16.
__device__ __forceinline__ void stage_out(uint8_t *dst, const uint8_t *buf, int len, int off)
{
    uint8_t *a = dst - off;
    const int total = off + len;
    const int nv = (total + 15) >> 4;
    for (int v = threadIdx.x; v < nv; v += blockDim.x) {
        const int b0 = v << 4;
        if (b0 >= off && b0 + 16 <= total) {
            *reinterpret_cast<uint4 *>(a + b0) = *reinterpret_cast<const uint4 *>(buf + b0);
        } else {
            const int lo = b0 > off ? b0 : off;
            const int hi = b0 + 16 < total ? b0 + 16 : total;
            for (int q = lo; q < hi; ++q)
                a[q] = buf[q];
        }
    }
}

// Sec. 1 forward map for one span from the anchor (0, 0), binary64, no FMA.
// A symbol >= N takes a NaN vertex, so its span's point comes out NaN.
template <typename Sym>
__device__ __forceinline__ double2 encode_span(const Sym *s, int m, const double2 *sV, int N, double r,
                                               double x, double y)
{
    for (int k = 0; k < m; ++k) {
        const unsigned c = s[k];
        const double2 v = c < static_cast<unsigned>(N) ? sV[c] : make_double2(__longlong_as_double(-1ll),
                                                                              __longlong_as_double(-1ll));
        const double dx = __dsub_rn(x, v.x);
        const double dy = __dsub_rn(y, v.y);
        const double tx = __dmul_rn(r, dx);
        const double ty = __dmul_rn(r, dy);
        x = __dadd_rn(v.x, tx);
        y = __dadd_rn(v.y, ty);
    }
    return make_double2(x, y);
}

template <typename Sym>
__global__ void __launch_bounds__(kThreads)
k_span_encode(const Sym *__restrict__ sym, int64_t n, int64_t sym_stride, int64_t spans, int bps,
              double2 *__restrict__ pts, int64_t pt_stride, const double2 *__restrict__ V, int N, double r, int L,
              unsigned *status)
{
    __shared__ __align__(16) uint8_t sbuf[stage_bytes<Sym>()];
    __shared__ double2 sV[vtab_len<Sym>()];
    const int64_t stream = blockIdx.x / bps;
    const int64_t s0 = static_cast<int64_t>(blockIdx.x % bps) * kThreads;
    for (int i = threadIdx.x; i < N; i += kThreads)
        sV[i] = V[i];
    const int64_t b = s0 * L;
    const int64_t e = min(n, (s0 + kThreads) * L);
    const int off = stage_in(sbuf, reinterpret_cast<const uint8_t *>(sym + stream * sym_stride + b),
                             static_cast<int>(e - b) * static_cast<int>(sizeof(Sym)));
    __syncthreads();
    const int64_t s = s0 + threadIdx.x;
    if (s < spans) {
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - s * L));
        const Sym *my = reinterpret_cast<const Sym *>(sbuf + off) + threadIdx.x * L;
        const double2 p = encode_span(my, m, sV, N, r, 0.0, 0.0);
        if (isnan(p.x))   // a symbol >= N reads a NaN vertex
            atomicOr(status, FKV_ST_CORRUPT);
        pts[stream * pt_stride + s] = p;
    }
}

// ------------------------------------------------------------- decoding
// (arithmetic in decode_core.cuh: exact Q1.62 walk, no division)

__host__ __device__ inline int tables_bytes(int N, int L)
{
    return (fkvdec::smem_bytes(N, L) + 15) & ~15;
}

// A persistent block's chunk (stream, span block), chunk = stream * bps +
// block, stepped gridDim.x chunks at a time without a division per step: the
// whole streams and remaining blocks of one step are worked out once.
struct ChunkWalk {
    int64_t stream, sb;
    unsigned dq, dr, bps;
    __device__ explicit ChunkWalk(int bps_) : bps(static_cast<unsigned>(bps_))
    {
        stream = blockIdx.x / bps;
        sb = blockIdx.x - static_cast<unsigned>(stream) * bps;
        dq = gridDim.x / bps;
        dr = gridDim.x - dq * bps;
    }
    __device__ void next()
    {
        sb += dr;
        stream += dq;
        if (sb >= bps) {
            sb -= bps;
            ++stream;
        }
    }
};

// Unsigned 32-bit division by an invariant d >= 1 as a multiply-high, a
// subtract, an add and two shifts (Granlund and Montgomery, "Division by
// invariant integers using multiplication", PLDI 1994, Sec. 4): with l =
// ceil(log2 d) and m = floor(2^32 (2^l - d) / d) + 1, t = mulhi(m, q) and
// q / d = (t + ((q - t) >> min(l, 1))) >> max(l - 1, 0) for every 32-bit q.
struct FastDiv {
    unsigned m;
    int sh1, sh2;
    __host__ static FastDiv make(unsigned d)
    {
        int l = 0;
        while ((1ull << l) < d)
            ++l;
        FastDiv f;
        f.m = static_cast<unsigned>((((1ull << l) - d) << 32) / d + 1);
        f.sh1 = l < 1 ? l : 1;
        f.sh2 = l - 1 > 0 ? l - 1 : 0;
        return f;
    }
    __device__ __forceinline__ unsigned div(unsigned q) const
    {
        const unsigned t = __umulhi(m, q);
        return (t + ((q - t) >> sh1)) >> sh2;
    }
};

// Decode span s of `stream` (one per thread): the walk's symbols go through
// `put(j, c)`, j = 0 .. m-1 from the span's last symbol back to its first,
// straight from registers to their place; a point whose walk does not end at
// the anchor sets the corrupt status.
template <class Put>
__device__ __forceinline__ void decode_span(const fkvdec::Tables &t, const double2 *__restrict__ pts, int64_t n,
                                            int64_t pt_stride, int64_t stream, int64_t s,
                                            const fkv_decconst *__restrict__ dc, int L, unsigned *status, Put put,
                                            int &m)
{
    m = static_cast<int>(min(static_cast<int64_t>(L), n - s * L));
    const double2 p = pts[stream * pt_stride + s];
    long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
    fkvdec::walk(t, X, Y, m, put);
    const long long lim = __ldg(&dc->alim[m]);
    if (X > lim || X < -lim || Y > lim || Y < -lim)
        atomicOr(status, FKV_ST_CORRUPT);
}

// Persistent: a block loads the decoder tables once and walks chunks of
// dec_threads spans (chunk = stream * bps + span block), blockIdx.x,
// + gridDim.x, ...; each thread stores its span's symbols directly, so the
// chunks need no block barrier.
template <typename Sym>
__global__ void __launch_bounds__(dec_threads<Sym>())
k_span_decode(const double2 *__restrict__ pts, int64_t n, int64_t pt_stride, int64_t spans, int bps,
              int64_t n_chunks, Sym *__restrict__ sym, int64_t sym_stride, const fkv_decconst *__restrict__ dc,
              const longlong2 *__restrict__ T, int N, int L, unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    __syncthreads();
    constexpr int TPB = dec_threads<Sym>();
    ChunkWalk w(bps);
    for (int64_t ck = blockIdx.x; ck < n_chunks; ck += gridDim.x, w.next()) {
        const int64_t s = w.sb * TPB + threadIdx.x;
        if (s >= spans)
            continue;
        Sym *dst = sym + w.stream * sym_stride + s * L;
        int m = 0;
        decode_span(t, pts, n, pt_stride, w.stream, s, dc, L, status,
                    [&](int j, int c) { dst[m - 1 - j] = static_cast<Sym>(c); }, m);
    }
}

// Decode 256 spans of one stream (chunk `ck` of the n_streams * bps chunks)
// into sbuf (one span per thread, symbol i of the chunk at sbuf[i]).
template <typename Sym>
__device__ __forceinline__ void decode_chunk(const fkvdec::Tables &t, const double2 *__restrict__ pts, int64_t n,
                                             int64_t pt_stride, int64_t spans, int64_t stream, int64_t s0,
                                             Sym *sbuf, const fkv_decconst *__restrict__ dc, int L,
                                             unsigned *status)
{
    const int64_t s = s0 + threadIdx.x;
    if (s < spans) {
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - s * L));
        const double2 p = pts[stream * pt_stride + s];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        Sym *my = sbuf + threadIdx.x * L;
        fkvdec::walk(t, X, Y, m, [&](int j, int c) { my[m - 1 - j] = static_cast<Sym>(c); });
        const long long lim = __ldg(&dc->alim[m]);
        if (X > lim || X < -lim || Y > lim || Y < -lim)
            atomicOr(status, FKV_ST_CORRUPT);
    }
}

// The stream decode for long spans (more than 8 symbols): a chunk's symbols
// are staged in shared memory and written out with aligned 16-byte stores,
// since a thread's own span would otherwise be a run of scattered byte
// stores.  Persistent: chunk = stream * bps + span block, blockIdx.x,
// + gridDim.x, ...
template <typename Sym>
__global__ void __launch_bounds__(dec_threads<Sym>())
k_span_decode_staged(const double2 *__restrict__ pts, int64_t n, int64_t pt_stride, int64_t spans, int bps,
              int64_t n_chunks, Sym *__restrict__ sym, int64_t sym_stride, const fkv_decconst *__restrict__ dc,
              const longlong2 *__restrict__ T, int N, int L, unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    uint8_t *sbuf = dsm + tables_bytes(N, L);
    __syncthreads();
    constexpr int TPB = dec_threads<Sym>();
    ChunkWalk w(bps);
    for (int64_t ck = blockIdx.x; ck < n_chunks; ck += gridDim.x, w.next()) {
        const int64_t stream = w.stream;
        const int64_t s0 = w.sb * TPB;
        const int64_t b = s0 * L;
        const int64_t e = min(n, (s0 + TPB) * L);
        uint8_t *dst = reinterpret_cast<uint8_t *>(sym + stream * sym_stride + b);
        const int off = static_cast<int>(reinterpret_cast<uintptr_t>(dst) & 15);
        decode_chunk(t, pts, n, pt_stride, spans, stream, s0, reinterpret_cast<Sym *>(sbuf + off), dc, L, status);
        __syncthreads();
        stage_out(dst, sbuf, static_cast<int>(e - b) * static_cast<int>(sizeof(Sym)), off);
        __syncthreads();
    }
}

// The same decode for a whole archive of token records, written out in the
// planar layout the archive gather reads: per stream, the H key planes
// (n_rec x S_K indices each, one plane per head) and then the H value planes
// (n_rec x S_V).  A block first tabulates, for each of the R symbols of a
// record, its offset inside its record's first plane row; a thread then places
// each symbol of its span as the walk yields it, last to first, at that
// offset plus record x stages, stepping back one symbol of the record (and a
// record at its start) per symbol.  Positions inside a stream are 32-bit (the
// launcher keeps a stream below 2^31 symbols) and the span's last record comes
// from a multiply-high division.
template <typename Sym>
__global__ void __launch_bounds__(dec_threads<Sym>())
k_span_decode_planar(const double2 *__restrict__ pts, unsigned n_rec, int64_t pt_stride, unsigned spans, int bps,
                     unsigned n_chunks, Sym *__restrict__ out, int H, int SK, int SV, FastDiv div_r,
                     const fkv_decconst *__restrict__ dc, const longlong2 *__restrict__ T, int N, int L,
                     unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    const int R = H * (SK + SV);
    const int nk = H * SK;
    const unsigned n = n_rec * static_cast<unsigned>(R);
    constexpr int TPB = dec_threads<Sym>();
    // symbol o of a record: plane offset (K planes, then V planes) + stage
    unsigned *poff = reinterpret_cast<unsigned *>(dsm + tables_bytes(N, L));
    for (int o = threadIdx.x; o < R; o += TPB) {
        const bool v = o >= nk;
        const int S = v ? SV : SK, oo = v ? o - nk : o;
        const int h = oo / S;
        poff[o] = (v ? static_cast<unsigned>(nk) * n_rec : 0u) + static_cast<unsigned>(h) * n_rec * S + (oo - h * S);
    }
    __syncthreads();
    const long long lim_full = __ldg(&dc->alim[L]);
    ChunkWalk w(bps);
    for (unsigned ck = blockIdx.x; ck < n_chunks; ck += gridDim.x, w.next()) {
        const unsigned s = static_cast<unsigned>(w.sb) * TPB + threadIdx.x;
        if (s >= spans)
            continue;
        const unsigned first = s * static_cast<unsigned>(L);
        const int m = n - first < static_cast<unsigned>(L) ? static_cast<int>(n - first) : L;
        const unsigned q = first + m - 1;             // the span's last symbol
        unsigned rec = div_r.div(q);
        int o = static_cast<int>(q - rec * static_cast<unsigned>(R));
        Sym *base = out + w.stream * static_cast<int64_t>(n);
        const double2 p = pts[w.stream * pt_stride + s];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        fkvdec::walk(t, X, Y, m, [&](int, int c) {
            const unsigned S = o < nk ? SK : SV;
            base[poff[o] + rec * S] = static_cast<Sym>(c);
            if (o == 0) {
                o = R;
                --rec;
            }
            --o;
        });
        const long long lim = m == L ? lim_full : __ldg(&dc->alim[m]);
        if (X > lim || X < -lim || Y > lim || Y < -lim)
            atomicOr(status, FKV_ST_CORRUPT);
    }
}

// Sec. 5 retrieval in place.  Persistent blocks scan their share of the
// stored points against the query's point (the query encoded from the
// origin by the Sec. 1 map, bit for bit as the encoder would): a point of a
// span of at least l symbols inside the 2 r^l ball is a candidate, and a
// candidate is walked back l steps by the exact decoder; it matches when
// those symbols are the query.  Matches are appended (stream, span) in any
// order; counts[0] counts matches (all of them, even past cap), counts[1]
// candidates.  GB300's FP64 pipe would bound a binary64 distance test of every
// point, so each point first passes an integer box test: the ball's bounding
// box, rounded outward, in an order-preserving integer image of binary64; only
// points inside the box take the binary64 test.  Four points per thread are
// in flight at once.
struct SuffixQuery {
    uint16_t sym[kMaxSpan];
    int len;
};

__global__ void __launch_bounds__(kThreads)
k_suffix_search(const double2 *__restrict__ pts, int64_t n_streams, int64_t n, int64_t pt_stride, int64_t spans,
                const SuffixQuery qy, double thr, double thr2, const double2 *__restrict__ V, double r,
                const fkv_decconst *__restrict__ dc, const longlong2 *__restrict__ T, int N, int L,
                long long *__restrict__ out, long long cap, unsigned long long *__restrict__ counts)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ double2 q_s;
    __shared__ long long box_s[4];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    // order-preserving integer image of a binary64 value (signed compare)
    auto okey = [](long long b) { return b ^ ((b >> 63) & 0x7FFFFFFFFFFFFFFFll); };
    if (threadIdx.x == 0) {
        const double2 qq = encode_span(qy.sym, qy.len, V, N, r, 0.0, 0.0);
        q_s = qq;
        const double tb = __dmul_ru(thr, 1.0 + 0x1p-40);           // the box contains the ball
        box_s[0] = okey(__double_as_longlong(__dsub_rd(qq.x, tb)));
        box_s[1] = okey(__double_as_longlong(__dadd_ru(qq.x, tb)));
        box_s[2] = okey(__double_as_longlong(__dsub_rd(qq.y, tb)));
        box_s[3] = okey(__double_as_longlong(__dadd_ru(qq.y, tb)));
    }
    __syncthreads();
    const double2 q = q_s;
    const long long bx0 = box_s[0], bx1 = box_s[1], by0 = box_s[2], by1 = box_s[3];
    const longlong2 *pk = reinterpret_cast<const longlong2 *>(pts);
    const int l = qy.len;
    // this block's contiguous share of the n_streams * spans points, walked
    // kThreads apart per thread without division
    const int64_t total = n_streams * spans;
    const int64_t hi = total * (blockIdx.x + 1) / gridDim.x;
    int64_t g = total * blockIdx.x / gridDim.x + threadIdx.x;
    int64_t stream = g / spans, u = g - stream * spans;
    const int64_t step_s = kThreads / spans, step_u = kThreads - step_s * spans;
    constexpr int kU = 4;
    while (g < hi) {
        longlong2 pb[kU];
        int64_t su[kU], uu[kU];
        bool live[kU];
#pragma unroll
        for (int i = 0; i < kU; ++i) {
            live[i] = g < hi;
            su[i] = stream;
            uu[i] = u;
            if (live[i])
                pb[i] = pk[stream * pt_stride + u];
            g += kThreads;
            u += step_u;
            stream += step_s;
            if (u >= spans) {
                u -= spans;
                ++stream;
            }
        }
#pragma unroll
        for (int i = 0; i < kU; ++i) {
            if (!live[i])
                break;
            const int m = static_cast<int>(min(static_cast<int64_t>(L), n - uu[i] * L));
            const long long kx = okey(pb[i].x), ky = okey(pb[i].y);
            if (m >= l && kx >= bx0 && kx <= bx1 && ky >= by0 && ky <= by1) {
                const double2 p = make_double2(__longlong_as_double(pb[i].x), __longlong_as_double(pb[i].y));
                const double dx = __dsub_rn(p.x, q.x), dy = __dsub_rn(p.y, q.y);
                const double d2 = __dadd_rn(__dmul_rn(dx, dx), __dmul_rn(dy, dy));
                if (d2 <= thr2) {
                    atomicAdd(&counts[1], 1ull);
                    long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
                    bool eq = true;
                    // step j recovers the span's symbol m - 1 - j, the query's l - 1 - j
                    fkvdec::walk(t, X, Y, l, [&](int j, int c) { eq = eq && c == qy.sym[l - 1 - j]; });
                    if (eq) {
                        const unsigned long long slot = atomicAdd(&counts[0], 1ull);
                        if (static_cast<long long>(slot) < cap) {
                            out[2 * slot] = su[i];
                            out[2 * slot + 1] = uu[i];
                        }
                    }
                }
            }
        }
    }
}

// Sec. 2 random access: one request per thread, decoding only its span down
// to the requested offset.  Persistent: a block loads the decoder tables once
// and takes requests blockIdx.x * TPB + threadIdx.x, + gridDim.x * TPB, ...
template <typename Sym>
__global__ void __launch_bounds__(dec_threads<Sym>())
k_read(const double2 *__restrict__ pts, int64_t n_streams, int64_t n, int64_t pt_stride,
       const int64_t *__restrict__ req, int64_t n_req, Sym *__restrict__ out,
       const fkv_decconst *__restrict__ dc, const longlong2 *__restrict__ T, int N, int L, unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    __syncthreads();
    constexpr int TPB = dec_threads<Sym>();
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * TPB + threadIdx.x; q < n_req;
         q += static_cast<int64_t>(gridDim.x) * TPB) {
        const int64_t st = req[2 * q], pos = req[2 * q + 1];
        if (st < 0 || st >= n_streams || pos < 0 || pos >= n) {
            out[q] = static_cast<Sym>(~0u);
            atomicOr(status, FKV_ST_RANGE);
            continue;
        }
        const int64_t u = pos / L;
        const int o = static_cast<int>(pos - u * L);
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
        const double2 p = pts[st * pt_stride + u];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        int sym = 0;
        fkvdec::walk(t, X, Y, m - o, [&](int j, int c) { sym = c; });
        out[q] = static_cast<Sym>(sym);
    }
}

// Sec. 2 append: one thread per (stream, span touched by the new symbols).
// The first touched span continues from the stored tail point when the old
// length is not a multiple of L; every later span starts at the anchor.
template <typename Sym>
__global__ void __launch_bounds__(kThreads)
k_append(double2 *__restrict__ pts, int64_t n_streams, int64_t pt_stride, int64_t n_old,
         const Sym *__restrict__ sym, int64_t m, int64_t sym_stride, int64_t u_first, int64_t cnt,
         const double2 *__restrict__ V, int N, double r, int L, unsigned *status)
{
    __shared__ double2 sV[vtab_len<Sym>()];
    for (int i = threadIdx.x; i < N; i += kThreads)
        sV[i] = V[i];
    __syncthreads();
    const int64_t t = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x;
    if (t >= n_streams * cnt)
        return;
    const int64_t stream = t / cnt;
    const int64_t u = u_first + (t - stream * cnt);
    const int64_t n_new = n_old + m;
    const int64_t b = max(u * L, n_old);
    const int64_t e = min((u + 1) * L, n_new);
    double2 p = make_double2(0.0, 0.0);
    if (u * L < n_old)
        p = pts[stream * pt_stride + u];
    Sym s[kMaxSpan];
    const Sym *src = sym + stream * sym_stride + (b - n_old);
    const int len = static_cast<int>(e - b);
    for (int k = 0; k < len; ++k)
        s[k] = src[k];
    p = encode_span(s, len, sV, N, r, p.x, p.y);
    if (isnan(p.x))
        atomicOr(status, FKV_ST_CORRUPT);
    pts[stream * pt_stride + u] = p;
}

// ------------------------------------------------------------ ragged batches
// Streams of different lengths in one call (the sequences of a serving batch
// rarely share a length): stream i holds len_i = so[i + 1] - so[i] symbols at
// sym + so[i] and owns point slots [po[i], po[i + 1]) of pts, at least
// ceil(len_i / L) of them.  so and po are device arrays of n_streams + 1
// offsets.  The kernels walk the point slots [po[0], po[n_streams])
// grid-stride, one span per thread, and find a slot's stream by binary search
// over po.  A stream whose offsets are inconsistent (a negative length, fewer
// point slots than spans) is left alone and reported by the range status bit;
// the check runs once per stream, so a stream with no slots is reported too.

// The stream owning point slot g: the largest i < n_streams with po[i] <= g
// (po nondecreasing; every index read stays in [0, n_streams]).
__device__ __forceinline__ int64_t ragged_stream(const int64_t *__restrict__ po, int64_t n_streams, int64_t g)
{
    int64_t lo = 0, hi = n_streams;
    while (hi - lo > 1) {
        const int64_t mid = (lo + hi) >> 1;
        if (__ldg(&po[mid]) <= g)
            lo = mid;
        else
            hi = mid;
    }
    return lo;
}

// Length of stream i and whether its offsets hold together.
__device__ __forceinline__ bool ragged_ok(const int64_t *__restrict__ so, const int64_t *__restrict__ po, int64_t i,
                                          int L, int64_t *len)
{
    const int64_t n = __ldg(&so[i + 1]) - __ldg(&so[i]);
    const int64_t slots = __ldg(&po[i + 1]) - __ldg(&po[i]);
    *len = n;
    return n >= 0 && slots >= 0 && slots >= (n + L - 1) / L;
}

// Every thread of the grid takes part in checking the streams' offsets.
__device__ __forceinline__ void ragged_check(const int64_t *__restrict__ so, const int64_t *__restrict__ po,
                                             int64_t n_streams, int L, unsigned *status)
{
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n_streams; i += stride) {
        int64_t n;
        if (!ragged_ok(so, po, i, L, &n))
            atomicOr(status, FKV_ST_RANGE);
    }
}

template <typename Sym>
__global__ void __launch_bounds__(kThreads)
k_span_encode_ragged(const Sym *__restrict__ sym, const int64_t *__restrict__ so, int64_t n_streams,
                     double2 *__restrict__ pts, const int64_t *__restrict__ po, const double2 *__restrict__ V,
                     int N, double r, int L, unsigned *status)
{
    __shared__ double2 sV[vtab_len<Sym>()];
    for (int i = threadIdx.x; i < N; i += kThreads)
        sV[i] = V[i];
    __syncthreads();
    ragged_check(so, po, n_streams, L, status);
    const int64_t g0 = __ldg(&po[0]), g1 = __ldg(&po[n_streams]);
    const int64_t stride = static_cast<int64_t>(gridDim.x) * kThreads;
    for (int64_t g = g0 + static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; g < g1; g += stride) {
        const int64_t i = ragged_stream(po, n_streams, g);
        int64_t n;
        if (!ragged_ok(so, po, i, L, &n))
            continue;
        const int64_t s = g - __ldg(&po[i]);
        if (s < 0 || s * L >= n)
            continue;                       // a slot past the stream's last span
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - s * L));
        const double2 p = encode_span(sym + __ldg(&so[i]) + s * L, m, sV, N, r, 0.0, 0.0);
        if (isnan(p.x))
            atomicOr(status, FKV_ST_CORRUPT);
        pts[g] = p;
    }
}

template <typename Sym>
__global__ void __launch_bounds__(dec_threads<Sym>())
k_span_decode_ragged(const double2 *__restrict__ pts, const int64_t *__restrict__ po, int64_t n_streams,
                     Sym *__restrict__ sym, const int64_t *__restrict__ so, const fkv_decconst *__restrict__ dc,
                     const longlong2 *__restrict__ T, int N, int L, unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    __syncthreads();
    ragged_check(so, po, n_streams, L, status);
    const int64_t g0 = __ldg(&po[0]), g1 = __ldg(&po[n_streams]);
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t g = g0 + static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; g < g1; g += stride) {
        const int64_t i = ragged_stream(po, n_streams, g);
        int64_t n;
        if (!ragged_ok(so, po, i, L, &n))
            continue;
        const int64_t s = g - __ldg(&po[i]);
        if (s < 0 || s * L >= n)
            continue;
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - s * L));
        const double2 p = pts[g];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        Sym *dst = sym + __ldg(&so[i]) + s * L;
        fkvdec::walk(t, X, Y, m, [&](int j, int c) { dst[m - 1 - j] = static_cast<Sym>(c); });
        const long long lim = __ldg(&dc->alim[m]);
        if (X > lim || X < -lim || Y > lim || Y < -lim)
            atomicOr(status, FKV_ST_CORRUPT);
    }
}

// Random access into a ragged batch: request q = (stream, position), the
// position checked against that stream's own length.
template <typename Sym>
__global__ void __launch_bounds__(dec_threads<Sym>())
k_read_ragged(const double2 *__restrict__ pts, const int64_t *__restrict__ po, const int64_t *__restrict__ so,
              int64_t n_streams, const int64_t *__restrict__ req, int64_t n_req, Sym *__restrict__ out,
              const fkv_decconst *__restrict__ dc, const longlong2 *__restrict__ T, int N, int L, unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(dc, T, N, L, dsm);
    __syncthreads();
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < n_req; q += stride) {
        const int64_t st = req[2 * q], pos = req[2 * q + 1];
        int64_t n = 0;
        if (st < 0 || st >= n_streams || !ragged_ok(so, po, st, L, &n) || pos < 0 || pos >= n) {
            out[q] = static_cast<Sym>(~0u);
            atomicOr(status, FKV_ST_RANGE);
            continue;
        }
        const int64_t u = pos / L;
        const int o = static_cast<int>(pos - u * L);
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
        const double2 p = pts[__ldg(&po[st]) + u];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        int c = 0;
        fkvdec::walk(t, X, Y, m - o, [&](int, int cc) { c = cc; });
        out[q] = static_cast<Sym>(c);
    }
}

inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// ------------------------------------------------------------- lossy archive
// Sec. 4: a span's stored point truncated to B bits per coordinate, the
// B-bit two's complement code k = floor(x 2^(B-1)); the spans of a stream
// older than its last keep_exact are kept as codes, packed into uint32 words
// (span u's x code at stream bit 2uB, its y code at 2uB + B, least
// significant bit first), the recent ones as exact points in a tail array.
struct LossyArgs {
    const uint32_t *codes;   // [n_streams][code_stride] words
    int64_t code_stride;
    int64_t words;           // words holding codes, per stream
    const double2 *tail;     // [n_streams][tail_stride] exact points of spans T ..
    int64_t tail_stride;
    int64_t T;               // truncated spans per stream
    int bits;
    double scale;            // 2^-(B-1)
};

// B-bit code of one coordinate: floor(x 2^(B-1)) (exact scaling, floor conversion).
__device__ __forceinline__ unsigned long long trunc_field(double x, double up, int bits)
{
    const long long k = __double2ll_rd(__dmul_rn(x, up));
    return static_cast<unsigned long long>(k) & ((1ull << bits) - 1);
}

// Warp per group of 32 spans of one stream: the group's 64 codes fill exactly
// 2B words (the group starts at stream bit 64 B g, a word boundary); each lane
// computes its span's two codes, then assembles words lane, lane + 32, ... of
// the group from the codes that overlap them, fetched by warp shuffles.
__global__ void __launch_bounds__(kThreads)
k_truncate(const double *__restrict__ pts, int64_t pt_stride, int64_t n_streams, int64_t T, int bits,
           uint32_t *__restrict__ codes, int64_t code_stride, int64_t words)
{
    const double up = static_cast<double>(1ull << (bits - 1));
    const int lane = threadIdx.x & 31;
    const int64_t gps = (T + 31) >> 5;                       // groups per stream
    const int64_t n_groups = n_streams * gps;
    const int64_t nw = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
    const int kmax = 32 / bits + 2;                          // codes overlapping one word, at most
    const int wpg = 2 * bits;                                // words per group
    for (int64_t g = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5; g < n_groups; g += nw) {
        const int64_t stream = g / gps, grp = g - stream * gps;
        const int64_t u = grp * 32 + lane;
        unsigned long long fx = 0, fy = 0;
        if (u < T) {
            const double2 p = reinterpret_cast<const double2 *>(pts)[stream * pt_stride + u];
            fx = trunc_field(p.x, up, bits);
            fy = trunc_field(p.y, up, bits);
        }
        const int64_t w0 = grp * wpg;
        const int64_t nwg = min(static_cast<int64_t>(wpg), words - w0);
        for (int j0 = 0; j0 < wpg; j0 += 32) {
            const int j = j0 + lane;
            const int bit0 = 32 * j;                         // relative to the group
            const int c0 = bit0 / bits;
            uint32_t out = 0;
            for (int k = 0; k < kmax; ++k) {
                const int ci = c0 + k;                       // code of the group: span ci / 2, x or y
                const int src = min(ci >> 1, 31);
                const unsigned long long vx = __shfl_sync(0xFFFFFFFFu, fx, src);
                const unsigned long long vy = __shfl_sync(0xFFFFFFFFu, fy, src);
                const unsigned long long f = (ci & 1) ? vy : vx;
                const int sh = ci * bits - bit0;
                if (ci < 64 && sh < 32)
                    out |= static_cast<uint32_t>(sh >= 0 ? f << sh : f >> (-sh));
            }
            if (j < nwg)
                codes[stream * code_stride + w0 + j] = out;
        }
    }
}

// The B-bit field at stream bit `pos`, sign-extended.
__device__ __forceinline__ long long read_field(const uint32_t *w, int64_t words, int64_t pos, int bits)
{
    const int64_t q = pos >> 5;
    const int off = static_cast<int>(pos & 31);
    unsigned long long v = __ldg(w + q);
    if (q + 1 < words)
        v |= static_cast<unsigned long long>(__ldg(w + q + 1)) << 32;
    v >>= off;
    if (off + bits > 64 && q + 2 < words)
        v |= static_cast<unsigned long long>(__ldg(w + q + 2)) << (64 - off);
    const int sh = 64 - bits;
    return static_cast<long long>(v << sh) >> sh;
}

// The point a lossy archive keeps for span u of a stream.
__device__ __forceinline__ double2 lossy_point(const LossyArgs &a, int64_t stream, int64_t u)
{
    if (u >= a.T)
        return a.tail[stream * a.tail_stride + (u - a.T)];
    const uint32_t *w = a.codes + stream * a.code_stride;
    const int64_t pos = 2 * u * a.bits;
    const long long kx = read_field(w, a.words, pos, a.bits);
    const long long ky = read_field(w, a.words, pos + a.bits, a.bits);
    return make_double2(__dmul_rn(static_cast<double>(kx), a.scale), __dmul_rn(static_cast<double>(ky), a.scale));
}

// Squared distance to a vertex as the paper's binary64 arithmetic forms it
// (two products and a sum, no FMA).
__device__ __forceinline__ double dist2(double2 v, double x, double y)
{
    const double dx = __dsub_rn(x, v.x), dy = __dsub_rn(y, v.y);
    return __dadd_rn(__dmul_rn(dx, dx), __dmul_rn(dy, dy));
}

// Sec. 1 cell test in binary64 for a point that need not be a code point:
// the vertex of least binary64 squared distance, lowest index on a tie.  The
// nearest vertex is the angularly nearest, so for |p|^2 in [2^-40, 2^60] only
// the three vertices around the fp32 angle are scored: every other vertex is
// farther by at least 2|p|(cos(pi/N) - cos(3 pi/N)) (7.5e-5 |p| at N = 1024),
// far above the rounding of the distances, so the choice equals a full scan's.
// Other points (tiny, huge, not finite) take the full scan.
__device__ __forceinline__ int nearest64(const double2 *sV, int N, double x, double y)
{
    const double rr = x * x + y * y;
    if (rr >= 0x1p-40 && rr <= 0x1p60) {
        const float a = atan2f(static_cast<float>(y), static_cast<float>(x)) *
                        (static_cast<float>(N) * 0.15915494309189535f);
        int c0 = static_cast<int>(rintf(a));
        c0 = c0 < 0 ? c0 + N : (c0 >= N ? c0 - N : c0);
        int best = -1;
        double bd = 0.0;
#pragma unroll
        for (int k = -1; k <= 1; ++k) {
            int c = c0 + k;
            c = c < 0 ? c + N : (c >= N ? c - N : c);
            const double d = dist2(sV[c], x, y);
            if (best < 0 || d < bd || (d == bd && c < best)) {
                bd = d;
                best = c;
            }
        }
        return best;
    }
    int best = 0;
    double bd = INFINITY;
    for (int c = 0; c < N; ++c) {
        const double d = dist2(sV[c], x, y);
        if (d < bd) {
            bd = d;
            best = c;
        }
    }
    return best;
}

// Backward walk from (x, y) in the paper's arithmetic: the cell, then
// p <- (p - w V(c)) / r with w = 1 - r (binary64 product, difference and
// IEEE division).  emit(j, c) receives the symbol of step j.
template <class Emit>
__device__ __forceinline__ void walk64(const double2 *sV, int N, double w, double r, double x, double y, int steps,
                                       Emit emit)
{
    for (int j = 0; j < steps; ++j) {
        const int c = nearest64(sV, N, x, y);
        emit(j, c);
        const double2 v = sV[c];
        x = __ddiv_rn(__dsub_rn(x, __dmul_rn(w, v.x)), r);
        y = __ddiv_rn(__dsub_rn(y, __dmul_rn(w, v.y)), r);
    }
}

// Bulk decode of a lossy archive: persistent blocks walk chunks of 256 spans
// (one per thread) and write the symbols through shared memory.
template <typename Sym>
__global__ void __launch_bounds__(kThreads)
k_lossy_decode(const LossyArgs a, int64_t n, int64_t spans, int bps, int64_t n_chunks, Sym *__restrict__ sym,
               int64_t sym_stride, const double2 *__restrict__ V, int N, double w, double r, int L)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    double2 *sV = reinterpret_cast<double2 *>(dsm);
    uint8_t *sbuf = dsm + N * 16;
    for (int i = threadIdx.x; i < N; i += kThreads)
        sV[i] = V[i];
    __syncthreads();
    ChunkWalk cw(bps);
    for (int64_t ck = blockIdx.x; ck < n_chunks; ck += gridDim.x, cw.next()) {
        const int64_t stream = cw.stream;
        const int64_t s0 = cw.sb * kThreads;
        const int64_t b = s0 * L;
        const int64_t e = min(n, (s0 + kThreads) * L);
        uint8_t *dst = reinterpret_cast<uint8_t *>(sym + stream * sym_stride + b);
        const int off = static_cast<int>(reinterpret_cast<uintptr_t>(dst) & 15);
        const int64_t s = s0 + threadIdx.x;
        if (s < spans) {
            const int m = static_cast<int>(min(static_cast<int64_t>(L), n - s * L));
            const double2 p = lossy_point(a, stream, s);
            Sym *my = reinterpret_cast<Sym *>(sbuf + off) + threadIdx.x * L;
            walk64(sV, N, w, r, p.x, p.y, m, [&](int j, int c) { my[m - 1 - j] = static_cast<Sym>(c); });
        }
        __syncthreads();
        stage_out(dst, sbuf, static_cast<int>(e - b) * static_cast<int>(sizeof(Sym)), off);
        __syncthreads();
    }
}

// Random reads from a lossy archive: one request per thread.
template <typename Sym>
__global__ void __launch_bounds__(kThreads)
k_lossy_read(const LossyArgs a, int64_t n_streams, int64_t n, const int64_t *__restrict__ req, int64_t n_req,
             Sym *__restrict__ out, const double2 *__restrict__ V, int N, double w, double r, int L,
             unsigned *status)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    double2 *sV = reinterpret_cast<double2 *>(dsm);
    for (int i = threadIdx.x; i < N; i += kThreads)
        sV[i] = V[i];
    __syncthreads();
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; q < n_req;
         q += static_cast<int64_t>(gridDim.x) * kThreads) {
        const int64_t st = req[2 * q], pos = req[2 * q + 1];
        if (st < 0 || st >= n_streams || pos < 0 || pos >= n) {
            out[q] = static_cast<Sym>(~0u);
            atomicOr(status, FKV_ST_RANGE);
            continue;
        }
        const int64_t u = pos / L;
        const int o = static_cast<int>(pos - u * L);
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
        const double2 p = lossy_point(a, st, u);
        int c = 0;
        walk64(sV, N, w, r, p.x, p.y, m - o, [&](int j, int cc) { c = cc; });
        out[q] = static_cast<Sym>(c);
    }
}

}  // namespace

// Symbol width of a context: 1 byte for N <= 256, else 2.
inline bool wide(const fkv_ctx *c) { return c->N > 256; }

int codec_smem_bytes(int N, int L)
{
    return tables_bytes(N, L) + (N > 256 ? dec_stage_bytes<uint16_t>(L) : dec_stage_bytes<uint8_t>(L));
}

template <typename Sym>
cudaError_t span_encode_t(const fkv_ctx *c, const Sym *sym, int64_t n_streams, int64_t n, int64_t sym_stride,
                          double *pts, int64_t pt_stride, cudaStream_t st)
{
    const int64_t spans = cdiv(n, c->L);
    const int64_t bps = cdiv(spans, kThreads);
    const int64_t blocks = n_streams * bps;
    if (blocks == 0)
        return cudaSuccess;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    k_span_encode<Sym><<<static_cast<unsigned>(blocks), kThreads, 0, st>>>(
        sym, n, sym_stride, spans, static_cast<int>(bps), reinterpret_cast<double2 *>(pts), pt_stride,
        c->d_V, c->N, c->r, c->L, c->d_status);
    return cudaGetLastError();
}

cudaError_t launch_span_encode(const fkv_ctx *c, const void *sym, int64_t n_streams, int64_t n,
                               int64_t sym_stride, double *pts, int64_t pt_stride, cudaStream_t st)
{
    if (wide(c))
        return span_encode_t(c, static_cast<const uint16_t *>(sym), n_streams, n, sym_stride, pts, pt_stride, st);
    return span_encode_t(c, static_cast<const uint8_t *>(sym), n_streams, n, sym_stride, pts, pt_stride, st);
}

// Persistent decode grid: as many blocks of `threads` as fit on the GPU at
// once, at most one per chunk.
cudaError_t decode_grid(const fkv_ctx *c, const void *kern, int smem, int64_t n_chunks, unsigned *grid,
                        int threads = kThreads)
{
    int sms = 0, per_sm = 0;
    cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess)
        return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
    if (e != cudaSuccess)
        return e;
    int64_t g = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1);
    if (g > n_chunks)
        g = n_chunks;
    *grid = static_cast<unsigned>(g);
    return cudaSuccess;
}

template <typename Sym>
cudaError_t span_decode_t(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n, int64_t pt_stride,
                          Sym *sym, int64_t sym_stride, cudaStream_t st)
{
    constexpr int TPB = dec_threads<Sym>();
    const int64_t spans = cdiv(n, c->L);
    const int64_t bps = cdiv(spans, TPB);
    const int64_t n_chunks = n_streams * bps;
    if (n_chunks == 0)
        return cudaSuccess;
    if (bps > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    // spans of up to 8 symbols: each thread stores its own; longer ones: staged
    const bool direct = c->L <= 8;
    const void *kern = direct ? reinterpret_cast<const void *>(k_span_decode<Sym>)
                              : reinterpret_cast<const void *>(k_span_decode_staged<Sym>);
    const int smem = tables_bytes(c->N, c->L) + (direct ? 0 : dec_stage_bytes<Sym>(c->L));
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    unsigned grid = 0;
    e = decode_grid(c, kern, smem, n_chunks, &grid, TPB);
    if (e != cudaSuccess)
        return e;
    const double2 *p2 = reinterpret_cast<const double2 *>(pts);
    if (direct)
        k_span_decode<Sym><<<grid, TPB, smem, st>>>(p2, n, pt_stride, spans, static_cast<int>(bps), n_chunks, sym,
                                                         sym_stride, c->d_dec, c->d_T, c->N, c->L, c->d_status);
    else
        k_span_decode_staged<Sym><<<grid, TPB, smem, st>>>(p2, n, pt_stride, spans, static_cast<int>(bps), n_chunks,
                                                                sym, sym_stride, c->d_dec, c->d_T, c->N, c->L,
                                                                c->d_status);
    return cudaGetLastError();
}

cudaError_t launch_span_decode(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n,
                               int64_t pt_stride, void *sym, int64_t sym_stride, cudaStream_t st)
{
    if (wide(c))
        return span_decode_t(c, pts, n_streams, n, pt_stride, static_cast<uint16_t *>(sym), sym_stride, st);
    return span_decode_t(c, pts, n_streams, n, pt_stride, static_cast<uint8_t *>(sym), sym_stride, st);
}

template <typename Sym>
cudaError_t span_decode_planar_t(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n_rec,
                                 int64_t pt_stride, Sym *out, cudaStream_t st)
{
    const int SK = c->cb[0].stages, SV = c->cb[1].stages;
    const int R = c->H * (SK + SV);
    const int64_t n = n_rec * R;
    constexpr int TPB = dec_threads<Sym>();
    const int64_t spans = cdiv(n, c->L);
    const int64_t bps = cdiv(spans, TPB);
    const int64_t n_chunks = n_streams * bps;
    if (n_chunks == 0)
        return cudaSuccess;
    // 32-bit positions inside a stream, and chunk numbers
    if (n > 0x7FFFFFFF || n_chunks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    const int smem = tables_bytes(c->N, c->L) + R * static_cast<int>(sizeof(unsigned));
    cudaError_t e = cudaFuncSetAttribute(k_span_decode_planar<Sym>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         smem);
    if (e != cudaSuccess)
        return e;
    unsigned grid = 0;
    e = decode_grid(c, reinterpret_cast<const void *>(k_span_decode_planar<Sym>), smem, n_chunks, &grid, TPB);
    if (e != cudaSuccess)
        return e;
    k_span_decode_planar<Sym><<<grid, TPB, smem, st>>>(
        reinterpret_cast<const double2 *>(pts), static_cast<unsigned>(n_rec), pt_stride,
        static_cast<unsigned>(spans), static_cast<int>(bps), static_cast<unsigned>(n_chunks), out, c->H, SK, SV,
        FastDiv::make(static_cast<unsigned>(R)), c->d_dec, c->d_T, c->N, c->L, c->d_status);
    return cudaGetLastError();
}

cudaError_t launch_span_decode_planar(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n_rec,
                                      int64_t pt_stride, void *out, cudaStream_t st)
{
    if (wide(c))
        return span_decode_planar_t(c, pts, n_streams, n_rec, pt_stride, static_cast<uint16_t *>(out), st);
    return span_decode_planar_t(c, pts, n_streams, n_rec, pt_stride, static_cast<uint8_t *>(out), st);
}

cudaError_t launch_suffix_search(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n,
                                 int64_t pt_stride, const uint16_t *query, int qlen, int64_t *out, int64_t cap,
                                 int64_t *counts, cudaStream_t st)
{
    cudaError_t e = cudaMemsetAsync(counts, 0, 2 * sizeof(int64_t), st);
    if (e != cudaSuccess)
        return e;
    const int64_t spans = cdiv(n, c->L);
    if (n_streams * spans == 0)
        return cudaSuccess;
    SuffixQuery qy;
    for (int i = 0; i < kMaxSpan; ++i)
        qy.sym[i] = i < qlen ? query[i] : 0;
    qy.len = qlen;
    // (2 r^l)^2 with r^l by l successive multiplications (the Sec. 5 ball)
    double rl = 1.0;
    for (int i = 0; i < qlen; ++i)
        rl = rl * c->r;
    const double t = 2.0 * rl;
    const double thr2 = t * t;
    const int smem = tables_bytes(c->N, c->L);
    e = cudaFuncSetAttribute(k_suffix_search, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    unsigned grid = 0;
    e = decode_grid(c, reinterpret_cast<const void *>(k_suffix_search), smem, cdiv(n_streams * spans, kThreads),
                    &grid);
    if (e != cudaSuccess)
        return e;
    k_suffix_search<<<grid, kThreads, smem, st>>>(reinterpret_cast<const double2 *>(pts), n_streams, n, pt_stride,
                                                  spans, qy, t, thr2, c->d_V, c->r, c->d_dec, c->d_T, c->N, c->L,
                                                  reinterpret_cast<long long *>(out), cap,
                                                  reinterpret_cast<unsigned long long *>(counts));
    return cudaGetLastError();
}

template <typename Sym>
cudaError_t read_t(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n, int64_t pt_stride,
                   const int64_t *req, int64_t n_req, Sym *out, cudaStream_t st)
{
    constexpr int TPB = dec_threads<Sym>();
    const int64_t blocks = cdiv(n_req, TPB);
    if (blocks == 0)
        return cudaSuccess;
    const int smem = tables_bytes(c->N, c->L);
    cudaError_t e = cudaFuncSetAttribute(k_read<Sym>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    unsigned grid = 0;
    e = decode_grid(c, reinterpret_cast<const void *>(k_read<Sym>), smem, blocks, &grid, TPB);
    if (e != cudaSuccess)
        return e;
    k_read<Sym><<<grid, TPB, smem, st>>>(
        reinterpret_cast<const double2 *>(pts), n_streams, n, pt_stride, req, n_req, out, c->d_dec, c->d_T,
        c->N, c->L, c->d_status);
    return cudaGetLastError();
}

cudaError_t launch_read(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n,
                        int64_t pt_stride, const int64_t *req, int64_t n_req, void *out,
                        cudaStream_t st)
{
    if (wide(c))
        return read_t(c, pts, n_streams, n, pt_stride, req, n_req, static_cast<uint16_t *>(out), st);
    return read_t(c, pts, n_streams, n, pt_stride, req, n_req, static_cast<uint8_t *>(out), st);
}

template <typename Sym>
cudaError_t append_t(const fkv_ctx *c, double *pts, int64_t n_streams, int64_t pt_stride, int64_t n_old,
                     const Sym *sym, int64_t m, int64_t sym_stride, cudaStream_t st)
{
    if (m <= 0 || n_streams <= 0)
        return cudaSuccess;
    const int L = c->L;
    int64_t head = 0;   // new symbols that finish the stored partial span
    if (n_old % L) {
        head = min(m, L - n_old % L);
        const int64_t blocks = cdiv(n_streams, kThreads);
        if (blocks > 0x7FFFFFFF)
            return cudaErrorInvalidConfiguration;
        k_append<Sym><<<static_cast<unsigned>(blocks), kThreads, 0, st>>>(
            reinterpret_cast<double2 *>(pts), n_streams, pt_stride, n_old, sym, head, sym_stride, n_old / L, 1,
            c->d_V, c->N, c->r, L, c->d_status);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess)
            return e;
    }
    if (m == head)
        return cudaSuccess;
    // every later span starts at the anchor: the bulk span encoder on the
    // remaining symbols, writing from span (n_old + head) / L on
    return span_encode_t(c, sym + head, n_streams, m - head, sym_stride, pts + 2 * ((n_old + head) / L),
                         pt_stride, st);
}

cudaError_t launch_append(const fkv_ctx *c, double *pts, int64_t n_streams, int64_t pt_stride,
                          int64_t n_old, const void *sym, int64_t m, int64_t sym_stride,
                          cudaStream_t st)
{
    if (wide(c))
        return append_t(c, pts, n_streams, pt_stride, n_old, static_cast<const uint16_t *>(sym), m, sym_stride,
                        st);
    return append_t(c, pts, n_streams, pt_stride, n_old, static_cast<const uint8_t *>(sym), m, sym_stride, st);
}

// ------------------------------------------------------------ lossy launches
namespace {

LossyArgs lossy_args(const fkv_ctx *c, const uint32_t *codes, int64_t code_stride, const double *tail,
                     int64_t tail_stride, int64_t n, int bits, int64_t keep_exact)
{
    LossyArgs a;
    const int64_t spans = cdiv(n, c->L);
    a.T = spans > keep_exact ? spans - keep_exact : 0;
    a.codes = codes;
    a.code_stride = code_stride;
    a.words = cdiv(2 * a.T * bits, 32);
    a.tail = reinterpret_cast<const double2 *>(tail);
    a.tail_stride = tail_stride;
    a.bits = bits;
    a.scale = ldexp(1.0, -(bits - 1));
    return a;
}

template <typename Sym>
cudaError_t lossy_decode_t(const fkv_ctx *c, const LossyArgs &a, int64_t n_streams, int64_t n, Sym *sym,
                           int64_t sym_stride, cudaStream_t st)
{
    const int64_t spans = cdiv(n, c->L);
    const int64_t bps = cdiv(spans, kThreads);
    const int64_t n_chunks = n_streams * bps;
    if (n_chunks == 0)
        return cudaSuccess;
    if (bps > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    const int smem = c->N * 16 + ((kThreads * c->L * static_cast<int>(sizeof(Sym)) + 32 + 15) & ~15);
    cudaError_t e = cudaFuncSetAttribute(k_lossy_decode<Sym>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    unsigned grid = 0;
    e = decode_grid(c, reinterpret_cast<const void *>(k_lossy_decode<Sym>), smem, n_chunks, &grid);
    if (e != cudaSuccess)
        return e;
    k_lossy_decode<Sym><<<grid, kThreads, smem, st>>>(a, n, spans, static_cast<int>(bps), n_chunks, sym, sym_stride,
                                                      c->d_V, c->N, 1.0 - c->r, c->r, c->L);
    return cudaGetLastError();
}

template <typename Sym>
cudaError_t lossy_read_t(const fkv_ctx *c, const LossyArgs &a, int64_t n_streams, int64_t n, const int64_t *req,
                         int64_t n_req, Sym *out, cudaStream_t st)
{
    const int64_t blocks = cdiv(n_req, kThreads);
    if (blocks == 0)
        return cudaSuccess;
    const int smem = c->N * 16;
    cudaError_t e = cudaFuncSetAttribute(k_lossy_read<Sym>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    unsigned grid = 0;
    e = decode_grid(c, reinterpret_cast<const void *>(k_lossy_read<Sym>), smem, blocks, &grid);
    if (e != cudaSuccess)
        return e;
    k_lossy_read<Sym><<<grid, kThreads, smem, st>>>(a, n_streams, n, req, n_req, out, c->d_V, c->N, 1.0 - c->r,
                                                    c->r, c->L, c->d_status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_truncate(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n, int64_t pt_stride,
                            int bits, int64_t keep_exact, uint32_t *codes, int64_t code_stride, double *tail,
                            int64_t tail_stride, cudaStream_t st)
{
    const int64_t spans = cdiv(n, c->L);
    const int64_t T = spans > keep_exact ? spans - keep_exact : 0;
    const int64_t words = cdiv(2 * T * bits, 32);
    if (n_streams > 0 && words > 0) {
        int sms = 0;
        cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
        if (e != cudaSuccess)
            return e;
        const int64_t blocks = min(cdiv(n_streams * cdiv(T, 32), kThreads / 32), static_cast<int64_t>(sms) * 8);
        k_truncate<<<static_cast<unsigned>(blocks), kThreads, 0, st>>>(pts, pt_stride, n_streams, T, bits, codes,
                                                                        code_stride, words);
        e = cudaGetLastError();
        if (e != cudaSuccess)
            return e;
    }
    if (tail && n_streams > 0 && spans > T)
        return cudaMemcpy2DAsync(tail, tail_stride * 16, pts + 2 * T, pt_stride * 16, (spans - T) * 16, n_streams,
                                 cudaMemcpyDeviceToDevice, st);
    return cudaSuccess;
}

cudaError_t launch_lossy_decode(const fkv_ctx *c, const uint32_t *codes, int64_t code_stride, const double *tail,
                                int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                                void *sym, int64_t sym_stride, cudaStream_t st)
{
    const LossyArgs a = lossy_args(c, codes, code_stride, tail, tail_stride, n, bits, keep_exact);
    if (wide(c))
        return lossy_decode_t(c, a, n_streams, n, static_cast<uint16_t *>(sym), sym_stride, st);
    return lossy_decode_t(c, a, n_streams, n, static_cast<uint8_t *>(sym), sym_stride, st);
}

cudaError_t launch_lossy_read(const fkv_ctx *c, const uint32_t *codes, int64_t code_stride, const double *tail,
                              int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                              const int64_t *req, int64_t n_req, void *out, cudaStream_t st)
{
    const LossyArgs a = lossy_args(c, codes, code_stride, tail, tail_stride, n, bits, keep_exact);
    if (wide(c))
        return lossy_read_t(c, a, n_streams, n, req, n_req, static_cast<uint16_t *>(out), st);
    return lossy_read_t(c, a, n_streams, n, req, n_req, static_cast<uint8_t *>(out), st);
}


// ------------------------------------------------------------ ragged launches
namespace {

// Persistent grid for the ragged kernels: the slot count lives on the device,
// so the grid is sized to fill the GPU and the kernels stride over the slots.
template <typename Sym>
cudaError_t ragged_decoder_grid(const fkv_ctx *c, const void *kern, int smem, unsigned *grid)
{
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    return decode_grid(c, kern, smem, 1ll << 40, grid, dec_threads<Sym>());
}

template <typename Sym>
cudaError_t encode_ragged_t(const fkv_ctx *c, const Sym *sym, const int64_t *so, int64_t n_streams, double *pts,
                            const int64_t *po, cudaStream_t st)
{
    unsigned grid = 0;
    cudaError_t e = decode_grid(c, reinterpret_cast<const void *>(k_span_encode_ragged<Sym>), 0, 1ll << 40, &grid);
    if (e != cudaSuccess)
        return e;
    k_span_encode_ragged<Sym><<<grid, kThreads, 0, st>>>(sym, so, n_streams, reinterpret_cast<double2 *>(pts), po,
                                                         c->d_V, c->N, c->r, c->L, c->d_status);
    return cudaGetLastError();
}

template <typename Sym>
cudaError_t decode_ragged_t(const fkv_ctx *c, const double *pts, const int64_t *po, int64_t n_streams, Sym *sym,
                            const int64_t *so, cudaStream_t st)
{
    const int smem = tables_bytes(c->N, c->L);
    unsigned grid = 0;
    cudaError_t e = ragged_decoder_grid<Sym>(c, reinterpret_cast<const void *>(k_span_decode_ragged<Sym>), smem,
                                             &grid);
    if (e != cudaSuccess)
        return e;
    k_span_decode_ragged<Sym><<<grid, dec_threads<Sym>(), smem, st>>>(reinterpret_cast<const double2 *>(pts), po,
                                                                      n_streams, sym, so, c->d_dec, c->d_T, c->N,
                                                                      c->L, c->d_status);
    return cudaGetLastError();
}

template <typename Sym>
cudaError_t read_ragged_t(const fkv_ctx *c, const double *pts, const int64_t *po, const int64_t *so,
                          int64_t n_streams, const int64_t *req, int64_t n_req, Sym *out, cudaStream_t st)
{
    const int smem = tables_bytes(c->N, c->L);
    unsigned grid = 0;
    cudaError_t e = ragged_decoder_grid<Sym>(c, reinterpret_cast<const void *>(k_read_ragged<Sym>), smem, &grid);
    if (e != cudaSuccess)
        return e;
    const int64_t need = cdiv(n_req, dec_threads<Sym>());
    if (static_cast<int64_t>(grid) > need)
        grid = static_cast<unsigned>(need);
    k_read_ragged<Sym><<<grid, dec_threads<Sym>(), smem, st>>>(reinterpret_cast<const double2 *>(pts), po, so,
                                                               n_streams, req, n_req, out, c->d_dec, c->d_T, c->N,
                                                               c->L, c->d_status);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_span_encode_ragged(const fkv_ctx *c, const void *sym, const int64_t *so, int64_t n_streams,
                                      double *pts, const int64_t *po, cudaStream_t st)
{
    if (wide(c))
        return encode_ragged_t(c, static_cast<const uint16_t *>(sym), so, n_streams, pts, po, st);
    return encode_ragged_t(c, static_cast<const uint8_t *>(sym), so, n_streams, pts, po, st);
}

cudaError_t launch_span_decode_ragged(const fkv_ctx *c, const double *pts, const int64_t *po, int64_t n_streams,
                                      void *sym, const int64_t *so, cudaStream_t st)
{
    if (wide(c))
        return decode_ragged_t(c, pts, po, n_streams, static_cast<uint16_t *>(sym), so, st);
    return decode_ragged_t(c, pts, po, n_streams, static_cast<uint8_t *>(sym), so, st);
}

cudaError_t launch_read_ragged(const fkv_ctx *c, const double *pts, const int64_t *po, const int64_t *so,
                               int64_t n_streams, const int64_t *req, int64_t n_req, void *out, cudaStream_t st)
{
    if (wide(c))
        return read_ragged_t(c, pts, po, so, n_streams, req, n_req, static_cast<uint16_t *>(out), st);
    return read_ragged_t(c, pts, po, so, n_streams, req, n_req, static_cast<uint8_t *>(out), st);
}

// ------------------------------------------------------------ FP64 probe
// Binary64 add/mul throughput with independent chains: every thread runs
// kChains chains of x <- x * a, x <- x + b (round to nearest, no FMA: the
// encoder's operation mix), whose fixed point b / (1 - a) keeps the values
// bounded.  The chains' sum is written only when it equals an impossible
// value, so the work stays live without a store per thread.
namespace {
constexpr int kFp64Chains = 8;
__device__ double g_fp64_sink;

__global__ void __launch_bounds__(256) k_fp64_rate(int iters, double a, double b)
{
    double x[kFp64Chains];
#pragma unroll
    for (int i = 0; i < kFp64Chains; ++i)
        x[i] = 1.0 + 1e-3 * i + 1e-7 * threadIdx.x;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < kFp64Chains; ++i) {
            x[i] = __dmul_rn(x[i], a);
            x[i] = __dadd_rn(x[i], b);
        }
    }
    double s = 0.0;
#pragma unroll
    for (int i = 0; i < kFp64Chains; ++i)
        s += x[i];
    if (s == -1.0)
        g_fp64_sink = s;
}
}  // namespace

cudaError_t measure_fp64_rate(int device, cudaStream_t st, double *ops_per_s)
{
    int sms = 0;
    cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess)
        return e;
    const int blocks = sms * 4, iters = 4096;
    cudaEvent_t t0, t1;
    if ((e = cudaEventCreate(&t0)) != cudaSuccess)
        return e;
    if ((e = cudaEventCreate(&t1)) != cudaSuccess) {
        cudaEventDestroy(t0);
        return e;
    }
    float best = 0.0f;
    for (int rep = 0; rep < 4 && e == cudaSuccess; ++rep) {   // the first launch warms up
        cudaEventRecord(t0, st);
        k_fp64_rate<<<blocks, 256, 0, st>>>(iters, 0.99999999, 1e-8);
        cudaEventRecord(t1, st);
        e = cudaGetLastError();
        if (e == cudaSuccess)
            e = cudaEventSynchronize(t1);
        float ms = 0.0f;
        if (e == cudaSuccess)
            e = cudaEventElapsedTime(&ms, t0, t1);
        if (e == cudaSuccess && rep > 0 && (best == 0.0f || ms < best))
            best = ms;
    }
    cudaEventDestroy(t0);
    cudaEventDestroy(t1);
    if (e != cudaSuccess)
        return e;
    *ops_per_s = 2.0 * kFp64Chains * static_cast<double>(iters) * blocks * 256 / (best * 1e-3);
    return cudaSuccess;
}
