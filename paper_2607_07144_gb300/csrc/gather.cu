// Codebook gather: K/V reconstruction from RVQ indices (Sec. 3 "Setup": the
// reconstruction is the sum of the selected centroids), for whole archives
// and for random record reads (Sec. 2).
//
// Whole archive: persistent blocks, each taking an equal share of the
// (codebook group, dimension slice, head sharing the group, vector) work.  A
// block holds the float32 codebooks of one group and one slice of the head
// dimension (all stages) in shared memory while it works on that slice, so
// HBM sees only the indices in and the rebuilt K/V out.  Codebooks of 256
// codewords take uint8 indices, of 1024 codewords uint16.  A thread rebuilds eight dimensions
// (two 16-byte granules of a slice row) of a vector, four in 16-float slices.  Sums run in float32, stage
// order, then round to nearest-even into the cache dtype.
//
// Each round of four vectors per thread prefetches the next round's index
// words into L1 (decode_kv on the Llama-shaped archive: 5.29 -> 4.70 ms).
//
// Shared-memory reads are conflict-free for any indices: a slice row spans a
// multiple of 128 bytes, so its granule g lies in bank group g % 8.  A thread
// owns granules 2q and 2q + 1; lanes 0-3 of a quarter warp read the even one
// first and lanes 4-7 the odd one, so each read covers the eight bank groups
// once (32-float rows: two vectors per quarter warp; 64-float rows: one).  A
// 16-float slice (two rows per bank line, for more than four stages) gives a
// thread one granule and permutes granules by an XOR of the row instead.
#include <type_traits>

#include "decode_core.cuh"

namespace {

constexpr int kThreads = 1024;

struct GatherArgs {
    const void *sym;       // the S indices of (b, l, h, rec) at sym + b ib + l il + h ih + rec ir + ioff (symbols)
    int64_t ib, il, ih, ir, ioff;
    int64_t n_rec, batch, t0;
    int n_layers, n_heads, D, S;
    int pooled;            // one codebook per layer (1) or per (layer, head) (0)
    const float *cb32;     // [G][S][KC][D]
    void *out;
    int dtype;
    int64_t s_layer, s_batch, s_head, s_pos;
    int parts, Dp;
};

__device__ __forceinline__ void store2(void *out, int dtype, int64_t elem, float a, float b)
{
    if (dtype == FKV_F32) {
        *reinterpret_cast<float2 *>(static_cast<float *>(out) + elem) = make_float2(a, b);
    } else if (dtype == FKV_F16) {
        *reinterpret_cast<__half2 *>(static_cast<__half *>(out) + elem) = __floats2half2_rn(a, b);
    } else {
        *reinterpret_cast<__nv_bfloat162 *>(static_cast<__nv_bfloat16 *>(out) + elem) =
            __floats2bfloat162_rn(a, b);
    }
}

__device__ __forceinline__ uint32_t pack2(int dtype, float a, float b)
{
    if (dtype == FKV_F16) {
        const __half2 v = __floats2half2_rn(a, b);
        return *reinterpret_cast<const uint32_t *>(&v);
    }
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&v);
}

// Eight consecutive elements at `elem` (16-byte aligned): lo then hi.
__device__ __forceinline__ void store8(void *out, int dtype, int64_t elem, float4 lo, float4 hi)
{
    if (dtype == FKV_F32) {
        float4 *p = reinterpret_cast<float4 *>(static_cast<float *>(out) + elem);
        p[0] = lo;
        p[1] = hi;
        return;
    }
    *reinterpret_cast<uint4 *>(static_cast<uint16_t *>(out) + elem) =
        make_uint4(pack2(dtype, lo.x, lo.y), pack2(dtype, lo.z, lo.w), pack2(dtype, hi.x, hi.y),
                   pack2(dtype, hi.z, hi.w));
}

// Four consecutive elements at `elem` (aligned to their size).
__device__ __forceinline__ void store4(void *out, int dtype, int64_t elem, float4 x)
{
    if (dtype == FKV_F32) {
        *reinterpret_cast<float4 *>(static_cast<float *>(out) + elem) = x;
        return;
    }
    *reinterpret_cast<uint2 *>(static_cast<uint16_t *>(out) + elem) = make_uint2(pack2(dtype, x.x, x.y),
                                                                                  pack2(dtype, x.z, x.w));
}

// x0 += c0, x1 += c1 as one packed fp32 add (each lane rounds like a scalar add).
__device__ __forceinline__ void add2(float &x0, float &x1, float c0, float c1)
{
    asm("{\n\t.reg .b64 u, w;\n\t"
        "mov.b64 u, {%0, %1};\n\t"
        "mov.b64 w, {%2, %3};\n\t"
        "add.rn.f32x2 u, u, w;\n\t"
        "mov.b64 {%0, %1}, u;\n\t}"
        : "+f"(x0), "+f"(x1)
        : "f"(c0), "f"(c1));
}

// The S stage indices of one vector, first stage in the low bits (8 or 16
// bits each, by symbol type): one load of the whole run when it is aligned
// (WIDE, a run of 2, 4 or 8 bytes), else one load per index.
template <int S, bool WIDE, typename Sym>
__device__ __forceinline__ uint64_t load_ids(const Sym *p)
{
    constexpr int bytes = S * static_cast<int>(sizeof(Sym));
    if (WIDE && bytes == 4)
        return __ldg(reinterpret_cast<const unsigned *>(p));
    if (WIDE && bytes == 2)
        return __ldg(reinterpret_cast<const unsigned short *>(p));
    if (WIDE && bytes == 8)
        return __ldg(reinterpret_cast<const unsigned long long *>(p));
    uint64_t w = 0;
#pragma unroll
    for (int s = 0; s < S; ++s)
        w |= static_cast<uint64_t>(__ldg(p + s)) << (8 * sizeof(Sym) * s);
    return w;
}

// The slice width: the widest of 64, 32 or 16 floats whose codebook slice
// (all stages, KC codewords each) fits 128 KB; rows of 64 or 32 floats span
// whole 128-byte bank lines.
__host__ __device__ constexpr int gather_dp(int S, int KC)
{
    return KC == 256 ? (S <= 2 ? 64 : (S <= 4 ? 32 : 16)) : (S <= 1 ? 32 : 16);
}

// The stage sum of one vector's eight dimensions (granules ga, gb of its
// slice row; q4 granules per row) from the codebook slice in shared memory:
// float32, stage order.  ids holds the S indices, the first in the low bits.
template <int S, int KC>
__device__ __forceinline__ void sum_stages8(const float4 *row0, uint64_t ids, int ga, int gb, float4 &x, float4 &y)
{
    constexpr int kBits = KC == 256 ? 8 : 16;
    constexpr uint64_t kMask = (1ull << kBits) - 1;
    constexpr int q4 = gather_dp(S, KC) / 4;
    x = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    y = x;
#pragma unroll
    for (int s = 0; s < S; ++s) {
        const int row = s * KC + static_cast<int>((ids >> (kBits * s)) & kMask);
        const float4 c = row0[row * q4 + ga];
        const float4 e = row0[row * q4 + gb];
        add2(x.x, x.y, c.x, c.y);
        add2(x.z, x.w, c.z, c.w);
        add2(y.x, y.y, e.x, e.y);
        add2(y.z, y.w, e.z, e.w);
    }
}

// The same for four dimensions of a 16-float slice row (granule dq; rows
// permute their granules by an XOR of the row).
template <int S, int KC>
__device__ __forceinline__ float4 sum_stages4(const float4 *row0, uint64_t ids, int dq)
{
    constexpr int kBits = KC == 256 ? 8 : 16;
    constexpr uint64_t kMask = (1ull << kBits) - 1;
    constexpr int Dp = gather_dp(S, KC);
    constexpr int q4 = Dp / 4;
    constexpr bool xor_rows = Dp < 32;
    float4 x = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
    for (int s = 0; s < S; ++s) {
        const int row = s * KC + static_cast<int>((ids >> (kBits * s)) & kMask);
        const int xq = xor_rows ? (row >> 1) & 3 : 0;
        const float4 c = row0[row * q4 + (dq ^ xq)];
        add2(x.x, x.y, c.x, c.y);
        add2(x.z, x.w, c.z, c.w);
    }
    return x;
}

// A (codebook group, dimension slice) of float32 codebooks (all S stages, KC
// codewords each, Dp floats of every row) into shared memory: every 16-byte
// copy in flight, one wait.  The block meets at both ends.
template <int S, int KC>
__device__ __forceinline__ void load_slice(float *scb, const float *src, int D)
{
    constexpr int Dp = gather_dp(S, KC);
    constexpr int q4 = Dp / 4;
    constexpr bool xor_rows = Dp < 32;
    __syncthreads();
    for (int i = threadIdx.x; i < S * KC * q4; i += blockDim.x) {
        const int row = i / q4, q = i - row * q4;
        const int pq = xor_rows ? q ^ ((row >> 1) & 3) : q;
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(fkvd::smem_u32(scb + 4 * (row * q4 + pq))),
                     "l"(src + static_cast<int64_t>(row) * D + 4 * q)
                     : "memory");
    }
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
    __syncthreads();
}

template <int S, bool WIDE, int KC>
__global__ void __launch_bounds__(kThreads, 1) k_gather(const GatherArgs a)
{
    using Sym = typename std::conditional<KC == 256, uint8_t, uint16_t>::type;
    constexpr int kBits = 8 * sizeof(Sym);
    extern __shared__ __align__(128) float scb[];   // [S][KC][Dp] floats
    constexpr int Dp = gather_dp(S, KC);
    const int D = a.D, parts = a.parts;
    constexpr int kDT = Dp >= 32 ? 8 : 4;    // dimensions a thread rebuilds
    constexpr int tpv = Dp / kDT;            // threads per vector
    constexpr int vpi = kThreads / tpv;      // vectors per pass
    const int dq = threadIdx.x % tpv;        // this thread's granule (pair) of the slice row
    // Two granules per thread: the upper four lanes of each quarter warp read
    // their pair in the opposite order, so each read instruction's quarter
    // warp covers the eight bank groups once whatever rows it reads
    const int ph = kDT == 8 ? (threadIdx.x >> 2) & 1 : 0;
    const int64_t n_rec = a.n_rec;
    // advancing by vpi vectors: step_r records and step_b sequences, plus one
    // more sequence when the record wraps
    const int step_b = static_cast<int>(vpi / n_rec), step_r = static_cast<int>(vpi - step_b * n_rec);
    const int64_t di_step = step_b * a.ib + step_r * a.ir, di_wrap = a.ib - n_rec * a.ir;
    const int64_t do_step = step_b * a.s_batch + step_r * a.s_pos, do_wrap = a.s_batch - n_rec * a.s_pos;
    // this block's share of the work: slots ((cgroup * parts + part) * HH +
    // head of the group) * nvec + vector, HH heads sharing a codebook group
    const int HH = a.pooled ? a.n_heads : 1;
    const int64_t nvec = a.batch * n_rec;
    const int64_t total = static_cast<int64_t>(a.n_layers) * a.n_heads * parts * nvec;
    int64_t lo = total * blockIdx.x / gridDim.x;
    const int64_t hi = total * (blockIdx.x + 1) / gridDim.x;
    int64_t cur = -1;                        // (group, part) whose slice is in shared memory
    while (lo < hi) {
        const int64_t gph = lo / nvec;
        const int64_t v0 = lo - gph * nvec;
        const int64_t v1 = min(nvec, v0 + (hi - lo));
        lo += v1 - v0;
        const int64_t gp = gph / HH;
        const int hh = static_cast<int>(gph - gp * HH);
        const int cgi = static_cast<int>(gp / parts), part = static_cast<int>(gp % parts);
        const int g = a.pooled ? cgi * a.n_heads + hh : cgi;
        const int l = g / a.n_heads, h = g % a.n_heads;
        const int d0 = part * Dp;
        if (gp != cur) {
            load_slice<S, KC>(scb, a.cb32 + static_cast<int64_t>(cgi) * S * KC * D + d0, D);
            cur = gp;
        }
        const int64_t v = v0 + threadIdx.x / tpv;
        if (v >= v1)
            continue;
        int n_it = static_cast<int>((v1 - v + vpi - 1) / vpi);
        const int64_t b = v / n_rec;
        int rec = static_cast<int>(v - b * n_rec);
        const Sym *ip = static_cast<const Sym *>(a.sym) + l * a.il + h * a.ih + a.ioff + b * a.ib + rec * a.ir;
        int64_t oe = l * a.s_layer + h * a.s_head + (a.t0 + rec) * a.s_pos + b * a.s_batch + d0 + dq * kDT;
        const float4 *row0 = reinterpret_cast<const float4 *>(scb);
        // kU vectors per round: their index loads are all issued before any is used
        constexpr int kU = 4;
        for (; n_it > 0; n_it -= kU) {
            using Ids = typename std::conditional<S * kBits <= 32, uint32_t, uint64_t>::type;
            Ids ids[kU];
            int64_t off[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                ids[u] = u < n_it ? static_cast<Ids>(load_ids<S, WIDE>(ip)) : 0;
                off[u] = oe;
                rec += step_r;
                ip += di_step;
                oe += do_step;
                if (rec >= n_rec) {
                    rec -= static_cast<int>(n_rec);
                    ip += di_wrap;
                    oe += do_wrap;
                }
            }
            // the next round's index words into L1 while this round's gathers
            // run: vectors of this thread's range whose record does not wrap
            // (their address is then ip + u * di_step exactly)
#pragma unroll
            for (int u = 0; u < kU; ++u)
                if (u + kU < n_it && rec + static_cast<int64_t>(u) * step_r < n_rec)
                    asm volatile("prefetch.global.L1 [%0];" ::"l"(ip + u * di_step));
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                if (u >= n_it)
                    break;
                if constexpr (kDT == 8) {
                    float4 x, y;
                    sum_stages8<S, KC>(row0, ids[u], 2 * dq + ph, 2 * dq + 1 - ph, x, y);
                    store8(a.out, a.dtype, off[u], ph ? y : x, ph ? x : y);
                } else {
                    store4(a.out, a.dtype, off[u], sum_stages4<S, KC>(row0, ids[u], dq));
                }
            }
        }
    }
}

template <int S, int KC>
void *gather_kernel(bool wide)
{
    constexpr int bytes = S * (KC == 256 ? 1 : 2);
    if ((bytes == 2 || bytes == 4 || bytes == 8) && wide)
        return reinterpret_cast<void *>(k_gather<S, true, KC>);
    return reinterpret_cast<void *>(k_gather<S, false, KC>);
}

// 256-codeword codebooks take 1..8 stages, 1024-codeword ones 1 or 2.
void *gather_kernel_for(int S, bool wide, int KC)
{
    if (KC == 1024)
        return S == 1 ? gather_kernel<1, 1024>(wide) : gather_kernel<2, 1024>(wide);
    switch (S) {
    case 1: return gather_kernel<1, 256>(wide);
    case 2: return gather_kernel<2, 256>(wide);
    case 3: return gather_kernel<3, 256>(wide);
    case 4: return gather_kernel<4, 256>(wide);
    case 5: return gather_kernel<5, 256>(wide);
    case 6: return gather_kernel<6, 256>(wide);
    case 7: return gather_kernel<7, 256>(wide);
    default: return gather_kernel<8, 256>(wide);
    }
}

// ------------------------------------------------------- random reads ---
constexpr int kReadWarps = 8;
constexpr int kMaxRecord = 1024;

struct ReadArgs {
    const double2 *pts;
    int64_t n_streams, n_rec, pt_stride;
    const int64_t *req;
    const int4 *order;             // (request, stream or -1, record, 0) grouped by layer, or null
    int64_t n_req;
    void *out;
    int dtype;
    int n_layers, n_heads, D, SK, SV, R, N, L;
    int KC, pooled;                // codewords per stage; one codebook per layer (1) or per head (0)
    const float *cbk, *cbv;
    const fkv_decconst *dec;
    const longlong2 *T;
    unsigned *status;
    void *scr;                     // staged reads: entry i's record symbols at scr + i R
};

__host__ __device__ inline int read_tables_bytes(int N, int L)
{
    return (fkvdec::smem_bytes(N, L) + 15) & ~15;
}

// One warp per request: its lanes decode the spans covering the record into
// shared memory, then rebuild the record's 2 * H head vectors, eight
// consecutive dimensions per lane and item (two 16-byte codeword loads per
// stage, four stages' loads issued before their sums).  Persistent: a block
// loads the decoder tables once and its warps take requests blockIdx.x *
// warps + warp, + gridDim.x * warps, ...  Three blocks per SM (80 registers,
// a few spilled to L1) beat two without spills: 1.12 against 1.20 ms for
// 262,144 Llama-shaped records.
template <typename Sym>
__global__ void __launch_bounds__(kReadWarps * 32, 3) k_read_kv(const ReadArgs a)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(a.dec, a.T, a.N, a.L, dsm);
    Sym *srec = reinterpret_cast<Sym *>(dsm + read_tables_bytes(a.N, a.L));
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int H = a.n_heads, D = a.D, R = a.R, L = a.L;
    const int64_t out_vec = static_cast<int64_t>(2) * H * D;
    const int gsh = D == 128 ? 4 : 3;             // log2 of the 8-dimension groups per head
    const int items = 2 * H << gsh;
    Sym *my = srec + warp * kMaxRecord;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * kReadWarps + warp; i < a.n_req;
         i += static_cast<int64_t>(gridDim.x) * kReadWarps) {
        int64_t q = i, st, rec;
        if (a.order) {
            const int4 e = a.order[i];
            q = e.x;
            st = e.y;
            rec = e.z;
        } else {
            st = a.req[2 * q];
            rec = a.req[2 * q + 1];
        }
        if (st < 0 || st >= a.n_streams || rec < 0 || rec >= a.n_rec) {
            for (int64_t i = lane; i < out_vec / 2; i += 32)
                store2(a.out, a.dtype, q * out_vec + 2 * i, 0.0f, 0.0f);
            if (lane == 0)
                atomicOr(a.status, FKV_ST_RANGE);
            continue;
        }
        const int64_t n = a.n_rec * R;
        const int64_t sym0 = rec * R;
        const int64_t u0 = sym0 / L, u1 = (sym0 + R - 1) / L;
        bool bad = false;
        for (int64_t u = u0 + lane; u <= u1; u += 32) {
            const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
            const double2 p = a.pts[st * a.pt_stride + u];
            long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
            const int64_t base = u * L - sym0;
            fkvdec::walk<true>(t, X, Y, m, [&](int j, int c) {
                const int64_t pos = base + m - 1 - j;
                if (pos >= 0 && pos < R)
                    my[pos] = static_cast<Sym>(c);
            });
            const long long lim = __ldg(&a.dec->alim[m]);
            bad |= X > lim || X < -lim || Y > lim || Y < -lim;
        }
        if (bad)
            atomicOr(a.status, FKV_ST_CORRUPT);
        __syncwarp();
        const int l = static_cast<int>(st % a.n_layers);
#pragma unroll 2
        for (int g = lane; g < items; g += 32) {
            const int kv = g >= (H << gsh) ? 1 : 0;
            const int gi = kv ? g - (H << gsh) : g;
            const int hh = gi >> gsh, d0 = (gi - (hh << gsh)) * 8;
            const int S = kv ? a.SV : a.SK;
            const float *cb = kv ? a.cbv : a.cbk;
            const int off = kv ? H * a.SK : 0;
            const int64_t cg = a.pooled ? l : static_cast<int64_t>(l) * H + hh;
            const float *gcb = cb + cg * S * a.KC * D + d0;
            float4 x = make_float4(0.0f, 0.0f, 0.0f, 0.0f), y = x;
            for (int s0 = 0; s0 < S; s0 += 4) {
                float4 c[8];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    if (s0 + k < S) {
                        const float4 *row = reinterpret_cast<const float4 *>(
                            gcb + (static_cast<int64_t>(s0 + k) * a.KC + my[off + hh * S + s0 + k]) * D);
                        c[2 * k] = __ldg(row);
                        c[2 * k + 1] = __ldg(row + 1);
                    }
                }
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    if (s0 + k < S) {
                        x.x += c[2 * k].x;
                        x.y += c[2 * k].y;
                        x.z += c[2 * k].z;
                        x.w += c[2 * k].w;
                        y.x += c[2 * k + 1].x;
                        y.y += c[2 * k + 1].y;
                        y.z += c[2 * k + 1].z;
                        y.w += c[2 * k + 1].w;
                    }
                }
            }
            store8(a.out, a.dtype, q * out_vec + (static_cast<int64_t>(kv) * H + hh) * D + d0, x, y);
        }
        __syncwarp();                             // the next request reuses `my`
    }
}

// Staged record reads, first step: the symbols of every entry's record into
// scr + i R, one thread per (entry, span covering the record) so that every
// lane walks a span (a record of R symbols spans about R / L of them); the
// decoder tables are loaded once per persistent block.  An out-of-range
// entry (stream -1, the last run) writes its request's zeros and sets
// FKV_ST_RANGE instead.
template <typename Sym>
__global__ void __launch_bounds__(256) k_read_syms(const ReadArgs a, int spr)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(a.dec, a.T, a.N, a.L, dsm);
    __syncthreads();
    const int R = a.R, L = a.L;
    const int64_t n = a.n_rec * R;
    const int64_t out_vec = static_cast<int64_t>(2) * a.n_heads * a.D;
    Sym *scr = static_cast<Sym *>(a.scr);
    const int64_t items = a.n_req * spr;
    for (int64_t it = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; it < items;
         it += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = it / spr;
        const int k = static_cast<int>(it - i * spr);
        const int4 e = a.order[i];
        if (e.y < 0) {
            // out of range: this thread's share of the request's zeros
            for (int64_t j = 2 * k; j < out_vec; j += 2 * spr)
                store2(a.out, a.dtype, e.x * out_vec + j, 0.0f, 0.0f);
            if (k == 0)
                atomicOr(a.status, FKV_ST_RANGE);
            continue;
        }
        const int64_t sym0 = static_cast<int64_t>(e.z) * R;
        const int64_t u = sym0 / L + k;
        if (u > (sym0 + R - 1) / L)
            continue;
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
        const double2 p = a.pts[e.y * a.pt_stride + u];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        const int64_t base = u * L - sym0;
        Sym *dst = scr + i * R;
        fkvdec::walk<true>(t, X, Y, m, [&](int j, int c) {
            const int64_t pos = base + m - 1 - j;
            if (pos >= 0 && pos < R)
                dst[pos] = static_cast<Sym>(c);
        });
        const long long lim = __ldg(&a.dec->alim[m]);
        if (X > lim || X < -lim || Y > lim || Y < -lim)
            atomicOr(a.status, FKV_ST_CORRUPT);
    }
}

// Staged record reads, second step: the K (kv 0) or V (kv 1) head vectors of
// every in-range request rebuilt like the whole-archive gather, from a
// (codebook group, dimension slice) held in shared memory.  Entries are the
// layer-ordered requests: entry i's symbols at scr + i R (the first step
// decoded them), its request at order[i].x, and layer l's entries end at
// ends[l].  Work items are (layer, head and slice, entry) in that order
// (slice-major over the heads when the layer's codebook is pooled, so the
// slice stays for all of them); each block takes an equal share and loads a
// slice when its group or slice changes.  With thousands of requests per
// layer each slice serves many vectors from shared memory instead of every
// vector reading its codeword rows from L2.
struct ReadGatherArgs {
    const void *scr;
    const int4 *order;
    const int *ends;
    const float *cb32;     // [G][S][KC][D]
    void *out;             // [n_req][2][H][D]
    int dtype;
    int n_layers, n_heads, D, R, off, kv, pooled, parts;
};

template <int S, bool WIDE, int KC>
__global__ void __launch_bounds__(kThreads, 1) k_read_gather(const ReadGatherArgs a)
{
    using Sym = typename std::conditional<KC == 256, uint8_t, uint16_t>::type;
    constexpr int kBits = 8 * sizeof(Sym);
    extern __shared__ __align__(128) float scb[];   // [S][KC][Dp] floats
    constexpr int Dp = gather_dp(S, KC);
    constexpr int kDT = Dp >= 32 ? 8 : 4;
    constexpr int tpv = Dp / kDT;
    constexpr int vpi = kThreads / tpv;
    constexpr int kU = 4;
    const int D = a.D, H = a.n_heads, parts = a.parts, R = a.R;
    const int GHP = H * parts;
    const int dq = threadIdx.x % tpv;
    const int ph = kDT == 8 ? (threadIdx.x >> 2) & 1 : 0;
    const int64_t out_vec = static_cast<int64_t>(2) * H * D;
    const int64_t total = static_cast<int64_t>(GHP) * __ldg(&a.ends[a.n_layers - 1]);
    int64_t lo = total * blockIdx.x / gridDim.x;
    const int64_t hi = total * (blockIdx.x + 1) / gridDim.x;
    int64_t cur = -1;
    int l = 0;
    int64_t start = 0, end = __ldg(&a.ends[0]);
    const Sym *scr = static_cast<const Sym *>(a.scr);
    const float4 *row0 = reinterpret_cast<const float4 *>(scb);
    while (lo < hi) {
        // layer l's items are [GHP start_l, GHP end_l); empty layers are passed over
        while (lo >= static_cast<int64_t>(GHP) * end) {
            ++l;
            start = end;
            end = __ldg(&a.ends[l]);
        }
        const int64_t n_l = end - start;
        const int64_t r = lo - static_cast<int64_t>(GHP) * start;
        const int seg = static_cast<int>(r / n_l);
        const int64_t j0 = r - seg * n_l;
        const int64_t j1 = min(n_l, j0 + (hi - lo));
        lo += j1 - j0;
        int h, part;
        if (a.pooled) {
            part = seg / H;
            h = seg - part * H;
        } else {
            h = seg / parts;
            part = seg - h * parts;
        }
        const int64_t cg = a.pooled ? l : static_cast<int64_t>(l) * H + h;
        if (cg * parts + part != cur) {
            load_slice<S, KC>(scb, a.cb32 + cg * S * KC * D + part * Dp, D);
            cur = cg * parts + part;
        }
        const int64_t ooff = static_cast<int64_t>(a.kv * H + h) * D + part * Dp + dq * kDT;
        for (int64_t j = j0 + threadIdx.x / tpv; j < j1; j += kU * vpi) {
            using Ids = typename std::conditional<S * kBits <= 32, uint32_t, uint64_t>::type;
            Ids ids[kU];
            int q[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int64_t e = start + j + u * vpi;
                if (j + u * vpi < j1) {
                    ids[u] = static_cast<Ids>(load_ids<S, WIDE>(scr + e * R + a.off + h * S));
                    q[u] = __ldg(&a.order[e].x);
                }
            }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                if (j + u * vpi >= j1)
                    break;
                const int64_t o = q[u] * out_vec + ooff;
                if constexpr (kDT == 8) {
                    float4 x, y;
                    sum_stages8<S, KC>(row0, ids[u], 2 * dq + ph, 2 * dq + 1 - ph, x, y);
                    store8(a.out, a.dtype, o, ph ? y : x, ph ? x : y);
                } else {
                    store4(a.out, a.dtype, o, sum_stages4<S, KC>(row0, ids[u], dq));
                }
            }
        }
    }
}

template <int S, int KC>
void *read_gather_kernel(bool wide)
{
    constexpr int bytes = S * (KC == 256 ? 1 : 2);
    if ((bytes == 2 || bytes == 4 || bytes == 8) && wide)
        return reinterpret_cast<void *>(k_read_gather<S, true, KC>);
    return reinterpret_cast<void *>(k_read_gather<S, false, KC>);
}

void *read_gather_kernel_for(int S, bool wide, int KC)
{
    if (KC == 1024)
        return S == 1 ? read_gather_kernel<1, 1024>(wide) : read_gather_kernel<2, 1024>(wide);
    switch (S) {
    case 1: return read_gather_kernel<1, 256>(wide);
    case 2: return read_gather_kernel<2, 256>(wide);
    case 3: return read_gather_kernel<3, 256>(wide);
    case 4: return read_gather_kernel<4, 256>(wide);
    case 5: return read_gather_kernel<5, 256>(wide);
    case 6: return read_gather_kernel<6, 256>(wide);
    case 7: return read_gather_kernel<7, 256>(wide);
    default: return read_gather_kernel<8, 256>(wide);
    }
}

// The layer of request q, or n_layers for an out-of-range request (taken last).
__device__ __forceinline__ int req_layer(const int64_t *req, int64_t q, int64_t n_streams, int64_t n_rec,
                                         int n_layers)
{
    const int64_t st = req[2 * q], rec = req[2 * q + 1];
    return st < 0 || st >= n_streams || rec < 0 || rec >= n_rec ? n_layers : static_cast<int>(st % n_layers);
}

// Counting sort of the requests by layer, step 1: per-layer counts (a
// shared-memory histogram per block, then one global add per layer).
__global__ void __launch_bounds__(256) k_order_count(const int64_t *__restrict__ req, int64_t n_req, int64_t n_streams,
                                                     int64_t n_rec, int n_layers, int *__restrict__ cnt)
{
    extern __shared__ int hist[];
    for (int i = threadIdx.x; i <= n_layers; i += blockDim.x)
        hist[i] = 0;
    __syncthreads();
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < n_req;
         q += static_cast<int64_t>(gridDim.x) * blockDim.x)
        atomicAdd(&hist[req_layer(req, q, n_streams, n_rec, n_layers)], 1);
    __syncthreads();
    for (int i = threadIdx.x; i <= n_layers; i += blockDim.x)
        if (hist[i])
            atomicAdd(&cnt[i], hist[i]);
}

// Step 2: counts -> first slot of each layer (exclusive prefix sum, one thread).
__global__ void k_order_scan(int *cnt, int n_layers)
{
    int sum = 0;
    for (int i = 0; i <= n_layers; ++i) {
        const int c = cnt[i];
        cnt[i] = sum;
        sum += c;
    }
}

// Step 3: each block counts its contiguous share of the requests per layer,
// reserves a run of slots per layer with one global add, and places its
// requests in those runs as (request, stream, record, 0), stream -1 for an
// out-of-range request.  The order inside a layer is arbitrary: every output
// goes to its own request's place.
__global__ void __launch_bounds__(256) k_order_scatter(const int64_t *__restrict__ req, int64_t n_req,
                                                       int64_t n_streams, int64_t n_rec, int n_layers,
                                                       int *__restrict__ slot, int4 *__restrict__ order)
{
    extern __shared__ int sh[];                  // [n_layers + 1] counts, then run starts
    int *cntl = sh, *base = sh + n_layers + 1;
    const int64_t q0 = n_req * blockIdx.x / gridDim.x, q1 = n_req * (blockIdx.x + 1) / gridDim.x;
    for (int i = threadIdx.x; i <= n_layers; i += blockDim.x)
        cntl[i] = 0;
    __syncthreads();
    for (int64_t q = q0 + threadIdx.x; q < q1; q += blockDim.x)
        atomicAdd(&cntl[req_layer(req, q, n_streams, n_rec, n_layers)], 1);
    __syncthreads();
    for (int i = threadIdx.x; i <= n_layers; i += blockDim.x) {
        base[i] = cntl[i] ? atomicAdd(&slot[i], cntl[i]) : 0;
        cntl[i] = 0;
    }
    __syncthreads();
    for (int64_t q = q0 + threadIdx.x; q < q1; q += blockDim.x) {
        const int ly = req_layer(req, q, n_streams, n_rec, n_layers);
        const int pos = base[ly] + atomicAdd(&cntl[ly], 1);
        order[pos] = ly < n_layers ? make_int4(static_cast<int>(q), static_cast<int>(req[2 * q]),
                                               static_cast<int>(req[2 * q + 1]), 0)
                                   : make_int4(static_cast<int>(q), -1, 0, 0);
    }
}

}  // namespace

// Staged reads (decode into a symbol buffer, then the codebook-slice gather)
// pay for loading every slice of the codebooks, so they serve batches of at
// least this many requests per layer; smaller batches read codeword rows from
// L2 one request per warp.
constexpr int64_t kStagedPerLayer = 512;

static bool read_staged(const fkv_ctx *c, int64_t n_req)
{
    return n_req >= kStagedPerLayer * c->Ly;
}

// Ints before the staged reads' symbol buffer: the entries and the layer
// counters, rounded up to 16 bytes.
static int64_t read_scr_ints(const fkv_ctx *c, int64_t n_req)
{
    return (4 * n_req + c->Ly + 1 + 3) & ~int64_t(3);
}

int64_t read_order_ints(const fkv_ctx *c, int64_t n_req)
{
    // 32-bit request, stream and record numbers in the entries; the
    // per-block counts and run starts in 48 KB of shared memory
    if (n_req <= 0 || n_req > 0x7FFFFFFF || 2 * (c->Ly + 1) > 12 * 1024)
        return 0;
    if (!read_staged(c, n_req))
        return 4 * n_req + c->Ly + 1;
    const int64_t R = static_cast<int64_t>(c->H) * (c->cb[0].stages + c->cb[1].stages);
    const int64_t esz = c->KC == 256 ? 1 : 2;
    return read_scr_ints(c, n_req) + (n_req * R * esz + 3) / 4;
}

cudaError_t launch_rvq_decode(const fkv_ctx *c, int kv, const void *sym, int layout, int64_t stream_stride,
                              int64_t n_rec, const fkv_cache *out, int64_t t0, cudaStream_t st)
{
    const fkv_cbset &cb = c->cb[kv];
    GatherArgs a;
    a.sym = sym;
    const int H = c->H, SK = c->cb[0].stages, S = cb.stages;
    if (layout == FKV_SYM_PLANAR) {
        a.il = stream_stride;
        a.ih = n_rec * S;
        a.ir = S;
        a.ioff = kv == 0 ? 0 : static_cast<int64_t>(H) * n_rec * SK;
    } else {
        a.il = stream_stride;
        a.ih = S;
        a.ir = static_cast<int64_t>(H) * (SK + c->cb[1].stages);
        a.ioff = kv == 0 ? 0 : static_cast<int64_t>(H) * SK;
    }
    a.ib = static_cast<int64_t>(c->Ly) * stream_stride;
    a.n_rec = n_rec;
    a.batch = out->batch;
    a.t0 = t0;
    a.n_layers = c->Ly;
    a.n_heads = H;
    a.D = c->D;
    a.S = S;
    a.pooled = c->pooled ? 1 : 0;
    a.cb32 = cb.cb32;
    a.out = out->data;
    a.dtype = out->dtype;
    a.s_layer = out->stride_layer;
    a.s_batch = out->stride_batch;
    a.s_head = out->stride_head;
    a.s_pos = out->stride_pos;
    a.Dp = gather_dp(a.S, c->KC);
    const int parts = c->D / a.Dp;
    a.parts = parts;
    const int64_t nvec = a.batch * n_rec;
    if (nvec <= 0)
        return cudaSuccess;
    const size_t smem = static_cast<size_t>(a.S) * c->KC * a.Dp * 4;
    // one load per vector's index run when every run is aligned to its size
    const int64_t Sv = a.S, esz = c->KC == 256 ? 1 : 2;
    const bool wide = reinterpret_cast<uintptr_t>(sym) % (Sv * esz) == 0 && a.ib % Sv == 0 && a.il % Sv == 0 &&
                      a.ih % Sv == 0 && a.ir % Sv == 0 && a.ioff % Sv == 0;
    const void *kern = gather_kernel_for(a.S, wide, c->KC);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem > 48 * 1024 ? smem : 48 * 1024));
    if (e != cudaSuccess)
        return e;
    // persistent: as many blocks as fit at once, each taking an equal share
    int sms = 0, per_sm = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess)
        return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, smem);
    if (e != cudaSuccess)
        return e;
    const int64_t work = static_cast<int64_t>(c->Ly) * c->H * parts * nvec;
    int64_t blocks = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1);
    if (blocks > work)
        blocks = work;
    void *args[] = {&a};
    e = cudaLaunchKernel(kern, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), args, smem, st);
    if (e != cudaSuccess)
        return e;
    return cudaGetLastError();
}

cudaError_t launch_read_kv(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n_rec,
                           int64_t pt_stride, const int64_t *req, int64_t n_req, void *out,
                           int dtype, int *order, cudaStream_t st)
{
    ReadArgs a;
    a.pts = reinterpret_cast<const double2 *>(pts);
    a.n_streams = n_streams;
    a.n_rec = n_rec;
    a.pt_stride = pt_stride;
    a.req = req;
    a.order = nullptr;
    a.n_req = n_req;
    a.out = out;
    a.dtype = dtype;
    a.n_layers = c->Ly;
    a.n_heads = c->H;
    a.D = c->D;
    a.SK = c->cb[0].stages;
    a.SV = c->cb[1].stages;
    a.R = c->H * (a.SK + a.SV);
    a.N = c->N;
    a.L = c->L;
    a.KC = c->KC;
    a.pooled = c->pooled ? 1 : 0;
    a.cbk = c->cb[0].cb32;
    a.cbv = c->cb[1].cb32;
    a.dec = c->d_dec;
    a.T = c->d_T;
    a.status = c->d_status;
    a.scr = nullptr;
    if (n_req <= 0)
        return cudaSuccess;
    const int esz = c->KC == 256 ? 1 : 2;
    const int smem = read_tables_bytes(a.N, a.L) + kReadWarps * kMaxRecord * esz;
    const void *kern = esz == 1 ? reinterpret_cast<const void *>(k_read_kv<uint8_t>)
                                : reinterpret_cast<const void *>(k_read_kv<uint16_t>);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    // persistent: as many blocks as fit at once, or one per eight requests
    int sms = 0, per_sm = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess)
        return e;
    if (order && n_streams <= 0x7FFFFFFF && n_rec <= 0x7FFFFFFF) {
        // requests grouped by layer: n_req int4 entries, the layer counters after them
        int4 *ent = reinterpret_cast<int4 *>(order);
        int *cnt = order + 4 * n_req;
        e = cudaMemsetAsync(cnt, 0, (c->Ly + 1) * sizeof(int), st);
        if (e != cudaSuccess)
            return e;
        const int64_t need = (n_req + 255) / 256;
        const unsigned g = static_cast<unsigned>(need < 4 * sms ? need : 4 * sms);
        const size_t hsm = (c->Ly + 1) * sizeof(int);
        k_order_count<<<g, 256, hsm, st>>>(req, n_req, n_streams, n_rec, c->Ly, cnt);
        k_order_scan<<<1, 1, 0, st>>>(cnt, c->Ly);
        k_order_scatter<<<g, 256, 2 * hsm, st>>>(req, n_req, n_streams, n_rec, c->Ly, cnt, ent);
        e = cudaGetLastError();
        if (e != cudaSuccess)
            return e;
        a.order = ent;
        if (read_staged(c, n_req))
            a.scr = order + read_scr_ints(c, n_req);
    }
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kReadWarps * 32, smem);
    if (e != cudaSuccess)
        return e;
    int64_t blocks = (n_req + kReadWarps - 1) / kReadWarps;
    const int64_t resident = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1);
    if (blocks > resident)
        blocks = resident;
    void *args[] = {&a};
    if (!a.scr) {
        e = cudaLaunchKernel(kern, dim3(static_cast<unsigned>(blocks)), dim3(kReadWarps * 32), args, smem, st);
        if (e != cudaSuccess)
            return e;
        return cudaGetLastError();
    }
    // staged: the records' symbols (a thread per entry and span covering its record) ...
    {
        const int tsm = read_tables_bytes(a.N, a.L);
        const void *sk = esz == 1 ? reinterpret_cast<const void *>(k_read_syms<uint8_t>)
                                  : reinterpret_cast<const void *>(k_read_syms<uint16_t>);
        e = cudaFuncSetAttribute(sk, cudaFuncAttributeMaxDynamicSharedMemorySize, tsm);
        if (e != cudaSuccess)
            return e;
        int sper = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&sper, sk, 256, tsm);
        if (e != cudaSuccess)
            return e;
        int spr = (a.R + a.L - 1) / a.L + (a.R % a.L ? 1 : 0);
        const int64_t items = n_req * spr;
        int64_t sblocks = static_cast<int64_t>(sms) * (sper > 0 ? sper : 1);
        if (sblocks > (items + 255) / 256)
            sblocks = (items + 255) / 256;
        void *sargs[] = {&a, &spr};
        e = cudaLaunchKernel(sk, dim3(static_cast<unsigned>(sblocks)), dim3(256), sargs, tsm, st);
        if (e != cudaSuccess)
            return e;
    }
    // ... then K and V rebuilt from codebook slices in shared memory
    for (int kv = 0; kv < 2; ++kv) {
        ReadGatherArgs g;
        g.scr = a.scr;
        g.order = a.order;
        g.ends = order + 4 * n_req;
        g.cb32 = c->cb[kv].cb32;
        g.out = out;
        g.dtype = dtype;
        g.n_layers = c->Ly;
        g.n_heads = c->H;
        g.D = c->D;
        g.R = a.R;
        g.off = kv ? c->H * a.SK : 0;
        g.kv = kv;
        g.pooled = a.pooled;
        const int S = c->cb[kv].stages;
        const int Dp = gather_dp(S, c->KC);
        g.parts = c->D / Dp;
        const size_t gsm = static_cast<size_t>(S) * c->KC * Dp * 4;
        const bool wide = a.R % S == 0 && g.off % S == 0;
        const void *gk = read_gather_kernel_for(S, wide, c->KC);
        e = cudaFuncSetAttribute(gk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(gsm > 48 * 1024 ? gsm : 48 * 1024));
        if (e != cudaSuccess)
            return e;
        int gper = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&gper, gk, kThreads, gsm);
        if (e != cudaSuccess)
            return e;
        void *gargs[] = {&g};
        e = cudaLaunchKernel(gk, dim3(static_cast<unsigned>(sms * (gper > 0 ? gper : 1))), dim3(kThreads), gargs, gsm,
                             st);
        if (e != cudaSuccess)
            return e;
    }
    return cudaGetLastError();
}
