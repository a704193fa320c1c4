// Per-head residual-VQ assignment on the 5th-generation tensor cores.
//
// Sec. 3 "Setup": each archived head vector is quantised stage by stage to
// the nearest of 256 codewords of its (layer, head, K/V, stage) codebook, the
// residual dropping the chosen codeword after each stage.
//
// One CTA owns a tile of 128 vectors of one codebook group and walks all of
// its stages:
//   * the residual tile lives in shared memory as two fp16 operands, hi and
//     lo (r * 2^-e_row = hi + lo), in the tcgen05 K-major 128-byte-swizzle
//     layout; e_row is a per-row power of two that keeps the row in range;
//   * the stage codebook arrives by TMA as fp16 hi/lo (scaled by 2^-e_stage);
//   * one elected thread issues tcgen05.mma (M = 128, N = 256, K = 16 per
//     instruction) for hi*hi + hi*lo + lo*hi into a 128 x 256 fp32
//     accumulator in tensor memory -- the dot products r . c_j to ~2^-21
//     relative, so the score ||c_j||^2 - 2 r . c_j is certain to well below
//     the 1e-4 ||r||^2 tie band;
//   * the four epilogue warps read their 32 lanes of tensor memory
//     (tcgen05.ld), form the scores, take the running argmin (lowest index on
//     ties), subtract the chosen float32 codeword and re-split the residual
//     into the operand tiles for the next stage.
#include "fkv_internal.h"

using namespace fkvd;

namespace {

constexpr int kRows = 128;          // vectors per tile (MMA M)
constexpr int kCodes = 256;         // codewords per stage (MMA N)
constexpr int kThreads = 128;       // 4 warps: one TMEM lane quadrant each
constexpr uint32_t kTmemCols = 256; // fp32 accumulator columns

struct RvqArgs {
    const void *x;
    int dtype;
    int64_t batch, n_pos, t0;
    int64_t s_layer, s_batch, s_head, s_pos;
    int n_layers, n_heads, S;
    const float *cb32;
    const float *cnorm;
    const int *escale;
    uint8_t *sym;
    int64_t stream_stride, rec0;
    int R, kv_off;
    int tiles_per_group;
    unsigned *status;
};

template <int D>
struct Layout {
    static constexpr int KB = D / 64;                 // 64-element K blocks
    static constexpr int A_BYTES = KB * kRows * 128;  // one of hi / lo
    static constexpr int B_BYTES = KB * kCodes * 128;
    static constexpr int AHI = 0;
    static constexpr int ALO = A_BYTES;
    static constexpr int BHI = 2 * A_BYTES;
    static constexpr int BLO = 2 * A_BYTES + B_BYTES;
    static constexpr int CN = 2 * A_BYTES + 2 * B_BYTES;   // 256 float
    static constexpr int BAR = CN + kCodes * 4;            // 2 mbarriers
    static constexpr int SLOT = BAR + 16;                  // tmem address
    static constexpr int FLAG = SLOT + 16;                 // abort flag
    static constexpr int END = FLAG + 16;
    static constexpr int SMEM = END + 1024;                // + alignment slack
};

// Byte offset of 16-byte chunk `kk` (0..7) of row `row` inside one
// 128-row-per-atom K block in the 128-byte swizzle layout.
__device__ __forceinline__ uint32_t swz(int row, int kk)
{
    return static_cast<uint32_t>((row >> 3) * 1024 + (row & 7) * 128 + ((kk ^ (row & 7)) << 4));
}

// Eight consecutive elements of a head vector as float.
__device__ __forceinline__ void load8(const uint8_t *p, int dtype, float *o)
{
    if (dtype == FKV_F32) {
        const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
        const float4 b = __ldg(reinterpret_cast<const float4 *>(p + 16));
        o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
        o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
    } else {
        const uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f;
            if (dtype == FKV_F16)
                f = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
            else
                f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[i]));
            o[2 * i] = f.x;
            o[2 * i + 1] = f.y;
        }
    }
}

// Power-of-two exponent e such that m * 2^-e lies in [2^14, 2^15) (0 for m = 0).
__device__ __forceinline__ int row_exp(float m)
{
    if (!(m > 0.0f))
        return 0;
    int E;
    frexpf(m, &E);      // m = f * 2^E, f in [0.5, 1)
    return E - 15;
}

// Split 8 scaled values into fp16 hi and lo and store them as chunk kk of
// K block kb of this row's operand tiles.  Returns whether any lo is nonzero.
__device__ __forceinline__ bool store_split8(uint8_t *ahi, uint8_t *alo, int row, int chunk,
                                             const float *v)
{
    __align__(16) __half hi[8];
    __align__(16) __half lo[8];
    bool nz = false;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        hi[i] = __float2half_rn(v[i]);
        lo[i] = __float2half_rn(v[i] - __half2float(hi[i]));
        nz |= __half2float(lo[i]) != 0.0f;
    }
    const int kb = chunk >> 3, kk = chunk & 7;
    const uint32_t off = static_cast<uint32_t>(kb * kRows * 128) + swz(row, kk);
    *reinterpret_cast<uint4 *>(ahi + off) = *reinterpret_cast<const uint4 *>(hi);
    *reinterpret_cast<uint4 *>(alo + off) = *reinterpret_cast<const uint4 *>(lo);
    return nz;
}

// hi + lo of chunk `chunk` of this row, unscaled by 2^e.
__device__ __forceinline__ void load_split8(const uint8_t *ahi, const uint8_t *alo, int row, int chunk,
                                            int e, float *o)
{
    const int kb = chunk >> 3, kk = chunk & 7;
    const uint32_t off = static_cast<uint32_t>(kb * kRows * 128) + swz(row, kk);
    const uint4 h = *reinterpret_cast<const uint4 *>(ahi + off);
    const uint4 l = *reinterpret_cast<const uint4 *>(alo + off);
    const __half *hh = reinterpret_cast<const __half *>(&h);
    const __half *ll = reinterpret_cast<const __half *>(&l);
#pragma unroll
    for (int i = 0; i < 8; ++i)
        o[i] = ldexpf(__half2float(hh[i]) + __half2float(ll[i]), e);
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t *r)
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Bounded wait that also gives up once another thread has flagged an abort.
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, unsigned *status,
                                              volatile int *abort_flag)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity))
            return true;
        if (*abort_flag)
            return false;
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
            atomicOr(status, FKV_ST_TIMEOUT);
            *abort_flag = 1;
            return false;
        }
    }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
k_rvq(const __grid_constant__ CUtensorMap tmap, const RvqArgs a)
{
    using Lay = Layout<D>;
    constexpr int CHUNKS = D / 8;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *ahi = base + Lay::AHI;
    uint8_t *alo = base + Lay::ALO;
    float *cn = reinterpret_cast<float *>(base + Lay::CN);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(base + Lay::FLAG);
    const uint32_t sbase = smem_u32(base);
    const uint32_t bar_b = sbase + Lay::BAR;
    const uint32_t bar_mma = sbase + Lay::BAR + 8;

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int g = blockIdx.x / a.tiles_per_group;
    const int tile = blockIdx.x % a.tiles_per_group;
    const int l = g / a.n_heads, h = g % a.n_heads;
    const int S = a.S;
    const int64_t nvec = a.batch * a.n_pos;
    const int64_t v = static_cast<int64_t>(tile) * kRows + tid;
    const bool valid = v < nvec;
    const int64_t b = valid ? v / a.n_pos : 0;
    const int64_t t = valid ? a.t0 + (v - b * a.n_pos) : 0;

    if (tid == 0) {
        mbar_init(bar_b, 1);
        mbar_init(bar_mma, 1);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap);
    }
    if (warp == 0)
        tmem_alloc(sbase + Lay::SLOT, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(base + Lay::SLOT);

    auto issue_codebook = [&](int s) {
        const int row0 = (g * S + s) * 2 * kCodes;
        mbar_arrive_expect_tx(bar_b, 2u * Lay::KB * kCodes * 128u);
#pragma unroll
        for (int kb = 0; kb < Lay::KB; ++kb) {
            tma_load_2d(sbase + Lay::BHI + kb * kCodes * 128, &tmap, kb * 64, row0, bar_b);
            tma_load_2d(sbase + Lay::BLO + kb * kCodes * 128, &tmap, kb * 64, row0 + kCodes, bar_b);
        }
    };
    if (tid == 0)
        issue_codebook(0);

    // Stage-0 residual = the input vector, split into the operand tiles.
    const uint8_t *xr = nullptr;
    const int esz = a.dtype == FKV_F32 ? 4 : 2;
    if (valid)
        xr = static_cast<const uint8_t *>(a.x) +
             (l * a.s_layer + b * a.s_batch + h * a.s_head + t * a.s_pos) * esz;
    float rmax = 0.0f;
    if (valid) {
        for (int c = 0; c < CHUNKS; ++c) {
            float f[8];
            load8(xr + c * 8 * esz, a.dtype, f);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                rmax = fmaxf(rmax, fabsf(f[i]));
        }
    }
    int ea = row_exp(rmax);
    bool lo_nz = false;
    for (int c = 0; c < CHUNKS; ++c) {
        float f[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        if (valid) {
            load8(xr + c * 8 * esz, a.dtype, f);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                f[i] = ldexpf(f[i], -ea);
        }
        lo_nz |= store_split8(ahi, alo, tid, c, f);
    }
    const float *cn_g = a.cnorm + static_cast<int64_t>(g) * S * kCodes;
    cn[tid] = cn_g[tid];
    cn[tid + kThreads] = cn_g[tid + kThreads];
    fence_proxy_async_smem();
    int lo_any = __syncthreads_or(lo_nz);

    uint8_t idx[8];
    const float *cb_g = a.cb32 + static_cast<int64_t>(g) * S * kCodes * D;
    const uint32_t idesc = idesc_f16_f32(kRows, kCodes);

    for (int s = 0; s < S; ++s) {
        // --- MMA: acc[row][j] = sum_k (hi*hi + hi*lo + lo*hi), all K blocks
        if (tid == 0) {
            if (wait_or_abort(bar_b, s & 1, a.status, abort_flag)) {
                tc_fence_after();
                uint32_t accum = 0;
#pragma unroll
                for (int kb = 0; kb < Lay::KB; ++kb) {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint32_t ka = kb * kRows * 128 + k * 32;
                        const uint32_t kbb = kb * kCodes * 128 + k * 32;
                        const uint64_t dah = sdesc_sw128(sbase + Lay::AHI + ka);
                        const uint64_t dal = sdesc_sw128(sbase + Lay::ALO + ka);
                        const uint64_t dbh = sdesc_sw128(sbase + Lay::BHI + kbb);
                        const uint64_t dbl = sdesc_sw128(sbase + Lay::BLO + kbb);
                        umma_f16(tmem, dah, dbh, idesc, accum);
                        accum = 1;
                        umma_f16(tmem, dah, dbl, idesc, 1);
                        if (lo_any)
                            umma_f16(tmem, dal, dbh, idesc, 1);
                    }
                }
                umma_commit(bar_mma);
            }
        }
        const bool ok = wait_or_abort(bar_mma, s & 1, a.status, abort_flag);
        if (!__syncthreads_and(ok))
            break;
        tc_fence_after();

        // --- epilogue: scores ||c||^2 - 2 r.c, argmin over this row's 256 columns
        const int eb = a.escale[g * S + s];
        const float sc = -ldexpf(1.0f, ea + eb + 1);
        float best = INFINITY;
        int bi = 0;
        const uint32_t trow = tmem + (static_cast<uint32_t>(warp * 32) << 16);
#pragma unroll 1
        for (int ch = 0; ch < kCodes / 32; ++ch) {
            uint32_t r[32];
            tmem_ld32(trow + ch * 32, r);
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const float score = fmaf(sc, __uint_as_float(r[j]), cn[ch * 32 + j]);
                if (score < best) {
                    best = score;
                    bi = ch * 32 + j;
                }
            }
        }
        idx[s] = static_cast<uint8_t>(bi);
        tc_fence_before();
        __syncthreads();   // TMEM read, operand tiles and codebook buffers free

        if (s + 1 < S) {
            if (tid == 0)
                issue_codebook(s + 1);
            // residual update: r <- r - C_s[bi], re-split with a fresh row exponent
            const float *crow = cb_g + (static_cast<int64_t>(s) * kCodes + bi) * D;
            float m2 = 0.0f;
            if (valid) {
                for (int c = 0; c < CHUNKS; ++c) {
                    float f[8];
                    load_split8(ahi, alo, tid, c, ea, f);
                    const float4 c0 = __ldg(reinterpret_cast<const float4 *>(crow + c * 8));
                    const float4 c1 = __ldg(reinterpret_cast<const float4 *>(crow + c * 8 + 4));
                    const float cc[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        m2 = fmaxf(m2, fabsf(f[i] - cc[i]));
                }
            }
            const int ea2 = row_exp(m2);
            lo_nz = false;
            for (int c = 0; c < CHUNKS; ++c) {
                float f[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                if (valid) {
                    load_split8(ahi, alo, tid, c, ea, f);
                    const float4 c0 = __ldg(reinterpret_cast<const float4 *>(crow + c * 8));
                    const float4 c1 = __ldg(reinterpret_cast<const float4 *>(crow + c * 8 + 4));
                    const float cc[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        f[i] = ldexpf(f[i] - cc[i], -ea2);
                }
                lo_nz |= store_split8(ahi, alo, tid, c, f);
            }
            ea = ea2;
            cn[tid] = cn_g[(s + 1) * kCodes + tid];
            cn[tid + kThreads] = cn_g[(s + 1) * kCodes + tid + kThreads];
            fence_proxy_async_smem();
            lo_any = __syncthreads_or(lo_nz);
        }
    }

    if (valid && !*abort_flag) {
        uint8_t *dst = a.sym + (b * a.n_layers + l) * a.stream_stride +
                       (a.rec0 + (t - a.t0)) * a.R + a.kv_off + h * S;
        for (int s = 0; s < S; ++s)
            dst[s] = idx[s];
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0)
        tmem_dealloc(tmem, kTmemCols);
}

}  // namespace

cudaError_t launch_rvq_encode(const fkv_ctx *c, int kv, const fkv_cache *x, int64_t t0, int64_t t1,
                              uint8_t *sym, int64_t stream_stride, int64_t rec0, cudaStream_t st)
{
    const fkv_cbset &cb = c->cb[kv];
    RvqArgs a;
    a.x = x->data;
    a.dtype = x->dtype;
    a.batch = x->batch;
    a.n_pos = t1 - t0;
    a.t0 = t0;
    a.s_layer = x->stride_layer;
    a.s_batch = x->stride_batch;
    a.s_head = x->stride_head;
    a.s_pos = x->stride_pos;
    a.n_layers = c->Ly;
    a.n_heads = c->H;
    a.S = cb.stages;
    a.cb32 = cb.cb32;
    a.cnorm = cb.cnorm;
    a.escale = cb.escale;
    a.sym = sym;
    a.stream_stride = stream_stride;
    a.rec0 = rec0;
    a.R = c->H * (c->cb[0].stages + c->cb[1].stages);
    a.kv_off = kv == 0 ? 0 : c->H * c->cb[0].stages;
    a.status = c->d_status;
    const int64_t nvec = a.batch * a.n_pos;
    if (nvec <= 0)
        return cudaSuccess;
    const int64_t tiles = (nvec + kRows - 1) / kRows;
    const int64_t blocks = tiles * c->Ly * c->H;
    if (tiles > 0x7FFFFFFF || blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    a.tiles_per_group = static_cast<int>(tiles);
    if (c->D == 64) {
        static bool attr = false;
        if (!attr) {
            cudaError_t e = cudaFuncSetAttribute(k_rvq<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 Layout<64>::SMEM);
            if (e != cudaSuccess)
                return e;
            attr = true;
        }
        k_rvq<64><<<static_cast<unsigned>(blocks), kThreads, Layout<64>::SMEM, st>>>(cb.tmap, a);
    } else {
        static bool attr = false;
        if (!attr) {
            cudaError_t e = cudaFuncSetAttribute(k_rvq<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 Layout<128>::SMEM);
            if (e != cudaSuccess)
                return e;
            attr = true;
        }
        k_rvq<128><<<static_cast<unsigned>(blocks), kThreads, Layout<128>::SMEM, st>>>(cb.tmap, a);
    }
    return cudaGetLastError();
}
