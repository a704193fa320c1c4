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
#include <type_traits>

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
    const int *escale_h;   // [Ly*H][S] escale of each head's codebook group
    const __half *cbaug;
    const __half *cb16;    // [G][S][2][KC][64] hi/lo of -2 c 2^-e (64-dim heads)
    int KC;                // codewords per stage: 256 or 1024
    int pooled;            // codebook group = layer (1) or (layer, head) (0)
    void *sym;             // uint8 indices for KC = 256, uint16 for KC = 1024
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

// 2^e as a float for e in [-126, 127] (clamped), built from its exponent bits.
__device__ __forceinline__ float pow2f(int e)
{
    e = e < -126 ? -126 : (e > 127 ? 127 : e);
    return __int_as_float((e + 127) << 23);
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
    const int cg = a.pooled ? l : g;          // codebook group
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
        const int row0 = (cg * S + s) * 2 * kCodes;
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
    const float *cn_g = a.cnorm + static_cast<int64_t>(cg) * S * kCodes;
    cn[tid] = cn_g[tid];
    cn[tid + kThreads] = cn_g[tid + kThreads];
    fence_proxy_async_smem();
    int lo_any = __syncthreads_or(lo_nz);

    uint8_t idx[8];
    const float *cb_g = a.cb32 + static_cast<int64_t>(cg) * S * kCodes * D;
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
        const int eb = a.escale[cg * S + s];
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
        uint8_t *dst = static_cast<uint8_t *>(a.sym) + (b * a.n_layers + l) * a.stream_stride +
                       (a.rec0 + (t - a.t0)) * a.R + a.kv_off + h * S;
        for (int s = 0; s < S; ++s)
            dst[s] = idx[s];
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0)
        tmem_dealloc(tmem, kTmemCols);
}

// ===================================================================
// Persistent, warp-specialised kernel for 64-dimensional heads.
//
// One CTA per SM walks pairs of tiles (2 x 128 vectors of one codebook
// group) through all stages.  Warp 0 streams the stage operands into a double
// buffer (fp16 hi/lo of -2 c' by TMA, the 256 x 16 norm operand by a bulk
// copy); warp 1 issues the MMAs; two 4-warp epilogue groups each own one tile:
// a 128 x 256 fp32 accumulator in tensor memory (2 x 256 of the 512 columns)
// and a hi/lo operand tile of the scaled residual r'.
//
// A (group, stage) is scaled by a power of two 2^-e (max |c'| in [2^3, 2^9),
// usually one e for all stages of a group), and an extra K = 16 MMA against a
// constant operand adds the codeword norms, so
//     acc_j = sum (r'_hi,lo) (-2 c'_hi,lo) + 2^10 sum_3 parts(||c'_j||^2 2^-10)
//           = ||r' - c'_j||^2 - ||r'||^2
// (hi*hi + hi*lo + lo*hi, ~22-bit operands; norms to ~33 bits).  The argmin
// over the 256 columns is exact on the fp32 accumulators: tcgen05.ld.red
// returns the minimum of every 16 columns with the load, which gives the
// best value and its 16-column chunk, and an elementwise minimum across the
// chunks gives its position inside the chunk; an exact tie (the minimum in two
// chunks or two positions) is rescanned column by column.  A row whose scaled
// residual reaches 2^14 (far outside the codebook) is scored exactly in fp32
// from the stage buffer instead.  The fp32 residual r' lives in registers and
// is updated with mixed-precision FMAs straight from the fp16 hi/lo codeword in
// the buffer; the next pair's 16-bit input rows are prefetched into registers
// during the last stage.  Both tiles of a pair share each stage's operands, so
// one tile's epilogue overlaps the other's MMAs.
namespace v2 {
constexpr int kWarps = 10;                   // 0 TMA, 1 MMA, 2..5 and 6..9 epilogue groups
constexpr int kThreads = kWarps * 32;
constexpr int A_TILE = kRows * 128;          // 16 KB: 128 rows x 64 fp16 (128-byte swizzle)
constexpr int A_SLOT = 2 * A_TILE;           // hi + lo
constexpr int A_AUG = kRows * 32;            // 4 KB: 128 rows x 16 fp16 (core-matrix layout), constant
constexpr int B_TILE = kCodes * 128;         // 32 KB
constexpr int B_AUG = kCodes * 32;           // 8 KB
constexpr int B_BUF = 2 * B_TILE + B_AUG;    // 72 KB
constexpr int OFF_A = 0;
constexpr int OFF_AAUG = 2 * A_SLOT;
constexpr int OFF_B = OFF_AAUG + A_AUG;      // 68 KB: 1024-aligned
constexpr int OFF_BAR = OFF_B + 2 * B_BUF;   // b_full[2], b_empty[2], a_ready[2], acc_full[2], drain
constexpr int OFF_SLOT = OFF_BAR + 80;
constexpr int OFF_LO = OFF_SLOT + 16;        // per slot: the pair whose first-stage lo operand is nonzero
constexpr int OFF_ABORT = OFF_LO + 16;
constexpr int END = OFF_ABORT + 16;
constexpr int SMEM = END + 1024;
constexpr float kFastLimit = 16384.0f;       // |r'| below 2^14: fp16 operands in range
}  // namespace v2

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// 1-D bulk copy global -> shared, completion counted on `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// Shared-memory descriptor of a K-major operand in the no-swizzle
// core-matrix layout: 128 B between the two 8x16 B core matrices along K,
// 256 B between 8-row groups.
__device__ __forceinline__ uint64_t sdesc_core16(uint32_t saddr)
{
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
    d |= static_cast<uint64_t>(128 >> 4) << 16;     // leading byte offset: along K
    d |= static_cast<uint64_t>(256 >> 4) << 32;     // stride byte offset: 8-row groups
    d |= static_cast<uint64_t>(1) << 46;            // descriptor version (sm_100 family)
    return d;                                       // swizzle mode 0: none
}

// 16-byte word of row `row`, columns 8h .. 8h+7, of a [rows x 16] operand.
__device__ __forceinline__ uint32_t core16_off(int row, int h)
{
    return static_cast<uint32_t>((row >> 3) * 256 + h * 128 + (row & 7) * 16);
}

__device__ __forceinline__ uint32_t pack_half2(float a, float b)
{
    const __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t *>(&h);
}

__device__ __forceinline__ float min3f(float a, float b, float c)
{
    float d;
    asm volatile("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ float max3f(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// x0 += w.lo / 2, x1 += w.hi / 2 for the two fp16 halves of w, each one
// mixed-precision FMA (exact product, one rounding).
__device__ __forceinline__ void add_half2_halved(uint32_t w, float &x0, float &x1)
{
    asm("{\n\t.reg .b16 l, h, c;\n\t"
        "mov.b32 {l, h}, %2;\n\t"
        "mov.b16 c, 0x3800;\n\t"
        "fma.rn.f32.f16 %0, l, c, %0;\n\t"
        "fma.rn.f32.f16 %1, h, c, %1;\n\t}"
        : "+f"(x0), "+f"(x1)
        : "r"(w));
}

// hi = fp16(a) (packed pair), lo = fp16(a - hi); a - hi is exact in fp32.
__device__ __forceinline__ void split_half2(float a0, float a1, uint32_t &hi, uint32_t &lo)
{
    asm("{\n\t.reg .b16 x, y, m;\n\t.reg .f32 d0, d1;\n\t"
        "cvt.rn.f16x2.f32 %0, %3, %2;\n\t"
        "mov.b32 {x, y}, %0;\n\t"
        "mov.b16 m, 0xBC00;\n\t"
        "fma.rn.f32.f16 d0, x, m, %2;\n\t"
        "fma.rn.f32.f16 d1, y, m, %3;\n\t"
        "cvt.rn.f16x2.f32 %1, d1, d0;\n\t}"
        : "=r"(hi), "=r"(lo)
        : "f"(a0), "f"(a1));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t *r)
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}

// Columns [c, c + 32) of this thread's accumulator row as two 16-column
// chunks a and b, with their minima ra and rb (tcgen05.ld.red), loads and
// wait in one statement.
__device__ __forceinline__ void tmem_red2x16(uint32_t taddr, float *a, float *b, float &ra, float &rb)
{
    asm volatile(
        "tcgen05.ld.red.sync.aligned.32x32b.x16.min.f32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, %32, [%34];\n\t"
        "tcgen05.ld.red.sync.aligned.32x32b.x16.min.f32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, %33, [%34+16];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=f"(a[0]), "=f"(a[1]), "=f"(a[2]), "=f"(a[3]), "=f"(a[4]), "=f"(a[5]), "=f"(a[6]), "=f"(a[7]), "=f"(a[8]), "=f"(a[9]), "=f"(a[10]), "=f"(a[11]), "=f"(a[12]), "=f"(a[13]), "=f"(a[14]), "=f"(a[15]), "=f"(b[0]), "=f"(b[1]), "=f"(b[2]), "=f"(b[3]), "=f"(b[4]), "=f"(b[5]), "=f"(b[6]), "=f"(b[7]), "=f"(b[8]), "=f"(b[9]), "=f"(b[10]), "=f"(b[11]), "=f"(b[12]), "=f"(b[13]), "=f"(b[14]), "=f"(b[15]),
          "=f"(ra), "=f"(rb)
        : "r"(taddr));
}

// Scale the residual row by a power of two.
__device__ __forceinline__ void scale_row(float *r, float f)
{
#pragma unroll
    for (int i = 0; i < 64; ++i)
        r[i] *= f;
}

// Store the hi/lo split of the scaled residual r' into this row of the
// operand tile.  *fast tells whether every |r'| stays below the fast-path
// limit; with NZ the return value tells whether any lo is nonzero.
template <bool NZ>
__device__ __forceinline__ bool write_operands(uint8_t *ahi, uint8_t *alo, int row, const float *r, bool *fast)
{
    uint32_t nz = 0;
    float mx = 0.0f;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        uint4 hv, lv;
        uint32_t *hw = &hv.x, *lw = &lv.x;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float a0 = r[c * 8 + 2 * i], a1 = r[c * 8 + 2 * i + 1];
            split_half2(a0, a1, hw[i], lw[i]);
            mx = max3f(mx, fabsf(a0), fabsf(a1));
            if (NZ)
                nz |= lw[i] & 0x7FFF7FFFu;   // either sign of zero counts as zero
        }
        const uint32_t off = swz(row, c);
        *reinterpret_cast<uint4 *>(ahi + off) = hv;
        *reinterpret_cast<uint4 *>(alo + off) = lv;
    }
    *fast = mx < v2::kFastLimit;
    return nz != 0;
}

template <int ESZ>
__device__ __forceinline__ void unpack_row64(const uint4 *xr, int dtype, float *r)
{
    if (ESZ == 4) {
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            r[4 * c] = __uint_as_float(xr[c].x);
            r[4 * c + 1] = __uint_as_float(xr[c].y);
            r[4 * c + 2] = __uint_as_float(xr[c].z);
            r[4 * c + 3] = __uint_as_float(xr[c].w);
        }
    } else {
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const uint32_t w[4] = {xr[c].x, xr[c].y, xr[c].z, xr[c].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float2 f;
                if (dtype == FKV_F16)
                    f = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
                else
                    f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[i]));
                r[8 * c + 2 * i] = f.x;
                r[8 * c + 2 * i + 1] = f.y;
            }
        }
    }
}

// Exact fp32 scoring of one scaled row against the 256 codewords of a buffer
// (c' = -(hi + lo) / 2), for rows outside the fast path.  Lowest index on ties;
// *dmin receives the best squared distance.
__device__ __forceinline__ int slow_argmin(const float *r, const uint8_t *bb, float *dmin)
{
    float best = INFINITY;
    int bidx = 0;
#pragma unroll 1
    for (int j = 0; j < kCodes; ++j) {
        float d = 0.0f;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const uint32_t off = swz(j, c);
            const uint4 hv = *reinterpret_cast<const uint4 *>(bb + off);
            const uint4 lv = *reinterpret_cast<const uint4 *>(bb + v2::B_TILE + off);
            const __half2 *hh = reinterpret_cast<const __half2 *>(&hv);
            const __half2 *ll = reinterpret_cast<const __half2 *>(&lv);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 h = __half22float2(hh[i]), l = __half22float2(ll[i]);
                const float t0 = r[c * 8 + 2 * i] + 0.5f * (h.x + l.x);
                const float t1 = r[c * 8 + 2 * i + 1] + 0.5f * (h.y + l.y);
                d = fmaf(t0, t0, d);
                d = fmaf(t1, t1, d);
            }
        }
        if (d < best) {
            best = d;
            bidx = j;
        }
    }
    *dmin = best;
    return bidx;
}

// Argmin of one accumulator row (warp-collective: every lane of the warp
// calls it).  Returns bc * 16 + p, where bc is the first 16-column chunk whose
// minimum (from tcgen05.ld.red) equals the row minimum and p the position at
// which the elementwise minimum across chunks equals it.  When the row minimum
// is held by exactly one chunk and one position, that column is the unique
// argmin; otherwise (an exact tie, or no finite value) *amb is set and the
// caller rescans.  *vmin receives the row minimum.
__device__ __forceinline__ int argmin_row(uint32_t trow, bool *amb, float *vmin)
{
    float m[16];
    float best = INFINITY;
    int bc = 0;
    bool tie = false;
#pragma unroll 1
    for (int c = 0; c < kCodes / 16; c += 2) {
        float a[16], b[16], ra, rb;
        tmem_red2x16(trow + c * 16, a, b, ra, rb);
#pragma unroll
        for (int p = 0; p < 16; ++p)
            m[p] = c == 0 ? fminf(a[p], b[p]) : min3f(m[p], a[p], b[p]);
        if (ra < best) {
            best = ra;
            bc = c;
            tie = false;
        } else if (ra == best) {
            tie = true;
        }
        if (rb < best) {
            best = rb;
            bc = c + 1;
            tie = false;
        } else if (rb == best) {
            tie = true;
        }
    }
    uint32_t pm = 0;
#pragma unroll
    for (int p = 0; p < 16; ++p)
        pm |= (m[p] == best ? 1u : 0u) << p;
    *amb = tie || pm == 0 || (pm & (pm - 1)) != 0;
    *vmin = best;
    return bc * 16 + (__ffs(pm) - 1);
}

// Exact argmin of an accumulator row (float compare, lowest index on ties).
__device__ __forceinline__ int exact_argmin_tmem(uint32_t trow)
{
    float best = INFINITY;
    int bidx = 0;
#pragma unroll 1
    for (int ch = 0; ch < kCodes / 16; ++ch) {
        uint32_t acc[16];
        tmem_ld16(trow + ch * 16, acc);
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const float d = __uint_as_float(acc[j]);
            if (d < best) {
                best = d;
                bidx = ch * 16 + j;
            }
        }
    }
    return bidx;
}

// NB = codewords per stage / 256: each stage runs as NB blocks of 256
// codewords through the same buffers, the running argmin carried across the
// blocks (a later block wins only with a strictly smaller score, so ties keep
// the lowest index) and the residual updated once, after the last block, from
// the chosen codeword's global fp16 hi/lo copy (the stage buffer that held it
// may already be reused).
template <int ESZ, int NB>
__global__ void __launch_bounds__(v2::kThreads, 1)
k_rvq64(const __grid_constant__ CUtensorMap tmap, const RvqArgs a, int pairs_per_group, int n_pairs)
{
    using namespace v2;
    using Sym = typename std::conditional<NB == 1, uint8_t, uint16_t>::type;
    constexpr int KC = NB * kCodes;              // codewords per stage
    constexpr int XN = 64 * ESZ / 16;            // 16-byte chunks per input row
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(base);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(base + OFF_ABORT);
    volatile int *lo_stamp = reinterpret_cast<volatile int *>(base + OFF_LO);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // barrier i: 0,1 b_full; 2,3 b_empty; 4,5 a_ready; 6,7 acc_full; 8 drain (MMA completion at exit)
    auto bar = [&](int i) { return sbase + OFF_BAR + 8u * i; };
    if (tid == 0) {
        mbar_init(bar(0), 1);
        mbar_init(bar(1), 1);
        mbar_init(bar(2), 256);
        mbar_init(bar(3), 256);
        mbar_init(bar(4), 128);
        mbar_init(bar(5), 128);
        mbar_init(bar(6), 1);
        mbar_init(bar(7), 1);
        mbar_init(bar(8), 1);
        lo_stamp[0] = 0;
        lo_stamp[1] = 0;
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap);
    }
    // the norm operand of A: columns 0..2 hold 2^10 (times the three parts of
    // ||c'||^2 2^-10 in B), the rest zero
    for (int i = tid; i < kRows; i += v2::kThreads) {
        *reinterpret_cast<uint4 *>(base + OFF_AAUG + core16_off(i, 0)) =
            make_uint4(pack_half2(1024.0f, 1024.0f), pack_half2(1024.0f, 0.0f), 0u, 0u);
        *reinterpret_cast<uint4 *>(base + OFF_AAUG + core16_off(i, 1)) = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();
    if (warp == 1)
        tmem_alloc(sbase + OFF_SLOT, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(base + OFF_SLOT);
    const int S = a.S;
    const int64_t nvec = a.batch * a.n_pos;
    const int tiles = a.tiles_per_group;
    // codebook group of head group g = (layer, head): the layer when pooled
    auto cgroup = [&](int g) { return a.pooled ? g / a.n_heads : g; };

    if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            int it = 0;
            int last[2] = {-1, -1};               // last iteration that loaded each buffer
            for (int p = blockIdx.x; p < n_pairs; p += gridDim.x) {
                const int cg = cgroup(p / pairs_per_group);
                bool ok = true;
                for (int s = 0; s < S && ok; ++s) {
                    for (int u = 0; u < NB; ++u, ++it) {
                        const int bi = it & 1;
                        const uint32_t ph = (it >> 1) & 1;
                        if (!wait_or_abort(bar(2 + bi), ph ^ 1, a.status, abort_flag)) {
                            ok = false;
                            break;
                        }
                        const uint32_t bb = sbase + OFF_B + bi * B_BUF;
                        const int row0 = (cg * S + s) * 2 * KC + u * kCodes;
                        mbar_arrive_expect_tx(bar(bi), 2u * B_TILE + B_AUG);
                        tma_load_2d(bb, &tmap, 0, row0, bar(bi));
                        tma_load_2d(bb + B_TILE, &tmap, 0, row0 + KC, bar(bi));
                        bulk_load(bb + 2 * B_TILE, a.cbaug + (static_cast<int64_t>(cg * S + s) * KC + u * kCodes) * 16,
                                  B_AUG, bar(bi));
                        last[bi] = it;
                    }
                }
                if (!ok)
                    break;
            }
            // no copy may still be landing in shared memory when the CTA exits
            // (after an abort the consumers may not have waited for them)
            for (int bi = 0; bi < 2; ++bi)
                if (last[bi] >= 0)
                    mbar_wait(bar(bi), (last[bi] >> 1) & 1, a.status);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_f32(kRows, kCodes);
            const uint64_t daug = sdesc_core16(sbase + OFF_AAUG);
            int it = 0;
            uint32_t aph[2] = {0, 0};
            int pc = 0;
            bool ok = true;
            for (int p = blockIdx.x; p < n_pairs && ok; p += gridDim.x) {
                ++pc;
                for (int s = 0; s < S && ok; ++s) {
                    for (int u = 0; u < NB && ok; ++u, ++it) {
                        const int bi = it & 1;
                        const uint32_t ph = (it >> 1) & 1;
                        ok = wait_or_abort(bar(bi), ph, a.status, abort_flag);
                        if (!ok)
                            break;
                        const uint32_t bb = sbase + OFF_B + bi * B_BUF;
                        for (int k = 0; k < 2; ++k) {
                            ok = wait_or_abort(bar(4 + k), aph[k], a.status, abort_flag);
                            if (!ok)
                                break;
                            aph[k] ^= 1;
                            tc_fence_after();
                            // the lo operand is nonzero after the first stage; at the
                            // first stage only if a row's input needs it
                            const bool lo = s > 0 || lo_stamp[k] == pc;
                            const uint32_t ab = sbase + OFF_A + k * A_SLOT;
                            const uint32_t acc = tmem + k * 256;
                            // codeword norms first (K = 16, no swizzle), then the split dot products
                            umma_f16(acc, daug, sdesc_core16(bb + 2 * B_TILE), idesc, 0);
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk) {
                                const uint64_t dah = sdesc_sw128(ab + kk * 32);
                                const uint64_t dal = sdesc_sw128(ab + A_TILE + kk * 32);
                                const uint64_t dbh = sdesc_sw128(bb + kk * 32);
                                const uint64_t dbl = sdesc_sw128(bb + B_TILE + kk * 32);
                                umma_f16(acc, dah, dbh, idesc, 1);
                                umma_f16(acc, dah, dbl, idesc, 1);
                                if (lo)
                                    umma_f16(acc, dal, dbh, idesc, 1);
                            }
                            umma_commit(bar(6 + k));
                        }
                    }
                }
            }
            // every MMA has completed before tensor memory is released
            umma_commit(bar(8));
            mbar_wait(bar(8), 0, a.status);
        }
    } else {
        // ---------------------------------------------------- epilogue groups
        const int k = (warp - 2) >> 2;           // tile slot 0 or 1
        const int quad = warp & 3;                // TMEM lane quadrant of this warp
        const int row = quad * 32 + lane;
        const uint32_t trow = tmem + k * 256 + (static_cast<uint32_t>(quad * 32) << 16);
        uint8_t *ahi = base + OFF_A + k * A_SLOT;
        uint8_t *alo = ahi + A_TILE;
        uint4 xr[XN];
        auto row_src = [&](int p, bool *in) -> const uint4 * {
            const int g = p / pairs_per_group, q = p - g * pairs_per_group;
            const int tile = 2 * q + k;
            const int64_t v = static_cast<int64_t>(tile) * kRows + row;
            *in = tile < tiles && v < nvec;
            if (!*in)
                return nullptr;
            const int l = g / a.n_heads, h = g - l * a.n_heads;
            const int64_t b = v / a.n_pos;
            const int64_t t = a.t0 + (v - b * a.n_pos);
            return reinterpret_cast<const uint4 *>(static_cast<const uint8_t *>(a.x) +
                                                   (l * a.s_layer + b * a.s_batch + h * a.s_head + t * a.s_pos) * ESZ);
        };
        auto load_row = [&](int p) {
            bool in;
            const uint4 *src = row_src(p, &in);
            if (in) {
#pragma unroll
                for (int c = 0; c < XN; ++c)
                    xr[c] = __ldg(src + c);
            } else {
#pragma unroll
                for (int c = 0; c < XN; ++c)
                    xr[c] = make_uint4(0, 0, 0, 0);
            }
        };
        int it = 0;
        uint32_t fph = 0;
        int pc = 0;
        if (static_cast<int>(blockIdx.x) < n_pairs)
            load_row(blockIdx.x);
        for (int p = blockIdx.x; p < n_pairs; p += gridDim.x) {
            const bool has_next = p + static_cast<int>(gridDim.x) < n_pairs;
            if (has_next) {
                // pull the next pair's input row into L2 now; it is loaded into
                // registers once this pair's last argmin no longer needs them
                bool in;
                const uint4 *src = row_src(p + gridDim.x, &in);
                if (in) {
#pragma unroll
                    for (int c = 0; c < XN; c += 8)
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(src + c));
                }
            }
            const int g = p / pairs_per_group, q = p - g * pairs_per_group;
            const int l = g / a.n_heads, h = g - l * a.n_heads;
            const int tile = 2 * q + k;
            const int64_t v = static_cast<int64_t>(tile) * kRows + row;
            const bool valid = tile < tiles && v < nvec;
            float r[64];
            unpack_row64<ESZ>(xr, a.dtype, r);
            int e = __ldg(&a.escale_h[g * S]);
            scale_row(r, pow2f(-e));
            bool fast;
            ++pc;
            if (write_operands<true>(ahi, alo, row, r, &fast))
                lo_stamp[k] = pc;
            fence_proxy_async_smem();
            mbar_arrive(bar(4 + k));
            Sym idx[8];
            bool ok = true;
            for (int s = 0; s < S; ++s) {
                const int e_next = s + 1 < S ? __ldg(&a.escale_h[g * S + s + 1]) : e;   // in flight during the waits
                float bv = INFINITY;
                int bidx = 0, bi = 0;
                const uint8_t *bb = nullptr;
                for (int u = 0; u < NB; ++u, ++it) {
                    bi = it & 1;
                    ok = wait_or_abort(bar(6 + k), fph, a.status, abort_flag) &&
                         wait_or_abort(bar(bi), (it >> 1) & 1, a.status, abort_flag);
                    // the tensor-memory loads below are warp-collective: the warp
                    // goes on, or leaves, as one
                    ok = __all_sync(0xFFFFFFFFu, ok);
                    if (!ok)
                        break;
                    fph ^= 1;
                    tc_fence_after();
                    bb = base + OFF_B + bi * B_BUF;
                    __syncwarp();
                    bool amb;
                    float vu;
                    int j = argmin_row(trow, &amb, &vu);
                    if (__any_sync(0xFFFFFFFFu, fast && amb)) {   // warp-collective loads: every lane takes part
                        const int jj = exact_argmin_tmem(trow);
                        if (amb)
                            j = jj;
                    }
                    tc_fence_before();
                    if (!fast)
                        j = slow_argmin(r, bb, &vu);
                    if (NB == 1 || u == 0 || vu < bv) {
                        bv = vu;
                        bidx = u * kCodes + j;
                    }
                    if (u + 1 < NB) {
                        // this block's scores are read: the buffer and the
                        // accumulator slot go back (the operands stay)
                        mbar_arrive(bar(2 + bi));
                        mbar_arrive(bar(4 + k));
                    }
                }
                if (!ok)
                    break;
                idx[s] = static_cast<Sym>(bidx);
                if (s == S - 1 && has_next)
                    load_row(p + gridDim.x);      // r is dead from here: the next input takes its registers
                if (s + 1 < S) {
                    // r' <- r' - c'_bidx = r' + (hi + lo) / 2, the codeword read from the
                    // stage buffer (one block) or from its global copy
                    const uint4 *gh = nullptr;
                    if (NB > 1)
                        gh = reinterpret_cast<const uint4 *>(a.cb16 +
                                                             ((static_cast<int64_t>(cgroup(g) * S + s) * 2) * KC + bidx) * 64);
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        uint4 hv, lv;
                        if (NB == 1) {
                            const uint32_t bo = swz(bidx, c);
                            hv = *reinterpret_cast<const uint4 *>(bb + bo);
                            lv = *reinterpret_cast<const uint4 *>(bb + B_TILE + bo);
                        } else {
                            hv = __ldg(gh + c);
                            lv = __ldg(gh + KC * 8 + c);
                        }
                        const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w};
                        const uint32_t lw[4] = {lv.x, lv.y, lv.z, lv.w};
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            add_half2_halved(hw[i], r[8 * c + 2 * i], r[8 * c + 2 * i + 1]);
                            add_half2_halved(lw[i], r[8 * c + 2 * i], r[8 * c + 2 * i + 1]);
                        }
                    }
                }
                mbar_arrive(bar(2 + bi));         // this thread is done with the stage buffer
                if (s + 1 < S) {
                    if (e_next != e) {            // uniform: one group per CTA at a time
                        scale_row(r, pow2f(e - e_next));
                        e = e_next;
                    }
                    if (!valid) {
#pragma unroll
                        for (int i = 0; i < 64; ++i)
                            r[i] = 0.0f;
                    }
                    write_operands<false>(ahi, alo, row, r, &fast);
                    fence_proxy_async_smem();
                    mbar_arrive(bar(4 + k));
                }
            }
            if (!ok)
                break;
            if (valid) {
                const int64_t b = v / a.n_pos;
                const int64_t t = a.t0 + (v - b * a.n_pos);
                Sym *dst = static_cast<Sym *>(a.sym) + (b * a.n_layers + l) * a.stream_stride +
                           (a.rec0 + (t - a.t0)) * a.R + a.kv_off + h * S;
                for (int s = 0; s < S; ++s)
                    dst[s] = idx[s];
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem, 512);
    }
}

}  // namespace

template <int ESZ, int NB>
cudaError_t launch_rvq64(const CUtensorMap &tmap, const RvqArgs &a, int ppg, int n_pairs, unsigned grid,
                         cudaStream_t st)
{
    cudaError_t e = cudaFuncSetAttribute(k_rvq64<ESZ, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, v2::SMEM);
    if (e != cudaSuccess)
        return e;
    k_rvq64<ESZ, NB><<<grid, v2::kThreads, v2::SMEM, st>>>(tmap, a, ppg, n_pairs);
    return cudaGetLastError();
}

cudaError_t launch_rvq_encode(const fkv_ctx *c, int kv, const fkv_cache *x, int64_t t0, int64_t t1,
                              void *sym, int64_t stream_stride, int64_t rec0, cudaStream_t st)
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
    a.escale_h = cb.escale_h;
    a.cbaug = cb.cbaug;
    a.cb16 = cb.cb16;
    a.KC = c->KC;
    a.pooled = c->pooled ? 1 : 0;
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
        const int64_t ppg = (tiles + 1) / 2;
        const int64_t n_pairs = ppg * c->Ly * c->H;
        if (n_pairs > 0x7FFFFFFF)
            return cudaErrorInvalidConfiguration;
        int sms = 0;
        cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
        if (e != cudaSuccess)
            return e;
        const unsigned grid = static_cast<unsigned>(n_pairs < sms ? n_pairs : sms);
        const int pp = static_cast<int>(ppg), np = static_cast<int>(n_pairs);
        if (c->KC == 1024)
            return x->dtype == FKV_F32 ? launch_rvq64<4, 4>(cb.tmap, a, pp, np, grid, st)
                                       : launch_rvq64<2, 4>(cb.tmap, a, pp, np, grid, st);
        return x->dtype == FKV_F32 ? launch_rvq64<4, 1>(cb.tmap, a, pp, np, grid, st)
                                   : launch_rvq64<2, 1>(cb.tmap, a, pp, np, grid, st);
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
