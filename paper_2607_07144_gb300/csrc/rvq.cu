// Residual-VQ assignment on the 5th-generation tensor cores.
//
// Sec. 3 "Setup": each archived head vector is quantised stage by stage to
// the nearest codeword of its (layer, head or pooled layer, K/V, stage)
// codebook, the residual dropping the chosen codeword after each stage.
//
// Two persistent, warp-specialised kernels, one CTA per SM: k_rvq64 for
// 64-dimensional heads (256 or 1024 codewords per stage) and k_rvq128 for
// 128-dimensional heads (256).  Warp 0 streams the stage codebook by TMA, warp
// 1 issues tcgen05.mma (M = 128, N = 256, K = 16) into fp32 accumulators in
// tensor memory, and two 4-warp epilogue groups each walk one 128-vector tile
// through the stages: exact argmin read out of tensor memory with
// tcgen05.ld.red, then the residual update in the fp16 hi/lo operand tiles.
#include <type_traits>

#include "fkv_internal.h"

using namespace fkvd;

namespace {

constexpr int kRows = 128;          // vectors per tile (MMA M)
constexpr int kCodes = 256;         // codewords per block (MMA N)

struct RvqArgs {
    const void *x;
    int dtype;
    int64_t batch, n_pos, t0;
    int64_t s_layer, s_batch, s_head, s_pos;
    int n_layers, n_heads, S;
    const float *cb32;
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

// Byte offset of 16-byte chunk `kk` (0..7) of row `row` inside one
// 128-row-per-atom K block in the 128-byte swizzle layout.
__device__ __forceinline__ uint32_t swz(int row, int kk)
{
    return static_cast<uint32_t>((row >> 3) * 1024 + (row & 7) * 128 + ((kk ^ (row & 7)) << 4));
}

// 2^e as a float for e in [-126, 127] (clamped), built from its exponent bits.
__device__ __forceinline__ float pow2f(int e)
{
    e = e < -126 ? -126 : (e > 127 ? 127 : e);
    return __int_as_float((e + 127) << 23);
}

// Bounded wait that also gives up once another thread has flagged an abort.
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, unsigned *status,
                                              volatile int *abort_flag, uint64_t limit_ns = kWaitLimitNs)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity))
            return true;
        if (*abort_flag)
            return false;
        if (globaltimer_ns() - t0 > limit_ns) {
            atomicOr(status, FKV_ST_TIMEOUT);
            *abort_flag = 1;
            return false;
        }
    }
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
// usually one e for all stages of a group) and a row by a further 2^-er,
// er >= 0 chosen when its pair starts so that the row's operand
// t = r 2^-(e + er) starts below 2^12; an extra K = 16 MMA against the row's
// norm operand (2^(10 - er) in columns 0..2) adds the codeword norms, so
//     acc_j = sum (t_hi,lo) (-2 c'_hi,lo) + 2^(10-er) sum_3 parts(||c'_j||^2 2^-10)
//           = 2^-er (||r' - c'_j||^2 - ||r'||^2)
// (hi*hi + hi*lo + lo*hi, ~22-bit operands; norms to ~33 bits), whose argmin
// over j is the nearest codeword for any input magnitude.  The argmin over
// the 256 columns is exact on the fp32 accumulators: tcgen05.ld.red returns
// the minimum of every 16 columns with the load (four loads in flight per
// wait), which gives the best value and its 16-column chunk, and an
// elementwise minimum across the chunks gives its position inside the chunk;
// an exact tie (the minimum in two chunks or two positions) is rescanned
// column by column.  The residual lives only in the operand tiles: each stage
// adds the chosen codeword's fp16 hi/lo halves (from the stage buffer) to
// hi + lo (exact in fp32) and splits the sum again, so |t| stays below
// 2^12 + S 2^9 < 2^14 and fp16 never overflows; a change of the stage scale
// e re-derives er.  The next pair's input rows are loaded into registers
// during the last stage.  Both tiles of a pair share each stage's operands, so
// one tile's epilogue overlaps the other's MMAs.
namespace v2 {
constexpr int kWarps = 10;                   // 0 TMA, 1 MMA, 2..5 and 6..9 epilogue groups
constexpr int kThreads = kWarps * 32;
constexpr int A_TILE = kRows * 128;          // 16 KB: 128 rows x 64 fp16 (128-byte swizzle)
constexpr int A_SLOT = 2 * A_TILE;           // hi + lo
constexpr int A_AUG = kRows * 32;            // 4 KB per slot: 128 rows x 16 fp16 (core-matrix layout)
constexpr int B_TILE = kCodes * 128;         // 32 KB
constexpr int B_AUG = kCodes * 32;           // 8 KB
constexpr int B_BUF = 2 * B_TILE + B_AUG;    // 72 KB
constexpr int OFF_A = 0;
constexpr int OFF_AAUG = 2 * A_SLOT;
constexpr int OFF_B = OFF_AAUG + 2 * A_AUG;  // 72 KB: 1024-aligned
constexpr int OFF_BAR = OFF_B + 2 * B_BUF;   // b_full[2], b_empty[2], a_ready[2], acc_full[2], drain
constexpr int OFF_SLOT = OFF_BAR + 80;
constexpr int OFF_LO = OFF_SLOT + 16;        // per slot: the pair whose first-stage lo operand is nonzero
constexpr int OFF_ABORT = OFF_LO + 16;
constexpr int END = OFF_ABORT + 16;
constexpr int SMEM = END + 1024;
constexpr int kRowLog = 12;                  // a row's operand starts below 2^12
constexpr int kAugMaxShift = 34;             // 2^(10 - er) stays an fp16 (2^-24 subnormal at most)
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

// Columns [c, c + 64) of this thread's accumulator row as four 16-column
// chunks with their minima (tcgen05.ld.red), all four loads in flight before
// the one wait.
__device__ __forceinline__ void tmem_red4x16(uint32_t taddr, float *a, float *b, float *c, float *d, float &ra,
                                             float &rb, float &rc, float &rd)
{
    asm volatile(
        "tcgen05.ld.red.sync.aligned.32x32b.x16.min.f32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, %64, [%68+0];\n\t"
        "tcgen05.ld.red.sync.aligned.32x32b.x16.min.f32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, %65, [%68+16];\n\t"
        "tcgen05.ld.red.sync.aligned.32x32b.x16.min.f32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47}, %66, [%68+32];\n\t"
        "tcgen05.ld.red.sync.aligned.32x32b.x16.min.f32 {%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, %67, [%68+48];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=f"(a[0]), "=f"(a[1]), "=f"(a[2]), "=f"(a[3]), "=f"(a[4]), "=f"(a[5]), "=f"(a[6]), "=f"(a[7]), "=f"(a[8]), "=f"(a[9]), "=f"(a[10]), "=f"(a[11]), "=f"(a[12]), "=f"(a[13]), "=f"(a[14]), "=f"(a[15]), "=f"(b[0]), "=f"(b[1]), "=f"(b[2]), "=f"(b[3]), "=f"(b[4]), "=f"(b[5]), "=f"(b[6]), "=f"(b[7]), "=f"(b[8]), "=f"(b[9]), "=f"(b[10]), "=f"(b[11]), "=f"(b[12]), "=f"(b[13]), "=f"(b[14]), "=f"(b[15]), "=f"(c[0]), "=f"(c[1]), "=f"(c[2]), "=f"(c[3]), "=f"(c[4]), "=f"(c[5]), "=f"(c[6]), "=f"(c[7]), "=f"(c[8]), "=f"(c[9]), "=f"(c[10]), "=f"(c[11]), "=f"(c[12]), "=f"(c[13]), "=f"(c[14]), "=f"(c[15]), "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3]), "=f"(d[4]), "=f"(d[5]), "=f"(d[6]), "=f"(d[7]), "=f"(d[8]), "=f"(d[9]), "=f"(d[10]), "=f"(d[11]), "=f"(d[12]), "=f"(d[13]), "=f"(d[14]), "=f"(d[15]), "=f"(ra), "=f"(rb), "=f"(rc), "=f"(rd)
        : "r"(taddr));
}

// Row shift er >= 0 that brings a row of magnitude m below 2^12 (0 when it
// already is, or when m is not a number).
__device__ __forceinline__ int row_shift(float m)
{
    if (!(m >= 4096.0f))
        return 0;
    if (isinf(m))
        return 116;
    int E;
    frexpf(m, &E);                         // m < 2^E
    return E - v2::kRowLog;
}

// The norm operand's row: columns 0..2 hold 2^(10 - er) (times the three
// parts of ||c'||^2 2^-10 in B), the rest zero; far-out rows (er > 34), whose
// norm term is below the accumulator's resolution, hold zero.
__device__ __forceinline__ void write_aug_row(uint8_t *aaug, int row, int er)
{
    const float s = er <= v2::kAugMaxShift ? ldexpf(1024.0f, -er) : 0.0f;
    *reinterpret_cast<uint4 *>(aaug + core16_off(row, 0)) =
        make_uint4(pack_half2(s, s), pack_half2(s, 0.0f), 0u, 0u);
    *reinterpret_cast<uint4 *>(aaug + core16_off(row, 1)) = make_uint4(0u, 0u, 0u, 0u);
}

// Store 8 values as chunk c of this row's hi/lo operand tiles; returns the
// nonzero bits of the lo halves.
__device__ __forceinline__ uint32_t store_chunk(uint8_t *ahi, uint8_t *alo, int row, int c, const float *v)
{
    uint4 hv, lv;
    uint32_t *hw = &hv.x, *lw = &lv.x;
    uint32_t nz = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        split_half2(v[2 * i], v[2 * i + 1], hw[i], lw[i]);
        nz |= lw[i] & 0x7FFF7FFFu;       // either sign of zero counts as zero
    }
    const uint32_t off = swz(row, c);
    *reinterpret_cast<uint4 *>(ahi + off) = hv;
    *reinterpret_cast<uint4 *>(alo + off) = lv;
    return nz;
}

// hi + lo of 16-bit halves as float32, exact (lo lies at least 11 bits below
// hi): one conversion and one mixed-precision multiply-add per element.
__device__ __forceinline__ void join_half2(uint32_t hw, uint32_t lw, float &v0, float &v1)
{
    asm("{\n\t.reg .b16 h0, h1, l0, l1, one;\n\t"
        "mov.b32 {h0, h1}, %2;\n\t"
        "mov.b32 {l0, l1}, %3;\n\t"
        "mov.b16 one, 0x3C00;\n\t"
        "cvt.f32.f16 %0, l0;\n\t"
        "cvt.f32.f16 %1, l1;\n\t"
        "fma.rn.f32.f16 %0, h0, one, %0;\n\t"
        "fma.rn.f32.f16 %1, h1, one, %1;\n\t}"
        : "=f"(v0), "=f"(v1)
        : "r"(hw), "r"(lw));
}

// Chunk c of this row's operand as 8 floats hi + lo (exact).
__device__ __forceinline__ void load_chunk(const uint8_t *ahi, const uint8_t *alo, int row, int c, float *v)
{
    const uint32_t off = swz(row, c);
    const uint4 hv = *reinterpret_cast<const uint4 *>(ahi + off);
    const uint4 lv = *reinterpret_cast<const uint4 *>(alo + off);
    join_half2(hv.x, lv.x, v[0], v[1]);
    join_half2(hv.y, lv.y, v[2], v[3]);
    join_half2(hv.z, lv.z, v[4], v[5]);
    join_half2(hv.w, lv.w, v[6], v[7]);
}

// v += (hi + lo) f for the 8 codeword halves of chunk hv/lv (hi + lo exact in
// fp32, one rounding per element).
__device__ __forceinline__ void add_codeword(uint4 hv, uint4 lv, float f, float *v)
{
    const uint32_t hw[4] = {hv.x, hv.y, hv.z, hv.w};
    const uint32_t lw[4] = {lv.x, lv.y, lv.z, lv.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float c0, c1;
        join_half2(hw[i], lw[i], c0, c1);
        v[2 * i] = fmaf(c0, f, v[2 * i]);
        v[2 * i + 1] = fmaf(c1, f, v[2 * i + 1]);
    }
}

// Chunk c of this row's operand plus f times 8 float32 codeword elements:
// v = (hi + lo) + c f, the hi + lo sum exact, then one rounding in the final
// multiply-add.
__device__ __forceinline__ void load_add_chunk(const uint8_t *ahi, const uint8_t *alo, int row, int c, float4 c0,
                                               float4 c1, float f, float *v)
{
    load_chunk(ahi, alo, row, c, v);
    const float cw[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
    for (int i = 0; i < 8; ++i)
        v[i] = fmaf(cw[i], f, v[i]);
}

// t <- t + c f for the 32 rows of one TMEM lane quadrant and one K block,
// the warp taking two rows at a time: half-warp h holds row 2p + h, its lane
// i (0..15) dimensions 4i .. 4i+3 of the block, so a row's codeword half
// (256 bytes of float32) is one 16-byte load per lane over two whole lines,
// and its operand words one conflict-free 128-byte access per half.  (Row
// per lane, each load would touch 32 lines for 16 bytes of each.)  bidx and
// f are this lane's own row's chosen codeword and factor, broadcast row by
// row (f is passed as uniform, UF, when every row's is the same); cbk points
// at the K block's first element of codeword 0 of the stage codebook.  Same
// arithmetic as load_add_chunk and store_chunk: hi + lo exact, one rounding
// in the multiply-add.  Software-pipelined over batches of 8 rows: the next
// batch's codeword loads are in flight while one batch is updated.
template <bool UF>
__device__ __forceinline__ void update_rows_t(uint8_t *ahi, uint8_t *alo, int quad, const float *cbk, int bidx,
                                              float f)
{
    const int lane = threadIdx.x & 31;
    const int hs = lane >> 4, li = lane & 15;
    const uint32_t cw = static_cast<uint32_t>(li >> 1), wo = static_cast<uint32_t>((li & 1) << 3);
    const float4 *cl = reinterpret_cast<const float4 *>(cbk) + li;
    uint8_t *qhi = ahi + quad * 32 * 128, *qlo = alo + quad * 32 * 128;
    float4 cv[2][4];
    float fm[2][4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int m = 2 * j + hs;
        fm[0][j] = UF ? f : __shfl_sync(0xFFFFFFFFu, f, m);
        cv[0][j] = __ldg(cl + __shfl_sync(0xFFFFFFFFu, bidx, m) * 32);
    }
#pragma unroll
    for (int b = 0; b < 4; ++b) {
        const int cur = b & 1, nxt = cur ^ 1;
        if (b < 3) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int m = 8 * (b + 1) + 2 * j + hs;
                fm[nxt][j] = UF ? f : __shfl_sync(0xFFFFFFFFu, f, m);
                cv[nxt][j] = __ldg(cl + __shfl_sync(0xFFFFFFFFu, bidx, m) * 32);
            }
        }
        uint2 hv[4], lv[4];
        uint32_t off[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int r7 = 2 * j + hs;                                    // row & 7
            off[j] = static_cast<uint32_t>((8 * b + r7) * 128) + ((cw ^ static_cast<uint32_t>(r7)) << 4) + wo;   // swz
            hv[j] = *reinterpret_cast<const uint2 *>(qhi + off[j]);
            lv[j] = *reinterpret_cast<const uint2 *>(qlo + off[j]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            float v0, v1, v2, v3;
            join_half2(hv[j].x, lv[j].x, v0, v1);
            join_half2(hv[j].y, lv[j].y, v2, v3);
            v0 = fmaf(cv[cur][j].x, fm[cur][j], v0);
            v1 = fmaf(cv[cur][j].y, fm[cur][j], v1);
            v2 = fmaf(cv[cur][j].z, fm[cur][j], v2);
            v3 = fmaf(cv[cur][j].w, fm[cur][j], v3);
            uint2 h, l;
            split_half2(v0, v1, h.x, l.x);
            split_half2(v2, v3, h.y, l.y);
            *reinterpret_cast<uint2 *>(qhi + off[j]) = h;
            *reinterpret_cast<uint2 *>(qlo + off[j]) = l;
        }
    }
}

// Eight consecutive input elements (chunk c of the row) as floats.
template <int ESZ>
__device__ __forceinline__ void unpack8(const uint4 *xr, int dtype, int c, float *v)
{
    if (ESZ == 4) {
        const uint4 a = xr[2 * c], b = xr[2 * c + 1];
        v[0] = __uint_as_float(a.x); v[1] = __uint_as_float(a.y);
        v[2] = __uint_as_float(a.z); v[3] = __uint_as_float(a.w);
        v[4] = __uint_as_float(b.x); v[5] = __uint_as_float(b.y);
        v[6] = __uint_as_float(b.z); v[7] = __uint_as_float(b.w);
    } else {
        const uint32_t w[4] = {xr[c].x, xr[c].y, xr[c].z, xr[c].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f;
            if (dtype == FKV_F16)
                f = __half22float2(*reinterpret_cast<const __half2 *>(&w[i]));
            else
                f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&w[i]));
            v[2 * i] = f.x;
            v[2 * i + 1] = f.y;
        }
    }
}

// Argmin of one accumulator row as argmin_row, reading four 16-column chunks
// per tensor-memory wait.
__device__ __forceinline__ int argmin_row4(uint32_t trow, bool *amb, float *vmin)
{
    float m[16];
    float best = INFINITY;
    int bc = 0;
    bool tie = false;
#pragma unroll 1
    for (int c = 0; c < kCodes / 16; c += 4) {
        float a[16], b[16], d[16], e[16], ra, rb, rd, re;
        tmem_red4x16(trow + c * 16, a, b, d, e, ra, rb, rd, re);
#pragma unroll
        for (int p = 0; p < 16; ++p) {
            const float t = fminf(min3f(a[p], b[p], d[p]), e[p]);
            m[p] = c == 0 ? t : fminf(m[p], t);
        }
        const float rr[4] = {ra, rb, rd, re};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (rr[i] < best) {
                best = rr[i];
                bc = c + i;
                tie = false;
            } else if (rr[i] == best) {
                tie = true;
            }
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
                            umma_f16(acc, sdesc_core16(sbase + OFF_AAUG + k * A_AUG), sdesc_core16(bb + 2 * B_TILE),
                                     idesc, 0);
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
        uint8_t *aaug = base + OFF_AAUG + k * A_AUG;
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
            // the row's operand t = x 2^-(e + er): e the stage scale of the
            // codebooks, er >= 0 the row shift keeping |t| below 2^12
            int e = __ldg(&a.escale_h[g * S]);
            int er;
            ++pc;
            {
                // one pass when the row needs no shift (the usual case); a row that
                // turns out larger is stored again, shifted
                const float se = pow2f(-e);
                float mx = 0.0f;
                uint32_t nz = 0;
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    float f[8];
                    unpack8<ESZ>(xr, a.dtype, c, f);
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        f[i] = f[i] * se;
                        mx = fmaxf(mx, fabsf(f[i]));
                    }
                    nz |= store_chunk(ahi, alo, row, c, f);
                }
                er = row_shift(mx);
                if (__any_sync(0xFFFFFFFFu, er != 0) && er != 0) {
                    const float sr = pow2f(-er);
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        float f[8];
                        unpack8<ESZ>(xr, a.dtype, c, f);
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            f[i] = f[i] * se * sr;
                        nz |= store_chunk(ahi, alo, row, c, f);
                    }
                }
                write_aug_row(aaug, row, er);
                if (nz)
                    lo_stamp[k] = pc;
            }
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
                    int j = argmin_row4(trow, &amb, &vu);
                    if (__any_sync(0xFFFFFFFFu, amb)) {   // warp-collective loads: every lane takes part
                        const int jj = exact_argmin_tmem(trow);
                        if (amb)
                            j = jj;
                    }
                    tc_fence_before();
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
                    load_row(p + gridDim.x);      // the next pair's input, while this pair finishes
                if (s + 1 < S && valid) {
                    // t <- t - c'_bidx 2^-er = t + (hi + lo) 2^(-1-er), the codeword read
                    // from the stage buffer (one block) or from its global copy
                    const float f = pow2f(-1 - er);
                    const uint4 *gh = nullptr;
                    if (NB > 1)
                        gh = reinterpret_cast<const uint4 *>(a.cb16 +
                                                             ((static_cast<int64_t>(cgroup(g) * S + s) * 2) * KC + bidx) * 64);
                    auto codeword = [&](int c, uint4 &hv, uint4 &lv) {
                        if (NB == 1) {
                            const uint32_t bo = swz(bidx, c);
                            hv = *reinterpret_cast<const uint4 *>(bb + bo);
                            lv = *reinterpret_cast<const uint4 *>(bb + B_TILE + bo);
                        } else {
                            hv = __ldg(gh + c);
                            lv = __ldg(gh + KC * 8 + c);
                        }
                    };
                    if (e_next == e) {
                        // |t| stays below 2^12 + S 2^9 < 2^14: the row shift holds
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            uint4 hv, lv;
                            load_chunk(ahi, alo, row, c, t);
                            codeword(c, hv, lv);
                            add_codeword(hv, lv, f, t);
                            store_chunk(ahi, alo, row, c, t);
                        }
                    } else {
                        // the next stage has another codebook scale: rescale the row and
                        // choose its shift again from the updated magnitude
                        float mx = 0.0f;
#pragma unroll 1
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            uint4 hv, lv;
                            load_chunk(ahi, alo, row, c, t);
                            codeword(c, hv, lv);
                            add_codeword(hv, lv, f, t);
#pragma unroll
                            for (int i = 0; i < 8; i += 2)
                                mx = max3f(mx, fabsf(t[i]), fabsf(t[i + 1]));
                        }
                        int E = 0;
                        if (mx > 0.0f)
                            frexpf(mx, &E);                      // |t| < 2^E in units 2^-(e + er)
                        const int tot = E + er + e - e_next;     // |r| < 2^tot in units 2^-e_next
                        const int er2 = tot > v2::kRowLog ? tot - v2::kRowLog : 0;
                        const float gsc = pow2f(er + e - e_next - er2);
#pragma unroll 1
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            uint4 hv, lv;
                            load_chunk(ahi, alo, row, c, t);
                            codeword(c, hv, lv);
                            add_codeword(hv, lv, f, t);
#pragma unroll
                            for (int i = 0; i < 8; ++i)
                                t[i] *= gsc;
                            store_chunk(ahi, alo, row, c, t);
                        }
                        er = er2;
                        write_aug_row(aaug, row, er);
                    }
                }
                mbar_arrive(bar(2 + bi));         // this thread is done with the stage buffer
                if (s + 1 < S) {
                    e = e_next;
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


// ===================================================================
// Persistent kernel for 128-dimensional heads.
//
// The k_rvq64 scheme (two tile slots, split-fp16 operands of -2 c', a per-row
// shift, the residual in the operand tiles, exact ld.red argmin) with the
// head dimension in two 64-wide K blocks.  A slot's hi and lo operand tiles
// take 64 KB, so the stage codebook does not fit twice: it streams through a
// ring of two 32 KB pieces, the hi and the lo half of each K block (256
// codewords x 64 dimensions; the 256 x 16 norm operand rides with a stage's
// first piece), so the next piece loads while the MMAs use the other.  Per
// stage the MMA warp runs slot 0's four pieces (hi piece: hi*hi and lo*hi; lo
// piece: hi*lo; the norm MMA first), committing its accumulator, then slot
// 1's: the stage codebook streams in once per slot, and slot 1's MMAs run
// during slot 0's epilogue (and slot 0's next stage during slot 1's).  Running
// both slots block by block had kept the two in step and left the tensor pipe
// idle through every epilogue (32.9 / 16.8 ms against 28.9 / 14.5 ms for the
// Llama-shaped key / value launches; with the ring 27.95 / 13.99 ms).  The
// buffers are the MMAs' alone: the epilogue reads the chosen codeword's row
// from the float32 codebook in global (L2) memory.  Four helper warps split the
// residual update with the slot warps: after its argmin a slot warp leaves its
// rows' chosen indices and shifts in shared memory and signals the quadrant's
// helper, then updates the first K block while the helper updates the second;
// a stage change of scale exchanges the two halves' row maxima through
// mbarriers, and the MMA warp waits for the helpers' own barrier before a
// slot's next stage (26.2 / 13.6 ms).
namespace v3 {
constexpr int kWarps = 14;                   // 0 TMA, 1 MMA, 2..5 and 6..9 epilogue groups, 10..13 update helpers
constexpr int kThreads = kWarps * 32;
constexpr int A_KB = kRows * 128;            // 16 KB: 128 rows x 64 fp16 (128-byte swizzle)
constexpr int A_HALF = 2 * A_KB;             // hi (or lo): both K blocks
constexpr int A_SLOT = 2 * A_HALF;           // 64 KB
constexpr int A_AUG = kRows * 32;            // 4 KB per slot
constexpr int B_TILE = kCodes * 128;         // 32 KB: 256 codewords x 64 fp16
constexpr int B_BUF = 2 * B_TILE;            // the ring: two 32 KB codebook pieces
constexpr int B_AUG = kCodes * 32;           // 8 KB
constexpr int OFF_A = 0;
constexpr int OFF_AAUG = 2 * A_SLOT;         // 128 KB
constexpr int OFF_B = OFF_AAUG + 2 * A_AUG;  // 136 KB: 1024-aligned
constexpr int OFF_BAUG = OFF_B + B_BUF;
constexpr int OFF_BAR = OFF_BAUG + B_AUG;    // ring_full[2], ring_empty[2], a_ready[2], acc_full[2], drain,
                                             // a_ready_h[2], hand[2][4], mx_e[2][4], mx_h[2][4]
constexpr int OFF_HX = OFF_BAR + 8 * 40;     // per slot and row: chosen index, row shift, partial maxima
constexpr int OFF_SLOT = OFF_HX + 2 * kRows * 16;
constexpr int OFF_LO = OFF_SLOT + 16;
constexpr int OFF_ABORT = OFF_LO + 16;
constexpr int END = OFF_ABORT + 16;
constexpr int SMEM = END + 1024;
static_assert(SMEM <= 232448, "shared memory");
}  // namespace v3

template <int ESZ>
__global__ void __launch_bounds__(v3::kThreads, 1)
k_rvq128(const __grid_constant__ CUtensorMap tmap, const RvqArgs a, int n_pairs)
{
    using namespace v3;
    constexpr int D = 128;
    constexpr int XC = D * ESZ / 16;             // 16-byte chunks per input row
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(base);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(base + OFF_ABORT);
    volatile int *lo_stamp = reinterpret_cast<volatile int *>(base + OFF_LO);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // barrier i: 0,1 ring_full; 2,3 ring_empty; 4,5 a_ready; 6,7 acc_full; 8 drain (MMA completion at exit);
    // 9,10 a_ready_h (helpers); 11 + 4k + q hand (slot k, quadrant q: chosen indices ready); 19 + 4k + q
    // mx_e and 27 + 4k + q mx_h (the two halves' row maxima when the next stage rescales)
    auto bar = [&](int i) { return sbase + OFF_BAR + 8u * i; };
    if (tid == 0) {
        mbar_init(bar(0), 1);
        mbar_init(bar(1), 1);
        mbar_init(bar(2), 1);
        mbar_init(bar(3), 1);
        mbar_init(bar(4), 128);
        mbar_init(bar(5), 128);
        mbar_init(bar(6), 1);
        mbar_init(bar(7), 1);
        mbar_init(bar(8), 1);
        mbar_init(bar(9), 128);                   // a_ready_h: the helpers' half of an update
        mbar_init(bar(10), 128);
        for (int i = 11; i < 35; ++i)             // hand, mx_e, mx_h: one warp each
            mbar_init(bar(i), 32);
        lo_stamp[0] = 0;
        lo_stamp[1] = 0;
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap);
    }
    if (warp == 1)
        tmem_alloc(sbase + OFF_SLOT, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(base + OFF_SLOT);
    const int S = a.S;
    const int64_t nvec = a.batch * a.n_pos;
    const int tiles = a.tiles_per_group;
    const int n_groups = a.n_layers * a.n_heads;
    auto cgroup = [&](int g) { return a.pooled ? g / a.n_heads : g; };
    // The tiles of all head groups in one sequence, paired in order: slot k of
    // pair p takes tile 2p + k, so a pair may straddle two groups (and a
    // group's last odd tile is no half-empty pair).  *lt = the tile within its
    // group; the group is clamped for the tile past the last one (its rows are
    // past the data), whose codebook reads then stay in range.
    auto slot_group = [&](int p, int k, int *lt) -> int {
        const int64_t tau = 2 * static_cast<int64_t>(p) + k;
        const int g = static_cast<int>(tau / tiles);
        *lt = static_cast<int>(tau - static_cast<int64_t>(g) * tiles);
        return g < n_groups ? g : n_groups - 1;
    };

    if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            // pieces of a slot's stage: q = 0 hi of K block 0 (with the slot's
            // norm operand), 1 its lo, 2 hi of K block 1, 3 its lo; piece n
            // goes to ring slot n & 1; each slot's codebook group is its tile's
            int n = 0;
            int last[2] = {-1, -1};
            bool ok = true;
            for (int p = blockIdx.x; p < n_pairs && ok; p += gridDim.x) {
                int lt;
                const int cgs[2] = {cgroup(slot_group(p, 0, &lt)), cgroup(slot_group(p, 1, &lt))};
                for (int s = 0; s < S && ok; ++s) {
                    for (int kq = 0; kq < 8; ++kq, ++n) {
                        const int k = kq >> 2, q = kq & 3, r = n & 1;
                        const int cg = cgs[k];
                        if (!wait_or_abort(bar(2 + r), ((n >> 1) & 1) ^ 1, a.status, abort_flag)) {
                            ok = false;
                            break;
                        }
                        const int row0 = (cg * S + s) * 2 * kCodes + (q & 1) * kCodes;
                        const bool aug = q == 0;
                        mbar_arrive_expect_tx(bar(r), B_TILE + (aug ? B_AUG : 0));
                        tma_load_2d(sbase + OFF_B + r * B_TILE, &tmap, (q >> 1) * 64, row0, bar(r));
                        if (aug)   // free: the other slot's norm MMA precedes the piece this ring slot held
                            bulk_load(sbase + OFF_BAUG, a.cbaug + static_cast<int64_t>(cg * S + s) * kCodes * 16,
                                      B_AUG, bar(r));
                        last[r] = n;
                    }
                }
            }
            // no copy may still be landing in shared memory when the CTA exits
            for (int r = 0; r < 2; ++r)
                if (last[r] >= 0)
                    mbar_wait(bar(r), (last[r] >> 1) & 1, a.status);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_f16_f32(kRows, kCodes);
            int n = 0;
            uint32_t aph[2] = {0, 0}, hph[2] = {0, 0};
            int pc = 0;
            bool ok = true;
            for (int p = blockIdx.x; p < n_pairs && ok; p += gridDim.x) {
                ++pc;
                for (int s = 0; s < S && ok; ++s) {
                    for (int kq = 0; kq < 8 && ok; ++kq, ++n) {
                        const int k = kq >> 2, q = kq & 3, r = n & 1;
                        ok = wait_or_abort(bar(r), (n >> 1) & 1, a.status, abort_flag);
                        if (!ok)
                            break;
                        if (q == 0) {
                            ok = wait_or_abort(bar(4 + k), aph[k], a.status, abort_flag);
                            if (ok && s > 0) {    // the helpers' half of the update
                                ok = wait_or_abort(bar(9 + k), hph[k], a.status, abort_flag);
                                hph[k] ^= 1;
                            }
                            if (!ok)
                                break;
                            aph[k] ^= 1;
                        }
                        tc_fence_after();
                        const bool lo = s > 0 || lo_stamp[k] == pc;
                        const uint32_t bb = sbase + OFF_B + r * B_TILE;
                        const uint32_t ab = sbase + OFF_A + k * A_SLOT + (q >> 1) * A_KB;
                        const uint32_t acc = tmem + k * 256;
                        if (q == 0)   // codeword norms first (K = 16, no swizzle)
                            umma_f16(acc, sdesc_core16(sbase + OFF_AAUG + k * A_AUG), sdesc_core16(sbase + OFF_BAUG),
                                     idesc, 0);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint64_t db = sdesc_sw128(bb + kk * 32);
                            umma_f16(acc, sdesc_sw128(ab + kk * 32), db, idesc, 1);     // hi*hi or hi*lo
                            if ((q & 1) == 0 && lo)
                                umma_f16(acc, sdesc_sw128(ab + A_HALF + kk * 32), db, idesc, 1);   // lo*hi
                        }
                        if (q == 3)
                            umma_commit(bar(6 + k));
                        umma_commit(bar(2 + r));          // the ring slot is free once these MMAs are done
                    }
                }
            }
            // every MMA has completed before tensor memory is released
            umma_commit(bar(8));
            mbar_wait(bar(8), 0, a.status);
        }
    } else if (warp >= 10) {
        // ---------------------------------------------------- update helpers
        // warp 10 + i serves quadrant (10 + i) & 3 of both slots: for every
        // update, the second K block (dimensions 64..127) of its 32 rows
        const int quad = warp & 3;
        const int row = quad * 32 + lane;
        uint8_t *hx0 = base + OFF_HX;
        uint32_t hp_[2] = {0, 0}, xp_[2] = {0, 0};
        bool ok = true;
        for (int p = blockIdx.x; p < n_pairs && ok; p += gridDim.x) {
            int lt;
            const int gs[2] = {slot_group(p, 0, &lt), slot_group(p, 1, &lt)};
            int es[2] = {__ldg(&a.escale_h[gs[0] * S]), __ldg(&a.escale_h[gs[1] * S])};
            for (int s = 0; s + 1 < S && ok; ++s) {
                for (int k = 0; k < 2 && ok; ++k) {
                    const int g = gs[k], e = es[k];
                    const int e_next = __ldg(&a.escale_h[g * S + s + 1]);
                    es[k] = e_next;
                    ok = wait_or_abort(bar(11 + 4 * k + quad), hp_[k], a.status, abort_flag);
                    ok = __all_sync(0xFFFFFFFFu, ok);
                    if (!ok)
                        break;
                    hp_[k] ^= 1;
                    uint8_t *hx = hx0 + (k * kRows + row) * 16;
                    const int bidx = hx[0];
                    const int er = *reinterpret_cast<const int *>(hx + 4);
                    uint8_t *ahi = base + OFF_A + k * A_SLOT + A_KB;
                    uint8_t *alo = ahi + A_HALF;
                    const float f = -pow2f(-e - er);
                    const float *cbs = a.cb32 + static_cast<int64_t>(cgroup(g) * S + s) * kCodes * D;
                    const float4 *gc = reinterpret_cast<const float4 *>(cbs + bidx * D) + 16;
                    if (e_next == e) {
                        if (__all_sync(0xFFFFFFFFu, er == 0))
                            update_rows_t<true>(ahi, alo, quad, cbs + 64, bidx, f);
                        else
                            update_rows_t<false>(ahi, alo, quad, cbs + 64, bidx, f);
                    } else {
                        float mx = 0.0f;
#pragma unroll 4
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            load_add_chunk(ahi, alo, row, c, __ldg(gc + 2 * c), __ldg(gc + 2 * c + 1), f, t);
#pragma unroll
                            for (int i = 0; i < 8; i += 2)
                                mx = max3f(mx, fabsf(t[i]), fabsf(t[i + 1]));
                            store_chunk(ahi, alo, row, c, t);
                        }
                        // the row's maximum over both halves: exchange with the slot's warp
                        *reinterpret_cast<float *>(hx + 12) = mx;
                        mbar_arrive(bar(27 + 4 * k + quad));
                        ok = wait_or_abort(bar(19 + 4 * k + quad), xp_[k], a.status, abort_flag);
                        ok = __all_sync(0xFFFFFFFFu, ok);
                        if (!ok)
                            break;
                        xp_[k] ^= 1;
                        mx = fmaxf(mx, *reinterpret_cast<const float *>(hx + 8));
                        int E = 0;
                        if (mx > 0.0f)
                            frexpf(mx, &E);
                        const int tot = E + er + e - e_next;
                        const int er2 = tot > v2::kRowLog ? tot - v2::kRowLog : 0;
                        const float gsc = pow2f(er + e - e_next - er2);
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            load_chunk(ahi, alo, row, c, t);
#pragma unroll
                            for (int i = 0; i < 8; ++i)
                                t[i] *= gsc;
                            store_chunk(ahi, alo, row, c, t);
                        }
                    }
                    fence_proxy_async_smem();
                    mbar_arrive(bar(9 + k));
                }
            }
        }
    } else {
        // ---------------------------------------------------- epilogue groups
        const int k = (warp - 2) >> 2;           // tile slot 0 or 1
        const int quad = warp & 3;                // TMEM lane quadrant of this warp
        const int row = quad * 32 + lane;
        const uint32_t trow = tmem + k * 256 + (static_cast<uint32_t>(quad * 32) << 16);
        uint8_t *ahi = base + OFF_A + k * A_SLOT;
        uint8_t *alo = ahi + A_HALF;
        uint8_t *aaug = base + OFF_AAUG + k * A_AUG;
        const int64_t all_tiles = static_cast<int64_t>(n_groups) * tiles;
        auto row_src = [&](int p, bool *in) -> const uint4 * {
            int tile;
            const int g = slot_group(p, k, &tile);
            const int64_t v = static_cast<int64_t>(tile) * kRows + row;
            *in = 2 * static_cast<int64_t>(p) + k < all_tiles && v < nvec;
            if (!*in)
                return nullptr;
            const int l = g / a.n_heads, h = g - l * a.n_heads;
            const int64_t b = v / a.n_pos;
            const int64_t t = a.t0 + (v - b * a.n_pos);
            return reinterpret_cast<const uint4 *>(static_cast<const uint8_t *>(a.x) +
                                                   (l * a.s_layer + b * a.s_batch + h * a.s_head + t * a.s_pos) * ESZ);
        };
        int it = 0;
        uint32_t fph = 0, xph = 0;
        int pc = 0;
        for (int p = blockIdx.x; p < n_pairs; p += gridDim.x) {
            int tile;
            const int g = slot_group(p, k, &tile);
            const int l = g / a.n_heads, h = g - l * a.n_heads;
            const int64_t v = static_cast<int64_t>(tile) * kRows + row;
            const bool valid = 2 * static_cast<int64_t>(p) + k < all_tiles && v < nvec;
            bool in;
            const uint4 *src = row_src(p, &in);
            // the row's operand t = x 2^-(e + er), er >= 0 keeping |t| below 2^12
            int e = __ldg(&a.escale_h[g * S]);
            int er;
            ++pc;
            {
                // one pass when the row needs no shift (its magnitude below 2^12 in
                // units of 2^-e, the usual case): the operand is stored as it is
                // read; a row that turns out larger is stored again, shifted
                const float se = pow2f(-e);
                float mx = 0.0f;
                uint32_t nz = 0;
#pragma unroll 4
                for (int c = 0; c < 16; ++c) {
                    float f[8];
                    uint4 xr[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)};
                    if (in) {
                        xr[0] = __ldg(src + c * (ESZ / 2));
                        if (ESZ == 4)
                            xr[1] = __ldg(src + c * 2 + 1);
                    }
                    unpack8<ESZ>(xr, a.dtype, 0, f);
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        f[i] = f[i] * se;
                        mx = fmaxf(mx, fabsf(f[i]));
                    }
                    nz |= store_chunk(ahi + (c >> 3) * A_KB, alo + (c >> 3) * A_KB, row, c & 7, f);
                }
                er = row_shift(mx);
                if (__any_sync(0xFFFFFFFFu, er != 0)) {
                    const float sr = pow2f(-er);
#pragma unroll 4
                    for (int c = 0; c < 16; ++c) {
                        if (er == 0)
                            continue;
                        float f[8];
                        uint4 xr[2] = {make_uint4(0, 0, 0, 0), make_uint4(0, 0, 0, 0)};
                        if (in) {
                            xr[0] = __ldg(src + c * (ESZ / 2));
                            if (ESZ == 4)
                                xr[1] = __ldg(src + c * 2 + 1);
                        }
                        unpack8<ESZ>(xr, a.dtype, 0, f);
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            f[i] = f[i] * se * sr;
                        nz |= store_chunk(ahi + (c >> 3) * A_KB, alo + (c >> 3) * A_KB, row, c & 7, f);
                    }
                }
                write_aug_row(aaug, row, er);
                if (nz)
                    lo_stamp[k] = pc;
            }
            fence_proxy_async_smem();
            mbar_arrive(bar(4 + k));
            if (p + static_cast<int>(gridDim.x) < n_pairs) {
                // the next pair's input row into L2 while this pair runs
                bool nin;
                const uint4 *nsrc = row_src(p + gridDim.x, &nin);
                if (nin)
                    for (int c = 0; c < XC; c += 8)
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(nsrc + c));
            }
            uint8_t idx[8];
            bool ok = true;
            for (int s = 0; s < S; ++s, ++it) {
                const int e_next = s + 1 < S ? __ldg(&a.escale_h[g * S + s + 1]) : e;
                ok = wait_or_abort(bar(6 + k), fph, a.status, abort_flag);
                // the tensor-memory loads below are warp-collective: the warp
                // goes on, or leaves, as one
                ok = __all_sync(0xFFFFFFFFu, ok);
                if (!ok)
                    break;
                fph ^= 1;
                tc_fence_after();
                __syncwarp();
                bool amb;
                float vu;
                int bidx = argmin_row4(trow, &amb, &vu);
                if (__any_sync(0xFFFFFFFFu, amb)) {   // warp-collective loads: every lane takes part
                    const int jj = exact_argmin_tmem(trow);
                    if (amb)
                        bidx = jj;
                }
                tc_fence_before();
                idx[s] = static_cast<uint8_t>(bidx);
                if (s + 1 < S) {
                    // t <- t - c 2^(-e-er) (t is the row in units of 2^-(e+er)),
                    // c the chosen codeword's float32 row; this warp takes the first
                    // K block, the quadrant's helper the second
                    uint8_t *hx = base + OFF_HX + (k * kRows + row) * 16;
                    hx[0] = static_cast<uint8_t>(bidx);
                    *reinterpret_cast<int *>(hx + 4) = er;
                    mbar_arrive(bar(11 + 4 * k + quad));
                    const float f = -pow2f(-e - er);
                    const float *cbs = a.cb32 + static_cast<int64_t>(cgroup(g) * S + s) * kCodes * D;
                    const float4 *gc = reinterpret_cast<const float4 *>(cbs + bidx * D);
                    if (e_next == e) {
                        if (__all_sync(0xFFFFFFFFu, er == 0))
                            update_rows_t<true>(ahi, alo, quad, cbs, bidx, f);
                        else
                            update_rows_t<false>(ahi, alo, quad, cbs, bidx, f);
                    } else {
                        float mx = 0.0f;
#pragma unroll 4
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            load_add_chunk(ahi, alo, row, c, __ldg(gc + 2 * c), __ldg(gc + 2 * c + 1), f, t);
#pragma unroll
                            for (int i = 0; i < 8; i += 2)
                                mx = max3f(mx, fabsf(t[i]), fabsf(t[i + 1]));
                            store_chunk(ahi, alo, row, c, t);
                        }
                        // the row's maximum over both halves: exchange with the helper
                        *reinterpret_cast<float *>(hx + 8) = mx;
                        mbar_arrive(bar(19 + 4 * k + quad));
                        ok = wait_or_abort(bar(27 + 4 * k + quad), xph, a.status, abort_flag);
                        ok = __all_sync(0xFFFFFFFFu, ok);
                        if (!ok)
                            break;
                        xph ^= 1;
                        mx = fmaxf(mx, *reinterpret_cast<const float *>(hx + 12));
                        int E = 0;
                        if (mx > 0.0f)
                            frexpf(mx, &E);
                        const int tot = E + er + e - e_next;
                        const int er2 = tot > v2::kRowLog ? tot - v2::kRowLog : 0;
                        const float gsc = pow2f(er + e - e_next - er2);
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            float t[8];
                            load_chunk(ahi, alo, row, c, t);
#pragma unroll
                            for (int i = 0; i < 8; ++i)
                                t[i] *= gsc;
                            store_chunk(ahi, alo, row, c, t);
                        }
                        er = er2;
                        write_aug_row(aaug, row, er);
                    }
                    e = e_next;
                    fence_proxy_async_smem();
                    mbar_arrive(bar(4 + k));
                }
            }
            if (!ok)
                break;
            if (valid) {
                const int64_t b = v / a.n_pos;
                const int64_t t = a.t0 + (v - b * a.n_pos);
                uint8_t *dst = static_cast<uint8_t *>(a.sym) + (b * a.n_layers + l) * a.stream_stride +
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

// ===================================================================
// The failure path of the kernels above, on barriers that never complete.
// Warp 1 holds TMEM as the MMA warp does; warp 0's lane 0 waits on bar 0,
// which nothing arrives on, gives up after limit_ns and raises the abort
// flag; warp 1's lane 0 waits on the same barrier with the library's full
// limit and must leave on the flag, well before its own timer.  Warp 2 checks
// that a plain bounded wait passes a completed phase and times out on an
// open one.  All warps then meet and TMEM is released, as in the kernels'
// teardown.  out: [0] warp 0's wait result, [1] warp 1's, [2] 1 if warp 1
// left within 2 x limit_ns (on the flag), [3] the completed phase's wait,
// [4] the open phase's wait, [5] 1 after the teardown.
__global__ void __launch_bounds__(96, 1) k_wait_check(unsigned *status, uint64_t limit_ns, int *out)
{
    __shared__ __align__(8) uint64_t bars[3];
    __shared__ int abort_word;
    __shared__ uint32_t tmem_slot;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int *abort_flag = &abort_word;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    if (threadIdx.x == 0) {
        for (int i = 0; i < 3; ++i)
            mbar_init(bar(i), 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1)
        tmem_alloc(smem_u32(&tmem_slot), 32);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t *>(&tmem_slot);
    if (lane == 0) {
        if (warp == 0) {
            out[0] = wait_or_abort(bar(0), 0, status, abort_flag, limit_ns) ? 1 : 0;
        } else if (warp == 1) {
            const uint64_t t0 = globaltimer_ns();
            out[1] = wait_or_abort(bar(0), 0, status, abort_flag) ? 1 : 0;
            out[2] = globaltimer_ns() - t0 < 2 * limit_ns ? 1 : 0;
        } else {
            mbar_arrive(bar(1));
            out[3] = mbar_wait(bar(1), 0, status, limit_ns) ? 1 : 0;
            out[4] = mbar_wait(bar(2), 0, status, limit_ns) ? 1 : 0;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem, 32);
    }
    if (threadIdx.x == 0)
        out[5] = 1;
}

}  // namespace

cudaError_t launch_wait_check(unsigned *status, uint64_t limit_ns, int *out_dev, cudaStream_t st)
{
    k_wait_check<<<1, 96, 0, st>>>(status, limit_ns, out_dev);
    return cudaGetLastError();
}

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
        // 128-dimensional heads: 256 codewords per stage, the tiles of all
        // head groups paired in order
        const int64_t n_pairs = (tiles * c->Ly * c->H + 1) / 2;
        if (n_pairs > 0x7FFFFFFF)
            return cudaErrorInvalidConfiguration;
        int sms = 0;
        cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c->device);
        if (e != cudaSuccess)
            return e;
        const unsigned grid = static_cast<unsigned>(n_pairs < sms ? n_pairs : sms);
        const int np = static_cast<int>(n_pairs);
        if (x->dtype == FKV_F32) {
            e = cudaFuncSetAttribute(k_rvq128<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, v3::SMEM);
            if (e != cudaSuccess)
                return e;
            k_rvq128<4><<<grid, v3::kThreads, v3::SMEM, st>>>(cb.tmap, a, np);
        } else {
            e = cudaFuncSetAttribute(k_rvq128<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, v3::SMEM);
            if (e != cudaSuccess)
                return e;
            k_rvq128<2><<<grid, v3::kThreads, v3::SMEM, st>>>(cb.tmap, a, np);
        }
    }
    return cudaGetLastError();
}
