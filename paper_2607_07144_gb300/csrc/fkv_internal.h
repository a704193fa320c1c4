// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "fkv.h"

// Device status bits (ctx->d_status); mapped to FKV_E* by fkv_sync_status.
#define FKV_ST_CORRUPT 1u
#define FKV_ST_TIMEOUT 2u
#define FKV_ST_RANGE 4u      // a request named a position or stream outside the archive

// Codebook-side constants of one K-or-V half of the archive.  G codebook
// groups (G = Ly * H per-head, Ly pooled), K = ctx->KC codewords per stage.
struct fkv_cbset {
    int stages = 0;
    float *cb32 = nullptr;    // [G][S][K][D] float32 (gather, residual update)
    __half *cb16 = nullptr;   // [G][S][2][K][D] fp16 hi/lo split, scaled by 2^-e
    int *escale = nullptr;    // [G][S] exponent e of the fp16 split
    int *escale_h = nullptr;  // [Ly*H][S] the same per head (its group's), for k_rvq64
    CUtensorMap tmap;         // TMA map over cb16 as [rows][D], box {64, 256}, 128B swizzle
    // 64-dimensional heads only (rvq.cu k_rvq64): cb16 holds the hi/lo split of
    // -2 c 2^-e with max |c 2^-e| in [2^3, 2^9), and cbaug the norm operand.
    __half *cbaug = nullptr;  // [G][S] blocks of K x 16 fp16 in core-matrix layout (32 B per codeword)
};

// Largest alphabet: symbols are uint8 up to N = 256 and uint16 above.
#define FKV_MAX_N 1024

// Decoder constants (see decode_core.cuh).  Fixed point is Q1.62 (value * 2^62).
struct fkv_decconst {
    long long vx[FKV_MAX_N], vy[FKV_MAX_N];    // V(c)
    float vfx[FKV_MAX_N], vfy[FKV_MAX_N];      // V(c) rounded to float
    long long alim[48];            // anchor limit 2^-4 r^m in Q1.62, per span length m
    float sect_thr;                // sector test threshold, N > 8 (decode_core.cuh classify)
};

struct fkv_ctx {
    int N = 0;
    double r = 0.0;
    int L = 0;
    int device = 0;
    double2 *d_V = nullptr;        // [N] vertices
    fkv_decconst *d_dec = nullptr; // decoder constants (device copy)
    longlong2 *d_T = nullptr;      // [L][N] (1-r) r^j V(c) in Q1.62
    unsigned *d_status = nullptr;
    // archive geometry and codebooks
    bool has_cb = false;
    int Ly = 0, H = 0, D = 0;
    int KC = 256;                  // codewords per stage (= N): 256 or 1024
    bool pooled = false;           // one codebook per layer shared by its heads
    fkv_cbset cb[2];
    uint8_t *d_scratch = nullptr;
    size_t scratch_bytes = 0;
    // record reads: request indices grouped by layer and the layer counters
    // (gather.cu launch_read_kv), grown on demand
    int *d_read_order = nullptr;
    size_t read_order_bytes = 0;
    // device address and size of the library's fixed scratch array on this
    // context's device (decode_static.cu), looked up once by fkv_create
    uint8_t *static_scratch = nullptr;
    size_t static_scratch_bytes = 0;
    std::string err;
};

struct fkv_streams {
    fkv_ctx *ctx = nullptr;
    int64_t n_streams = 0;
    int64_t length = 0;          // symbols per stream
    int64_t cap_spans = 0;       // point stride
    double *d_pts = nullptr;     // [n_streams][cap_spans][2]
};

// ---------------------------------------------------------------- launches
// codec.cu
// Dynamic shared memory the codec's decoding kernels take for (N, L): the
// decoder tables plus one chunk of staged symbols.
int codec_smem_bytes(int N, int L);
constexpr int kMaxDynSmem = 232448;   // 227 KB per block on sm_103a

// Symbols are uint8 when c->N <= 256, else uint16; strides count symbols.
cudaError_t launch_span_encode(const fkv_ctx *c, const void *sym, int64_t n_streams, int64_t n,
                               int64_t sym_stride, double *pts, int64_t pt_stride, cudaStream_t st);
cudaError_t launch_span_decode(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n,
                               int64_t pt_stride, void *sym, int64_t sym_stride, cudaStream_t st);
cudaError_t launch_read(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n,
                        int64_t pt_stride, const int64_t *req, int64_t n_req, void *out,
                        cudaStream_t st);
// Ragged batches: stream i's symbols at sym + so[i], len_i = so[i+1] - so[i];
// its points in slots [po[i], po[i+1]) of pts (device offset arrays).
cudaError_t launch_span_encode_ragged(const fkv_ctx *c, const void *sym, const int64_t *so, int64_t n_streams,
                                      double *pts, const int64_t *po, cudaStream_t st);
cudaError_t launch_span_decode_ragged(const fkv_ctx *c, const double *pts, const int64_t *po, int64_t n_streams,
                                      void *sym, const int64_t *so, cudaStream_t st);
cudaError_t launch_read_ragged(const fkv_ctx *c, const double *pts, const int64_t *po, const int64_t *so,
                               int64_t n_streams, const int64_t *req, int64_t n_req, void *out, cudaStream_t st);
cudaError_t launch_suffix_search(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n,
                                 int64_t pt_stride, const uint16_t *query, int qlen, int64_t *out, int64_t cap,
                                 int64_t *counts, cudaStream_t st);
cudaError_t launch_append(const fkv_ctx *c, double *pts, int64_t n_streams, int64_t pt_stride,
                          int64_t n_old, const void *sym, int64_t m, int64_t sym_stride,
                          cudaStream_t st);
// Sec. 4 lossy archive: B-bit codes of the spans older than the last
// keep_exact, packed (words of uint32 per stream), plus the exact tail points.
cudaError_t launch_truncate(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n, int64_t pt_stride,
                            int bits, int64_t keep_exact, uint32_t *codes, int64_t code_stride, double *tail,
                            int64_t tail_stride, cudaStream_t st);
cudaError_t launch_lossy_decode(const fkv_ctx *c, const uint32_t *codes, int64_t code_stride, const double *tail,
                                int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                                void *sym, int64_t sym_stride, cudaStream_t st);
cudaError_t launch_lossy_read(const fkv_ctx *c, const uint32_t *codes, int64_t code_stride, const double *tail,
                              int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                              const int64_t *req, int64_t n_req, void *out, cudaStream_t st);
// Binary64 add/mul instructions per second of the current device, measured
// by independent chains (the span encoder's roofline denominator).
cudaError_t measure_fp64_rate(int device, cudaStream_t st, double *ops_per_s);
// One CTA that runs the RVQ kernels' bounded waits against barriers that
// never complete (limit_ns for the first waiter) and their teardown: results
// to out_dev[0..5] (device ints), the timeout bit to *status.
cudaError_t launch_wait_check(unsigned *status, uint64_t limit_ns, int *out_dev, cudaStream_t st);
// ac.cu (Sec. 6 probability-weighted maps): words that always hold the code
// of n symbols, and the warp-per-stream coder
int64_t ac_capacity_words(int N, int64_t n);
cudaError_t launch_ac_encode(const fkv_ctx *c, const void *sym, int64_t n_streams, int64_t n, int64_t sym_stride,
                             int adaptive, uint32_t *words, int64_t word_stride, int64_t *nbits, cudaStream_t st);
cudaError_t launch_ac_decode(const fkv_ctx *c, const uint32_t *words, int64_t word_stride, const int64_t *nbits,
                             int64_t n_streams, int64_t n, int adaptive, void *sym, int64_t sym_stride, cudaStream_t st);
// rvq.cu
cudaError_t launch_rvq_encode(const fkv_ctx *c, int kv, const fkv_cache *x, int64_t t0, int64_t t1,
                              void *sym, int64_t stream_stride, int64_t rec0, cudaStream_t st);
// Decoded archive symbols in one of two layouts: the token records of the
// stream itself (stream_stride symbols per stream), or planar (per stream of
// n_rec * R symbols: H key planes of n_rec x S_K, then H value planes of
// n_rec x S_V), which launch_span_decode_planar writes for the gather.
enum { FKV_SYM_RECORDS = 0, FKV_SYM_PLANAR = 1 };
cudaError_t launch_span_decode_planar(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n_rec,
                                      int64_t pt_stride, void *out, cudaStream_t st);
// fkv_api.cu: both output views (either may be null) hold [t0, t0 + n_rec);
// the planar decode of a whole archive into `scratch` (n_streams * n_rec * R
// symbols) and the K/V gathers from it, once every argument has been checked.
bool check_outputs(const fkv_ctx *ctx, const fkv_cache *k_out, const fkv_cache *v_out, int64_t n_rec, int64_t t0);
int decode_archive(fkv_ctx *ctx, const double *pts, int64_t n_streams, int64_t n_rec, int64_t pt_stride,
                   void *scratch, const fkv_cache *k_out, const fkv_cache *v_out, int64_t t0, cudaStream_t st);
// decode_static.cu: look up the fixed scratch array's device address for the
// current device (context creation only)
int static_scratch_resolve(fkv_ctx *ctx);
// gather.cu
cudaError_t launch_rvq_decode(const fkv_ctx *c, int kv, const void *sym, int layout, int64_t stream_stride,
                              int64_t n_rec, const fkv_cache *out, int64_t t0, cudaStream_t st);
// order: null, or room for read_order_ints(c, n_req) ints, 16-byte aligned
// (requests then taken grouped by layer)
cudaError_t launch_read_kv(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n_rec,
                           int64_t pt_stride, const int64_t *req, int64_t n_req, void *out,
                           int dtype, int *order, cudaStream_t st);
// ints of the record reads' order buffer for n_req requests, or 0 when the
// requests are taken in their given order (too many requests or layers)
int64_t read_order_ints(const fkv_ctx *c, int64_t n_req);

// ------------------------------------------------------- device helpers
#ifdef __CUDACC__
namespace fkvd {

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Every device wait in the library gives up after this long and records
// FKV_ST_TIMEOUT instead of spinning forever.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait on an mbarrier phase; false (and a status bit) on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned *status,
                                          uint64_t limit_ns = kWaitLimitNs)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity))
            return true;
        if (globaltimer_ns() - t0 > limit_ns) {
            atomicOr(status, FKV_ST_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 2-D TMA tile load into shared memory, completion counted on `bar`.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int c0, int c1,
                                            uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void prefetch_tmap(const CUtensorMap *map)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---- tcgen05 (5th-generation tensor core, accumulators in tensor memory)
__device__ __forceinline__ void tmem_alloc(uint32_t slot_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot_smem),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (fp16 or bf16 in, fp32 accumulate).
__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive on `bar` once every previously issued tcgen05.mma of this thread is done.
__device__ __forceinline__ void umma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// Shared-memory matrix descriptor: K-major operand in the 128-byte swizzle
// layout (rows of 64 16-bit elements, 8-row / 1024-byte swizzle atoms).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr)
{
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);   // start address
    d |= static_cast<uint64_t>(1) << 16;                    // leading byte offset (unused here)
    d |= static_cast<uint64_t>(1024 >> 4) << 32;            // stride byte offset: 8 rows x 128 B
    d |= static_cast<uint64_t>(1) << 46;                    // descriptor version (sm_100 family)
    d |= static_cast<uint64_t>(2) << 61;                    // swizzle mode: 128 B
    return d;
}

// Instruction descriptor, kind::f16: fp16 A and B (K-major), fp32 D, M x N.
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N)
{
    return (1u << 4)                                   // D format: f32
           | (0u << 7) | (0u << 10)                    // A, B format: f16
           | (static_cast<uint32_t>(N >> 3) << 17)     // N / 8
           | (static_cast<uint32_t>(M >> 4) << 24);    // M / 16
}

}  // namespace fkvd
#endif
