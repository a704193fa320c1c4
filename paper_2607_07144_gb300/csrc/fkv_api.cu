// Host side of the C ABI declared in include/fkv.h: argument checks, the
// context (vertex table, decoder constants, codebook copies), stream sets,
// and the launches of the kernels in codec.cu, rvq.cu and gather.cu.
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <cstdlib>
#include <mutex>
#include <vector>

#include "fkv_internal.h"

namespace {

const char *kNoCtx = "no context";

int fail(fkv_ctx *c, int code, const char *msg)
{
    if (c)
        c->err = msg;
    return code;
}

int cuda_fail(fkv_ctx *c, cudaError_t e, const char *where)
{
    if (c) {
        c->err = std::string(where) + ": " + cudaGetErrorString(e);
    }
    return e == cudaErrorMemoryAllocation ? FKV_ENOMEM : FKV_ECUDA;
}

#define CK(call, where)                              \
    do {                                             \
        cudaError_t e_ = (call);                     \
        if (e_ != cudaSuccess)                       \
            return cuda_fail(ctx, e_, where);        \
    } while (0)

// Sec. 1 vertex table: unit circumradius, V(0) = (1, 0), counter-clockwise,
// the angle 2*pi*c/N in binary64; quarter turns are exactly 0 and +-1.
void vertex(int N, int c, double *x, double *y)
{
    if ((4 * c) % N == 0) {
        const int q = (4 * c) / N;
        *x = q == 0 ? 1.0 : (q == 2 ? -1.0 : 0.0);
        *y = q == 1 ? 1.0 : (q == 3 ? -1.0 : 0.0);
        return;
    }
    const double theta = 2.0 * M_PI * c / N;
    *x = cos(theta);
    *y = sin(theta);
}

long long q_round(long double v, int frac_bits)
{
    return llroundl(ldexpl(v, frac_bits));
}

// Bytes per symbol: uint8 up to N = 256, uint16 above.
int sym_size(const fkv_ctx *c)
{
    return c->N > 256 ? 2 : 1;
}

void destroy_cbset(fkv_cbset &s)
{
    cudaFree(s.cb32);
    cudaFree(s.cb16);
    cudaFree(s.escale);
    cudaFree(s.escale_h);
    cudaFree(s.cbaug);
    s = fkv_cbset();
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// Byte offset of element (row, k) of a [rows x 16] fp16 operand in the
// no-swizzle K-major core-matrix layout (8 x 16-byte core matrices; 128 B
// between the two along K, 256 B between 8-row groups).
size_t core16_offset(int row, int k)
{
    return static_cast<size_t>(row / 8) * 256 + (k / 8) * 128 + (row % 8) * 16 + (k % 8) * 2;
}

// Three fp16 parts whose sum is v to about 33 bits.
void split3(double v, __half *out)
{
    double rest = v;
    for (int i = 0; i < 3; ++i) {
        out[i] = __double2half(rest);
        rest -= static_cast<double>(__half2float(out[i]));
    }
}

// Upload one K-or-V half of the codebooks: float32 copy, squared norms and
// the fp16 operands of the tensor-core RVQ kernels with their TMA map:
//   hi/lo split of -2 c 2^-e, max |c 2^-e| in [2^3, 2^9)
//   (in [2^8, 2^9) at a group's first stage; later stages keep the previous
//   e while they can), and a K x 16 norm operand per (group, stage):
//   columns 0-2 hold three fp16 parts of ||c 2^-e||^2 2^-10, the rest zero.
// G = Ly * H codebook groups per-head, Ly pooled; K = ctx->KC codewords.
int upload_cbset(fkv_ctx *ctx, int kv, const float *host, int stages)
{
    fkv_cbset &s = ctx->cb[kv];
    s.stages = stages;
    const int G = ctx->Ly * (ctx->pooled ? 1 : ctx->H), D = ctx->D, K = ctx->KC;
    const size_t ncode = static_cast<size_t>(G) * stages * K;
    std::vector<int> es(static_cast<size_t>(G) * stages);
    std::vector<__half> c16(ncode * 2 * D);
    std::vector<__half> caug(ncode * 16, __float2half(0.0f));
    for (int gs = 0; gs < G * stages; ++gs) {
        const float *cb = host + static_cast<size_t>(gs) * K * D;
        float m = 0.0f;
        for (int i = 0; i < K * D; ++i) {
            if (!isfinite(cb[i]))
                return fail(ctx, FKV_EINVAL, "codebook holds a non-finite value");
            m = fmaxf(m, fabsf(cb[i]));
        }
        int E = 0;
        if (m > 0.0f)
            frexpf(m, &E);
        int e = m > 0.0f ? E - 9 : 0;
        if (gs % stages != 0) {
            // keep the previous stage's scale while this stage's max |c| 2^-e
            // stays in [2^3, 2^9), so the kernels rescale the residual only
            // between stages of very different magnitude
            const int prev = es[gs - 1];
            const float q = ldexpf(m, -prev);
            if (q >= 8.0f && q < 512.0f)
                e = prev;
        }
        es[gs] = e;
        const float mul = -2.0f;
        for (int j = 0; j < K; ++j) {
            double ns = 0.0;
            for (int d = 0; d < D; ++d) {
                const double vs = ldexp(static_cast<double>(cb[j * D + d]), -e);
                ns += vs * vs;
                const float sv = mul * ldexpf(cb[j * D + d], -e);
                const __half hi = __float2half_rn(sv);
                const __half lo = __float2half_rn(sv - __half2float(hi));
                c16[((static_cast<size_t>(gs) * 2 + 0) * K + j) * D + d] = hi;
                c16[((static_cast<size_t>(gs) * 2 + 1) * K + j) * D + d] = lo;
            }
            // K rows in the core-matrix layout: 256-row blocks of 8 KB, back to back
            __half *blk = caug.data() + static_cast<size_t>(gs) * K * 16;
            __half parts[3];
            split3(ldexp(ns, -10), parts);
            for (int k = 0; k < 16; ++k) {
                const __half val = k < 3 ? parts[k] : __float2half(0.0f);
                blk[core16_offset(j, k) / 2] = val;
            }
        }
    }
    CK(cudaMalloc(&s.cb32, ncode * D * sizeof(float)), "codebook alloc");
    CK(cudaMalloc(&s.cb16, ncode * 2 * D * sizeof(__half)), "codebook alloc");
    CK(cudaMalloc(&s.escale, es.size() * sizeof(int)), "codebook alloc");
    CK(cudaMemcpy(s.cb32, host, ncode * D * sizeof(float), cudaMemcpyHostToDevice), "codebook copy");
    CK(cudaMemcpy(s.cb16, c16.data(), c16.size() * sizeof(__half), cudaMemcpyHostToDevice), "codebook copy");
    CK(cudaMemcpy(s.escale, es.data(), es.size() * sizeof(int), cudaMemcpyHostToDevice), "codebook copy");
    {
        // each head's copy of its codebook group's scales
        const int GH = ctx->Ly * ctx->H;
        std::vector<int> eh(static_cast<size_t>(GH) * stages);
        for (int g = 0; g < GH; ++g)
            for (int st = 0; st < stages; ++st)
                eh[static_cast<size_t>(g) * stages + st] = es[static_cast<size_t>(ctx->pooled ? g / ctx->H : g) * stages + st];
        CK(cudaMalloc(&s.escale_h, eh.size() * sizeof(int)), "codebook alloc");
        CK(cudaMemcpy(s.escale_h, eh.data(), eh.size() * sizeof(int), cudaMemcpyHostToDevice), "codebook copy");
    }
    CK(cudaMalloc(&s.cbaug, caug.size() * sizeof(__half)), "codebook alloc");
    CK(cudaMemcpy(s.cbaug, caug.data(), caug.size() * sizeof(__half), cudaMemcpyHostToDevice), "codebook copy");
    EncodeTiledFn enc = encode_tiled();
    if (!enc)
        return fail(ctx, FKV_ECUDA, "cuTensorMapEncodeTiled unavailable");
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(ncode * 2)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(D) * sizeof(__half)};
    const cuuint32_t box[2] = {64, 256};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&s.tmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, s.cb16, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(ctx, FKV_ECUDA, "cuTensorMapEncodeTiled failed");
    return FKV_OK;
}

bool check_cache(const fkv_ctx *ctx, const fkv_cache *c)
{
    if (!c || !c->data || c->batch <= 0 || c->seq <= 0)
        return false;
    if (c->dtype != FKV_F32 && c->dtype != FKV_F16 && c->dtype != FKV_BF16)
        return false;
    const int64_t esz = c->dtype == FKV_F32 ? 4 : 2;
    // head vectors start on 16-byte boundaries (vector loads and stores)
    if (reinterpret_cast<uintptr_t>(c->data) % 16)
        return false;
    const int64_t s[4] = {c->stride_layer, c->stride_batch, c->stride_head, c->stride_pos};
    for (int i = 0; i < 4; ++i)
        if (s[i] < 0 || (s[i] * esz) % 16)
            return false;
    (void)ctx;
    return true;
}

cudaStream_t as_stream(void *s) { return static_cast<cudaStream_t>(s); }

}  // namespace

// Both output views (either may be null) hold [t0, t0 + n_rec).
bool check_outputs(const fkv_ctx *ctx, const fkv_cache *k_out, const fkv_cache *v_out, int64_t n_rec, int64_t t0)
{
    const fkv_cache *outs[2] = {k_out, v_out};
    for (const fkv_cache *c : outs)
        if (c && (!check_cache(ctx, c) || t0 < 0 || t0 + n_rec > c->seq))
            return false;
    return true;
}

int decode_archive(fkv_ctx *ctx, const double *pts, int64_t n_streams, int64_t n_rec, int64_t pt_stride,
                   void *scratch, const fkv_cache *k_out, const fkv_cache *v_out, int64_t t0, cudaStream_t st)
{
    const int64_t stride = n_rec * fkv_record_len(ctx);
    CK(launch_span_decode_planar(ctx, pts, n_streams, n_rec, pt_stride, scratch, st), "span decode launch");
    const fkv_cache *outs[2] = {k_out, v_out};
    for (int kv = 0; kv < 2; ++kv)
        if (outs[kv])
            CK(launch_rvq_decode(ctx, kv, scratch, FKV_SYM_PLANAR, stride, n_rec, outs[kv], t0, st), "gather launch");
    return FKV_OK;
}

namespace {

// Geometry of a lossy archive: truncated spans T and code words per stream.
void lossy_geometry(const fkv_ctx *ctx, int64_t n, int bits, int64_t keep_exact, int64_t *T, int64_t *words,
                    int64_t *tail_spans)
{
    const int64_t spans = (n + ctx->L - 1) / ctx->L;
    *T = spans > keep_exact ? spans - keep_exact : 0;
    *words = (2 * *T * bits + 31) / 32;
    *tail_spans = spans - *T;
}

// Shared checks of the lossy calls; null on success, else the reason.
const char *check_lossy(const fkv_ctx *ctx, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                        const void *codes, int64_t code_stride, const void *tail, int64_t tail_stride, bool need_tail)
{
    if (n_streams < 0 || n < 0 || keep_exact < 0)
        return "negative size";
    if (bits < 2 || bits > 53)
        return "bits outside [2, 53]";
    int64_t T, words, tail_spans;
    lossy_geometry(ctx, n, bits, keep_exact, &T, &words, &tail_spans);
    if (n_streams > 0 && words > 0 && (!codes || code_stride < words || reinterpret_cast<uintptr_t>(codes) % 4))
        return "bad code buffer or stride";
    if (n_streams > 0 && tail_spans > 0 && (need_tail || tail) &&
        (!tail || tail_stride < tail_spans || reinterpret_cast<uintptr_t>(tail) % 16))
        return "bad tail buffer or stride";
    return nullptr;
}

}  // namespace

extern "C" {

double fkv_packing_ratio(int N)
{
    if (N < 3 || N > FKV_MAX_N)
        return 0.0;
    double s = 0.0;
    for (int k = 1; k <= N / 4; ++k) {
        double x, y;
        vertex(N, k, &x, &y);
        s += x;
    }
    return 1.0 / (2.0 * (1.0 + s));
}

int fkv_max_span_len(double r)
{
    if (!(r > 0.0 && r <= 0.5))
        return 0;
    return static_cast<int>(floor(44.0 / log2(1.0 / r)));
}

int fkv_create(int N, double r, int span_len, const fkv_codebooks *cb, fkv_ctx **out)
{
    if (!out)
        return FKV_EINVAL;
    *out = nullptr;
    fkv_ctx *ctx = new fkv_ctx();
    auto bail = [&](int code) {
        fkv_destroy(ctx);
        return code;
    };
    if (N < 3 || N > FKV_MAX_N)
        return bail(FKV_EINVAL);
    const double rN = fkv_packing_ratio(N);
    if (!(r > 0.0) || r > rN * (1.0 + 1e-12))
        return bail(FKV_EINVAL);
    const int Lmax = fkv_max_span_len(r);
    if (span_len < 1 || span_len > Lmax || span_len > 44)
        return bail(FKV_EINVAL);
    // the decoder tables must fit one block (always true: r <= r_N bounds
    // span_len by 44 / log2(1 / r_N), 6 symbols for every N > 256)
    if (codec_smem_bytes(N, span_len) > kMaxDynSmem)
        return bail(FKV_EINVAL);
    ctx->N = N;
    ctx->r = r;
    ctx->L = span_len;
    if (cudaGetDevice(&ctx->device) != cudaSuccess)
        return bail(FKV_ECUDA);

    // vertex table (the encoders give a symbol >= N a NaN vertex)
    std::vector<double2> V(N);
    for (int c = 0; c < N; ++c)
        vertex(N, c, &V[c].x, &V[c].y);
    // decoder constants: vertices in Q1.62 and float, the step table
    // T[j][c] = (1 - r) r^j V(c) in Q1.62, and the anchor limits 2^-4 r^m
    fkv_decconst dec;
    memset(&dec, 0, sizeof(dec));
    std::vector<longlong2> T(static_cast<size_t>(span_len) * N);
    for (int c = 0; c < N; ++c) {
        dec.vx[c] = q_round(V[c].x, 62);
        dec.vy[c] = q_round(V[c].y, 62);
        dec.vfx[c] = static_cast<float>(V[c].x);
        dec.vfy[c] = static_cast<float>(V[c].y);
    }
    long double rj = 1.0L;
    for (int j = 0; j < span_len; ++j) {
        const long double coef = (1.0L - static_cast<long double>(r)) * rj;
        for (int c = 0; c < N; ++c) {
            T[static_cast<size_t>(j) * N + c].x = q_round(coef * V[c].x, 62);
            T[static_cast<size_t>(j) * N + c].y = q_round(coef * V[c].y, 62);
        }
        rj *= static_cast<long double>(r);
    }
    rj = 1.0L;
    for (int m = 0; m < 48; ++m) {
        dec.alim[m] = q_round(0.0625L * rj, 62);
        rj *= static_cast<long double>(r);
    }
    // the fp32 sector angle's error, in sector widths: 1.2e-5 rad (arctangent
    // polynomial) + 1.5e-6 rad (direction, division, reflections), times
    // N / (2 pi), + N 2^-24 (scaling); fractions within twice that of a
    // boundary take the exact test
    const double sect_err = N * (1.2e-5 + 1.5e-6) / (2.0 * 3.14159265358979) + N * 0x1p-24;
    dec.sect_thr = static_cast<float>(0.5 - 2.0 * sect_err);
    CK(cudaMalloc(&ctx->d_V, N * sizeof(double2)), "vertex alloc");
    CK(cudaMemcpy(ctx->d_V, V.data(), N * sizeof(double2), cudaMemcpyHostToDevice), "vertex copy");
    CK(cudaMalloc(&ctx->d_dec, sizeof(fkv_decconst)), "decoder alloc");
    CK(cudaMemcpy(ctx->d_dec, &dec, sizeof(dec), cudaMemcpyHostToDevice), "decoder copy");
    CK(cudaMalloc(&ctx->d_T, T.size() * sizeof(longlong2)), "decoder alloc");
    CK(cudaMemcpy(ctx->d_T, T.data(), T.size() * sizeof(longlong2), cudaMemcpyHostToDevice), "decoder copy");
    CK(cudaMalloc(&ctx->d_status, sizeof(unsigned)), "status alloc");
    CK(cudaMemset(ctx->d_status, 0, sizeof(unsigned)), "status init");

    if (cb) {
        // the allocation-free archive read's fixed scratch: its address is
        // looked up here, so that call itself never loads a module
        const int src = static_scratch_resolve(ctx);
        if (src != FKV_OK)
            return bail(src);
        const int K = cb->codewords == 0 ? 256 : cb->codewords;
        const int smax = K == 256 ? 8 : 2;
        if (N != K || (K != 256 && K != 1024) || (cb->pooled != 0 && cb->pooled != 1) || cb->n_layers < 1 ||
            cb->n_heads < 1 || (cb->dim != 64 && cb->dim != 128) || (K == 1024 && cb->dim != 64) ||
            cb->stages_k < 1 || cb->stages_k > smax || cb->stages_v < 1 || cb->stages_v > smax || !cb->k ||
            !cb->v)
            return bail(FKV_EINVAL);
        if (cb->n_heads * (cb->stages_k + cb->stages_v) > 1024)
            return bail(FKV_EINVAL);
        ctx->has_cb = true;
        ctx->Ly = cb->n_layers;
        ctx->H = cb->n_heads;
        ctx->D = cb->dim;
        ctx->KC = K;
        ctx->pooled = cb->pooled != 0;
        int rc = upload_cbset(ctx, 0, cb->k, cb->stages_k);
        if (rc == FKV_OK)
            rc = upload_cbset(ctx, 1, cb->v, cb->stages_v);
        if (rc != FKV_OK)
            return bail(rc);
    }
    *out = ctx;
    return FKV_OK;
}

int fkv_destroy(fkv_ctx *ctx)
{
    if (!ctx)
        return FKV_OK;
    cudaDeviceSynchronize();
    cudaFree(ctx->d_V);
    cudaFree(ctx->d_dec);
    cudaFree(ctx->d_T);
    cudaFree(ctx->d_status);
    cudaFree(ctx->d_scratch);
    cudaFree(ctx->d_read_order);
    destroy_cbset(ctx->cb[0]);
    destroy_cbset(ctx->cb[1]);
    delete ctx;
    return FKV_OK;
}

int fkv_vertices(const fkv_ctx *ctx, double *out)
{
    if (!ctx || !out)
        return FKV_EINVAL;
    for (int c = 0; c < ctx->N; ++c)
        vertex(ctx->N, c, &out[2 * c], &out[2 * c + 1]);
    return FKV_OK;
}

int fkv_params(const fkv_ctx *ctx, int *N, double *r, int *span_len)
{
    if (!ctx)
        return FKV_EINVAL;
    if (N)
        *N = ctx->N;
    if (r)
        *r = ctx->r;
    if (span_len)
        *span_len = ctx->L;
    return FKV_OK;
}

int fkv_symbol_bytes(const fkv_ctx *ctx)
{
    return ctx ? sym_size(ctx) : 0;
}

const char *fkv_last_error(const fkv_ctx *ctx)
{
    return ctx ? ctx->err.c_str() : kNoCtx;
}

int fkv_sync_status(fkv_ctx *ctx, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    unsigned st = 0;
    CK(cudaStreamSynchronize(as_stream(stream)), "stream sync");
    CK(cudaMemcpy(&st, ctx->d_status, sizeof(st), cudaMemcpyDeviceToHost), "status read");
    CK(cudaMemset(ctx->d_status, 0, sizeof(unsigned)), "status clear");
    if (st & FKV_ST_TIMEOUT)
        return fail(ctx, FKV_ETIMEOUT, "a device wait timed out");
    if (st & FKV_ST_CORRUPT)
        return fail(ctx, FKV_ECORRUPT, "corrupt point or symbol (anchor check failed)");
    if (st & FKV_ST_RANGE)
        return fail(ctx, FKV_ERANGE, "a request named a position or stream outside the archive");
    return FKV_OK;
}

int fkv_span_encode(fkv_ctx *ctx, const void *sym_dev, int64_t n_streams, int64_t n,
                    int64_t sym_stride, double *pts_dev, int64_t pt_stride, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_streams < 0 || n < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (n_streams == 0 || n == 0)
        return FKV_OK;
    if (!sym_dev || !pts_dev || sym_stride < n || pt_stride < (n + ctx->L - 1) / ctx->L)
        return fail(ctx, FKV_EINVAL, "bad pointer or stride");
    if (reinterpret_cast<uintptr_t>(pts_dev) % 16)
        return fail(ctx, FKV_EINVAL, "points must be 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "uint16 symbols must be 2-byte aligned");
    CK(launch_span_encode(ctx, sym_dev, n_streams, n, sym_stride, pts_dev, pt_stride, as_stream(stream)),
       "span encode launch");
    return FKV_OK;
}

int fkv_span_decode(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n,
                    int64_t pt_stride, void *sym_dev, int64_t sym_stride, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_streams < 0 || n < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (n_streams == 0 || n == 0)
        return FKV_OK;
    if (!sym_dev || !pts_dev || sym_stride < n || pt_stride < (n + ctx->L - 1) / ctx->L)
        return fail(ctx, FKV_EINVAL, "bad pointer or stride");
    if (reinterpret_cast<uintptr_t>(pts_dev) % 16)
        return fail(ctx, FKV_EINVAL, "points must be 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "uint16 symbols must be 2-byte aligned");
    CK(launch_span_decode(ctx, pts_dev, n_streams, n, pt_stride, sym_dev, sym_stride, as_stream(stream)),
       "span decode launch");
    return FKV_OK;
}

int fkv_read(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n, int64_t pt_stride,
             const int64_t *req_dev, int64_t n_req, void *out_dev, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_req < 0 || n_streams < 0 || n < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (n_req == 0)
        return FKV_OK;
    if (!pts_dev || !req_dev || !out_dev || pt_stride < (n + ctx->L - 1) / ctx->L)
        return fail(ctx, FKV_EINVAL, "bad pointer or stride");
    if (reinterpret_cast<uintptr_t>(pts_dev) % 16 || reinterpret_cast<uintptr_t>(req_dev) % 8 ||
        reinterpret_cast<uintptr_t>(out_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "misaligned buffer");
    CK(launch_read(ctx, pts_dev, n_streams, n, pt_stride, req_dev, n_req, out_dev, as_stream(stream)),
       "read launch");
    return FKV_OK;
}

namespace {

// Host checks shared by the ragged calls (the offsets themselves live on the
// device and are checked there).
const char *check_ragged(const fkv_ctx *ctx, const void *sym, const int64_t *so, int64_t n_streams,
                         const double *pts, const int64_t *po)
{
    if (n_streams < 0)
        return "negative stream count";
    if (!so || !po || (n_streams > 0 && (!sym || !pts)))
        return "null pointer";
    if (reinterpret_cast<uintptr_t>(so) % 8 || reinterpret_cast<uintptr_t>(po) % 8)
        return "offset arrays must be 8-byte aligned";
    if (reinterpret_cast<uintptr_t>(pts) % 16)
        return "points must be 16-byte aligned";
    if (reinterpret_cast<uintptr_t>(sym) % sym_size(ctx))
        return "uint16 symbols must be 2-byte aligned";
    return nullptr;
}

}  // namespace

int fkv_span_encode_ragged(fkv_ctx *ctx, const void *sym_dev, const int64_t *sym_off_dev, int64_t n_streams,
                           double *pts_dev, const int64_t *pt_off_dev, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (const char *why = check_ragged(ctx, sym_dev, sym_off_dev, n_streams, pts_dev, pt_off_dev))
        return fail(ctx, FKV_EINVAL, why);
    if (n_streams == 0)
        return FKV_OK;
    CK(launch_span_encode_ragged(ctx, sym_dev, sym_off_dev, n_streams, pts_dev, pt_off_dev, as_stream(stream)),
       "ragged span encode launch");
    return FKV_OK;
}

int fkv_span_decode_ragged(fkv_ctx *ctx, const double *pts_dev, const int64_t *pt_off_dev, int64_t n_streams,
                           void *sym_dev, const int64_t *sym_off_dev, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (const char *why = check_ragged(ctx, sym_dev, sym_off_dev, n_streams, pts_dev, pt_off_dev))
        return fail(ctx, FKV_EINVAL, why);
    if (n_streams == 0)
        return FKV_OK;
    CK(launch_span_decode_ragged(ctx, pts_dev, pt_off_dev, n_streams, sym_dev, sym_off_dev, as_stream(stream)),
       "ragged span decode launch");
    return FKV_OK;
}

int fkv_read_ragged(fkv_ctx *ctx, const double *pts_dev, const int64_t *pt_off_dev, const int64_t *sym_off_dev,
                    int64_t n_streams, const int64_t *req_dev, int64_t n_req, void *out_dev, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_req < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (n_req == 0)
        return FKV_OK;
    if (const char *why = check_ragged(ctx, out_dev, sym_off_dev, n_streams, pts_dev, pt_off_dev))
        return fail(ctx, FKV_EINVAL, why);
    if (!req_dev || !out_dev || reinterpret_cast<uintptr_t>(req_dev) % 8)
        return fail(ctx, FKV_EINVAL, "bad request buffer");
    CK(launch_read_ragged(ctx, pts_dev, pt_off_dev, sym_off_dev, n_streams, req_dev, n_req, out_dev,
                          as_stream(stream)),
       "ragged read launch");
    return FKV_OK;
}

int fkv_suffix_search(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n, int64_t pt_stride,
                      const void *query, int qlen, int64_t *match_dev, int64_t cap, int64_t *counts_dev,
                      void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_streams < 0 || n < 0 || cap < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (qlen < 1 || qlen > ctx->L || !query)
        return fail(ctx, FKV_EINVAL, "query length outside [1, span_len]");
    uint16_t q16[64];
    for (int i = 0; i < qlen; ++i) {
        q16[i] = ctx->N > 256 ? static_cast<const uint16_t *>(query)[i] : static_cast<const uint8_t *>(query)[i];
        if (q16[i] >= ctx->N)
            return fail(ctx, FKV_EINVAL, "query symbol outside the alphabet");
    }
    if (!counts_dev || (cap > 0 && !match_dev) || (n_streams > 0 && n > 0 && !pts_dev) ||
        pt_stride < (n + ctx->L - 1) / ctx->L)
        return fail(ctx, FKV_EINVAL, "bad pointer or stride");
    if (reinterpret_cast<uintptr_t>(pts_dev) % 16 || reinterpret_cast<uintptr_t>(match_dev) % 8 ||
        reinterpret_cast<uintptr_t>(counts_dev) % 8)
        return fail(ctx, FKV_EINVAL, "misaligned buffer");
    CK(launch_suffix_search(ctx, pts_dev, n_streams, n, pt_stride, q16, qlen, match_dev, cap, counts_dev,
                            as_stream(stream)),
       "suffix search launch");
    return FKV_OK;
}


int fkv_truncate(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n, int64_t pt_stride, int bits,
                 int64_t keep_exact, uint32_t *codes_dev, int64_t code_stride, double *tail_dev, int64_t tail_stride,
                 void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (const char *why = check_lossy(ctx, n_streams, n, bits, keep_exact, codes_dev, code_stride, tail_dev,
                                      tail_stride, false))
        return fail(ctx, FKV_EINVAL, why);
    if (n_streams == 0 || n == 0)
        return FKV_OK;
    if (!pts_dev || pt_stride < (n + ctx->L - 1) / ctx->L || reinterpret_cast<uintptr_t>(pts_dev) % 16)
        return fail(ctx, FKV_EINVAL, "bad point buffer or stride");
    CK(launch_truncate(ctx, pts_dev, n_streams, n, pt_stride, bits, keep_exact, codes_dev, code_stride, tail_dev,
                       tail_stride, as_stream(stream)),
       "truncate launch");
    return FKV_OK;
}

int fkv_lossy_decode(fkv_ctx *ctx, const uint32_t *codes_dev, int64_t code_stride, const double *tail_dev,
                     int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact, void *sym_dev,
                     int64_t sym_stride, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (const char *why = check_lossy(ctx, n_streams, n, bits, keep_exact, codes_dev, code_stride, tail_dev,
                                      tail_stride, true))
        return fail(ctx, FKV_EINVAL, why);
    if (n_streams == 0 || n == 0)
        return FKV_OK;
    if (!sym_dev || sym_stride < n || reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "bad symbol buffer or stride");
    CK(launch_lossy_decode(ctx, codes_dev, code_stride, tail_dev, tail_stride, n_streams, n, bits, keep_exact,
                           sym_dev, sym_stride, as_stream(stream)),
       "lossy decode launch");
    return FKV_OK;
}

int fkv_lossy_read(fkv_ctx *ctx, const uint32_t *codes_dev, int64_t code_stride, const double *tail_dev,
                   int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                   const int64_t *req_dev, int64_t n_req, void *out_dev, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_req < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (const char *why = check_lossy(ctx, n_streams, n, bits, keep_exact, codes_dev, code_stride, tail_dev,
                                      tail_stride, true))
        return fail(ctx, FKV_EINVAL, why);
    if (n_req == 0)
        return FKV_OK;
    if (!req_dev || !out_dev || reinterpret_cast<uintptr_t>(req_dev) % 8 ||
        reinterpret_cast<uintptr_t>(out_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "bad request or output buffer");
    CK(launch_lossy_read(ctx, codes_dev, code_stride, tail_dev, tail_stride, n_streams, n, bits, keep_exact, req_dev,
                         n_req, out_dev, as_stream(stream)),
       "lossy read launch");
    return FKV_OK;
}

int64_t fkv_ac_capacity_words(const fkv_ctx *ctx, int64_t n)
{
    if (!ctx || n < 0)
        return 0;
    return ac_capacity_words(ctx->N, n);
}

int fkv_ac_encode(fkv_ctx *ctx, const void *sym_dev, int64_t n_streams, int64_t n, int64_t sym_stride, int adaptive,
                  uint32_t *words_dev, int64_t word_stride, int64_t *nbits_dev, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_streams < 0 || n < 0 || n >= (int64_t(1) << 29))
        return fail(ctx, FKV_EINVAL, "size outside [0, 2^29)");
    if (adaptive != 0 && adaptive != 1)
        return fail(ctx, FKV_EINVAL, "adaptive must be 0 or 1");
    if (n_streams == 0)
        return FKV_OK;
    if ((n > 0 && (!sym_dev || sym_stride < n || reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))) ||
        !words_dev || word_stride < ac_capacity_words(ctx->N, n) || reinterpret_cast<uintptr_t>(words_dev) % 4 ||
        !nbits_dev || reinterpret_cast<uintptr_t>(nbits_dev) % 8)
        return fail(ctx, FKV_EINVAL, "bad buffer, stride or alignment");
    CK(launch_ac_encode(ctx, sym_dev, n_streams, n, sym_stride, adaptive, words_dev, word_stride, nbits_dev,
                        as_stream(stream)),
       "arithmetic encode launch");
    return FKV_OK;
}

int fkv_ac_decode(fkv_ctx *ctx, const uint32_t *words_dev, int64_t word_stride, const int64_t *nbits_dev,
                  int64_t n_streams, int64_t n, int adaptive, void *sym_dev, int64_t sym_stride, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (n_streams < 0 || n < 0 || n >= (int64_t(1) << 29))
        return fail(ctx, FKV_EINVAL, "size outside [0, 2^29)");
    if (adaptive != 0 && adaptive != 1)
        return fail(ctx, FKV_EINVAL, "adaptive must be 0 or 1");
    if (n_streams == 0 || n == 0)
        return FKV_OK;
    if (!sym_dev || sym_stride < n || reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx) || !words_dev ||
        word_stride < 1 || reinterpret_cast<uintptr_t>(words_dev) % 4 || !nbits_dev ||
        reinterpret_cast<uintptr_t>(nbits_dev) % 8)
        return fail(ctx, FKV_EINVAL, "bad buffer, stride or alignment");
    CK(launch_ac_decode(ctx, words_dev, word_stride, nbits_dev, n_streams, n, adaptive, sym_dev, sym_stride,
                        as_stream(stream)),
       "arithmetic decode launch");
    return FKV_OK;
}

int fkv_measure_fp64_rate(double *ops_per_s, void *stream)
{
    if (!ops_per_s)
        return FKV_EINVAL;
    *ops_per_s = 0.0;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return FKV_ECUDA;
    return measure_fp64_rate(dev, as_stream(stream), ops_per_s) == cudaSuccess ? FKV_OK : FKV_ECUDA;
}

int fkv_check_bounded_wait(fkv_ctx *ctx, int64_t limit_ns, int32_t *result, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!result)
        return fail(ctx, FKV_EINVAL, "null result");
    if (limit_ns < 100000 || limit_ns > 1000000000)
        return fail(ctx, FKV_EINVAL, "limit_ns outside [1e5, 1e9]");
    cudaStream_t st = as_stream(stream);
    int *d = nullptr;
    CK(cudaMalloc(&d, 6 * sizeof(int)), "wait check: malloc");
    cudaError_t e = cudaMemsetAsync(d, 0, 6 * sizeof(int), st);
    if (e == cudaSuccess)
        e = launch_wait_check(ctx->d_status, static_cast<uint64_t>(limit_ns), d, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(result, d, 6 * sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess)
        e = cudaStreamSynchronize(st);
    const cudaError_t ef = cudaFree(d);
    CK(e, "wait check");
    CK(ef, "wait check: free");
    return FKV_OK;
}

int fkv_record_len(const fkv_ctx *ctx)
{
    if (!ctx || !ctx->has_cb)
        return 0;
    return ctx->H * (ctx->cb[0].stages + ctx->cb[1].stages);
}

int fkv_rvq_encode(fkv_ctx *ctx, int kv, const fkv_cache *x, int64_t t0, int64_t t1, void *sym_dev,
                   int64_t stream_stride, int64_t rec0, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!ctx->has_cb)
        return fail(ctx, FKV_EINVAL, "context has no codebooks");
    if (kv != 0 && kv != 1)
        return fail(ctx, FKV_EINVAL, "kv must be 0 (keys) or 1 (values)");
    if (!check_cache(ctx, x))
        return fail(ctx, FKV_EINVAL, "bad cache view (dtype, alignment or strides)");
    if (t0 < 0 || t1 < t0 || t1 > x->seq || rec0 < 0 || !sym_dev)
        return fail(ctx, FKV_EINVAL, "bad position range");
    if (reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "uint16 symbols must be 2-byte aligned");
    if (t1 == t0)
        return FKV_OK;
    const int64_t R = fkv_record_len(ctx);
    if (stream_stride < (rec0 + (t1 - t0)) * R)
        return fail(ctx, FKV_EINVAL, "stream stride too small for the records");
    CK(launch_rvq_encode(ctx, kv, x, t0, t1, sym_dev, stream_stride, rec0, as_stream(stream)),
       "rvq encode launch");
    return FKV_OK;
}

int fkv_rvq_decode(fkv_ctx *ctx, const void *sym_dev, int64_t stream_stride, int64_t n_rec,
                   fkv_cache *k_out, fkv_cache *v_out, int64_t t0, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!ctx->has_cb)
        return fail(ctx, FKV_EINVAL, "context has no codebooks");
    if (!sym_dev || n_rec < 0 || t0 < 0 || reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))
        return fail(ctx, FKV_EINVAL, "bad arguments");
    const int64_t R = fkv_record_len(ctx);
    if (stream_stride < n_rec * R)
        return fail(ctx, FKV_EINVAL, "stream stride too small for the records");
    if (!check_outputs(ctx, k_out, v_out, n_rec, t0))
        return fail(ctx, FKV_EINVAL, "bad output cache view");
    if (n_rec == 0)
        return FKV_OK;
    fkv_cache *outs[2] = {k_out, v_out};
    for (int kv = 0; kv < 2; ++kv)
        if (outs[kv])
            CK(launch_rvq_decode(ctx, kv, sym_dev, FKV_SYM_RECORDS, stream_stride, n_rec, outs[kv], t0,
                                 as_stream(stream)),
               "gather launch");
    return FKV_OK;
}

int fkv_decode_kv(fkv_ctx *ctx, const double *pts_dev, int64_t n_rec, int64_t pt_stride, fkv_cache *k_out,
                  fkv_cache *v_out, int64_t t0, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!ctx->has_cb)
        return fail(ctx, FKV_EINVAL, "context has no codebooks");
    const fkv_cache *ref = k_out ? k_out : v_out;
    if (!ref || !pts_dev || n_rec < 0)
        return fail(ctx, FKV_EINVAL, "bad arguments");
    if (k_out && v_out && k_out->batch != v_out->batch)
        return fail(ctx, FKV_EINVAL, "K and V batch differ");
    // every view is checked before anything is launched
    if (!check_outputs(ctx, k_out, v_out, n_rec, t0))
        return fail(ctx, FKV_EINVAL, "bad output cache view");
    if (n_rec == 0)
        return FKV_OK;
    const int64_t R = fkv_record_len(ctx);
    const int64_t n_streams = ref->batch * ctx->Ly;
    const int64_t n = n_rec * R;
    if (pt_stride < (n + ctx->L - 1) / ctx->L || reinterpret_cast<uintptr_t>(pts_dev) % 16)
        return fail(ctx, FKV_EINVAL, "bad point stride or alignment");
    const size_t need = static_cast<size_t>(n_streams) * static_cast<size_t>(n) * sym_size(ctx);
    if (need > ctx->scratch_bytes) {
        CK(cudaStreamSynchronize(as_stream(stream)), "scratch sync");
        cudaFree(ctx->d_scratch);
        ctx->d_scratch = nullptr;
        ctx->scratch_bytes = 0;
        CK(cudaMalloc(&ctx->d_scratch, need), "scratch alloc");
        ctx->scratch_bytes = need;
    }
    return decode_archive(ctx, pts_dev, n_streams, n_rec, pt_stride, ctx->d_scratch, k_out, v_out, t0,
                          as_stream(stream));
}

int fkv_cache_upload(fkv_ctx *ctx, const fkv_cache *src_host, const fkv_cache *dst_dev, int64_t t0, int64_t t1,
                     void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!ctx->has_cb)
        return fail(ctx, FKV_EINVAL, "context has no codebooks");
    if (!src_host || !dst_dev || !src_host->data || !dst_dev->data || src_host->dtype != dst_dev->dtype ||
        src_host->batch != dst_dev->batch || src_host->batch <= 0)
        return fail(ctx, FKV_EINVAL, "bad cache views");
    if (t0 < 0 || t1 < t0 || t1 > src_host->seq || t1 > dst_dev->seq)
        return fail(ctx, FKV_EINVAL, "bad position range");
    const int64_t D = ctx->D;
    if (src_host->stride_pos != D || dst_dev->stride_pos != D)
        return fail(ctx, FKV_EINVAL, "positions must be contiguous (stride_pos = dim)");
    if (t1 == t0)
        return FKV_OK;
    const int64_t esz = src_host->dtype == FKV_F32 ? 4 : 2;
    const int64_t L = ctx->Ly, B = src_host->batch, H = ctx->H;
    const int64_t width = (t1 - t0) * D * esz;
    const uint8_t *s = static_cast<const uint8_t *>(src_host->data);
    uint8_t *d = static_cast<uint8_t *>(dst_dev->data);
    auto uniform = [&](const fkv_cache *c) {
        return c->stride_batch == H * c->stride_head && c->stride_layer == B * c->stride_batch;
    };
    if (uniform(src_host) && uniform(dst_dev)) {
        // every (layer, sequence, head) row at one pitch: a single 2-D copy
        CK(cudaMemcpy2DAsync(d + t0 * D * esz, dst_dev->stride_head * esz, s + t0 * D * esz,
                             src_host->stride_head * esz, width, L * B * H, cudaMemcpyHostToDevice,
                             as_stream(stream)),
           "cache upload");
        return FKV_OK;
    }
    for (int64_t l = 0; l < L; ++l)
        for (int64_t b = 0; b < B; ++b)
            CK(cudaMemcpy2DAsync(d + (l * dst_dev->stride_layer + b * dst_dev->stride_batch + t0 * D) * esz,
                                 dst_dev->stride_head * esz,
                                 s + (l * src_host->stride_layer + b * src_host->stride_batch + t0 * D) * esz,
                                 src_host->stride_head * esz, width, H, cudaMemcpyHostToDevice, as_stream(stream)),
               "cache upload");
    return FKV_OK;
}

int fkv_read_kv(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n_rec, int64_t pt_stride,
                const int64_t *req_dev, int64_t n_req, void *out_dev, int dtype, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!ctx->has_cb)
        return fail(ctx, FKV_EINVAL, "context has no codebooks");
    if (n_req < 0 || n_streams < 0 || n_rec < 0)
        return fail(ctx, FKV_EINVAL, "negative size");
    if (n_req == 0)
        return FKV_OK;
    if (!pts_dev || !req_dev || !out_dev || (dtype != FKV_F32 && dtype != FKV_F16 && dtype != FKV_BF16))
        return fail(ctx, FKV_EINVAL, "bad arguments");
    const int64_t R = fkv_record_len(ctx);
    if (pt_stride < (n_rec * R + ctx->L - 1) / ctx->L)
        return fail(ctx, FKV_EINVAL, "point stride too small");
    if (reinterpret_cast<uintptr_t>(out_dev) % 16 || reinterpret_cast<uintptr_t>(pts_dev) % 16)
        return fail(ctx, FKV_EINVAL, "misaligned buffer");
    const size_t need = static_cast<size_t>(read_order_ints(ctx, n_req)) * sizeof(int);
    if (need > ctx->read_order_bytes) {
        CK(cudaStreamSynchronize(as_stream(stream)), "read order sync");
        cudaFree(ctx->d_read_order);
        ctx->d_read_order = nullptr;
        ctx->read_order_bytes = 0;
        CK(cudaMalloc(&ctx->d_read_order, need), "read order alloc");
        ctx->read_order_bytes = need;
    }
    CK(launch_read_kv(ctx, pts_dev, n_streams, n_rec, pt_stride, req_dev, n_req, out_dev, dtype,
                      need ? ctx->d_read_order : nullptr, as_stream(stream)),
       "read_kv launch");
    return FKV_OK;
}

int fkv_streams_create(fkv_ctx *ctx, int64_t n_streams, int64_t capacity_symbols, fkv_streams **out)
{
    if (!ctx || !out)
        return FKV_EINVAL;
    *out = nullptr;
    if (n_streams < 1 || capacity_symbols < 0)
        return fail(ctx, FKV_EINVAL, "bad stream-set size");
    fkv_streams *s = new fkv_streams();
    s->ctx = ctx;
    s->n_streams = n_streams;
    s->cap_spans = capacity_symbols / ctx->L + 1;
    cudaError_t e = cudaMalloc(&s->d_pts, static_cast<size_t>(n_streams) * s->cap_spans * 16);
    if (e != cudaSuccess) {
        delete s;
        return cuda_fail(ctx, e, "stream alloc");
    }
    *out = s;
    return FKV_OK;
}

int fkv_streams_destroy(fkv_streams *s)
{
    if (!s)
        return FKV_OK;
    cudaDeviceSynchronize();
    cudaFree(s->d_pts);
    delete s;
    return FKV_OK;
}

int fkv_streams_reset(fkv_streams *s)
{
    if (!s)
        return FKV_EINVAL;
    s->length = 0;
    return FKV_OK;
}

int fkv_streams_info(const fkv_streams *s, int64_t *n_streams, int64_t *length, int64_t *pt_stride,
                     double **pts_dev)
{
    if (!s)
        return FKV_EINVAL;
    if (n_streams)
        *n_streams = s->n_streams;
    if (length)
        *length = s->length;
    if (pt_stride)
        *pt_stride = s->cap_spans;
    if (pts_dev)
        *pts_dev = s->d_pts;
    return FKV_OK;
}

int fkv_append(fkv_ctx *ctx, fkv_streams *s, const void *sym_dev, int64_t m, int64_t sym_stride,
               void *stream)
{
    if (!ctx || !s || s->ctx != ctx)
        return fail(ctx, FKV_EINVAL, "bad stream set");
    if (m < 0 || (m > 0 && (!sym_dev || sym_stride < m || reinterpret_cast<uintptr_t>(sym_dev) % sym_size(ctx))))
        return fail(ctx, FKV_EINVAL, "bad symbols");
    if (m == 0)
        return FKV_OK;
    const int64_t n_new = s->length + m;
    const int64_t need = (n_new + ctx->L - 1) / ctx->L;
    if (need > s->cap_spans) {
        int64_t cap = s->cap_spans * 2;
        if (cap < need)
            cap = need;
        double *np = nullptr;
        CK(cudaMalloc(&np, static_cast<size_t>(s->n_streams) * cap * 16), "stream grow");
        const int64_t used = (s->length + ctx->L - 1) / ctx->L;
        cudaError_t e = cudaSuccess;
        if (used > 0)
            e = cudaMemcpy2DAsync(np, cap * 16, s->d_pts, s->cap_spans * 16, used * 16, s->n_streams,
                                  cudaMemcpyDeviceToDevice, as_stream(stream));
        if (e == cudaSuccess)
            e = cudaStreamSynchronize(as_stream(stream));
        if (e != cudaSuccess) {
            // the set keeps its old buffer; the new one is given back
            cudaFree(np);
            return cuda_fail(ctx, e, "stream grow copy");
        }
        cudaFree(s->d_pts);
        s->d_pts = np;
        s->cap_spans = cap;
    }
    CK(launch_append(ctx, s->d_pts, s->n_streams, s->cap_spans, s->length, sym_dev, m, sym_stride,
                     as_stream(stream)),
       "append launch");
    s->length = n_new;
    return FKV_OK;
}

int fkv_streams_export(const fkv_streams *s, int64_t *length, double *host_pts, void *stream)
{
    if (!s)
        return FKV_EINVAL;
    fkv_ctx *ctx = s->ctx;
    const int64_t used = (s->length + ctx->L - 1) / ctx->L;
    if (length)
        *length = s->length;
    if (host_pts && used > 0) {
        CK(cudaMemcpy2DAsync(host_pts, used * 16, s->d_pts, s->cap_spans * 16, used * 16, s->n_streams,
                             cudaMemcpyDeviceToHost, as_stream(stream)),
           "export copy");
        CK(cudaStreamSynchronize(as_stream(stream)), "export sync");
    }
    return FKV_OK;
}

int fkv_streams_import(fkv_ctx *ctx, int64_t n_streams, int64_t length, const double *host_pts,
                       fkv_streams **out)
{
    if (!ctx || !out || length < 0 || (length > 0 && !host_pts))
        return fail(ctx, FKV_EINVAL, "bad import arguments");
    int rc = fkv_streams_create(ctx, n_streams, length, out);
    if (rc != FKV_OK)
        return rc;
    fkv_streams *s = *out;
    const int64_t used = (length + ctx->L - 1) / ctx->L;
    if (used > 0) {
        cudaError_t e = cudaMemcpy2D(s->d_pts, s->cap_spans * 16, host_pts, used * 16, used * 16, n_streams,
                                     cudaMemcpyHostToDevice);
        if (e != cudaSuccess) {
            fkv_streams_destroy(s);
            *out = nullptr;
            return cuda_fail(ctx, e, "import copy");
        }
    }
    s->length = length;
    return FKV_OK;
}

}  // extern "C"
