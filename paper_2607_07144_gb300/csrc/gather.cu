// Codebook gather: K/V reconstruction from RVQ indices (Sec. 3 "Setup": the
// reconstruction is the sum of the selected centroids), for whole archives
// and for random record reads (Sec. 2).
//
// Whole archive: a block owns one codebook group (layer, head), a slice of
// the head dimension and a run of vectors; the group's float32 codebooks for
// that slice sit in shared memory, so HBM sees only the index bytes in and
// the rebuilt K/V out.  Sums run in float32, stage order, then round to
// nearest-even into the cache dtype.
#include "fkv_internal.h"

namespace {

constexpr int kThreads = 256;
constexpr int kSmemBudget = 64 * 1024;   // codebook slice per block
constexpr int64_t kChunk = 4096;         // vectors per block

struct GatherArgs {
    const uint8_t *sym;
    int64_t stream_stride, n_rec, batch, t0;
    int n_layers, n_heads, D, S, R, kv_off;
    const float *cb32;     // [Ly*H][S][256][D]
    void *out;
    int dtype;
    int64_t s_layer, s_batch, s_head, s_pos;
    int parts, Dp, chunks;
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

__global__ void __launch_bounds__(kThreads) k_gather(const GatherArgs a)
{
    extern __shared__ __align__(16) float scb[];   // [S][256][Dp]
    const int chunk = blockIdx.x % a.chunks;
    const int part = (blockIdx.x / a.chunks) % a.parts;
    const int g = blockIdx.x / (a.chunks * a.parts);
    const int l = g / a.n_heads, h = g % a.n_heads;
    const int Dp = a.Dp, S = a.S, D = a.D;
    const int d0 = part * Dp;
    // codebook slice -> shared memory (float4 granules; Dp is a multiple of 4)
    const float *src = a.cb32 + static_cast<int64_t>(g) * S * 256 * D;
    const int q4 = Dp / 4;
    for (int i = threadIdx.x; i < S * 256 * q4; i += kThreads) {
        const int row = i / q4, q = i - row * q4;
        reinterpret_cast<float4 *>(scb)[i] = __ldg(reinterpret_cast<const float4 *>(src + static_cast<int64_t>(row) * D + d0) + q);
    }
    __syncthreads();
    const int tpv = Dp / 2;                  // threads per vector (two dims each)
    const int vpi = kThreads / tpv;          // vectors per pass
    const int dd = (threadIdx.x % tpv) * 2;
    const int64_t nvec = a.batch * a.n_rec;
    const int64_t v_beg = static_cast<int64_t>(chunk) * kChunk;
    const int64_t v_end = min(nvec, v_beg + kChunk);
    for (int64_t v = v_beg + threadIdx.x / tpv; v < v_end; v += vpi) {
        const int64_t b = v / a.n_rec;
        const int64_t rec = v - b * a.n_rec;
        const uint8_t *ids = a.sym + (b * a.n_layers + l) * a.stream_stride + rec * a.R + a.kv_off + h * S;
        float x = 0.0f, y = 0.0f;
        for (int s = 0; s < S; ++s) {
            const float2 c = *reinterpret_cast<const float2 *>(scb + (s * 256 + ids[s]) * Dp + dd);
            x += c.x;
            y += c.y;
        }
        const int64_t e = l * a.s_layer + b * a.s_batch + h * a.s_head + (a.t0 + rec) * a.s_pos + d0 + dd;
        store2(a.out, a.dtype, e, x, y);
    }
}

// ------------------------------------------------------- random reads ---
struct DecTables {
    long long vx[256], vy[256], wx[256], wy[256], hn[256];
};

__device__ __forceinline__ long long vscore(const DecTables &d, long long X, long long Y, int c)
{
    return __mul64hi(X, d.vx[c]) + __mul64hi(Y, d.vy[c]) - d.hn[c];
}

__device__ __forceinline__ int classify(const DecTables &d, long long X, long long Y, int N)
{
    if (N <= 8) {
        int best = 0;
        long long bs = vscore(d, X, Y, 0);
        for (int c = 1; c < N; ++c) {
            const long long s = vscore(d, X, Y, c);
            if (s > bs) {
                bs = s;
                best = c;
            }
        }
        return best;
    }
    const float xf = static_cast<float>(static_cast<int>(X >> 32));
    const float yf = static_cast<float>(static_cast<int>(Y >> 32));
    int c0 = __float2int_rn(atan2f(yf, xf) * (static_cast<float>(N) * 0.15915494309189535f));
    if (c0 < 0)
        c0 += N;
    if (c0 >= N)
        c0 -= N;
    const int cm = c0 == 0 ? N - 1 : c0 - 1;
    const int cp = c0 == N - 1 ? 0 : c0 + 1;
    int best = c0;
    long long bs = vscore(d, X, Y, c0);
    long long s = vscore(d, X, Y, cm);
    if (s > bs) {
        bs = s;
        best = cm;
    }
    s = vscore(d, X, Y, cp);
    if (s > bs)
        best = cp;
    return best;
}

__device__ __forceinline__ long long mulshift(long long v, long long rinv, int k)
{
    const unsigned long long lo = static_cast<unsigned long long>(v) * static_cast<unsigned long long>(rinv);
    const long long hi = __mul64hi(v, rinv);
    return static_cast<long long>((lo >> k) | (static_cast<unsigned long long>(hi) << (64 - k)));
}

constexpr int kReadWarps = 8;
constexpr int kMaxRecord = 1024;

struct ReadArgs {
    const double2 *pts;
    int64_t n_streams, n_rec, pt_stride;
    const int64_t *req;
    int64_t n_req;
    void *out;
    int dtype;
    int n_layers, n_heads, D, SK, SV, R, N, L;
    const float *cbk, *cbv;
    const fkv_decconst *dec;
    unsigned *status;
};

// One warp per request: its lanes decode the spans covering the record into
// shared memory, then gather the record's 2 * H head vectors.
__global__ void __launch_bounds__(kReadWarps * 32) k_read_kv(const ReadArgs a)
{
    __shared__ DecTables sd;
    __shared__ uint8_t srec[kReadWarps][kMaxRecord];
    for (int i = threadIdx.x; i < 256; i += blockDim.x) {
        sd.vx[i] = a.dec->vx[i];
        sd.vy[i] = a.dec->vy[i];
        sd.wx[i] = a.dec->wx[i];
        sd.wy[i] = a.dec->wy[i];
        sd.hn[i] = a.dec->hn[i];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t q = static_cast<int64_t>(blockIdx.x) * kReadWarps + warp;
    if (q >= a.n_req)
        return;
    const long long rinv = a.dec->rinv;
    const int rsh = a.dec->rshift;
    const int64_t st = a.req[2 * q], rec = a.req[2 * q + 1];
    const int H = a.n_heads, D = a.D, R = a.R, L = a.L;
    const int64_t out_vec = static_cast<int64_t>(2) * H * D;
    if (st < 0 || st >= a.n_streams || rec < 0 || rec >= a.n_rec) {
        for (int64_t i = lane; i < out_vec / 2; i += 32)
            store2(a.out, a.dtype, q * out_vec + 2 * i, 0.0f, 0.0f);
        if (lane == 0)
            atomicOr(a.status, FKV_ST_CORRUPT);
        return;
    }
    const int64_t n = a.n_rec * R;
    const int64_t sym0 = rec * R;
    const int64_t u0 = sym0 / L, u1 = (sym0 + R - 1) / L;
    uint8_t *my = srec[warp];
    bool bad = false;
    for (int64_t u = u0 + lane; u <= u1; u += 32) {
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
        const double2 p = a.pts[st * a.pt_stride + u];
        long long X = __double2ll_rn(p.x * 4611686018427387904.0);
        long long Y = __double2ll_rn(p.y * 4611686018427387904.0);
        for (int k = m - 1; k >= 0; --k) {
            const int c = classify(sd, X, Y, a.N);
            const int64_t pos = u * L + k - sym0;
            if (pos >= 0 && pos < R)
                my[pos] = static_cast<uint8_t>(c);
            X = mulshift(static_cast<long long>(static_cast<unsigned long long>(X) - static_cast<unsigned long long>(sd.wx[c])), rinv, rsh);
            Y = mulshift(static_cast<long long>(static_cast<unsigned long long>(Y) - static_cast<unsigned long long>(sd.wy[c])), rinv, rsh);
        }
        const long long lim = 1ll << 58;
        bad |= X > lim || X < -lim || Y > lim || Y < -lim;
    }
    if (bad)
        atomicOr(a.status, FKV_ST_CORRUPT);
    __syncwarp();
    const int l = static_cast<int>(st % a.n_layers);
    for (int kv = 0; kv < 2; ++kv) {
        const int S = kv == 0 ? a.SK : a.SV;
        const float *cb = kv == 0 ? a.cbk : a.cbv;
        const int off = kv == 0 ? 0 : H * a.SK;
        for (int hh = 0; hh < H; ++hh) {
            const float *gcb = cb + (static_cast<int64_t>(l) * H + hh) * S * 256 * D;
            const int64_t obase = q * out_vec + (static_cast<int64_t>(kv) * H + hh) * D;
            for (int d = lane * 2; d < D; d += 64) {
                float x = 0.0f, y = 0.0f;
                for (int s = 0; s < S; ++s) {
                    const float2 c = __ldg(reinterpret_cast<const float2 *>(
                        gcb + (static_cast<int64_t>(s) * 256 + my[off + hh * S + s]) * D + d));
                    x += c.x;
                    y += c.y;
                }
                store2(a.out, a.dtype, obase + d, x, y);
            }
        }
    }
}

}  // namespace

cudaError_t launch_rvq_decode(const fkv_ctx *c, int kv, const uint8_t *sym, int64_t stream_stride,
                              int64_t n_rec, const fkv_cache *out, int64_t t0, cudaStream_t st)
{
    const fkv_cbset &cb = c->cb[kv];
    GatherArgs a;
    a.sym = sym;
    a.stream_stride = stream_stride;
    a.n_rec = n_rec;
    a.batch = out->batch;
    a.t0 = t0;
    a.n_layers = c->Ly;
    a.n_heads = c->H;
    a.D = c->D;
    a.S = cb.stages;
    a.R = c->H * (c->cb[0].stages + c->cb[1].stages);
    a.kv_off = kv == 0 ? 0 : c->H * c->cb[0].stages;
    a.cb32 = cb.cb32;
    a.out = out->data;
    a.dtype = out->dtype;
    a.s_layer = out->stride_layer;
    a.s_batch = out->stride_batch;
    a.s_head = out->stride_head;
    a.s_pos = out->stride_pos;
    int parts = 1;
    while (static_cast<int64_t>(a.S) * 256 * (c->D / parts) * 4 > kSmemBudget && c->D / parts > 4)
        parts *= 2;
    a.parts = parts;
    a.Dp = c->D / parts;
    const int64_t nvec = a.batch * n_rec;
    if (nvec <= 0)
        return cudaSuccess;
    const int64_t chunks = (nvec + kChunk - 1) / kChunk;
    const int64_t blocks = chunks * parts * c->Ly * c->H;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    a.chunks = static_cast<int>(chunks);
    const size_t smem = static_cast<size_t>(a.S) * 256 * a.Dp * 4;
    cudaError_t e = cudaFuncSetAttribute(k_gather, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem > 48 * 1024 ? smem : 48 * 1024));
    if (e != cudaSuccess)
        return e;
    k_gather<<<static_cast<unsigned>(blocks), kThreads, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_read_kv(const fkv_ctx *c, const double *pts, int64_t n_streams, int64_t n_rec,
                           int64_t pt_stride, const int64_t *req, int64_t n_req, void *out,
                           int dtype, cudaStream_t st)
{
    ReadArgs a;
    a.pts = reinterpret_cast<const double2 *>(pts);
    a.n_streams = n_streams;
    a.n_rec = n_rec;
    a.pt_stride = pt_stride;
    a.req = req;
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
    a.cbk = c->cb[0].cb32;
    a.cbv = c->cb[1].cb32;
    a.dec = c->d_dec;
    a.status = c->d_status;
    if (n_req <= 0)
        return cudaSuccess;
    const int64_t blocks = (n_req + kReadWarps - 1) / kReadWarps;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    k_read_kv<<<static_cast<unsigned>(blocks), kReadWarps * 32, 0, st>>>(a);
    return cudaGetLastError();
}
