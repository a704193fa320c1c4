// Codebook gather: K/V reconstruction from RVQ indices (Sec. 3 "Setup": the
// reconstruction is the sum of the selected centroids), for whole archives
// and for random record reads (Sec. 2).
//
// Whole archive: a block owns one codebook group (layer, head), a slice of
// the head dimension and a run of vectors; the group's float32 codebooks for
// that slice sit in shared memory, so HBM sees only the index bytes in and
// the rebuilt K/V out.  Sums run in float32, stage order, then round to
// nearest-even into the cache dtype.
#include "decode_core.cuh"

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
    extern __shared__ __align__(16) float scb[];   // [S][256][Dp] floats, then offsets and indices
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
    // this block's indices and output offsets -> shared memory (independent
    // loads, many in flight; 32-bit index arithmetic, checked on the host)
    int64_t *soff = reinterpret_cast<int64_t *>(scb + S * 256 * Dp);
    uint8_t *sids = reinterpret_cast<uint8_t *>(soff + kChunk);
    const int nvec = static_cast<int>(a.batch * a.n_rec);
    const int v_beg = chunk * static_cast<int>(kChunk);
    const int nv = min(nvec - v_beg, static_cast<int>(kChunk));
    const unsigned n_rec = static_cast<unsigned>(a.n_rec);
    for (int vi = threadIdx.x; vi < nv; vi += kThreads) {
        const unsigned v = static_cast<unsigned>(v_beg + vi);
        const unsigned b = v / n_rec;
        const unsigned rec = v - b * n_rec;
        const uint8_t *ids = a.sym + (static_cast<int64_t>(b) * a.n_layers + l) * a.stream_stride +
                             static_cast<int64_t>(rec) * a.R + a.kv_off + h * S;
        for (int s = 0; s < S; ++s)
            sids[vi * S + s] = __ldg(ids + s);
        soff[vi] = l * a.s_layer + b * a.s_batch + h * a.s_head + (a.t0 + rec) * a.s_pos + d0;
    }
    __syncthreads();
    const int tpv = Dp / 2;                  // threads per vector (two dims each)
    const int vpi = kThreads / tpv;          // vectors per pass
    const int dd = (threadIdx.x % tpv) * 2;
#pragma unroll 2
    for (int vi = threadIdx.x / tpv; vi < nv; vi += vpi) {
        float x = 0.0f, y = 0.0f;
        for (int s = 0; s < S; ++s) {
            const float2 c = *reinterpret_cast<const float2 *>(scb + (s * 256 + sids[vi * S + s]) * Dp + dd);
            x += c.x;
            y += c.y;
        }
        store2(a.out, a.dtype, soff[vi] + dd, x, y);
    }
}

// ------------------------------------------------------- random reads ---
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
    const longlong2 *T;
    unsigned *status;
};

__host__ __device__ inline int read_tables_bytes(int N, int L)
{
    return (fkvdec::smem_bytes(N, L) + 15) & ~15;
}

// One warp per request: its lanes decode the spans covering the record into
// shared memory, then gather the record's 2 * H head vectors.
__global__ void __launch_bounds__(kReadWarps * 32) k_read_kv(const ReadArgs a)
{
    extern __shared__ __align__(16) uint8_t dsm[];
    const fkvdec::Tables t = fkvdec::load(a.dec, a.T, a.N, a.L, dsm);
    uint8_t *srec = dsm + read_tables_bytes(a.N, a.L);
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t q = static_cast<int64_t>(blockIdx.x) * kReadWarps + warp;
    if (q >= a.n_req)
        return;
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
    uint8_t *my = srec + warp * kMaxRecord;
    bool bad = false;
    for (int64_t u = u0 + lane; u <= u1; u += 32) {
        const int m = static_cast<int>(min(static_cast<int64_t>(L), n - u * L));
        const double2 p = a.pts[st * a.pt_stride + u];
        long long X = fkvdec::to_q62(p.x), Y = fkvdec::to_q62(p.y);
        const int64_t base = u * L - sym0;
        fkvdec::walk(t, X, Y, m, [&](int j, int c) {
            const int64_t pos = base + m - 1 - j;
            if (pos >= 0 && pos < R)
                my[pos] = static_cast<uint8_t>(c);
        });
        const long long lim = __ldg(&a.dec->alim[m]);
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
    if (nvec > 0x7FFFFFFF)
        return cudaErrorInvalidValue;   // vector indices are 32-bit in the kernel
    const int64_t chunks = (nvec + kChunk - 1) / kChunk;
    const int64_t blocks = chunks * parts * c->Ly * c->H;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    a.chunks = static_cast<int>(chunks);
    const size_t smem = static_cast<size_t>(a.S) * 256 * a.Dp * 4 + static_cast<size_t>(kChunk) * (8 + a.S);
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
    a.T = c->d_T;
    a.status = c->d_status;
    if (n_req <= 0)
        return cudaSuccess;
    const int64_t blocks = (n_req + kReadWarps - 1) / kReadWarps;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    const int smem = read_tables_bytes(a.N, a.L) + kReadWarps * kMaxRecord;
    cudaError_t e = cudaFuncSetAttribute(k_read_kv, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    k_read_kv<<<static_cast<unsigned>(blocks), kReadWarps * 32, smem, st>>>(a);
    return cudaGetLastError();
}
