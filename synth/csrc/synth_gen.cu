// Device-side twin of synth/__init__.py: the same seeded inputs, generated
// on the GPU for configurations too large to build on the host.  Philox4x32-10
// as published by Salmon, Moraes, Dror and Shaw (SC'11); no archive
// arithmetic lives here.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace {

struct U4 {
    uint32_t x, y, z, w;
};

__device__ __forceinline__ U4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0, uint32_t k1)
{
    const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u, W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(M0, c0), lo0 = M0 * c0;
        const uint32_t hi1 = __umulhi(M1, c2), lo1 = M1 * c2;
        const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
        k0 += W0;
        k1 += W1;
    }
    return {c0, c1, c2, c3};
}

__device__ __forceinline__ int irwin_hall(uint64_t e, uint32_t tid, uint32_t k0, uint32_t k1)
{
    const U4 w = philox(static_cast<uint32_t>(e), static_cast<uint32_t>(e >> 32), tid, 0u, k0, k1);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
    int z = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i)
        z += static_cast<int>(ws[i] & 0xFFFFu) + static_cast<int>(ws[i] >> 16);
    return z - 262140;
}

// Positions [t0, t0 + C) of the cache [Ly][B][H][T][D] into out [Ly][B][H][C][D];
// every element keeps its flat index in the whole cache; scale [Ly][H][D] float32.
__global__ void k_gen_kv(void *out, int dtype, int64_t B, int64_t H, int64_t T, int64_t D, int64_t t0, int64_t C,
                         int64_t total, uint32_t tid, uint32_t k0, uint32_t k1, const float *scale)
{
    for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < total;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t d = e % D;
        const int64_t t = (e / D) % C;
        const int64_t row = e / (D * C);               // (l * B + b) * H + h
        const int64_t h = row % H;
        const int64_t l = row / (H * B);
        const int64_t ef = (row * T + t0 + t) * D + d; // flat index in the whole cache
        const float x = __fmul_rn(static_cast<float>(irwin_hall(static_cast<uint64_t>(ef), tid, k0, k1)),
                                  scale[(l * H + h) * D + d]);
        if (dtype == 0)
            static_cast<float *>(out)[e] = x;
        else if (dtype == 1)
            static_cast<__half *>(out)[e] = __float2half_rn(x);
        else
            static_cast<__nv_bfloat16 *>(out)[e] = __float2bfloat16_rn(x);
    }
}

// symbols of one stream: uniform floor(w N / 2^32) or Zipf inverse CDF.
// One byte per symbol for N <= 256, else two (uint16).
__global__ void k_gen_sym(void *out, int64_t n, uint64_t stream, uint32_t tid, uint32_t N, int zipf,
                          const uint32_t *thr, uint32_t k0, uint32_t k1)
{
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const uint64_t e = static_cast<uint64_t>(i) + (stream << 40);
        const uint32_t w = philox(static_cast<uint32_t>(e), static_cast<uint32_t>(e >> 32), tid, 0u, k0, k1).x;
        uint32_t s;
        if (!zipf) {
            s = static_cast<uint32_t>((static_cast<uint64_t>(w) * N) >> 32);
        } else {
            uint32_t lo = 0, hi = N - 1;   // count of thresholds <= w among thr[0..N-2]
            while (lo < hi) {
                const uint32_t mid = (lo + hi) >> 1;
                if (thr[mid] <= w)
                    lo = mid + 1;
                else
                    hi = mid;
            }
            s = lo;
        }
        if (N <= 256)
            static_cast<uint8_t *>(out)[i] = static_cast<uint8_t>(s);
        else
            static_cast<uint16_t *>(out)[i] = static_cast<uint16_t>(s);
    }
}

__global__ void k_gen_pos(int64_t *out, int64_t count, uint64_t stream, uint32_t tid, uint64_t n, uint32_t k0,
                          uint32_t k1, int64_t stride, int64_t col)
{
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < count;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const uint64_t e = static_cast<uint64_t>(i) + (stream << 40);
        const uint32_t w = philox(static_cast<uint32_t>(e), static_cast<uint32_t>(e >> 32), tid, 0u, k0, k1).x;
        out[i * stride + col] = static_cast<int64_t>((static_cast<uint64_t>(w) * n) >> 32);
    }
}

unsigned grid_for(int64_t n)
{
    int64_t g = (n + 255) / 256;
    return static_cast<unsigned>(g > 152 * 64 ? 152 * 64 : (g < 1 ? 1 : g));
}

}  // namespace

extern "C" {

int synth_gen_kv(void *out, int dtype, int64_t Ly, int64_t B, int64_t H, int64_t T, int64_t D, int64_t t0,
                 int64_t C, uint32_t tid, uint32_t k0, uint32_t k1, const float *scale, void *stream)
{
    const int64_t total = Ly * B * H * C * D;
    k_gen_kv<<<grid_for(total), 256, 0, static_cast<cudaStream_t>(stream)>>>(out, dtype, B, H, T, D, t0, C, total,
                                                                             tid, k0, k1, scale);
    return static_cast<int>(cudaGetLastError());
}

int synth_gen_symbols(void *out, int64_t n, uint64_t stream_id, uint32_t tid, uint32_t N, int zipf,
                      const uint32_t *thr, uint32_t k0, uint32_t k1, void *stream)
{
    k_gen_sym<<<grid_for(n), 256, 0, static_cast<cudaStream_t>(stream)>>>(out, n, stream_id, tid, N, zipf, thr,
                                                                          k0, k1);
    return static_cast<int>(cudaGetLastError());
}

int synth_gen_positions(int64_t *out, int64_t count, uint64_t stream_id, uint32_t tid, uint64_t n, uint32_t k0,
                        uint32_t k1, int64_t stride, int64_t col, void *stream)
{
    k_gen_pos<<<grid_for(count), 256, 0, static_cast<cudaStream_t>(stream)>>>(out, count, stream_id, tid, n, k0,
                                                                               k1, stride, col);
    return static_cast<int>(cudaGetLastError());
}

}  // extern "C"
