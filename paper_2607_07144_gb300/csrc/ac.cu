// Probability-weighted maps (Sec. 6 eq. (1)): the arithmetic-coding form of
// the iterated map, in which symbol c shrinks the interval [lo, hi] to its
// sub-interval of width p(c) at offset F(c).  Decoding is sequential within a
// stream, so the GPU codes independent streams side by side: one warp per
// stream.  The model's counts live in the warp's registers, CPL symbols per
// lane (symbol c in lane c / CPL, slot c % CPL), with each lane's count total
// and the count total of the lanes below it kept current, so the cumulative
// count of a symbol is one shuffle away and no scan is needed per step.  The
// interval arithmetic runs redundantly in every lane (it is warp-uniform), so
// the renormalisation loop never diverges; lane 0 packs the output bits.
//
// Integer form (32-bit interval, 64-bit products): with w = hi - lo + 1 and T
// the count total, lo' = lo + floor(w cum(c) / T), hi' = lo + floor(w (cum(c) +
// cnt(c)) / T) - 1; a settled half emits its bit (and the pending opposite
// bits), a middle-half straddle adds a pending bit, and the interval doubles.
// Counts start at 1 and, adaptively, the coded symbol's count grows by one
// (add-one prequential model); otherwise p(c) = 1/N throughout, which is the
// uniform code of Sec. 1.  Bits are written most significant first.
#include "fkv_internal.h"

namespace {

constexpr int kWarpsPerBlock = 4;
constexpr unsigned long long kHalf = 0x80000000ull, kQtr = 0x40000000ull, k3Qtr = 0xC0000000ull;

template <int CPL>
struct Model {
    uint32_t cnt[CPL];     // this lane's counts: symbols lane * CPL + j
    uint32_t lt;           // their sum
    uint32_t base;         // the count total of the lanes below this one
    uint32_t total;

    __device__ __forceinline__ void init(int lane, int N)
    {
        lt = 0;
#pragma unroll
        for (int j = 0; j < CPL; ++j) {
            cnt[j] = lane * CPL + j < N ? 1u : 0u;
            lt += cnt[j];
        }
        base = min(lane * CPL, N);
        total = N;
    }
    // cumulative count of slot `off` of this lane and the count there
    __device__ __forceinline__ void local(int off, uint32_t &cum, uint32_t &f) const
    {
        cum = base;
        f = 0;
#pragma unroll
        for (int j = 0; j < CPL; ++j) {
            cum += j < off ? cnt[j] : 0u;
            f = j == off ? cnt[j] : f;
        }
    }
    // after coding symbol c (owner lane o, slot off)
    __device__ __forceinline__ void bump(int lane, int o, int off)
    {
        if (lane == o) {
#pragma unroll
            for (int j = 0; j < CPL; ++j)
                cnt[j] += j == off ? 1u : 0u;
            lt += 1;
        }
        base += lane > o ? 1u : 0u;
        total += 1;
    }
};

template <typename Sym, int CPL>
__global__ void __launch_bounds__(kWarpsPerBlock * 32)
k_ac_encode(const Sym *__restrict__ sym, int64_t n_streams, int64_t n, int64_t sym_stride, int N, int adaptive,
            uint32_t *__restrict__ words, int64_t word_stride, int64_t *__restrict__ nbits, unsigned *status)
{
    const int lane = threadIdx.x & 31;
    const int64_t stream = static_cast<int64_t>(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
    if (stream >= n_streams)
        return;
    const Sym *src = sym + stream * sym_stride;
    uint32_t *out = words + stream * word_stride;
    const int64_t cap_bits = word_stride * 32;
    Model<CPL> m;
    m.init(lane, N);
    unsigned long long lo = 0, hi = 0xFFFFFFFFull;
    int64_t follow = 0, nb = 0;
    uint32_t acc = 0;
    bool overflow = false, bad = false;
    auto put = [&](uint32_t b) {               // warp-uniform; lane 0 stores full words
        if (nb >= cap_bits) {
            overflow = true;
            return;
        }
        acc = (acc << 1) | b;
        ++nb;
        if ((nb & 31) == 0 && lane == 0)
            out[(nb >> 5) - 1] = acc;
    };
    Sym next = 0;
    for (int64_t k = 0; k < n; ++k) {
        if ((k & 31) == 0)
            next = k + lane < n ? src[k + lane] : Sym(0);   // 32 symbols per load
        int c = static_cast<int>(__shfl_sync(0xFFFFFFFFu, static_cast<uint32_t>(next), static_cast<int>(k & 31)));
        if (c >= N) {                             // not a symbol: coded as N - 1, reported
            bad = true;
            c = N - 1;
        }
        const int o = c / CPL, off = c - o * CPL;
        uint32_t cl, fl;
        m.local(off, cl, fl);
        const unsigned long long cum = __shfl_sync(0xFFFFFFFFu, cl, o);
        const unsigned long long f = __shfl_sync(0xFFFFFFFFu, fl, o);
        const unsigned long long w = hi - lo + 1;
        hi = lo + w * (cum + f) / m.total - 1;
        lo = lo + w * cum / m.total;
        for (;;) {
            if (hi < kHalf) {
                put(0);
                for (; follow > 0; --follow)
                    put(1);
            } else if (lo >= kHalf) {
                put(1);
                for (; follow > 0; --follow)
                    put(0);
                lo -= kHalf;
                hi -= kHalf;
            } else if (lo >= kQtr && hi < k3Qtr) {
                ++follow;
                lo -= kQtr;
                hi -= kQtr;
            } else {
                break;
            }
            lo = 2 * lo;
            hi = 2 * hi + 1;
        }
        if (adaptive)
            m.bump(lane, o, off);
    }
    ++follow;
    const uint32_t b = lo >= kQtr;
    put(b);
    for (; follow > 0; --follow)
        put(b ^ 1u);
    if (lane == 0) {
        if (nb & 31)
            out[nb >> 5] = acc << (32 - (nb & 31));   // the last, partial word
        nbits[stream] = overflow ? -1 : nb;
        if (overflow || bad)
            atomicOr(status, FKV_ST_CORRUPT);
    }
}

template <typename Sym, int CPL>
__global__ void __launch_bounds__(kWarpsPerBlock * 32)
k_ac_decode(const uint32_t *__restrict__ words, int64_t word_stride, const int64_t *__restrict__ nbits,
            int64_t n_streams, int64_t n, int N, int adaptive, Sym *__restrict__ sym, int64_t sym_stride,
            unsigned *status)
{
    const int lane = threadIdx.x & 31;
    const int64_t stream = static_cast<int64_t>(blockIdx.x) * kWarpsPerBlock + (threadIdx.x >> 5);
    if (stream >= n_streams)
        return;
    const uint32_t *in = words + stream * word_stride;
    Sym *dst = sym + stream * sym_stride;
    int64_t nb = nbits[stream];
    if (nb < 0 || nb > word_stride * 32) {        // not a code this call can read
        if (lane == 0)
            atomicOr(status, FKV_ST_CORRUPT);
        nb = 0;
    }
    int64_t pos = 0;
    auto bit = [&]() -> unsigned long long {
        const unsigned long long b = pos < nb ? (__ldg(in + (pos >> 5)) >> (31 - (pos & 31))) & 1u : 0u;
        ++pos;
        return b;
    };
    Model<CPL> m;
    m.init(lane, N);
    bool bad = false;
    unsigned long long lo = 0, hi = 0xFFFFFFFFull, val = 0;
    for (int i = 0; i < 32; ++i)
        val = 2 * val + bit();
    Sym pending = 0;
    for (int64_t k = 0; k < n; ++k) {
        const unsigned long long w = hi - lo + 1;
        unsigned long long target = ((val - lo + 1) * m.total - 1) / w;
        if (target >= m.total) {                  // bits that no code produces: keep the interval valid
            bad = true;
            target = m.total - 1;
        }
        // the lane whose counts hold the target, then the slot inside it
        const bool mine = target >= m.base && target < static_cast<unsigned long long>(m.base) + m.lt;
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, mine);
        const int o = bal ? __ffs(bal) - 1 : 0;
        int off = 0;
        uint32_t cl = m.base, fl = 0;
        if (lane == o) {
            uint32_t run = m.base;
            bool found = false;
#pragma unroll
            for (int j = 0; j < CPL; ++j) {
                const bool here = !found && target < static_cast<unsigned long long>(run) + m.cnt[j];
                off = here ? j : off;
                cl = here ? run : cl;
                fl = here ? m.cnt[j] : fl;
                found = found || here;
                run += m.cnt[j];
            }
        }
        off = __shfl_sync(0xFFFFFFFFu, off, o);
        const unsigned long long cum = __shfl_sync(0xFFFFFFFFu, cl, o);
        const unsigned long long f = __shfl_sync(0xFFFFFFFFu, fl, o);
        const int c = min(o * CPL + off, N - 1);
        if (lane == static_cast<int>(k & 31))
            pending = static_cast<Sym>(c);
        if ((k & 31) == 31 || k == n - 1) {       // 32 symbols per store
            const int64_t k0 = k & ~int64_t(31);
            if (lane <= static_cast<int>(k - k0))
                dst[k0 + lane] = pending;
        }
        hi = lo + w * (cum + f) / m.total - 1;
        lo = lo + w * cum / m.total;
        for (;;) {
            if (hi < kHalf) {
            } else if (lo >= kHalf) {
                lo -= kHalf;
                hi -= kHalf;
                val -= kHalf;
            } else if (lo >= kQtr && hi < k3Qtr) {
                lo -= kQtr;
                hi -= kQtr;
                val -= kQtr;
            } else {
                break;
            }
            lo = 2 * lo;
            hi = 2 * hi + 1;
            val = 2 * val + bit();
        }
        if (adaptive)
            m.bump(lane, o, off);
    }
    if (bad && lane == 0)
        atomicOr(status, FKV_ST_CORRUPT);
}

template <typename Sym>
cudaError_t ac_encode_t(const fkv_ctx *c, const Sym *sym, int64_t n_streams, int64_t n, int64_t sym_stride,
                        int adaptive, uint32_t *words, int64_t word_stride, int64_t *nbits, cudaStream_t st)
{
    const int64_t blocks = (n_streams + kWarpsPerBlock - 1) / kWarpsPerBlock;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    if (c->N <= 256)
        k_ac_encode<Sym, 8><<<static_cast<unsigned>(blocks), kWarpsPerBlock * 32, 0, st>>>(
            sym, n_streams, n, sym_stride, c->N, adaptive, words, word_stride, nbits, c->d_status);
    else
        k_ac_encode<Sym, 32><<<static_cast<unsigned>(blocks), kWarpsPerBlock * 32, 0, st>>>(
            sym, n_streams, n, sym_stride, c->N, adaptive, words, word_stride, nbits, c->d_status);
    return cudaGetLastError();
}

template <typename Sym>
cudaError_t ac_decode_t(const fkv_ctx *c, const uint32_t *words, int64_t word_stride, const int64_t *nbits,
                        int64_t n_streams, int64_t n, int adaptive, Sym *sym, int64_t sym_stride, cudaStream_t st)
{
    const int64_t blocks = (n_streams + kWarpsPerBlock - 1) / kWarpsPerBlock;
    if (blocks > 0x7FFFFFFF)
        return cudaErrorInvalidConfiguration;
    if (c->N <= 256)
        k_ac_decode<Sym, 8><<<static_cast<unsigned>(blocks), kWarpsPerBlock * 32, 0, st>>>(
            words, word_stride, nbits, n_streams, n, c->N, adaptive, sym, sym_stride, c->d_status);
    else
        k_ac_decode<Sym, 32><<<static_cast<unsigned>(blocks), kWarpsPerBlock * 32, 0, st>>>(
            words, word_stride, nbits, n_streams, n, c->N, adaptive, sym, sym_stride, c->d_status);
    return cudaGetLastError();
}

}  // namespace

int64_t ac_capacity_words(int N, int64_t n)
{
    int per = 1;
    while ((int64_t(1) << per) < N + n)
        ++per;
    return (n * (per + 1) + 2 + 31) / 32 + 1;
}

cudaError_t launch_ac_encode(const fkv_ctx *c, const void *sym, int64_t n_streams, int64_t n, int64_t sym_stride,
                             int adaptive, uint32_t *words, int64_t word_stride, int64_t *nbits, cudaStream_t st)
{
    if (n_streams <= 0)
        return cudaSuccess;
    if (c->N > 256)
        return ac_encode_t(c, static_cast<const uint16_t *>(sym), n_streams, n, sym_stride, adaptive, words,
                           word_stride, nbits, st);
    return ac_encode_t(c, static_cast<const uint8_t *>(sym), n_streams, n, sym_stride, adaptive, words, word_stride,
                       nbits, st);
}

cudaError_t launch_ac_decode(const fkv_ctx *c, const uint32_t *words, int64_t word_stride, const int64_t *nbits,
                             int64_t n_streams, int64_t n, int adaptive, void *sym, int64_t sym_stride, cudaStream_t st)
{
    if (n_streams <= 0 || n <= 0)
        return cudaSuccess;
    if (c->N > 256)
        return ac_decode_t(c, words, word_stride, nbits, n_streams, n, adaptive, static_cast<uint16_t *>(sym),
                           sym_stride, st);
    return ac_decode_t(c, words, word_stride, nbits, n_streams, n, adaptive, static_cast<uint8_t *>(sym), sym_stride,
                       st);
}
