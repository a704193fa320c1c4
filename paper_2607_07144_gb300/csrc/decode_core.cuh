// Span decoding core shared by the bulk decoder, the random reads and the
// record reads (Sec. 1 "The code": the symbol is the cell holding the point,
// then p_{k-1} = (p_k - (1-r) V(c_k)) / r).
//
// The decoder never divides.  With m the span length and Q_k = r^(m-k) p_k,
//     Q_m = stored point,   Q_{k-1} = Q_k - (1-r) r^(m-k) V(c_k),
// and Q_0 = r^m p_0 must be back at the anchor (the origin).  Nearest-vertex
// classification of p_k (= cell containment for r <= r_N) is the argmax over
// c of p_k . V(c) because every vertex lies on the unit circle, and that is
// scale-free: argmax_c Q_k . V(c).  The margin of the true point to a cell
// boundary is about r^m in Q space at every step, so Q is kept in exact
// Q1.62 fixed point (int64, units of 2^-62) and the step is one table load
// of T[j][c] = round((1-r) r^j V(c) 2^62), j = m - k, and two subtractions.
//
// Classification takes an fp32 fast path with a certified margin and falls
// back to integer dot products in the rare near-boundary case: the high words
// of the 64x64->128-bit products, each dropping less than 2^-60, so a
// difference of two such dot products is off by less than 2^-59 (and by
// 2^-61 more from the vertices' Q1.62 rounding).  The decision it makes is
// the sign of Q . (V(a) - V(b)) for neighbouring vertices a, b, whose
// magnitude for a point of the true cell is at least
//     r^(m-1) (1 - cos(2 pi / N)) (1 - 2 r)
// (the point after the span's first symbol, (1 - r) V(c), is the closest
// case; a later point's own offset costs at most the factor 1 - 2 r).  With
// span lengths up to 44 / log2(1/r), r^(m-1) >= 2^-44 / r, and r_N ~ pi / N,
// that is at least about 2^-44 * 2 pi / N >= 2^-51.3 for every N <= 1024,
// 2^7 above the error (at N = 1024, L = 5 the bound is 2^-49.1, and that
// value is reached by alternating-neighbour spans):
//   * N = 4: the vertices are the axis directions, exact integer compares;
//   * N <= 8: fp32 scores q . V(c); exact scores when the best two are closer
//     than a bound far above the fp32 error;
//   * N > 8: Voronoi regions of the vertices are angular sectors, so the fp32
//     angle picks the sector; within twice the angle's error bound of a
//     boundary (the bound: 1.2e-5 rad for the arctangent polynomial plus
//     1.5e-6 rad for the fp32 direction, division and reflections, plus
//     N 2^-24 sector widths for the scaling) the two neighbouring sectors are
//     decided by the sign of Q . (V(a) - V(b)); the record reads take the
//     angle from atan2f instead (a shorter dependency chain) with a band of
//     1e-3 sector widths.
#pragma once

#include <climits>

#include "fkv_internal.h"

namespace fkvdec {

// atan u ~ u (a1 + a3 u^2 + a5 u^4 + a7 u^6 + a9 u^8) on [0, 1], from
// fit_atan.py: float32 Horner evaluation within 1.18e-5 rad of atan
__device__ constexpr float kAtan[5] = {9.998637438e-01f, -3.302824795e-01f, 1.800999194e-01f, -8.509350568e-02f,
                                       2.082198113e-02f};

struct Tables {
    const longlong2 *T;   // [L][N] (x, y), shared memory
    const long long *vx;  // [N] V(c) in Q1.62, shared memory
    const long long *vy;
    const float2 *vf;     // [N] V(c) as float, shared memory
    int N;
    float sect_thr;       // sector test: |fraction| below this is decided in fp32
};

// Shared-memory footprint of the tables for (N, L).
__host__ __device__ inline int smem_bytes(int N, int L)
{
    return L * N * 16 + N * 16 + N * 8;
}

// Block-cooperative copy of the tables into `sm` (16-byte aligned).
__device__ inline Tables load(const fkv_decconst *__restrict__ g, const longlong2 *__restrict__ Tg, int N, int L,
                              uint8_t *sm)
{
    longlong2 *T = reinterpret_cast<longlong2 *>(sm);
    long long *vx = reinterpret_cast<long long *>(sm + L * N * 16);
    long long *vy = vx + N;
    float2 *vf = reinterpret_cast<float2 *>(sm + L * N * 16 + N * 16);
    for (int i = threadIdx.x; i < L * N; i += blockDim.x)
        T[i] = Tg[i];
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        vx[i] = g->vx[i];
        vy[i] = g->vy[i];
        vf[i] = make_float2(g->vfx[i], g->vfy[i]);
    }
    return Tables{T, vx, vy, vf, N, g->sect_thr};
}

// Q . V(c) in units of 2^-60: the high words of the two 128-bit products
// (the error bound is in the header comment).
__device__ __forceinline__ long long exact_dot(const Tables &t, long long X, long long Y, int c)
{
    return __mul64hi(X, t.vx[c]) + __mul64hi(Y, t.vy[c]);
}

static __device__ __noinline__ int classify_exact_all(const Tables &t, long long X, long long Y)
{
    int best = 0;
    long long bs = exact_dot(t, X, Y, 0);
    for (int c = 1; c < t.N; ++c) {
        const long long s = exact_dot(t, X, Y, c);
        if (s > bs) {
            bs = s;
            best = c;
        }
    }
    return best;
}

// fp32 image (qx, qy) of the direction of (X, Y): both scaled by one power of
// two that puts the larger magnitude's top bit at bit 62, then their high
// 32-bit words converted.  Relative to the larger magnitude the image is off
// by at most 2^-30 (the dropped low word) plus one fp32 rounding, like a
// direct conversion; only integer ops and 32-bit conversions are used,
// because 64-bit integer conversions issue at the FP64 rate on this GPU.
__device__ __forceinline__ void direction(long long X, long long Y, float &qx, float &qy)
{
    const unsigned long long ax = X < 0 ? 0ull - static_cast<unsigned long long>(X) : static_cast<unsigned long long>(X);
    const unsigned long long ay = Y < 0 ? 0ull - static_cast<unsigned long long>(Y) : static_cast<unsigned long long>(Y);
    const int sh = max(__clzll(static_cast<long long>(ax | ay)) - 1, 0);
    const unsigned long long xs = static_cast<unsigned long long>(X) << sh;
    const unsigned long long ys = static_cast<unsigned long long>(Y) << sh;
    qx = __int2float_rn(static_cast<int>(static_cast<unsigned>(xs >> 32)));
    qy = __int2float_rn(static_cast<int>(static_cast<unsigned>(ys >> 32)));
}

// kShortChain: the sector angle from the library's atan2f, whose dependency
// chain is shorter than the polynomial's (record reads, where one walk per
// lane is the whole latency); otherwise from the polynomial, which issues
// fewer instructions (bulk decoders, many walks in flight).
template <bool kShortChain = false>
__device__ __forceinline__ int classify(const Tables &t, long long X, long long Y)
{
    const int N = t.N;
    if (N == 4) {
        const long long ax = X < 0 ? -X : X, ay = Y < 0 ? -Y : Y;
        if (ax >= ay)
            return X >= 0 ? 0 : 2;
        return Y >= 0 ? 1 : 3;
    }
    float qx, qy;
    direction(X, Y, qx, qy);
    if (N <= 8) {
        float b1 = -INFINITY, b2 = -INFINITY;
        int bi = 0;
        for (int c = 0; c < N; ++c) {
            const float s = fmaf(qx, t.vf[c].x, qy * t.vf[c].y);
            if (s > b1) {
                b2 = b1;
                b1 = s;
                bi = c;
            } else if (s > b2) {
                b2 = s;
            }
        }
        if (b1 - b2 > 0x1p-18f * (fabsf(qx) + fabsf(qy)))
            return bi;
        return classify_exact_all(t, X, Y);
    }
    float ph, thr;
    if constexpr (kShortChain) {
        // atan2f is within a few ulp: 1e-3 sector widths covers it at any N
        ph = atan2f(qy, qx);
        thr = 0.499f;
    } else {
        // the angle of (qx, qy): octant reduction to u in [0, 1], atan u
        // from the odd polynomial of fit_atan.py (error below 1.2e-5 rad),
        // then the octant's reflections, giving an angle in [-pi, pi]
        const float ax = fabsf(qx), ay = fabsf(qy);
        const float mx = fmaxf(ax, ay), mn = fminf(ax, ay);
        const float u = mx > 0.0f ? __fdividef(mn, mx) : 0.0f;
        const float u2 = u * u;
        ph = u * fmaf(fmaf(fmaf(fmaf(kAtan[4], u2, kAtan[3]), u2, kAtan[2]), u2, kAtan[1]), u2, kAtan[0]);
        if (ay > ax)
            ph = 1.57079637f - ph;
        if (qx < 0.0f)
            ph = 3.14159274f - ph;
        if (qy < 0.0f)
            ph = -ph;
        thr = t.sect_thr;
    }
    const float a = ph * (static_cast<float>(N) * 0.159154937f);
    const float ar = rintf(a);
    const float f = a - ar;                        // in [-0.5, 0.5]
    int c0 = static_cast<int>(ar);
    if (c0 < 0)
        c0 += N;
    if (c0 >= N)
        c0 -= N;
    // away from a sector boundary by more than the angle's error allows
    if (fabsf(f) < thr)
        return c0;
    int c1 = f > 0.0f ? c0 + 1 : c0 - 1;           // the neighbour across the near boundary
    if (c1 < 0)
        c1 += N;
    if (c1 >= N)
        c1 -= N;
    const long long d = exact_dot(t, X, Y, c0) - exact_dot(t, X, Y, c1);
    if (d > 0)
        return c0;
    if (d < 0)
        return c1;
    return c0 < c1 ? c0 : c1;
}

// round(v * 2^62) to nearest, ties to even, saturated to int64 (NaN gives
// INT64_MIN), from the binary64 fields with integer ops: v = m 2^(e - 1075),
// so v 2^62 = m 2^(e - 1013), a left shift or a rounded right shift of m.
__device__ __forceinline__ long long to_q62(double v)
{
    const unsigned long long b = static_cast<unsigned long long>(__double_as_longlong(v));
    const int e = static_cast<int>((b >> 52) & 0x7FF);
    const unsigned long long frac = b & 0xFFFFFFFFFFFFFull;
    const bool neg = (b >> 63) != 0;
    if (e >= 1024) {                           // |v| >= 2, infinity or NaN
        if (e == 2047 && frac)
            return LLONG_MIN;
        return neg ? LLONG_MIN : LLONG_MAX;
    }
    if (e == 0)                                // zero or subnormal: |v 2^62| < 2^-960
        return 0;
    const unsigned long long m = frac | (1ull << 52);
    const int s = e - 1013;
    unsigned long long mag;
    if (s >= 0) {
        mag = m << s;                          // s <= 10: below 2^63
    } else if (s > -54) {
        const int k = -s;
        const unsigned long long q = m >> k, rem = m & ((1ull << k) - 1), half = 1ull << (k - 1);
        mag = q + ((rem > half || (rem == half && (q & 1))) ? 1 : 0);
    } else {
        mag = 0;                               // below half a unit
    }
    return neg ? -static_cast<long long>(mag) : static_cast<long long>(mag);
}

// Decode `steps` symbols backward from Q (the span's stored point in Q1.62):
// step j = 0 .. steps-1 emits the symbol at offset m-1-j of the span.
// `emit(j, c)` receives each symbol.
template <bool kShortChain = false, class Emit>
__device__ __forceinline__ void walk(const Tables &t, long long &X, long long &Y, int steps, Emit emit)
{
    const int N = t.N;
    for (int j = 0; j < steps; ++j) {
        const int c = classify<kShortChain>(t, X, Y);
        emit(j, c);
        const longlong2 w = t.T[j * N + c];
        X = static_cast<long long>(static_cast<unsigned long long>(X) - static_cast<unsigned long long>(w.x));
        Y = static_cast<long long>(static_cast<unsigned long long>(Y) - static_cast<unsigned long long>(w.y));
    }
}

}  // namespace fkvdec
