/*
 * fkv_oracle.c -- TEST INFRASTRUCTURE, not part of the library.
 *
 * A plain, slow, float64 CPU restatement of what the fractal KV-cache archive
 * computes, written from the paper (arXiv 2607.07144) and used only to check
 * the CUDA library: tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
 * leg are its only callers.  It shares no code, header, table or constant
 * generator with the CUDA path.
 *
 * Build: gcc -O2 -ffp-contract=off -fno-fast-math -fopenmp -fPIC -shared
 * (no FMA contraction, so every a*b+c below is two IEEE-754 binary64 roundings,
 * exactly as written).  OpenMP only splits independent spans / vectors.
 *
 * Functions and the passage each follows:
 *   oracle_vertices       -- Sec. 1 "The code": regular N-gon, one vertex per symbol.
 *   oracle_packing_ratio  -- Sec. 1 and Fig. 1 caption: the kissing ratio r_N below
 *                            which the N cells are disjoint (formula not printed; the
 *                            N-flake ratio is the reading taken, pinned by brute force).
 *   oracle_max_span_len   -- Sec. 1: one double carries about 44/log2(1/r) symbols.
 *   oracle_span_encode    -- Sec. 1 forward map p_k = V(c_k) + r (p_{k-1} - V(c_k)),
 *                            one stored point per fixed-length span, from the anchor.
 *   oracle_span_decode    -- Sec. 1 inverse: the symbol is the cell holding the point
 *                            (nearest vertex for r <= r_N), p_{k-1} = (p_k-(1-r)V)/r.
 *   oracle_rvq_encode     -- Sec. 3 "Setup": residual VQ of depth s, nearest codeword
 *                            of the running residual at each stage.
 *   oracle_rvq_decode     -- Sec. 3 "Setup": the reconstruction is the sum of the
 *                            s selected centroids.
 *   oracle_ac_encode/decode -- Sec. 6 eq. (1): probability-weighted maps, i.e.
 *                            arithmetic coding: [lo, hi) shrinks to the symbol's
 *                            sub-interval of width p(c) at offset F(c), with p from
 *                            add-one counts (adaptive) or 1/N (the uniform code).
 * Parity pins for every function live in tests/test_oracle_*.py.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#ifndef M_PI
#define M_PI 3.14159265358979323846
#endif

/* Sec. 1: a regular N-gon, one vertex per symbol.  Reading: unit circumradius,
 * V(0) = (1, 0), counter-clockwise, angle 2*pi*c/N evaluated left to right in
 * binary64 with the C library's cos/sin; quarter turns (4c = 0 mod N) are the
 * exact values 0 and +-1.  V is written as [N][2] (x, y). */
void oracle_vertices(int N, double *V)
{
    for (int c = 0; c < N; ++c) {
        if ((4 * c) % N == 0) {
            int q = (4 * c) / N; /* 0..3 quarter turns */
            static const double qx[4] = {1.0, 0.0, -1.0, 0.0};
            static const double qy[4] = {0.0, 1.0, 0.0, -1.0};
            V[2 * c] = qx[q];
            V[2 * c + 1] = qy[q];
        } else {
            double theta = 2.0 * M_PI * c / N;
            V[2 * c] = cos(theta);
            V[2 * c + 1] = sin(theta);
        }
    }
}

/* Sec. 1 / Fig. 1 caption: the packing ("kissing") ratio.  Adjacent cells
 * V(c) + r (P - V(c)) of the unit N-gon P first touch when
 *     r_N = 1 / (2 (1 + sum_{k=1}^{floor(N/4)} cos(2 pi k / N))),
 * (the N-flake ratio); r_3 = r_4 = 1/2 as the paper states.  The cosines are the
 * x coordinates of oracle_vertices so the exact quarter-turn zero is used. */
double oracle_packing_ratio(int N)
{
    double s = 0.0;
    for (int k = 1; k <= N / 4; ++k) {
        if ((4 * k) % N == 0)
            s += 0.0; /* cos(pi/2), exact */
        else
            s += cos(2.0 * M_PI * k / N);
    }
    return 1.0 / (2.0 * (1.0 + s));
}

/* Sec. 1: one IEEE-754 double reliably carries about 44/log2(1/r) symbols; the
 * span length is the floor of that. */
int oracle_max_span_len(double r)
{
    return (int)floor(44.0 / log2(1.0 / r));
}

/* Sec. 1: forward contraction, span by span.  Each span starts at the anchor
 * (0, 0) and applies, per symbol c and per coordinate, d = p - V(c);
 * t = r * d; p = V(c) + t (three binary64 roundings, no FMA).  The point after
 * the span's last symbol is stored; the last span holds n mod L symbols when
 * that is nonzero.  pts is [ceil(n/L)][2]. */
void oracle_span_encode(const double *V, double r, int L,
                        const int32_t *sym, int64_t n, double *pts)
{
    int64_t spans = (n + L - 1) / L;
#pragma omp parallel for schedule(static)
    for (int64_t s = 0; s < spans; ++s) {
        int64_t b = s * L;
        int64_t e = b + L < n ? b + L : n;
        double x = 0.0, y = 0.0;
        for (int64_t k = b; k < e; ++k) {
            int c = sym[k];
            double vx = V[2 * c], vy = V[2 * c + 1];
            double dx = x - vx, dy = y - vy;
            double tx = r * dx, ty = r * dy;
            x = vx + tx;
            y = vy + ty;
        }
        pts[2 * s] = x;
        pts[2 * s + 1] = y;
    }
}

/* Nearest vertex of p, lowest index on a tie.  For r <= r_N every cell lies in
 * its vertex's Voronoi region, so this is the cell-containment test of Sec. 1. */
static int nearest_vertex(const double *V, int N, double x, double y)
{
    int best = 0;
    double bd = INFINITY;
    for (int c = 0; c < N; ++c) {
        double dx = x - V[2 * c], dy = y - V[2 * c + 1];
        double d = dx * dx + dy * dy;
        if (d < bd) {
            bd = d;
            best = c;
        }
    }
    return best;
}

/* Sec. 1: decoding inverts the map span by span, last symbol first:
 * c = cell containing p, then p <- (p - (1 - r) V(c)) / r with (1 - r) and
 * (1 - r) V(c) as binary64 products and an IEEE division.  After the span's
 * first symbol the point should be back at the anchor; anchor[s] receives
 * max(|x|, |y|) of that residual point (the anchor check).  Returns the number
 * of spans whose residual exceeds tol. */
int64_t oracle_span_decode(const double *V, int N, double r, int L,
                           const double *pts, int64_t n, int32_t *sym,
                           double *anchor, double tol)
{
    int64_t spans = (n + L - 1) / L;
    int64_t bad = 0;
    double w = 1.0 - r;
#pragma omp parallel for schedule(static) reduction(+ : bad)
    for (int64_t s = 0; s < spans; ++s) {
        int64_t b = s * L;
        int64_t e = b + L < n ? b + L : n;
        double x = pts[2 * s], y = pts[2 * s + 1];
        for (int64_t k = e - 1; k >= b; --k) {
            int c = nearest_vertex(V, N, x, y);
            sym[k] = c;
            double wx = w * V[2 * c], wy = w * V[2 * c + 1];
            x = (x - wx) / r;
            y = (y - wy) / r;
        }
        double a = fabs(x) > fabs(y) ? fabs(x) : fabs(y);
        if (anchor)
            anchor[s] = a;
        if (!(a <= tol))
            bad += 1;
    }
    return bad;
}

/* Sec. 3 "Setup": residual vector quantization.  For each vector, stage by
 * stage, the index is the codeword nearest (squared L2 summed directly in
 * float64 over the D coordinates, lowest index on a tie) to the running
 * residual, and the residual then drops that codeword.  x is [n][D] float64,
 * cb is [S][K][D] float32 (K codewords per stage), idx is [n][S].  Symbols
 * everywhere in this file are int32 so any alphabet size fits.  gap[n][S]
 * (may be NULL) receives (second-best - best distance) / ||residual||^2, the
 * quantity the parity criterion is stated on. */
void oracle_rvq_encode(const double *x, int64_t n, int D, const float *cb,
                       int S, int K, int32_t *idx, double *gap)
{
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t i = 0; i < n; ++i) {
        double res[1024];
        for (int k = 0; k < D; ++k)
            res[k] = x[i * D + k];
        for (int s = 0; s < S; ++s) {
            const float *C = cb + (int64_t)s * K * D;
            int best = 0;
            double bd = INFINITY, second = INFINITY;
            for (int j = 0; j < K; ++j) {
                double d = 0.0;
                for (int k = 0; k < D; ++k) {
                    double t = res[k] - (double)C[(int64_t)j * D + k];
                    d += t * t;
                }
                if (d < bd) {
                    second = bd;
                    bd = d;
                    best = j;
                } else if (d < second) {
                    second = d;
                }
            }
            idx[i * S + s] = best;
            if (gap) {
                double rn = 0.0;
                for (int k = 0; k < D; ++k)
                    rn += res[k] * res[k];
                gap[i * S + s] = rn > 0.0 ? (second - bd) / rn : INFINITY;
            }
            for (int k = 0; k < D; ++k)
                res[k] -= (double)C[(int64_t)best * D + k];
        }
    }
}

/* Sec. 3 "Setup": depth-s RVQ reconstructs a vector as the sum of its s
 * centroids, added in stage order in float64.  y is [n][D]. */
void oracle_rvq_decode(const int32_t *idx, int64_t n, int D, const float *cb,
                       int S, int K, double *y)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        for (int k = 0; k < D; ++k)
            y[i * D + k] = 0.0;
        for (int s = 0; s < S; ++s) {
            const float *C = cb + ((int64_t)s * K + idx[i * S + s]) * D;
            for (int k = 0; k < D; ++k)
                y[i * D + k] += (double)C[k];
        }
    }
}

/* Sec. 6 eq. (1): the probability-weighted map.  Encoding keeps an interval
 * [lo, hi] and replaces it, for symbol c, by lo' = lo + w F(c),
 * hi' = lo + w (F(c) + p(c)) - 1 with w = hi - lo + 1 -- the paper's recursion
 * in 32-bit integer arithmetic (the finite-precision arithmetic coder of
 * Witten, Neal and Cleary, CACM 1987): F(c) and p(c) are the cumulative count
 * and count of c over the total T, so w F(c) is floor(w cum(c) / T).
 * Whenever the interval lies in one half of [0, 2^32), the half's bit is
 * settled: it is emitted, followed by any pending opposite bits, and the
 * interval doubles; an interval straddling the middle inside the middle half
 * doubles around it and adds one pending bit.  After the last symbol two bits
 * (plus the pending ones) single out a point inside the final interval.
 * Model: counts start at 1 for all N symbols and, when adaptive, the coded
 * symbol's count grows by one after each step (the prequential add-one model);
 * otherwise every p(c) stays 1/N, which is the uniform code.  Bits are written
 * most significant first: stream bit i is bit 31 - i % 32 of word i / 32.
 * Returns the number of bits, or -1 when out (cap words) is too small. */
#define AC_HALF 0x80000000ull
#define AC_QTR 0x40000000ull
#define AC_3QTR 0xC0000000ull

static int ac_put(uint32_t *out, int64_t cap, int64_t *nb, int bit)
{
    if (*nb >= cap * 32)
        return -1;
    if (bit)
        out[*nb >> 5] |= 1u << (31 - (*nb & 31));
    *nb += 1;
    return 0;
}

int64_t oracle_ac_encode(const int32_t *sym, int64_t n, int N, int adaptive, uint32_t *out, int64_t cap)
{
    uint64_t lo = 0, hi = 0xFFFFFFFFull, total = (uint64_t)N;
    int64_t follow = 0, nb = 0;
    uint32_t cnt[4096];
    if (N > 4096)
        return -1;
    for (int c = 0; c < N; ++c)
        cnt[c] = 1;
    for (int64_t i = 0; i < cap; ++i)
        out[i] = 0;
    for (int64_t k = 0; k < n; ++k) {
        int c = sym[k];
        uint64_t cum = 0;
        for (int j = 0; j < c; ++j)
            cum += cnt[j];
        uint64_t w = hi - lo + 1;
        hi = lo + w * (cum + cnt[c]) / total - 1;
        lo = lo + w * cum / total;
        for (;;) {
            if (hi < AC_HALF) {
                if (ac_put(out, cap, &nb, 0)) return -1;
                for (; follow > 0; --follow)
                    if (ac_put(out, cap, &nb, 1)) return -1;
            } else if (lo >= AC_HALF) {
                if (ac_put(out, cap, &nb, 1)) return -1;
                for (; follow > 0; --follow)
                    if (ac_put(out, cap, &nb, 0)) return -1;
                lo -= AC_HALF;
                hi -= AC_HALF;
            } else if (lo >= AC_QTR && hi < AC_3QTR) {
                follow += 1;
                lo -= AC_QTR;
                hi -= AC_QTR;
            } else {
                break;
            }
            lo = 2 * lo;
            hi = 2 * hi + 1;
        }
        if (adaptive) {
            cnt[c] += 1;
            total += 1;
        }
    }
    follow += 1;
    int b = lo >= AC_QTR;
    if (ac_put(out, cap, &nb, b)) return -1;
    for (; follow > 0; --follow)
        if (ac_put(out, cap, &nb, !b)) return -1;
    return nb;
}

/* The inverse of oracle_ac_encode: the decoder holds the 32 stream bits that
 * follow its interval's origin (bits past the end read as zero), finds the
 * symbol whose sub-interval holds them and applies the same interval steps. */
int oracle_ac_decode(const uint32_t *in, int64_t nbits, int64_t n, int N, int adaptive, int32_t *sym)
{
    uint64_t lo = 0, hi = 0xFFFFFFFFull, total = (uint64_t)N, val = 0;
    int64_t pos = 0;
    uint32_t cnt[4096];
    if (N > 4096)
        return -1;
    for (int c = 0; c < N; ++c)
        cnt[c] = 1;
    for (int i = 0; i < 32; ++i, ++pos)
        val = 2 * val + (pos < nbits ? (in[pos >> 5] >> (31 - (pos & 31))) & 1 : 0);
    for (int64_t k = 0; k < n; ++k) {
        uint64_t w = hi - lo + 1;
        uint64_t target = ((val - lo + 1) * total - 1) / w;
        int c = 0;
        uint64_t cum = 0;
        while (cum + cnt[c] <= target) {
            cum += cnt[c];
            ++c;
        }
        sym[k] = c;
        hi = lo + w * (cum + cnt[c]) / total - 1;
        lo = lo + w * cum / total;
        for (;;) {
            if (hi < AC_HALF) {
            } else if (lo >= AC_HALF) {
                lo -= AC_HALF;
                hi -= AC_HALF;
                val -= AC_HALF;
            } else if (lo >= AC_QTR && hi < AC_3QTR) {
                lo -= AC_QTR;
                hi -= AC_QTR;
                val -= AC_QTR;
            } else {
                break;
            }
            lo = 2 * lo;
            hi = 2 * hi + 1;
            val = 2 * val + (pos < nbits ? (in[pos >> 5] >> (31 - (pos & 31))) & 1 : 0);
            ++pos;
        }
        if (adaptive) {
            cnt[c] += 1;
            total += 1;
        }
    }
    return 0;
}

/* Thread count the OpenMP runtime will use (reported beside CPU timings). */
int oracle_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}
