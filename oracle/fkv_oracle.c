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
