/*
 * fkv.h -- C ABI of the GB300 fractal KV-cache archive.
 *
 * The archive of arXiv 2607.07144: archived K/V head vectors are reduced to
 * per-head residual-VQ indices (Sec. 3 "Setup"), the indices of each
 * (sequence, layer) form a symbol stream, and the stream is stored by the
 * contractive iterated-map code of Sec. 1 "The code" -- one float64 point per
 * fixed-length span -- which gives lossless, linear-time encoding, O(1)
 * random access and O(1) amortised append (Sec. 2, Table 1).
 *
 * Conventions for every call
 *   - Return value: FKV_OK (0) or a negative FKV_E* code; on error the reason
 *     is available from fkv_last_error(ctx) and nothing was launched.
 *   - Pointers named *_dev (and every data pointer unless stated "host") are
 *     CUDA device pointers owned by the caller; the library never frees them.
 *   - `stream` is a cudaStream_t passed as void*; NULL is the legacy default
 *     stream.  Every call is asynchronous on that stream.
 *   - Errors found on the device (corrupt points, a failed anchor check) are
 *     recorded in a per-context status word; fkv_sync_status() waits for the
 *     stream and returns (and clears) it.  Kernels never trap.
 *   - A context is not thread-safe: calls on one context must be serialised.
 *   - Symbols are uint8 for alphabets N <= 256 (the paper's k = 256
 *     codebooks) and uint16 (native byte order, 2-byte aligned) for
 *     256 < N <= 1024 (the k = 1024 rows of Table 2); fkv_symbol_bytes()
 *     gives the width.  Symbol strides and counts are in symbols.
 *   - A point is two float64 (x, y), 16 bytes; one point per span.
 */
#ifndef FKV_H
#define FKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FKV_OK 0
#define FKV_EINVAL (-1)      /* bad argument: range, null pointer, shape */
#define FKV_ERANGE (-2)      /* a position or record index outside a stream */
#define FKV_ENOMEM (-3)      /* device or host allocation failed */
#define FKV_ECUDA (-4)       /* a CUDA runtime/driver call failed */
#define FKV_ECORRUPT (-5)    /* device status: anchor check failed / bad point */
#define FKV_ETIMEOUT (-6)    /* device status: a bounded device wait ran out */

/* Element types of K/V caches. */
#define FKV_F32 0
#define FKV_F16 1
#define FKV_BF16 2

typedef struct fkv_ctx fkv_ctx;
typedef struct fkv_streams fkv_streams;

/* ------------------------------------------------------------ geometry --- */

/* Sec. 1 and Fig. 1 caption: the packing ("kissing") ratio r_N, the largest
 * contraction ratio for which the N cells V(c) + r (P - V(c)) of the regular
 * N-gon P are disjoint.  The paper prints no formula; this library uses the
 * touching ratio of adjacent cells,
 *     r_N = 1 / (2 (1 + sum_{k=1}^{floor(N/4)} cos(2 pi k / N))),
 * which is exactly 1/2 for N = 3 and N = 4 as the paper states.
 * Returns 0.0 for N < 3 or N > 1024. */
double fkv_packing_ratio(int N);

/* Sec. 1: inversion amplifies rounding by 1/r per step, so one IEEE-754
 * double carries about 44 / log2(1/r) symbols.  Returns
 * floor(44 / log2(1/r)), or 0 when r is outside (0, 1/2]. */
int fkv_max_span_len(double r);

/* ----------------------------------------------------------- context --- */

/* Residual-VQ codebooks (Sec. 3 "Setup", Table 2): K codewords per stage
 * (K = codewords), one codebook per layer, K or V, stage and either KV head
 * (per-head, pooled = 0) or the whole layer (pooled = 1: all heads of a layer
 * share it).  With Hc = pooled ? 1 : n_heads, all host memory, float32,
 * row-major:
 *   k: [n_layers][Hc][stages_k][K][dim]
 *   v: [n_layers][Hc][stages_v][K][dim]
 * K = 256 (0 is read as 256): dim 64 or 128, stages_k, stages_v in [1, 8].
 * K = 1024 (uint16 symbols): dim 64, stages_k, stages_v in [1, 2]. */
typedef struct {
    int n_layers;
    int n_heads;
    int dim;
    int stages_k;
    int stages_v;
    const float *k;
    const float *v;
    int codewords;
    int pooled;
} fkv_codebooks;

/* Create a context for alphabet size N in [3, 1024], contraction ratio r in
 * (0, r_N] (r_N per fkv_packing_ratio, with a relative slack of 1e-12) and
 * span length span_len in [1, fkv_max_span_len(r)] (Sec. 1; at most 5
 * symbols for N = 1024).  cb may be NULL
 * for a symbol-only codec; when given, its codebooks are copied to the
 * current CUDA device (the caller keeps ownership of cb's arrays) and N must
 * equal its codewords per stage.  The context owns the vertex table V(c) (Sec. 1: unit circumradius,
 * V(0) = (1, 0), counter-clockwise), the codebook copies and a status word.
 * *out receives the context, or NULL on failure.  Synchronous. */
int fkv_create(int N, double r, int span_len, const fkv_codebooks *cb, fkv_ctx **out);

/* Free a context and everything it owns.  NULL is accepted.  Synchronises
 * the device. */
int fkv_destroy(fkv_ctx *ctx);

/* Copy the vertex table V(c), c = 0..N-1, to host memory out[N][2]. */
int fkv_vertices(const fkv_ctx *ctx, double *out);

/* Alphabet size, ratio and span length of a context (any pointer may be NULL). */
int fkv_params(const fkv_ctx *ctx, int *N, double *r, int *span_len);

/* Bytes per symbol in every symbol array of the context: 1 (uint8) for
 * N <= 256, 2 (uint16) above; 0 for a NULL context. */
int fkv_symbol_bytes(const fkv_ctx *ctx);

/* Last error message of the context (static storage, never NULL). */
const char *fkv_last_error(const fkv_ctx *ctx);

/* Wait for `stream`, then return and clear the device status word:
 * FKV_OK, or the first of FKV_ETIMEOUT (a bounded device wait ran out),
 * FKV_ECORRUPT (a corrupt point or symbol) and FKV_ERANGE (a request named a
 * position, record or stream outside the archive) that was recorded. */
int fkv_sync_status(fkv_ctx *ctx, void *stream);

/* -------------------------------------------------- bulk symbol codec --- */

/* Sec. 1 / Sec. 2: span-parallel encoding.  Encodes n_streams streams of n
 * symbols each.  Stream i's symbols are sym_dev[i * sym_stride + k],
 * k < n (sym_dev typed per fkv_symbol_bytes; sym_stride in symbols, >= n).  Every span of span_len symbols starts
 * at the anchor (0, 0) and applies, per symbol c, p <- V(c) + r (p - V(c))
 * as the binary64 sequence d = p - V(c), t = r * d, p = V(c) + t (no FMA);
 * the point after the span's last symbol is stored.  The last span of a
 * stream holds n mod span_len symbols when that is nonzero.  Output: stream i,
 * span j is the point at pts_dev[2 * (i * pt_stride + j)] (x then y),
 * pt_stride (in points) >= ceil(n / span_len).  Symbols >= N are reported as
 * FKV_ECORRUPT in the status word (their span's point is written as NaN). */
int fkv_span_encode(fkv_ctx *ctx, const void *sym_dev, int64_t n_streams, int64_t n,
                    int64_t sym_stride, double *pts_dev, int64_t pt_stride, void *stream);

/* Sec. 1: span-parallel decoding, the inverse of fkv_span_encode (same
 * layouts).  Each span is decoded from its stored point, last symbol first:
 * the symbol is the vertex whose cell holds the point (the nearest vertex,
 * since r <= r_N puts every cell inside its vertex's Voronoi region), then
 * p <- (p - (1 - r) V(c)) / r.  After a span's first symbol the point must be
 * back at the anchor: a residual above 2^-4 in either coordinate sets
 * FKV_ECORRUPT in the status word (the symbols are still written). */
int fkv_span_decode(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n,
                    int64_t pt_stride, void *sym_dev, int64_t sym_stride, void *stream);

/* Sec. 2, Table 1: O(1) random access.  For each request q < n_req,
 * req_dev[2q] = stream index, req_dev[2q + 1] = symbol position, writes the
 * symbol at that position to out_dev[q] by decoding only the span holding it
 * (at most span_len backward steps).  Points laid out as in fkv_span_encode.
 * out_dev holds symbols of the context's width.  A request outside
 * [0, n_streams) x [0, n) writes all ones (0xFF or 0xFFFF) to out_dev[q] and
 * sets FKV_ERANGE in the status word. */
int fkv_read(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n, int64_t pt_stride,
             const int64_t *req_dev, int64_t n_req, void *out_dev, void *stream);

/* The same three calls for a ragged batch: streams of different lengths in
 * one call, as the sequences of a serving batch are (Sec. 2 applies the code
 * per sequence; nothing in it ties the streams' lengths together).
 *   sym_off_dev: int64 [n_streams + 1], DEVICE memory, caller-owned: stream
 *                i's symbols are sym_dev[sym_off_dev[i] .. sym_off_dev[i+1])
 *                (symbols of the context's width), len_i their count;
 *   pt_off_dev:  int64 [n_streams + 1], DEVICE memory, caller-owned: stream
 *                i's points occupy point slots [pt_off_dev[i],
 *                pt_off_dev[i+1]) of pts_dev (slot g at pts_dev[2 g]), at
 *                least ceil(len_i / span_len) of them; slots past the
 *                stream's last span are left untouched.
 * Both arrays must be nondecreasing.  The host checks pointers and alignment
 * (FKV_EINVAL, nothing launched); the offsets are read on the device, where a
 * stream with a negative length or too few point slots is skipped and sets
 * FKV_ERANGE in the status word.  Span contents, arithmetic and the corrupt
 * status are those of fkv_span_encode / fkv_span_decode.  fkv_read_ragged
 * takes requests req_dev[2q] = stream, req_dev[2q + 1] = position within
 * that stream; a request outside [0, n_streams) x [0, len_i) writes all ones
 * to out_dev[q] and sets FKV_ERANGE. */
int fkv_span_encode_ragged(fkv_ctx *ctx, const void *sym_dev, const int64_t *sym_off_dev, int64_t n_streams,
                           double *pts_dev, const int64_t *pt_off_dev, void *stream);
int fkv_span_decode_ragged(fkv_ctx *ctx, const double *pts_dev, const int64_t *pt_off_dev, int64_t n_streams,
                           void *sym_dev, const int64_t *sym_off_dev, void *stream);
int fkv_read_ragged(fkv_ctx *ctx, const double *pts_dev, const int64_t *pt_off_dev, const int64_t *sym_off_dev,
                    int64_t n_streams, const int64_t *req_dev, int64_t n_req, void *out_dev, void *stream);

/* Sec. 5: in-place suffix retrieval over the stored points, with no
 * decompression of the archive.  query (host memory, the context's symbol
 * width) holds qlen symbols, 1 <= qlen <= span_len, each < N; it is encoded
 * from the origin by the Sec. 1 map.  Two positions sharing an l-symbol
 * suffix have points within 2 r^l, so every stored point of a span of at
 * least qlen symbols with |p - q|^2 <= (2 r^qlen)^2 (binary64, r^qlen by
 * successive multiplication) is a candidate; a candidate is verified by walking its span back qlen steps
 * with the exact decoder and matches when those symbols are the query.  A
 * span-end point carries only its own span's symbols, so a match means: the
 * last qlen symbols of span (stream, span) equal the query.
 *   match_dev: int64 [cap][2], device, caller-owned: (stream, span) of each
 *              match, in no particular order; only the first cap are written;
 *   counts_dev: int64 [2], device, caller-owned: [0] the number of matches
 *              (all of them, even past cap), [1] the number of candidates.
 * Points laid out as in fkv_span_encode.  Returns FKV_EINVAL for a bad qlen,
 * a symbol >= N, a null or misaligned pointer or a negative size. */
int fkv_suffix_search(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n, int64_t pt_stride,
                      const void *query, int qlen, int64_t *match_dev, int64_t cap, int64_t *counts_dev,
                      void *stream);

/* ------------------------------------------------------ lossy archive --- */

/* Sec. 4: lossy operation, with precision allocated across spans by recency.
 * A stream of n symbols has S = ceil(n / span_len) spans; its last keep_exact
 * spans stay exact and the T = max(0, S - keep_exact) older ones are truncated:
 * each coordinate x of the span's point becomes the B-bit two's complement
 * code k = floor(x * 2^(B-1)) (B = bits in [2, 53]; the kept value k 2^-(B-1)
 * is x with the bits below 2^-(B-1) dropped).  Truncation perturbs the point
 * by less than 2^-(B-1) and decoding amplifies that by 1/r per step, so a
 * truncated span keeps its last symbols exact and loses its first ones:
 * roughly (B - 1) / log2(1/r) - 1 trailing symbols survive on random data.
 * Layout: codes_dev is uint32 [n_streams][code_stride], code_stride >=
 * ceil(2 T B / 32) words; span u's x code occupies bits [2uB, 2uB + B) and its
 * y code bits [2uB + B, 2uB + 2B) of the stream's words (bit i of the stream is
 * bit i % 32 of word i / 32), least significant bit first.  tail_dev is
 * float64 [n_streams][tail_stride][2], tail_stride >= S - T: the exact points
 * of spans T .. S-1.  Together they replace the 16 S bytes of points per
 * stream with 4 code_stride + 16 (S - T).
 *
 * fkv_truncate writes the codes of spans 0 .. T-1 from a point array laid out
 * as in fkv_span_encode, and copies spans T .. S-1 to tail_dev when it is not
 * NULL.  Returns FKV_EINVAL for bits outside [2, 53], a negative size, a short
 * stride or a misaligned buffer. */
int fkv_truncate(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n, int64_t pt_stride, int bits,
                 int64_t keep_exact, uint32_t *codes_dev, int64_t code_stride, double *tail_dev,
                 int64_t tail_stride, void *stream);

/* Sec. 4 decode of a lossy archive: every span is decoded from its kept point
 * (the truncated value k 2^-(B-1) or the exact tail point) by the Sec. 1
 * inverse map in the paper's binary64 arithmetic: the nearest vertex (least
 * binary64 squared distance, lowest index on a tie), then
 * p <- (p - (1 - r) V(c)) / r with an IEEE division.  Symbols are written as
 * in fkv_span_decode; no anchor check (a truncated span does not return to
 * the anchor). */
int fkv_lossy_decode(fkv_ctx *ctx, const uint32_t *codes_dev, int64_t code_stride, const double *tail_dev,
                     int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                     void *sym_dev, int64_t sym_stride, void *stream);

/* Sec. 2 random access into a lossy archive: requests as in fkv_read (an
 * out-of-range request writes all ones and sets FKV_ERANGE), each decoded
 * from its span's kept point as fkv_lossy_decode does. */
int fkv_lossy_read(fkv_ctx *ctx, const uint32_t *codes_dev, int64_t code_stride, const double *tail_dev,
                   int64_t tail_stride, int64_t n_streams, int64_t n, int bits, int64_t keep_exact,
                   const int64_t *req_dev, int64_t n_req, void *out_dev, void *stream);

/* ------------------------------------------ probability-weighted maps --- */

/* Sec. 6 eq. (1): the iterated map with maps sized by a source model, i.e.
 * arithmetic coding.  Each of n_streams streams of n symbols (laid out as in
 * fkv_span_encode) is coded on its own, the streams side by side (decoding is
 * sequential within a stream: there is no random access, append or in-place
 * search on this form).  Integer form: a 32-bit interval [lo, hi]; symbol c
 * with cumulative count cum(c), count cnt(c) and count total T gives, with
 * w = hi - lo + 1, lo' = lo + floor(w cum(c) / T) and
 * hi' = lo + floor(w (cum(c) + cnt(c)) / T) - 1; whenever the interval lies in
 * one half of [0, 2^32) that half's bit is emitted (followed by the bits held
 * back for a middle straddle) and the interval doubles; an interval inside the
 * middle half doubles around the middle and holds back one bit; after the last
 * symbol two bits (plus those held back) pick a point inside the interval.
 * Model: counts start at 1 for all N symbols; adaptive = 1 adds one to the
 * coded symbol's count after each step (add-one prequential model, code
 * length close to -sum log2 p(c_k)); adaptive = 0 keeps p(c) = 1/N, the
 * uniform code (log2 N bits per symbol).  n < 2^29.
 * Output: words_dev uint32 [n_streams][word_stride], word_stride >=
 * fkv_ac_capacity_words(ctx, n); stream bit i is bit 31 - i % 32 of word
 * i / 32 (most significant first); nbits_dev int64 [n_streams] receives each
 * stream's bit count.  A symbol >= N is coded as N - 1 and sets FKV_ECORRUPT. */
int64_t fkv_ac_capacity_words(const fkv_ctx *ctx, int64_t n);
int fkv_ac_encode(fkv_ctx *ctx, const void *sym_dev, int64_t n_streams, int64_t n, int64_t sym_stride, int adaptive,
                  uint32_t *words_dev, int64_t word_stride, int64_t *nbits_dev, void *stream);

/* The inverse of fkv_ac_encode: n symbols per stream from the codes (bits past
 * a stream's nbits read as zero).  Bits that no code produces decode to some
 * symbols and set FKV_ECORRUPT. */
int fkv_ac_decode(fkv_ctx *ctx, const uint32_t *words_dev, int64_t word_stride, const int64_t *nbits_dev,
                  int64_t n_streams, int64_t n, int adaptive, void *sym_dev, int64_t sym_stride, void *stream);

/* Measurement utility (no counterpart in the paper): binary64 add and
 * multiply instructions per second of the current device, measured by
 * independent chains of round-to-nearest multiplies and adds (no FMA), the
 * operation mix of the span encoder (Sec. 1: six such operations per
 * symbol).  It is the measured denominator of span encoding's roofline on a
 * GPU whose FP64 rate, not memory, bounds it.  Launches about 30 ms of work
 * on `stream` and waits for it; writes the rate to *ops_per_s (host). */
int fkv_measure_fp64_rate(double *ops_per_s, void *stream);

/* Failure-path check (no counterpart in the paper): runs, in one CTA on
 * `stream`, the bounded device waits of the RVQ kernels against mbarriers
 * that nothing completes, with their teardown (TMEM held and released as the
 * MMA warp does).  The first waiter gives up after limit_ns (1e5..1e9 ns,
 * else FKV_EINVAL) and raises the kernel's abort flag; a second waiter on
 * the same barrier, under the library's full 2 s limit, must leave on that
 * flag.  Waits for the kernel and writes to result[0..5] (host):
 * [0] the first waiter's result (0 = gave up), [1] the second's, [2] 1 if
 * the second left within 2 x limit_ns, [3] a bounded wait on a completed
 * phase (1), [4] one on an open phase (0), [5] 1 once the teardown ran.
 * The timeouts set FKV_ETIMEOUT in ctx's status word: fkv_sync_status()
 * reports and clears it, and the context stays usable. */
int fkv_check_bounded_wait(fkv_ctx *ctx, int64_t limit_ns, int32_t *result, void *stream);

/* -------------------------------------------------- K/V archive path ---- */

/* A K or V cache tensor on the device: head vectors of `dim` contiguous
 * elements indexed by (layer, sequence, head, position) with the element
 * strides below.  The usual layout [n_layers][batch][n_heads][seq][dim] has
 * stride_pos = dim, stride_head = seq * dim, and so on. */
typedef struct {
    void *data;
    int dtype;              /* FKV_F32, FKV_F16 or FKV_BF16 */
    int64_t batch;          /* sequences */
    int64_t seq;            /* positions per (layer, sequence, head) */
    int64_t stride_layer;
    int64_t stride_batch;
    int64_t stride_head;
    int64_t stride_pos;
} fkv_cache;

/* Symbols per token record: n_heads * (stages_k + stages_v). */
int fkv_record_len(const fkv_ctx *ctx);

/* Sec. 3 "Setup": residual-VQ assignment of every archived vector.
 * kv = 0 quantises keys (stages_k stages), kv = 1 values (stages_v).  For
 * each layer l, sequence b, head h and position t in [t0, t1) of `x`, stage
 * by stage the index is the codeword of codebook (l, h or, pooled, l alone,
 * kv, stage) nearest in
 * squared L2 to the running residual (lowest index on a tie), and the
 * residual then drops that codeword.  Indices (symbols of the context's
 * width) are written in token-record order (the paper does not fix one):
 * stream (b * n_layers + l) starts at sym_dev + (b * n_layers + l) *
 * stream_stride (in symbols); the record of position t is
 * record rec0 + (t - t0) of R = fkv_record_len symbols, holding the key
 * indices of heads 0..H-1 (stages inner) then the value indices likewise.
 * Only the kv half of each record is written.  Runs on the tensor cores
 * (tcgen05) with split-fp16 operands whose score error is below 5e-5 of the
 * residual's squared norm; ties closer than that may differ from a float64
 * search. */
int fkv_rvq_encode(fkv_ctx *ctx, int kv, const fkv_cache *x, int64_t t0, int64_t t1,
                   void *sym_dev, int64_t stream_stride, int64_t rec0, void *stream);

/* Sec. 3 "Setup": the reconstruction is the sum of the selected centroids.
 * Rebuilds positions [t0, t0 + n_rec) of every (layer, sequence, head) of
 * k_out and v_out (either may be NULL) from records 0..n_rec-1 of the symbol
 * streams laid out as in fkv_rvq_encode: sum of the stage codewords in
 * float32, stage order, rounded to nearest-even into the cache dtype. */
int fkv_rvq_decode(fkv_ctx *ctx, const void *sym_dev, int64_t stream_stride, int64_t n_rec,
                   fkv_cache *k_out, fkv_cache *v_out, int64_t t0, void *stream);

/* Sec. 1-3: full archive read.  Decodes records 0..n_rec-1 of the
 * batch * n_layers streams (stream (b * n_layers + l) holds n_rec * R symbols,
 * its points at pts_dev + 2 * (b * n_layers + l) * pt_stride) and writes the
 * reconstructed K and V at positions [t0, t0 + n_rec), as fkv_span_decode
 * followed by fkv_rvq_decode.  Uses a context-owned scratch buffer of
 * batch * n_layers * n_rec * R symbols, grown on demand (a synchronous
 * allocation the first time a larger archive is decoded). */
int fkv_decode_kv(fkv_ctx *ctx, const double *pts_dev, int64_t n_rec, int64_t pt_stride,
                  fkv_cache *k_out, fkv_cache *v_out, int64_t t0, void *stream);

/* Allocation-free variant of fkv_decode_kv (the paper has no counterpart;
 * it exists for callers that must not allocate device memory, such as a
 * serving loop whose device memory belongs to its own pool allocator, or a
 * decode step that cannot take the implicit synchronisation of cudaMalloc).
 * Same arguments, layouts and results as fkv_decode_kv, but the decoded
 * symbols go through a 16 MiB scratch array compiled into the library
 * instead of a context-owned buffer: it calls no cudaMalloc or cudaFree.
 * Limit: batch * n_layers * n_rec * fkv_record_len(ctx) *
 * fkv_symbol_bytes(ctx) <= 16 MiB, else
 * FKV_EINVAL with nothing launched (decode fewer sequences per call).  The
 * first call on a device looks up the array's device address (once per
 * device, with that device current); make that first call before any stream
 * capture.  All calls share the array and it keeps the previous call's
 * contents, so calls that can overlap on the GPU race and must be ordered by
 * the caller. */
int fkv_decode_kv_static(fkv_ctx *ctx, const double *pts_dev, int64_t n_rec, int64_t pt_stride,
                         fkv_cache *k_out, fkv_cache *v_out, int64_t t0, void *stream);

/* Host-to-device transfer of the positions that leave the exact window:
 * copies positions [t0, t1) of every (layer, sequence, head) of src_host (a
 * cache view of HOST memory, pinned for full speed) into the same positions
 * of dst_dev (device), n_layers and n_heads from the context, asynchronously
 * on `stream`; both views hold positions contiguously (stride_pos = dim) and
 * share dtype and batch.  The archive path reads only these positions
 * (Sec. 3 "Setup": the 4 sinks and the 32 recent positions stay exact), so an
 * archive write need not move the rest of the cache.  One 2-D copy when the
 * (layer, sequence, head) rows share one pitch on both sides, else one per
 * (layer, sequence). */
int fkv_cache_upload(fkv_ctx *ctx, const fkv_cache *src_host, const fkv_cache *dst_dev, int64_t t0, int64_t t1,
                     void *stream);

/* Sec. 2 random access at record granularity: for each request q,
 * req_dev[2q] = stream (b * n_layers + l), req_dev[2q + 1] = record index,
 * decode only the spans of that record and write its K and V head vectors to
 * out_dev, laid out [n_req][2 (K, V)][n_heads][dim] in `dtype`.  Streams hold
 * n_rec records each, points as in fkv_decode_kv.  Out-of-range requests
 * write zeros and set FKV_ERANGE.  The requests are taken grouped by layer
 * (a counting sort of their indices on the device, so that one layer's
 * codebooks serve the requests in flight).  A batch of at least 512 requests
 * per layer is staged: its records' symbols are decoded into a buffer first,
 * then rebuilt from (codebook group, dimension slice) copies in shared memory
 * as in fkv_decode_kv; smaller batches rebuild each record from codeword rows
 * in L2.  Both give the same values.  The context keeps the index (and symbol)
 * buffer, allocating it on first use and whenever n_req outgrows it (after a
 * synchronisation of `stream`). */
int fkv_read_kv(fkv_ctx *ctx, const double *pts_dev, int64_t n_streams, int64_t n_rec,
                int64_t pt_stride, const int64_t *req_dev, int64_t n_req, void *out_dev,
                int dtype, void *stream);

/* ------------------------------------------------- appendable streams --- */

/* A set of n_streams symbol streams of equal length, owned by the library on
 * the device: points [n_streams][capacity_spans][2] float64, the last point
 * of a stream being its partial tail span's point.  Initial length 0. */
int fkv_streams_create(fkv_ctx *ctx, int64_t n_streams, int64_t capacity_symbols,
                       fkv_streams **out);
int fkv_streams_destroy(fkv_streams *s);

/* Empty every stream of the set (length 0), keeping its device buffer. */
int fkv_streams_reset(fkv_streams *s);

/* Current geometry: symbols per stream, point stride (points between
 * streams) and the device point buffer (valid until the next append that
 * grows the set).  Any output pointer may be NULL. */
int fkv_streams_info(const fkv_streams *s, int64_t *n_streams, int64_t *length,
                     int64_t *pt_stride, double **pts_dev);

/* Sec. 2, Table 1: O(1) amortised append.  Appends m symbols to every stream:
 * stream i's new symbols are sym_dev[i * sym_stride + k], k < m.  Only the
 * tail is re-walked: the partial last span continues from its stored point,
 * later spans start at the anchor; sealed spans are never touched.  The
 * result is bit-identical to encoding the extended streams from scratch.
 * The point buffer grows geometrically (x2) when full, with a device copy. */
int fkv_append(fkv_ctx *ctx, fkv_streams *s, const void *sym_dev, int64_t m,
               int64_t sym_stride, void *stream);

/* Checkpoint: copy a stream set's length and points to host memory
 * (host_pts: [n_streams][ceil(length / span_len)][2]), and rebuild a set
 * from such a copy.  The archive is its own serialised form. */
int fkv_streams_export(const fkv_streams *s, int64_t *length, double *host_pts, void *stream);
int fkv_streams_import(fkv_ctx *ctx, int64_t n_streams, int64_t length, const double *host_pts,
                       fkv_streams **out);

#ifdef __cplusplus
}
#endif
#endif /* FKV_H */
