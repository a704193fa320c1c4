// fkv_decode_kv_static: the full archive read of fkv_decode_kv, for callers
// that must not allocate device memory.
//
// fkv_decode_kv keeps the decoded symbols between its two kernels in a
// context-owned buffer that it (re)allocates with cudaMalloc when an archive
// is larger than any seen before -- a call that also synchronises the stream.
// Some callers cannot accept that: a serving loop whose device memory all
// belongs to its own pool allocator (memory taken behind the pool's back can
// make the pool's later requests fail), or a latency-critical decode step that
// may not stall on an implicit device-wide synchronisation.  This entry point
// uses instead a fixed scratch array compiled into the library, so it never
// calls cudaMalloc, cudaFree or any allocating routine.
//
// The array lives for the life of the process on every GPU that loads this
// library and holds kStaticScratchBytes (16 MiB) of decoded symbols: at most
// batch * n_layers * n_rec * R bytes per call (R = fkv_record_len).  It is
// taken from device memory when fkv_create first looks up its address on a
// device (static_scratch_resolve below), not by this entry point.  Every
// call shares it, so calls whose kernels overlap on the GPU (different
// streams without ordering) race on it and must be serialised by the caller.
// It keeps whatever the previous call left; nothing here needs it zeroed,
// because the decode kernel overwrites every byte the gather then reads.
#include "fkv_internal.h"

namespace {

constexpr size_t kStaticScratchBytes = 16u << 20;

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

}  // namespace

// Called by fkv_create with the context's device current.  In host code the
// symbol g_static_scratch is a host-side stand-in and must never be handed to
// a kernel; its device address comes from cudaGetSymbolAddress.  Under lazy
// module loading that first lookup is what loads this file's module and
// takes the 16 MiB array from device memory, so it happens here, inside the
// (synchronous, allocating) context creation, and never inside
// fkv_decode_kv_static.  The address is kept in the context, whose lifetime
// ends before any reset of the device could invalidate it.
int static_scratch_resolve(fkv_ctx *ctx)
{
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess || !p) {
        ctx->err = std::string("static scratch: cudaGetSymbolAddress: ") + cudaGetErrorString(e);
        return FKV_ECUDA;
    }
    ctx->static_scratch = static_cast<uint8_t *>(p);
    ctx->static_scratch_bytes = kStaticScratchBytes;
    return FKV_OK;
}

extern "C" int fkv_decode_kv_static(fkv_ctx *ctx, const double *pts_dev, int64_t n_rec, int64_t pt_stride,
                                    fkv_cache *k_out, fkv_cache *v_out, int64_t t0, void *stream)
{
    if (!ctx)
        return FKV_EINVAL;
    if (!ctx->has_cb) {
        ctx->err = "context has no codebooks";
        return FKV_EINVAL;
    }
    const fkv_cache *ref = k_out ? k_out : v_out;
    if (!ref || !pts_dev || n_rec < 0 || t0 < 0) {
        ctx->err = "bad arguments";
        return FKV_EINVAL;
    }
    if (k_out && v_out && k_out->batch != v_out->batch) {
        ctx->err = "K and V batch differ";
        return FKV_EINVAL;
    }
    if (n_rec == 0)
        return FKV_OK;
    const int64_t R = fkv_record_len(ctx);
    const int64_t n_streams = ref->batch * ctx->Ly;
    const int64_t n = n_rec * R;
    if (n_streams <= 0 || n > static_cast<int64_t>(ctx->static_scratch_bytes) / fkv_symbol_bytes(ctx) / n_streams) {
        ctx->err = "fkv_decode_kv_static: batch * n_layers * n_rec * record_len symbols exceed the 16 MiB static "
                   "scratch; decode fewer sequences per call";
        return FKV_EINVAL;
    }
    if (pt_stride < (n + ctx->L - 1) / ctx->L) {
        ctx->err = "point stride too small";
        return FKV_EINVAL;
    }
    if (reinterpret_cast<uintptr_t>(pts_dev) % 16) {
        ctx->err = "points must be 16-byte aligned";
        return FKV_EINVAL;
    }
    // output views are checked before anything is launched
    if (!check_outputs(ctx, k_out, v_out, n_rec, t0)) {
        ctx->err = "bad output cache view";
        return FKV_EINVAL;
    }
    uint8_t *scratch = ctx->static_scratch;
    if (!scratch) {
        ctx->err = "fkv_decode_kv_static: the context has no static scratch address";
        return FKV_ECUDA;
    }
    // the same planar decode and gathers as fkv_decode_kv, through the static scratch
    return decode_archive(ctx, pts_dev, n_streams, n_rec, pt_stride, scratch, k_out, v_out, t0,
                          static_cast<cudaStream_t>(stream));
}
