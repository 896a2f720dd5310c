// noalloc.cu -- lm_head_stats without a caller-provided workspace.
//
// Some callers cannot allocate device memory at all: code running inside a
// host framework that owns every allocation, a plugin sandbox that forbids
// cudaMalloc, or a process whose memory pool is already carved up.  For them
// the LM-head kernel can run with its scratch (per-tile partial statistics and
// arrival counters) in a fixed array that lives inside this library, declared
// below.  Every GPU that loads the library holds that array until the process
// exits.
#include <mutex>

#include "kernels.cuh"

namespace tv {

// 16 MiB of partials.  The plan needs one partial per 128 vocabulary entries
// (two per 256-entry tile of a CTA pair) for every row (rows padded to 16, 24
// bytes each): 10 MiB at 256 rows and vocab 200000, 16 MiB up to a vocabulary
// of about 330 000.
constexpr size_t kNoAllocScratchBytes = 16u << 20;
constexpr size_t kNoAllocCounterBytes = 4096;  // 1024 counters, cleared on every call
constexpr int kNoAllocStatusWord = kNoAllocCounterBytes / 4 - 1;  // last counter word: device-detected errors

static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes + kNoAllocCounterBytes];

static std::mutex g_noalloc_mu;
static void *g_noalloc_ptr[256];  // last device address of g_noalloc_scratch seen per device ordinal

// Host code cannot use g_noalloc_scratch as a device address (on the host it
// names a shadow variable).  Outside stream capture the address is looked up
// on every call, so a context that was reset and recreated is seen; while
// `stream` is being captured the address of the last call on this device is
// used, so a first call must come before any capture.
static tb_status noalloc_scratch(cudaStream_t stream, void **out, const char *fn)
{
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return record_error(TB_ECUDA, "%s: no current device: %s", fn, cudaGetErrorString(e));
    if (dev < 0 || dev >= 256)
        return record_error(TB_EINVAL, "%s: device ordinal %d", fn, dev);
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if ((e = cudaStreamIsCapturing(stream, &cap)) != cudaSuccess)
        return record_error(TB_ECUDA, "%s: cudaStreamIsCapturing: %s", fn, cudaGetErrorString(e));
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (cap == cudaStreamCaptureStatusNone) {
        void *p = nullptr;
        if ((e = cudaGetSymbolAddress(&p, g_noalloc_scratch)) != cudaSuccess)
            return record_error(TB_ECUDA, "%s: cudaGetSymbolAddress: %s", fn, cudaGetErrorString(e));
        g_noalloc_ptr[dev] = p;
    } else if (!g_noalloc_ptr[dev]) {
        return record_error(TB_EINVAL, "%s: first call on device %d made during stream capture; make one call "
                                       "outside capture first", fn, dev);
    }
    *out = g_noalloc_ptr[dev];
    return TB_OK;
}

}  // namespace tv

using namespace tv;

extern "C" tb_status lm_head_stats_noalloc(const void *hidden, int n_rows, const void *lm_head, int d_model,
                                           int vocab, int32_t *argmax, float *top1, float *entropy, int flags,
                                           tb_stream stream)
{
    const char *fn = "lm_head_stats_noalloc";
    LmPlan pl;
    tb_status st = lm_validate(hidden, n_rows, lm_head, d_model, vocab, argmax, top1, entropy, fn, &pl);
    if (st != TB_OK)
        return st;
    if (flags & ~TB_DEBUG_EXPIRE_WAIT)
        return record_error(TB_EINVAL, "%s: flags 0x%x (0 or TB_DEBUG_EXPIRE_WAIT)", fn, flags);
    if (pl.ws_bytes > kNoAllocScratchBytes || pl.n_counters > kNoAllocStatusWord)
        return record_error(TB_ECAPACITY, "%s: %d rows x vocab %d need %zu scratch bytes; the built-in array holds %zu",
                            fn, n_rows, vocab, pl.ws_bytes, kNoAllocScratchBytes);
    void *base = nullptr;
    if ((st = noalloc_scratch((cudaStream_t)stream, &base, fn)) != TB_OK)
        return st;
    uint8_t *parts = static_cast<uint8_t *>(base);
    int *counters = reinterpret_cast<int *>(parts + kNoAllocScratchBytes);
    // The array keeps whatever the previous call left; the arrival counters
    // and the status word must start at zero.
    cudaError_t e = cudaMemsetAsync(counters, 0, kNoAllocCounterBytes, (cudaStream_t)stream);
    if (e != cudaSuccess)
        return record_error(TB_ECUDA, "%s: clearing counters: %s", fn, cudaGetErrorString(e));
    int n_sm = 0;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return record_error(TB_ECUDA, "%s: no current device", fn);
    const char *err = "";
    e = lm_head_launch(hidden, n_rows, lm_head, d_model, vocab, argmax, top1, entropy, parts, counters,
                       counters + kNoAllocStatusWord, n_sm, (cudaStream_t)stream, &err,
                       (flags & TB_DEBUG_EXPIRE_WAIT) ? 1 : 0);
    if (e != cudaSuccess)
        return record_error(e == cudaErrorInvalidValue ? TB_EINVAL : TB_ECUDA, "%s: %s", fn,
                            err[0] ? err : cudaGetErrorString(e));
    return record_error(TB_OK, "");
}

extern "C" tb_status lm_head_stats_noalloc_status(int32_t *status, tb_stream stream)
{
    const char *fn = "lm_head_stats_noalloc_status";
    if (!status)
        return record_error(TB_EINVAL, "%s: status is NULL", fn);
    int32_t w = 0;
    cudaError_t e = cudaMemcpyFromSymbolAsync(&w, g_noalloc_scratch, sizeof w,
                                              kNoAllocScratchBytes + (size_t)kNoAllocStatusWord * 4,
                                              cudaMemcpyDeviceToHost, (cudaStream_t)stream);
    if (e == cudaSuccess)
        e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess)
        return record_error(TB_ECUDA, "%s: %s", fn, cudaGetErrorString(e));
    *status = (w & kStatusTimeout) ? TB_ETIMEOUT : TB_OK;
    return record_error(TB_OK, "");
}
