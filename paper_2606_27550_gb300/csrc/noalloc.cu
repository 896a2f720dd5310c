// noalloc.cu -- lm_head_stats without a caller-provided workspace.
//
// Some callers cannot allocate device memory at all: code running inside a
// host framework that owns every allocation, a plugin sandbox that forbids
// cudaMalloc, or a process whose memory pool is already carved up.  For them
// the LM-head kernel can run with its scratch (per-tile partial statistics,
// group partials and arrival counters) in a fixed array that lives inside
// this library, declared below.  Every GPU that loads the library holds that
// array until the process exits.
#include <mutex>

#include "kernels.cuh"

namespace tv {

// 4 MiB of partials: (CTAs + merge groups) x rows (padded to 16) x 24 bytes,
// whatever the vocabulary: about 2 MiB for 256 rows on a GPU with 152 SMs.
constexpr size_t kNoAllocScratchBytes = 4u << 20;
constexpr size_t kNoAllocCounterBytes = 4096;  // 1024 counters, cleared on every call

static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes + kNoAllocCounterBytes];

static std::mutex g_noalloc_mu;
static void *g_noalloc_ptr[256];  // device address of g_noalloc_scratch, per device ordinal

// Host code cannot use g_noalloc_scratch as a device address (on the host it
// names a shadow variable).  Look the device address up once per device.
static cudaError_t noalloc_scratch(void **out)
{
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    if (dev < 0 || dev >= 256)
        return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess)
            return e;
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

}  // namespace tv

using namespace tv;

extern "C" tb_status lm_head_stats_noalloc(const void *hidden, int n_rows, const void *lm_head, int d_model,
                                           int vocab, int32_t *argmax, float *top1, float *entropy, tb_stream stream)
{
    if (!hidden || !lm_head || !argmax || !top1 || !entropy)
        return record_error(TB_EINVAL, "lm_head_stats_noalloc: NULL argument");
    if ((reinterpret_cast<uintptr_t>(hidden) | reinterpret_cast<uintptr_t>(lm_head)) & 15u)
        return record_error(TB_EINVAL, "lm_head_stats_noalloc: hidden / lm_head not 16-byte aligned");
    if (n_rows < 1 || n_rows > 256 || d_model < 8 || d_model % 8 || vocab < 1)
        return record_error(TB_EINVAL, "lm_head_stats_noalloc: n_rows %d (1..256), d_model %d (multiple of 8), vocab %d",
                            n_rows, d_model, vocab);
    int dev = 0, n_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) !=
                                                  cudaSuccess)
        return record_error(TB_ECUDA, "lm_head_stats_noalloc: no current device");
    const LmPlan pl = lm_plan(n_rows, d_model, vocab, n_sm);
    if (pl.ws_bytes > kNoAllocScratchBytes || pl.n_counters + 1 > (int)(kNoAllocCounterBytes / 4))
        return record_error(TB_ECAPACITY,
                            "lm_head_stats_noalloc: %d rows x vocab %d need %zu scratch bytes; the built-in array "
                            "holds %zu",
                            n_rows, vocab, pl.ws_bytes, kNoAllocScratchBytes);
    void *base = nullptr;
    cudaError_t e = noalloc_scratch(&base);
    if (e != cudaSuccess)
        return record_error(TB_ECUDA, "lm_head_stats_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    uint8_t *parts = static_cast<uint8_t *>(base);
    int *counters = reinterpret_cast<int *>(parts + kNoAllocScratchBytes);
    // The array keeps whatever the previous call left; the arrival counters
    // and the status word must start at zero.
    e = cudaMemsetAsync(counters, 0, kNoAllocCounterBytes, (cudaStream_t)stream);
    if (e != cudaSuccess)
        return record_error(TB_ECUDA, "lm_head_stats_noalloc: clearing counters: %s", cudaGetErrorString(e));
    const char *err = "";
    int *status = counters + (kNoAllocCounterBytes / 4 - 1);  // last word: device-detected errors
    e = lm_head_launch(hidden, n_rows, lm_head, d_model, vocab, argmax, top1, entropy, parts, counters, status, n_sm,
                       (cudaStream_t)stream, &err);
    if (e != cudaSuccess)
        return record_error(e == cudaErrorInvalidValue ? TB_EINVAL : TB_ECUDA, "lm_head_stats_noalloc: %s",
                            err[0] ? err : cudaGetErrorString(e));
    return record_error(TB_OK, "");
}
