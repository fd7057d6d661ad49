// An entry point for callers that cannot allocate device memory: the final
// RMSNorm + LM head + greedy argmax over a caller-given hidden vector, with
// its scratch in a fixed array that lives in this library's device image.
#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdio.h>

#include <mutex>

#include "../../include/wici.h"
#include "common.cuh"
#include "kernels.h"

using namespace wici;

namespace {

// Scratch of the no-allocation LM head: the control words (ticket, token,
// position), one history word and one argmax partial per CTA.  Every GPU that
// loads the library holds this array until the process exits.
constexpr int kNoAllocMaxCtas = 1024;
struct NoAllocScratch {
    int ctrl[CTRL_WORDS];
    int hist[64];
    int2 partials[kNoAllocMaxCtas];
};
static __device__ __align__(256) NoAllocScratch g_noalloc_scratch;

constexpr int kMaxDevices = 64;
std::mutex g_mu;
NoAllocScratch *g_scratch_ptr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};

// errors are reported through wici_last_error(NULL), like wici_create's
int fail(int code, const char *fmt, ...) {
    char buf[256];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_thread_error(buf);
    return code;
}

// Once per device, with that device current: the device address of the
// scratch array (in host code the symbol itself is only a stand-in) and the
// kernels' shared-memory limits.
int setup_device(int dev, NoAllocScratch **out, int *nsm) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) return fail(WICI_E_CUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        if ((e = setup_kernels()) != cudaSuccess)
            return fail(WICI_E_CUDA, "kernel attributes: %s", cudaGetErrorString(e));
        int v = 0;
        if ((e = cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
            return fail(WICI_E_CUDA, "SM count: %s", cudaGetErrorString(e));
        g_scratch_ptr[dev] = (NoAllocScratch *)p;
        g_num_sms[dev] = v;
    }
    *out = g_scratch_ptr[dev];
    *nsm = g_num_sms[dev];
    return WICI_OK;
}

// Hands the token to the caller, or -1 when a bounded wait inside the LM-head
// kernel gave up (its logits are then incomplete and its token meaningless).
__global__ void noalloc_publish_token(const int *ctrl, int32_t *token) {
    token[0] = ctrl[CTRL_ERR] != 0 ? -1 : ctrl[CTRL_TOKEN];
}

}  // namespace

extern "C" int wici_lm_head_argmax_noalloc(void *cuda_stream, const void *lm_head_dev, const void *norm_gain_dev,
                                           const float *x_dev, int32_t hidden, int32_t vocab, float rms_eps,
                                           float *logits_dev, int32_t *token_dev) {
    if (!lm_head_dev || !norm_gain_dev || !x_dev || !logits_dev || !token_dev)
        return fail(WICI_E_ARG, "null pointer argument");
    if (hidden < 8 || hidden > 16384 || hidden % 8 != 0)
        return fail(WICI_E_ARG, "hidden must be a multiple of 8 in [8, 16384], got %d", hidden);
    if (vocab < 1) return fail(WICI_E_ARG, "vocab must be >= 1, got %d", vocab);
    if (!(rms_eps > 0.f)) return fail(WICI_E_ARG, "rms_eps must be > 0");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(WICI_E_CUDA, "no CUDA device: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices) return fail(WICI_E_ARG, "device ordinal %d beyond %d", dev, kMaxDevices);
    NoAllocScratch *sc = nullptr;
    int nsm = 0;
    if (int rc = setup_device(dev, &sc, &nsm)) return rc;
    const int grid = nsm < vocab ? nsm : vocab;
    if (grid > kNoAllocMaxCtas)
        return fail(WICI_E_ARG, "needs %d argmax partials, the fixed scratch holds %d", grid, kNoAllocMaxCtas);
    cudaStream_t st = (cudaStream_t)cuda_stream;
    // the ticket, position, token and error words must start at zero on every call
    if ((e = cudaMemsetAsync(sc->ctrl, 0, sizeof sc->ctrl, st)) != cudaSuccess)
        return fail(WICI_E_CUDA, "clear scratch: %s", cudaGetErrorString(e));
    if ((e = enqueue_lm_head_argmax_raw((const uint16_t *)lm_head_dev, (const uint16_t *)norm_gain_dev, x_dev,
                                        hidden, vocab, rms_eps, logits_dev, sc->ctrl, sc->partials, sc->hist, grid,
                                        st)) != cudaSuccess)
        return fail(WICI_E_CUDA, "launch: %s", cudaGetErrorString(e));
    noalloc_publish_token<<<1, 1, 0, st>>>(sc->ctrl, token_dev);
    if ((e = cudaGetLastError()) != cudaSuccess) return fail(WICI_E_CUDA, "token publish: %s", cudaGetErrorString(e));
    return WICI_OK;
}
