// C ABI of the CNN-training sample's convolution layer (include/wici.h):
// tensor maps, tile counts and launches of conv_tc_kernel.
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdio.h>

#include <mutex>

#include "../../include/wici.h"
#include "conv_tc.cuh"
#include "kernels.h"

using namespace wici;

namespace {

constexpr size_t kConvErrBytes = 256;   // the error word, then the transposed filter

int fail(int code, const char *fmt, ...) {
    char buf[256];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_thread_error(buf);
    return code;
}

const char *check_shape(const wici_conv_shape *s) {
    if (!s) return "null shape";
    if (s->n < 1 || s->c < 1 || s->k < 1 || s->h < 2 || s->w < 2) return "non-positive dimension";
    if (s->c % CV_BN || s->k % CV_BN) return "c and k must be multiples of 256";
    if (s->h % 2 || s->w % 2) return "h and w must be even";
    return nullptr;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

std::mutex g_mu;
int g_attr_device = -1;

cudaError_t setup(int *nsm) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_attr_device != dev) {
        if ((e = cudaFuncSetAttribute(conv_tc_kernel<CONV_FWD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CV_SMEM)) != cudaSuccess ||
            (e = cudaFuncSetAttribute(conv_tc_kernel<CONV_DGRAD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CV_SMEM)) != cudaSuccess ||
            (e = cudaFuncSetAttribute(conv_tc_kernel<CONV_WGRAD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)CV_SMEM)) != cudaSuccess)
            return e;
        g_attr_device = dev;
    }
    return cudaSuccess;
}

ConvArgs make_args(const wici_conv_shape *s, float *out, void *ws) {
    ConvArgs a = {};
    a.n = s->n; a.c = s->c; a.h = s->h; a.w = s->w; a.k = s->k;
    a.p = s->h / 2; a.q = s->w / 2;
    a.pt = (a.p + 7) / 8;
    a.qt = (a.q + 15) / 16;
    a.out = out;
    a.err = (int *)ws;
    return a;
}

// x [n][h][w][c] with element strides 2 in w and h: boxes of 64 c x `wbox` w x `hbox` h
bool map_x_strided(CUtensorMap *m, const void *x, const wici_conv_shape *s, int wbox, int hbox) {
    const uint64_t dims[4] = {(uint64_t)s->c, (uint64_t)s->w, (uint64_t)s->h, (uint64_t)s->n};
    const uint64_t st[3] = {(uint64_t)s->c * 2, (uint64_t)s->w * s->c * 2, (uint64_t)s->h * s->w * s->c * 2};
    const uint32_t box[4] = {64, (uint32_t)wbox, (uint32_t)hbox, 1};
    const uint32_t es[4] = {1, 2, 2, 1};
    return encode_tiled(m, 4, x, dims, st, box, es);
}

// dy [n][p][q][k]: boxes of 64 k x 16 q x `pbox` p
bool map_dy(CUtensorMap *m, const void *dy, const wici_conv_shape *s, int pbox) {
    const int p = s->h / 2, q = s->w / 2;
    const uint64_t dims[4] = {(uint64_t)s->k, (uint64_t)q, (uint64_t)p, (uint64_t)s->n};
    const uint64_t st[3] = {(uint64_t)s->k * 2, (uint64_t)q * s->k * 2, (uint64_t)p * q * s->k * 2};
    const uint32_t box[4] = {64, 16, (uint32_t)pbox, 1};
    const uint32_t es[4] = {1, 1, 1, 1};
    return encode_tiled(m, 4, dy, dims, st, box, es);
}

// a row-major bf16 matrix [rows][cols]: boxes of 64 columns x 256 rows
bool map_rows(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols) {
    const uint64_t dims[2] = {cols, rows};
    const uint64_t st[1] = {cols * 2};
    const uint32_t box[2] = {64, (uint32_t)CV_BN};
    const uint32_t es[2] = {1, 1};
    return encode_tiled(m, 2, ptr, dims, st, box, es);
}

template <int MODE>
cudaError_t launch(const CUtensorMap &ma, const CUtensorMap &mb, ConvArgs a, int nsm, cudaStream_t st) {
    const int grid = a.ntiles < nsm ? a.ntiles : nsm;
    conv_tc_kernel<MODE><<<grid, CV_THREADS, CV_SMEM, st>>>(ma, mb, a);
    return cudaGetLastError();
}

}  // namespace

extern "C" {

int wici_conv_workspace_bytes(const wici_conv_shape *s, size_t *bytes) {
    if (const char *m = check_shape(s)) return fail(WICI_E_ARG, "conv: %s", m);
    if (!bytes) return fail(WICI_E_ARG, "conv: null output");
    *bytes = kConvErrBytes + (size_t)9 * s->c * s->k * 2;
    return WICI_OK;
}

int wici_conv_forward(void *cuda_stream, const wici_conv_shape *s, const void *x, const void *w, float *y,
                      void *workspace) {
    if (const char *m = check_shape(s)) return fail(WICI_E_ARG, "conv: %s", m);
    if (!aligned16(x) || !aligned16(w) || !aligned16(y) || !aligned16(workspace) || !workspace)
        return fail(WICI_E_ARG, "conv: null or unaligned buffer");
    int nsm = 0;
    cudaError_t e = setup(&nsm);
    if (e != cudaSuccess) return fail(WICI_E_CUDA, "conv: %s", cudaGetErrorString(e));
    CUtensorMap ma, mb;
    if (!map_x_strided(&ma, x, s, 32, 16) || !map_rows(&mb, w, (uint64_t)s->k, (uint64_t)9 * s->c))
        return fail(WICI_E_CUDA, "conv: cuTensorMapEncodeTiled failed");
    ConvArgs a = make_args(s, y, workspace);
    a.ntiles = a.n * a.pt * a.qt * (a.k / CV_BN);
    if ((e = launch<CONV_FWD>(ma, mb, a, nsm, (cudaStream_t)cuda_stream)) != cudaSuccess)
        return fail(WICI_E_CUDA, "conv forward: %s", cudaGetErrorString(e));
    return WICI_OK;
}

int wici_conv_backward_data(void *cuda_stream, const wici_conv_shape *s, const void *dy, const void *w, float *dx,
                            void *workspace) {
    if (const char *m = check_shape(s)) return fail(WICI_E_ARG, "conv: %s", m);
    if (!aligned16(dy) || !aligned16(w) || !aligned16(dx) || !aligned16(workspace) || !workspace)
        return fail(WICI_E_ARG, "conv: null or unaligned buffer");
    int nsm = 0;
    cudaError_t e = setup(&nsm);
    if (e != cudaSuccess) return fail(WICI_E_CUDA, "conv: %s", cudaGetErrorString(e));
    cudaStream_t st = (cudaStream_t)cuda_stream;
    uint16_t *wt = (uint16_t *)((uint8_t *)workspace + kConvErrBytes);
    conv_transpose_filter_kernel<<<dim3((s->c + 31) / 32, (s->k + 31) / 32, 9), dim3(32, 8), 0, st>>>(
        (const uint16_t *)w, wt, s->k, s->c);
    if ((e = cudaGetLastError()) != cudaSuccess) return fail(WICI_E_CUDA, "conv transpose: %s", cudaGetErrorString(e));
    CUtensorMap ma, mb;
    if (!map_dy(&ma, dy, s, 8) || !map_rows(&mb, wt, (uint64_t)9 * s->c, (uint64_t)s->k))
        return fail(WICI_E_CUDA, "conv: cuTensorMapEncodeTiled failed");
    ConvArgs a = make_args(s, dx, workspace);
    a.ntiles = 4 * a.n * a.pt * a.qt * (a.c / CV_BN);
    if ((e = launch<CONV_DGRAD>(ma, mb, a, nsm, st)) != cudaSuccess)
        return fail(WICI_E_CUDA, "conv data gradient: %s", cudaGetErrorString(e));
    return WICI_OK;
}

int wici_conv_backward_filter(void *cuda_stream, const wici_conv_shape *s, const void *x, const void *dy, float *dw,
                              void *workspace) {
    if (const char *m = check_shape(s)) return fail(WICI_E_ARG, "conv: %s", m);
    if (!aligned16(x) || !aligned16(dy) || !aligned16(dw) || !aligned16(workspace) || !workspace)
        return fail(WICI_E_ARG, "conv: null or unaligned buffer");
    int nsm = 0;
    cudaError_t e = setup(&nsm);
    if (e != cudaSuccess) return fail(WICI_E_CUDA, "conv: %s", cudaGetErrorString(e));
    CUtensorMap ma, mb;
    if (!map_dy(&ma, dy, s, 4) || !map_x_strided(&mb, x, s, 32, 8))
        return fail(WICI_E_CUDA, "conv: cuTensorMapEncodeTiled failed");
    ConvArgs a = make_args(s, dw, workspace);
    a.ntiles = 9 * (a.k / CV_BM) * (a.c / CV_BN);
    if ((e = launch<CONV_WGRAD>(ma, mb, a, nsm, (cudaStream_t)cuda_stream)) != cudaSuccess)
        return fail(WICI_E_CUDA, "conv filter gradient: %s", cudaGetErrorString(e));
    return WICI_OK;
}

int wici_conv_status(void *cuda_stream, void *workspace) {
    if (!workspace) return fail(WICI_E_ARG, "conv: null workspace");
    int h = 0;
    cudaStream_t st = (cudaStream_t)cuda_stream;
    cudaError_t e = cudaMemcpyAsync(&h, workspace, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return fail(WICI_E_CUDA, "conv status: %s", cudaGetErrorString(e));
    if (h != 0) {
        cudaMemsetAsync(workspace, 0, sizeof(int), st);
        cudaStreamSynchronize(st);
        return fail(WICI_E_TIMEOUT, "conv: a device-side wait gave up (site %d)", h);
    }
    return WICI_OK;
}

}  // extern "C"
