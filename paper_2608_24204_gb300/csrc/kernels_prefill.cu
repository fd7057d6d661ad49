// Prefill kernels: a chunk of T prompt tokens at positions P..P+T-1 through
// every layer, fp32 activations.  The matrix products here are CUDA-core
// tiled GEMMs with fused epilogues (RoPE + KV append, residual add, SwiGLU).
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace wici {

// ----------------------------------------------------------- embed / norm ----
__global__ void embed_rows_kernel(const uint16_t *E, const int *tok, float *X, int H) {
    const int t = blockIdx.x;
    const uint16_t *row = E + (size_t)tok[t] * H;
    for (int i = threadIdx.x; i < H; i += blockDim.x) X[(size_t)t * H + i] = bf16_to_f32(row[i]);
}

// A[t] = X[t] / sqrt(mean(X[t]^2) + eps) * g
__global__ void rmsnorm_rows_kernel(const float *X, const uint16_t *g, float *A, int H, float eps) {
    __shared__ float s_part[32];
    const int t = blockIdx.x;
    const float *x = X + (size_t)t * H;
    float ss = 0.f;
    for (int i = threadIdx.x; i < H; i += blockDim.x) ss = fmaf(x[i], x[i], ss);
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += s_part[w];
    const float rinv = 1.0f / sqrtf(tot / (float)H + eps);
    for (int i = threadIdx.x; i < H; i += blockDim.x)
        A[(size_t)t * H + i] = x[i] * rinv * bf16_to_f32(g[i]);
}

// --------------------------------------------------------------- epilogues ----
// unit(t, c, v): row t, output columns (c, c+1) with values v[0], v[1]
struct PEpiQKV {  // packed QKV columns -> Q (fp32) and K/V pages (bf16)
    float *Q;
    uint16_t *kv;
    const int *pages;
    const float2 *rope;
    const uint16_t *bias;
    int P, qdim, kvdim, d, nkv;
    size_t page_elems;
    __device__ void pair(int t, int c, float a, float b) const {
        if (bias) {
            a += bf16_to_f32(bias[c]);
            b += bf16_to_f32(bias[c + 1]);
        }
        const int pos = P + t;
        uint16_t *page = kv + (size_t)pages[pos / kPage] * page_elems;
        const int slot = pos % kPage;
        if (c < qdim + kvdim) {
            const int hd = c / d, i = (c % d) >> 1, half = d >> 1;
            const float2 cs = rope[(size_t)pos * half + i];
            const float ra = a * cs.x - b * cs.y;
            const float rb = b * cs.x + a * cs.y;
            if (c < qdim) {
                float *qr = Q + (size_t)t * qdim + hd * d;
                qr[i] = ra;
                qr[i + half] = rb;
            } else {
                uint16_t *kr = page + ((size_t)(hd - qdim / d) * kPage + slot) * d;
                kr[i] = f32_to_bf16(ra);
                kr[i + half] = f32_to_bf16(rb);
            }
        } else {
            const int j = c - qdim - kvdim, vh = j / d, e = j % d;
            uint16_t *vr = page + (size_t)nkv * kPage * d + ((size_t)vh * kPage + slot) * d;
            vr[e] = f32_to_bf16(a);
            vr[e + 1] = f32_to_bf16(b);
        }
    }
};

struct PEpiResidual {  // X[t][c] += v
    float *X;
    int ld;
    __device__ void pair(int t, int c, float a, float b) const {
        X[(size_t)t * ld + c] += a;
        X[(size_t)t * ld + c + 1] += b;
    }
};

struct PEpiSwiGLU {  // interleaved (gate, up) columns -> M[t][c/2] = silu(g) * u
    float *M;
    int ld;
    __device__ void pair(int t, int c, float a, float b) const {
        M[(size_t)t * ld + (c >> 1)] = a / (1.0f + expf(-a)) * b;
    }
};

// ---------------------------------------------------------------- GEMM ------
// C[T][N] = A[T][K] (fp32) . W[N][K]^T (bf16), fp32 accumulation.
// 64x64 output tile, 256 threads, 4x4 outputs per thread.
constexpr int GBM = 64, GBN = 64, GBK = 16;

template <class Epi>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const float *A, const uint16_t *W, int T,
                                                        int N, int K, const Epi epi) {
    __shared__ float As[GBK][GBM + 4];
    __shared__ float Ws[GBK][GBN + 4];
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const int m0 = blockIdx.y * GBM, n0 = blockIdx.x * GBN;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += GBK) {
        for (int i = tid; i < GBM * GBK; i += 256) {
            const int r = i / GBK, k = i % GBK;
            const int gm = m0 + r, gk = k0 + k;
            As[k][r] = (gm < T && gk < K) ? A[(size_t)gm * K + gk] : 0.f;
            const int gn = n0 + r;
            Ws[k][r] = (gn < N && gk < K) ? bf16_to_f32(W[(size_t)gn * K + gk]) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < GBK; ++k) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                a[i] = As[k][ty * 4 + i];
                b[i] = Ws[k][tx * 4 + i];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int t = m0 + ty * 4 + i;
        if (t >= T) continue;
#pragma unroll
        for (int j = 0; j < 4; j += 2) {
            const int c = n0 + tx * 4 + j;
            if (c < N) epi.pair(t, c, acc[i][j], acc[i][j + 1]);
        }
    }
}

// ------------------------------------------------------------ attention -----
// O[t][head] = softmax over keys 0..P+t of (Q[t][head] . K) / sqrt(d), times V.
// One warp per (token, query head); keys read through the page table.
template <int D>
__global__ void __launch_bounds__(128) attn_prefill_kernel(const float *Q, const uint16_t *kv,
                                                           const int *pages, float *O, int P, int T,
                                                           int nq, int nkv, size_t page_elems,
                                                           float qscale) {
    constexpr int EPL = D / 32;
    const int t = blockIdx.x;
    const int head = blockIdx.y * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (head >= nq) return;
    const int g = head / (nq / nkv);
    const int qdim = nq * D;
    float qv[EPL], acc[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
        qv[e] = Q[(size_t)t * qdim + head * D + lane * EPL + e] * qscale;
        acc[e] = 0.f;
    }
    float m = -INFINITY, l = 0.f;
    const int nkeys = P + t + 1;
    for (int s = 0; s < nkeys; ++s) {
        const uint16_t *pg = kv + (size_t)pages[s / kPage] * page_elems;
        const uint16_t *kr = pg + ((size_t)g * kPage + (s % kPage)) * D + lane * EPL;
        const uint16_t *vr = kr + (size_t)nkv * kPage * D;
        float part = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) part = fmaf(qv[e], bf16_to_f32(kr[e]), part);
        const float sc = warp_sum(part);
        const float mx = fmaxf(m, sc);
        const float corr = exp2f(m - mx);
        const float pt = exp2f(sc - mx);
        l = l * corr + pt;
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] = fmaf(pt, bf16_to_f32(vr[e]), acc[e] * corr);
        m = mx;
    }
    const float inv = 1.0f / l;
#pragma unroll
    for (int e = 0; e < EPL; ++e) O[(size_t)t * qdim + head * D + lane * EPL + e] = acc[e] * inv;
}

// --------------------------------------------------------------- RoPE table --
__global__ void rope_table_kernel(float2 *rope, int n_pos, int half, double theta) {
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= n_pos * half) return;
    const int p = idx / half, i = idx % half;
    const double freq = pow(theta, -2.0 * (double)i / (double)(2 * half));
    double s, c;
    sincos((double)p * freq, &s, &c);
    rope[idx] = make_float2((float)c, (float)s);
}

// ================================================================ host =======

template <class Epi>
static cudaError_t gemm(const float *A, const uint16_t *W, int T, int N, int K, const Epi &epi,
                        cudaStream_t st, LaunchHook *hook, const char *name) {
    if (hook) hook->before(name);
    dim3 grid((N + GBN - 1) / GBN, (T + GBM - 1) / GBM);
    gemm_simt_kernel<Epi><<<grid, 256, 0, st>>>(A, W, T, N, K, epi);
    if (hook) hook->after(name);
    return cudaGetLastError();
}

cudaError_t enqueue_prefill_chunk(const Plan &p, const Bufs &b, cudaStream_t st, int P, int T,
                                  int lm_pos_add, LaunchHook *hook) {
    cudaError_t e;
    const float qscale = 1.4426950408889634f / sqrtf((float)p.d);
    embed_rows_kernel<<<T, 256, 0, st>>>(b.W + p.w_embed, b.tok, b.X, p.H);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    for (int l = 0; l < p.L; ++l) {
        const LayerOffsets &lo = p.layer[l];
        uint16_t *kvl = b.KV + (size_t)l * p.kv_layer_elems;
        rmsnorm_rows_kernel<<<T, 256, 0, st>>>(b.X, b.W + lo.attn_norm, b.A, p.H, p.cfg.rms_eps);
        PEpiQKV eq = {b.Q, kvl, b.pages, b.rope, p.cfg.qkv_bias ? b.W + lo.bqkv : nullptr, P, p.qdim,
                      p.kvdim, p.d, p.nkv, p.kv_page_elems};
        if ((e = gemm(b.A, b.W + lo.wqkv, T, p.nqkv, p.H, eq, st, hook, "prefill_qkv")) != cudaSuccess)
            return e;
        dim3 ag(T, (p.nq + 3) / 4);
        if (hook) hook->before("prefill_attention");
        if (p.d == 128)
            attn_prefill_kernel<128><<<ag, 128, 0, st>>>(b.Q, kvl, b.pages, b.O, P, T, p.nq, p.nkv,
                                                        p.kv_page_elems, qscale);
        else
            attn_prefill_kernel<64><<<ag, 128, 0, st>>>(b.Q, kvl, b.pages, b.O, P, T, p.nq, p.nkv,
                                                       p.kv_page_elems, qscale);
        if (hook) hook->after("prefill_attention");
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        if ((e = gemm(b.O, b.W + lo.wo, T, p.H, p.qdim, PEpiResidual{b.X, p.H}, st, hook,
                      "prefill_o_proj")) != cudaSuccess)
            return e;
        rmsnorm_rows_kernel<<<T, 256, 0, st>>>(b.X, b.W + lo.ffn_norm, b.A, p.H, p.cfg.rms_eps);
        if ((e = gemm(b.A, b.W + lo.wgu, T, 2 * p.F, p.H, PEpiSwiGLU{b.M, p.F}, st, hook,
                      "prefill_gate_up")) != cudaSuccess)
            return e;
        if ((e = gemm(b.M, b.W + lo.wd, T, p.H, p.F, PEpiResidual{b.X, p.H}, st, hook,
                      "prefill_down")) != cudaSuccess)
            return e;
    }
    if (lm_pos_add > 0) {
        if ((e = cudaMemcpyAsync(b.x, b.X + (size_t)(T - 1) * p.H, (size_t)p.H * sizeof(float),
                                 cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
            return e;
        return enqueue_lm_head(p, b, st, false, lm_pos_add, hook);
    }
    return cudaSuccess;
}

cudaError_t enqueue_rope_table(const Plan &p, const Bufs &b, cudaStream_t st) {
    const int half = p.d / 2;
    const int n = p.cfg.max_tokens * half;
    rope_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(b.rope, p.cfg.max_tokens, half, p.cfg.rope_theta);
    return cudaGetLastError();
}

}  // namespace wici
