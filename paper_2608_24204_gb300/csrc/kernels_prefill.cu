// Prefill: a chunk of T prompt tokens at positions P..P+T-1 through every
// layer.  The four linear maps of a layer run on the tcgen05 GEMM (gemm_tc.cuh)
// with fused epilogues (bias + RoPE + paged KV append, residual add, SwiGLU)
// and the causal attention on the tcgen05 attention kernel (attn_tc.cuh); the
// kernels around them produce the tensor-core operands as bf16 hi/lo pairs.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "common.cuh"
#include "attn_tc.cuh"
#include "gemm_tc.cuh"
#include "kernels.h"

namespace wici {

// output-tile widths of the prefill GEMMs: 128 x 192 tiles (three 72 KB ring
// stages) or 128 x 128 tiles (three 64 KB stages), chosen per weight matrix
// for the fewest whole waves of tiles at the largest chunk
// output-tile width: the fewest columns per SM over the waves of tiles, a
// 128-column tile charged 10% for reading its A operand more often per FLOP;
// 224 only for GEMMs of two activation terms (three leave too few ring stages)
static int pick_bn(int T, int N, int sms, bool allow224) {
    const int tm = (T + TC_BM - 1) / TC_BM;
    int best = 0;
    double best_cost = 0.0;
    for (int bn : {128, 192, 224}) {
        if (bn == 224 && !allow224) continue;
        const int waves = (tm * ((N + bn - 1) / bn) + sms - 1) / sms;
        const double cost = (double)waves * bn * (bn == 128 ? 1.1 : 1.0);
        if (best == 0 || cost < best_cost) {
            best = bn;
            best_cost = cost;
        }
    }
    return best;
}

// store a as its three bf16 terms
__device__ __forceinline__ void split_store(uint16_t *const *t, size_t i, float a) {
    uint16_t t0, t1, t2;
    split_bf16x3(a, t0, t1, t2);
    t[0][i] = t0;
    t[1][i] = t1;
    t[2][i] = t2;
}

struct Terms {   // kTerms pointers passed by value to kernels
    uint16_t *p[kTerms];
};

// ----------------------------------------------------------- embed / norm ----
__global__ void embed_rows_kernel(const uint16_t *E, const int *tok, float *X, int H) {
    const int t = blockIdx.x;
    const uint16_t *row = E + (size_t)tok[t] * H;
    for (int i = threadIdx.x; i < H; i += blockDim.x) X[(size_t)t * H + i] = bf16_to_f32(row[i]);
}

// A[t] = X[t] / sqrt(mean(X[t]^2) + eps) * g, stored as three bf16 terms
// One CTA per row t: RMSNorm of x_t with gain g, stored as the first `nterms`
// bf16 terms of the next GEMM's operand (its kATerms).  H % 8 == 0: 8-element
// chunks, one 16-byte store per term.
__global__ void rmsnorm_rows_kernel(const float *X, const uint16_t *g, const Terms A, int H, float eps,
                                    int nterms) {
    __shared__ float s_part[32];
    const int t = blockIdx.x;
    const float4 *x = reinterpret_cast<const float4 *>(X + (size_t)t * H);
    const int nc = H >> 3;
    float ss = 0.f;
    for (int c = threadIdx.x; c < nc; c += blockDim.x) {
        const float4 u = x[2 * c], v = x[2 * c + 1];
        ss = fmaf(u.x, u.x, ss); ss = fmaf(u.y, u.y, ss); ss = fmaf(u.z, u.z, ss); ss = fmaf(u.w, u.w, ss);
        ss = fmaf(v.x, v.x, ss); ss = fmaf(v.y, v.y, ss); ss = fmaf(v.z, v.z, ss); ss = fmaf(v.w, v.w, ss);
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += s_part[w];
    const float rinv = 1.0f / sqrtf(tot / (float)H + eps);
    for (int c = threadIdx.x; c < nc; c += blockDim.x) {
        const float4 u = x[2 * c], v = x[2 * c + 1];
        const uint4 gw = reinterpret_cast<const uint4 *>(g)[c];
        const float y[8] = {u.x * rinv * bf16lo(gw.x), u.y * rinv * bf16hi(gw.x), u.z * rinv * bf16lo(gw.y),
                            u.w * rinv * bf16hi(gw.y), v.x * rinv * bf16lo(gw.z), v.y * rinv * bf16hi(gw.z),
                            v.z * rinv * bf16lo(gw.w), v.w * rinv * bf16hi(gw.w)};
        uint32_t w[kTerms][4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            uint16_t a0[kTerms], a1[kTerms];
            split_bf16x3(y[2 * e], a0[0], a0[1], a0[2]);
            split_bf16x3(y[2 * e + 1], a1[0], a1[1], a1[2]);
#pragma unroll
            for (int q = 0; q < kTerms; ++q) w[q][e] = (uint32_t)a0[q] | ((uint32_t)a1[q] << 16);
        }
        const size_t o = (size_t)t * H + 8 * (size_t)c;
#pragma unroll
        for (int q = 0; q < kTerms; ++q)
            if (q < nterms) *reinterpret_cast<uint4 *>(A.p[q] + o) = make_uint4(w[q][0], w[q][1], w[q][2], w[q][3]);
    }
}

// --------------------------------------------------------------- epilogues ----
// pair(t, c, a, b): GEMM output row t, columns (c, c + 1)
struct PEpiQKV {  // packed QKV columns -> Q (three bf16 terms) and K/V pages (bf16)
    static constexpr bool kRow = true;
    static constexpr int kATerms = kTerms;   // activation terms the GEMM multiplies
    Terms Q;
    uint16_t *kv;
    const int *pages;
    const float2 *rope;
    const uint16_t *bias;
    int P, qdim, kvdim, d, nkv;
    size_t page_elems;
    float *raw;      // qk_norm: q | k of row t land here as they are ([t][qdim + kvdim], natural order)
    __device__ void pair(int t, int c, float a, float b) const {
        if (bias) {
            a += bf16_to_f32(bias[c]);
            b += bf16_to_f32(bias[c + 1]);
        }
        const int pos = P + t;
        uint16_t *page = kv + (size_t)pages[pos / kPage] * page_elems;
        const int slot = pos % kPage;
        if (raw && c < qdim + kvdim) {
            const int hd = c / d, i = (c % d) >> 1, half = d >> 1;
            float *dst = raw + (size_t)t * (qdim + kvdim) + hd * d;
            dst[i] = a;
            dst[i + half] = b;
        } else if (c < qdim + kvdim) {
            const int hd = c / d, i = (c % d) >> 1, half = d >> 1;
            const float2 cs = rope[(size_t)pos * half + i];
            const float ra = a * cs.x - b * cs.y;
            const float rb = b * cs.x + a * cs.y;
            if (c < qdim) {
                const size_t qo = (size_t)t * qdim + hd * d + i;
                split_store(Q.p, qo, ra);
                split_store(Q.p, qo + half, rb);
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
    // 16 columns at a time: one head and one of q / k / v (head_dim, qdim and
    // kvdim are multiples of 64), 16-byte stores
    template <int NC>
    __device__ __forceinline__ void row(int t, int c0, const float (&v)[NC], int n) const {
        const int pos = P + t;
        uint16_t *page = kv + (size_t)pages[pos / kPage] * page_elems;
        const int slot = pos % kPage, half = d >> 1;
#pragma unroll
        for (int g = 0; g < NC; g += 16) {
            const int c = c0 + g;
            if (g + 16 > n) {
#pragma unroll
                for (int k = 0; k < 16; k += 2)
                    if (g + k + 1 < n) pair(t, c + k, v[g + k], v[g + k + 1]);
                continue;
            }
            float x[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) x[k] = v[g + k] + (bias ? bf16_to_f32(bias[c + k]) : 0.f);
            if (raw && c < qdim + kvdim) {
                // 8 RoPE pairs (i0 + k, i0 + k + d/2) of one head, unnormalised
                const int hd = c / d, i0 = (c % d) >> 1;
                float *dst = raw + (size_t)t * (qdim + kvdim) + hd * d + i0;
                *reinterpret_cast<float4 *>(dst) = make_float4(x[0], x[2], x[4], x[6]);
                *reinterpret_cast<float4 *>(dst + 4) = make_float4(x[8], x[10], x[12], x[14]);
                *reinterpret_cast<float4 *>(dst + half) = make_float4(x[1], x[3], x[5], x[7]);
                *reinterpret_cast<float4 *>(dst + half + 4) = make_float4(x[9], x[11], x[13], x[15]);
            } else if (c < qdim + kvdim) {
                const int hd = c / d, i0 = (c % d) >> 1;
                float ra[8], rb[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const float2 cs = rope[(size_t)pos * half + i0 + k];
                    ra[k] = x[2 * k] * cs.x - x[2 * k + 1] * cs.y;
                    rb[k] = x[2 * k + 1] * cs.x + x[2 * k] * cs.y;
                }
                if (c < qdim) {
                    const size_t qo = (size_t)t * qdim + hd * d + i0;
                    uint32_t wa[kTerms][4], wb[kTerms][4];
#pragma unroll
                    for (int k = 0; k < 8; k += 2) {
                        uint16_t a0[kTerms], a1[kTerms], b0[kTerms], b1[kTerms];
                        split_bf16x3(ra[k], a0[0], a0[1], a0[2]);
                        split_bf16x3(ra[k + 1], a1[0], a1[1], a1[2]);
                        split_bf16x3(rb[k], b0[0], b0[1], b0[2]);
                        split_bf16x3(rb[k + 1], b1[0], b1[1], b1[2]);
#pragma unroll
                        for (int q = 0; q < kTerms; ++q) {
                            wa[q][k >> 1] = (uint32_t)a0[q] | ((uint32_t)a1[q] << 16);
                            wb[q][k >> 1] = (uint32_t)b0[q] | ((uint32_t)b1[q] << 16);
                        }
                    }
#pragma unroll
                    for (int q = 0; q < kTerms; ++q) {
                        *reinterpret_cast<uint4 *>(Q.p[q] + qo) = make_uint4(wa[q][0], wa[q][1], wa[q][2], wa[q][3]);
                        *reinterpret_cast<uint4 *>(Q.p[q] + qo + half) =
                            make_uint4(wb[q][0], wb[q][1], wb[q][2], wb[q][3]);
                    }
                } else {
                    uint16_t *kr = page + ((size_t)(hd - qdim / d) * kPage + slot) * d + i0;
                    uint32_t wa[4], wb[4];
#pragma unroll
                    for (int k = 0; k < 8; k += 2) {
                        wa[k >> 1] = (uint32_t)f32_to_bf16(ra[k]) | ((uint32_t)f32_to_bf16(ra[k + 1]) << 16);
                        wb[k >> 1] = (uint32_t)f32_to_bf16(rb[k]) | ((uint32_t)f32_to_bf16(rb[k + 1]) << 16);
                    }
                    *reinterpret_cast<uint4 *>(kr) = make_uint4(wa[0], wa[1], wa[2], wa[3]);
                    *reinterpret_cast<uint4 *>(kr + half) = make_uint4(wb[0], wb[1], wb[2], wb[3]);
                }
            } else {
                const int j = c - qdim - kvdim, vh = j / d, e0 = j % d;
                uint16_t *vr = page + (size_t)nkv * kPage * d + ((size_t)vh * kPage + slot) * d + e0;
                uint32_t w[8];
#pragma unroll
                for (int k = 0; k < 16; k += 2)
                    w[k >> 1] = (uint32_t)f32_to_bf16(x[k]) | ((uint32_t)f32_to_bf16(x[k + 1]) << 16);
                *reinterpret_cast<uint4 *>(vr) = make_uint4(w[0], w[1], w[2], w[3]);
                *reinterpret_cast<uint4 *>(vr + 8) = make_uint4(w[4], w[5], w[6], w[7]);
            }
        }
    }
};

// row(t, c0, v, n): output row t, columns c0 .. c0 + n of one thread's span
// (NC consecutive columns, c0 a multiple of 32), written with 16-byte stores
struct PEpiResidual {  // X[t][c] += v
    float *X;
    int ld;
    static constexpr bool kRow = true;
    // the O and down GEMMs multiply two terms of their activations (o, m): with
    // gate/up also at two terms, measured at 1.36e-2 max-abs against the fp64
    // oracle at the Qwen2.5-14B shape (1.30e-2 with three); the QKV GEMM keeps
    // three terms (two there fail the 2e-2 tolerance)
    static constexpr int kATerms = 2;
    __device__ void pair(int t, int c, float a, float b) const {
        float2 *p = reinterpret_cast<float2 *>(X + (size_t)t * ld + c);
        float2 v = *p;
        v.x += a;
        v.y += b;
        *p = v;
    }
    template <int NC>
    __device__ __forceinline__ void row(int t, int c0, const float (&v)[NC], int n) const {
        float *x = X + (size_t)t * ld + c0;
#pragma unroll
        for (int j = 0; j < NC; j += 4) {
            if (j + 4 <= n) {
                float4 *p = reinterpret_cast<float4 *>(x + j);
                float4 a = *p;
                a.x += v[j]; a.y += v[j + 1]; a.z += v[j + 2]; a.w += v[j + 3];
                *p = a;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (j + e < n) x[j + e] += v[j + e];
            }
        }
    }
};

struct PEpiSwiGLU {  // interleaved (gate, up) columns -> M[t][c/2] = silu(g) * u as three terms
    Terms M;
    int ld;
    static constexpr bool kRow = true;
    // the gate/up GEMM multiplies two terms of its activation (16 significant bits):
    // measured against the fp64 oracle at the 8B and 14B shapes, it moves the
    // logits by less than 1e-4, where two terms in every GEMM fail the tolerance
    static constexpr int kATerms = 2;
    __device__ void pair(int t, int c, float a, float b) const {
        split_store(M.p, (size_t)t * ld + (c >> 1), a / (1.0f + expf(-a)) * b);
    }
    template <int NC>
    __device__ __forceinline__ void row(int t, int c0, const float (&v)[NC], int n) const {
        const size_t o = (size_t)t * ld + (c0 >> 1);
#pragma unroll
        for (int j = 0; j < NC; j += 16) {   // 8 outputs: one 16-byte store per term
            if (j + 16 <= n) {
                uint32_t w[kTerms][4];
#pragma unroll
                for (int k = 0; k < 8; k += 2) {
                    const float g0 = v[j + 2 * k], u0 = v[j + 2 * k + 1];
                    const float g1 = v[j + 2 * k + 2], u1 = v[j + 2 * k + 3];
                    uint16_t a[kTerms], b[kTerms];
                    split_bf16x3(g0 / (1.0f + expf(-g0)) * u0, a[0], a[1], a[2]);
                    split_bf16x3(g1 / (1.0f + expf(-g1)) * u1, b[0], b[1], b[2]);
#pragma unroll
                    for (int q = 0; q < kTerms; ++q) w[q][k >> 1] = (uint32_t)a[q] | ((uint32_t)b[q] << 16);
                }
#pragma unroll
                for (int q = 0; q < kTerms; ++q)
                    *reinterpret_cast<uint4 *>(M.p[q] + o + (j >> 1)) = make_uint4(w[q][0], w[q][1], w[q][2], w[q][3]);
            } else {
#pragma unroll
                for (int k = 0; k < 16; k += 2)
                    if (j + k + 1 < n) pair(t, c0 + j + k, v[j + k], v[j + k + 1]);
            }
        }
    }
};

// ------------------------------------------------- Qwen3 q/k norm (prefill) --
// One warp per (row t, head): the head of raw q (or k) RMS-normalised over
// head_dim with its gain, RoPE at position P + t, then q as three bf16 terms in
// Q[t] or k as bf16 in its page slot.  Lane l holds elements l*EPL ..; the RoPE
// partner of element i < d/2 is i + d/2, in lane l + 16.
template <int D>
__global__ void qk_norm_rope_kernel(const float *raw, const uint16_t *qn, const uint16_t *kn, const float2 *rope,
                                    Terms Q, uint16_t *kv, const int *pages, size_t page_elems, int P, int nq,
                                    int nkv, float eps) {
    constexpr int EPL = D / 32, HALF = D / 2;
    const int t = blockIdx.x, lane = threadIdx.x & 31;
    const int hd = blockIdx.y * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (hd >= nq + nkv) return;
    const int qdim = nq * D, kvdim = nkv * D;
    const float *src = raw + (size_t)t * (qdim + kvdim) + (size_t)hd * D + lane * EPL;
    const uint16_t *gain = hd < nq ? qn : kn;
    float v[EPL];
    float ss = 0.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
        v[e] = src[e];
        ss = fmaf(v[e], v[e], ss);
    }
    const float rinv = 1.0f / sqrtf(warp_sum(ss) / (float)D + eps);
    const int pos = P + t;
#pragma unroll
    for (int e = 0; e < EPL; ++e) v[e] = v[e] * rinv * bf16_to_f32(gain[lane * EPL + e]);
    float r[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
        const float other = __shfl_xor_sync(0xffffffffu, v[e], 16);
        const float2 cs = rope[(size_t)pos * HALF + (lane * EPL + e) % HALF];
        r[e] = lane < 16 ? v[e] * cs.x - other * cs.y : v[e] * cs.x + other * cs.y;
    }
    if (hd < nq) {
        const size_t o = (size_t)t * qdim + (size_t)hd * D + lane * EPL;
#pragma unroll
        for (int e = 0; e < EPL; ++e) split_store(Q.p, o + e, r[e]);
    } else {
        uint16_t *kr = kv + (size_t)pages[pos / kPage] * page_elems + ((size_t)(hd - nq) * kPage + pos % kPage) * D +
                       lane * EPL;
#pragma unroll
        for (int e = 0; e < EPL; ++e) kr[e] = f32_to_bf16(r[e]);
    }
}

// ------------------------------------------------ 8-bit block format (prefill) --
// W[r][c] = d[r][c / 32] * code[r][c] of `rows` arena rows (int8 codes, then
// the row's fp16 block scales), written as three bf16 terms of a
// row-major [rows][K] matrix.  The product is exact in fp32 (at most 18
// significant bits), and so is its split into three terms.  8 elements per
// thread: one 8-byte code load, one scale, one 16-byte store per term.
__global__ void q8_dequant_terms_kernel(const uint8_t *src, int rows, int K, const Terms out, int nterms) {
    const int per_row = K / 8;
    const size_t rb = (size_t)K + (size_t)K / 16;
    const long long n = (long long)rows * per_row;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const long long r = i / per_row;
        const int c = (int)(i - r * per_row);
        const uint8_t *row = src + (size_t)r * rb;
        const uint2 w = *reinterpret_cast<const uint2 *>(row + (size_t)c * 8);
        const float d = __half2float(__ushort_as_half(*reinterpret_cast<const unsigned short *>(row + K + (c >> 2) * 2)));
        uint32_t t[kTerms][4];
#pragma unroll
        for (int k = 0; k < 8; k += 2) {
            const uint32_t word = k < 4 ? w.x : w.y;
            const float a = d * (float)(int8_t)(word >> (8 * (k & 3)));
            const float b = d * (float)(int8_t)(word >> (8 * ((k & 3) + 1)));
            uint16_t ta[kTerms], tb[kTerms];
            split_bf16x3(a, ta[0], ta[1], ta[2]);
            split_bf16x3(b, tb[0], tb[1], tb[2]);
#pragma unroll
            for (int q = 0; q < kTerms; ++q) t[q][k >> 1] = (uint32_t)ta[q] | ((uint32_t)tb[q] << 16);
        }
        const size_t o = (size_t)r * K + (size_t)c * 8;
#pragma unroll
        for (int q = 0; q < kTerms; ++q)
            if (q < nterms) *reinterpret_cast<uint4 *>(out.p[q] + o) = make_uint4(t[q][0], t[q][1], t[q][2], t[q][3]);
    }
}

static cudaError_t dequant_terms(const Plan &p, const Bufs &b, const uint16_t *W, int rows, int K, int nterms,
                                 cudaStream_t st, LaunchHook *hook) {
    const long long n = (long long)rows * (K / 8);
    const int grid = (int)((n + 255) / 256 < 8 * p.num_sms ? (n + 255) / 256 : 8 * p.num_sms);
    if (hook) hook->before("prefill_q8_dequant");
    q8_dequant_terms_kernel<<<grid, 256, 0, st>>>(reinterpret_cast<const uint8_t *>(W), rows, K,
                                                 Terms{{b.Wt[0], b.Wt[1], b.Wt[2]}}, nterms);
    if (hook) hook->after("prefill_q8_dequant");
    return cudaGetLastError();
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

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

bool encode_tiled(CUtensorMap *m, int rank, const void *ptr, const uint64_t *dims, const uint64_t *strides_bytes,
                  const uint32_t *box, const uint32_t *elem_strides) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t d[5], st[4];
    cuuint32_t b[5], e[5];
    for (int i = 0; i < rank; ++i) {
        d[i] = dims[i];
        b[i] = box[i];
        e[i] = elem_strides[i];
        if (i + 1 < rank) st[i] = strides_bytes[i];
    }
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void *>(ptr), d, st, b, e,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D map over a row-major bf16 matrix [rows][K]; boxes of 64 x box_rows, 128 B swizzle
static bool encode_2d(CUtensorMap *m, const void *ptr, int rows, int K, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    cuuint32_t box[2] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// the KV pool of every layer as [page (layer-major)][K|V][kv head][16 slots][d]:
// boxes of 64 d x 16 slots of one (page, K|V, head)
static bool encode_kv(CUtensorMap *m, const void *ptr, const Plan &p) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[5] = {(cuuint64_t)p.d, (cuuint64_t)kPage, (cuuint64_t)p.nkv, 2,
                          (cuuint64_t)p.L * (cuuint64_t)p.max_pages};
    cuuint64_t strides[4] = {(cuuint64_t)p.d * 2, (cuuint64_t)kPage * p.d * 2, (cuuint64_t)p.nkv * kPage * p.d * 2,
                             (cuuint64_t)2 * p.nkv * kPage * p.d * 2};
    cuuint32_t box[5] = {64, (cuuint32_t)kPage, 1, 1, 1};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(ptr), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

const char *make_prefill_maps(const Plan &p, const Bufs &b, PrefillMaps *m) {
    const int T = p.max_chunk;
    bool ok = true;
    for (int t = 0; t < kTerms; ++t)
        ok = ok && encode_2d(&m->a[t], b.A[t], T, p.H, TC_BM) && encode_2d(&m->o[t], b.O[t], T, p.qdim, TC_BM) &&
             encode_2d(&m->m[t], b.M[t], T, p.F, TC_BM);
    if (!ok) return "cuTensorMapEncodeTiled failed for an activation operand";
    ok = encode_kv(&m->kv, b.KV, p);
    if (!ok) return "cuTensorMapEncodeTiled failed for the attention operands";
    m->bn_qkv = pick_bn(T, p.nqkv, p.num_sms, PEpiQKV::kATerms == 2);
    m->bn_o = pick_bn(T, p.H, p.num_sms, PEpiResidual::kATerms == 2);
    m->bn_gu = pick_bn(T, 2 * p.F, p.num_sms, PEpiSwiGLU::kATerms == 2);
    m->bn_d = pick_bn(T, p.H, p.num_sms, PEpiResidual::kATerms == 2);
    if (p.q8) {
        // the 8-bit format: every GEMM reads the one dequantised matrix in the workspace
        for (int t = 0; t < kTerms; ++t) {
            ok = encode_2d(&m->wt_qkv[t], b.Wt[t], p.nqkv, p.H, m->bn_qkv) &&
                 encode_2d(&m->wt_o[t], b.Wt[t], p.H, p.qdim, m->bn_o) &&
                 encode_2d(&m->wt_gu[t], b.Wt[t], 2 * p.F, p.H, m->bn_gu) &&
                 encode_2d(&m->wt_d[t], b.Wt[t], p.H, p.F, m->bn_d);
            if (!ok) return "cuTensorMapEncodeTiled failed for a dequantised weight matrix";
        }
    }
    m->wqkv.resize(p.q8 ? 0 : p.L);
    m->wo.resize(p.q8 ? 0 : p.L);
    m->wgu.resize(p.q8 ? 0 : p.L);
    m->wd.resize(p.q8 ? 0 : p.L);
    for (int l = 0; l < (p.q8 ? 0 : p.L); ++l) {
        const LayerOffsets &lo = p.layer[l];
        ok = encode_2d(&m->wqkv[l], b.W + lo.wqkv, p.nqkv, p.H, m->bn_qkv) &&
             encode_2d(&m->wo[l], b.W + lo.wo, p.H, p.qdim, m->bn_o) &&
             encode_2d(&m->wgu[l], b.W + lo.wgu, 2 * p.F, p.H, m->bn_gu) &&
             encode_2d(&m->wd[l], b.W + lo.wd, p.H, p.F, m->bn_d);
        if (!ok) return "cuTensorMapEncodeTiled failed for a weight matrix";
    }
    static bool attrs = false;
    if (!attrs) {
        const auto attr = [](const void *f, int bytes) {
            return cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) == cudaSuccess;
        };
#define WICI_GEMM_ATTR(BN, WT, E) attr((const void *)gemm_tc_kernel<BN, WT, E>, (int)TcTile<BN, E::kATerms>::SMEM)
        if (!WICI_GEMM_ATTR(192, 1, PEpiQKV) || !WICI_GEMM_ATTR(192, 1, PEpiResidual) ||
            !WICI_GEMM_ATTR(192, 1, PEpiSwiGLU) || !WICI_GEMM_ATTR(128, 1, PEpiQKV) ||
            !WICI_GEMM_ATTR(128, 1, PEpiResidual) || !WICI_GEMM_ATTR(128, 1, PEpiSwiGLU) ||
            !WICI_GEMM_ATTR(192, kTerms, PEpiQKV) || !WICI_GEMM_ATTR(192, kTerms, PEpiResidual) ||
            !WICI_GEMM_ATTR(192, kTerms, PEpiSwiGLU) || !WICI_GEMM_ATTR(128, kTerms, PEpiQKV) ||
            !WICI_GEMM_ATTR(128, kTerms, PEpiResidual) || !WICI_GEMM_ATTR(128, kTerms, PEpiSwiGLU) ||
            !WICI_GEMM_ATTR(224, 1, PEpiResidual) || !WICI_GEMM_ATTR(224, 1, PEpiSwiGLU) ||
            !WICI_GEMM_ATTR(224, kTerms, PEpiResidual) || !WICI_GEMM_ATTR(224, kTerms, PEpiSwiGLU) ||
            cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(AttnSmem<128>::TOTAL + 1024)) != cudaSuccess ||
            cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(AttnSmem<64>::TOTAL + 1024)) != cudaSuccess)
            return "cannot raise the shared-memory limit of the tensor-core GEMM";
#undef WICI_GEMM_ATTR
        attrs = true;
    }
    return nullptr;
}

// causal GQA attention of chunk rows [0, T) at positions P.. on the tensor cores
cudaError_t launch_attn_tc(const Plan &p, const Bufs &b, const PrefillMaps &mp, int layer, int P, int T,
                           cudaStream_t st) {
    AttnArgs a;
    for (int t = 0; t < AT_TERMS; ++t) a.Q[t] = b.Q[t];
    for (int t = 0; t < kTerms; ++t) a.O[t] = b.O[t];
    a.pages = b.pages;
    a.err = b.ctrl + CTRL_ERR;
    a.P = P;
    a.T = T;
    a.nq = p.nq;
    a.group = p.group;
    a.tpt = attn_tokens_per_tile(p.group);
    a.layer = layer;
    a.max_pages = p.max_pages;
    a.scale_log2 = 1.4426950408889634f / sqrtf((float)p.d);
    dim3 grid(((T + a.tpt - 1) / a.tpt) * p.nkv);
    if (p.d == 128)
        attn_tc_kernel<128><<<grid, AT_THREADS, AttnSmem<128>::TOTAL + 1024, st>>>(mp.kv, a);
    else
        attn_tc_kernel<64><<<grid, AT_THREADS, AttnSmem<64>::TOTAL + 1024, st>>>(mp.kv, a);
    return cudaGetLastError();
}

// the weight operand of one GEMM: one exact bf16 matrix, or three terms
struct WOperand {
    const CUtensorMap *w[kTerms];
    int terms;
};

template <int BN, class Epi>
static void launch_gemm(const Plan &p, const CUtensorMap *a, const WOperand &w, int T, int N, int K, int *err,
                        const Epi &epi, cudaStream_t st) {
    const int tiles = ((T + TC_BM - 1) / TC_BM) * ((N + BN - 1) / BN);
    const int grid = tiles < p.num_sms ? tiles : p.num_sms;   // persistent: at most one CTA per SM
    if (w.terms == 1)
        gemm_tc_kernel<BN, 1, Epi><<<grid, TC_THREADS, TcTile<BN, Epi::kATerms>::SMEM, st>>>(a[0], a[1], a[2], *w.w[0], *w.w[1],
                                                                              *w.w[2], T, N, K, err, epi);
    else
        gemm_tc_kernel<BN, kTerms, Epi><<<grid, TC_THREADS, TcTile<BN, Epi::kATerms>::SMEM, st>>>(
            a[0], a[1], a[2], *w.w[0], *w.w[1], *w.w[2], T, N, K, err, epi);
}

template <class Epi>
static cudaError_t gemm(const Plan &p, int bn, const CUtensorMap *a, const WOperand &w, int T, int N, int K,
                        int *err, const Epi &epi, cudaStream_t st, LaunchHook *hook, const char *name) {
    if (hook) hook->before(name);
    if (bn == 128)
        launch_gemm<128>(p, a, w, T, N, K, err, epi, st);
    else if (bn == 192)
        launch_gemm<192>(p, a, w, T, N, K, err, epi, st);
    else if constexpr (Epi::kATerms == 2)
        launch_gemm<224>(p, a, w, T, N, K, err, epi, st);
    else
        return cudaErrorInvalidValue;   // pick_bn never picks 224 for three terms
    if (hook) hook->after(name);
    return cudaGetLastError();
}

// bf16: the layer's own matrix; 8-bit format: dequantise the layer's rows into
// the workspace terms first (stream order makes the previous GEMM finish reading them)
template <class Epi>
static cudaError_t weight_operand(const Plan &p, const Bufs &b, const CUtensorMap &bf16_map,
                                  const CUtensorMap *terms, const uint16_t *rows, int n_rows, int K, cudaStream_t st,
                                  LaunchHook *hook, WOperand *w) {
    if (!p.q8) {
        *w = WOperand{{&bf16_map, &bf16_map, &bf16_map}, 1};
        return cudaSuccess;
    }
    *w = WOperand{{&terms[0], &terms[1], &terms[2]}, kTerms};
    return dequant_terms(p, b, rows, n_rows, K, Epi::kATerms, st, hook);   // the weight terms the GEMM uses
}

cudaError_t enqueue_prefill_chunk(const Plan &p, const Bufs &b, const PrefillMaps &mp, cudaStream_t st, int P,
                                  int T, int lm_pos_add, LaunchHook *hook) {
    cudaError_t e;
    int *err = b.ctrl + CTRL_ERR;
    embed_rows_kernel<<<T, 256, 0, st>>>(b.W + p.w_embed, b.tok, b.X, p.H);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    for (int l = 0; l < p.L; ++l) {
        const LayerOffsets &lo = p.layer[l];
        uint16_t *kvl = b.KV + (size_t)l * p.kv_layer_elems;
        // A3 + A4: RMSNorm, QKV (+bias), RoPE, paged KV append
        const Terms A = {{b.A[0], b.A[1], b.A[2]}};
        rmsnorm_rows_kernel<<<T, 256, 0, st>>>(b.X, b.W + lo.attn_norm, A, p.H, p.cfg.rms_eps, PEpiQKV::kATerms);
        PEpiQKV eq = {{{b.Q[0], b.Q[1], b.Q[2]}}, kvl, b.pages, b.rope, p.cfg.qkv_bias ? b.W + lo.bqkv : nullptr, P, p.qdim,
                      p.kvdim, p.d, p.nkv, p.kv_page_elems, p.qk_norm ? b.QKraw : nullptr};
        WOperand w;
        if ((e = weight_operand<PEpiQKV>(p, b, p.q8 ? mp.wt_qkv[0] : mp.wqkv[l], mp.wt_qkv, b.W + lo.wqkv, p.nqkv, p.H, st,
                                hook, &w)) != cudaSuccess)
            return e;
        if ((e = gemm(p, mp.bn_qkv, mp.a, w, T, p.nqkv, p.H, err, eq, st, hook, "prefill_qkv")) != cudaSuccess)
            return e;
        if (p.qk_norm) {
            // Qwen3 block: per-head q/k norm, then RoPE and the operand / page stores
            const Terms Qt = {{b.Q[0], b.Q[1], b.Q[2]}};
            const dim3 grid(T, (p.nq + p.nkv + 7) / 8);
            if (hook) hook->before("prefill_qk_norm_rope");
            if (p.d == 128)
                qk_norm_rope_kernel<128><<<grid, 256, 0, st>>>(b.QKraw, b.W + lo.qn, b.W + lo.kn, b.rope, Qt, kvl,
                                                               b.pages, p.kv_page_elems, P, p.nq, p.nkv, p.cfg.rms_eps);
            else
                qk_norm_rope_kernel<64><<<grid, 256, 0, st>>>(b.QKraw, b.W + lo.qn, b.W + lo.kn, b.rope, Qt, kvl,
                                                              b.pages, p.kv_page_elems, P, p.nq, p.nkv, p.cfg.rms_eps);
            if (hook) hook->after("prefill_qk_norm_rope");
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
        }
        // A5: causal attention over the cache (earlier chunks + this one), tensor cores
        if (hook) hook->before("prefill_attention");
        e = launch_attn_tc(p, b, mp, l, P, T, st);
        if (hook) hook->after("prefill_attention");
        if (e != cudaSuccess) return e;
        // A6: O projection + residual
        if ((e = weight_operand<PEpiResidual>(p, b, p.q8 ? mp.wt_o[0] : mp.wo[l], mp.wt_o, b.W + lo.wo, p.H, p.qdim, st, hook,
                                &w)) != cudaSuccess)
            return e;
        if ((e = gemm(p, mp.bn_o, mp.o, w, T, p.H, p.qdim, err, PEpiResidual{b.X, p.H}, st, hook,
                      "prefill_o_proj")) != cudaSuccess)
            return e;
        // A7: RMSNorm + gate/up + SwiGLU
        rmsnorm_rows_kernel<<<T, 256, 0, st>>>(b.X, b.W + lo.ffn_norm, A, p.H, p.cfg.rms_eps, PEpiSwiGLU::kATerms);
        const Terms M = {{b.M[0], b.M[1], b.M[2]}};
        if ((e = weight_operand<PEpiSwiGLU>(p, b, p.q8 ? mp.wt_gu[0] : mp.wgu[l], mp.wt_gu, b.W + lo.wgu, 2 * p.F, p.H, st,
                                hook, &w)) != cudaSuccess)
            return e;
        if ((e = gemm(p, mp.bn_gu, mp.a, w, T, 2 * p.F, p.H, err, PEpiSwiGLU{M, p.F}, st, hook,
                      "prefill_gate_up")) != cudaSuccess)
            return e;
        // A8: down projection + residual
        if ((e = weight_operand<PEpiResidual>(p, b, p.q8 ? mp.wt_d[0] : mp.wd[l], mp.wt_d, b.W + lo.wd, p.H, p.F, st, hook,
                                &w)) != cudaSuccess)
            return e;
        if ((e = gemm(p, mp.bn_d, mp.m, w, T, p.H, p.F, err, PEpiResidual{b.X, p.H}, st, hook,
                      "prefill_down")) != cudaSuccess)
            return e;
    }
    if (lm_pos_add > 0) {
        // A9 on the chunk's last row only
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
