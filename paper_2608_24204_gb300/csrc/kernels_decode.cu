// Decode-step kernels (batch 1): weight-streaming GEMVs with fused prologues
// and epilogues, and split-K flash-decode over the paged KV cache.
//
// A decode step is HBM-bound: every weight byte is read once per token
// (arithmetic intensity ~1 FLOP/byte).  The GEMV streams each CTA's rows through
// a 3-stage ring in shared memory with 1-D TMA bulk copies (cp.async.bulk,
// completion on mbarriers); one producer warp issues the copies, eight consumer
// warps do the dot products with the input vector held in registers.  The
// producer starts before griddepcontrol.wait, so under programmatic dependent
// launch a GEMV's first weight tiles stream in while its predecessor finishes.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

namespace wici {

// wait-site ids recorded in ctrl[CTRL_ERR]
enum : int { SITE_GEMV_EMPTY = 11, SITE_GEMV_FULL = 12, SITE_GEMV_DRAIN = 13, SITE_PROBE = 99 };

struct GemvIn {
    const uint16_t *W;      // rows of this matrix, [n_units * rpu][K]
    int K, n_units, rpu, ups;
    const float *in;        // input vector (x when gain != nullptr)
    const uint16_t *gain;   // RMSNorm gain (bf16) or nullptr for a plain input
    const uint16_t *embed;  // non-null: the input is embed[ctrl[CTRL_TOKEN]] (layer 0)
    float *x_out;           // embed variant: CTA 0 stores the embedded row here
    int *ctrl;
    float eps;
};

// ---------------------------------------------------------------- epilogues --
// unit(u, v): v[0..rpu) are the finished dot products of unit u's rows.

struct EpiResidual {  // x[u] += W x_in   (O projection, down projection)
    float *x;
    static constexpr bool kArgmax = false;
    __device__ void unit(int u, const float *v) { x[u] += v[0]; }
};

struct EpiSwiGLU {    // rows (2u, 2u+1) are (gate_u, up_u): m[u] = silu(g) * u
    float *m;
    static constexpr bool kArgmax = false;
    __device__ void unit(int u, const float *v) {
        const float gt = v[0];
        m[u] = gt / (1.0f + expf(-gt)) * v[1];
    }
};

// Packed QKV rows: for every q and k head the rows are paired (i, i + d/2) as
// adjacent rows (2i, 2i + 1), so one unit holds one RoPE pair; v rows are in
// natural order, two per unit.
struct EpiQKV {
    float *q;
    uint16_t *kv;          // this layer's pages
    const int *pages;
    const float2 *rope;
    const int *ctrl;
    const uint16_t *bias;  // packed like the rows, or nullptr
    int qdim, kvdim, d, nkv;
    size_t page_elems;
    static constexpr bool kArgmax = false;
    __device__ void unit(int u, const float *v) {
        const int r0 = 2 * u;
        float a = v[0], b = v[1];
        if (bias) {
            a += bf16_to_f32(bias[r0]);
            b += bf16_to_f32(bias[r0 + 1]);
        }
        const int pos = ctrl[CTRL_POS];
        uint16_t *page = kv + (size_t)pages[pos / kPage] * page_elems;
        const int slot = pos % kPage;
        if (r0 < qdim + kvdim) {
            const int hd = r0 / d, i = (r0 % d) >> 1, half = d >> 1;
            const float2 cs = rope[(size_t)pos * half + i];
            const float ra = a * cs.x - b * cs.y;
            const float rb = b * cs.x + a * cs.y;
            if (r0 < qdim) {
                q[hd * d + i] = ra;
                q[hd * d + i + half] = rb;
            } else {
                const int kh = hd - qdim / d;
                uint16_t *kr = page + ((size_t)kh * kPage + slot) * d;
                kr[i] = f32_to_bf16(ra);
                kr[i + half] = f32_to_bf16(rb);
            }
        } else {
            const int j = r0 - qdim - kvdim, vh = j / d, e = j % d;
            uint16_t *vr = page + (size_t)nkv * kPage * d + ((size_t)vh * kPage + slot) * d;
            vr[e] = f32_to_bf16(a);
            vr[e + 1] = f32_to_bf16(b);
        }
    }
};

struct EpiArgmax {    // logits[u] = v; greedy argmax (lowest index on ties) across the grid
    float *logits;
    int2 *partial;
    int *ctrl;
    int *hist;
    int pos_add;
    float best;
    int bidx;
    static constexpr bool kArgmax = true;
    __device__ void unit(int u, const float *v) {
        logits[u] = v[0];
        if (v[0] > best || (v[0] == best && u < bidx)) {
            best = v[0];
            bidx = u;
        }
    }
};

__device__ __forceinline__ bool better(float av, int ai, float bv, int bi) {
    return av > bv || (av == bv && ai < bi);
}

__device__ __forceinline__ void consumer_bar() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__device__ __forceinline__ float dot8(const uint4 w, const float *h) {
    float s = bf16lo(w.x) * h[0];
    s = fmaf(bf16hi(w.x), h[1], s);
    s = fmaf(bf16lo(w.y), h[2], s);
    s = fmaf(bf16hi(w.y), h[3], s);
    s = fmaf(bf16lo(w.z), h[4], s);
    s = fmaf(bf16hi(w.z), h[5], s);
    s = fmaf(bf16lo(w.w), h[6], s);
    s = fmaf(bf16hi(w.w), h[7], s);
    return s;
}

constexpr size_t kGemvSmem =
    (size_t)kGemvStages * kGemvStageMax + 2 * kGemvStages * 8 + 2 * 8 * kGemvMaxRows * 4;

// ------------------------------------------------------------------- GEMV ----
// Grid: num_sms CTAs, each owning a contiguous, balanced range of units.
template <int NCH, class Epi>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_kernel(const GemvIn g, const Epi epi_in) {
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *ring = smem;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + (size_t)kGemvStages * kGemvStageMax);
    float *red = reinterpret_cast<float *>(bars + 2 * kGemvStages);  // [2][8][kGemvMaxRows]
    __shared__ float s_part[8];
    __shared__ int s_abort;
    __shared__ float s_bv[8];
    __shared__ int s_bi[8];
    __shared__ int s_last;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = gridDim.x;
    const int u0 = (int)(((long long)blockIdx.x * g.n_units) / G);
    const int u1 = (int)(((long long)(blockIdx.x + 1) * g.n_units) / G);
    const int nunits = u1 - u0;
    const int nst = (nunits + g.ups - 1) / g.ups;
    const uint32_t unit_bytes = (uint32_t)g.rpu * (uint32_t)g.K * 2u;
    int *err = g.ctrl + CTRL_ERR;

    const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kGemvStages);
    if (tid == 0) {
        for (int s = 0; s < kGemvStages; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 8);
        }
        fence_barrier_init();
        s_abort = 0;
    }
    __syncthreads();
    griddep_launch_dependents();

    if (warp == 8) {  // ------------------------------------------ producer
        if (lane == 0) {
            const uint64_t pol = l2_evict_first();
            const uint32_t ring0 = smem_u32(ring);
            int issued = 0;
            for (int s = 0; s < nst; ++s) {
                const int slot = s % kGemvStages;
                if (s >= kGemvStages &&
                    !mbar_wait(empty0 + 8 * slot, ((s / kGemvStages) + 1) & 1, err, SITE_GEMV_EMPTY))
                    break;
                const int un = min(g.ups, nunits - s * g.ups);
                const uint32_t bytes = (uint32_t)un * unit_bytes;
                mbar_arrive_expect_tx(full0 + 8 * slot, bytes);
                bulk_g2s(ring0 + slot * kGemvStageMax,
                         g.W + (size_t)(u0 + s * g.ups) * g.rpu * g.K, bytes, full0 + 8 * slot, pol);
                issued = s + 1;
            }
            // no copy may still be landing in this CTA's shared memory when it exits
            for (int s = max(0, issued - kGemvStages); s < issued; ++s)
                mbar_wait(full0 + 8 * (s % kGemvStages), (s / kGemvStages) & 1, err, SITE_GEMV_DRAIN);
        }
        return;
    }

    // --------------------------------------------------------------- consumers
    Epi epi = epi_in;
    griddep_wait();
    const int nchunks = g.K >> 3;
    float h[NCH][8];
    float ss = 0.f;
    const int tok = g.embed ? g.ctrl[CTRL_TOKEN] : 0;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
        const int c = tid + 256 * j;
        if (c < nchunks) {
            if (g.embed) {
                const uint4 w = *reinterpret_cast<const uint4 *>(g.embed + (size_t)tok * g.K + c * 8);
                h[j][0] = bf16lo(w.x); h[j][1] = bf16hi(w.x);
                h[j][2] = bf16lo(w.y); h[j][3] = bf16hi(w.y);
                h[j][4] = bf16lo(w.z); h[j][5] = bf16hi(w.z);
                h[j][6] = bf16lo(w.w); h[j][7] = bf16hi(w.w);
                if (blockIdx.x == 0) {
                    float4 *dst = reinterpret_cast<float4 *>(g.x_out + c * 8);
                    dst[0] = make_float4(h[j][0], h[j][1], h[j][2], h[j][3]);
                    dst[1] = make_float4(h[j][4], h[j][5], h[j][6], h[j][7]);
                }
            } else {
                const float4 a = *reinterpret_cast<const float4 *>(g.in + c * 8);
                const float4 b = *reinterpret_cast<const float4 *>(g.in + c * 8 + 4);
                h[j][0] = a.x; h[j][1] = a.y; h[j][2] = a.z; h[j][3] = a.w;
                h[j][4] = b.x; h[j][5] = b.y; h[j][6] = b.z; h[j][7] = b.w;
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) ss = fmaf(h[j][e], h[j][e], ss);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) h[j][e] = 0.f;
        }
    }
    if (g.gain) {  // RMSNorm prologue: every CTA reduces the whole vector in the same order
        ss = warp_sum(ss);
        if (lane == 0) s_part[warp] = ss;
        consumer_bar();
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) tot += s_part[w];
        const float rinv = 1.0f / sqrtf(tot / (float)g.K + g.eps);
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int c = tid + 256 * j;
            if (c < nchunks) {
                const uint4 gw = *reinterpret_cast<const uint4 *>(g.gain + c * 8);
                const float gg[8] = {bf16lo(gw.x), bf16hi(gw.x), bf16lo(gw.y), bf16hi(gw.y),
                                     bf16lo(gw.z), bf16hi(gw.z), bf16lo(gw.w), bf16hi(gw.w)};
#pragma unroll
                for (int e = 0; e < 8; ++e) h[j][e] = h[j][e] * rinv * gg[e];
            }
        }
    }

    int buf = 0;
    for (int s = 0; s < nst; ++s) {
        const int slot = s % kGemvStages;
        const int un = min(g.ups, nunits - s * g.ups);
        const int rows = un * g.rpu;
        const bool ok = mbar_wait(full0 + 8 * slot, (s / kGemvStages) & 1, err, SITE_GEMV_FULL);
        if (!ok) s_abort = 1;
        if (ok) {
            const uint8_t *st = ring + (size_t)slot * kGemvStageMax;
            float *rb = red + (size_t)(buf * 8 + warp) * kGemvMaxRows;
            for (int r = 0; r < rows; ++r) {
                const uint8_t *row = st + (size_t)r * g.K * 2;
                float acc = 0.f;
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    const int c = tid + 256 * j;
                    if (c < nchunks) acc += dot8(*reinterpret_cast<const uint4 *>(row + c * 16), h[j]);
                }
                acc = warp_sum(acc);
                if (lane == 0) rb[r] = acc;
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * slot);
        consumer_bar();
        if (s_abort) break;
        if (tid < un) {
            float v[2];
            for (int j = 0; j < g.rpu; ++j) {
                float t = 0.f;
#pragma unroll
                for (int w = 0; w < 8; ++w) t += red[(size_t)(buf * 8 + w) * kGemvMaxRows + tid * g.rpu + j];
                v[j] = t;
            }
            epi.unit(u0 + s * g.ups + tid, v);
        }
        buf ^= 1;
    }

    if constexpr (Epi::kArgmax) {
        // CTA argmax, then the last CTA to finish reduces all CTAs' results in index order
        float bv = epi.best;
        int bi = epi.bidx;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
        }
        if (lane == 0) { s_bv[warp] = bv; s_bi[warp] = bi; }
        consumer_bar();
        if (tid == 0) {
            for (int w = 1; w < 8; ++w)
                if (better(s_bv[w], s_bi[w], bv, bi)) { bv = s_bv[w]; bi = s_bi[w]; }
            epi.partial[blockIdx.x] = make_int2(__float_as_int(bv), bi);
            __threadfence();
            const int t = atomicAdd(epi.ctrl + CTRL_LM_TICKET, 1);
            s_last = (t == G - 1);
        }
        consumer_bar();
        if (s_last && tid == 0) {
            __threadfence();
            float fv = -INFINITY;
            int fi = 0x7fffffff;
            for (int c = 0; c < G; ++c) {
                const int2 pr = __ldcg(epi.partial + c);
                const float pv = __int_as_float(pr.x);
                if (better(pv, pr.y, fv, fi)) { fv = pv; fi = pr.y; }
            }
            if (fi == 0x7fffffff) fi = 0;
            const int np = epi.ctrl[CTRL_POS] + epi.pos_add;
            epi.ctrl[CTRL_TOKEN] = fi;
            epi.ctrl[CTRL_POS] = np;
            epi.hist[np] = fi;
            epi.ctrl[CTRL_LM_TICKET] = 0;
        }
    }
}

// ------------------------------------------------------------ flash-decode ----
// Grid (splits, nkv); block = 32 * group threads, warp w = query head g*group+w.
// Each CTA covers a contiguous range of KV pages of head g (length taken from the
// device position, so one captured graph serves every step), keeps a warp-level
// online softmax per query head, writes (m, l, acc[d]) partials, and the last
// CTA of each KV head combines the partials in split order.
struct FDArgs {
    const float *q;
    const uint16_t *kv;  // this layer's pages
    const int *pages;
    int *ctrl;
    float *part;
    float *o;
    int nkv, group, splits;
    size_t page_elems;
    float qscale;        // log2(e) / sqrt(d)
};

template <int D>
__global__ void __launch_bounds__(256) flash_decode_kernel(const FDArgs a) {
    constexpr int EPL = D / 32;
    __shared__ int s_last;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.y, split = blockIdx.x;
    const int head = g * a.group + w;
    griddep_launch_dependents();
    griddep_wait();

    const int len = a.ctrl[CTRL_POS] + 1;
    const int npages = (len + kPage - 1) / kPage;
    const int pps = (npages + a.splits - 1) / a.splits;
    const int p0 = split * pps, p1 = min(npages, p0 + pps);

    float qv[EPL], acc[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
        qv[e] = a.q[head * D + lane * EPL + e] * a.qscale;
        acc[e] = 0.f;
    }
    float m = -INFINITY, l = 0.f;
    for (int p = p0; p < p1; ++p) {
        const uint16_t *Kb = a.kv + (size_t)a.pages[p] * a.page_elems + (size_t)g * kPage * D;
        const uint16_t *Vb = Kb + (size_t)a.nkv * kPage * D;
        const int ntok = min(kPage, len - p * kPage);
        float sc[kPage];
        float mx = m;
#pragma unroll
        for (int t = 0; t < kPage; ++t) {
            float s = -INFINITY;
            if (t < ntok) {
                const uint16_t *kr = Kb + t * D + lane * EPL;
                float part = 0.f;
                if constexpr (EPL == 4) {
                    const uint2 kw = *reinterpret_cast<const uint2 *>(kr);
                    part = qv[0] * bf16lo(kw.x) + qv[1] * bf16hi(kw.x) + qv[2] * bf16lo(kw.y) +
                           qv[3] * bf16hi(kw.y);
                } else {
                    const uint32_t kw = *reinterpret_cast<const uint32_t *>(kr);
                    part = qv[0] * bf16lo(kw) + qv[1] * bf16hi(kw);
                }
                s = warp_sum(part);
            }
            sc[t] = s;
            mx = fmaxf(mx, s);
        }
        const float corr = exp2f(m - mx);
        l *= corr;
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] *= corr;
#pragma unroll
        for (int t = 0; t < kPage; ++t) {
            if (t < ntok) {
                const float pt = exp2f(sc[t] - mx);
                l += pt;
                const uint16_t *vr = Vb + t * D + lane * EPL;
                if constexpr (EPL == 4) {
                    const uint2 vw = *reinterpret_cast<const uint2 *>(vr);
                    acc[0] = fmaf(pt, bf16lo(vw.x), acc[0]);
                    acc[1] = fmaf(pt, bf16hi(vw.x), acc[1]);
                    acc[2] = fmaf(pt, bf16lo(vw.y), acc[2]);
                    acc[3] = fmaf(pt, bf16hi(vw.y), acc[3]);
                } else {
                    const uint32_t vw = *reinterpret_cast<const uint32_t *>(vr);
                    acc[0] = fmaf(pt, bf16lo(vw), acc[0]);
                    acc[1] = fmaf(pt, bf16hi(vw), acc[1]);
                }
            }
        }
        m = mx;
    }
    float *pp = a.part + ((size_t)(g * a.splits + split) * a.group + w) * (D + 2);
#pragma unroll
    for (int e = 0; e < EPL; ++e) pp[lane * EPL + e] = acc[e];
    if (lane == 0) {
        pp[D] = m;
        pp[D + 1] = l;
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        const int t = atomicAdd(a.ctrl + CTRL_ATTN_TICKET0 + g, 1);
        s_last = (t == a.splits - 1);
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    float M = -INFINITY;
    for (int s = 0; s < a.splits; ++s) {
        const float *ps = a.part + ((size_t)(g * a.splits + s) * a.group + w) * (D + 2);
        M = fmaxf(M, __ldcg(ps + D));
    }
    float L = 0.f, out[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) out[e] = 0.f;
    for (int s = 0; s < a.splits; ++s) {
        const float *ps = a.part + ((size_t)(g * a.splits + s) * a.group + w) * (D + 2);
        const float f = exp2f(__ldcg(ps + D) - M);
        L = fmaf(__ldcg(ps + D + 1), f, L);
#pragma unroll
        for (int e = 0; e < EPL; ++e) out[e] = fmaf(__ldcg(ps + lane * EPL + e), f, out[e]);
    }
    const float inv = 1.0f / L;
#pragma unroll
    for (int e = 0; e < EPL; ++e) a.o[head * D + lane * EPL + e] = out[e] * inv;
    if (threadIdx.x == 0) a.ctrl[CTRL_ATTN_TICKET0 + g] = 0;
}

// ------------------------------------------------------------ probe kernel ----
__global__ void bounded_wait_probe_kernel(int *err, long long limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait(smem_u32(&bar), 0, err, SITE_PROBE, (uint64_t)limit_ns);
}

// ============================================================ host side ====

template <typename Kern, typename... Args>
static cudaError_t launch(Kern kern, dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl,
                          Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

template <class Epi>
static void *gemv_fn(int nch) {
    switch (nch) {
        case 1: return (void *)gemv_kernel<1, Epi>;
        case 2: return (void *)gemv_kernel<2, Epi>;
        case 3: return (void *)gemv_kernel<3, Epi>;
        case 4: return (void *)gemv_kernel<4, Epi>;
        case 5: return (void *)gemv_kernel<5, Epi>;
        case 6: return (void *)gemv_kernel<6, Epi>;
        case 7: return (void *)gemv_kernel<7, Epi>;
        case 8: return (void *)gemv_kernel<8, Epi>;
    }
    return nullptr;
}

template <class Epi>
static cudaError_t set_gemv_attrs() {
    for (int n = 1; n <= 8; ++n) {
        cudaError_t e = cudaFuncSetAttribute(gemv_fn<Epi>(n), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kGemvSmem);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t setup_kernels() {
    cudaError_t e;
    if ((e = set_gemv_attrs<EpiResidual>()) != cudaSuccess) return e;
    if ((e = set_gemv_attrs<EpiSwiGLU>()) != cudaSuccess) return e;
    if ((e = set_gemv_attrs<EpiQKV>()) != cudaSuccess) return e;
    if ((e = set_gemv_attrs<EpiArgmax>()) != cudaSuccess) return e;
    return cudaSuccess;
}

// units per stage: as many whole units as fit one stage, at most kGemvMaxRows rows
static int units_per_stage(int K, int rpu) {
    const int unit_bytes = rpu * K * 2;
    int ups = (int)(kGemvStageMax / (uint32_t)unit_bytes);
    ups = ups < 1 ? 1 : ups;
    while (ups * rpu > kGemvMaxRows) --ups;
    return ups;
}

template <class Epi>
static cudaError_t launch_gemv(const Plan &p, GemvIn g, Epi epi, cudaStream_t st, bool pdl,
                               LaunchHook *hook, const char *name) {
    g.ups = units_per_stage(g.K, g.rpu);
    const int nch = (g.K / 8 + 255) / 256;
    if (nch < 1 || nch > 8) return cudaErrorInvalidValue;
    const int grid = p.num_sms;
    if (hook) hook->before(name);
    cudaError_t e = launch(reinterpret_cast<void (*)(const GemvIn, const Epi)>(gemv_fn<Epi>(nch)),
                           dim3(grid), dim3(kGemvThreads), kGemvSmem, st, pdl, g, epi);
    if (hook) hook->after(name);
    return e;
}

static GemvIn gemv_in(const Plan &p, const Bufs &b, const uint16_t *W, int K, int n_units, int rpu,
                      const float *in, const uint16_t *gain) {
    GemvIn g = {};
    g.W = W;
    g.K = K;
    g.n_units = n_units;
    g.rpu = rpu;
    g.in = in;
    g.gain = gain;
    g.ctrl = b.ctrl;
    g.eps = p.cfg.rms_eps;
    return g;
}

cudaError_t enqueue_lm_head(const Plan &p, const Bufs &b, cudaStream_t st, bool pdl, int pos_add,
                            LaunchHook *hook) {
    GemvIn g = gemv_in(p, b, b.W + p.w_lm, p.H, p.V, 1, b.x, b.W + p.w_final_norm);
    EpiArgmax e = {};
    e.logits = b.logits;
    e.partial = b.amax;
    e.ctrl = b.ctrl;
    e.hist = b.hist;
    e.pos_add = pos_add;
    e.best = -INFINITY;
    e.bidx = 0x7fffffff;
    return launch_gemv(p, g, e, st, pdl, hook, "lm_head_argmax");
}

cudaError_t enqueue_decode_step(const Plan &p, const Bufs &b, cudaStream_t st, bool pdl,
                                LaunchHook *hook) {
    cudaError_t e;
    const float qscale = 1.4426950408889634f / sqrtf((float)p.d);
    for (int l = 0; l < p.L; ++l) {
        const LayerOffsets &lo = p.layer[l];
        uint16_t *kvl = b.KV + (size_t)l * p.kv_layer_elems;
        // A3 + A4: RMSNorm, QKV, RoPE, KV append (layer 0 also gathers the embedding, A2)
        GemvIn g = gemv_in(p, b, b.W + lo.wqkv, p.H, p.nqkv / 2, 2, b.x, b.W + lo.attn_norm);
        if (l == 0) {
            g.embed = b.W + p.w_embed;
            g.x_out = b.x;
        }
        EpiQKV eq = {};
        eq.q = b.q;
        eq.kv = kvl;
        eq.pages = b.pages;
        eq.rope = b.rope;
        eq.ctrl = b.ctrl;
        eq.bias = p.cfg.qkv_bias ? b.W + lo.bqkv : nullptr;
        eq.qdim = p.qdim;
        eq.kvdim = p.kvdim;
        eq.d = p.d;
        eq.nkv = p.nkv;
        eq.page_elems = p.kv_page_elems;
        if ((e = launch_gemv(p, g, eq, st, pdl && l > 0, hook, "qkv_rope_kvappend")) != cudaSuccess) return e;
        // A5: attention
        FDArgs fa = {b.q, kvl, b.pages, b.ctrl, b.attn, b.o, p.nkv, p.group, p.attn_splits,
                     p.kv_page_elems, qscale};
        if (hook) hook->before("flash_decode");
        if (p.d == 128)
            e = launch(flash_decode_kernel<128>, dim3(p.attn_splits, p.nkv), dim3(32 * p.group), 0, st,
                       pdl, fa);
        else
            e = launch(flash_decode_kernel<64>, dim3(p.attn_splits, p.nkv), dim3(32 * p.group), 0, st,
                       pdl, fa);
        if (hook) hook->after("flash_decode");
        if (e != cudaSuccess) return e;
        // A6: O projection + residual
        g = gemv_in(p, b, b.W + lo.wo, p.qdim, p.H, 1, b.o, nullptr);
        if ((e = launch_gemv(p, g, EpiResidual{b.x}, st, pdl, hook, "o_proj_residual")) != cudaSuccess)
            return e;
        // A7: RMSNorm + gate/up + SwiGLU
        g = gemv_in(p, b, b.W + lo.wgu, p.H, p.F, 2, b.x, b.W + lo.ffn_norm);
        if ((e = launch_gemv(p, g, EpiSwiGLU{b.m}, st, pdl, hook, "gate_up_swiglu")) != cudaSuccess)
            return e;
        // A8: down projection + residual
        g = gemv_in(p, b, b.W + lo.wd, p.F, p.H, 1, b.m, nullptr);
        if ((e = launch_gemv(p, g, EpiResidual{b.x}, st, pdl, hook, "down_residual")) != cudaSuccess)
            return e;
    }
    // A9: final norm + LM head + greedy argmax; advances the position by one
    return enqueue_lm_head(p, b, st, pdl, 1, hook);
}

cudaError_t enqueue_bounded_wait_probe(int *err, int64_t limit_ns, cudaStream_t st) {
    bounded_wait_probe_kernel<<<1, 32, 0, st>>>(err, (long long)limit_ns);
    return cudaGetLastError();
}

}  // namespace wici
