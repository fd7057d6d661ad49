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
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace wici {

// wait-site ids recorded in ctrl[CTRL_ERR]
enum : int { SITE_GEMV_EMPTY = 11, SITE_GEMV_FULL = 12, SITE_GEMV_DRAIN = 13, SITE_PROBE = 99 };

struct GemvIn {
    const uint16_t *W;      // rows of this matrix, [n_units * rpu][K]
    int K, n_units, rpu, ups;
    int stages;             // ring slots (<= kGemvMaxStages)
    uint32_t slot_bytes;    // bytes per ring slot (>= ups * rpu * K * 2, multiple of 128)
    const float *in;        // input vector (x when gain != nullptr)
    const uint16_t *gain;   // RMSNorm gain (bf16) or nullptr for a plain input
    const uint16_t *embed;  // non-null: the input is embed[ctrl[CTRL_TOKEN]] (layer 0)
    float *x_out;           // embed variant: CTA 0 stores the embedded row here
    int *ctrl;
    float eps;
    // the GEMV launched after this one: the producer moves the first rows of
    // this CTA's share of it into L2 once its own rows are issued
    const uint16_t *next_W;  // nullptr: none
    int next_K, next_n_units, next_rpu;
};

// ---------------------------------------------------------------- epilogues --
// unit(u, v): v[0..rpu) are the finished dot products of unit u's rows.

struct EpiResidual {  // x[u] += W x_in   (O projection, down projection)
    float *x;
    static constexpr bool kArgmax = false;
    // x is read at L2 (.cg): inside the persistent decode kernel other SMs write it
    __device__ void unit(int u, const float *v) { x[u] = __ldcg(x + u) + v[0]; }
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
    float *kraw;           // qk_norm: q and k leave unnormalised and without RoPE (k here)
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
        if (kraw && r0 < qdim + kvdim) {
            // the per-head norm needs the whole head: the attention phase finishes q and k
            const int hd = r0 / d, i = (r0 % d) >> 1, half = d >> 1;
            float *dst = r0 < qdim ? q + hd * d : kraw + (hd - qdim / d) * d;
            dst[i] = a;
            dst[i + half] = b;
        } else if (r0 < qdim + kvdim) {
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


constexpr int kRedRows = 128;  // rows of partial sums per reduction batch
constexpr int kGemvMaxStages = 8;
// dynamic shared memory: [reduction scratch 2 x 8 warps x kRedRows fp32][ring]
constexpr size_t kGemvRedBytes = 2 * 8 * kRedRows * 4;
static inline size_t gemv_smem_bytes(int stages, uint32_t slot_bytes) {
    return kGemvRedBytes + (size_t)stages * slot_bytes;
}

// ------------------------------------------------------------------- GEMV ----
// Grid: num_sms CTAs, each owning a contiguous, balanced range of units.  Each
// consumer thread holds NCH 8-element chunks of the input vector in registers
// (chunk c = tid + 256 j) and, for every row of a stage, contributes the dot
// product over its chunks; warp sums go to shared memory and are reduced over
// the 8 warps (fixed order) once per batch of up to kRedRows rows.
// Shapes: every slot holds RPS rows (RPS a power of two, at most 8, RPS x K x 2
// <= 32 KB, a multiple of the unit); consumer thread t covers the 8-element
// chunks c = t + 256 j, j < NCH; FULL when the chunks cover K exactly (no tail
// check in the inner loop).
__host__ __device__ constexpr int gemv_rps(int K) {
    return 2 * K * 8 <= 32768 ? 8 : 2 * K * 4 <= 32768 ? 4 : 2 * K * 2 <= 32768 ? 2 : 1;
}
__host__ __device__ constexpr int gemv_nch(int K) { return (K / 8 + 255) / 256; }

constexpr int kGemvConsumers = 256;
constexpr int kGemvWarps = 8;

__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

// consumer barrier that also returns the OR of every consumer thread's flag, so
// all of them take the same branch afterwards
__device__ __forceinline__ bool consumer_sync_or(bool v) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 q, %1, 0;\n\t"
        "bar.red.or.pred p, 1, 256, q;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)v)
        : "memory");
    return r != 0;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 r;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "r"(addr));
    return r;
}

// a + (8 bf16 weights) . (8 fp32 inputs)
__device__ __forceinline__ float dot8(const uint4 w, const float *h, float a) {
    a = fmaf(bf16lo(w.x), h[0], a);
    a = fmaf(bf16hi(w.x), h[1], a);
    a = fmaf(bf16lo(w.y), h[2], a);
    a = fmaf(bf16hi(w.y), h[3], a);
    a = fmaf(bf16lo(w.z), h[4], a);
    a = fmaf(bf16hi(w.z), h[5], a);
    a = fmaf(bf16lo(w.w), h[6], a);
    a = fmaf(bf16hi(w.w), h[7], a);
    return a;
}

// Warp sums of a slot's RPS rows (each lane holds its partial of every row),
// stored to rb[0, rows): a transposed butterfly.  R = RPS rounded up to a power
// of two; at each of the first log2(R) levels a lane keeps one half of its rows
// and trades the other half with its partner, so one shuffle moves one row (R - 1
// shuffles in all instead of 5 R); plain butterflies finish the sum.  Lane l then
// holds the row whose index is spelled by lane bits 4, 3, ... (most significant
// first), and the lanes whose remaining low bits are zero store it.
template <int RPS>
__device__ __forceinline__ void warp_rows_store(const float (&acc)[RPS], float *rb, int rows, int lane) {
    constexpr int R = RPS <= 1 ? 1 : RPS <= 2 ? 2 : RPS <= 4 ? 4 : 8;
    static_assert(RPS <= 8, "at most 8 rows per slot");
    float v[R];
#pragma unroll
    for (int i = 0; i < R; ++i) v[i] = i < RPS ? acc[i] : 0.f;
    int row = 0;
#pragma unroll
    for (int o = 16, cnt = R; o > 0; o >>= 1) {
        if (cnt > 1) {
            const bool up = (lane & o) != 0;
#pragma unroll
            for (int t = 0; t < cnt / 2; ++t) {
                const float send = up ? v[t] : v[t + cnt / 2];
                const float keep = up ? v[t + cnt / 2] : v[t];
                v[t] = keep + __shfl_xor_sync(0xffffffffu, send, o);
            }
            if (up) row += cnt / 2;
            cnt >>= 1;
        } else {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
        }
    }
    if ((lane & (32 / R - 1)) == 0 && row < rows) rb[row] = v[0];
}

// ------------------------------------------------- 8-bit block rows (decode) --
// A row of the 8-bit block format in shared memory: K int8 codes (two's
// complement), then the row's K/32 fp16 block scales.
//
// The input vector of a phase is put once into fixed point, X[c] = rint(h[c] *
// 2^E) with |X| < 2^23 (three byte digits) or 2^15 (two), E from the vector's
// largest magnitude (one rounding of at most 2^-24, or 2^-16, of it), and X is
// cut into byte digits, e.g. X = 65536 X2 + 256 X1 + X0 (X2 signed, the others
// unsigned).  The
// integer dot products of 16 codes with each digit (dp4a, exact in int32) make
// the chunk's exact sum q . X, which one fp32 rounding carries into the row's
// fp32 accumulator with the block scale; 2^-E is applied once per row.  That is
// 12 dp4a and a handful of fp32 operations per 16 codes, where converting every
// code to fp32 costs three operations per code.
__device__ __forceinline__ int dp4a_ss(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.s32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}
__device__ __forceinline__ int dp4a_su(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.s32.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}
// exact int -> fp32 for |v| < 2^22: the integer added under the exponent of 1.5 * 2^23
__device__ __forceinline__ float small_int_to_f32(int v) {
    return __int_as_float(0x4B400000 + v) - 12582912.0f;
}

__device__ __forceinline__ float lds_f16(uint32_t addr) {
    unsigned short v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(addr));
    return __half2float(__ushort_as_half(v));
}

// ------------------------------------------------------------------- GEMV ----
// Grid: num_sms CTAs, each owning a contiguous, balanced range of units.  The
// producer warp streams the CTA's rows, RPS per slot, through the ring; each of
// the 8 consumer warps adds its chunks of every row and reduces the slot's RPS
// rows with interleaved butterflies; warp sums go to shared memory and are
// reduced over the warps (fixed order) once per kRedRows rows, then passed to
// the epilogue.
template <int NCH, int RPS, bool FULL, class Epi>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_kernel(const GemvIn g, const Epi epi_in) {
    extern __shared__ __align__(128) uint8_t smem[];
    float *red = reinterpret_cast<float *>(smem);  // [2][kGemvWarps][kRedRows]
    uint8_t *ring = smem + kGemvRedBytes;
    __shared__ __align__(8) uint64_t bars[2 * kGemvMaxStages];  // full[S], empty[S]
    __shared__ float s_part[kGemvWarps];
    __shared__ int s_abort;
    __shared__ float s_bv[kGemvWarps];
    __shared__ int s_bi[kGemvWarps];
    __shared__ int s_last;
    const int S = g.stages;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = gridDim.x;
    const int u0 = (int)(((long long)blockIdx.x * g.n_units) / G);
    const int u1 = (int)(((long long)(blockIdx.x + 1) * g.n_units) / G);
    const int nunits = u1 - u0;
    const int total_rows = nunits * g.rpu;
    const int nst = (total_rows + RPS - 1) / RPS;
    int *err = g.ctrl + CTRL_ERR;

    const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + kGemvMaxStages);
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, kGemvWarps);
        }
        fence_barrier_init();
        s_abort = 0;
    }
    __syncthreads();
    griddep_launch_dependents();

    if (warp == kGemvWarps) {  // ------------------------------------ producer
        if (lane == 0) {
            const uint64_t pol = l2_evict_first();
            const uint32_t ring0 = smem_u32(ring);
            const uint16_t *src = g.W + (size_t)u0 * g.rpu * g.K;
            int issued = 0;
            for (int s = 0; s < nst; ++s) {
                const int slot = s % S;
                if (s >= S && !mbar_wait(empty0 + 8 * slot, ((s / S) + 1) & 1, err, SITE_GEMV_EMPTY)) break;
                const int rows = min(RPS, total_rows - s * RPS);
                const uint32_t bytes = (uint32_t)rows * (uint32_t)g.K * 2u;
                mbar_arrive_expect_tx(full0 + 8 * slot, bytes);
                bulk_g2s(ring0 + slot * g.slot_bytes, src + (size_t)s * RPS * g.K, bytes, full0 + 8 * slot, pol);
                issued = s + 1;
            }
            if (g.next_W) {
                // the next kernel's CTA of the same index streams units [nu0, nu1); its
                // first ring-full is fetched while this CTA drains, so the HBM stays busy
                // across the kernel boundary
                const int nu0 = (int)(((long long)blockIdx.x * g.next_n_units) / G);
                const int nu1 = (int)(((long long)(blockIdx.x + 1) * g.next_n_units) / G);
                const size_t total = (size_t)(nu1 - nu0) * g.next_rpu * g.next_K * 2;
                const size_t want = total < (size_t)kGemvRingBytes ? total : (size_t)kGemvRingBytes;
                const uint8_t *src = reinterpret_cast<const uint8_t *>(g.next_W + (size_t)nu0 * g.next_rpu * g.next_K);
                for (size_t off = 0; off < want; off += 32768)
                    bulk_prefetch_l2(src + off, (uint32_t)(want - off < 32768 ? want - off : 32768));
            }
            // no copy may still be landing in this CTA's shared memory when it exits
            for (int s = max(0, issued - S); s < issued; ++s)
                mbar_wait(full0 + 8 * (s % S), (s / S) & 1, err, SITE_GEMV_DRAIN);
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
        const int c = tid + kGemvConsumers * j;
        if (FULL || c < nchunks) {
            if (g.embed) {
                const uint4 w = *reinterpret_cast<const uint4 *>(g.embed + (size_t)tok * g.K + c * 8);
                h[j][0] = bf16lo(w.x); h[j][1] = bf16hi(w.x); h[j][2] = bf16lo(w.y); h[j][3] = bf16hi(w.y);
                h[j][4] = bf16lo(w.z); h[j][5] = bf16hi(w.z); h[j][6] = bf16lo(w.w); h[j][7] = bf16hi(w.w);
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
        consumer_sync();
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < kGemvWarps; ++w) tot += s_part[w];
        const float rinv = 1.0f / sqrtf(tot / (float)g.K + g.eps);
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int c = tid + kGemvConsumers * j;
            if (FULL || c < nchunks) {
                const uint4 gw = *reinterpret_cast<const uint4 *>(g.gain + c * 8);
                const float gg[8] = {bf16lo(gw.x), bf16hi(gw.x), bf16lo(gw.y), bf16hi(gw.y),
                                     bf16lo(gw.z), bf16hi(gw.z), bf16lo(gw.w), bf16hi(gw.w)};
#pragma unroll
                for (int e = 0; e < 8; ++e) h[j][e] = h[j][e] * rinv * gg[e];
            }
        }
    }

    const uint32_t row_bytes = (uint32_t)g.K * 2u;
    const uint32_t my0 = smem_u32(ring) + (uint32_t)tid * 16u;   // this thread's chunk 0 in slot 0
    const bool tail_ok = FULL || tid + kGemvConsumers * (NCH - 1) < nchunks;
    int buf = 0, brow = 0, bunit0 = 0, slot = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int s = 0; s < nst; ++s) {
        const int rows = min(RPS, total_rows - s * RPS);
        ok = ok && !*reinterpret_cast<volatile int *>(&s_abort) &&
             mbar_wait(full0 + 8 * slot, phase, err, SITE_GEMV_FULL);
        if (!ok) s_abort = 1;
        float acc[RPS];
#pragma unroll
        for (int r = 0; r < RPS; ++r) acc[r] = 0.f;
        if (ok) {
            const uint32_t sb = my0 + (uint32_t)slot * g.slot_bytes;
            if (rows == RPS) {
#pragma unroll
                for (int r = 0; r < RPS; ++r)
#pragma unroll
                    for (int j = 0; j < NCH; ++j)
                        if (j < NCH - 1 || tail_ok)
                            acc[r] = dot8(lds128(sb + r * row_bytes + j * kGemvConsumers * 16), h[j], acc[r]);
            } else {   // the CTA's last slot may hold fewer rows
#pragma unroll
                for (int r = 0; r < RPS; ++r)
                    if (r < rows)
#pragma unroll
                        for (int j = 0; j < NCH; ++j)
                            if (j < NCH - 1 || tail_ok)
                                acc[r] = dot8(lds128(sb + r * row_bytes + j * kGemvConsumers * 16), h[j], acc[r]);
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * slot);
        if (++slot == S) {
            slot = 0;
            phase ^= 1u;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
#pragma unroll
            for (int r = 0; r < RPS; ++r) acc[r] += __shfl_xor_sync(0xffffffffu, acc[r], o);
        if (lane == 0) {
            float *rb = red + (size_t)(buf * kGemvWarps + warp) * kRedRows + brow;
#pragma unroll
            for (int r = 0; r < RPS; ++r)
                if (r < rows) rb[r] = acc[r];
        }
        brow += rows;
        if (s == nst - 1 || brow + RPS > kRedRows) {
            consumer_sync();
            if (s_abort) break;
            const int bunits = brow / g.rpu;
            for (int t = tid; t < bunits; t += kGemvConsumers) {
                float v[2];
                for (int j = 0; j < g.rpu; ++j) {
                    float sum = 0.f;
#pragma unroll
                    for (int w = 0; w < kGemvWarps; ++w)
                        sum += red[(size_t)(buf * kGemvWarps + w) * kRedRows + t * g.rpu + j];
                    v[j] = sum;
                }
                epi.unit(u0 + bunit0 + t, v);
            }
            bunit0 += bunits;
            brow = 0;
            buf ^= 1;
        }
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
        consumer_sync();
        if (tid == 0) {
            for (int w = 1; w < kGemvWarps; ++w)
                if (better(s_bv[w], s_bi[w], bv, bi)) { bv = s_bv[w]; bi = s_bi[w]; }
            epi.partial[blockIdx.x] = make_int2(__float_as_int(bv), bi);
            __threadfence();
            const int t = atomicAdd(epi.ctrl + CTRL_LM_TICKET, 1);
            s_last = (t == G - 1);
        }
        consumer_sync();
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
// Split-K attention of one query token over the paged cache (Sec. 5.1 decode
// step).  Grid (S, nkv): CTA (r, g) covers split r of KV head g, a contiguous
// range of the cached pages; block = group x wph query warps + 1 producer warp.
// The producer streams the range's pages (the K and V blocks of head g, 16 x d
// bf16 each, contiguous in a page) through a small TMA ring; query warp
// (j, set) runs an online softmax for query head g*group + j over the pages
// i = set (mod wph) of the range, and the wph states of a head are merged in
// shared memory.  Each CTA writes its per-head state (acc, m, l) to global
// memory and takes a ticket; the last CTA of head g combines the splits in
// split order, so the result does not depend on which CTA finishes last.
//
// No cluster and a small footprint (<= 288 threads, 32 KB ring): the CTAs fit
// beside a GEMV CTA on the same SM, so under programmatic dependent launch the
// kernel starts streaming pages while the QKV GEMV still runs, and the O
// projection's weight ring fills while the attention finishes.  The length comes
// from the device position, so one captured graph serves every step; the split
// count adapts to it at run time (at most gridDim.x splits).
constexpr uint32_t kFdRingBytes = 32768;
constexpr int kFdMaxQueryWarps = 8;
constexpr int kFdMaxSplits = 32;

struct FDArgs {
    const float *q;
    const uint16_t *kv;  // this layer's pages
    const int *pages;
    int *ctrl;
    float *o;
    float *part;         // [nkv][splits][group][d + 4]: acc[d], m, l of each split
    int nkv, group, wph;
    size_t page_elems;
    float qscale;        // log2(e) / sqrt(d)
};

enum : int { SITE_FD_EMPTY = 31, SITE_FD_FULL = 32, SITE_FD_DRAIN = 33 };

// (m, l, acc) online-softmax merge of b into a (log2 domain)
// An empty state (no keys seen) has m = -inf, l = 0, acc = 0 and is skipped:
// exp2(m - M) with both maxima -inf would be NaN.
template <int EPL>
__device__ __forceinline__ void fd_merge(float &m, float &l, float *acc, float mb, float lb, const float *accb) {
    if (mb == -INFINITY) return;
    if (m == -INFINITY) {
        m = mb;
        l = lb;
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] = accb[e];
        return;
    }
    const float M = fmaxf(m, mb);
    const float fa = exp2f(m - M), fb = exp2f(mb - M);
    l = l * fa + lb * fb;
#pragma unroll
    for (int e = 0; e < EPL; ++e) acc[e] = acc[e] * fa + accb[e] * fb;
    m = M;
}

template <int D>
__global__ void __launch_bounds__(32 * (kFdMaxQueryWarps + 1)) flash_decode_kernel(const FDArgs a) {
    constexpr int EPL = D / 32;
    constexpr uint32_t BLK = kPage * D * 2;              // bytes of one K (or V) block of a page
    constexpr int STAGES = (int)(kFdRingBytes / (2 * BLK));
    constexpr int STRIDE = D + 4;                        // floats per state: acc[D], m, l, pad
    extern __shared__ __align__(128) uint8_t fsm[];      // [STAGES][K block | V block]
    __shared__ __align__(8) uint64_t full_bar[STAGES], empty_bar[STAGES];
    __shared__ __align__(16) float s_state[kFdMaxQueryWarps][STRIDE];
    __shared__ int s_last;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nq = a.group * a.wph;   // query warps
    const int g = blockIdx.y;
    const int r = blockIdx.x;
    int *err = a.ctrl + CTRL_ERR;

    // the position is only advanced at the end of a step, so it is stable here
    const int len = *reinterpret_cast<volatile int *>(a.ctrl + CTRL_POS) + 1;
    const int npages = (len + kPage - 1) / kPage;
    const int pps = (npages + (int)gridDim.x - 1) / (int)gridDim.x;
    const int splits = (npages + pps - 1) / pps;          // every split below this has pages
    if (r >= splits) return;                              // idle CTA: no state, no ticket
    const int p0 = r * pps;
    const int n = min(npages, p0 + pps) - p0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), a.group);
        }
        fence_barrier_init();
    }
    __syncthreads();
    griddep_launch_dependents();

    if (w == nq) {  // ---------------------------------------------- producer
        // the whole warp walks the pages so that 32 page-table entries are read at
        // once (one coalesced load) and handed out by shuffle; lane 0 issues
        const uint32_t ring0 = smem_u32(fsm);
        int issued = 0, my_page = 0;
        bool waited = false;
        for (int i = 0; i < n; ++i) {
            if ((i & 31) == 0 && i + lane < n) my_page = a.pages[p0 + i + lane];
            const int page = __shfl_sync(0xffffffffu, my_page, i & 31);
            const int s = i % STAGES;
            bool ok = true;
            if (lane == 0 && i >= STAGES)
                ok = mbar_wait(smem_u32(&empty_bar[s]), ((i / STAGES) + 1) & 1, err, SITE_FD_EMPTY);
            if (!__shfl_sync(0xffffffffu, (int)ok, 0)) break;
            // the page holding the current position is written by the preceding kernel
            if (!waited && p0 + i == npages - 1) {
                griddep_wait();
                waited = true;
            }
            if (lane == 0) {
                const uint16_t *Kb = a.kv + (size_t)page * a.page_elems + (size_t)g * kPage * D;
                const uint16_t *Vb = Kb + (size_t)a.nkv * kPage * D;
                const uint32_t fb = smem_u32(&full_bar[s]);
                mbar_arrive_expect_tx(fb, 2 * BLK);
                bulk_g2s(ring0 + s * 2 * BLK, Kb, BLK, fb);
                bulk_g2s(ring0 + s * 2 * BLK + BLK, Vb, BLK, fb);
            }
            issued = i + 1;
        }
        if (lane == 0)
            for (int i = max(0, issued - STAGES); i < issued; ++i)
                mbar_wait(smem_u32(&full_bar[i % STAGES]), (i / STAGES) & 1, err, SITE_FD_DRAIN);
        __syncwarp();
        return;   // the producer takes no part in the named barriers below
    }

    // ------------------------------------------------------------ query warps
    griddep_wait();
    const int j = w % a.group, set = w / a.group;
    const int head = g * a.group + j;
    float qv[EPL], acc[EPL];
    if constexpr (EPL == 4) {
        const float4 q4 = *reinterpret_cast<const float4 *>(a.q + head * D + lane * 4);
        qv[0] = q4.x * a.qscale; qv[1] = q4.y * a.qscale; qv[2] = q4.z * a.qscale; qv[3] = q4.w * a.qscale;
    } else {
        const float2 q2 = *reinterpret_cast<const float2 *>(a.q + head * D + lane * 2);
        qv[0] = q2.x * a.qscale; qv[1] = q2.y * a.qscale;
    }
#pragma unroll
    for (int e = 0; e < EPL; ++e) acc[e] = 0.f;
    float m = -INFINITY, l = 0.f;
    const int key = lane >> 1;   // the key whose score this lane ends with
    bool ok = true;
    for (int i = set; i < n && ok; i += a.wph) {
        const int s = i % STAGES;
        ok = mbar_wait(smem_u32(&full_bar[s]), (i / STAGES) & 1, err, SITE_FD_FULL);
        if (!ok) break;
        const uint8_t *Ks = fsm + (size_t)s * 2 * BLK;
        const uint8_t *Vs = Ks + BLK;
        const int ntok = min(kPage, len - (p0 + i) * kPage);
        // partial dot products of this lane's d-slice with the 16 keys
        float sc[kPage];
#pragma unroll
        for (int t = 0; t < kPage; ++t) {
            const uint8_t *kr = Ks + (t * D + lane * EPL) * 2;
            if constexpr (EPL == 4) {
                const uint2 kw = *reinterpret_cast<const uint2 *>(kr);
                sc[t] = qv[0] * bf16lo(kw.x) + qv[1] * bf16hi(kw.x) + qv[2] * bf16lo(kw.y) + qv[3] * bf16hi(kw.y);
            } else {
                const uint32_t kw = *reinterpret_cast<const uint32_t *>(kr);
                sc[t] = qv[0] * bf16lo(kw) + qv[1] * bf16hi(kw);
            }
        }
        // transposed butterfly: lanes 2k and 2k+1 end with the full score of key k
#pragma unroll
        for (int o = 16, cnt = kPage; o > 0; o >>= 1) {
            if (cnt > 1) {
                const bool up = (lane & o) != 0;
#pragma unroll
                for (int t = 0; t < cnt / 2; ++t) {
                    const float send = up ? sc[t] : sc[t + cnt / 2];
                    const float keep = up ? sc[t + cnt / 2] : sc[t];
                    sc[t] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                }
                cnt >>= 1;
            } else {
                sc[0] += __shfl_xor_sync(0xffffffffu, sc[0], o);
            }
        }
        const float my = key < ntok ? sc[0] : -INFINITY;   // slots past the length are masked
        const float mx = fmaxf(m, warp_max(my));
        const float corr = exp2f(m - mx);
        const float pme = exp2f(my - mx);                  // 0 for masked keys
        l = l * corr + pme;   // per-lane share of the denominator (every key is held by two lanes)
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] *= corr;
#pragma unroll
        for (int t = 0; t < kPage; ++t) {
            // slots past the length are never used: they may hold stale values
            const bool valid = t < ntok;
            const float pt = __shfl_sync(0xffffffffu, pme, 2 * t);
            const uint8_t *vr = Vs + (t * D + lane * EPL) * 2;
            if constexpr (EPL == 4) {
                uint2 vw = *reinterpret_cast<const uint2 *>(vr);
                if (!valid) vw = make_uint2(0u, 0u);
                acc[0] = fmaf(pt, bf16lo(vw.x), acc[0]);
                acc[1] = fmaf(pt, bf16hi(vw.x), acc[1]);
                acc[2] = fmaf(pt, bf16lo(vw.y), acc[2]);
                acc[3] = fmaf(pt, bf16hi(vw.y), acc[3]);
            } else {
                uint32_t vw = *reinterpret_cast<const uint32_t *>(vr);
                if (!valid) vw = 0u;
                acc[0] = fmaf(pt, bf16lo(vw), acc[0]);
                acc[1] = fmaf(pt, bf16hi(vw), acc[1]);
            }
        }
        m = mx;
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&empty_bar[s]));
    }
    l = warp_sum(l) * 0.5f;
    if (a.wph > 1) {
#pragma unroll
        for (int e = 0; e < EPL; ++e) s_state[w][lane * EPL + e] = acc[e];
        if (lane == 0) {
            s_state[w][D] = m;
            s_state[w][D + 1] = l;
        }
        // merge the wph page sets of each head into set 0 (fixed set order)
        asm volatile("bar.sync 1, %0;" ::"r"(32 * nq) : "memory");
        if (set == 0)
            for (int t = 1; t < a.wph; ++t) {
                const float *o = s_state[t * a.group + j];
                float ob[EPL];
#pragma unroll
                for (int e = 0; e < EPL; ++e) ob[e] = o[lane * EPL + e];
                fd_merge<EPL>(m, l, acc, o[D], o[D + 1], ob);
            }
    }
    // this split's state of head j -> global; then the ticket
    float *mine = a.part + ((size_t)(g * gridDim.x + r) * a.group + j) * STRIDE;
    if (set == 0) {
        if constexpr (EPL == 4)
            *reinterpret_cast<float4 *>(mine + lane * 4) = make_float4(acc[0], acc[1], acc[2], acc[3]);
        else
            *reinterpret_cast<float2 *>(mine + lane * 2) = make_float2(acc[0], acc[1]);
        if (lane == 0) *reinterpret_cast<float2 *>(mine + D) = make_float2(m, l);
    }
    // the CTA barrier orders every warp's stores before thread 0's fence, which
    // publishes them at GPU scope ahead of the ticket (and, for the last CTA, orders
    // the other splits' stores before the loads below)
    asm volatile("bar.sync 1, %0;" ::"r"(32 * nq) : "memory");
    if (threadIdx.x == 0) {
        __threadfence();
        const int t = atomicAdd(a.ctrl + CTRL_ATTN_TICKET0 + g, 1);
        s_last = (t == splits - 1);
        if (s_last) __threadfence();
    }
    asm volatile("bar.sync 1, %0;" ::"r"(32 * nq) : "memory");
    if (!s_last || set != 0) return;

    // ------------------------------------------- last CTA of head g: combine
    const float *base = a.part + ((size_t)g * gridDim.x * a.group + j) * STRIDE;
    const size_t sstride = (size_t)a.group * STRIDE;     // floats between splits of one head
    float2 ml = make_float2(-INFINITY, 0.f);
    if (lane < splits) ml = __ldcg(reinterpret_cast<const float2 *>(base + lane * sstride + D));
    const float M = warp_max(ml.x);
    const float f = lane < splits ? exp2f(ml.x - M) : 0.f;
    const float L = warp_sum(ml.y * f);
    float out[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) out[e] = 0.f;
    for (int s0 = 0; s0 < splits; s0 += 8) {
        float v[8][EPL];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int sp = min(s0 + u, splits - 1);
            const float *src = base + sp * sstride + lane * EPL;
            if constexpr (EPL == 4) {
                const float4 t4 = __ldcg(reinterpret_cast<const float4 *>(src));
                v[u][0] = t4.x; v[u][1] = t4.y; v[u][2] = t4.z; v[u][3] = t4.w;
            } else {
                const float2 t2 = __ldcg(reinterpret_cast<const float2 *>(src));
                v[u][0] = t2.x; v[u][1] = t2.y;
            }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const float fs = __shfl_sync(0xffffffffu, f, (s0 + u) & 31);
            if (s0 + u < splits)
#pragma unroll
                for (int e = 0; e < EPL; ++e) out[e] = fmaf(v[u][e], fs, out[e]);
        }
    }
    const float inv = 1.0f / L;
    if constexpr (EPL == 4)
        *reinterpret_cast<float4 *>(a.o + head * D + lane * 4) =
            make_float4(out[0] * inv, out[1] * inv, out[2] * inv, out[3] * inv);
    else
        *reinterpret_cast<float2 *>(a.o + head * D + lane * 2) = make_float2(out[0] * inv, out[1] * inv);
    if (j == 0 && lane == 0) a.ctrl[CTRL_ATTN_TICKET0 + g] = 0;   // ready for the next layer
}

// ======================================================= persistent decode ====
// The whole decode step (Sec. 5.1: one forward pass per generated token) as one
// cooperative kernel, one CTA per SM.  Weight streaming does not depend on the
// data, so the producer warp walks the step's weights (per layer: this CTA's
// rows of Wqkv, its KV pages, its rows of Wo, Wg|Wu and Wd; then the LM head)
// through one TMA ring without ever waiting on a data dependency, only on free
// ring slots.  The eight consumer warps run the phases in order and meet at a
// grid barrier wherever a phase needs every CTA's output (the normalised
// residual, the attention output, the SwiGLU vector).  While the consumers wait
// at a barrier the ring keeps filling, so the HBM stays busy across the phase
// boundaries that separate kernels in the multi-launch path.
//
// Data written by one CTA and read by another inside the launch (x, q, o, m,
// the attention split states, this step's K/V row) is read at L2 (.cg loads),
// never from a possibly stale L1 line.
constexpr int kMegaSlots = 6;
constexpr uint32_t kMegaSlotBytes = 32768;
constexpr size_t kMegaSmem = kGemvRedBytes + (size_t)kMegaSlots * kMegaSlotBytes;
constexpr size_t kMegaPrefetchBytes = 196608;
constexpr int kMegaMaxCtas = 256;   // grid size limit (one CTA per SM)   // gate/up bytes per CTA moved into L2 during attention

enum : int { SITE_MEGA_EMPTY = 51, SITE_MEGA_FULL = 52, SITE_MEGA_DRAIN = 53, SITE_MEGA_GRID = 54 };

template <int NCH_, int RPS_, bool FULL_>
struct GShape {
    static constexpr int NCH = NCH_, RPS = RPS_;
    static constexpr bool FULL = FULL_;
};

struct MegaArgs {
    const uint16_t *W;          // weight arena
    float *kraw;                // qk_norm: this step's k before its norm and RoPE [kvdim], else nullptr
    size_t lstride;             // elements between the same tensor of consecutive layers
    LayerOffsets l0;            // layer 0 offsets
    size_t w_embed, w_final_norm, w_lm;
    uint16_t *KV;
    size_t kv_layer_elems, page_elems;
    int *ctrl, *hist;
    float *x, *q, *o, *m, *logits;
    int2 *amax;
    const float2 *rope;
    const int *pages;
    float *part;                // attention split states [nkv][splits][group][d + 4]
    uint32_t *bound;            // [grid + 1] share boundaries of the GEMV phases (2^24 = all rows)
    float *cta_time;            // [grid] each CTA's gate/up streaming time in the last step (us)
    int L, H, F, V, nqkv, qdim, kvdim, d, nkv, group, wph, splits;
    int bias;
    float eps, qscale;
};

struct MegaRing {
    uint32_t full0, empty0, data0;   // shared-memory addresses
    const uint8_t *ring;             // generic pointer to slot 0
    int n;   // slots issued (producer) or consumed (consumer) so far
    int *abort;                      // shared flag: a consumer wait gave up
    uint32_t b0, b1;                 // this CTA's share of every GEMV phase: [b0, b1) / 2^24
};

// units [u0, u1) of an n-unit phase for the share [b0, b1) (fixed point, 2^24 = all)
__device__ __forceinline__ int mega_unit(uint32_t b, int n_units) {
    return (int)(((unsigned long long)b * (unsigned long long)n_units) >> 24);
}

// ----------------------------------------------------------- producer side --
// this CTA's rows of an n_units-unit matrix whose rows are row_bytes long (bf16:
// 2K; the 8-bit block format: q8_row_bytes(K)), RPS rows per ring slot
__device__ bool mp_rows(MegaRing &R, const uint16_t *W, uint32_t row_bytes, int n_units, int rpu, int RPS,
                        int *err, uint64_t pol) {
    const int u0 = mega_unit(R.b0, n_units);
    const int u1 = mega_unit(R.b1, n_units);
    const int total_rows = (u1 - u0) * rpu;
    const int nst = (total_rows + RPS - 1) / RPS;
    const uint8_t *src = reinterpret_cast<const uint8_t *>(W) + (size_t)u0 * rpu * row_bytes;
    for (int s = 0; s < nst; ++s) {
        const int slot = R.n % kMegaSlots;
        if (R.n >= kMegaSlots &&
            !mbar_wait(R.empty0 + 8 * slot, ((R.n / kMegaSlots) + 1) & 1, err, SITE_MEGA_EMPTY))
            return false;
        const int rows = min(RPS, total_rows - s * RPS);
        const uint32_t bytes = (uint32_t)rows * row_bytes;
        mbar_arrive_expect_tx(R.full0 + 8 * slot, bytes);
        bulk_g2s(R.data0 + slot * kMegaSlotBytes, src + (size_t)s * RPS * row_bytes, bytes, R.full0 + 8 * slot, pol);
        ++R.n;
    }
    return true;
}

// move rows [skip, skip + bytes) of this CTA's share of a GEMV phase into L2
__device__ void mp_prefetch(const MegaRing &R, const uint16_t *W, uint32_t row_bytes, int n_units, int rpu,
                            size_t skip, size_t bytes) {
    const int u0 = mega_unit(R.b0, n_units);
    const int u1 = mega_unit(R.b1, n_units);
    const size_t row = row_bytes;
    const size_t own = (size_t)(u1 - u0) * rpu * row;
    skip -= skip % row;
    const size_t end = own < skip + bytes ? own : skip + bytes;
    const uint8_t *src = reinterpret_cast<const uint8_t *>(W) + (size_t)u0 * rpu * row;
    for (size_t off = skip; off < end; off += 32768)
        bulk_prefetch_l2(src + off, (uint32_t)(end - off < 32768 ? end - off : 32768));
}

// the pages of this CTA's attention split (its K and V blocks), one page per slot
struct MegaSplit {
    int g, r, p0, n, npages, splits;
    bool active;
};

__device__ __forceinline__ MegaSplit mega_split(const MegaArgs &a, int len) {
    MegaSplit sp;
    const int unit = blockIdx.x;
    sp.npages = (len + kPage - 1) / kPage;
    const int pps = (sp.npages + a.splits - 1) / a.splits;
    sp.splits = (sp.npages + pps - 1) / pps;
    sp.g = unit / a.splits;
    sp.r = unit % a.splits;
    sp.active = unit < a.nkv * a.splits && sp.r < sp.splits;
    sp.p0 = sp.r * pps;
    sp.n = sp.active ? min(sp.npages, sp.p0 + pps) - sp.p0 : 0;
    return sp;
}

template <int D>
__device__ bool mp_pages(MegaRing &R, const MegaArgs &a, const uint16_t *kvl, const MegaSplit &sp, int *err) {
    constexpr uint32_t BLK = kPage * D * 2;
    for (int i = 0; i < sp.n; ++i) {
        const int slot = R.n % kMegaSlots;
        if (R.n >= kMegaSlots &&
            !mbar_wait(R.empty0 + 8 * slot, ((R.n / kMegaSlots) + 1) & 1, err, SITE_MEGA_EMPTY))
            return false;
        const int page = a.pages[sp.p0 + i];
        const uint16_t *Kb = kvl + (size_t)page * a.page_elems + (size_t)sp.g * kPage * D;
        const uint16_t *Vb = Kb + (size_t)a.nkv * kPage * D;
        mbar_arrive_expect_tx(R.full0 + 8 * slot, 2 * BLK);
        bulk_g2s(R.data0 + slot * kMegaSlotBytes, Kb, BLK, R.full0 + 8 * slot);
        bulk_g2s(R.data0 + slot * kMegaSlotBytes + BLK, Vb, BLK, R.full0 + 8 * slot);
        ++R.n;
    }
    return true;
}

// ----------------------------------------------------------- consumer side --
// consumers only (8 warps): bar.sync 1, 256 is consumer_sync()

// Grid barrier number k (1-based): every CTA's consumer writes so far are visible
// to every CTA afterwards.  Gives up after kWaitLimitNs, or at once when another
// CTA has recorded an error.
__device__ bool mega_grid_sync(int *ctrl, int k, int *s_flag) {
    consumer_sync();
    if (threadIdx.x == 0) {
        int *ctr = ctrl + CTRL_GRID_BAR;
        const int target = k * (int)gridDim.x;
        // release: every consumer store of this CTA (ordered before this thread by
        // the barrier above) is visible to a CTA whose acquire load sees the count
        asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(ctr) : "memory");
        bool ok = false;
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0; it < 0x7FFFFFFFu; ++it) {
            int v;
            asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
            if (v >= target) {
                ok = true;
                break;
            }
            if (*reinterpret_cast<volatile int *>(ctrl + CTRL_ERR) != 0) break;
            if ((it & 15u) == 15u && globaltimer_ns() - t0 > kWaitLimitNs) {
                atomicCAS(ctrl + CTRL_ERR, 0, SITE_MEGA_GRID);
                break;
            }
            __nanosleep(20);
        }
        *s_flag = ok ? 1 : 0;
    }
    consumer_sync();
    return *s_flag != 0;
}

// One GEMV phase of the consumers: the rows of units [u0, u1) of a K-column matrix
// against `in` (RMSNorm'd with `gain` when given; layer 0 reads embed[token]).
template <class SH, class Epi>
__device__ bool mc_gemv(MegaRing &R, float *red, int K, int n_units, int rpu, const float *in,
                        const uint16_t *gain, const uint16_t *embed, float *x_out, float eps, int *ctrl, Epi &epi,
                        float *s_part) {
    constexpr int NCH = SH::NCH, RPS = SH::RPS;
    constexpr bool FULL = SH::FULL;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int u0 = mega_unit(R.b0, n_units);
    const int u1 = mega_unit(R.b1, n_units);
    const int total_rows = (u1 - u0) * rpu;
    const int nst = (total_rows + RPS - 1) / RPS;
    int *err = ctrl + CTRL_ERR;
    const int nchunks = K >> 3;
    float h[NCH][8];
    float ss = 0.f;
    const int tok = embed ? ctrl[CTRL_TOKEN] : 0;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
        const int c = tid + kGemvConsumers * j;
        if (FULL || c < nchunks) {
            if (embed) {
                const uint4 w = *reinterpret_cast<const uint4 *>(embed + (size_t)tok * K + c * 8);
                h[j][0] = bf16lo(w.x); h[j][1] = bf16hi(w.x); h[j][2] = bf16lo(w.y); h[j][3] = bf16hi(w.y);
                h[j][4] = bf16lo(w.z); h[j][5] = bf16hi(w.z); h[j][6] = bf16lo(w.w); h[j][7] = bf16hi(w.w);
                if (blockIdx.x == 0) {
                    float4 *dst = reinterpret_cast<float4 *>(x_out + c * 8);
                    dst[0] = make_float4(h[j][0], h[j][1], h[j][2], h[j][3]);
                    dst[1] = make_float4(h[j][4], h[j][5], h[j][6], h[j][7]);
                }
            } else {
                const float4 a = __ldcg(reinterpret_cast<const float4 *>(in + c * 8));
                const float4 b = __ldcg(reinterpret_cast<const float4 *>(in + c * 8 + 4));
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
    if (gain) {
        ss = warp_sum(ss);
        if (lane == 0) s_part[warp] = ss;
        consumer_sync();
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < kGemvWarps; ++w) tot += s_part[w];
        const float rinv = 1.0f / sqrtf(tot / (float)K + eps);
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int c = tid + kGemvConsumers * j;
            if (FULL || c < nchunks) {
                const uint4 gw = *reinterpret_cast<const uint4 *>(gain + c * 8);
                const float gg[8] = {bf16lo(gw.x), bf16hi(gw.x), bf16lo(gw.y), bf16hi(gw.y),
                                     bf16lo(gw.z), bf16hi(gw.z), bf16lo(gw.w), bf16hi(gw.w)};
#pragma unroll
                for (int e = 0; e < 8; ++e) h[j][e] = h[j][e] * rinv * gg[e];
            }
        }
    }

    const uint32_t row_bytes = (uint32_t)K * 2u;
    const bool tail_ok = FULL || tid + kGemvConsumers * (NCH - 1) < nchunks;
    int buf = 0, brow = 0, bunit0 = 0;
    bool ok = true;
    for (int s = 0; s < nst; ++s) {
        const int slot = R.n % kMegaSlots;
        const int rows = min(RPS, total_rows - s * RPS);
        // after a wait gives up every thread still reaches the same barriers; they
        // leave together at the next flush
        ok = ok && !*reinterpret_cast<volatile int *>(R.abort) &&
             mbar_wait(R.full0 + 8 * slot, (R.n / kMegaSlots) & 1, err, SITE_MEGA_FULL);
        if (!ok) *R.abort = 1;
        float acc[RPS];
#pragma unroll
        for (int r = 0; r < RPS; ++r) acc[r] = 0.f;
        const uint32_t sb = R.data0 + (uint32_t)slot * kMegaSlotBytes + (uint32_t)tid * 16u;
        if (!ok) {
        } else if (rows == RPS) {
#pragma unroll
            for (int r = 0; r < RPS; ++r)
#pragma unroll
                for (int j = 0; j < NCH; ++j)
                    if (j < NCH - 1 || tail_ok)
                        acc[r] = dot8(lds128(sb + r * row_bytes + j * kGemvConsumers * 16), h[j], acc[r]);
        } else {
#pragma unroll
            for (int r = 0; r < RPS; ++r)
                if (r < rows)
#pragma unroll
                    for (int j = 0; j < NCH; ++j)
                        if (j < NCH - 1 || tail_ok)
                            acc[r] = dot8(lds128(sb + r * row_bytes + j * kGemvConsumers * 16), h[j], acc[r]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(R.empty0 + 8 * slot);
        ++R.n;
        warp_rows_store<RPS>(acc, red + (size_t)(buf * kGemvWarps + warp) * kRedRows + brow, rows, lane);
        brow += rows;
        if (s == nst - 1 || brow + RPS > kRedRows) {
            if (consumer_sync_or(!ok)) return false;
            const int bunits = brow / rpu;
            for (int t = tid; t < bunits; t += kGemvConsumers) {
                float v[2];
                for (int j = 0; j < rpu; ++j) {
                    float sum = 0.f;
#pragma unroll
                    for (int w = 0; w < kGemvWarps; ++w)
                        sum += red[(size_t)(buf * kGemvWarps + w) * kRedRows + t * rpu + j];
                    v[j] = sum;
                }
                epi.unit(u0 + bunit0 + t, v);
            }
            bunit0 += bunits;
            brow = 0;
            buf ^= 1;
        }
    }
    return true;
}

// One GEMV phase over a matrix in the 8-bit block format (rows of
// q8_row_bytes(K) bytes), same role as mc_gemv.  Thread t owns the 16-element
// chunks c = t + 256 j of the input, as byte digits of its fixed-point form.
// ND: byte digits of the fixed-point input (3: 24 bits; 2: 16 bits)
template <class QS, int ND, class Epi>
__device__ bool mc_gemv_q8(MegaRing &R, float *red, int K, int n_units, int rpu, const float *in,
                           const uint16_t *gain, const uint16_t *embed, float *x_out, float eps, int *ctrl, Epi &epi,
                           float *s_part) {
    static_assert(ND == 2 || ND == 3, "two or three input digits");
    constexpr int NCH = QS::NCH, RPS = QS::RPS;
    constexpr bool FULL = QS::FULL;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int u0 = mega_unit(R.b0, n_units);
    const int u1 = mega_unit(R.b1, n_units);
    const int total_rows = (u1 - u0) * rpu;
    const int nst = (total_rows + RPS - 1) / RPS;
    int *err = ctrl + CTRL_ERR;
    const int nchunks = K >> 4;
    float h[NCH][16];
    float ss = 0.f;
    const int tok = embed ? ctrl[CTRL_TOKEN] : 0;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
        const int c = tid + kGemvConsumers * j;
        if (FULL || c < nchunks) {
            if (embed) {
#pragma unroll
                for (int hv = 0; hv < 2; ++hv) {
                    const uint4 w = *reinterpret_cast<const uint4 *>(embed + (size_t)tok * K + c * 16 + hv * 8);
                    float *d = h[j] + hv * 8;
                    d[0] = bf16lo(w.x); d[1] = bf16hi(w.x); d[2] = bf16lo(w.y); d[3] = bf16hi(w.y);
                    d[4] = bf16lo(w.z); d[5] = bf16hi(w.z); d[6] = bf16lo(w.w); d[7] = bf16hi(w.w);
                }
                if (blockIdx.x == 0) {
                    float4 *dst = reinterpret_cast<float4 *>(x_out + c * 16);
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        dst[q] = make_float4(h[j][4 * q], h[j][4 * q + 1], h[j][4 * q + 2], h[j][4 * q + 3]);
                }
            } else {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float4 a = __ldcg(reinterpret_cast<const float4 *>(in + c * 16 + 4 * q));
                    h[j][4 * q] = a.x; h[j][4 * q + 1] = a.y; h[j][4 * q + 2] = a.z; h[j][4 * q + 3] = a.w;
                }
            }
#pragma unroll
            for (int e = 0; e < 16; ++e) ss = fmaf(h[j][e], h[j][e], ss);
        } else {
#pragma unroll
            for (int e = 0; e < 16; ++e) h[j][e] = 0.f;
        }
    }
    // with the RMSNorm gain applied (before the common factor 1/rms), and the
    // largest magnitude for the fixed point: one reduction of (sum of squares, max)
    float mx = 0.f;
    if (gain) {
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int c = tid + kGemvConsumers * j;
            if (FULL || c < nchunks) {
#pragma unroll
                for (int hv = 0; hv < 2; ++hv) {
                    const uint4 gw = *reinterpret_cast<const uint4 *>(gain + c * 16 + hv * 8);
                    const float gg[8] = {bf16lo(gw.x), bf16hi(gw.x), bf16lo(gw.y), bf16hi(gw.y),
                                         bf16lo(gw.z), bf16hi(gw.z), bf16lo(gw.w), bf16hi(gw.w)};
#pragma unroll
                    for (int e = 0; e < 8; ++e) h[j][hv * 8 + e] *= gg[e];
                }
            }
        }
    }
#pragma unroll
    for (int j = 0; j < NCH; ++j)
#pragma unroll
        for (int e = 0; e < 16; ++e) mx = fmaxf(mx, fabsf(h[j][e]));
    ss = warp_sum(ss);
    mx = warp_max(mx);
    if (lane == 0) {
        s_part[warp] = ss;
        s_part[kGemvWarps + warp] = mx;
    }
    consumer_sync();
    float tot = 0.f, M = 0.f;
#pragma unroll
    for (int w = 0; w < kGemvWarps; ++w) {
        tot += s_part[w];
        M = fmaxf(M, s_part[kGemvWarps + w]);
    }
    if (gain) {
        const float rinv = 1.0f / sqrtf(tot / (float)K + eps);
        M *= rinv;
#pragma unroll
        for (int j = 0; j < NCH; ++j)
#pragma unroll
            for (int e = 0; e < 16; ++e) h[j][e] *= rinv;
    }
    // fixed point: M * 2^E just below 2^(8 ND - 1) for the largest magnitude M
    // (values that round past the limit are clamped to it)
    constexpr int XBITS = 8 * ND - 1;
    const int E = M > 0.f ? min(XBITS - 1 - ilogbf(M), 120) : 0;
    const float to_fixed = ldexpf(1.0f, E), from_fixed = ldexpf(1.0f, -E);
    // byte digits, most significant (signed) first: X = sum_i X_i 256^(ND-1-i)
    uint32_t dg[NCH][ND][4];   // [chunk][digit][4 words of 4 byte digits]
#pragma unroll
    for (int j = 0; j < NCH; ++j)
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            uint32_t w[ND];
#pragma unroll
            for (int i = 0; i < ND; ++i) w[i] = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const int X = max(min(__float2int_rn(h[j][4 * k + b] * to_fixed), (1 << XBITS) - 1), -(1 << XBITS) + 1);
#pragma unroll
                for (int i = 0; i < ND; ++i) w[i] |= ((uint32_t)(X >> (8 * (ND - 1 - i))) & 0xFFu) << (8 * b);
            }
#pragma unroll
            for (int i = 0; i < ND; ++i) dg[j][i][k] = w[i];
        }

    const uint32_t row_bytes = (uint32_t)q8_row_bytes((size_t)K);
    const bool tail_ok = FULL || tid + kGemvConsumers * (NCH - 1) < nchunks;
    int buf = 0, brow = 0, bunit0 = 0;
    bool ok = true;
    for (int s = 0; s < nst; ++s) {
        const int slot = R.n % kMegaSlots;
        const int rows = min(RPS, total_rows - s * RPS);
        ok = ok && !*reinterpret_cast<volatile int *>(R.abort) &&
             mbar_wait(R.full0 + 8 * slot, (R.n / kMegaSlots) & 1, err, SITE_MEGA_FULL);
        if (!ok) *R.abort = 1;
        float acc[RPS];
#pragma unroll
        for (int r = 0; r < RPS; ++r) acc[r] = 0.f;
        // chunk c: codes at byte 16 c of the row, its block's scale at byte K + 2 (c / 2)
        const uint32_t s0 = R.data0 + (uint32_t)slot * kMegaSlotBytes;
        const uint32_t sb = s0 + (uint32_t)tid * 16u;
        const uint32_t sc = s0 + (uint32_t)K + (uint32_t)(tid >> 1) * 2u;
        if (ok) {
#pragma unroll
            for (int r = 0; r < RPS; ++r)
                if (rows == RPS || r < rows)
#pragma unroll
                    for (int j = 0; j < NCH; ++j)
                        if (j < NCH - 1 || tail_ok) {
                            const uint4 w = lds128(sb + r * row_bytes + j * kGemvConsumers * 16);
                            const float d = lds_f16(sc + r * row_bytes + j * (kGemvConsumers / 2) * 2);
                            const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
                            int a[ND];
#pragma unroll
                            for (int i = 0; i < ND; ++i) a[i] = 0;
#pragma unroll
                            for (int k = 0; k < 4; ++k)
#pragma unroll
                                for (int i = 0; i < ND; ++i)
                                    a[i] = i == 0 ? dp4a_ss(ws[k], dg[j][i][k], a[i]) : dp4a_su(ws[k], dg[j][i][k], a[i]);
                            float cv = small_int_to_f32(a[0]);
#pragma unroll
                            for (int i = 1; i < ND; ++i) cv = fmaf(cv, 256.0f, small_int_to_f32(a[i]));
                            acc[r] = fmaf(d, cv, acc[r]);
                        }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(R.empty0 + 8 * slot);
        ++R.n;
        warp_rows_store<RPS>(acc, red + (size_t)(buf * kGemvWarps + warp) * kRedRows + brow, rows, lane);
        brow += rows;
        if (s == nst - 1 || brow + RPS > kRedRows) {
            if (consumer_sync_or(!ok)) return false;
            const int bunits = brow / rpu;
            for (int t = tid; t < bunits; t += kGemvConsumers) {
                float v[2];
                for (int j = 0; j < rpu; ++j) {
                    float sum = 0.f;
#pragma unroll
                    for (int w = 0; w < kGemvWarps; ++w)
                        sum += red[(size_t)(buf * kGemvWarps + w) * kRedRows + t * rpu + j];
                    v[j] = sum * from_fixed;
                }
                epi.unit(u0 + bunit0 + t, v);
            }
            bunit0 += bunits;
            brow = 0;
            buf ^= 1;
        }
    }
    return true;
}

// Input digits of the 8-bit GEMV phases: three (24 bits) for QKV, whose outputs
// become the bf16 K/V and the queries, and kQ8RestDigits for O, gate/up, down.
#ifndef WICI_Q8_REST_DIGITS
#define WICI_Q8_REST_DIGITS 3
#endif
constexpr int kQ8QkvDigits = 3, kQ8RestDigits = WICI_Q8_REST_DIGITS;

// a per-layer GEMV phase in the layer matrices' format
template <bool Q8, class S, int ND = kQ8RestDigits, class Epi>
__device__ __forceinline__ bool mc_layer_gemv(MegaRing &R, float *red, int K, int n_units, int rpu, const float *in,
                                              const uint16_t *gain, const uint16_t *embed, float *x_out, float eps,
                                              int *ctrl, Epi &epi, float *s_part) {
    if constexpr (Q8)
        return mc_gemv_q8<S, ND>(R, red, K, n_units, rpu, in, gain, embed, x_out, eps, ctrl, epi, s_part);
    else
        return mc_gemv<S>(R, red, K, n_units, rpu, in, gain, embed, x_out, eps, ctrl, epi, s_part);
}

// Attention of the current token for this CTA's split (KV head g, pages
// [p0, p0 + n)), then the split state to global memory and the ticket; the last
// split of head g combines the states in split order into o.  Warp (j, set) with
// j = warp % group handles query head g*group + j on pages i = set (mod wph);
// warps beyond group * wph only keep the ring in step.
// Qwen3 block, for one head held by a warp (lane l has elements l*EPL ..): RMS
// norm over the head with the gain, then rotate-half RoPE at position pos (the
// partner of element i < D/2 is i + D/2, EPL elements further in lane l + 16).
template <int D>
__device__ __forceinline__ void head_norm_rope(float *v, const uint16_t *gain, float eps, const float2 *rope,
                                               int pos, int lane) {
    constexpr int EPL = D / 32, HALF = D / 2;
    float ss = 0.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e) ss = fmaf(v[e], v[e], ss);
    const float rinv = 1.0f / sqrtf(warp_sum(ss) / (float)D + eps);
#pragma unroll
    for (int e = 0; e < EPL; ++e) v[e] = v[e] * rinv * bf16_to_f32(gain[lane * EPL + e]);
    const bool lower = lane < 16;
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
        const float other = __shfl_xor_sync(0xffffffffu, v[e], 16);
        const int i = (lane * EPL + e) % HALF;
        const float2 cs = rope[(size_t)pos * HALF + i];
        v[e] = lower ? v[e] * cs.x - other * cs.y : v[e] * cs.x + other * cs.y;
    }
}

template <int D>
__device__ bool mc_attn(MegaRing &R, const MegaArgs &a, const uint16_t *kvl, const MegaSplit &sp, int len,
                        float (*s_state)[D + 4], int *s_last, const uint16_t *qn, const uint16_t *kn) {
    constexpr int EPL = D / 32;
    constexpr uint32_t BLK = kPage * D * 2;
    constexpr int STRIDE = D + 4;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nq = a.group * a.wph;
    int *err = a.ctrl + CTRL_ERR;
    if (!sp.active) return true;
    const int j = w % a.group, set = w / a.group;
    const bool qwarp = w < nq;
    const int head = sp.g * a.group + j;
    float qv[EPL], acc[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) acc[e] = 0.f;
    if (qwarp) {
        if constexpr (EPL == 4) {
            const float4 q4 = __ldcg(reinterpret_cast<const float4 *>(a.q + head * D + lane * 4));
            qv[0] = q4.x; qv[1] = q4.y; qv[2] = q4.z; qv[3] = q4.w;
        } else {
            const float2 q2 = __ldcg(reinterpret_cast<const float2 *>(a.q + head * D + lane * 2));
            qv[0] = q2.x; qv[1] = q2.y;
        }
        if (qn) head_norm_rope<D>(qv, qn, a.eps, a.rope, len - 1, lane);
#pragma unroll
        for (int e = 0; e < EPL; ++e) qv[e] *= a.qscale;
    }
    // this step's K/V row was written by another CTA during the QKV phase, possibly
    // after the producer copied its page: it is read from L2 instead of the ring
    // (with qk_norm the key is finished here from its raw form and written to the page)
    const int cur_slot = (len - 1) % kPage;
    uint32_t kcur[EPL / 2], vcur[EPL / 2];
    if (qwarp && sp.p0 + sp.n == sp.npages) {
        const int page = a.pages[sp.npages - 1];
        uint16_t *kr = const_cast<uint16_t *>(kvl) + (size_t)page * a.page_elems + ((size_t)sp.g * kPage + cur_slot) * D +
                       lane * EPL;
        const uint16_t *vr = kr + (size_t)a.nkv * kPage * D;
        if (kn) {
            float kv_[EPL];
#pragma unroll
            for (int e = 0; e < EPL; ++e) kv_[e] = __ldcg(a.kraw + sp.g * D + lane * EPL + e);
            head_norm_rope<D>(kv_, kn, a.eps, a.rope, len - 1, lane);
#pragma unroll
            for (int e = 0; e < EPL; e += 2)
                kcur[e >> 1] = (uint32_t)f32_to_bf16(kv_[e]) | ((uint32_t)f32_to_bf16(kv_[e + 1]) << 16);
            if (w == 0) {
#pragma unroll
                for (int e = 0; e < EPL; e += 2) reinterpret_cast<uint32_t *>(kr)[e >> 1] = kcur[e >> 1];
            }
            if constexpr (EPL == 4) {
                const uint2 v2 = __ldcg(reinterpret_cast<const uint2 *>(vr));
                vcur[0] = v2.x; vcur[1] = v2.y;
            } else {
                vcur[0] = __ldcg(reinterpret_cast<const unsigned int *>(vr));
            }
        } else if constexpr (EPL == 4) {
            const uint2 k2 = __ldcg(reinterpret_cast<const uint2 *>(kr));
            const uint2 v2 = __ldcg(reinterpret_cast<const uint2 *>(vr));
            kcur[0] = k2.x; kcur[1] = k2.y; vcur[0] = v2.x; vcur[1] = v2.y;
        } else {
            kcur[0] = __ldcg(reinterpret_cast<const unsigned int *>(kr));
            vcur[0] = __ldcg(reinterpret_cast<const unsigned int *>(vr));
        }
    }
    float m = -INFINITY, l = 0.f;
    const int key = lane >> 1;
    bool ok = true;
    for (int i = 0; i < sp.n; ++i) {
        const int slot = R.n % kMegaSlots;
        ok = ok && !*reinterpret_cast<volatile int *>(R.abort) &&
             mbar_wait(R.full0 + 8 * slot, (R.n / kMegaSlots) & 1, err, SITE_MEGA_FULL);
        if (!ok) *R.abort = 1;
        if (ok && qwarp && (i % a.wph) == set) {
            const uint8_t *Ks = R.ring + (size_t)slot * kMegaSlotBytes;
            const uint8_t *Vs = Ks + BLK;
            const int ntok = min(kPage, len - (sp.p0 + i) * kPage);
            const int ct = (sp.p0 + i == sp.npages - 1) ? cur_slot : -1;
            float sc[kPage];
#pragma unroll
            for (int t = 0; t < kPage; ++t) {
                const uint8_t *kr = Ks + (t * D + lane * EPL) * 2;
                if constexpr (EPL == 4) {
                    uint2 kw = *reinterpret_cast<const uint2 *>(kr);
                    if (t == ct) kw = make_uint2(kcur[0], kcur[1]);
                    sc[t] = qv[0] * bf16lo(kw.x) + qv[1] * bf16hi(kw.x) + qv[2] * bf16lo(kw.y) +
                            qv[3] * bf16hi(kw.y);
                } else {
                    uint32_t kw = *reinterpret_cast<const uint32_t *>(kr);
                    if (t == ct) kw = kcur[0];
                    sc[t] = qv[0] * bf16lo(kw) + qv[1] * bf16hi(kw);
                }
            }
#pragma unroll
            for (int o = 16, cnt = kPage; o > 0; o >>= 1) {
                if (cnt > 1) {
                    const bool up = (lane & o) != 0;
#pragma unroll
                    for (int t = 0; t < cnt / 2; ++t) {
                        const float send = up ? sc[t] : sc[t + cnt / 2];
                        const float keep = up ? sc[t + cnt / 2] : sc[t];
                        sc[t] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                    }
                    cnt >>= 1;
                } else {
                    sc[0] += __shfl_xor_sync(0xffffffffu, sc[0], o);
                }
            }
            const float my = key < ntok ? sc[0] : -INFINITY;
            const float mx = fmaxf(m, warp_max(my));
            const float corr = exp2f(m - mx);
            const float pme = exp2f(my - mx);
            l = l * corr + pme;
#pragma unroll
            for (int e = 0; e < EPL; ++e) acc[e] *= corr;
#pragma unroll
            for (int t = 0; t < kPage; ++t) {
                const bool valid = t < ntok;
                const float pt = __shfl_sync(0xffffffffu, pme, 2 * t);
                const uint8_t *vr = Vs + (t * D + lane * EPL) * 2;
                if constexpr (EPL == 4) {
                    uint2 vw = *reinterpret_cast<const uint2 *>(vr);
                    if (t == ct) vw = make_uint2(vcur[0], vcur[1]);
                    if (!valid) vw = make_uint2(0u, 0u);
                    acc[0] = fmaf(pt, bf16lo(vw.x), acc[0]);
                    acc[1] = fmaf(pt, bf16hi(vw.x), acc[1]);
                    acc[2] = fmaf(pt, bf16lo(vw.y), acc[2]);
                    acc[3] = fmaf(pt, bf16hi(vw.y), acc[3]);
                } else {
                    uint32_t vw = *reinterpret_cast<const uint32_t *>(vr);
                    if (t == ct) vw = vcur[0];
                    if (!valid) vw = 0u;
                    acc[0] = fmaf(pt, bf16lo(vw), acc[0]);
                    acc[1] = fmaf(pt, bf16hi(vw), acc[1]);
                }
            }
            m = mx;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(R.empty0 + 8 * slot);
        ++R.n;
    }
    if (consumer_sync_or(!ok)) return false;
    l = warp_sum(l) * 0.5f;
    if (a.wph > 1) {
        if (qwarp) {
#pragma unroll
            for (int e = 0; e < EPL; ++e) s_state[w][lane * EPL + e] = acc[e];
            if (lane == 0) {
                s_state[w][D] = m;
                s_state[w][D + 1] = l;
            }
        }
        consumer_sync();
        if (qwarp && set == 0)
            for (int t = 1; t < a.wph; ++t) {
                const float *o = s_state[t * a.group + j];
                float ob[EPL];
#pragma unroll
                for (int e = 0; e < EPL; ++e) ob[e] = o[lane * EPL + e];
                fd_merge<EPL>(m, l, acc, o[D], o[D + 1], ob);
            }
    }
    const bool writer = qwarp && set == 0;
    if (writer) {
        float *mine = a.part + ((size_t)(sp.g * a.splits + sp.r) * a.group + j) * STRIDE;
        if constexpr (EPL == 4)
            *reinterpret_cast<float4 *>(mine + lane * 4) = make_float4(acc[0], acc[1], acc[2], acc[3]);
        else
            *reinterpret_cast<float2 *>(mine + lane * 2) = make_float2(acc[0], acc[1]);
        if (lane == 0) *reinterpret_cast<float2 *>(mine + D) = make_float2(m, l);
    }
    consumer_sync();
    if (threadIdx.x == 0) {
        __threadfence();
        const int t = atomicAdd(a.ctrl + CTRL_ATTN_TICKET0 + sp.g, 1);
        *s_last = (t == sp.splits - 1);
        if (*s_last) __threadfence();
    }
    consumer_sync();
    if (!*s_last || !writer) return true;

    const float *base = a.part + ((size_t)sp.g * a.splits * a.group + j) * STRIDE;
    const size_t sstride = (size_t)a.group * STRIDE;
    float2 ml = make_float2(-INFINITY, 0.f);
    if (lane < sp.splits) ml = __ldcg(reinterpret_cast<const float2 *>(base + lane * sstride + D));
    const float M = warp_max(ml.x);
    const float f = lane < sp.splits ? exp2f(ml.x - M) : 0.f;
    const float Lsum = warp_sum(ml.y * f);
    float out[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) out[e] = 0.f;
    for (int s0 = 0; s0 < sp.splits; s0 += 8) {
        float v[8][EPL];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int si = min(s0 + u, sp.splits - 1);
            const float *src = base + si * sstride + lane * EPL;
            if constexpr (EPL == 4) {
                const float4 t4 = __ldcg(reinterpret_cast<const float4 *>(src));
                v[u][0] = t4.x; v[u][1] = t4.y; v[u][2] = t4.z; v[u][3] = t4.w;
            } else {
                const float2 t2 = __ldcg(reinterpret_cast<const float2 *>(src));
                v[u][0] = t2.x; v[u][1] = t2.y;
            }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const float fs = __shfl_sync(0xffffffffu, f, (s0 + u) & 31);
            if (s0 + u < sp.splits)
#pragma unroll
                for (int e = 0; e < EPL; ++e) out[e] = fmaf(v[u][e], fs, out[e]);
        }
    }
    const float inv = 1.0f / Lsum;
    if constexpr (EPL == 4)
        *reinterpret_cast<float4 *>(a.o + head * D + lane * 4) =
            make_float4(out[0] * inv, out[1] * inv, out[2] * inv, out[3] * inv);
    else
        *reinterpret_cast<float2 *>(a.o + head * D + lane * 2) = make_float2(out[0] * inv, out[1] * inv);
    if (j == 0 && lane == 0) a.ctrl[CTRL_ATTN_TICKET0 + sp.g] = 0;
    return true;
}

// The SMs do not draw equal HBM bandwidth, and which SMs are slow stays the same
// from step to step, so the GEMV rows are split in proportion to each CTA's
// measured speed instead of evenly.  Run by the consumers of the last CTA of a
// step: the new share of CTA b blends its old share with old share / time of
// its gate/up phases (normalised), half and half, with a floor of a quarter of
// an even share.  Which CTA streams which rows changes no result.
__device__ void mega_rebalance(const MegaArgs &a, float *rate) {
    const int G = gridDim.x, tid = threadIdx.x;
    for (int b = tid; b < G; b += kGemvConsumers) {
        const float share = (float)(__ldcg(a.bound + b + 1) - __ldcg(a.bound + b)) * (1.0f / 16777216.0f);
        const float t = __ldcg(a.cta_time + b);
        rate[b] = t > 0.f ? share / t : 0.f;
        rate[kMegaMaxCtas + b] = share;
    }
    consumer_sync();
    if (tid == 0) {
        float tot = 0.f;
        for (int b = 0; b < G; ++b) tot += rate[b];
        if (tot > 0.f) {
            const float floor_share = 0.25f / (float)G;
            float sum = 0.f;
            for (int b = 0; b < G; ++b) {
                const float ns = fmaxf(0.5f * rate[kMegaMaxCtas + b] + 0.5f * rate[b] / tot, floor_share);
                rate[b] = ns;
                sum += ns;
            }
            float acc = 0.f;
            a.bound[0] = 0;
            for (int b = 1; b < G; ++b) {
                acc += rate[b - 1] / sum;
                a.bound[b] = (uint32_t)fminf(acc * 16777216.0f, 16777216.0f);
            }
            a.bound[G] = 1u << 24;
        }
    }
}

// SH, SF: GEMV shapes of K = hidden and K = ffn for bf16 rows; with Q8 the seven
// per-layer matrices are in the 8-bit block format and stream with the shapes
// QH, QF (16-element chunks, rows per slot sized for the shorter rows), while
// the LM head stays bf16 (SH).
template <int D, class SH, class SF, bool Q8, class QH, class QF>
__global__ void __launch_bounds__(kGemvThreads, 1) decode_step_kernel(const MegaArgs a) {
    using LH = std::conditional_t<Q8, QH, SH>;   // layer matrices with K = hidden (and K = n_q * d)
    using LF = std::conditional_t<Q8, QF, SF>;   // the down projection, K = ffn
    const uint32_t rb_h = Q8 ? (uint32_t)q8_row_bytes((size_t)a.H) : (uint32_t)a.H * 2u;
    const uint32_t rb_q = Q8 ? (uint32_t)q8_row_bytes((size_t)a.qdim) : (uint32_t)a.qdim * 2u;
    const uint32_t rb_f = Q8 ? (uint32_t)q8_row_bytes((size_t)a.F) : (uint32_t)a.F * 2u;
    extern __shared__ __align__(128) uint8_t smem[];
    float *red = reinterpret_cast<float *>(smem);
    __shared__ __align__(8) uint64_t bars[2 * kMegaSlots];
    __shared__ __align__(16) float s_state[kFdMaxQueryWarps][D + 4];
    __shared__ float s_part[2 * kGemvWarps];  // per-warp partials: sums, then maxima (8-bit phases)
    __shared__ float s_bv[kGemvWarps];
    __shared__ int s_bi[kGemvWarps];
    __shared__ int s_flag, s_last, s_abort;
    __shared__ float s_part_rate[2 * kMegaMaxCtas];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int *err = a.ctrl + CTRL_ERR;

    MegaRing R;
    R.full0 = smem_u32(bars);
    R.empty0 = smem_u32(bars + kMegaSlots);
    R.data0 = smem_u32(smem + kGemvRedBytes);
    R.ring = smem + kGemvRedBytes;
    R.n = 0;
    R.abort = &s_abort;
    // the table changes only at the very end of a step, after every CTA read it here
    R.b0 = a.bound[blockIdx.x];
    R.b1 = a.bound[blockIdx.x + 1];
    if (tid == 0) {
        s_abort = 0;
        for (int s = 0; s < kMegaSlots; ++s) {
            mbar_init(R.full0 + 8 * s, 1);
            mbar_init(R.empty0 + 8 * s, kGemvWarps);
        }
        fence_barrier_init();
    }
    __syncthreads();

    // the position only changes at the very end of the step (last LM-head CTA)
    const int len = *reinterpret_cast<volatile int *>(a.ctrl + CTRL_POS) + 1;
    const MegaSplit sp = mega_split(a, len);

    if (warp == kGemvWarps) {  // ------------------------------------ producer
        if (lane == 0) {
            const uint64_t pol = l2_evict_first();
            bool ok = true;
            for (int l = 0; l < a.L && ok; ++l) {
                const size_t lo = (size_t)l * a.lstride;
                ok = mp_rows(R, a.W + a.l0.wqkv + lo, rb_h, a.nqkv / 2, 2, LH::RPS, err, pol) &&
                     mp_pages<D>(R, a, a.KV + (size_t)l * a.kv_layer_elems, sp, err) &&
                     mp_rows(R, a.W + a.l0.wo + lo, rb_q, a.H, 1, LH::RPS, err, pol) &&
                     mp_rows(R, a.W + a.l0.wgu + lo, rb_h, a.F, 2, LH::RPS, err, pol) &&
                     mp_rows(R, a.W + a.l0.wd + lo, rb_f, a.H, 1, LF::RPS, err, pol);
            }
            if (ok) mp_rows(R, a.W + a.w_lm, (uint32_t)a.H * 2u, a.V, 1, SH::RPS, err, pol);
            // no copy may still be landing in shared memory when the CTA exits
            for (int s = max(0, R.n - kMegaSlots); s < R.n; ++s)
                mbar_wait(R.full0 + 8 * (s % kMegaSlots), (s / kMegaSlots) & 1, err, SITE_MEGA_DRAIN);
        }
        return;
    }

    // ---------------------------------------------------------------- consumers
    int k = 0;   // grid barriers passed
    bool ok = true;
    uint64_t gu_ns = 0;   // this CTA's time in the gate/up phases (thread 0's clock)
    for (int l = 0; l < a.L && ok; ++l) {
        const size_t lo = (size_t)l * a.lstride;
        uint16_t *kvl = a.KV + (size_t)l * a.kv_layer_elems;
        if (l > 0) ok = mega_grid_sync(a.ctrl, ++k, &s_flag);
        if (!ok) break;
        EpiQKV eq;
        eq.q = a.q; eq.kv = kvl; eq.pages = a.pages; eq.rope = a.rope; eq.ctrl = a.ctrl;
        eq.bias = a.bias ? a.W + a.l0.bqkv + lo : nullptr;
        eq.kraw = a.kraw;
        eq.qdim = a.qdim; eq.kvdim = a.kvdim; eq.d = a.d; eq.nkv = a.nkv; eq.page_elems = a.page_elems;
        ok = mc_layer_gemv<Q8, LH, kQ8QkvDigits>(R, red, a.H, a.nqkv / 2, 2, a.x, a.W + a.l0.attn_norm + lo,
                                   l == 0 ? a.W + a.w_embed : nullptr, a.x, a.eps, a.ctrl, eq, s_part) &&
             mega_grid_sync(a.ctrl, ++k, &s_flag);
        if (!ok) break;
        // the attention phase leaves the HBM nearly idle: move the first gate/up rows
        // of this CTA into L2 meanwhile (its O rows are already filling the ring)
        if (tid == 0) mp_prefetch(R, a.W + a.l0.wgu + lo, rb_h, a.F, 2, 0, kMegaPrefetchBytes);
        ok = mc_attn<D>(R, a, kvl, sp, len, s_state, &s_last, a.kraw ? a.W + a.l0.qn + lo : nullptr,
                        a.kraw ? a.W + a.l0.kn + lo : nullptr) &&
             mega_grid_sync(a.ctrl, ++k, &s_flag);
        if (!ok) break;
        EpiResidual er{a.x};
        ok = mc_layer_gemv<Q8, LH>(R, red, a.qdim, a.H, 1, a.o, nullptr, nullptr, nullptr, a.eps, a.ctrl, er,
                                   s_part) &&
             mega_grid_sync(a.ctrl, ++k, &s_flag);
        if (!ok) break;
        EpiSwiGLU es{a.m};
        const uint64_t t_gu = globaltimer_ns();
        ok = mc_layer_gemv<Q8, LH>(R, red, a.H, a.F, 2, a.x, a.W + a.l0.ffn_norm + lo, nullptr, nullptr, a.eps,
                                   a.ctrl, es, s_part);
        gu_ns += globaltimer_ns() - t_gu;
        ok = ok && mega_grid_sync(a.ctrl, ++k, &s_flag);
        if (!ok) break;
        ok = mc_layer_gemv<Q8, LF>(R, red, a.F, a.H, 1, a.m, nullptr, nullptr, nullptr, a.eps, a.ctrl, er, s_part);
    }
    if (tid == 0) a.cta_time[blockIdx.x] = (float)gu_ns * 1e-3f;
    if (ok) ok = mega_grid_sync(a.ctrl, ++k, &s_flag);
    if (!ok) return;
    EpiArgmax ea;
    ea.logits = a.logits; ea.partial = a.amax; ea.ctrl = a.ctrl; ea.hist = a.hist; ea.pos_add = 1;
    ea.best = -INFINITY; ea.bidx = 0x7fffffff;
    if (!mc_gemv<SH>(R, red, a.H, a.V, 1, a.x, a.W + a.w_final_norm, nullptr, nullptr, a.eps, a.ctrl, ea, s_part))
        return;
    // CTA argmax, then the last CTA reduces every CTA's result in index order
    float bv = ea.best;
    int bi = ea.bidx;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
    }
    if (lane == 0) { s_bv[warp] = bv; s_bi[warp] = bi; }
    consumer_sync();
    if (tid == 0) {
        for (int w = 1; w < kGemvWarps; ++w)
            if (better(s_bv[w], s_bi[w], bv, bi)) { bv = s_bv[w]; bi = s_bi[w]; }
        a.amax[blockIdx.x] = make_int2(__float_as_int(bv), bi);
        __threadfence();
        const int t = atomicAdd(a.ctrl + CTRL_LM_TICKET, 1);
        if (t == (int)gridDim.x - 1) {
            __threadfence();
            float fv = -INFINITY;
            int fi = 0x7fffffff;
            for (int c = 0; c < (int)gridDim.x; ++c) {
                const int2 pr = __ldcg(a.amax + c);
                const float pv = __int_as_float(pr.x);
                if (better(pv, pr.y, fv, fi)) { fv = pv; fi = pr.y; }
            }
            if (fi == 0x7fffffff) fi = 0;
            const int np = a.ctrl[CTRL_POS] + 1;
            a.ctrl[CTRL_TOKEN] = fi;
            a.ctrl[CTRL_POS] = np;
            a.hist[np] = fi;
            a.ctrl[CTRL_LM_TICKET] = 0;
            // every CTA has passed the last grid barrier (it took a ticket after it):
            // the arrival counter starts the next step at zero without a memset in the
            // stream (a memset would queue behind other streams' copies and kernels)
            a.ctrl[CTRL_GRID_BAR] = 0;
        }
        s_last = (t == (int)gridDim.x - 1);
    }
    consumer_sync();
    if (s_last) mega_rebalance(a, s_part_rate);
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

// query warps per head: at most kFdMaxQueryWarps query warps per CTA
static int fd_wph(int group) { return group >= kFdMaxQueryWarps ? 1 : kFdMaxQueryWarps / group; }

int fd_splits(int max_pages) {
    const int s = (max_pages + 3) / 4;   // about four pages per split at the largest length
    return s < 1 ? 1 : (s > kFdMaxSplits ? kFdMaxSplits : s);
}

size_t fd_part_floats(int nkv, int group, int d, int max_pages) {
    (void)max_pages;   // room for the largest split count of either decode path
    return (size_t)nkv * kFdMaxSplits * group * (d + 4);
}

template <int D>
static cudaError_t launch_fd(const Plan &p, const FDArgs &fa, cudaStream_t st, bool pdl) {
    constexpr uint32_t BLK = kPage * D * 2;
    return launch(flash_decode_kernel<D>, dim3(fd_splits(p.max_pages), p.nkv), dim3(32 * (fa.group * fa.wph + 1)),
                  (size_t)(kFdRingBytes / (2 * BLK)) * 2 * BLK, st, pdl, fa);
}

// the (NCH, RPS, FULL) shapes of every supported K (K % 8 == 0, K <= 16384)
#define WICI_GEMV_SHAPES(X)                                                                     \
    X(1, 8, true) X(1, 8, false) X(2, 4, true) X(2, 4, false) X(3, 2, true) X(3, 2, false)     \
    X(4, 2, true) X(4, 2, false) X(5, 1, true) X(5, 1, false) X(6, 1, true) X(6, 1, false)     \
    X(7, 1, true) X(7, 1, false) X(8, 1, true) X(8, 1, false)

template <class Epi>
static void *gemv_fn(int K) {
    const int nch = gemv_nch(K), rps = gemv_rps(K);
    const bool full = (K / 8) == nch * kGemvConsumers;
#define WICI_PICK(N, R, F) \
    if (nch == N && rps == R && full == F) return (void *)gemv_kernel<N, R, F, Epi>;
    WICI_GEMV_SHAPES(WICI_PICK)
#undef WICI_PICK
    return nullptr;
}

template <class Epi>
static cudaError_t set_gemv_attrs() {
#define WICI_ATTR(N, R, F)                                                                              \
    {                                                                                                   \
        cudaError_t e = cudaFuncSetAttribute(gemv_kernel<N, R, F, Epi>,                                \
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,              \
                                             (int)gemv_smem_bytes(1, kGemvRingBytes));                 \
        if (e != cudaSuccess) return e;                                                                 \
    }
    WICI_GEMV_SHAPES(WICI_ATTR)
#undef WICI_ATTR
    return cudaSuccess;
}

// The instantiated shapes: (head dim, GEMV shape of K = hidden, GEMV shape of K = ffn)
using MegaH4096 = GShape<2, 4, true>;     // Llama-3-8B widths: hidden 4096, ffn 14336
using MegaF14336 = GShape<7, 1, true>;
using MegaH2048 = GShape<1, 8, true>;     // Llama-3.2-1B widths: hidden 2048, ffn 8192
using MegaF8192 = GShape<4, 2, true>;
using MegaH5120 = GShape<3, 2, false>;    // Qwen2.5-14B widths: hidden 5120, ffn 13824
using MegaF13824 = GShape<7, 1, false>;
using MegaSmall = GShape<1, 8, false>;    // hidden and ffn below 2048 (e.g. 256 / 688)
using MegaF12288 = GShape<6, 1, true>;    // Qwen3-8B widths: hidden 4096, ffn 12288
// 8-bit block format: 16-element chunks per thread (NCH = ceil(K / 4096)), and
// rows of q8_row_bytes(K) bytes per 32 KB slot: as many as fit, even where a
// unit is a row pair
using Q8H4096 = GShape<1, 7, true>;       // 7 x 4352 B
using Q8F14336 = GShape<4, 2, false>;     // 2 x 15232 B; 896 chunks
using Q8Small = GShape<1, 8, false>;      // 8 x <= 1904 B (K < 2048)
using Q8F12288 = GShape<3, 2, true>;      // 2 x 13056 B
// (head dim, bf16 shape K = hidden, bf16 shape K = ffn, 8-bit format, its shapes)
#define WICI_MEGA_SHAPES(X)                                       \
    X(128, MegaH4096, MegaF14336, false, MegaH4096, MegaF14336)   \
    X(64, MegaH2048, MegaF8192, false, MegaH2048, MegaF8192)      \
    X(128, MegaH5120, MegaF13824, false, MegaH5120, MegaF13824)   \
    X(64, MegaSmall, MegaSmall, false, MegaSmall, MegaSmall)      \
    X(128, MegaH4096, MegaF12288, false, MegaH4096, MegaF12288)   \
    X(128, MegaH4096, MegaF14336, true, Q8H4096, Q8F14336)        \
    X(128, MegaH4096, MegaF12288, true, Q8H4096, Q8F12288)        \
    X(64, MegaSmall, MegaSmall, true, Q8Small, Q8Small)

cudaError_t setup_kernels() {
    cudaError_t e;
#define WICI_MEGA_ATTR(DD, SH, SF, Q8, QH, QF)                                                        \
    if ((e = cudaFuncSetAttribute(decode_step_kernel<DD, SH, SF, Q8, QH, QF>,                          \
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMegaSmem)) != cudaSuccess) \
        return e;
    WICI_MEGA_SHAPES(WICI_MEGA_ATTR)
#undef WICI_MEGA_ATTR
    if ((e = set_gemv_attrs<EpiResidual>()) != cudaSuccess) return e;
    if ((e = set_gemv_attrs<EpiSwiGLU>()) != cudaSuccess) return e;
    if ((e = set_gemv_attrs<EpiQKV>()) != cudaSuccess) return e;
    if ((e = set_gemv_attrs<EpiArgmax>()) != cudaSuccess) return e;
    return cudaSuccess;
}

// Ring geometry: slots of gemv_rps(K) rows, as many as fit kGemvRingBytes (2 to 8).
static void ring_geometry(GemvIn &g) {
    const int rps = gemv_rps(g.K);
    g.ups = rps / g.rpu;
    g.slot_bytes = ((uint32_t)rps * (uint32_t)g.K * 2u + 127u) & ~127u;
    int st = (int)(kGemvRingBytes / g.slot_bytes);
    g.stages = st < 2 ? 2 : (st > kGemvMaxStages ? kGemvMaxStages : st);
}

template <class Epi>
static cudaError_t launch_gemv(const Plan &p, GemvIn g, Epi epi, cudaStream_t st, bool pdl,
                               LaunchHook *hook, const char *name) {
    ring_geometry(g);
    void *fn = gemv_fn<Epi>(g.K);
    if (!fn || g.ups < 1) return cudaErrorInvalidValue;
    const int grid = p.num_sms * kGemvCtasPerSm;
    if (hook) hook->before(name);
    cudaError_t e = launch(reinterpret_cast<void (*)(const GemvIn, const Epi)>(fn),
                           dim3(grid), dim3(kGemvThreads), gemv_smem_bytes(g.stages, g.slot_bytes), st, pdl,
                           g, epi);
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

// Decode-step GEMVs in launch order: per layer QKV, O, gate/up, down; then the LM head.
enum GemvId : int { G_QKV = 0, G_O = 1, G_GU = 2, G_DOWN = 3, G_LM = 4 };

static void set_next(const Plan &p, const Bufs &b, GemvIn &g, int layer, int id) {
    if (id == G_LM) {
        layer = 0;
        id = G_QKV;        // the next step starts with layer 0
    } else if (id == G_DOWN) {
        if (++layer == p.L) id = G_LM;
        else id = G_QKV;
    } else {
        ++id;
    }
    if (id == G_LM) {
        g.next_W = b.W + p.w_lm; g.next_K = p.H; g.next_n_units = p.V; g.next_rpu = 1;
        return;
    }
    const LayerOffsets &lo = p.layer[layer];
    switch (id) {
        case G_QKV: g.next_W = b.W + lo.wqkv; g.next_K = p.H; g.next_n_units = p.nqkv / 2; g.next_rpu = 2; break;
        case G_O: g.next_W = b.W + lo.wo; g.next_K = p.qdim; g.next_n_units = p.H; g.next_rpu = 1; break;
        case G_GU: g.next_W = b.W + lo.wgu; g.next_K = p.H; g.next_n_units = p.F; g.next_rpu = 2; break;
        default: g.next_W = b.W + lo.wd; g.next_K = p.F; g.next_n_units = p.H; g.next_rpu = 1; break;
    }
}

cudaError_t enqueue_lm_head(const Plan &p, const Bufs &b, cudaStream_t st, bool pdl, int pos_add,
                            LaunchHook *hook) {
    GemvIn g = gemv_in(p, b, b.W + p.w_lm, p.H, p.V, 1, b.x, b.W + p.w_final_norm);
    set_next(p, b, g, p.L - 1, G_LM);   // a decode step (layer 0) follows
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

cudaError_t enqueue_lm_head_argmax_raw(const uint16_t *W, const uint16_t *gain, const float *x, int H, int V,
                                       float eps, float *logits, int *ctrl, int2 *partials, int *hist, int grid,
                                       cudaStream_t st) {
    GemvIn g = {};
    g.W = W;
    g.K = H;
    g.n_units = V;
    g.rpu = 1;
    g.in = x;
    g.gain = gain;
    g.ctrl = ctrl;
    g.eps = eps;
    ring_geometry(g);
    void *fn = gemv_fn<EpiArgmax>(g.K);
    if (!fn || g.ups < 1) return cudaErrorInvalidValue;
    EpiArgmax e = {};
    e.logits = logits;
    e.partial = partials;
    e.ctrl = ctrl;
    e.hist = hist;
    e.pos_add = 0;
    e.best = -INFINITY;
    e.bidx = 0x7fffffff;
    return launch(reinterpret_cast<void (*)(const GemvIn, const EpiArgmax)>(fn), dim3(grid), dim3(kGemvThreads),
                  gemv_smem_bytes(g.stages, g.slot_bytes), st, false, g, e);
}


// ------------------------------------------------------- persistent decode: host
typedef cudaError_t (*MegaLaunch)(const MegaArgs &, int grid, cudaStream_t);

template <int D, class SH, class SF, bool Q8, class QH, class QF>
static cudaError_t launch_mega(const MegaArgs &a, int grid, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kGemvThreads);
    cfg.dynamicSmemBytes = kMegaSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;   // every CTA resident: the grid barriers need it
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decode_step_kernel<D, SH, SF, Q8, QH, QF>, a);
}

template <class S>
static bool shape_is(int K) {
    return gemv_nch(K) == S::NCH && gemv_rps(K) == S::RPS && ((K / 8) == S::NCH * kGemvConsumers) == S::FULL;
}

// 8-bit block rows: 16-element chunks, and S::RPS rows of the format in a slot
template <class S>
static bool q8_shape_is(int K) {
    const int nch = (K / 16 + kGemvConsumers - 1) / kGemvConsumers;
    return nch == S::NCH && ((K / 16) == nch * kGemvConsumers) == S::FULL &&
           (size_t)S::RPS * q8_row_bytes((size_t)K) <= kMegaSlotBytes;
}

static MegaLaunch mega_launcher(const Plan &p) {
    if (p.qdim != p.H || p.nkv > 64 || p.num_sms > kMegaMaxCtas) return nullptr;
    // every layer's tensors must sit at one fixed stride
    if (p.L > 1) {
        const size_t st = p.layer[1].wqkv - p.layer[0].wqkv;
        for (int l = 0; l < p.L; ++l) {
            const LayerOffsets &a = p.layer[l], &b = p.layer[0];
            const size_t o = st * (size_t)l;
            if (a.attn_norm != b.attn_norm + o || a.wqkv != b.wqkv + o || a.wo != b.wo + o ||
                a.ffn_norm != b.ffn_norm + o || a.wgu != b.wgu + o || a.wd != b.wd + o ||
                (p.cfg.qkv_bias && a.bqkv != b.bqkv + o) || (p.qk_norm && (a.qn != b.qn + o || a.kn != b.kn + o)))
                return nullptr;
        }
    }
#define WICI_MEGA_PICK(DD, SH, SF, Q8, QH, QF)                                                       \
    if (p.q8 == Q8 && p.d == DD && shape_is<SH>(p.H) && shape_is<SF>(p.F) &&                            \
        (!Q8 || (q8_shape_is<QH>(p.H) && q8_shape_is<QF>(p.F))))                                        \
        return launch_mega<DD, SH, SF, Q8, QH, QF>;
    WICI_MEGA_SHAPES(WICI_MEGA_PICK)
#undef WICI_MEGA_PICK
    return nullptr;
}

bool decode_is_persistent(const Plan &p) { return mega_launcher(p) != nullptr; }

static cudaError_t enqueue_mega(const Plan &p, const Bufs &b, cudaStream_t st, MegaLaunch fn) {
    MegaArgs a = {};
    a.W = b.W;
    a.kraw = p.qk_norm ? b.kraw : nullptr;
    a.lstride = p.L > 1 ? p.layer[1].wqkv - p.layer[0].wqkv : 0;
    a.l0 = p.layer[0];
    a.w_embed = p.w_embed;
    a.w_final_norm = p.w_final_norm;
    a.w_lm = p.w_lm;
    a.KV = b.KV;
    a.kv_layer_elems = p.kv_layer_elems;
    a.page_elems = p.kv_page_elems;
    a.ctrl = b.ctrl;
    a.hist = b.hist;
    a.x = b.x; a.q = b.q; a.o = b.o; a.m = b.m; a.logits = b.logits;
    a.amax = b.amax;
    a.rope = b.rope;
    a.pages = b.pages;
    a.part = b.fd_part;
    a.bound = b.mega_bound;
    a.cta_time = b.mega_time;
    a.L = p.L; a.H = p.H; a.F = p.F; a.V = p.V;
    a.nqkv = p.nqkv; a.qdim = p.qdim; a.kvdim = p.kvdim; a.d = p.d; a.nkv = p.nkv; a.group = p.group;
    a.wph = fd_wph(p.group);
    const int grid = p.num_sms;
    a.splits = grid / p.nkv < kFdMaxSplits ? grid / p.nkv : kFdMaxSplits;
    a.bias = p.cfg.qkv_bias;
    a.eps = p.cfg.rms_eps;
    a.qscale = 1.4426950408889634f / sqrtf((float)p.d);
    // the grid-barrier counter is zero here: set at create, reset by the last CTA of
    // every step, and by the host after a step that gave up
    return fn(a, grid, st);
}

cudaError_t enqueue_decode_step(const Plan &p, const Bufs &b, cudaStream_t st, bool pdl,
                                LaunchHook *hook) {
    if (MegaLaunch fn = mega_launcher(p)) {
        if (hook) hook->before("decode_step");
        cudaError_t e = enqueue_mega(p, b, st, fn);
        if (hook) hook->after("decode_step");
        return e;
    }
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
        set_next(p, b, g, l, G_QKV);
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
        FDArgs fa = {b.q, kvl, b.pages, b.ctrl, b.o, b.fd_part, p.nkv, p.group, fd_wph(p.group), p.kv_page_elems,
                     qscale};
        if (hook) hook->before("flash_decode");
        if (p.d == 128)
            e = launch_fd<128>(p, fa, st, pdl);
        else
            e = launch_fd<64>(p, fa, st, pdl);
        if (hook) hook->after("flash_decode");
        if (e != cudaSuccess) return e;
        // A6: O projection + residual
        g = gemv_in(p, b, b.W + lo.wo, p.qdim, p.H, 1, b.o, nullptr);
        set_next(p, b, g, l, G_O);
        if ((e = launch_gemv(p, g, EpiResidual{b.x}, st, pdl, hook, "o_proj_residual")) != cudaSuccess)
            return e;
        // A7: RMSNorm + gate/up + SwiGLU
        g = gemv_in(p, b, b.W + lo.wgu, p.H, p.F, 2, b.x, b.W + lo.ffn_norm);
        set_next(p, b, g, l, G_GU);
        if ((e = launch_gemv(p, g, EpiSwiGLU{b.m}, st, pdl, hook, "gate_up_swiglu")) != cudaSuccess)
            return e;
        // A8: down projection + residual
        g = gemv_in(p, b, b.W + lo.wd, p.F, p.H, 1, b.m, nullptr);
        set_next(p, b, g, l, G_DOWN);
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
