// Prefill GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   C[T][N] = (A_0 + A_1 + A_2)[T][K] . W[N][K]^T,  fp32 accumulation in TMEM
//
// A is an fp32 activation carried as kTerms = 3 bf16 terms (split_bf16x3); W is
// bf16 and exact.  The three products accumulate into one fp32 TMEM
// accumulator, so the activations keep fp32 precision on bf16 MMAs (the bf16x3
// scheme of Henry, Tang & Heinecke, ARITH 2019, applied to one operand).
//
// Accumulation: one tcgen05 accumulator that absorbs the whole K dimension adds
// each MMA's result with the tensor core's internal alignment, and over K/16
// k-steps x 3 terms that error grows well past fp32 summation (measured: 4x the
// logits error of the fp32 CUDA-core path at the Llama-3-8B shape).  So the MMAs
// accumulate only TC_GROUP k-blocks into one of two TMEM buffers; the epilogue
// warps fold each finished group into fp32 registers (round-to-nearest adds)
// while the next group accumulates into the other buffer.
//
// Weights in the 8-bit block format arrive dequantised as WT = 3 bf16 terms
// W = W_0 + W_1 + W_2 (exact: a code times an fp16 scale has at most 18
// significant bits).  The K loop then runs once per weight term j < AT, issuing
// the products A_i W_j with i + j < AT, AT the activation terms of the GEMM:
// with AT = 3 that is 3 + 2 + 1 MMAs per k-step (the dropped products lie below
// 2^-24 of the result); with AT = 2 it is 2 + 1, the weight then carried at the
// activations' own 16 significant bits.
//
// Persistent: one CTA per SM walks the output tiles (M tiles fastest, so the
// CTAs that run together share a weight tile through L2) with three warp roles:
//   warp 0      TMA producer: 2-D tiled loads (128-byte swizzle) of the three A
//               terms and the W k-block into a shared-memory ring;
//   warp 1      allocates 512 TMEM columns and issues tcgen05.mma (one thread);
//               each stage is released by tcgen05.commit to its "empty" barrier;
//   warps 2..9  tcgen05.ld of one TMEM lane quadrant and half of the tile's
//               columns each (one output row per thread), group sums in
//               registers, then the fused epilogue on column pairs.  The
//               epilogue of one tile overlaps the MMAs of the next.
// Every mbarrier wait is bounded; a wait that gives up records its site in
// *err and the CTA still drains its copies, frees TMEM and exits.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace wici {

constexpr int TC_BM = 128, TC_BK = 64, TC_THREADS = 320, TC_EPI_WARPS = 8;
constexpr int TC_GROUP = 4;                                             // k-blocks per TMEM accumulation
constexpr uint32_t TC_A_BYTES = TC_BM * TC_BK * 2;                      // 16 KB per term
constexpr uint32_t TC_TMEM_COLS = 512;                                  // two accumulator buffers
constexpr size_t TC_SMEM_BUDGET = 216 * 1024;                           // ring bytes

// geometry of a 128 x BN output tile whose stages hold AT activation terms
template <int BN, int AT = kTerms>
struct TcTile {
    static_assert(BN % 32 == 0 && BN <= 256, "BN: a multiple of 32 up to 256");
    static constexpr uint32_t B_BYTES = BN * TC_BK * 2;
    static constexpr uint32_t STAGE_BYTES = AT * TC_A_BYTES + B_BYTES;
    static constexpr int STAGES = (int)(TC_SMEM_BUDGET / STAGE_BYTES);
    static constexpr size_t SMEM = (size_t)STAGES * STAGE_BYTES + 1024;
    static constexpr int EPI_COLS = BN / 2;                               // columns per epilogue warp
    static constexpr uint32_t ACC_STRIDE = TC_TMEM_COLS / 2;              // TMEM columns between the two buffers
    static_assert(STAGES >= 3, "at least three ring stages");
};

enum : int { SITE_TC_EMPTY = 21, SITE_TC_FULL = 22, SITE_TC_ACCUM = 23, SITE_TC_DRAIN = 24, SITE_TC_FREE = 25 };

// instruction descriptor of tcgen05.mma.kind::f16: D fp32, A and B bf16, both
// K-major, M = 128, N = n
__host__ __device__ constexpr uint32_t tc_idesc(int n) {
    return (1u << 4)                      // D format: f32
           | (1u << 7)                    // A format: bf16
           | (1u << 10)                   // B format: bf16
           | ((uint32_t)(n >> 3) << 17)
           | ((uint32_t)(TC_BM >> 4) << 24);
}

// shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row groups 1024 bytes apart
__device__ __forceinline__ uint64_t tc_desc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);   // start address
    d |= (uint64_t)1 << 16;                     // leading byte offset (unused with this swizzle)
    d |= (uint64_t)(1024 >> 4) << 32;           // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1 << 46;                     // descriptor version for tcgen05
    d |= (uint64_t)2 << 61;                     // swizzle mode: 128 B
    return d;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tc_mma(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// 16 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void tc_ld16(uint32_t taddr, float *v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// 32 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void tc_ld32(uint32_t taddr, float *v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Epi::pair(t, c, v0, v1): output row t, columns (c, c + 1); Epi::row (when
// Epi::kRow): the thread's whole span of columns at once, with vector stores
template <int BN, int WT, class Epi>
__global__ void __launch_bounds__(TC_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap map_a0, const __grid_constant__ CUtensorMap map_a1,
                   const __grid_constant__ CUtensorMap map_a2, const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_w1, const __grid_constant__ CUtensorMap map_w2, int T,
                   int N, int K, int *err, const Epi epi) {
    static_assert(WT == 1 || WT == kTerms, "one exact bf16 weight term, or three");
    constexpr int AT = Epi::kATerms;   // activation terms multiplied (and loaded)
    static_assert(AT >= 1 && AT <= kTerms, "activation terms");
    using G = TcTile<BN, AT>;
    constexpr int S = G::STAGES;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[S], empty_bar[S], acc_full[2], acc_free[2];
    __shared__ uint32_t s_tmem;
    __shared__ int s_issued;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntm = (T + TC_BM - 1) / TC_BM, ntn = (N + BN - 1) / BN;
    const int ntiles = ntm * ntn;
    const int nk = (K + TC_BK - 1) / TC_BK;
    constexpr int WU = WT == 1 ? 1 : Epi::kATerms;  // weight terms used
    const int nkk = nk * WU;                      // k-blocks of all weight terms
    const int ngroups = (nkk + TC_GROUP - 1) / TC_GROUP;
    const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_free[b]), TC_EPI_WARPS);
        }
        fence_barrier_init();
        s_issued = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                     "r"(TC_TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;

    if (warp == 0) {
        if (lane == 0) {  // ------------------------------------------- TMA producer
            int it = 0;   // k-blocks issued over all tiles
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
                const int m0 = (tile % ntm) * TC_BM, n0 = (tile / ntm) * BN;
                for (int kk = 0; kk < nkk; ++kk, ++it) {
                    const int s = it % S;
                    if (it >= S && !(ok = mbar_wait(smem_u32(&empty_bar[s]), ((it / S) + 1) & 1, err, SITE_TC_EMPTY)))
                        break;
                    const int j = WT == 1 ? 0 : kk / nk, kb = kk - j * nk;     // weight term, k-block
                    const uint32_t st = base + (uint32_t)s * G::STAGE_BYTES;
                    const uint32_t fb = smem_u32(&full_bar[s]);
                    // term j meets the activation terms i <= 2 - j only
                    const int na = AT - j;
                    mbar_arrive_expect_tx(fb, (uint32_t)na * TC_A_BYTES + G::B_BYTES);
                    tma_load_2d(st, &map_a0, kb * TC_BK, m0, fb);
                    if (na > 1) tma_load_2d(st + TC_A_BYTES, &map_a1, kb * TC_BK, m0, fb);
                    if (na > 2) tma_load_2d(st + 2 * TC_A_BYTES, &map_a2, kb * TC_BK, m0, fb);
                    tma_load_2d(st + AT * TC_A_BYTES, j == 0 ? &map_w : j == 1 ? &map_w1 : &map_w2, kb * TC_BK, n0,
                                fb);
                    s_issued = it + 1;
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ------------------------------------------- MMA issuer
            constexpr uint32_t idesc = tc_idesc(BN);
            bool ok = true;
            int it = 0, gg = 0;   // k-blocks and groups consumed over all tiles
            for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
                for (int gi = 0; gi < ngroups && ok; ++gi, ++gg) {
                    const int b = gg & 1;
                    // the epilogue must have read this buffer's previous group
                    if (gg >= 2 && !(ok = mbar_wait(smem_u32(&acc_free[b]), ((gg / 2) + 1) & 1, err, SITE_TC_FREE)))
                        break;
                    tc_fence_after();
                    const uint32_t acc = tmem + (uint32_t)b * G::ACC_STRIDE;
                    const int kk1 = min(nkk, (gi + 1) * TC_GROUP);
                    for (int kk = gi * TC_GROUP; kk < kk1; ++kk, ++it) {
                        const int s = it % S;
                        ok = mbar_wait(smem_u32(&full_bar[s]), (it / S) & 1, err, SITE_TC_FULL);
                        if (!ok) break;
                        tc_fence_after();
                        const int nt = WT == 1 ? AT : AT - kk / nk;   // activation terms meeting this weight term
                        const uint32_t st = base + (uint32_t)s * G::STAGE_BYTES;
                        // descriptors of k-step 0; each k-step of 16 elements is 32 bytes further
                        const uint64_t bd0 = tc_desc_sw128(st + AT * TC_A_BYTES);
                        const uint64_t ad0 = tc_desc_sw128(st);
#pragma unroll
                        for (int k = 0; k < TC_BK / 16; ++k)
#pragma unroll
                            for (int t = 0; t < kTerms; ++t)
                                if (t < nt)
                                    tc_mma(acc, ad0 + (uint64_t)((t * TC_A_BYTES + 32 * k) >> 4),
                                           bd0 + (uint64_t)(2 * k), idesc, (kk != gi * TC_GROUP || k != 0 || t != 0));
                        tc_commit(smem_u32(&empty_bar[s]));
                    }
                    tc_commit(smem_u32(&acc_full[b]));  // fires when this group's MMAs have completed
                }
            }
        }
    } else {  // ------------------------------------------------------- epilogue
        const int q = warp & 3;                          // TMEM lane quadrant of this warp
        const int half = (warp - 2) >> 2;                // which half of the tile's columns
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        bool ok = true;
        int gg = 0;
        for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
            const int m0 = (tile % ntm) * TC_BM, n0 = (tile / ntm) * BN;
            const int t = m0 + q * 32 + lane;
            float sum[G::EPI_COLS];
#pragma unroll
            for (int c = 0; c < G::EPI_COLS; ++c) sum[c] = 0.f;
            for (int gi = 0; gi < ngroups; ++gi, ++gg) {
                const int b = gg & 1;
                ok = mbar_wait(smem_u32(&acc_full[b]), (gg / 2) & 1, err, SITE_TC_ACCUM);
                if (!ok) break;
                tc_fence_after();
                const uint32_t ta = tmem + lane_base + (uint32_t)b * G::ACC_STRIDE + (uint32_t)(half * G::EPI_COLS);
#pragma unroll
                for (int c0 = 0; c0 + 32 <= G::EPI_COLS; c0 += 32) {
                    float v[32];
                    tc_ld32(ta + (uint32_t)c0, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) sum[c0 + i] += v[i];
                }
                if constexpr (G::EPI_COLS % 32 != 0) {   // a last 16 columns
                    constexpr int c0 = G::EPI_COLS - 16;
                    float v[16];
                    tc_ld16(ta + (uint32_t)c0, v);
#pragma unroll
                    for (int i = 0; i < 16; ++i) sum[c0 + i] += v[i];
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&acc_free[b]));
            }
            if (ok && t < T) {
                const int c0 = n0 + half * G::EPI_COLS;
                if constexpr (Epi::kRow) {
                    epi.row(t, c0, sum, N - c0);
                } else {
#pragma unroll
                    for (int j = 0; j < G::EPI_COLS; j += 2)
                        if (c0 + j < N) epi.pair(t, c0 + j, sum[j], sum[j + 1]);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0 && lane == 0) {
        // nothing may still land in shared memory after exit (all stages were
        // consumed on the normal path; this only matters after a wait gave up)
        const int issued = s_issued;
        for (int kb = issued - S < 0 ? 0 : issued - S; kb < issued; ++kb)
            mbar_wait(smem_u32(&full_bar[kb % S]), (kb / S) & 1, err, SITE_TC_DRAIN);
    }
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TC_TMEM_COLS)
                     : "memory");
    }
}

}  // namespace wici
