// Prefill GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   C[T][N] = (A_hi + A_lo)[T][K] . W[N][K]^T,  fp32 accumulation in TMEM
//
// A is an fp32 activation split into two bf16 terms (hi = bf16(a),
// lo = bf16(a - hi)); W is bf16 and exact.  Both products accumulate into one
// 128x256 fp32 accumulator, giving ~16-bit activation precision on bf16 MMAs
// (the bf16x2 scheme of Henry, Tang & Heinecke, ARITH 2019, on one operand).
//
// One CTA computes one 128x256 output tile with three warp roles:
//   warp 0      TMA producer: 2-D tiled loads (128-byte swizzle) of A_hi, A_lo
//               and W k-blocks into a 3-stage shared-memory ring;
//   warp 1      allocates 256 TMEM columns and issues tcgen05.mma (one thread);
//               each stage is released by tcgen05.commit to its "empty" barrier;
//   warps 2..5  epilogue: tcgen05.ld of their 32 TMEM lanes (one output row per
//               thread) and the fused epilogue functor on column pairs.
// Every mbarrier wait is bounded; a wait that gives up records its site in
// *err and the CTA still drains its copies, frees TMEM and exits.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace wici {

constexpr int TC_BM = 128, TC_BN = 256, TC_BK = 64, TC_STAGES = 3, TC_THREADS = 192;
constexpr uint32_t TC_A_BYTES = TC_BM * TC_BK * 2;                 // 16 KB
constexpr uint32_t TC_B_BYTES = TC_BN * TC_BK * 2;                 // 32 KB
constexpr uint32_t TC_STAGE_BYTES = 2 * TC_A_BYTES + TC_B_BYTES;   // 64 KB
constexpr size_t TC_SMEM = (size_t)TC_STAGES * TC_STAGE_BYTES + 1024;
constexpr uint32_t TC_TMEM_COLS = 256;

enum : int { SITE_TC_EMPTY = 21, SITE_TC_FULL = 22, SITE_TC_ACCUM = 23, SITE_TC_DRAIN = 24 };

// instruction descriptor of tcgen05.mma.kind::f16: D fp32, A and B bf16, both
// K-major, M = 128, N = 256
__host__ __device__ constexpr uint32_t tc_idesc() {
    return (1u << 4)                      // D format: f32
           | (1u << 7)                    // A format: bf16
           | (1u << 10)                   // B format: bf16
           | ((uint32_t)(TC_BN >> 3) << 17)
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

// Epi::pair(t, c, v0, v1): output row t, columns (c, c + 1)
template <class Epi>
__global__ void __launch_bounds__(TC_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap map_ahi, const __grid_constant__ CUtensorMap map_alo,
                   const __grid_constant__ CUtensorMap map_w, int T, int N, int K, int *err, const Epi epi) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[TC_STAGES], empty_bar[TC_STAGES], accum_bar;
    __shared__ uint32_t s_tmem;
    __shared__ int s_issued;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n0 = blockIdx.x * TC_BN, m0 = blockIdx.y * TC_BM;
    const int nk = (K + TC_BK - 1) / TC_BK;
    const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;

    if (threadIdx.x == 0) {
        for (int s = 0; s < TC_STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        mbar_init(smem_u32(&accum_bar), 1);
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
            int issued = 0;
            for (int kb = 0; kb < nk; ++kb) {
                const int s = kb % TC_STAGES;
                if (kb >= TC_STAGES &&
                    !mbar_wait(smem_u32(&empty_bar[s]), ((kb / TC_STAGES) + 1) & 1, err, SITE_TC_EMPTY))
                    break;
                const uint32_t st = base + (uint32_t)s * TC_STAGE_BYTES;
                const uint32_t fb = smem_u32(&full_bar[s]);
                mbar_arrive_expect_tx(fb, TC_STAGE_BYTES);
                tma_load_2d(st, &map_ahi, kb * TC_BK, m0, fb);
                tma_load_2d(st + TC_A_BYTES, &map_alo, kb * TC_BK, m0, fb);
                tma_load_2d(st + 2 * TC_A_BYTES, &map_w, kb * TC_BK, n0, fb);
                issued = kb + 1;
            }
            s_issued = issued;
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ------------------------------------------- MMA issuer
            constexpr uint32_t idesc = tc_idesc();
            bool ok = true;
            for (int kb = 0; kb < nk && ok; ++kb) {
                const int s = kb % TC_STAGES;
                ok = mbar_wait(smem_u32(&full_bar[s]), (kb / TC_STAGES) & 1, err, SITE_TC_FULL);
                if (!ok) break;
                tc_fence_after();
                const uint32_t st = base + (uint32_t)s * TC_STAGE_BYTES;
#pragma unroll
                for (int k = 0; k < TC_BK / 16; ++k) {
                    const uint64_t bd = tc_desc_sw128(st + 2 * TC_A_BYTES + 32 * k);
                    tc_mma(tmem, tc_desc_sw128(st + 32 * k), bd, idesc, (kb | k) != 0);
                    tc_mma(tmem, tc_desc_sw128(st + TC_A_BYTES + 32 * k), bd, idesc, 1);
                }
                tc_commit(smem_u32(&empty_bar[s]));
            }
            tc_commit(smem_u32(&accum_bar));  // fires when every MMA issued above has completed
        }
    } else {  // ------------------------------------------------------- epilogue
        const bool ok = mbar_wait(smem_u32(&accum_bar), 0, err, SITE_TC_ACCUM);
        tc_fence_after();
        const int q = warp & 3;                 // TMEM lane quadrant of this warp
        const int t = m0 + q * 32 + lane;
        for (int c0 = 0; c0 < TC_BN; c0 += 32) {
            float v[32];
            tc_ld32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, v);
            if (ok && t < T) {
#pragma unroll
                for (int j = 0; j < 32; j += 2) {
                    const int c = n0 + c0 + j;
                    if (c < N) epi.pair(t, c, v[j], v[j + 1]);
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
        for (int kb = issued - TC_STAGES < 0 ? 0 : issued - TC_STAGES; kb < issued; ++kb)
            mbar_wait(smem_u32(&full_bar[kb % TC_STAGES]), (kb / TC_STAGES) & 1, err, SITE_TC_DRAIN);
    }
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TC_TMEM_COLS)
                     : "memory");
    }
}

}  // namespace wici
