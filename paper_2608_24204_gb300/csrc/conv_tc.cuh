// One 3x3, stride-2, padding-1 convolution layer on the tensor cores, forward
// and both gradients of backpropagation, as implicit GEMMs (the paper's second
// evaluated application, NVIDIA's CNN-training sample, Sec. 5.4).  Channels
// last: x [N][H][W][C], w [K][3][3][C], y and dy [N][P][Q][K], P = H/2, Q = W/2,
// all bf16 except the fp32 outputs.  bf16 operands are exact, products are
// exact, and each output accumulates in fp32 in TMEM over its whole reduction.
//
//   forward    y[pix][k]  = sum_{tap, c} X_tap[pix][c] w[k][tap][c]
//              M = output pixels (tiles of 8 rows x 16 columns), N = K, reduction
//              9 taps x C.  X_tap is x at (2p + r - 1, 2q + s - 1): one TMA box
//              with element strides 2 in h and w, zero outside the image.
//   data grad  dx[h][v][c] = sum dy[p][q][k] w[k][r][s][c] over 2p + r - 1 = h,
//              2q + s - 1 = v.  The output pixels split into four parity classes
//              (h even/odd x v even/odd); in each, a tap (r, s) reads dy at a
//              fixed offset (p = i + (ph + 1 - r) / 2 for h = 2i + ph), so every
//              class is a plain implicit GEMM over its 1, 2, 2 or 4 taps with the
//              filter transposed to [tap][c][k] (K-major B).
//   filter grad dw[k][tap][c] = sum_pix dy[pix][k] X_tap[pix][c]: per tap a GEMM
//              M = K, N = C, reduction over the N P Q pixels in blocks of 64
//              (4 output rows x 16 columns).  Both operands are pixel-by-channel
//              tiles, i.e. MN-major for tcgen05.
//
// Persistent, one CTA per SM, three warp roles as in the prefill GEMM: warp 0
// issues the TMA loads into a 4-stage ring (16 KB A + 32 KB B a stage), warp 1
// allocates 512 TMEM columns (two 256-column accumulators) and issues
// tcgen05.mma, warps 2..9 read a finished accumulator (lane quadrant x column
// half) and store fp32 rows while the next tile accumulates.  Waits are bounded.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "gemm_tc.cuh"

namespace wici {

enum ConvMode : int { CONV_FWD = 0, CONV_DGRAD = 1, CONV_WGRAD = 2 };

constexpr int CV_BM = 128, CV_BN = 256, CV_BK = 64, CV_STAGES = 4, CV_THREADS = 320;
constexpr uint32_t CV_A_BYTES = CV_BM * CV_BK * 2;        // 16 KB
constexpr uint32_t CV_B_BYTES = CV_BN * CV_BK * 2;        // 32 KB
constexpr uint32_t CV_STAGE_BYTES = CV_A_BYTES + CV_B_BYTES;
constexpr size_t CV_SMEM = (size_t)CV_STAGES * CV_STAGE_BYTES + 1024;
constexpr uint32_t CV_BOX_BYTES = 64 * 64 * 2;            // one 64-pixel x 64-channel box (filter grad)

enum : int { SITE_CV_EMPTY = 71, SITE_CV_FULL = 72, SITE_CV_ACCUM = 73, SITE_CV_FREE = 74, SITE_CV_DRAIN = 75 };

struct ConvArgs {
    int n, c, h, w, k, p, q;
    int pt, qt;          // output-row tiles (8 rows) and column tiles (16 columns)
    int ntiles;
    float *out;          // y [N][P][Q][K], dx [N][H][W][C] or dw [K][3][3][C]
    int *err;
};

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, int c0, int c1, int c2, int c3,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], "
        "[%6];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

// MN-major operand, 128-byte swizzle: rows are reduction indices (pixels) of 64
// consecutive M/N values; 8-row groups 1024 B apart, the next 64 values `lbo` further
__device__ __forceinline__ uint64_t cv_desc_mn(uint32_t saddr, uint32_t lbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// kind::f16: D fp32, A and B bf16, M = 128, N = 256; MN-major A and B when mn
__host__ __device__ constexpr uint32_t cv_idesc(bool mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((mn ? 1u : 0u) << 15) | ((mn ? 1u : 0u) << 16) |
           ((uint32_t)(CV_BN >> 3) << 17) | ((uint32_t)(CV_BM >> 4) << 24);
}

// the data-gradient parity classes, heaviest first: (ph, pw) and their tap count
__device__ __forceinline__ void cv_class(int cls, int &ph, int &pw) {
    ph = cls == 0 || cls == 1 ? 1 : 0;     // classes: (1,1) 4 taps, (1,0) 2, (0,1) 2, (0,0) 1
    pw = cls == 0 || cls == 2 ? 1 : 0;
}
__device__ __forceinline__ int cv_ntaps_1d(int ph) { return ph ? 2 : 1; }
// i-th tap index along one axis of a class: even phase -> r = 1; odd -> r = 0, 2
__device__ __forceinline__ int cv_tap_1d(int ph, int i) { return ph ? 2 * i : 1; }

// tile -> (mode-specific) coordinates; the reduction length in 64-wide blocks
struct CvTile {
    int n, p0, q0, nt;     // forward / data grad: image, first output row / column, N tile
    int cls, ph, pw;       // data grad
    int tap, mt;           // filter grad: tap, M (k) tile
    int nkb;               // reduction blocks
};

template <int MODE>
__device__ __forceinline__ CvTile cv_tile(const ConvArgs &a, int t) {
    CvTile s = {};
    if constexpr (MODE == CONV_FWD) {
        const int ntn = a.k / CV_BN;
        s.nt = t % ntn;
        int m = t / ntn;
        s.q0 = (m % a.qt) * 16;
        m /= a.qt;
        s.p0 = (m % a.pt) * 8;
        s.n = m / a.pt;
        s.nkb = 9 * (a.c / CV_BK);
    } else if constexpr (MODE == CONV_DGRAD) {
        const int ntn = a.c / CV_BN, per_class = a.n * a.pt * a.qt * ntn;
        s.cls = t / per_class;
        int m = t % per_class;
        s.nt = m % ntn;
        m /= ntn;
        s.q0 = (m % a.qt) * 16;
        m /= a.qt;
        s.p0 = (m % a.pt) * 8;
        s.n = m / a.pt;
        cv_class(s.cls, s.ph, s.pw);
        s.nkb = cv_ntaps_1d(s.ph) * cv_ntaps_1d(s.pw) * (a.k / CV_BK);
    } else {
        const int ntn = a.c / CV_BN, ntm = a.k / CV_BM;
        s.nt = t % ntn;
        s.mt = (t / ntn) % ntm;
        s.tap = t / (ntn * ntm);
        s.nkb = a.n * ((a.p + 3) / 4) * a.qt;
    }
    return s;
}

// TMA loads of reduction block kb of a tile into stage buffers (A at sa, B at sb)
template <int MODE>
__device__ __forceinline__ void cv_load(const ConvArgs &a, const CvTile &s, int kb, const CUtensorMap *ma,
                                        const CUtensorMap *mb, uint32_t sa, uint32_t sb, uint32_t bar) {
    if constexpr (MODE == CONV_FWD) {
        const int cbs = a.c / CV_BK, tap = kb / cbs, c0 = (kb % cbs) * CV_BK, r = tap / 3, ss = tap % 3;
        // x at rows 2p + r - 1, columns 2q + s - 1 (element strides 2): 8 x 16 pixels x 64 channels
        tma_load_4d(sa, ma, c0, 2 * s.q0 + ss - 1, 2 * s.p0 + r - 1, s.n, bar);
        tma_load_2d(sb, mb, tap * a.c + c0, s.nt * CV_BN, bar);                 // w[k][tap][c]
    } else if constexpr (MODE == CONV_DGRAD) {
        const int kbs = a.k / CV_BK, ti = kb / kbs, k0 = (kb % kbs) * CV_BK;
        const int nts = cv_ntaps_1d(s.pw);
        const int r = cv_tap_1d(s.ph, ti / nts), ss = cv_tap_1d(s.pw, ti % nts);
        const int dp = (s.ph + 1 - r) / 2, dq = (s.pw + 1 - ss) / 2;
        tma_load_4d(sa, ma, k0, s.q0 + dq, s.p0 + dp, s.n, bar);              // dy at (i + dp, j + dq)
        tma_load_2d(sb, mb, k0, (r * 3 + ss) * a.c + s.nt * CV_BN, bar);       // w^T[tap][c][k]
    } else {
        const int pbs = (a.p + 3) / 4, pb = kb % (pbs * a.qt);
        const int n = kb / (pbs * a.qt), p0 = (pb / a.qt) * 4, q0 = (pb % a.qt) * 16;
        const int r = s.tap / 3, ss = s.tap % 3;
        // A: dy pixels x 128 channels k (two 64-channel boxes); B: x pixels x 256 channels c
#pragma unroll
        for (int i = 0; i < CV_BM / 64; ++i) tma_load_4d(sa + i * CV_BOX_BYTES, ma, s.mt * CV_BM + 64 * i, q0, p0, n, bar);
#pragma unroll
        for (int i = 0; i < CV_BN / 64; ++i)
            tma_load_4d(sb + i * CV_BOX_BYTES, mb, s.nt * CV_BN + 64 * i, 2 * q0 + ss - 1, 2 * p0 + r - 1, n, bar);
    }
}

template <int MODE>
__global__ void __launch_bounds__(CV_THREADS, 1)
    conv_tc_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                   const ConvArgs a) {
    constexpr bool MN = MODE == CONV_WGRAD;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[CV_STAGES], empty_bar[CV_STAGES], acc_full[2], acc_free[2];
    __shared__ uint32_t s_tmem;
    __shared__ int s_issued;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;

    if (threadIdx.x == 0) {
        for (int s = 0; s < CV_STAGES; ++s) {
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
                     "r"(512)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;

    if (warp == 0) {
        if (lane == 0) {  // ------------------------------------------- TMA producer
            int it = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < a.ntiles && ok; t += gridDim.x) {
                const CvTile s = cv_tile<MODE>(a, t);
                for (int kb = 0; kb < s.nkb; ++kb, ++it) {
                    const int st = it % CV_STAGES;
                    if (it >= CV_STAGES &&
                        !(ok = mbar_wait(smem_u32(&empty_bar[st]), ((it / CV_STAGES) + 1) & 1, a.err, SITE_CV_EMPTY)))
                        break;
                    const uint32_t sa = base + (uint32_t)st * CV_STAGE_BYTES;
                    const uint32_t fb = smem_u32(&full_bar[st]);
                    mbar_arrive_expect_tx(fb, CV_STAGE_BYTES);
                    cv_load<MODE>(a, s, kb, &map_a, &map_b, sa, sa + CV_A_BYTES, fb);
                    s_issued = it + 1;
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ------------------------------------------- MMA issuer
            constexpr uint32_t idesc = cv_idesc(MN);
            bool ok = true;
            int it = 0, tt = 0;
            for (int t = blockIdx.x; t < a.ntiles && ok; t += gridDim.x, ++tt) {
                const CvTile s = cv_tile<MODE>(a, t);
                const int b = tt & 1;
                if (tt >= 2 && !(ok = mbar_wait(smem_u32(&acc_free[b]), ((tt / 2) + 1) & 1, a.err, SITE_CV_FREE)))
                    break;
                tc_fence_after();
                const uint32_t acc = tmem + (uint32_t)(b * CV_BN);
                for (int kb = 0; kb < s.nkb; ++kb, ++it) {
                    const int st = it % CV_STAGES;
                    ok = mbar_wait(smem_u32(&full_bar[st]), (it / CV_STAGES) & 1, a.err, SITE_CV_FULL);
                    if (!ok) break;
                    tc_fence_after();
                    const uint32_t sa = base + (uint32_t)st * CV_STAGE_BYTES, sb = sa + CV_A_BYTES;
#pragma unroll
                    for (int k = 0; k < CV_BK / 16; ++k) {
                        uint64_t ad, bd;
                        if constexpr (MN) {   // 16 pixels = 16 rows of 128 B further
                            ad = cv_desc_mn(sa + 2048u * k, CV_BOX_BYTES);
                            bd = cv_desc_mn(sb + 2048u * k, CV_BOX_BYTES);
                        } else {              // 16 channels = 32 B further inside the swizzled rows
                            ad = tc_desc_sw128(sa + 32u * k);
                            bd = tc_desc_sw128(sb + 32u * k);
                        }
                        tc_mma(acc, ad, bd, idesc, (kb | k) != 0);
                    }
                    tc_commit(smem_u32(&empty_bar[st]));
                }
                if (!ok) break;
                tc_commit(smem_u32(&acc_full[b]));
            }
        }
    } else {  // ------------------------------------------------------- epilogue
        const int qd = warp & 3, half = (warp - 2) >> 2;
        const int m = qd * 32 + lane;                   // tile row = TMEM lane
        const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
        int tt = 0;
        for (int t = blockIdx.x; t < a.ntiles; t += gridDim.x, ++tt) {
            const CvTile s = cv_tile<MODE>(a, t);
            const int b = tt & 1;
            if (!mbar_wait(smem_u32(&acc_full[b]), (tt / 2) & 1, a.err, SITE_CV_ACCUM)) break;
            tc_fence_after();
            float *row = nullptr;     // this thread's output row, columns from the tile's first
            if constexpr (MODE == CONV_FWD) {
                const int p = s.p0 + m / 16, q = s.q0 + m % 16;
                if (p < a.p && q < a.q) row = a.out + (((size_t)s.n * a.p + p) * a.q + q) * a.k + s.nt * CV_BN;
            } else if constexpr (MODE == CONV_DGRAD) {
                const int i = s.p0 + m / 16, j = s.q0 + m % 16;
                if (i < a.p && j < a.q)
                    row = a.out + (((size_t)s.n * a.h + 2 * i + s.ph) * a.w + 2 * j + s.pw) * a.c + s.nt * CV_BN;
            } else {
                row = a.out + ((size_t)(s.mt * CV_BM + m) * 9 + s.tap) * a.c + s.nt * CV_BN;
            }
#pragma unroll
            for (int c0 = 0; c0 < CV_BN / 2; c0 += 32) {
                float v[32];
                tc_ld32(tmem + lane_base + (uint32_t)(b * CV_BN + half * (CV_BN / 2) + c0), v);
                if (row) {
                    float4 *dst = reinterpret_cast<float4 *>(row + half * (CV_BN / 2) + c0);
#pragma unroll
                    for (int i = 0; i < 8; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&acc_free[b]));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0 && lane == 0) {
        const int issued = s_issued;
        for (int kb = issued - CV_STAGES < 0 ? 0 : issued - CV_STAGES; kb < issued; ++kb)
            mbar_wait(smem_u32(&full_bar[kb % CV_STAGES]), (kb / CV_STAGES) & 1, a.err, SITE_CV_DRAIN);
    }
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(512) : "memory");
    }
}

// w [K][9][C] -> w^T [9][C][K] (the data gradient's K-major B operand), 32 x 32 tiles
__global__ void conv_transpose_filter_kernel(const uint16_t *w, uint16_t *wt, int K, int C) {
    __shared__ uint16_t tile[32][33];
    const int tap = blockIdx.z, k0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int k = k0 + i, c = c0 + threadIdx.x;
        tile[i][threadIdx.x] = (k < K && c < C) ? w[((size_t)k * 9 + tap) * C + c] : 0;
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int c = c0 + i, k = k0 + threadIdx.x;
        if (c < C && k < K) wt[((size_t)tap * C + c) * K + k] = tile[threadIdx.x][i];
    }
}

}  // namespace wici
