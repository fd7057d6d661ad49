// Prefill attention on the tcgen05 tensor cores.
//
// One CTA computes causal GQA attention for a tile of query rows of one KV
// head g: the rows pack TPT tokens x `group` query heads (row r = token r/group,
// head g*group + r%group), so each K/V tile serves the whole group.  Keys come
// from the paged cache in blocks of 64 (four 16-key pages, fetched by 5-D TMA
// through the page table).  Per block:
//   S  = (Q_0 + Q_1) K^T          tcgen05.mma, M=128 rows, N=64 keys, fp32 in TMEM
//   softmax (one row per thread, read from TMEM): online max/sum, P = exp2(s - m)
//   O_blk = (P_0 + P_1) V         tcgen05.mma, N=d, V read as an MN-major operand
//   O = O * corr + O_blk          in registers
// Q and P are carried as two bf16 terms (hi + lo: 16 significant bits), K and V
// are exact bf16: the products only meet bf16 K and V, whose own rounding is 2^-9,
// and the two-term tiles leave room for a three-stage K/V ring (the kernel is
// bound by the K/V bytes it keeps in flight).  Warp roles: 0 TMA producer,
// 1 TMEM owner + MMA issuer, 2..5
// softmax / output (TMEM lane quadrant = warp % 4).  Every wait is bounded.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "gemm_tc.cuh"

namespace wici {

constexpr int AT_ROWS = 128;           // query rows per tile (TMEM lanes)
constexpr int AT_KEYS = 64;            // keys per block
constexpr int AT_STAGES = 3;           // K/V ring depth
constexpr int AT_TERMS = 2;            // bf16 terms of the Q and P operands
constexpr int AT_THREADS = 192;
constexpr uint32_t AT_TMEM_COLS = 256; // S: [0, 64), O block: [128, 128 + d)

enum : int { SITE_AT_Q = 41, SITE_AT_KVE = 42, SITE_AT_KVF = 43, SITE_AT_S = 44, SITE_AT_P = 45, SITE_AT_O = 46,
             SITE_AT_DRAIN = 47 };

template <int D>
struct AttnSmem {
    static constexpr int DCH = D / 64;                                   // 64-element d chunks
    static constexpr uint32_t Q_BYTES = AT_ROWS * D * 2;                 // one term
    static constexpr uint32_t KV_BYTES = AT_KEYS * D * 2;                // K (or V) of a block
    static constexpr uint32_t P_BYTES = AT_ROWS * AT_KEYS * 2;           // one term
    static constexpr uint32_t OFF_Q = 0;                                 // [term]
    static constexpr uint32_t OFF_KV = AT_TERMS * Q_BYTES;               // [stage][K | V]
    static constexpr uint32_t OFF_P = OFF_KV + AT_STAGES * 2 * KV_BYTES; // [term]
    static constexpr uint32_t TOTAL = OFF_P + AT_TERMS * P_BYTES;
};

// K-major, 128-byte swizzle, 8-row groups 1024 B apart (Q, K and P operands)
__device__ __forceinline__ uint64_t at_desc_k(uint32_t saddr) { return tc_desc_sw128(saddr); }

// MN-major, 128-byte swizzle (V as the B operand of P.V): rows are keys (the K
// dimension) of 64 consecutive d values; 8-key groups are 1024 B apart (stride
// byte offset) and the next 64 d values are `lbo` bytes further (leading byte offset)
__device__ __forceinline__ uint64_t at_desc_mn(uint32_t saddr, uint32_t lbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// kind::f16 instruction descriptor: D fp32, A/B bf16, M = 128, N = n; b_mn selects an MN-major B
__host__ __device__ constexpr uint32_t at_idesc(int n, bool b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn ? 1u : 0u) << 16) | ((uint32_t)(n >> 3) << 17) |
           ((uint32_t)(AT_ROWS >> 4) << 24);
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int x, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap *map, int c0, int c1, int c2, int c3, int c4,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// tokens per 128-row tile: the group's query heads of each token share a tile
__host__ __device__ constexpr int attn_tokens_per_tile(int group) { return AT_ROWS / group; }

struct AttnArgs {
    uint16_t *O[kTerms];  // [T][nq * d] output terms
    const int *pages;     // logical -> physical page
    int *err;
    int P, T;             // cached positions before the chunk, chunk length
    int nq, group, tpt;   // query heads, heads per KV head, tokens per tile
    int layer, max_pages;
    float scale_log2;     // log2(e) / sqrt(d)
};

template <int D>
__global__ void __launch_bounds__(AT_THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_q0, const __grid_constant__ CUtensorMap map_q1,
                   const __grid_constant__ CUtensorMap map_kv,
                   const AttnArgs a) {
    using L = AttnSmem<D>;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t q_full, kv_full[AT_STAGES], kv_empty[AT_STAGES], s_full, p_full, o_full;
    __shared__ uint32_t s_tmem;
    __shared__ int s_issued;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.y;
    const int tile = gridDim.x - 1 - blockIdx.x;     // heaviest (latest) tiles first
    const int t0 = tile * a.tpt;
    const int t_end = min(a.T, t0 + a.tpt);
    const int nkeys = a.P + t_end;                    // keys the tile's last token sees
    const int nb = (nkeys + AT_KEYS - 1) / AT_KEYS;
    const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;
    const uint32_t q_bytes_box = 64u * (uint32_t)a.group * (uint32_t)a.tpt * 2u;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&q_full), 1);
        for (int s = 0; s < AT_STAGES; ++s) {
            mbar_init(smem_u32(&kv_full[s]), 1);
            mbar_init(smem_u32(&kv_empty[s]), 1);
        }
        mbar_init(smem_u32(&s_full), 1);
        mbar_init(smem_u32(&p_full), 4);
        mbar_init(smem_u32(&o_full), 1);
        fence_barrier_init();
        s_issued = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                     "r"(AT_TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    const uint32_t tm_s = tmem, tm_o = tmem + 128;

    if (warp == 0) {
        if (lane == 0) {  // ----------------------------------------------- TMA producer
            const uint32_t qb = smem_u32(&q_full);
            mbar_arrive_expect_tx(qb, (uint32_t)AT_TERMS * L::DCH * q_bytes_box);
            for (int c = 0; c < L::DCH; ++c) {
                tma_load_3d(base + L::OFF_Q + c * AT_ROWS * 128, &map_q0, c * 64, g * a.group, t0, qb);
                tma_load_3d(base + L::OFF_Q + L::Q_BYTES + c * AT_ROWS * 128, &map_q1, c * 64, g * a.group, t0, qb);
            }
            int issued = 0;
            for (int j = 0; j < nb; ++j) {
                const int s = j % AT_STAGES;
                if (j >= AT_STAGES &&
                    !mbar_wait(smem_u32(&kv_empty[s]), ((j / AT_STAGES) + 1) & 1, a.err, SITE_AT_KVE))
                    break;
                const uint32_t fb = smem_u32(&kv_full[s]);
                mbar_arrive_expect_tx(fb, 2u * L::KV_BYTES);
                const uint32_t kdst = base + L::OFF_KV + (uint32_t)s * 2 * L::KV_BYTES;
                const uint32_t vdst = kdst + L::KV_BYTES;
                for (int pg = 0; pg < AT_KEYS / 16; ++pg) {
                    int lp = j * (AT_KEYS / 16) + pg;              // logical page
                    const int pp = lp < a.max_pages ? a.pages[lp] : 0;   // past the table: masked keys
                    const int page = a.layer * a.max_pages + pp;
                    for (int c = 0; c < L::DCH; ++c) {
                        // chunk c holds d values [64c, 64c+64) of all 64 keys (rows of 128 B)
                        tma_load_5d(kdst + c * (AT_KEYS * 128) + pg * 16 * 128, &map_kv, c * 64, 0, g, 0, page, fb);
                        tma_load_5d(vdst + c * (AT_KEYS * 128) + pg * 16 * 128, &map_kv, c * 64, 0, g, 1, page, fb);
                    }
                }
                issued = j + 1;
            }
            s_issued = issued;
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ----------------------------------------------- MMA issuer
            constexpr uint32_t idesc_s = at_idesc(AT_KEYS, false);
            constexpr uint32_t idesc_o = at_idesc(D, true);
            bool ok = mbar_wait(smem_u32(&q_full), 0, a.err, SITE_AT_Q);
            auto issue_s = [&](int j) {
                const int s = j % AT_STAGES;
                ok = ok && mbar_wait(smem_u32(&kv_full[s]), (j / AT_STAGES) & 1, a.err, SITE_AT_KVF);
                if (!ok) return;
                tc_fence_after();
                const uint32_t kb = base + L::OFF_KV + (uint32_t)s * 2 * L::KV_BYTES;
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    const uint32_t off = (uint32_t)(k / 4) * (AT_ROWS * 128) + 32u * (k % 4);
                    const uint32_t koff = (uint32_t)(k / 4) * (AT_KEYS * 128) + 32u * (k % 4);
                    const uint64_t bd = at_desc_k(kb + koff);
#pragma unroll
                    for (int t = 0; t < AT_TERMS; ++t)
                        tc_mma(tm_s, at_desc_k(base + L::OFF_Q + t * L::Q_BYTES + off), bd, idesc_s, (k | t) != 0);
                }
                tc_commit(smem_u32(&s_full));
            };
            if (nb > 0) issue_s(0);
            for (int j = 0; j < nb && ok; ++j) {
                const int s = j % AT_STAGES;
                ok = mbar_wait(smem_u32(&p_full), j & 1, a.err, SITE_AT_P);   // P_j written, S_j read
                if (!ok) break;
                tc_fence_after();
                const uint32_t vb = base + L::OFF_KV + (uint32_t)s * 2 * L::KV_BYTES + L::KV_BYTES;
#pragma unroll
                for (int k = 0; k < AT_KEYS / 16; ++k) {
                    // 16 keys = two 8-key groups of V rows; P columns 16k..16k+15
                    const uint64_t vd = at_desc_mn(vb + 2048u * k, AT_KEYS * 128);
#pragma unroll
                    for (int t = 0; t < AT_TERMS; ++t)
                        tc_mma(tm_o, at_desc_k(base + L::OFF_P + t * L::P_BYTES + 32u * k), vd, idesc_o, (k | t) != 0);
                }
                tc_commit(smem_u32(&o_full));
                tc_commit(smem_u32(&kv_empty[s]));
                if (j + 1 < nb) issue_s(j + 1);
            }
        }
    } else {  // ------------------------------------------------------- softmax / output
        const int qd = warp & 3;                   // TMEM lane quadrant
        const int r = qd * 32 + lane;              // tile row
        const bool row_ok = r < a.tpt * a.group;
        const int tok = t0 + r / a.group;          // chunk token of this row
        const int qpos = a.P + tok;                // its absolute position
        const int head = g * a.group + r % a.group;
        const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
        float o[D];
#pragma unroll
        for (int i = 0; i < D; ++i) o[i] = 0.f;
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        uint8_t *pbase = smem_raw + (base - smem_u32(smem_raw)) + L::OFF_P;
        for (int j = 0; j < nb && ok; ++j) {
            ok = mbar_wait(smem_u32(&s_full), j & 1, a.err, SITE_AT_S);
            tc_fence_after();
            float sv[AT_KEYS];
            tc_ld32(tm_s + lane_base, sv);
            tc_ld32(tm_s + lane_base + 32, sv + 32);
            float bm = -INFINITY;
#pragma unroll
            for (int c = 0; c < AT_KEYS; ++c) {
                const int key = j * AT_KEYS + c;
                sv[c] = (row_ok && key <= qpos) ? sv[c] * a.scale_log2 : -INFINITY;
                bm = fmaxf(bm, sv[c]);
            }
            const float mn = fmaxf(m, bm);
            const float msafe = mn == -INFINITY ? 0.f : mn;   // rows with nothing visible yet
            const float corr = exp2f(m - msafe);
            float ps = 0.f;
            // P row r as two bf16 terms, 128-byte swizzled rows (16-byte piece i at i ^ (r % 8))
            uint8_t *prow = pbase + r * 128;
#pragma unroll
            for (int piece = 0; piece < AT_KEYS / 8; ++piece) {
                uint32_t w0[4], w1[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float p0 = exp2f(sv[piece * 8 + 2 * e] - msafe);
                    const float p1 = exp2f(sv[piece * 8 + 2 * e + 1] - msafe);
                    ps += p0 + p1;
                    const uint16_t a0 = f32_to_bf16(p0), b0 = f32_to_bf16(p1);
                    const uint16_t a1 = f32_to_bf16(p0 - bf16_to_f32(a0)), b1 = f32_to_bf16(p1 - bf16_to_f32(b0));
                    w0[e] = (uint32_t)a0 | ((uint32_t)b0 << 16);
                    w1[e] = (uint32_t)a1 | ((uint32_t)b1 << 16);
                }
                const int sp = (piece ^ (r & 7)) * 16;
                *reinterpret_cast<uint4 *>(prow + sp) = make_uint4(w0[0], w0[1], w0[2], w0[3]);
                *reinterpret_cast<uint4 *>(prow + L::P_BYTES + sp) = make_uint4(w1[0], w1[1], w1[2], w1[3]);
            }
            l = l * corr + ps;
            m = mn;
            fence_proxy_async_smem();   // generic-proxy writes of P before the MMA reads them
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&p_full));
            ok = ok && mbar_wait(smem_u32(&o_full), j & 1, a.err, SITE_AT_O);
            tc_fence_after();
#pragma unroll
            for (int c0 = 0; c0 < D; c0 += 32) {
                float ov[32];
                tc_ld32(tm_o + lane_base + c0, ov);
#pragma unroll
                for (int i = 0; i < 32; ++i) o[c0 + i] = fmaf(o[c0 + i], corr, ov[i]);
            }
        }
        if (ok && row_ok && tok < a.T) {
            const float inv = 1.0f / l;
            const size_t off = (size_t)tok * a.nq * D + (size_t)head * D;
#pragma unroll
            for (int c = 0; c < D; c += 8) {
                uint32_t w0[4], w1[4], w2[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    uint16_t a0, a1, a2, b0, b1, b2;
                    split_bf16x3(o[c + 2 * e] * inv, a0, a1, a2);
                    split_bf16x3(o[c + 2 * e + 1] * inv, b0, b1, b2);
                    w0[e] = (uint32_t)a0 | ((uint32_t)b0 << 16);
                    w1[e] = (uint32_t)a1 | ((uint32_t)b1 << 16);
                    w2[e] = (uint32_t)a2 | ((uint32_t)b2 << 16);
                }
                *reinterpret_cast<uint4 *>(a.O[0] + off + c) = make_uint4(w0[0], w0[1], w0[2], w0[3]);
                *reinterpret_cast<uint4 *>(a.O[1] + off + c) = make_uint4(w1[0], w1[1], w1[2], w1[3]);
                *reinterpret_cast<uint4 *>(a.O[2] + off + c) = make_uint4(w2[0], w2[1], w2[2], w2[3]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0 && lane == 0) {
        // nothing may still land in shared memory after exit
        mbar_wait(smem_u32(&q_full), 0, a.err, SITE_AT_DRAIN);
        const int issued = s_issued;
        for (int j = issued - AT_STAGES < 0 ? 0 : issued - AT_STAGES; j < issued; ++j)
            mbar_wait(smem_u32(&kv_full[j % AT_STAGES]), (j / AT_STAGES) & 1, a.err, SITE_AT_DRAIN);
    }
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(AT_TMEM_COLS)
                     : "memory");
    }
}

}  // namespace wici
