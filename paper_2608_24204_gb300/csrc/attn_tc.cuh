// Prefill attention on the tcgen05 tensor cores.
//
// One CTA computes causal GQA attention for a tile of query rows of one KV
// head g: the rows pack TPT tokens x `group` query heads (row r = token r/group,
// head g*group + r%group), so each K/V tile serves the whole group.  Keys come
// from the paged cache in blocks of 128 (eight 16-key pages, fetched by 5-D TMA
// through the page table).  Per block j:
//   S_j  = (Q_0 + Q_1) K_j^T      tcgen05.mma, M=128 rows, N=128 keys, fp32 in TMEM
//   softmax (one row per thread pair, read from TMEM): P_j = exp2(s - m), with m
//          the row's reference maximum, stored over S_j in TMEM
//   O   += (P_0 + P_1) V_j        tcgen05.mma, N=d, V read as an MN-major operand,
//          accumulated in TMEM over all blocks
// Both A operands live in tensor memory: the softmax warps store the tile's Q
// terms there once, and each block's P terms over its S.  Shared memory only
// holds the K/V ring, and the tensor cores read only K and V from it.  N=128
// MMAs run at the full tensor rate (an N=64 one takes about 1.4 times its share).
// The reference maximum only moves when a block's maximum exceeds it by more
// than 2^8 (so P <= 256): then the softmax rescales its rows of the TMEM
// accumulator and its row sums by exp2(m_old - m_new), between P_{j-1} V_{j-1}
// and P_j V_j; the result O / l is the same softmax in exact arithmetic.
// S / P is double-buffered, so the tensor cores work ahead of the softmax: the
// MMA warp issues S_{j+2} into buffer j % 2 right after P_j V_j (the tensor core
// runs one thread's MMAs in issue order, so P_j is read before S_{j+2} lands),
// and P_j V_j runs while the softmax computes P_{j+1}.
// Q and P are carried as two bf16 terms (hi + lo: 16 significant bits), K and V
// are exact bf16: the products only meet bf16 K and V, whose own rounding is 2^-9.
// Warp roles: 0 TMA producer, 1 TMEM owner + MMA issuer, 2..9 softmax / output:
// two warps per TMEM lane quadrant (warp % 4), one for keys 0..63, d values
// [0, d/2) of Q and output columns [0, d/2) of its 32 rows, the other for keys
// 64..127 and the upper halves; the pair exchanges each block's row maxima
// through shared memory.  Every wait is bounded.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "gemm_tc.cuh"

namespace wici {

constexpr int AT_ROWS = 128;           // query rows per tile (TMEM lanes)
constexpr int AT_KEYS = 128;           // keys per block
constexpr int AT_STAGES = 3;           // K/V ring depth
constexpr int AT_TERMS = 2;            // bf16 terms of the Q and P operands
constexpr int AT_THREADS = 320;        // producer, MMA, 8 softmax warps (two per TMEM lane quadrant)
constexpr uint32_t AT_TMEM_COLS = 512;
constexpr float AT_RESCALE_LOG2 = 8.f; // the reference maximum trails the row maximum by at most this

enum : int { SITE_AT_Q = 41, SITE_AT_KVE = 42, SITE_AT_KVF = 43, SITE_AT_S = 44, SITE_AT_P = 45, SITE_AT_O = 46,
             SITE_AT_DRAIN = 47 };

// TMEM columns (one 32-bit column holds two bf16 of a row): Q terms [0, d);
// S / P buffers [d, d + 128) and [d + 128, d + 256), each holding S (128 fp32
// columns) and then P (term t in columns [64 t, 64 t + 64)); the O accumulator
// [d + 256, 2d + 256)
template <int D>
struct AttnTmem {
    static constexpr uint32_t Q = 0, SP = D, O = D + 2 * AT_KEYS;
    static_assert(2 * D + 2 * AT_KEYS <= (int)AT_TMEM_COLS, "tensor memory");
};

template <int D>
struct AttnSmem {
    static constexpr int DCH = D / 64;                                   // 64-element d chunks
    static constexpr uint32_t KV_BYTES = AT_KEYS * D * 2;                // K (or V) of a block
    static constexpr uint32_t OFF_KV = 0;                                // [stage][K | V]
    static constexpr uint32_t TOTAL = AT_STAGES * 2 * KV_BYTES;
};

// K-major, 128-byte swizzle, 8-row groups 1024 B apart (the K operand)
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

__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap *map, int c0, int c1, int c2, int c3, int c4,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
        "l"((uint64_t)map), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(bar)
        : "memory");
}

// 32 lanes x 32 (16) columns of 32-bit words into TMEM (this warp's lane quadrant); complete at tc_wait_st
__device__ __forceinline__ void tc_st32(uint32_t taddr, const uint32_t *v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]),
        "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]),
        "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
}
__device__ __forceinline__ void tc_st16(uint32_t taddr, const uint32_t *v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}
template <int N>
__device__ __forceinline__ void tc_st_cols(uint32_t taddr, const uint32_t *v) {
    static_assert(N == 16 || N == 32, "16 or 32 columns");
    if constexpr (N == 32)
        tc_st32(taddr, v);
    else
        tc_st16(taddr, v);
}

// D (+)= A B with the A operand (M = 128 rows on the TMEM lanes, K-major bf16 pairs) in tensor memory
__device__ __forceinline__ void tc_mma_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(tmem_d),
        "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
// 2^x (PTX ex2.approx, flush-to-zero): 2^-inf = 0
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// two floats -> two bf16 (round to nearest even) in one word, lo in bits 0..15
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t w;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(w) : "f"(hi), "f"(lo));
    return w;
}

// tokens per 128-row tile: the group's query heads of each token share a tile
__host__ __device__ constexpr int attn_tokens_per_tile(int group) { return AT_ROWS / group; }

struct AttnArgs {
    const uint16_t *Q[AT_TERMS];  // [T][nq * d] query terms
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
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_kv, const AttnArgs a) {
    using L = AttnSmem<D>;
    using TM = AttnTmem<D>;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t q_ready, kv_full[AT_STAGES], kv_empty[AT_STAGES], s_full[2], p_full[2], o_full;
    __shared__ uint32_t s_tmem;
    __shared__ int s_issued;
    __shared__ float s_rowmax[2][AT_ROWS];      // [key half][row]: each block's row maxima, the row sums at the end

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // CTAs in launch order take the tiles heaviest (latest) first across all KV
    // heads, so the last wave holds the lightest tiles of every head
    const int nkv = a.nq / a.group;
    const int g = (int)blockIdx.x % nkv;
    const int tile = (int)(gridDim.x / nkv) - 1 - (int)blockIdx.x / nkv;
    const int t0 = tile * a.tpt;
    const int t_end = min(a.T, t0 + a.tpt);
    const int nkeys = a.P + t_end;                    // keys the tile's last token sees
    const int nb = (nkeys + AT_KEYS - 1) / AT_KEYS;
    const uint32_t base = (smem_u32(smem_raw) + 1023u) & ~1023u;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&q_ready), 8);
        for (int s = 0; s < AT_STAGES; ++s) {
            mbar_init(smem_u32(&kv_full[s]), 1);
            mbar_init(smem_u32(&kv_empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&s_full[b]), 1);
            mbar_init(smem_u32(&p_full[b]), 8);
        }
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
    const uint32_t tm_q = tmem + TM::Q, tm_sp = tmem + TM::SP, tm_o = tmem + TM::O;

    if (warp == 0) {
        if (lane == 0) {  // ----------------------------------------------- TMA producer
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
                        // chunk c holds d values [64c, 64c+64) of the block's keys (rows of 128 B)
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
            bool ok = mbar_wait(smem_u32(&q_ready), 0, a.err, SITE_AT_Q);
            auto issue_s = [&](int j) {
                const int s = j % AT_STAGES;
                ok = ok && mbar_wait(smem_u32(&kv_full[s]), (j / AT_STAGES) & 1, a.err, SITE_AT_KVF);
                if (!ok) return;
                tc_fence_after();
                const uint32_t kb = base + L::OFF_KV + (uint32_t)s * 2 * L::KV_BYTES;
                const uint32_t sacc = tm_sp + (uint32_t)AT_KEYS * (uint32_t)(j & 1);
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    // d values 16k..16k+15: 8 TMEM columns of each Q term, 32 bytes of each K row
                    const uint32_t koff = (uint32_t)(k / 4) * (AT_KEYS * 128) + 32u * (k % 4);
                    const uint64_t bd = at_desc_k(kb + koff);
#pragma unroll
                    for (int t = 0; t < AT_TERMS; ++t)
                        tc_mma_ts(sacc, tm_q + (uint32_t)(t * (D / 2) + 8 * k), bd, idesc_s, (k | t) != 0);
                }
                tc_commit(smem_u32(&s_full[j & 1]));
            };
            if (nb > 0) issue_s(0);
            if (nb > 1) issue_s(1);
            for (int j = 0; j < nb && ok; ++j) {
                const int s = j % AT_STAGES, b = j & 1;
                // P_j stored over S_j (and O rescaled if its reference maximum moved) by the softmax
                ok = mbar_wait(smem_u32(&p_full[b]), (j >> 1) & 1, a.err, SITE_AT_P);
                if (!ok) break;
                tc_fence_after();
                const uint32_t vb = base + L::OFF_KV + (uint32_t)s * 2 * L::KV_BYTES + L::KV_BYTES;
                const uint32_t pb = tm_sp + (uint32_t)AT_KEYS * (uint32_t)b;
#pragma unroll
                for (int k = 0; k < AT_KEYS / 16; ++k) {
                    // 16 keys = two 8-key groups of V rows; P columns 8k..8k+7 of each term
                    const uint64_t vd = at_desc_mn(vb + 2048u * k, AT_KEYS * 128);
#pragma unroll
                    for (int t = 0; t < AT_TERMS; ++t)
                        tc_mma_ts(tm_o, pb + (uint32_t)(AT_KEYS / 2) * t + 8u * k, vd, idesc_o, (j | k | t) != 0);
                }
                tc_commit(smem_u32(&kv_empty[s]));
                // the softmax waits for O only before its last block and at the end; earlier
                // rescales wait for S_{j+1}, which lands after P_{j-1} V_{j-1}
                if (j >= nb - 2) tc_commit(smem_u32(&o_full));
                if (j + 2 < nb) issue_s(j + 2);   // S buffer b was read before P_j was posted
            }
        }
    } else {  // ------------------------------------------------------- softmax / output
        constexpr int HK = AT_KEYS / 2, HD = D / 2;   // keys, d values and output columns per warp of a pair
        const int qd = warp & 3;                   // TMEM lane quadrant
        const int hc = (warp - 2) >> 2;            // which half of the keys, of Q and of the output columns
        const int r = qd * 32 + lane;              // tile row
        const bool row_ok = r < a.tpt * a.group;
        const int tok = t0 + r / a.group;          // chunk token of this row
        const int qpos = a.P + tok;                // its absolute position
        const int head = g * a.group + r % a.group;
        const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
        const uint32_t pair_bar = 1 + qd;          // named barrier of the two warps of this quadrant
        const size_t row_off = (size_t)tok * a.nq * D + (size_t)head * D + hc * HD;
        {   // this row's half of the Q terms into TMEM (zeros past the chunk)
            const bool q_ok = row_ok && tok < a.T;
#pragma unroll
            for (int t = 0; t < AT_TERMS; ++t) {
                uint32_t qw[HD / 2];
#pragma unroll
                for (int c = 0; c < HD / 8; ++c) {
                    const uint4 v = q_ok ? *reinterpret_cast<const uint4 *>(a.Q[t] + row_off + 8 * c)
                                         : make_uint4(0u, 0u, 0u, 0u);
                    qw[4 * c] = v.x;
                    qw[4 * c + 1] = v.y;
                    qw[4 * c + 2] = v.z;
                    qw[4 * c + 3] = v.w;
                }
                tc_st_cols<HD / 2>(tm_q + lane_base + (uint32_t)(t * (D / 2) + hc * (HD / 2)), qw);
            }
            tc_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&q_ready));
        }
        // blocks before this one are visible to every row of the tile: no causal mask
        const int first_masked = a.tpt * a.group == AT_ROWS ? (a.P + t0 + 1) / AT_KEYS : 0;
        float m = -INFINITY, l = 0.f;   // reference maximum (log2 units) and row sum in its scale
        bool ok = true;
        const uint32_t tm_orow = tm_o + lane_base + hc * HD;
        for (int j = 0; j < nb; ++j) {
            const uint32_t sp = tm_sp + (uint32_t)AT_KEYS * (uint32_t)(j & 1) + lane_base;
            ok = ok && mbar_wait(smem_u32(&s_full[j & 1]), (j >> 1) & 1, a.err, SITE_AT_S);
            tc_fence_after();
            float sv[HK];
#pragma unroll
            for (int c0 = 0; c0 < HK; c0 += 32) tc_ld32(sp + hc * HK + c0, sv + c0);
            if (j >= first_masked) {
#pragma unroll
                for (int c = 0; c < HK; ++c) {
                    const int key = j * AT_KEYS + hc * HK + c;
                    if (!(row_ok && key <= qpos)) sv[c] = -INFINITY;
                }
            }
            float bm = sv[0];
#pragma unroll
            for (int c = 1; c + 1 < HK; c += 2) bm = fmax3(bm, sv[c], sv[c + 1]);
            if ((HK & 1) == 0) bm = fmaxf(bm, sv[HK - 1]);
            // the row's block maximum over both halves (raw scores: the scale is positive)
            s_rowmax[hc][r] = bm;
            // the pair leaves the loop together: the barrier also ANDs the two warps'
            // wait results, so a wait that gave up in one warp never strands the other.
            // Past it both warps hold their S values in registers, so P may overwrite S.
            uint32_t both_ok;
            asm volatile(
                "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 q, %1, 0;\n\t"
                "bar.red.and.pred p, %2, 64, q;\n\tselp.u32 %0, 1, 0, p;\n\t}"
                : "=r"(both_ok)
                : "r"((uint32_t)ok), "r"(pair_bar)
                : "memory");
            if (!both_ok) {
                ok = false;
                break;
            }
            bm = fmaxf(bm, s_rowmax[hc ^ 1][r]) * a.scale_log2;
            // both have read before either writes the next block's value
            asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
            // a new reference maximum only when this block's exceeds it by more than 2^8
            const bool grow = bm > m + AT_RESCALE_LOG2;
            const float mn = grow ? bm : m;
            const float corr = grow ? fast_exp2(m - mn) : 1.f;
            const float nms = mn == -INFINITY ? 0.f : -mn;   // rows with nothing visible yet
            float ps0 = 0.f, ps1 = 0.f;
            // P as two bf16 terms over S: this half's 64 keys are 32 columns of each term,
            // written 16 columns (32 keys) at a time
#pragma unroll
            for (int c0 = 0; c0 < HK; c0 += 32) {
                uint32_t w0[16], w1[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const float p0 = fast_exp2(fmaf(sv[c0 + 2 * e], a.scale_log2, nms));
                    const float p1 = fast_exp2(fmaf(sv[c0 + 2 * e + 1], a.scale_log2, nms));
                    ps0 += p0;
                    ps1 += p1;
                    w0[e] = pack_bf16x2(p0, p1);
                    w1[e] = pack_bf16x2(p0 - bf16lo(w0[e]), p1 - bf16hi(w0[e]));
                }
                const uint32_t pc = sp + (uint32_t)(hc * (HK / 2) + c0 / 2);
                tc_st16(pc, w0);
                tc_st16(pc + AT_KEYS / 2, w1);
            }
            // O is rescaled once P_{j-1} V_{j-1} has landed and before P_j V_j is issued.
            // Before block nb - 1, S_{j+1} completing implies it (S_{j+1} was issued after
            // it; P_{j+1} is not posted, so that parity wait is exact).  The last block
            // always waits for the first of the two o_full phases (P_{nb-2} V_{nb-2}),
            // which keeps the final wait for the second one exact.
            const bool any_grow = __any_sync(0xFFFFFFFFu, grow);
            if (j > 0 && (any_grow || j == nb - 1)) {
                if (j + 1 < nb)
                    ok = ok && mbar_wait(smem_u32(&s_full[(j + 1) & 1]), ((j + 1) >> 1) & 1, a.err, SITE_AT_O);
                else
                    ok = ok && mbar_wait(smem_u32(&o_full), 0, a.err, SITE_AT_O);
                tc_fence_after();
                if (any_grow) {
#pragma unroll
                    for (int c0 = 0; c0 < HD; c0 += 32) {
                        float ov[32];
                        uint32_t ow[32];
                        tc_ld32(tm_orow + c0, ov);
#pragma unroll
                        for (int i = 0; i < 32; ++i) ow[i] = __float_as_uint(ov[i] * corr);
                        tc_st32(tm_orow + c0, ow);
                    }
                }
            }
            tc_wait_st();
            l = l * corr + (ps0 + ps1);   // this half's share of the row sum, in the reference scale
            m = mn;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&p_full[j & 1]));
        }
        // the last P.V: O complete in TMEM
        float o[HD];
#pragma unroll
        for (int i = 0; i < HD; ++i) o[i] = 0.f;
        if (ok && nb > 0) {
            // o_full completes after P_{nb-2} V_{nb-2} (when nb > 1; waited for in the last
            // block) and after P_{nb-1} V_{nb-1}
            ok = mbar_wait(smem_u32(&o_full), nb > 1 ? 1 : 0, a.err, SITE_AT_O);
            tc_fence_after();
#pragma unroll
            for (int c0 = 0; c0 < HD; c0 += 32) tc_ld32(tm_orow + c0, o + c0);
        }
        // the row sum of both halves (the last maxima were read before the pair's last barrier)
        s_rowmax[hc][r] = l;
        asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
        l += s_rowmax[hc ^ 1][r];
        if (ok && row_ok && tok < a.T) {
            const float inv = 1.0f / l;
#pragma unroll
            for (int c = 0; c < HD; c += 8) {
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
                *reinterpret_cast<uint4 *>(a.O[0] + row_off + c) = make_uint4(w0[0], w0[1], w0[2], w0[3]);
                *reinterpret_cast<uint4 *>(a.O[1] + row_off + c) = make_uint4(w1[0], w1[1], w1[2], w1[3]);
                *reinterpret_cast<uint4 *>(a.O[2] + row_off + c) = make_uint4(w2[0], w2[1], w2[2], w2[3]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0 && lane == 0) {
        // nothing may still land in shared memory after exit
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
