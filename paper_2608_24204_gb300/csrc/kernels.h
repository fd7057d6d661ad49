// Device buffers and the enqueue functions of the decode and prefill paths.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

#include "common.cuh"
#include "plan.h"

namespace wici {

// Device pointers derived from the three caller-owned buffers and the plan.
struct Bufs {
    uint16_t *W;      // packed weight arena (bf16 bits)
    uint16_t *KV;     // paged KV pool (bf16 bits)
    int *ctrl;        // control words (CtrlSlot)
    int *hist;        // hist[p] = greedy token produced for position p   [max_tokens + 1]
    float *x;         // decode residual stream                             [H]
    float *q;         // decode query after RoPE                            [qdim]
    float *o;         // decode attention output                            [qdim]
    float *m;         // decode SwiGLU output                               [F]
    float *logits;    // last logits                                        [V]
    int2 *amax;       // per-CTA argmax partials (value bits, index)        [num_sms]
    float *fd_part;   // flash-decode split states                           [nkv][splits][group][d + 4]
    uint32_t *mega_bound; // persistent decode: row-share boundaries (2^24 = all) [num_sms + 1]
    float *mega_time;     // persistent decode: gate/up time per CTA, last step (us) [num_sms]
    float2 *rope;     // (cos, sin) of p * theta^(-2i/d)                     [max_tokens][d/2]
    int *pages;       // logical -> physical KV page                         [max_pages]
    int *tok;         // prefill chunk tokens                                [max_chunk]
    float *X;         // prefill residual stream                             [max_chunk][H]
    // prefill tensor-core operands: each fp32 activation as kTerms bf16 terms
    uint16_t *Q[kTerms];  // queries after RoPE                               [max_chunk][qdim]
    uint16_t *A[kTerms];  // RMSNorm output                                   [max_chunk][H]
    uint16_t *O[kTerms];  // attention output                                 [max_chunk][qdim]
    uint16_t *M[kTerms];  // SwiGLU output                                    [max_chunk][F]
    // 8-bit block format only: the matrix of the next prefill GEMM dequantised
    // as three bf16 terms (exact: a code times an fp16 scale has <= 18 significant bits)
    uint16_t *Wt[kTerms]; //                                                    [wt_elems]
    // qk_norm only: k of this decode step before its norm and RoPE            [kvdim]
    // and the prefill chunk's q | k before their norms and RoPE               [max_chunk][qdim + kvdim]
    float *kraw, *QKraw;
};

// TMA descriptors of the prefill GEMM operands (built once per context).
struct PrefillMaps {
    CUtensorMap a[kTerms], o[kTerms], m[kTerms];       // GEMM activations, 128-row boxes
    CUtensorMap kv;                                    // the whole KV pool: [page][K|V][kv_head][16][d]
    std::vector<CUtensorMap> wqkv, wo, wgu, wd;        // per layer weights, boxes of bn_* rows
    CUtensorMap wt_qkv[kTerms], wt_o[kTerms], wt_gu[kTerms], wt_d[kTerms];  // 8-bit format: the dequantised terms
    int bn_qkv, bn_o, bn_gu, bn_d;                     // output-tile width of each matrix's GEMM
};


// A bf16 tensor map with 128-byte swizzle: dims / box / element strides innermost
// first, strides_bytes[i] the byte stride of dimension i + 1 (false on failure).
bool encode_tiled(CUtensorMap *m, int rank, const void *ptr, const uint64_t *dims, const uint64_t *strides_bytes,
                  const uint32_t *box, const uint32_t *elem_strides);

// Encodes every tensor map of `m`; returns an error message or nullptr.
const char *make_prefill_maps(const Plan &p, const Bufs &b, PrefillMaps *m);

// Called around every launch when profiling (eager mode).
struct LaunchHook {
    virtual void before(const char *name) = 0;
    virtual void after(const char *name) = 0;
    virtual ~LaunchHook() {}
};

// Flash-decode split count for a context of max_pages pages, and the floats
// of its split-state buffer.
int fd_splits(int max_pages);
size_t fd_part_floats(int nkv, int group, int d, int max_pages);

// One-time per-process kernel attributes (dynamic shared memory limits).
cudaError_t setup_kernels();

// Final RMSNorm + LM head + argmax of a caller-given row x [H] against W [V][H]
// with caller-given scratch: ctrl (CTRL_WORDS ints, zeroed), partials (grid
// int2) and hist (>= 1 int).  The token lands in ctrl[CTRL_TOKEN].
cudaError_t enqueue_lm_head_argmax_raw(const uint16_t *W, const uint16_t *gain, const float *x, int H, int V,
                                       float eps, float *logits, int *ctrl, int2 *partials, int *hist, int grid,
                                       cudaStream_t st);

// True when the decode step runs as one persistent kernel for this plan.
bool decode_is_persistent(const Plan &p);

// Whole decode step for the token in ctrl[CTRL_TOKEN] at position ctrl[CTRL_POS]:
// 5 launches per layer + the LM head.  `pdl` enables programmatic dependent launch.
cudaError_t enqueue_decode_step(const Plan &p, const Bufs &b, cudaStream_t st, bool pdl,
                                LaunchHook *hook);

// Final RMSNorm + LM head + argmax of the row in b.x; the last CTA writes
// ctrl[CTRL_TOKEN], hist[pos + pos_add] and advances ctrl[CTRL_POS] by pos_add.
cudaError_t enqueue_lm_head(const Plan &p, const Bufs &b, cudaStream_t st, bool pdl, int pos_add,
                            LaunchHook *hook);

// Prefill of the chunk b.tok[0..T) at positions P..P+T-1 through every layer.
// With lm_pos_add > 0 it then copies the chunk's last row to b.x and runs the
// LM head, which advances ctrl[CTRL_POS] by lm_pos_add.
cudaError_t enqueue_prefill_chunk(const Plan &p, const Bufs &b, const PrefillMaps &maps,
                                  cudaStream_t st, int P, int T, int lm_pos_add, LaunchHook *hook);

// Sets the per-thread message returned by wici_last_error(NULL).
void set_thread_error(const char *msg);

// RoPE table for positions [0, max_tokens).
cudaError_t enqueue_rope_table(const Plan &p, const Bufs &b, cudaStream_t st);

// One CTA waiting on an mbarrier that never completes; writes the wait's
// site id to *err when it gives up after limit_ns.
cudaError_t enqueue_bounded_wait_probe(int *err, int64_t limit_ns, cudaStream_t st);

}  // namespace wici
