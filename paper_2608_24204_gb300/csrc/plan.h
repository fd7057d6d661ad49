// Buffer plan: where every tensor lives in the caller-owned weight arena,
// KV pool and workspace.  Host-side only; shared by the launch code.
#pragma once
#include <stddef.h>
#include <stdint.h>

#include <vector>

#include "../../include/wici.h"

namespace wici {

constexpr int kPage = 16;          // tokens per KV page
constexpr int kGemvThreads = 288;  // 8 consumer warps + 1 producer warp
#ifndef WICI_GEMV_RING_BYTES
#define WICI_GEMV_RING_BYTES 98304
#endif
#ifndef WICI_GEMV_CTAS_PER_SM
#define WICI_GEMV_CTAS_PER_SM 1
#endif
constexpr uint32_t kGemvRingBytes = WICI_GEMV_RING_BYTES;   // shared-memory ring per CTA
constexpr int kGemvCtasPerSm = WICI_GEMV_CTAS_PER_SM;       // GEMV grid = SMs x this
constexpr uint32_t kGemvStageMax = 32768;  // one unit (<= 2 rows of hidden <= 8192, or a row of K <= 16384)

// Bytes of one matrix row of K input columns in the 8-bit block format as the
// decode kernel streams it: K int8 codes followed by the row's K/32 fp16 block
// scales.  K % 256 == 0 keeps every row 16-byte aligned.
constexpr size_t q8_row_bytes(size_t K) { return K + K / 16; }

struct LayerOffsets {       // bf16 element offsets into the weight arena
    size_t attn_norm, wqkv, bqkv, qn, kn, wo, ffn_norm, wgu, wd;   // qn, kn: q/k norm gains (qk_norm)
};

struct Plan {
    wici_config cfg;
    int L, H, F, V, nq, nkv, d, qdim, kvdim, nqkv, group, max_pages, max_chunk;
    bool q8;                // the per-layer matrices are in the 8-bit block format
    bool qk_norm;           // Qwen3 block: per-head RMSNorm of q and k before RoPE
    // weight arena (bf16 elements)
    size_t w_embed, w_final_norm, w_lm;
    std::vector<LayerOffsets> layer;
    size_t weight_elems;
    // KV pool (bf16 elements)
    size_t kv_page_elems;   // one page: [K|V][nkv][16][d]
    size_t kv_layer_elems;  // max_pages pages
    size_t kv_elems;
    // workspace (byte offsets)
    size_t ws_ctrl, ws_hist, ws_x, ws_q, ws_o, ws_m, ws_logits, ws_amax, ws_rope,
        ws_pages, ws_tok, ws_X, ws_fd_part, ws_mega_bound, ws_mega_time;
    size_t ws_Q[3], ws_A[3], ws_O[3], ws_M[3];   // one buffer per bf16 term
    size_t ws_Wt[3];        // 8-bit format only: one matrix dequantised as three bf16 terms (prefill)
    size_t ws_kraw, ws_QKraw;   // qk_norm only: this step's k before its norm (decode), the chunk's q|k (prefill)
    size_t wt_elems;        // elements of the largest per-layer matrix
    size_t ws_bytes;
    int num_sms;
};

// Fills `p` from `cfg`; returns an error message or nullptr.
const char *make_plan(const wici_config *cfg, int num_sms, Plan *p);

}  // namespace wici
