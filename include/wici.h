/*
 * wici.h - C ABI of the GB300-native batch-1 decoder forward pass.
 *
 * The library computes the per-token GPU work that WiCi (arxiv 2608.24204)
 * offloads from a mobile client: T_Local of Eq. 1 (Sec. 3.3), i.e. the
 * prefill over a prompt (time to first token) and then one forward step per
 * generated token, each step repeating the same computation with a new input
 * token (Sec. 4.2.2).  Model: Llama-style decoder (RMSNorm, rotate-half RoPE,
 * grouped-query causal attention over a paged bf16 KV cache, SwiGLU MLP,
 * greedy argmax); weights are bf16, row-major [out, in], y = W x.
 *
 * Conventions for every entry point
 *   - Return value: WICI_OK (0) or a negative wici_status; the message is in
 *     wici_last_error(ctx) (ctx may be NULL for wici_create/wici_get_sizes
 *     failures: the message is then per calling thread).
 *   - On any error the KV length and the cached K/V of positions < kv_len are
 *     unchanged.  Capacity and arguments are checked before any launch.
 *   - Device buffers (weights arena, KV pool, workspace) are allocated by the
 *     caller with the sizes from wici_get_sizes and borrowed by the context
 *     until wici_destroy; the library owns only its streams, events, CUDA
 *     graph and a small pinned staging buffer.
 *   - Host buffers (token arrays, logits) are owned by the caller and are
 *     read or written before the call returns: every call that produces
 *     output synchronises its stream before returning.
 *   - A context is not thread-safe; use one per thread (the paper's router
 *     serves each client from its own thread, Sec. 3.2).
 *   - Device-side waits are bounded in time; a wait that gives up makes the
 *     call return WICI_E_TIMEOUT and leaves the context usable.
 */
#ifndef WICI_H
#define WICI_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct wici_ctx wici_ctx;

typedef enum wici_status {
    WICI_OK = 0,
    WICI_E_ARG = -1,      /* bad pointer, size, name or configuration */
    WICI_E_STATE = -2,    /* call not valid now (e.g. decode before prefill, weights missing) */
    WICI_E_CAPACITY = -3, /* the tokens would not fit in max_tokens KV positions */
    WICI_E_CUDA = -4,     /* a CUDA runtime call failed */
    WICI_E_TIMEOUT = -5   /* a bounded device-side wait gave up */
} wici_status;

/* Model shape and capacity.  Constraints: hidden, ffn_dim and n_q_heads*head_dim
 * multiples of 8; head_dim 64 or 128; n_q_heads a multiple of n_kv_heads with at
 * most 8 query heads per KV head; page_tokens == 16; 1 <= max_chunk <= max_tokens. */
typedef struct wici_config {
    int32_t n_layers, hidden, n_q_heads, n_kv_heads, head_dim, ffn_dim, vocab;
    int32_t max_tokens;      /* KV capacity in positions */
    int32_t max_chunk;       /* tokens processed per prefill pass; longer prompts are split */
    int32_t page_tokens;     /* KV page size in tokens (16) */
    float rms_eps;
    double rope_theta;
    int32_t tied_embeddings; /* 1: the LM head is the embedding table */
    int32_t qkv_bias;        /* 1: bq, bk, bv are present (added before RoPE) */
    int32_t weight_format;   /* WICI_WEIGHTS_BF16, or WICI_WEIGHTS_Q8: the seven per-layer
                                matrices in the 8-bit block format (see wici_load_weights_q8) */
    int32_t qk_norm;         /* 1: Qwen3 block: each head of q and of k is RMS-normalised over
                                head_dim with its own gain ("layers.<l>.q_norm" / ".k_norm",
                                [1, head_dim]) before RoPE (the paper's models are Qwen3,
                                Sec. 5.1, Tab. 1) */
    int32_t max_sms;         /* SM share: the context's kernels use at most this many SMs
                                (0: all).  Several contexts whose shares add up to at most
                                the GPU's SM count decode concurrently, each on its own
                                stream (Sec. 5.4, multiple clients; Sec. 7, task scheduling:
                                the caller's stream priorities order the tenants). */
} wici_config;

/* Storage format of the per-layer matrices wq, wk, wv, wo, wg, wu, wd.  The
 * embedding, norms, biases and LM head are bf16 in both. */
enum { WICI_WEIGHTS_BF16 = 0, WICI_WEIGHTS_Q8 = 1 };

/* Device bytes the caller allocates (each buffer 256-byte aligned). */
typedef struct wici_sizes {
    size_t weight_bytes;     /* packed bf16 weight arena */
    size_t kv_bytes;         /* paged bf16 K/V pool: [layer][page][K|V][kv_head][16][head_dim] */
    size_t workspace_bytes;  /* activations, partials, RoPE table, page table, control words */
} wici_sizes;

/* One named weight tensor, bf16 row-major [rows, cols].  Names:
 *   "embed" [vocab, hidden]; "final_norm" [1, hidden]; "lm_head" [vocab, hidden] (untied);
 *   "layers.<l>.attn_norm" [1, hidden]; "layers.<l>.wq" [n_q*d, hidden];
 *   "layers.<l>.wk" / ".wv" [n_kv*d, hidden]; "layers.<l>.bq" [1, n_q*d] and
 *   ".bk" / ".bv" [1, n_kv*d] (qkv_bias only); "layers.<l>.wo" [hidden, n_q*d];
 *   "layers.<l>.ffn_norm" [1, hidden]; "layers.<l>.wg" / ".wu" [ffn, hidden];
 *   "layers.<l>.wd" [hidden, ffn]; "layers.<l>.q_norm" / ".k_norm" [1, head_dim] (qk_norm only).
 * `data` is a host pointer (on_device = 0) or a device pointer (on_device = 1);
 * it is read during the call and not kept.  The paper's frameworks load a model
 * "tensor by tensor" (Sec. 4.1); so does this call. */
typedef struct wici_tensor {
    const char *name;
    const void *data;
    int64_t rows, cols;
    int32_t on_device;
} wici_tensor;

/* Sizes of the three caller-owned device buffers for `cfg`.  WICI_E_ARG on an
 * invalid configuration.  (Sec. 3.2, context management: the application's
 * own memory on the server's native CUDA context holds the model; here the
 * caller allocates it, the library only lays it out.) */
int wici_get_sizes(const wici_config *cfg, wici_sizes *out);

/* Create a context on the current CUDA device (Sec. 3.2: each client is served
 * by its own server thread on the native CUDA context; one wici_ctx per
 * client thread).  `cuda_stream` (a cudaStream_t,
 * may be NULL for the legacy stream) orders every launch of this context; the
 * three buffers must be at least wici_get_sizes() bytes and 256-byte aligned.
 * The KV page table starts as the identity.  *out receives the context. */
int wici_create(const wici_config *cfg, void *cuda_stream, void *weight_dev, void *kv_dev,
                void *workspace_dev, wici_ctx **out);

/* Copy `n` named tensors into the packed weight arena (rows of Wq/Wk are paired
 * for RoPE, Wg/Wu rows are interleaved, Wq/Wk/Wv are concatenated).  May be
 * called several times; prefill/decode require every tensor to have been loaded. */
int wici_load_weights(wici_ctx *ctx, const wici_tensor *t, int32_t n);

/* One per-layer matrix in the 8-bit block format, GGUF-style (the paper's
 * models are GGUF files at about 8.5 bits per parameter, Sec. 5.1 and Tab. 1):
 * row r of a [rows, cols] matrix is cut into blocks of 32 consecutive input
 * columns; block b holds 32 int8 codes (two's complement, in [-127, 127]) and
 * one fp16 scale d[r][b], and stands for W[r][c] = d[r][c / 32] * code[r][c].
 *   codes   int8 [rows, cols], row-major;   scales  fp16 bits [rows, cols / 32]
 * Names and shapes are those of wici_tensor's per-layer matrices ("layers.<l>.wq",
 * ".wk", ".wv", ".wo", ".wg", ".wu", ".wd").  `codes` and `scales` are host
 * (on_device = 0) or device (on_device = 1) pointers, read during the call. */
typedef struct wici_q8_tensor {
    const char *name;
    const void *codes;
    const void *scales;
    int64_t rows, cols;
    int32_t on_device;
} wici_q8_tensor;

/* Copy `n` matrices in the 8-bit block format into the weight arena of a
 * context created with weight_format = WICI_WEIGHTS_Q8 (the row pairings of
 * wici_load_weights apply; each row's codes and scales are stored side by
 * side).  Such a context takes the seven per-layer matrices only through this
 * call, and the other tensors through wici_load_weights.  WICI_E_ARG for a
 * bf16 context, an unknown name or a wrong shape; nothing is copied then.
 * Constraints of the format here: hidden, ffn_dim and n_q_heads*head_dim
 * multiples of 256. */
int wici_load_weights_q8(wici_ctx *ctx, const wici_q8_tensor *t, int32_t n);

/* Append `n` >= 1 host tokens at positions kv_len..kv_len+n-1 (Sec. 5.1 TTFT
 * path; a later call after decode steps is a chunked prefill onto the live cache).
 * logits_out (nullable, host float[vocab]) receives the last position's logits;
 * token_out (nullable) its greedy token.  WICI_E_CAPACITY if kv_len+n > max_tokens,
 * WICI_E_ARG if a token is outside [0, vocab). */
int wici_prefill(wici_ctx *ctx, const int32_t *tokens, int32_t n, float *logits_out,
                 int32_t *token_out);

/* One decode step: feed `token_in` (>= 0), or the last greedy token when
 * token_in < 0, at position kv_len; kv_len += 1.  Outputs as for wici_prefill.
 * Runs the captured CUDA graph of the whole step.  WICI_E_STATE before the
 * first prefill.  (T_Local of Eq. 1, Sec. 3.3: the GPU time of one generated
 * token; Sec. 4.2.2, trace replay: every token repeats the same computation
 * with only the input token changing, so one recorded graph is replayed.) */
int wici_decode_step(wici_ctx *ctx, int32_t token_in, float *logits_out, int32_t *token_out);

/* Sec. 4.2.2 (trace replay without a round trip per token):
 * `n_steps` greedy decode steps back to back on the device (each step feeds
 * the previous step's argmax; the first feeds token_in, or the last greedy
 * token if token_in < 0).  tokens_out (nullable, host int32[n_steps]) receives
 * the generated tokens. */
int wici_decode(wici_ctx *ctx, int32_t n_steps, int32_t token_in, int32_t *tokens_out);

/* Forget the cached tokens (kv_len := 0); weights stay loaded.  (Sec. 5.1:
 * every evaluated sample is a new request on the already loaded model.) */
int wici_reset(wici_ctx *ctx);

/* Replace the logical->physical KV page map (host int32[n], n = max_tokens/16
 * rounded up, a permutation of 0..n-1).  Only valid when kv_len == 0.  The
 * paper has no counterpart: the paged cache is this library's layout. */
int wici_set_page_table(wici_ctx *ctx, const int32_t *pages, int32_t n);

/* Number of cached positions, or a negative status (bookkeeping; no paper
 * counterpart). */
int32_t wici_kv_len(const wici_ctx *ctx);

/* Message of the last error on ctx (or of this thread when ctx is NULL). */
const char *wici_last_error(const wici_ctx *ctx);

/* Measurement of T_Local (Eq. 1, Sec. 3.3) per kernel.
 * Per-kernel timing of `n_steps` decode steps run as individual launches, each
 * bracketed by CUDA events on the context's stream (for roofline accounting).
 * For each kernel kind i < *n_kinds: names[i] (static string), launches[i] and
 * total_ms[i].  Arrays have room for `cap` entries.  Advances kv_len by n_steps
 * like wici_decode.  Where the step runs as one persistent kernel there is a
 * single kind, "decode_step"; otherwise one kind per layer operation
 * ("qkv_rope_kvappend", "flash_decode", "o_proj_residual", "gate_up_swiglu",
 * "down_residual") plus "lm_head_argmax". */
int wici_profile_decode(wici_ctx *ctx, int32_t n_steps, const char **names, int32_t *launches,
                        double *total_ms, int32_t cap, int32_t *n_kinds);

/* Measurement of the prefill's kernels (Sec. 5.1, TTFT), like wici_profile_decode:
 * appends the n host tokens exactly as wici_prefill does (kv_len += n), with
 * every launch bracketed by CUDA events on the context's stream.  For each
 * kernel kind i < *n_kinds: names[i] ("prefill_qkv", "prefill_attention",
 * "prefill_o_proj", "prefill_gate_up", "prefill_down", ...; static strings),
 * launches[i] and total_ms[i].  Arrays have room for `cap` entries. */
int wici_profile_prefill(wici_ctx *ctx, const int32_t *tokens, int32_t n, const char **names, int32_t *launches,
                         double *total_ms, int32_t cap, int32_t *n_kinds);

/* Failure detection (no paper counterpart).
 * Self-test of the bounded device wait: launches one CTA that waits on an
 * mbarrier nobody arrives at, giving up after `limit_ns` nanoseconds.  Returns
 * WICI_E_TIMEOUT when the wait gave up as designed (the expected result). */
int wici_check_bounded_wait(void *cuda_stream, int64_t limit_ns);

/* Final RMSNorm + LM head + greedy argmax of one hidden vector, for callers
 * that cannot allocate device memory.  The paper has no counterpart: WiCi's
 * GPU work runs inside the application's own allocations.
 *
 * Who needs it: a caller whose device memory is owned by someone else, e.g.
 * an engine or framework that hands out every byte from its own pool and
 * forbids side allocations, or a latency-critical thread where cudaMalloc's
 * possible implicit synchronisation or failure cannot be afforded.  Such a
 * caller can still pass its input and output buffers, but cannot give the
 * kernel scratch space; here the scratch (control words and one argmax
 * partial per CTA, about 9 KB) is a fixed array compiled into the library,
 * which every GPU that loads the library keeps until the process exits.
 *
 *   lm_head_dev    device bf16 [vocab, hidden], row-major (y = W x)
 *   norm_gain_dev  device bf16 [hidden], final RMSNorm gain
 *   x_dev          device fp32 [hidden], the hidden vector
 *   logits_dev     device fp32 [vocab], receives W . RMSNorm(x)
 *   token_dev      device int32 [1], receives the argmax (lowest index on ties)
 * All work is enqueued on cuda_stream (a cudaStream_t, NULL for the legacy
 * stream); the call does not synchronise.  The device is the current one.
 * The call returns before the GPU has run, so a device-side failure cannot
 * reach its return code: if a bounded wait inside the kernel gives up,
 * *token_dev receives -1 instead of a vocabulary index, and the logits are
 * then incomplete.  Check the token for -1 before using either output.
 * Limits: hidden a multiple of 8 in [8, 16384]; vocab >= 1; the current GPU
 * may have at most 1024 SMs (one scratch partial per CTA); anything else
 * returns WICI_E_ARG with the reason in wici_last_error(NULL).
 * The call allocates nothing: no cudaMalloc, no cudaFree, no allocating
 * library routine.  The first call on a device looks up the scratch array's
 * device address for that device (make that first call before any stream
 * capture).  Calls share the one scratch array, which keeps the last call's
 * contents (the ticket word is cleared at the start of every call), so calls
 * that can overlap on the GPU race: order them on one stream. */
int wici_lm_head_argmax_noalloc(void *cuda_stream, const void *lm_head_dev, const void *norm_gain_dev,
                                const float *x_dev, int32_t hidden, int32_t vocab, float rms_eps,
                                float *logits_dev, int32_t *token_dev);

/* ---------------------------------------------------------------------------
 * CNN-training sample (Sec. 5.4, "Multiple applications": NVIDIA's CNN training
 * sample, input 4 x 1024 x 224 x 224, 3x3 filter, stride 2).  One convolution
 * layer, 3x3, stride 2, zero padding 1 (readings: padding 1, no bias), forward
 * and the two gradients of backpropagation, on the tensor cores.  Channels last,
 * row-major, device pointers, 16-byte aligned:
 *   x  bf16 [n][h][w][c]      w  bf16 [k][3][3][c]     dy bf16 [n][h/2][w/2][k]
 *   y  fp32 [n][h/2][w/2][k]  dx fp32 [n][h][w][c]     dw fp32 [k][3][3][c]
 * Constraints: c and k multiples of 256; h and w even; n >= 1 (else WICI_E_ARG,
 * message in wici_last_error(NULL)).  Each call is enqueued on cuda_stream and
 * returns without synchronising; `workspace` (wici_conv_workspace_bytes, zeroed
 * once by the caller before its first use) holds the error word and, for the
 * data gradient, the transposed filter.  Calls sharing a workspace must be
 * ordered on one stream. */
typedef struct wici_conv_shape {
    int32_t n, c, h, w, k;
} wici_conv_shape;

/* Bytes of the workspace for `s`. */
int wici_conv_workspace_bytes(const wici_conv_shape *s, size_t *bytes);

/* y[pix][k] = sum over taps and c of x at (2p + r - 1, 2q + s - 1) times w[k][r][s][c]. */
int wici_conv_forward(void *cuda_stream, const wici_conv_shape *s, const void *x, const void *w, float *y,
                      void *workspace);

/* dx = the gradient of sum(y * dy) with respect to x. */
int wici_conv_backward_data(void *cuda_stream, const wici_conv_shape *s, const void *dy, const void *w, float *dx,
                            void *workspace);

/* dw = the gradient of sum(y * dy) with respect to w. */
int wici_conv_backward_filter(void *cuda_stream, const wici_conv_shape *s, const void *x, const void *dy, float *dw,
                              void *workspace);

/* Synchronises cuda_stream and reports whether a bounded device wait of an
 * earlier convolution call on `workspace` gave up (WICI_E_TIMEOUT; the word is
 * then cleared) or not (WICI_OK). */
int wici_conv_status(void *cuda_stream, void *workspace);

/* Destroy the context (frees only what the library allocated).  (Sec. 5.4,
 * multiple clients: a client that disconnects releases its server thread.) */
void wici_destroy(wici_ctx *ctx);

#ifdef __cplusplus
}
#endif

#endif /* WICI_H */
