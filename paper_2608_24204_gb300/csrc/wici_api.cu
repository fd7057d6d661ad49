// C ABI (include/wici.h): buffer plan, weight packing, prefill and decode
// orchestration, CUDA-graph capture of the decode step.
#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <string>
#include <vector>

#include "../../include/wici.h"
#include "common.cuh"
#include "kernels.h"

using namespace wici;

static thread_local std::string g_thread_err;

// lets other translation units report an error for wici_last_error(NULL)
void wici::set_thread_error(const char *msg) { g_thread_err = msg; }

struct wici_ctx {
    Plan plan;
    Bufs bufs;
    cudaStream_t stream = nullptr;
    int device = 0;
    int32_t kv_len = 0;
    bool prefilled = false;          // a greedy token exists to feed
    std::vector<char> loaded;        // per canonical tensor
    int n_required = 0, n_loaded = 0;
    cudaGraphExec_t step_exec = nullptr;
    cudaEvent_t step_done[2] = {nullptr, nullptr};  // SM-share contexts: after every decode step
    long long steps_launched = 0;
    PrefillMaps maps;
    int32_t *pinned = nullptr;       // host staging: [0] token in, [1] token out, [2] err
    std::string err;
};

// --------------------------------------------------------------- helpers ----
static int fail(wici_ctx *c, int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c)
        c->err = buf;
    else
        g_thread_err = buf;
    return code;
}

#define CUDA_TRY(c, call)                                                                  \
    do {                                                                                   \
        cudaError_t e_ = (call);                                                           \
        if (e_ != cudaSuccess)                                                             \
            return fail((c), WICI_E_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_)); \
    } while (0)

static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

const char *wici::make_plan(const wici_config *cfg, int num_sms, Plan *p) {
    if (!cfg) return "null config";
    const wici_config &c = *cfg;
    if (c.n_layers < 1 || c.hidden < 8 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.ffn_dim < 8 ||
        c.vocab < 1 || c.max_tokens < 1)
        return "non-positive dimension";
    if (c.head_dim != 64 && c.head_dim != 128) return "head_dim must be 64 or 128";
    if (c.hidden % 8 || c.ffn_dim % 8) return "hidden and ffn_dim must be multiples of 8";
    // one GEMV unit (two rows of K = hidden, or one row of K = ffn_dim / n_q*d)
    // must fit one 32 KB ring stage
    if (c.hidden > 8192 || c.ffn_dim > 16384 || c.n_q_heads * c.head_dim > 16384)
        return "hidden must be <= 8192; ffn_dim and n_q_heads*head_dim <= 16384";
    if (c.n_q_heads % c.n_kv_heads) return "n_q_heads must be a multiple of n_kv_heads";
    if (c.n_q_heads / c.n_kv_heads > 8) return "at most 8 query heads per KV head";
    if (c.n_kv_heads > 64) return "at most 64 KV heads";
    if (c.page_tokens != kPage) return "page_tokens must be 16";
    if (c.max_chunk < 1 || c.max_chunk > c.max_tokens) return "max_chunk must be in [1, max_tokens]";
    if (!(c.rms_eps > 0.f) || !(c.rope_theta > 1.0)) return "rms_eps > 0 and rope_theta > 1 required";
    if (c.qkv_bias != 0 && c.qkv_bias != 1) return "qkv_bias must be 0 or 1";
    if (c.tied_embeddings != 0 && c.tied_embeddings != 1) return "tied_embeddings must be 0 or 1";
    if (c.max_sms < 0) return "max_sms must be >= 0 (0: every SM)";
    if (c.qk_norm != 0 && c.qk_norm != 1) return "qk_norm must be 0 or 1";
    if (c.weight_format != WICI_WEIGHTS_BF16 && c.weight_format != WICI_WEIGHTS_Q8)
        return "weight_format must be WICI_WEIGHTS_BF16 or WICI_WEIGHTS_Q8";
    if (c.weight_format == WICI_WEIGHTS_Q8 &&
        (c.hidden % 256 || c.ffn_dim % 256 || (c.n_q_heads * c.head_dim) % 256))
        return "the 8-bit block format needs hidden, ffn_dim and n_q_heads*head_dim multiples of 256";

    Plan &P = *p;
    P.cfg = c;
    P.L = c.n_layers; P.H = c.hidden; P.F = c.ffn_dim; P.V = c.vocab;
    P.nq = c.n_q_heads; P.nkv = c.n_kv_heads; P.d = c.head_dim;
    P.qdim = P.nq * P.d; P.kvdim = P.nkv * P.d; P.nqkv = P.qdim + 2 * P.kvdim;
    P.group = P.nq / P.nkv;
    P.max_pages = (c.max_tokens + kPage - 1) / kPage;
    P.max_chunk = c.max_chunk;
    P.num_sms = num_sms > 0 ? num_sms : 1;
    if (c.max_sms > 0 && c.max_sms < P.num_sms) P.num_sms = c.max_sms;   // this tenant's SM share
    P.q8 = c.weight_format == WICI_WEIGHTS_Q8;
    P.qk_norm = c.qk_norm == 1;

    // weight arena: every tensor starts on a 128-byte boundary
    size_t off = 0;
    auto take = [&](size_t elems) { size_t o = off; off = align_up(off + elems, 64); return o; };
    const size_t H = P.H, F = P.F, V = P.V;
    // a per-layer matrix [rows, K]: bf16, or rows of the 8-bit block format (in bf16 units)
    auto mat = [&](size_t rows, size_t K) { return P.q8 ? rows * q8_row_bytes(K) / 2 : rows * K; };
    P.w_embed = take(V * H);
    P.layer.resize(P.L);
    for (int l = 0; l < P.L; ++l) {
        LayerOffsets &lo = P.layer[l];
        lo.attn_norm = take(H);
        lo.wqkv = take(mat(P.nqkv, H));
        lo.bqkv = c.qkv_bias ? take((size_t)P.nqkv) : 0;
        lo.qn = P.qk_norm ? take((size_t)P.d) : 0;
        lo.kn = P.qk_norm ? take((size_t)P.d) : 0;
        lo.wo = take(mat(H, P.qdim));
        lo.ffn_norm = take(H);
        lo.wgu = take(mat(2 * F, H));
        lo.wd = take(mat(H, F));
    }
    P.w_final_norm = take(H);
    P.w_lm = c.tied_embeddings ? P.w_embed : take(V * H);
    P.weight_elems = off;

    P.kv_page_elems = (size_t)2 * P.nkv * kPage * P.d;
    P.kv_layer_elems = P.kv_page_elems * P.max_pages;
    P.kv_elems = P.kv_layer_elems * P.L;


    size_t w = 0;
    auto ws = [&](size_t bytes) { size_t o = w; w = align_up(w + bytes, 256); return o; };
    const size_t T = (size_t)P.max_chunk;
    P.ws_ctrl = ws(CTRL_WORDS * sizeof(int));
    P.ws_hist = ws(((size_t)c.max_tokens + 1) * sizeof(int));
    P.ws_x = ws(H * 4);
    P.ws_q = ws((size_t)P.qdim * 4);
    P.ws_o = ws((size_t)P.qdim * 4);
    P.ws_m = ws(F * 4);
    P.ws_logits = ws(V * 4);
    P.ws_amax = ws((size_t)P.num_sms * sizeof(int2));
    P.ws_fd_part = ws(fd_part_floats(P.nkv, P.group, P.d, P.max_pages) * sizeof(float));
    P.ws_mega_bound = ws(((size_t)P.num_sms + 1) * sizeof(uint32_t));
    P.ws_mega_time = ws((size_t)P.num_sms * sizeof(float));
    P.ws_rope = ws((size_t)c.max_tokens * (P.d / 2) * sizeof(float2));
    P.ws_pages = ws((size_t)P.max_pages * 4);
    P.ws_tok = ws(T * 4);
    P.ws_X = ws(T * H * 4);
    for (int t = 0; t < kTerms; ++t) {
        P.ws_Q[t] = ws(T * P.qdim * 2);
        P.ws_A[t] = ws(T * H * 2);
        P.ws_O[t] = ws(T * P.qdim * 2);
        P.ws_M[t] = ws(T * F * 2);
    }
    P.wt_elems = 0;
    for (size_t e : {(size_t)P.nqkv * H, H * (size_t)P.qdim, 2 * F * H, H * F}) P.wt_elems = e > P.wt_elems ? e : P.wt_elems;
    for (int t = 0; t < kTerms; ++t) P.ws_Wt[t] = P.q8 ? ws(P.wt_elems * 2) : 0;
    P.ws_kraw = P.qk_norm ? ws((size_t)P.kvdim * 4) : 0;
    P.ws_QKraw = P.qk_norm ? ws(T * (size_t)(P.qdim + P.kvdim) * 4) : 0;
    P.ws_bytes = w;
    return nullptr;
}

static Bufs make_bufs(const Plan &p, void *W, void *KV, void *WS) {
    Bufs b;
    uint8_t *ws = (uint8_t *)WS;
    b.W = (uint16_t *)W;
    b.KV = (uint16_t *)KV;
    b.ctrl = (int *)(ws + p.ws_ctrl);
    b.hist = (int *)(ws + p.ws_hist);
    b.x = (float *)(ws + p.ws_x);
    b.q = (float *)(ws + p.ws_q);
    b.o = (float *)(ws + p.ws_o);
    b.m = (float *)(ws + p.ws_m);
    b.logits = (float *)(ws + p.ws_logits);
    b.amax = (int2 *)(ws + p.ws_amax);
    b.fd_part = (float *)(ws + p.ws_fd_part);
    b.mega_bound = (uint32_t *)(ws + p.ws_mega_bound);
    b.mega_time = (float *)(ws + p.ws_mega_time);
    b.rope = (float2 *)(ws + p.ws_rope);
    b.pages = (int *)(ws + p.ws_pages);
    b.tok = (int *)(ws + p.ws_tok);
    b.X = (float *)(ws + p.ws_X);
    for (int t = 0; t < kTerms; ++t) {
        b.Q[t] = (uint16_t *)(ws + p.ws_Q[t]);
        b.A[t] = (uint16_t *)(ws + p.ws_A[t]);
        b.O[t] = (uint16_t *)(ws + p.ws_O[t]);
        b.M[t] = (uint16_t *)(ws + p.ws_M[t]);
        b.Wt[t] = p.q8 ? (uint16_t *)(ws + p.ws_Wt[t]) : nullptr;
    }
    b.kraw = p.qk_norm ? (float *)(ws + p.ws_kraw) : nullptr;
    b.QKraw = p.qk_norm ? (float *)(ws + p.ws_QKraw) : nullptr;
    return b;
}

// canonical tensor index of a name, or -1; fills rows/cols expected and the layer
struct TensorSlot { int kind; int layer; int64_t rows, cols; };
enum { T_EMBED, T_FINAL_NORM, T_LM_HEAD, T_ATTN_NORM, T_WQ, T_WK, T_WV, T_BQ, T_BK, T_BV, T_WO,
       T_FFN_NORM, T_WG, T_WU, T_WD, T_QN, T_KN, T_KINDS };
static const char *kLayerNames[] = {nullptr, nullptr, nullptr, "attn_norm", "wq", "wk", "wv", "bq",
                                    "bk", "bv", "wo", "ffn_norm", "wg", "wu", "wd", "q_norm", "k_norm"};
static const int kLayerKinds = 14;  // T_ATTN_NORM .. T_KN

static bool parse_name(const Plan &p, const char *name, TensorSlot *s) {
    const int64_t H = p.H, F = p.F, V = p.V;
    if (!strcmp(name, "embed")) { *s = {T_EMBED, -1, V, H}; return true; }
    if (!strcmp(name, "final_norm")) { *s = {T_FINAL_NORM, -1, 1, H}; return true; }
    if (!strcmp(name, "lm_head")) {
        if (p.cfg.tied_embeddings) return false;
        *s = {T_LM_HEAD, -1, V, H};
        return true;
    }
    if (strncmp(name, "layers.", 7)) return false;
    char *end = nullptr;
    long l = strtol(name + 7, &end, 10);
    if (end == name + 7 || *end != '.' || l < 0 || l >= p.L) return false;
    const char *leaf = end + 1;
    for (int k = T_ATTN_NORM; k < T_KINDS; ++k) {
        if (strcmp(leaf, kLayerNames[k])) continue;
        if ((k == T_BQ || k == T_BK || k == T_BV) && !p.cfg.qkv_bias) return false;
        if ((k == T_QN || k == T_KN) && !p.qk_norm) return false;
        int64_t r = 0, c = 0;
        switch (k) {
            case T_ATTN_NORM: case T_FFN_NORM: r = 1; c = H; break;
            case T_WQ: r = p.qdim; c = H; break;
            case T_WK: case T_WV: r = p.kvdim; c = H; break;
            case T_BQ: r = 1; c = p.qdim; break;
            case T_BK: case T_BV: r = 1; c = p.kvdim; break;
            case T_WO: r = H; c = p.qdim; break;
            case T_WG: case T_WU: r = F; c = H; break;
            case T_WD: r = H; c = F; break;
            case T_QN: case T_KN: r = 1; c = p.d; break;
        }
        *s = {k, (int)l, r, c};
        return true;
    }
    return false;
}

static bool is_q8_kind(int kind) {
    return kind == T_WQ || kind == T_WK || kind == T_WV || kind == T_WO || kind == T_WG || kind == T_WU ||
           kind == T_WD;
}

static int slot_index(const Plan &p, const TensorSlot &s) {
    if (s.layer < 0) return s.kind;  // 0..2
    return 3 + s.layer * kLayerKinds + (s.kind - T_ATTN_NORM);
}

// copy `rows` rows of `cols` bf16 from src (row pitch cols) to dst with row pitch dpitch_elems
static cudaError_t copy_rows(uint16_t *dst, size_t dpitch_elems, const uint16_t *src, int64_t rows,
                             int64_t cols, size_t spitch_elems, cudaStream_t st) {
    return cudaMemcpy2DAsync(dst, dpitch_elems * 2, src, spitch_elems * 2, (size_t)cols * 2,
                             (size_t)rows, cudaMemcpyDefault, st);
}

// Wq/Wk rows (and biases): for each head, rows i and i + d/2 become adjacent rows 2i, 2i+1
static cudaError_t copy_rope_paired(uint16_t *dst, const uint16_t *src, int heads, int d, int64_t cols,
                                    cudaStream_t st) {
    const int half = d / 2;
    for (int h = 0; h < heads; ++h) {
        const uint16_t *s = src + (size_t)h * d * cols;
        uint16_t *t = dst + (size_t)h * d * cols;
        cudaError_t e = copy_rows(t, 2 * cols, s, half, cols, cols, st);
        if (e != cudaSuccess) return e;
        e = copy_rows(t + cols, 2 * cols, s + (size_t)half * cols, half, cols, cols, st);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// ------------------------------------------------------------------ ABI ----
extern "C" {

int wici_get_sizes(const wici_config *cfg, wici_sizes *out) {
    if (!cfg || !out) return fail(nullptr, WICI_E_ARG, "null argument");
    Plan p;
    int nsm = 152;
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0) nsm = v;
    } else {
        cudaGetLastError();
    }
    if (const char *m = make_plan(cfg, nsm, &p)) return fail(nullptr, WICI_E_ARG, "config: %s", m);
    out->weight_bytes = p.weight_elems * 2;
    out->kv_bytes = p.kv_elems * 2;
    out->workspace_bytes = p.ws_bytes;
    return WICI_OK;
}

int wici_create(const wici_config *cfg, void *cuda_stream, void *weight_dev, void *kv_dev,
                void *workspace_dev, wici_ctx **out) {
    if (!cfg || !out || !weight_dev || !kv_dev || !workspace_dev)
        return fail(nullptr, WICI_E_ARG, "null argument");
    if (((uintptr_t)weight_dev | (uintptr_t)kv_dev | (uintptr_t)workspace_dev) & 255)
        return fail(nullptr, WICI_E_ARG, "device buffers must be 256-byte aligned");
    *out = nullptr;
    int dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return fail(nullptr, WICI_E_CUDA, "no CUDA device: %s", cudaGetErrorString(e));
    wici_ctx *c = new wici_ctx();
    if (const char *m = make_plan(cfg, nsm, &c->plan)) {
        delete c;
        return fail(nullptr, WICI_E_ARG, "config: %s", m);
    }
    if (c->plan.qk_norm && !decode_is_persistent(c->plan)) {
        delete c;
        return fail(nullptr, WICI_E_ARG,
                    "config: the per-head q/k norm is built into the one-launch decode step, which needs "
                    "n_q_heads * head_dim == hidden and an instantiated width");
    }
    if (c->plan.q8 && !decode_is_persistent(c->plan)) {
        delete c;
        return fail(nullptr, WICI_E_ARG,
                    "config: the 8-bit block format is built for hidden 4096 / ffn 14336 (head_dim 128) and for "
                    "hidden, ffn below 2048 (head_dim 64), with n_q_heads * head_dim == hidden");
    }
    c->device = dev;
    c->stream = (cudaStream_t)cuda_stream;
    c->bufs = make_bufs(c->plan, weight_dev, kv_dev, workspace_dev);
    const Plan &p = c->plan;
    c->loaded.assign(3 + (size_t)p.L * kLayerKinds, 0);
    c->n_required = 2 + (p.cfg.tied_embeddings ? 0 : 1) + p.L * (9 + (p.cfg.qkv_bias ? 3 : 0) + (p.qk_norm ? 2 : 0));
    int rc = WICI_OK;
    do {
        if ((e = setup_kernels()) != cudaSuccess) break;
        if ((e = cudaHostAlloc((void **)&c->pinned, 64, cudaHostAllocDefault)) != cudaSuccess) break;
        if (p.cfg.max_sms > 0 &&
            ((e = cudaEventCreateWithFlags(&c->step_done[0], cudaEventDisableTiming)) != cudaSuccess ||
             (e = cudaEventCreateWithFlags(&c->step_done[1], cudaEventDisableTiming)) != cudaSuccess))
            break;
        if ((e = cudaMemsetAsync(c->bufs.ctrl, 0, CTRL_WORDS * sizeof(int), c->stream)) != cudaSuccess) break;
        // cache slots past the length are read (and weighted by zero) by the
        // tensor-core attention: they must hold finite values from the start
        if ((e = cudaMemsetAsync(c->bufs.KV, 0, p.kv_elems * 2, c->stream)) != cudaSuccess) break;
        {   // even row shares to start with; the decode kernel refines them step by step
            std::vector<uint32_t> bound(p.num_sms + 1);
            for (int i = 0; i <= p.num_sms; ++i)
                bound[i] = (uint32_t)(((unsigned long long)i << 24) / (unsigned long long)p.num_sms);
            if ((e = cudaMemcpy(c->bufs.mega_bound, bound.data(), bound.size() * sizeof(uint32_t),
                                cudaMemcpyHostToDevice)) != cudaSuccess)
                break;
            if ((e = cudaMemsetAsync(c->bufs.mega_time, 0, (size_t)p.num_sms * sizeof(float), c->stream)) !=
                cudaSuccess)
                break;
        }
        std::vector<int> pages(p.max_pages);
        for (int i = 0; i < p.max_pages; ++i) pages[i] = i;
        if ((e = cudaMemcpyAsync(c->bufs.pages, pages.data(), pages.size() * 4, cudaMemcpyHostToDevice,
                                 c->stream)) != cudaSuccess)
            break;
        if ((e = enqueue_rope_table(p, c->bufs, c->stream)) != cudaSuccess) break;
        if (const char *m = make_prefill_maps(p, c->bufs, &c->maps)) {
            int rc2 = fail(nullptr, WICI_E_CUDA, "create: %s", m);
            wici_destroy(c);
            return rc2;
        }
        e = cudaStreamSynchronize(c->stream);
    } while (0);
    if (e != cudaSuccess) {
        rc = fail(nullptr, WICI_E_CUDA, "create: %s", cudaGetErrorString(e));
        wici_destroy(c);
        return rc;
    }
    *out = c;
    return WICI_OK;
}

int wici_load_weights(wici_ctx *c, const wici_tensor *t, int32_t n) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (!t || n < 0) return fail(c, WICI_E_ARG, "bad tensor list");
    const Plan &p = c->plan;
    // validate everything first: nothing is copied when one entry is wrong
    for (int i = 0; i < n; ++i) {
        TensorSlot s;
        if (!t[i].name || !t[i].data) return fail(c, WICI_E_ARG, "tensor %d: null name or data", i);
        if (!parse_name(p, t[i].name, &s)) return fail(c, WICI_E_ARG, "unknown tensor name '%s'", t[i].name);
        if (p.q8 && is_q8_kind(s.kind))
            return fail(c, WICI_E_ARG, "'%s' is in the 8-bit block format here: load it with wici_load_weights_q8",
                        t[i].name);
        if (t[i].rows != s.rows || t[i].cols != s.cols)
            return fail(c, WICI_E_ARG, "tensor '%s': shape [%lld, %lld], expected [%lld, %lld]", t[i].name,
                        (long long)t[i].rows, (long long)t[i].cols, (long long)s.rows, (long long)s.cols);
    }
    uint16_t *W = c->bufs.W;
    const int64_t H = p.H;
    for (int i = 0; i < n; ++i) {
        TensorSlot s;
        parse_name(p, t[i].name, &s);
        const uint16_t *src = (const uint16_t *)t[i].data;
        cudaError_t e = cudaSuccess;
        if (s.layer < 0) {
            const size_t dst = s.kind == T_EMBED ? p.w_embed : s.kind == T_FINAL_NORM ? p.w_final_norm : p.w_lm;
            e = cudaMemcpyAsync(W + dst, src, (size_t)s.rows * s.cols * 2, cudaMemcpyDefault, c->stream);
        } else {
            const LayerOffsets &lo = p.layer[s.layer];
            switch (s.kind) {
                case T_ATTN_NORM:
                    e = cudaMemcpyAsync(W + lo.attn_norm, src, H * 2, cudaMemcpyDefault, c->stream); break;
                case T_FFN_NORM:
                    e = cudaMemcpyAsync(W + lo.ffn_norm, src, H * 2, cudaMemcpyDefault, c->stream); break;
                case T_WQ: e = copy_rope_paired(W + lo.wqkv, src, p.nq, p.d, H, c->stream); break;
                case T_WK:
                    e = copy_rope_paired(W + lo.wqkv + (size_t)p.qdim * H, src, p.nkv, p.d, H, c->stream);
                    break;
                case T_WV:
                    e = cudaMemcpyAsync(W + lo.wqkv + (size_t)(p.qdim + p.kvdim) * H, src,
                                        (size_t)p.kvdim * H * 2, cudaMemcpyDefault, c->stream);
                    break;
                case T_BQ: e = copy_rope_paired(W + lo.bqkv, src, p.nq, p.d, 1, c->stream); break;
                case T_BK: e = copy_rope_paired(W + lo.bqkv + p.qdim, src, p.nkv, p.d, 1, c->stream); break;
                case T_BV:
                    e = cudaMemcpyAsync(W + lo.bqkv + p.qdim + p.kvdim, src, (size_t)p.kvdim * 2,
                                        cudaMemcpyDefault, c->stream);
                    break;
                case T_WO:
                    e = cudaMemcpyAsync(W + lo.wo, src, (size_t)H * p.qdim * 2, cudaMemcpyDefault, c->stream);
                    break;
                case T_WG: e = copy_rows(W + lo.wgu, 2 * H, src, p.F, H, H, c->stream); break;
                case T_WU: e = copy_rows(W + lo.wgu + H, 2 * H, src, p.F, H, H, c->stream); break;
                case T_WD:
                    e = cudaMemcpyAsync(W + lo.wd, src, (size_t)H * p.F * 2, cudaMemcpyDefault, c->stream);
                    break;
                case T_QN: e = cudaMemcpyAsync(W + lo.qn, src, (size_t)p.d * 2, cudaMemcpyDefault, c->stream); break;
                case T_KN: e = cudaMemcpyAsync(W + lo.kn, src, (size_t)p.d * 2, cudaMemcpyDefault, c->stream); break;
            }
        }
        if (e != cudaSuccess) return fail(c, WICI_E_CUDA, "copy of '%s': %s", t[i].name, cudaGetErrorString(e));
        const int si = slot_index(p, s);
        if (!c->loaded[si]) {
            c->loaded[si] = 1;
            ++c->n_loaded;
        }
    }
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));
    return WICI_OK;
}

// Rows of one matrix in the 8-bit block format: codes and scales of source row
// r go to arena row dst_row(r) (codes first, then the K/32 scales); the RoPE
// pairing of wq/wk and the gate/up interleaving are the bf16 loader's.
static cudaError_t copy_q8_rows(uint8_t *dst, size_t drow_bytes, int dst_step, const uint8_t *codes,
                                const uint8_t *scales, int64_t rows, int64_t K, cudaStream_t st) {
    cudaError_t e = cudaMemcpy2DAsync(dst, drow_bytes * dst_step, codes, (size_t)K, (size_t)K, (size_t)rows,
                                      cudaMemcpyDefault, st);
    if (e != cudaSuccess) return e;
    return cudaMemcpy2DAsync(dst + K, drow_bytes * dst_step, scales, (size_t)K / 16, (size_t)K / 16, (size_t)rows,
                             cudaMemcpyDefault, st);
}

static cudaError_t load_q8(const Plan &p, uint16_t *W, const TensorSlot &s, const wici_q8_tensor &t,
                           cudaStream_t st) {
    const LayerOffsets &lo = p.layer[s.layer];
    const int64_t K = s.cols;
    const size_t rb = q8_row_bytes((size_t)K);
    uint8_t *base = nullptr;   // the matrix's first arena row
    int step = 1;              // arena rows per source row
    int64_t row0 = 0;          // first arena row of this tensor inside `base`
    switch (s.kind) {
        case T_WQ: base = (uint8_t *)(W + lo.wqkv); break;
        case T_WK: base = (uint8_t *)(W + lo.wqkv); row0 = p.qdim; break;
        case T_WV: base = (uint8_t *)(W + lo.wqkv); row0 = p.qdim + p.kvdim; break;
        case T_WO: base = (uint8_t *)(W + lo.wo); break;
        case T_WG: base = (uint8_t *)(W + lo.wgu); step = 2; break;
        case T_WU: base = (uint8_t *)(W + lo.wgu); step = 2; row0 = 1; break;
        case T_WD: base = (uint8_t *)(W + lo.wd); break;
    }
    const uint8_t *codes = (const uint8_t *)t.codes, *scales = (const uint8_t *)t.scales;
    cudaError_t e = cudaSuccess;
    if (s.kind == T_WQ || s.kind == T_WK) {
        // per head: rows i and i + d/2 become adjacent arena rows 2i, 2i + 1
        const int heads = (int)(s.rows / p.d), half = p.d / 2;
        for (int h = 0; h < heads && e == cudaSuccess; ++h) {
            uint8_t *dst = base + (size_t)(row0 + (int64_t)h * p.d) * rb;
            const size_t sr = (size_t)h * p.d;
            e = copy_q8_rows(dst, rb, 2, codes + sr * K, scales + sr * (K / 16), half, K, st);
            if (e == cudaSuccess)
                e = copy_q8_rows(dst + rb, rb, 2, codes + (sr + half) * K, scales + (sr + half) * (K / 16), half, K,
                                 st);
        }
    } else {
        e = copy_q8_rows(base + (size_t)row0 * rb, rb, step, codes, scales, s.rows, K, st);
    }
    return e;
}

int wici_load_weights_q8(wici_ctx *c, const wici_q8_tensor *t, int32_t n) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (!t || n < 0) return fail(c, WICI_E_ARG, "bad tensor list");
    const Plan &p = c->plan;
    if (!p.q8) return fail(c, WICI_E_ARG, "the context holds bf16 matrices (weight_format = WICI_WEIGHTS_BF16)");
    for (int i = 0; i < n; ++i) {
        TensorSlot s;
        if (!t[i].name || !t[i].codes || !t[i].scales)
            return fail(c, WICI_E_ARG, "tensor %d: null name, codes or scales", i);
        if (!parse_name(p, t[i].name, &s) || !is_q8_kind(s.kind))
            return fail(c, WICI_E_ARG, "'%s' is not a per-layer matrix of the 8-bit format", t[i].name);
        if (t[i].rows != s.rows || t[i].cols != s.cols)
            return fail(c, WICI_E_ARG, "tensor '%s': shape [%lld, %lld], expected [%lld, %lld]", t[i].name,
                        (long long)t[i].rows, (long long)t[i].cols, (long long)s.rows, (long long)s.cols);
    }
    for (int i = 0; i < n; ++i) {
        TensorSlot s;
        parse_name(p, t[i].name, &s);
        cudaError_t e = load_q8(p, c->bufs.W, s, t[i], c->stream);
        if (e != cudaSuccess) return fail(c, WICI_E_CUDA, "copy of '%s': %s", t[i].name, cudaGetErrorString(e));
        const int si = slot_index(p, s);
        if (!c->loaded[si]) {
            c->loaded[si] = 1;
            ++c->n_loaded;
        }
    }
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));
    return WICI_OK;
}

static int check_ready(wici_ctx *c) {
    if (c->n_loaded < c->n_required)
        return fail(c, WICI_E_STATE, "weights not loaded (%d of %d tensors)", c->n_loaded, c->n_required);
    return WICI_OK;
}

// read back token + error word, clear a set error, restore the device position
static int finish_call(wici_ctx *c, int32_t new_kv_len, int32_t *token_out) {
    CUDA_TRY(c, cudaMemcpyAsync(c->pinned + 1, c->bufs.ctrl + CTRL_TOKEN, 2 * sizeof(int),
                                cudaMemcpyDeviceToHost, c->stream));
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));
    const int errw = c->pinned[2];
    if (errw != 0) {
        c->pinned[3] = 0;
        c->pinned[4] = c->kv_len;
        cudaMemcpyAsync(c->bufs.ctrl + CTRL_ERR, c->pinned + 3, sizeof(int), cudaMemcpyHostToDevice, c->stream);
        cudaMemcpyAsync(c->bufs.ctrl + CTRL_POS, c->pinned + 4, sizeof(int), cudaMemcpyHostToDevice, c->stream);
        cudaMemsetAsync(c->bufs.ctrl + CTRL_LM_TICKET, 0, sizeof(int), c->stream);
        cudaMemsetAsync(c->bufs.ctrl + CTRL_GRID_BAR, 0, sizeof(int), c->stream);
        cudaMemsetAsync(c->bufs.ctrl + CTRL_ATTN_TICKET0, 0, 64 * sizeof(int), c->stream);
        cudaStreamSynchronize(c->stream);
        return fail(c, WICI_E_TIMEOUT, "a device-side wait gave up (site %d)", errw);
    }
    c->kv_len = new_kv_len;
    if (token_out) *token_out = c->pinned[1];
    return WICI_OK;
}

int wici_prefill(wici_ctx *c, const int32_t *tokens, int32_t n, float *logits_out, int32_t *token_out) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (!tokens || n < 1) return fail(c, WICI_E_ARG, "need n >= 1 tokens");
    if (int rc = check_ready(c)) return rc;
    const Plan &p = c->plan;
    if ((int64_t)c->kv_len + n > p.cfg.max_tokens)
        return fail(c, WICI_E_CAPACITY, "kv_len %d + %d tokens exceeds max_tokens %d", c->kv_len, n,
                    p.cfg.max_tokens);
    for (int i = 0; i < n; ++i)
        if (tokens[i] < 0 || tokens[i] >= p.V) return fail(c, WICI_E_ARG, "token %d out of range", tokens[i]);
    for (int off = 0; off < n; off += p.max_chunk) {
        const int T = n - off < p.max_chunk ? n - off : p.max_chunk;
        CUDA_TRY(c, cudaMemcpyAsync(c->bufs.tok, tokens + off, (size_t)T * 4, cudaMemcpyHostToDevice, c->stream));
        const bool last = off + T == n;
        CUDA_TRY(c, enqueue_prefill_chunk(p, c->bufs, c->maps, c->stream, c->kv_len + off, T, last ? n : 0, nullptr));
        if (!last) CUDA_TRY(c, cudaStreamSynchronize(c->stream));  // tok buffer is reused by the next chunk
    }
    if (logits_out)
        CUDA_TRY(c, cudaMemcpyAsync(logits_out, c->bufs.logits, (size_t)p.V * 4, cudaMemcpyDeviceToHost, c->stream));
    int rc = finish_call(c, c->kv_len + n, token_out);
    if (rc == WICI_OK) c->prefilled = true;
    return rc;
}

static int ensure_graph(wici_ctx *c) {
    if (c->step_exec) return WICI_OK;
    cudaStream_t cap;
    CUDA_TRY(c, cudaStreamCreateWithFlags(&cap, cudaStreamNonBlocking));
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamBeginCapture(cap, cudaStreamCaptureModeThreadLocal);
    if (e == cudaSuccess) {
        cudaError_t e2 = enqueue_decode_step(c->plan, c->bufs, cap, true, nullptr);
        e = cudaStreamEndCapture(cap, &g);
        if (e2 != cudaSuccess) e = e2;
    }
    if (e == cudaSuccess) e = cudaGraphInstantiate(&c->step_exec, g, 0);
    if (g) cudaGraphDestroy(g);
    cudaStreamDestroy(cap);
    if (e != cudaSuccess) {
        c->step_exec = nullptr;
        return fail(c, WICI_E_CUDA, "decode graph capture: %s", cudaGetErrorString(e));
    }
    return WICI_OK;
}

static int begin_decode(wici_ctx *c, int32_t n_steps, int32_t token_in) {
    if (int rc = check_ready(c)) return rc;
    if (!c->prefilled) return fail(c, WICI_E_STATE, "decode before prefill");
    const Plan &p = c->plan;
    if ((int64_t)c->kv_len + n_steps > p.cfg.max_tokens)
        return fail(c, WICI_E_CAPACITY, "kv_len %d + %d steps exceeds max_tokens %d", c->kv_len, n_steps,
                    p.cfg.max_tokens);
    if (token_in >= p.V) return fail(c, WICI_E_ARG, "token %d out of range", token_in);
    if (int rc = ensure_graph(c)) return rc;
    if (token_in >= 0) {
        c->pinned[0] = token_in;
        CUDA_TRY(c, cudaMemcpyAsync(c->bufs.ctrl + CTRL_TOKEN, c->pinned, sizeof(int), cudaMemcpyHostToDevice,
                                    c->stream));
    }
    return WICI_OK;
}

// One decode step on the stream: the captured graph, or, for a context on an SM
// share, the step kernel launched directly (graph replays of different contexts
// were measured to run one after the other, while direct launches of the
// persistent step kernel on disjoint SM shares run at the same time).
// At most this many decode steps of an SM-share context are queued at once:
// with deep queues the steps of two tenants were measured to alternate on the
// GPU instead of overlapping.
constexpr int kShareDepth = 2;

static cudaError_t launch_step(wici_ctx *c) {
    if (c->plan.cfg.max_sms > 0 && decode_is_persistent(c->plan)) {
        cudaEvent_t ev = c->step_done[c->steps_launched % kShareDepth];
        cudaError_t e = c->steps_launched >= kShareDepth ? cudaEventSynchronize(ev) : cudaSuccess;
        if (e == cudaSuccess) e = enqueue_decode_step(c->plan, c->bufs, c->stream, false, nullptr);
        if (e == cudaSuccess) e = cudaEventRecord(ev, c->stream);
        if (e == cudaSuccess) ++c->steps_launched;
        return e;
    }
    return cudaGraphLaunch(c->step_exec, c->stream);
}

int wici_decode_step(wici_ctx *c, int32_t token_in, float *logits_out, int32_t *token_out) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (int rc = begin_decode(c, 1, token_in)) return rc;
    CUDA_TRY(c, launch_step(c));
    if (logits_out)
        CUDA_TRY(c, cudaMemcpyAsync(logits_out, c->bufs.logits, (size_t)c->plan.V * 4, cudaMemcpyDeviceToHost,
                                    c->stream));
    return finish_call(c, c->kv_len + 1, token_out);
}

int wici_decode(wici_ctx *c, int32_t n_steps, int32_t token_in, int32_t *tokens_out) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (n_steps < 1) return fail(c, WICI_E_ARG, "n_steps must be >= 1");
    if (int rc = begin_decode(c, n_steps, token_in)) return rc;
    for (int i = 0; i < n_steps; ++i) CUDA_TRY(c, launch_step(c));
    if (tokens_out)
        CUDA_TRY(c, cudaMemcpyAsync(tokens_out, c->bufs.hist + c->kv_len + 1, (size_t)n_steps * 4,
                                    cudaMemcpyDeviceToHost, c->stream));
    return finish_call(c, c->kv_len + n_steps, nullptr);
}

int wici_reset(wici_ctx *c) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    c->pinned[0] = 0;
    CUDA_TRY(c, cudaMemcpyAsync(c->bufs.ctrl + CTRL_POS, c->pinned, sizeof(int), cudaMemcpyHostToDevice, c->stream));
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));
    c->kv_len = 0;
    c->prefilled = false;
    return WICI_OK;
}

int wici_set_page_table(wici_ctx *c, const int32_t *pages, int32_t n) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    const Plan &p = c->plan;
    if (!pages || n != p.max_pages) return fail(c, WICI_E_ARG, "page table must have %d entries", p.max_pages);
    if (c->kv_len != 0) return fail(c, WICI_E_STATE, "page table can only change when kv_len == 0");
    std::vector<char> seen(n, 0);
    for (int i = 0; i < n; ++i) {
        if (pages[i] < 0 || pages[i] >= n || seen[pages[i]])
            return fail(c, WICI_E_ARG, "page table is not a permutation of 0..%d", n - 1);
        seen[pages[i]] = 1;
    }
    CUDA_TRY(c, cudaMemcpyAsync(c->bufs.pages, pages, (size_t)n * 4, cudaMemcpyHostToDevice, c->stream));
    CUDA_TRY(c, cudaStreamSynchronize(c->stream));
    return WICI_OK;
}

int32_t wici_kv_len(const wici_ctx *c) { return c ? c->kv_len : WICI_E_ARG; }

const char *wici_last_error(const wici_ctx *c) { return c ? c->err.c_str() : g_thread_err.c_str(); }

struct EventHook : LaunchHook {
    cudaStream_t st;
    std::vector<std::string> names;
    std::vector<cudaEvent_t> ev;  // pairs
    std::vector<int> which;
    cudaError_t err = cudaSuccess;
    void before(const char *name) override {
        cudaEvent_t e0;
        if (cudaEventCreate(&e0) != cudaSuccess) { err = cudaErrorUnknown; return; }
        cudaEventRecord(e0, st);
        ev.push_back(e0);
        int k = -1;
        for (size_t i = 0; i < names.size(); ++i)
            if (names[i] == name) k = (int)i;
        if (k < 0) { names.push_back(name); k = (int)names.size() - 1; }
        which.push_back(k);
    }
    void after(const char *) override {
        cudaEvent_t e1;
        if (cudaEventCreate(&e1) != cudaSuccess) { err = cudaErrorUnknown; return; }
        cudaEventRecord(e1, st);
        ev.push_back(e1);
    }
};

// per-kind launches and milliseconds of a finished EventHook into the caller's arrays
static void report_hook(EventHook &hook, const char **names, int32_t *launches, double *total_ms, int32_t cap,
                        int32_t *n_kinds) {
    std::vector<double> ms(hook.names.size(), 0.0);
    std::vector<int> cnt(hook.names.size(), 0);
    for (size_t i = 0; i < hook.which.size(); ++i) {
        float t = 0.f;
        cudaEventElapsedTime(&t, hook.ev[2 * i], hook.ev[2 * i + 1]);
        ms[hook.which[i]] += t;
        cnt[hook.which[i]] += 1;
    }
    for (cudaEvent_t e : hook.ev) cudaEventDestroy(e);
    const int k = (int)hook.names.size() < cap ? (int)hook.names.size() : cap;
    static std::vector<std::string> keep;  // names outlive the call
    for (int i = 0; i < k; ++i) {
        bool found = false;
        for (auto &s : keep) if (s == hook.names[i]) found = true;
        if (!found) keep.push_back(hook.names[i]);
    }
    for (int i = 0; i < k; ++i) {
        for (auto &s : keep)
            if (s == hook.names[i]) names[i] = s.c_str();
        launches[i] = cnt[i];
        total_ms[i] = ms[i];
    }
    *n_kinds = k;
}

int wici_profile_decode(wici_ctx *c, int32_t n_steps, const char **names, int32_t *launches, double *total_ms,
                        int32_t cap, int32_t *n_kinds) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (n_steps < 1 || !names || !launches || !total_ms || !n_kinds || cap < 1)
        return fail(c, WICI_E_ARG, "bad profile arguments");
    if (int rc = begin_decode(c, n_steps, -1)) return rc;
    EventHook hook;
    hook.st = c->stream;
    for (int i = 0; i < n_steps; ++i) {
        cudaError_t e = enqueue_decode_step(c->plan, c->bufs, c->stream, false, &hook);
        if (e != cudaSuccess) return fail(c, WICI_E_CUDA, "profile launch: %s", cudaGetErrorString(e));
    }
    int rc = finish_call(c, c->kv_len + n_steps, nullptr);
    report_hook(hook, names, launches, total_ms, cap, n_kinds);
    return rc;
}

int wici_profile_prefill(wici_ctx *c, const int32_t *tokens, int32_t n, const char **names, int32_t *launches,
                         double *total_ms, int32_t cap, int32_t *n_kinds) {
    if (!c) return fail(nullptr, WICI_E_ARG, "null context");
    if (!tokens || n < 1 || !names || !launches || !total_ms || !n_kinds || cap < 1)
        return fail(c, WICI_E_ARG, "bad profile arguments");
    if (int rc = check_ready(c)) return rc;
    const Plan &p = c->plan;
    if ((int64_t)c->kv_len + n > p.cfg.max_tokens)
        return fail(c, WICI_E_CAPACITY, "kv_len %d + %d tokens exceeds max_tokens %d", c->kv_len, n,
                    p.cfg.max_tokens);
    for (int i = 0; i < n; ++i)
        if (tokens[i] < 0 || tokens[i] >= p.V) return fail(c, WICI_E_ARG, "token %d out of range", tokens[i]);
    EventHook hook;
    hook.st = c->stream;
    for (int off = 0; off < n; off += p.max_chunk) {
        const int T = n - off < p.max_chunk ? n - off : p.max_chunk;
        CUDA_TRY(c, cudaMemcpyAsync(c->bufs.tok, tokens + off, (size_t)T * 4, cudaMemcpyHostToDevice, c->stream));
        const bool last = off + T == n;
        CUDA_TRY(c, enqueue_prefill_chunk(p, c->bufs, c->maps, c->stream, c->kv_len + off, T, last ? n : 0, &hook));
        if (!last) CUDA_TRY(c, cudaStreamSynchronize(c->stream));
    }
    int rc = finish_call(c, c->kv_len + n, nullptr);
    if (rc == WICI_OK) c->prefilled = true;
    report_hook(hook, names, launches, total_ms, cap, n_kinds);
    return rc;
}

int wici_check_bounded_wait(void *cuda_stream, int64_t limit_ns) {
    cudaStream_t st = (cudaStream_t)cuda_stream;
    int *d_err = nullptr;
    int h_err = 0;
    if (limit_ns < 0) return fail(nullptr, WICI_E_ARG, "limit_ns must be >= 0");
    cudaError_t e = cudaMallocAsync((void **)&d_err, sizeof(int), st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d_err, 0, sizeof(int), st);
    if (e == cudaSuccess) e = enqueue_bounded_wait_probe(d_err, limit_ns, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&h_err, d_err, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (d_err) {
        cudaFreeAsync(d_err, st);
        cudaStreamSynchronize(st);
    }
    if (e != cudaSuccess) return fail(nullptr, WICI_E_CUDA, "bounded-wait probe: %s", cudaGetErrorString(e));
    if (h_err != 0) return fail(nullptr, WICI_E_TIMEOUT, "wait gave up as designed (site %d)", h_err);
    return WICI_OK;
}

void wici_destroy(wici_ctx *c) {
    if (!c) return;
    if (c->stream) cudaStreamSynchronize(c->stream);
    if (c->step_exec) cudaGraphExecDestroy(c->step_exec);
    for (cudaEvent_t e : c->step_done)
        if (e) cudaEventDestroy(e);
    if (c->pinned) cudaFreeHost(c->pinned);
    delete c;
}

}  // extern "C"
