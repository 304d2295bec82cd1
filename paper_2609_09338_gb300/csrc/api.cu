// C ABI: argument validation, workspace layout and launch sequencing.
#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>

#include "common.cuh"
#include "draft.cuh"
#include "tc.cuh"
#include "internal.h"
#include "tma.cuh"
#include "osprey.h"

namespace osp {

static std::atomic<long long> g_launches{0};
void count_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

static thread_local char g_err[512] = "";

static int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return code;
}

void set_last_error(const char *msg) { snprintf(g_err, sizeof g_err, "%s", msg); }

static int cuda_fail(cudaError_t e, const char *what) {
    return fail(OSPREY_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace osp

using namespace osp;

struct osprey_ctx {
    osprey_config cfg;
    osprey_weights w;
    Dims dim;
    int sms;
    int attn_cs;    // cluster size of the attention kernel (0: split partials in global memory)
    bool tc;        // batched rows (3..80) run their projections on tcgen05
    bool fused_mlp; // batch-1 chain steps run O-proj, gate/up and down as one launch
    bool fused_layer; // batch-1 chain steps run each whole layer as one launch
    CUtensorMap tm_c, tm_lm, tm_qkv[OSPREY_MAX_LAYERS], tm_o[OSPREY_MAX_LAYERS], tm_gate[OSPREY_MAX_LAYERS],
        tm_up[OSPREY_MAX_LAYERS], tm_down[OSPREY_MAX_LAYERS];
    double inv_freq[64];
    int n_probe;
    int probe_kind;   // OSPREY_PROBE_LM_HEAD or OSPREY_PROBE_ATTENTION
    cudaEvent_t *probe_begin, *probe_end;
};

extern "C" const char *osprey_last_error(void) { return g_err; }
extern "C" int64_t osprey_launch_count(void) { return g_launches.load(); }

// One block waiting on an mbarrier that nothing arrives on, bounded like every
// wait of the library; on expiry it reports the timeout and returns.
__global__ void selftest_wait_kernel(long long limit_cycles, int32_t *status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        osp::mbar_init(&bar, 1);
        osp::mbar_fence_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !osp::mbar_wait(&bar, 0, limit_cycles)) osp::set_status(status, OSPREY_ERR_TIMEOUT);
}

extern "C" int osprey_selftest_wait_timeout(int64_t limit_cycles, int32_t *dev_status, void *stream) {
    g_err[0] = 0;
    if (limit_cycles < 1 || limit_cycles > 2000000000LL || !dev_status)
        return fail(OSPREY_ERR_INVALID_ARG, "limit_cycles in 1..2e9 and a status word required");
    selftest_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>((long long)limit_cycles, dev_status);
    osp::count_launch();
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? OSPREY_OK : cuda_fail(e, "self-test launch");
}

static bool is_pow2_multiple(int x, int m) { return x > 0 && x % m == 0; }

extern "C" int osprey_create(const osprey_config *cfg, const osprey_weights *w, osprey_ctx **out) {
    g_err[0] = 0;
    if (!cfg || !w || !out) return fail(OSPREY_ERR_INVALID_ARG, "null argument");
    *out = nullptr;
    const osprey_config &c = *cfg;
    if (c.n_layers < 1 || c.n_layers > OSPREY_MAX_LAYERS)
        return fail(OSPREY_ERR_SHAPE, "n_layers must be in 1..%d", OSPREY_MAX_LAYERS);
    if (!is_pow2_multiple(c.d_model, 256)) return fail(OSPREY_ERR_SHAPE, "d_model must be a multiple of 256");
    if (c.head_dim != 64 && c.head_dim != 128) return fail(OSPREY_ERR_SHAPE, "head_dim must be 64 or 128");
    if (c.n_kv_heads < 1 || c.n_q_heads < c.n_kv_heads || c.n_q_heads % c.n_kv_heads)
        return fail(OSPREY_ERR_SHAPE, "n_q_heads must be a positive multiple of n_kv_heads");
    const int G = c.n_q_heads / c.n_kv_heads;
    if (G != 1 && G != 2 && G != 4 && G != 8) return fail(OSPREY_ERR_SHAPE, "n_q_heads/n_kv_heads must be 1, 2, 4 or 8");
    if ((c.n_q_heads * c.head_dim) % 256) return fail(OSPREY_ERR_SHAPE, "n_q_heads*head_dim must be a multiple of 256");
    if (!is_pow2_multiple(c.ffn_dim, 256)) return fail(OSPREY_ERR_SHAPE, "ffn_dim must be a multiple of 256");
    if (!is_pow2_multiple(c.feat_dim, 256)) return fail(OSPREY_ERR_SHAPE, "feat_dim must be a multiple of 256");
    if (c.feat_dim > 100 * 1024) return fail(OSPREY_ERR_SHAPE, "feat_dim above 102400 is not supported");
    if (c.vocab < 1) return fail(OSPREY_ERR_SHAPE, "vocab must be positive");
    if (c.page_size != 16) return fail(OSPREY_ERR_SHAPE, "page_size must be 16");
    if (!(c.rms_eps > 0.f) || !(c.rope_theta > 1.f)) return fail(OSPREY_ERR_INVALID_ARG, "rms_eps and rope_theta must be positive");
    if (!w->W_c || !w->embed || !w->final_norm || !w->lm_head) return fail(OSPREY_ERR_INVALID_ARG, "null weight pointer");
    for (int l = 0; l < c.n_layers; ++l)
        if (!w->attn_norm[l] || !w->W_qkv[l] || !w->W_o[l] || !w->ffn_norm[l] || !w->W_gate[l] ||
            !w->W_up[l] || !w->W_down[l])
            return fail(OSPREY_ERR_INVALID_ARG, "null weight pointer in layer %d", l);
    const void *ptrs[] = {w->W_c, w->embed, w->final_norm, w->lm_head};
    for (const void *p : ptrs)
        if ((uintptr_t)p % 16) return fail(OSPREY_ERR_INVALID_ARG, "weights must be 16-byte aligned");
    for (int l = 0; l < c.n_layers; ++l) {
        const void *lp[] = {w->attn_norm[l], w->W_qkv[l], w->W_o[l], w->ffn_norm[l], w->W_gate[l], w->W_up[l],
                            w->W_down[l]};
        for (const void *p : lp)
            if ((uintptr_t)p % 16) return fail(OSPREY_ERR_INVALID_ARG, "weights must be 16-byte aligned");
    }
    osprey_ctx *ctx = new (std::nothrow) osprey_ctx();
    if (!ctx) return fail(OSPREY_ERR_INVALID_ARG, "out of host memory");
    ctx->cfg = c;
    ctx->w = *w;
    ctx->dim = Dims{c.d_model, c.n_layers, c.n_q_heads, c.n_kv_heads, c.head_dim, c.ffn_dim,
                    c.vocab, c.feat_dim, c.page_size, c.rms_eps};
    for (int i = 0; i < c.head_dim / 2; ++i)
        ctx->inv_freq[i] = std::pow((double)c.rope_theta, -2.0 * i / c.head_dim);
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = draft_set_attributes();
    if (e == cudaSuccess) e = stream_set_attributes();
    if (e == cudaSuccess) {
        // OSPREY_ATTN_CLUSTER=0 selects the attention kernel that merges split
        // partials through global memory (also used where clusters cannot run)
        const char *env = std::getenv("OSPREY_ATTN_CLUSTER");
        ctx->attn_cs = env && env[0] == '0' ? 0 : attn_cluster_size(ctx->dim);
        // OSPREY_TC=0 keeps batched rows on the CUDA-core GEMV
        const char *tenv = std::getenv("OSPREY_TC");
        const Dims &D = ctx->dim;
        const osprey_weights &W = ctx->w;
        bool tc = !(tenv && tenv[0] == '0') && tc_available() && tc_set_attributes() == cudaSuccess;
        tc = tc && tc_encode_weight(&ctx->tm_c, W.W_c, D.d, D.feat) && tc_encode_weight(&ctx->tm_lm, W.lm_head, D.V, D.d);
        for (int l = 0; tc && l < D.L; ++l)
            tc = tc_encode_weight(&ctx->tm_qkv[l], W.W_qkv[l], (D.Hq + 2 * D.Hkv) * D.hd, 2 * D.d) &&
                 tc_encode_weight(&ctx->tm_o[l], W.W_o[l], D.d, D.Hq * D.hd) &&
                 tc_encode_weight(&ctx->tm_gate[l], W.W_gate[l], D.F, D.d) &&
                 tc_encode_weight(&ctx->tm_up[l], W.W_up[l], D.F, D.d) &&
                 tc_encode_weight(&ctx->tm_down[l], W.W_down[l], D.d, D.F);
        ctx->tc = tc;
        // OSPREY_FUSED_MLP=1 runs O-proj, gate/up and down of a batch-1 chain
        // step as one launch with grid barriers (not yet the default)
        const char *menv = std::getenv("OSPREY_FUSED_MLP");
        ctx->fused_mlp = menv && menv[0] == '1' && mlp_fused_supported(D, ctx->sms);
        // OSPREY_FUSED_LAYER=1 runs each whole layer of a batch-1 chain step as
        // one launch with grid barriers (not yet the default)
        const char *lenv = std::getenv("OSPREY_FUSED_LAYER");
        ctx->fused_layer = lenv && lenv[0] == '1' && layer_fused_supported(D, ctx->sms);
        cudaGetLastError();
    }
    if (e != cudaSuccess) {
        cudaGetLastError();   // do not leave the error pending for the caller's next CUDA call
        delete ctx;
        return cuda_fail(e, "device query");
    }
    *out = ctx;
    return OSPREY_OK;
}

static void probe_release(osprey_ctx *ctx) {
    for (int i = 0; i < ctx->n_probe; ++i) {
        cudaEventDestroy(ctx->probe_begin[i]);
        cudaEventDestroy(ctx->probe_end[i]);
    }
    delete[] ctx->probe_begin;
    delete[] ctx->probe_end;
    ctx->probe_begin = ctx->probe_end = nullptr;
    ctx->n_probe = 0;
}

extern "C" void osprey_destroy(osprey_ctx *ctx) {
    if (!ctx) return;
    probe_release(ctx);
    delete ctx;
}

extern "C" int osprey_probe_enable(osprey_ctx *ctx, int n) {
    if (!ctx || n < 0) return fail(OSPREY_ERR_INVALID_ARG, "bad probe arguments");
    probe_release(ctx);
    if (n == 0) return OSPREY_OK;
    ctx->probe_begin = new cudaEvent_t[n];
    ctx->probe_end = new cudaEvent_t[n];
    for (int i = 0; i < n; ++i) {
        cudaError_t e = cudaEventCreate(&ctx->probe_begin[i]);
        if (e == cudaSuccess) e = cudaEventCreate(&ctx->probe_end[i]);
        if (e != cudaSuccess) {
            ctx->n_probe = i;
            probe_release(ctx);
            return cuda_fail(e, "cudaEventCreate");
        }
        ctx->n_probe = i + 1;
    }
    return OSPREY_OK;
}

extern "C" int osprey_probe_select(osprey_ctx *ctx, int kind) {
    if (!ctx || (kind != OSPREY_PROBE_LM_HEAD && kind != OSPREY_PROBE_ATTENTION))
        return fail(OSPREY_ERR_INVALID_ARG, "bad probe kind");
    ctx->probe_kind = kind;
    return OSPREY_OK;
}

extern "C" int osprey_probe_read(osprey_ctx *ctx, float *ms, int n) {
    if (!ctx || !ms || n < 0 || n > ctx->n_probe) return fail(OSPREY_ERR_INVALID_ARG, "bad probe read");
    for (int i = 0; i < n; ++i) {
        cudaError_t e = cudaEventElapsedTime(&ms[i], ctx->probe_begin[i], ctx->probe_end[i]);
        if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
    }
    return OSPREY_OK;
}

static cudaError_t probe_record(cudaEvent_t ev, cudaStream_t s) {
    cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(s, &st);
    if (e != cudaSuccess) return e;
    return st == cudaStreamCaptureStatusActive ? cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal)
                                               : cudaEventRecord(ev, s);
}

// ------------------------------------------------------------------ workspace
// block: the layout of a block-drafting call (every extend row is sampled, so
// the sampler buffers hold B * max_new rows instead of B)
static size_t draft_layout(const osprey_ctx *ctx, int B, int K, int max_new, int max_pages,
                           DraftWs *ws, void *base, bool block = false) {
    const Dims &D = ctx->dim;
    const long long R_ext = (long long)B * max_new;
    const long long R_lm = block ? R_ext : B;
    const int max_ctx = max_pages * D.P;
    const int ns = std::max(attn_splits((int)R_ext, D.Hkv, max_ctx, ctx->sms),
                            attn_splits(B, D.Hkv, max_ctx, ctx->sms));
    const int lm_warps = lm_blocks(D.V, ctx->sms) * 8;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align256(off + bytes); return o; };
    size_t o_valid = take(4ull * B), o_pos0 = take(4ull * B), o_nn = take(4ull * B);
    // arrival counters and the grid barrier, one contiguous block of int32
    // words that the call's first kernel zeroes
    const size_t o_at = off, n_at = (size_t)R_ext * D.Hkv;
    const size_t o_lt = o_at + 4 * n_at, o_gb = o_lt + 4ull * B, o_rt = o_gb + 8;
    const size_t n_counters = n_at + B + 2 + R_lm;
    take(4 * n_counters);
    size_t o_xe = take(4ull * R_ext * D.d), o_se = take(4ull * R_ext * D.d);
    size_t o_xc = take(4ull * B * D.d), o_sc = take(4ull * B * D.d);
    size_t o_q = take(4ull * R_ext * D.Hq * D.hd);
    size_t o_ap = take(4ull * R_ext * D.Hq * ns * (D.hd + 2));
    size_t o_ao = take(4ull * R_ext * D.Hq * D.hd);
    size_t o_fh = take(4ull * R_ext * D.F);
    size_t o_ls = take(16ull * B * lm_warps);
    const StreamPlan lmp = stream_plan(G_LM, D, ctx->sms);
    size_t o_lsup = take(8ull * B * lmp.blocks * lmp.nsup);   // the streamed LM head's run statistics (rows <= 2)
    size_t o_lc = take(16ull * B * lmp.blocks);
    // tensor-core path: bf16 operand planes, QKV output, row-sampler partials
    const long long tc_rows = std::min<long long>(std::max<long long>(R_ext, B), TC_MAX_ROWS);
    const long long np = (tc_rows + 15) / 16 * 16;
    const long long nqkv = (long long)(D.Hq + 2 * D.Hkv) * D.hd;
    const bool tcw = ctx->tc;
    size_t o_xq = take(tcw ? 2ull * TC_PLANES * np * 2 * D.d : 0), o_yq = take(tcw ? 4ull * np * nqkv : 0);
    size_t o_xo = take(tcw ? 2ull * TC_PLANES * np * D.Hq * D.hd : 0), o_xg = take(tcw ? 2ull * TC_PLANES * np * D.d : 0);
    size_t o_xh = take(tcw ? 2ull * TC_PLANES * np * D.F : 0), o_xl = take(tcw ? 2ull * TC_PLANES * np * D.d : 0);
    const long long lm_nsub = (D.V + TC_LM_GROUP - 1) / TC_LM_GROUP;
    size_t o_rp = take(tcw ? 16ull * R_lm * lm_nsub : 0);
    // split-K partials: the largest nsplit x rows x outputs of the call's projections
    long long part = 0;
    if (tcw) {
        const long long rows = tc_rows;
        auto need = [&](int nout, int K_) {
            const int ns = tc_nsplit(nout, K_, ctx->sms);
            if (ns > 1) part = std::max(part, (long long)ns * rows * nout);
        };
        need(D.d, D.feat);
        need((D.Hq + 2 * D.Hkv) * D.hd, 2 * D.d);
        need(D.d, D.Hq * D.hd);
        // gate/up: one GEMM whose partials always go through the buffer
        part = std::max(part, (long long)std::max(tc_nsplit(2 * D.F, D.d, ctx->sms), 1) * rows * 2 * D.F);
        need(D.d, D.F);
        need(D.V, D.d);
    }
    size_t o_tp = take(4ull * part);
    if (ws && base) {
        char *p = (char *)base;
        ws->seq_valid = (int *)(p + o_valid);
        ws->seq_pos0 = (int *)(p + o_pos0);
        ws->seq_nnew = (int *)(p + o_nn);
        ws->attn_ticket = (int *)(p + o_at);
        ws->lm_ticket = (int *)(p + o_lt);
        ws->grid_bar = (unsigned *)(p + o_gb);
        ws->x_ext = (float *)(p + o_xe);
        ws->s_ext = (float *)(p + o_se);
        ws->x_chain = (float *)(p + o_xc);
        ws->s_chain = (float *)(p + o_sc);
        ws->q = (float *)(p + o_q);
        ws->attn_part = (float *)(p + o_ap);
        ws->attn_out = (float *)(p + o_ao);
        ws->ffn_h = (float *)(p + o_fh);
        ws->lm_stats = (float4 *)(p + o_ls);
        ws->lm_sup = (float2 *)(p + o_lsup);
        ws->lm_cta_stats = (float4 *)(p + o_lc);
        ws->tc_xq = (uint16_t *)(p + o_xq);
        ws->tc_yq = (float *)(p + o_yq);
        ws->tc_xo = (uint16_t *)(p + o_xo);
        ws->tc_xg = (uint16_t *)(p + o_xg);
        ws->tc_xh = (uint16_t *)(p + o_xh);
        ws->tc_xl = (uint16_t *)(p + o_xl);
        ws->rs_part = (float4 *)(p + o_rp);
        ws->rs_ticket = (int *)(p + o_rt);
        ws->counters = (int *)(p + o_at);
        ws->n_counters = (int)n_counters;
        ws->tc_part = (float *)(p + o_tp);
        ws->tc_part_cap = part;
        ws->n_splits_max = ns;
        ws->lm_warps_max = lm_warps;
    }
    (void)K;
    return off;
}

static bool draft_args_ok(const osprey_ctx *ctx, int B, int K, int max_new, int max_pages) {
    return ctx && B >= 1 && B <= 65535 && K >= 1 && K <= 64 && max_new >= 1 && max_new <= 64 &&
           max_pages >= 1 && (long long)max_pages * ctx->dim.P < (1LL << 30);
}

extern "C" size_t osprey_draft_workspace_bytes(const osprey_ctx *ctx, int B, int K, int max_new,
                                               int max_pages_per_seq) {
    if (!draft_args_ok(ctx, B, K, max_new, max_pages_per_seq)) return 0;
    return draft_layout(ctx, B, K, max_new, max_pages_per_seq, nullptr, nullptr);
}

// ------------------------------------------------------------------ kv append
extern "C" int osprey_kv_append(const osprey_ctx *ctx, const osprey_kv *kv, int B, const int32_t *n_rows,
                                int64_t total_rows, const void *k_rows, const void *v_rows,
                                int32_t *dev_status, void *stream) {
    g_err[0] = 0;
    if (!ctx || !kv) return fail(OSPREY_ERR_INVALID_ARG, "null context or kv");
    if (B == 0) return OSPREY_OK;
    if (B < 0 || B > 4096) return fail(OSPREY_ERR_INVALID_ARG, "B must be in 0..4096");
    if (total_rows < 0) return fail(OSPREY_ERR_INVALID_ARG, "total_rows must be >= 0");
    if (!n_rows || !kv->k_pages || !kv->v_pages || !kv->page_table || !kv->seq_len)
        return fail(OSPREY_ERR_INVALID_ARG, "null pointer");
    if (total_rows > 0 && (!k_rows || !v_rows)) return fail(OSPREY_ERR_INVALID_ARG, "null rows");
    if (kv->max_pages_per_seq < 1 || kv->n_pages < 1) return fail(OSPREY_ERR_INVALID_ARG, "empty page pool");
    if (((uintptr_t)k_rows | (uintptr_t)v_rows | (uintptr_t)kv->k_pages | (uintptr_t)kv->v_pages) % 16)
        return fail(OSPREY_ERR_INVALID_ARG, "K/V buffers must be 16-byte aligned");
    KvAppendArgs a{};
    a.k_pages = kv->k_pages;
    a.v_pages = kv->v_pages;
    a.page_table = kv->page_table;
    a.seq_len = kv->seq_len;
    a.n_rows = n_rows;
    a.k_rows = k_rows;
    a.v_rows = v_rows;
    a.total_rows = total_rows;
    a.B = B;
    a.L = ctx->dim.L;
    a.Hkv = ctx->dim.Hkv;
    a.hd = ctx->dim.hd;
    a.P = ctx->dim.P;
    a.max_pages = kv->max_pages_per_seq;
    a.n_pages = kv->n_pages;
    a.status = dev_status;
    cudaError_t e = launch_kv_append(a, (cudaStream_t)stream);
    return e == cudaSuccess ? OSPREY_OK : cuda_fail(e, "kv_append launch");
}

// ------------------------------------------------------------------ draft step
// block: a block-drafting call (EAGLE-style DFlash): K = 1, every one of the
// max_new extend rows of a sequence is sampled (row j's output proposes the
// token at j + 1) into draft_* [B][max_new], and only the first row (the
// anchor) is committed.
static int draft_step_impl(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int max_new,
                           const int32_t *n_new, const int32_t *tokens, const void *feats, float temperature,
                           const float *u_draft, int32_t *draft_tokens, float *draft_qx, float *draft_stats,
                           float *draft_logits, float *draft_hidden, void *workspace, size_t workspace_bytes,
                           int32_t *dev_status, void *stream, bool block = false, int topk = 1) {
    g_err[0] = 0;
    if (!ctx || !kv) return fail(OSPREY_ERR_INVALID_ARG, "null context or kv");
    if (B == 0) return OSPREY_OK;
    if (!draft_args_ok(ctx, B, K, max_new, kv->max_pages_per_seq))
        return fail(OSPREY_ERR_INVALID_ARG, "B in 1..65535, K and max_new in 1..64, max_pages_per_seq >= 1 required");
    if (!(temperature >= 0.f) || !std::isfinite(temperature))
        return fail(OSPREY_ERR_INVALID_ARG, "temperature must be finite and >= 0");
    if (!n_new || !tokens || !feats || !draft_tokens || !workspace || !kv->k_pages || !kv->v_pages ||
        !kv->page_table || !kv->seq_len)
        return fail(OSPREY_ERR_INVALID_ARG, "null pointer");
    if (temperature > 0.f && !u_draft) return fail(OSPREY_ERR_INVALID_ARG, "u_draft is required when temperature > 0");
    if (kv->n_pages < 1) return fail(OSPREY_ERR_INVALID_ARG, "empty page pool");
    if (((uintptr_t)feats | (uintptr_t)workspace | (uintptr_t)draft_hidden) % 16)
        return fail(OSPREY_ERR_INVALID_ARG, "feats, workspace and draft_hidden must be 16-byte aligned");
    DraftWs ws{};
    const size_t need = draft_layout(ctx, B, K, max_new, kv->max_pages_per_seq, &ws, workspace, block);
    if (workspace_bytes < need)
        return fail(OSPREY_ERR_CAPACITY, "workspace too small: %zu < %zu bytes", workspace_bytes, need);
    if (block && (K != 1 || !ctx->tc || B * max_new < 3 || B * max_new > TC_MAX_ROWS))
        return fail(OSPREY_ERR_SHAPE, "block drafting runs 3..%d rows per group on the tensor cores", TC_MAX_ROWS);
    if (topk > 1 && (!ctx->tc || B > TC_MAX_ROWS))
        return fail(OSPREY_ERR_SHAPE, "topk > 1 samples on the tensor-core LM head: at most %d sequences and a "
                                      "device with tcgen05 (not OSPREY_TC=0)", TC_MAX_ROWS);

    cudaStream_t s = (cudaStream_t)stream;
    const Dims &D = ctx->dim;
    const osprey_weights &W = ctx->w;
    const size_t layer_pages = (size_t)kv->n_pages * D.Hkv * D.P * D.hd;
    const int max_ctx = kv->max_pages_per_seq * D.P;
    cudaError_t e;

    PrepArgs pa{B, K, max_new, kv->max_pages_per_seq, kv->n_pages, D.P, D.V,
                kv->seq_len, n_new, tokens, kv->page_table,
                ws.seq_valid, ws.seq_pos0, ws.seq_nnew, draft_tokens, dev_status, ws.counters, ws.n_counters,
                block ? 1 : 0, block ? max_new : (topk > 1 ? K * topk : 0)};
    if ((e = launch_prepare(pa, s)) != cudaSuccess) return cuda_fail(e, "prepare launch");

    GemvArgs g{};
    g.dim = D;
    g.map = RowMap{ws.seq_valid, ws.seq_pos0, ws.seq_nnew, max_new, 0};
    g.R = B * max_new;
    g.W = (const uint16_t *)W.W_c;
    g.embed = (const uint16_t *)W.embed;
    g.tokens = tokens;
    g.feats = (const uint16_t *)feats;
    g.max_new = max_new;
    g.x = ws.x_ext;
    g.s = ws.s_ext;
    g.page_table = kv->page_table;
    g.max_pages = kv->max_pages_per_seq;
    g.n_pages = kv->n_pages;
    for (int i = 0; i < D.hd / 2; ++i) g.inv_freq[i] = ctx->inv_freq[i];
    // tensor-core path for 3..TC_MAX_ROWS activation rows
    auto tc_rows = [&](int rows) { return ctx->tc && rows >= 3 && rows <= TC_MAX_ROWS; };
    auto npad_of = [](int rows) { return (rows + 15) / 16 * 16; };
    // the next GEMM's operand planes, written by a residual GEMM's reduction when it has one
    struct NextPlanes {
        uint16_t *dst;
        const uint16_t *gain;
        int ld, col0, npl, map, rows_per_seq, npad;
    };
    auto tc_gemm = [&](int epi, int rows, int K_, int nout, int planes, const CUtensorMap &wa,
                       const void *xbuf, bool in_place_rows, float *y, int ldy, uint16_t *h,
                       const char *what, const CUtensorMap *wb = nullptr, const NextPlanes *nxt = nullptr,
                       bool *nxt_done = nullptr, const QkvPostArgs *rope = nullptr) -> int {
        const int np = npad_of(rows);
        CUtensorMap xm;
        const bool ok = in_place_rows ? tc_encode_rows(&xm, xbuf, rows, np, K_) : tc_encode_operand(&xm, xbuf, planes, np, K_);
        if (!ok) return fail(OSPREY_ERR_INVALID_ARG, "%s: tensor map encoding failed", what);
        TcArgs ta{};
        ta.epi = epi;
        ta.R = rows;
        ta.npad = np;
        ta.K = K_;
        ta.nout = nout;
        ta.planes = planes;
        ta.y = y;
        ta.x = y;
        ta.ldy = ldy;
        ta.h = h;
        ta.status = dev_status;
        ta.part = ws.tc_part;
        ta.part_cap = ws.tc_part_cap;
        ta.nout_a = wb ? nout / 2 : nout;
        if (nxt) {
            ta.pl_dst = nxt->dst;
            ta.pl_gain = nxt->gain;
            ta.pl_eps = D.eps;
            ta.pl_ld = nxt->ld;
            ta.pl_col0 = nxt->col0;
            ta.pl_npl = nxt->npl;
            ta.pl_npad = nxt->npad;
            ta.pl_map = nxt->map;
            ta.pl_rows_per_seq = nxt->rows_per_seq;
            ta.pl_max_new = max_new;
            ta.pl_valid = ws.seq_valid;
            ta.pl_nnew = ws.seq_nnew;
        }
        const cudaError_t e2 = launch_tc2(ta, wa, wb ? *wb : wa, xm, ctx->sms, s, nxt_done, rope);
        return e2 == cudaSuccess ? OSPREY_OK : cuda_fail(e2, what);
    };
    // the LM head of `rows` operand rows in ws.tc_xl on the tensor cores, with the
    // sampling partials in its epilogue (logits stored only into z, when given),
    // then one pick block per row
    auto tc_lm = [&](int rows, float *z, long long ldz, const LmPickArgs &pick_in) -> int {
        const int np = npad_of(rows);
        CUtensorMap xm;
        if (!tc_encode_operand(&xm, ws.tc_xl, TC_LM_PLANES, np, D.d))
            return fail(OSPREY_ERR_INVALID_ARG, "lm head: tensor map encoding failed");
        TcArgs ta{};
        ta.epi = TC_LM;
        ta.R = rows;
        ta.npad = np;
        ta.K = D.d;
        ta.nout = D.V;
        ta.planes = TC_LM_PLANES;
        ta.y = z;
        ta.ldy = (int)ldz;
        ta.status = dev_status;
        ta.lm_part = ws.rs_part;
        ta.lm_nsub = (D.V + TC_LM_GROUP - 1) / TC_LM_GROUP;
        ta.lm_invT = temperature > 0.f ? 1.f / temperature : 1.f;
        cudaError_t e2 = launch_tc(ta, ctx->tm_lm, xm, ctx->sms, s);
        if (e2 != cudaSuccess) return cuda_fail(e2, "lm head launch");
        LmPickArgs pk = pick_in;
        pk.dim = D;
        pk.part = ws.rs_part;
        pk.nsub = ta.lm_nsub;
        pk.planes = ws.tc_xl;
        pk.npad = np;
        pk.W = (const uint16_t *)W.lm_head;
        pk.temperature = temperature;
        pk.u_draft = u_draft;
        pk.embed = (const uint16_t *)W.embed;
        e2 = launch_lm_pick(pk, s);
        return e2 == cudaSuccess ? OSPREY_OK : cuda_fail(e2, "sampler launch");
    };
    auto planes = [&](const float *src, const uint16_t *gain, int d_, int rows, int ld, int col0, uint16_t *dst,
                      int rows_per_seq, bool last_of_seq, const char *what, int npl = TC_PLANES,
                      const float *src2 = nullptr, int col2 = 0) -> int {
        PlaneArgs pl{};
        pl.npl = npl;
        pl.src2 = src2;
        pl.col2 = col2;
        pl.src = src;
        pl.gain = gain;
        pl.eps = D.eps;
        pl.d = d_;
        pl.R = rows;
        pl.npad = npad_of(rows);
        pl.ld = ld;
        pl.col0 = col0;
        pl.dst = dst;
        pl.nnew = ws.seq_nnew;
        pl.max_new = max_new;
        pl.last_of_seq = last_of_seq;
        pl.valid = ws.seq_valid;
        pl.rows_per_seq = rows_per_seq;
        const cudaError_t e2 = launch_planes(pl, s);
        return e2 == cudaSuccess ? OSPREY_OK : cuda_fail(e2, what);
    };
    if (tc_rows(B * max_new)) {
        EmbedArgs ea{D.d, B * max_new, max_new, ws.seq_valid, ws.seq_nnew, tokens, (const uint16_t *)W.embed, ws.x_ext};
        if ((e = launch_embed_rows(ea, s)) != cudaSuccess) return cuda_fail(e, "embedding launch");
        const int rc = tc_gemm(TC_STORE, B * max_new, D.feat, D.d, 1, ctx->tm_c, feats, true, ws.s_ext, D.d,
                               nullptr, "feature projection launch");
        if (rc != OSPREY_OK) return rc;
    } else if ((e = launch_gemv(G_FEAT, g, gemv_rg(G_FEAT, D, g.R), ctx->sms, s)) != cudaSuccess) {
        return cuda_fail(e, "feature projection launch");
    }

    // measurement hook: events around the attention launch of (step, layer)
    auto attn_probe = [&](int slot, bool begin) -> cudaError_t {
        if (ctx->probe_kind != OSPREY_PROBE_ATTENTION || slot >= ctx->n_probe) return cudaSuccess;
        return probe_record(begin ? ctx->probe_begin[slot] : ctx->probe_end[slot], s);
    };
    // the LM head's operand comes from the tensor-core planes (block drafting, or
    // the tensor-core LM head) rather than the streamed or CUDA-core heads
    const bool lm_tc = block || (!(topk <= 1 && B <= 2 && stream_supported(G_LM, D, B, ctx->sms)) &&
                                 (tc_rows(B) || topk > 1));
    bool xq_next = false;   // the previous step's pick wrote this step's first QKV operand
    for (int step = 0; step < K; ++step) {
        const bool ext = step == 0;
        const int rows_per_seq = ext ? max_new : 1;
        const int R = B * rows_per_seq;
        // operand planes already written by an earlier kernel (a reduction, the pick)
        bool xq_ready = xq_next, xl_ready = false;
        xq_next = false;
        RowMap map{ws.seq_valid, ws.seq_pos0, ws.seq_nnew, rows_per_seq, step};
        float *x = ext ? ws.x_ext : ws.x_chain;
        float *sb = ext ? ws.s_ext : ws.s_chain;
        const int ns = attn_splits(R, D.Hkv, max_ctx, ctx->sms);
        // the on-chip-merge attention pays off while its clusters fit in one wave
        // (one block per SM); beyond that the global-partials kernel keeps more
        // loads in flight
        const bool clu = ctx->attn_cs && (long long)R * D.Hkv * ctx->attn_cs <= ctx->sms;
        // activation rows per launch: the streamed kernels serve one or two
        const bool streamed = R <= 2;
        StreamArgs sa{};
        sa.dim = D;
        sa.map = map;
        sa.R = R;
        sa.B = B;
        sa.K = K;
        sa.step = step;
        sa.max_new = max_new;
        sa.embed = (const uint16_t *)W.embed;
        sa.x = x;
        sa.s = sb;
        sa.q = ws.q;
        sa.page_table = kv->page_table;
        sa.max_pages = kv->max_pages_per_seq;
        sa.status = dev_status;
        for (int i = 0; i < D.hd / 2; ++i) sa.inv_freq[i] = ctx->inv_freq[i];
        auto plan_into = [&](GemvMode m) {
            const StreamPlan p = stream_plan(m, D, ctx->sms);
            sa.mode = m;
            sa.items = p.items;
            sa.n_items = p.n_items;
            sa.n_stages = p.n_stages;
            sa.stage_bytes = p.stage_bytes;
            sa.blocks = p.blocks;
        };
        auto gemv = [&](GemvMode m, const char *what) -> int {
            const int rg = streamed ? R : gemv_rg(m, D, R);
            cudaError_t e2;
            if (streamed && stream_supported(m, D, rg, ctx->sms)) {
                plan_into(m);
                sa.W = g.W;
                sa.W2 = g.W2;
                sa.gain = g.gain;
                sa.xin = g.xin;
                sa.out = g.out;
                sa.k_pages = g.k_pages;
                sa.v_pages = g.v_pages;
                e2 = launch_stream(m, sa, rg, s);
            } else {
                e2 = launch_gemv(m, g, rg, ctx->sms, s);
            }
            return e2 == cudaSuccess ? OSPREY_OK : cuda_fail(e2, what);
        };
        const bool tcp = !streamed && tc_rows(R);
        for (int l = 0; l < D.L && tcp; ++l) {
            uint16_t *kp = (uint16_t *)kv->k_pages + l * layer_pages;
            uint16_t *vp = (uint16_t *)kv->v_pages + l * layer_pages;
            const int nqkv = (D.Hq + 2 * D.Hkv) * D.hd;
            int rc;
            // [s; RMSNorm(x)] -> QKV (Eq. 2-3) -> RoPE and the paged K/V rows; the s half
            // of the operand is the same for every layer of the step, and the x half of
            // a later layer comes from the previous layer's down-projection reduction
            QkvPostArgs qp{};
            qp.dim = D;
            qp.map = map;
            qp.R = R;
            qp.y = ws.tc_yq;
            qp.q = ws.q;
            qp.k_pages = kp;
            qp.v_pages = vp;
            qp.page_table = kv->page_table;
            qp.max_pages = kv->max_pages_per_seq;
            for (int i = 0; i < D.hd / 2; ++i) qp.inv_freq[i] = ctx->inv_freq[i];
            // the QKV GEMM's reduction does RoPE and the K/V write when it runs
            bool rope_done = false;
            if ((!xq_ready &&
                 (rc = planes(x, (const uint16_t *)W.attn_norm[l], D.d, R, 2 * D.d, D.d, ws.tc_xq, rows_per_seq, false,
                              "qkv operand", TC_PLANES, l == 0 ? sb : nullptr, 0)) != OSPREY_OK) ||
                (rc = tc_gemm(TC_STORE, R, 2 * D.d, nqkv, TC_PLANES, ctx->tm_qkv[l], ws.tc_xq, false, ws.tc_yq, nqkv,
                              nullptr, "qkv launch", nullptr, nullptr, &rope_done, &qp)) != OSPREY_OK)
                return rc;
            if (!rope_done && (e = launch_qkv_post(qp, s)) != cudaSuccess) return cuda_fail(e, "rope launch");
            AttnArgs at{};
            at.dim = D;
            at.map = map;
            at.R = R;
            at.n_splits = clu ? ctx->attn_cs : ns;
            at.split_len = attn_split_len(max_ctx, at.n_splits);
            at.q = ws.q;
            at.k_pages = kp;
            at.v_pages = vp;
            at.page_table = kv->page_table;
            at.max_pages = kv->max_pages_per_seq;
            at.part = ws.attn_part;
            at.out = ws.attn_out;
            at.out_planes = ws.tc_xo;   // the O projection's operand, written by attention itself
            at.npad = npad_of(R);
            at.ticket = ws.attn_ticket;
            at.status = dev_status;
            if ((e = attn_probe(step * D.L + l, true)) != cudaSuccess) return cuda_fail(e, "probe record");
            e = clu ? launch_attn_cluster(at, ctx->attn_cs, s) : launch_attn(at, s);
            if (e != cudaSuccess) return cuda_fail(e, "attention launch");
            if ((e = attn_probe(step * D.L + l, false)) != cudaSuccess) return cuda_fail(e, "probe record");
            // x += W_o attn;  x += W_down (silu(W_g n) * W_u n),  n = RMSNorm(x)
            const int ha = D.Hq * D.hd;
            const NextPlanes ffn{ws.tc_xg, (const uint16_t *)W.ffn_norm[l], D.d, 0, TC_PLANES, 0, rows_per_seq,
                                 npad_of(R)};
            bool ffn_ready = false;
            if ((rc = tc_gemm(TC_RESID, R, ha, D.d, TC_PLANES, ctx->tm_o[l], ws.tc_xo, false, x, D.d, nullptr,
                              "o-proj launch", nullptr, &ffn, &ffn_ready)) != OSPREY_OK ||
                (!ffn_ready && (rc = planes(x, (const uint16_t *)W.ffn_norm[l], D.d, R, D.d, 0, ws.tc_xg, rows_per_seq,
                                            false, "gate/up operand")) != OSPREY_OK) ||
                (rc = tc_gemm(TC_GLU, R, D.d, 2 * D.F, TC_PLANES, ctx->tm_gate[l], ws.tc_xg, false, nullptr, 0,
                              ws.tc_xh, "gate/up launch", &ctx->tm_up[l])) != OSPREY_OK)
                return rc;
            // the down projection's reduction prepares the next layer's x half, or the
            // LM head's operand rows after the last layer
            NextPlanes nxt{};
            const NextPlanes *nxtp = nullptr;
            if (l + 1 < D.L) {
                nxt = NextPlanes{ws.tc_xq, (const uint16_t *)W.attn_norm[l + 1], 2 * D.d, D.d, TC_PLANES, 0,
                                 rows_per_seq, npad_of(R)};
                nxtp = &nxt;
            } else if (lm_tc) {
                const bool last_rows = ext && !block;   // one LM row per sequence: its last new row
                nxt = NextPlanes{ws.tc_xl, (const uint16_t *)W.final_norm, D.d, 0, TC_LM_PLANES, last_rows ? 1 : 0,
                                 rows_per_seq, npad_of(last_rows ? B : R)};
                nxtp = &nxt;
            }
            bool nxt_ready = false;
            if ((rc = tc_gemm(TC_RESID, R, D.F, D.d, TC_PLANES, ctx->tm_down[l], ws.tc_xh, false, x, D.d, nullptr,
                              "down launch", nullptr, nxtp, &nxt_ready)) != OSPREY_OK)
                return rc;
            xq_ready = nxt_ready && l + 1 < D.L;
            xl_ready = nxt_ready && l + 1 == D.L;
        }
        for (int l = 0; l < D.L && !tcp; ++l) {
            if (streamed && R == 1 && ctx->fused_layer) {
                LayerArgs la{};
                la.dim = D;
                la.map = map;
                la.W_qkv = (const uint16_t *)W.W_qkv[l];
                la.attn_norm = (const uint16_t *)W.attn_norm[l];
                la.W_o = (const uint16_t *)W.W_o[l];
                la.W_gate = (const uint16_t *)W.W_gate[l];
                la.W_up = (const uint16_t *)W.W_up[l];
                la.W_down = (const uint16_t *)W.W_down[l];
                la.ffn_norm = (const uint16_t *)W.ffn_norm[l];
                la.x = x;
                la.s = sb;
                la.q = ws.q;
                la.k_pages = (uint16_t *)kv->k_pages + l * layer_pages;
                la.v_pages = (uint16_t *)kv->v_pages + l * layer_pages;
                la.page_table = kv->page_table;
                la.max_pages = kv->max_pages_per_seq;
                la.n_splits = layer_fused_splits(D, max_ctx, ctx->sms);
                la.split_len = attn_split_len(max_ctx, la.n_splits);
                la.attn_part = ws.attn_part;
                la.attn_out = ws.attn_out;
                la.attn_ticket = ws.attn_ticket;
                la.h = ws.ffn_h;
                la.bar_count = ws.grid_bar;
                la.bar_gen = ws.grid_bar + 1;
                la.status = dev_status;
                for (int i = 0; i < D.hd / 2; ++i) la.inv_freq[i] = ctx->inv_freq[i];
                if ((e = launch_layer_fused(la, ctx->sms, s)) != cudaSuccess) return cuda_fail(e, "fused layer launch");
                continue;
            }
            g.map = map;
            g.R = R;
            g.x = x;
            g.s = sb;
            g.W = (const uint16_t *)W.W_qkv[l];
            g.W2 = nullptr;
            g.gain = (const uint16_t *)W.attn_norm[l];
            g.q = ws.q;
            g.k_pages = (uint16_t *)kv->k_pages + l * layer_pages;
            g.v_pages = (uint16_t *)kv->v_pages + l * layer_pages;
            int rc;
            if ((rc = gemv(G_QKV, "qkv launch")) != OSPREY_OK) return rc;
            AttnArgs at{};
            at.dim = D;
            at.map = map;
            at.R = R;
            at.n_splits = clu ? ctx->attn_cs : ns;
            at.split_len = attn_split_len(max_ctx, at.n_splits);
            at.q = ws.q;
            at.k_pages = g.k_pages;
            at.v_pages = g.v_pages;
            at.page_table = kv->page_table;
            at.max_pages = kv->max_pages_per_seq;
            at.part = ws.attn_part;
            at.out = ws.attn_out;
            at.ticket = ws.attn_ticket;
            at.status = dev_status;
            if ((e = attn_probe(step * D.L + l, true)) != cudaSuccess) return cuda_fail(e, "probe record");
            e = clu ? launch_attn_cluster(at, ctx->attn_cs, s) : launch_attn(at, s);
            if (e != cudaSuccess) return cuda_fail(e, "attention launch");
            if ((e = attn_probe(step * D.L + l, false)) != cudaSuccess) return cuda_fail(e, "probe record");
            if (streamed && R == 1 && ctx->fused_mlp) {
                MlpArgs ma{};
                ma.dim = D;
                ma.map = map;
                ma.W_o = (const uint16_t *)W.W_o[l];
                ma.W_gate = (const uint16_t *)W.W_gate[l];
                ma.W_up = (const uint16_t *)W.W_up[l];
                ma.W_down = (const uint16_t *)W.W_down[l];
                ma.ffn_norm = (const uint16_t *)W.ffn_norm[l];
                ma.attn = ws.attn_out;
                ma.x = x;
                ma.h = ws.ffn_h;
                ma.bar_count = ws.grid_bar;
                ma.bar_gen = ws.grid_bar + 1;
                ma.status = dev_status;
                if ((e = launch_mlp_fused(ma, ctx->sms, s)) != cudaSuccess) return cuda_fail(e, "fused mlp launch");
                continue;
            }
            g.W = (const uint16_t *)W.W_o[l];
            g.xin = ws.attn_out;
            if ((rc = gemv(G_OPROJ, "o-proj launch")) != OSPREY_OK) return rc;
            g.W = (const uint16_t *)W.W_gate[l];
            g.W2 = (const uint16_t *)W.W_up[l];
            g.gain = (const uint16_t *)W.ffn_norm[l];
            g.out = ws.ffn_h;
            if ((rc = gemv(G_GATEUP, "gate/up launch")) != OSPREY_OK) return rc;
            g.W = (const uint16_t *)W.W_down[l];
            g.W2 = nullptr;
            g.xin = ws.ffn_h;
            if ((rc = gemv(G_DOWN, "down launch")) != OSPREY_OK) return rc;
        }
        if (draft_hidden &&
            (e = launch_keep_hidden(x, ext, B, K, step, max_new, D.d, ws.seq_valid, ws.seq_nnew, draft_hidden, s)) !=
                cudaSuccess)
            return cuda_fail(e, "keep-hidden launch");
        const bool probe = ctx->probe_kind == OSPREY_PROBE_LM_HEAD && step < ctx->n_probe;
        if (probe && (e = probe_record(ctx->probe_begin[step], s)) != cudaSuccess)
            return cuda_fail(e, "probe record");
        if (block) {
            // every extend row: final RMSNorm -> LM head -> its own draw (row r of
            // sequence r / max_new proposes the token after it)
            const int rows = B * max_new;
            int rc;
            if (!xl_ready && (rc = planes(x, (const uint16_t *)W.final_norm, D.d, rows, D.d, 0, ws.tc_xl, max_new, false,
                                          "lm operand", TC_LM_PLANES)) != OSPREY_OK)
                return rc;
            LmPickArgs pk{};
            pk.B = rows;
            pk.K = 1;
            pk.step = 0;
            pk.max_new = max_new;
            pk.rows_per_valid = max_new;
            pk.valid = ws.seq_valid;
            pk.nnew = ws.seq_nnew;
            pk.tokens = draft_tokens;
            pk.qx = draft_qx;
            pk.stats = draft_stats;
            if ((rc = tc_lm(rows, draft_logits, D.V, pk)) != OSPREY_OK) return rc;
        } else if (topk <= 1 && B <= 2 && stream_supported(G_LM, D, B, ctx->sms)) {
            plan_into(G_LM);
            sa.W = (const uint16_t *)W.lm_head;
            sa.gain = (const uint16_t *)W.final_norm;
            sa.x_in = x;
            sa.src_is_ext = ext;
            sa.x_chain = ws.x_chain;
            sa.s_chain = ws.s_chain;
            sa.temperature = temperature;
            sa.u_draft = u_draft;
            sa.tokens = draft_tokens;
            sa.qx = draft_qx;
            sa.stats = draft_stats;
            sa.logits = draft_logits;
            sa.sup = ws.lm_sup;
            const StreamPlan lp = stream_plan(G_LM, D, ctx->sms);
            sa.nsup = lp.nsup;
            sa.run = lp.run;
            sa.cta_stats = ws.lm_cta_stats;
            sa.ticket = ws.lm_ticket;
            if ((e = launch_stream(G_LM, sa, B, s)) != cudaSuccess) return cuda_fail(e, "lm head launch");
        } else if (tc_rows(B) || topk > 1) {
            // final RMSNorm rows -> LM head with the sampling partials in its
            // epilogue (logits stored only into draft_logits) -> one pick per row
            // (topk candidates per row when drafting a tree)
            int rc;
            if (!xl_ready && (rc = planes(x, (const uint16_t *)W.final_norm, D.d, B, D.d, 0, ws.tc_xl, 1, ext,
                                          "lm operand", TC_LM_PLANES)) != OSPREY_OK)
                return rc;
            LmPickArgs pk{};
            pk.B = B;
            pk.K = K;
            pk.step = step;
            pk.max_new = max_new;
            pk.src_is_ext = ext;
            pk.topk = topk;
            pk.valid = ws.seq_valid;
            pk.nnew = ws.seq_nnew;
            pk.tokens = draft_tokens;
            pk.qx = draft_qx;
            pk.stats = draft_stats;
            pk.x_in = x;
            pk.x_chain = ws.x_chain;
            pk.s_chain = ws.s_chain;
            if (step + 1 < K && B > 2 && tc_rows(B)) {   // the next step's layers run on the tensor cores
                pk.qkv_planes = ws.tc_xq;
                pk.qkv_gain = (const uint16_t *)W.attn_norm[0];
                pk.eps = D.eps;
                pk.qkv_npad = npad_of(B);
                xq_next = true;
            }
            if ((rc = tc_lm(B, draft_logits ? draft_logits + (size_t)step * D.V : nullptr, (long long)K * D.V, pk)) !=
                OSPREY_OK)
                return rc;
        } else {
            LmArgs lm{};
            lm.dim = D;
            lm.map = map;
            lm.B = B;
            lm.K = K;
            lm.step = step;
            lm.max_new = max_new;
            lm.W = (const uint16_t *)W.lm_head;
            lm.gain = (const uint16_t *)W.final_norm;
            lm.embed = (const uint16_t *)W.embed;
            lm.x_in = x;
            lm.src_is_ext = ext;
            lm.x_chain = ws.x_chain;
            lm.s_chain = ws.s_chain;
            lm.temperature = temperature;
            lm.u_draft = u_draft;
            lm.tokens = draft_tokens;
            lm.qx = draft_qx;
            lm.stats = draft_stats;
            lm.logits = draft_logits;
            lm.warp_stats = ws.lm_stats;
            lm.ticket = ws.lm_ticket;
            const int blocks = lm_blocks(D.V, ctx->sms);
            lm.warps_total = blocks * 8;
            int rg = 1;
            while (rg < B && rg < 8) rg <<= 1;
            if ((e = launch_lm(lm, rg, blocks, s)) != cudaSuccess) return cuda_fail(e, "lm head launch");
        }
        if (probe && (e = probe_record(ctx->probe_end[step], s)) != cudaSuccess)
            return cuda_fail(e, "probe record");
    }
    return OSPREY_OK;
}

extern "C" int osprey_draft_step(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int max_new,
                                 const int32_t *n_new, const int32_t *tokens, const void *feats,
                                 float temperature, const float *u_draft, int32_t *draft_tokens,
                                 float *draft_qx, float *draft_stats, float *draft_logits,
                                 void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                 void *stream) {
    return draft_step_impl(ctx, kv, B, K, max_new, n_new, tokens, feats, temperature, u_draft, draft_tokens, draft_qx,
                           draft_stats, draft_logits, nullptr, workspace, workspace_bytes, dev_status, stream);
}

extern "C" int osprey_draft_step_hidden(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int max_new,
                                        const int32_t *n_new, const int32_t *tokens, const void *feats,
                                        float temperature, const float *u_draft, int32_t *draft_tokens,
                                        float *draft_qx, float *draft_stats, float *draft_hidden,
                                        void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                        void *stream) {
    if (!draft_hidden) {
        g_err[0] = 0;
        return fail(OSPREY_ERR_INVALID_ARG, "draft_hidden is required");
    }
    return draft_step_impl(ctx, kv, B, K, max_new, n_new, tokens, feats, temperature, u_draft, draft_tokens, draft_qx,
                           draft_stats, nullptr, draft_hidden, workspace, workspace_bytes, dev_status, stream);
}

extern "C" int osprey_draft_step_topk(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int topk, int max_new,
                                      const int32_t *n_new, const int32_t *tokens, const void *feats,
                                      float temperature, const float *u_draft, int32_t *cand, float *cand_qx,
                                      float *draft_stats, float *draft_logits, void *workspace,
                                      size_t workspace_bytes, int32_t *dev_status, void *stream) {
    if (topk < 1 || topk > 8) {
        g_err[0] = 0;
        return fail(OSPREY_ERR_INVALID_ARG, "topk must be in 1..8");
    }
    return draft_step_impl(ctx, kv, B, K, max_new, n_new, tokens, feats, temperature, u_draft, cand, cand_qx,
                           draft_stats, draft_logits, nullptr, workspace, workspace_bytes, dev_status, stream, false,
                           topk);
}

// ------------------------------------------------------------------ block drafting
// Sequences are drafted in groups whose block rows fit one tensor-core tile
// (TC_MAX_ROWS rows); each group's call re-reads the weights once.  Workspace:
// the block-mode draft layout of one group, then the group's token array
// [n][P], n_new [n] and broadcast features [n][P][feat_dim] bf16.
static int block_group(int B, int P) {
    const int g = TC_MAX_ROWS / P;
    return g < 1 ? 1 : (g < B ? g : B);
}

static size_t block_layout(const osprey_ctx *ctx, int n, int P, int max_pages, DraftWs *ws, void *base,
                           int32_t **tok, int32_t **nnew, uint16_t **feats) {
    size_t off = align256(draft_layout(ctx, n, 1, P, max_pages, ws, base, true));
    const size_t o_t = off;
    off = align256(off + 4ull * n * P);
    const size_t o_n = off;
    off = align256(off + 4ull * n);
    const size_t o_f = off;
    off = align256(off + 2ull * n * P * ctx->dim.feat);
    if (base) {
        *tok = (int32_t *)((char *)base + o_t);
        *nnew = (int32_t *)((char *)base + o_n);
        *feats = (uint16_t *)((char *)base + o_f);
    }
    return off;
}

static bool block_args_ok(const osprey_ctx *ctx, int B, int block, int max_pages) {
    return ctx && B >= 1 && B <= 65535 && block >= 4 && block <= TC_MAX_ROWS + 1 && max_pages >= 1 &&
           (long long)max_pages * ctx->dim.P < (1LL << 30);
}

extern "C" size_t osprey_dflash_workspace_bytes(const osprey_ctx *ctx, int B, int block, int max_pages_per_seq) {
    if (!block_args_ok(ctx, B, block, max_pages_per_seq)) return 0;
    const int P = block - 1;
    return block_layout(ctx, block_group(B, P), P, max_pages_per_seq, nullptr, nullptr, nullptr, nullptr, nullptr);
}

extern "C" int osprey_dflash_step(osprey_ctx *ctx, const osprey_kv *kv, int B, int block, const int32_t *anchors,
                                  int32_t mask_token, const void *feats, float temperature, const float *u_draft,
                                  int32_t *draft_tokens, float *draft_qx, float *draft_stats, float *draft_logits,
                                  void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream) {
    g_err[0] = 0;
    if (!ctx || !kv) return fail(OSPREY_ERR_INVALID_ARG, "null context or kv");
    if (B == 0) return OSPREY_OK;
    if (!block_args_ok(ctx, B, block, kv->max_pages_per_seq))
        return fail(OSPREY_ERR_INVALID_ARG, "B in 1..65535, block in 4..%d and max_pages_per_seq >= 1 required",
                    TC_MAX_ROWS + 1);
    if (!ctx->tc)
        return fail(OSPREY_ERR_SHAPE, "block drafting runs on the tensor cores; this context has none "
                                      "(OSPREY_TC=0 or no tcgen05)");
    if (mask_token < 0 || mask_token >= ctx->dim.V) return fail(OSPREY_ERR_INVALID_ARG, "mask_token out of range");
    if (!(temperature >= 0.f) || !std::isfinite(temperature))
        return fail(OSPREY_ERR_INVALID_ARG, "temperature must be finite and >= 0");
    if (!anchors || !feats || !draft_tokens || !workspace || !kv->k_pages || !kv->v_pages || !kv->page_table ||
        !kv->seq_len)
        return fail(OSPREY_ERR_INVALID_ARG, "null pointer");
    if (temperature > 0.f && !u_draft) return fail(OSPREY_ERR_INVALID_ARG, "u_draft is required when temperature > 0");
    if (((uintptr_t)feats | (uintptr_t)workspace) % 16)
        return fail(OSPREY_ERR_INVALID_ARG, "feats and workspace must be 16-byte aligned");
    const int P = block - 1, G = block_group(B, P);
    const Dims &D = ctx->dim;
    DraftWs ws{};
    int32_t *tok = nullptr, *nnew = nullptr;
    uint16_t *frep = nullptr;
    const size_t need = block_layout(ctx, G, P, kv->max_pages_per_seq, &ws, workspace, &tok, &nnew, &frep);
    if (workspace_bytes < need)
        return fail(OSPREY_ERR_CAPACITY, "workspace too small: %zu < %zu bytes", workspace_bytes, need);
    cudaStream_t s = (cudaStream_t)stream;
    for (int b0 = 0; b0 < B; b0 += G) {
        const int n = B - b0 < G ? B - b0 : G;
        BlockInArgs bi{n, P, D.feat, anchors + b0, mask_token, (const uint16_t *)feats + (size_t)b0 * D.feat,
                       tok, nnew, frep};
        cudaError_t e = launch_block_inputs(bi, s);
        if (e != cudaSuccess) return cuda_fail(e, "block inputs launch");
        osprey_kv kg = *kv;
        kg.page_table = kv->page_table + (size_t)b0 * kv->max_pages_per_seq;
        kg.seq_len = kv->seq_len + b0;
        const size_t o = (size_t)b0 * P;
        const int rc = draft_step_impl(ctx, &kg, n, 1, P, nnew, tok, frep, temperature, u_draft ? u_draft + o : nullptr,
                                       draft_tokens + o, draft_qx ? draft_qx + o : nullptr,
                                       draft_stats ? draft_stats + 2 * o : nullptr,
                                       draft_logits ? draft_logits + o * D.V : nullptr, nullptr, workspace,
                                       workspace_bytes, dev_status, stream, true);
        if (rc != OSPREY_OK) return rc;
    }
    return OSPREY_OK;
}

// ------------------------------------------------------------------ verify
extern "C" size_t osprey_verify_workspace_bytes(int B, int K, int V) {
    if (B < 1 || K < 1 || K > 15 || V < 1) return 0;
    return verify_workspace_layout(B, K, V, nullptr, nullptr);
}

extern "C" int osprey_verify(int B, int K, int V, int logits_dtype, const void *target_logits,
                             const void *draft_logits, const int32_t *draft_tokens, float temperature,
                             const float *u_accept, const float *u_sample, int32_t *out_tokens,
                             int32_t *n_accepted, uint8_t *flags, float *probs, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, void *stream) {
    g_err[0] = 0;
    if (B == 0) return OSPREY_OK;
    if (B < 0 || K < 1 || K > 15 || V < 1)
        return fail(OSPREY_ERR_INVALID_ARG, "B >= 0, K in 1..15 and V >= 1 required");
    if (logits_dtype != OSPREY_F32 && logits_dtype != OSPREY_BF16)
        return fail(OSPREY_ERR_DTYPE, "logits_dtype must be OSPREY_F32 or OSPREY_BF16");
    if (!(temperature >= 0.f) || !std::isfinite(temperature))
        return fail(OSPREY_ERR_INVALID_ARG, "temperature must be finite and >= 0");
    if (!target_logits || !draft_tokens || !out_tokens || !n_accepted || !flags || !workspace)
        return fail(OSPREY_ERR_INVALID_ARG, "null pointer");
    if (temperature > 0.f && (!draft_logits || !u_accept || !u_sample))
        return fail(OSPREY_ERR_INVALID_ARG, "draft_logits, u_accept and u_sample are required when temperature > 0");
    if ((long long)V * (K + 1) * B > (1LL << 40)) return fail(OSPREY_ERR_SHAPE, "logits too large");
    if ((long long)((V + 8191) / 8192) * (K + 1) * B >= (1LL << 31))
        return fail(OSPREY_ERR_SHAPE, "too many (sequence, row, chunk) blocks");
    VerifyArgs a{};
    const size_t need = verify_workspace_layout(B, K, V, &a, workspace);
    if (workspace_bytes < need)
        return fail(OSPREY_ERR_CAPACITY, "workspace too small: %zu < %zu bytes", workspace_bytes, need);
    a.B = B;
    a.K = K;
    a.V = V;
    a.dtype = logits_dtype;
    a.temperature = temperature;
    a.target = target_logits;
    a.draft = draft_logits;
    a.tokens = draft_tokens;
    a.u_accept = u_accept;
    a.u_sample = u_sample;
    a.out_tokens = out_tokens;
    a.n_accepted = n_accepted;
    a.flags = flags;
    a.probs = probs;
    a.status = dev_status;
    // the arrival counters start at zero on every call, so a call that ran out
    // of a bounded wait leaves nothing stale for the next one
    cudaError_t e = cudaMemsetAsync(a.ticket1, 0, a.counter_bytes, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "clearing the verify counters");
    e = launch_verify(a, (cudaStream_t)stream);
    return e == cudaSuccess ? OSPREY_OK : cuda_fail(e, "verify launch");
}

// ------------------------------------------------------------------ tree verify
extern "C" int osprey_verify_tree(int B, int K, int topk, int V, int logits_dtype, const void *target_logits,
                                  const void *draft_logits, const int32_t *cand, float temperature,
                                  const float *u_accept, const float *u_sample, int32_t *out_tokens,
                                  int32_t *n_accepted, int32_t *branch, uint8_t *flags, int32_t *dev_status,
                                  void *stream) {
    g_err[0] = 0;
    if (B == 0) return OSPREY_OK;
    if (B < 0 || B > 65535 || K < 1 || K > 64 || topk < 1 || topk > 8 || V < 1 || V > (1 << 20))
        return fail(OSPREY_ERR_INVALID_ARG, "B in 0..65535, K in 1..64, topk in 1..8 and V in 1..2^20 required");
    if (logits_dtype != OSPREY_F32 && logits_dtype != OSPREY_BF16)
        return fail(OSPREY_ERR_DTYPE, "logits_dtype must be OSPREY_F32 or OSPREY_BF16");
    if (!(temperature >= 0.f) || !std::isfinite(temperature))
        return fail(OSPREY_ERR_INVALID_ARG, "temperature must be finite and >= 0");
    if (!target_logits || !cand || !out_tokens || !n_accepted || !branch || !flags)
        return fail(OSPREY_ERR_INVALID_ARG, "null pointer");
    if (temperature > 0.f && (!draft_logits || !u_accept || !u_sample))
        return fail(OSPREY_ERR_INVALID_ARG, "draft_logits, u_accept and u_sample are required when temperature > 0");
    VerifyTreeArgs a{B, K, topk, V, logits_dtype, temperature, target_logits, draft_logits, cand, u_accept, u_sample,
                     out_tokens, n_accepted, branch, flags, dev_status};
    const cudaError_t e = launch_verify_tree(a, (cudaStream_t)stream);
    return e == cudaSuccess ? OSPREY_OK : cuda_fail(e, "tree verify launch");
}

// ------------------------------------------------------------------ logits-free verify
// Workspace: the verify layout (counters, partials, decisions, chunk sums), then
// for one group of up to TC_MAX_ROWS sequences the gathered kept states
// [rows][d] float, their operand planes [TC_PLANES][npad][d] bf16, the
// recomputed decision-row logits [rows][V] float (the draft step's LM-head GEMM:
// the same operand planes, unsplit, so the rows come out the same).
struct HiddenWs {
    float *rows;
    uint16_t *planes;
    float *z;
    int group, npad;
};

static size_t verify_hidden_layout(const osprey_ctx *ctx, int B, int K, VerifyArgs *a, void *base, HiddenWs *hw) {
    const Dims &D = ctx->dim;
    size_t off = align256(verify_workspace_layout(B, K, D.V, a, base));
    const int group = B < TC_MAX_ROWS ? B : TC_MAX_ROWS;
    const int npad = (group + 15) / 16 * 16;
    const size_t o_r = off;
    off = align256(off + 4ull * group * D.d);
    const size_t o_p = off;
    off = align256(off + 2ull * TC_PLANES * npad * D.d);
    const size_t o_z = off;
    off = align256(off + 4ull * group * D.V);
    if (hw && base) {
        char *p = (char *)base;
        hw->rows = (float *)(p + o_r);
        hw->planes = (uint16_t *)(p + o_p);
        hw->z = (float *)(p + o_z);
        hw->group = group;
        hw->npad = npad;
    }
    return off;
}

extern "C" size_t osprey_verify_hidden_workspace_bytes(const osprey_ctx *ctx, int B, int K) {
    if (!ctx || B < 1 || K < 1 || K > 15) return 0;
    return verify_hidden_layout(ctx, B, K, nullptr, nullptr, nullptr);
}

extern "C" int osprey_verify_hidden(osprey_ctx *ctx, int B, int K, int logits_dtype, const void *target_logits,
                                    const float *draft_hidden, const float *draft_qx, const float *draft_stats,
                                    const int32_t *draft_tokens, float temperature, const float *u_accept,
                                    const float *u_sample, int32_t *out_tokens, int32_t *n_accepted, uint8_t *flags,
                                    float *probs, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                    void *stream) {
    g_err[0] = 0;
    if (!ctx) return fail(OSPREY_ERR_INVALID_ARG, "null context");
    if (B == 0) return OSPREY_OK;
    const Dims &D = ctx->dim;
    const int V = D.V;
    if (B < 0 || K < 1 || K > 15) return fail(OSPREY_ERR_INVALID_ARG, "B >= 0 and K in 1..15 required");
    if (logits_dtype != OSPREY_F32 && logits_dtype != OSPREY_BF16)
        return fail(OSPREY_ERR_DTYPE, "logits_dtype must be OSPREY_F32 or OSPREY_BF16");
    if (!(temperature > 0.f) || !std::isfinite(temperature))
        return fail(OSPREY_ERR_INVALID_ARG,
                    "temperature must be finite and > 0 (greedy verification reads no draft rows: osprey_verify)");
    if (!target_logits || !draft_hidden || !draft_qx || !draft_stats || !draft_tokens || !u_accept || !u_sample ||
        !out_tokens || !n_accepted || !flags || !workspace)
        return fail(OSPREY_ERR_INVALID_ARG, "null pointer");
    if ((uintptr_t)workspace % 16) return fail(OSPREY_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
    if (!ctx->tc)
        return fail(OSPREY_ERR_SHAPE, "the decision rows are recomputed on the tensor cores; this context has no "
                                      "tensor-core path (OSPREY_TC=0 or no tcgen05)");
    if ((long long)V * (K + 1) * B > (1LL << 40)) return fail(OSPREY_ERR_SHAPE, "logits too large");
    if ((long long)((V + 8191) / 8192) * (K + 1) * B >= (1LL << 31))
        return fail(OSPREY_ERR_SHAPE, "too many (sequence, row, chunk) blocks");
    VerifyArgs a{};
    HiddenWs hw{};
    const size_t need = verify_hidden_layout(ctx, B, K, &a, workspace, &hw);
    if (workspace_bytes < need)
        return fail(OSPREY_ERR_CAPACITY, "workspace too small: %zu < %zu bytes", workspace_bytes, need);
    a.B = B;
    a.K = K;
    a.V = V;
    a.dtype = logits_dtype;
    a.temperature = temperature;
    a.target = target_logits;
    a.draft = nullptr;
    a.tokens = draft_tokens;
    a.u_accept = u_accept;
    a.u_sample = u_sample;
    a.out_tokens = out_tokens;
    a.n_accepted = n_accepted;
    a.flags = flags;
    a.probs = probs;
    a.status = dev_status;
    a.qx_in = draft_qx;
    a.stats_in = draft_stats;
    a.zrec = hw.z;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(a.ticket1, 0, a.counter_bytes, s);   // counters start at zero on every call
    if (e != cudaSuccess) return cuda_fail(e, "clearing the verify counters");
    // 1. target row statistics, the acceptance chain and the decision row r
    if ((e = launch_verify_hidden_stats(a, s)) != cudaSuccess) return cuda_fail(e, "verify launch");
    for (int b0 = 0; b0 < B; b0 += hw.group) {
        const int n = B - b0 < hw.group ? B - b0 : hw.group;
        const int npad = (n + 15) / 16 * 16;
        // 2. the kept state of each decision row -> final RMSNorm -> bf16 planes
        if ((e = launch_decision_rows(a.dec, draft_hidden, K, D.d, b0, n, hw.rows, s)) != cudaSuccess)
            return cuda_fail(e, "decision-row launch");
        PlaneArgs pl{};
        pl.src = hw.rows;
        pl.gain = (const uint16_t *)ctx->w.final_norm;
        pl.eps = D.eps;
        pl.d = D.d;
        pl.R = n;
        pl.npad = npad;
        pl.ld = D.d;
        pl.col0 = 0;
        pl.dst = hw.planes;
        pl.max_new = 1;
        pl.rows_per_seq = 1;
        pl.npl = TC_LM_PLANES;
        if ((e = launch_planes(pl, s)) != cudaSuccess) return cuda_fail(e, "decision-row operand launch");
        // 3. their draft logits on the tensor cores (the draft step's LM head GEMM)
        CUtensorMap xm;
        if (!tc_encode_operand(&xm, hw.planes, TC_LM_PLANES, npad, D.d))
            return fail(OSPREY_ERR_INVALID_ARG, "decision-row tensor map encoding failed");
        TcArgs ta{};
        ta.epi = TC_STORE;
        ta.R = n;
        ta.npad = npad;
        ta.K = D.d;
        ta.nout = V;
        ta.planes = TC_LM_PLANES;
        ta.y = hw.z;
        ta.x = hw.z;
        ta.ldy = V;
        ta.status = dev_status;   // unsplit, like the draft step's LM head: the same logits bit for bit
        if ((e = launch_tc(ta, ctx->tm_lm, xm, ctx->sms, s)) != cudaSuccess) return cuda_fail(e, "decision-row lm head");
        // 4. the emitted token of each sequence of the group
        if ((e = launch_verify_hidden_sample(a, b0, n, s)) != cudaSuccess) return cuda_fail(e, "verify sample launch");
    }
    return OSPREY_OK;
}
