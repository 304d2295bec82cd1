// Draft-step kernel interface (CUDA-core GEMV path for up to 8 rows per group).
// Activations between kernels are float32; weights and the KV cache are bf16.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "osprey.h"

namespace osp {

struct Dims {
    int d, L, Hq, Hkv, hd, F, V, feat, P;
    float eps;
};

// Workspace views of one draft call.
struct DraftWs {
    int *seq_valid, *seq_pos0, *seq_nnew;  // [B]
    int *attn_ticket;                      // [R_ext * Hkv]
    int *lm_ticket;                        // [groups]
    unsigned *grid_bar;                    // [2] grid barrier (count, generation)
    float *x_ext;                          // [B*max_new][d]  residual stream, extend rows
    float *s_ext;                          // [B*max_new][d]  context slot (c)
    float *x_chain;                        // [B][d]          residual stream, chain rows
    float *s_chain;                        // [B][d]          context slot (fed-back x_L)
    float *q;                              // [R_ext][Hq*hd]  rotated queries
    float *attn_part;                      // [R_ext][Hq][n_splits][hd+2]
    float *attn_out;                       // [R_ext][Hq*hd]
    float *ffn_h;                          // [R_ext][F]
    float4 *lm_stats;                      // [B][lm_warps]
    float2 *lm_sup;                        // [B][blocks][nsup] run statistics of the streamed LM head
    float4 *lm_cta_stats;                  // [B][sms]
    // tensor-core path (rows padded to np <= 80): bf16 operand planes [TC_PLANES][np][...]
    uint16_t *tc_xq;                       // [P][np][2d]    [s; RMSNorm(x)] for QKV
    float *tc_yq;                          // [np][(Hq+2Hkv)hd] QKV output before RoPE
    uint16_t *tc_xo;                       // [P][np][Hq*hd] attention output
    uint16_t *tc_xg;                       // [P][np][d]     RMSNorm(x) for gate/up
    float *tc_part;                        // split-K partials of the projections
    long long tc_part_cap;
    uint16_t *tc_xh;                       // [P][np][F]     SwiGLU hidden (down operand)
    uint16_t *tc_xl;                       // [P][np][d]     final RMSNorm rows for the LM head
    float4 *rs_part;                       // [B][V/4096]    row-sampler chunk partials
    int *rs_ticket;                        // [B]
    int *counters;                         // attn_ticket .. rs_ticket: one contiguous block
    int n_counters;
    int n_splits_max, lm_warps_max;
};

// Which rows a launch works on: extend rows (step 0, rows_per_seq = max_new,
// row r = b*max_new + j, active for j < n_new[b]) or the chain row of step k
// (rows_per_seq = 1, row r = b, position pos0 + n_new + k - 1).
struct RowMap {
    const int *valid, *pos0, *nnew;
    int rows_per_seq, step;
    __device__ __forceinline__ bool row(int r, int &b, int &pos) const {
        b = r / rows_per_seq;
        const int j = r - b * rows_per_seq;
        if (!valid[b]) return false;
        const int nn = nnew[b];
        if (step == 0) {
            if (j >= nn) return false;
            pos = pos0[b] + j;
        } else {
            pos = pos0[b] + nn + step - 1;
        }
        return true;
    }
};

struct GemvArgs {
    Dims dim;
    RowMap map;
    int R;                        // rows of this step (B * rows_per_seq)
    const uint16_t *W, *W2;       // weight matrix (and the up matrix for gate/up)
    const uint16_t *gain;         // RMSNorm gain of the prologue (qkv, gate/up)
    const uint16_t *embed;        // feature projection: embedding gather
    const int32_t *tokens;        // [B][max_new]
    const uint16_t *feats;        // [B][max_new][feat]
    int max_new;
    float *x;                     // residual stream of this step
    float *s;                     // context slot of this step
    const float *xin;             // activation input (attn_out / ffn_h)
    float *out;                   // gate/up output (ffn_h)
    float *q;                     // rotated queries
    uint16_t *k_pages, *v_pages;  // this layer's pages
    const int32_t *page_table;
    int max_pages, n_pages;
    double inv_freq[64];          // theta^(-2i/hd)
};

struct AttnArgs {
    Dims dim;
    RowMap map;
    int R, n_splits, split_len;
    const float *q;
    const uint16_t *k_pages, *v_pages;
    const int32_t *page_table;
    int max_pages;
    float *part;
    float *out;
    // when set, the output rows go to the O projection's tensor-core operand
    // instead of out: three bf16 planes [3][npad][Hq hd]
    uint16_t *out_planes;
    int npad;
    int *ticket;
    int32_t *status;
};

struct LmArgs {
    Dims dim;
    RowMap map;
    int B, K, step, max_new;
    const uint16_t *W, *gain, *embed;
    const float *x_in;            // residual of the step's rows (x_ext or x_chain)
    int src_is_ext;               // extend step: read row b*max_new + n_new[b] - 1
    float *x_chain;
    float *s_chain;
    float temperature;
    const float *u_draft;
    int32_t *tokens;
    float *qx, *stats, *logits;
    float4 *warp_stats;
    int *ticket;
    int warps_total;              // gridDim.x * 8 (stats entries per row)
};

struct PrepArgs {
    int B, K, max_new, max_pages, n_pages, P, V;
    int32_t *seq_len;
    const int32_t *n_new, *tokens, *page_table;
    int *valid, *pos0, *nnew;
    int32_t *draft_tokens;
    int32_t *status;
    // the call's arrival counters and grid-barrier words, zeroed here so that a
    // call that ran out of a bounded wait leaves no stale count to the next one
    int *counters;
    int n_counters;
    int commit;    // rows committed per sequence (0: all n_new rows)
    int n_out;     // draft tokens per sequence set to -1 for a skipped sequence (0: K)
};

enum GemvMode { G_FEAT = 0, G_QKV = 1, G_OPROJ = 2, G_GATEUP = 3, G_DOWN = 4, G_LM = 5 };

// Arguments of the TMA-streamed GEMV (stream.cu): one or two activation rows.
struct StreamArgs {
    Dims dim;
    RowMap map;
    int mode, R, B, K, step, max_new;
    const uint16_t *W, *W2, *gain, *embed;
    float *x;                     // residual stream (read by qkv/gateup, += by oproj/down)
    const float *s;               // context slot (qkv)
    const float *xin;             // attention output (oproj) / SwiGLU hidden (down)
    float *out;                   // SwiGLU hidden (gateup)
    float *q;
    uint16_t *k_pages, *v_pages;
    const int32_t *page_table;
    int max_pages;
    double inv_freq[64];
    // LM head
    const float *x_in;
    int src_is_ext;
    float *x_chain, *s_chain;
    float temperature;
    const float *u_draft;
    int32_t *tokens;
    float *qx, *stats, *logits;   // logits: the caller's draft_logits (optional output)
    float2 *sup;                  // [B][blocks][nsup] (max, sum exp) of logits/T per run of `run` stages
    int nsup, run;                // runs per block (entries reserved per block in sup), stages per run
    float4 *cta_stats;            // [B][blocks]
    int *ticket;                  // [groups]
    int32_t *status;
    // plan (stream_plan)
    int items, n_items, n_stages, stage_bytes, blocks;
};

struct StreamPlan {
    int items, n_items, n_stages, stage_bytes, blocks;
    int nsup;   // LM head: runs of stages per block (second sampling level, <= 32)
    int run;    // LM head: stages per run
    size_t smem;
};

// Batch-1 chain steps: O-proj + residual, RMSNorm + gate/up + SwiGLU and
// down + residual of one layer in one launch (one block per SM, every block's
// weight slices requested before griddepcontrol.wait, two grid barriers).
struct MlpArgs {
    Dims dim;
    RowMap map;                       // row 0 of the step
    const uint16_t *W_o, *W_gate, *W_up, *W_down, *ffn_norm;
    const float *attn;                // [Hq hd] attention output of the row
    float *x;                         // [d] residual stream of the row
    float *h;                         // [F] SwiGLU hidden (scratch)
    unsigned *bar_count, *bar_gen;    // grid barrier words; count zero between uses
    int32_t *status;
};
bool mlp_fused_supported(const Dims &D, int sms);
cudaError_t launch_mlp_fused(const MlpArgs &a, int sms, cudaStream_t s);

// Batch-1 chain steps: a whole drafter layer in one launch (one block per SM):
// RMSNorm + expanded QKV + RoPE + K/V write | split-KV attention (the last
// split of a KV head merges) | O-proj + residual | RMSNorm + gate/up + SwiGLU |
// down + residual, each '|' a grid barrier.
struct LayerArgs {
    Dims dim;
    RowMap map;                       // row 0 of the step
    const uint16_t *W_qkv, *attn_norm, *W_o, *W_gate, *W_up, *W_down, *ffn_norm;
    float *x;                         // [d] residual stream of the row
    const float *s;                   // [d] context slot of the row
    float *q;                         // [Hq hd] rotated queries (scratch)
    uint16_t *k_pages, *v_pages;      // this layer's pages
    const int32_t *page_table;
    int max_pages;
    int n_splits, split_len;          // attention: key ranges per KV head (Hkv x n_splits <= grid)
    float *attn_part;                 // [Hq][n_splits][hd + 2]
    float *attn_out;                  // [Hq hd]
    int *attn_ticket;                 // [Hkv], zero between uses
    float *h;                         // [F] SwiGLU hidden (scratch)
    unsigned *bar_count, *bar_gen;    // grid barrier words; count zero between uses
    int32_t *status;
    double inv_freq[64];
};
bool layer_fused_supported(const Dims &D, int sms);
int layer_fused_splits(const Dims &D, int max_ctx, int sms);
cudaError_t launch_layer_fused(const LayerArgs &a, int sms, cudaStream_t s);

StreamPlan stream_plan(GemvMode mode, const Dims &D, int sms);
bool stream_supported(GemvMode mode, const Dims &D, int rg, int sms);
cudaError_t launch_stream(GemvMode mode, const StreamArgs &a, int rg, cudaStream_t s);
cudaError_t stream_set_attributes();

cudaError_t launch_prepare(const PrepArgs &a, cudaStream_t s);
// hidden[b][step] <- the last layer's output row that feeds draft token `step`
// of sequence b (extend step: row b*max_new + n_new[b] - 1; chain: row b);
// zeros for a sequence the call skipped
cudaError_t launch_keep_hidden(const float *x, bool ext, int B, int K, int step, int max_new, int d,
                               const int *valid, const int *nnew, float *hidden, cudaStream_t s);
cudaError_t launch_gemv(GemvMode mode, const GemvArgs &a, int rg, int sms, cudaStream_t s);
cudaError_t launch_attn(const AttnArgs &a, cudaStream_t s);
// Cluster size (16 or 8) the on-chip-merge attention can run with on the
// current device for this shape, 0 if clusters are not available.
int attn_cluster_size(const Dims &D);
cudaError_t launch_attn_cluster(const AttnArgs &a, int cs, cudaStream_t s);
cudaError_t launch_lm(const LmArgs &a, int rg, int blocks, cudaStream_t s);
int attn_splits(int R, int Hkv, int max_ctx, int sms);
int attn_split_len(int max_ctx, int n_splits);
int lm_blocks(int V, int sms);
size_t gemv_smem(GemvMode mode, const Dims &d, int rg);
int gemv_rg(GemvMode mode, const Dims &d, int R);
cudaError_t draft_set_attributes();

}  // namespace osp
