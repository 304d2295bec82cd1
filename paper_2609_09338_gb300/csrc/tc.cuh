// Batched-row draft step on the 5th-generation tensor cores (tcgen05): the
// projections of Sec. 3.3 (Eq. 1-3, the MLP and the LM head) as streamed
// swap-AB GEMMs, Y[R x Nout] = X[R x K] . W[Nout x K]^T, for 3..80 rows.
//
// Weights are the M = 128 operand, streamed tile by tile with 2-D TMA (128-byte
// swizzle); the R activation rows are the N operand (padded to a multiple of
// 16).  The LM head multiplies two weight tiles against each stage's operand
// planes (twice the weight bytes in flight per byte of operand reloaded).  Activations are float32 between kernels; for the tensor cores each is
// split into three bf16 planes, q0 = bf16(x), q1 = bf16(x - q0), q2 =
// bf16(x - q0 - q1), and every k-step issues one MMA per plane into the same
// float32 accumulator, so the product keeps the 24 mantissa bits of x (bf16
// inputs such as the target features use a single plane).  Two planes (16
// bits) were not enough: attention over thousands of cached keys turns a 1e-5
// relative error in q into logit errors two orders above the float32 path's.  The reduction is accumulated in segments of
// 512 (a fresh TMEM accumulator each) whose float32 sum the epilogue keeps, so
// no accumulation chain in the tensor core is longer than 32 MMA steps per
// plane (a long chain loses precision against a float32 tree sum).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "draft.cuh"

namespace osp {

// TC_LM: the LM head; per row and 32-id group of the vocabulary the epilogue
// keeps only (max of logits/T, sum of exp(logits/T - max), argmax logit and its
// id), and stores the logits only when y is given.
enum TcEpi { TC_STORE = 0, TC_RESID = 1, TC_GLU = 2, TC_LM = 3 };
constexpr int TC_LM_GROUP = 32;    // vocabulary ids per LM-head partial (one epilogue warp's lanes)
// The LM head's operand rows enter as two bf16 planes (16 significant bits):
// a logit's error from the dropped bits is a sum of d random terms of
// 2^-17 |h_k| |W_jk|, about 5e-6 at d 1024, the float32 GEMV's own level; the
// smaller stage lets three weight tiles per CTA be in flight instead of two.
constexpr int TC_LM_PLANES = 2;

constexpr int TC_MAX_ROWS = 80;    // activation rows per GEMM: three accumulators fit a CTA's 256 TMEM columns
constexpr int TC_PLANES = 3;       // bf16 planes of a float32 operand

struct TcArgs {
    int epi;           // TcEpi
    int R, npad;       // rows, rows padded to a multiple of 16
    int K;             // reduction length (multiple of 64)
    int nout;          // output features (tiles of 128, the last one may be partial)
    int nout_a;        // features [0, nout_a) from the first weight map, the rest from the second
    int planes;        // 1 (bf16 input) or TC_PLANES (split float32 input)
    float *y;          // TC_STORE: [R][ldy] float32 output
    int ldy;
    float *x;          // TC_RESID: [R][ldy] float32, +=
    uint16_t *h;       // TC_GLU: [TC_PLANES][npad][nout_a] bf16 planes of silu(gate) * up
    int32_t *status;
    // TC_LM: partials [R][lm_nsub] (lm_nsub = ceil(nout / 32)), 1/T (1 for greedy)
    float4 *lm_part;
    int lm_nsub;
    float lm_invT;
    // TC_RESID with a split-K reduction and pl_dst set: the reduction runs one
    // block per row and also writes the updated rows' RMS-normalised planes for
    // the next GEMM (gain pl_gain, pl_npl planes [pl_npl][pl_npad][pl_ld] from
    // column pl_col0).  pl_map 0: row n to planes row n (zeros unless sequence
    // n / pl_rows_per_seq is valid and, with several rows per sequence, n is one
    // of its new rows); 1: the last new row of each sequence to its planes row
    // (zeros for an invalid sequence).
    uint16_t *pl_dst;
    const uint16_t *pl_gain;
    float pl_eps;
    int pl_ld, pl_col0, pl_npl, pl_npad, pl_map, pl_rows_per_seq, pl_max_new;
    const int *pl_valid, *pl_nnew;
    // split-K: per-range float32 partials [nsplit][R][nout] (null: no split)
    float *part;
    long long part_cap;   // floats available in part
    int nsplit, kbps;     // set by launch_tc
    int segkb;            // k-blocks per accumulation segment, set by launch_tc
};

// Host side.  Tensor maps: weights [rows][K] bf16 with a 64 x 128 box, operand
// planes [planes * npad][K] bf16 with a 64 x npad box, both 128-byte swizzled.
bool tc_available();   // the driver exposes tensor-map encoding and the device is sm_100+
bool tc_encode_weight(CUtensorMap *m, const void *w, int rows, int K);
bool tc_encode_operand(CUtensorMap *m, const void *x, int planes, int npad, int K);
// a single bf16 plane of `rows` rows read in place (rows past `rows` read as zero)
bool tc_encode_rows(CUtensorMap *m, const void *x, int rows, int npad, int K);
size_t tc_smem_bytes(int npad, int planes, int na);
cudaError_t tc_set_attributes();
// SwiGLU runs as one GEMM over the gate rows (map wa) and the up rows (map wb),
// nout = 2 nout_a; its partials always go to `part`, and the reduction forms
// silu(gate) * up.  Outputs narrower than the CTA slots are split along K
// (tc_nsplit ranges per 128-feature tile); the float32 partials are then summed
// in range order by a reduction kernel that applies the epilogue.
int tc_nsplit(int nout, int K, int sms);
cudaError_t launch_tc(const TcArgs &a, const CUtensorMap &wa, const CUtensorMap &xm, int sms, cudaStream_t s);
// *planes_done (when given) tells whether the reduction did the follow-up work:
// wrote the pl_* planes (TC_RESID), or RoPE and the K/V write of `rope`
// (TC_STORE of the QKV projection) instead of storing y.  Otherwise the caller
// does it itself.
struct QkvPostArgs;
cudaError_t launch_tc2(const TcArgs &a, const CUtensorMap &wa, const CUtensorMap &wb, const CUtensorMap &xm, int sms,
                       cudaStream_t s, bool *planes_done = nullptr, const QkvPostArgs *rope = nullptr);

// Operand preparation: rows of float32 (optionally RMS-normalised with a bf16
// gain) written as bf16 planes [TC_PLANES][npad][ld] starting at column col0.
struct PlaneArgs {
    const float *src;          // row r at src + src_row(r) * d
    const uint16_t *gain;      // RMSNorm gain, or null for a plain copy
    float eps;
    int d, R, npad, ld, col0;
    uint16_t *dst;
    // row selection: r itself, or (LM at the extend step) b*max_new + n_new[b] - 1
    const int *nnew;
    int max_new, last_of_seq;
    const int *valid;          // rows of invalid sequences are written as zeros (may be null)
    int rows_per_seq;
    int npl;                   // planes written (0: TC_PLANES)
    const float *src2;         // optional second source, same rows, written plain at column col2
    int col2;
};
cudaError_t launch_planes(const PlaneArgs &a, cudaStream_t s);

// RoPE and the paged K/V write from the QKV GEMM output y [R][(Hq+2Hkv)hd].
struct QkvPostArgs {
    Dims dim;
    RowMap map;
    int R;
    const float *y;
    float *q;
    uint16_t *k_pages, *v_pages;
    const int32_t *page_table;
    int max_pages;
    double inv_freq[64];       // rotary frequencies theta^(-2i/hd)
};
cudaError_t launch_qkv_post(const QkvPostArgs &a, cudaStream_t s);

// Sampling each LM-head row (Sec. 3.1 draft distribution q = softmax(z / T))
// from the TC_LM partials: the inverse CDF at u_draft[b][step] over ascending
// ids picks a 32-id group from the partials, then the id inside it from that
// group's logits, recomputed from the LM head's operand planes; T = 0 takes the
// argmax (lowest id).  Writes the token, q(token), (max, log-sum-exp) and, when
// a next chain step follows, the next chain row (context slot = x_L, residual =
// E[token]).  Row b belongs to sequence b / rows_per_valid (0 or 1: itself).
// topk > 1 (tree drafting): k candidates per row, [B][K][k] in tokens and qx;
// sampled: k independent inverse-CDF draws at u_draft[b][step][j]; greedy: the
// k highest logits in descending order (ties to the lowest id).  Candidate 0
// continues the chain.
struct LmPickArgs {
    Dims dim;
    int B, K, step, max_new, src_is_ext, rows_per_valid;
    int topk;                  // candidates per row (0 or 1: one)
    const int *valid, *nnew;
    const float4 *part;        // [B][nsub] TC_LM partials
    int nsub;
    const uint16_t *planes;    // [TC_PLANES][npad][d] bf16 planes of the LM head's rows
    int npad;
    const uint16_t *W;         // LM head [V][d]
    float temperature;
    const float *u_draft;
    int32_t *tokens;
    float *qx, *stats;
    const float *x_in;         // residual rows of the step (x_ext or x_chain)
    float *x_chain, *s_chain;
    const uint16_t *embed;
    // when set (chain drafting on the tensor cores), the next chain row's QKV
    // operand too: [TC_PLANES][qkv_npad][2 d] bf16 planes of [s; RMSNorm(x) * qkv_gain]
    uint16_t *qkv_planes;
    const uint16_t *qkv_gain;
    float eps;
    int qkv_npad;
};
cudaError_t launch_lm_pick(const LmPickArgs &a, cudaStream_t s);
// Block drafting inputs (EAGLE-style DFlash): for row r = b*P + j of n
// sequences, tokens[r] = anchor[b] (j = 0) or mask (j > 0); feats_rep[r] =
// feats[b] (feat_dim bf16, broadcast over the block); nnew[b] = P.
struct BlockInArgs {
    int n, P, feat;
    const int32_t *anchors;
    int32_t mask;
    const uint16_t *feats;
    int32_t *tokens, *nnew;
    uint16_t *feats_rep;
};
cudaError_t launch_block_inputs(const BlockInArgs &a, cudaStream_t s);
// x[r] = E[tokens[r]] (float32) for the active extend rows r = b*max_new + j, j < n_new[b].
struct EmbedArgs {
    int d, R, max_new;
    const int *valid, *nnew;
    const int32_t *tokens;
    const uint16_t *embed;
    float *x;
};
cudaError_t launch_embed_rows(const EmbedArgs &a, cudaStream_t s);

}  // namespace osp
