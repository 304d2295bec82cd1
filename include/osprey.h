/*
 * osprey.h - C ABI of the speculative-decoding hot path (draft step + verify)
 * for Osprey-style drafters on one NVIDIA GB300 (sm_103a).
 *
 * The path, after the paper:
 *   - Sec. 3.1: a drafter q proposes K tokens after a prefix; the frozen target p
 *     verifies them in one pass with the standard speculative-sampling rule
 *     (Leviathan et al.), which Osprey does not modify.
 *   - Sec. 3.3, Eq. 1: c_t = W_c [h_low; h_mid; h_high] projects three target
 *     hidden states into the drafter width and feeds every attention layer.
 *   - Sec. 3.3, Eq. 2-3: each layer's QKV projection reads [c_{t-1}; z_t]
 *     through W~_qkv = [W_ctx  W_qkv] (context columns first).
 *   - Sec. 3.4: inside a chain the drafter's own hidden state (the last layer's
 *     residual output, before the final norm) takes the context slot.
 *   - Sec. 4 (inference settings): chain drafting with topk = 1.
 *
 * Conventions for every entry point:
 *   - All tensor arguments are DEVICE pointers owned by the caller and borrowed
 *     for the duration of the (asynchronous) call.  The library allocates no
 *     device memory on these paths; scratch comes from a caller workspace.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and returns before it completes.  Nothing is synchronised.
 *   - The return value is OSPREY_OK or a negative OSPREY_ERR_* code.  Argument
 *     errors the host can see are reported before anything is launched;
 *     osprey_last_error() then holds a message (thread-local).
 *   - Errors only the device can see (a token id out of range, a sequence whose
 *     pages cannot hold the rows) are written to the caller's int32
 *     `dev_status` word (first error wins; it is never cleared by the library:
 *     the caller zeroes it).  The affected sequence's outputs are filled with
 *     -1 / 0 and the other sequences are unaffected.
 *   - A workspace needs no initialisation: every call clears the arrival
 *     counters it uses, on its stream, before the kernels that count (the
 *     draft step in its first kernel, verification with a memset), so a call
 *     that ran out of a bounded wait leaves nothing stale for the next one.  A
 *     workspace must not be shared by calls that can run at the same time.
 *   - bf16 is IEEE-754 binary32 truncated to its top 16 bits (round to nearest
 *     even by the producer); all row-major, no padding.
 */
#ifndef OSPREY_H
#define OSPREY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define OSPREY_MAX_LAYERS 8

enum {
    OSPREY_OK = 0,
    OSPREY_ERR_INVALID_ARG = -1, /* null pointer, bad count, bad enum */
    OSPREY_ERR_SHAPE = -2,       /* a dimension the kernels do not support */
    OSPREY_ERR_DTYPE = -3,       /* unknown logits dtype */
    OSPREY_ERR_CAPACITY = -4,    /* pages or workspace too small */
    OSPREY_ERR_CUDA = -5,        /* a CUDA runtime call failed */
    OSPREY_ERR_TIMEOUT = -6      /* a bounded device wait ran out (dev_status) */
};

enum { OSPREY_F32 = 0, OSPREY_BF16 = 1 };

/* Drafter shape.  d_model, head_dim and feat_dim multiples of 256, 64 and 256;
 * n_q_heads a multiple of n_kv_heads; ffn_dim a multiple of 256.
 * rms_eps: RMSNorm epsilon (1e-6).  rope_theta: rotary base (rotate-half
 * convention, angle pos * theta^(-2i/head_dim)). */
typedef struct osprey_config {
    int32_t d_model, n_layers, n_q_heads, n_kv_heads, head_dim, ffn_dim, vocab, feat_dim;
    int32_t page_size; /* KV page length in positions; must be 16 */
    float rms_eps, rope_theta;
} osprey_config;

/* Drafter weights, bf16, device, borrowed for the context's lifetime.
 *   W_c        [d][feat_dim]                 Eq. 1, no bias
 *   embed      [vocab][d]
 *   final_norm [d]
 *   lm_head    [vocab][d]
 * per layer l < n_layers:
 *   attn_norm  [d]
 *   W_qkv      [(Hq + 2 Hkv) head_dim][2 d]  Eq. 2: columns 0..d-1 read the
 *              context slot (c or the fed-back hidden state), d..2d-1 read
 *              RMSNorm(x); rows are Q heads, then K heads, then V heads
 *   W_o        [d][Hq head_dim]
 *   ffn_norm   [d]
 *   W_gate, W_up [ffn][d];  W_down [d][ffn]                                  */
typedef struct osprey_weights {
    const void *W_c, *embed, *final_norm, *lm_head;
    const void *attn_norm[OSPREY_MAX_LAYERS], *W_qkv[OSPREY_MAX_LAYERS], *W_o[OSPREY_MAX_LAYERS];
    const void *ffn_norm[OSPREY_MAX_LAYERS], *W_gate[OSPREY_MAX_LAYERS], *W_up[OSPREY_MAX_LAYERS];
    const void *W_down[OSPREY_MAX_LAYERS];
} osprey_weights;

/* Paged drafter KV cache (bf16, device, caller-owned).
 *   k_pages, v_pages [n_layers][n_pages][n_kv_heads][page_size][head_dim]
 *   page_table [B][max_pages_per_seq] int32: position t of sequence b lives in
 *              page page_table[b][t / page_size], slot t % page_size
 *   seq_len    [B] int32: committed positions of each sequence                */
typedef struct osprey_kv {
    void *k_pages, *v_pages;
    int32_t *page_table, *seq_len;
    int32_t max_pages_per_seq, n_pages;
} osprey_kv;

typedef struct osprey_ctx osprey_ctx;

/* Thread-local message for the last error returned on this thread ("" if none). */
const char *osprey_last_error(void);

/* Validate the shape and weight pointers and make a context (host memory only).
 * The context picks the kernels a draft call uses:
 *   rows <= 2 per chain step: TMA-streamed GEMVs (weights read once per step);
 *   3..80 rows: tcgen05 tensor-core GEMMs, float32 activations split into three
 *     bf16 planes (24 mantissa bits) so results match the GEMV path's (the LM
 *     head's operand into two planes, 16 bits: its logits differ from the
 *     GEMV path's by rounding of the operand's last bits);
 *   attention: clusters merged on chip while they fit one wave, else global
 *     partials.
 * Two environment variables, read here, select the alternatives for testing:
 * OSPREY_TC=0 (CUDA-core GEMVs for batched rows) and OSPREY_ATTN_CLUSTER=0
 * (global-partials attention).  Two more select fused batch-1 chain steps,
 * off by default: OSPREY_FUSED_MLP=1 (O-proj, gate/up and down of a layer as
 * one launch) and OSPREY_FUSED_LAYER=1 (the whole layer as one launch, for
 * shapes whose per-SM weight slices fit shared memory); both use one block per
 * SM and bounded grid barriers.
 * Errors: INVALID_ARG (null), SHAPE (unsupported dimension). */
int osprey_create(const osprey_config *cfg, const osprey_weights *w, osprey_ctx **out);
void osprey_destroy(osprey_ctx *ctx);

/* Bytes of workspace osprey_draft_step needs for a batch of B sequences, chains
 * of K tokens, up to max_new extend rows per sequence and page tables of
 * max_pages_per_seq pages.  0 on bad arguments. */
size_t osprey_draft_workspace_bytes(const osprey_ctx *ctx, int B, int K, int max_new,
                                    int max_pages_per_seq);

/* Write K/V rows into the paged cache after each sequence's committed length
 * and advance seq_len (the prefix fill of a draft session).
 *   n_rows [B] int32 (device): rows for sequence b, summing to total_rows
 *   k_rows, v_rows [n_layers][total_rows][n_kv_heads][head_dim] bf16 (keys
 *   already rotated), rows of sequence b after those of sequences < b.
 * Device errors: CAPACITY (rows past the page table or a page id outside
 * [0, n_pages)), INVALID_ARG (n_rows negative or not summing to total_rows);
 * such a sequence is left untouched. */
int osprey_kv_append(const osprey_ctx *ctx, const osprey_kv *kv, int B, const int32_t *n_rows,
                     int64_t total_rows, const void *k_rows, const void *v_rows,
                     int32_t *dev_status, void *stream);

/* One draft call: extend, then a K-token chain (Sec. 3.1, Eq. 1-3, Sec. 3.4).
 *   n_new  [B] int32 (device), 1 <= n_new[b] <= max_new: extend rows of b
 *   tokens [B][max_new] int32: extend row j is token tokens[b][j] at position
 *          seq_len[b] + j ...
 *   feats  [B][max_new][feat_dim] bf16: ... paired with the concatenated target
 *          hidden states of the previous position (Eq. 2 pairs x_t with c_{t-1})
 *   temperature: draft distribution q = softmax(logits / T); T == 0 is greedy
 *          (argmax, lowest id on ties)
 *   u_draft [B][K] float in [0,1): token k is the smallest id j with
 *          u * S < C_j (C the inclusive cumulative of exp(logits/T - M) over ids
 *          in ascending order, S its total)
 * Outputs (device):
 *   draft_tokens [B][K] int32
 *   draft_qx     [B][K] float, q(token) (1 for greedy); may be NULL
 *   draft_stats  [B][K][2] float, (M, log S) of logits/T (of logits when
 *                greedy); may be NULL
 *   draft_logits [B][K][vocab] float, raw logits; NULL to keep them on chip
 * Effects: the extend rows' K/V are committed and seq_len[b] += n_new[b]; the
 * chain rows' K/V are written speculatively after them (not committed; the
 * next call's extend rows overwrite them).  The pages must hold
 * seq_len[b] + n_new[b] + K - 1 positions (else dev_status = CAPACITY and the
 * sequence is skipped: tokens -1, seq_len unchanged).
 * Host errors: INVALID_ARG, SHAPE, CAPACITY (workspace_bytes too small). */
int osprey_draft_step(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int max_new,
                      const int32_t *n_new, const int32_t *tokens, const void *feats,
                      float temperature, const float *u_draft, int32_t *draft_tokens,
                      float *draft_qx, float *draft_stats, float *draft_logits,
                      void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream);

/* osprey_draft_step with draft_logits NULL that also keeps, for every draft
 * token, the state it was drafted from, for osprey_verify_hidden:
 *   draft_hidden [B][K][d_model] float (device, 16-byte aligned): row k of
 *          sequence b is the last layer's residual output before the final
 *          norm (Sec. 3.4's g) of the row whose LM head drew token k; zeros
 *          for a sequence the call skipped.
 * Everything else as osprey_draft_step (same workspace size). */
int osprey_draft_step_hidden(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int max_new,
                             const int32_t *n_new, const int32_t *tokens, const void *feats,
                             float temperature, const float *u_draft, int32_t *draft_tokens,
                             float *draft_qx, float *draft_stats, float *draft_hidden,
                             void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream);

/* Tree drafting (topk > 1; the paper serves chains, topk = 1, Sec. 4 inference
 * settings): osprey_draft_step whose LM head draws topk candidates per chain
 * step.  Candidate j of step k is the inverse CDF of q_k at u_draft[b][k][j]
 * (independent draws; at T = 0 the topk highest logits in descending order,
 * ties to the lowest id); candidate 0 continues the chain (Sec. 3.4), the
 * others are leaves of the branching chain that osprey_verify_tree checks.
 *   topk 1 .. 8; topk > 1 needs the tensor-core LM head (B <= 80 and a device
 *        with tcgen05, else SHAPE)
 *   u_draft [B][K][topk]; cand [B][K][topk] int32; cand_qx [B][K][topk] q of
 *   each candidate (1 for greedy; may be NULL); draft_stats [B][K][2] and
 *   draft_logits [B][K][V] as osprey_draft_step.  Workspace: as
 *   osprey_draft_step (osprey_draft_workspace_bytes). */
int osprey_draft_step_topk(osprey_ctx *ctx, const osprey_kv *kv, int B, int K, int topk, int max_new,
                           const int32_t *n_new, const int32_t *tokens, const void *feats, float temperature,
                           const float *u_draft, int32_t *cand, float *cand_qx, float *draft_stats,
                           float *draft_logits, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                           void *stream);

/* Verification of a draft tree (the multi-candidate form of the Sec. 3.1 rule;
 * topk = 1 gives osprey_verify's result).  The tree is a branching chain: at
 * depth i < K the topk candidates cand[b][i][*] were drawn from the drafter's
 * q_i = softmax(draft_logits[b][i] / T); candidate 0 continues the chain.
 *   target_logits [B][1 + K*topk][V]: row 0 is the target's distribution after
 *          the verified prefix, row 1 + i*topk + j the one after the path to
 *          candidate j of depth i
 *   draft_logits [B][K][V] (NULL iff T == 0), same dtype
 *   u_accept [B][K][topk], u_sample [B][K+1] float in [0,1)
 * The walk: at depth i, with p the current node's row and the residual r = p,
 * candidate j is accepted iff u_accept[i][j] < r(x) / q_i(x), and a rejection
 * sets r = norm(max(0, r - q_i)).  An accepted candidate 0 below depth K - 1
 * moves on to depth i + 1; an accepted leaf or depth K - 1 ends the walk with a
 * draw from that node's row at u_sample[i + 1]; topk rejections end it with a
 * draw from r at u_sample[i].  Greedy: the current node's argmax is accepted
 * when it is a candidate (the first such).  Draws are inverse CDFs over
 * ascending ids.
 * Outputs (device): out_tokens [B][K+1] (accepted candidates, the drawn
 *   token, then -1), n_accepted [B], branch [B] (the candidate index accepted
 *   at the last accepted depth, -1 if none), flags [B][K+1] (bit 3: a residual
 *   without float32 mass, p sampled instead; bit 4: the draw clamped to the
 *   last id with weight).
 * No workspace: one block per sequence keeps its walk on chip; rows off the
 * walked path are never read.  V <= 2^20.
 * Device errors: INVALID_ARG for a candidate outside [0, V) (that sequence gets
 * n_accepted 0 and out_tokens -1). */
int osprey_verify_tree(int B, int K, int topk, int V, int logits_dtype, const void *target_logits,
                       const void *draft_logits, const int32_t *cand, float temperature, const float *u_accept,
                       const float *u_sample, int32_t *out_tokens, int32_t *n_accepted, int32_t *branch,
                       uint8_t *flags, int32_t *dev_status, void *stream);

/* Bytes of workspace osprey_dflash_step needs.  0 on bad arguments. */
size_t osprey_dflash_workspace_bytes(const osprey_ctx *ctx, int B, int block, int max_pages_per_seq);

/* Block drafting with the EAGLE-style DFlash interface (Appendix, "EAGLE-Style
 * Target Interface for DFlash"): one drafter forward over a block of `block`
 * positions per sequence - the verified anchor token at position seq_len[b],
 * then the mask placeholder token at the next block - 1 positions - with causal
 * attention inside the block, and with the target feature gathered at the
 * anchor fed to every position through the expanded QKV projection (its
 * target-side columns are Eq. 2's context columns, zero at initialisation).
 * Labels are shifted by one: the output at block position j proposes the
 * token at j + 1, so positions 0..block-2 give block - 1 proposals, each drawn
 * from its own q_j = softmax(logits_j / T) by the inverse CDF at u_draft[b][j]
 * (argmax at T = 0).  The proposals are verified like a chain of block - 1
 * draft tokens (osprey_verify with K = block - 1).
 *   block  4 .. 81 (3 .. 80 proposals); sequences are processed in groups of
 *          floor(80 / (block - 1)), each group one tensor-core pass over the
 *          weights (SHAPE if the context has no tensor-core path)
 *   anchors [B] int32 (device), mask_token in [0, vocab)
 *   feats  [B][feat_dim] bf16: the concatenated target hidden states gathered
 *          at the anchor (c = W_c feats, Eq. 1, broadcast over the block)
 *   u_draft [B][block-1] float in [0,1) (may be NULL when T == 0)
 * Outputs (device): draft_tokens [B][block-1] int32, draft_qx [B][block-1],
 *   draft_stats [B][block-1][2] (as osprey_draft_step; qx and stats may be
 *   NULL), draft_logits [B][block-1][vocab] float (NULL to keep them in the
 *   workspace)
 * Effects: the anchor's K/V row is committed (seq_len[b] += 1); the mask rows'
 * K/V are written speculatively after it (the next call overwrites them).  The
 * pages must hold seq_len[b] + block - 1 positions (else dev_status = CAPACITY
 * and the sequence is skipped: tokens -1, seq_len unchanged).
 * Host errors: INVALID_ARG, SHAPE, CAPACITY (workspace_bytes too small). */
int osprey_dflash_step(osprey_ctx *ctx, const osprey_kv *kv, int B, int block, const int32_t *anchors,
                       int32_t mask_token, const void *feats, float temperature, const float *u_draft,
                       int32_t *draft_tokens, float *draft_qx, float *draft_stats, float *draft_logits,
                       void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream);

/* Bytes of workspace osprey_verify_hidden needs.  0 on bad arguments. */
size_t osprey_verify_hidden_workspace_bytes(const osprey_ctx *ctx, int B, int K);

/* Sampled verification (the rule of osprey_verify, temperature > 0) without
 * draft logits in memory.  The acceptance test at i reads the draft step's own
 * q_i(x_i) (draft_qx); the one draft row the rule needs in full, q_r at the
 * first rejected position r < K, is recomputed on the tensor cores from the
 * kept state (draft_hidden row r) through ctx's final RMSNorm and LM head, and
 * normalised with the draft step's (M, log S) of that row (draft_stats).  The
 * draft logits, B*K*V floats, are neither written by the draft step nor read
 * here; the LM head is read once per 80 sequences instead.
 *   ctx: the drafter whose draft step produced the inputs (V = its vocab)
 *   target_logits [B][K+1][V], logits_dtype OSPREY_F32 or OSPREY_BF16
 *   draft_hidden [B][K][d_model], draft_qx [B][K], draft_stats [B][K][2]
 *          float: as written by osprey_draft_step_hidden at the same T
 *   draft_tokens, u_accept, u_sample, out_tokens, n_accepted, flags, probs:
 *          as osprey_verify (probs' q column is draft_qx)
 *   workspace: osprey_verify_hidden_workspace_bytes(ctx, B, K) bytes
 * Host errors: INVALID_ARG (null pointer, T <= 0), SHAPE (the context has no
 * tensor-core path: OSPREY_TC=0 or a device without tcgen05), CAPACITY. */
int osprey_verify_hidden(osprey_ctx *ctx, int B, int K, int logits_dtype, const void *target_logits,
                         const float *draft_hidden, const float *draft_qx, const float *draft_stats,
                         const int32_t *draft_tokens, float temperature, const float *u_accept,
                         const float *u_sample, int32_t *out_tokens, int32_t *n_accepted, uint8_t *flags,
                         float *probs, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                         void *stream);

/* Bytes of workspace osprey_verify needs.  0 on bad arguments. */
size_t osprey_verify_workspace_bytes(int B, int K, int V);

/* Speculative-sampling verification of B chains of K draft tokens (Sec. 3.1).
 *   logits_dtype: OSPREY_F32 or OSPREY_BF16 for both logits arrays
 *   target_logits [B][K+1][V], draft_logits [B][K][V] (may be NULL iff T == 0)
 *   draft_tokens [B][K] int32 in [0, V)
 *   temperature: p_i = softmax(target_i / T), q_i = softmax(draft_i / T);
 *          T == 0 is greedy: accept while argmax p_i == token_i, then emit
 *          argmax p_r (raw logits, lowest id on ties)
 *   u_accept [B][K]: accept token i iff u_accept[i] < p_i(x_i) / q_i(x_i)
 *   u_sample [B][K+1]: the token emitted at the first rejected position r is
 *          drawn from norm(max(0, p_r - q_r)) (r < K) or from p_K (all
 *          accepted) by the same inverse CDF as osprey_draft_step, at
 *          u_sample[r]
 * Outputs (device):
 *   out_tokens [B][K+1] int32: accepted tokens, then the emitted one, then -1
 *   n_accepted [B] int32
 *   flags [B][K+1] uint8: bit 3 = the residual had no mass in float32 and p_r
 *          was sampled instead; bit 4 = the inverse-CDF point fell past the last
 *          cumulative sum after rounding and the last token with mass was taken
 *   probs [B][K][2] float: (p_i(x_i), q_i(x_i)); may be NULL (greedy: unused)
 * Device errors: INVALID_ARG for a draft token outside [0, V) (that sequence
 * gets n_accepted 0 and out_tokens -1). */
int osprey_verify(int B, int K, int V, int logits_dtype, const void *target_logits,
                  const void *draft_logits, const int32_t *draft_tokens, float temperature,
                  const float *u_accept, const float *u_sample, int32_t *out_tokens,
                  int32_t *n_accepted, uint8_t *flags, float *probs, void *workspace,
                  size_t workspace_bytes, int32_t *dev_status, void *stream);

/* Allocation-free variant of osprey_verify (the paper has no counterpart; this is
 * for callers that cannot allocate device memory).  Some callers must not call
 * cudaMalloc: an engine that has already reserved nearly all HBM for weights and
 * its KV cache (an extra allocation fails or fragments its pool), or code on a
 * latency-critical path where cudaMalloc/cudaFree may block or synchronise the
 * device.  This entry point takes the same arguments as osprey_verify minus the
 * workspace and uses instead a scratch array of OSPREY_VERIFY_STATIC_SCRATCH_BYTES
 * that the library keeps in device global memory (every GPU that loads the
 * library holds it until the process exits).
 *   - It allocates nothing: no cudaMalloc/cudaFree, no allocating library call.
 *   - The first call on a device may load the library's device code into the
 *     current context (the runtime does this lazily); make that first call
 *     before any stream capture.
 *   - Requests whose scratch would exceed the array (see
 *     osprey_verify_workspace_bytes) return OSPREY_ERR_CAPACITY with a message.
 *   - All calls share the one array: calls whose work can overlap on the GPU
 *     (different streams, or different host threads) race and must be
 *     serialised by the caller.  The counters that must start at zero are
 *     cleared on the call's stream before its kernels run.
 *   - The array's device address is looked up (cudaGetSymbolAddress, which
 *     allocates nothing) with the caller's device current on every call. */
#define OSPREY_VERIFY_STATIC_SCRATCH_BYTES (4u << 20)
int osprey_verify_static(int B, int K, int V, int logits_dtype, const void *target_logits,
                         const void *draft_logits, const int32_t *draft_tokens, float temperature,
                         const float *u_accept, const float *u_sample, int32_t *out_tokens,
                         int32_t *n_accepted, uint8_t *flags, float *probs, int32_t *dev_status,
                         void *stream);

/* ---- measurement hooks (not part of the method) ------------------------------
 * osprey_probe_enable: make n_slots pairs of timing events in the context (n = 0
 * releases them).  While enabled, osprey_draft_step records pair k around its
 * k-th launch of the selected kernel (k < n_slots), also under stream capture
 * (as external event nodes).  osprey_probe_select picks that kernel:
 * OSPREY_PROBE_LM_HEAD (the default; pair k = chain step k's LM head) or
 * OSPREY_PROBE_ATTENTION (pair step * n_layers + layer = that attention launch;
 * none where a fused layer kernel runs the attention).  osprey_probe_read
 * writes the elapsed milliseconds of the first n pairs after the caller has
 * synchronised.  osprey_launch_count: kernels the library has launched (or
 * captured) in this process. */
enum { OSPREY_PROBE_LM_HEAD = 0, OSPREY_PROBE_ATTENTION = 1 };
int osprey_probe_enable(osprey_ctx *ctx, int n_slots);
int osprey_probe_select(osprey_ctx *ctx, int kind);
int osprey_probe_read(osprey_ctx *ctx, float *ms, int n);
int64_t osprey_launch_count(void);

/* ---- self-test of the failure path (not part of the method) ------------------
 * Every device-side wait of the library (mbarrier phases of the TMA rings,
 * tensor-core commits, grid barriers) is bounded: when the limit runs out the
 * kernel writes OSPREY_ERR_TIMEOUT to the caller's status word and returns, so
 * the context stays usable.  This call launches one block that waits on a
 * barrier nothing completes, for about limit_cycles SM clocks (1 .. 2e9), and
 * then takes that path: dev_status (device int32, first error wins) reads
 * OSPREY_ERR_TIMEOUT once the stream reaches it.
 * Host errors: INVALID_ARG (limit out of range, null status). */
int osprey_selftest_wait_timeout(int64_t limit_cycles, int32_t *dev_status, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* OSPREY_H */
