// Launchers shared between the C-ABI translation unit and the kernel units.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>

#include <atomic>
#include <stdint.h>

#include "osprey.h"

namespace osp {

// Counts every kernel the library launches (or captures), for measurement.
void count_launch(int n = 1);

// Sets the message osprey_last_error() returns on this thread.
void set_last_error(const char *msg);

// Runs set() (a cudaFuncSetAttribute call) the first time it is reached with a
// device current, per flag array.  set() must be idempotent: host threads that
// race here may both run it, but no thread reads a flag torn by another.
constexpr int kMaxDevices = 256;
template <typename F>
cudaError_t once_per_device(std::atomic<int> (&done)[kMaxDevices], F set) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const bool tracked = dev >= 0 && dev < kMaxDevices;
    if (tracked && done[dev].load(std::memory_order_acquire)) return cudaSuccess;
    e = set();
    if (e == cudaSuccess && tracked) done[dev].store(1, std::memory_order_release);
    return e;
}

// Lets a kernel use all the opt-in shared memory left after its static part
// (the same value every time, so a repeated call is harmless).
template <typename F>
cudaError_t allow_smem(F *kernel) {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    cudaFuncAttributes fa{};
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, kernel);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
    return e;
}

// True when `grid` blocks of `threads` threads and `smem` bytes of dynamic
// shared memory can all be resident at once on `sms` SMs of the current
// device (what a grid-wide barrier needs).  Call after allow_smem(kernel).
template <typename F>
bool grid_fits_resident(F *kernel, int threads, size_t smem, int grid, int sms) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return per_sm >= 1 && (long long)per_sm * sms >= grid;
}

// ---------------------------------------------------------------- verify
struct Decision {
    int r;          // first rejected position (K = all accepted), -1 = invalid sequence
    float Mp, Sp;   // normalisers of target row r (logits / T)
    float Mq, Sq;   // of draft row r (r < K)
    int pad[3];
};

struct VerifyArgs {
    int B, K, V, dtype;
    float temperature;
    const void *target, *draft;
    const int32_t *tokens;
    const float *u_accept, *u_sample;
    int32_t *out_tokens, *n_accepted;
    uint8_t *flags;
    float *probs;
    int32_t *status;
    // workspace views
    void *part;     // [B][K+1][nch] 16-byte partials
    void *dec;      // [B] decisions
    void *csum;     // [B][nch] float2 chunk sums
    int *ticket1;   // [B]
    int *ticket2;   // [B]
    int nch;
    // streamed path (vstream.cu): per-tile partials, 4 KB row chunks
    void *tpart;    // [B][K+1][nch3] float4
    void *tsum;     // [B][nch3] float2
    int *trow;      // [B][K+1] per-row arrival counters
    void *rowstat;  // [B][K+1] float4 row summaries
    int nch3;
    size_t counter_bytes;   // ticket1, ticket2 and trow are one block from ticket1 on
    // logits-free form: q_i(x_i) [B][K] and (M, log S) [B][K][2] from the draft
    // step; the decision rows' draft logits of sequences b0.. are rows of zrec [.][V]
    const float *qx_in, *stats_in;
    const float *zrec;
    int b0;
};
cudaError_t launch_verify_stream(const VerifyArgs &a, int sms, cudaStream_t s);
bool verify_stream_ok(const VerifyArgs &a);
size_t verify_workspace_layout(int B, int K, int V, VerifyArgs *a, void *base);
cudaError_t launch_verify(const VerifyArgs &a, cudaStream_t s);
// logits-free form: target statistics and the decision for every sequence, then
// per group of n sequences from b0 (after zrec holds their decision rows) the draw
cudaError_t launch_verify_hidden_stats(const VerifyArgs &a, cudaStream_t s);
cudaError_t launch_verify_hidden_sample(const VerifyArgs &a, int b0, int n, cudaStream_t s);
// the kept state of each sequence's decision row r < K (zeros otherwise) as
// rows 0..n-1 of dst [n][d], for the sequences b0..b0+n-1
cudaError_t launch_decision_rows(const void *dec, const float *hidden, int K, int d, int b0, int n, float *dst,
                                 cudaStream_t s);

// ---------------------------------------------------------------- tree verify
struct VerifyTreeArgs {
    int B, K, k, V, dtype;
    float temperature;
    const void *target;   // [B][1 + K k][V]: the root, then node (i, j) at row 1 + i k + j
    const void *draft;    // [B][K][V] (null when greedy)
    const int32_t *cand;  // [B][K][k]
    const float *u_accept, *u_sample;   // [B][K][k], [B][K+1]
    int32_t *out_tokens, *n_accepted, *branch;
    uint8_t *flags;
    int32_t *status;
};
cudaError_t launch_verify_tree(const VerifyTreeArgs &a, cudaStream_t s);

// ---------------------------------------------------------------- kv append
struct KvAppendArgs {
    void *k_pages, *v_pages;
    const int32_t *page_table;
    int32_t *seq_len;
    const int32_t *n_rows;
    const void *k_rows, *v_rows;
    int64_t total_rows;
    int B, L, Hkv, hd, P, max_pages, n_pages;
    int32_t *status;
};
cudaError_t launch_kv_append(const KvAppendArgs &a, cudaStream_t s);

}  // namespace osp
