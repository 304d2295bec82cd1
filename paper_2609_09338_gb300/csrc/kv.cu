// Paged KV-cache append: scatter caller-provided K/V rows into the pages after
// each sequence's committed length, then advance the committed lengths.
#include "common.cuh"
#include "internal.h"

namespace osp {

constexpr int KV_THREADS = 256;
constexpr int KV_ROWS_PER_BLOCK = 8;
constexpr int KV_MAX_B = 4096;

// One block per KV_ROWS_PER_BLOCK flattened rows.  Every block rebuilds the
// per-sequence row offsets (B is small) and binary-searches its rows' owner.
__global__ void __launch_bounds__(KV_THREADS) kv_scatter(KvAppendArgs a) {
    __shared__ int64_t off[KV_MAX_B + 1];
    __shared__ int bad;
    if (threadIdx.x == 0) {
        int64_t acc = 0;
        int neg = 0;
        for (int b = 0; b < a.B; ++b) {
            off[b] = acc;
            int n = a.n_rows[b];
            neg |= n < 0;
            acc += n;
        }
        off[a.B] = acc;
        bad = neg || acc != a.total_rows;
    }
    __syncthreads();
    if (bad) return;   // reported by kv_advance
    const int64_t r0 = (int64_t)blockIdx.x * KV_ROWS_PER_BLOCK;
    const int chunks = a.Hkv * a.hd / 8;           // 16-byte pieces of one row of one layer
    const int per_row = 2 * a.L * chunks;
    for (int rr = 0; rr < KV_ROWS_PER_BLOCK; ++rr) {
        const int64_t r = r0 + rr;
        if (r >= a.total_rows) break;
        int lo = 0, hi = a.B - 1;                  // owner: last b with off[b] <= r
        while (lo < hi) {
            int mid = (lo + hi + 1) >> 1;
            if (off[mid] <= r) lo = mid; else hi = mid - 1;
        }
        const int b = lo;
        const int n = (int)(off[b + 1] - off[b]);
        const int L0 = a.seq_len[b];
        const int64_t pos = (int64_t)L0 + (r - off[b]);
        const bool seq_fits = L0 >= 0 && (int64_t)L0 + n <= (int64_t)a.max_pages * a.P;
        if (!seq_fits) continue;
        const int page = a.page_table[(size_t)b * a.max_pages + pos / a.P];
        if (page < 0 || page >= a.n_pages) continue;
        const int slot = (int)(pos % a.P);
        for (int c = threadIdx.x; c < per_row; c += blockDim.x) {
            const int kvsel = c / (a.L * chunks);
            const int rem = c % (a.L * chunks);
            const int l = rem / chunks, hc = rem % chunks;
            const int h = hc / (a.hd / 8), dpart = hc % (a.hd / 8);
            const uint16_t *src = (const uint16_t *)(kvsel ? a.v_rows : a.k_rows) +
                                  (((size_t)l * a.total_rows + r) * a.Hkv + h) * a.hd + dpart * 8;
            uint16_t *dst = (uint16_t *)(kvsel ? a.v_pages : a.k_pages) +
                            ((((size_t)l * a.n_pages + page) * a.Hkv + h) * a.P + slot) * a.hd +
                            dpart * 8;
            *(uint4 *)dst = ld_stream(src);
        }
    }
}

// One block: checks the row counts, then advances each sequence whose rows all
// fit (capacity and valid page ids); reports the first failure in *status.
__global__ void __launch_bounds__(1024) kv_advance(KvAppendArgs a) {
    __shared__ long long tot;
    __shared__ int neg;
    if (threadIdx.x == 0) { tot = 0; neg = 0; }
    __syncthreads();
    long long mine = 0;
    int mneg = 0;
    for (int b = threadIdx.x; b < a.B; b += blockDim.x) {
        int n = a.n_rows[b];
        mneg |= n < 0;
        mine += n;
    }
    atomicAdd((unsigned long long *)&tot, (unsigned long long)mine);
    if (mneg) atomicOr(&neg, 1);
    __syncthreads();
    if (neg || tot != a.total_rows) {
        if (threadIdx.x == 0) set_status(a.status, OSPREY_ERR_INVALID_ARG);
        return;
    }
    for (int b = threadIdx.x; b < a.B; b += blockDim.x) {
        const int n = a.n_rows[b], L0 = a.seq_len[b];
        bool ok = L0 >= 0 && (int64_t)L0 + n <= (int64_t)a.max_pages * a.P;
        if (ok && n > 0) {
            for (int pg = L0 / a.P; pg <= (L0 + n - 1) / a.P; ++pg) {
                int page = a.page_table[(size_t)b * a.max_pages + pg];
                if (page < 0 || page >= a.n_pages) { ok = false; break; }
            }
        }
        if (ok) a.seq_len[b] = L0 + n;
        else set_status(a.status, OSPREY_ERR_CAPACITY);
    }
}

cudaError_t launch_kv_append(const KvAppendArgs &a, cudaStream_t s) {
    if (a.total_rows > 0) {
        int64_t blocks = (a.total_rows + KV_ROWS_PER_BLOCK - 1) / KV_ROWS_PER_BLOCK;
        kv_scatter<<<(unsigned)blocks, KV_THREADS, 0, s>>>(a);
        count_launch();
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    kv_advance<<<1, 1024, 0, s>>>(a);
    count_launch();
    return cudaGetLastError();
}

}  // namespace osp
