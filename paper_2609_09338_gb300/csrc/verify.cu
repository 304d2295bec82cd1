// Speculative-sampling verification (Sec. 3.1: the unmodified rule of
// Leviathan et al.) as two streaming kernels.
//
// verify_stats: one block per (vocab chunk, row i, sequence b) reads the chunk
//   of target row i and, for i < K, of draft row i exactly once with 16-byte
//   coalesced loads, and publishes (max, sum exp) of logits/T for both (argmax
//   in greedy mode).  The last block of a sequence to finish (atomic ticket, no
//   waiting) combines the partials into the row normalisers, evaluates
//   p_i(x_i), q_i(x_i), runs the acceptance chain and fixes the decision row r.
// verify_sample (sampled mode only): one block per (vocab chunk, sequence)
//   re-reads only row r and sums the weights max(0, p_r - q_r) (or p_K for the
//   bonus) per chunk; the last block picks the chunk holding u * S and scans it
//   in id order for the token.
// Logits-free form (HIDDEN): no draft rows in memory.  verify_stats reads the
//   target rows only and the decision takes q_i(x_i) from the draft step;
//   verify_sample reads the decision row's draft logits from `zrec`, recomputed
//   for a group of sequences by the tensor-core LM head (api.cu).
#include <float.h>
#include <math.h>

#include <cstdio>
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace osp {

constexpr int VT = 256;                 // threads per block
constexpr int VCHUNK = 8192;            // logits of one row per block
constexpr int VPER = VCHUNK / VT;       // logits per thread

template <typename T> struct Vec;
template <> struct Vec<float> { static constexpr int W = 4; };
template <> struct Vec<uint16_t> { static constexpr int W = 8; };

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(uint16_t x) { return bf_to_f(x); }

// Element index of value j (0..VPER-1) of this thread inside its chunk: the
// thread's vectors are strided across the block so every load is coalesced.
template <typename T, bool VEC>
__device__ __forceinline__ int chunk_index(int j) {
    constexpr int W = VEC ? Vec<T>::W : 1;
    return ((j / W) * VT + threadIdx.x) * W + (j % W);
}

// Load this thread's VPER values of a chunk; positions past V read -inf.
template <typename T, bool VEC>
__device__ __forceinline__ void load_chunk(const T *row, int start, int V, float (&f)[VPER]) {
    if (VEC) {
        constexpr int W = Vec<T>::W;
        constexpr int NV = VPER / W;
        uint4 raw[NV];
#pragma unroll
        for (int it = 0; it < NV; ++it) {
            int e = start + (it * VT + threadIdx.x) * W;
            raw[it] = e < V ? ld_stream(row + e) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int it = 0; it < NV; ++it) {
            int e = start + (it * VT + threadIdx.x) * W;
            if (W == 4) {
                f[it * 4 + 0] = __uint_as_float(raw[it].x);
                f[it * 4 + 1] = __uint_as_float(raw[it].y);
                f[it * 4 + 2] = __uint_as_float(raw[it].z);
                f[it * 4 + 3] = __uint_as_float(raw[it].w);
            } else {
                float g[8];
                unpack8(raw[it], g);
#pragma unroll
                for (int j = 0; j < 8; ++j) f[it * 8 + j] = g[j];
            }
            if (e >= V) {
#pragma unroll
                for (int j = 0; j < W; ++j) f[it * W + j] = -INFINITY;
            }
        }
    } else {
#pragma unroll
        for (int j = 0; j < VPER; ++j) {
            int e = start + j * VT + threadIdx.x;
            f[j] = e < V ? to_f(row[e]) : -INFINITY;
        }
    }
}

template <typename T, bool VEC>
__device__ __forceinline__ int elem_index(int start, int j) {
    return VEC ? start + chunk_index<T, true>(j) : start + j * VT + threadIdx.x;
}

// Load this thread's VPER values of a float32 row in the element order that
// load_chunk<T, VEC> gives a row of T (so that value j of both loads is the
// same id): the logits-free draw pairs bf16 target rows with float32 draft rows.
template <typename T, bool VEC>
__device__ __forceinline__ void load_chunk_f32_as(const float *row, int start, int V, float (&f)[VPER]) {
    if (!VEC || Vec<T>::W == 4) {
        load_chunk<float, VEC>(row, start, V, f);
        return;
    }
    constexpr int NV = VPER / 8;   // T has 8 values per 16-byte vector: two float4 loads each
    uint4 lo[NV], hi[NV];
#pragma unroll
    for (int it = 0; it < NV; ++it) {
        const int e = start + (it * VT + threadIdx.x) * 8;
        lo[it] = e < V ? ld_stream(row + e) : make_uint4(0, 0, 0, 0);
        hi[it] = e < V ? ld_stream(row + e + 4) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int it = 0; it < NV; ++it) {
        const int e = start + (it * VT + threadIdx.x) * 8;
        const uint32_t w[8] = {lo[it].x, lo[it].y, lo[it].z, lo[it].w, hi[it].x, hi[it].y, hi[it].z, hi[it].w};
#pragma unroll
        for (int j = 0; j < 8; ++j) f[it * 8 + j] = e < V ? __uint_as_float(w[j]) : -INFINITY;
    }
}

__device__ __forceinline__ MS thread_ms(const float (&f)[VPER], float invT) {
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < VPER; ++j) m = fmaxf(m, f[j] * invT);
    if (m == -INFINITY) return {m, 0.f};
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < VPER; ++j) s += __expf(f[j] * invT - m);
    return {m, s};
}

__device__ __forceinline__ float ld_logit(const void *base, int dtype, size_t idx) {
    return dtype == OSPREY_F32 ? __ldg((const float *)base + idx)
                               : bf_to_f(__ldg((const uint16_t *)base + idx));
}

// The last block of sequence b: combine the partials of all K+1 rows, run the
// acceptance chain and write everything but the token emitted at r.
template <bool GREEDY, bool HIDDEN>
__device__ void decide(const VerifyArgs &a, int b) {
    __shared__ float sMp[16], sSp[16], sMq[16], sSq[16];
    __shared__ int sAm[16];
    const int K = a.K, V = a.V, nch = a.nch;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float4 *part = (const float4 *)a.part + (size_t)b * (K + 1) * nch;
    for (int i = w; i <= K; i += VT / 32) {
        if (GREEDY) {
            AM am{-INFINITY, 0x7fffffff};
            for (int c = lane; c < nch; c += 32) {
                float4 p = __ldcg(part + (size_t)i * nch + c);
                am = am_combine(am, AM{p.x, __float_as_int(p.y)});
            }
            am = warp_am(am);
            if (lane == 0) sAm[i] = am.i;
        } else {
            MS p{-INFINITY, 0.f}, q{-INFINITY, 0.f};
            for (int c = lane; c < nch; c += 32) {
                float4 v = __ldcg(part + (size_t)i * nch + c);
                p = ms_combine(p, MS{v.x, v.y});
                q = ms_combine(q, MS{v.z, v.w});
            }
            p = warp_ms(p);
            q = warp_ms(q);
            if (lane == 0) {
                sMp[i] = p.m; sSp[i] = p.s; sMq[i] = q.m; sSq[i] = q.s;
            }
        }
    }
    __syncthreads();
    if (w != 0) return;
    // warp 0: lane i evaluates position i; the chain is a ballot.  All loads
    // below are independent, so the decision costs one round of latency.
    const int32_t *x = a.tokens + (size_t)b * K;
    int32_t *out = a.out_tokens + (size_t)b * (K + 1);
    uint8_t *fl = a.flags + (size_t)b * (K + 1);
    Decision *dec = (Decision *)a.dec + b;
    const int xi = lane < K ? x[lane] : 0;
    const bool ok = __all_sync(0xffffffffu, lane >= K || (xi >= 0 && xi < V));
    if (lane <= K) fl[lane] = 0;
    if (!ok) {
        if (lane == 0) {
            set_status(a.status, OSPREY_ERR_INVALID_ARG);
            a.n_accepted[b] = 0;
            dec->r = -1;
        }
        if (lane <= K) out[lane] = -1;
        return;
    }
    bool accept = false;
    if (GREEDY) {
        accept = lane < K && sAm[lane] == xi;
    } else if (lane < K) {
        const float invT = 1.f / a.temperature;
        const size_t rowp = ((size_t)b * (K + 1) + lane) * V, rowq = ((size_t)b * K + lane) * V;
        const float px = expf(ld_logit(a.target, a.dtype, rowp + xi) * invT - sMp[lane]) / sSp[lane];
        const float qx = HIDDEN ? a.qx_in[(size_t)b * K + lane]
                                : expf(ld_logit(a.draft, a.dtype, rowq + xi) * invT - sMq[lane]) / sSq[lane];
        if (a.probs) {
            a.probs[((size_t)b * K + lane) * 2 + 0] = px;
            a.probs[((size_t)b * K + lane) * 2 + 1] = qx;
        }
        accept = a.u_accept[(size_t)b * K + lane] < px / qx;
    }
    const unsigned rej = ~__ballot_sync(0xffffffffu, accept) & ((1u << K) - 1u);
    const int r = rej ? __ffs(rej) - 1 : K;
    if (lane < r) out[lane] = xi;
    else if (lane == r) out[lane] = GREEDY ? sAm[r] : -1;   // sampled: written by verify_sample
    else if (lane <= K) out[lane] = -1;
    if (lane == 0) {
        a.n_accepted[b] = r;
        if (!GREEDY) {
            dec->r = r;
            dec->Mp = sMp[r]; dec->Sp = sSp[r];
            if (HIDDEN) {   // (M, log S) of the draft row, from the draft step
                dec->Mq = r < K ? a.stats_in[((size_t)b * K + r) * 2 + 0] : 0.f;
                dec->Sq = r < K ? expf(a.stats_in[((size_t)b * K + r) * 2 + 1]) : 1.f;
            } else {
                dec->Mq = r < K ? sMq[r] : 0.f;
                dec->Sq = r < K ? sSq[r] : 1.f;
            }
        }
    }
}

template <typename T, bool VEC, bool GREEDY, bool HIDDEN = false>
__global__ void __launch_bounds__(VT) verify_stats(VerifyArgs a) {
    __shared__ MS shm[VT / 32];
    __shared__ AM sha[VT / 32];
    // flattened grid: x = (b * (K+1) + i) * nch + c
    const int K = a.K, V = a.V;
    const int c = (int)(blockIdx.x % a.nch);
    const int i = (int)((blockIdx.x / a.nch) % (K + 1));
    const int b = (int)(blockIdx.x / ((unsigned)a.nch * (K + 1)));
    const int start = c * VCHUNK;
    const T *zp = (const T *)a.target + ((size_t)b * (K + 1) + i) * V;
    float4 *part = (float4 *)a.part + ((size_t)b * (K + 1) + i) * a.nch + c;
    if (GREEDY) {
        float f[VPER];
        load_chunk<T, VEC>(zp, start, V, f);
        AM am{-INFINITY, 0x7fffffff};
#pragma unroll
        for (int j = 0; j < VPER; ++j) am = am_combine(am, AM{f[j], elem_index<T, VEC>(start, j)});
        am = block_am(am, sha);
        if (threadIdx.x == 0) *part = make_float4(am.v, __int_as_float(am.i), 0.f, 0.f);
    } else {
        const float invT = 1.f / a.temperature;
        float f[VPER], g[VPER];
        load_chunk<T, VEC>(zp, start, V, f);
        const bool has_q = !HIDDEN && i < K;
        if (has_q) load_chunk<T, VEC>((const T *)a.draft + ((size_t)b * K + i) * V, start, V, g);
        MS p = block_ms(thread_ms(f, invT), shm);
        MS q{-INFINITY, 0.f};
        if (has_q) q = block_ms(thread_ms(g, invT), shm);
        if (threadIdx.x == 0) *part = make_float4(p.m, p.s, q.m, q.s);
    }
    if (arrive_last(a.ticket1 + b, a.nch * (K + 1))) decide<GREEDY, HIDDEN>(a, b);
}

// Weight of id e in the decision row's draw: max(0, p - q) (residual) or p.
__device__ __forceinline__ float sample_weight(float zp, float zq, const Decision &d, float invT,
                                               bool residual, bool use_p) {
    float p = __expf(zp * invT - d.Mp) * (1.f / d.Sp);
    if (use_p || !residual) return p;
    float q = __expf(zq * invT - d.Mq) * (1.f / d.Sq);
    return fmaxf(0.f, p - q);
}

// HIDDEN: blocks cover the group of sequences b0 .. b0 + n - 1 and the draft
// row r of sequence b is row b - b0 of zrec (float32 logits, TQ = float).
template <typename T, bool VEC, typename TQ = T, bool HIDDEN = false>
__global__ void __launch_bounds__(VT) verify_sample(VerifyArgs a) {
    __shared__ float sh[33];
    __shared__ float2 shs[VT / 32];
    __shared__ int s_chunk, s_tok, s_flag;
    __shared__ float s_t, s_before;
    const int K = a.K, V = a.V, nch = a.nch;
    const int c = (int)(blockIdx.x % nch), b = (HIDDEN ? a.b0 : 0) + (int)(blockIdx.x / nch);
    const Decision d = ((const Decision *)a.dec)[b];   // written by verify_stats
    const float invT = 1.f / a.temperature;
    // a decision outside [-1, K] means the workspace was not produced by
    // verify_stats (e.g. counters not zeroed): read nothing through it
    const bool valid = d.r >= 0 && d.r <= K;
    if (!valid && d.r != -1 && threadIdx.x == 0) set_status(a.status, OSPREY_ERR_INVALID_ARG);
    const int r = valid ? d.r : 0;
    const bool residual = r < K;
    const T *zp = (const T *)a.target + ((size_t)b * (K + 1) + r) * V;
    const TQ *zq = HIDDEN ? (residual ? (const TQ *)a.zrec + (size_t)(b - a.b0) * V : nullptr)
                          : (residual ? (const TQ *)a.draft + ((size_t)b * K + r) * V : (const TQ *)zp);
    const int start = c * VCHUNK;
    float2 *csum = (float2 *)a.csum + (size_t)b * nch;
    if (valid) {
        float f[VPER], g[VPER];
        load_chunk<T, VEC>(zp, start, V, f);
        if (residual) {
            if constexpr (std::is_same<T, TQ>::value) load_chunk<TQ, VEC>(zq, start, V, g);
            else load_chunk_f32_as<T, VEC>(zq, start, V, g);
        }
        float sw = 0.f, sp = 0.f;
#pragma unroll
        for (int j = 0; j < VPER; ++j) {
            if (f[j] == -INFINITY) continue;
            sw += sample_weight(f[j], residual ? g[j] : 0.f, d, invT, residual, false);
            sp += sample_weight(f[j], 0.f, d, invT, false, true);
        }
        sw = warp_sum(sw);
        sp = warp_sum(sp);
        if ((threadIdx.x & 31) == 0) shs[threadIdx.x >> 5] = make_float2(sw, sp);
        __syncthreads();
        if (threadIdx.x == 0) {
            float2 t = make_float2(0.f, 0.f);
            for (int w = 0; w < VT / 32; ++w) { t.x += shs[w].x; t.y += shs[w].y; }
            csum[c] = t;
        }
    }
    if (!arrive_last(a.ticket2 + b, nch) || !valid) return;

    // ---- last block: choose the chunk, then the id inside it (ascending ids)
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        float tot_w = 0.f;
        for (int base = 0; base < nch; base += 32) {
            float v = base + lane < nch ? __ldcg(&csum[base + lane].x) : 0.f;
            tot_w += warp_sum(v);
        }
        const bool fallback = !(tot_w > 0.f) || !isfinite(tot_w);
        float S = 0.f;
        for (int base = 0; base < nch; base += 32) {
            float v = base + lane < nch ? (fallback ? __ldcg(&csum[base + lane].y)
                                                    : __ldcg(&csum[base + lane].x)) : 0.f;
            S += warp_sum(v);
        }
        const float t = a.u_sample[(size_t)b * (K + 1) + r] * S;
        float run = 0.f;
        int chunk = -1, last_pos = 0;
        float before = 0.f;
        for (int base = 0; base < nch && chunk < 0; base += 32) {
            float v = base + lane < nch ? (fallback ? __ldcg(&csum[base + lane].y)
                                                    : __ldcg(&csum[base + lane].x)) : 0.f;
            float inc = warp_incl_scan(v) + run;
            unsigned hit = __ballot_sync(0xffffffffu, base + lane < nch && t < inc);
            unsigned pos = __ballot_sync(0xffffffffu, base + lane < nch && v > 0.f);
            if (pos) last_pos = base + 31 - __clz(pos);
            if (hit) {
                int l = __ffs(hit) - 1;
                chunk = base + l;
                before = __shfl_sync(0xffffffffu, inc - v, l);
            }
            run = __shfl_sync(0xffffffffu, inc, 31);
        }
        if (lane == 0) {
            s_flag = fallback ? 8 : 0;
            if (chunk < 0) {   // u*S past the last cumulative sum after rounding
                chunk = last_pos;
                s_flag |= 16;
                before = 0.f;
                for (int k2 = 0; k2 < chunk; ++k2)
                    before += fallback ? __ldcg(&csum[k2].y) : __ldcg(&csum[k2].x);
            }
            s_chunk = chunk;
            s_t = t;
            s_before = before;
            s_tok = 0x7fffffff;
        }
    }
    __syncthreads();
    const bool fallback = s_flag & 8;
    // each thread scans a contiguous run of ids inside the chosen chunk
    const int cs = s_chunk * VCHUNK;
    const int e0 = cs + threadIdx.x * VPER;
    float wv[VPER];
    float mine = 0.f;
#pragma unroll
    for (int j = 0; j < VPER; ++j) {
        int e = e0 + j;
        float w = 0.f;
        if (e < V) {
            float zpv = to_f(zp[e]);
            float zqv = residual ? to_f(zq[e]) : 0.f;
            w = sample_weight(zpv, zqv, d, invT, residual, fallback);
        }
        wv[j] = w;
        mine += w;
    }
    float total;
    float ex = block_excl_scan(mine, sh, &total);
    float run = s_before + ex;
    int found = 0x7fffffff, lastpos = -1;
#pragma unroll
    for (int j = 0; j < VPER; ++j) {
        run += wv[j];
        if (found == 0x7fffffff && wv[j] > 0.f && s_t < run) found = e0 + j;
        if (wv[j] > 0.f) lastpos = e0 + j;
    }
    atomicMin(&s_tok, found);
    __syncthreads();
    if (s_tok == 0x7fffffff) {   // rounding left u*S past this chunk: last id with weight
        __shared__ int s_last;
        if (threadIdx.x == 0) s_last = -1;
        __syncthreads();
        atomicMax(&s_last, lastpos);
        __syncthreads();
        if (threadIdx.x == 0) {
            s_tok = s_last >= 0 ? s_last : cs;
            s_flag |= 16;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        a.out_tokens[(size_t)b * (K + 1) + r] = s_tok;
        a.flags[(size_t)b * (K + 1) + r] = (uint8_t)s_flag;
    }
}

size_t verify_workspace_layout(int B, int K, int V, VerifyArgs *a, void *base) {
    const int nch = (V + VCHUNK - 1) / VCHUNK;
    const int nch3 = (V + 1023) / 1024;   // 4 KB chunks of float32 rows (bf16 rows use half)
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    size_t off = 0;
    // arrival counters first, in one block (they must start at zero)
    const size_t o_t1 = 0, o_t2 = sizeof(int) * (size_t)B, o_tr = 2 * sizeof(int) * (size_t)B;
    const size_t ctr = o_tr + sizeof(int) * (size_t)B * (K + 1);
    off = al(ctr);
    size_t o_rs = off; off = al(off + (size_t)16 * B * (K + 1));
    size_t o_part = off; off = al(off + (size_t)16 * B * (K + 1) * nch);
    size_t o_dec = off; off = al(off + sizeof(Decision) * B);
    size_t o_cs = off; off = al(off + (size_t)8 * B * nch);
    size_t o_tp = off; off = al(off + (size_t)16 * B * (K + 1) * nch3);
    size_t o_ts = off; off = al(off + (size_t)8 * B * nch3);
    if (a && base) {
        char *p = (char *)base;
        a->ticket1 = (int *)(p + o_t1);
        a->ticket2 = (int *)(p + o_t2);
        a->part = p + o_part;
        a->dec = p + o_dec;
        a->csum = p + o_cs;
        a->nch = nch;
        a->tpart = p + o_tp;
        a->tsum = p + o_ts;
        a->trow = (int *)(p + o_tr);
        a->rowstat = p + o_rs;
        a->nch3 = nch3;
        a->counter_bytes = ctr;
    }
    return off;
}

template <typename T, bool VEC>
static cudaError_t launch_t(const VerifyArgs &a, cudaStream_t s) {
    const unsigned g1 = (unsigned)a.nch * (a.K + 1) * a.B;
    if (a.temperature == 0.f) {
        verify_stats<T, VEC, true><<<g1, VT, 0, s>>>(a);
        count_launch();
        return cudaGetLastError();
    }
    verify_stats<T, VEC, false><<<g1, VT, 0, s>>>(a);
    count_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    verify_sample<T, VEC><<<(unsigned)a.nch * a.B, VT, 0, s>>>(a);
    count_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------- logits-free form
static bool hidden_vec(const VerifyArgs &a) {
    // both element types vectorised: 8 bf16 or 2 x 4 float per 16 bytes
    return a.V % 8 == 0 && ((uintptr_t)a.target % 16) == 0 && ((uintptr_t)a.zrec % 16) == 0;
}

cudaError_t launch_verify_hidden_stats(const VerifyArgs &a, cudaStream_t s) {
    const unsigned g1 = (unsigned)a.nch * (a.K + 1) * a.B;
    const bool vec = hidden_vec(a);
    if (a.dtype == OSPREY_F32) {
        if (vec) verify_stats<float, true, false, true><<<g1, VT, 0, s>>>(a);
        else verify_stats<float, false, false, true><<<g1, VT, 0, s>>>(a);
    } else {
        if (vec) verify_stats<uint16_t, true, false, true><<<g1, VT, 0, s>>>(a);
        else verify_stats<uint16_t, false, false, true><<<g1, VT, 0, s>>>(a);
    }
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_verify_hidden_sample(const VerifyArgs &a_in, int b0, int n, cudaStream_t s) {
    VerifyArgs a = a_in;
    a.b0 = b0;
    const unsigned g2 = (unsigned)a.nch * n;
    const bool vec = hidden_vec(a);
    if (a.dtype == OSPREY_F32) {
        if (vec) verify_sample<float, true, float, true><<<g2, VT, 0, s>>>(a);
        else verify_sample<float, false, float, true><<<g2, VT, 0, s>>>(a);
    } else {
        if (vec) verify_sample<uint16_t, true, float, true><<<g2, VT, 0, s>>>(a);
        else verify_sample<uint16_t, false, float, true><<<g2, VT, 0, s>>>(a);
    }
    count_launch();
    return cudaGetLastError();
}

__global__ void __launch_bounds__(256) decision_rows_kernel(const Decision *dec, const float *hidden, int K, int d,
                                                            int b0, float *dst) {
    const int j = blockIdx.x, b = b0 + j;
    const int r = dec[b].r;   // written by verify_stats
    const bool act = r >= 0 && r < K;
    const float *src = hidden + ((size_t)b * K + (act ? r : 0)) * d;
    float *out = dst + (size_t)j * d;
    for (int k = threadIdx.x; k < d; k += blockDim.x) out[k] = act ? src[k] : 0.f;
}

cudaError_t launch_decision_rows(const void *dec, const float *hidden, int K, int d, int b0, int n, float *dst,
                                 cudaStream_t s) {
    decision_rows_kernel<<<n, 256, 0, s>>>((const Decision *)dec, hidden, K, d, b0, dst);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_verify(const VerifyArgs &a, cudaStream_t s) {
    if (verify_stream_ok(a)) {
        int dev = 0, sms = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        return launch_verify_stream(a, sms, s);
    }
    const bool f32 = a.dtype == OSPREY_F32;
    const int W = f32 ? 4 : 8;
    bool vec = (a.V % W) == 0 && ((uintptr_t)a.target % 16) == 0 &&
               (a.draft == nullptr || ((uintptr_t)a.draft % 16) == 0);
    if (f32) return vec ? launch_t<float, true>(a, s) : launch_t<float, false>(a, s);
    return vec ? launch_t<uint16_t, true>(a, s) : launch_t<uint16_t, false>(a, s);
}

}  // namespace osp

// ---------------------------------------------------------------------------
// Allocation-free verify: the scratch lives in this file-scope device array
// instead of a caller workspace.  Host code may not use the array's name as a
// device address (on the host it names a stand-in), so its device address is
// looked up with cudaGetSymbolAddress, with the caller's device current, on
// every call: the address belongs to the current context (a context torn down
// and made again loads the module again), and the lookup allocates nothing.
namespace osp {

static __device__ __align__(256) unsigned char g_verify_scratch[OSPREY_VERIFY_STATIC_SCRATCH_BYTES];

}  // namespace osp

extern "C" int osprey_verify_static(int B, int K, int V, int logits_dtype, const void *target_logits,
                                    const void *draft_logits, const int32_t *draft_tokens, float temperature,
                                    const float *u_accept, const float *u_sample, int32_t *out_tokens,
                                    int32_t *n_accepted, uint8_t *flags, float *probs, int32_t *dev_status,
                                    void *stream) {
    using namespace osp;
    if (B == 0) return OSPREY_OK;
    const size_t need = osprey_verify_workspace_bytes(B, K, V);
    if (need == 0)   // bad B, K or V: let the regular entry point report it
        return osprey_verify(B, K, V, logits_dtype, target_logits, draft_logits, draft_tokens, temperature,
                             u_accept, u_sample, out_tokens, n_accepted, flags, probs, nullptr, 0, dev_status,
                             stream);
    if (need > OSPREY_VERIFY_STATIC_SCRATCH_BYTES) {
        char msg[256];
        snprintf(msg, sizeof msg,
                 "osprey_verify_static: B=%d, K=%d, V=%d needs %zu bytes of scratch; the static scratch holds %u",
                 B, K, V, need, (unsigned)OSPREY_VERIFY_STATIC_SCRATCH_BYTES);
        set_last_error(msg);
        return OSPREY_ERR_CAPACITY;
    }
    void *base = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&base, g_verify_scratch);
    if (e != cudaSuccess || !base) {
        cudaGetLastError();
        set_last_error("osprey_verify_static: cudaGetSymbolAddress of the scratch array failed");
        return OSPREY_ERR_CUDA;
    }
    // osprey_verify clears the arrival counters on the stream before its
    // kernels; everything else is written before it is read
    return osprey_verify(B, K, V, logits_dtype, target_logits, draft_logits, draft_tokens, temperature, u_accept,
                         u_sample, out_tokens, n_accepted, flags, probs, base, OSPREY_VERIFY_STATIC_SCRATCH_BYTES,
                         dev_status, stream);
}
