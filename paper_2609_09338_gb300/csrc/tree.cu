// Verification of a draft tree (topk > 1): the multi-candidate form of the
// Sec. 3.1 rule over a branching chain.  At depth i the k candidates x_{i,j}
// (independent draws from the drafter's q_i; candidate 0 continues the chain)
// are tried in order against the residual r of the current node's target
// distribution p: x is accepted iff u_accept < r(x) / q_i(x), and a rejection
// replaces r by norm(max(0, r - q_i)).  Written as r = max(0, p - c q_i) / W,
// a rejection is c <- c + W, W <- sum_x max(0, p(x) - c q_i(x)) (one pass over
// the two rows), starting from c = 0, W = 1 (r = p).  An accepted chain
// candidate moves the walk one depth down; an accepted leaf, or the last
// depth, ends it with a draw from the accepted node's target row; k rejections
// end it with a draw from the last residual.  Greedy: the node's argmax is
// accepted if it is a candidate (the first such).
//
// One block (512 threads) per sequence walks its tree.  A node's row statistics
// are computed when the walk reaches it (rows off the path are never read); every pass
// streams one or two rows with 16-byte loads, 256 ids per warp-iteration
// ("chunk"), several chunks per warp in flight.  A draw keeps its chunk sums
// in shared memory, picks the chunk by a block scan and the id by a warp scan.
#include <math.h>

#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

namespace osp {

constexpr int TR_THREADS = 512;
constexpr int TR_WARPS = TR_THREADS / 32;
constexpr int TR_CH = 256;       // ids per chunk: 32 lanes x 8
constexpr int TR_U = 4;          // chunks a warp loads before using them
constexpr float TR_LOG2E = 1.4426950408889634f;

__device__ __forceinline__ float tr_ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <typename T> __device__ __forceinline__ float tr_f(T v);
template <> __device__ __forceinline__ float tr_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float tr_f<uint16_t>(uint16_t v) { return bf_to_f(v); }

// The lane's 8 logits of chunk c (ids c*256 + 8*lane ..), -inf past V.
template <typename T, bool VEC>
__device__ __forceinline__ void tr_load8(const T *row, int c, int V, float (&f)[8]) {
    const int e0 = c * TR_CH + (threadIdx.x & 31) * 8;
    if (VEC) {   // V % 8 == 0 and 16-byte rows: a vector is wholly in or out
        if (e0 < V) {
            if (sizeof(T) == 4) {
                const uint4 a = ld_stream(row + e0), b = ld_stream(row + e0 + 4);
                f[0] = __uint_as_float(a.x); f[1] = __uint_as_float(a.y);
                f[2] = __uint_as_float(a.z); f[3] = __uint_as_float(a.w);
                f[4] = __uint_as_float(b.x); f[5] = __uint_as_float(b.y);
                f[6] = __uint_as_float(b.z); f[7] = __uint_as_float(b.w);
            } else {
                unpack8(ld_stream(row + e0), f);
            }
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) f[e] = -INFINITY;
        }
    } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) f[e] = e0 + e < V ? tr_f<T>(row[e0 + e]) : -INFINITY;
    }
}

template <typename T>
__device__ __forceinline__ float tr_at(const T *row, int x) { return tr_f<T>(row[x]); }

struct TrNorm {   // p(x) = 2^(z c2 - mp) / Sp (and q alike), c2 = log2(e) / T
    float c2, mp, isp, mq, isq;
};

// (max, sum exp) of y = z / T over row p (and row q when q != null).
template <typename T, bool VEC>
__device__ void tr_stats(const T *zp, const T *zq, int V, float invT, MS *shm, MS &P, MS &Q) {
    const int warp = threadIdx.x >> 5, nch = (V + TR_CH - 1) / TR_CH;
    float mp = -INFINITY, sp = 0.f, mq = -INFINITY, sq = 0.f;
    for (int c0 = warp; c0 < nch; c0 += TR_WARPS * TR_U) {
        float f[TR_U][8], g[TR_U][8];
#pragma unroll
        for (int u = 0; u < TR_U; ++u) {
            const int c = c0 + u * TR_WARPS;
            tr_load8<T, VEC>(zp, c < nch ? c : nch, V, f[u]);
            if (zq) tr_load8<T, VEC>(zq, c < nch ? c : nch, V, g[u]);
        }
#pragma unroll
        for (int u = 0; u < TR_U; ++u) {
            float lm = -INFINITY;
#pragma unroll
            for (int e = 0; e < 8; ++e) lm = fmaxf(lm, f[u][e] * invT);
            if (lm > mp) {
                sp = mp == -INFINITY ? 0.f : sp * tr_ex2((mp - lm) * TR_LOG2E);
                mp = lm;
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) sp += f[u][e] == -INFINITY ? 0.f : tr_ex2((f[u][e] * invT - mp) * TR_LOG2E);
            if (zq) {
                float lq = -INFINITY;
#pragma unroll
                for (int e = 0; e < 8; ++e) lq = fmaxf(lq, g[u][e] * invT);
                if (lq > mq) {
                    sq = mq == -INFINITY ? 0.f : sq * tr_ex2((mq - lq) * TR_LOG2E);
                    mq = lq;
                }
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    sq += g[u][e] == -INFINITY ? 0.f : tr_ex2((g[u][e] * invT - mq) * TR_LOG2E);
            }
        }
    }
    P = block_ms(MS{mp, sp}, shm);
    Q = zq ? block_ms(MS{mq, sq}, shm) : MS{-INFINITY, 0.f};
}

// argmax (lowest id on ties) of a row
template <typename T, bool VEC>
__device__ int tr_argmax(const T *z, int V, AM *sha) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nch = (V + TR_CH - 1) / TR_CH;
    AM am{-INFINITY, 0x7fffffff};
    for (int c0 = warp; c0 < nch; c0 += TR_WARPS * TR_U) {
        float f[TR_U][8];
#pragma unroll
        for (int u = 0; u < TR_U; ++u) tr_load8<T, VEC>(z, min(c0 + u * TR_WARPS, nch), V, f[u]);
#pragma unroll
        for (int u = 0; u < TR_U; ++u) {
            const int base = (c0 + u * TR_WARPS) * TR_CH + lane * 8;
#pragma unroll
            for (int e = 0; e < 8; ++e)
                if (f[u][e] > am.v) am = AM{f[u][e], base + e};
        }
    }
    return block_am(am, sha).i;
}

// Weight of one id in a draw: the residual max(0, p - c q) (c > 0) or p.
__device__ __forceinline__ float tr_weight(float zp, float zq, const TrNorm &n, float c) {
    const float p = zp == -INFINITY ? 0.f : tr_ex2(zp * n.c2 - n.mp) * n.isp;
    if (c == 0.f) return p;
    const float q = zq == -INFINITY ? 0.f : tr_ex2(zq * n.c2 - n.mq) * n.isq;
    return fmaxf(0.f, p - c * q);
}

// sum over the ids of tr_weight; with csum, each chunk's sum is kept there
template <typename T, bool VEC>
__device__ float tr_mass(const T *zp, const T *zq, int V, const TrNorm &n, float c, float *csum, float *shf) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nch = (V + TR_CH - 1) / TR_CH;
    float acc = 0.f;
    for (int c0 = warp; c0 < nch; c0 += TR_WARPS * TR_U) {
        float f[TR_U][8], g[TR_U][8];
#pragma unroll
        for (int u = 0; u < TR_U; ++u) {
            const int ch = min(c0 + u * TR_WARPS, nch);
            tr_load8<T, VEC>(zp, ch, V, f[u]);
            if (c != 0.f) tr_load8<T, VEC>(zq, ch, V, g[u]);
        }
#pragma unroll
        for (int u = 0; u < TR_U; ++u) {
            float s = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) s += tr_weight(f[u][e], c != 0.f ? g[u][e] : -INFINITY, n, c);
            if (csum) {
                s = warp_sum(s);
                if (lane == 0 && c0 + u * TR_WARPS < nch) csum[c0 + u * TR_WARPS] = s;
            }
            acc += s;
        }
    }
    // with csum every lane holds its warp's chunk sums: count them once
    if (csum) acc = lane == 0 ? acc : 0.f;
    float tot = 0.f;
    {
        const float w = warp_sum(acc);
        if (lane == 0) shf[warp] = w;
        __syncthreads();
        if (threadIdx.x < 32) {
            float v = threadIdx.x < TR_WARPS ? shf[threadIdx.x] : 0.f;
            v = warp_sum(v);
            if (threadIdx.x == 0) shf[32] = v;
        }
        __syncthreads();
        tot = shf[32];
        __syncthreads();
    }
    return tot;
}

// Inverse CDF over ascending ids of tr_weight at u (a mass pass with chunk
// sums first).  flag |= 16 when rounding leaves u*S past the last sum (the
// last id with weight is taken).
template <typename T, bool VEC>
__device__ int tr_draw(const T *zp, const T *zq, int V, const TrNorm &n, float c, float u, float *csum, float *shf,
                       int *shi, int &flag) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nch = (V + TR_CH - 1) / TR_CH;
    const float S = tr_mass<T, VEC>(zp, zq, V, n, c, csum, shf);
    const float target = u * S;
    // chunks per thread, in order
    const int per = (nch + TR_THREADS - 1) / TR_THREADS;
    const int k0 = min(nch, threadIdx.x * per), k1 = min(nch, k0 + per);
    float mine = 0.f;
    for (int k = k0; k < k1; ++k) mine += csum[k];
    float tot;
    const float ex = block_excl_scan(mine, shf, &tot);
    if (threadIdx.x == 0) { shi[0] = 0x7fffffff; shi[1] = -1; }
    __syncthreads();
    if (mine > 0.f && target < ex + mine) atomicMin(&shi[0], (int)threadIdx.x);
    if (mine > 0.f) atomicMax(&shi[1], (int)threadIdx.x);
    __syncthreads();
    const int ct = shi[0] != 0x7fffffff ? shi[0] : (shi[1] >= 0 ? shi[1] : 0);
    const bool past = shi[0] == 0x7fffffff;
    __syncthreads();
    if ((int)threadIdx.x == ct) {
        float cum = ex;
        int ch = -1, lastc = k0;
        float lastb = ex;
        for (int k = k0; k < k1; ++k) {
            if (csum[k] > 0.f) { lastc = k; lastb = cum; }
            if (csum[k] > 0.f && target < cum + csum[k]) { ch = k; break; }
            cum += csum[k];
        }
        shi[2] = ch >= 0 ? ch : lastc;
        shf[33] = ch >= 0 ? cum : lastb;
        shi[3] = ch < 0 || past;
    }
    __syncthreads();
    if (warp == 0) {
        const int ch = shi[2];
        float f[8], g[8];
        tr_load8<T, VEC>(zp, ch, V, f);
        if (c != 0.f) tr_load8<T, VEC>(zq, ch, V, g);
        float w[8], s = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            w[e] = tr_weight(f[e], c != 0.f ? g[e] : -INFINITY, n, c);
            s += w[e];
        }
        const float incl = warp_incl_scan(s);
        const float before = shf[33] + incl - s;
        int found = -1, lastp = -1;
        float run = before;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            run += w[e];
            if (w[e] > 0.f) lastp = e;
            if (found < 0 && w[e] > 0.f && target < run) found = e;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, found >= 0);
        const unsigned pos = __ballot_sync(0xffffffffu, lastp >= 0);
        const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
        if (lane == l) {
            const int e = found >= 0 ? found : (lastp >= 0 ? lastp : 0);
            shi[4] = ch * TR_CH + l * 8 + e;
            if (!hit || shi[3]) shi[5] = 16;
            else shi[5] = 0;
        }
    }
    __syncthreads();
    flag |= shi[5];
    const int tok = shi[4];
    __syncthreads();
    return tok;
}

template <typename T, bool VEC, bool GREEDY>
__global__ void __launch_bounds__(TR_THREADS) tree_verify_kernel(const VerifyTreeArgs a) {
    extern __shared__ float csum[];   // [chunks of a row]
    __shared__ MS shm[32];
    __shared__ AM sha[32];
    __shared__ float shf[34];
    __shared__ int shi[8];
    __shared__ int s_acc;
    const int b = blockIdx.x, K = a.K, k = a.k, V = a.V;
    const size_t nrow = (size_t)(1 + K * k);
    const T *tp = (const T *)a.target + (size_t)b * nrow * V;
    const T *dq = GREEDY ? nullptr : (const T *)a.draft + (size_t)b * K * V;
    const int32_t *cand = a.cand + (size_t)b * K * k;
    int32_t *out = a.out_tokens + (size_t)b * (K + 1);
    uint8_t *fl = a.flags + (size_t)b * (K + 1);
    pdl_trigger();
    pdl_wait();
    // candidate ids outside [0, V): the sequence is reported and skipped
    bool ok = true;
    for (int i = threadIdx.x; i < K * k; i += TR_THREADS) ok &= cand[i] >= 0 && cand[i] < V;
    ok = __syncthreads_and(ok);
    if (threadIdx.x <= K) {
        out[threadIdx.x] = -1;
        fl[threadIdx.x] = 0;
    }
    if (!ok) {
        if (threadIdx.x == 0) {
            set_status(a.status, OSPREY_ERR_INVALID_ARG);
            a.n_accepted[b] = 0;
            a.branch[b] = -1;
        }
        return;
    }
    const float invT = GREEDY ? 1.f : 1.f / a.temperature;
    int row = 0, nacc = 0, br = -1;
    for (int i = 0; i < K; ++i) {
        const T *zp = tp + (size_t)row * V;
        if (GREEDY) {
            const int y = tr_argmax<T, VEC>(zp, V, sha);
            int j = -1;
            for (int jj = 0; jj < k && j < 0; ++jj)
                if (cand[i * k + jj] == y) j = jj;
            if (threadIdx.x == 0) out[i] = y;
            if (j < 0) break;
            ++nacc;
            br = j;
            row = 1 + i * k + j;
            if (j > 0 || i == K - 1) {
                const int z = tr_argmax<T, VEC>(tp + (size_t)row * V, V, sha);
                if (threadIdx.x == 0) out[i + 1] = z;
                break;
            }
            continue;
        }
        const T *zq = dq + (size_t)i * V;
        MS P, Q;
        tr_stats<T, VEC>(zp, zq, V, invT, shm, P, Q);
        TrNorm n{invT * TR_LOG2E, P.m * TR_LOG2E, 1.f / P.s, Q.m * TR_LOG2E, 1.f / Q.s};
        float c = 0.f, W = 1.f;
        int flag = 0;
        if (threadIdx.x == 0) s_acc = -1;
        __syncthreads();
        for (int j = 0; j < k; ++j) {
            const int x = cand[i * k + j];
            const float px = tr_ex2(tr_at<T>(zp, x) * n.c2 - n.mp) * n.isp;
            const float qx = tr_ex2(tr_at<T>(zq, x) * n.c2 - n.mq) * n.isq;
            const float r = fmaxf(0.f, px - c * qx) / W;
            const float u = a.u_accept[((size_t)b * K + i) * k + j];
            if (u < r / qx) {
                if (threadIdx.x == 0) s_acc = j;
                break;
            }
            // rejected: the next residual
            c += W;
            W = tr_mass<T, VEC>(zp, zq, V, n, c, nullptr, shf);
            if (!(W > 0.f)) {   // no mass left in float32: sample p instead
                c = 0.f;
                W = 1.f;
                flag |= 8;
            }
        }
        __syncthreads();
        const int acc = s_acc;
        if (acc < 0) {   // every candidate rejected: a draw from the residual
            const int t = tr_draw<T, VEC>(zp, zq, V, n, c, a.u_sample[(size_t)b * (K + 1) + i], csum, shf, shi,
                                          flag);
            if (threadIdx.x == 0) {
                out[i] = t;
                fl[i] = (uint8_t)flag;
            }
            break;
        }
        if (threadIdx.x == 0) {
            out[i] = cand[i * k + acc];
            fl[i] = (uint8_t)flag;
        }
        ++nacc;
        br = acc;
        row = 1 + i * k + acc;
        if (acc > 0 || i == K - 1) {   // a leaf or the last depth: the next token from the node's row
            const T *zn = tp + (size_t)row * V;
            MS Pn, Qn;
            tr_stats<T, VEC>(zn, (const T *)nullptr, V, invT, shm, Pn, Qn);
            TrNorm nn{invT * TR_LOG2E, Pn.m * TR_LOG2E, 1.f / Pn.s, 0.f, 0.f};
            int f2 = 0;
            const int t = tr_draw<T, VEC>(zn, (const T *)nullptr, V, nn, 0.f,
                                          a.u_sample[(size_t)b * (K + 1) + i + 1], csum, shf, shi, f2);
            if (threadIdx.x == 0) {
                out[i + 1] = t;
                fl[i + 1] = (uint8_t)f2;
            }
            break;
        }
    }
    if (threadIdx.x == 0) {
        a.n_accepted[b] = nacc;
        a.branch[b] = br;
    }
}

template <typename T, bool VEC>
static cudaError_t tree_launch(const VerifyTreeArgs &a, cudaStream_t s) {
    const size_t smem = (size_t)((a.V + TR_CH - 1) / TR_CH) * sizeof(float);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.B);
    cfg.blockDim = dim3(TR_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = a.temperature == 0.f ? cudaLaunchKernelEx(&cfg, tree_verify_kernel<T, VEC, true>, a)
                                         : cudaLaunchKernelEx(&cfg, tree_verify_kernel<T, VEC, false>, a);
    count_launch();
    return e;
}

cudaError_t launch_verify_tree(const VerifyTreeArgs &a, cudaStream_t s) {
    const int es = a.dtype == OSPREY_F32 ? 4 : 2;
    const bool vec = a.V % 8 == 0 && (uintptr_t)a.target % 16 == 0 &&
                     (a.draft == nullptr || (uintptr_t)a.draft % 16 == 0) && ((size_t)a.V * es) % 16 == 0;
    if (a.dtype == OSPREY_F32) return vec ? tree_launch<float, true>(a, s) : tree_launch<float, false>(a, s);
    return vec ? tree_launch<uint16_t, true>(a, s) : tree_launch<uint16_t, false>(a, s);
}

}  // namespace osp
