// Draft step on CUDA cores: HBM-bound GEMV kernels with fused prologues and
// epilogues, split-KV GQA decode attention over the paged cache, and an LM
// head that samples on chip.
//
// Per chain step and layer (Sec. 3.3 Eq. 1-3, Sec. 3.4):
//   qkv     z = RMSNorm(x); [q;k;v] = W~_qkv [s; z]; rotary on q,k; k,v -> pages
//   attn    split-KV partial softmax per (row, KV head, split); the last split
//           block of a (row, KV head) merges the partials
//   oproj   x += W_o attn
//   gateup  h = silu(W_gate n) * (W_up n), n = RMSNorm(x)
//   down    x += W_down h
// then lm_head: logits = W_lm RMSNorm(x_L) by warp ranges of the vocabulary,
// each warp keeping (max, sum exp) and argmax of its range; the last block
// picks the range that holds u * S, recomputes only that range's logits and
// scans them in id order.  The logits never leave the chip unless asked for.
#include <math.h>

#include "common.cuh"
#include "draft.cuh"
#include "internal.h"
#include "tma.cuh"

#include <cooperative_groups.h>

namespace osp {

constexpr int GT = 256;          // threads per GEMV / LM-head block
constexpr int GW = GT / 32;      // warps per block
constexpr int AT = 128;          // threads per attention block
constexpr int ATTN_MAX_SPLITS = 128;

// ---------------------------------------------------------------------------
// One warp computes TR dot products of length Kd (bf16 weights streamed from
// HBM, 16 bytes per lane per load, NB loads per row in flight) against RG
// float32 activation rows held in shared memory.  Every (row, activation) pair is
// accumulated in the same order (ascending k, fmaf) whatever TR, NB and RG are,
// so a recomputed logit is bitwise equal to the first one.
template <int TR, int RG, int NB>
__device__ __forceinline__ void warp_dot(const uint16_t *const (&w)[TR], const float *xs, int Kd,
                                         float (&acc)[TR][RG]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int t = 0; t < TR; ++t)
#pragma unroll
        for (int r = 0; r < RG; ++r) acc[t][r] = 0.f;
    for (int base = 0; base < Kd; base += NB * 256) {
        uint4 wv[TR][NB];
#pragma unroll
        for (int i = 0; i < NB; ++i) {
            const int k = base + i * 256 + lane * 8;
#pragma unroll
            for (int t = 0; t < TR; ++t)
                wv[t][i] = (base + i * 256 < Kd) ? ld_stream(w[t] + k) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int i = 0; i < NB; ++i) {
            if (base + i * 256 < Kd) {
                const int k = base + i * 256 + lane * 8;
                float wf[TR][8];
#pragma unroll
                for (int t = 0; t < TR; ++t) unpack8(wv[t][i], wf[t]);
#pragma unroll
                for (int r = 0; r < RG; ++r) {
                    const float4 x0 = *(const float4 *)(xs + (size_t)r * Kd + k);
                    const float4 x1 = *(const float4 *)(xs + (size_t)r * Kd + k + 4);
                    const float xf[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
                    for (int t = 0; t < TR; ++t)
#pragma unroll
                        for (int e = 0; e < 8; ++e) acc[t][r] = fmaf(wf[t][e], xf[e], acc[t][r]);
                }
            }
        }
    }
#pragma unroll
    for (int t = 0; t < TR; ++t)
#pragma unroll
        for (int r = 0; r < RG; ++r) acc[t][r] = warp_sum(acc[t][r]);
}

// ---- prologue helpers -------------------------------------------------------------
// dst[k] = src[k] for a float32 row (zeros when src is null).
__device__ __forceinline__ void stage_copy(float *dst, const float *src, int n) {
    for (int c = threadIdx.x; c < n / 4; c += blockDim.x)
        ((float4 *)dst)[c] = src ? *((const float4 *)src + c) : make_float4(0.f, 0.f, 0.f, 0.f);
}

// dst[k] = widen(src[k]) for a bf16 row (zeros when src is null).
__device__ __forceinline__ void stage_widen(float *dst, const uint16_t *src, int n) {
    for (int c = threadIdx.x; c < n / 8; c += blockDim.x) {
        float f[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (src) unpack8(*((const uint4 *)src + c), f);
        ((float4 *)dst)[2 * c] = make_float4(f[0], f[1], f[2], f[3]);
        ((float4 *)dst)[2 * c + 1] = make_float4(f[4], f[5], f[6], f[7]);
    }
}

// dst[k] = x[k] / sqrt(mean(x^2) + eps) * gain[k] (zeros when x is null).
__device__ __forceinline__ void stage_rmsnorm(float *dst, const float *x, const uint16_t *gain,
                                              int d, float eps, float *red) {
    float ss = 0.f;
    if (x)
        for (int k = threadIdx.x; k < d; k += blockDim.x) {
            float v = x[k];
            ss = fmaf(v, v, ss);
        }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
        red[32] = rsqrtf(t / (float)d + eps);
    }
    __syncthreads();
    const float inv = red[32];
    for (int k = threadIdx.x; k < d; k += blockDim.x)
        dst[k] = x ? x[k] * inv * bf_to_f(gain[k]) : 0.f;
    __syncthreads();
}

__device__ __forceinline__ void rope_cs(double inv_freq, int pos, float &c, float &s) {
    // angle reduced modulo 2*pi in double before the float sin/cos
    const double turns = (double)pos * inv_freq * 0.15915494309189535;
    const double frac = turns - floor(turns);
    sincosf((float)(frac * 6.283185307179586), &s, &c);
}

// ---------------------------------------------------------------------------
template <int MODE, int RG>
__global__ void __launch_bounds__(GT) gemv_kernel(const GemvArgs a) {
    extern __shared__ __align__(16) float xs[];
    __shared__ float red[33];
    __shared__ int s_b[RG], s_pos[RG], s_act[RG];
    const Dims &D = a.dim;
    const int r0 = blockIdx.y * RG;
    if (threadIdx.x < RG) {
        int b = 0, pos = 0;
        const int r = r0 + threadIdx.x;
        const bool act = r < a.R && a.map.row(r, b, pos);
        s_b[threadIdx.x] = b;
        s_pos[threadIdx.x] = pos;
        s_act[threadIdx.x] = act;
    }
    __syncthreads();

    int Kd, n_tasks;
    if (MODE == G_FEAT) { Kd = D.feat; n_tasks = D.d; }
    else if (MODE == G_QKV) { Kd = 2 * D.d; n_tasks = (D.Hq + 2 * D.Hkv) * D.hd / 2; }
    else if (MODE == G_OPROJ) { Kd = D.Hq * D.hd; n_tasks = D.d; }
    else if (MODE == G_GATEUP) { Kd = D.d; n_tasks = D.F; }
    else { Kd = D.F; n_tasks = D.d; }

    // ---- prologue: stage the activation rows (float32) in shared memory
    for (int rr = 0; rr < RG; ++rr) {
        const int r = r0 + rr;
        const bool act = s_act[rr];
        float *row = xs + (size_t)rr * Kd;
        if (MODE == G_FEAT) {
            stage_widen(row, act ? a.feats + (size_t)r * D.feat : nullptr, Kd);
            if (blockIdx.x == 0 && act) {     // residual stream of layer 0 starts at E[x]
                const uint16_t *e = a.embed + (size_t)a.tokens[r] * D.d;
                for (int k = threadIdx.x; k < D.d; k += blockDim.x) a.x[(size_t)r * D.d + k] = bf_to_f(e[k]);
            }
        } else if (MODE == G_QKV) {
            stage_copy(row, act ? a.s + (size_t)r * D.d : nullptr, D.d);
            stage_rmsnorm(row + D.d, act ? a.x + (size_t)r * D.d : nullptr, a.gain, D.d, D.eps, red);
        } else if (MODE == G_OPROJ) {
            stage_copy(row, act ? a.xin + (size_t)r * Kd : nullptr, Kd);
        } else if (MODE == G_GATEUP) {
            stage_rmsnorm(row, act ? a.x + (size_t)r * D.d : nullptr, a.gain, D.d, D.eps, red);
        } else {
            stage_copy(row, act ? a.xin + (size_t)r * Kd : nullptr, Kd);
        }
    }
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int task = blockIdx.x * GW + warp; task < n_tasks; task += gridDim.x * GW) {
        if (MODE == G_QKV || MODE == G_GATEUP) {
            const uint16_t *w[2];
            int h = 0, i = 0;
            if (MODE == G_QKV) {
                h = task / (D.hd / 2);
                i = task % (D.hd / 2);
                w[0] = a.W + ((size_t)h * D.hd + i) * Kd;
                w[1] = a.W + ((size_t)h * D.hd + i + D.hd / 2) * Kd;
            } else {
                w[0] = a.W + (size_t)task * Kd;
                w[1] = a.W2 + (size_t)task * Kd;
            }
            float acc[2][RG];
            warp_dot<2, RG, 8>(w, xs, Kd, acc);
#pragma unroll
            for (int rr = 0; rr < RG; ++rr) {
                if (lane != rr || !s_act[rr]) continue;
                const int r = r0 + rr;
                if (MODE == G_GATEUP) {
                    const float g = acc[0][rr], u = acc[1][rr];
                    a.out[(size_t)r * D.F + task] = g / (1.f + expf(-g)) * u;
                } else {
                    const int b = s_b[rr], pos = s_pos[rr];
                    float x1 = acc[0][rr], x2 = acc[1][rr];
                    if (h < D.Hq + D.Hkv) {       // rotary on q and k (rotate-half pairs)
                        float c, s;
                        rope_cs(a.inv_freq[i], pos, c, s);
                        const float y1 = x1 * c - x2 * s, y2 = x2 * c + x1 * s;
                        x1 = y1;
                        x2 = y2;
                    }
                    if (h < D.Hq) {
                        float *q = a.q + (size_t)r * D.Hq * D.hd + (size_t)h * D.hd;
                        q[i] = x1;
                        q[i + D.hd / 2] = x2;
                    } else {
                        const bool is_k = h < D.Hq + D.Hkv;
                        const int kvh = is_k ? h - D.Hq : h - D.Hq - D.Hkv;
                        const int page = a.page_table[(size_t)b * a.max_pages + pos / D.P];
                        uint16_t *dst = (is_k ? a.k_pages : a.v_pages) +
                                        (((size_t)page * D.Hkv + kvh) * D.P + pos % D.P) * D.hd;
                        dst[i] = f_to_bf(x1);
                        dst[i + D.hd / 2] = f_to_bf(x2);
                    }
                }
            }
        } else {
            const uint16_t *w[1] = {a.W + (size_t)task * Kd};
            float acc[1][RG];
            warp_dot<1, RG, 16>(w, xs, Kd, acc);
#pragma unroll
            for (int rr = 0; rr < RG; ++rr) {
                if (lane != rr || !s_act[rr]) continue;
                const int r = r0 + rr;
                if (MODE == G_FEAT) a.s[(size_t)r * D.d + task] = acc[0][rr];
                else a.x[(size_t)r * D.d + task] += acc[0][rr];   // residual add (oproj, down)
            }
        }
    }
}

// Attention output element (row r, column col of the Hq hd heads): float32
// into out, or the three bf16 planes x ~= q0 + q1 + q2 (q_i the bf16 rounding of
// what the earlier planes leave) of the O projection's tensor-core operand.
__device__ __forceinline__ void attn_store(const AttnArgs &a, int r, int col, float v) {
    const int ha = a.dim.Hq * a.dim.hd;
    if (!a.out_planes) {
        a.out[(size_t)r * ha + col] = v;
        return;
    }
    const size_t plane = (size_t)a.npad * ha;
    uint16_t *p = a.out_planes + (size_t)r * ha + col;
    float rem = v;
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        const uint16_t q = f_to_bf(rem);
        p[i * plane] = q;
        rem -= bf_to_f(q);
    }
}

// ---------------------------------------------------------------------------
// Split-KV GQA decode attention (Sec. 4, paged serving).  Both kernels below
// give a block (key range, KV head, row) and its warps the range's pages
// round-robin (attn_warp_pages); HD/8 lanes share one key (8 dims, 16 bytes
// each).  attn_kernel merges the ranges through global partials (the last block
// of a (row, KV head) merges); attn_cluster_kernel merges them on chip.
__device__ __forceinline__ void cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Transposed butterfly over a group of 2*O lanes holding N partial sums each:
// every level hands half of the lane's values to its partner and adds the half
// it receives, so after log2(2*O) levels each lane holds N / (2*O) complete
// sums (for N < 2*O, one sum shared by 2*O / N lanes).  That is N - 1 shuffles
// in place of N * log2(2*O).
template <int N, int O, int NVV>
struct AttnTrReduce {
    static __device__ __forceinline__ void run(float (&v)[NVV], int lane) {
        if constexpr (O >= 1) {
            if constexpr (N >= 2) {
                constexpr int H = N / 2;
                const bool up = (lane & O) != 0;
#pragma unroll
                for (int i = 0; i < H; ++i) {
                    const float send = up ? v[i] : v[i + H];
                    const float keep = up ? v[i + H] : v[i];
                    v[i] = keep + __shfl_xor_sync(0xffffffffu, send, O);
                }
                AttnTrReduce<H, O / 2, NVV>::run(v, lane);
            } else {
                v[0] += __shfl_xor_sync(0xffffffffu, v[0], O);
                AttnTrReduce<1, O / 2, NVV>::run(v, lane);
            }
        }
    }
};

// One warp's share of a key range [k_begin, k_end) of row r, KV head kvh: its
// pages (warp, warp + NW, ...) stream through the warp's own NSPW shared-memory
// stages with 1-D bulk copies; pages wholly below pos0 (the context committed
// before this draft call, which no kernel of the call writes) are requested
// before griddepcontrol.wait, which this function executes.  Per page each K/V
// chunk is unpacked once for the G query heads and the q.k sums are completed
// by a transposed butterfly (one score per lane).  Leaves the warp's partial
// (max, sum, G x HD accumulator) in sm_m / sm_l / sm_acc[warp].
// QCG: read q through L2 (q written by other blocks of the same grid).
template <int HD, int G, int NW, int NSPW, bool QCG = false>
__device__ __forceinline__ void attn_warp_pages(const AttnArgs &a, int b, int r, int kvh, int qh0, int k_begin,
                                                int k_end, int pos0, uint8_t *ring, uint64_t (*full)[NSPW],
                                                float (*sm_m)[G], float (*sm_l)[G], float (*sm_acc)[G][HD]) {
    constexpr int LPK = HD / 8;
    constexpr int KPL = 32 / LPK;
    constexpr int NIT = 16 / KPL;     // row loads per page (16 positions)
    constexpr int PB = 16 * HD * 2;   // bytes of one page of one head (K or V)
    const Dims &D = a.dim;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int pg0 = k_begin / 16;
    const int npg = k_end > k_begin ? (k_end - k_begin + 15) / 16 : 0;
    const int my_pages = npg > warp ? (npg - warp + NW - 1) / NW : 0;   // local pages warp + j * NW
    const int kg = lane / LPK, dl = (lane % LPK) * 8;
    const float scale = rsqrtf((float)HD);
    const size_t head_stride = (size_t)D.P * HD;
    uint8_t *wring = ring + (size_t)warp * NSPW * 2 * PB;
    const int32_t *ptab = a.page_table + (size_t)b * a.max_pages + pg0;

    // lane i holds the page id of the warp's i-th page (the page table is fixed for the call)
    const int my_pid = lane < my_pages ? __ldg(ptab + warp + lane * NW) : 0;
    auto issue = [&](int j, int page) {   // lane 0: page j of this warp into stage j % NSPW
        const int st = j % NSPW;
        uint8_t *dst = wring + (size_t)st * 2 * PB;
        mbar_arrive_expect_tx(&full[warp][st], 2 * PB);
        bulk_g2s(dst, a.k_pages + ((size_t)page * D.Hkv + kvh) * head_stride, PB, &full[warp][st]);
        bulk_g2s(dst + PB, a.v_pages + ((size_t)page * D.Hkv + kvh) * head_stride, PB, &full[warp][st]);
    };
    auto pid_of = [&](int j) {   // warp-wide
        const int p = __shfl_sync(0xffffffffu, my_pid, j & 31);
        return j < 32 ? p : __ldg(ptab + warp + j * NW);
    };
    const int first = min(NSPW, my_pages);
    int pids[NSPW];
#pragma unroll
    for (int j = 0; j < NSPW; ++j) pids[j] = pid_of(j);
    int issued = 0;
    if (lane == 0) {
        for (int st = 0; st < NSPW; ++st) mbar_init(&full[warp][st], 1);
        mbar_fence_init();
        // committed pages: every position of the page below pos0
#pragma unroll
        for (int j = 0; j < NSPW; ++j)
            if (j == issued && j < first && (pg0 + warp + j * NW + 1) * 16 <= pos0) issue(issued++, pids[j]);
    }
    pdl_wait();   // q and this call's K/V rows come from the QKV kernels
    if (lane == 0) {
#pragma unroll
        for (int j = 0; j < NSPW; ++j)
            if (j >= issued && j < first) issue(j, pids[j]);
        issued = first;
    }
    __syncwarp();

    constexpr int NV = G * NIT;                    // partial dot products per lane and page
    constexpr int NF = NV >= LPK ? NV / LPK : 1;   // complete scores per lane after the reduction
    constexpr int REP = NV >= LPK ? 1 : LPK / NV;  // lanes holding the same score
    constexpr int LPG = LPK / G;                   // lanes of a key group per query head
    static_assert(G <= LPK && NF <= NIT, "score layout");
    const int sbase = ((lane % LPK) / REP) * NF;   // the lane's scores: head sbase / NIT
    float q[G][8], acc[G][8], m_run[G];
    float m_own_run = -INFINITY, l_own = 0.f;      // the lane's head: running max, partial sum
#pragma unroll
    for (int g = 0; g < G; ++g) {
        const float *qp = a.q + (size_t)r * D.Hq * HD + (size_t)(qh0 + g) * HD + dl;
        const float4 q0 = QCG ? __ldcg((const float4 *)qp) : *(const float4 *)qp;
        const float4 q1 = QCG ? __ldcg((const float4 *)(qp + 4)) : *(const float4 *)(qp + 4);
        q[g][0] = q0.x * scale; q[g][1] = q0.y * scale; q[g][2] = q0.z * scale; q[g][3] = q0.w * scale;
        q[g][4] = q1.x * scale; q[g][5] = q1.y * scale; q[g][6] = q1.z * scale; q[g][7] = q1.w * scale;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[g][e] = 0.f;
        m_run[g] = -INFINITY;
    }
    int consumed = 0;
    for (int j = 0; j < my_pages; ++j) {
        const int st = j % NSPW;
        if (!__all_sync(0xffffffffu, mbar_wait(&full[warp][st], (uint32_t)(j / NSPW) & 1))) {   // warp-uniform exit
            if (lane == 0) set_status(a.status, OSPREY_ERR_TIMEOUT);
            break;
        }
        consumed = j + 1;
        const uint16_t *ks = (const uint16_t *)(wring + (size_t)st * 2 * PB);
        const uint16_t *vs = ks + 16 * HD;
        uint4 kr[NIT], vr[NIT];
#pragma unroll
        for (int it = 0; it < NIT; ++it) {
            const int slot = it * KPL + kg;
            kr[it] = *(const uint4 *)(ks + slot * HD + dl);
            vr[it] = *(const uint4 *)(vs + slot * HD + dl);
        }
        if (j + NSPW < my_pages) {   // refill the stage once every lane has read it
            const int pn = pid_of(j + NSPW);
            __syncwarp();
            if (lane == 0) {
                fence_proxy_async_smem();
                issue(j + NSPW, pn);
                issued = j + NSPW + 1;
            }
        }
        const int key0 = (pg0 + warp + j * NW) * 16;
        // partial q.k over the lane's HD / LPK dimensions, each K chunk unpacked once
        float v[NV];
#pragma unroll
        for (int it = 0; it < NIT; ++it) {
            float kf[8];
            unpack8(kr[it], kf);
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float d = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) d = fmaf(q[g][e], kf[e], d);
                v[g * NIT + it] = d;
            }
        }
        // complete the sums across the LPK lanes of each key group, leaving the
        // lane NF consecutive scores (indices sbase .. sbase + NF - 1 of g * NIT + it)
        AttnTrReduce<NV, LPK / 2, NV>::run(v, lane);
        float mloc = -INFINITY;
#pragma unroll
        for (int i = 0; i < NF; ++i) {
            const int key = key0 + ((sbase + i) % NIT) * KPL + kg;
            v[i] = key < k_end ? v[i] : -INFINITY;
            mloc = fmaxf(mloc, v[i]);
        }
        // page maximum of the lane's head, then of every head
#pragma unroll
        for (int o = 1; o < LPG; o <<= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
#pragma unroll
        for (int o = LPK; o < 32; o <<= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
        float corr[G];
#pragma unroll
        for (int g = 0; g < G; ++g) {
            const float mn = fmaxf(m_run[g], __shfl_sync(0xffffffffu, mloc, g * LPG));
            corr[g] = mn == -INFINITY ? 1.f : __expf(m_run[g] - mn);
            m_run[g] = mn;
        }
        const float m_own = fmaxf(m_own_run, mloc);
        l_own *= m_own == -INFINITY ? 1.f : __expf(m_own_run - m_own);
        m_own_run = m_own;
        float p[NF];
#pragma unroll
        for (int i = 0; i < NF; ++i) {
            p[i] = v[i] == -INFINITY ? 0.f : __expf(v[i] - m_own);
            l_own += p[i];
        }
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[g][e] *= corr[g];
        // p . V: each V chunk unpacked once, each weight fetched from the lane holding it
#pragma unroll
        for (int it = 0; it < NIT; ++it) {
            float vf[8];
            unpack8(vr[it], vf);
#pragma unroll
            for (int g = 0; g < G; ++g) {
                const int vi = g * NIT + it;
                const float pp = __shfl_sync(0xffffffffu, p[vi % NF], (lane & ~(LPK - 1)) | ((vi / NF) * REP));
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[g][e] = fmaf(pp, vf[e], acc[g][e]);
            }
        }
    }
    // after a timed-out wait: let the copies already requested land before the block can exit
    if (lane == 0)
        for (int j = consumed; j < issued; ++j) mbar_wait(&full[warp][j % NSPW], (uint32_t)(j / NSPW) & 1, 200000000LL);
    // the warp's sums per head (REP lanes hold each score), then merge the key
    // groups of the warp and the warps of the block
#pragma unroll
    for (int o = 1; o < LPG; o <<= 1) l_own += __shfl_xor_sync(0xffffffffu, l_own, o);
#pragma unroll
    for (int o = LPK; o < 32; o <<= 1) l_own += __shfl_xor_sync(0xffffffffu, l_own, o);
    float l[G];
#pragma unroll
    for (int g = 0; g < G; ++g) l[g] = __shfl_sync(0xffffffffu, l_own, g * LPG) * (1.f / REP);
#pragma unroll
    for (int g = 0; g < G; ++g) {
#pragma unroll
        for (int o = LPK; o < 32; o <<= 1) {
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[g][e] += __shfl_xor_sync(0xffffffffu, acc[g][e], o);
        }
        if (lane < LPK) {
#pragma unroll
            for (int e = 0; e < 8; ++e) sm_acc[warp][g][dl + e] = acc[g][e];
        }
        if (lane == 0) { sm_m[warp][g] = m_run[g]; sm_l[warp][g] = l[g]; }
    }
}

// Stages per warp of the global-partials attention (4 warps per block): two
// or three blocks fit an SM next to the ring.
template <int HD>
struct AttnSplit {
    static constexpr int PB = 16 * HD * 2;
    static constexpr int NSPW = HD == 128 ? 2 : 4;
    static constexpr int RING = (AT / 32) * NSPW * 2 * PB;
};

template <int HD, int G>
__global__ void __launch_bounds__(AT) attn_kernel(const AttnArgs a) {
    constexpr int NW = AT / 32, NSPW = AttnSplit<HD>::NSPW;
    extern __shared__ __align__(128) uint8_t ring[];   // [NW][NSPW][K | V][PB]
    __shared__ __align__(8) uint64_t full[NW][NSPW];
    __shared__ float sm_m[NW][G], sm_l[NW][G];
    __shared__ float sm_acc[NW][G][HD];
    const Dims &D = a.dim;
    const int split = blockIdx.x, kvh = blockIdx.y, r = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    pdl_trigger();   // the next projection may start streaming its weights
    int b, pos;
    if (!a.map.row(r, b, pos)) return;   // the row map was written by the prepare kernel
    const int n_keys = pos + 1, pos0 = a.map.pos0[b];
    const int k_begin = split * a.split_len;   // a multiple of the page size
    const int k_end = min(n_keys, k_begin + a.split_len);
    attn_warp_pages<HD, G, NW, NSPW>(a, b, r, kvh, kvh * G, k_begin, k_end, pos0, ring, full, sm_m, sm_l, sm_acc);
    __syncthreads();
    const int Hq = D.Hq;
    for (int idx = threadIdx.x; idx < G * HD; idx += AT) {
        const int g = idx / HD, dim = idx % HD;
        float M = -INFINITY;
        for (int w = 0; w < AT / 32; ++w) M = fmaxf(M, sm_m[w][g]);
        float num = 0.f, den = 0.f;
        if (M != -INFINITY)
            for (int w = 0; w < AT / 32; ++w) {
                const float f = __expf(sm_m[w][g] - M);
                num = fmaf(f, sm_acc[w][g][dim], num);
                den = fmaf(f, sm_l[w][g], den);
            }
        float *pp = a.part + (((size_t)r * Hq + kvh * G + g) * a.n_splits + split) * (HD + 2);
        pp[2 + dim] = num;
        if (dim == 0) { pp[0] = M; pp[1] = den; }
    }
    if (!arrive_last(a.ticket + (size_t)r * D.Hkv + kvh, a.n_splits)) return;
    // last split block of this (row, KV head): merge the split partials.  A
    // thread issues every load it needs at once (split maxima and sums, and its
    // accumulator values for up to SPR splits), so up to SPR splits cost one
    // round trip to L2.
    constexpr int IPT = (G * HD + AT - 1) / AT;            // (head, dim) items per thread
    constexpr int SPR = IPT >= 8 ? 8 : (IPT >= 4 ? 16 : 32);  // splits per pass, <= 64 values held
    __shared__ float s_w[G][ATTN_MAX_SPLITS], s_l[G][ATTN_MAX_SPLITS];
    __shared__ float s_den[G];
    const int ns = a.n_splits;
    const float *base = a.part + ((size_t)r * Hq + kvh * G) * ns * (HD + 2);
    for (int idx = threadIdx.x; idx < G * ns; idx += AT) {
        const int g = idx / ns, sp = idx % ns;
        const float *pp = base + ((size_t)g * ns + sp) * (HD + 2);
        s_w[g][sp] = __ldcg(pp);
        s_l[g][sp] = __ldcg(pp + 1);
    }
    float v[IPT][SPR];
    auto load_pass = [&](int s0) {
#pragma unroll
        for (int it = 0; it < IPT; ++it) {
            const int idx = threadIdx.x + it * AT;
            const int g = idx / HD, dim = idx % HD;
#pragma unroll
            for (int k = 0; k < SPR; ++k)
                v[it][k] = idx < G * HD && s0 + k < ns
                               ? __ldcg(base + ((size_t)g * ns + s0 + k) * (HD + 2) + 2 + dim)
                               : 0.f;
        }
    };
    load_pass(0);
    __syncthreads();
    for (int g = warp; g < G; g += AT / 32) {
        float M = -INFINITY;
        for (int sp = lane; sp < ns; sp += 32) M = fmaxf(M, s_w[g][sp]);
        M = warp_max(M);
        float den = 0.f;
        for (int sp = lane; sp < ns; sp += 32) {
            const float ms = s_w[g][sp];
            const float f = ms == -INFINITY ? 0.f : __expf(ms - M);
            den = fmaf(f, s_l[g][sp], den);
            s_w[g][sp] = f;
        }
        den = warp_sum(den);
        if (lane == 0) s_den[g] = den;
    }
    __syncthreads();
    float num[IPT];
#pragma unroll
    for (int it = 0; it < IPT; ++it) num[it] = 0.f;
    for (int s0 = 0; s0 < ns; s0 += SPR) {
        if (s0 > 0) load_pass(s0);
#pragma unroll
        for (int it = 0; it < IPT; ++it) {
            const int g = (threadIdx.x + it * AT) / HD;
            if (g >= G) continue;
#pragma unroll
            for (int k = 0; k < SPR; ++k)
                if (s0 + k < ns) num[it] = fmaf(s_w[g][s0 + k], v[it][k], num[it]);
        }
    }
#pragma unroll
    for (int it = 0; it < IPT; ++it) {
        const int idx = threadIdx.x + it * AT;
        if (idx >= G * HD) continue;
        const int g = idx / HD, dim = idx % HD;
        attn_store(a, r, (kvh * G + g) * HD + dim, num[it] / s_den[g]);
    }
}

// ---------------------------------------------------------------------------
// Split-KV GQA decode attention with the split merge kept on chip.  A cluster
// of CS blocks takes one (row, KV head); block k of the cluster takes the k-th
// key range, its warps the range's pages round-robin (attn_warp_pages: each
// warp streams its pages through its own AttnCluster::NSPW shared-memory stages
// with 1-D bulk copies, one page of one head being P x HD contiguous bf16 for K
// and again for V).  Each block reduces its warps in shared memory and pushes its partial
// (max, sum, G x HD accumulator) into block 0's shared memory through
// distributed shared memory; block 0 merges the CS partials after one cluster
// barrier.  Every block of a cluster shares the row, so either all of them
// reach the barriers or the whole cluster returns before the first.
#ifndef OSP_ATTN_CS
#define OSP_ATTN_CS 8       // blocks per cluster (16 needs the non-portable cluster size)
#endif
#ifndef OSP_ATTN_RING_KB
#define OSP_ATTN_RING_KB 220   // shared memory budget of a block (ring + partials)
#endif
#ifndef OSP_ATTN_WARPS
#define OSP_ATTN_WARPS 16   // warps per block for groups of up to two query heads (8 beyond)
#endif

template <int HD, int G, int CS>
struct AttnCluster {
    // groups of <= 2 heads fit 128 registers: 16 warps, every page of a 2k-key
    // range in flight at once; larger groups keep 8 warps and more stages each
    static constexpr int NW = G <= 2 ? OSP_ATTN_WARPS : 8;
    static constexpr int THREADS = NW * 32;
    static constexpr int PB = 16 * HD * 2;   // bytes of one page of one head (K or V)
    static constexpr int STATIC = NW * G * HD * 4 + CS * G * HD * 4 + 2 * (NW + CS) * G * 4 + 256;
    static constexpr int FIT = (OSP_ATTN_RING_KB * 1024 - STATIC) / (NW * 2 * PB);
    static constexpr int NSPW = FIT > 4 ? 4 : (FIT < 1 ? 1 : FIT);   // stages per warp
    static constexpr int RING = NW * NSPW * 2 * PB;
};

template <int HD, int G, int CS>
__global__ void __launch_bounds__(AttnCluster<HD, G, CS>::THREADS, 1) attn_cluster_kernel(const AttnArgs a) {
    namespace cg = cooperative_groups;
    using C = AttnCluster<HD, G, CS>;
    constexpr int NW = C::NW, NSPW = C::NSPW;
    extern __shared__ __align__(128) uint8_t ring[];   // [NW][NSPW][K | V][PB]
    __shared__ __align__(8) uint64_t full[NW][NSPW];
    __shared__ float sm_m[NW][G], sm_l[NW][G];
    __shared__ float sm_acc[NW][G][HD];
    __shared__ float gm[CS][G], gl[CS][G];   // block 0: the partials of the cluster
    __shared__ float gacc[CS][G][HD];
    cg::cluster_group cluster = cg::this_cluster();
    const Dims &D = a.dim;
    const int split = (int)cluster.block_rank(), r = blockIdx.z;
    const int qh0 = blockIdx.y * G, kvh = qh0 / (D.Hq / D.Hkv);   // the block's G query heads share a KV head
    cluster_arrive_relaxed();   // this block has started: its shared memory may be written by the cluster
    pdl_trigger();              // the next projection may start streaming its weights
    int b, pos;
    if (!a.map.row(r, b, pos)) return;   // the whole cluster (same row) leaves here
    const int n_keys = pos + 1, pos0 = a.map.pos0[b];
    const int k_begin = split * a.split_len;   // a multiple of the page size
    const int k_end = min(n_keys, k_begin + a.split_len);
    attn_warp_pages<HD, G, NW, NSPW>(a, b, r, kvh, qh0, k_begin, k_end, pos0, ring, full, sm_m, sm_l, sm_acc);
    __syncthreads();
    cluster_wait_acquire();   // every block of the cluster has started
    float *r_acc = cluster.map_shared_rank(&gacc[split][0][0], 0);
    float *r_m = cluster.map_shared_rank(&gm[split][0], 0);
    float *r_l = cluster.map_shared_rank(&gl[split][0], 0);
    for (int idx = threadIdx.x; idx < G * HD; idx += C::THREADS) {
        const int g = idx / HD, dim = idx % HD;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NW; ++w) M = fmaxf(M, sm_m[w][g]);
        float num = 0.f, den = 0.f;
        if (M != -INFINITY)
#pragma unroll
            for (int w = 0; w < NW; ++w) {
                const float f = sm_m[w][g] == -INFINITY ? 0.f : __expf(sm_m[w][g] - M);
                num = fmaf(f, sm_acc[w][g][dim], num);
                den = fmaf(f, sm_l[w][g], den);
            }
        r_acc[idx] = num;
        if (dim == 0) { r_m[g] = M; r_l[g] = den; }
    }
    cluster_arrive_release();   // the pushed partial is visible to block 0 once it waits
    if (split != 0) return;
    cluster_wait_acquire();
    for (int idx = threadIdx.x; idx < G * HD; idx += C::THREADS) {
        const int g = idx / HD, dim = idx % HD;
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < CS; ++k) M = fmaxf(M, gm[k][g]);
        float num = 0.f, den = 0.f;
#pragma unroll
        for (int k = 0; k < CS; ++k) {
            const float f = gm[k][g] == -INFINITY ? 0.f : __expf(gm[k][g] - M);
            num = fmaf(f, gacc[k][g][dim], num);
            den = fmaf(f, gl[k][g], den);
        }
        attn_store(a, r, (qh0 + g) * HD + dim, num / den);
    }
}

// ---------------------------------------------------------------------------
// LM head + on-chip sampling.
__device__ __forceinline__ void warp_range(int V, int warps_total, int gw, int &lo, int &hi) {
    lo = (int)(((long long)V * gw) / warps_total);
    hi = (int)(((long long)V * (gw + 1)) / warps_total);
}

template <int RG>
__device__ void lm_sample(const LmArgs &a, int b, int rr, int src_row, const float *xs,
                          float *ybuf) {
    __shared__ MS shm[GW];
    __shared__ AM sha[GW];
    __shared__ float sh_scan[33];
    __shared__ int s_pick, s_last, s_tok;
    __shared__ float s_before, s_before_last, s_e;
    const Dims &D = a.dim;
    const int V = D.V, Wt = a.warps_total;
    const bool greedy = a.temperature == 0.f;
    const float invT = greedy ? 1.f : 1.f / a.temperature;
    const float4 *st = a.warp_stats + (size_t)b * Wt;
    const int per = (Wt + GT - 1) / GT;
    const int e0 = threadIdx.x * per, e1 = min(Wt, e0 + per);

    MS ms{-INFINITY, 0.f};
    AM am{-INFINITY, 0x7fffffff};
    for (int e = e0; e < e1; ++e) {
        const float4 v = __ldcg(st + e);
        ms = ms_combine(ms, MS{v.x, v.y});
        am = am_combine(am, AM{v.z, __float_as_int(v.w)});
    }
    const MS tot = block_ms(ms, shm);
    const AM best = block_am(am, sha);
    const float M = tot.m;
    int token;
    float qx, S;
    if (greedy) {
        token = best.i;
        qx = 1.f;
        S = tot.s;
    } else {
        // contributions of the warp ranges, in id order
        float mine = 0.f;
        for (int e = e0; e < e1; ++e) {
            const float4 v = __ldcg(st + e);
            mine += v.x == -INFINITY ? 0.f : v.y * __expf(v.x - M);
        }
        float Ssum;
        const float ex = block_excl_scan(mine, sh_scan, &Ssum);
        S = Ssum;
        const float t = a.u_draft[(size_t)b * a.K + a.step] * S;
        if (threadIdx.x == 0) { s_pick = 0x7fffffff; s_last = -1; }
        __syncthreads();
        float run = ex;
        int found = 0x7fffffff, lastpos = -1;
        float before = 0.f, before_last = 0.f;
        for (int e = e0; e < e1; ++e) {
            const float4 v = __ldcg(st + e);
            const float c = v.x == -INFINITY ? 0.f : v.y * __expf(v.x - M);
            if (c > 0.f) { lastpos = e; before_last = run; }
            if (found == 0x7fffffff && c > 0.f && t < run + c) { found = e; before = run; }
            run += c;
        }
        atomicMin(&s_pick, found);
        atomicMax(&s_last, lastpos);
        __syncthreads();
        if (found != 0x7fffffff && found == s_pick) s_before = before;
        if (s_pick == 0x7fffffff && lastpos >= 0 && lastpos == s_last) s_before_last = before_last;
        __syncthreads();
        const int pick = s_pick != 0x7fffffff ? s_pick : s_last;
        const float cbefore = s_pick != 0x7fffffff ? s_before : s_before_last;
        // recompute the chosen range's logits (same arithmetic as the first pass)
        int lo, hi;
        warp_range(V, Wt, pick, lo, hi);
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        for (int n = lo + warp; n < hi; n += GW) {
            const uint16_t *w[1] = {a.W + (size_t)n * D.d};
            float acc[1][RG];
            warp_dot<1, RG, 16>(w, xs, D.d, acc);
            if (lane == 0) ybuf[n - lo] = acc[0][rr] * invT;
        }
        __syncthreads();
        if (warp == 0) {
            float run2 = cbefore;
            int tok = -1, lastp = -1;
            float etok = 0.f, elast = 0.f;
            for (int base = lo; base < hi && tok < 0; base += 32) {
                const int n = base + lane;
                const float e = n < hi ? __expf(ybuf[n - lo] - M) : 0.f;
                const float inc = warp_incl_scan(e) + run2;
                const unsigned hit = __ballot_sync(0xffffffffu, n < hi && e > 0.f && t < inc);
                const unsigned pos = __ballot_sync(0xffffffffu, n < hi && e > 0.f);
                if (pos) {
                    const int l2 = 31 - __clz(pos);
                    lastp = base + l2;
                    elast = __shfl_sync(0xffffffffu, e, l2);
                }
                if (hit) {
                    const int l2 = __ffs(hit) - 1;
                    tok = base + l2;
                    etok = __shfl_sync(0xffffffffu, e, l2);
                }
                run2 = __shfl_sync(0xffffffffu, inc, 31);
            }
            if (lane == 0) {
                if (tok < 0) { tok = lastp >= 0 ? lastp : lo; etok = elast; }
                s_tok = tok;
                s_e = etok;
            }
        }
        __syncthreads();
        token = s_tok;
        qx = s_e / S;
    }
    if (threadIdx.x == 0) {
        a.tokens[(size_t)b * a.K + a.step] = token;
        if (a.qx) a.qx[(size_t)b * a.K + a.step] = qx;
        if (a.stats) {
            a.stats[((size_t)b * a.K + a.step) * 2 + 0] = M;
            a.stats[((size_t)b * a.K + a.step) * 2 + 1] = logf(S);
        }
    }
    if (a.step + 1 < a.K) {
        // next chain row: context slot <- x_L (Sec. 3.4), residual <- E[token]
        const float *xl = a.x_in + (size_t)src_row * D.d;
        for (int k = threadIdx.x; k < D.d; k += blockDim.x)
            a.s_chain[(size_t)b * D.d + k] = xl[k];
        __syncthreads();
        const uint16_t *e = a.embed + (size_t)token * D.d;
        for (int k = threadIdx.x; k < D.d; k += blockDim.x)
            a.x_chain[(size_t)b * D.d + k] = bf_to_f(e[k]);
    }
    __syncthreads();
}

template <int RG>
__global__ void __launch_bounds__(GT) lm_head_kernel(const LmArgs a) {
    extern __shared__ __align__(16) float xs[];   // [RG][d] float32, then the range's logits
    __shared__ float red[33];
    __shared__ int s_src[RG], s_act[RG];
    const Dims &D = a.dim;
    const int b0 = blockIdx.y * RG;
    if (threadIdx.x < RG) {
        const int b = b0 + threadIdx.x;
        const bool act = b < a.B && a.map.valid[b];
        s_act[threadIdx.x] = act;
        s_src[threadIdx.x] = act ? (a.src_is_ext ? b * a.max_new + a.map.nnew[b] - 1 : b) : 0;
    }
    __syncthreads();
    for (int rr = 0; rr < RG; ++rr)
        stage_rmsnorm(xs + (size_t)rr * D.d, s_act[rr] ? a.x_in + (size_t)s_src[rr] * D.d : nullptr,
                      a.gain, D.d, D.eps, red);
    float *ybuf = xs + (size_t)RG * D.d;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gw = blockIdx.x * GW + warp;
    int lo, hi;
    warp_range(D.V, a.warps_total, gw, lo, hi);
    const float invT = a.temperature == 0.f ? 1.f : 1.f / a.temperature;
    float m[RG], s[RG], bv[RG];
    int bi[RG];
#pragma unroll
    for (int rr = 0; rr < RG; ++rr) { m[rr] = -INFINITY; s[rr] = 0.f; bv[rr] = -INFINITY; bi[rr] = 0x7fffffff; }
    auto consume = [&](int n, int rr, float z) {
        if (a.logits && lane == 0 && s_act[rr])
            a.logits[((size_t)(b0 + rr) * a.K + a.step) * D.V + n] = z;
        const float y = z * invT;
        if (y > m[rr]) { s[rr] = s[rr] * __expf(m[rr] - y) + 1.f; m[rr] = y; }
        else s[rr] += __expf(y - m[rr]);
        if (z > bv[rr]) { bv[rr] = z; bi[rr] = n; }
    };
    int n = lo;
    for (; n + 4 <= hi; n += 4) {
        const uint16_t *w[4] = {a.W + (size_t)n * D.d, a.W + (size_t)(n + 1) * D.d,
                                a.W + (size_t)(n + 2) * D.d, a.W + (size_t)(n + 3) * D.d};
        float acc[4][RG];
        warp_dot<4, RG, 4>(w, xs, D.d, acc);
#pragma unroll
        for (int t = 0; t < 4; ++t)
#pragma unroll
            for (int rr = 0; rr < RG; ++rr) consume(n + t, rr, acc[t][rr]);
    }
    for (; n < hi; ++n) {
        const uint16_t *w[1] = {a.W + (size_t)n * D.d};
        float acc[1][RG];
        warp_dot<1, RG, 16>(w, xs, D.d, acc);
#pragma unroll
        for (int rr = 0; rr < RG; ++rr) consume(n, rr, acc[0][rr]);
    }
    if (lane == 0) {
#pragma unroll
        for (int rr = 0; rr < RG; ++rr)
            if (b0 + rr < a.B)
                a.warp_stats[(size_t)(b0 + rr) * a.warps_total + gw] =
                    make_float4(m[rr], s[rr], bv[rr], __int_as_float(bi[rr]));
    }
    if (!arrive_last(a.ticket + blockIdx.y, gridDim.x)) return;
    for (int rr = 0; rr < RG; ++rr)
        if (s_act[rr]) lm_sample<RG>(a, b0 + rr, rr, s_src[rr], xs, ybuf);
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128) prepare_kernel(const PrepArgs a) {
    __shared__ int ok, code;
    const int b = blockIdx.x;
    // every kernel of the call starts after this one has finished (it is
    // launched without early dependents), so the counters read zero for all
    for (int i = b * blockDim.x + threadIdx.x; i < a.n_counters; i += gridDim.x * blockDim.x) a.counters[i] = 0;
    const int L0 = a.seq_len[b], nn = a.n_new[b];
    if (threadIdx.x == 0) {
        const bool n_ok = nn >= 1 && nn <= a.max_new;
        const bool cap = L0 >= 0 && (long long)L0 + nn + a.K - 1 <= (long long)a.max_pages * a.P;
        ok = n_ok && cap;
        code = !n_ok ? OSPREY_ERR_INVALID_ARG : (!cap ? OSPREY_ERR_CAPACITY : 0);
    }
    __syncthreads();
    if (ok) {
        const int npages = (L0 + nn + a.K - 1 + a.P - 1) / a.P;
        for (int pg = threadIdx.x; pg < npages; pg += blockDim.x) {
            const int page = a.page_table[(size_t)b * a.max_pages + pg];
            if (page < 0 || page >= a.n_pages) { ok = 0; atomicCAS(&code, 0, OSPREY_ERR_CAPACITY); }
        }
        for (int j = threadIdx.x; j < nn; j += blockDim.x) {
            const int t = a.tokens[(size_t)b * a.max_new + j];
            if (t < 0 || t >= a.V) { ok = 0; atomicCAS(&code, 0, OSPREY_ERR_INVALID_ARG); }
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        a.valid[b] = ok;
        a.pos0[b] = L0;
        a.nnew[b] = nn;
        if (ok) a.seq_len[b] = L0 + (a.commit > 0 ? a.commit : nn);
        else set_status(a.status, code);
    }
    const int n_out = a.n_out > 0 ? a.n_out : a.K;
    if (!ok)
        for (int k = threadIdx.x; k < n_out; k += blockDim.x) a.draft_tokens[(size_t)b * n_out + k] = -1;
}

// ---------------------------------------------------------------------------
// host side

// Splits per (row, KV head): about four blocks per SM over the whole grid, at
// most 1024 keys per block, at least 64 keys (one page per warp) per block.
int attn_splits(int R, int Hkv, int max_ctx, int sms) {
    auto cdiv = [](long long x, long long y) { return (int)((x + y - 1) / y); };
    int want = cdiv(4LL * sms, (long long)R * Hkv);
    int by_len = cdiv(max_ctx, 1024);
    int s = want > by_len ? want : by_len;
    int cap = cdiv(max_ctx, 64);
    if (s > cap) s = cap;
    if (s > ATTN_MAX_SPLITS) s = ATTN_MAX_SPLITS;
    return s < 1 ? 1 : s;
}

int attn_split_len(int max_ctx, int n_splits) {
    int len = (max_ctx + n_splits - 1) / n_splits;
    return (len + 15) / 16 * 16;
}

int lm_blocks(int V, int sms) {
    int want = 2 * sms;
    int cap = (V + GW * 16 - 1) / (GW * 16);   // at least ~16 rows per warp range
    return want < cap ? want : (cap < 1 ? 1 : cap);
}

static int gemv_kd(GemvMode mode, const Dims &d) {
    switch (mode) {
    case G_FEAT: return d.feat;
    case G_QKV: return 2 * d.d;
    case G_OPROJ: return d.Hq * d.hd;
    case G_GATEUP: return d.d;
    default: return d.F;
    }
}

int gemv_rg(GemvMode mode, const Dims &d, int R) {
    int rg = 1;
    while (rg < R && rg < 8) rg <<= 1;
    const size_t limit = 200 * 1024;
    while (rg > 1 && (size_t)rg * gemv_kd(mode, d) * 4 > limit) rg >>= 1;
    return rg;
}

size_t gemv_smem(GemvMode mode, const Dims &d, int rg) { return (size_t)rg * gemv_kd(mode, d) * 4; }

template <int MODE>
static cudaError_t launch_gemv_m(const GemvArgs &a, int rg, int sms, cudaStream_t s) {
    const Dims &D = a.dim;
    int n_tasks;
    if (MODE == G_QKV) n_tasks = (D.Hq + 2 * D.Hkv) * D.hd / 2;
    else if (MODE == G_GATEUP) n_tasks = D.F;
    else n_tasks = D.d;
    int blocks = (n_tasks + GW - 1) / GW;
    if (blocks > 4 * sms) blocks = 4 * sms;
    const int groups = (a.R + rg - 1) / rg;
    const size_t smem = gemv_smem((GemvMode)MODE, D, rg);
    dim3 grid(blocks, groups);
    switch (rg) {
    case 1: gemv_kernel<MODE, 1><<<grid, GT, smem, s>>>(a); break;
    case 2: gemv_kernel<MODE, 2><<<grid, GT, smem, s>>>(a); break;
    case 4: gemv_kernel<MODE, 4><<<grid, GT, smem, s>>>(a); break;
    default: gemv_kernel<MODE, 8><<<grid, GT, smem, s>>>(a); break;
    }
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_gemv(GemvMode mode, const GemvArgs &a, int rg, int sms, cudaStream_t s) {
    switch (mode) {
    case G_FEAT: return launch_gemv_m<G_FEAT>(a, rg, sms, s);
    case G_QKV: return launch_gemv_m<G_QKV>(a, rg, sms, s);
    case G_OPROJ: return launch_gemv_m<G_OPROJ>(a, rg, sms, s);
    case G_GATEUP: return launch_gemv_m<G_GATEUP>(a, rg, sms, s);
    default: return launch_gemv_m<G_DOWN>(a, rg, sms, s);
    }
}

template <int HD, int G>
static cudaError_t launch_attn_t(const AttnArgs &a, cudaStream_t s) {
    static std::atomic<int> done[kMaxDevices];   // the ring's dynamic shared memory, opted into once per device
    cudaError_t e = once_per_device(done, [] {
        return cudaFuncSetAttribute(attn_kernel<HD, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    AttnSplit<HD>::RING);
    });
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_splits, a.dim.Hkv, a.R);
    cfg.blockDim = dim3(AT);
    cfg.dynamicSmemBytes = AttnSplit<HD>::RING;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, attn_kernel<HD, G>, a);
}

cudaError_t launch_attn(const AttnArgs &a, cudaStream_t s) {
    const int G = a.dim.Hq / a.dim.Hkv;
    cudaError_t e;
    if (a.dim.hd == 128) {
        switch (G) {
        case 1: e = launch_attn_t<128, 1>(a, s); break;
        case 2: e = launch_attn_t<128, 2>(a, s); break;
        case 4: e = launch_attn_t<128, 4>(a, s); break;
        default: e = launch_attn_t<128, 8>(a, s); break;
        }
    } else {
        switch (G) {
        case 1: e = launch_attn_t<64, 1>(a, s); break;
        case 2: e = launch_attn_t<64, 2>(a, s); break;
        case 4: e = launch_attn_t<64, 4>(a, s); break;
        default: e = launch_attn_t<64, 8>(a, s); break;
        }
    }
    count_launch();
    return e;
}

template <int HD, int G, int CS>
static cudaLaunchConfig_t attn_cluster_cfg(const AttnArgs &a, cudaStream_t s, cudaLaunchAttribute (&attr)[2]) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(CS, a.dim.Hq / G, a.R);
    cfg.blockDim = dim3(AttnCluster<HD, G, CS>::THREADS);
    cfg.dynamicSmemBytes = AttnCluster<HD, G, CS>::RING;
    cfg.stream = s;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cfg;
}

// Whether clusters of CS blocks of this kernel can be resident on the device
// (sets the non-portable size attribute when CS > 8).
template <int HD, int G, int CS>
static bool attn_cluster_ok(const Dims &D) {
    auto k = attn_cluster_kernel<HD, G, CS>;
    if (CS > 8 && cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, AttnCluster<HD, G, CS>::RING) !=
        cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (D.P != 16) return false;   // the page loop takes 16 positions per page
    AttnArgs a{};
    a.dim = D;
    a.R = 1;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = attn_cluster_cfg<HD, G, CS>(a, nullptr, attr);
    cfg.numAttrs = 1;   // the occupancy query takes the cluster shape only
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return n >= 1;
}

template <int HD, int G>
static int attn_cluster_size_t(const Dims &D) {
    if (OSP_ATTN_CS == 16 && attn_cluster_ok<HD, G, 16>(D)) return 16;
    if (attn_cluster_ok<HD, G, 8>(D)) return 8;
    return 0;
}

int attn_cluster_size(const Dims &D) {
    const int G = D.Hq / D.Hkv;
    if (D.hd == 128) {
        switch (G) {
        case 1: return attn_cluster_size_t<128, 1>(D);
        case 2: return attn_cluster_size_t<128, 2>(D);
        case 4: return attn_cluster_size_t<128, 4>(D);
        default: return attn_cluster_size_t<128, 8>(D);
        }
    }
    switch (G) {
    case 1: return attn_cluster_size_t<64, 1>(D);
    case 2: return attn_cluster_size_t<64, 2>(D);
    case 4: return attn_cluster_size_t<64, 4>(D);
    default: return attn_cluster_size_t<64, 8>(D);
    }
}

template <int HD, int G>
static cudaError_t launch_attn_cluster_t(const AttnArgs &a, int cs, cudaStream_t s) {
    cudaLaunchAttribute attr[2];
    if (cs == 16) {
        cudaLaunchConfig_t cfg = attn_cluster_cfg<HD, G, 16>(a, s, attr);
        return cudaLaunchKernelEx(&cfg, attn_cluster_kernel<HD, G, 16>, a);
    }
    cudaLaunchConfig_t cfg = attn_cluster_cfg<HD, G, 8>(a, s, attr);
    return cudaLaunchKernelEx(&cfg, attn_cluster_kernel<HD, G, 8>, a);
}

cudaError_t launch_attn_cluster(const AttnArgs &a, int cs, cudaStream_t s) {
    const int G = a.dim.Hq / a.dim.Hkv;
    cudaError_t e;
    if (a.dim.hd == 128) {
        switch (G) {
        case 1: e = launch_attn_cluster_t<128, 1>(a, cs, s); break;
        case 2: e = launch_attn_cluster_t<128, 2>(a, cs, s); break;
        case 4: e = launch_attn_cluster_t<128, 4>(a, cs, s); break;
        default: e = launch_attn_cluster_t<128, 8>(a, cs, s); break;
        }
    } else {
        switch (G) {
        case 1: e = launch_attn_cluster_t<64, 1>(a, cs, s); break;
        case 2: e = launch_attn_cluster_t<64, 2>(a, cs, s); break;
        case 4: e = launch_attn_cluster_t<64, 4>(a, cs, s); break;
        default: e = launch_attn_cluster_t<64, 8>(a, cs, s); break;
        }
    }
    count_launch();
    return e;
}

cudaError_t launch_lm(const LmArgs &a, int rg, int blocks, cudaStream_t s) {
    const int groups = (a.B + rg - 1) / rg;
    const int range_max = (a.dim.V + a.warps_total - 1) / a.warps_total + 1;
    const size_t smem = (size_t)rg * a.dim.d * 4 + (size_t)range_max * 4;
    dim3 grid(blocks, groups);
    switch (rg) {
    case 1: lm_head_kernel<1><<<grid, GT, smem, s>>>(a); break;
    case 2: lm_head_kernel<2><<<grid, GT, smem, s>>>(a); break;
    case 4: lm_head_kernel<4><<<grid, GT, smem, s>>>(a); break;
    default: lm_head_kernel<8><<<grid, GT, smem, s>>>(a); break;
    }
    count_launch();
    return cudaGetLastError();
}

__global__ void __launch_bounds__(256) keep_hidden_kernel(const float *x, int ext, int K, int step, int max_new,
                                                          int d, const int *valid, const int *nnew, float *hidden) {
    const int b = blockIdx.x;
    const bool ok = valid[b] != 0;   // then 1 <= nnew[b] <= max_new
    const float *src = x + (size_t)(ok ? (ext ? b * max_new + nnew[b] - 1 : b) : 0) * d;
    float *dst = hidden + ((size_t)b * K + step) * d;
    for (int k = threadIdx.x * 4; k < d; k += blockDim.x * 4)   // d is a multiple of 256
        *(float4 *)(dst + k) = ok ? *(const float4 *)(src + k) : make_float4(0.f, 0.f, 0.f, 0.f);
}

cudaError_t launch_keep_hidden(const float *x, bool ext, int B, int K, int step, int max_new, int d,
                               const int *valid, const int *nnew, float *hidden, cudaStream_t s) {
    keep_hidden_kernel<<<B, 256, 0, s>>>(x, ext ? 1 : 0, K, step, max_new, d, valid, nnew, hidden);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_prepare(const PrepArgs &a, cudaStream_t s) {
    prepare_kernel<<<a.B, 128, 0, s>>>(a);
    count_launch();
    return cudaGetLastError();
}

template <int MODE>
static cudaError_t set_gemv_attr() {
    cudaError_t e;
    if ((e = allow_smem(gemv_kernel<MODE, 1>))) return e;
    if ((e = allow_smem(gemv_kernel<MODE, 2>))) return e;
    if ((e = allow_smem(gemv_kernel<MODE, 4>))) return e;
    return allow_smem(gemv_kernel<MODE, 8>);
}

cudaError_t draft_set_attributes() {
    cudaError_t e;
    if ((e = set_gemv_attr<G_FEAT>())) return e;
    if ((e = set_gemv_attr<G_QKV>())) return e;
    if ((e = set_gemv_attr<G_OPROJ>())) return e;
    if ((e = set_gemv_attr<G_GATEUP>())) return e;
    if ((e = set_gemv_attr<G_DOWN>())) return e;
    if ((e = allow_smem(lm_head_kernel<1>))) return e;
    if ((e = allow_smem(lm_head_kernel<2>))) return e;
    if ((e = allow_smem(lm_head_kernel<4>))) return e;
    return allow_smem(lm_head_kernel<8>);
}

// ---------------------------------------------------------------------------
// Fused batch-1 layer: a whole drafter layer of one chain row (Sec. 3.3 Eq. 2-3
// and the transferred block) in one launch, one block per SM.  Block c owns
// pair units [u0, u1) of the expanded QKV rows (rows i and i + hd/2 of a head,
// so the rotation stays in the block), KV head c / n_splits and key range
// c % n_splits of the attention (blocks past Hkv x n_splits skip it), rows
// [o0, o1) of W_o and W_down and SwiGLU units [f0, f1).  Phases, each ending in
// a grid barrier:
//   A  z = RMSNorm(x); the block's q/k/v pairs of W~_qkv [s; z]; RoPE; k, v to
//      the page
//   B  attention partial of the block's key range; the last range of a KV head
//      merges the ranges
//   C  x += W_o attn (own rows)
//   D  n = RMSNorm(x); h = silu(W_g n) * (W_u n) (own units)
//   E  x += W_down h (own rows)
// Shared memory regions:
//   A  QKV pair rows (requested before griddepcontrol.wait), then the gate/up
//      rows (requested when phase A is done), then the down rows (requested
//      when phase D is done)
//   B  W_o rows (requested before griddepcontrol.wait)
//   C  [s; z], then the attention pages, then the activation of C-E
// Values written by other blocks are read through L2 (ld.global.cg), or by
// bulk copies after proxy fences on both sides of the barrier.
constexpr int LY_THREADS = 256;
constexpr int LY_WARPS = LY_THREADS / 32;
constexpr int LY_NSPW = 1;   // attention pages in flight per warp

struct LayerPlan {
    int nu, up, ro, rf;   // pair units (all), per block at most; O/down rows, SwiGLU units per block at most
    size_t a_bytes, b_bytes, c_bytes, smem;
};

static __host__ __device__ size_t ly_round(size_t x) { return (x + 127) / 128 * 128; }

static __host__ __device__ LayerPlan layer_plan(const Dims &D, int grid) {
    LayerPlan p{};
    p.nu = (D.Hq + 2 * D.Hkv) * (D.hd / 2);
    p.up = (p.nu + grid - 1) / grid;
    p.ro = (D.d + grid - 1) / grid;
    p.rf = (D.F + grid - 1) / grid;
    const int Ko = D.Hq * D.hd;
    const size_t qkv = (size_t)2 * p.up * 2 * D.d * 2, gu = (size_t)2 * p.rf * D.d * 2;
    const size_t dn = (size_t)p.ro * D.F * 2;
    size_t a = qkv > gu ? qkv : gu;
    a = a > dn ? a : dn;
    const size_t ring = (size_t)LY_WARPS * LY_NSPW * 2 * 16 * D.hd * 2;
    int act = 2 * D.d > Ko ? 2 * D.d : Ko;
    act = act > D.F ? act : D.F;
    p.a_bytes = ly_round(a);
    p.b_bytes = ly_round((size_t)p.ro * Ko * 2);
    p.c_bytes = ly_round(ring > (size_t)act * 4 ? ring : (size_t)act * 4);
    p.smem = p.a_bytes + p.b_bytes + p.c_bytes;
    return p;
}

// v[0, d) <- RMSNorm(v) * gain, in place, by the whole block.
__device__ __forceinline__ void ly_rmsnorm(float *v, const uint16_t *gain, int d, float eps, float *red) {
    __syncthreads();   // v was written by other threads
    float ss = 0.f;
    for (int i = threadIdx.x; i < d; i += LY_THREADS) ss = fmaf(v[i], v[i], ss);
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < LY_WARPS; ++w) t += red[w];
    const float inv = rsqrtf(t / (float)d + eps);
    for (int i = threadIdx.x; i < d; i += LY_THREADS) v[i] = v[i] * inv * bf_to_f(gain[i]);
    __syncthreads();
}

__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

template <int HD, int G>
__global__ void __launch_bounds__(LY_THREADS, 1) layer_fused_kernel(const LayerArgs a) {
    constexpr int NW = LY_WARPS;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar[4];   // QKV rows, W_o rows, gate/up rows, down rows
    __shared__ __align__(8) uint64_t full[NW][LY_NSPW];
    __shared__ float sm_m[NW][G], sm_l[NW][G];
    __shared__ float sm_acc[NW][G][HD];
    __shared__ float red[NW];
    const Dims &D = a.dim;
    const int d = D.d, F = D.F, Ko = D.Hq * HD, half = HD / 2;
    const int nb = gridDim.x, c = blockIdx.x;
    const LayerPlan p = layer_plan(D, nb);
    uint8_t *regA = smem, *regB = smem + p.a_bytes, *regC = regB + p.b_bytes;
    const int u0 = (int)((long long)p.nu * c / nb), u1 = (int)((long long)p.nu * (c + 1) / nb), nu = u1 - u0;
    const int o0 = (int)((long long)d * c / nb), o1 = (int)((long long)d * (c + 1) / nb), no = o1 - o0;
    const int f0 = (int)((long long)F * c / nb), f1 = (int)((long long)F * (c + 1) / nb), nf = f1 - f0;
    uint16_t *wq_lo = (uint16_t *)regA;                    // [up][2d]: row i of the unit's head
    uint16_t *wq_hi = wq_lo + (size_t)p.up * 2 * d;         // [up][2d]: row i + hd/2
    uint16_t *wg = (uint16_t *)regA;                        // [rf][d]
    uint16_t *wu = wg + (size_t)p.rf * d;                   // [rf][d]
    uint16_t *wd = (uint16_t *)regA;                        // [ro][F]
    uint16_t *wo = (uint16_t *)regB;                        // [ro][Ko]
    float *act = (float *)regC;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int issued = 0;   // thread 0: barriers 0 .. issued-1 have copies requested

    if (threadIdx.x == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bar[i], 1);
        mbar_fence_init();
        // the weights do not depend on earlier kernels: request them now
        const uint32_t row_b = (uint32_t)4 * d;   // one expanded QKV row: 2d bf16
        mbar_arrive_expect_tx(&bar[0], (uint32_t)nu * 2 * row_b);
        for (int u = u0; u < u1;) {   // the units of one head at a time: two row ranges each
            const int h = u / half, i = u - h * half;
            const int n = min(u1 - u, half - i);
            const size_t lo = (size_t)h * HD + i;
            if (OSP_BOUNDS_OK(u - u0 + n <= p.up && lo + half + n <= (size_t)(D.Hq + 2 * D.Hkv) * HD &&
                                  p.smem <= dynamic_smem_bytes(),
                              a.status)) {
                bulk_g2s(wq_lo + (size_t)(u - u0) * 2 * d, a.W_qkv + lo * 2 * d, (uint32_t)n * row_b, &bar[0]);
                bulk_g2s(wq_hi + (size_t)(u - u0) * 2 * d, a.W_qkv + (lo + half) * 2 * d, (uint32_t)n * row_b,
                         &bar[0]);
            }
            u += n;
        }
        const uint32_t bo = (uint32_t)no * Ko * 2;
        mbar_arrive_expect_tx(&bar[1], bo);
        if (bo && OSP_BOUNDS_OK(no <= p.ro && o1 <= d, a.status)) bulk_g2s(wo, a.W_o + (size_t)o0 * Ko, bo, &bar[1]);
        issued = 2;
    }
    pdl_trigger();
    int b = 0, pos = 0;
    const bool live = a.map.row(0, b, pos);   // the row map was written before the chain
    __syncthreads();
    pdl_wait();   // the residual, the context slot and this call's K/V rows come from earlier kernels
    bool ok = true;

    // ---- A. [s; RMSNorm(x) gamma] -> the block's q/k/v pairs, RoPE, K/V rows
    float *u_s = act;   // [2d]
    if (live) {
        for (int i = threadIdx.x * 4; i < d; i += LY_THREADS * 4) {
            *(float4 *)(u_s + i) = __ldcg((const float4 *)(a.s + i));
            *(float4 *)(u_s + d + i) = __ldcg((const float4 *)(a.x + i));
        }
        ly_rmsnorm(u_s + d, a.attn_norm, d, D.eps, red);
    }
    ok = ok && __syncthreads_and(mbar_wait(&bar[0], 0));
    if (ok && live)
        for (int k = warp; k < nu; k += NW) {
            const float y1 = warp_smem_dot(wq_lo + (size_t)k * 2 * d, u_s, 2 * d);
            const float y2 = warp_smem_dot(wq_hi + (size_t)k * 2 * d, u_s, 2 * d);
            if (lane == 0) {
                const int unit = u0 + k, h = unit / half, i = unit - h * half;
                float x1 = y1, x2 = y2;
                if (h < D.Hq + D.Hkv) {   // rotate-half RoPE on q and k
                    float cs, sn;
                    rope_cs2(a.inv_freq[i], pos, cs, sn);
                    x1 = y1 * cs - y2 * sn;
                    x2 = y2 * cs + y1 * sn;
                }
                if (h < D.Hq) {
                    a.q[(size_t)h * HD + i] = x1;
                    a.q[(size_t)h * HD + i + half] = x2;
                } else {
                    const bool is_k = h < D.Hq + D.Hkv;
                    const int kvh = is_k ? h - D.Hq : h - D.Hq - D.Hkv;
                    if (OSP_BOUNDS_OK(pos / D.P < a.max_pages, a.status)) {
                        const int page = a.page_table[(size_t)b * a.max_pages + pos / D.P];
                        uint16_t *dst = (is_k ? a.k_pages : a.v_pages) +
                                        (((size_t)page * D.Hkv + kvh) * D.P + pos % D.P) * HD;
                        dst[i] = f_to_bf(x1);
                        dst[i + half] = f_to_bf(x2);
                    }
                }
            }
        }
    fence_proxy_async_global();   // the K/V rows are read by other blocks' bulk copies
    ok = ok && grid_sync(a.bar_count, a.bar_gen, a.status);   // a block that timed out stops

    // ---- B. attention partial of the block's key range; gate/up rows requested
    fence_proxy_async_global();
    fence_proxy_async_smem();     // regions A and C are refilled by bulk copies
    __syncthreads();
    if (threadIdx.x == 0 && ok) {
        const uint32_t bf = (uint32_t)nf * d * 2;
        mbar_arrive_expect_tx(&bar[2], 2 * bf);
        if (bf && OSP_BOUNDS_OK(nf <= p.rf && f1 <= F, a.status)) {
            bulk_g2s(wg, a.W_gate + (size_t)f0 * d, bf, &bar[2]);
            bulk_g2s(wu, a.W_up + (size_t)f0 * d, bf, &bar[2]);
        }
        issued = 3;
    }
    const int units = D.Hkv * a.n_splits;
    if (ok && live && c < units) {
        const int kvh = c / a.n_splits, split = c - kvh * a.n_splits;
        const int n_keys = pos + 1, pos0 = a.map.pos0[b];
        const int k_begin = split * a.split_len;   // a multiple of the page size
        const int k_end = min(n_keys, k_begin + a.split_len);
        AttnArgs at{};
        at.dim = D;
        at.q = a.q;
        at.k_pages = a.k_pages;
        at.v_pages = a.v_pages;
        at.page_table = a.page_table;
        at.max_pages = a.max_pages;
        at.status = a.status;
        attn_warp_pages<HD, G, NW, LY_NSPW, true>(at, b, 0, kvh, kvh * G, k_begin, k_end, pos0, regC, full, sm_m,
                                                  sm_l, sm_acc);
        __syncthreads();
        for (int idx = threadIdx.x; idx < G * HD; idx += LY_THREADS) {
            const int g = idx / HD, dim = idx - g * HD;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < NW; ++w) M = fmaxf(M, sm_m[w][g]);
            float num = 0.f, den = 0.f;
            if (M != -INFINITY)
#pragma unroll
                for (int w = 0; w < NW; ++w) {
                    const float f = sm_m[w][g] == -INFINITY ? 0.f : __expf(sm_m[w][g] - M);
                    num = fmaf(f, sm_acc[w][g][dim], num);
                    den = fmaf(f, sm_l[w][g], den);
                }
            float *pp = a.attn_part + ((size_t)(kvh * G + g) * a.n_splits + split) * (HD + 2);
            pp[2 + dim] = num;
            if (dim == 0) { pp[0] = M; pp[1] = den; }
        }
        if (arrive_last(a.attn_ticket + kvh, a.n_splits)) {
            // the last key range of this KV head merges the ranges
            for (int idx = threadIdx.x; idx < G * HD; idx += LY_THREADS) {
                const int g = idx / HD, dim = idx - g * HD;
                const float *base = a.attn_part + (size_t)(kvh * G + g) * a.n_splits * (HD + 2);
                float M = -INFINITY;
                for (int sp = 0; sp < a.n_splits; ++sp) M = fmaxf(M, __ldcg(base + (size_t)sp * (HD + 2)));
                float num = 0.f, den = 0.f;
                for (int sp = 0; sp < a.n_splits; ++sp) {
                    const float *pp = base + (size_t)sp * (HD + 2);
                    const float ms = __ldcg(pp);
                    const float f = ms == -INFINITY ? 0.f : __expf(ms - M);
                    num = fmaf(f, __ldcg(pp + 2 + dim), num);
                    den = fmaf(f, __ldcg(pp + 1), den);
                }
                a.attn_out[(size_t)(kvh * G + g) * HD + dim] = num / den;
            }
        }
    }
    ok = ok && grid_sync(a.bar_count, a.bar_gen, a.status);   // a block that timed out stops

    // ---- C. O-proj and residual
    if (ok && live)
        for (int i = threadIdx.x * 4; i < Ko; i += LY_THREADS * 4)
            *(float4 *)(act + i) = __ldcg((const float4 *)(a.attn_out + i));
    __syncthreads();
    ok = ok && __syncthreads_and(mbar_wait(&bar[1], 0));
    if (ok && live)
        for (int j = warp; j < no; j += NW) {
            const float acc = warp_smem_dot(wo + (size_t)j * Ko, act, Ko);
            if (lane == 0) a.x[o0 + j] = __ldcg(a.x + o0 + j) + acc;
        }
    ok = ok && grid_sync(a.bar_count, a.bar_gen, a.status);   // a block that timed out stops

    // ---- D. RMSNorm of the whole residual, gate/up and SwiGLU
    if (ok && live) {
        for (int i = threadIdx.x * 4; i < d; i += LY_THREADS * 4)
            *(float4 *)(act + i) = __ldcg((const float4 *)(a.x + i));
        ly_rmsnorm(act, a.ffn_norm, d, D.eps, red);
    }
    __syncthreads();
    ok = ok && __syncthreads_and(mbar_wait(&bar[2], 0));
    if (ok && live)
        for (int j = warp; j < nf; j += NW) {
            const float g = warp_smem_dot(wg + (size_t)j * d, act, d);
            const float u = warp_smem_dot(wu + (size_t)j * d, act, d);
            if (lane == 0) a.h[f0 + j] = g / (1.f + expf(-g)) * u;
        }
    fence_proxy_async_smem();   // region A takes the down rows next
    __syncthreads();
    if (threadIdx.x == 0 && ok) {
        const uint32_t bd = (uint32_t)no * F * 2;
        mbar_arrive_expect_tx(&bar[3], bd);
        if (bd && OSP_BOUNDS_OK((size_t)bd <= p.a_bytes && o1 <= d, a.status))
            bulk_g2s(wd, a.W_down + (size_t)o0 * F, bd, &bar[3]);
        issued = 4;
    }
    ok = ok && grid_sync(a.bar_count, a.bar_gen, a.status);   // a block that timed out stops

    // ---- E. down and residual
    if (ok && live)
        for (int i = threadIdx.x * 4; i < F; i += LY_THREADS * 4)
            *(float4 *)(act + i) = __ldcg((const float4 *)(a.h + i));
    __syncthreads();
    ok = ok && __syncthreads_and(mbar_wait(&bar[3], 0));
    if (ok && live)
        for (int j = warp; j < no; j += NW) {
            const float acc = warp_smem_dot(wd + (size_t)j * F, act, F);
            if (lane == 0) a.x[o0 + j] = __ldcg(a.x + o0 + j) + acc;
        }
    if (!ok) {
        if (threadIdx.x == 0) {
            set_status(a.status, OSPREY_ERR_TIMEOUT);
            for (int i = 0; i < issued; ++i) mbar_wait(&bar[i], 0, 200000000LL);   // copies land before exit
        }
        __syncthreads();
    }
}

int layer_fused_splits(const Dims &D, int max_ctx, int sms) {
    int ns = sms / D.Hkv;
    const int cap = attn_splits(1, D.Hkv, max_ctx, sms);
    if (ns > cap) ns = cap;
    return ns < 1 ? 1 : ns;
}

template <int HD, int G>
static bool layer_fits(const LayerPlan &p, int sms) {
    int dev = 0, optin = 0;
    cudaFuncAttributes fa{};
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
        cudaFuncGetAttributes(&fa, layer_fused_kernel<HD, G>) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    if (p.smem + fa.sharedSizeBytes > (size_t)optin) return false;
    // the grid barriers need every block resident at once: one per SM
    if (allow_smem(layer_fused_kernel<HD, G>) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return grid_fits_resident(layer_fused_kernel<HD, G>, LY_THREADS, p.smem, sms, sms);
}

bool layer_fused_supported(const Dims &D, int sms) {
    const int G = D.Hq / D.Hkv;
    if ((D.hd != 64 && D.hd != 128) || (G != 1 && G != 2 && G != 4 && G != 8) || D.P != 16) return false;
    if (D.d % 256 || D.F % 256 || (D.Hq * D.hd) % 256 || D.Hkv > sms) return false;
    const LayerPlan p = layer_plan(D, sms);
    // each mbarrier phase counts fewer than 2^20 bytes
    if ((size_t)p.up * 2 * 4 * D.d >= (1u << 20) || (size_t)p.ro * D.Hq * D.hd * 2 >= (1u << 20) ||
        (size_t)2 * p.rf * D.d * 2 >= (1u << 20) || (size_t)p.ro * D.F * 2 >= (1u << 20))
        return false;
#define OSP_LY_FITS(hd_, g_) \
    if (D.hd == hd_ && G == g_) return layer_fits<hd_, g_>(p, sms);
    OSP_LY_FITS(64, 1) OSP_LY_FITS(64, 2) OSP_LY_FITS(64, 4) OSP_LY_FITS(64, 8)
    OSP_LY_FITS(128, 1) OSP_LY_FITS(128, 2) OSP_LY_FITS(128, 4) OSP_LY_FITS(128, 8)
#undef OSP_LY_FITS
    return false;
}

template <int HD, int G>
static cudaError_t launch_layer_t(const LayerArgs &a, int sms, cudaStream_t s) {
    // the shared-memory opt-in and the residency check ran when the context chose
    // this path (layer_fused_supported, with the same grid)
    const LayerPlan p = layer_plan(a.dim, sms);
    cudaError_t e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(sms);
    cfg.blockDim = dim3(LY_THREADS);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, layer_fused_kernel<HD, G>, a);
    count_launch();
    return e;
}

cudaError_t launch_layer_fused(const LayerArgs &a, int sms, cudaStream_t s) {
    const int G = a.dim.Hq / a.dim.Hkv;
    if (a.n_splits < 1 || a.dim.Hkv * a.n_splits > sms || a.split_len % 16) return cudaErrorInvalidValue;
#define OSP_LY_LAUNCH(hd_, g_) \
    if (a.dim.hd == hd_ && G == g_) return launch_layer_t<hd_, g_>(a, sms, s);
    OSP_LY_LAUNCH(64, 1) OSP_LY_LAUNCH(64, 2) OSP_LY_LAUNCH(64, 4) OSP_LY_LAUNCH(64, 8)
    OSP_LY_LAUNCH(128, 1) OSP_LY_LAUNCH(128, 2) OSP_LY_LAUNCH(128, 4) OSP_LY_LAUNCH(128, 8)
#undef OSP_LY_LAUNCH
    return cudaErrorInvalidValue;
}

}  // namespace osp
