// TMA-streamed GEMV for one or two activation rows (the single-stream decode
// regime, HBM-bound).
//
// Block = 8 consumer warps + 1 producer warp.  The weight rows a block owns
// are cut into stages (8-16 KB); the producer streams them with 1-D bulk
// copies (cp.async.bulk) into an 8-slot shared-memory ring, slot w being
// consumed by warp w, with full/empty mbarriers (every wait bounded).  The
// activation rows are staged once in shared memory as float32.  Launches use
// programmatic dependent launch: the producer starts streaming weights before
// the previous kernel has finished; the consumers wait for it
// (griddepcontrol.wait) before they read activations.
//
// Modes (Sec. 3.3 Eq. 1-3 per layer; LM head per chain step):
//   QKV     [q;k;v] = W~_qkv [s; RMSNorm(x)], rotary on q,k; k,v -> pages
//   OPROJ   x += W_o attn              DOWN  x += W_down h
//   GATEUP  h = silu(W_gate n) * (W_up n), n = RMSNorm(x)
//   LM      logits = W_lm RMSNorm(x_L), never written out (unless the caller
//           asks for draft_logits): per-block (max, sum exp, argmax), and per
//           run of stages (at most 32 runs a block: max, sum exp); the last block draws the token
//           by inverse CDF: block -> run -> that run's logits, recomputed from
//           W_lm with the main pass's arithmetic (bitwise equal) -> id.
#include <math.h>

#include "common.cuh"
#include "draft.cuh"
#include "internal.h"
#include "tma.cuh"

namespace osp {

// Tuning knobs (compile-time): ring slots per block, stage bytes for the LM
// head and for the per-layer projections, order in which a block walks its
// stages (0: ascending; 1: ascending from a per-block rotation), blocks per SM.
#ifndef OSP_SG_NST
#define OSP_SG_NST 8
#endif
#ifndef OSP_SG_LM_STAGE
#define OSP_SG_LM_STAGE 8192
#endif
#ifndef OSP_SG_STAGE
#define OSP_SG_STAGE 4096
#endif
#ifndef OSP_SG_ORDER
#define OSP_SG_ORDER 0
#endif
#ifndef OSP_SG_BLOCKS_PER_SM
#define OSP_SG_BLOCKS_PER_SM 2
#endif
#ifndef OSP_SG_GEMV_BPS
#define OSP_SG_GEMV_BPS OSP_SG_BLOCKS_PER_SM   // blocks per SM of the layer GEMVs
#endif
#ifndef OSP_SG_MIN_BLOCKS
#define OSP_SG_MIN_BLOCKS 2   // register budget: this many blocks (of any stream kernel) per SM
#endif
#ifndef OSP_SG_NPROD
#define OSP_SG_NPROD 1   // producer lanes; lane p issues stages p, p + NPROD, ...
#endif
// L2 priority of the weight streams: the LM head is loaded evict-first (it is
// read once per chain step and does not fit in L2); layer weights at normal
// priority.  Evict-last would keep layer weights in L2 across the chain steps
// of a call, but such lines also survive later traffic (a flush of twice the
// L2 size left about a third of them resident), and the layer weights are
// fetched while the previous kernel finishes, off the critical path, anyway.


constexpr int SG_CW = 8;                      // consumer warps
constexpr int SG_THREADS = (SG_CW + 1) * 32;  // + one producer warp
constexpr int SG_NST = OSP_SG_NST;            // ring slots; warp w consumes slots w, w + 8, ... in turn
constexpr int SG_MAXR = 8;                    // weight rows per stage at most
static_assert(SG_NST % SG_CW == 0, "ring slots must be a multiple of the consumer warps");

__device__ __forceinline__ int sg_kd(const StreamArgs &a) {
    const Dims &D = a.dim;
    switch (a.mode) {
    case G_QKV: return 2 * D.d;
    case G_OPROJ: return D.Hq * D.hd;
    case G_GATEUP: return D.d;
    case G_DOWN: return D.F;
    default: return D.d;   // G_LM
    }
}

__device__ __forceinline__ bool sg_pair(int mode) { return mode == G_QKV || mode == G_GATEUP; }

// Dot of one bf16 weight row in shared memory with RG float32 rows: lane l
// takes elements base + 8l .. base + 8l + 7 of every 256-wide chunk, in
// ascending order, then a butterfly sum (the order warp_dot uses on global
// memory, so a recomputed value is bitwise equal).
template <int RG>
__device__ __forceinline__ void smem_dot(const uint16_t *w, const float *xs, int Kd, float (&acc)[RG]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int r = 0; r < RG; ++r) acc[r] = 0.f;
#pragma unroll 4
    for (int base = 0; base < Kd; base += 256) {
        const uint4 wv = *(const uint4 *)(w + base + lane * 8);
        float wf[8];
        unpack8(wv, wf);
#pragma unroll
        for (int r = 0; r < RG; ++r) {
            const float4 x0 = *(const float4 *)(xs + (size_t)r * Kd + base + lane * 8);
            const float4 x1 = *(const float4 *)(xs + (size_t)r * Kd + base + lane * 8 + 4);
            const float xf[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[r] = fmaf(wf[e], xf[e], acc[r]);
        }
    }
#pragma unroll
    for (int r = 0; r < RG; ++r) acc[r] = warp_sum(acc[r]);
}

// NR rows at once (rows past `cnt` skipped): independent accumulators, the
// activation chunk read once for all rows, butterflies interleaved.  Each
// row's value is computed in exactly the order smem_dot / global_dot use.
template <int NR, int RG>
__device__ __forceinline__ void smem_dot_rows(const uint16_t *w, unsigned valid, const float *xs, int Kd,
                                              float (&acc)[NR][RG]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int i = 0; i < NR; ++i)
#pragma unroll
        for (int r = 0; r < RG; ++r) acc[i][r] = 0.f;
#pragma unroll 2
    for (int base = 0; base < Kd; base += 256) {
        uint4 wv[NR];
#pragma unroll
        for (int i = 0; i < NR; ++i)
            wv[i] = ((valid >> i) & 1u) ? *(const uint4 *)(w + (size_t)i * Kd + base + lane * 8)
                                        : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int r = 0; r < RG; ++r) {
            const float4 x0 = *(const float4 *)(xs + (size_t)r * Kd + base + lane * 8);
            const float4 x1 = *(const float4 *)(xs + (size_t)r * Kd + base + lane * 8 + 4);
            const float xf[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int i = 0; i < NR; ++i) {
                float wf[8];
                unpack8(wv[i], wf);
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[i][r] = fmaf(wf[e], xf[e], acc[i][r]);
            }
        }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1)
#pragma unroll
        for (int i = 0; i < NR; ++i)
#pragma unroll
            for (int r = 0; r < RG; ++r) acc[i][r] += __shfl_xor_sync(0xffffffffu, acc[i][r], o);
}

// Same arithmetic reading the row from global memory (LM-head recompute).
template <int RG>
__device__ __forceinline__ void global_dot(const uint16_t *w, const float *xs, int Kd, float (&acc)[RG]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int r = 0; r < RG; ++r) acc[r] = 0.f;
#pragma unroll 4
    for (int base = 0; base < Kd; base += 256) {
        const uint4 wv = ld_stream(w + base + lane * 8);
        float wf[8];
        unpack8(wv, wf);
#pragma unroll
        for (int r = 0; r < RG; ++r) {
            const float4 x0 = *(const float4 *)(xs + (size_t)r * Kd + base + lane * 8);
            const float4 x1 = *(const float4 *)(xs + (size_t)r * Kd + base + lane * 8 + 4);
            const float xf[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[r] = fmaf(wf[e], xf[e], acc[r]);
        }
    }
#pragma unroll
    for (int r = 0; r < RG; ++r) acc[r] = warp_sum(acc[r]);
}

// RMSNorm of a float32 row into shared memory by the consumer threads only.
__device__ __forceinline__ void consumer_rmsnorm(float *dst, const float *x, const uint16_t *gain, int d,
                                                 float eps, float *red) {
    const int nt = SG_CW * 32;
    float ss = 0.f;
    if (x)
        for (int k = threadIdx.x; k < d; k += nt) ss = fmaf(x[k], x[k], ss);
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    named_sync(1, nt);
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < SG_CW; ++w) t += red[w];
        red[32] = rsqrtf(t / (float)d + eps);
    }
    named_sync(1, nt);
    const float inv = red[32];
    for (int k = threadIdx.x; k < d; k += nt) dst[k] = x ? x[k] * inv * bf_to_f(gain[k]) : 0.f;
    named_sync(1, nt);
}

// Register-held variant for d <= SG_PV * 4 * 256: the caller issues the loads
// of x (and of the gain, before griddepcontrol.wait) together, so the
// normalisation costs a single round trip.
constexpr int SG_PV = 4;   // float4 of a d-vector per consumer thread
__device__ __forceinline__ void load_vec4(float4 (&v)[SG_PV], const float *src, int n4) {
#pragma unroll
    for (int k = 0; k < SG_PV; ++k) {
        const int c = threadIdx.x + k * SG_CW * 32;
        v[k] = src && c < n4 ? ((const float4 *)src)[c] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
}
__device__ __forceinline__ void load_gain4(uint2 (&g)[SG_PV], const uint16_t *gain, int n4) {
#pragma unroll
    for (int k = 0; k < SG_PV; ++k) {
        const int c = threadIdx.x + k * SG_CW * 32;
        g[k] = c < n4 ? ((const uint2 *)gain)[c] : make_uint2(0u, 0u);
    }
}
__device__ __forceinline__ void store_vec4(float *dst, const float4 (&v)[SG_PV], int n4) {
#pragma unroll
    for (int k = 0; k < SG_PV; ++k) {
        const int c = threadIdx.x + k * SG_CW * 32;
        if (c < n4) ((float4 *)dst)[c] = v[k];
    }
}
__device__ __forceinline__ void consumer_rmsnorm_regs(float *dst, const float4 (&x)[SG_PV], const uint2 (&g)[SG_PV],
                                                      int d, float eps, float *red) {
    const int nt = SG_CW * 32;
    float ss = 0.f;
#pragma unroll
    for (int k = 0; k < SG_PV; ++k) ss += x[k].x * x[k].x + x[k].y * x[k].y + x[k].z * x[k].z + x[k].w * x[k].w;
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    named_sync(1, nt);
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < SG_CW; ++w) t += red[w];
    const float inv = rsqrtf(t / (float)d + eps);
#pragma unroll
    for (int k = 0; k < SG_PV; ++k) {
        const int c = threadIdx.x + k * nt;
        if (c < d / 4)
            ((float4 *)dst)[c] = make_float4(x[k].x * inv * bf_lo(g[k].x), x[k].y * inv * bf_hi(g[k].x),
                                             x[k].z * inv * bf_lo(g[k].y), x[k].w * inv * bf_hi(g[k].y));
    }
    named_sync(1, nt);
}

__device__ __forceinline__ void consumer_copy(float *dst, const float *src, int n) {
    for (int c = threadIdx.x; c < n / 4; c += SG_CW * 32)
        ((float4 *)dst)[c] = src ? ((const float4 *)src)[c] : make_float4(0.f, 0.f, 0.f, 0.f);
}


struct StageGeom {
    int i0, cnt;                  // first item, items in this stage
    const uint16_t *src0, *src1;  // segment sources (src1: pair modes)
    uint32_t seg_bytes;           // bytes of one segment
};

__device__ __forceinline__ StageGeom stage_geom(const StreamArgs &a, int st, int Kd) {
    StageGeom g;
    g.i0 = st * a.items;
    g.cnt = min(a.items, a.n_items - g.i0);
    g.seg_bytes = (uint32_t)g.cnt * Kd * 2;
    if (a.mode == G_QKV) {
        const int half = a.dim.hd / 2;
        const int h = g.i0 / half, i = g.i0 % half;
        g.src0 = a.W + ((size_t)h * a.dim.hd + i) * Kd;
        g.src1 = a.W + ((size_t)h * a.dim.hd + half + i) * Kd;
    } else if (a.mode == G_GATEUP) {
        g.src0 = a.W + (size_t)g.i0 * Kd;
        g.src1 = a.W2 + (size_t)g.i0 * Kd;
    } else {
        g.src0 = a.W + (size_t)g.i0 * Kd;
        g.src1 = nullptr;
    }
    return g;
}

// ---------------------------------------------------------------------------
// Ordered inverse-CDF pick over n weighted entries (ids in ascending order):
// the smallest i with target < C_i, C the inclusive cumulative weight.  Each
// thread holds at most PER consecutive weights (w[]), loaded once.  Returns i
// (or, if rounding left target past the last sum, the last entry with weight)
// and the cumulative weight before it.  *total receives the sum of all weights
// (as the scan computed it).
// target_or_u: the target itself, or (scale_by_total) a uniform u whose target
// is u times the total this scan computes.
template <int PER>
__device__ int cdf_pick_regs(const float (&w)[PER], int e0, int n, float target_or_u, bool scale_by_total,
                             float *before, float *total, float *sh) {
    __shared__ int s_pick, s_last;
    __shared__ float s_before;
    float mine = 0.f;
#pragma unroll
    for (int k = 0; k < PER; ++k) mine += w[k];
    float tot;
    const float ex = block_excl_scan(mine, sh, &tot);
    const float target = scale_by_total ? target_or_u * tot : target_or_u;
    if (threadIdx.x == 0) { s_pick = 0x7fffffff; s_last = -1; }
    __syncthreads();
    float run = ex, bfound = 0.f, blast = 0.f;
    int found = 0x7fffffff, last = -1;
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        const int e = e0 + k;
        const float c = w[k];
        if (e < n && c > 0.f) { last = e; blast = run; }
        if (e < n && found == 0x7fffffff && c > 0.f && target < run + c) { found = e; bfound = run; }
        run += c;
    }
    if (found != 0x7fffffff) atomicMin(&s_pick, found);
    if (last >= 0) atomicMax(&s_last, last);
    __syncthreads();
    const int chosen = s_pick != 0x7fffffff ? s_pick : (s_last >= 0 ? s_last : 0);
    if (s_pick != 0x7fffffff && found == chosen) s_before = bfound;
    if (s_pick == 0x7fffffff && last == chosen) s_before = blast;
    if (s_pick == 0x7fffffff && s_last < 0 && threadIdx.x == 0) s_before = 0.f;
    __syncthreads();
    *before = s_before;
    *total = tot;
    __syncthreads();
    return chosen;
}

constexpr int SG_PICK_PER = 2;    // block entries per thread in the first pick (blocks <= 2 x 288)
constexpr int SG_LM_MAXLOC = 1024;   // stages per block at most (per-stage statistics in shared memory)
constexpr int SG_RUN_IDS = 32;    // ids of one run at most (stages per run x items)


// Inverse CDF over one weight per lane (in lane order) at `target`: the first
// lane whose cumulative weight passes it (the last lane with weight when
// rounding leaves the target past the total); *before = the weight before it.
__device__ __forceinline__ int warp_cdf_pick(float c, bool valid, float target, float *before) {
    const int lane = threadIdx.x & 31;
    const float incl = warp_incl_scan(c);
    const unsigned hit = __ballot_sync(0xffffffffu, valid && c > 0.f && target < incl);
    const unsigned pos = __ballot_sync(0xffffffffu, valid && c > 0.f);
    const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
    *before = __shfl_sync(0xffffffffu, incl - c, l);
    return l;
}

// Logits of ids [lo, hi) (at most SG_RUN_IDS) into z, each computed as
// global_dot computes it (so bitwise equal to the main pass): warp w takes ids
// lo + w, lo + w + SG_CW + 1, ...; the loads of all its ids for a 1024-wide
// stretch of the row are issued before any is used.
__device__ __forceinline__ void lm_recompute_run(const StreamArgs &a, int lo, int hi, const float *x, float *z) {
    constexpr int NW = SG_THREADS / 32, PW = (SG_RUN_IDS + NW - 1) / NW;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, d = a.dim.d;
    float acc[PW];
#pragma unroll
    for (int i = 0; i < PW; ++i) acc[i] = 0.f;
    for (int b0 = 0; b0 < d; b0 += 1024) {
        uint4 wv[PW][4];
#pragma unroll
        for (int i = 0; i < PW; ++i) {
            const int id = lo + warp + i * NW;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int base = b0 + 256 * c;
                wv[i][c] = id < hi && base < d ? ld_stream(a.W + (size_t)id * d + base + lane * 8) : make_uint4(0, 0, 0, 0);
            }
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int base = b0 + 256 * c;
            if (base >= d) break;
            const float4 x0 = *(const float4 *)(x + base + lane * 8);
            const float4 x1 = *(const float4 *)(x + base + lane * 8 + 4);
            const float xf[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int i = 0; i < PW; ++i) {
                float wf[8];
                unpack8(wv[i][c], wf);
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[i] = fmaf(wf[e], xf[e], acc[i]);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < PW; ++i) {
        const float v = warp_sum(acc[i]);
        const int id = lo + warp + i * NW;
        if (lane == 0 && id < hi) z[id - lo] = v;
    }
}

template <int RG>
__device__ void lm_sample_stream(const StreamArgs &a, int b, int rr, int src_row, const float *xs, float *ybuf,
                                 int nblk) {
    __shared__ MS shm[SG_CW + 1];
    __shared__ AM sha[SG_CW + 1];
    __shared__ float sh_scan[33];
    __shared__ float s_e, s_pickb;
    __shared__ int s_pick[2];
    __shared__ float s_run[SG_RUN_IDS];
    const Dims &D = a.dim;
    const bool greedy = a.temperature == 0.f;
    const float invT = greedy ? 1.f : 1.f / a.temperature;
    const int t = threadIdx.x;
    const float4 *cst = a.cta_stats + (size_t)b * nblk;
    const float u = greedy ? 0.f : a.u_draft[(size_t)b * a.K + a.step];

    // level 1: one load per block entry; (max, sum) and argmax over all blocks
    const int e0 = t * SG_PICK_PER;
    float4 v[SG_PICK_PER];
    MS ms{-INFINITY, 0.f};
    AM am{-INFINITY, 0x7fffffff};
#pragma unroll
    for (int k = 0; k < SG_PICK_PER; ++k) {
        v[k] = e0 + k < nblk ? __ldcg(cst + e0 + k) : make_float4(-INFINITY, 0.f, -INFINITY, __int_as_float(0x7fffffff));
        ms = ms_combine(ms, MS{v[k].x, v[k].y});
        am = am_combine(am, AM{v[k].z, __float_as_int(v[k].w)});
    }
    const float M = block_ms(ms, shm).m;
    int token;
    float qx, S;
    if (greedy) {
        token = block_am(am, sha).i;
        qx = 1.f;
        // S relative to M of the raw logits, for the stats output
        float c[SG_PICK_PER];
#pragma unroll
        for (int k = 0; k < SG_PICK_PER; ++k) c[k] = v[k].x == -INFINITY ? 0.f : v[k].y * __expf(v[k].x - M);
        float mine = 0.f;
#pragma unroll
        for (int k = 0; k < SG_PICK_PER; ++k) mine += c[k];
        block_excl_scan(mine, sh_scan, &S);
    } else {
        float c1[SG_PICK_PER];
#pragma unroll
        for (int k = 0; k < SG_PICK_PER; ++k) c1[k] = v[k].x == -INFINITY ? 0.f : v[k].y * __expf(v[k].x - M);
        // the target u * S needs the total: the pick's own scan provides it
        float before1;
        const int blk = cdf_pick_regs<SG_PICK_PER>(c1, e0, nblk, u, true, &before1, &S, sh_scan);
        const float target = u * S;
        // level 2: the chosen block's runs of a.run stages (at most 32: one warp)
        const float2 *sp = a.sup + ((size_t)b * nblk + blk) * a.nsup;
        const int st0 = (int)((long long)a.n_stages * blk / nblk);
        const int st1 = (int)((long long)a.n_stages * (blk + 1) / nblk);
        const int nrun = (st1 - st0 + a.run - 1) / a.run;
        const int warp = t >> 5, lane = t & 31;
        if (warp == 0) {
            const float2 e = lane < nrun ? __ldcg(sp + lane) : make_float2(-INFINITY, 0.f);
            const float c = e.x == -INFINITY ? 0.f : e.y * __expf(e.x - M);
            float bef;
            const int run = warp_cdf_pick(c, lane < nrun, target - before1, &bef);
            if (lane == 0) { s_pick[0] = run; s_pickb = bef; }
        }
        __syncthreads();
        const int run = s_pick[0];
        const float before2 = s_pickb;
        // level 3: that run's logits, recomputed with the main pass's arithmetic
        const int lo = (st0 + run * a.run) * a.items;
        const int hi = min(D.V, min(st1, st0 + (run + 1) * a.run) * a.items);
        lm_recompute_run(a, lo, hi, xs + (size_t)rr * D.d, s_run);
        __syncthreads();
        if (warp == 0) {
            const float c = lane < hi - lo ? __expf(s_run[lane] * invT - M) : 0.f;
            float bef;
            const int id = warp_cdf_pick(c, lane < hi - lo, target - before1 - before2, &bef);
            if (lane == id) s_e = c;
            if (lane == 0) s_pick[1] = id;
        }
        __syncthreads();
        const int idx = s_pick[1];
        token = lo + idx;
        qx = s_e / S;
    }
    if (t == 0) {
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
        const uint16_t *e = a.embed + (size_t)token * D.d;
        for (int k = 4 * t; k < D.d; k += 4 * blockDim.x) {   // d is a multiple of 256
            const float4 xv = __ldcg((const float4 *)(xl + k));
            const uint2 ev = *(const uint2 *)(e + k);
            *(float4 *)(a.s_chain + (size_t)b * D.d + k) = xv;
            *(float4 *)(a.x_chain + (size_t)b * D.d + k) =
                make_float4(bf_lo(ev.x), bf_hi(ev.x), bf_lo(ev.y), bf_hi(ev.y));
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// NRS = weight rows per stage (single modes: items; pair modes: 2 * items, the
// second segment at row `items` of the slot).
template <int MODE, int RG, int NRS>
__global__ void __launch_bounds__(SG_THREADS, OSP_SG_MIN_BLOCKS) stream_kernel(const StreamArgs a) {
    constexpr bool PAIR = MODE == G_QKV || MODE == G_GATEUP;
    constexpr int NI = PAIR ? NRS / 2 : NRS;   // items per full stage
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t full[SG_NST], empty[SG_NST];
    __shared__ float red[33];
    __shared__ int s_b[RG], s_pos[RG], s_act[RG], s_src[RG], s_abort;
    __shared__ float4 s_wstats[SG_CW][RG];
    __shared__ float2 s_stst[MODE == G_LM ? SG_LM_MAXLOC : 1][RG];   // LM: (max, sum exp) of each local stage
    const Dims &D = a.dim;
    const int Kd = sg_kd(a);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t *ring = smem;
    float *xs = (float *)(smem + (size_t)SG_NST * a.stage_bytes);
    float *ybuf = xs + (size_t)RG * Kd;
    const int nblk = gridDim.x;
    const int st0 = (int)((long long)a.n_stages * blockIdx.x / nblk);
    const int st1 = (int)((long long)a.n_stages * (blockIdx.x + 1) / nblk);
    const int nloc = st1 - st0;
    const int r0 = blockIdx.y * RG;
    const int rot = OSP_SG_ORDER == 1 && nloc > 0 ? (int)((blockIdx.x * 2654435761u) % (unsigned)nloc) : 0;
    auto stage_of = [&](int j) { return st0 + (j + rot >= nloc ? j + rot - nloc : j + rot); };

    if (threadIdx.x == 0) {
        for (int i = 0; i < SG_NST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        s_abort = 0;
        mbar_fence_init();
    }
    __syncthreads();
    pdl_trigger();

    if (warp == SG_CW) {
        // ---- producer: weights do not depend on the previous kernel
        if (lane < OSP_SG_NPROD) {
            const uint64_t pol = policy_evict_first();
            int issued = 0;
            for (int j = lane; j < nloc; j += OSP_SG_NPROD) {
                const int slot = j % SG_NST;
                if (j >= SG_NST && !mbar_wait(&empty[slot], ((j / SG_NST) - 1) & 1)) {
                    set_status(a.status, OSPREY_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                    break;
                }
                if (s_abort) break;
                const StageGeom g = stage_geom(a, stage_of(j), Kd);
                uint8_t *dst = ring + (size_t)slot * a.stage_bytes;
                mbar_arrive_expect_tx(&full[slot], PAIR ? 2 * g.seg_bytes : g.seg_bytes);
                if (MODE == G_LM) {
                    bulk_g2s_hint(dst, g.src0, g.seg_bytes, &full[slot], pol);
                } else {
                    bulk_g2s(dst, g.src0, g.seg_bytes, &full[slot]);
                    if (PAIR) bulk_g2s(dst + (size_t)NI * Kd * 2, g.src1, g.seg_bytes, &full[slot]);
                }
                issued = j + 1;
            }
            if (s_abort) {
                // let every copy this lane issued land before the block can exit
                for (int j = lane; j < issued; j += OSP_SG_NPROD)
                    if (j + SG_NST >= issued) mbar_wait(&full[j % SG_NST], (j / SG_NST) & 1, 200000000LL);
            }
        }
    } else {
        // ---- consumers
        // the row map and the norm gain were written before the chain started:
        // read them while the previous kernel finishes
        if (threadIdx.x < RG) {
            int b = 0, pos = 0, src = 0;
            bool act;
            if (MODE == G_LM) {
                b = r0 + threadIdx.x;
                act = b < a.B && a.map.valid[b];
                src = act ? (a.src_is_ext ? b * a.max_new + a.map.nnew[b] - 1 : b) : 0;
            } else {
                const int r = r0 + threadIdx.x;
                act = r < a.R && a.map.row(r, b, pos);
                src = r;
            }
            s_b[threadIdx.x] = b;
            s_pos[threadIdx.x] = pos;
            s_act[threadIdx.x] = act;
            s_src[threadIdx.x] = src;
        }
        constexpr bool NORM = MODE == G_QKV || MODE == G_GATEUP || MODE == G_LM;
        const bool regs = D.d <= SG_PV * 4 * SG_CW * 32;
        uint2 gv[SG_PV];
        if (NORM && regs) load_gain4(gv, a.gain, D.d / 4);
        named_sync(1, SG_CW * 32);
        pdl_wait();
        for (int rr = 0; rr < RG; ++rr) {
            const bool act = s_act[rr];
            const int r = s_src[rr];
            float *row = xs + (size_t)rr * Kd;
            if (NORM && regs) {
                // every load of the row issued at once: x (and the context slot for qkv)
                const float *xsrc = MODE == G_LM ? a.x_in : a.x;
                float4 xv[SG_PV], sv[SG_PV];
                load_vec4(xv, act ? xsrc + (size_t)r * D.d : nullptr, D.d / 4);
                if (MODE == G_QKV) load_vec4(sv, act ? a.s + (size_t)r * D.d : nullptr, D.d / 4);
                consumer_rmsnorm_regs(MODE == G_QKV ? row + D.d : row, xv, gv, D.d, D.eps, red);
                if (MODE == G_QKV) store_vec4(row, sv, D.d / 4);
            } else if (MODE == G_QKV) {
                consumer_copy(row, act ? a.s + (size_t)r * D.d : nullptr, D.d);
                consumer_rmsnorm(row + D.d, act ? a.x + (size_t)r * D.d : nullptr, a.gain, D.d, D.eps, red);
            } else if (MODE == G_GATEUP) {
                consumer_rmsnorm(row, act ? a.x + (size_t)r * D.d : nullptr, a.gain, D.d, D.eps, red);
            } else if (MODE == G_LM) {
                consumer_rmsnorm(row, act ? a.x_in + (size_t)r * D.d : nullptr, a.gain, D.d, D.eps, red);
            } else {
                consumer_copy(row, act ? a.xin + (size_t)r * Kd : nullptr, Kd);
            }
        }
        named_sync(1, SG_CW * 32);

        const float invT = (MODE == G_LM && a.temperature > 0.f) ? 1.f / a.temperature : 1.f;
        float wm[RG], ws[RG], wbv[RG];
        int wbi[RG];
#pragma unroll
        for (int rr = 0; rr < RG; ++rr) { wm[rr] = -INFINITY; ws[rr] = 0.f; wbv[rr] = -INFINITY; wbi[rr] = 0x7fffffff; }

        for (int j = warp; j < nloc; j += SG_CW) {
            const int slot = j % SG_NST;
            if (!mbar_wait(&full[slot], (j / SG_NST) & 1)) {
                set_status(a.status, OSPREY_ERR_TIMEOUT);
                atomicExch(&s_abort, 1);
                mbar_wait(&full[slot], (j / SG_NST) & 1, 200000000LL);   // bounded drain
                break;
            }
            const int st = stage_of(j);
            const StageGeom g = stage_geom(a, st, Kd);
            const uint16_t *rows = (const uint16_t *)(ring + (size_t)slot * a.stage_bytes);
            unsigned valid = (1u << g.cnt) - 1u;
            if (PAIR) valid |= valid << NI;
            float acc[NRS][RG];
            smem_dot_rows<NRS, RG>(rows, valid, xs, Kd, acc);
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);   // the slot can be refilled

            if (PAIR) {
#pragma unroll
                for (int i = 0; i < NI; ++i) {
                    if (i >= g.cnt) break;
                    const int item = g.i0 + i;
#pragma unroll
                    for (int rr = 0; rr < RG; ++rr) {
                        if (lane != rr || !s_act[rr]) continue;
                        const int r = r0 + rr;
                        if (MODE == G_GATEUP) {
                            const float gv = acc[i][rr], uv = acc[i + NI][rr];
                            a.out[(size_t)r * D.F + item] = gv / (1.f + expf(-gv)) * uv;
                        } else {
                            const int half = D.hd / 2;
                            const int h = item / half, ii = item % half;
                            const int b = s_b[rr], pos = s_pos[rr];
                            float x1 = acc[i][rr], x2 = acc[i + NI][rr];
                            if (h < D.Hq + D.Hkv) {
                                float c, sn;
                                rope_cs2(a.inv_freq[ii], pos, c, sn);
                                const float y1 = x1 * c - x2 * sn, y2 = x2 * c + x1 * sn;
                                x1 = y1;
                                x2 = y2;
                            }
                            if (h < D.Hq) {
                                float *q = a.q + (size_t)r * D.Hq * D.hd + (size_t)h * D.hd;
                                q[ii] = x1;
                                q[ii + half] = x2;
                            } else {
                                const bool is_k = h < D.Hq + D.Hkv;
                                const int kvh = is_k ? h - D.Hq : h - D.Hq - D.Hkv;
                                const int page = a.page_table[(size_t)b * a.max_pages + pos / D.P];
                                uint16_t *dst = (is_k ? a.k_pages : a.v_pages) +
                                                (((size_t)page * D.Hkv + kvh) * D.P + pos % D.P) * D.hd;
                                dst[ii] = f_to_bf(x1);
                                dst[ii + half] = f_to_bf(x2);
                            }
                        }
                    }
                }
            } else if (MODE == G_LM) {
                float tm[RG], ts[RG], tbv[RG];
                int tbi[RG];
#pragma unroll
                for (int rr = 0; rr < RG; ++rr) { tm[rr] = -INFINITY; ts[rr] = 0.f; tbv[rr] = -INFINITY; tbi[rr] = 0x7fffffff; }
#pragma unroll
                for (int i = 0; i < NI; ++i) {
                    if (i >= g.cnt) break;
                    const int item = g.i0 + i;
#pragma unroll
                    for (int rr = 0; rr < RG; ++rr) {
                        const float z = acc[i][rr];
                        if (lane == 0 && s_act[rr] && a.logits)
                            a.logits[((size_t)(r0 + rr) * a.K + a.step) * D.V + item] = z;
                        const float y = z * invT;
                        if (y > tm[rr]) { ts[rr] = ts[rr] * __expf(tm[rr] - y) + 1.f; tm[rr] = y; }
                        else ts[rr] += __expf(y - tm[rr]);
                        if (z > tbv[rr]) { tbv[rr] = z; tbi[rr] = item; }
                    }
                }
#pragma unroll
                for (int rr = 0; rr < RG; ++rr) {
                    if (lane == 0) s_stst[st - st0][rr] = make_float2(tm[rr], ts[rr]);
                    const MS c = ms_combine(MS{wm[rr], ws[rr]}, MS{tm[rr], ts[rr]});
                    wm[rr] = c.m;
                    ws[rr] = c.s;
                    const AM m2 = am_combine(AM{wbv[rr], wbi[rr]}, AM{tbv[rr], tbi[rr]});
                    wbv[rr] = m2.v;
                    wbi[rr] = m2.i;
                }
            } else {
#pragma unroll
                for (int i = 0; i < NI; ++i) {
                    if (i >= g.cnt) break;
#pragma unroll
                    for (int rr = 0; rr < RG; ++rr)
                        if (lane == rr && s_act[rr]) a.x[(size_t)s_src[rr] * D.d + g.i0 + i] += acc[i][rr];
                }
            }
        }
        if (MODE == G_LM && lane == 0)
#pragma unroll
            for (int rr = 0; rr < RG; ++rr) s_wstats[warp][rr] = make_float4(wm[rr], ws[rr], wbv[rr], __int_as_float(wbi[rr]));
    }
    if (MODE != G_LM) return;
    __syncthreads();
    if (warp > 0) {   // the block's runs of a.run stages
        const int nrun = (nloc + a.run - 1) / a.run;
        for (int e = threadIdx.x - 32; e < nrun * RG; e += SG_THREADS - 32) {
            const int k = e / RG, rr = e - k * RG;
            MS m{-INFINITY, 0.f};
            for (int q = k * a.run; q < min(nloc, (k + 1) * a.run); ++q)
                m = ms_combine(m, MS{s_stst[q][rr].x, s_stst[q][rr].y});
            if (r0 + rr < a.B) a.sup[((size_t)(r0 + rr) * nblk + blockIdx.x) * a.nsup + k] = make_float2(m.m, m.s);
        }
    }
    if (warp == 0) {
#pragma unroll
        for (int rr = 0; rr < RG; ++rr) {
            float4 v = lane < SG_CW ? s_wstats[lane][rr] : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
            if (lane >= SG_CW) v.w = __int_as_float(0x7fffffff);
            const MS m = warp_ms(MS{v.x, v.y});
            const AM am = warp_am(AM{v.z, __float_as_int(v.w)});
            if (lane == 0 && r0 + rr < a.B)
                a.cta_stats[(size_t)(r0 + rr) * nblk + blockIdx.x] = make_float4(m.m, m.s, am.v, __int_as_float(am.i));
        }
    }
    if (!arrive_last(a.ticket + blockIdx.y, nblk)) return;
    for (int rr = 0; rr < RG; ++rr)
        if (s_act[rr]) lm_sample_stream<RG>(a, r0 + rr, rr, s_src[rr], xs, ybuf, nblk);
}

// ---------------------------------------------------------------------------
// host side

static int pow2_floor(int x) {
    int p = 1;
    while (p * 2 <= x) p *= 2;
    return p;
}

static int host_kd(GemvMode mode, const Dims &D) {
    switch (mode) {
    case G_QKV: return 2 * D.d;
    case G_OPROJ: return D.Hq * D.hd;
    case G_GATEUP: return D.d;
    case G_DOWN: return D.F;
    default: return D.d;
    }
}

StreamPlan stream_plan(GemvMode mode, const Dims &D, int sms) {
    StreamPlan p{};
    const int Kd = host_kd(mode, D);
    const int row_bytes = Kd * 2;
    const int target = mode == G_LM ? OSP_SG_LM_STAGE : OSP_SG_STAGE;   // bytes per stage
    // the LM head rounds to the nearest whole row (d 2560: two 5 KB rows, not one)
    int rows = mode == G_LM ? (target + row_bytes / 2) / row_bytes : target / row_bytes;
    const bool pair = mode == G_QKV || mode == G_GATEUP;
    rows = rows < (pair ? 2 : 1) ? (pair ? 2 : 1) : rows;
    rows = rows > SG_MAXR ? SG_MAXR : (!pair && rows >= 6 ? 6 : pow2_floor(rows));
    if (pair) {
        int sp = rows / 2;
        if (mode == G_QKV && sp > D.hd / 2) sp = D.hd / 2;
        p.items = sp;
        p.n_items = mode == G_QKV ? (D.Hq + 2 * D.Hkv) * D.hd / 2 : D.F;
        p.stage_bytes = 2 * sp * row_bytes;
    } else {
        p.items = rows;
        p.n_items = mode == G_LM ? D.V : D.d;
        p.stage_bytes = rows * row_bytes;
    }
    p.n_stages = (p.n_items + p.items - 1) / p.items;
    const int bps = mode == G_LM ? OSP_SG_BLOCKS_PER_SM : OSP_SG_GEMV_BPS;
    p.blocks = p.n_stages < sms * bps ? p.n_stages : sms * bps;
    // LM head runs: the fewest stages per run that leave at most 32 runs a block
    const int maxloc = (p.n_stages + p.blocks - 1) / p.blocks;
    p.run = (maxloc + 31) / 32;
    p.nsup = (maxloc + p.run - 1) / p.run;
    p.smem = (size_t)SG_NST * p.stage_bytes;
    return p;
}

static size_t stream_smem(GemvMode mode, const Dims &D, int rg, const StreamPlan &p) {
    const int range = mode == G_LM ? p.items : 0;
    return (size_t)SG_NST * p.stage_bytes + (size_t)rg * host_kd(mode, D) * 4 + (size_t)(range + 4) * 4;
}

bool stream_supported(GemvMode mode, const Dims &D, int rg, int sms) {
    if (rg < 1 || rg > 2 || mode == G_FEAT) return false;
    const StreamPlan p = stream_plan(mode, D, sms);
    if (stream_smem(mode, D, rg, p) > 200 * 1024) return false;
    // the LM head's sampler: blocks at most SG_PICK_PER per thread; a block's
    // stages within its statistics array; a run's ids within the recompute buffer
    // (the plan keeps the runs of a block at most 32)
    if (mode == G_LM) {
        const int maxloc = (p.n_stages + p.blocks - 1) / p.blocks;
        if (p.blocks > SG_PICK_PER * SG_THREADS || maxloc > SG_LM_MAXLOC ||
            p.run * p.items > SG_RUN_IDS)
            return false;
    }
    return true;
}

template <int MODE, int RG, int NRS>
static cudaError_t launch_stream_t(const StreamArgs &a, int groups, int blocks, size_t smem, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks, groups);
    cfg.blockDim = dim3(SG_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, stream_kernel<MODE, RG, NRS>, a);
    count_launch();
    return e;
}

template <int MODE, int RG>
static cudaError_t launch_stream_nrs(const StreamArgs &a, int nrs, int groups, int blocks, size_t smem,
                                     cudaStream_t s) {
    switch (nrs) {
    case 1: return (MODE == G_QKV || MODE == G_GATEUP) ? cudaErrorInvalidValue
                                                       : launch_stream_t<MODE, RG, 1>(a, groups, blocks, smem, s);
    case 2: return launch_stream_t<MODE, RG, 2>(a, groups, blocks, smem, s);
    case 4: return launch_stream_t<MODE, RG, 4>(a, groups, blocks, smem, s);
    case 6: return (MODE == G_QKV || MODE == G_GATEUP) ? cudaErrorInvalidValue
                                                       : launch_stream_t<MODE, RG, 6>(a, groups, blocks, smem, s);
    case 8: return launch_stream_t<MODE, RG, 8>(a, groups, blocks, smem, s);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_stream(GemvMode mode, const StreamArgs &a, int rg, cudaStream_t s) {
    const int rows = mode == G_LM ? a.B : a.R;
    const int groups = (rows + rg - 1) / rg;
    StreamPlan p{a.items, a.n_items, a.n_stages, a.stage_bytes, a.blocks, 0, 0};
    const size_t smem = stream_smem(mode, a.dim, rg, p);
    const int blocks = a.n_stages < a.blocks ? a.n_stages : a.blocks;
    const bool pair = mode == G_QKV || mode == G_GATEUP;
    const int nrs = pair ? 2 * a.items : a.items;
#define OSP_STREAM_CASE(M)                                                                          \
    case M:                                                                                         \
        return rg == 1 ? launch_stream_nrs<M, 1>(a, nrs, groups, blocks, smem, s)                   \
                       : launch_stream_nrs<M, 2>(a, nrs, groups, blocks, smem, s);
    switch (mode) {
        OSP_STREAM_CASE(G_QKV)
        OSP_STREAM_CASE(G_OPROJ)
        OSP_STREAM_CASE(G_GATEUP)
        OSP_STREAM_CASE(G_DOWN)
        OSP_STREAM_CASE(G_LM)
    default: return cudaErrorInvalidValue;
    }
#undef OSP_STREAM_CASE
}

template <typename F>
static cudaError_t allow_smem_s(F *kernel) {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    cudaFuncAttributes fa{};
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, kernel);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
    return e;
}

template <int MODE, int RG>
static cudaError_t attr_all() {
    cudaError_t e;
    if (!(MODE == G_QKV || MODE == G_GATEUP)) {
        if ((e = allow_smem_s(stream_kernel<MODE, RG, 1>)) != cudaSuccess) return e;
        if ((e = allow_smem_s(stream_kernel<MODE, RG, 6>)) != cudaSuccess) return e;
    }
    if ((e = allow_smem_s(stream_kernel<MODE, RG, 2>)) != cudaSuccess) return e;
    if ((e = allow_smem_s(stream_kernel<MODE, RG, 4>)) != cudaSuccess) return e;
    return allow_smem_s(stream_kernel<MODE, RG, 8>);
}

cudaError_t stream_set_attributes() {
    cudaError_t e;
#define OSP_ATTR(M)                                                   \
    if ((e = attr_all<M, 1>()) != cudaSuccess) return e;             \
    if ((e = attr_all<M, 2>()) != cudaSuccess) return e;
    OSP_ATTR(G_QKV)
    OSP_ATTR(G_OPROJ)
    OSP_ATTR(G_GATEUP)
    OSP_ATTR(G_DOWN)
    OSP_ATTR(G_LM)
#undef OSP_ATTR
    return cudaSuccess;
}

}  // namespace osp
