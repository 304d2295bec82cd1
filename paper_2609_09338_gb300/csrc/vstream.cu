// Streamed speculative-sampling verification (Sec. 3.1) for 16-byte-aligned
// logits: persistent blocks (8 consumer warps + 1 producer warp, three per SM)
// pull 4 KB chunks of the target row (and of the draft row, for rows i < K)
// through an 8-slot shared-memory ring with 1-D bulk copies (TMA): the copies
// of the other warps' tiles stay in flight while a warp works on its own, 24
// slots per SM in all (three blocks fit the SM's registers and shared memory;
// two blocks of 12 slots kept fewer warps resident and were slower).  The
// fence and atomic that publish a result happen after the slot is freed, once
// per run of tiles.
//
// vs_stats:  a tile is (sequence b, row i, chunk c).  The owning warp reduces
//   it to (max, sum exp) of logits/T for p and q (argmax in greedy mode) and
//   writes one partial.  Per run of tiles of one row a warp adds the run's
//   length to the row's counter; the warp that completes a row reduces its
//   partials to a row summary (all loads in flight at once), then counts the
//   row for its sequence; the warp that completes a sequence reads the K+1
//   row summaries (one load per lane), evaluates p_i(x_i) and q_i(x_i) and
//   decides the first rejection with a ballot.  The serial tail is thus three
//   dependent round trips, whatever V and K.
// vs_sample: a tile is (sequence b, chunk c) of the decision row r only.  The
//   warp sums the draw weights max(0, p_r - q_r) (p_K for the bonus) and p_r;
//   the warp that completes the sequence's count walks the chunk sums in id
//   order, loads the chosen chunk (two halves of loads in flight) and walks its
//   8 segments, then its lanes, then one lane's elements (inverse CDF at
//   u_sample[r]).
// Both kernels are launched as programmatic dependents: barrier set-up overlaps
// the previous kernel's tail, and every global read follows griddepcontrol.wait.
#include <math.h>

#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

namespace osp {

#ifndef OSP_VS_BPS
#define OSP_VS_BPS 3   // resident blocks per SM (grid = OSP_VS_BPS x SMs at most)
#endif

#ifndef OSP_VS_NST
#define OSP_VS_NST 8   // ring slots per block: 3 x 8 x 8 KB of the SM's shared memory
#endif
#ifndef OSP_VS_EARLY
#define OSP_VS_EARLY 0   // 1: a consumer copies both rows of its tile to registers and frees the slot first
#endif
#ifndef OSP_VS_ROWB
#define OSP_VS_ROWB 4096   // bytes of one row chunk (the workspace holds 4 KB float32 chunks at least)
#endif

constexpr int VS_CW = 8;
constexpr int VS_THREADS = (VS_CW + 1) * 32;
constexpr int VS_NST = OSP_VS_NST;
constexpr int VS_ROWB = OSP_VS_ROWB;       // bytes of one row chunk
static_assert(VS_ROWB % 4096 == 0, "row chunks are whole multiples of 4 KB");
// Slot s serves tiles s, s + NST, s + 2 NST, ... and tile j belongs to warp
// j % CW, so consecutive uses of a slot can belong to different warps.  A wait
// on a phase parity is exact only while the barrier is at most one phase
// behind: a warp reaching use u of a slot first waits for use u - 1 to be freed
// (vs_wait_slot).  That wait is itself exact because use u - 2 belongs to the
// same warp, which has freed it: 2 NST must be a multiple of CW.
static_assert((2 * VS_NST) % VS_CW == 0, "ring slots: 2 x slots must be a multiple of the consumer warps");
constexpr int VS_SLOT = 2 * VS_ROWB;       // target chunk + draft chunk
constexpr int VS_NV = VS_ROWB / 16 / 32;   // 16-byte vectors per lane per row chunk (8)

// 2^x on the special-function unit (PTX ex2.approx, flush-to-zero)
__device__ __forceinline__ float vs_ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
constexpr float VS_LOG2E = 1.4426950408889634f;

// Consumer wait for tile j of a block: the slot's previous use (another warp's
// tile) freed, then tile j's copy complete.  False when a bounded wait ran out.
__device__ __forceinline__ bool vs_wait_slot(uint64_t *full, uint64_t *empty, int j) {
    const int slot = j % VS_NST, use = j / VS_NST;
    if (use > 0 && !mbar_wait(&empty[slot], (use - 1) & 1)) return false;
    return mbar_wait(&full[slot], use & 1);
}

// Position of tile t = (row * nch + c) with row = b * rows_per_seq + i, advanced
// incrementally: the 64-bit divisions run once per launch and once per row,
// not once per tile.
struct VsCur {
    long long row;
    int b, i, c;
    __device__ __forceinline__ void set_row(int rows_per_seq) {
        b = (int)(row / rows_per_seq);
        i = (int)(row - (long long)b * rows_per_seq);
    }
    __device__ __forceinline__ void init(long long t, int nch, int rows_per_seq) {
        row = t / nch;
        c = (int)(t - row * nch);
        set_row(rows_per_seq);
    }
    __device__ __forceinline__ void step(int n, int nch, int rows_per_seq) {
        c += n;
        if (c < nch) return;
        do {
            c -= nch;
            ++row;
        } while (c >= nch);
        set_row(rows_per_seq);
    }
};

template <typename T> struct VsT;
template <> struct VsT<float> {
    static constexpr int EL = VS_ROWB / 4;   // elements per chunk
    static constexpr int VW = 4;             // elements per 16-byte vector
    static constexpr uint32_t NEG = 0xff800000u;   // -inf
    __device__ static void unpack(const uint4 v, float (&f)[VW]) {
        f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
    }
    __device__ static float vmax(const uint4 (&r)[VS_NV]) {
        float m[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int k = 0; k < VS_NV; ++k) {
            m[0] = fmaxf(m[0], __uint_as_float(r[k].x)); m[1] = fmaxf(m[1], __uint_as_float(r[k].y));
            m[2] = fmaxf(m[2], __uint_as_float(r[k].z)); m[3] = fmaxf(m[3], __uint_as_float(r[k].w));
        }
        return fmaxf(fmaxf(m[0], m[1]), fmaxf(m[2], m[3]));
    }
};
template <> struct VsT<uint16_t> {
    static constexpr int EL = VS_ROWB / 2;
    static constexpr int VW = 8;
    static constexpr uint32_t NEG = 0xff80ff80u;   // two bf16 -inf
    __device__ static void unpack(const uint4 v, float (&f)[VW]) { unpack8(v, f); }
    __device__ static uint32_t max2(uint32_t a, uint32_t b) {
        uint32_t d;
        asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
        return d;
    }
    // max of the packed pairs, widened once at the end
    __device__ static float vmax(const uint4 (&r)[VS_NV]) {
        uint32_t m[4] = {r[0].x, r[0].y, r[0].z, r[0].w};
#pragma unroll
        for (int k = 1; k < VS_NV; ++k) {
            m[0] = max2(m[0], r[k].x); m[1] = max2(m[1], r[k].y);
            m[2] = max2(m[2], r[k].z); m[3] = max2(m[3], r[k].w);
        }
        const uint32_t w = max2(max2(m[0], m[1]), max2(m[2], m[3]));
        return fmaxf(bf_lo(w), bf_hi(w));
    }
};

// Overwrite the lane's vectors at or past element nel with -inf (nel is a
// multiple of the vector width, so a vector is wholly in or wholly out).
template <typename T>
__device__ __forceinline__ void vs_mask(uint4 (&r)[VS_NV], int lane, int nel) {
    using L = VsT<T>;
#pragma unroll
    for (int k = 0; k < VS_NV; ++k)
        if ((lane + 32 * k) * L::VW >= nel) r[k] = make_uint4(L::NEG, L::NEG, L::NEG, L::NEG);
}

// Sum over the lane's vectors of 2^(x*c - mc) = exp((x - m) / T) with c =
// log2(e)/T and mc = m*c.
template <typename T>
__device__ __forceinline__ float vs_sum_exp(const uint4 (&r)[VS_NV], float c, float mc) {
    using L = VsT<T>;
    float s0 = 0.f, s1 = 0.f;
#pragma unroll
    for (int k = 0; k < VS_NV; ++k) {
        float f[L::VW];
        L::unpack(r[k], f);
#pragma unroll
        for (int e = 0; e < L::VW; e += 2) {
            s0 += vs_ex2(fmaf(f[e], c, -mc));
            s1 += vs_ex2(fmaf(f[e + 1], c, -mc));
        }
    }
    return s0 + s1;
}

__device__ __forceinline__ float vs_logit(const void *base, int dtype, size_t i) {
    return dtype == OSPREY_F32 ? __ldg((const float *)base + i) : bf_to_f(__ldg((const uint16_t *)base + i));
}

// Copy one row chunk (lane's 8 vectors, interleaved by 32 lanes) from the ring.
__device__ __forceinline__ void vs_stage(const uint8_t *chunk, int lane, uint4 (&r)[VS_NV]) {
#pragma unroll
    for (int k = 0; k < VS_NV; ++k) r[k] = ((const uint4 *)chunk)[lane + 32 * k];
}

// ---------------------------------------------------------------------------
// Branch-free warp combine of (max, sum exp) pairs: the warp maximum first,
// then each lane's sum rescaled once to it.  An empty lane has m = -inf, s = 0.
__device__ __forceinline__ MS vs_warp_ms(float m, float s) {
    const float M = warp_max(m);
    const float r = m == -INFINITY ? 0.f : s * vs_ex2((m - M) * VS_LOG2E);
    return MS{M, warp_sum(r)};
}

// The warp that completes row (b, i): reduce the row's nch tile partials to one
// summary (greedy: the argmax, lowest id on ties).  A lane's loads (8 at a
// time) are all issued before any is used.
template <bool GREEDY>
__device__ void vs_row_reduce(const VerifyArgs &a, size_t row) {
    constexpr int CPL = 8;
    const int lane = threadIdx.x & 31, nch = a.nch3;
    const float4 *tp = (const float4 *)a.tpart + row * nch;
    float4 out;
    if (GREEDY) {
        AM am{-INFINITY, 0x7fffffff};
        for (int c0 = 0; c0 < nch; c0 += 32 * CPL) {
            float4 v[CPL];
#pragma unroll
            for (int k = 0; k < CPL; ++k) {
                const int c = c0 + lane + 32 * k;
                v[k] = c < nch ? __ldcg(tp + c) : make_float4(-INFINITY, __int_as_float(0x7fffffff), 0.f, 0.f);
            }
#pragma unroll
            for (int k = 0; k < CPL; ++k) am = am_combine(am, AM{v[k].x, __float_as_int(v[k].y)});
        }
        am = warp_am(am);
        out = make_float4(am.v, __int_as_float(am.i), 0.f, 0.f);
    } else {
        float mp = -INFINITY, sp = 0.f, mq = -INFINITY, sq = 0.f;
        for (int c0 = 0; c0 < nch; c0 += 32 * CPL) {
            float4 v[CPL];
#pragma unroll
            for (int k = 0; k < CPL; ++k) {
                const int c = c0 + lane + 32 * k;
                v[k] = c < nch ? __ldcg(tp + c) : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
            }
            float np = mp, nq = mq;
#pragma unroll
            for (int k = 0; k < CPL; ++k) { np = fmaxf(np, v[k].x); nq = fmaxf(nq, v[k].z); }
            sp = mp == -INFINITY ? 0.f : sp * vs_ex2((mp - np) * VS_LOG2E);
            sq = mq == -INFINITY ? 0.f : sq * vs_ex2((mq - nq) * VS_LOG2E);
#pragma unroll
            for (int k = 0; k < CPL; ++k) {
                sp += v[k].x == -INFINITY ? 0.f : v[k].y * vs_ex2((v[k].x - np) * VS_LOG2E);
                sq += v[k].z == -INFINITY ? 0.f : v[k].w * vs_ex2((v[k].z - nq) * VS_LOG2E);
            }
            mp = np;
            mq = nq;
        }
        const MS p = vs_warp_ms(mp, sp), q = vs_warp_ms(mq, sq);
        out = make_float4(p.m, p.s, q.m, q.s);
    }
    if (lane == 0) ((float4 *)a.rowstat)[row] = out;
}

// The warp that completes sequence b: lane i holds row i's summary; accept
// while u_i < p_i(x_i) / q_i(x_i) (greedy: while argmax p_i == x_i).
template <bool GREEDY>
__device__ void vs_decide(const VerifyArgs &a, int b) {
    const int lane = threadIdx.x & 31;
    const int K = a.K, V = a.V;
    const int xi = lane < K ? __ldg(a.tokens + (size_t)b * K + lane) : 0;
    const bool ok = __all_sync(0xffffffffu, lane >= K || (xi >= 0 && xi < V));
    // everything below but the summaries is independent of the reduction: load it together
    float zpx = 0.f, zqx = 0.f, ua = 0.f;
    if (!GREEDY && ok && lane < K) {
        zpx = vs_logit(a.target, a.dtype, ((size_t)b * (K + 1) + lane) * V + xi);
        zqx = vs_logit(a.draft, a.dtype, ((size_t)b * K + lane) * V + xi);
        ua = __ldg(a.u_accept + (size_t)b * K + lane);
    }
    const float4 rs = lane <= K ? __ldcg((const float4 *)a.rowstat + (size_t)b * (K + 1) + lane)
                                : make_float4(0.f, 1.f, 0.f, 1.f);
    const float rMp = rs.x, rSp = rs.y, rMq = rs.z, rSq = rs.w;
    const int ram = __float_as_int(rs.y);
    int32_t *out = a.out_tokens + (size_t)b * (K + 1);
    uint8_t *fl = a.flags + (size_t)b * (K + 1);
    Decision *dec = (Decision *)a.dec + b;
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
        accept = lane < K && ram == xi;
    } else if (lane < K) {
        const float invT = 1.f / a.temperature;
        const float px = expf(zpx * invT - rMp) / rSp;
        const float qx = expf(zqx * invT - rMq) / rSq;
        if (a.probs) {
            a.probs[((size_t)b * K + lane) * 2 + 0] = px;
            a.probs[((size_t)b * K + lane) * 2 + 1] = qx;
        }
        accept = ua < px / qx;
    }
    const unsigned rej = ~__ballot_sync(0xffffffffu, accept) & ((1u << K) - 1u);
    const int r = rej ? __ffs(rej) - 1 : K;
    const int am_r = __shfl_sync(0xffffffffu, ram, r);
    const float Mp = __shfl_sync(0xffffffffu, rMp, r), Sp = __shfl_sync(0xffffffffu, rSp, r);
    const float Mq = __shfl_sync(0xffffffffu, rMq, r), Sq = __shfl_sync(0xffffffffu, rSq, r);
    if (lane < r) out[lane] = xi;
    else if (lane == r) out[lane] = GREEDY ? am_r : -1;   // sampled: written by vs_sample
    else if (lane <= K) out[lane] = -1;
    if (lane == 0) {
        a.n_accepted[b] = r;
        dec->r = r;
        dec->Mp = Mp;
        dec->Sp = Sp;
        dec->Mq = r < K ? Mq : 0.f;
        dec->Sq = r < K ? Sq : 1.f;
    }
}

// Adds a run of `pend` finished tiles to sequence b's counter; true in every
// lane for the warp that completes the count (which resets it to zero).
__device__ __forceinline__ bool vs_arrive(int *counter, int pend, int total) {
    int last = 0;
    if ((threadIdx.x & 31) == 0) {
        __threadfence();
        last = atomicAdd(counter, pend) + pend == total;
        if (last) {
            atomicExch(counter, 0);
            __threadfence();
        }
    }
    return __shfl_sync(0xffffffffu, last, 0);
}

// A warp finished `pend` tiles of row `row`: count them; the warp completing
// the row summarises it, and the one completing the sequence decides.
template <bool GREEDY>
__device__ __forceinline__ void vs_row_done(const VerifyArgs &a, size_t row, int pend) {
    if (!vs_arrive(a.trow + row, pend, a.nch3)) return;
    vs_row_reduce<GREEDY>(a, row);
    const int b = (int)(row / (a.K + 1));
    if (vs_arrive(a.ticket1 + b, 1, a.K + 1)) vs_decide<GREEDY>(a, b);
}

template <typename T, bool GREEDY>
__global__ void __launch_bounds__(VS_THREADS, OSP_VS_BPS) vs_stats(const VerifyArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t full[VS_NST], empty[VS_NST];
    __shared__ int s_abort;
    using L = VsT<T>;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = a.K, V = a.V, nch = a.nch3;
    const long long NT = (long long)a.B * (K + 1) * nch;
    const long long t0 = NT * blockIdx.x / gridDim.x, t1 = NT * (blockIdx.x + 1) / gridDim.x;
    const int n = (int)(t1 - t0);
    if (threadIdx.x == 0) {
        for (int i = 0; i < VS_NST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        s_abort = 0;
        mbar_fence_init();
    }
    __syncthreads();
    pdl_trigger();
    pdl_wait();
    if (warp == VS_CW) {
        if (lane == 0) {
            const uint64_t pol = policy_evict_first();
            int issued = 0;
            VsCur cur;
            cur.init(t0, nch, K + 1);
            for (int j = 0; j < n; ++j, cur.step(1, nch, K + 1)) {
                const int slot = j % VS_NST;
                if (j >= VS_NST && !mbar_wait(&empty[slot], ((j / VS_NST) - 1) & 1)) {
                    set_status(a.status, OSPREY_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                    break;
                }
                const int b = cur.b, i = cur.i, c = cur.c;
                const int nel = min(L::EL, V - c * L::EL);
                uint8_t *dst = smem + (size_t)slot * VS_SLOT;
                issued = j + 1;
                if (nel <= 0) {   // never issue a copy outside the row
                    set_status(a.status, OSPREY_ERR_INVALID_ARG);
                    mbar_arrive_expect_tx(&full[slot], 0);
                    continue;
                }
                const uint32_t bytes = (uint32_t)nel * sizeof(T);
                const bool has_q = !GREEDY && i < K;
                mbar_arrive_expect_tx(&full[slot], has_q ? 2 * bytes : bytes);
                bulk_g2s_hint(dst, (const T *)a.target + ((size_t)b * (K + 1) + i) * V + (size_t)c * L::EL, bytes,
                              &full[slot], pol);
                if (has_q)
                    bulk_g2s_hint(dst + VS_ROWB, (const T *)a.draft + ((size_t)b * K + i) * V + (size_t)c * L::EL,
                                  bytes, &full[slot], pol);
            }
            if (s_abort)
                for (int j = max(0, issued - VS_NST); j < issued; ++j)
                    mbar_wait(&full[j % VS_NST], (j / VS_NST) & 1, 200000000LL);
        }
        return;
    }
    const float invT = GREEDY ? 1.f : 1.f / a.temperature;
    const float cexp = invT * VS_LOG2E;
    long long cur_row = -1;
    int pend = 0;
    bool aborted = false;
    VsCur cur;
    cur.init(t0 + warp, nch, K + 1);
    for (int j = warp; j < n; j += VS_CW, cur.step(VS_CW, nch, K + 1)) {
        const int i = cur.i, c = cur.c;
        const long long row = cur.row;
        if (row != cur_row) {
            if (pend) vs_row_done<GREEDY>(a, (size_t)cur_row, pend);
            cur_row = row;
            pend = 0;
        }
        const int slot = j % VS_NST;
        if (!vs_wait_slot(full, empty, j)) {
            set_status(a.status, OSPREY_ERR_TIMEOUT);
            atomicExch(&s_abort, 1);
            mbar_wait(&full[slot], (j / VS_NST) & 1, 200000000LL);
            aborted = true;
            break;
        }
        const int nel = min(L::EL, V - c * L::EL);
        const bool whole = nel == L::EL;
        const bool has_q = !GREEDY && i < K;
        const uint8_t *chunk = smem + (size_t)slot * VS_SLOT;
        // one row at a time through registers; the slot is freed after both
        float4 part;
        uint4 rv[VS_NV];
        vs_stage(chunk, lane, rv);
        if (!whole) vs_mask<T>(rv, lane, nel);
        if (GREEDY) {
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
            AM am{-INFINITY, 0x7fffffff};
#pragma unroll
            for (int k = 0; k < VS_NV; ++k) {
                float f[L::VW];
                L::unpack(rv[k], f);
#pragma unroll
                for (int e = 0; e < L::VW; ++e)
                    if (f[e] > am.v) am = AM{f[e], c * L::EL + (lane + 32 * k) * L::VW + e};
            }
            am = warp_am(am);
            part = make_float4(am.v, __int_as_float(am.i), 0.f, 0.f);
        } else if (OSP_VS_EARLY) {
            // both rows to registers, the slot freed, then the sums
            uint4 rq[VS_NV];
            if (has_q) {
                vs_stage(chunk + VS_ROWB, lane, rq);
                if (!whole) vs_mask<T>(rq, lane, nel);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
            const float xp = L::vmax(rv);
            const float sp = xp == -INFINITY ? 0.f : vs_sum_exp<T>(rv, cexp, xp * cexp);
            float xq = -INFINITY, sq = 0.f;
            if (has_q) {
                xq = L::vmax(rq);
                sq = xq == -INFINITY ? 0.f : vs_sum_exp<T>(rq, cexp, xq * cexp);
            }
            const MS p = vs_warp_ms(xp * invT, sp);
            const MS q = has_q ? vs_warp_ms(xq * invT, sq) : MS{-INFINITY, 0.f};
            part = make_float4(p.m, p.s, q.m, q.s);
        } else {
            // maxima of the raw logits (order is kept by the positive 1/T), then
            // sums of exp((z - max) / T)
            const float xp = L::vmax(rv);
            const float sp = xp == -INFINITY ? 0.f : vs_sum_exp<T>(rv, cexp, xp * cexp);
            float xq = -INFINITY, sq = 0.f;
            if (has_q) {
                vs_stage(chunk + VS_ROWB, lane, rv);
                if (!whole) vs_mask<T>(rv, lane, nel);
                xq = L::vmax(rv);
                sq = xq == -INFINITY ? 0.f : vs_sum_exp<T>(rv, cexp, xq * cexp);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
            const MS p = vs_warp_ms(xp * invT, sp);
            const MS q = has_q ? vs_warp_ms(xq * invT, sq) : MS{-INFINITY, 0.f};
            part = make_float4(p.m, p.s, q.m, q.s);
        }
        if (lane == 0) ((float4 *)a.tpart)[t0 + j] = part;
        ++pend;
    }
    if (!aborted && pend) vs_row_done<GREEDY>(a, (size_t)cur_row, pend);
}

// ---------------------------------------------------------------------------
// Normalisers of the decision row in exp2 form: p(z) = 2^(z c - Mp log2 e) / Sp.
struct VsNorm {
    float c, mcp, mcq, isp, isq;
};
__device__ __forceinline__ VsNorm vs_norm(const Decision &d, float temperature) {
    return VsNorm{VS_LOG2E / temperature, d.Mp * VS_LOG2E, d.Mq * VS_LOG2E, 1.f / d.Sp, 1.f / d.Sq};
}
// p and the draw weight (max(0, p - q) on a rejection, p for the bonus draw),
// computed the same way by the tile sums and by the final walk.
__device__ __forceinline__ float vs_pw(float zp, float zq, const VsNorm &n, bool residual, float &p) {
    p = vs_ex2(fmaf(zp, n.c, -n.mcp)) * n.isp;
    return residual ? fmaxf(0.f, p - vs_ex2(fmaf(zq, n.c, -n.mcq)) * n.isq) : p;
}
__device__ __forceinline__ float vs_weight(float zp, float zq, const VsNorm &n, bool residual, bool use_p) {
    float p;
    const float w = vs_pw(zp, zq, n, residual, p);
    return use_p ? p : w;
}

// The sampling warp of sequence b (inverse CDF at t = u_sample[r] * S over
// ascending ids): pick the chunk by the chunk sums, then load the chunk once
// and walk its 8 segments (segment k = the k-th vector of every lane, 32 x VW
// consecutive ids), then the lanes of the chosen segment, then one lane's VW
// elements.  Two dependent loads in all.
template <typename T>
__device__ void vs_pick(const VerifyArgs &a, int b, const Decision &d) {
    using L = VsT<T>;
    constexpr int CPL = 8;   // chunk sums a lane holds per round (256 chunks a round)
    const int lane = threadIdx.x & 31;
    const int K = a.K, V = a.V, nch = a.nch3, r = d.r;
    const bool residual = r < K;
    const VsNorm nrm = vs_norm(d, a.temperature);
    const float2 *ts = (const float2 *)a.tsum + (size_t)b * nch;
    const float u = __ldg(a.u_sample + (size_t)b * (K + 1) + r);
    // totals of both weight kinds
    float tw = 0.f, tp = 0.f;
    for (int c0 = 0; c0 < nch; c0 += 32 * CPL) {
        float2 s[CPL];
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = c0 + lane * CPL + k;
            s[k] = c < nch ? __ldcg(ts + c) : make_float2(0.f, 0.f);
        }
#pragma unroll
        for (int k = 0; k < CPL; ++k) { tw += s[k].x; tp += s[k].y; }
    }
    tw = warp_sum(tw);
    tp = warp_sum(tp);
    const bool fallback = !(tw > 0.f) || !isfinite(tw);
    const float S = fallback ? tp : tw;
    const float t = u * S;
    // chunk walk in id order: lane l of a round owns chunks [c0 + l*CPL, c0 + (l+1)*CPL)
    float run = 0.f, before = 0.f;
    int chunk = -1, last_pos = 0;
    for (int c0 = 0; c0 < nch && chunk < 0; c0 += 32 * CPL) {
        float v[CPL], mine = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = c0 + lane * CPL + k;
            v[k] = c < nch ? (fallback ? __ldcg(&ts[c].y) : __ldcg(&ts[c].x)) : 0.f;
            mine += v[k];
        }
        const float incl = warp_incl_scan(mine);
        float cum = run + incl - mine;
        int hit = -1, lastp = -1;
        float hit_before = 0.f;
#pragma unroll
        for (int k = 0; k < CPL; ++k) {
            const int c = c0 + lane * CPL + k;
            if (c < nch && v[k] > 0.f) lastp = c;
            if (hit < 0 && c < nch && t < cum + v[k]) { hit = c; hit_before = cum; }
            cum += v[k];
        }
        const unsigned lp = __ballot_sync(0xffffffffu, lastp >= 0);
        if (lp) last_pos = __shfl_sync(0xffffffffu, lastp, 31 - __clz(lp));
        const unsigned h = __ballot_sync(0xffffffffu, hit >= 0);
        if (h) {
            const int l = __ffs(h) - 1;
            chunk = __shfl_sync(0xffffffffu, hit, l);
            before = __shfl_sync(0xffffffffu, hit_before, l);
        }
        run = __shfl_sync(0xffffffffu, run + incl, 31);
    }
    int flag = fallback ? 8 : 0;
    if (chunk < 0) {   // u*S past the last cumulative sum after rounding
        chunk = last_pos;
        flag |= 16;
        float bsum = 0.f;
        for (int c = lane; c < chunk; c += 32) bsum += fallback ? __ldcg(&ts[c].y) : __ldcg(&ts[c].x);
        before = warp_sum(bsum);
    }
    // the chosen chunk, once: lane l holds vectors l + 32k, k < 8
    const size_t rowp = ((size_t)b * (K + 1) + r) * V + (size_t)chunk * L::EL;
    const size_t rowq = ((size_t)b * K + r) * V + (size_t)chunk * L::EL;
    const uint4 *gp = (const uint4 *)((const T *)a.target + rowp);
    const uint4 *gq = (const uint4 *)((const T *)a.draft + rowq);
    const int nel = min(L::EL, V - chunk * L::EL);   // a multiple of VW (rows are 16-byte multiples)
    // in two halves, so that the loads in flight stay in registers next to the
    // walk's state (the kernel keeps two blocks per SM)
    float seg[VS_NV];
#pragma unroll
    for (int h = 0; h < VS_NV; h += VS_NV / 2) {
        uint4 vp[VS_NV / 2], vq[VS_NV / 2];
#pragma unroll
        for (int k = 0; k < VS_NV / 2; ++k) {
            const bool in = (lane + 32 * (h + k)) * L::VW < nel;
            vp[k] = in ? __ldg(gp + lane + 32 * (h + k)) : make_uint4(0, 0, 0, 0);
            vq[k] = in && residual ? __ldg(gq + lane + 32 * (h + k)) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int k = 0; k < VS_NV / 2; ++k) {
            float f[L::VW], g[L::VW];
            L::unpack(vp[k], f);
            L::unpack(vq[k], g);
            float w = 0.f;
            if ((lane + 32 * (h + k)) * L::VW < nel) {
#pragma unroll
                for (int e = 0; e < L::VW; ++e) w += vs_weight(f[e], g[e], nrm, residual, fallback);
            }
            seg[h + k] = w;
        }
    }
    // segment walk (every lane holds every segment's total)
    int sk = -1, last_seg = -1;
    float segbefore = before, acc = before;
#pragma unroll
    for (int k = 0; k < VS_NV; ++k) {
        const float tot = warp_sum(seg[k]);
        if (tot > 0.f) last_seg = k;
        if (sk < 0 && t < acc + tot) { sk = k; segbefore = acc; }
        acc += tot;
    }
    if (sk < 0) {   // past the chunk's total after rounding: its last segment with mass
        flag |= 16;
        sk = last_seg < 0 ? 0 : last_seg;
        segbefore = before;
#pragma unroll
        for (int k = 0; k < VS_NV; ++k)
            if (k < sk) segbefore += warp_sum(seg[k]);
    }
    // lane walk inside segment sk
    float mine = 0.f;
#pragma unroll
    for (int k = 0; k < VS_NV; ++k)
        if (k == sk) mine = seg[k];
    const float incl = warp_incl_scan(mine);
    const unsigned hit = __ballot_sync(0xffffffffu, mine > 0.f && t < segbefore + incl);
    const unsigned pos = __ballot_sync(0xffffffffu, mine > 0.f);
    int hl;
    if (hit) {
        hl = __ffs(hit) - 1;
    } else {
        hl = pos ? 31 - __clz(pos) : 0;
        flag |= 16;
    }
    const float lane_before = __shfl_sync(0xffffffffu, segbefore + incl - mine, hl);
    // element walk inside lane hl's vector (re-read, an L1 hit)
    int tok = 0;
    if (lane == hl) {
        const int vi = hl + 32 * sk;
        float f[L::VW], g[L::VW];
        L::unpack(__ldg(gp + vi), f);
        if (residual) L::unpack(__ldg(gq + vi), g);
        float cum = lane_before;
        int found = -1, lastp = 0;
#pragma unroll
        for (int e = 0; e < L::VW; ++e) {
            const float w = vs_weight(f[e], residual ? g[e] : 0.f, nrm, residual, fallback);
            cum += w;
            if (w > 0.f) lastp = e;
            if (found < 0 && w > 0.f && t < cum) found = e;
        }
        if (found < 0) {
            found = lastp;
            flag |= 16;
        }
        tok = vi * L::VW + found;
        a.out_tokens[(size_t)b * (K + 1) + r] = chunk * L::EL + tok;
        a.flags[(size_t)b * (K + 1) + r] = (uint8_t)flag;
    }
}

template <typename T>
__global__ void __launch_bounds__(VS_THREADS, OSP_VS_BPS) vs_sample(const VerifyArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t full[VS_NST], empty[VS_NST];
    __shared__ int s_abort;
    using L = VsT<T>;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = a.K, V = a.V, nch = a.nch3;
    const long long NT = (long long)a.B * nch;
    const long long t0 = NT * blockIdx.x / gridDim.x, t1 = NT * (blockIdx.x + 1) / gridDim.x;
    const int n = (int)(t1 - t0);
    const Decision *decs = (const Decision *)a.dec;
    if (threadIdx.x == 0) {
        for (int i = 0; i < VS_NST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        s_abort = 0;
        mbar_fence_init();
    }
    __syncthreads();
    pdl_trigger();
    pdl_wait();
    if (warp == VS_CW) {
        if (lane == 0) {
            const uint64_t pol = policy_evict_first();
            int issued = 0, rb = -1, r = -1;
            VsCur cur;
            cur.init(t0, nch, 1);
            for (int j = 0; j < n; ++j, cur.step(1, nch, 1)) {
                const int slot = j % VS_NST;
                if (j >= VS_NST && !mbar_wait(&empty[slot], ((j / VS_NST) - 1) & 1)) {
                    set_status(a.status, OSPREY_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                    break;
                }
                const int b = (int)cur.row, c = cur.c;
                if (b != rb) {
                    r = __ldcg(&decs[b].r);
                    rb = b;
                    if (r < -1 || r > K) {   // not written by vs_stats: read nothing through it
                        set_status(a.status, OSPREY_ERR_INVALID_ARG);
                        r = -1;
                    }
                }
                uint8_t *dst = smem + (size_t)slot * VS_SLOT;
                const int nel = min(L::EL, V - c * L::EL);
                issued = j + 1;
                if (r < 0 || nel <= 0) {   // nothing to copy: complete the slot's phase
                    if (nel <= 0) set_status(a.status, OSPREY_ERR_INVALID_ARG);
                    mbar_arrive_expect_tx(&full[slot], 0);
                    continue;
                }
                const uint32_t bytes = (uint32_t)nel * sizeof(T);
                const bool has_q = r < K;
                mbar_arrive_expect_tx(&full[slot], has_q ? 2 * bytes : bytes);
                bulk_g2s_hint(dst, (const T *)a.target + ((size_t)b * (K + 1) + r) * V + (size_t)c * L::EL, bytes,
                              &full[slot], pol);
                if (has_q)
                    bulk_g2s_hint(dst + VS_ROWB, (const T *)a.draft + ((size_t)b * K + r) * V + (size_t)c * L::EL,
                                  bytes, &full[slot], pol);
            }
            if (s_abort)
                for (int j = max(0, issued - VS_NST); j < issued; ++j)
                    mbar_wait(&full[j % VS_NST], (j / VS_NST) & 1, 200000000LL);
        }
        return;
    }
    int cur_b = -1, pend = 0;
    bool aborted = false;
    Decision d{};
    // the consumer warps divide per tile: with the incremental cursor here the
    // sampling walk's loads of the chosen chunk measured 4.9 us instead of 1.4 us
    // at batch 1 (cause not identified)
    for (int j = warp; j < n; j += VS_CW) {
        const long long t = t0 + j;
        const int b = (int)(t / nch), c = (int)(t % nch);
        if (b != cur_b) {
            if (pend && vs_arrive(a.ticket2 + cur_b, pend, nch) && d.r >= 0) vs_pick<T>(a, cur_b, d);
            cur_b = b;
            pend = 0;
            d = decs[b];
            if (d.r > K) d.r = -1;   // corrupt decision (reported by the producer)
        }
        const int slot = j % VS_NST;
        if (!vs_wait_slot(full, empty, j)) {
            set_status(a.status, OSPREY_ERR_TIMEOUT);
            atomicExch(&s_abort, 1);
            mbar_wait(&full[slot], (j / VS_NST) & 1, 200000000LL);
            aborted = true;
            break;
        }
        float2 sums = make_float2(0.f, 0.f);
        if (d.r >= 0) {
            const bool residual = d.r < K;
            const int nel = min(L::EL, V - c * L::EL);
            const bool whole = nel == L::EL;
            const uint8_t *chunk = smem + (size_t)slot * VS_SLOT;
            // the vectors are read straight from the slot, which is freed afterwards
            const VsNorm nrm = vs_norm(d, a.temperature);
            float sw = 0.f, sp = 0.f;
#pragma unroll 4
            for (int k = 0; k < VS_NV; ++k) {
                if (!whole && (lane + 32 * k) * L::VW >= nel) continue;
                float f[L::VW], g[L::VW];
                L::unpack(((const uint4 *)chunk)[lane + 32 * k], f);
                if (residual) L::unpack(((const uint4 *)(chunk + VS_ROWB))[lane + 32 * k], g);
#pragma unroll
                for (int e = 0; e < L::VW; ++e) {
                    float p;
                    sw += vs_pw(f[e], residual ? g[e] : 0.f, nrm, residual, p);
                    sp += p;
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
            sums = make_float2(warp_sum(sw), warp_sum(sp));
        } else {
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
        }
        if (lane == 0) ((float2 *)a.tsum)[t] = sums;
        ++pend;
    }
    if (!aborted && pend && vs_arrive(a.ticket2 + cur_b, pend, nch) && d.r >= 0) vs_pick<T>(a, cur_b, d);
}

// ---------------------------------------------------------------------------
bool verify_stream_ok(const VerifyArgs &a) {
    const int s = a.dtype == OSPREY_F32 ? 4 : 2;
    const size_t row = (size_t)a.V * s;
    return row % 16 == 0 && (uintptr_t)a.target % 16 == 0 && (a.draft == nullptr || (uintptr_t)a.draft % 16 == 0) &&
           a.K + 1 <= 32;
}

// Opt each kernel into the ring's shared memory once per device.  The flag
// lives in a per-kernel template (the kernels share one function type).
template <auto Kernel>
static cudaError_t vs_allow_smem() {
    static std::atomic<int> done[kMaxDevices];
    return once_per_device(done, [] {
        return cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, VS_NST * VS_SLOT);
    });
}

template <auto Kernel>
static cudaError_t vs_launch(const VerifyArgs &a, int blocks, cudaStream_t s) {
    cudaError_t e = vs_allow_smem<Kernel>();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks);
    cfg.blockDim = dim3(VS_THREADS);
    cfg.dynamicSmemBytes = (size_t)VS_NST * VS_SLOT;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, Kernel, a);
    count_launch();
    return e;
}

template <typename T>
static cudaError_t launch_vs(const VerifyArgs &a, int sms, cudaStream_t s) {
    const long long nt1 = (long long)a.B * (a.K + 1) * a.nch3, nt2 = (long long)a.B * a.nch3;
    const long long cap = (long long)OSP_VS_BPS * sms;
    const int g1 = (int)(nt1 < cap ? nt1 : cap), g2 = (int)(nt2 < cap ? nt2 : cap);
    if (a.temperature == 0.f) return vs_launch<vs_stats<T, true>>(a, g1, s);
    cudaError_t e = vs_launch<vs_stats<T, false>>(a, g1, s);
    if (e != cudaSuccess) return e;
    return vs_launch<vs_sample<T>>(a, g2, s);
}

cudaError_t launch_verify_stream(const VerifyArgs &a, int sms, cudaStream_t s) {
    // chunks per row for this dtype (the workspace holds enough for float32)
    VerifyArgs b = a;
    if (a.dtype == OSPREY_F32) {
        b.nch3 = (a.V + VsT<float>::EL - 1) / VsT<float>::EL;
        return launch_vs<float>(b, sms, s);
    }
    b.nch3 = (a.V + VsT<uint16_t>::EL - 1) / VsT<uint16_t>::EL;
    return launch_vs<uint16_t>(b, sms, s);
}

}  // namespace osp
