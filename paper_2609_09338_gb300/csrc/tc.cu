// Batched-row draft step on tcgen05 tensor cores: streamed swap-AB GEMMs for
// the projections of Sec. 3.3 (Eq. 1-3, MLP, LM head), operand preparation,
// RoPE + paged K/V write, and per-row sampling of the draft token (Sec. 3.1).
//
// tc_kernel: persistent, two CTAs per SM, 6 warps.
//   warp 0     issues 2-D TMA copies of one 128-row weight tile and the
//              activation planes per 64-wide k-block into
//              an nst-slot shared-memory ring (128-byte swizzle);
//   warp 1     issues tcgen05.mma (M 128, N npad, K 16, bf16 in, float32
//              accumulate in TMEM) per k-block and plane, then commits the
//              k-block to the slot's "empty" barrier and the tile to the
//              accumulator's "full" barrier;
//   warps 2-5  read the accumulator (tcgen05.ld, TMEM lane group = warp % 4)
//              and run the epilogue while the next tile accumulates into the
//              other TMEM buffer.
// Every wait is bounded; on expiry the CTA records OSPREY_ERR_TIMEOUT, stops
// issuing, lets its copies and MMAs land and frees its TMEM.
#include <cooperative_groups.h>
#include <cudaTypedefs.h>
#include <math.h>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"
#include "tma.cuh"

namespace osp {

namespace cg = cooperative_groups;

constexpr int TC_THREADS = 192;
constexpr int TC_ABYTES = 128 * 128;    // weight tile: 128 rows x 64 bf16
constexpr int TC_MAXST = 8;
#ifndef OSP_TC_CTAS_PER_SM
#define OSP_TC_CTAS_PER_SM 2   // two CTAs per SM: two TMA producers and two MMA chains per SM
#endif
constexpr size_t TC_SMEM_CAP = (OSP_TC_CTAS_PER_SM == 1 ? 200 : 100) * 1024;
#ifndef OSP_TC_SEGKB
#define OSP_TC_SEGKB 8   // k-blocks (64 wide) per accumulation segment
#endif
#ifndef OSP_TC_LM_NA
#define OSP_TC_LM_NA 2   // LM head: weight tiles per stage that share one operand stage
#endif

// ---------------------------------------------------------------- tcgen05 PTX
__device__ __forceinline__ void tma_2d(void *dst, const CUtensorMap *m, int x, int y, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_u32(dst)),
        "l"(m), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}
// Shared-memory matrix descriptor: K-major tile, rows 128 bytes apart inside
// 8-row (1024-byte) swizzle atoms.
__device__ __forceinline__ uint64_t tc_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;              // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;    // stride byte offset: one 8-row atom
    d |= (uint64_t)1 << 46;              // descriptor version
    d |= (uint64_t)2 << 61;              // 128-byte swizzle
    return d;
}
// Instruction descriptor, kind::f16: bf16 A and B (K-major), float32 D.
__host__ __device__ constexpr uint32_t tc_idesc(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void tc_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\ntcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d),
                 "l"(a), "l"(b), "r"(idesc), "r"(acc)
                 : "memory");
}
__device__ __forceinline__ void tc_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[j]);
}
__device__ __forceinline__ void tc_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tc_st16(uint32_t taddr, const float (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
            taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
        "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
        "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15]))
        : "memory");
}
__device__ __forceinline__ void tc_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// x ~= q0 + q1 + q2 with q_i = bf16(x - q0 - ... - q_{i-1}): 8 significant bits
// per plane, so three planes carry a float32 value's 24 (up to the last rounding).
__device__ __forceinline__ void tc_split(float x, uint16_t (&q)[TC_PLANES]) {
    float r = x;
#pragma unroll
    for (int i = 0; i < TC_PLANES; ++i) {
        q[i] = f_to_bf(r);
        r -= bf_to_f(q[i]);
    }
}

// Merges two (argmax logit a with its id i, sum s of exp((z - a) / T)) pairs
// into the first: the larger logit wins (the lower id on ties) and the
// other's sum is rescaled to it.
__device__ __forceinline__ void lm_combine(float &a1, int &i1, float &s1, float a2, int i2, float s2, float invT) {
    const bool two = a2 > a1 || (a2 == a1 && i2 < i1);
    const float aw = two ? a2 : a1, al = two ? a1 : a2;
    const float sw = two ? s2 : s1, sl = two ? s1 : s2;
    const float f = al == -INFINITY ? 0.f : __expf((al - aw) * invT);
    a1 = aw;
    i1 = two ? i2 : i1;
    s1 = sw + sl * f;
}

// ---------------------------------------------------------------- GEMM kernel
// NA weight tiles (NA x 128 output features) share each stage's operand
// planes: one work item is NA adjacent tiles, accumulated side by side in TMEM.
// Output features [0, nout_a) come from the weights of map wa, the rest from
// wb (row f - nout_a): the SwiGLU gate and up projections run as one GEMM.
template <int EPI, int NA>
__global__ void __launch_bounds__(TC_THREADS, OSP_TC_CTAS_PER_SM)
    tc_kernel(const __grid_constant__ CUtensorMap wa, const __grid_constant__ CUtensorMap wb,
              const __grid_constant__ CUtensorMap xm, const TcArgs a, int nst) {
    extern __shared__ uint8_t raw[];
    uint8_t *sm = (uint8_t *)(((uintptr_t)raw + 1023) & ~(uintptr_t)1023);
    __shared__ __align__(8) uint64_t full[TC_MAXST], empty[TC_MAXST], accf[2], acce[2], fin;
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // work item = (NA output tiles of 128 features, k-range); items of a CTA are contiguous
    const int segkb = a.segkb;
    const int n_items = (a.nout + 128 * NA - 1) / (128 * NA) * a.nsplit;
    const int i0 = (int)((long long)n_items * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)n_items * (blockIdx.x + 1) / gridDim.x);
    const int nloc = i1 - i0, nkb = a.K / 64, npad = a.npad;
    auto krange = [&](int item, int &lo, int &hi) {
        const int sp = item % a.nsplit;
        lo = sp * a.kbps;
        hi = min(nkb, lo + a.kbps);
    };
    const uint32_t bbytes = (uint32_t)a.planes * npad * 128;
    const uint32_t stage = NA * TC_ABYTES + bbytes;
    // TMEM: two segment buffers and (when a tile has several segments) the
    // running float32 total of the tile
    const uint32_t acc_cols = NA * npad;
    const int nseg_max = (min(nkb, a.kbps) + segkb - 1) / segkb;
    uint32_t ncols = 32;
    while (ncols < (nseg_max > 1 ? 3 : 2) * acc_cols) ncols <<= 1;

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s_tmem)),
                     "r"(ncols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (threadIdx.x == 32) {
        for (int i = 0; i < nst; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&accf[i], 1);
            mbar_init(&acce[i], 4);
        }
        mbar_init(&fin, 1);
        s_abort = 0;
        mbar_fence_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    pdl_trigger();
    // the activation planes and the residual come from earlier kernels; the
    // producer first requests the weight tiles of the ring's first stages,
    // which do not, and waits after that
    if (warp != 0) pdl_wait();

    if (warp == 0) {
        if (lane == 0) {
            auto weights = [&](uint8_t *st, int y, int kb, uint64_t *bar) {
#pragma unroll
                for (int t = 0; t < NA; ++t) {
                    const int f = y + 128 * t;   // tiles never straddle nout_a (a multiple of 128)
                    tma_2d(st + t * TC_ABYTES, f < a.nout_a ? &wa : &wb, kb * 64, f < a.nout_a ? f : f - a.nout_a, bar);
                }
            };
            long long npre = 0;   // stages whose weights were requested before the wait
            for (int it = 0; it < nloc && npre < nst; ++it) {
                const int y = (i0 + it) / a.nsplit * 128 * NA;
                int klo, khi;
                krange(i0 + it, klo, khi);
                for (int kb = klo; kb < khi && npre < nst; ++kb, ++npre) {
                    mbar_expect_tx(&full[npre], NA * TC_ABYTES);
                    weights(sm + (size_t)npre * stage, y, kb, &full[npre]);
                }
            }
            pdl_wait();
            long long g = 0;
            bool stop = false;
            for (int it = 0; it < nloc && !stop; ++it) {
                const int y = (i0 + it) / a.nsplit * 128 * NA;
                int klo, khi;
                krange(i0 + it, klo, khi);
                for (int kb = klo; kb < khi; ++kb, ++g) {
                    const int s = (int)(g % nst);
                    if (g >= nst && !mbar_wait(&empty[s], (uint32_t)((g / nst) - 1) & 1)) {
                        set_status(a.status, OSPREY_ERR_TIMEOUT);
                        atomicExch(&s_abort, 1);
                        stop = true;
                        break;
                    }
                    if (*(volatile int *)&s_abort) { stop = true; break; }
                    uint8_t *st = sm + (size_t)s * stage;
                    if (g < npre) {
                        mbar_arrive_expect_tx(&full[s], bbytes);
                    } else {
                        mbar_arrive_expect_tx(&full[s], stage);
                        weights(st, y, kb, &full[s]);
                    }
                    for (int p = 0; p < a.planes; ++p)
                        tma_2d(st + NA * TC_ABYTES + (size_t)p * npad * 128, &xm, kb * 64, p * npad, &full[s]);
                }
            }
            if (stop) {   // let the copies this thread issued land before the CTA can exit
                // stages whose weights were requested early but never armed: arrive, so
                // that their phase completes when the weights land
                for (long long q = g; q < npre; ++q) mbar_arrive(&full[q]);
                const long long end = g > npre ? g : npre;
                for (long long q = end - nst > 0 ? end - nst : 0; q < end; ++q)
                    mbar_wait(&full[q % nst], (uint32_t)(q / nst) & 1, 200000000LL);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // one accumulation unit = one segment of one tile, into buffer u & 1
            const uint32_t idesc = tc_idesc(128, npad);
            long long g = 0, u = 0;
            bool stop = false;
            for (int it = 0; it < nloc && !stop; ++it) {
                int klo, khi;
                krange(i0 + it, klo, khi);
                const int nseg = (khi - klo + segkb - 1) / segkb;
                for (int sg = 0; sg < nseg && !stop; ++sg, ++u) {
                    const int buf = (int)(u & 1);
                    if (u >= 2 && !mbar_wait(&acce[buf], (uint32_t)((u >> 1) - 1) & 1)) {
                        set_status(a.status, OSPREY_ERR_TIMEOUT);
                        atomicExch(&s_abort, 1);
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d0 = tmem + (uint32_t)buf * acc_cols;
                    const int kb0 = klo + sg * segkb, kb1 = min(khi, kb0 + segkb);
                    for (int kb = kb0; kb < kb1; ++kb, ++g) {
                        const int s = (int)(g % nst);
                        if (!mbar_wait(&full[s], (uint32_t)(g / nst) & 1) || *(volatile int *)&s_abort) {
                            set_status(a.status, OSPREY_ERR_TIMEOUT);
                            atomicExch(&s_abort, 1);
                            stop = true;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t st = smem_u32(sm + (size_t)s * stage);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            for (int p = 0; p < a.planes; ++p) {
                                const uint64_t db = tc_desc(st + NA * TC_ABYTES + (uint32_t)p * npad * 128);
                                const uint32_t acc = (kb != kb0) || kk || p;
#pragma unroll
                                for (int t = 0; t < NA; ++t)
                                    tc_mma(d0 + (uint32_t)(t * npad), tc_desc(st + t * TC_ABYTES) + 2 * kk, db + 2 * kk,
                                           idesc, acc);
                            }
                        }
                        tc_commit(&empty[s]);
                    }
                    if (!stop) tc_commit(&accf[buf]);
                }
            }
            tc_commit(&fin);
            mbar_wait(&fin, 0, 400000000LL);   // every MMA of this CTA has completed
        }
    } else {
        // epilogue: TMEM lanes (warp % 4) * 32 .. + 31 hold output features m.
        // Each segment's partial is added into the tile's running total in float32;
        // the last segment's sum goes through the epilogue.
        const int lg = (warp & 3) * 32;
        const int m = lg + lane;
        long long u = 0;
        bool stop = false;
        for (int it = 0; it < nloc && !stop; ++it) {
            const int col0 = (i0 + it) / a.nsplit * 128 * NA + m, sp = (i0 + it) % a.nsplit;
            const uint32_t tt = tmem + ((uint32_t)lg << 16) + 2u * acc_cols;
            int klo, khi;
            krange(i0 + it, klo, khi);
            const int nseg = (khi - klo + segkb - 1) / segkb;
            for (int sg = 0; sg < nseg; ++sg, ++u) {
                const int buf = (int)(u & 1);
                if (!mbar_wait(&accf[buf], (uint32_t)(u >> 1) & 1) || *(volatile int *)&s_abort) {
                    set_status(a.status, OSPREY_ERR_TIMEOUT);
                    atomicExch(&s_abort, 1);
                    stop = true;
                    break;
                }
                tc_fence_after();
                const bool last = sg == nseg - 1;
                const uint32_t t0 = tmem + ((uint32_t)lg << 16) + (uint32_t)buf * acc_cols;
                for (int cc = 0; cc < NA * npad; cc += 16) {
                    // accumulator columns [t npad, (t + 1) npad) hold tile t's rows
                    const int tile = cc / npad, c0 = cc - tile * npad;
                    const int col = col0 + 128 * tile;
                    const bool colok = col < a.nout;
                    float v[16], tv[16];
                    tc_ld16(t0 + (uint32_t)cc, v);
                    if (sg > 0) tc_ld16(tt + (uint32_t)cc, tv);
                    tc_ld_wait();
                    if (sg > 0) {
#pragma unroll
                        for (int j = 0; j < 16; ++j) v[j] += tv[j];
                    }
                    if (!last) {
                        tc_st16(tt + (uint32_t)cc, v);
                        continue;
                    }
                    if constexpr (EPI == TC_LM) {
                        // per row: (argmax z, sum exp((z - max z) / T)) over this warp's 32
                        // ids, for the 16 rows c0.. at once: each butterfly round halves the
                        // rows a lane carries (it keeps one half and receives the partner's
                        // share of it), so after four rounds lane l holds row l / 2 over 16
                        // lanes and one more exchange completes it over all 32
                        const int sub = (int)(((long long)((i0 + it) / a.nsplit) * 128 * NA + 128 * tile + lg) /
                                              TC_LM_GROUP);
                        float av[16], sv[16];
                        int ai[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            av[j] = colok ? v[j] : -INFINITY;
                            ai[j] = colok ? col : 0x7fffffff;
                            sv[j] = colok ? 1.f : 0.f;
                            if (a.y && colok && c0 + j < a.R) a.y[(size_t)(c0 + j) * a.ldy + col] = v[j];
                        }
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            const int off = 16 >> r, w = 8 >> r;
                            const bool up = lane & off;
#pragma unroll
                            for (int i = 0; i < w; ++i) {
                                const float ra = __shfl_xor_sync(0xffffffffu, up ? av[i] : av[i + w], off);
                                const int ri = __shfl_xor_sync(0xffffffffu, up ? ai[i] : ai[i + w], off);
                                const float rs = __shfl_xor_sync(0xffffffffu, up ? sv[i] : sv[i + w], off);
                                float ka = up ? av[i + w] : av[i], ks = up ? sv[i + w] : sv[i];
                                int ki = up ? ai[i + w] : ai[i];
                                lm_combine(ka, ki, ks, ra, ri, rs, a.lm_invT);
                                av[i] = ka;
                                ai[i] = ki;
                                sv[i] = ks;
                            }
                        }
                        {
                            const float ra = __shfl_xor_sync(0xffffffffu, av[0], 1);
                            const int ri = __shfl_xor_sync(0xffffffffu, ai[0], 1);
                            const float rs = __shfl_xor_sync(0xffffffffu, sv[0], 1);
                            lm_combine(av[0], ai[0], sv[0], ra, ri, rs, a.lm_invT);
                        }
                        const int n = c0 + (lane >> 1);
                        if (!(lane & 1) && n < a.R && sub < a.lm_nsub)
                            a.lm_part[(size_t)n * a.lm_nsub + sub] =
                                make_float4(av[0] * a.lm_invT, sv[0], av[0], __int_as_float(ai[0]));
                    } else {
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const int n = c0 + j;
                            if (n >= a.R || !colok) continue;
                            if (a.nsplit > 1 || EPI == TC_GLU) {   // partial of this k-range; tc_reduce applies the epilogue
                                a.part[((size_t)sp * a.R + n) * a.nout + col] = v[j];
                            } else if (EPI == TC_STORE) {
                                a.y[(size_t)n * a.ldy + col] = v[j];
                            } else if (EPI == TC_RESID) {
                                a.x[(size_t)n * a.ldy + col] += v[j];
                            }
                        }
                    }
                }
                if (!last) tc_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acce[buf]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols));
}

// ---------------------------------------------------------------- split-K reduction
// out[n][col] = sum over the k-ranges (in order) of the partials, then the
// GEMM's epilogue.  TC_GLU: gate = output col, up = output nout_a + col, and
// the planes of h = silu(gate) * up go to h [TC_PLANES][npad][nout_a].
template <int EPI>
__global__ void __launch_bounds__(256) tc_reduce_kernel(const TcArgs a) {
    pdl_trigger();
    pdl_wait();
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const int w = EPI == TC_GLU ? a.nout_a : a.nout;
    if (idx >= (long long)a.R * w) return;
    const int n = (int)(idx / w), col = (int)(idx % w);
    float v = 0.f;
    for (int sp = 0; sp < a.nsplit; ++sp) v += __ldcg(a.part + ((size_t)sp * a.R + n) * a.nout + col);
    if (EPI == TC_STORE) {
        a.y[(size_t)n * a.ldy + col] = v;
    } else if (EPI == TC_RESID) {
        a.x[(size_t)n * a.ldy + col] += v;
    } else {
        float u = 0.f;
        for (int sp = 0; sp < a.nsplit; ++sp) u += __ldcg(a.part + ((size_t)sp * a.R + n) * a.nout + w + col);
        const float h = v / (1.f + expf(-v)) * u;
        uint16_t q[TC_PLANES];
        tc_split(h, q);
#pragma unroll
        for (int i = 0; i < TC_PLANES; ++i) a.h[((size_t)i * a.npad + n) * w + col] = q[i];
    }
}

// TC_RESID reduction with the next operand's planes: a cluster of RP_CS blocks
// per row n, each summing the partials (in range order) of its share of the
// columns into x[n]; the blocks' sums of squares are exchanged through
// distributed shared memory, then each writes the RMS-normalised planes of its
// columns.
constexpr int RP_CS = 8;     // blocks per row (one cluster)
constexpr int RP_VPT = 4;    // columns per thread at most (nout <= RP_CS * 256 * RP_VPT)
__device__ __forceinline__ void rp_cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void rp_cluster_arrive_release() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void rp_cluster_wait_acquire() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__global__ void __launch_bounds__(256) tc_resid_planes_kernel(const TcArgs a) {
    __shared__ float red[8];
    __shared__ float css[RP_CS];   // every block's sum of squares, pushed by its owner
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank(), n = blockIdx.y, t = threadIdx.x;
    rp_cluster_arrive_relaxed();   // started: the cluster may write this block's shared memory
    pdl_trigger();
    pdl_wait();
    int prow = -1;
    bool act = false;
    if (a.pl_map == 0) {
        const int b = n / a.pl_rows_per_seq, j = n - b * a.pl_rows_per_seq;
        act = a.pl_valid[b] && (a.pl_rows_per_seq == 1 || j < a.pl_nnew[b]);
        prow = n;
    } else {
        const int b = n / a.pl_max_new, j = n - b * a.pl_max_new;
        if (a.pl_valid[b] ? j == a.pl_nnew[b] - 1 : j == 0) {
            prow = b;
            act = a.pl_valid[b] != 0;
        }
    }
    const int per = (a.nout + RP_CS - 1) / RP_CS;
    const int c0 = rank * per, c1 = min(a.nout, c0 + per);
    float xv[RP_VPT];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < RP_VPT; ++i) {
        const int col = c0 + t + 256 * i;
        xv[i] = 0.f;
        if (col >= c1) continue;
        float v = 0.f;
        for (int sp = 0; sp < a.nsplit; ++sp) v += __ldcg(a.part + ((size_t)sp * a.R + n) * a.nout + col);
        const float xn = a.x[(size_t)n * a.ldy + col] + v;
        a.x[(size_t)n * a.ldy + col] = xn;
        xv[i] = xn;
        ss = fmaf(xn, xn, ss);
    }
    if (prow < 0) return;   // the whole cluster (same row) leaves here
    ss = warp_sum(ss);
    if ((t & 31) == 0) red[t >> 5] = ss;
    __syncthreads();
    rp_cluster_wait_acquire();   // every block of the cluster has started
    if (t == 0) {
        float tot = 0.f;
        for (int w = 0; w < 8; ++w) tot += red[w];
        for (int k = 0; k < RP_CS; ++k) *cluster.map_shared_rank(&css[rank], k) = tot;
    }
    rp_cluster_arrive_release();
    rp_cluster_wait_acquire();   // every block's sum has arrived here
    float tot = 0.f;
#pragma unroll
    for (int k = 0; k < RP_CS; ++k) tot += css[k];
    const float inv = rsqrtf(tot / (float)a.nout + a.pl_eps);
    uint16_t *p0 = a.pl_dst + (size_t)prow * a.pl_ld + a.pl_col0;
    const size_t plane = (size_t)a.pl_npad * a.pl_ld;
#pragma unroll
    for (int i = 0; i < RP_VPT; ++i) {
        const int col = c0 + t + 256 * i;
        if (col >= c1) continue;
        const float v = act ? xv[i] * inv * bf_to_f(a.pl_gain[col]) : 0.f;
        uint16_t q[TC_PLANES];
        tc_split(v, q);
#pragma unroll
        for (int j = 0; j < TC_PLANES; ++j)
            if (j < a.pl_npl) p0[j * plane + col] = q[j];
    }
}

// ---------------------------------------------------------------- operand planes
__global__ void __launch_bounds__(256) planes_kernel(const PlaneArgs a) {
    __shared__ float red[33];
    const int r = blockIdx.x;
    pdl_trigger();
    pdl_wait();
    bool act;
    int srow;
    if (a.last_of_seq) {
        act = !a.valid || a.valid[r];
        srow = act ? r * a.max_new + a.nnew[r] - 1 : 0;
    } else {
        const int b = r / a.rows_per_seq, j = r - b * a.rows_per_seq;
        act = (!a.valid || a.valid[b]) && (a.rows_per_seq == 1 || j < a.nnew[b]);
        srow = r;
    }
    const float *x = a.src + (size_t)srow * a.d;
    float inv = 1.f;
    if (a.gain) {
        float ss = 0.f;
        if (act)
            for (int k = threadIdx.x; k < a.d; k += blockDim.x) ss = fmaf(x[k], x[k], ss);
        ss = warp_sum(ss);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
        __syncthreads();
        if (threadIdx.x == 0) {
            float t = 0.f;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
            red[32] = rsqrtf(t / (float)a.d + a.eps);
        }
        __syncthreads();
        inv = red[32];
    }
    uint16_t *p0 = a.dst + (size_t)r * a.ld + a.col0;
    const size_t plane = (size_t)a.npad * a.ld;
    const int npl = a.npl > 0 ? a.npl : TC_PLANES;
    for (int k = threadIdx.x; k < a.d; k += blockDim.x) {
        float v = act ? x[k] : 0.f;
        if (a.gain) v = v * inv * bf_to_f(a.gain[k]);
        uint16_t q[TC_PLANES];
        tc_split(v, q);
#pragma unroll
        for (int i = 0; i < TC_PLANES; ++i)
            if (i < npl) p0[i * plane + k] = q[i];
    }
    if (a.src2) {   // a second part of the row, copied without normalisation
        const float *x2 = a.src2 + (size_t)srow * a.d;
        uint16_t *p2 = a.dst + (size_t)r * a.ld + a.col2;
        for (int k = threadIdx.x; k < a.d; k += blockDim.x) {
            uint16_t q[TC_PLANES];
            tc_split(act ? x2[k] : 0.f, q);
#pragma unroll
            for (int i = 0; i < TC_PLANES; ++i)
                if (i < npl) p2[i * plane + k] = q[i];
        }
    }
}

// ---------------------------------------------------------------- RoPE + K/V write
__global__ void __launch_bounds__(256) qkv_post_kernel(const QkvPostArgs a) {
    const Dims &D = a.dim;
    const int half = D.hd / 2;
    const int per_row = (D.Hq + 2 * D.Hkv) * half;
    pdl_trigger();
    pdl_wait();
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)a.R * per_row) return;
    const int r = (int)(idx / per_row), item = (int)(idx % per_row);
    int b, pos;
    if (!a.map.row(r, b, pos)) return;
    const int h = item / half, ii = item % half;
    const float *yr = a.y + (size_t)r * (D.Hq + 2 * D.Hkv) * D.hd + (size_t)h * D.hd;
    float x1 = yr[ii], x2 = yr[ii + half];
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
        uint16_t *dst = (is_k ? a.k_pages : a.v_pages) + (((size_t)page * D.Hkv + kvh) * D.P + pos % D.P) * D.hd;
        dst[ii] = f_to_bf(x1);
        dst[ii + half] = f_to_bf(x2);
    }
}

// The QKV GEMM's split-K reduction with RoPE and the paged K/V write folded
// in: each thread sums the partials (in range order) of one rotary pair
// (ii, ii + hd / 2) of one head, then does what qkv_post_kernel does with it.
__global__ void __launch_bounds__(256) tc_reduce_rope_kernel(const TcArgs a, const QkvPostArgs p) {
    const Dims &D = p.dim;
    const int half = D.hd / 2;
    const int per_row = (D.Hq + 2 * D.Hkv) * half;
    pdl_trigger();
    pdl_wait();
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)a.R * per_row) return;
    const int r = (int)(idx / per_row), item = (int)(idx % per_row);
    int b, pos;
    if (!p.map.row(r, b, pos)) return;
    const int h = item / half, ii = item % half;
    const int col = h * D.hd + ii;
    float x1 = 0.f, x2 = 0.f;
    for (int sp = 0; sp < a.nsplit; ++sp) {
        const float *pr = a.part + ((size_t)sp * a.R + r) * a.nout;
        x1 += __ldcg(pr + col);
        x2 += __ldcg(pr + col + half);
    }
    if (h < D.Hq + D.Hkv) {
        float c, sn;
        rope_cs2(p.inv_freq[ii], pos, c, sn);
        const float y1 = x1 * c - x2 * sn, y2 = x2 * c + x1 * sn;
        x1 = y1;
        x2 = y2;
    }
    if (h < D.Hq) {
        float *q = p.q + (size_t)r * D.Hq * D.hd + (size_t)h * D.hd;
        q[ii] = x1;
        q[ii + half] = x2;
    } else {
        const bool is_k = h < D.Hq + D.Hkv;
        const int kvh = is_k ? h - D.Hq : h - D.Hq - D.Hkv;
        const int page = p.page_table[(size_t)b * p.max_pages + pos / D.P];
        uint16_t *dst = (is_k ? p.k_pages : p.v_pages) + (((size_t)page * D.Hkv + kvh) * D.P + pos % D.P) * D.hd;
        dst[ii] = f_to_bf(x1);
        dst[ii + half] = f_to_bf(x2);
    }
}

// ---------------------------------------------------------------- LM-head pick
constexpr int PK_THREADS = 1024;   // each thread walks about V / 32 / 1024 partials

constexpr int PK_MAXK = 8;   // candidates per row at most

// Recomputes the 32 logits of group g (ids 32 g ..): 8 warps x 4 ids, lanes
// split the reduction over the row's operand in shared memory.
__device__ __forceinline__ void pk_group_logits(const LmPickArgs &a, const float *hrow, int g, float *z) {
    const Dims &D = a.dim;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int PER = TC_LM_GROUP / (PK_THREADS / 32);
    for (int i = 0; i < PER; ++i) {
        const int id = g * TC_LM_GROUP + warp * PER + i;
        float acc = 0.f;
        if (id < D.V) {
            const uint16_t *wr = a.W + (size_t)id * D.d;
            for (int k = lane * 8; k < D.d; k += 256) {
                float wf[8];
                unpack8(ld_stream(wr + k), wf);
#pragma unroll
                for (int e = 0; e < 8; ++e) acc = fmaf(wf[e], hrow[k + e], acc);
            }
        }
        acc = warp_sum(acc);
        if (lane == 0) z[warp * PER + i] = id < D.V ? acc : -INFINITY;
    }
}

// One block per row.  Level 1: the row's 32-id partials, a contiguous run per
// thread, give M = max y, S = sum exp(y - M) and, per draw, the group holding
// u * S.  Level 2: that group's 32 logits, recomputed as dot products of the
// LM-head rows with the row's operand (the sum of its bf16 planes), scanned in
// ascending ids.  Greedy: the argmax from the partials; with topk > 1 the next
// candidates come from the topk groups of largest maximum (the only groups
// that can hold one of the topk largest logits), recomputed and ranked.
__global__ void __launch_bounds__(PK_THREADS) lm_pick_kernel(const LmPickArgs a) {
    extern __shared__ float hrow[];   // [d] the row's LM-head operand
    __shared__ MS sm_ms[PK_THREADS / 32];
    __shared__ AM sm_am[PK_THREADS / 32];
    __shared__ float sh[34];
    __shared__ int si[2];
    __shared__ float s_z[PK_MAXK * TC_LM_GROUP];
    __shared__ int s_grp[PK_MAXK], s_tok[PK_MAXK];
    __shared__ float s_before, s_e[PK_MAXK];
    const Dims &D = a.dim;
    const int b = blockIdx.x, t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int topk = a.topk > 1 ? a.topk : 1;
    pdl_trigger();
    pdl_wait();
    if (!a.valid[a.rows_per_valid > 1 ? b / a.rows_per_valid : b]) return;
    const bool greedy = a.temperature == 0.f;
    const float invT = greedy ? 1.f : 1.f / a.temperature;
    const float4 *pp = a.part + (size_t)b * a.nsub;
    const int per = (a.nsub + PK_THREADS - 1) / PK_THREADS;
    const int j0 = min(a.nsub, t * per), j1 = min(a.nsub, j0 + per);
    // one pass over the thread's run: its argmax and its (max, sum) rescaled online
    float m = -INFINITY, sm = 0.f;
    AM am{-INFINITY, 0x7fffffff};
    for (int j = j0; j < j1; ++j) {
        const float4 p = __ldcg(pp + j);
        am = am_combine(am, AM{p.z, __float_as_int(p.w)});
        if (p.x == -INFINITY) continue;
        if (p.x > m) {
            sm = (m == -INFINITY ? 0.f : sm * __expf(m - p.x)) + p.y;
            m = p.x;
        } else {
            sm += p.y * __expf(p.x - m);
        }
    }
    const MS tot = block_ms(MS{m, sm}, sm_ms);
    const float M = tot.m, S = tot.s;
    const float w = m == -INFINITY ? 0.f : sm * __expf(m - M);   // the run's weight
    if (topk > 1 || !greedy) {
        // the row's operand: the sum of its planes (the values the tensor cores multiplied)
        const size_t plane = (size_t)a.npad * D.d;
        const uint16_t *q = a.planes + (size_t)b * D.d;
        for (int k = t; k < D.d; k += PK_THREADS) {
            float h = 0.f;
#pragma unroll
            for (int i = 0; i < TC_LM_PLANES; ++i) h += bf_to_f(q[i * plane + k]);
            hrow[k] = h;
        }
    }
    if (greedy) {
        const AM top = block_am(am, sm_am);   // candidate 0: the argmax of the tensor-core logits
        if (t == 0) { s_tok[0] = top.i; s_e[0] = 1.f; }
        if (topk > 1) {
            // the topk groups of largest maximum, one block argmax per round
            for (int r = 0; r < topk; ++r) {
                AM loc{-INFINITY, 0x7fffffff};
                for (int j = j0; j < j1; ++j) {
                    bool taken = false;
                    for (int rr = 0; rr < r; ++rr) taken |= s_grp[rr] == j;
                    const float4 p = __ldcg(pp + j);
                    if (!taken) loc = am_combine(loc, AM{p.z, j});
                }
                const AM g = block_am(loc, sm_am);
                if (t == 0) s_grp[r] = g.v == -INFINITY ? -1 : g.i;
                __syncthreads();
            }
            __syncthreads();
            for (int r = 0; r < topk; ++r)
                if (s_grp[r] >= 0) pk_group_logits(a, hrow, s_grp[r], s_z + r * TC_LM_GROUP);
                else if (t < TC_LM_GROUP) s_z[r * TC_LM_GROUP + t] = -INFINITY;
            __syncthreads();
            // rank: candidates 1.. are the largest recomputed logits other than candidate 0
            for (int c = 1; c < topk; ++c) {
                AM loc{-INFINITY, 0x7fffffff};
                if (t < topk * TC_LM_GROUP) {
                    const int r = t / TC_LM_GROUP, l = t - r * TC_LM_GROUP;
                    const int id = s_grp[r] < 0 ? -1 : s_grp[r] * TC_LM_GROUP + l;
                    bool taken = id < 0;
                    for (int cc = 0; cc < c; ++cc) taken |= s_tok[cc] == id;
                    if (!taken) loc = AM{s_z[t], id};
                }
                const AM best = block_am(loc, sm_am);
                if (t == 0) { s_tok[c] = best.i == 0x7fffffff ? s_tok[0] : best.i; s_e[c] = 1.f; }
                __syncthreads();
            }
        }
        __syncthreads();
    } else {
        // each draw: its group from the partials, then its id inside the recomputed group
        float tot;
        const float ex = block_excl_scan(w, sh, &tot);
        for (int c = 0; c < topk; ++c) {
            const float target = a.u_draft[((size_t)b * a.K + a.step) * topk + c] * S;
            if (t == 0) { si[0] = 0x7fffffff; si[1] = -1; }
            __syncthreads();
            if (w > 0.f && target < ex + w) atomicMin(&si[0], t);
            if (w > 0.f) atomicMax(&si[1], t);
            __syncthreads();
            const int ct = si[0] != 0x7fffffff ? si[0] : (si[1] >= 0 ? si[1] : 0);
            if (t == ct) {   // this thread's run holds the point: find its group
                float cum = ex;
                int grp = -1, lastg = -1;
                float lastb = ex;
                for (int j = j0; j < j1; ++j) {
                    const float4 p = __ldcg(pp + j);
                    const float wj = p.x != -INFINITY ? p.y * __expf(p.x - M) : 0.f;
                    if (wj > 0.f) { lastg = j; lastb = cum; }
                    if (wj > 0.f && target < cum + wj) { grp = j; break; }
                    cum += wj;
                }
                s_grp[c] = grp >= 0 ? grp : (lastg >= 0 ? lastg : j0);
                s_before = grp >= 0 ? cum : lastb;
            }
            __syncthreads();
            pk_group_logits(a, hrow, s_grp[c], s_z);
            __syncthreads();
            if (warp == 0) {
                const int id = s_grp[c] * TC_LM_GROUP + lane;
                const float e = id < D.V ? __expf(s_z[lane] * invT - M) : 0.f;
                const float cum = s_before + warp_incl_scan(e);
                const unsigned hit = __ballot_sync(0xffffffffu, e > 0.f && target < cum);
                const unsigned pos = __ballot_sync(0xffffffffu, e > 0.f);
                const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
                if (lane == l) { s_tok[c] = id; s_e[c] = e; }
            }
            __syncthreads();
        }
    }
    const size_t o = (size_t)b * a.K + a.step;
    if (t < topk) {
        a.tokens[o * topk + t] = s_tok[t];
        if (a.qx) a.qx[o * topk + t] = greedy ? 1.f : s_e[t] / S;
    }
    if (t == 0 && a.stats) {
        a.stats[o * 2 + 0] = M;
        a.stats[o * 2 + 1] = logf(S);
    }
    const int token = s_tok[0];
    if (a.step + 1 < a.K) {
        // next chain row: context slot <- x_L (Sec. 3.4), residual <- E[candidate 0]
        const int src = a.src_is_ext ? b * a.max_new + a.nnew[b] - 1 : b;
        const float *xl = a.x_in + (size_t)src * D.d;
        const uint16_t *er = a.embed + (size_t)token * D.d;
        float ss = 0.f;
        for (int k = t; k < D.d; k += PK_THREADS) {
            const float e = bf_to_f(er[k]);
            a.s_chain[(size_t)b * D.d + k] = xl[k];
            a.x_chain[(size_t)b * D.d + k] = e;
            ss = fmaf(e, e, ss);
        }
        if (a.qkv_planes) {   // and its first layer's operand, [s; RMSNorm(x)]
            ss = warp_sum(ss);
            if (lane == 0) sh[warp] = ss;
            __syncthreads();
            if (t == 0) {
                float tot = 0.f;
                for (int w = 0; w < PK_THREADS / 32; ++w) tot += sh[w];
                sh[33] = rsqrtf(tot / (float)D.d + a.eps);
            }
            __syncthreads();
            const float inv = sh[33];
            const size_t ld = 2 * (size_t)D.d, plane = (size_t)a.qkv_npad * ld;
            uint16_t *p0 = a.qkv_planes + (size_t)b * ld;
            for (int k = t; k < D.d; k += PK_THREADS) {
                // the s half from this thread's own copy in s_chain: x_in may be x_chain,
                // whose row b now holds the embedding
                uint16_t q[TC_PLANES];
                tc_split(a.s_chain[(size_t)b * D.d + k], q);
#pragma unroll
                for (int i = 0; i < TC_PLANES; ++i) p0[i * plane + k] = q[i];
                tc_split(bf_to_f(er[k]) * inv * bf_to_f(a.qkv_gain[k]), q);
#pragma unroll
                for (int i = 0; i < TC_PLANES; ++i) p0[i * plane + D.d + k] = q[i];
            }
        }
    }
}

// ---------------------------------------------------------------- embedding rows
__global__ void __launch_bounds__(256) embed_rows_kernel(const EmbedArgs a) {
    const int r = blockIdx.x, b = r / a.max_new, j = r - b * a.max_new;
    pdl_trigger();
    pdl_wait();
    if (!a.valid[b] || j >= a.nnew[b]) return;
    const uint16_t *e = a.embed + (size_t)a.tokens[r] * a.d;   // ids checked by the prepare kernel
    for (int k = threadIdx.x; k < a.d; k += blockDim.x) a.x[(size_t)r * a.d + k] = bf_to_f(e[k]);
}

// ---------------------------------------------------------------- block inputs
__global__ void __launch_bounds__(256) block_inputs_kernel(const BlockInArgs a) {
    const int r = blockIdx.x, b = r / a.P, j = r - b * a.P;
    if (threadIdx.x == 0) {
        a.tokens[r] = j == 0 ? a.anchors[b] : a.mask;
        if (j == 0) a.nnew[b] = a.P;
    }
    const uint4 *src = (const uint4 *)(a.feats + (size_t)b * a.feat);
    uint4 *dst = (uint4 *)(a.feats_rep + (size_t)r * a.feat);
    for (int k = threadIdx.x; k < a.feat / 8; k += blockDim.x) dst[k] = src[k];
}

cudaError_t launch_block_inputs(const BlockInArgs &a, cudaStream_t s) {
    // a normal launch: the draft call's prepare kernel reads these arrays
    block_inputs_kernel<<<a.n * a.P, 256, 0, s>>>(a);
    count_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------- host side
static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

// The driver's tensor-map encoder and a device with tcgen05 (compute
// capability 10 or above); looked up once, thread-safely (a function-local
// static is initialised exactly once).
bool tc_available() {
    static const bool ok = [] {
        cudaDriverEntryPointQueryResult q;
        void *fn = nullptr;
        const cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        g_encode = e == cudaSuccess && q == cudaDriverEntryPointSuccess ? (PFN_cuTensorMapEncodeTiled_v12000)fn : nullptr;
        if (e != cudaSuccess) cudaGetLastError();
        int dev = 0, major = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) {
            cudaGetLastError();
            major = 0;
        }
        return g_encode != nullptr && major >= 10;
    }();
    return ok;
}

static bool encode2d(CUtensorMap *m, const void *base, uint64_t inner, uint64_t rows, uint32_t box_rows) {
    if (!tc_available()) return false;
    if (((uintptr_t)base & 15) || (inner * 2) % 16) return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t es[2] = {1, 1};
    return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool tc_encode_weight(CUtensorMap *m, const void *w, int rows, int K) { return encode2d(m, w, K, rows, 128); }
bool tc_encode_rows(CUtensorMap *m, const void *x, int rows, int npad, int K) { return encode2d(m, x, K, rows, npad); }
bool tc_encode_operand(CUtensorMap *m, const void *x, int planes, int npad, int K) {
    return encode2d(m, x, K, (uint64_t)planes * npad, npad);
}

static int tc_stages(int npad, int planes, int na) {
    const size_t stage = (size_t)na * TC_ABYTES + (size_t)planes * npad * 128;
    int n = (int)((TC_SMEM_CAP - 1024) / stage);
    return n > TC_MAXST ? TC_MAXST : n;
}
size_t tc_smem_bytes(int npad, int planes, int na) {
    const size_t stage = (size_t)na * TC_ABYTES + (size_t)planes * npad * 128;
    return (size_t)tc_stages(npad, planes, na) * stage + 1024;
}

cudaError_t tc_set_attributes() {
    const int bytes = (int)TC_SMEM_CAP;
    cudaError_t e = cudaFuncSetAttribute(tc_kernel<TC_STORE, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(tc_kernel<TC_RESID, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(tc_kernel<TC_GLU, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(tc_kernel<TC_LM, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && OSP_TC_LM_NA > 1)
        e = cudaFuncSetAttribute(tc_kernel<TC_LM, OSP_TC_LM_NA>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) e = allow_smem(lm_pick_kernel);
    return e;
}

template <typename... P, typename... A>
static cudaError_t pdl_launch(void (*k)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, const A &...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, k, args...);
    count_launch();
    return e;
}

// k-ranges per output tile so that tiles x ranges fill the CTA slots (few
// output tiles, long K: the layer projections); 1 for wide outputs.
#ifndef OSP_TC_MIN_KB
#define OSP_TC_MIN_KB 1   // k-blocks (of 64) per range at least: fewer, longer ranges write fewer partials
#endif
int tc_nsplit(int nout, int K, int sms) {
    const int tiles = (nout + 127) / 128, nkb = K / 64;
    // at most one item per CTA slot: one item more than the slots would take two
    // item times for barely more than one wave of work
    int want = OSP_TC_CTAS_PER_SM * sms / tiles;
    if (want < 1) want = 1;
    if (want > nkb / OSP_TC_MIN_KB) want = nkb / OSP_TC_MIN_KB > 1 ? nkb / OSP_TC_MIN_KB : 1;
    const int kbps = (nkb + want - 1) / want;
    return (nkb + kbps - 1) / kbps;
}

cudaError_t launch_tc(const TcArgs &a_in, const CUtensorMap &wa, const CUtensorMap &xm, int sms, cudaStream_t s) {
    TcArgs a = a_in;
    a.nout_a = a.nout;
    return launch_tc2(a, wa, wa, xm, sms, s);
}

cudaError_t launch_tc2(const TcArgs &a_in, const CUtensorMap &wa, const CUtensorMap &wb, const CUtensorMap &xm, int sms,
                       cudaStream_t s, bool *planes_done, const QkvPostArgs *rope) {
    TcArgs a = a_in;
    if (planes_done) *planes_done = false;
    if (a.npad % 16 || a.npad < 16 || a.npad > TC_MAX_ROWS || a.K % 64 || a.R > a.npad) return cudaErrorInvalidValue;
    if (a.nout_a < 1 || a.nout_a > a.nout || (a.nout_a < a.nout && a.nout_a % 128)) return cudaErrorInvalidValue;
    if (a.epi == TC_GLU && (a.nout != 2 * a.nout_a || !a.part || !a.h)) return cudaErrorInvalidValue;
    const int nkb = a.K / 64;
    if (a.epi == TC_LM && (!a.lm_part || a.lm_nsub != (a.nout + TC_LM_GROUP - 1) / TC_LM_GROUP))
        return cudaErrorInvalidValue;
    a.nsplit = a.part && a.epi != TC_LM ? tc_nsplit(a.nout, a.K, sms) : 1;   // the LM epilogue needs whole sums
    if ((long long)a.nsplit * a.R * a.nout > a.part_cap) a.nsplit = 1;
    if (a.epi == TC_GLU && (long long)a.nsplit * a.R * a.nout > a.part_cap) return cudaErrorInvalidValue;
    a.kbps = (nkb + a.nsplit - 1) / a.nsplit;
    a.segkb = OSP_TC_SEGKB;
    constexpr int tmem_cols = 512 / OSP_TC_CTAS_PER_SM;
    // the LM head takes OSP_TC_LM_NA weight tiles per stage when two stages fit
    // and the double-buffered accumulators fit TMEM in one segment (the LM head's
    // reduction over d is short: one segment keeps its MMA chain at 4 d / 64 steps
    // per plane)
    int na = 1;
    if (a.epi == TC_LM && OSP_TC_LM_NA > 1 && tc_stages(a.npad, a.planes, OSP_TC_LM_NA) >= 2 &&
        2 * OSP_TC_LM_NA * a.npad <= tmem_cols && a.kbps <= 32) {
        na = OSP_TC_LM_NA;
        a.segkb = a.kbps;
    }
    const int nst = tc_stages(a.npad, a.planes, na);
    if (nst < 2) return cudaErrorInvalidValue;
    const int nseg = (a.kbps + a.segkb - 1) / a.segkb;
    if ((nseg > 1 ? 3 : 2) * na * a.npad > tmem_cols) return cudaErrorInvalidValue;   // TMEM columns
    const int items = (a.nout + 128 * na - 1) / (128 * na) * a.nsplit;
    const int grid = items < OSP_TC_CTAS_PER_SM * sms ? items : OSP_TC_CTAS_PER_SM * sms;
    const size_t smem = tc_smem_bytes(a.npad, a.planes, na);
    cudaError_t e;
    switch (a.epi) {
    case TC_STORE:
        e = pdl_launch(tc_kernel<TC_STORE, 1>, dim3(grid), dim3(TC_THREADS), smem, s, wa, wb, xm, a, nst);
        break;
    case TC_RESID:
        e = pdl_launch(tc_kernel<TC_RESID, 1>, dim3(grid), dim3(TC_THREADS), smem, s, wa, wb, xm, a, nst);
        break;
    case TC_GLU: e = pdl_launch(tc_kernel<TC_GLU, 1>, dim3(grid), dim3(TC_THREADS), smem, s, wa, wb, xm, a, nst); break;
    default:
        e = na > 1
                ? pdl_launch(tc_kernel<TC_LM, OSP_TC_LM_NA>, dim3(grid), dim3(TC_THREADS), smem, s, wa, wb, xm, a, nst)
                : pdl_launch(tc_kernel<TC_LM, 1>, dim3(grid), dim3(TC_THREADS), smem, s, wa, wb, xm, a, nst);
        break;
    }
    if (e != cudaSuccess || (a.nsplit == 1 && a.epi != TC_GLU)) return e;
    if (a.epi == TC_RESID && a.pl_dst && a.nout <= RP_CS * 256 * RP_VPT) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(RP_CS, a.R);
        cfg.blockDim = dim3(256);
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = RP_CS;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 2;
        e = cudaLaunchKernelEx(&cfg, tc_resid_planes_kernel, a);
        count_launch();
        if (e == cudaSuccess && planes_done) *planes_done = true;
        return e;
    }
    if (a.epi == TC_STORE && rope) {
        const long long n = (long long)a.R * (rope->dim.Hq + 2 * rope->dim.Hkv) * (rope->dim.hd / 2);
        e = pdl_launch(tc_reduce_rope_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, a, *rope);
        if (e == cudaSuccess && planes_done) *planes_done = true;
        return e;
    }
    const unsigned rblocks =
        (unsigned)(((long long)a.R * (a.epi == TC_GLU ? a.nout_a : a.nout) + 255) / 256);
    switch (a.epi) {
    case TC_STORE: return pdl_launch(tc_reduce_kernel<TC_STORE>, dim3(rblocks), dim3(256), 0, s, a);
    case TC_RESID: return pdl_launch(tc_reduce_kernel<TC_RESID>, dim3(rblocks), dim3(256), 0, s, a);
    default: return pdl_launch(tc_reduce_kernel<TC_GLU>, dim3(rblocks), dim3(256), 0, s, a);
    }
}

cudaError_t launch_planes(const PlaneArgs &a, cudaStream_t s) {
    return pdl_launch(planes_kernel, dim3(a.R), dim3(256), 0, s, a);
}

cudaError_t launch_qkv_post(const QkvPostArgs &a, cudaStream_t s) {
    const long long n = (long long)a.R * (a.dim.Hq + 2 * a.dim.Hkv) * (a.dim.hd / 2);
    return pdl_launch(qkv_post_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, a);
}

cudaError_t launch_embed_rows(const EmbedArgs &a, cudaStream_t s) {
    return pdl_launch(embed_rows_kernel, dim3(a.R), dim3(256), 0, s, a);
}

cudaError_t launch_lm_pick(const LmPickArgs &a, cudaStream_t s) {
    return pdl_launch(lm_pick_kernel, dim3(a.B), dim3(PK_THREADS), (size_t)a.dim.d * 4, s, a);
}

}  // namespace osp
