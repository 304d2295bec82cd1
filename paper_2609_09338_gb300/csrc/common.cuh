// Device helpers shared by the draft-step, verify and KV kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "osprey.h"

namespace osp {

constexpr int kWarp = 32;

// ---- bf16 <-> f32 ----------------------------------------------------------
// bf16 is the top half of a binary32, so widening is a shift.
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float bf_to_f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

// binary32 -> bf16, round to nearest even (finite inputs).
__device__ __forceinline__ uint16_t f_to_bf(float x) {
    uint32_t u = __float_as_uint(x);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}
__device__ __forceinline__ uint32_t pack_bf2(float lo, float hi) {
    return (uint32_t)f_to_bf(lo) | ((uint32_t)f_to_bf(hi) << 16);
}

__device__ __forceinline__ void unpack8(const uint4 v, float (&f)[8]) {
    f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
    f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
}

// ---- loads -------------------------------------------------------------------
// Weights and logits are read once per launch: keep them out of L1.
__device__ __forceinline__ uint4 ld_stream(const void *p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}
// Data written by other CTAs of the same launch: read from L2 (bypass L1).
__device__ __forceinline__ float ld_cg(const float *p) { return __ldcg(p); }
__device__ __forceinline__ int ld_cg(const int *p) { return __ldcg(p); }

// ---- warp / block reductions ------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// (max, sum of exp(y - max)) pairs; an empty side has m = -inf, s = 0.
struct MS {
    float m, s;
};
__device__ __forceinline__ MS ms_combine(MS a, MS b) {
    if (a.m == -INFINITY) return b;
    if (b.m == -INFINITY) return a;
    float m = fmaxf(a.m, b.m);
    return {m, a.s * __expf(a.m - m) + b.s * __expf(b.m - m)};
}
__device__ __forceinline__ MS warp_ms(MS v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        MS w{__shfl_xor_sync(0xffffffffu, v.m, o), __shfl_xor_sync(0xffffffffu, v.s, o)};
        v = ms_combine(v, w);
    }
    return v;
}

// argmax with the lowest index on ties
struct AM {
    float v;
    int i;
};
__device__ __forceinline__ AM am_combine(AM a, AM b) {
    if (b.v > a.v || (b.v == a.v && b.i < a.i)) return b;
    return a;
}
__device__ __forceinline__ AM warp_am(AM v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        AM w{__shfl_xor_sync(0xffffffffu, v.v, o), __shfl_xor_sync(0xffffffffu, v.i, o)};
        v = am_combine(v, w);
    }
    return v;
}

// Block-wide reductions; `sh` holds one entry per warp.
__device__ __forceinline__ MS block_ms(MS v, MS *sh) {
    v = warp_ms(v);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) sh[w] = v;
    __syncthreads();
    if (w == 0) {
        MS t = lane < (blockDim.x >> 5) ? sh[lane] : MS{-INFINITY, 0.f};
        t = warp_ms(t);
        if (lane == 0) sh[0] = t;
    }
    __syncthreads();
    MS r = sh[0];
    __syncthreads();
    return r;
}

__device__ __forceinline__ AM block_am(AM v, AM *sh) {
    v = warp_am(v);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) sh[w] = v;
    __syncthreads();
    if (w == 0) {
        AM t = lane < (blockDim.x >> 5) ? sh[lane] : AM{-INFINITY, 0x7fffffff};
        t = warp_am(t);
        if (lane == 0) sh[0] = t;
    }
    __syncthreads();
    AM r = sh[0];
    __syncthreads();
    return r;
}

// Inclusive prefix sum across a warp.
__device__ __forceinline__ float warp_incl_scan(float v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        float n = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += n;
    }
    return v;
}

// Block-wide exclusive prefix of one float per thread (blockDim.x <= 1024, a
// multiple of 32).  Returns the exclusive prefix; *total receives the sum.
// `sh` needs 33 floats of shared memory.
__device__ __forceinline__ float block_excl_scan(float v, float *sh, float *total) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    float inc = warp_incl_scan(v);
    if (lane == 31) sh[w] = inc;
    __syncthreads();
    if (w == 0) {
        float t = lane < nw ? sh[lane] : 0.f;
        float ti = warp_incl_scan(t);
        if (lane < nw) sh[lane] = ti - t;
        if (lane == nw - 1) sh[32] = ti;
    }
    __syncthreads();
    float ex = sh[w] + inc - v;
    *total = sh[32];
    __syncthreads();
    return ex;
}

// ---- "last block to arrive" ticket -------------------------------------------------
// Every block of a group calls this once after publishing its partial results.
// Returns true (in all threads) for exactly one block: the last one.  The
// counter is reset to zero by that block, so the workspace stays reusable.
__device__ __forceinline__ bool arrive_last(int *counter, int total) {
    __shared__ int s_last;
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        int t = atomicAdd(counter, 1);
        s_last = (t == total - 1);
        if (s_last) atomicExch(counter, 0);
    }
    __syncthreads();
    if (s_last) __threadfence();
    return s_last;
}

// cos and sin of the rotary angle pos * inv_freq: the angle is reduced to
// [0, 2 pi) in double (whole turns removed) before the float sincos.
__device__ __forceinline__ void rope_cs2(double inv_freq, int pos, float &c, float &s) {
    const double turns = (double)pos * inv_freq * 0.15915494309189535;
    const double frac = turns - floor(turns);
    sincosf((float)(frac * 6.283185307179586), &s, &c);
}

// One warp: dot of a bf16 weight row with a float32 row, both in shared
// memory.  Lane l takes elements base + 8l .. base + 8l + 7 of every 256-wide
// chunk in ascending order, then a butterfly sum.  Kd is a multiple of 256.
__device__ __forceinline__ float warp_smem_dot(const uint16_t *w, const float *xs, int Kd) {
    const int lane = threadIdx.x & 31;
    float acc = 0.f;
#pragma unroll 4
    for (int base = 0; base < Kd; base += 256) {
        const uint4 wv = *(const uint4 *)(w + base + lane * 8);
        float wf[8];
        unpack8(wv, wf);
        const float4 x0 = *(const float4 *)(xs + base + lane * 8);
        const float4 x1 = *(const float4 *)(xs + base + lane * 8 + 4);
        const float xf[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) acc = fmaf(wf[e], xf[e], acc);
    }
    return warp_sum(acc);
}

__device__ __forceinline__ void set_status(int32_t *status, int code) {
    if (status) atomicCAS((int *)status, 0, code);
}

// Bounds-checked debug build (nvcc -DOSP_BOUNDS=1, e.g. through
// OSPREY_NVCC_DEFINES): OSP_BOUNDS_OK(cond, status) is false when cond fails,
// after writing -(1000 + source line) to the status word (first error wins), and
// the caller skips the access it guards.  A skipped copy leaves its barrier
// short, so the bounded wait on it runs out and the kernel returns.  In the
// default build the macro is the constant true.
#ifndef OSP_BOUNDS
#define OSP_BOUNDS 0
#endif
#if OSP_BOUNDS
#define OSP_BOUNDS_OK(cond, status) ((cond) || (::osp::set_status((status), -1000 - __LINE__), false))
#else
#define OSP_BOUNDS_OK(cond, status) true
#endif

// Bytes of dynamic shared memory the running block was launched with.
__device__ __forceinline__ unsigned dynamic_smem_bytes() {
    unsigned v;
    asm("mov.u32 %0, %%dynamic_smem_size;" : "=r"(v));
    return v;
}

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned *p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release_gpu(unsigned *p, unsigned v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Barrier over every block of a grid whose blocks are all resident at once.
// `count` is zero between uses (the last block to arrive resets it) and `gen`
// advances once per use; a block reads `gen` before arriving, so the release
// cannot be missed.  The wait is bounded (about a second of SM clocks): on
// expiry the status word gets OSPREY_ERR_TIMEOUT and the call returns false in
// every thread of the block, which then stops (after draining its own copies).
// The count may then stay short; the draft call's first kernel zeroes both
// words, so the next call starts clean.
__device__ __forceinline__ bool grid_sync(unsigned *count, unsigned *gen, int32_t *status) {
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        const unsigned g = ld_acquire_gpu(gen);
        __threadfence();   // this block's writes, ordered before the arrival
        if (atomicAdd(count, 1u) == gridDim.x - 1) {
            atomicExch(count, 0u);
            __threadfence();
            st_release_gpu(gen, g + 1u);
        } else {
            const long long t0 = clock64();
            while (ld_acquire_gpu(gen) == g) {
                if (clock64() - t0 > 2000000000LL) {
                    set_status(status, OSPREY_ERR_TIMEOUT);
                    ok = 0;
                    break;
                }
                __nanosleep(64);
            }
        }
        __threadfence();
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
}

}  // namespace osp
