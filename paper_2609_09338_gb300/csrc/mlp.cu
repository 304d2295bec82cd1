// Batch-1 chain steps of the drafter (Sec. 3.3): the layer's O-proj +
// residual, RMSNorm + gate/up + SwiGLU and down + residual as one launch.
#include <math.h>

#include "common.cuh"
#include "draft.cuh"
#include "internal.h"
#include "tma.cuh"

namespace osp {

// Fused O-proj / gate-up / down of one layer for one activation row (batch-1
// chain steps).  Block c owns output rows [o0, o1) of W_o and W_down and
// SwiGLU units [f0, f1) of W_gate / W_up; all four slices are contiguous in
// memory and are requested with one bulk copy each before
// griddepcontrol.wait.  Phases, each ending in a grid barrier:
//   1. x[o] += W_o[o] . attn                  (own rows of the residual)
//   2. n = RMSNorm(x) gamma; h[f] = silu(W_g[f] . n) * (W_u[f] . n)
//   3. x[o] += W_down[o] . h
// Values written by other blocks are read through L2 (ld.global.cg).  Every
// block is resident at once (one per SM; the grid is the SM count).
constexpr int MLP_THREADS = 256;

struct MlpPlan {
    int ro, rf;          // rows per block at most (O / down rows, SwiGLU units)
    size_t smem;
};

static __host__ __device__ MlpPlan mlp_plan(const Dims &D, int grid) {
    MlpPlan p{};
    p.ro = (D.d + grid - 1) / grid;
    p.rf = (D.F + grid - 1) / grid;
    const int Ko = D.Hq * D.hd;
    int act = Ko > D.d ? Ko : D.d;
    act = act > D.F ? act : D.F;
    p.smem = (size_t)p.ro * Ko * 2 + (size_t)2 * p.rf * D.d * 2 + (size_t)p.ro * D.F * 2 + (size_t)act * 4;
    return p;
}

__global__ void __launch_bounds__(MLP_THREADS, 1) mlp_fused_kernel(const MlpArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar[3];
    __shared__ float red[MLP_THREADS / 32];
    const Dims &D = a.dim;
    const int d = D.d, F = D.F, Ko = D.Hq * D.hd;
    const int nb = gridDim.x, c = blockIdx.x;
    const MlpPlan p = mlp_plan(D, nb);
    const int o0 = (int)((long long)d * c / nb), o1 = (int)((long long)d * (c + 1) / nb), no = o1 - o0;
    const int f0 = (int)((long long)F * c / nb), f1 = (int)((long long)F * (c + 1) / nb), nf = f1 - f0;
    uint16_t *wo = (uint16_t *)smem;              // [no][Ko]
    uint16_t *wg = wo + (size_t)p.ro * Ko;        // [nf][d]
    uint16_t *wu = wg + (size_t)p.rf * d;         // [nf][d]
    uint16_t *wd = wu + (size_t)p.rf * d;         // [no][F]
    float *act = (float *)(wd + (size_t)p.ro * F);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int NW = MLP_THREADS / 32;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 3; ++i) mbar_init(&bar[i], 1);
        mbar_fence_init();
        // the weights do not depend on earlier kernels: request them now
        const uint32_t bo = (uint32_t)no * Ko * 2, bf = (uint32_t)nf * d * 2, bd = (uint32_t)no * F * 2;
        const bool fits = OSP_BOUNDS_OK(p.smem <= dynamic_smem_bytes() && no <= p.ro && nf <= p.rf, a.status);
        mbar_arrive_expect_tx(&bar[0], bo);
        if (bo && fits) bulk_g2s(wo, a.W_o + (size_t)o0 * Ko, bo, &bar[0]);
        mbar_arrive_expect_tx(&bar[1], 2 * bf);
        if (bf && fits) {
            bulk_g2s(wg, a.W_gate + (size_t)f0 * d, bf, &bar[1]);
            bulk_g2s(wu, a.W_up + (size_t)f0 * d, bf, &bar[1]);
        }
        mbar_arrive_expect_tx(&bar[2], bd);
        if (bd && fits) bulk_g2s(wd, a.W_down + (size_t)o0 * F, bd, &bar[2]);
    }
    pdl_trigger();
    int b, pos;
    const bool live = a.map.row(0, b, pos);   // the row map was written before the chain
    __syncthreads();
    pdl_wait();   // the attention output and the residual come from earlier kernels
    bool ok = true;

    // 1. O-proj and residual
    if (live)
        for (int i = threadIdx.x * 4; i < Ko; i += MLP_THREADS * 4)
            *(float4 *)(act + i) = __ldcg((const float4 *)(a.attn + i));
    __syncthreads();
    ok = ok && __syncthreads_and(mbar_wait(&bar[0], 0));
    if (ok && live)
        for (int j = warp; j < no; j += NW) {
            const float acc = warp_smem_dot(wo + (size_t)j * Ko, act, Ko);
            if (lane == 0) a.x[o0 + j] = __ldcg(a.x + o0 + j) + acc;
        }
    ok = ok && grid_sync(a.bar_count, a.bar_gen, a.status);   // a block that timed out stops

    // 2. RMSNorm of the whole residual, gate/up and SwiGLU
    if (ok && live) {
        float ss = 0.f;
        for (int i = threadIdx.x * 4; i < d; i += MLP_THREADS * 4) {
            const float4 v = __ldcg((const float4 *)(a.x + i));
            *(float4 *)(act + i) = v;
            ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
        ss = warp_sum(ss);
        if (lane == 0) red[warp] = ss;
        __syncthreads();
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) t += red[w];
        const float inv = rsqrtf(t / (float)d + D.eps);
        for (int i = threadIdx.x; i < d; i += MLP_THREADS) act[i] = act[i] * inv * bf_to_f(a.ffn_norm[i]);
    }
    __syncthreads();
    ok = ok && __syncthreads_and(mbar_wait(&bar[1], 0));
    if (ok && live)
        for (int j = warp; j < nf; j += NW) {
            const float g = warp_smem_dot(wg + (size_t)j * d, act, d);
            const float u = warp_smem_dot(wu + (size_t)j * d, act, d);
            if (lane == 0) a.h[f0 + j] = g / (1.f + expf(-g)) * u;
        }
    ok = ok && grid_sync(a.bar_count, a.bar_gen, a.status);   // a block that timed out stops

    // 3. down and residual
    if (ok && live)
        for (int i = threadIdx.x * 4; i < F; i += MLP_THREADS * 4)
            *(float4 *)(act + i) = __ldcg((const float4 *)(a.h + i));
    __syncthreads();
    ok = ok && __syncthreads_and(mbar_wait(&bar[2], 0));
    if (ok && live)
        for (int j = warp; j < no; j += NW) {
            const float acc = warp_smem_dot(wd + (size_t)j * F, act, F);
            if (lane == 0) a.x[o0 + j] = __ldcg(a.x + o0 + j) + acc;
        }
    if (!ok) {
        if (threadIdx.x == 0) {
            set_status(a.status, OSPREY_ERR_TIMEOUT);
            for (int i = 0; i < 3; ++i) mbar_wait(&bar[i], 0, 200000000LL);   // copies land before exit
        }
        __syncthreads();
    }
}

bool mlp_fused_supported(const Dims &D, int sms) {
    const MlpPlan p = mlp_plan(D, sms);
    int dev = 0, optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    // whole 16-byte vectors everywhere; one block per SM fits
    // (each mbarrier phase counts fewer than 2^20 bytes)
    if (!(D.d % 256 == 0 && D.F % 256 == 0 && (D.Hq * D.hd) % 256 == 0 && p.smem + 1024 <= (size_t)optin &&
          (size_t)p.ro * D.Hq * D.hd * 2 < (1u << 20) && (size_t)p.rf * D.d * 2 * 2 < (1u << 20) &&
          (size_t)p.ro * D.F * 2 < (1u << 20)))
        return false;
    // the grid barriers need every block resident at once: one per SM
    if (allow_smem(mlp_fused_kernel) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return grid_fits_resident(mlp_fused_kernel, MLP_THREADS, p.smem, sms, sms);
}

cudaError_t launch_mlp_fused(const MlpArgs &a, int sms, cudaStream_t s) {
    // the shared-memory opt-in and the residency check ran when the context chose
    // this path (mlp_fused_supported, with the same grid)
    const MlpPlan p = mlp_plan(a.dim, sms);
    cudaError_t e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(sms);
    cfg.blockDim = dim3(MLP_THREADS);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, mlp_fused_kernel, a);
    count_launch();
    return e;
}

}  // namespace osp
