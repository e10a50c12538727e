// optimizer.cu -- the optimizer step of the target layers on their fp32 master
// copies (Sec. 3.1: AdamW with weight decay, SGD with momentum; App. A: fp32
// masters cast to the working dtype, and each step's relative clip to
// clip_frac * ||W||_F, on the step itself or on the gradient).
//
// bf16 with the step clip: the GEMM's epilogue (EpiOptStep) advances the state and leaves
// the unclipped steps and their norm partials to opt_step_scale + opt_step_apply below.
// Otherwise, from the pseudogradients G_l (fp32, written by the grouped GEMM):
//   pass 1  optim_norms    per layer, partial sums of ||W||^2, ||G||^2 and
//                          ||step||^2 (step = the unclipped optimizer step)
//   pass 2  optim_scale    per layer, the clip factor from those sums
//   pass 3  optim_apply    W <- W + s * step(c * G), optimizer state, W_out
// Passes 1-2 are skipped without a clip.  HBM-bound: 16-byte loads, grid of
// blocks x layers, fp32 per thread, fp64 per block, fixed-order reductions.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "internal.h"
#include "optim_math.cuh"

namespace fpo {
namespace {

constexpr int kOptThreads = 256;
constexpr int kOptBlocksPerLayerMax = 512;
constexpr int kMaxLayers = 64;

struct LayerPtrs {
    float* G[kMaxLayers];
    float* W[kMaxLayers];
    void* Wo[kMaxLayers];
    float* s1[kMaxLayers];
    float* s2[kMaxLayers];
};

__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__global__ void __launch_bounds__(kOptThreads)
    optim_norms_kernel(const __grid_constant__ LayerPtrs lp, size_t n, const OptimParams op,
                       double* __restrict__ partials) {
    const int layer = blockIdx.y;
    const float* G = lp.G[layer];
    const float* W = lp.W[layer];
    const float* S1 = lp.s1[layer];
    const float* S2 = lp.s2[layer];
    float ww = 0.f, gg = 0.f, dd = 0.f;
    const size_t stride = static_cast<size_t>(gridDim.x) * kOptThreads;
    for (size_t i = blockIdx.x * static_cast<size_t>(kOptThreads) + threadIdx.x; i < n; i += stride) {
        const float g = G[i], w = W[i];
        float s1 = S1 ? S1[i] : 0.f, s2 = S2 ? S2[i] : 0.f;
        const float st = opt_step(op, g, w, s1, s2);
        ww = fmaf(w, w, ww);
        gg = fmaf(g, g, gg);
        dd = fmaf(st, st, dd);
    }
    __shared__ double sh[3][kOptThreads / 32];
    double a = warp_sum_d(ww), b = warp_sum_d(gg), c = warp_sum_d(dd);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sh[0][wid] = a;
        sh[1][wid] = b;
        sh[2][wid] = c;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double x = 0, y = 0, z = 0;
        for (int k = 0; k < kOptThreads / 32; ++k) {
            x += sh[0][k];
            y += sh[1][k];
            z += sh[2][k];
        }
        double* p = partials + (static_cast<size_t>(layer) * gridDim.x + blockIdx.x) * 3;
        p[0] = x;
        p[1] = y;
        p[2] = z;
    }
}

__global__ void optim_scale_kernel(const double* __restrict__ partials, int blocks,
                                   const OptimParams op, float* __restrict__ scales) {
    const int layer = blockIdx.x;
    if (threadIdx.x != 0) return;
    double ww = 0, gg = 0, dd = 0;
    const double* p = partials + static_cast<size_t>(layer) * blocks * 3;
    for (int b = 0; b < blocks; ++b) {
        ww += p[3 * b];
        gg += p[3 * b + 1];
        dd += p[3 * b + 2];
    }
    const double lim = static_cast<double>(op.clip_frac) * sqrt(ww);
    double s = 1.0;
    if (op.clip == 1 && sqrt(dd) > lim) s = lim / sqrt(dd);
    if (op.clip == 2 && sqrt(gg) > lim) s = lim / sqrt(gg);
    scales[layer] = static_cast<float>(s);
}

template <bool kBf16Out>
__global__ void __launch_bounds__(kOptThreads)
    optim_apply_kernel(const __grid_constant__ LayerPtrs lp, size_t n, const OptimParams op,
                       const float* __restrict__ scales) {
    const int layer = blockIdx.y;
    const float* G = lp.G[layer];
    float* W = lp.W[layer];
    float* S1 = lp.s1[layer];
    float* S2 = lp.s2[layer];
    void* Wo = lp.Wo[layer];
    const float sc = scales ? scales[layer] : 1.f;
    const float gscale = op.clip == 2 ? sc : 1.f;
    const float sscale = op.clip == 1 ? sc : 1.f;
    const size_t stride = static_cast<size_t>(gridDim.x) * kOptThreads;
    for (size_t i = blockIdx.x * static_cast<size_t>(kOptThreads) + threadIdx.x; i < n; i += stride) {
        const float g = gscale * G[i];
        const float w = W[i];
        float s1 = S1 ? S1[i] : 0.f, s2 = S2 ? S2[i] : 0.f;
        const float st = opt_step(op, g, w, s1, s2);
        const float wn = fmaf(sscale, st, w);
        W[i] = wn;
        if (S1) S1[i] = s1;
        if (S2) S2[i] = s2;
        if (Wo) {
            if constexpr (kBf16Out)
                static_cast<__nv_bfloat16*>(Wo)[i] = __float2bfloat16_rn(wn);
            else
                static_cast<float*>(Wo)[i] = wn;
        }
    }
}

// Step clip after the fused epilogue (EpiOptStep): one block per layer adds the layer's
// (||W||^2, ||d||^2) slot pairs in a fixed order (thread-strided fp64 sums, a fixed
// butterfly per warp, then the warps' sums in warp order; 256 threads keep many loads
// in flight, where one warp waited on one load at a time) and writes the layer's scale
// min(1, clip_frac ||W|| / ||d||).
constexpr int kScaleThreads = 256;

__global__ void __launch_bounds__(kScaleThreads)
    opt_step_scale_kernel(const float* __restrict__ part, int slots, const OptimParams op,
                          float* __restrict__ scales) {
    const int layer = blockIdx.x;
    const float2* p = reinterpret_cast<const float2*>(part) + static_cast<size_t>(layer) * slots;
    double ww = 0.0, dd = 0.0;
#pragma unroll 4
    for (int i = threadIdx.x; i < slots; i += kScaleThreads) {
        const float2 v = p[i];
        ww += v.x;
        dd += v.y;
    }
    ww = warp_sum_d(ww);
    dd = warp_sum_d(dd);
    __shared__ double sh[2][kScaleThreads / 32];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sh[0][wid] = ww;
        sh[1][wid] = dd;
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    ww = dd = 0.0;
    for (int k = 0; k < kScaleThreads / 32; ++k) {
        ww += sh[0][k];
        dd += sh[1][k];
    }
    const double lim = static_cast<double>(op.clip_frac) * sqrt(ww);
    scales[layer] = static_cast<float>(sqrt(dd) > lim ? lim / sqrt(dd) : 1.0);
}

// W <- W + s d with the layer's scale, and W_out = bf16(W) (16-byte vectors).
__global__ void __launch_bounds__(kOptThreads)
    opt_step_apply_kernel(const __grid_constant__ LayerPtrs lp, size_t n,
                          const float* __restrict__ scales) {
    const int layer = blockIdx.y;
    const float4* D = reinterpret_cast<const float4*>(lp.G[layer]);
    float4* W = reinterpret_cast<float4*>(lp.W[layer]);
    uint2* Wo = static_cast<uint2*>(lp.Wo[layer]);
    const float s = scales[layer];
    const size_t n4 = n / 4;  // n = d d_ff, a multiple of 8
    const size_t stride = static_cast<size_t>(gridDim.x) * kOptThreads;
    for (size_t i = blockIdx.x * static_cast<size_t>(kOptThreads) + threadIdx.x; i < n4; i += stride) {
        const float4 dv = D[i];
        float4 w = W[i];
        w.x = fmaf(s, dv.x, w.x);
        w.y = fmaf(s, dv.y, w.y);
        w.z = fmaf(s, dv.z, w.z);
        w.w = fmaf(s, dv.w, w.w);
        W[i] = w;
        if (Wo) {
            const __nv_bfloat162 lo = __floats2bfloat162_rn(w.x, w.y);
            const __nv_bfloat162 hi = __floats2bfloat162_rn(w.z, w.w);
            Wo[i] = make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                               *reinterpret_cast<const uint32_t*>(&hi));
        }
    }
}

int blocks_per_layer(int n_layers) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    int b = (sms * 8) / (n_layers > 0 ? n_layers : 1);
    if (b < 1) b = 1;
    return b < kOptBlocksPerLayerMax ? b : kOptBlocksPerLayerMax;
}

}  // namespace

size_t optim_partials_bytes(int n_layers) {
    return static_cast<size_t>(n_layers) * kOptBlocksPerLayerMax * 3 * sizeof(double);
}

cudaError_t launch_optimizer(int dtype, int n_layers, size_t n_elem, const OptimParams& op,
                             float* const* G, float* const* W_master, void* const* W_out,
                             float* const* s1, float* const* s2, double* partials, float* scales,
                             cudaStream_t st) {
    if (n_layers < 1 || n_layers > kMaxLayers) return cudaErrorInvalidValue;
    if (n_elem == 0) return cudaSuccess;
    LayerPtrs lp;
    for (int l = 0; l < kMaxLayers; ++l) {
        const bool in = l < n_layers;
        lp.G[l] = in ? G[l] : nullptr;
        lp.W[l] = in ? W_master[l] : nullptr;
        lp.Wo[l] = in && W_out ? W_out[l] : nullptr;
        lp.s1[l] = in && s1 ? s1[l] : nullptr;
        lp.s2[l] = in && s2 ? s2[l] : nullptr;
    }
    const int bpl = blocks_per_layer(n_layers);
    const dim3 grid(bpl, n_layers);
    if (op.clip != 0) {
        optim_norms_kernel<<<grid, kOptThreads, 0, st>>>(lp, n_elem, op, partials),
            ::fpo::note_launch();
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        optim_scale_kernel<<<n_layers, 32, 0, st>>>(partials, bpl, op, scales),
            ::fpo::note_launch();
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (dtype == 1)
        optim_apply_kernel<true><<<grid, kOptThreads, 0, st>>>(lp, n_elem, op,
                                                               op.clip != 0 ? scales : nullptr),
            ::fpo::note_launch();
    else
        optim_apply_kernel<false><<<grid, kOptThreads, 0, st>>>(lp, n_elem, op,
                                                                op.clip != 0 ? scales : nullptr),
            ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_opt_step_clip(int n_layers, size_t n_elem, const OptimParams& op,
                                 const float* part, int slots, float* const* D,
                                 float* const* W_master, void* const* W_out, float* scales,
                                 cudaStream_t st) {
    if (n_layers < 1 || n_layers > kMaxLayers) return cudaErrorInvalidValue;
    if (n_elem == 0) return cudaSuccess;
    LayerPtrs lp;
    for (int l = 0; l < kMaxLayers; ++l) {
        const bool in = l < n_layers;
        lp.G[l] = in ? D[l] : nullptr;
        lp.W[l] = in ? W_master[l] : nullptr;
        lp.Wo[l] = in && W_out ? W_out[l] : nullptr;
        lp.s1[l] = lp.s2[l] = nullptr;
    }
    opt_step_scale_kernel<<<n_layers, kScaleThreads, 0, st>>>(part, slots, op, scales),
        ::fpo::note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const dim3 grid(blocks_per_layer(n_layers), n_layers);
    opt_step_apply_kernel<<<grid, kOptThreads, 0, st>>>(lp, n_elem, scales), ::fpo::note_launch();
    return cudaGetLastError();
}

}  // namespace fpo
