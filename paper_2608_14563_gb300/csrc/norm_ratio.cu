// norm_ratio.cu -- the update-magnitude ratio of App. C and the learning rate it
// implies (Sec. C.2): for every target layer l,
//   ||G_l||_F^2, ||W_l||_F^2,
//   r_l  = ||G_l||_F / ||W_l||_F   (fractional weight change per unit learning rate;
//                                   G_l = g~ (x) h in the paper's notation)
//   lr_l = rel / r_l               (the SGD rate whose step is rel ||W_l||_F)
//
// Pass 1: a grid of (blocks, layers) streams G_l and W_l 8 elements per thread per
// step (one 16-byte load for bf16, two for fp32), sums squares in fp32 over runs
// of 128 elements and in fp64 across runs, and reduces each block in fp64.  Pass 2: one
// thread per layer adds its block partials in a fixed order (deterministic) and
// forms r_l and lr_l.  HBM-bound: 2 or 4 bytes of G and of W per element.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "internal.h"

namespace fpo {
namespace {

constexpr int kNrThreads = 256;

struct NrPtrs {
    const void* G[kNrMaxLayers];
    const void* W[kNrMaxLayers];
};

template <typename TT>
__device__ __forceinline__ void load8(const TT* p, float (&v)[8]);

template <>
__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
    const float4 a = __ldcs(reinterpret_cast<const float4*>(p));
    const float4 b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

template <>
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
    const uint4 a = __ldcs(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        v[2 * k] = __uint_as_float(w[k] << 16);
        v[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
    }
}

__device__ __forceinline__ float load1(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float load1(const __nv_bfloat16* p, int64_t i) {
    return __bfloat162float(p[i]);
}

__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

template <typename TG, typename TW>
__global__ void __launch_bounds__(kNrThreads)
    norm_ratio_partial_kernel(const __grid_constant__ NrPtrs ptrs, int64_t n,
                              double* __restrict__ partial) {
    const int layer = blockIdx.y;
    const TG* G = static_cast<const TG*>(ptrs.G[layer]);
    const TW* W = static_cast<const TW*>(ptrs.W[layer]);
    // fp32 over up to 128 elements (8 iterations of two 8-element vectors), then fp64:
    // GB300's fp64 rate is far below what one add per vector would need at HBM speed
    double gg = 0.0, ww = 0.0;
    float a = 0.f, b = 0.f;
    auto add8 = [&](const float (&g)[8], const float (&w)[8]) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            a = fmaf(g[k], g[k], a);
            b = fmaf(w[k], w[k], b);
        }
    };
    const int64_t nvec = n / 8;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * kNrThreads;
    int64_t i = static_cast<int64_t>(blockIdx.x) * kNrThreads + threadIdx.x;
    int since_flush = 0;
    for (; i + stride < nvec; i += 2 * stride) {  // two vectors of each in flight
        float g0[8], w0[8], g1[8], w1[8];
        load8(G + i * 8, g0);
        load8(W + i * 8, w0);
        load8(G + (i + stride) * 8, g1);
        load8(W + (i + stride) * 8, w1);
        add8(g0, w0);
        add8(g1, w1);
        if (++since_flush == 8) {
            gg += a;
            ww += b;
            a = b = 0.f;
            since_flush = 0;
        }
    }
    if (i < nvec) {
        float g0[8], w0[8];
        load8(G + i * 8, g0);
        load8(W + i * 8, w0);
        add8(g0, w0);
    }
    gg += a;
    ww += b;
    if (blockIdx.x == 0) {  // the last n % 8 elements
        const int64_t j = nvec * 8 + threadIdx.x;
        if (j < n) {
            const double g = load1(G, j), w = load1(W, j);
            gg += g * g;
            ww += w * w;
        }
    }
    __shared__ double sh[2][kNrThreads / 32];
    const double sg = warp_sum_d(gg), sw = warp_sum_d(ww);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sh[0][wid] = sg;
        sh[1][wid] = sw;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double x = 0.0, y = 0.0;
        for (int k = 0; k < kNrThreads / 32; ++k) {
            x += sh[0][k];
            y += sh[1][k];
        }
        double* p = partial + (static_cast<size_t>(layer) * gridDim.x + blockIdx.x) * 2;
        p[0] = x;
        p[1] = y;
    }
}

__global__ void norm_ratio_final_kernel(const double* __restrict__ partial, int blocks,
                                        int n_layers, double rel, double* __restrict__ out) {
    const int layer = blockIdx.x * blockDim.x + threadIdx.x;
    if (layer >= n_layers) return;
    const double* p = partial + static_cast<size_t>(layer) * blocks * 2;
    double gg = 0.0, ww = 0.0;
    for (int b = 0; b < blocks; ++b) {
        gg += p[2 * b];
        ww += p[2 * b + 1];
    }
    const double r = sqrt(gg) / sqrt(ww);
    out[4 * layer + 0] = gg;
    out[4 * layer + 1] = ww;
    out[4 * layer + 2] = r;
    out[4 * layer + 3] = rel / r;
}

template <typename TG, typename TW>
cudaError_t run(const NrPtrs& ptrs, int n_layers, int64_t n, int blocks, double rel,
                double* partial, double* out, cudaStream_t st) {
    norm_ratio_partial_kernel<TG, TW>
        <<<dim3(static_cast<unsigned>(blocks), static_cast<unsigned>(n_layers)), kNrThreads, 0,
           st>>>(ptrs, n, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    norm_ratio_final_kernel<<<(n_layers + 63) / 64, 64, 0, st>>>(partial, blocks, n_layers, rel,
                                                                 out);
    return cudaGetLastError();
}

}  // namespace

int norm_ratio_blocks(int n_layers, int64_t n) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    // about 8 resident blocks of 256 threads per SM over all layers, at most one block
    // per 2048 vectors of a layer
    int64_t b = (static_cast<int64_t>(sms) * 8 + n_layers - 1) / n_layers;
    const int64_t cap = (n / 8 + 2047) / 2048;
    if (b > cap) b = cap;
    if (b < 1) b = 1;
    if (b > 1024) b = 1024;
    return static_cast<int>(b);
}

cudaError_t launch_norm_ratio(int g_dtype, int w_dtype, int n_layers, int64_t n,
                              const void* const* G, const void* const* W, double rel,
                              double* partial, int blocks, double* out, cudaStream_t st) {
    if (n_layers < 1 || n_layers > kNrMaxLayers) return cudaErrorInvalidValue;
    NrPtrs ptrs{};
    for (int l = 0; l < n_layers; ++l) {
        ptrs.G[l] = G[l];
        ptrs.W[l] = W[l];
    }
    if (g_dtype == 1 && w_dtype == 0)
        return run<__nv_bfloat16, float>(ptrs, n_layers, n, blocks, rel, partial, out, st);
    if (g_dtype == 0 && w_dtype == 0)
        return run<float, float>(ptrs, n_layers, n, blocks, rel, partial, out, st);
    if (g_dtype == 1 && w_dtype == 1)
        return run<__nv_bfloat16, __nv_bfloat16>(ptrs, n_layers, n, blocks, rel, partial, out,
                                                 st);
    return run<float, __nv_bfloat16>(ptrs, n_layers, n, blocks, rel, partial, out, st);
}

}  // namespace fpo
