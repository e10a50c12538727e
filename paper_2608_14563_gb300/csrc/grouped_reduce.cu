// grouped_reduce.cu -- per-layer reductions over every target layer in one launch
// pair (HBM-bound):
//
//   norm ratio (App. C update-magnitude ratios, Sec. C.2): for G_l, W_l
//     ||G_l||^2, ||W_l||^2, r_l = ||G_l|| / ||W_l|| (fractional weight change per unit
//     learning rate, G_l = g~ (x) h), rel / r_l (the SGD rate of a step rel ||W_l||)
//   cosine (Sec. 2.2, Eq. (cosine)): for X_l, Y_l
//     <X_l, Y_l>, ||X_l||^2, ||Y_l||^2, cos_l  (cos = 0 if a norm is 0)
//
// Pass 1: a grid of (blocks, layers) streams both tensors, four 8-element vectors of
// each per thread in flight (one 16-byte load per vector for bf16, two for fp32),
// sums in fp32 over runs of 128 elements and in fp64 across runs, and reduces each
// block in fp64.  Pass 2: one
// warp per layer adds its block partials in a fixed order (deterministic).
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

// Eight consecutive elements held as loaded (raw), converted to fp32 only when used,
// so that several vectors per thread can be in flight in few registers.
template <typename TT>
struct Raw8;

template <>
struct Raw8<float> {
    float4 a, b;
    __device__ __forceinline__ void load(const float* p) {
        a = __ldcs(reinterpret_cast<const float4*>(p));
        b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
    }
    __device__ __forceinline__ void to(float (&v)[8]) const {
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
};

template <>
struct Raw8<__nv_bfloat16> {
    uint4 a;
    __device__ __forceinline__ void load(const __nv_bfloat16* p) {
        a = __ldcs(reinterpret_cast<const uint4*>(p));
    }
    __device__ __forceinline__ void to(float (&v)[8]) const {
        const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            v[2 * k] = __uint_as_float(w[k] << 16);
            v[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
        }
    }
};

__device__ __forceinline__ float load1(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float load1(const __nv_bfloat16* p, int64_t i) {
    return __bfloat162float(p[i]);
}

__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

template <typename TG, typename TW, bool kDot>
__global__ void __launch_bounds__(kNrThreads)
    grouped_partial_kernel(const __grid_constant__ NrPtrs ptrs, int64_t n,
                           double* __restrict__ partial) {
    const int layer = blockIdx.y;
    const TG* G = static_cast<const TG*>(ptrs.G[layer]);
    const TW* W = static_cast<const TW*>(ptrs.W[layer]);
    // fp32 over runs of at most 128 elements, then fp64: GB300's fp64 rate is far below
    // what one fp64 add per vector would need at HBM speed
    double gg = 0.0, ww = 0.0, gw = 0.0;
    float a = 0.f, b = 0.f, c = 0.f;
    auto add8 = [&](const float (&g)[8], const float (&w)[8]) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            a = fmaf(g[k], g[k], a);
            b = fmaf(w[k], w[k], b);
            if constexpr (kDot) c = fmaf(g[k], w[k], c);
        }
    };
    auto flush = [&]() {
        gg += a;
        ww += b;
        gw += c;
        a = b = c = 0.f;
    };
    constexpr int kU = 4;  // vectors of each tensor in flight per thread
    const int64_t nvec = n / 8;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * kNrThreads;
    int64_t i = static_cast<int64_t>(blockIdx.x) * kNrThreads + threadIdx.x;
    int since_flush = 0;
    for (; i + (kU - 1) * stride < nvec; i += kU * stride) {
        Raw8<TG> rg[kU];
        Raw8<TW> rw[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            rg[u].load(G + (i + u * stride) * 8);
            rw[u].load(W + (i + u * stride) * 8);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            float g0[8], w0[8];
            rg[u].to(g0);
            rw[u].to(w0);
            add8(g0, w0);
        }
        if (++since_flush == 4) {  // 4 x 4 vectors = 128 elements per fp32 run
            flush();
            since_flush = 0;
        }
    }
    flush();
    for (; i < nvec; i += stride) {  // at most kU - 1 vectors left per thread
        Raw8<TG> rg;
        Raw8<TW> rw;
        rg.load(G + i * 8);
        rw.load(W + i * 8);
        float g0[8], w0[8];
        rg.to(g0);
        rw.to(w0);
        add8(g0, w0);
    }
    flush();
    if (blockIdx.x == 0) {  // the last n % 8 elements
        const int64_t j = nvec * 8 + threadIdx.x;
        if (j < n) {
            const double g = load1(G, j), w = load1(W, j);
            gg += g * g;
            ww += w * w;
            gw += g * w;
        }
    }
    __shared__ double sh[3][kNrThreads / 32];
    const double s0 = warp_sum_d(gg), s1 = warp_sum_d(ww), s2 = warp_sum_d(gw);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sh[0][wid] = s0;
        sh[1][wid] = s1;
        sh[2][wid] = s2;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double x = 0.0, y = 0.0, z = 0.0;
        for (int k = 0; k < kNrThreads / 32; ++k) {
            x += sh[0][k];
            y += sh[1][k];
            z += sh[2][k];
        }
        double* p = partial + (static_cast<size_t>(layer) * gridDim.x + blockIdx.x) * 3;
        p[0] = x;
        p[1] = y;
        p[2] = z;
    }
}

// mode 0: norm ratio {gg, ww, r, rel / r};  mode 1: cosine {gw, gg, ww, cos}
// One warp per layer: lane i adds the partials i, i + 32, ... in order, then the lanes'
// sums meet in a fixed butterfly (a fixed order for a given block count).  A single
// thread adding up to a thousand partials in a dependent fp64 chain took ~0.1 ms.
__device__ __forceinline__ double warp_sum_f64(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__global__ void grouped_final_kernel(const double* __restrict__ partial, int blocks,
                                     int n_layers, int mode, double rel,
                                     double* __restrict__ out) {
    const int layer = blockIdx.x;
    const int lane = threadIdx.x;
    const double* p = partial + static_cast<size_t>(layer) * blocks * 3;
    double gg = 0.0, ww = 0.0, gw = 0.0;
    for (int b = lane; b < blocks; b += 32) {
        gg += p[3 * b];
        ww += p[3 * b + 1];
        gw += p[3 * b + 2];
    }
    gg = warp_sum_f64(gg);
    ww = warp_sum_f64(ww);
    gw = warp_sum_f64(gw);
    if (lane != 0) return;
    double* o = out + 4 * layer;
    if (mode == 0) {
        const double r = sqrt(gg) / sqrt(ww);
        o[0] = gg;
        o[1] = ww;
        o[2] = r;
        o[3] = rel / r;
    } else {
        o[0] = gw;
        o[1] = gg;
        o[2] = ww;
        o[3] = (gg > 0.0 && ww > 0.0) ? gw / (sqrt(gg) * sqrt(ww)) : 0.0;
    }
}

template <typename TG, typename TW, bool kDot>
cudaError_t run(const NrPtrs& ptrs, int n_layers, int64_t n, int blocks, int mode, double rel,
                double* partial, double* out, cudaStream_t st) {
    grouped_partial_kernel<TG, TW, kDot>
        <<<dim3(static_cast<unsigned>(blocks), static_cast<unsigned>(n_layers)), kNrThreads, 0,
           st>>>(ptrs, n, partial), ::fpo::note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    grouped_final_kernel<<<n_layers, 32, 0, st>>>(partial, blocks, n_layers, mode, rel, out),
        ::fpo::note_launch();
    return cudaGetLastError();
}

NrPtrs pack(int n_layers, const void* const* G, const void* const* W) {
    NrPtrs ptrs{};
    for (int l = 0; l < n_layers; ++l) {
        ptrs.G[l] = G[l];
        ptrs.W[l] = W[l];
    }
    return ptrs;
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
    const NrPtrs ptrs = pack(n_layers, G, W);
    if (g_dtype == 1 && w_dtype == 0)
        return run<__nv_bfloat16, float, false>(ptrs, n_layers, n, blocks, 0, rel, partial, out,
                                                st);
    if (g_dtype == 0 && w_dtype == 0)
        return run<float, float, false>(ptrs, n_layers, n, blocks, 0, rel, partial, out, st);
    if (g_dtype == 1 && w_dtype == 1)
        return run<__nv_bfloat16, __nv_bfloat16, false>(ptrs, n_layers, n, blocks, 0, rel,
                                                        partial, out, st);
    return run<float, __nv_bfloat16, false>(ptrs, n_layers, n, blocks, 0, rel, partial, out, st);
}

cudaError_t launch_cosine_grouped(int dtype, int n_layers, int64_t n, const void* const* X,
                                  const void* const* Y, double* partial, int blocks, double* out,
                                  cudaStream_t st) {
    if (n_layers < 1 || n_layers > kNrMaxLayers) return cudaErrorInvalidValue;
    const NrPtrs ptrs = pack(n_layers, X, Y);
    if (dtype == 1)
        return run<__nv_bfloat16, __nv_bfloat16, true>(ptrs, n_layers, n, blocks, 1, 0.0,
                                                       partial, out, st);
    return run<float, float, true>(ptrs, n_layers, n, blocks, 1, 0.0, partial, out, st);
}

}  // namespace fpo
