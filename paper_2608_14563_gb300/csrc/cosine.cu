// cosine.cu -- the layer-viability diagnostic's reduction (Sec. 2.2,
// Eq. (cosine)): <X,Y>, ||X||^2, ||Y||^2 and cos over n elements.
//
// Pass 1: a grid of 2 x SM-count blocks streams X and Y with 16-byte loads
// (two vectors per operand in flight per thread), accumulates fp32 partial
// sums per thread, and reduces each block in fp64 to one triple.
// Pass 2: one block adds the triples in a fixed order (deterministic result)
// and forms the cosine.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "internal.h"

namespace fpo {
namespace {

constexpr int kCosThreads = 512;

template <typename TT>
struct CosVec;

template <>
struct CosVec<float> {
    static constexpr int kN = 4;
    __device__ static void load(const float* p, float (&v)[4]) {
        float4 a = __ldcs(reinterpret_cast<const float4*>(p));
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    }
};

template <>
struct CosVec<__nv_bfloat16> {
    static constexpr int kN = 8;
    __device__ static void load(const __nv_bfloat16* p, float (&v)[8]) {
        uint4 a = __ldcs(reinterpret_cast<const uint4*>(p));
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&a);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            float2 f = __bfloat1622float2(h2[k]);
            v[2 * k] = f.x;
            v[2 * k + 1] = f.y;
        }
    }
};

__device__ __forceinline__ float to_float(float x) { return x; }
__device__ __forceinline__ float to_float(__nv_bfloat16 x) { return __bfloat162float(x); }

__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// Block-wide fp64 sum of three values; result valid in thread 0.
__device__ __forceinline__ void block_sum3(double& a, double& b, double& c) {
    __shared__ double sh[3][32];
    a = warp_sum_d(a);
    b = warp_sum_d(b);
    c = warp_sum_d(c);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sh[0][wid] = a;
        sh[1][wid] = b;
        sh[2][wid] = c;
    }
    __syncthreads();
    if (wid == 0) {
        const int nw = blockDim.x >> 5;
        a = lane < nw ? sh[0][lane] : 0.0;
        b = lane < nw ? sh[1][lane] : 0.0;
        c = lane < nw ? sh[2][lane] : 0.0;
        a = warp_sum_d(a);
        b = warp_sum_d(b);
        c = warp_sum_d(c);
    }
}

template <typename TT>
__global__ void __launch_bounds__(kCosThreads)
    cosine_partial_kernel(const TT* __restrict__ X, const TT* __restrict__ Y, int64_t n,
                          double* __restrict__ partial) {
    constexpr int kV = CosVec<TT>::kN;
    float xy = 0.f, xx = 0.f, yy = 0.f;
    const int64_t nvec = n / kV;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    for (; i + stride < nvec; i += 2 * stride) {
        float a0[kV], b0[kV], a1[kV], b1[kV];
        CosVec<TT>::load(X + i * kV, a0);
        CosVec<TT>::load(Y + i * kV, b0);
        CosVec<TT>::load(X + (i + stride) * kV, a1);
        CosVec<TT>::load(Y + (i + stride) * kV, b1);
#pragma unroll
        for (int k = 0; k < kV; ++k) {
            xy = fmaf(a0[k], b0[k], xy);
            xx = fmaf(a0[k], a0[k], xx);
            yy = fmaf(b0[k], b0[k], yy);
        }
#pragma unroll
        for (int k = 0; k < kV; ++k) {
            xy = fmaf(a1[k], b1[k], xy);
            xx = fmaf(a1[k], a1[k], xx);
            yy = fmaf(b1[k], b1[k], yy);
        }
    }
    if (i < nvec) {
        float a0[kV], b0[kV];
        CosVec<TT>::load(X + i * kV, a0);
        CosVec<TT>::load(Y + i * kV, b0);
#pragma unroll
        for (int k = 0; k < kV; ++k) {
            xy = fmaf(a0[k], b0[k], xy);
            xx = fmaf(a0[k], a0[k], xx);
            yy = fmaf(b0[k], b0[k], yy);
        }
    }
    // scalar tail (fewer than kV elements), handled by block 0
    if (blockIdx.x == 0) {
        const int64_t j = nvec * kV + threadIdx.x;
        if (j < n) {
            const float a = to_float(X[j]), b = to_float(Y[j]);
            xy = fmaf(a, b, xy);
            xx = fmaf(a, a, xx);
            yy = fmaf(b, b, yy);
        }
    }
    double dxy = xy, dxx = xx, dyy = yy;
    block_sum3(dxy, dxx, dyy);
    if (threadIdx.x == 0) {
        partial[3 * blockIdx.x + 0] = dxy;
        partial[3 * blockIdx.x + 1] = dxx;
        partial[3 * blockIdx.x + 2] = dyy;
    }
}

__global__ void __launch_bounds__(kCosThreads)
    cosine_final_kernel(const double* __restrict__ partial, int blocks, double* __restrict__ out) {
    double xy = 0.0, xx = 0.0, yy = 0.0;
    for (int b = threadIdx.x; b < blocks; b += blockDim.x) {
        xy += partial[3 * b + 0];
        xx += partial[3 * b + 1];
        yy += partial[3 * b + 2];
    }
    block_sum3(xy, xx, yy);
    if (threadIdx.x == 0) {
        out[0] = xy;
        out[1] = xx;
        out[2] = yy;
        out[3] = (xx > 0.0 && yy > 0.0) ? xy / (sqrt(xx) * sqrt(yy)) : 0.0;
    }
}

}  // namespace

int cosine_blocks(int64_t n) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    const int64_t want = (n + 8LL * kCosThreads - 1) / (8LL * kCosThreads);
    const int64_t cap = 2LL * sms;
    return static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
}

cudaError_t launch_cosine(int dtype, int64_t n, const void* X, const void* Y, double* partial,
                          int blocks, double* out, cudaStream_t st) {
    if (dtype == 1)
        cosine_partial_kernel<__nv_bfloat16><<<blocks, kCosThreads, 0, st>>>(
            static_cast<const __nv_bfloat16*>(X), static_cast<const __nv_bfloat16*>(Y), n, partial),
            ::fpo::note_launch();
    else
        cosine_partial_kernel<float><<<blocks, kCosThreads, 0, st>>>(
            static_cast<const float*>(X), static_cast<const float*>(Y), n, partial),
            ::fpo::note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    cosine_final_kernel<<<1, kCosThreads, 0, st>>>(partial, blocks, out), ::fpo::note_launch();
    return cudaGetLastError();
}

}  // namespace fpo

// ---------------------------------------------------------------------------
// fpo_cosine_noalloc: the same two-pass reduction, for callers that cannot
// allocate device memory (no cudaMalloc, no caching allocator, no caller-side
// workspace), with its scratch -- one fp64 triple of partial sums per block of
// pass 1 -- in a fixed, file-scope device array instead of a workspace.
#include <mutex>

#include "../../include/fpo.h"

namespace fpo {
namespace {

// Partial-sum slots the static scratch holds: pass 1 of a call uses
// cosine_blocks(n) <= 2 x SM count of them (304 on a 152-SM GB300).
constexpr int kNoAllocSlots = 1024;

// 24 KiB of device memory, held by every GPU that loads the library until exit.
static __device__ __align__(256) double g_cosine_noalloc_scratch[3 * kNoAllocSlots];

// Device address of the static scratch per device, once looked up successfully.
std::mutex g_noalloc_mu;
double* g_noalloc_scratch[64] = {};

// Device address of the static scratch on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up with that
// device current.  Only a successful lookup is kept: a failed one (e.g. a first call
// made during a stream capture) is retried on the next call.
cudaError_t noalloc_scratch(double** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_scratch[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_cosine_noalloc_scratch);
        if (e != cudaSuccess) {
            cudaGetLastError();  // leave no sticky-free error behind for the caller
            return e;
        }
        g_noalloc_scratch[dev] = static_cast<double*>(p);
    }
    *out = g_noalloc_scratch[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace fpo

extern "C" int32_t fpo_cosine_noalloc(int64_t n, int32_t dtype, const void* X, const void* Y,
                                      double* out, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n < 0) return FPO_ERR_SHAPE;
    if (!out || (n > 0 && (!X || !Y))) return FPO_ERR_NULL;
    if ((reinterpret_cast<uintptr_t>(X) & 15u) || (reinterpret_cast<uintptr_t>(Y) & 15u) ||
        (reinterpret_cast<uintptr_t>(out) & 7u))
        return FPO_ERR_ALIGN;
    fpo::DevInfo di;
    if (!fpo::current_device_info(&di)) return FPO_ERR_CUDA;
    if (di.major != 10 || di.minor != 3) return FPO_ERR_ARCH;
    const int blocks = fpo::cosine_blocks(n);
    if (blocks > fpo::kNoAllocSlots) return FPO_ERR_WORKSPACE;  // more partials than slots
    double* scratch = nullptr;
    if (fpo::noalloc_scratch(&scratch) != cudaSuccess) return FPO_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (n == 0)
        return cudaMemsetAsync(out, 0, 4 * sizeof(double), st) == cudaSuccess ? FPO_OK
                                                                               : FPO_ERR_CUDA;
    return fpo::launch_cosine(dtype, n, X, Y, scratch, blocks, out, st) == cudaSuccess
               ? FPO_OK
               : FPO_ERR_CUDA;
}
