// rowwise.cu -- bandwidth-bound per-token kernels of the error signal.
//
//   rmsnorm_fwd   rho_t = sqrt(mean_j h_tj^2 + eps), yhat_t = w (.) h_t / rho_t
//                 (the final RMSNorm forward of App. E), plus the target-range
//                 check of every token and, for the direct algorithm, the
//                 anchor c_t = <yhat_t, W_U[y_t]> (the target logit)
//   lse_combine   lse_t from the per-vocabulary-tile (max, sum exp) partials
//   direct_combine  the same, plus the direct algorithm's row factors
//                 alpha_t, beta_t and the list of rows outside the anchor window
//   gather_rows   gathers the yhat rows of those rows for their tensor-core
//                 recomputation anchored at lse_t (gemm_bf16.cu)
//   mean          mean of a vector in a fixed order (the mean cross-entropy)
//   rmsnorm_vjp   App. E Eq. (rmsnorm-vjp) with the min-RMS clamp:
//                 g~ = (w (.) g - xhat <xhat, w (.) g> / d) / max(rho, rho_min)
//
// bf16 rows of up to 8192 elements: one block per row, the row kept in registers
// (each input read once); otherwise one warp per row (two passes over the row),
// 16-byte vector loads, shuffle reductions.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "error_math.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace fpo {
namespace {

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

// Load / store VEC consecutive elements as floats (VEC * sizeof(T) is 16 bytes
// for the vector forms, or VEC = 1).
template <int VEC>
__device__ __forceinline__ void ld_vec(const float* p, float (&v)[VEC]) {
    if constexpr (VEC == 4) {
        float4 a = *reinterpret_cast<const float4*>(p);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    } else if constexpr (VEC == 8) {
        float4 a = *reinterpret_cast<const float4*>(p);
        float4 b = *reinterpret_cast<const float4*>(p + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    } else {
#pragma unroll
        for (int k = 0; k < VEC; ++k) v[k] = p[k];
    }
}

template <int VEC>
__device__ __forceinline__ void ld_vec(const __nv_bfloat16* p, float (&v)[VEC]) {
    static_assert(VEC == 8, "bf16 rows are read 8 elements (16 bytes) at a time");
    uint4 a = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&a);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        float2 f = __bfloat1622float2(h2[k]);
        v[2 * k] = f.x;
        v[2 * k + 1] = f.y;
    }
}

template <int VEC>
__device__ __forceinline__ void st_vec(float* p, const float (&v)[VEC]) {
    if constexpr (VEC == 4) {
        *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    } else {
#pragma unroll
        for (int k = 0; k < VEC; ++k) p[k] = v[k];
    }
}

template <int VEC>
__device__ __forceinline__ void st_vec(__nv_bfloat16* p, const float (&v)[VEC]) {
    static_assert(VEC == 8, "bf16 rows are written 8 elements (16 bytes) at a time");
    uint4 a;
    __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(&a);
#pragma unroll
    for (int k = 0; k < 4; ++k) h2[k] = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
    *reinterpret_cast<uint4*>(p) = a;
}

// x rounded to the storage type TT and back.
template <typename TT>
__device__ __forceinline__ float round_to(float x) {
    if constexpr (sizeof(TT) == 2)
        return __bfloat162float(__float2bfloat16_rn(x));
    else
        return x;
}

constexpr int kRowThreads = 256;  // 8 warps, one row each

template <typename TT, int VEC>
__global__ void __launch_bounds__(kRowThreads)
    rmsnorm_fwd_kernel(const TT* __restrict__ h, const TT* __restrict__ w, int T, int d, float eps,
                       TT* __restrict__ yhat, float* __restrict__ rho, const int32_t* __restrict__ y,
                       int V, unsigned* status, const TT* __restrict__ W_U,
                       float* __restrict__ anchor) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    for (int row = blockIdx.x * wpb + (threadIdx.x >> 5); row < T; row += gridDim.x * wpb) {
        const TT* hr = h + static_cast<size_t>(row) * d;
        const int t = y[row];
        const bool t_ok = t >= 0 && t < V;
        // the target's unembedding row, read only for an in-range target
        const TT* ur = (anchor && t_ok) ? W_U + static_cast<size_t>(t) * d : nullptr;
        float ss = 0.f;
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float x[VEC];
            ld_vec<VEC>(hr + j, x);
#pragma unroll
            for (int k = 0; k < VEC; ++k) ss = fmaf(x[k], x[k], ss);
        }
        ss = warp_sum(ss);
        const float r = sqrtf(ss / static_cast<float>(d) + eps);
        const float inv = 1.0f / r;
        TT* yr = yhat + static_cast<size_t>(row) * d;
        float zt = 0.f;
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float x[VEC], wv[VEC], o[VEC];
            ld_vec<VEC>(hr + j, x);
            ld_vec<VEC>(w + j, wv);
#pragma unroll
            for (int k = 0; k < VEC; ++k) o[k] = wv[k] * (x[k] * inv);
            st_vec<VEC>(yr + j, o);
            if (ur) {
                float u[VEC];
                ld_vec<VEC>(ur + j, u);
#pragma unroll
                for (int k = 0; k < VEC; ++k) zt = fmaf(round_to<TT>(o[k]), u[k], zt);
            }
        }
        if (anchor) zt = warp_sum(zt);
        if (lane == 0) {
            rho[row] = r;
            if (!t_ok) atomicOr(status, kDevTargetRange);
            if (anchor) anchor[row] = zt;
        }
    }
}

// ---------------------------------------------------------------------------
// One block per row (bf16, d <= 256 EPT): the row stays in registers, so each
// input is read from HBM once (the warp-per-row kernels above read the row twice:
// a reduction pass, then the output pass).  Element k of thread j's v-th vector is
// (v * 256 + j) * 8 + i: every vector load of the block is one contiguous 4 KB span.
constexpr int kBlkThreads = 256;

// Block-wide sum of two values; every thread gets both results.
__device__ __forceinline__ float2 block_sum2(float a, float b) {
    __shared__ float2 red[kBlkThreads / 32];
    a = warp_sum(a);
    b = warp_sum(b);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    __syncthreads();  // the previous call's readers are done with red
    if (lane == 0) red[wid] = make_float2(a, b);
    __syncthreads();
    float2 t = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < kBlkThreads / 32; ++i) {
        t.x += red[i].x;
        t.y += red[i].y;
    }
    return t;
}

template <int EPT>
__global__ void __launch_bounds__(kBlkThreads)
    rmsnorm_fwd_row_kernel(const __nv_bfloat16* __restrict__ h, const __nv_bfloat16* __restrict__ w,
                           int T, int d, float eps, __nv_bfloat16* __restrict__ yhat,
                           float* __restrict__ rho, const int32_t* __restrict__ y, int V,
                           unsigned* status, const __nv_bfloat16* __restrict__ W_U,
                           float* __restrict__ anchor) {
    constexpr int NV = EPT / 8;
    for (int row = blockIdx.x; row < T; row += gridDim.x) {
        const __nv_bfloat16* hr = h + static_cast<size_t>(row) * d;
        const int t = y[row];
        const bool t_ok = t >= 0 && t < V;
        // the target's unembedding row, read only for an in-range target, loaded with h
        const __nv_bfloat16* ur = (anchor && t_ok) ? W_U + static_cast<size_t>(t) * d : nullptr;
        uint4 hx[NV], ux[NV];
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            hx[v] = k < d ? *reinterpret_cast<const uint4*>(hr + k) : make_uint4(0, 0, 0, 0);
            ux[v] = (ur && k < d) ? *reinterpret_cast<const uint4*>(ur + k) : make_uint4(0, 0, 0, 0);
        }
        float ss = 0.f;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const uint32_t q4[4] = {hx[v].x, hx[v].y, hx[v].z, hx[v].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float lo = __uint_as_float(q4[q] << 16), hi = __uint_as_float(q4[q] & 0xffff0000u);
                ss = fmaf(lo, lo, ss);
                ss = fmaf(hi, hi, ss);
            }
        }
        const float r = sqrtf(block_sum2(ss, 0.f).x / static_cast<float>(d) + eps);
        const float inv = 1.0f / r;
        __nv_bfloat16* yr = yhat + static_cast<size_t>(row) * d;
        float zt = 0.f;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            if (k < d) {
                float wv[8], o[8];
                ld_vec<8>(w + k, wv);
                const uint32_t q4[4] = {hx[v].x, hx[v].y, hx[v].z, hx[v].w};
                const uint32_t u4[4] = {ux[v].x, ux[v].y, ux[v].z, ux[v].w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    o[2 * q] = wv[2 * q] * (__uint_as_float(q4[q] << 16) * inv);
                    o[2 * q + 1] = wv[2 * q + 1] * (__uint_as_float(q4[q] & 0xffff0000u) * inv);
                    zt = fmaf(round_to<__nv_bfloat16>(o[2 * q]), __uint_as_float(u4[q] << 16), zt);
                    zt = fmaf(round_to<__nv_bfloat16>(o[2 * q + 1]),
                              __uint_as_float(u4[q] & 0xffff0000u), zt);
                }
                st_vec<8>(yr + k, o);
            }
        }
        if (anchor) zt = block_sum2(zt, 0.f).x;
        if (threadIdx.x == 0) {
            rho[row] = r;
            if (!t_ok) atomicOr(status, kDevTargetRange);
            if (anchor) anchor[row] = zt;
        }
    }
}

template <int EPT>
__global__ void __launch_bounds__(kBlkThreads)
    rmsnorm_vjp_row_kernel(const float* __restrict__ g, const __nv_bfloat16* __restrict__ h,
                           const __nv_bfloat16* __restrict__ w, const float* __restrict__ rho,
                           int T, int d, float min_rms, __nv_bfloat16* __restrict__ out) {
    constexpr int NV = EPT / 8;
    for (int row = blockIdx.x; row < T; row += gridDim.x) {
        const float r = rho[row];
        const float inv_r = 1.0f / r;
        const float* gr = g + static_cast<size_t>(row) * d;
        const __nv_bfloat16* hr = h + static_cast<size_t>(row) * d;
        float wg[EPT], xh[EPT];
        float c = 0.f;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            float gv[8], x[8], wv[8];
            if (k < d) {
                ld_vec<8>(gr + k, gv);
                ld_vec<8>(hr + k, x);
                ld_vec<8>(w + k, wv);
            } else {
#pragma unroll
                for (int q = 0; q < 8; ++q) gv[q] = x[q] = wv[q] = 0.f;
            }
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                wg[8 * v + q] = wv[q] * gv[q];
                xh[8 * v + q] = x[q] * inv_r;
                c = fmaf(xh[8 * v + q], wg[8 * v + q], c);
            }
        }
        const float kd = block_sum2(c, 0.f).x / static_cast<float>(d);
        const float pref = 1.0f / fmaxf(r, min_rms);
        __nv_bfloat16* orow = out + static_cast<size_t>(row) * d;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            if (k < d) {
                float o[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) o[q] = (wg[8 * v + q] - xh[8 * v + q] * kd) * pref;
                st_vec<8>(orow + k, o);
            }
        }
    }
}

template <int EPT>
__global__ void __launch_bounds__(kBlkThreads)
    rmsnorm_vjp_at_row_kernel(const __nv_bfloat16* __restrict__ g,
                              const __nv_bfloat16* __restrict__ x,
                              const __nv_bfloat16* __restrict__ gamma, int T, int d, float eps,
                              float min_rms, __nv_bfloat16* __restrict__ out) {
    constexpr int NV = EPT / 8;
    for (int row = blockIdx.x; row < T; row += gridDim.x) {
        const __nv_bfloat16* gr = g + static_cast<size_t>(row) * d;
        const __nv_bfloat16* xr = x + static_cast<size_t>(row) * d;
        float wg[EPT], xv[EPT];
        float ss = 0.f, xg = 0.f;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            float gv[8], xx[8], wv[8];
            if (k < d) {
                ld_vec<8>(gr + k, gv);
                ld_vec<8>(xr + k, xx);
                ld_vec<8>(gamma + k, wv);
            } else {
#pragma unroll
                for (int q = 0; q < 8; ++q) gv[q] = xx[q] = wv[q] = 0.f;
            }
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                wg[8 * v + q] = wv[q] * gv[q];
                xv[8 * v + q] = xx[q];
                ss = fmaf(xx[q], xx[q], ss);
                xg = fmaf(xx[q], wg[8 * v + q], xg);
            }
        }
        const float2 sums = block_sum2(ss, xg);
        const float r = sqrtf(sums.x / static_cast<float>(d) + eps);
        const float inv_r = 1.0f / r;
        const float kd = (sums.y * inv_r) / static_cast<float>(d);
        const float pref = 1.0f / fmaxf(r, min_rms);
        __nv_bfloat16* orow = out + static_cast<size_t>(row) * d;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            if (k < d) {
                float o[8];
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    o[q] = (wg[8 * v + q] - (xv[8 * v + q] * inv_r) * kd) * pref;
                st_vec<8>(orow + k, o);
            }
        }
    }
}

// Elements per thread of the block-per-row kernels for a bf16 row of d, or 0 when
// the row does not fit (the warp-per-row kernels take it).
int row_ept(int d) {
    if (d <= 8 * kBlkThreads) return 8;
    if (d <= 16 * kBlkThreads) return 16;
    if (d <= 32 * kBlkThreads) return 32;
    return 0;
}

int blk_grid(int T) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    return T < sms * 8 ? T : sms * 8;
}

template <typename TT, int VEC>
__global__ void __launch_bounds__(kRowThreads)
    rmsnorm_vjp_kernel(const float* __restrict__ g, const TT* __restrict__ h,
                       const TT* __restrict__ w, const float* __restrict__ rho, int T, int d,
                       float min_rms, TT* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    for (int row = blockIdx.x * wpb + (threadIdx.x >> 5); row < T; row += gridDim.x * wpb) {
        const float r = rho[row];
        const float inv_r = 1.0f / r;
        const float* gr = g + static_cast<size_t>(row) * d;
        const TT* hr = h + static_cast<size_t>(row) * d;
        float c = 0.f;
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float gv[VEC], x[VEC], wv[VEC];
            ld_vec<VEC>(gr + j, gv);
            ld_vec<VEC>(hr + j, x);
            ld_vec<VEC>(w + j, wv);
#pragma unroll
            for (int k = 0; k < VEC; ++k) c = fmaf(x[k] * inv_r, wv[k] * gv[k], c);
        }
        c = warp_sum(c);
        const float kd = c / static_cast<float>(d);
        const float pref = 1.0f / fmaxf(r, min_rms);
        TT* orow = out + static_cast<size_t>(row) * d;
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float gv[VEC], x[VEC], wv[VEC], o[VEC];
            ld_vec<VEC>(gr + j, gv);
            ld_vec<VEC>(hr + j, x);
            ld_vec<VEC>(w + j, wv);
#pragma unroll
            for (int k = 0; k < VEC; ++k) o[k] = (wv[k] * gv[k] - (x[k] * inv_r) * kd) * pref;
            st_vec<VEC>(orow + j, o);
        }
    }
}

// RMSNorm VJP at a norm input x whose rho is recomputed from x: one pass for
// sum x^2 and sum x gamma g, then the output pass (App. E Eq. rmsnorm-vjp).
template <typename TT, int VEC>
__global__ void __launch_bounds__(kRowThreads)
    rmsnorm_vjp_at_kernel(const TT* __restrict__ g, const TT* __restrict__ x,
                          const TT* __restrict__ gamma, int T, int d, float eps, float min_rms,
                          TT* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    for (int row = blockIdx.x * wpb + (threadIdx.x >> 5); row < T; row += gridDim.x * wpb) {
        const TT* gr = g + static_cast<size_t>(row) * d;
        const TT* xr = x + static_cast<size_t>(row) * d;
        float ss = 0.f, xg = 0.f;
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float gv[VEC], xv[VEC], wv[VEC];
            ld_vec<VEC>(gr + j, gv);
            ld_vec<VEC>(xr + j, xv);
            ld_vec<VEC>(gamma + j, wv);
#pragma unroll
            for (int k = 0; k < VEC; ++k) {
                ss = fmaf(xv[k], xv[k], ss);
                xg = fmaf(xv[k], wv[k] * gv[k], xg);
            }
        }
        ss = warp_sum(ss);
        xg = warp_sum(xg);
        const float r = sqrtf(ss / static_cast<float>(d) + eps);
        const float inv_r = 1.0f / r;
        const float kd = (xg * inv_r) / static_cast<float>(d);
        const float pref = 1.0f / fmaxf(r, min_rms);
        TT* orow = out + static_cast<size_t>(row) * d;
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float gv[VEC], xv[VEC], wv[VEC], o[VEC];
            ld_vec<VEC>(gr + j, gv);
            ld_vec<VEC>(xr + j, xv);
            ld_vec<VEC>(gamma + j, wv);
#pragma unroll
            for (int k = 0; k < VEC; ++k) o[k] = (wv[k] * gv[k] - (xv[k] * inv_r) * kd) * pref;
            st_vec<VEC>(orow + j, o);
        }
    }
}

__global__ void __launch_bounds__(kRowThreads)
    lse_combine_kernel(const float2* __restrict__ part, int n_tiles, int T,
                       const float* __restrict__ zy, float* __restrict__ lse, float* __restrict__ ce) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    for (int row = blockIdx.x * wpb + (threadIdx.x >> 5); row < T; row += gridDim.x * wpb) {
        const float2* pr = part + static_cast<size_t>(row) * n_tiles;
        float m = -INFINITY;
        for (int i = lane; i < n_tiles; i += 32) m = fmaxf(m, pr[i].x);
        m = warp_max(m);
        float s = 0.f;
        for (int i = lane; i < n_tiles; i += 32) {
            const float2 p = pr[i];
            if (p.y > 0.f) s += p.y * expf(p.x - m);
        }
        s = warp_sum(s);
        const float l = m + logf(s);
        if (lane == 0) {
            lse[row] = l;
            if (ce) ce[row] = l - zy[row];
        }
    }
}

// Direct algorithm, per token: S_t = sum of the tiles' p~ = exp(z - c_t) (target
// excluded), S'_t the same sum of the bf16-rounded p~ and Qz_t = sum of the rounded
// p~ times z, in a fixed order (fp32; the cancelling difference Qz_t - c_t S'_t and
// the factors in fp64).  The target's own term is exp(0) = 1, so
//   lse_t = c_t + log(1 + S_t),  ce_t = log(1 + S_t),
// and the row factors of the projection are
//   alpha_t = s exp(c_t - lse_t) = s / (1 + S_t),  beta_t = -alpha_t S'_t,
// with the final-norm VJP's row term cv_t = <yhat_t, g_t> = alpha_t (Qz_t - c_t S'_t).
// The anchor window: with c_t the target logit, p~ holds every probability that
// matters as a normal bf16 number, and the projection's fp32 sums stay finite, while
// 2^-80 <= S'_t <= 2^80.  A row outside it (or with a non-finite S'_t) gets
// alpha_t = beta_t = 0 here and is appended to `fix` for the fixup passes, which also
// form its lse and ce; a row with an out-of-range target gets zeros and no fixup.
constexpr double kWindowHi = 1.2089258196146292e24;   // 2^80
constexpr double kWindowLo = 8.271806125530277e-25;  // 2^-80

__global__ void __launch_bounds__(kRowThreads)
    direct_combine_kernel(const float* __restrict__ su, const float* __restrict__ sx,
                          const float* __restrict__ qz, int n_tiles, int T, int V,
                          const int32_t* __restrict__ y,
                          const float* __restrict__ anchor, float s, float* __restrict__ lse,
                          float* __restrict__ ce, float* __restrict__ alpha,
                          float* __restrict__ beta, float* __restrict__ cv,
                          int* __restrict__ fix, int* __restrict__ fix_count) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    for (int row = blockIdx.x * wpb + (threadIdx.x >> 5); row < T; row += gridDim.x * wpb) {
        const float* ur = su + static_cast<size_t>(row) * n_tiles;
        const float* xr = sx + static_cast<size_t>(row) * n_tiles;
        const float* qr = qz + static_cast<size_t>(row) * n_tiles;
        float su_ = 0.f, sx_ = 0.f, q_ = 0.f;
        for (int i = lane; i < n_tiles; i += 32) {
            su_ += ur[i];
            sx_ += xr[i];
            q_ += qr[i];
        }
        const double Su = warp_sum(su_), S = warp_sum(sx_), Q = warp_sum(q_);
        if (lane == 0) {
            const int t = y[row];
            float a = 0.f, b = 0.f, c = 0.f;
            if (t >= 0 && t < V) {
                const bool inside = S <= kWindowHi && (S >= kWindowLo || V == 1);
                if (inside) {
                    const float c_t = anchor[row];
                    const float l1p = log1pf(static_cast<float>(Su));
                    lse[row] = c_t + l1p;
                    if (ce) ce[row] = l1p;
                    a = s / (1.0f + static_cast<float>(Su));
                    b = -a * static_cast<float>(S);
                    c = a * static_cast<float>(Q - static_cast<double>(c_t) * S);
                } else {
                    fix[atomicAdd(fix_count, 1)] = row;
                }
            } else {
                lse[row] = 0.f;
                if (ce) ce[row] = 0.f;
            }
            alpha[row] = a;
            beta[row] = b;
            cv[row] = c;
        }
    }
}

// Rows outside the anchor window: their yhat rows gathered into a compact [count, d]
// matrix for the tensor-core recomputation (16-byte vectors; the row count is read on
// the device, so with no such row the launch returns at once).
__global__ void __launch_bounds__(kRowThreads)
    gather_rows_kernel(const uint4* __restrict__ src, const int* __restrict__ fix,
                       const int* __restrict__ count, int v8, uint4* __restrict__ dst) {
    const long long n = static_cast<long long>(*count) * v8;
    for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
         i += static_cast<long long>(gridDim.x) * blockDim.x) {
        const long long r = i / v8;
        dst[i] = src[static_cast<long long>(fix[r]) * v8 + (i - r * v8)];
    }
}

// lse and ce of the rows outside the anchor window, from the (max, sum exp) partials of
// the first fixup pass: lse = m + log sum_tiles s_i exp(m_i - m), ce = lse - c.
__global__ void __launch_bounds__(kRowThreads)
    direct_fixup_lse_kernel(const float2* __restrict__ part, const int* __restrict__ fix,
                            const int* __restrict__ fix_count, int n_tiles,
                            const float* __restrict__ anchor, float* __restrict__ lse,
                            float* __restrict__ ce) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    const int n = *fix_count;
    for (int i = blockIdx.x * wpb + (threadIdx.x >> 5); i < n; i += gridDim.x * wpb) {
        const int row = fix[i];
        const float2* pr = part + static_cast<size_t>(row) * n_tiles;
        float m = -INFINITY;
        for (int k = lane; k < n_tiles; k += 32) m = fmaxf(m, pr[k].x);
        m = warp_max(m);
        float e = 0.f;
        for (int k = lane; k < n_tiles; k += 32) {
            const float2 p = pr[k];
            if (p.y > 0.f) e += p.y * expf(p.x - m);
        }
        e = warp_sum(e);
        if (lane == 0) {
            const float l = m + logf(e);
            lse[row] = l;
            if (ce) ce[row] = l - anchor[row];
        }
    }
}

// Row factors of the fixed rows (anchored at lse: alpha = s, beta = -s S', and the
// VJP's row term cv = s (Qz - c S')).
__global__ void __launch_bounds__(kRowThreads)
    direct_fixup_factors_kernel(const float* __restrict__ sx, const float* __restrict__ qz,
                                const int* __restrict__ fix, const int* __restrict__ fix_count,
                                int n_tiles, const float* __restrict__ anchor, float s,
                                float* __restrict__ alpha, float* __restrict__ beta,
                                float* __restrict__ cv) {
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    const int n = *fix_count;
    for (int i = blockIdx.x * wpb + (threadIdx.x >> 5); i < n; i += gridDim.x * wpb) {
        const int row = fix[i];
        const float* xr = sx + static_cast<size_t>(row) * n_tiles;
        const float* qr = qz + static_cast<size_t>(row) * n_tiles;
        float sx_ = 0.f, q_ = 0.f;
        for (int k = lane; k < n_tiles; k += 32) {
            sx_ += xr[k];
            q_ += qr[k];
        }
        const double S = warp_sum(sx_), Q = warp_sum(q_);
        if (lane == 0) {
            alpha[row] = s;
            beta[row] = static_cast<float>(-static_cast<double>(s) * S);
            cv[row] = static_cast<float>(static_cast<double>(s) *
                                         (Q - static_cast<double>(anchor[row]) * S));
        }
    }
}

constexpr int kMeanThreads = 1024;

__global__ void __launch_bounds__(kMeanThreads) mean_kernel(const float* __restrict__ x, int n,
                                                            float* __restrict__ out) {
    __shared__ double buf[kMeanThreads];
    double acc = 0.0;
    for (int i = threadIdx.x; i < n; i += kMeanThreads) acc += static_cast<double>(x[i]);
    buf[threadIdx.x] = acc;
    __syncthreads();
    for (int s = kMeanThreads / 2; s > 0; s >>= 1) {
        if (threadIdx.x < s) buf[threadIdx.x] += buf[threadIdx.x + s];
        __syncthreads();
    }
    if (threadIdx.x == 0) out[0] = static_cast<float>(buf[0] / static_cast<double>(n));
}

__global__ void cast_f32_kernel(const float* __restrict__ src, size_t n, __nv_bfloat16* __restrict__ dst) {
    for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<size_t>(gridDim.x) * blockDim.x)
        dst[i] = __float2bfloat16_rn(src[i]);
}

// One block per row (grid-stride over rows): 8 logits per thread per step,
// two 16-byte loads of z and one 16-byte (bf16) or two (fp32) stores of E.
constexpr int kErrThreads = 256;

template <bool kBf16>
__global__ void __launch_bounds__(kErrThreads)
    error_from_logits_kernel(const float* __restrict__ z, const float* __restrict__ lse,
                             const int32_t* __restrict__ y, int M, int V, float s,
                             void* __restrict__ E) {
    for (int row = blockIdx.x; row < M; row += gridDim.x) {
        const float l = lse[row];
        const float l2 = l * kLog2e;
        const int yt = y[row];
        const float* zr = z + static_cast<size_t>(row) * V;
        for (int c = threadIdx.x * 8; c < V; c += kErrThreads * 8) {
            const float4 a = __ldcs(reinterpret_cast<const float4*>(zr + c));
            const float4 b = __ldcs(reinterpret_cast<const float4*>(zr + c + 4));
            const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
            if constexpr (kBf16) {
                uint32_t w[4];
#pragma unroll
                for (int k = 0; k < 8; k += 2)
                    w[k / 2] = pack_bf16x2(error_value(v[k], l2, c + k == yt, s),
                                           error_value(v[k + 1], l2, c + k + 1 == yt, s));
                *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(E) +
                                          static_cast<size_t>(row) * V + c) =
                    make_uint4(w[0], w[1], w[2], w[3]);
            } else {
                float o[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) o[k] = error_value_f32(v[k], l, c + k == yt, s);
                float* dst = static_cast<float*>(E) + static_cast<size_t>(row) * V + c;
                *reinterpret_cast<float4*>(dst) = make_float4(o[0], o[1], o[2], o[3]);
                *reinterpret_cast<float4*>(dst + 4) = make_float4(o[4], o[5], o[6], o[7]);
            }
        }
    }
}

// Scalar variant for fp32 rows whose length is not a multiple of 8.
__global__ void __launch_bounds__(kErrThreads)
    error_from_logits_scalar_kernel(const float* __restrict__ z, const float* __restrict__ lse,
                                    const int32_t* __restrict__ y, int M, int V, float s,
                                    float* __restrict__ E) {
    for (int row = blockIdx.x; row < M; row += gridDim.x) {
        const float l = lse[row];
        const int yt = y[row];
        for (int c = threadIdx.x; c < V; c += kErrThreads)
            E[static_cast<size_t>(row) * V + c] =
                error_value_f32(z[static_cast<size_t>(row) * V + c], l, c == yt, s);
    }
}

// A wait on an mbarrier that no thread arrives on: ends by its time limit.
__global__ void wait_timeout_kernel(unsigned* status, unsigned long long limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const WaitGuard g{&abort_flag, status, limit_ns};
        mbar_wait(smem_u32(&bar), 0, g);
    }
}

int row_grid(int T) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    const int wpb = kRowThreads / 32;
    int blocks = (T + wpb - 1) / wpb;
    const int cap = sms * 8;
    return blocks < cap ? (blocks > 0 ? blocks : 1) : cap;
}

}  // namespace

cudaError_t launch_rmsnorm_fwd(int dtype, const void* h, const void* w, int T, int d, float eps,
                               void* yhat, float* rho, const int32_t* y, int V, unsigned* status,
                               cudaStream_t st, const void* W_U, float* anchor) {
    if (T <= 0) return cudaSuccess;
    const int grid = row_grid(T);
    const int ept = dtype == 1 ? row_ept(d) : 0;
    if (ept) {
        const auto* hh = static_cast<const __nv_bfloat16*>(h);
        const auto* ww = static_cast<const __nv_bfloat16*>(w);
        auto* yy = static_cast<__nv_bfloat16*>(yhat);
        const auto* wu = static_cast<const __nv_bfloat16*>(W_U);
        if (ept == 8)
            rmsnorm_fwd_row_kernel<8><<<blk_grid(T), kBlkThreads, 0, st>>>(
                hh, ww, T, d, eps, yy, rho, y, V, status, wu, anchor), ::fpo::note_launch();
        else if (ept == 16)
            rmsnorm_fwd_row_kernel<16><<<blk_grid(T), kBlkThreads, 0, st>>>(
                hh, ww, T, d, eps, yy, rho, y, V, status, wu, anchor), ::fpo::note_launch();
        else
            rmsnorm_fwd_row_kernel<32><<<blk_grid(T), kBlkThreads, 0, st>>>(
                hh, ww, T, d, eps, yy, rho, y, V, status, wu, anchor), ::fpo::note_launch();
    } else if (dtype == 1) {
        rmsnorm_fwd_kernel<__nv_bfloat16, 8><<<grid, kRowThreads, 0, st>>>(
            static_cast<const __nv_bfloat16*>(h), static_cast<const __nv_bfloat16*>(w), T, d, eps,
            static_cast<__nv_bfloat16*>(yhat), rho, y, V, status,
            static_cast<const __nv_bfloat16*>(W_U), anchor), ::fpo::note_launch();
    } else if (d % 4 == 0) {
        rmsnorm_fwd_kernel<float, 4><<<grid, kRowThreads, 0, st>>>(
            static_cast<const float*>(h), static_cast<const float*>(w), T, d, eps,
            static_cast<float*>(yhat), rho, y, V, status, static_cast<const float*>(W_U), anchor),
            ::fpo::note_launch();
    } else {
        rmsnorm_fwd_kernel<float, 1><<<grid, kRowThreads, 0, st>>>(
            static_cast<const float*>(h), static_cast<const float*>(w), T, d, eps,
            static_cast<float*>(yhat), rho, y, V, status, static_cast<const float*>(W_U), anchor),
            ::fpo::note_launch();
    }
    return cudaGetLastError();
}

cudaError_t launch_direct_combine(const float* su, const float* sx, const float* qz, int n_tiles,
                                  int T, int V, const int32_t* y, const float* anchor, float s,
                                  float* lse, float* ce, float* alpha, float* beta, float* cv,
                                  int* fix, int* fix_count, cudaStream_t st) {
    if (T <= 0) return cudaSuccess;
    direct_combine_kernel<<<row_grid(T), kRowThreads, 0, st>>>(
        su, sx, qz, n_tiles, T, V, y, anchor, s, lse, ce, alpha, beta, cv, fix, fix_count),
        ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const void* yhat, const int* fix, const int* fix_count, int d,
                               void* out, cudaStream_t st) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    gather_rows_kernel<<<4 * sms, kRowThreads, 0, st>>>(static_cast<const uint4*>(yhat), fix,
                                                        fix_count, d / 8, static_cast<uint4*>(out)),
        ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_direct_fixup_lse(const float2* part, const int* fix, const int* fix_count,
                                    int n_tiles, const float* anchor, float* lse, float* ce,
                                    cudaStream_t st) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    direct_fixup_lse_kernel<<<sms, kRowThreads, 0, st>>>(part, fix, fix_count, n_tiles, anchor,
                                                        lse, ce), ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_direct_fixup_factors(const float* sx, const float* qz, const int* fix,
                                        const int* fix_count, int n_tiles, const float* anchor,
                                        float s, float* alpha, float* beta, float* cv,
                                        cudaStream_t st) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    direct_fixup_factors_kernel<<<sms, kRowThreads, 0, st>>>(sx, qz, fix, fix_count, n_tiles,
                                                            anchor, s, alpha, beta, cv),
        ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_rmsnorm_vjp(int dtype, const float* g, const void* h, const void* w,
                               const float* rho, int T, int d, float min_rms, void* out,
                               cudaStream_t st) {
    if (T <= 0) return cudaSuccess;
    const int grid = row_grid(T);
    const int ept = dtype == 1 ? row_ept(d) : 0;
    if (ept) {
        const auto* hh = static_cast<const __nv_bfloat16*>(h);
        const auto* ww = static_cast<const __nv_bfloat16*>(w);
        auto* oo = static_cast<__nv_bfloat16*>(out);
        if (ept == 8)
            rmsnorm_vjp_row_kernel<8><<<blk_grid(T), kBlkThreads, 0, st>>>(g, hh, ww, rho, T, d,
                                                                        min_rms, oo),
                ::fpo::note_launch();
        else if (ept == 16)
            rmsnorm_vjp_row_kernel<16><<<blk_grid(T), kBlkThreads, 0, st>>>(g, hh, ww, rho, T, d,
                                                                         min_rms, oo),
                ::fpo::note_launch();
        else
            rmsnorm_vjp_row_kernel<32><<<blk_grid(T), kBlkThreads, 0, st>>>(g, hh, ww, rho, T, d,
                                                                         min_rms, oo),
                ::fpo::note_launch();
    } else if (dtype == 1) {
        rmsnorm_vjp_kernel<__nv_bfloat16, 8><<<grid, kRowThreads, 0, st>>>(
            g, static_cast<const __nv_bfloat16*>(h), static_cast<const __nv_bfloat16*>(w), rho, T,
            d, min_rms, static_cast<__nv_bfloat16*>(out)), ::fpo::note_launch();
    } else if (d % 4 == 0) {
        rmsnorm_vjp_kernel<float, 4><<<grid, kRowThreads, 0, st>>>(
            g, static_cast<const float*>(h), static_cast<const float*>(w), rho, T, d, min_rms,
            static_cast<float*>(out)), ::fpo::note_launch();
    } else {
        rmsnorm_vjp_kernel<float, 1><<<grid, kRowThreads, 0, st>>>(
            g, static_cast<const float*>(h), static_cast<const float*>(w), rho, T, d, min_rms,
            static_cast<float*>(out)), ::fpo::note_launch();
    }
    return cudaGetLastError();
}

cudaError_t launch_cast_f32(int dtype, const float* src, size_t n, void* dst, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (dtype != 1) return cudaMemcpyAsync(dst, src, n * sizeof(float), cudaMemcpyDeviceToDevice, st);
    cast_f32_kernel<<<row_grid(static_cast<int>((n + 255) / 256 * 8)), kRowThreads, 0, st>>>(
        src, n, static_cast<__nv_bfloat16*>(dst)), ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_error_from_logits(int dtype, const float* z, const float* lse, const int32_t* y,
                                     int M, int V, float s, void* E, cudaStream_t st) {
    if (M <= 0) return cudaSuccess;
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    const int grid = M < sms * 8 ? M : sms * 8;
    if (dtype == 1)
        error_from_logits_kernel<true><<<grid, kErrThreads, 0, st>>>(z, lse, y, M, V, s, E),
            ::fpo::note_launch();
    else if (V % 8 == 0)
        error_from_logits_kernel<false><<<grid, kErrThreads, 0, st>>>(z, lse, y, M, V, s, E),
            ::fpo::note_launch();
    else
        error_from_logits_scalar_kernel<<<grid, kErrThreads, 0, st>>>(z, lse, y, M, V, s,
                                                                      static_cast<float*>(E)),
            ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_wait_timeout(unsigned* status, uint64_t limit_ns, cudaStream_t st) {
    wait_timeout_kernel<<<1, 32, 0, st>>>(status, limit_ns), ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_rmsnorm_vjp_at(int dtype, const void* g, const void* x, const void* gamma,
                                  int T, int d, float eps, float min_rms, void* out,
                                  cudaStream_t st) {
    if (T <= 0) return cudaSuccess;
    const int grid = row_grid(T);
    const int ept = dtype == 1 ? row_ept(d) : 0;
    if (ept) {
        const auto* gg = static_cast<const __nv_bfloat16*>(g);
        const auto* xx = static_cast<const __nv_bfloat16*>(x);
        const auto* ga = static_cast<const __nv_bfloat16*>(gamma);
        auto* oo = static_cast<__nv_bfloat16*>(out);
        if (ept == 8)
            rmsnorm_vjp_at_row_kernel<8><<<blk_grid(T), kBlkThreads, 0, st>>>(gg, xx, ga, T, d, eps,
                                                                           min_rms, oo),
                ::fpo::note_launch();
        else if (ept == 16)
            rmsnorm_vjp_at_row_kernel<16><<<blk_grid(T), kBlkThreads, 0, st>>>(gg, xx, ga, T, d,
                                                                            eps, min_rms, oo),
                ::fpo::note_launch();
        else
            rmsnorm_vjp_at_row_kernel<32><<<blk_grid(T), kBlkThreads, 0, st>>>(gg, xx, ga, T, d,
                                                                            eps, min_rms, oo),
                ::fpo::note_launch();
    } else if (dtype == 1) {
        rmsnorm_vjp_at_kernel<__nv_bfloat16, 8><<<grid, kRowThreads, 0, st>>>(
            static_cast<const __nv_bfloat16*>(g), static_cast<const __nv_bfloat16*>(x),
            static_cast<const __nv_bfloat16*>(gamma), T, d, eps, min_rms,
            static_cast<__nv_bfloat16*>(out)), ::fpo::note_launch();
    } else if (d % 4 == 0) {
        rmsnorm_vjp_at_kernel<float, 4><<<grid, kRowThreads, 0, st>>>(
            static_cast<const float*>(g), static_cast<const float*>(x),
            static_cast<const float*>(gamma), T, d, eps, min_rms, static_cast<float*>(out)),
            ::fpo::note_launch();
    } else {
        rmsnorm_vjp_at_kernel<float, 1><<<grid, kRowThreads, 0, st>>>(
            static_cast<const float*>(g), static_cast<const float*>(x),
            static_cast<const float*>(gamma), T, d, eps, min_rms, static_cast<float*>(out)),
            ::fpo::note_launch();
    }
    return cudaGetLastError();
}

cudaError_t launch_lse_combine(const float2* part, int n_tiles, int T, const float* zy, float* lse,
                               float* ce, cudaStream_t st) {
    if (T <= 0) return cudaSuccess;
    lse_combine_kernel<<<row_grid(T), kRowThreads, 0, st>>>(part, n_tiles, T, zy, lse, ce),
        ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_mean(const float* x, int n, float* out, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    mean_kernel<<<1, kMeanThreads, 0, st>>>(x, n, out), ::fpo::note_launch();
    return cudaGetLastError();
}

}  // namespace fpo
