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
//   layer_signal  the same expression at a layer's post-FFN and / or pre-MLP norm,
//                 composed per target layer (Sec. 3.2); fpo_rmsnorm_vjp runs its
//                 one-norm form
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
template <int THREADS = kBlkThreads>
__device__ __forceinline__ float2 block_sum2(float a, float b) {
    __shared__ float2 red[THREADS / 32];
    a = warp_sum(a);
    b = warp_sum(b);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    __syncthreads();  // the previous call's readers are done with red
    if (lane == 0) red[wid] = make_float2(a, b);
    __syncthreads();
    float2 t = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < THREADS / 32; ++i) {
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
    // h row r and, for an in-range target, the target's unembedding row (the anchor's
    // operand); the next row's are loaded before the current row is computed
    auto load_row = [&](int r, int& t, uint4 (&hx)[NV], uint4 (&ux)[NV]) {
        t = y[r];
        const __nv_bfloat16* hr = h + static_cast<size_t>(r) * d;
        const __nv_bfloat16* ur =
            (anchor && t >= 0 && t < V) ? W_U + static_cast<size_t>(t) * d : nullptr;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * kBlkThreads + threadIdx.x) * 8;
            hx[v] = k < d ? *reinterpret_cast<const uint4*>(hr + k) : make_uint4(0, 0, 0, 0);
            ux[v] = (ur && k < d) ? *reinterpret_cast<const uint4*>(ur + k) : make_uint4(0, 0, 0, 0);
        }
    };
    int t_next = 0;
    uint4 hx_next[NV], ux_next[NV];
    if (blockIdx.x < T) load_row(blockIdx.x, t_next, hx_next, ux_next);
    for (int row = blockIdx.x; row < T; row += gridDim.x) {
        const int t = t_next;
        uint4 hx[NV], ux[NV];
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            hx[v] = hx_next[v];
            ux[v] = ux_next[v];
        }
        if (row + static_cast<int>(gridDim.x) < T)
            load_row(row + gridDim.x, t_next, hx_next, ux_next);
        const bool t_ok = t >= 0 && t < V;
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
    // thread i adds x[i], x[i + kMeanThreads], ... in that order; eight loads are issued
    // before their adds, so the loop waits once per eight elements, not once per element
    constexpr int kBatch = 8;
    double acc = 0.0;
    long long i = threadIdx.x;
    for (; i + (kBatch - 1) * static_cast<long long>(kMeanThreads) < n; i += kBatch * kMeanThreads) {
        float v[kBatch];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) v[k] = x[i + k * kMeanThreads];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) acc += static_cast<double>(v[k]);
    }
    for (; i < n; i += kMeanThreads) acc += static_cast<double>(x[i]);
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

// ---------------------------------------------------------------------------
// Layer-specific signals (Sec. 3.1 step 4, Sec. 3.2, App. E): for target layer l and
// token t, the shared signal g (after the final norm's Jacobian) composed with the
// post-feedforward RMSNorm Jacobian at m_l, then with the pre-MLP one at x_l:
//   u   = (gp (.) g - mhat <mhat, gp (.) g> / d) / max(rho_m, rho_min)    (POST)
//   out = (gq (.) u - xhat <xhat, gq (.) u> / d) / max(rho_x, rho_min)    (PRE)
// Each stage's sums in fp32; u stays in registers (fp32) between the stages.  Grid x
// runs over the layers, grid y over the rows.
constexpr int kSigThreads = 256;  // block size of the block-per-row kernel (512: slower)

struct LayerSignalPtrs {
    const void* m[kNrMaxLayers];
    const void* gp[kNrMaxLayers];
    const void* x[kNrMaxLayers];
    const void* gq[kNrMaxLayers];
    void* out[kNrMaxLayers];
};

// Block-wide sums of N values (warp butterflies, then the warps' partials in order).
template <int N, int THREADS>
__device__ __forceinline__ void block_sum_n(float (&v)[N]) {
    __shared__ float red[THREADS / 32][N];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] = warp_sum(v[i]);
    __syncthreads();  // the previous call's readers are done with red
    if (lane == 0) {
#pragma unroll
        for (int i = 0; i < N; ++i) red[wid][i] = v[i];
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < N; ++i) {
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < THREADS / 32; ++w) t += red[w][i];
        v[i] = t;
    }
}

// This thread's NV 16-byte vectors of a bf16 row (elements (v THREADS + tid) 8 ..),
// zeros past d; converted to fp32 only where used, so that every row the block needs is
// in flight at once.
template <int NV, int THREADS>
__device__ __forceinline__ void ld_row_raw(const __nv_bfloat16* __restrict__ p, int d,
                                           uint4 (&r)[NV]) {
#pragma unroll
    for (int v = 0; v < NV; ++v) {
        const int k = (v * THREADS + threadIdx.x) * 8;
        r[v] = k < d ? __ldg(reinterpret_cast<const uint4*>(p + k)) : make_uint4(0u, 0u, 0u, 0u);
    }
}

__device__ __forceinline__ void raw_to_f32(const uint4& a, float (&v)[8]) {
    const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&a);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 f = __bfloat1622float2(h2[k]);
        v[2 * k] = f.x;
        v[2 * k + 1] = f.y;
    }
}

// Elements 2k, 2k + 1 of a loaded 16-byte bf16 vector as a float pair.
__device__ __forceinline__ float2 bf16x2_at(const uint4& a, int k) {
    const uint32_t w = k == 0 ? a.x : k == 1 ? a.y : k == 2 ? a.z : a.w;
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// One Jacobian stage on a register-held row (block per row): u <- VJP of u at the norm
// input row xr with weight gam (both as loaded), in packed f32x2 arithmetic:
//   a = gam (.) u,  sums <x, x>, <x, a>;  u = a pref - x (inv_r kd pref)
template <int NV, int THREADS>
__device__ __forceinline__ void vjp_stage_row(float (&u)[NV * 8], const uint4 (&xr)[NV],
                                              const uint4 (&gam)[NV], int d, float eps,
                                              float min_rms) {
    float2 sxx = make_float2(0.f, 0.f), sxa = make_float2(0.f, 0.f);
#pragma unroll
    for (int v = 0; v < NV; ++v) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 x2 = bf16x2_at(xr[v], k);
            const float2 a2 = __fmul2_rn(bf16x2_at(gam[v], k), make_float2(u[8 * v + 2 * k],
                                                                           u[8 * v + 2 * k + 1]));
            u[8 * v + 2 * k] = a2.x;
            u[8 * v + 2 * k + 1] = a2.y;
            sxx = __ffma2_rn(x2, x2, sxx);
            sxa = __ffma2_rn(x2, a2, sxa);
        }
    }
    const float2 sums = block_sum2<THREADS>(sxx.x + sxx.y, sxa.x + sxa.y);
    const float r = sqrtf(sums.x / static_cast<float>(d) + eps);
    const float inv_r = 1.0f / r;
    const float kd = (sums.y * inv_r) / static_cast<float>(d);
    const float pref = 1.0f / fmaxf(r, min_rms);
    const float2 P = make_float2(pref, pref);
    const float nc = -(inv_r * kd) * pref;
    const float2 NC = make_float2(nc, nc);
#pragma unroll
    for (int v = 0; v < NV; ++v) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 o = __ffma2_rn(make_float2(u[8 * v + 2 * k], u[8 * v + 2 * k + 1]), P,
                                        __fmul2_rn(bf16x2_at(xr[v], k), NC));
            u[8 * v + 2 * k] = o.x;
            u[8 * v + 2 * k + 1] = o.y;
        }
    }
}

// Stages of rows in flight per block of the block-per-row kernel (shared memory:
// kSigStages x (1 + POST + PRE) rows of d bf16).
constexpr int kSigStages = 3;

// Block per (row, layer), the rows staged in shared memory by cp.async kSigStages - 1
// rows ahead of the one being computed (each thread copies, then reads, the same
// 16-byte chunks, so its own cp.async.wait_group is all the synchronisation the staging
// needs).  The layer's norm weights are held in registers.
template <int EPT, int THREADS, bool POST, bool PRE>
__global__ void __launch_bounds__(THREADS)
    layer_signal_row_kernel(const __nv_bfloat16* __restrict__ g,
                            const __grid_constant__ LayerSignalPtrs p, int T, int d, float eps,
                            float min_rms) {
    constexpr int NV = EPT / 8;
    constexpr int NT = 1 + (POST ? 1 : 0) + (PRE ? 1 : 0);  // staged rows per token
    extern __shared__ __align__(128) uint8_t sig_smem[];
    const int l = blockIdx.x;  // layers fastest: the blocks of all layers of a row are
                               // resident together and share its g row in L2
    const auto* m = static_cast<const __nv_bfloat16*>(p.m[l]);
    const auto* x = static_cast<const __nv_bfloat16*>(p.x[l]);
    auto* out = static_cast<__nv_bfloat16*>(p.out[l]);
    uint4 gp[NV], gq[NV];  // the layer's norm weights, loaded once
    if constexpr (POST) ld_row_raw<NV, THREADS>(static_cast<const __nv_bfloat16*>(p.gp[l]), d, gp);
    if constexpr (PRE) ld_row_raw<NV, THREADS>(static_cast<const __nv_bfloat16*>(p.gq[l]), d, gq);
    const uint32_t sbase = smem_u32(sig_smem);
    const uint32_t row_bytes = static_cast<uint32_t>(d) * 2u;  // a multiple of 16
    auto stage_row = [&](int s, int t) { return sbase + static_cast<uint32_t>(s * NT + t) * row_bytes; };
    auto copy_row = [&](uint32_t dst, const __nv_bfloat16* src) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * THREADS + threadIdx.x) * 8;
            if (k < d) cp_async16(dst + static_cast<uint32_t>(k) * 2u, src + k);
        }
    };
    auto issue = [&](int row, int s) {
        const size_t off = static_cast<size_t>(row) * d;
        copy_row(stage_row(s, 0), g + off);
        if constexpr (POST) copy_row(stage_row(s, 1), m + off);
        if constexpr (PRE) copy_row(stage_row(s, NT - 1), x + off);
    };
    auto read_row = [&](uint32_t src, uint4 (&r)[NV]) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * THREADS + threadIdx.x) * 8;
            if (k < d) {
                asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                             : "=r"(r[v].x), "=r"(r[v].y), "=r"(r[v].z), "=r"(r[v].w)
                             : "r"(src + static_cast<uint32_t>(k) * 2u)
                             : "memory");
            } else {
                r[v] = make_uint4(0u, 0u, 0u, 0u);
            }
        }
    };
    const int G = gridDim.y;
#pragma unroll
    for (int s = 0; s < kSigStages - 1; ++s) {
        const int r = blockIdx.y + s * G;
        if (r < T) issue(r, s);
        cp_async_commit();
    }
    int k_it = 0;
    for (int row = blockIdx.y; row < T; row += G, ++k_it) {
        const int rn = row + (kSigStages - 1) * G;
        if (rn < T) issue(rn, (k_it + kSigStages - 1) % kSigStages);
        cp_async_commit();
        cp_async_wait<kSigStages - 1>();  // this thread's copies of `row` have landed
        const int s = k_it % kSigStages;
        const size_t off = static_cast<size_t>(row) * d;
        uint4 graw[NV], mraw[NV], xraw[NV];
        read_row(stage_row(s, 0), graw);
        if constexpr (POST) read_row(stage_row(s, 1), mraw);
        if constexpr (PRE) read_row(stage_row(s, NT - 1), xraw);
        float u[EPT];
        if constexpr (POST && PRE) {
            // Both stages from one block reduction: with a = gp (.) g and
            // u = (a - m inv1 kd1) pref1, the pre-MLP stage's sum <x, gq (.) u> is
            // pref1 (<x gq, a> - inv1 kd1 <x gq, m>), so all five sums are taken in one
            // pass over the row (one barrier round per row instead of two).
            float2 S[5];
#pragma unroll
            for (int i = 0; i < 5; ++i) S[i] = make_float2(0.f, 0.f);
#pragma unroll
            for (int v = 0; v < NV; ++v) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float2 m2 = bf16x2_at(mraw[v], k), x2 = bf16x2_at(xraw[v], k);
                    const float2 a2 = __fmul2_rn(bf16x2_at(gp[v], k), bf16x2_at(graw[v], k));
                    const float2 b2 = __fmul2_rn(x2, bf16x2_at(gq[v], k));
                    S[0] = __ffma2_rn(m2, m2, S[0]);
                    S[1] = __ffma2_rn(m2, a2, S[1]);
                    S[2] = __ffma2_rn(x2, x2, S[2]);
                    S[3] = __ffma2_rn(b2, a2, S[3]);
                    S[4] = __ffma2_rn(b2, m2, S[4]);
                }
            }
            float s5[5];
#pragma unroll
            for (int i = 0; i < 5; ++i) s5[i] = S[i].x + S[i].y;
            block_sum_n<5, THREADS>(s5);
            const float r1 = sqrtf(s5[0] / static_cast<float>(d) + eps);
            const float inv1 = 1.0f / r1;
            const float kd1 = (s5[1] * inv1) / static_cast<float>(d);
            const float pref1 = 1.0f / fmaxf(r1, min_rms);
            const float r2 = sqrtf(s5[2] / static_cast<float>(d) + eps);
            const float inv2 = 1.0f / r2;
            const float xu = pref1 * (s5[3] - (inv1 * kd1) * s5[4]);
            const float kd2 = (xu * inv2) / static_cast<float>(d);
            const float pref2 = 1.0f / fmaxf(r2, min_rms);
            // u = a pref1 - m (inv1 kd1 pref1);  out = (gq (.) u) pref2 - x (inv2 kd2 pref2)
            const float2 P1 = make_float2(pref1, pref1), P2 = make_float2(pref2, pref2);
            const float c1 = -(inv1 * kd1) * pref1, c2 = -(inv2 * kd2) * pref2;
            const float2 C1 = make_float2(c1, c1), C2 = make_float2(c2, c2);
#pragma unroll
            for (int v = 0; v < NV; ++v) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float2 a2 = __fmul2_rn(bf16x2_at(gp[v], k), bf16x2_at(graw[v], k));
                    const float2 u2 = __ffma2_rn(a2, P1, __fmul2_rn(bf16x2_at(mraw[v], k), C1));
                    const float2 o2 = __ffma2_rn(__fmul2_rn(bf16x2_at(gq[v], k), u2), P2,
                                                 __fmul2_rn(bf16x2_at(xraw[v], k), C2));
                    u[8 * v + 2 * k] = o2.x;
                    u[8 * v + 2 * k + 1] = o2.y;
                }
            }
        } else {
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                float gv[8];
                raw_to_f32(graw[v], gv);
#pragma unroll
                for (int q = 0; q < 8; ++q) u[8 * v + q] = gv[q];
            }
            if constexpr (POST) vjp_stage_row<NV, THREADS>(u, mraw, gp, d, eps, min_rms);
            if constexpr (PRE) vjp_stage_row<NV, THREADS>(u, xraw, gq, d, eps, min_rms);
        }
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int k = (v * THREADS + threadIdx.x) * 8;
            if (k < d) {
                float o[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) o[q] = u[8 * v + q];
                st_vec<8>(out + off + k, o);
            }
        }
    }
    cp_async_wait<0>();
}

// Rows too long for registers, and fp32: one warp per row, three passes over the row
// (the post-FFN sums; the pre-MLP sums over u recomputed elementwise; the output).
template <typename TT, int VEC, bool POST, bool PRE>
__global__ void __launch_bounds__(kRowThreads)
    layer_signal_kernel(const TT* __restrict__ g, const __grid_constant__ LayerSignalPtrs p, int T,
                        int d, float eps, float min_rms) {
    const int l = blockIdx.x;
    const TT* m = static_cast<const TT*>(p.m[l]);
    const TT* gp = static_cast<const TT*>(p.gp[l]);
    const TT* x = static_cast<const TT*>(p.x[l]);
    const TT* gq = static_cast<const TT*>(p.gq[l]);
    TT* out = static_cast<TT*>(p.out[l]);
    const int lane = threadIdx.x & 31;
    const int wpb = blockDim.x >> 5;
    for (int row = blockIdx.y * wpb + (threadIdx.x >> 5); row < T; row += gridDim.y * wpb) {
        const size_t off = static_cast<size_t>(row) * d;
        float inv1 = 0.f, kd1 = 0.f, pref1 = 1.f;
        if constexpr (POST) {
            float ss = 0.f, mg = 0.f;
            for (int j = lane * VEC; j < d; j += 32 * VEC) {
                float gv[VEC], mv[VEC], wv[VEC];
                ld_vec<VEC>(g + off + j, gv);
                ld_vec<VEC>(m + off + j, mv);
                ld_vec<VEC>(gp + j, wv);
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    ss = fmaf(mv[k], mv[k], ss);
                    mg = fmaf(mv[k], wv[k] * gv[k], mg);
                }
            }
            ss = warp_sum(ss);
            mg = warp_sum(mg);
            const float r = sqrtf(ss / static_cast<float>(d) + eps);
            inv1 = 1.0f / r;
            kd1 = (mg * inv1) / static_cast<float>(d);
            pref1 = 1.0f / fmaxf(r, min_rms);
        }
        // u at elements j .. j + VEC - 1 (the post-FFN stage, or g itself)
        auto u_at = [&](int j, float (&u)[VEC]) {
            ld_vec<VEC>(g + off + j, u);
            if constexpr (POST) {
                float mv[VEC], wv[VEC];
                ld_vec<VEC>(m + off + j, mv);
                ld_vec<VEC>(gp + j, wv);
#pragma unroll
                for (int k = 0; k < VEC; ++k) u[k] = (wv[k] * u[k] - (mv[k] * inv1) * kd1) * pref1;
            }
        };
        float inv2 = 0.f, kd2 = 0.f, pref2 = 1.f;
        if constexpr (PRE) {
            float ss = 0.f, xu = 0.f;
            for (int j = lane * VEC; j < d; j += 32 * VEC) {
                float u[VEC], xv[VEC], wv[VEC];
                u_at(j, u);
                ld_vec<VEC>(x + off + j, xv);
                ld_vec<VEC>(gq + j, wv);
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    ss = fmaf(xv[k], xv[k], ss);
                    xu = fmaf(xv[k], wv[k] * u[k], xu);
                }
            }
            ss = warp_sum(ss);
            xu = warp_sum(xu);
            const float r = sqrtf(ss / static_cast<float>(d) + eps);
            inv2 = 1.0f / r;
            kd2 = (xu * inv2) / static_cast<float>(d);
            pref2 = 1.0f / fmaxf(r, min_rms);
        }
        for (int j = lane * VEC; j < d; j += 32 * VEC) {
            float u[VEC];
            u_at(j, u);
            if constexpr (PRE) {
                float xv[VEC], wv[VEC];
                ld_vec<VEC>(x + off + j, xv);
                ld_vec<VEC>(gq + j, wv);
#pragma unroll
                for (int k = 0; k < VEC; ++k) u[k] = (wv[k] * u[k] - (xv[k] * inv2) * kd2) * pref2;
            }
            st_vec<VEC>(out + off + j, u);
        }
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

namespace {

// The block-per-row kernel with its shared-memory size; the limit is raised once per
// instantiation and device to the largest staging it can need (rows of EPT x kSigThreads
// elements).
template <int EPT, bool POST, bool PRE>
cudaError_t launch_sig_rows(dim3 grid, size_t smem, cudaStream_t st, const __nv_bfloat16* g,
                            const LayerSignalPtrs& p, int T, int d, float eps, float min_rms) {
    constexpr auto kern = layer_signal_row_kernel<EPT, kSigThreads, POST, PRE>;
    constexpr int kNT = 1 + (POST ? 1 : 0) + (PRE ? 1 : 0);
    const cudaError_t attr = set_smem_limit<kern>(kSigStages * kNT * EPT * kSigThreads * 2);
    if (attr != cudaSuccess) return attr;
    kern<<<grid, kSigThreads, smem, st>>>(g, p, T, d, eps, min_rms);
    return cudaSuccess;
}

template <bool POST, bool PRE>
cudaError_t run_layer_signals(int dtype, int n_layers, const void* g, const LayerSignalPtrs& p,
                              int T, int d, float eps, float min_rms, cudaStream_t st) {
    DevInfo di;
    const int sms = current_device_info(&di) ? di.sm_count : 148;
    const int per_layer = (sms * 8 + n_layers - 1) / n_layers;  // ~8 blocks per SM in all
    // bf16 rows up to 32 x kSigThreads elements: block per row, the rows in registers
    const int ept = dtype != 1             ? 0
                    : d <= 8 * kSigThreads  ? 8
                    : d <= 16 * kSigThreads ? 16
                    : d <= 32 * kSigThreads ? 32
                                            : 0;
    if (ept) {
        const dim3 grid(static_cast<unsigned>(n_layers),
                        static_cast<unsigned>(T < per_layer ? T : per_layer));
        const auto* gg = static_cast<const __nv_bfloat16*>(g);
        constexpr int kNT = 1 + (POST ? 1 : 0) + (PRE ? 1 : 0);
        const size_t smem = static_cast<size_t>(kSigStages) * kNT * d * 2;
        cudaError_t e = cudaSuccess;
        if (ept == 8)
            e = launch_sig_rows<8, POST, PRE>(grid, smem, st, gg, p, T, d, eps, min_rms);
        else if (ept == 16)
            e = launch_sig_rows<16, POST, PRE>(grid, smem, st, gg, p, T, d, eps, min_rms);
        else
            e = launch_sig_rows<32, POST, PRE>(grid, smem, st, gg, p, T, d, eps, min_rms);
        if (e != cudaSuccess) return e;
    } else {
        const int wpb = kRowThreads / 32;
        const int need = (T + wpb - 1) / wpb;
        const dim3 grid(static_cast<unsigned>(n_layers),
                        static_cast<unsigned>(need < per_layer ? need : per_layer));
        if (dtype == 1)
            layer_signal_kernel<__nv_bfloat16, 8, POST, PRE><<<grid, kRowThreads, 0, st>>>(
                static_cast<const __nv_bfloat16*>(g), p, T, d, eps, min_rms);
        else if (d % 4 == 0)
            layer_signal_kernel<float, 4, POST, PRE><<<grid, kRowThreads, 0, st>>>(
                static_cast<const float*>(g), p, T, d, eps, min_rms);
        else
            layer_signal_kernel<float, 1, POST, PRE><<<grid, kRowThreads, 0, st>>>(
                static_cast<const float*>(g), p, T, d, eps, min_rms);
    }
    ::fpo::note_launch();
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_layer_signals(int dtype, int n_layers, const void* g, const void* const* m,
                                 const void* const* gamma_post, const void* const* x,
                                 const void* const* gamma_pre, void* const* out, int T, int d,
                                 float eps, float min_rms, cudaStream_t st) {
    if (n_layers < 1 || n_layers > kNrMaxLayers || (!m && !x)) return cudaErrorInvalidValue;
    if (T <= 0) return cudaSuccess;
    LayerSignalPtrs p{};
    for (int l = 0; l < n_layers; ++l) {
        p.m[l] = m ? m[l] : nullptr;
        p.gp[l] = m ? gamma_post[l] : nullptr;
        p.x[l] = x ? x[l] : nullptr;
        p.gq[l] = x ? gamma_pre[l] : nullptr;
        p.out[l] = out[l];
    }
    if (m && x) return run_layer_signals<true, true>(dtype, n_layers, g, p, T, d, eps, min_rms, st);
    if (m) return run_layer_signals<true, false>(dtype, n_layers, g, p, T, d, eps, min_rms, st);
    return run_layer_signals<false, true>(dtype, n_layers, g, p, T, d, eps, min_rms, st);
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
