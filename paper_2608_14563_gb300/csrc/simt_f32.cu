// simt_f32.cu -- true-fp32 (FFMA, no TF32) GEMMs of the FPO step for dtype
// FPO_F32, with the same four epilogues as the tensor-core path:
//
//   C[m, n] = sum_k A(m, k) B(n, k),  A(m,k) = A[m*sam + k*sak], B(n,k) = B[n*sbn + k*sbk]
//
// 64 x 64 output tile per 256-thread block, 16-deep k slices staged in shared
// memory, 4 x 4 outputs per thread; blockIdx.z selects the group (layer).
// Any shape is accepted; every load and store is bounds-checked.
#include <cuda_runtime.h>
#include <math.h>

#include <type_traits>

#include "error_math.cuh"
#include "internal.h"

namespace fpo {
namespace {

constexpr int kT = kSimtTile;  // 64
constexpr int kKs = 16;
constexpr int kThreads = 256;
constexpr int kMaxG = 64;

struct SimtOps {
    const float* A[kMaxG];
    long long sam, sak;
    const float* B[kMaxG];
    long long sbn, sbk;
    int M, N, K;
};

// ------------------------------------------------------------------ epilogues
struct SEpiLse {  // per (row, 64-column tile): (max, sum exp(z - max)) and z_{t,y_t}
    float2* part;
    int part_ld;
    float* zy;
    const int32_t* y;
    float* z;       // [M, ldz] logits for the stored-logits algorithm, or null
    long long ldz;
};
struct SEpiError {  // E = s (exp(z - lse) - [col == y])
    float* E;
    long long ldE;
    const float* lse;
    const int32_t* y;
    float s;
};
struct SEpiStore {
    float* C;
    long long ld;
};
struct SEpiSwiglu {  // dA = e b silu'(a), dB = e silu(a) from e = g W3 and cached a, b
    float* dA;
    float* dB;
    const float* a;
    const float* b;
    long long ld;
};
struct SEpiUpdate {
    float* W_master[kMaxG];
    float* W_out[kMaxG];
    float* G_out[kMaxG];
    long long ld;
    float neg_lr;
};

__device__ __forceinline__ float hmax16(float x) {
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}
__device__ __forceinline__ float hsum16(float x) {
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

template <class Epi>
__global__ void __launch_bounds__(kThreads)
    simt_gemm_kernel(const SimtOps ops, const Epi ep) {
    __shared__ float As[kKs][kT + 4];
    __shared__ float Bs[kKs][kT + 4];
    const int g = blockIdx.z;
    const int m0 = blockIdx.y * kT, n0 = blockIdx.x * kT;
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const float* A = ops.A[g];
    const float* B = ops.B[g];
    float acc[4][4] = {};

    for (int k0 = 0; k0 < ops.K; k0 += kKs) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int idx = tid + kThreads * r;
            int mm, kk;
            if (ops.sak == 1) { kk = idx & 15; mm = idx >> 4; } else { mm = idx & 63; kk = idx >> 6; }
            const int gm = m0 + mm, gk = k0 + kk;
            As[kk][mm] = (gm < ops.M && gk < ops.K) ? A[gm * ops.sam + gk * ops.sak] : 0.f;
            int nn, kb;
            if (ops.sbk == 1) { kb = idx & 15; nn = idx >> 4; } else { nn = idx & 63; kb = idx >> 6; }
            const int gn = n0 + nn, gk2 = k0 + kb;
            Bs[kb][nn] = (gn < ops.N && gk2 < ops.K) ? B[gn * ops.sbn + gk2 * ops.sbk] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kKs; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }

#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int row = m0 + ty * 4 + i;
        const bool rv = row < ops.M;
        if constexpr (std::is_same_v<Epi, SEpiLse>) {
            // all 16 threads sharing this row take part in the reductions
            const int yt = rv ? ep.y[row] : -1;
            float mx = -INFINITY;
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (n0 + tx * 4 + j < ops.N) mx = fmaxf(mx, acc[i][j]);
            mx = hmax16(mx);
            float s = 0.f;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int col = n0 + tx * 4 + j;
                if (col < ops.N) {
                    s += expf(acc[i][j] - mx);
                    if (rv && col == yt && ep.zy) ep.zy[row] = acc[i][j];
                    if (rv && ep.z) ep.z[row * ep.ldz + col] = acc[i][j];
                }
            }
            s = hsum16(s);
            if (rv && tx == 0) ep.part[static_cast<long long>(row) * ep.part_ld + blockIdx.x] = make_float2(mx, s);
        } else {
            if (!rv) continue;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int col = n0 + tx * 4 + j;
                if (col >= ops.N) continue;
                const float v = acc[i][j];
                if constexpr (std::is_same_v<Epi, SEpiError>) {
                    ep.E[row * ep.ldE + col] = error_value_f32(v, ep.lse[row], col == ep.y[row], ep.s);
                } else if constexpr (std::is_same_v<Epi, SEpiStore>) {
                    ep.C[row * ep.ld + col] = v;
                } else if constexpr (std::is_same_v<Epi, SEpiSwiglu>) {
                    const long long off = row * ep.ld + col;
                    const float x = ep.a[off];
                    const float sg = 1.f / (1.f + expf(-x));
                    ep.dA[off] = v * ep.b[off] * sg * fmaf(x, 1.f - sg, 1.f);
                    ep.dB[off] = v * x * sg;
                } else {
                    const long long off = row * ep.ld + col;
                    if (float* wm = ep.W_master[g]) {
                        const float nw = fmaf(ep.neg_lr, v, wm[off]);
                        wm[off] = nw;
                        if (ep.W_out[g]) ep.W_out[g][off] = nw;
                    }
                    if (ep.G_out[g]) ep.G_out[g][off] = v;
                }
            }
        }
    }
}

template <class Epi>
cudaError_t run(const SimtOps& ops, const Epi& ep, int groups, cudaStream_t st) {
    if (ops.M <= 0 || ops.N <= 0) return cudaSuccess;
    dim3 grid((ops.N + kT - 1) / kT, (ops.M + kT - 1) / kT, groups);
    simt_gemm_kernel<Epi><<<grid, kThreads, 0, st>>>(ops, ep), ::fpo::note_launch();
    return cudaGetLastError();
}

SimtOps ops_of(const float* A, long long sam, long long sak, const float* B, long long sbn,
               long long sbk, int M, int N, int K) {
    SimtOps o;
    for (int i = 0; i < kMaxG; ++i) o.A[i] = A;
    o.sam = sam;
    o.sak = sak;
    for (int i = 0; i < kMaxG; ++i) o.B[i] = B;
    o.sbn = sbn;
    o.sbk = sbk;
    o.M = M;
    o.N = N;
    o.K = K;
    return o;
}

}  // namespace

cudaError_t launch_lse_partial_f32(const float* yhat, const float* W_U, const int32_t* y, int T,
                                   int d, int V, float2* part, int part_ld, float* zy, float* z,
                                   cudaStream_t st) {
    SEpiLse ep{part, part_ld, zy, y, z, V};
    return run(ops_of(yhat, d, 1, W_U, d, 1, T, V, d), ep, 1, st);
}

cudaError_t launch_error_f32(const float* yhat, const float* W_U, const int32_t* y,
                             const float* lse, int Tc, int d, int V, float s, float* E,
                             cudaStream_t st) {
    SEpiError ep{E, V, lse, y, s};
    return run(ops_of(yhat, d, 1, W_U, d, 1, Tc, V, d), ep, 1, st);
}

cudaError_t launch_proj_f32(const float* E, const float* W_U, int Tc, int d, int V, float* g,
                            cudaStream_t st) {
    // g[t, j] = sum_v E[t, v] W_U[v, j]: B(n=j, k=v) = W_U[v*d + j]
    SEpiStore ep{g, d};
    return run(ops_of(E, V, 1, W_U, 1, d, Tc, d, V), ep, 1, st);
}

cudaError_t launch_swiglu_f32(int T, int d, int d_ff, const float* g, const float* W3,
                              const float* a, const float* b, float* dA, float* dB,
                              cudaStream_t st) {
    // e[t, f] = sum_j g[t, j] W3[j, f]: A(m=t, k=j) = g[t*d + j], B(n=f, k=j) = W3[j*d_ff + f]
    SEpiSwiglu ep{dA, dB, a, b, d_ff};
    return run(ops_of(g, d, 1, W3, 1, d_ff, T, d_ff, d), ep, 1, st);
}

cudaError_t launch_update_f32(int n, int T, int d, int d_ff, const float* const* g,
                              const float* const* A, float lr, float* const* W_master,
                              float* const* W_out, float* const* G_out, cudaStream_t st) {
    if (n < 1 || n > kMaxG) return cudaErrorInvalidValue;
    // G[i, j] = sum_t g[t, i] A[t, j]: A-operand(m=i, k=t) = g[t*d + i], B(n=j, k=t) = A[t*d_ff + j]
    SimtOps ops = ops_of(g[0], 1, d, A[0], 1, d_ff, d, d_ff, T);
    SEpiUpdate ep;
    for (int l = 0; l < kMaxG; ++l) {
        const bool in = l < n;
        ops.A[l] = in ? g[l] : g[0];
        ops.B[l] = in ? A[l] : A[0];
        ep.W_master[l] = in && W_master ? W_master[l] : nullptr;
        ep.W_out[l] = in && W_out ? W_out[l] : nullptr;
        ep.G_out[l] = in && G_out ? G_out[l] : nullptr;
    }
    ep.ld = d_ff;
    ep.neg_lr = -lr;
    return run(ops, ep, n, st);
}

}  // namespace fpo
