// epilogues.cuh -- per-row epilogues of the tcgen05 GEMM.
//
// Each epilogue thread owns one output row of a 128 x BN tile and receives its
// fp32 accumulator 32 columns at a time: Epi(params, group, row, n0), then
// chunk(params, v[32], col_of_v0, col_offset_in_tile, io) for each 32-column
// chunk in order, then finish(params, n_block).  Rows >= M and columns >= N
// belong to the zero-filled tile overhang and are never written.  Dense
// outputs go through the warp's swizzled staging buffers and TMA stores
// (one 32-row x 128-byte box per store; the TMA engine clips the overhang).
#pragma once

#include <cuda_bf16.h>
#include <math.h>

#include "error_math.cuh"
#include "ptx.cuh"
#include "tc_gemm.cuh"

namespace fpo {

// ---------------------------------------------------------------------------
// Logits pass (Sec. 3.1 step 2): per (row, vocabulary tile) the running max and
// sum of exponentials of z = yhat W_U^T over the tile's valid columns, plus the
// target logit z_{t, y_t} when the target falls inside the tile.  With kStoreZ
// the fp32 logits are also written to z [M, ldz] (stored-logits algorithm).
template <bool kStoreZ>
struct EpiLsePartialT {
    struct Params {
        CUtensorMap zmap;  // fp32 logits [M, N], box 32 x 32 (kStoreZ only)
        float2* part;      // [M, part_ld]: (max, sum exp(z - max)) per vocabulary tile
        int part_ld;
        float* zy;         // [M] target logit, or null
        const int* y;      // [M] targets
        int M, N;
    };
    float m, s, zt;
    int yoff;
    int row;
    bool valid, has_t;

    __device__ __forceinline__ EpiLsePartialT(const Params& p, int, int row_, int n0)
        : m(-INFINITY), s(0.f), zt(0.f), row(row_), has_t(false) {
        valid = row_ < p.M;
        yoff = valid ? __ldg(p.y + row_) - n0 : -1;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int c0,
                                          EpiIO& io) {
        const int lim = p.N - col0;  // valid columns in this chunk (may be <= 0)
        if (lim <= 0) return;
        if constexpr (kStoreZ) {
            if (io.row0 < p.M) {
                const uint32_t buf = out_acquire(io);
                uint32_t w[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) w[j] = __float_as_uint(v[j]);
                out_stage_row(buf, io.lane, w);
                out_commit(io, &p.zmap, buf, col0, io.row0);
            }
        }
        float cm = -INFINITY;
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (j < lim) cm = fmaxf(cm, v[j]);
        const float nm = fmaxf(m, cm);
        const float nml = nm * kLog2e;
        float acc = (m == -INFINITY) ? 0.f : s * ex2_approx(m * kLog2e - nml);
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (j < lim) acc += ex2_approx(fmaf(v[j], kLog2e, -nml));
        s = acc;
        m = nm;
        const int r = yoff - c0;
        if (static_cast<unsigned>(r) < 32u) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (j == r) zt = v[j];
            has_t = true;
        }
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        if (!valid) return;
        p.part[static_cast<long long>(row) * p.part_ld + nb] = make_float2(m, s);
        if (has_t && p.zy) p.zy[row] = zt;
    }
};
using EpiLsePartial = EpiLsePartialT<false>;
using EpiLseStoreZ = EpiLsePartialT<true>;

// ---------------------------------------------------------------------------
// Logits pass of the direct algorithm (Sec. 3.1 step 2 rewritten around a
// per-token anchor c_t): besides the (max, sum exp) partial and the target
// logit of EpiLsePartial, every valid non-target logit leaves
//   p~_tj = exp(z_tj - c_t) = exp(z_tj - m) exp(m - c_t)   (m: the running max)
// rounded to bf16 into P [M, N] (the target column and the overhang are written
// as 0), and the tile's sum of those rounded values, S'_t partial, goes to
// sx [M, part_ld].  Two 32-column chunks fill one 64-column bf16 staging row
// before each TMA store.
struct EpiLseProb {
    struct Params {
        CUtensorMap pmap;     // bf16 P [M, N], box 64 x 32
        float2* part;         // [M, part_ld] (max, sum exp(z - max))
        float* sx;            // [M, part_ld] sum of the rounded p~ of the tile
        int part_ld;
        float* zy;            // [M] target logit, or null
        const int* y;         // [M] targets
        const float* anchor;  // [M] c_t
        int M, N;
    };
    float m, s, zt, sxs, c2;
    int yoff;
    int row;
    bool valid, has_t, pair_out;
    uint32_t w[32];

    __device__ __forceinline__ EpiLseProb(const Params& p, int, int row_, int n0)
        : m(-INFINITY), s(0.f), zt(0.f), sxs(0.f), row(row_), has_t(false), pair_out(false) {
        valid = row_ < p.M;
        yoff = valid ? __ldg(p.y + row_) - n0 : -1;
        c2 = valid ? __ldg(p.anchor + row_) * kLog2e : 0.f;
    }

    // p~ of logits j, j+1 of the chunk from their exponentials e relative to the running
    // max (0 for the target and for columns >= lim, where e is 0), scaled by
    // f = exp(max - c); packed to bf16, the rounded values added to the tile sum.
    __device__ __forceinline__ uint32_t prob_pair(const float (&e)[32], float f, int j, int r) {
        const float a = j != r ? e[j] * f : 0.f;
        const float b = j + 1 != r ? e[j + 1] * f : 0.f;
        const uint32_t pk = pack_bf16x2(a, b);
        sxs += __uint_as_float(pk << 16) + __uint_as_float(pk & 0xffff0000u);
        return pk;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int c0,
                                          EpiIO& io) {
        const bool second = (c0 & 32) != 0;
        if (!second) pair_out = col0 >= p.N || io.row0 >= p.M;
        const int lim = p.N - col0;  // valid columns in this chunk (may be <= 0)
        const int r = yoff - c0;     // target position in this chunk, if in [0, 32)
        float e[32];
        float f = 0.f;
        if (lim > 0) {
            float cm = -INFINITY;
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (j < lim) cm = fmaxf(cm, v[j]);
            const float nm = fmaxf(m, cm);
            const float nml = nm * kLog2e;
            float acc = (m == -INFINITY) ? 0.f : s * ex2_approx(m * kLog2e - nml);
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                e[j] = j < lim ? ex2_approx(fmaf(v[j], kLog2e, -nml)) : 0.f;
                acc += e[j];
            }
            s = acc;
            m = nm;
            f = ex2_approx(nml - c2);
            if (static_cast<unsigned>(r) < 32u) {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (j == r) zt = v[j];
                has_t = true;
            }
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) e[j] = 0.f;
        }
        if (pair_out) return;
        if (!second) {
#pragma unroll
            for (int j = 0; j < 32; j += 2) w[j / 2] = prob_pair(e, f, j, r);
        } else {
#pragma unroll
            for (int j = 0; j < 32; j += 2) w[16 + j / 2] = prob_pair(e, f, j, r);
            const uint32_t buf = out_acquire(io);
            out_stage_row(buf, io.lane, w);
            out_commit(io, &p.pmap, buf, col0 - 32, io.row0);
        }
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        if (!valid) return;
        const long long o = static_cast<long long>(row) * p.part_ld + nb;
        p.part[o] = make_float2(m, s);
        p.sx[o] = sxs;
        if (has_t && p.zy) p.zy[row] = zt;
    }
};

// ---------------------------------------------------------------------------
// Direct algorithm, rows outside the anchor window (Sec. 3.1 step 2 with the
// anchor at lse_t): the GEMM's rows are the yhat rows gathered from fix[0, count);
// each logit z of such a row becomes p~ = exp(z - lse_t), 0 at the target,
// rounded to bf16 and stored into that row of P with plain 16-byte stores; the
// row's sum of the rounded values over the tile goes to sx[row, tile].
struct EpiFixProb {
    struct Params {
        __nv_bfloat16* P;    // [T, N] rows of the chunk, row stride N
        float* sx;           // [T, n_tiles]
        const int* fix;      // gathered row -> row of the chunk
        const int* count;    // gathered rows (device)
        const int32_t* y;    // [T] targets
        const float* lse;    // [T]
        int n_tiles, N;
    };
    int orig, yt;
    float lse2, sxs;
    bool valid;

    __device__ __forceinline__ EpiFixProb(const Params& p, int, int row_, int) : sxs(0.f) {
        valid = row_ < *p.count;
        orig = valid ? p.fix[row_] : 0;
        yt = valid ? p.y[orig] : -1;
        lse2 = valid ? p.lse[orig] * kLog2e : 0.f;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO&) {
        const int lim = p.N - col0;  // valid columns of the chunk
        if (!valid || lim <= 0) return;
        const int r = yt - col0;
        uint32_t w[16];
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const float a = (j < lim && j != r) ? ex2_approx(fmaf(v[j], kLog2e, -lse2)) : 0.f;
            const float b =
                (j + 1 < lim && j + 1 != r) ? ex2_approx(fmaf(v[j + 1], kLog2e, -lse2)) : 0.f;
            const uint32_t pk = pack_bf16x2(a, b);
            sxs += __uint_as_float(pk << 16) + __uint_as_float(pk & 0xffff0000u);
            w[j / 2] = pk;
        }
        uint4* dst = reinterpret_cast<uint4*>(p.P + static_cast<size_t>(orig) * p.N + col0);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (q * 8 < lim) dst[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        if (valid) p.sx[static_cast<size_t>(orig) * p.n_tiles + nb] = sxs;
    }
};

// ---------------------------------------------------------------------------
// Recompute pass (Sec. 3.1 step 2): e = s (exp(z - lse) - [col == y]) rounded
// to bf16 into the error matrix E [M, N]; two 32-column chunks fill one
// 64-column bf16 staging row before each TMA store.
struct EpiError {
    struct Params {
        CUtensorMap Emap;  // bf16 E [M, N], box 64 x 32
        const float* lse;  // [M]
        const int* y;      // [M]
        int M, N;
        float s;
    };
    int row, yt;
    float lse2;
    bool pair_out;  // the current 64-column pair lies beyond N
    uint32_t w[32];

    __device__ __forceinline__ EpiError(const Params& p, int, int row_, int) : row(row_) {
        const bool valid = row_ < p.M;
        yt = valid ? __ldg(p.y + row_) : -1;
        lse2 = valid ? __ldg(p.lse + row_) * kLog2e : 0.f;
        pair_out = false;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int c0,
                                          EpiIO& io) {
        const bool second = (c0 & 32) != 0;
        if (!second) pair_out = col0 >= p.N || io.row0 >= p.M;
        if (pair_out) return;
        if (!second) {
#pragma unroll
            for (int j = 0; j < 32; j += 2)
                w[j / 2] = pack_bf16x2(error_value(v[j], lse2, col0 + j == yt, p.s),
                                       error_value(v[j + 1], lse2, col0 + j + 1 == yt, p.s));
        } else {
#pragma unroll
            for (int j = 0; j < 32; j += 2)
                w[16 + j / 2] = pack_bf16x2(error_value(v[j], lse2, col0 + j == yt, p.s),
                                            error_value(v[j + 1], lse2, col0 + j + 1 == yt, p.s));
            const uint32_t buf = out_acquire(io);
            out_stage_row(buf, io.lane, w);
            out_commit(io, &p.Emap, buf, col0 - 32, io.row0);
        }
    }

    __device__ __forceinline__ void finish(const Params&, int) {}
};

// ---------------------------------------------------------------------------
// Plain fp32 store of C [M, N]: the projection g = E W_U (Eq. gproj).
struct EpiStoreF32 {
    struct Params {
        CUtensorMap Cmap;  // fp32 C [M, N], box 32 x 32
        int M, N;
    };

    __device__ __forceinline__ EpiStoreF32(const Params&, int, int, int) {}

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO& io) {
        if (col0 >= p.N || io.row0 >= p.M) return;
        const uint32_t buf = out_acquire(io);
        uint32_t w[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) w[j] = __float_as_uint(v[j]);
        out_stage_row(buf, io.lane, w);
        out_commit(io, &p.Cmap, buf, col0, io.row0);
    }

    __device__ __forceinline__ void finish(const Params&, int) {}
};

// ---------------------------------------------------------------------------
// Projection of the direct algorithm: with acc = P W_U (target column of P
// zero), the unnormalised error signal of token t is
//   g_t = alpha_t acc_t + beta_t W_U[y_t],   alpha_t = s exp(c_t - lse_t),
//   beta_t = -alpha_t S'_t,
// which is s (softmax(z_t) - 1_{y_t}) W_U written with the anchor c_t.  A row
// with alpha_t == 0 is written as zeros (rows the fixup kernel recomputes, or
// s == 0); beta_t == 0 skips the read of the target's W_U row.
struct EpiProjDirect {
    struct Params {
        CUtensorMap Cmap;  // fp32 g [M, N], box 32 x 32
        const float* alpha;
        const float* beta;
        const int* y;
        const __nv_bfloat16* W_U;  // [V, N]
        int M, N;
    };
    float a, b;
    const __nv_bfloat16* wy;

    __device__ __forceinline__ EpiProjDirect(const Params& p, int, int row, int) {
        const bool valid = row < p.M;
        a = valid ? __ldg(p.alpha + row) : 0.f;
        b = valid ? __ldg(p.beta + row) : 0.f;
        wy = (a != 0.f && b != 0.f) ? p.W_U + static_cast<long long>(__ldg(p.y + row)) * p.N
                                    : nullptr;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO& io) {
        if (col0 >= p.N || io.row0 >= p.M) return;
        const int lim = p.N - col0;  // a multiple of 8: N % 8 == 0 and col0 % 32 == 0
        uint32_t o[32];
        if (a == 0.f) {
#pragma unroll
            for (int j = 0; j < 32; ++j) o[j] = 0u;
        } else if (wy) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint4 u = make_uint4(0, 0, 0, 0);
                if (q * 8 < lim) u = __ldg(reinterpret_cast<const uint4*>(wy + col0) + q);
                const uint32_t h[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int j = 8 * q + 2 * k;
                    o[j] = __float_as_uint(fmaf(a, v[j], b * __uint_as_float(h[k] << 16)));
                    o[j + 1] =
                        __float_as_uint(fmaf(a, v[j + 1], b * __uint_as_float(h[k] & 0xffff0000u)));
                }
            }
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) o[j] = __float_as_uint(a * v[j]);
        }
        const uint32_t buf = out_acquire(io);
        out_stage_row(buf, io.lane, o);
        out_commit(io, &p.Cmap, buf, col0, io.row0);
    }

    __device__ __forceinline__ void finish(const Params&, int) {}
};

// ---------------------------------------------------------------------------
// Pseudogradient update (Eq. w3update, App. A): for group (layer) g,
//   W_master[g] -= lr * G ;  W_out[g] = bf16(W_master[g]) ;  G_out[g] = bf16(G)
// Any of the three pointers may be null for a layer.
struct EpiUpdate {
    struct Params {
        float* W_master[kMaxGroups];
        __nv_bfloat16* W_out[kMaxGroups];
        __nv_bfloat16* G_out[kMaxGroups];
        long long ld;
        int M, N;
        float neg_lr;
    };
    int row, g;
    bool valid;

    __device__ __forceinline__ EpiUpdate(const Params& p, int g_, int row_, int) : row(row_), g(g_) {
        valid = row_ < p.M;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO&) {
        const int lim = p.N - col0;
        if (!valid || lim <= 0) return;
        const long long off = row * p.ld + col0;
        float* wm = p.W_master[g];
        __nv_bfloat16* wo = p.W_out[g];
        __nv_bfloat16* go = p.G_out[g];
        if (wm) {
            float4* wp = reinterpret_cast<float4*>(wm + off);
            uint4* op = reinterpret_cast<uint4*>(wo + off);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (q * 8 >= lim) break;
                float4 a = wp[2 * q], b = wp[2 * q + 1];
                a.x = fmaf(p.neg_lr, v[8 * q + 0], a.x);
                a.y = fmaf(p.neg_lr, v[8 * q + 1], a.y);
                a.z = fmaf(p.neg_lr, v[8 * q + 2], a.z);
                a.w = fmaf(p.neg_lr, v[8 * q + 3], a.w);
                b.x = fmaf(p.neg_lr, v[8 * q + 4], b.x);
                b.y = fmaf(p.neg_lr, v[8 * q + 5], b.y);
                b.z = fmaf(p.neg_lr, v[8 * q + 6], b.z);
                b.w = fmaf(p.neg_lr, v[8 * q + 7], b.w);
                wp[2 * q] = a;
                wp[2 * q + 1] = b;
                if (wo)
                    op[q] = make_uint4(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w),
                                       pack_bf16x2(b.x, b.y), pack_bf16x2(b.z, b.w));
            }
        }
        if (go) {
            uint4* gp = reinterpret_cast<uint4*>(go + off);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                if (q * 8 < lim)
                    gp[q] = make_uint4(pack_bf16x2(v[8 * q], v[8 * q + 1]),
                                       pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                                       pack_bf16x2(v[8 * q + 4], v[8 * q + 5]),
                                       pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
        }
    }

    __device__ __forceinline__ void finish(const Params&, int) {}
};

// ---------------------------------------------------------------------------
// Pseudogradient only, fp32, one output per group (layer): G[g] = g~^T A_l, for
// the optimizers that need the whole G (and its norm) before they step.
struct EpiStoreGroupF32 {
    struct Params {
        float* G[kMaxGroups];
        long long ld;
        int M, N;
    };
    int row, g;
    bool valid;

    __device__ __forceinline__ EpiStoreGroupF32(const Params& p, int g_, int row_, int)
        : row(row_), g(g_) {
        valid = row_ < p.M;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO&) {
        const int lim = p.N - col0;
        if (!valid || lim <= 0) return;
        float4* dst = reinterpret_cast<float4*>(p.G[g] + row * p.ld + col0);
#pragma unroll
        for (int q = 0; q < 8; ++q)
            if (q * 4 < lim) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    }

    __device__ __forceinline__ void finish(const Params&, int) {}
};

// ---------------------------------------------------------------------------
// Gate / up signals of a SwiGLU MLP (Sec. 3.1 step 5, Eq. errh): the GEMM gives
// error_h = g W3_init; with the cached pre-activations a (gate) and b (up),
//   dA = error_h (.) b (.) silu'(a),  dB = error_h (.) silu(a)   (bf16 out)
// Each 64-column pair of chunks fills one dA and one dB staging buffer (the
// warp's two buffers), stored by two TMA stores in one bulk group.
struct EpiSwiglu {
    struct Params {
        CUtensorMap dAmap;  // bf16 [M, N], box 64 x 32
        CUtensorMap dBmap;
        const __nv_bfloat16* a;  // [M, N]
        const __nv_bfloat16* b;
        long long ld;
        int M, N;
    };
    static constexpr int kTileN = 256;  // columns of the tiles it runs on (both GEMM kernels)
    int row, n_end;
    bool valid, pair_out;
    // a and b of the chunk the next chunk() call works on: loaded one chunk ahead, so
    // their latency overlaps the arithmetic of the chunk before (the first chunk's loads
    // are issued by the constructor)
    uint4 ua[4], ub[4];

    __device__ __forceinline__ void fetch(const Params& p, int col0) {
        const int lim = p.N - col0;
        const uint4* pa = reinterpret_cast<const uint4*>(p.a + row * p.ld + col0);
        const uint4* pb = reinterpret_cast<const uint4*>(p.b + row * p.ld + col0);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const bool in = valid && q * 8 < lim;
            ua[q] = in ? pa[q] : make_uint4(0, 0, 0, 0);
            ub[q] = in ? pb[q] : make_uint4(0, 0, 0, 0);
        }
    }

    __device__ __forceinline__ EpiSwiglu(const Params& p, int, int row_, int n0) : row(row_) {
        valid = row_ < p.M;
        pair_out = false;
        n_end = n0 + kTileN;
        fetch(p, n0);
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int c0,
                                          EpiIO& io) {
        const bool second = (c0 & 32) != 0;
        uint4 ca[4], cb[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            ca[q] = ua[q];
            cb[q] = ub[q];
        }
        if (col0 + 32 < n_end) fetch(p, col0 + 32);
        if (!second) {
            pair_out = col0 >= p.N || io.row0 >= p.M;
            if (pair_out) return;
            if (io.lane == 0) bulk_wait_group_read<0>();  // both buffers free again
            __syncwarp();
        }
        if (pair_out) return;
        uint32_t wa[16], wb[16];
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const __nv_bfloat162 ha = reinterpret_cast<const __nv_bfloat162*>(&ca[j / 8])[(j % 8) / 2];
            const __nv_bfloat162 hb = reinterpret_cast<const __nv_bfloat162*>(&cb[j / 8])[(j % 8) / 2];
            const float2 fa = __bfloat1622float2(ha), fb = __bfloat1622float2(hb);
            const float xa[2] = {fa.x, fa.y}, xb[2] = {fb.x, fb.y};
            float da[2], db[2];
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                // sigmoid with the fast intrinsic divide: its few-ulp fp32 error is far
                // below the bf16 rounding of dA and dB (for x < -87 it gives 0, as the
                // exact value is below bf16's range there too)
                const float x = xa[k];
                const float sg = __fdividef(1.f, 1.f + __expf(-x));
                da[k] = v[j + k] * xb[k] * sg * fmaf(x, 1.f - sg, 1.f);
                db[k] = v[j + k] * x * sg;
            }
            wa[j / 2] = pack_bf16x2(da[0], da[1]);
            wb[j / 2] = pack_bf16x2(db[0], db[1]);
        }
        const uint32_t bufA = io.out, bufB = io.out + kOutBufBytes;
        out_stage_half(bufA, io.lane, second ? 1 : 0, wa);
        out_stage_half(bufB, io.lane, second ? 1 : 0, wb);
        if (second) {
            fence_proxy_async_smem();
            __syncwarp();
            if (io.lane == 0) {
                tma_store_2d(&p.dAmap, bufA, col0 - 32, io.row0);
                tma_store_2d(&p.dBmap, bufB, col0 - 32, io.row0);
                bulk_commit_group();
            }
        }
    }

    __device__ __forceinline__ void finish(const Params&, int) {}
};

}  // namespace fpo
