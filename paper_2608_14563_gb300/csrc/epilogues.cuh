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
#include "optim_math.cuh"
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
// per-token anchor c_t, the target logit): every valid non-target logit leaves
//   p~_tj = exp(z_tj - c_t)
// rounded to bf16 into P [M, N] (the target column and the overhang are written
// as 0), and per (row, 256-column tile) three sums:
//   su = sum_j p~_tj          (unrounded: lse_t = c_t + log(1 + S_t), the target's
//                              own term being exp(0) = 1)
//   sx = sum_j p^_tj          (p^ the rounded values: the tile's part of S'_t, which
//                              makes the target entry of e the exact negative sum)
//   qz = sum_j p^_tj z_tj     (for the final-norm VJP fused into the projection:
//                              <yhat_t, g_t> = sum_v e_tv z_tv = alpha_t (Qz_t - c_t S'_t))
// No running maximum is kept: a row whose S'_t leaves the window [2^-80, 2^80]
// (where the anchored sums could overflow, or hold no significant digit) is
// recomputed by the fixup path, which takes its lse from a max-based pass
// (EpiFixLse, then EpiFixProb).
// Chunks that hold neither a target nor the vocabulary's ragged end (all but a few
// per row) take a branch-free path on packed f32x2 arithmetic; two 32-column chunks
// fill one 64-column bf16 staging row before each TMA store.
struct EpiAnchorProb {
    struct Params {
        CUtensorMap pmap;     // bf16 P [M, N], box 64 x 32
        float* su;            // [M, part_ld] sum of p~ over the tile
        float* sx;            // [M, part_ld] sum of the rounded p~ of the tile
        float* qz;            // [M, part_ld] sum of the rounded p~ times z over the tile
        int part_ld;
        const int* y;         // [M] targets
        const float* anchor;  // [M] c_t
        int M, N;
    };
    float2 u0, u1, s0, s1, q0, q1;  // two accumulators each: shorter dependency chains
    float2 nc2;             // (-c_t log2 e) twice
    int yoff, row;
    bool valid, pair_out;
    uint32_t w[32];

    __device__ __forceinline__ EpiAnchorProb(const Params& p, int, int row_, int n0)
        : row(row_), pair_out(false) {
        valid = row_ < p.M;
        yoff = valid ? __ldg(p.y + row_) - n0 : -1;
        const float nc = valid ? -__ldg(p.anchor + row_) * kLog2e : 0.f;
        nc2 = make_float2(nc, nc);
        u0 = u1 = s0 = s1 = q0 = q1 = make_float2(0.f, 0.f);
    }

    // p^ of the pair (j, j + 1) and its contribution to the sums; kMask: zero the
    // target (position r) and the columns >= lim.
    template <bool kMask>
    __device__ __forceinline__ uint32_t pair(const float (&v)[32], int j, int r, int lim) {
        const float2 z = make_float2(v[j], v[j + 1]);
        const float2 arg = __ffma2_rn(z, make_float2(kLog2e, kLog2e), nc2);
        float pa = ex2_approx(arg.x), pb = ex2_approx(arg.y);
        if constexpr (kMask) {
            pa = (j < lim && j != r) ? pa : 0.f;
            pb = (j + 1 < lim && j + 1 != r) ? pb : 0.f;
        }
        const uint32_t pk = pack_bf16x2(pa, pb);
        const float2 rp = make_float2(__uint_as_float(pk << 16), __uint_as_float(pk & 0xffff0000u));
        if ((j / 2) & 1) {
            u1 = __fadd2_rn(u1, make_float2(pa, pb));
            s1 = __fadd2_rn(s1, rp);
            q1 = __ffma2_rn(rp, z, q1);
        } else {
            u0 = __fadd2_rn(u0, make_float2(pa, pb));
            s0 = __fadd2_rn(s0, rp);
            q0 = __ffma2_rn(rp, z, q0);
        }
        return pk;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int c0,
                                          EpiIO& io) {
        const bool second = (c0 & 32) != 0;
        if (!second) pair_out = col0 >= p.N || io.row0 >= p.M;
        const int lim = p.N - col0;  // valid columns in this chunk (may be <= 0)
        const int r = yoff - c0;     // target position in this chunk, if in [0, 32)
        uint32_t pk[16];
        // warp-uniform: a chunk holding any lane's target, or the ragged end, is masked
        if (lim < 32 || __any_sync(0xffffffffu, static_cast<unsigned>(r) < 32u)) {
#pragma unroll
            for (int j = 0; j < 32; j += 2) pk[j / 2] = pair<true>(v, j, r, lim);
        } else {
#pragma unroll
            for (int j = 0; j < 32; j += 2) pk[j / 2] = pair<false>(v, j, r, lim);
        }
        if (pair_out) return;
        if (!second) {
#pragma unroll
            for (int i = 0; i < 16; ++i) w[i] = pk[i];
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) w[16 + i] = pk[i];
            const uint32_t buf = out_acquire(io);
            out_stage_row(buf, io.lane, w);
            out_commit(io, &p.pmap, buf, col0 - 32, io.row0);
        }
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        if (!valid) return;
        const long long o = static_cast<long long>(row) * p.part_ld + nb;
        const float2 u = __fadd2_rn(u0, u1), s = __fadd2_rn(s0, s1), q = __fadd2_rn(q0, q1);
        p.su[o] = u.x + u.y;
        p.sx[o] = s.x + s.y;
        p.qz[o] = q.x + q.y;
    }
};

// ---------------------------------------------------------------------------
// Direct algorithm, rows outside the anchor window, first pass: the logits of the
// gathered rows (the GEMM's rows are fix[0, count)) reduced to a running max and
// sum of exponentials per (row, 256-column tile), written to part[row of the chunk,
// tile], from which lse is formed before the second pass (EpiFixProb).
struct EpiFixLse {
    struct Params {
        float2* part;        // [T, part_ld] (max, sum exp(z - max))
        int part_ld;
        const int* fix;      // gathered row -> row of the chunk
        const int* count;    // gathered rows (device)
        int N;
    };
    float m, s;
    int orig;
    bool valid;

    __device__ __forceinline__ EpiFixLse(const Params& p, int, int row_, int)
        : m(-INFINITY), s(0.f) {
        valid = row_ < *p.count;
        orig = valid ? p.fix[row_] : 0;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO&) {
        const int lim = p.N - col0;
        if (!valid || lim <= 0) return;
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
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        if (valid) p.part[static_cast<size_t>(orig) * p.part_ld + nb] = make_float2(m, s);
    }
};

// ---------------------------------------------------------------------------
// Direct algorithm, rows outside the anchor window, second pass (Sec. 3.1 step 2
// with the anchor at lse_t): the GEMM's rows are the yhat rows gathered from
// fix[0, count); each logit z of such a row becomes p~ = exp(z - lse_t), 0 at the
// target, rounded to bf16 and stored into that row of P with plain 16-byte stores;
// the row's sums over the tile of the rounded values and of the rounded values
// times z go to sx[row, tile] and qz[row, tile], as EpiAnchorProb leaves them.
struct EpiFixProb {
    struct Params {
        __nv_bfloat16* P;    // [T, N] rows of the chunk, row stride N
        float* sx;           // [T, n_tiles]
        float* qz;           // [T, n_tiles]
        const int* fix;      // gathered row -> row of the chunk
        const int* count;    // gathered rows (device)
        const int32_t* y;    // [T] targets
        const float* lse;    // [T]
        int n_tiles, N;
    };
    int orig, yt;
    float lse2, sxs, qs;
    bool valid;

    __device__ __forceinline__ EpiFixProb(const Params& p, int, int row_, int)
        : sxs(0.f), qs(0.f) {
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
            const float ra = __uint_as_float(pk << 16), rb = __uint_as_float(pk & 0xffff0000u);
            sxs += ra + rb;
            qs = fmaf(ra, v[j], qs);
            qs = fmaf(rb, v[j + 1], qs);
            w[j / 2] = pk;
        }
        uint4* dst = reinterpret_cast<uint4*>(p.P + static_cast<size_t>(orig) * p.N + col0);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            if (q * 8 < lim) dst[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        if (valid) {
            p.sx[static_cast<size_t>(orig) * p.n_tiles + nb] = sxs;
            p.qz[static_cast<size_t>(orig) * p.n_tiles + nb] = qs;
        }
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
// Projection of the direct algorithm with the final-norm VJP (App. E,
// Eq. rmsnorm-vjp) fused in.  With acc = P W_U (target column of P zero), the
// unnormalised error signal of token t is
//   g_t = alpha_t acc_t + beta_t W_U[y_t],   alpha_t = s exp(c_t - lse_t),
//   beta_t = -alpha_t S'_t,
// which is s (softmax(z_t) - 1_{y_t}) W_U written with the anchor c_t, and the
// epilogue writes, in bf16,
//   g~_t = (w (.) g_t - x^_t k_t) / max(rho_t, rho_min),   x^_t = h_t / rho_t,
// where k_t = <x^_t, w (.) g_t> / d arrives as cv_t / d: cv_t = alpha_t (Qz_t - c_t S'_t)
// from the logits pass (EpiAnchorProb), the same inner product taken through the
// logits (<yhat_t, W_U[v]> = z_tv), so no tile needs the whole row of g.
// A row with alpha_t == 0 is written as zeros (s == 0, or an out-of-range
// target); beta_t == 0 skips the read of the target's W_U row.  The h, w and
// W_U[y] values of the next 32-column chunk are loaded while the current one is
// processed; two chunks fill one 64-column bf16 staging row per TMA store.
struct EpiProjVjp {
    struct Params {
        CUtensorMap omap;           // bf16 g~ [M, N], box 64 x 32
        const float* alpha;         // [M]
        const float* beta;          // [M]
        const float* cv;            // [M] <yhat_t, g_t>
        const float* rho;           // [M] RMS of h_t (forward pass)
        const int* y;               // [M]
        const __nv_bfloat16* W_U;   // [V, N]
        const __nv_bfloat16* h;     // [M, N] pre-norm residual
        const __nv_bfloat16* w;     // [N] final RMSNorm weight
        float min_rms, inv_d;
        int M, N;
        int tile_n;                 // columns of the kernel's tiles (one epilogue object each)
    };
    float a;
    float2 a2, b2, nk2;  // per row, twice: alpha pref, beta pref, -(cv / d) pref / rho
    const __nv_bfloat16* wy;
    const __nv_bfloat16* hr;
    bool valid, pair_out;
    int n_end;
    uint4 uh[4], uw[4], uy[4];  // h, w, W_U[y] of the chunk the next chunk() call uses
    uint32_t o[32];

    __device__ __forceinline__ void fetch(const Params& p, int col0) {
        const int lim = p.N - col0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const bool in = q * 8 < lim;
            uh[q] = (valid && in) ? __ldg(reinterpret_cast<const uint4*>(hr + col0) + q)
                                  : make_uint4(0, 0, 0, 0);
            uw[q] = in ? __ldg(reinterpret_cast<const uint4*>(p.w + col0) + q)
                       : make_uint4(0, 0, 0, 0);
            uy[q] = (wy && in) ? __ldg(reinterpret_cast<const uint4*>(wy + col0) + q)
                               : make_uint4(0, 0, 0, 0);
        }
    }

    __device__ __forceinline__ EpiProjVjp(const Params& p, int, int row, int n0)
        : pair_out(false) {
        valid = row < p.M;
        a = valid ? __ldg(p.alpha + row) : 0.f;
        const float b = valid ? __ldg(p.beta + row) : 0.f;
        const float r = valid ? __ldg(p.rho + row) : 1.f;
        const float kd = valid ? __ldg(p.cv + row) * p.inv_d : 0.f;
        const float pref = 1.0f / fmaxf(r, p.min_rms);
        // g~_j = w_j (a pref acc_j + b pref W_U[y]_j) - h_j (kd pref / rho)
        a2 = make_float2(a * pref, a * pref);
        b2 = make_float2(b * pref, b * pref);
        const float nk = -(kd * (1.0f / r)) * pref;
        nk2 = make_float2(nk, nk);
        wy = (a != 0.f && b != 0.f) ? p.W_U + static_cast<long long>(__ldg(p.y + row)) * p.N
                                    : nullptr;
        hr = p.h + static_cast<long long>(valid ? row : 0) * p.N;
        n_end = min(n0 + p.tile_n, p.N);
        if (n0 < p.N) fetch(p, n0);
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int c0,
                                          EpiIO& io) {
        const bool second = (c0 & 32) != 0;
        uint4 ch[4], cw[4], cy[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            ch[q] = uh[q];
            cw[q] = uw[q];
            cy[q] = uy[q];
        }
        if (col0 + 32 < n_end) fetch(p, col0 + 32);
        if (!second) pair_out = col0 >= p.N || io.row0 >= p.M;
        if (pair_out) return;
        uint32_t r[16];
        if (a == 0.f) {  // s == 0 or an out-of-range target: g = 0 and cv = 0, so g~ = 0
#pragma unroll
            for (int i = 0; i < 16; ++i) r[i] = 0u;
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint32_t hh[4] = {ch[q].x, ch[q].y, ch[q].z, ch[q].w};
                const uint32_t ww[4] = {cw[q].x, cw[q].y, cw[q].z, cw[q].w};
                const uint32_t yy[4] = {cy[q].x, cy[q].y, cy[q].z, cy[q].w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int j = 8 * q + 2 * k;
                    const float2 hv = make_float2(__uint_as_float(hh[k] << 16),
                                                  __uint_as_float(hh[k] & 0xffff0000u));
                    const float2 wv = make_float2(__uint_as_float(ww[k] << 16),
                                                  __uint_as_float(ww[k] & 0xffff0000u));
                    const float2 uv = make_float2(__uint_as_float(yy[k] << 16),
                                                  __uint_as_float(yy[k] & 0xffff0000u));
                    const float2 t = __ffma2_rn(b2, uv, __fmul2_rn(a2, make_float2(v[j], v[j + 1])));
                    const float2 out = __ffma2_rn(wv, t, __fmul2_rn(nk2, hv));
                    r[j / 2] = pack_bf16x2(out.x, out.y);
                }
            }
        }
        if (!second) {
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] = r[i];
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) o[16 + i] = r[i];
            const uint32_t buf = out_acquire(io);
            out_stage_row(buf, io.lane, o);
            out_commit(io, &p.omap, buf, col0 - 32, io.row0);
        }
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
            // every master load of the chunk is issued before the first store (which the
            // compiler cannot reorder across, as W_out might alias W_master): one memory
            // round trip per chunk instead of four
            float4 ma[4], mb[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (q * 8 < lim) {
                    ma[q] = wp[2 * q];
                    mb[q] = wp[2 * q + 1];
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (q * 8 >= lim) break;
                float4 a = ma[q], b = mb[q];
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
// Pseudogradients with the layer-viability diagnostic's cosine (Sec. 2.2 Eq. (cosine),
// Eq. (w3update)): for group (layer) g, G_out[g] = bf16(G), and the three sums of the
// cosine of that stored G against Y[g] (<G, Y>, ||G||^2, ||Y||^2) over the thread's
// row of the tile, summed over the warp's 32 rows (a fixed butterfly) and written as one
// triple per (layer, 256-row block, column tile, 32-row slot):
//   part[(((g m256 + row / 256) n_blocks + nb) 8 + (row mod 256) / 32) 3 + {0, 1, 2}]
// so the cosine needs no second pass over G.  The Y values of the next 32-column chunk
// are loaded while the current one is processed.
struct EpiGradCos {
    struct Params {
        __nv_bfloat16* G_out[kMaxGroups];
        const __nv_bfloat16* Y[kMaxGroups];
        float* part;     // [groups][m256][n_blocks][8][3]
        long long ld;
        int M, N;
        int m256, n_blocks;
    };
    static constexpr int kTileN = 256;  // columns of the tiles it runs on (both GEMM kernels)
    int row, g, n_end;
    bool valid;
    float2 s_gy, s_gg, s_yy;
    uint4 uy[4];  // Y of the chunk the next chunk() call works on

    __device__ __forceinline__ void fetch(const Params& p, int col0) {
        const int lim = p.N - col0;
        const uint4* py = reinterpret_cast<const uint4*>(p.Y[g] + row * p.ld + col0);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            uy[q] = (valid && q * 8 < lim) ? __ldg(py + q) : make_uint4(0, 0, 0, 0);
    }

    __device__ __forceinline__ EpiGradCos(const Params& p, int g_, int row_, int n0)
        : row(row_), g(g_) {
        valid = row_ < p.M;
        n_end = n0 + kTileN;
        s_gy = s_gg = s_yy = make_float2(0.f, 0.f);
        if (n0 < p.N) fetch(p, n0);
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO&) {
        uint4 cy[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) cy[q] = uy[q];
        if (col0 + 32 < n_end && col0 + 32 < p.N) fetch(p, col0 + 32);
        const int lim = p.N - col0;
        if (!valid || lim <= 0) return;
        uint4* gp = reinterpret_cast<uint4*>(p.G_out[g] + row * p.ld + col0);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t pk[4] = {pack_bf16x2(v[8 * q], v[8 * q + 1]),
                                    pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                                    pack_bf16x2(v[8 * q + 4], v[8 * q + 5]),
                                    pack_bf16x2(v[8 * q + 6], v[8 * q + 7])};
            if (q * 8 < lim) gp[q] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            // columns >= N: G is 0 there (zero-filled operand) and Y was loaded as 0
            const uint32_t yk[4] = {cy[q].x, cy[q].y, cy[q].z, cy[q].w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 gr = make_float2(__uint_as_float(pk[k] << 16),
                                              __uint_as_float(pk[k] & 0xffff0000u));
                const float2 yr = make_float2(__uint_as_float(yk[k] << 16),
                                              __uint_as_float(yk[k] & 0xffff0000u));
                s_gy = __ffma2_rn(gr, yr, s_gy);
                s_gg = __ffma2_rn(gr, gr, s_gg);
                s_yy = __ffma2_rn(yr, yr, s_yy);
            }
        }
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        float gy = s_gy.x + s_gy.y, gg = s_gg.x + s_gg.y, yy = s_yy.x + s_yy.y;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            gy += __shfl_xor_sync(0xffffffffu, gy, o);
            gg += __shfl_xor_sync(0xffffffffu, gg, o);
            yy += __shfl_xor_sync(0xffffffffu, yy, o);
        }
        if ((threadIdx.x & 31) == 0) {
            const long long slot =
                ((static_cast<long long>(g) * p.m256 + row / 256) * p.n_blocks + nb) * 8 +
                (row % 256) / 32;
            float* o = p.part + slot * 3;
            o[0] = gy;
            o[1] = gg;
            o[2] = yy;
        }
    }
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
// The optimizer's first pass in the pseudogradient GEMM's epilogue, for the relative
// clip on the step (Sec. 3.1: SGD, SGD with momentum, AdamW on the fp32 masters; App. A:
// ||dW|| <= clip_frac ||W||).  With G from the accumulator, each element's optimizer state
// advances and its unclipped step d = opt_step(G, W, s1, s2) is stored (fp32, D[g]; the
// state sees the unclipped gradient), and ||W||^2, ||d||^2 of the warp's 32 rows of the
// tile are written as one pair per (layer, 256-row block, column tile, 32-row slot); a
// kernel then scales each layer's steps by min(1, clip_frac ||W|| / ||d||) and applies
// them (W is not written here, so its norm is the pre-step one).  Without a clip the
// stand-alone passes are used: taking the whole step here made the update faster but
// the power-capped step slower (its epilogue then held the tensor pipe back at full
// draw).
struct EpiOptStep {
    struct Params {
        const float* W_master[kMaxGroups];
        float* s1[kMaxGroups];             // momentum / AdamW first moment (or null)
        float* s2[kMaxGroups];             // AdamW second moment (or null)
        float* D[kMaxGroups];              // the unclipped steps
        float* part;                       // [groups][m256][n_blocks][8][2]
        OptimParams op;
        long long ld;
        int M, N;
        int m256, n_blocks;
    };
    int row, g;
    bool valid;
    float s_ww, s_dd;

    __device__ __forceinline__ EpiOptStep(const Params& p, int g_, int row_, int)
        : row(row_), g(g_), s_ww(0.f), s_dd(0.f) {
        valid = row_ < p.M;
    }

    __device__ __forceinline__ void chunk(const Params& p, const float (&v)[32], int col0, int,
                                          EpiIO&) {
        const int lim = p.N - col0;
        if (!valid || lim <= 0) return;
        const long long off = row * p.ld + col0;
        const float4* wp = reinterpret_cast<const float4*>(p.W_master[g] + off);
        float4* p1 = p.s1[g] ? reinterpret_cast<float4*>(p.s1[g] + off) : nullptr;
        float4* p2 = p.s2[g] ? reinterpret_cast<float4*>(p.s2[g] + off) : nullptr;
#pragma unroll
        for (int h = 0; h < 2; ++h) {  // 16 columns at a time
            if (h * 16 >= lim) break;
            float w[16], a[16], b[16];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int c4 = 4 * h + q;  // float4 index in the chunk
                if (c4 * 4 < lim) {
                    const float4 x = wp[c4];
                    w[4 * q] = x.x; w[4 * q + 1] = x.y; w[4 * q + 2] = x.z; w[4 * q + 3] = x.w;
                    const float4 y = p1 ? p1[c4] : make_float4(0.f, 0.f, 0.f, 0.f);
                    a[4 * q] = y.x; a[4 * q + 1] = y.y; a[4 * q + 2] = y.z; a[4 * q + 3] = y.w;
                    const float4 z = p2 ? p2[c4] : make_float4(0.f, 0.f, 0.f, 0.f);
                    b[4 * q] = z.x; b[4 * q + 1] = z.y; b[4 * q + 2] = z.z; b[4 * q + 3] = z.w;
                }
            }
            float out[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                out[e] = opt_step(p.op, v[16 * h + e], w[e], a[e], b[e]);
                if (16 * h + e < lim) {  // (columns past N were not loaded)
                    s_ww = fmaf(w[e], w[e], s_ww);
                    s_dd = fmaf(out[e], out[e], s_dd);
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int c4 = 4 * h + q;
                if (c4 * 4 >= lim) break;
                reinterpret_cast<float4*>(p.D[g] + off)[c4] =
                    make_float4(out[4 * q], out[4 * q + 1], out[4 * q + 2], out[4 * q + 3]);
                if (p1) p1[c4] = make_float4(a[4 * q], a[4 * q + 1], a[4 * q + 2], a[4 * q + 3]);
                if (p2) p2[c4] = make_float4(b[4 * q], b[4 * q + 1], b[4 * q + 2], b[4 * q + 3]);
            }
        }
    }

    __device__ __forceinline__ void finish(const Params& p, int nb) {
        float ww = s_ww, dd = s_dd;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            ww += __shfl_xor_sync(0xffffffffu, ww, o);
            dd += __shfl_xor_sync(0xffffffffu, dd, o);
        }
        if ((threadIdx.x & 31) == 0) {
            const long long slot =
                ((static_cast<long long>(g) * p.m256 + row / 256) * p.n_blocks + nb) * 8 +
                (row % 256) / 32;
            float* o = p.part + slot * 2;
            o[0] = ww;
            o[1] = dd;
        }
    }
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
