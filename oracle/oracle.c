/*
 * oracle.c -- plain, slow, fp64 CPU oracle for the FPO pseudogradient update.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  The
 * product path (libfpo.so and its Python binding) never calls it, and this
 * file shares no code, header, table or helper with the CUDA sources.
 *
 * Every function is the plain definition of one step of the method of
 * "Forward Pass Domain Adaptation (Without Cross-Layer Backpropagation)"
 * written out in fp64, with no blocking, fusion or reordering:
 *
 *   oracle_error_signal  Sec. 3.1 steps 2-4, Eq. (gproj), App. E Eq. (rmsnorm-vjp)
 *                        and the min-RMS clamp (Sec. 3.2 / App. E)
 *   oracle_rmsnorm_vjp   App. E Eq. (rmsnorm-vjp) at any norm (post-FFN, Sec. 3.2)
 *   oracle_layer_signal  Sec. 3.1 step 4 and Sec. 3.2: the per-layer composition with the
 *                        post-feedforward and / or pre-MLP RMSNorm Jacobians
 *   oracle_gate_up_signals  Sec. 3.1 step 5, Eq. (errh): W1/W2 signals of a SwiGLU MLP
 *   oracle_pseudograd    Sec. 3.1 step 5, Eq. (w3update): G = g~^T h_mid
 *   oracle_sgd_update    App. A (fp32 master weights, cast to bf16)
 *   oracle_optimizer_step  Sec. 3.1 (AdamW / SGD with momentum) + App. A relative clip
 *   oracle_cosine        Sec. 2.2, Eq. (cosine)
 *   oracle_norm_ratio    App. C (update-magnitude ratios) and Sec. C.2: ||G||/||W||
 *                        and the SGD learning rate of a relative step
 *
 * Inputs are the exact stored values (fp32, bf16 or fp64) upcast to fp64 as
 * they are read.  OpenMP parallelises only over independent tokens / output
 * rows; every sum runs in index order inside one thread.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORC_F32 = 0, ORC_BF16 = 1, ORC_F64 = 2 };

/* Upcast element i of a typed array to fp64.  bf16 is the upper half of an
 * IEEE binary32, so its value is that binary32 with a zero lower half. */
static inline double orc_load(int dt, const void* p, int64_t i) {
    if (dt == ORC_F64) return ((const double*)p)[i];
    if (dt == ORC_F32) return (double)((const float*)p)[i];
    uint32_t bits = (uint32_t)((const uint16_t*)p)[i] << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

int oracle_abi_version(void) { return 1; }

/*
 * Steps 1-5 of the error signal, one token at a time (tokens are independent
 * until the contraction over T in Eq. (w3update)).
 *
 * For token t (rows[r] when rows != NULL, else r):
 *   rho   = sqrt(mean_j h_tj^2 + eps)                       App. E, below Eq. (rmsnorm-vjp)
 *   xhat  = h_t / rho ;  yhat = w (.) xhat                  final RMSNorm forward
 *   z_v   = <yhat, W_U[v,:]>                                logits (Sec. 3.1 step 2)
 *   lse   = m + log sum_v exp(z_v - m),  m = max_v z_v
 *   e_v   = s * (exp(z_v - lse) - [v == y_t])              softmax(z) - 1_y, loss scale s
 *           (the target entry as -s sum_{v != y_t} exp(z_v - lse): the softmax
 *           sums to one, so this is the same number, and it keeps its digits
 *           when 1 - p_y is below the fp64 ulp of lse, where p_y - 1 has none)
 *   g_j   = sum_v e_v W_U[v,j]                              Eq. (gproj)
 *   c     = <xhat, w (.) g>
 *   g~_j  = (w_j g_j - xhat_j c / d) / max(rho, rho_min)    Eq. (rmsnorm-vjp) + min-RMS clamp
 *
 * The clamp replaces rho only in the 1/rho prefactor; xhat keeps the true rho
 * (the reading under which the clamp "caps the 1/rho amplification" and the
 * projection term stays exact).
 *
 * Outputs (each optional, NULL to skip) are indexed by r, the position in the
 * row list: rho[r], lse[r], zy[r] = z_{t,y_t}, g[r*d + j], g_tilde[r*d + j],
 * e[r*V + v].  Returns 0, or -1 for a bad argument, or -2 when a target is
 * outside [0, V) (that token's outputs are left untouched).
 */
int oracle_error_signal(int64_t T, int64_t d, int64_t V, int dt,
                        const void* h, const void* w, const void* W_U,
                        const int32_t* y, double eps, double min_rms, double s,
                        const int64_t* rows, int64_t n_rows,
                        double* rho, double* lse, double* zy, double* g,
                        double* g_tilde, double* e) {
    if (T < 0 || d <= 0 || V <= 0 || !h || !w || !W_U || !y) return -1;
    if (!rows) n_rows = T;
    int bad_target = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad_target)
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t t = rows ? rows[r] : r;
        if (t < 0 || t >= T) { bad_target = 1; continue; }
        int32_t yt = y[t];
        if (yt < 0 || yt >= V) { bad_target = 1; continue; }

        double* xhat = (double*)malloc(sizeof(double) * (size_t)d);
        double* yhat = (double*)malloc(sizeof(double) * (size_t)d);
        double* z = (double*)malloc(sizeof(double) * (size_t)V);
        double* gt = (double*)malloc(sizeof(double) * (size_t)d);

        double ss = 0.0;
        for (int64_t j = 0; j < d; ++j) {
            double x = orc_load(dt, h, t * d + j);
            ss += x * x;
        }
        double rh = sqrt(ss / (double)d + eps);
        for (int64_t j = 0; j < d; ++j) {
            xhat[j] = orc_load(dt, h, t * d + j) / rh;
            yhat[j] = orc_load(dt, w, j) * xhat[j];
        }

        double m = -INFINITY;
        for (int64_t v = 0; v < V; ++v) {
            double acc = 0.0;
            for (int64_t j = 0; j < d; ++j) acc += yhat[j] * orc_load(dt, W_U, v * d + j);
            z[v] = acc;
            if (acc > m) m = acc;
        }
        double se = 0.0;
        for (int64_t v = 0; v < V; ++v) se += exp(z[v] - m);
        double l = m + log(se);

        /* e overwrites z in place: e_v = s p_v off the target, and
         * e_y = -s sum_{v != y} p_v (summed in index order). */
        if (zy) zy[r] = z[yt];
        double rest = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            if (v == yt) continue;
            double p = exp(z[v] - l);
            rest += p;
            z[v] = s * p;
        }
        z[yt] = -s * rest;
        if (e) memcpy(e + r * V, z, sizeof(double) * (size_t)V);

        for (int64_t j = 0; j < d; ++j) gt[j] = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            double ev = z[v];
            for (int64_t j = 0; j < d; ++j) gt[j] += ev * orc_load(dt, W_U, v * d + j);
        }
        if (g) memcpy(g + r * d, gt, sizeof(double) * (size_t)d);

        if (g_tilde) {
            double c = 0.0;
            for (int64_t j = 0; j < d; ++j) c += xhat[j] * orc_load(dt, w, j) * gt[j];
            double denom = rh > min_rms ? rh : min_rms;
            for (int64_t j = 0; j < d; ++j)
                g_tilde[r * d + j] =
                    (orc_load(dt, w, j) * gt[j] - xhat[j] * c / (double)d) / denom;
        }
        if (rho) rho[r] = rh;
        if (lse) lse[r] = l;

        free(xhat);
        free(yhat);
        free(z);
        free(gt);
    }
    return bad_target ? -2 : 0;
}

/*
 * App. E Eq. (rmsnorm-vjp), the closed-form RMSNorm Jacobian applied to an
 * upstream gradient g at a cached norm input x with weight gamma (the same
 * expression the paper composes at every norm it corrects for: the final norm,
 * and per layer the post-feedforward norm of OLMo-2 / Gemma 3, Sec. 3.2):
 *   rho  = sqrt(mean_j x_j^2 + eps),  xhat = x / rho
 *   c    = <xhat, gamma (.) g>
 *   out  = (gamma (.) g - xhat c / d) / max(rho, rho_min)
 * g, x: [T, d] (dtypes dt_g, dt_x); gamma: [d] (dt_x); out: [T, d] fp64.
 */
int oracle_rmsnorm_vjp(int64_t T, int64_t d, int dt_g, const void* g, int dt_x, const void* x,
                       const void* gamma, double eps, double min_rms, double* out) {
    if (T < 0 || d <= 0 || !out || (T > 0 && (!g || !x || !gamma))) return -1;
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < T; ++t) {
        double ss = 0.0;
        for (int64_t j = 0; j < d; ++j) {
            double v = orc_load(dt_x, x, t * d + j);
            ss += v * v;
        }
        double rh = sqrt(ss / (double)d + eps);
        double c = 0.0;
        for (int64_t j = 0; j < d; ++j)
            c += (orc_load(dt_x, x, t * d + j) / rh) * orc_load(dt_x, gamma, j) *
                 orc_load(dt_g, g, t * d + j);
        double denom = rh > min_rms ? rh : min_rms;
        for (int64_t j = 0; j < d; ++j)
            out[t * d + j] = (orc_load(dt_x, gamma, j) * orc_load(dt_g, g, t * d + j) -
                              (orc_load(dt_x, x, t * d + j) / rh) * c / (double)d) / denom;
    }
    return 0;
}

/*
 * App. E Eq. (rmsnorm-vjp) on one fp64 row u at norm input row x (element offset
 * off of a typed [T, d] array) with weight gamma:
 *   rho = sqrt(mean_j x_j^2 + eps), xhat = x / rho, c = <xhat, gamma (.) u>,
 *   v   = (gamma (.) u - xhat c / d) / max(rho, rho_min)
 */
static void orc_vjp_row(int64_t d, const double* u, int dt, const void* x, int64_t off,
                        const void* gamma, double eps, double min_rms, double* v) {
    double ss = 0.0;
    for (int64_t j = 0; j < d; ++j) {
        double xv = orc_load(dt, x, off + j);
        ss += xv * xv;
    }
    double rh = sqrt(ss / (double)d + eps);
    double c = 0.0;
    for (int64_t j = 0; j < d; ++j) c += (orc_load(dt, x, off + j) / rh) * orc_load(dt, gamma, j) * u[j];
    double denom = rh > min_rms ? rh : min_rms;
    for (int64_t j = 0; j < d; ++j)
        v[j] = (orc_load(dt, gamma, j) * u[j] - (orc_load(dt, x, off + j) / rh) * c / (double)d) / denom;
}

/*
 * The layer-specific signal of one target layer (Sec. 3.1 step 4, Sec. 3.2, App. E
 * table of norms per family).  Starting from g (the signal after the final norm's
 * Jacobian), in the paper's order:
 *   1. post-feedforward RMSNorm (OLMo-2, Gemma 3): compose with its Jacobian at the
 *      layer's MLP output m with weight gamma_post;
 *   2. pre-MLP RMSNorm (Qwen3, Gemma 3): additionally compose with its Jacobian at
 *      the norm's input x (the residual stream entering the MLP block) with weight
 *      gamma_pre.
 * Each is App. E Eq. (rmsnorm-vjp) with its own rho and the min-RMS clamp; a norm
 * whose input is NULL is not composed (both NULL: out = g).  The intermediate signal
 * stays in fp64.  g: [T, d] (dt_g); m, x: [T, d] and gammas: [d] (dt_n); out: fp64.
 */
int oracle_layer_signal(int64_t T, int64_t d, int dt_g, const void* g, int dt_n, const void* m,
                        const void* gamma_post, const void* x, const void* gamma_pre, double eps,
                        double min_rms, double* out) {
    if (T < 0 || d <= 0 || !out || (T > 0 && !g) || (m && !gamma_post) || (x && !gamma_pre))
        return -1;
#pragma omp parallel
    {
        double* u = (double*)malloc((size_t)d * sizeof(double));
        double* v = (double*)malloc((size_t)d * sizeof(double));
#pragma omp for schedule(static)
        for (int64_t t = 0; t < T; ++t) {
            if (!u || !v) continue;
            for (int64_t j = 0; j < d; ++j) u[j] = orc_load(dt_g, g, t * d + j);
            if (m) {
                orc_vjp_row(d, u, dt_n, m, t * d, gamma_post, eps, min_rms, v);
                memcpy(u, v, (size_t)d * sizeof(double));
            }
            if (x) {
                orc_vjp_row(d, u, dt_n, x, t * d, gamma_pre, eps, min_rms, v);
                memcpy(u, v, (size_t)d * sizeof(double));
            }
            memcpy(out + t * d, u, (size_t)d * sizeof(double));
        }
        free(u);
        free(v);
    }
    return 0;
}

/*
 * Gate / up signals of a SwiGLU MLP (Sec. 3.1 step 5, Eq. (errh)):
 *   error_h = g W3_init                        [T, d_ff]   (g [T, d], W3_init [d, d_ff])
 * and, with the cached gate and up pre-activations a, b ([T, d_ff];
 * h_mid = silu(a) (.) b, silu(a) = a sigma(a)):
 *   dA = error_h (.) b (.) silu'(a),  silu'(a) = sigma(a) (1 + a (1 - sigma(a)))
 *   dB = error_h (.) silu(a)
 * so that G1 = dA^T x and G2 = dB^T x (x the MLP input) are the W1 / W2
 * pseudogradients.  Outputs fp64 [T, d_ff].
 */
int oracle_gate_up_signals(int64_t T, int64_t d, int64_t d_ff, int dt, const void* g,
                           const void* W3, const void* a, const void* b, double* dA, double* dB) {
    if (T < 0 || d <= 0 || d_ff <= 0 || !dA || !dB || (T > 0 && (!g || !W3 || !a || !b))) return -1;
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < T; ++t) {
        for (int64_t f = 0; f < d_ff; ++f) {
            double e = 0.0;
            for (int64_t j = 0; j < d; ++j) e += orc_load(dt, g, t * d + j) * orc_load(dt, W3, j * d_ff + f);
            const double av = orc_load(dt, a, t * d_ff + f), bv = orc_load(dt, b, t * d_ff + f);
            const double sg = 1.0 / (1.0 + exp(-av));
            dA[t * d_ff + f] = e * bv * sg * (1.0 + av * (1.0 - sg));
            dB[t * d_ff + f] = e * av * sg;
        }
    }
    return 0;
}

/*
 * Eq. (w3update): G[i,j] = sum_t g~[t,i] * A[t,j]  (g~ is [T,d], A is [T,d_ff],
 * G is [d,d_ff], the nn.Linear layout of the down-projection weight).
 * With ii == NULL every entry is written to G[i*d_ff + j]; otherwise only the
 * n_pairs entries (ii[k], jj[k]) are computed, into G[k].
 */
int oracle_pseudograd(int64_t T, int64_t d, int64_t d_ff, int dt_g, const void* gt,
                      int dt_a, const void* A, const int64_t* ii, const int64_t* jj,
                      int64_t n_pairs, double* G) {
    if (T < 0 || d <= 0 || d_ff <= 0 || !G || (T > 0 && (!gt || !A))) return -1;
    if (!ii) {
#pragma omp parallel for schedule(static)
        for (int64_t i = 0; i < d; ++i) {
            double* row = G + i * d_ff;
            for (int64_t j = 0; j < d_ff; ++j) row[j] = 0.0;
            for (int64_t t = 0; t < T; ++t) {
                double gi = orc_load(dt_g, gt, t * d + i);
                for (int64_t j = 0; j < d_ff; ++j) row[j] += gi * orc_load(dt_a, A, t * d_ff + j);
            }
        }
        return 0;
    }
    int bad = 0;
#pragma omp parallel for schedule(static) reduction(| : bad)
    for (int64_t k = 0; k < n_pairs; ++k) {
        int64_t i = ii[k], j = jj[k];
        if (i < 0 || i >= d || j < 0 || j >= d_ff) { bad = 1; continue; }
        double acc = 0.0;
        for (int64_t t = 0; t < T; ++t)
            acc += orc_load(dt_g, gt, t * d + i) * orc_load(dt_a, A, t * d_ff + j);
        G[k] = acc;
    }
    return bad ? -1 : 0;
}

/* IEEE binary64 -> binary32, round to nearest even (the C cast does this under
 * the default rounding mode). */
static inline float orc_to_f32(double x) { return (float)x; }

/* binary32 -> bfloat16, round to nearest even, from the definition: keep the
 * upper 16 bits; round up when the discarded half is above one half ulp, or
 * exactly one half ulp and the kept part is odd.  NaN stays a quiet NaN. */
static inline uint16_t orc_f32_to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu)) return (uint16_t)((u >> 16) | 0x40u);
    uint32_t upper = u >> 16, lower = u & 0xffffu;
    if (lower > 0x8000u || (lower == 0x8000u && (upper & 1u))) upper += 1u;
    return (uint16_t)upper;
}

/*
 * App. A: the fp32 master copy receives the step and the bf16 working weight
 * is its cast.  W_new = RN32(W - lr * G) evaluated in fp64, W_bf16 = RNE16(W_new).
 * Either output may be NULL.
 */
void oracle_sgd_update(int64_t n, const float* W, const double* G, double lr,
                       float* W_new, uint16_t* W_bf16) {
#pragma omp parallel for schedule(static)
    for (int64_t k = 0; k < n; ++k) {
        float wn = orc_to_f32((double)W[k] - lr * G[k]);
        if (W_new) W_new[k] = wn;
        if (W_bf16) W_bf16[k] = orc_f32_to_bf16(wn);
    }
}

/*
 * One optimizer step on the fp32 master copy of one layer (Sec. 3.1: AdamW with
 * weight decay 0.01 or SGD with momentum 0.9; App. A: fp32 master weights, and
 * a relative clip of each step to frac * ||W||_F).  kind: 0 SGD, 1 SGD with
 * momentum (buf = mu buf + G, step = -lr buf), 2 AdamW (m = b1 m + (1-b1) G,
 * v = b2 v + (1-b2) G^2, step = -lr (mhat / (sqrt(vhat) + eps) + wd W) with
 * mhat = m / (1 - b1^t), vhat = v / (1 - b2^t)).
 * clip: 0 none; 1 the step itself is scaled so ||step||_F <= frac ||W||_F (the
 * optimizer state is updated with the unscaled gradient); 2 the gradient is
 * scaled so ||G||_F <= frac ||W||_F before the optimizer sees it.
 * Norms are of the fp32 master W before the step.  Everything is evaluated in
 * fp64 from the stored fp32 values; outputs (W, state) are rounded to fp32 and
 * W_bf16 = RNE16(W_new).  s1 (momentum buffer / m) and s2 (v) may be NULL when
 * the kind has no such state.  Returns the clip factor applied (1 if none).
 */
double oracle_optimizer_step(int64_t n, int kind, double lr, double mu, double b1, double b2,
                             double eps, double wd, int64_t t, int clip, double frac,
                             const float* W, const double* G, const float* s1, const float* s2,
                             float* W_new, uint16_t* W_bf16, float* s1_new, float* s2_new) {
    double ww = 0.0, gg = 0.0;
    for (int64_t k = 0; k < n; ++k) {
        ww += (double)W[k] * (double)W[k];
        gg += G[k] * G[k];
    }
    const double wnorm = sqrt(ww);
    double gscale = 1.0;
    if (clip == 2 && sqrt(gg) > frac * wnorm) gscale = frac * wnorm / sqrt(gg);
    const double bc1 = 1.0 - pow(b1, (double)t), bc2 = 1.0 - pow(b2, (double)t);
    double* step = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    double dd = 0.0;
    for (int64_t k = 0; k < n; ++k) {
        const double g = gscale * G[k];
        double st;
        if (kind == 0) {
            st = -lr * g;
        } else if (kind == 1) {
            const double buf = mu * (double)s1[k] + g;
            if (s1_new) s1_new[k] = (float)buf;
            st = -lr * buf;
        } else {
            const double m = b1 * (double)s1[k] + (1.0 - b1) * g;
            const double v = b2 * (double)s2[k] + (1.0 - b2) * g * g;
            if (s1_new) s1_new[k] = (float)m;
            if (s2_new) s2_new[k] = (float)v;
            st = -lr * ((m / bc1) / (sqrt(v / bc2) + eps) + wd * (double)W[k]);
        }
        step[k] = st;
        dd += st * st;
    }
    double sscale = 1.0;
    if (clip == 1 && sqrt(dd) > frac * wnorm) sscale = frac * wnorm / sqrt(dd);
    for (int64_t k = 0; k < n; ++k) {
        const float wn = (float)((double)W[k] + sscale * step[k]);
        if (W_new) W_new[k] = wn;
        if (W_bf16) W_bf16[k] = orc_f32_to_bf16(wn);
    }
    free(step);
    return clip == 2 ? gscale : sscale;
}

/* Plain RNE conversion of an fp32 array to bf16 bits (test helper for the
 * update's bf16 output). */
void oracle_f32_to_bf16(int64_t n, const float* x, uint16_t* out) {
    for (int64_t k = 0; k < n; ++k) out[k] = orc_f32_to_bf16(x[k]);
}

/*
 * Eq. (cosine): out = { <X,Y>, ||X||^2, ||Y||^2, <X,Y> / (||X|| ||Y||) }.
 * Sequential fp64 sums in index order.
 */
void oracle_cosine(int64_t n, int dt, const void* X, const void* Y, double* out) {
    double xy = 0.0, xx = 0.0, yy = 0.0;
    for (int64_t k = 0; k < n; ++k) {
        double a = orc_load(dt, X, k), b = orc_load(dt, Y, k);
        xy += a * b;
        xx += a * a;
        yy += b * b;
    }
    out[0] = xy;
    out[1] = xx;
    out[2] = yy;
    out[3] = (xx > 0.0 && yy > 0.0) ? xy / (sqrt(xx) * sqrt(yy)) : 0.0;
}

/* Mean cross-entropy over tokens, (1/T) sum_t (lse_t - z_{t,y_t}), from the
 * per-token values returned by oracle_error_signal. */
double oracle_mean_ce(int64_t n, const double* lse, const double* zy) {
    double acc = 0.0;
    for (int64_t k = 0; k < n; ++k) acc += lse[k] - zy[k];
    return n > 0 ? acc / (double)n : 0.0;
}

/*
 * Update-magnitude ratio of App. C: for layer l, the fractional weight change
 * per unit learning rate ||g~ (x) h||_F / ||W||_F with g~ (x) h = G_l, and the
 * plain-SGD learning rate whose step -lr G_l has norm rel * ||W_l||_F (rel =
 * 0.01: the table's "1% step" column).  out[4 l + {0,1,2,3}] =
 * { ||G_l||^2, ||W_l||^2, ||G_l|| / ||W_l||, rel / (||G_l|| / ||W_l||) },
 * fp64 sums in index order (IEEE division: x/0 = inf, 0/0 = NaN).
 */
void oracle_norm_ratio(int64_t n_layers, int64_t n, int g_dt, const void* const* G, int w_dt,
                       const void* const* W, double rel, double* out) {
    for (int64_t l = 0; l < n_layers; ++l) {
        double gg = 0.0, ww = 0.0;
        for (int64_t k = 0; k < n; ++k) {
            double g = orc_load(g_dt, G[l], k), w = orc_load(w_dt, W[l], k);
            gg += g * g;
            ww += w * w;
        }
        double r = sqrt(gg) / sqrt(ww);
        out[4 * l + 0] = gg;
        out[4 * l + 1] = ww;
        out[4 * l + 2] = r;
        out[4 * l + 3] = rel / r;
    }
}
