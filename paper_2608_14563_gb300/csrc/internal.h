// internal.h -- launchers shared between the C-ABI layer and the kernel
// translation units.  Every launcher enqueues on `stream` and returns a
// cudaError_t (cudaSuccess when the launch was accepted).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace fpo {

// Device status bits, OR-ed into the status word at offset 0 of a workspace.
enum : unsigned int {
    kDevTargetRange = 1u,
    kDevTimeout = 2u,
};

struct DevInfo {
    int sm_count;
    int major, minor;
};
// Cached properties of the current device; false if the query failed.
bool current_device_info(DevInfo* out);

constexpr int kMaxDevices = 64;
// The current device's index, or -1 if it cannot be read (or is >= kMaxDevices).
int current_device();

// Raises Kern's dynamic shared-memory limit to `bytes` in the current device's context.
// A function attribute belongs to each context's copy of the module, so this runs once
// per device; a failed attempt is not remembered, and the next launch tries again.
template <auto Kern>
cudaError_t set_smem_limit(int bytes) {
    static std::atomic<bool> done[kMaxDevices];
    const int dev = current_device();
    if (dev < 0) return cudaErrorInvalidDevice;
    if (done[dev].load(std::memory_order_acquire)) return cudaSuccess;
    const cudaError_t e =
        cudaFuncSetAttribute(Kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) done[dev].store(true, std::memory_order_release);
    return e;
}

uint64_t wait_limit_ns();

// Counts one kernel launch of this library (process-wide); launches() reads the count.
void note_launch();
uint64_t launches();

// ------------------------------------------------------------ bf16 (tcgen05)
// Logits pass: part[T, n_tiles] (max, sum exp), zy[T] (target logits) and, when z is
// non-null, the fp32 logits z[T, V] (stored-logits algorithm).
cudaError_t launch_lse_partial_bf16(const void* yhat, const void* W_U, const int32_t* y, int T,
                                    int d, int V, float2* part, int part_ld, float* zy, float* z,
                                    unsigned* status, cudaStream_t s);
int lse_tile_n_bf16();

// Recompute pass for rows [0, Tc) of yhat: E[Tc, V] = s (softmax - onehot) in bf16.
cudaError_t launch_error_bf16(const void* yhat, const void* W_U, const int32_t* y, const float* lse,
                              int Tc, int d, int V, float s, void* E, unsigned* status,
                              cudaStream_t st);

// Projection: g[Tc, d] = E[Tc, V] W_U (fp32 out).  sk_scratch: proj_sk_scratch_bytes() of
// device memory for the split-K tail of the 256 x 512 kernel (or null: whole tiles only).
cudaError_t launch_proj_bf16(const void* E, const void* W_U, int Tc, int d, int V, float* g,
                             float* sk_scratch, unsigned* status, cudaStream_t st);
size_t proj_sk_scratch_bytes();

// Direct algorithm, logits pass anchored at c = anchor[t] (z never stored):
// P[T, V] = exp(z - c) in bf16 with the target column zero, and per (row, 256-column
// tile) the sums of P before rounding, su[T, part_ld], of the rounded P, sx[T, part_ld],
// and of the rounded P times z, qz[T, part_ld].
cudaError_t launch_anchor_prob_bf16(const void* yhat, const void* W_U, const int32_t* y,
                                    const float* anchor, int T, int d, int V, float* su, float* sx,
                                    float* qz, int part_ld, void* P, unsigned* status,
                                    cudaStream_t st);
// Direct algorithm, rows outside the anchor window (yfix[*fix_count, d], the gathered
// yhat rows, capacity Tc; the row count is read on the device, none: the kernels return
// at once).  First pass: part[fix[i], tile] = (max, sum exp(z - max)) of every tile.
cudaError_t launch_fixup_lse_bf16(const void* yfix, const void* W_U, const int* fix,
                                  const int* fix_count, int Tc, int d, int V, float2* part,
                                  int part_ld, unsigned* status, cudaStream_t st);
// Second pass, once lse is known: P[fix[i], :] = exp(z - lse) in bf16 with the target
// column zero, and the sx, qz sums of those rows as the logits pass leaves them.
cudaError_t launch_fixup_logits_bf16(const void* yfix, const void* W_U, const int* fix,
                                     const int* fix_count, const int32_t* y, const float* lse,
                                     int Tc, int d, int V, void* P, float* sx, float* qz,
                                     int n_tiles, unsigned* status, cudaStream_t st);
// Direct algorithm, projection with the final-norm VJP fused in: per row
// g = alpha (.) (P W_U) + beta (.) W_U[y] and g~[Tc, d] (bf16) =
// (w (.) g - (h / rho) cv / d) / max(rho, min_rms).
cudaError_t launch_proj_vjp_bf16(const void* P, const void* W_U, const int32_t* y,
                                 const float* alpha, const float* beta, const float* cv,
                                 const float* rho, const void* h, const void* w, float min_rms,
                                 int Tc, int d, int V, void* g_tilde, float* sk_scratch,
                                 unsigned* status, cudaStream_t st);

// Grouped pseudogradient update over n layers, layer l with signal g[l] (host array).
cudaError_t launch_update_bf16(int n, int T, int d, int d_ff, const void* const* g,
                               const void* const* A, float lr, float* const* W_master,
                               void* const* W_out, void* const* G_out, unsigned* status,
                               cudaStream_t st);

// Grouped pseudogradients only: G_out[l] (fp32 [d, d_ff]) = g[l]^T A[l].
cudaError_t launch_grad_bf16(int n, int T, int d, int d_ff, const void* const* g,
                             const void* const* A, float* const* G_out, unsigned* status,
                             cudaStream_t st);

// Grouped pseudogradients with the diagnostic's cosine: G_out[l] (bf16 [d, d_ff]) =
// g[l]^T A[l], and out[4 l ..] = <G_l, Y_l>, ||G_l||^2, ||Y_l||^2, cos_l of the stored
// G_l against Y[l] (bf16), from per-(tile, warp) partial sums in `part`
// (grad_cosine_partial_bytes) without a second pass over G.
size_t grad_cosine_partial_bytes(int n, int d, int d_ff);
cudaError_t launch_grad_cosine_bf16(int n, int T, int d, int d_ff, const void* const* g,
                                    const void* const* A, const void* const* Y,
                                    void* const* G_out, float* part, double* out,
                                    unsigned* status, cudaStream_t st);

// SwiGLU gate / up signals: dA, dB [T, d_ff] from error_h = g W3 (W3 [d, d_ff]) and the
// cached pre-activations a, b [T, d_ff].
cudaError_t launch_swiglu_bf16(int T, int d, int d_ff, const void* g, const void* W3,
                               const void* a, const void* b, void* dA, void* dB, unsigned* status,
                               cudaStream_t st);
cudaError_t launch_swiglu_f32(int T, int d, int d_ff, const float* g, const float* W3,
                              const float* a, const float* b, float* dA, float* dB,
                              cudaStream_t st);

// Optimizer step of n layers of n_elem elements from fp32 G (optimizer.cu).
struct OptimParams {
    int kind;          // 0 SGD, 1 SGD with momentum, 2 AdamW
    int clip;          // 0 none, 1 the step, 2 the gradient
    float lr, momentum, beta1, beta2, eps, weight_decay, clip_frac;
    float inv_bc1, inv_sqrt_bc2;  // AdamW bias corrections 1/(1-b1^t), 1/sqrt(1-b2^t)
};
size_t optim_partials_bytes(int n_layers);
// The step clip's first optimizer pass fused into the pseudogradient GEMM (bf16): the
// state advanced, the unclipped steps in D and (||W||^2, ||d||^2) per (layer, 256 rows,
// column tile, 32 rows) in part, for launch_opt_step_clip.
cudaError_t launch_opt_step_bf16(int n, int T, int d, int d_ff, const void* const* g,
                                 const void* const* A, const OptimParams& op,
                                 float* const* W_master, float* const* s1, float* const* s2,
                                 float* const* D, float* part, unsigned* status, cudaStream_t st);
size_t opt_step_partial_bytes(int n_layers, int d, int d_ff);
cudaError_t launch_opt_step_clip(int n_layers, size_t n_elem, const OptimParams& op,
                                 const float* part, int slots, float* const* D,
                                 float* const* W_master, void* const* W_out, float* scales,
                                 cudaStream_t st);
cudaError_t launch_optimizer(int dtype, int n_layers, size_t n_elem, const OptimParams& op,
                             float* const* G, float* const* W_master, void* const* W_out,
                             float* const* s1, float* const* s2, double* partials, float* scales,
                             cudaStream_t st);

// Which tcgen05 GEMM kernel the launchers use: 0 = single-CTA 128 x 256 tiles,
// 1 = CTA-pair 256 x 256 tiles.
void set_gemm_variant(int v);
int gemm_variant();
// Override of the L2 rasterisation band height in tiles (0 = default).
void set_band_override(int b);

// Plain GEMM with an fp32 store epilogue (test entry point).
cudaError_t launch_test_gemm_bf16(int M, int N, int K, bool a_mn, bool b_mn, const void* A,
                                  const void* B, float* C, unsigned* status, cudaStream_t st);

// ------------------------------------------------------------ row-wise kernels
// With anchor non-null (direct algorithm) also anchor[t] = <yhat_t, W_U[y_t]>.
cudaError_t launch_rmsnorm_fwd(int dtype, const void* h, const void* w, int T, int d, float eps,
                               void* yhat, float* rho, const int32_t* y, int V, unsigned* status,
                               cudaStream_t st, const void* W_U = nullptr,
                               float* anchor = nullptr);
// Direct algorithm (bf16), per token of a chunk with S = sum su, S' = sum sx and
// Qz = sum qz over the tiles: rows inside the anchor window get lse = c + log(1 + S),
// ce = log(1 + S), the projection's row factors alpha = s / (1 + S), beta = -alpha S'
// and the VJP's row term cv = alpha (Qz - c S'); the others are appended to
// fix[0 .. *fix_count) (atomically).
cudaError_t launch_direct_combine(const float* su, const float* sx, const float* qz, int n_tiles,
                                  int T, int V,
                                  const int32_t* y, const float* anchor, float s, float* lse,
                                  float* ce, float* alpha, float* beta, float* cv, int* fix,
                                  int* fix_count, cudaStream_t st);
// Rows outside the anchor window: out[i, :] = yhat[fix[i], :] for i < *fix_count (bf16,
// d a multiple of 8); after the first fixup pass their lse and ce from the (max, sum)
// partials; after the second their row factors alpha = s, beta = -s S' and
// cv = s (Qz - c S').
cudaError_t launch_gather_rows(const void* yhat, const int* fix, const int* fix_count, int d,
                               void* out, cudaStream_t st);
cudaError_t launch_direct_fixup_lse(const float2* part, const int* fix, const int* fix_count,
                                    int n_tiles, const float* anchor, float* lse, float* ce,
                                    cudaStream_t st);
cudaError_t launch_direct_fixup_factors(const float* sx, const float* qz, const int* fix,
                                        const int* fix_count, int n_tiles, const float* anchor,
                                        float s, float* alpha, float* beta, float* cv,
                                        cudaStream_t st);
cudaError_t launch_lse_combine(const float2* part, int n_tiles, int T, const float* zy,
                               float* lse, float* ce, cudaStream_t st);
cudaError_t launch_mean(const float* x, int n, float* out, cudaStream_t st);
// Stored-logits algorithm: E[M, V] = s (exp(z - lse) - onehot(y)) from z[M, V] fp32, in
// dtype (bf16 through the same formula as the recompute epilogue, or fp32).
cudaError_t launch_error_from_logits(int dtype, const float* z, const float* lse, const int32_t* y,
                                     int M, int V, float s, void* E, cudaStream_t st);
// dst[n] = src[n] rounded to dtype (a plain copy for fp32).
cudaError_t launch_cast_f32(int dtype, const float* src, size_t n, void* dst, cudaStream_t st);
cudaError_t launch_rmsnorm_vjp(int dtype, const float* g, const void* h, const void* w,
                               const float* rho, int T, int d, float min_rms, void* out,
                               cudaStream_t st);
// Layer-specific signals: out[l] = pre-MLP VJP at x[l] of (post-FFN VJP at m[l] of g), either
// stage skipped when its array is null (not both); one launch for all layers.
cudaError_t launch_layer_signals(int dtype, int n_layers, const void* g, const void* const* m,
                                 const void* const* gamma_post, const void* const* x,
                                 const void* const* gamma_pre, void* const* out, int T, int d,
                                 float eps, float min_rms, cudaStream_t st);

// One block waiting on an mbarrier nothing arrives on, bounded by limit_ns.
cudaError_t launch_wait_timeout(unsigned* status, uint64_t limit_ns, cudaStream_t st);

// ------------------------------------------------------------ grouped per-layer reductions
constexpr int kNrMaxLayers = 64;
// Blocks per layer of the first pass; partial needs n_layers * blocks * 3 doubles.
int norm_ratio_blocks(int n_layers, int64_t n);
// out[4 l ..] = ||G_l||^2, ||W_l||^2, ||G_l|| / ||W_l||, rel / ratio (device, fp64);
// dtypes 0 = fp32, 1 = bf16.
cudaError_t launch_norm_ratio(int g_dtype, int w_dtype, int n_layers, int64_t n,
                              const void* const* G, const void* const* W, double rel,
                              double* partial, int blocks, double* out, cudaStream_t st);
// out[4 l ..] = <X_l,Y_l>, ||X_l||^2, ||Y_l||^2, cos_l for every layer (dtype of both).
cudaError_t launch_cosine_grouped(int dtype, int n_layers, int64_t n, const void* const* X,
                                  const void* const* Y, double* partial, int blocks, double* out,
                                  cudaStream_t st);

// ------------------------------------------------------------ cosine
int cosine_blocks(int64_t n);
cudaError_t launch_cosine(int dtype, int64_t n, const void* X, const void* Y, double* partial,
                          int blocks, double* out, cudaStream_t st);

// ------------------------------------------------------------ fp32 SIMT path
constexpr int kSimtTile = 64;
cudaError_t launch_lse_partial_f32(const float* yhat, const float* W_U, const int32_t* y, int T,
                                   int d, int V, float2* part, int part_ld, float* zy, float* z,
                                   cudaStream_t st);
cudaError_t launch_error_f32(const float* yhat, const float* W_U, const int32_t* y,
                             const float* lse, int Tc, int d, int V, float s, float* E,
                             cudaStream_t st);
cudaError_t launch_proj_f32(const float* E, const float* W_U, int Tc, int d, int V, float* g,
                            cudaStream_t st);
cudaError_t launch_update_f32(int n, int T, int d, int d_ff, const float* const* g,
                              const float* const* A, float lr, float* const* W_master,
                              float* const* W_out, float* const* G_out, cudaStream_t st);

}  // namespace fpo
