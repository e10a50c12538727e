/*
 * fpo.h -- C ABI of libfpo, the GB300 (sm_103a) implementation of the
 * per-step pseudogradient update of Forward-Pass-Only MLP training (FPO) from
 * "Forward Pass Domain Adaptation (Without Cross-Layer Backpropagation)".
 *
 * One FPO step on the down-projections is
 *
 *     fpo_error_signal(...)            Sec. 3.1 steps 2-4 + App. E
 *     for each target layer l:
 *         fpo_layer_update(...)        Sec. 3.1 step 5, Eq. (w3update), App. A
 *     (or one fpo_layer_update_grouped call for all target layers)
 *
 * and the layer-viability diagnostic of Sec. 2.2 reduces pairs of gradients
 * with fpo_cosine (one pair) or fpo_cosine_grouped (every layer in one call).
 * Further entry points cover the rest of the method around that step: the
 * post-FFN and pre-MLP RMSNorm VJPs and per-layer signals (fpo_rmsnorm_vjp,
 * fpo_layer_signals, fpo_layer_update_grouped_signals), optimizers with the relative clip
 * (fpo_layer_optimize_grouped), the gate/up signals through the cached
 * W3_init (fpo_gate_up_signals) and the App. C update-magnitude ratio
 * (fpo_norm_ratio).  fpo_h2d_copy stages a step's inputs from host memory.
 *
 * Conventions (all entry points)
 * ------------------------------
 * - Tensor arguments are CUDA device pointers to dense row-major arrays,
 *   16-byte aligned.  The caller owns every buffer; the library allocates
 *   and frees no memory and never synchronises, except fpo_get_device_status.
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   Every call only enqueues work on it and returns.
 * - The return value reports errors the host can see (null pointers, shapes,
 *   dtype, alignment, workspace size, device architecture, CUDA launch
 *   errors).  After such an error nothing was enqueued.
 * - Errors only the device can see (a target id outside [0, V), a bounded
 *   wait inside a kernel that ran out) set bits of a status word at offset 0
 *   of the call's workspace.  Each call clears that word when it starts;
 *   fpo_get_device_status reads it after the call.
 * - dtype FPO_BF16: every floating-point tensor argument except the fp32
 *   master weights and lse/loss outputs is bf16; arithmetic is bf16 tensor-core
 *   MMA with fp32 accumulation and fp32 elementwise math.  d, V and d_ff must be
 *   multiples of 8 (16-byte rows for the TMA engine).
 *   dtype FPO_F32: every floating-point tensor is fp32 and all arithmetic is
 *   fp32 FFMA (no TF32); any positive shape is accepted.
 * - The library only runs on compute capability 10.3 (GB300); any other
 *   device returns FPO_ERR_ARCH.
 * - Every call runs on the calling thread's current device.  One process may
 *   drive several GPUs: a kernel's launch setup (its shared-memory limit, the
 *   clusters resident at once) is made once per device, on that device's
 *   first call.
 */
#ifndef FPO_H_
#define FPO_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FPO_ABI_VERSION 2

/* Largest number of layers one fpo_layer_update_grouped call accepts. */
#define FPO_MAX_GROUPED_LAYERS 64

/* Largest number of buffers one fpo_h2d_copy call accepts. */
#define FPO_MAX_COPY_BUFFERS 64

typedef enum fpo_dtype {
    FPO_F32 = 0,
    FPO_BF16 = 1
} fpo_dtype;

typedef enum fpo_status {
    FPO_OK = 0,
    FPO_ERR_NULL = 1,          /* a required pointer is NULL */
    FPO_ERR_SHAPE = 2,         /* a size is negative, unsupported, or too large */
    FPO_ERR_DTYPE = 3,         /* unknown dtype */
    FPO_ERR_ALIGN = 4,         /* a tensor pointer is not 16-byte aligned */
    FPO_ERR_WORKSPACE = 5,     /* workspace NULL or smaller than the query returned */
    FPO_ERR_ARCH = 6,          /* current device is not compute capability 10.3 */
    FPO_ERR_CUDA = 7,          /* a CUDA runtime/driver call failed */
    FPO_ERR_TARGET_RANGE = 8,  /* device: a target id was outside [0, V) */
    FPO_ERR_TIMEOUT = 9,       /* device: a bounded wait inside a kernel ran out */
    FPO_ERR_ARG = 10           /* any other invalid argument */
} fpo_status;

/*
 * How fpo_error_signal forms the error matrix E = s (softmax(z) - 1_y) without
 * ever holding all T x V logits:
 *  FPO_ES_RECOMPUTE      a logits pass keeps only per-(token, vocabulary tile)
 *                        max / sum-exp partials; a second pass recomputes the
 *                        logits GEMM and writes E (bf16) for one token chunk.
 *  FPO_ES_STORED_LOGITS  the logits pass also stores the chunk's fp32 logits; a
 *                        bandwidth-bound kernel turns them into E once the
 *                        log-sum-exp is known (one GEMM instead of two, at the
 *                        cost of T_chunk x V x 4 bytes of workspace and ~3 passes
 *                        over it in HBM).
 *  FPO_ES_DIRECT         (bf16 only) no E at all.  With the anchor c_t =
 *                        <xhat_t (.) norm_w, W_U[y_t]> (the target logit, from the
 *                        RMSNorm forward), the logits pass writes
 *                        P_tj = exp(z_tj - c_t) in bf16 with the target column 0,
 *                        lse_t = c_t + log(1 + sum_j P_tj) before rounding, and
 *                        the projection forms
 *                          g_t = s e^{c_t - lse_t} (P_t W_U - S'_t W_U[y_t]),
 *                        S'_t the sum of row t of the rounded P.
 *                        This equals e_t W_U exactly in real arithmetic (the
 *                        target entry of e_t is -sum of the others), rounds each
 *                        probability to bf16 once like E, and saves the E pass:
 *                        T_chunk x V x 2 bytes of workspace.  The projection's
 *                        epilogue also applies the final-norm VJP, writing g~
 *                        directly: the row term <xhat_t, norm_w (.) g_t> is
 *                        s e^{c_t - lse_t} sum_j P_tj (z_tj - c_t), with sums the
 *                        logits pass keeps (<yhat_t, W_U[j]> = z_tj).  Rows
 *                        with S'_t outside [2^-80, 2^80] (token cross-entropy
 *                        beyond ~55 nats, or 1 - p_target below ~1e-24) are
 *                        gathered and recomputed by the same tensor-core logits
 *                        GEMM, first for a max-based lse_t, then anchored at
 *                        lse_t, before the projection (their row count read on
 *                        the device).  A row with an out-of-range target gets
 *                        g~ = 0, and lse 0 and loss term 0.
 *  FPO_ES_AUTO           the library's choice: FPO_ES_DIRECT for bf16,
 *                        FPO_ES_STORED_LOGITS for fp32 (where DIRECT also runs
 *                        the stored-logits algorithm).
 * RECOMPUTE and STORED_LOGITS compute every value with the same arithmetic:
 * their outputs are bit-identical.  DIRECT agrees with them to the bf16
 * rounding of the probabilities.  Results are deterministic; across t_chunk
 * values they are bit-identical while the projection has whole tiles (fewer
 * than one wave), and otherwise agree to rounding (its last partial wave is
 * split into k ranges).
 */

/* Tokens per error-matrix chunk when fpo_error_signal_desc.t_chunk is 0. */
#define FPO_AUTO_T_CHUNK 8192
typedef enum fpo_es_algo {
    FPO_ES_AUTO = 0,
    FPO_ES_RECOMPUTE = 1,
    FPO_ES_STORED_LOGITS = 2,
    FPO_ES_DIRECT = 3
} fpo_es_algo;

/* Error-signal problem description (Sec. 3.1 steps 2-4, App. E). */
typedef struct fpo_error_signal_desc {
    int64_t T;          /* tokens (B x L flattened), >= 0; T = 0 launches no
                           kernel (the status word and loss_out are zeroed)      */
    int64_t d;          /* model width (RMSNorm size, unembedding input)          */
    int64_t V;          /* vocabulary size                                        */
    int32_t dtype;      /* fpo_dtype of h, norm_w, W_U and g_out                  */
    float eps;          /* RMSNorm epsilon, inside the square root (App. E)      */
    float min_rms;      /* floor on rho in the 1/rho prefactor of the VJP (0.5)  */
    float loss_scale;   /* s in e = s (softmax(z) - 1_y); 1/T = mean-reduced CE */
    int32_t algo;       /* fpo_es_algo                                            */
    int64_t t_chunk;    /* tokens per error-matrix chunk; 0 = FPO_AUTO_T_CHUNK    */
    void* const* stage_events;  /* NULL, or caller-created cudaEvent_t recorded on
                                   the stream at the stage boundaries (profiling;
                                   see below)                                     */
    int32_t stage_events_per_chunk; /* 0: FPO_STAGE_EVENTS events; 1: the stages of
                                   every token chunk, fpo_error_signal_stage_events()
                                   events (see below)                             */
} fpo_error_signal_desc;

/*
 * Stage boundaries of fpo_error_signal at which desc->stage_events[i] is
 * recorded: 0 start, 1 after the RMSNorm forward, 2 after the logits pass (of
 * the last token chunk for FPO_ES_STORED_LOGITS), 3 after the log-sum-exp
 * combine (and loss), 4 after the recompute pass (FPO_ES_RECOMPUTE), the
 * logits-to-E conversion (FPO_ES_STORED_LOGITS) or the anchor-window fixup
 * (FPO_ES_DIRECT; with the loss mean) of the last token chunk, 5
 * after the projection of the last token chunk, 6 after the final-norm VJP
 * (under FPO_ES_DIRECT the projection applies the VJP: 5 to 6 is empty).
 * With one chunk, consecutive events bracket one kernel each (plus the loss
 * mean in [2]-[3]).
 * With stage_events_per_chunk = 1 and n token chunks the events are 3 + 4 n:
 * 0 start, 1 after the RMSNorm forward, then for chunk c = 0 .. n-1:
 * 2 + 4c after its logits pass, 3 + 4c after its combine (and, last chunk and
 * not FPO_ES_DIRECT, the loss mean), 4 + 4c after its E / fixup stage (and,
 * last chunk and FPO_ES_DIRECT, the loss mean), 5 + 4c after its projection;
 * and 2 + 4n after the VJP.  (FPO_ES_RECOMPUTE runs one logits pass and one
 * combine over all tokens: they fill chunk 0's first two slots; the other
 * chunks record those two at the chunk's start.)
 */
#define FPO_STAGE_EVENTS 7

/* Number of stage events `desc` asks for (FPO_STAGE_EVENTS, or 3 + 4 n with
 * stage_events_per_chunk), or 0 on a bad desc. */
int32_t fpo_error_signal_stage_events(const fpo_error_signal_desc* desc);

/* Bytes of workspace fpo_error_signal needs for `desc` (0 on a bad desc). */
size_t fpo_error_signal_workspace(const fpo_error_signal_desc* desc);

/*
 * fpo_error_signal -- output-layer error projected to the residual stream and
 * through the final RMSNorm's Jacobian (Sec. 3.1 steps 2-4; Eq. (gproj);
 * App. E Eq. (rmsnorm-vjp) with the min-RMS clamp).
 *
 * For every token t:
 *   rho_t = sqrt(mean_j h_tj^2 + eps),  xhat_t = h_t / rho_t
 *   z_t   = (norm_w (.) xhat_t) W_U^T                        (logits, never stored)
 *   e_t   = s (softmax(z_t) - onehot(targets[t]))
 *   g_t   = e_t W_U                                          (Eq. gproj)
 *   g~_t  = (norm_w (.) g_t - xhat_t <xhat_t, norm_w (.) g_t> / d) / max(rho_t, min_rms)
 *
 * h        [T, d]   final pre-norm residual (dtype)
 * norm_w   [d]      final RMSNorm weight (dtype)
 * W_U      [V, d]   unembedding, nn.Linear layout (dtype)
 * targets  [T]      int32 next-token ids in [0, V); out-of-range ids set
 *                   FPO_ERR_TARGET_RANGE in the device status
 * g_out    [T, d]   g~ (dtype)
 * lse_out  [T]      fp32 log-sum-exp of each token's logits, or NULL
 * loss_out [1]      fp32 mean cross-entropy (1/T) sum_t (lse_t - z_t,y_t), or NULL
 * workspace         device scratch of fpo_error_signal_workspace(desc) bytes,
 *                   256-byte aligned; owned by the caller, must not be shared
 *                   with a call that runs concurrently
 */
int32_t fpo_error_signal(const fpo_error_signal_desc* desc, const void* h, const void* norm_w,
                         const void* W_U, const int32_t* targets, void* g_out, float* lse_out,
                         float* loss_out, void* workspace, size_t workspace_bytes, void* stream);

/* Bytes of workspace fpo_layer_update / fpo_layer_update_grouped need. */
size_t fpo_layer_update_workspace(void);

/*
 * fpo_layer_update -- pseudogradient of one target layer's down-projection and
 * its plain-SGD step on the fp32 master copy (Sec. 3.1 step 5, Eq. (w3update);
 * App. A, fp32 master weights cast to the working dtype).
 *
 *   G = g~^T A                    [d, d_ff], fp32 accumulation over T
 *   W_master <- W_master - lr G   (fp32, one rounding)
 *   W_out    <- W_master          (rounded to dtype, nearest-even)
 *
 * g        [T, d]      g~ from fpo_error_signal (dtype)
 * A        [T, d_ff]   the layer's cached down-projection input h_mid (dtype)
 * W_master [d, d_ff]   fp32, updated in place; NULL computes G only
 * W_out    [d, d_ff]   updated weight in dtype, or NULL; needs W_master
 * G_out    [d, d_ff]   G in dtype, or NULL
 * workspace            fpo_layer_update_workspace() bytes (device status word)
 * At least one of W_master and G_out must be non-NULL.  lr = 0 leaves
 * W_master bit-identical.
 */
int32_t fpo_layer_update(int64_t T, int64_t d, int64_t d_ff, int32_t dtype, const void* g,
                         const void* A, float lr, float* W_master, void* W_out, void* G_out,
                         void* workspace, size_t workspace_bytes, void* stream);

/*
 * fpo_layer_update_grouped -- fpo_layer_update for n_layers target layers that
 * share g~ and the shapes, in one launch (1 <= n_layers <= FPO_MAX_GROUPED_LAYERS).
 * A, W_master, W_out and G_out are HOST arrays of n_layers device pointers;
 * W_master, W_out or G_out may be NULL as a whole (no such output for any
 * layer), and individual entries may be NULL with the same meaning per layer.
 */
int32_t fpo_layer_update_grouped(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                 int32_t dtype, const void* g, const void* const* A, float lr,
                                 float* const* W_master, void* const* W_out,
                                 void* const* G_out, void* workspace, size_t workspace_bytes,
                                 void* stream);

/*
 * fpo_layer_update_grouped_signals -- fpo_layer_update_grouped where layer l
 * has its own signal g[l] (HOST array of n_layers device pointers, [T, d]
 * each): the layer-specific g~^(l) of Sec. 3.1 step 4 for architectures with a
 * per-layer post-feedforward and / or pre-MLP RMSNorm (OLMo-2, Qwen3, Gemma 3),
 * obtained from g~ with fpo_layer_signals (or fpo_rmsnorm_vjp at that layer's cached
 * MLP output).  Entries may repeat.
 */
int32_t fpo_layer_update_grouped_signals(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                         int32_t dtype, const void* const* g,
                                         const void* const* A, float lr, float* const* W_master,
                                         void* const* W_out, void* const* G_out, void* workspace,
                                         size_t workspace_bytes, void* stream);

/*
 * fpo_layer_signals -- the layer-specific signals g~^(l) (Sec. 3.1 step 4; Sec. 3.2 and
 * the App. E table of norms per model family) for n_layers target layers in one launch
 * (1 <= n_layers <= FPO_MAX_GROUPED_LAYERS).  For layer l and every token, starting from
 * the shared signal g (g~ after the final norm's Jacobian, [T, d]):
 *
 *   u        = post-FFN RMSNorm VJP of g at m[l] with weight gamma_post[l]   (m given)
 *   g_out[l] = pre-MLP RMSNorm VJP of u at x[l] with weight gamma_pre[l]     (x given)
 *
 * each the expression of fpo_rmsnorm_vjp with its own rho = sqrt(mean x^2 + eps) and
 * the min-RMS clamp; OLMo-2 composes the post-FFN norm only, Qwen3 the pre-MLP norm
 * only, Gemma 3 both, in this order.  m[l] is the layer's cached MLP output (the input
 * of its post-feedforward norm), x[l] the input of its pre-MLP norm (the residual stream
 * entering the MLP block).  The intermediate u stays in fp32 registers: each row of g,
 * m[l] and x[l] is read once per layer (rows up to 8192 bf16 elements; longer bf16 rows
 * and fp32 rows are read in three passes) and g_out[l] written once.
 *
 * m, gamma_post, x, gamma_pre and g_out are HOST arrays of n_layers device pointers
 * ([T, d] rows and [d] weights, all in dtype).  m and gamma_post are both NULL (no
 * post-FFN norm) or both given, likewise x and gamma_pre, and at least one norm is
 * given (else FPO_ERR_ARG).  Entries of an input array may repeat; g_out[l] may not
 * alias g, any input, or another g_out.  bf16 needs d % 8 == 0; every pointer 16-byte
 * aligned (FPO_ERR_ALIGN).  fp32 accumulation; no workspace; asynchronous on `stream`.
 */
int32_t fpo_layer_signals(int32_t n_layers, int64_t T, int64_t d, int32_t dtype, const void* g,
                          const void* const* m, const void* const* gamma_post,
                          const void* const* x, const void* const* gamma_pre, float eps,
                          float min_rms, void* const* g_out, void* stream);

/*
 * fpo_rmsnorm_vjp -- the closed-form RMSNorm Jacobian applied to an upstream
 * gradient (App. E Eq. (rmsnorm-vjp) with the min-RMS clamp), at any norm the
 * method corrects for; for the post-feedforward norm of OLMo-2 / Gemma 3
 * (Sec. 3.2) x is the layer's cached MLP output and gamma its post-FFN weight:
 *
 *   rho = sqrt(mean_j x_j^2 + eps),  xhat = x / rho
 *   g_out = (gamma (.) g - xhat <xhat, gamma (.) g> / d) / max(rho, min_rms)
 *
 * g, x, g_out [T, d] and gamma [d] in dtype; g_out may not alias g or x.
 * fp32 accumulation; no workspace; asynchronous on `stream`.
 */
int32_t fpo_rmsnorm_vjp(int64_t T, int64_t d, int32_t dtype, const void* g, const void* x,
                        const void* gamma, float eps, float min_rms, void* g_out, void* stream);

/* Optimizers of Sec. 3.1 on the fp32 master copies. */
typedef enum fpo_optimizer_kind {
    FPO_OPT_SGD = 0,           /* step = -lr G                                           */
    FPO_OPT_SGD_MOMENTUM = 1,  /* buf = mu buf + G; step = -lr buf                       */
    FPO_OPT_ADAMW = 2          /* m, v moments; step = -lr (mhat/(sqrt(vhat)+eps) + wd W) */
} fpo_optimizer_kind;

/* The relative clip of App. A, ||.||_F <= clip_frac ||W||_F (W before the step). */
typedef enum fpo_clip_mode {
    FPO_CLIP_NONE = 0,
    FPO_CLIP_STEP = 1,      /* scale the optimizer's step (the update Delta W) */
    FPO_CLIP_GRADIENT = 2   /* scale G before the optimizer sees it            */
} fpo_clip_mode;

typedef struct fpo_optimizer_desc {
    int32_t kind;          /* fpo_optimizer_kind                                  */
    int32_t clip;          /* fpo_clip_mode                                       */
    float lr;
    float momentum;        /* SGD with momentum: mu (0.9)                         */
    float beta1, beta2;    /* AdamW moment decays (0.9, 0.999)                    */
    float adam_eps;        /* AdamW epsilon (1e-8)                                */
    float weight_decay;    /* AdamW decoupled weight decay (0.01)                 */
    float clip_frac;       /* relative clip bound (0.01)                          */
    int64_t step;          /* AdamW step index t >= 1, for the bias corrections   */
} fpo_optimizer_desc;

/* Bytes of workspace fpo_layer_optimize_grouped needs. */
size_t fpo_layer_optimize_workspace(int32_t n_layers, int64_t d, int64_t d_ff);

/*
 * fpo_layer_optimize_grouped -- the pseudogradient of every target layer
 * (Eq. (w3update), as in fpo_layer_update_grouped_signals) followed by an
 * optimizer step on its fp32 master (Sec. 3.1: SGD with momentum 0.9 or AdamW
 * with weight decay 0.01) with the relative clip of App. A:
 *   G_l = g[l]^T A[l]                 fp32, in the workspace
 *   c   = clip factor from ||G_l||, ||step_l|| and ||W_l|| (see fpo_clip_mode)
 *   state_l, W_master,l updated; W_out,l = W_master,l rounded to dtype.
 * state1[l] is the momentum buffer (SGD_MOMENTUM) or the first moment (ADAMW),
 * state2[l] the second moment (ADAMW); fp32 [d, d_ff], updated in place (NULL
 * arrays when the optimizer has no such state).  W_out may be NULL.  The clip
 * needs all of G_l (or of the steps) before any element steps, so the workspace
 * holds n_layers x d x d_ff x 4 bytes: G_l, or with bf16 and FPO_CLIP_STEP the
 * unclipped steps, which the GEMM's epilogue forms from G_l (and the state) without
 * storing G_l.  g, A, W_out: as fpo_layer_update_grouped_signals.
 */
int32_t fpo_layer_optimize_grouped(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                   int32_t dtype, const void* const* g, const void* const* A,
                                   const fpo_optimizer_desc* opt, float* const* W_master,
                                   void* const* W_out, float* const* state1,
                                   float* const* state2, void* workspace, size_t workspace_bytes,
                                   void* stream);

/*
 * fpo_gate_up_signals -- the hidden-space signals for the gate (W1) and up (W2)
 * projections of one SwiGLU target layer (Sec. 3.1 step 5, Eq. (errh)), with the
 * cached W3_init as the fixed feedback matrix:
 *
 *   error_h = g W3_init                                   [T, d_ff]
 *   dA = error_h (.) b (.) silu'(a),  dB = error_h (.) silu(a)
 *
 * where a = x W1^T and b = x W2^T are the layer's cached gate and up
 * pre-activations (h_mid = silu(a) (.) b) and silu'(a) = sigma(a)(1 + a(1 - sigma(a))).
 * The W1 / W2 pseudogradients are then G1 = dA^T x, G2 = dB^T x ([d_ff, d], the
 * nn.Linear layout of W1, W2), i.e. fpo_layer_update_grouped_signals with
 * signals {dA, dB} and "activations" {x, x} (x: the MLP input [T, d]).
 * The paper leaves the activation derivative to the MLP; these are SwiGLU's.
 *
 * g [T, d], W3_init [d, d_ff], a, b, dA, dB [T, d_ff], all in dtype.
 * workspace: fpo_layer_update_workspace() bytes (device status word).
 */
int32_t fpo_gate_up_signals(int64_t T, int64_t d, int64_t d_ff, int32_t dtype, const void* g,
                            const void* W3_init, const void* a, const void* b, void* dA, void* dB,
                            void* workspace, size_t workspace_bytes, void* stream);

/* Bytes of workspace fpo_cosine needs for n elements. */
size_t fpo_cosine_workspace(int64_t n);

/*
 * fpo_cosine -- the layer-viability diagnostic's reduction (Sec. 2.2,
 * Eq. (cosine)): cos = <X, Y> / (||X|| ||Y||) over n elements.
 *
 * X, Y  [n]  dtype (e.g. a pseudogradient and a true gradient, flattened)
 * out   [4]  device fp64: <X,Y>, ||X||^2, ||Y||^2, cos (cos = 0 if a norm is 0)
 * Per-thread partial sums are fp32, everything after is fp64, and the
 * reduction order is fixed, so repeated calls give identical bits.
 */
int32_t fpo_cosine(int64_t n, int32_t dtype, const void* X, const void* Y, double* out,
                   void* workspace, size_t workspace_bytes, void* stream);

/*
 * fpo_cosine_noalloc -- fpo_cosine for callers that cannot allocate device
 * memory: code running where cudaMalloc is off limits or would break the
 * caller's own memory accounting (inside another runtime's fixed memory pool,
 * a custom allocator, an embedded or real-time loop), which also has no
 * workspace to hand in.  The paper has no counterpart; this is a property of
 * the library, not of the method.
 *
 * Same inputs, output and result as fpo_cosine (bit-identical: the same
 * kernels, block count and summation order), but the pass-1 partial sums live
 * in a static device array inside libfpo of 1024 fp64 triples (24 KiB, held by
 * every GPU that loads the library until the process exits).  A call needs
 * cosine-blocks(n) <= 2 x SM count slots (304 on GB300, for any n); a device
 * whose launch would need more than 1024 returns FPO_ERR_WORKSPACE and
 * enqueues nothing.  The call allocates nothing: no cudaMalloc, no cudaFree,
 * no allocating library routine.
 *
 * - The first call on each device looks up the array's device address
 *   (cudaGetSymbolAddress) with that device current; make that first call
 *   before any stream capture.  A lookup that fails returns FPO_ERR_CUDA and is
 *   retried by the next call; only a successful one is kept.
 * - All calls on a device share the one array, which keeps the last call's
 *   partials.  Every slot a call reads is written by the same call first, so
 *   nothing needs clearing, but two calls that overlap on the GPU (different
 *   streams, or different host threads) race on the array: serialise them.
 */
int32_t fpo_cosine_noalloc(int64_t n, int32_t dtype, const void* X, const void* Y, double* out,
                           void* stream);

/* Bytes of workspace fpo_cosine_grouped needs (0 for an invalid n_layers or n). */
size_t fpo_cosine_grouped_workspace(int32_t n_layers, int64_t n);

/*
 * fpo_cosine_grouped -- fpo_cosine (Sec. 2.2, Eq. (cosine)) for n_layers pairs
 * of equal size in one launch pair, e.g. every target layer's pseudogradient
 * against its true gradient in the layer-viability diagnostic:
 *   out[4 l + {0,1,2,3}] = <X_l, Y_l>, ||X_l||^2, ||Y_l||^2, cos_l (0 if a norm is 0)
 * X, Y: host arrays of n_layers device pointers to n elements of dtype, 16-byte
 * aligned; out: device, 4 x n_layers fp64, 8-byte aligned; 1 <= n_layers <=
 * FPO_MAX_GROUPED_LAYERS.  Sums run in fp32 over runs of at most 128 elements and
 * in fp64 after that, in a fixed order (repeat calls give identical bits; the
 * order differs from fpo_cosine's, so the two agree to rounding, not bitwise).
 */
int32_t fpo_cosine_grouped(int32_t n_layers, int64_t n, int32_t dtype, const void* const* X,
                           const void* const* Y, double* out, void* workspace,
                           size_t workspace_bytes, void* stream);

/* Bytes of workspace fpo_layer_grad_cosine_grouped needs (0 on invalid sizes). */
size_t fpo_layer_grad_cosine_workspace(int32_t n_layers, int64_t d, int64_t d_ff);

/*
 * fpo_layer_grad_cosine_grouped -- the layer-viability diagnostic in one grouped GEMM
 * (Sec. 2.2, Eq. (cosine) over the pseudogradients of Eq. (w3update)): for every layer l
 *   G_out[l] = g^T A_l                                   [d, d_ff] (dtype), as
 *                                                        fpo_layer_update_grouped writes it
 *   out[4 l + {0,1,2,3}] = <G_l, Y_l>, ||G_l||^2, ||Y_l||^2, cos_l   of the stored G_l
 *                                                        (cos = 0 if a norm is 0)
 * with Y_l [d, d_ff] (dtype) the gradient G_l is compared with.  bf16: the GEMM's
 * epilogue adds up the three sums as it writes G_l (per tile and warp, in fp32 over a
 * warp's 32 x 256 block, then in fp64 in a fixed order), so G_l is not read back; fp32:
 * the update writes G_l and fpo_cosine_grouped reduces it.
 * g [T, d], A_l [T, d_ff] (dtype); 1 <= n_layers <= FPO_MAX_GROUPED_LAYERS; pointers
 * 16-byte aligned, out (device, 4 x n_layers fp64) 8-byte aligned; bf16 needs d and d_ff
 * multiples of 8.  T = 0 gives G = 0 and cos 0.  workspace:
 * fpo_layer_grad_cosine_workspace(n_layers, d, d_ff) bytes, 256-byte aligned (the device
 * status word, then the partial sums).  Results are deterministic; they agree with
 * fpo_layer_update_grouped + fpo_cosine_grouped bitwise on G and to rounding on the sums.
 */
int32_t fpo_layer_grad_cosine_grouped(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                      int32_t dtype, const void* g, const void* const* A,
                                      const void* const* Y, void* const* G_out, double* out,
                                      void* workspace, size_t workspace_bytes, void* stream);

/* Bytes of workspace fpo_norm_ratio needs (0 for an invalid n_layers or n). */
size_t fpo_norm_ratio_workspace(int32_t n_layers, int64_t n);

/*
 * fpo_norm_ratio -- the update-magnitude ratio of App. C ("Update-magnitude
 * ratios": the fractional weight change per unit learning rate,
 * ||g~ (x) h|| / ||W_3||) and the learning rate it implies (Sec. C.2), for
 * n_layers target layers in one call:
 *   out[4 l + 0] = ||G_l||_F^2        out[4 l + 1] = ||W_l||_F^2
 *   out[4 l + 2] = r_l = ||G_l||_F / ||W_l||_F
 *   out[4 l + 3] = rel_step / r_l     (the plain-SGD rate whose step -lr G_l has
 *                                      norm rel_step ||W_l||_F; 0.01 = the
 *                                      paper's "1% step")
 * IEEE division (x / 0 = inf, 0 / 0 = NaN), so r_l = NaN for n = 0.
 *
 * G, W     host arrays of n_layers device pointers, each to n elements: G_l in
 *          g_dtype (a pseudogradient, e.g. G_out of fpo_layer_update_grouped),
 *          W_l in w_dtype (the fp32 master, or the bf16 weight); 16-byte aligned
 * out      device, 4 x n_layers fp64, 8-byte aligned
 * 1 <= n_layers <= FPO_MAX_GROUPED_LAYERS.  Squares are summed in fp32 over
 * runs of at most 128 elements and in fp64 after that, in a fixed order (repeat
 * calls give identical bits).  workspace: fpo_norm_ratio_workspace(n_layers, n) bytes.
 */
int32_t fpo_norm_ratio(int32_t n_layers, int64_t n, int32_t g_dtype, const void* const* G,
                       int32_t w_dtype, const void* const* W, double rel_step, double* out,
                       void* workspace, size_t workspace_bytes, void* stream);

/*
 * Host-to-device copy of n buffers by SM loads, for steps whose inputs (h, the
 * targets, the cached activations A_l) arrive in host memory.  The paper has no
 * counterpart.  One kernel launch copies every buffer; its threads read the host
 * memory through its device mapping, so the copy does not use the copy engines
 * and runs beside kernels on other streams (one 256-thread block per SM, no
 * shared memory).
 *
 * src[i]    host, 16-byte aligned, inside page-locked memory that is mapped into
 *           the device address space (cudaHostAlloc / cudaMallocHost memory, or
 *           memory registered with cudaHostRegister and cudaHostRegisterMapped)
 * dst[i]    device, 16-byte aligned, bytes[i] bytes; no overlap with any other
 *           dst or src of the call
 * bytes[i]  any size (a tail under 16 bytes is copied bytewise); 0 skips the pair
 * 0 <= n <= FPO_MAX_COPY_BUFFERS; n == 0 enqueues nothing.  Host memory must stay
 * valid and unchanged until the copy has completed on `stream`.
 * Errors: FPO_ERR_SHAPE (n out of range), FPO_ERR_NULL, FPO_ERR_ALIGN, FPO_ERR_ARG
 * (the first or last byte of src[i] is not in page-locked, device-mapped host memory
 * -- pageable memory is rejected even where a kernel could read it -- or the two do
 * not map to one contiguous device range).
 */
int32_t fpo_h2d_copy(int32_t n, void* const* dst, const void* const* src, const size_t* bytes,
                     void* stream);

/*
 * Synchronise `stream`, read the device status word of `workspace` (set by the
 * last call that used it), clear it, and return FPO_OK, FPO_ERR_TARGET_RANGE
 * or FPO_ERR_TIMEOUT (the first of the two when both are set).
 */
int32_t fpo_get_device_status(void* workspace, void* stream);

/* Upper bound, in nanoseconds, on every wait inside a kernel (default 2 s). */
void fpo_set_wait_limit_ns(uint64_t ns);

/* Static, human-readable name of a status code. */
const char* fpo_status_string(int32_t status);

/* FPO_ABI_VERSION of the loaded library. */
int32_t fpo_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* FPO_H_ */
