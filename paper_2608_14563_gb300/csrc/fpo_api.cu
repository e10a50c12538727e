// fpo_api.cu -- the C ABI declared in include/fpo.h: argument checks,
// workspace layout and the launch sequence of each entry point.  All device
// work is enqueued on the caller's stream; nothing here allocates device
// memory or synchronises (except fpo_get_device_status).
#include <cuda_runtime.h>

#include <atomic>
#include <climits>
#include <cmath>
#include <mutex>

#include "../../include/fpo.h"
#include "../../include/fpo_testing.h"
#include "internal.h"

namespace fpo {

namespace {
std::atomic<uint64_t> g_wait_limit_ns{2000000000ull};
std::atomic<uint64_t> g_launches{0};

struct DevCache {
    std::once_flag once;
    DevInfo info;
    bool ok = false;
};
DevCache g_dev[kMaxDevices];
}  // namespace

uint64_t wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

uint64_t launches() { return g_launches.load(std::memory_order_relaxed); }

int current_device() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
    return dev;
}

bool current_device_info(DevInfo* out) {
    const int dev = current_device();
    if (dev < 0) return false;
    DevCache& c = g_dev[dev];
    std::call_once(c.once, [&] {
        int sms = 0, maj = 0, min = 0;
        c.ok = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
               cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev) == cudaSuccess &&
               cudaDeviceGetAttribute(&min, cudaDevAttrComputeCapabilityMinor, dev) == cudaSuccess;
        c.info = DevInfo{sms, maj, min};
    });
    if (c.ok) *out = c.info;
    return c.ok;
}

}  // namespace fpo

using namespace fpo;

namespace {

constexpr size_t kAlign = 256;
constexpr size_t kStatusBytes = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int32_t check_arch() {
    DevInfo di;
    if (!current_device_info(&di)) return FPO_ERR_CUDA;
    if (di.major != 10 || di.minor != 3) return FPO_ERR_ARCH;
    return FPO_OK;
}

int32_t cuda_status(cudaError_t e) { return e == cudaSuccess ? FPO_OK : FPO_ERR_CUDA; }

#define FPO_TRY(expr)                                \
    do {                                             \
        cudaError_t e_ = (expr);                     \
        if (e_ != cudaSuccess) return FPO_ERR_CUDA;  \
    } while (0)

// ------------------------------------------------------------------ error signal
struct EsLayout {
    size_t yhat, rho, lse, zy, ce, part, g, E, z, anchor, su, sx, q, alpha, beta, cv, fix, yfix,
        fix_count, sk, total;
    int n_tiles;
    int64_t Tc;
    int algo;  // the algorithm that runs: FPO_ES_RECOMPUTE, _STORED_LOGITS or _DIRECT
};

// The algorithm a descriptor selects: AUTO is the direct algorithm for bf16; the
// fp32 path has no direct form and runs the stored-logits algorithm for it.
int es_algo(const fpo_error_signal_desc* d) {
    if (d->algo == FPO_ES_RECOMPUTE) return FPO_ES_RECOMPUTE;
    if (d->dtype == FPO_BF16 && (d->algo == FPO_ES_AUTO || d->algo == FPO_ES_DIRECT))
        return FPO_ES_DIRECT;
    return FPO_ES_STORED_LOGITS;
}

int32_t es_check_desc(const fpo_error_signal_desc* d) {
    if (!d) return FPO_ERR_NULL;
    if (d->dtype != FPO_F32 && d->dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (d->T < 0 || d->d <= 0 || d->V <= 0 || d->t_chunk < 0) return FPO_ERR_SHAPE;
    if (d->T > INT_MAX || d->d > INT_MAX || d->V > INT_MAX) return FPO_ERR_SHAPE;
    if (d->dtype == FPO_BF16 && (d->d % 8 != 0 || d->V % 8 != 0)) return FPO_ERR_SHAPE;
    if (!(d->eps >= 0.f) || !(d->min_rms >= 0.f)) return FPO_ERR_ARG;
    if (d->stage_events_per_chunk != 0 && d->stage_events_per_chunk != 1) return FPO_ERR_ARG;
    if (d->algo != FPO_ES_AUTO && d->algo != FPO_ES_RECOMPUTE && d->algo != FPO_ES_STORED_LOGITS &&
        d->algo != FPO_ES_DIRECT)
        return FPO_ERR_ARG;
    return FPO_OK;
}

EsLayout es_layout(const fpo_error_signal_desc* d) {
    EsLayout L{};
    const size_t esz = d->dtype == FPO_BF16 ? 2 : 4;
    const size_t T = static_cast<size_t>(d->T), D = static_cast<size_t>(d->d),
                 V = static_cast<size_t>(d->V);
    const int tile_n = d->dtype == FPO_BF16 ? lse_tile_n_bf16() : kSimtTile;
    L.n_tiles = static_cast<int>((d->V + tile_n - 1) / tile_n);
    // Chunks of 8192 tokens by default: the logits pass and the projection alternating
    // per chunk ran 0.6-2.5% faster per step than over all tokens at once on GB300 (the
    // power-capped clock settles higher), and the chunk buffers shrink accordingly.
    const int64_t chunk = d->t_chunk > 0 ? d->t_chunk : FPO_AUTO_T_CHUNK;
    L.Tc = d->T == 0 ? 0 : (chunk < d->T ? chunk : d->T);
    size_t off = kStatusBytes;
    L.yhat = off; off = align_up(off + T * D * esz);
    L.rho = off;  off = align_up(off + T * 4);
    L.lse = off;  off = align_up(off + T * 4);
    L.zy = off;   off = align_up(off + T * 4);
    L.ce = off;   off = align_up(off + T * 4);
    L.part = off; off = align_up(off + T * static_cast<size_t>(L.n_tiles) * 8);
    L.algo = es_algo(d);
    const bool stored = L.algo == FPO_ES_STORED_LOGITS, direct = L.algo == FPO_ES_DIRECT;
    // g in fp32 for the separate VJP (the direct algorithm writes g~ from the projection)
    L.g = off;    off = align_up(off + (direct ? 0 : T * D * 4));
    L.E = off;    off = align_up(off + static_cast<size_t>(L.Tc) * V * esz);
    L.z = off;    off = align_up(off + (stored ? static_cast<size_t>(L.Tc) * V * 4 : 0));
    const size_t Tdir = direct ? T : 0, Tcdir = direct ? static_cast<size_t>(L.Tc) : 0;
    L.anchor = off;    off = align_up(off + Tdir * 4);
    L.su = off;        off = align_up(off + Tdir * static_cast<size_t>(L.n_tiles) * 4);
    L.sx = off;        off = align_up(off + Tdir * static_cast<size_t>(L.n_tiles) * 4);
    L.q = off;         off = align_up(off + Tdir * static_cast<size_t>(L.n_tiles) * 4);
    L.alpha = off;     off = align_up(off + Tdir * 4);
    L.beta = off;      off = align_up(off + Tdir * 4);
    L.cv = off;        off = align_up(off + Tdir * 4);
    L.fix = off;       off = align_up(off + Tcdir * 4);
    L.yfix = off;      off = align_up(off + Tcdir * D * esz);
    L.fix_count = off; off = align_up(off + (direct ? 4 : 0));
    // the projection's split-K tail (the fp32 partial sums of the last wave's split tiles)
    L.sk = off;        off = align_up(off + (d->dtype == FPO_BF16 ? proj_sk_scratch_bytes() : 0));
    L.total = off;
    return L;
}

}  // namespace

extern "C" {

int32_t fpo_abi_version(void) { return FPO_ABI_VERSION; }

void fpo_set_wait_limit_ns(uint64_t ns) {
    g_wait_limit_ns.store(ns > 0 ? ns : 1, std::memory_order_relaxed);
}

const char* fpo_status_string(int32_t s) {
    switch (s) {
        case FPO_OK: return "FPO_OK";
        case FPO_ERR_NULL: return "FPO_ERR_NULL: a required pointer is NULL";
        case FPO_ERR_SHAPE: return "FPO_ERR_SHAPE: unsupported or invalid size";
        case FPO_ERR_DTYPE: return "FPO_ERR_DTYPE: unknown dtype";
        case FPO_ERR_ALIGN: return "FPO_ERR_ALIGN: tensor pointer not 16-byte aligned";
        case FPO_ERR_WORKSPACE: return "FPO_ERR_WORKSPACE: workspace missing or too small";
        case FPO_ERR_ARCH: return "FPO_ERR_ARCH: device is not compute capability 10.3";
        case FPO_ERR_CUDA: return "FPO_ERR_CUDA: CUDA call failed";
        case FPO_ERR_TARGET_RANGE: return "FPO_ERR_TARGET_RANGE: a target id is outside [0, V)";
        case FPO_ERR_TIMEOUT: return "FPO_ERR_TIMEOUT: a bounded wait inside a kernel ran out";
        case FPO_ERR_ARG: return "FPO_ERR_ARG: invalid argument";
        default: return "unknown fpo status";
    }
}

size_t fpo_error_signal_workspace(const fpo_error_signal_desc* desc) {
    if (es_check_desc(desc) != FPO_OK) return 0;
    return es_layout(desc).total;
}

int32_t fpo_error_signal_stage_events(const fpo_error_signal_desc* desc) {
    if (es_check_desc(desc) != FPO_OK) return 0;
    if (!desc->stage_events_per_chunk) return FPO_STAGE_EVENTS;
    const EsLayout L = es_layout(desc);
    const int64_t n = L.Tc > 0 ? (desc->T + L.Tc - 1) / L.Tc : 0;
    return static_cast<int32_t>(3 + 4 * n);
}

int32_t fpo_error_signal(const fpo_error_signal_desc* desc, const void* h, const void* norm_w,
                         const void* W_U, const int32_t* targets, void* g_out, float* lse_out,
                         float* loss_out, void* workspace, size_t workspace_bytes, void* stream) {
    int32_t rc = es_check_desc(desc);
    if (rc != FPO_OK) return rc;
    if (!workspace) return FPO_ERR_WORKSPACE;
    if (desc->T > 0 && (!h || !norm_w || !W_U || !targets || !g_out)) return FPO_ERR_NULL;
    if (!aligned16(h) || !aligned16(norm_w) || !aligned16(W_U) || !aligned16(g_out) ||
        (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0 ||
        (reinterpret_cast<uintptr_t>(targets) & 3u) || (reinterpret_cast<uintptr_t>(lse_out) & 3u) ||
        (reinterpret_cast<uintptr_t>(loss_out) & 3u))
        return FPO_ERR_ALIGN;
    const EsLayout L = es_layout(desc);
    if (workspace_bytes < L.total) return FPO_ERR_WORKSPACE;
    if ((rc = check_arch()) != FPO_OK) return rc;

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    unsigned* status = reinterpret_cast<unsigned*>(ws);
    FPO_TRY(cudaMemsetAsync(status, 0, sizeof(unsigned), st));
    const int T = static_cast<int>(desc->T), d = static_cast<int>(desc->d),
              V = static_cast<int>(desc->V);
    if (T == 0) {
        if (loss_out) FPO_TRY(cudaMemsetAsync(loss_out, 0, sizeof(float), st));
        return FPO_OK;
    }
    const bool bf16 = desc->dtype == FPO_BF16;
    const size_t esz = bf16 ? 2 : 4;
    void* yhat = ws + L.yhat;
    float* rho = reinterpret_cast<float*>(ws + L.rho);
    float* lse = lse_out ? lse_out : reinterpret_cast<float*>(ws + L.lse);
    float* zy = loss_out ? reinterpret_cast<float*>(ws + L.zy) : nullptr;
    float* ce = loss_out ? reinterpret_cast<float*>(ws + L.ce) : nullptr;
    float2* part = reinterpret_cast<float2*>(ws + L.part);
    float* g = reinterpret_cast<float*>(ws + L.g);
    void* E = ws + L.E;
    float* sk = reinterpret_cast<float*>(ws + L.sk);

    // Stage events (profiling): ev(i) records event i; cmark(c, k) the boundary k (2 logits,
    // 3 combine, 4 E / fixup, 5 projection) of token chunk c, every chunk's in the
    // per-chunk layout, else only the last chunk's.
    const bool per_chunk = desc->stage_events && desc->stage_events_per_chunk;
    const int64_t n_chunks = L.Tc > 0 ? (T + L.Tc - 1) / L.Tc : 0;
    auto ev = [&](int64_t i) -> cudaError_t {
        if (!desc->stage_events || !desc->stage_events[i]) return cudaSuccess;
        return cudaEventRecord(static_cast<cudaEvent_t>(desc->stage_events[i]), st);
    };
    auto cmark = [&](int64_t c, int k) -> cudaError_t {
        if (per_chunk) return ev(k + 4 * c);
        return c == n_chunks - 1 ? ev(k) : cudaSuccess;
    };
    auto mark = [&](int i) -> cudaError_t { return ev(i); };
    const bool direct = L.algo == FPO_ES_DIRECT;
    float* anchor = reinterpret_cast<float*>(ws + L.anchor);
    FPO_TRY(mark(0));
    // 1. final RMSNorm forward: rho, yhat (and the target-range check; the anchor
    //    c_t = <yhat_t, W_U[y_t]> for the direct algorithm)
    FPO_TRY(launch_rmsnorm_fwd(desc->dtype, h, norm_w, T, d, desc->eps, yhat, rho, targets, V,
                               status, st, direct ? W_U : nullptr, direct ? anchor : nullptr));
    FPO_TRY(mark(1));
    if (direct) {
        // 2.-5. per token chunk: logits pass anchored at the target logit, writing
        //       P = exp(z - c) and the per-tile sums -> lse, loss and row factors -> the
        //       rows outside the anchor window: their lse by a max-based pass, then P
        //       anchored at lse -> g = alpha P W_U + beta W_U[y] with the final-norm VJP
        //       in the projection's epilogue -> g~
        float* su = reinterpret_cast<float*>(ws + L.su);
        float* sx = reinterpret_cast<float*>(ws + L.sx);
        float* qz = reinterpret_cast<float*>(ws + L.q);
        float* alpha = reinterpret_cast<float*>(ws + L.alpha);
        float* beta = reinterpret_cast<float*>(ws + L.beta);
        float* cv = reinterpret_cast<float*>(ws + L.cv);
        int* fix = reinterpret_cast<int*>(ws + L.fix);
        int* fix_count = reinterpret_cast<int*>(ws + L.fix_count);
        void* yfix = ws + L.yfix;
        for (int64_t c0 = 0, ci = 0; c0 < T; c0 += L.Tc, ++ci) {
            const int tc = static_cast<int>(L.Tc < T - c0 ? L.Tc : T - c0);
            const bool last = c0 + tc >= T;
            const void* yh = static_cast<const uint8_t*>(yhat) + static_cast<size_t>(c0) * d * esz;
            float2* pc = part + static_cast<size_t>(c0) * L.n_tiles;
            float* suc = su + static_cast<size_t>(c0) * L.n_tiles;
            float* sxc = sx + static_cast<size_t>(c0) * L.n_tiles;
            float* qc = qz + static_cast<size_t>(c0) * L.n_tiles;
            float* cec = ce ? ce + c0 : nullptr;
            FPO_TRY(cudaMemsetAsync(fix_count, 0, sizeof(int), st));
            FPO_TRY(launch_anchor_prob_bf16(yh, W_U, targets + c0, anchor + c0, tc, d, V, suc, sxc,
                                            qc, L.n_tiles, E, status, st));
            FPO_TRY(cmark(ci, 2));
            FPO_TRY(launch_direct_combine(suc, sxc, qc, L.n_tiles, tc, V, targets + c0, anchor + c0,
                                          desc->loss_scale, lse + c0, cec, alpha + c0, beta + c0,
                                          cv + c0, fix, fix_count, st));
            FPO_TRY(cmark(ci, 3));
            FPO_TRY(launch_gather_rows(yh, fix, fix_count, d, yfix, st));
            FPO_TRY(launch_fixup_lse_bf16(yfix, W_U, fix, fix_count, tc, d, V, pc, L.n_tiles,
                                          status, st));
            FPO_TRY(launch_direct_fixup_lse(pc, fix, fix_count, L.n_tiles, anchor + c0, lse + c0,
                                            cec, st));
            FPO_TRY(launch_fixup_logits_bf16(yfix, W_U, fix, fix_count, targets + c0, lse + c0, tc,
                                             d, V, E, sxc, qc, L.n_tiles, status, st));
            FPO_TRY(launch_direct_fixup_factors(sxc, qc, fix, fix_count, L.n_tiles, anchor + c0,
                                                desc->loss_scale, alpha + c0, beta + c0, cv + c0,
                                                st));
            if (last && loss_out) FPO_TRY(launch_mean(ce, T, loss_out, st));
            FPO_TRY(cmark(ci, 4));
            FPO_TRY(launch_proj_vjp_bf16(
                E, W_U, targets + c0, alpha + c0, beta + c0, cv + c0, rho + c0,
                static_cast<const uint8_t*>(h) + static_cast<size_t>(c0) * d * esz, norm_w,
                desc->min_rms, tc, d, V,
                static_cast<uint8_t*>(g_out) + static_cast<size_t>(c0) * d * esz, sk, status, st));
            FPO_TRY(cmark(ci, 5));
        }
    } else if (L.algo == FPO_ES_RECOMPUTE) {
        // 2. logits pass over all tokens: per-vocabulary-tile (max, sum exp) partials -> lse
        if (bf16)
            FPO_TRY(launch_lse_partial_bf16(yhat, W_U, targets, T, d, V, part, L.n_tiles, zy,
                                            nullptr, status, st));
        else
            FPO_TRY(launch_lse_partial_f32(static_cast<const float*>(yhat),
                                           static_cast<const float*>(W_U), targets, T, d, V, part,
                                           L.n_tiles, zy, nullptr, st));
        FPO_TRY(per_chunk ? ev(2) : mark(2));
        FPO_TRY(launch_lse_combine(part, L.n_tiles, T, zy, lse, ce, st));
        if (loss_out) FPO_TRY(launch_mean(ce, T, loss_out, st));
        FPO_TRY(per_chunk ? ev(3) : mark(3));
        // 3./4. per token chunk: recompute the logits -> E, then g = E W_U
        for (int64_t c0 = 0, ci = 0; c0 < T; c0 += L.Tc, ++ci) {
            const int tc = static_cast<int>(L.Tc < T - c0 ? L.Tc : T - c0);
            const void* yh = static_cast<const uint8_t*>(yhat) + static_cast<size_t>(c0) * d * esz;
            if (per_chunk && ci > 0) {  // no logits pass or combine of its own
                FPO_TRY(ev(2 + 4 * ci));
                FPO_TRY(ev(3 + 4 * ci));
            }
            if (bf16) {
                FPO_TRY(launch_error_bf16(yh, W_U, targets + c0, lse + c0, tc, d, V,
                                          desc->loss_scale, E, status, st));
                FPO_TRY(cmark(ci, 4));
                FPO_TRY(launch_proj_bf16(E, W_U, tc, d, V, g + c0 * d, sk, status, st));
            } else {
                FPO_TRY(launch_error_f32(static_cast<const float*>(yh),
                                         static_cast<const float*>(W_U), targets + c0, lse + c0,
                                         tc, d, V, desc->loss_scale, static_cast<float*>(E), st));
                FPO_TRY(cmark(ci, 4));
                FPO_TRY(launch_proj_f32(static_cast<const float*>(E), static_cast<const float*>(W_U),
                                        tc, d, V, g + c0 * d, st));
            }
            FPO_TRY(cmark(ci, 5));
        }
    } else {
        // 2.-4. per token chunk: logits pass storing z -> lse -> E from z -> g = E W_U
        float* z = reinterpret_cast<float*>(ws + L.z);
        for (int64_t c0 = 0, ci = 0; c0 < T; c0 += L.Tc, ++ci) {
            const int tc = static_cast<int>(L.Tc < T - c0 ? L.Tc : T - c0);
            const bool last = c0 + tc >= T;
            const void* yh = static_cast<const uint8_t*>(yhat) + static_cast<size_t>(c0) * d * esz;
            float2* pc = part + static_cast<size_t>(c0) * L.n_tiles;
            float* zyc = zy ? zy + c0 : nullptr;
            float* cec = ce ? ce + c0 : nullptr;
            if (bf16)
                FPO_TRY(launch_lse_partial_bf16(yh, W_U, targets + c0, tc, d, V, pc, L.n_tiles, zyc,
                                                z, status, st));
            else
                FPO_TRY(launch_lse_partial_f32(static_cast<const float*>(yh),
                                               static_cast<const float*>(W_U), targets + c0, tc, d,
                                               V, pc, L.n_tiles, zyc, z, st));
            FPO_TRY(cmark(ci, 2));
            FPO_TRY(launch_lse_combine(pc, L.n_tiles, tc, zyc, lse + c0, cec, st));
            if (last && loss_out) FPO_TRY(launch_mean(ce, T, loss_out, st));
            FPO_TRY(cmark(ci, 3));
            FPO_TRY(launch_error_from_logits(desc->dtype, z, lse + c0, targets + c0, tc, V,
                                             desc->loss_scale, E, st));
            FPO_TRY(cmark(ci, 4));
            if (bf16)
                FPO_TRY(launch_proj_bf16(E, W_U, tc, d, V, g + c0 * d, sk, status, st));
            else
                FPO_TRY(launch_proj_f32(static_cast<const float*>(E), static_cast<const float*>(W_U),
                                        tc, d, V, g + c0 * d, st));
            FPO_TRY(cmark(ci, 5));
        }
    }
    // 5. final-norm VJP with the min-RMS clamp -> g~ (already in the direct algorithm's
    //    projection epilogue; the stage is then empty)
    if (!direct)
        FPO_TRY(launch_rmsnorm_vjp(desc->dtype, g, h, norm_w, rho, T, d, desc->min_rms, g_out,
                                   st));
    FPO_TRY(per_chunk ? ev(2 + 4 * n_chunks) : mark(6));
    return FPO_OK;
}

size_t fpo_layer_update_workspace(void) { return kStatusBytes; }

int32_t fpo_layer_update_grouped_signals(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                         int32_t dtype, const void* const* g,
                                         const void* const* A, float lr, float* const* W_master,
                                         void* const* W_out, void* const* G_out, void* workspace,
                                         size_t workspace_bytes, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS) return FPO_ERR_SHAPE;
    if (T < 0 || d <= 0 || d_ff <= 0 || T > INT_MAX || d > INT_MAX || d_ff > INT_MAX)
        return FPO_ERR_SHAPE;
    if (dtype == FPO_BF16 && (d % 8 != 0 || d_ff % 8 != 0)) return FPO_ERR_SHAPE;
    if (!(lr == lr)) return FPO_ERR_ARG;
    if (!workspace || workspace_bytes < kStatusBytes) return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    if (!A || !g) return FPO_ERR_NULL;
    for (int l = 0; l < n_layers; ++l) {
        float* wm = W_master ? W_master[l] : nullptr;
        void* wo = W_out ? W_out[l] : nullptr;
        void* go = G_out ? G_out[l] : nullptr;
        if (T > 0 && (!A[l] || !g[l])) return FPO_ERR_NULL;
        if (!wm && !go) return FPO_ERR_NULL;
        if (wo && !wm) return FPO_ERR_NULL;
        if (!aligned16(g[l]) || !aligned16(A[l]) || !aligned16(wm) || !aligned16(wo) ||
            !aligned16(go))
            return FPO_ERR_ALIGN;
    }
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned* status = static_cast<unsigned*>(workspace);
    FPO_TRY(cudaMemsetAsync(status, 0, sizeof(unsigned), st));
    const int Ti = static_cast<int>(T), di = static_cast<int>(d), fi = static_cast<int>(d_ff);
    if (T == 0) {
        // G = 0: the master is unchanged, W_out is its cast, G_out is zero.
        const size_t n = static_cast<size_t>(d) * static_cast<size_t>(d_ff);
        for (int l = 0; l < n_layers; ++l) {
            void* go = G_out ? G_out[l] : nullptr;
            void* wo = W_out ? W_out[l] : nullptr;
            if (go) FPO_TRY(cudaMemsetAsync(go, 0, n * (dtype == FPO_BF16 ? 2 : 4), st));
            if (wo) FPO_TRY(launch_cast_f32(dtype, W_master[l], n, wo, st));
        }
        return FPO_OK;
    }
    if (dtype == FPO_BF16)
        return cuda_status(launch_update_bf16(n_layers, Ti, di, fi, g, A, lr, W_master, W_out,
                                              G_out, status, st));
    return cuda_status(launch_update_f32(
        n_layers, Ti, di, fi, reinterpret_cast<const float* const*>(g),
        reinterpret_cast<const float* const*>(A), lr, W_master,
        reinterpret_cast<float* const*>(W_out), reinterpret_cast<float* const*>(G_out), st));
}

int32_t fpo_layer_update_grouped(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                 int32_t dtype, const void* g, const void* const* A, float lr,
                                 float* const* W_master, void* const* W_out, void* const* G_out,
                                 void* workspace, size_t workspace_bytes, void* stream) {
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS) return FPO_ERR_SHAPE;
    if (T > 0 && !g) return FPO_ERR_NULL;
    const void* gs[FPO_MAX_GROUPED_LAYERS];
    for (int l = 0; l < n_layers; ++l) gs[l] = g;
    return fpo_layer_update_grouped_signals(n_layers, T, d, d_ff, dtype, gs, A, lr, W_master,
                                            W_out, G_out, workspace, workspace_bytes, stream);
}

size_t fpo_layer_grad_cosine_workspace(int32_t n_layers, int64_t d, int64_t d_ff) {
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS || d <= 0 || d_ff <= 0 ||
        d > INT_MAX || d_ff > INT_MAX)
        return 0;
    // bf16: the per-(tile, warp) triples of the fused epilogue; fp32: the partials of the
    // separate grouped cosine (the larger of the two, so one size serves both)
    const size_t fused = grad_cosine_partial_bytes(n_layers, static_cast<int>(d),
                                                   static_cast<int>(d_ff));
    const size_t sep = fpo_cosine_grouped_workspace(n_layers, d * d_ff);
    return kStatusBytes + align_up(fused > sep ? fused : sep);
}

int32_t fpo_layer_grad_cosine_grouped(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                      int32_t dtype, const void* g, const void* const* A,
                                      const void* const* Y, void* const* G_out, double* out,
                                      void* workspace, size_t workspace_bytes, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS) return FPO_ERR_SHAPE;
    if (T < 0 || d <= 0 || d_ff <= 0 || T > INT_MAX || d > INT_MAX || d_ff > INT_MAX)
        return FPO_ERR_SHAPE;
    if (dtype == FPO_BF16 && (d % 8 != 0 || d_ff % 8 != 0)) return FPO_ERR_SHAPE;
    if (!A || !Y || !G_out || !out || (T > 0 && !g)) return FPO_ERR_NULL;
    if (!aligned16(g) || (reinterpret_cast<uintptr_t>(out) & 7u)) return FPO_ERR_ALIGN;
    for (int l = 0; l < n_layers; ++l) {
        if ((T > 0 && !A[l]) || !Y[l] || !G_out[l]) return FPO_ERR_NULL;
        if (!aligned16(A[l]) || !aligned16(Y[l]) || !aligned16(G_out[l])) return FPO_ERR_ALIGN;
    }
    if (!workspace || workspace_bytes < fpo_layer_grad_cosine_workspace(n_layers, d, d_ff))
        return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    unsigned* status = reinterpret_cast<unsigned*>(ws);
    FPO_TRY(cudaMemsetAsync(status, 0, sizeof(unsigned), st));
    const int Ti = static_cast<int>(T), di = static_cast<int>(d), fi = static_cast<int>(d_ff);
    const size_t n = static_cast<size_t>(d) * static_cast<size_t>(d_ff);
    if (T == 0) {
        // G = 0: the cosine of every layer is 0, ||Y||^2 by the grouped reduction
        for (int l = 0; l < n_layers; ++l)
            FPO_TRY(cudaMemsetAsync(G_out[l], 0, n * (dtype == FPO_BF16 ? 2 : 4), st));
        return cuda_status(launch_cosine_grouped(
            dtype, n_layers, static_cast<int64_t>(n), const_cast<const void* const*>(G_out), Y,
            reinterpret_cast<double*>(ws + kStatusBytes), norm_ratio_blocks(n_layers, n), out,
            st));
    }
    const void* gs[FPO_MAX_GROUPED_LAYERS];
    for (int l = 0; l < n_layers; ++l) gs[l] = g;
    if (dtype == FPO_BF16)
        return cuda_status(launch_grad_cosine_bf16(n_layers, Ti, di, fi, gs, A, Y, G_out,
                                                   reinterpret_cast<float*>(ws + kStatusBytes),
                                                   out, status, st));
    // fp32: the SIMT update writes G, then the grouped cosine reads it back
    FPO_TRY(launch_update_f32(n_layers, Ti, di, fi, reinterpret_cast<const float* const*>(gs),
                              reinterpret_cast<const float* const*>(A), 0.f, nullptr, nullptr,
                              reinterpret_cast<float* const*>(G_out), st));
    return cuda_status(launch_cosine_grouped(
        dtype, n_layers, static_cast<int64_t>(n), const_cast<const void* const*>(G_out), Y,
        reinterpret_cast<double*>(ws + kStatusBytes), norm_ratio_blocks(n_layers, n), out, st));
}

// Bytes of the optimizer's norm partials: those of the stand-alone passes or of the
// fused epilogue's (layer, 256 rows, column tile, 32 rows) slots, whichever is larger.
static size_t optimize_partials_area(int32_t n_layers, int64_t d, int64_t d_ff) {
    const size_t a = optim_partials_bytes(n_layers);
    const size_t b = opt_step_partial_bytes(n_layers, static_cast<int>(d), static_cast<int>(d_ff));
    return align_up(a > b ? a : b);
}

size_t fpo_layer_optimize_workspace(int32_t n_layers, int64_t d, int64_t d_ff) {
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS || d <= 0 || d_ff <= 0) return 0;
    if (d > INT_MAX || d_ff > INT_MAX) return 0;
    return kStatusBytes + align_up(static_cast<size_t>(n_layers) * static_cast<size_t>(d) *
                                   static_cast<size_t>(d_ff) * 4) +
           optimize_partials_area(n_layers, d, d_ff) + align_up(static_cast<size_t>(n_layers) * 4);
}

int32_t fpo_layer_optimize_grouped(int32_t n_layers, int64_t T, int64_t d, int64_t d_ff,
                                   int32_t dtype, const void* const* g, const void* const* A,
                                   const fpo_optimizer_desc* opt, float* const* W_master,
                                   void* const* W_out, float* const* state1,
                                   float* const* state2, void* workspace, size_t workspace_bytes,
                                   void* stream) {
    if (!opt) return FPO_ERR_NULL;
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS) return FPO_ERR_SHAPE;
    if (T < 0 || d <= 0 || d_ff <= 0 || T > INT_MAX || d > INT_MAX || d_ff > INT_MAX)
        return FPO_ERR_SHAPE;
    if (dtype == FPO_BF16 && (d % 8 != 0 || d_ff % 8 != 0)) return FPO_ERR_SHAPE;
    if (opt->kind < FPO_OPT_SGD || opt->kind > FPO_OPT_ADAMW || opt->clip < FPO_CLIP_NONE ||
        opt->clip > FPO_CLIP_GRADIENT || !(opt->lr == opt->lr) || !(opt->clip_frac >= 0.f) ||
        (opt->kind == FPO_OPT_ADAMW && (opt->step < 1 || !(opt->beta1 >= 0.f && opt->beta1 < 1.f) ||
                                       !(opt->beta2 >= 0.f && opt->beta2 < 1.f))))
        return FPO_ERR_ARG;
    if (!A || !g || !W_master) return FPO_ERR_NULL;
    if ((opt->kind != FPO_OPT_SGD && !state1) || (opt->kind == FPO_OPT_ADAMW && !state2))
        return FPO_ERR_NULL;
    const size_t need = fpo_layer_optimize_workspace(n_layers, d, d_ff);
    if (!workspace || workspace_bytes < need) return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    for (int l = 0; l < n_layers; ++l) {
        if ((T > 0 && (!A[l] || !g[l])) || !W_master[l]) return FPO_ERR_NULL;
        if (opt->kind != FPO_OPT_SGD && !state1[l]) return FPO_ERR_NULL;
        if (opt->kind == FPO_OPT_ADAMW && !state2[l]) return FPO_ERR_NULL;
        if (!aligned16(g[l]) || !aligned16(A[l]) || !aligned16(W_master[l]) ||
            !aligned16(W_out ? W_out[l] : nullptr) || !aligned16(state1 ? state1[l] : nullptr) ||
            !aligned16(state2 ? state2[l] : nullptr))
            return FPO_ERR_ALIGN;
    }
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    unsigned* status = reinterpret_cast<unsigned*>(ws);
    FPO_TRY(cudaMemsetAsync(status, 0, sizeof(unsigned), st));
    const size_t n = static_cast<size_t>(d) * static_cast<size_t>(d_ff);
    float* Gbuf = reinterpret_cast<float*>(ws + kStatusBytes);
    double* partials = reinterpret_cast<double*>(ws + kStatusBytes + align_up(n_layers * n * 4));
    float* scales = reinterpret_cast<float*>(ws + kStatusBytes + align_up(n_layers * n * 4) +
                                             optimize_partials_area(n_layers, d, d_ff));
    float* G[FPO_MAX_GROUPED_LAYERS];
    for (int l = 0; l < n_layers; ++l) G[l] = Gbuf + static_cast<size_t>(l) * n;

    OptimParams op;
    op.kind = opt->kind;
    op.clip = opt->clip;
    op.lr = opt->lr;
    op.momentum = opt->momentum;
    op.beta1 = opt->beta1;
    op.beta2 = opt->beta2;
    op.eps = opt->adam_eps;
    op.weight_decay = opt->weight_decay;
    op.clip_frac = opt->clip_frac;
    const double t = static_cast<double>(opt->step < 1 ? 1 : opt->step);
    op.inv_bc1 = static_cast<float>(1.0 / (1.0 - pow(static_cast<double>(opt->beta1), t)));
    op.inv_sqrt_bc2 = static_cast<float>(1.0 / sqrt(1.0 - pow(static_cast<double>(opt->beta2), t)));
    if (opt->kind != FPO_OPT_ADAMW) op.inv_bc1 = op.inv_sqrt_bc2 = 1.f;
    float* const* s1 = opt->kind != FPO_OPT_SGD ? state1 : nullptr;
    float* const* s2 = opt->kind == FPO_OPT_ADAMW ? state2 : nullptr;

    if (dtype == FPO_BF16 && T > 0 && opt->clip == FPO_CLIP_STEP) {
        // the step clip's first pass in the GEMM's epilogue: the state advanced, the
        // unclipped steps (in the G buffer) and their norm partials; then a scale and an
        // apply pass (measured: the AdamW + step-clip step 0.6% faster than with G stored
        // and three passes; without a clip the stand-alone passes are faster overall)
        float* part = reinterpret_cast<float*>(partials);
        FPO_TRY(launch_opt_step_bf16(n_layers, static_cast<int>(T), static_cast<int>(d),
                                     static_cast<int>(d_ff), g, A, op, W_master, s1, s2, G, part,
                                     status, st));
        const int slots = static_cast<int>(opt_step_partial_bytes(1, static_cast<int>(d),
                                                                  static_cast<int>(d_ff)) /
                                           (2 * sizeof(float)));
        return cuda_status(launch_opt_step_clip(n_layers, n, op, part, slots, G, W_master, W_out,
                                                scales, st));
    }

    // 1. G_l = g_l^T A_l (fp32)
    if (T == 0) {
        FPO_TRY(cudaMemsetAsync(Gbuf, 0, n_layers * n * 4, st));
    } else if (dtype == FPO_BF16) {
        FPO_TRY(launch_grad_bf16(n_layers, static_cast<int>(T), static_cast<int>(d),
                                 static_cast<int>(d_ff), g, A, G, status, st));
    } else {
        FPO_TRY(launch_update_f32(n_layers, static_cast<int>(T), static_cast<int>(d),
                                  static_cast<int>(d_ff), reinterpret_cast<const float* const*>(g),
                                  reinterpret_cast<const float* const*>(A), 0.f, nullptr, nullptr,
                                  G, st));
    }
    // 2. clip factor and optimizer step on the fp32 masters
    return cuda_status(launch_optimizer(dtype, n_layers, n, op, G, W_master, W_out, s1, s2,
                                        partials, scales, st));
}

int32_t fpo_gate_up_signals(int64_t T, int64_t d, int64_t d_ff, int32_t dtype, const void* g,
                            const void* W3_init, const void* a, const void* b, void* dA, void* dB,
                            void* workspace, size_t workspace_bytes, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (T < 0 || d <= 0 || d_ff <= 0 || T > INT_MAX || d > INT_MAX || d_ff > INT_MAX)
        return FPO_ERR_SHAPE;
    if (dtype == FPO_BF16 && (d % 8 != 0 || d_ff % 8 != 0)) return FPO_ERR_SHAPE;
    if (T > 0 && (!g || !W3_init || !a || !b || !dA || !dB)) return FPO_ERR_NULL;
    if (!aligned16(g) || !aligned16(W3_init) || !aligned16(a) || !aligned16(b) || !aligned16(dA) ||
        !aligned16(dB))
        return FPO_ERR_ALIGN;
    if (!workspace || workspace_bytes < kStatusBytes) return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned* status = static_cast<unsigned*>(workspace);
    FPO_TRY(cudaMemsetAsync(status, 0, sizeof(unsigned), st));
    if (T == 0) return FPO_OK;
    const int Ti = static_cast<int>(T), di = static_cast<int>(d), fi = static_cast<int>(d_ff);
    if (dtype == FPO_BF16)
        return cuda_status(launch_swiglu_bf16(Ti, di, fi, g, W3_init, a, b, dA, dB, status, st));
    return cuda_status(launch_swiglu_f32(Ti, di, fi, static_cast<const float*>(g),
                                         static_cast<const float*>(W3_init),
                                         static_cast<const float*>(a), static_cast<const float*>(b),
                                         static_cast<float*>(dA), static_cast<float*>(dB), st));
}

int32_t fpo_rmsnorm_vjp(int64_t T, int64_t d, int32_t dtype, const void* g, const void* x,
                        const void* gamma, float eps, float min_rms, void* g_out, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (T < 0 || d <= 0 || T > INT_MAX || d > INT_MAX) return FPO_ERR_SHAPE;
    if (dtype == FPO_BF16 && d % 8 != 0) return FPO_ERR_SHAPE;
    if (!(eps >= 0.f) || !(min_rms >= 0.f)) return FPO_ERR_ARG;
    if (T > 0 && (!g || !x || !gamma || !g_out)) return FPO_ERR_NULL;
    if (!aligned16(g) || !aligned16(x) || !aligned16(gamma) || !aligned16(g_out))
        return FPO_ERR_ALIGN;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    if (T == 0) return FPO_OK;
    // one norm of fpo_layer_signals: its pre-MLP stage alone, for one layer
    const void* xs[1] = {x};
    const void* gs[1] = {gamma};
    void* outs[1] = {g_out};
    return cuda_status(launch_layer_signals(dtype, 1, g, nullptr, nullptr, xs, gs, outs,
                                            static_cast<int>(T), static_cast<int>(d), eps, min_rms,
                                            static_cast<cudaStream_t>(stream)));
}

int32_t fpo_layer_signals(int32_t n_layers, int64_t T, int64_t d, int32_t dtype, const void* g,
                          const void* const* m, const void* const* gamma_post,
                          const void* const* x, const void* const* gamma_pre, float eps,
                          float min_rms, void* const* g_out, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS) return FPO_ERR_SHAPE;
    if (T < 0 || d <= 0 || T > INT_MAX || d > INT_MAX) return FPO_ERR_SHAPE;
    if (dtype == FPO_BF16 && d % 8 != 0) return FPO_ERR_SHAPE;
    if (!(eps >= 0.f) || !(min_rms >= 0.f)) return FPO_ERR_ARG;
    if ((!m) != (!gamma_post) || (!x) != (!gamma_pre) || (!m && !x)) return FPO_ERR_ARG;
    if (!g_out) return FPO_ERR_NULL;
    if (T > 0) {
        if (!g || !aligned16(g)) return g ? FPO_ERR_ALIGN : FPO_ERR_NULL;
        const void* const* arrays[4] = {m, gamma_post, x, gamma_pre};
        for (int l = 0; l < n_layers; ++l) {
            for (const void* const* a : arrays) {
                if (!a) continue;
                if (!a[l]) return FPO_ERR_NULL;
                if (!aligned16(a[l])) return FPO_ERR_ALIGN;
            }
            if (!g_out[l]) return FPO_ERR_NULL;
            if (!aligned16(g_out[l])) return FPO_ERR_ALIGN;
        }
    }
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    if (T == 0) return FPO_OK;
    return cuda_status(launch_layer_signals(dtype, n_layers, g, m, gamma_post, x, gamma_pre, g_out,
                                            static_cast<int>(T), static_cast<int>(d), eps, min_rms,
                                            static_cast<cudaStream_t>(stream)));
}

int32_t fpo_layer_update(int64_t T, int64_t d, int64_t d_ff, int32_t dtype, const void* g,
                         const void* A, float lr, float* W_master, void* W_out, void* G_out,
                         void* workspace, size_t workspace_bytes, void* stream) {
    const void* As[1] = {A};
    float* Wm[1] = {W_master};
    void* Wo[1] = {W_out};
    void* Go[1] = {G_out};
    return fpo_layer_update_grouped(1, T, d, d_ff, dtype, g, As, lr, Wm, Wo, Go, workspace,
                                    workspace_bytes, stream);
}

size_t fpo_cosine_workspace(int64_t n) {
    if (n < 0) return 0;
    return kStatusBytes + align_up(static_cast<size_t>(cosine_blocks(n)) * 3 * sizeof(double));
}

int32_t fpo_cosine(int64_t n, int32_t dtype, const void* X, const void* Y, double* out,
                   void* workspace, size_t workspace_bytes, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n < 0) return FPO_ERR_SHAPE;
    if (!out || (n > 0 && (!X || !Y))) return FPO_ERR_NULL;
    if (!aligned16(X) || !aligned16(Y) || (reinterpret_cast<uintptr_t>(out) & 7u)) return FPO_ERR_ALIGN;
    if (!workspace) return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    const size_t need = fpo_cosine_workspace(n);
    if (workspace_bytes < need) return FPO_ERR_WORKSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    FPO_TRY(cudaMemsetAsync(ws, 0, sizeof(unsigned), st));
    if (n == 0) {
        FPO_TRY(cudaMemsetAsync(out, 0, 4 * sizeof(double), st));
        return FPO_OK;
    }
    const int blocks = cosine_blocks(n);
    return cuda_status(launch_cosine(dtype, n, X, Y, reinterpret_cast<double*>(ws + kStatusBytes),
                                     blocks, out, st));
}

size_t fpo_norm_ratio_workspace(int32_t n_layers, int64_t n) {
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS || n < 0) return 0;
    return kStatusBytes +
           align_up(static_cast<size_t>(n_layers) * norm_ratio_blocks(n_layers, n) * 3 *
                    sizeof(double));
}

int32_t fpo_norm_ratio(int32_t n_layers, int64_t n, int32_t g_dtype, const void* const* G,
                       int32_t w_dtype, const void* const* W, double rel_step, double* out,
                       void* workspace, size_t workspace_bytes, void* stream) {
    if ((g_dtype != FPO_F32 && g_dtype != FPO_BF16) || (w_dtype != FPO_F32 && w_dtype != FPO_BF16))
        return FPO_ERR_DTYPE;
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS || n < 0) return FPO_ERR_SHAPE;
    if (!G || !W || !out) return FPO_ERR_NULL;
    for (int l = 0; l < n_layers; ++l) {
        if (n > 0 && (!G[l] || !W[l])) return FPO_ERR_NULL;
        if (!aligned16(G[l]) || !aligned16(W[l])) return FPO_ERR_ALIGN;
    }
    if (reinterpret_cast<uintptr_t>(out) & 7u) return FPO_ERR_ALIGN;
    if (!workspace) return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    if (workspace_bytes < fpo_norm_ratio_workspace(n_layers, n)) return FPO_ERR_WORKSPACE;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    FPO_TRY(cudaMemsetAsync(ws, 0, sizeof(unsigned), st));
    return cuda_status(launch_norm_ratio(g_dtype, w_dtype, n_layers, n, G, W, rel_step,
                                         reinterpret_cast<double*>(ws + kStatusBytes),
                                         norm_ratio_blocks(n_layers, n), out, st));
}

size_t fpo_cosine_grouped_workspace(int32_t n_layers, int64_t n) {
    return fpo_norm_ratio_workspace(n_layers, n);  // same partial layout
}

int32_t fpo_cosine_grouped(int32_t n_layers, int64_t n, int32_t dtype, const void* const* X,
                           const void* const* Y, double* out, void* workspace,
                           size_t workspace_bytes, void* stream) {
    if (dtype != FPO_F32 && dtype != FPO_BF16) return FPO_ERR_DTYPE;
    if (n_layers < 1 || n_layers > FPO_MAX_GROUPED_LAYERS || n < 0) return FPO_ERR_SHAPE;
    if (!X || !Y || !out) return FPO_ERR_NULL;
    for (int l = 0; l < n_layers; ++l) {
        if (n > 0 && (!X[l] || !Y[l])) return FPO_ERR_NULL;
        if (!aligned16(X[l]) || !aligned16(Y[l])) return FPO_ERR_ALIGN;
    }
    if (reinterpret_cast<uintptr_t>(out) & 7u) return FPO_ERR_ALIGN;
    if (!workspace) return FPO_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return FPO_ERR_ALIGN;
    if (workspace_bytes < fpo_cosine_grouped_workspace(n_layers, n)) return FPO_ERR_WORKSPACE;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    FPO_TRY(cudaMemsetAsync(ws, 0, sizeof(unsigned), st));
    return cuda_status(launch_cosine_grouped(dtype, n_layers, n, X, Y,
                                             reinterpret_cast<double*>(ws + kStatusBytes),
                                             norm_ratio_blocks(n_layers, n), out, st));
}

int32_t fpo_testing_gemm_bf16(int64_t M, int64_t N, int64_t K, int32_t a_mn, int32_t b_mn,
                              const void* A, const void* B, float* C, void* workspace,
                              size_t workspace_bytes, void* stream) {
    if (M <= 0 || N <= 0 || K <= 0 || M > INT_MAX || N > INT_MAX || K > INT_MAX) return FPO_ERR_SHAPE;
    if (a_mn && !b_mn) return FPO_ERR_ARG;
    if ((a_mn ? M : K) % 8 != 0 || (b_mn ? N : K) % 8 != 0 || N % 8 != 0) return FPO_ERR_SHAPE;
    if (!A || !B || !C) return FPO_ERR_NULL;
    if (!aligned16(A) || !aligned16(B) || !aligned16(C)) return FPO_ERR_ALIGN;
    if (!workspace || workspace_bytes < kStatusBytes) return FPO_ERR_WORKSPACE;
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned* status = static_cast<unsigned*>(workspace);
    FPO_TRY(cudaMemsetAsync(status, 0, sizeof(unsigned), st));
    return cuda_status(launch_test_gemm_bf16(static_cast<int>(M), static_cast<int>(N),
                                             static_cast<int>(K), a_mn != 0, b_mn != 0, A, B, C,
                                             status, st));
}

int32_t fpo_testing_set_gemm_variant(int32_t variant) {
    const int32_t prev = gemm_variant();
    set_gemm_variant(variant);
    return prev;
}

void fpo_testing_set_band(int32_t band) { set_band_override(band); }

uint64_t fpo_testing_kernel_launches(void) { return fpo::launches(); }

int64_t fpo_testing_direct_fixup_rows(const fpo_error_signal_desc* desc, const void* workspace,
                                      void* stream) {
    if (es_check_desc(desc) != FPO_OK || !workspace || desc->T == 0) return -1;
    const EsLayout L = es_layout(desc);
    if (L.algo != FPO_ES_DIRECT) return -1;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return -1;
    int n = 0;
    if (cudaMemcpy(&n, static_cast<const uint8_t*>(workspace) + L.fix_count, sizeof n,
                   cudaMemcpyDeviceToHost) != cudaSuccess)
        return -1;
    return n;
}

int32_t fpo_testing_wait_timeout(uint64_t limit_ns, void* workspace, size_t workspace_bytes,
                                 void* stream) {
    if (!workspace || workspace_bytes < kStatusBytes) return FPO_ERR_WORKSPACE;
    if (limit_ns == 0 || limit_ns > 10000000000ull) return FPO_ERR_ARG;  // at most 10 s
    int32_t rc = check_arch();
    if (rc != FPO_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    FPO_TRY(cudaMemsetAsync(workspace, 0, sizeof(unsigned), st));
    return cuda_status(launch_wait_timeout(static_cast<unsigned*>(workspace), limit_ns, st));
}

int32_t fpo_get_device_status(void* workspace, void* stream) {
    if (!workspace) return FPO_ERR_WORKSPACE;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(st) != cudaSuccess) return FPO_ERR_CUDA;
    unsigned word = 0;
    if (cudaMemcpy(&word, workspace, sizeof word, cudaMemcpyDeviceToHost) != cudaSuccess)
        return FPO_ERR_CUDA;
    if (cudaMemset(workspace, 0, sizeof word) != cudaSuccess) return FPO_ERR_CUDA;
    if (word & kDevTargetRange) return FPO_ERR_TARGET_RANGE;
    if (word & kDevTimeout) return FPO_ERR_TIMEOUT;
    return FPO_OK;
}

}  // extern "C"
