// gemm_bf16.cu -- host launchers of the four tcgen05 GEMMs of the FPO step.
//
//   logits pass      z = yhat W_U^T      M=T  N=V    K=d   A K-major, B K-major
//   recompute pass   same GEMM, epilogue writes E = s (softmax - onehot)
//   direct logits    same GEMM, epilogue writes P = exp(z - c) (target zero)
//   projection       g = E W_U           M=T  N=d    K=V   A K-major, B MN-major
//                    (or g = alpha P W_U + beta W_U[y] in the direct algorithm, whose
//                    epilogue applies the final-norm VJP and writes g~)
//   update           G = g~^T A_l        M=d  N=d_ff K=T   A MN-major, B MN-major
//
// Tensor maps are encoded per call (a few microseconds of host work) through
// the driver entry point of cuTensorMapEncodeTiled, so the library does not
// link libcuda directly.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <mutex>

#include <atomic>

#include "epilogues.cuh"
#include "internal.h"
#include "tc_gemm.cuh"
#include "tc_gemm_pair.cuh"

namespace fpo {
namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 2-D tensor [outer, inner] of bf16 (esz 2) or fp32 (esz 4) with row stride
// `ld` elements, box {box_inner, box_outer}, 128-byte swizzle, zero fill
// outside the tensor on loads (and clipping on stores).  L2 promotion of 128 bytes:
// one box row; 256-byte promotion fetched 15-55% more from DRAM in the step's GEMMs
// for the same time.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t ld,
              uint32_t box_inner, uint32_t box_outer, int esz = 2) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {ld * static_cast<uint64_t>(esz)};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    const CUtensorMapDataType dt =
        esz == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output maps of the epilogues: 32 rows x 128 bytes per store.
bool map_out_f32(CUtensorMap* m, void* base, int rows, int cols) {
    return make_map(m, base, cols, rows, cols, 32, 32, 4);
}
bool map_out_bf16(CUtensorMap* m, void* base, int rows, int cols) {
    return make_map(m, base, cols, rows, cols, 64, 32, 2);
}

// K-major operand [rows, K]: box {64 (K), rows_per_tile}
bool map_kmajor(CUtensorMap* m, const void* base, int rows, int K, int box_rows) {
    return make_map(m, base, K, rows, K, kBK, box_rows);
}
// MN-major operand [K, mn]: box {64 (MN), 64 (K)}
bool map_mnmajor(CUtensorMap* m, const void* base, int K, int mn) {
    return make_map(m, base, mn, K, mn, 64, kBK);
}

GemmShape make_shape(int M, int N, int K, int BN, int groups, int band, int BM = kBM) {
    GemmShape sh;
    sh.M = M;
    sh.N = N;
    sh.K = K;
    sh.m_blocks = (M + BM - 1) / BM;
    sh.n_blocks = (N + BN - 1) / BN;
    sh.k_blocks = (K + kBK - 1) / kBK;
    sh.groups = groups;
    sh.band = band;
    sh.tiles = static_cast<long long>(groups) * sh.m_blocks * sh.n_blocks;
    sh.tail_tiles = 0;
    sh.tail_split = 0;
    sh.sk_scratch = nullptr;
    sh.m_dev = nullptr;
    return sh;
}

template <int BN, bool A_MN, bool B_MN, int STAGES, int MAXG, class Epi>
cudaError_t run_gemm(const GemmMaps<MAXG>& maps, const typename Epi::Params& ep,
                     const GemmShape& sh, unsigned* status, cudaStream_t st) {
    if (sh.tiles <= 0 || sh.k_blocks <= 0) return cudaSuccess;
    using L = GemmSmem<BN, STAGES>;
    constexpr auto kern = tc_gemm_kernel<BN, A_MN, B_MN, STAGES, MAXG, Epi>;
    const cudaError_t attr_err = set_smem_limit<kern>(L::kBytes);
    if (attr_err != cudaSuccess) return attr_err;
    DevInfo di;
    if (!current_device_info(&di)) return cudaErrorUnknown;
    const long long grid = sh.tiles < di.sm_count ? sh.tiles : di.sm_count;
    kern<<<static_cast<unsigned>(grid), kGemmThreads, L::kBytes, st>>>(maps, ep, sh, status,
                                                                      wait_limit_ns()),
        ::fpo::note_launch();
    return cudaGetLastError();
}

// Clusters (of `cta` CTAs, the kernel's cluster size) that can be resident at once for a
// pair-kernel instantiation.
template <class Kern>
int pair_clusters(Kern kern, int smem_bytes, int sm_count, int cta) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(sm_count / cta * cta), 1, 1);
    cfg.blockDim = dim3(kGemmThreads, 1, 1);
    cfg.dynamicSmemBytes = static_cast<size_t>(smem_bytes);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1) {
        cudaGetLastError();
        n = sm_count / cta;
    }
    return n;
}

// pair_clusters for the current device, computed once per device (after the kernel's
// shared-memory limit is raised there).
template <auto Kern>
int resident_clusters(int smem_bytes, int sm_count, int cta) {
    static std::atomic<int> cache[kMaxDevices];
    const int dev = current_device();
    if (dev < 0) return sm_count / cta;
    int n = cache[dev].load(std::memory_order_relaxed);
    if (n > 0) return n;
    n = pair_clusters(Kern, smem_bytes, sm_count, cta);
    cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

// Split-K tail of one launch: tail_tiles tiles, each in tail_split k ranges (0: whole).
struct SkPlan {
    long long tail_tiles = 0;
    int tail_split = 0;
};

// Units of split tail tiles a scratch area must hold: up to three waves of pair clusters.
constexpr int kTailWaves = 3;

// The split of the last partial wave of `tiles` tiles over `clusters` clusters: R tail
// tiles in S k ranges, S chosen so that the R S units fill whole waves as nearly as
// possible (at most kTailWaves waves, at least 8 k-blocks per range); none if no split
// beats the plain partial wave.
SkPlan tail_plan(long long tiles, long long clusters, int k_blocks) {
    SkPlan p;
    const long long R = tiles % clusters;
    if (tiles < clusters || R == 0) return p;
    double best = static_cast<double>(R) / clusters;  // busy fraction of the plain last wave
    for (int S = 2; S <= 64; ++S) {
        if (R * S > kTailWaves * clusters || k_blocks / S < 8) break;
        const long long waves = (R * S + clusters - 1) / clusters;
        const double eff = static_cast<double>(R * S) / (waves * clusters);
        if (eff > best + 1e-9) {
            best = eff;
            p.tail_tiles = R;
            p.tail_split = S;
        }
    }
    return p;
}

// With sk_scratch non-null, the tiles of the last partial wave are split by tail_plan
// (SegCursor); the caller then runs sk_fixup over them (plan->tail_tiles > 0).
// sk_scratch holds kTailWaves x clusters x 256 x BN fp32.
template <int BN, bool A_MN, bool B_MN, int STAGES, int MAXG, class Epi>
cudaError_t run_gemm_pair(const GemmMaps<MAXG>& maps, const typename Epi::Params& ep,
                          const GemmShape& sh_in, unsigned* status, cudaStream_t st,
                          float* sk_scratch = nullptr, SkPlan* plan = nullptr) {
    if (plan) *plan = SkPlan{};
    if (sh_in.tiles <= 0 || sh_in.k_blocks <= 0) return cudaSuccess;
    using L = GemmPairSmem<BN, STAGES, pair_ksub<BN, A_MN, B_MN>()>;
    static_assert(L::kBytes <= 227 * 1024, "stages exceed the shared memory of a CTA");
    constexpr auto kern = tc_gemm_pair_kernel<BN, A_MN, B_MN, STAGES, MAXG, Epi>;
    const cudaError_t attr_err = set_smem_limit<kern>(L::kBytes);
    if (attr_err != cudaSuccess) return attr_err;
    DevInfo di;
    if (!current_device_info(&di)) return cudaErrorUnknown;
    const int max_clusters = resident_clusters<kern>(L::kBytes, di.sm_count, 2);
    const long long clusters = sh_in.tiles < max_clusters ? sh_in.tiles : max_clusters;
    GemmShape sh = sh_in;
    if (sk_scratch) {
        const SkPlan p = tail_plan(sh.tiles, clusters, sh.k_blocks);
        if (p.tail_tiles > 0) {
            sh.tail_tiles = p.tail_tiles;
            sh.tail_split = p.tail_split;
            sh.sk_scratch = sk_scratch;
            if (plan) *plan = p;
        }
    }
    kern<<<static_cast<unsigned>(2 * clusters), kGemmThreads, L::kBytes, st>>>(maps, ep, sh, status,
                                                                              wait_limit_ns()),
        ::fpo::note_launch();
    return cudaGetLastError();
}

// Fixups of the split-K tail: sum the tail_split k-range partials of every split tail
// tile in range order, then apply the epilogue the whole tiles got.
// Grid (tail tiles, 256 rows / rows per block): one thread per 4 columns of a row.
constexpr int kFixupThreads = 256;

// The summed partials of this thread's 4 columns; false outside the matrix.
template <int BN>
__device__ __forceinline__ bool sk_tail_sum(const GemmShape& sh, const float* __restrict__ scratch,
                                            int& row, int& n, float (&s4)[4]) {
    constexpr int kThreadsPerRow = BN / 4;
    constexpr int kRowsPerBlock = kFixupThreads / kThreadsPerRow;
    const long long R = sh.tail_tiles;
    const long long r_tile = blockIdx.x;
    const int r = blockIdx.y * kRowsPerBlock + threadIdx.x / kThreadsPerRow;
    const int col = (threadIdx.x % kThreadsPerRow) * 4;
    int g, mp, nb;
    tile_coords(sh.tiles - R + r_tile, sh, g, mp, nb);
    row = mp * kPairBM + r;
    n = nb * BN + col;
    if (row >= sh.M || n >= sh.N) return false;  // N % 8 == 0: whole groups of 4
    s4[0] = s4[1] = s4[2] = s4[3] = 0.f;
    for (int q = 0; q < sh.tail_split; ++q) {
        const float4 u = *reinterpret_cast<const float4*>(
            scratch + ((static_cast<size_t>(q) * R + r_tile) * kPairBM + r) * BN + col);
        s4[0] += u.x;
        s4[1] += u.y;
        s4[2] += u.z;
        s4[3] += u.w;
    }
    return true;
}

// Plain fp32 sums, as EpiStoreF32 writes whole tiles (the projection g = E W_U).
template <int BN>
__global__ void __launch_bounds__(kFixupThreads)
    sk_fixup_kernel(const GemmShape sh, const float* __restrict__ scratch, float* __restrict__ C) {
    int row, n;
    float s4[4];
    if (!sk_tail_sum<BN>(sh, scratch, row, n, s4)) return;
    *reinterpret_cast<float4*>(C + static_cast<size_t>(row) * sh.N + n) =
        make_float4(s4[0], s4[1], s4[2], s4[3]);
}

// The direct algorithm's projection with the final-norm VJP fused in, as EpiProjVjp
// writes whole tiles: g = alpha sum + beta W_U[y], out = bf16 of
// (w g - (h / rho) cv / d) / max(rho, min_rms).
struct VjpArgs {
    const float* alpha;
    const float* beta;
    const float* cv;
    const float* rho;
    const int* y;
    const __nv_bfloat16* W_U;
    const __nv_bfloat16* h;
    const __nv_bfloat16* w;
    float min_rms, inv_d;
};

template <int BN>
__global__ void __launch_bounds__(kFixupThreads)
    sk_fixup_vjp_kernel(const GemmShape sh, const float* __restrict__ scratch,
                        __nv_bfloat16* __restrict__ out, const VjpArgs va) {
    int row, n;
    float s4[4];
    if (!sk_tail_sum<BN>(sh, scratch, row, n, s4)) return;
    const float a = va.alpha[row], bb = va.beta[row];
    const float rr = va.rho[row];
    const float kd = va.cv[row] * va.inv_d;
    const float pref = 1.0f / fmaxf(rr, va.min_rms);
    // the same association as EpiProjVjp: w (a pref sum + b pref W_U[y]) - h (kd pref / rho)
    const float ap = a * pref, bp = bb * pref, nk = -(kd * (1.0f / rr)) * pref;
    const __nv_bfloat16* wy =
        (a != 0.f && bb != 0.f) ? va.W_U + static_cast<long long>(va.y[row]) * sh.N : nullptr;
    const __nv_bfloat16* hr = va.h + static_cast<long long>(row) * sh.N;
    float o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float yv = wy ? __bfloat162float(wy[n + j]) : 0.f;
        const float t = fmaf(bp, yv, ap * s4[j]);
        o[j] = a == 0.f ? 0.f
                        : fmaf(__bfloat162float(va.w[n + j]), t,
                               nk * __bfloat162float(hr[n + j]));
    }
    *reinterpret_cast<uint2*>(out + static_cast<size_t>(row) * sh.N + n) =
        make_uint2(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]));
}

template <int BN>
dim3 sk_fixup_grid(const SkPlan& plan) {
    constexpr int kRowsPerBlock = kFixupThreads / (BN / 4);
    return dim3(static_cast<unsigned>(plan.tail_tiles), kPairBM / kRowsPerBlock);
}

GemmShape sk_fixup_shape(const SkPlan& plan, const GemmShape& sh_in) {
    GemmShape sh = sh_in;
    sh.tail_tiles = plan.tail_tiles;
    sh.tail_split = plan.tail_split;
    return sh;
}

template <int BN>
cudaError_t launch_sk_fixup(const SkPlan& plan, const GemmShape& sh, const float* scratch,
                            float* C, cudaStream_t st) {
    if (plan.tail_tiles <= 0) return cudaSuccess;
    sk_fixup_kernel<BN><<<sk_fixup_grid<BN>(plan), kFixupThreads, 0, st>>>(
        sk_fixup_shape(plan, sh), scratch, C), ::fpo::note_launch();
    return cudaGetLastError();
}

template <int BN>
cudaError_t launch_sk_fixup_vjp(const SkPlan& plan, const GemmShape& sh, const float* scratch,
                                void* out, const VjpArgs& va, cudaStream_t st) {
    if (plan.tail_tiles <= 0) return cudaSuccess;
    sk_fixup_vjp_kernel<BN><<<sk_fixup_grid<BN>(plan), kFixupThreads, 0, st>>>(
        sk_fixup_shape(plan, sh), scratch, static_cast<__nv_bfloat16*>(out), va),
        ::fpo::note_launch();
    return cudaGetLastError();
}

constexpr int kPairStages = 3;   // 256 x 256 pair tiles: 64 KB stages of two k-blocks
constexpr int kWideBN = 512;     // pair tiles 256 x 512: 48 KB stages
constexpr int kWideStages = 4;

// 0 = single-CTA tiles, 1 = CTA-pair tiles, 2 = CTA-pair tiles with 256 x 512 tiles for
// the projection (default: its K loop runs over the whole vocabulary, so the epilogue
// that the single accumulator cannot overlap costs ~1%, while a quarter less operand
// traffic per FLOP made the projection 6-7% faster)
std::atomic<int> g_gemm_variant{2};
std::atomic<int> g_band_override{0};  // > 0: rasterisation band height (tests / tuning)

bool use_pair() { return g_gemm_variant.load(std::memory_order_relaxed) >= 1; }
bool wide_proj() { return g_gemm_variant.load(std::memory_order_relaxed) >= 2; }

// Rasterisation band in tile rows, unless overridden: 16 tile rows, i.e. 2048
// output rows of single-CTA tiles and 4096 of pair tiles.  With pair tiles the
// 4096-row band gave the lowest DRAM traffic of the three GEMMs of the OLMo-2-7B
// shape (band heights 2 to 32 measured).
constexpr int kBandTiles = 16;
int band_for(bool) {
    const int o = g_band_override.load(std::memory_order_relaxed);
    return o > 0 ? o : kBandTiles;
}

}  // namespace

void set_band_override(int b) { g_band_override.store(b > 0 ? b : 0, std::memory_order_relaxed); }

void set_gemm_variant(int v) {
    g_gemm_variant.store(v >= 0 && v <= 2 ? v : 0, std::memory_order_relaxed);
}
int gemm_variant() { return g_gemm_variant.load(std::memory_order_relaxed); }

size_t proj_sk_scratch_bytes() {
    // kTailWaves x clusters units of 256 x 512 fp32; clusters of the 256 x 512 pair kernel
    // on the current device, or an upper bound of 128 without one
    using L = GemmPairSmem<kWideBN, kWideStages, pair_ksub<kWideBN, false, true>()>;
    constexpr auto kern = tc_gemm_pair_kernel<kWideBN, false, true, kWideStages, 1, EpiProjVjp>;
    DevInfo di;
    long long c = 128;
    if (current_device_info(&di) && set_smem_limit<kern>(L::kBytes) == cudaSuccess)
        c = resident_clusters<kern>(L::kBytes, di.sm_count, 2);
    cudaGetLastError();
    return static_cast<size_t>(kTailWaves) * c * kPairBM * kWideBN * sizeof(float);
}

constexpr int kLseBN = 256;
constexpr int kLseStages = 4;
int lse_tile_n_bf16() { return kLseBN; }

cudaError_t launch_lse_partial_bf16(const void* yhat, const void* W_U, const int32_t* y, int T,
                                    int d, int V, float2* part, int part_ld, float* zy, float* z,
                                    unsigned* status, cudaStream_t st) {
    const bool pair = use_pair();
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], yhat, T, d, kBM) ||
        !map_kmajor(&maps.b[0], W_U, V, d, pair ? kLseBN / 2 : kLseBN))
        return cudaErrorInvalidValue;
    const GemmShape sh = make_shape(T, V, d, kLseBN, 1, band_for(pair), pair ? kPairBM : kBM);
    if (z) {
        EpiLseStoreZ::Params ep;
        if (!map_out_f32(&ep.zmap, z, T, V)) return cudaErrorInvalidValue;
        ep.part = part;
        ep.part_ld = part_ld;
        ep.zy = zy;
        ep.y = y;
        ep.M = T;
        ep.N = V;
        if (pair)
            return run_gemm_pair<kLseBN, false, false, kPairStages, 1, EpiLseStoreZ>(maps, ep, sh,
                                                                                     status, st);
        return run_gemm<kLseBN, false, false, kLseStages, 1, EpiLseStoreZ>(maps, ep, sh, status, st);
    }
    EpiLsePartial::Params ep;
    ep.zmap = maps.a[0];  // unused
    ep.part = part;
    ep.part_ld = part_ld;
    ep.zy = zy;
    ep.y = y;
    ep.M = T;
    ep.N = V;
    if (pair)
        return run_gemm_pair<kLseBN, false, false, kPairStages, 1, EpiLsePartial>(maps, ep, sh,
                                                                                  status, st);
    return run_gemm<kLseBN, false, false, kLseStages, 1, EpiLsePartial>(maps, ep, sh, status, st);
}

cudaError_t launch_error_bf16(const void* yhat, const void* W_U, const int32_t* y, const float* lse,
                              int Tc, int d, int V, float s, void* E, unsigned* status,
                              cudaStream_t st) {
    const bool pair = use_pair();
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], yhat, Tc, d, kBM) ||
        !map_kmajor(&maps.b[0], W_U, V, d, pair ? kLseBN / 2 : kLseBN))
        return cudaErrorInvalidValue;
    EpiError::Params ep;
    if (!map_out_bf16(&ep.Emap, E, Tc, V)) return cudaErrorInvalidValue;
    ep.lse = lse;
    ep.y = y;
    ep.M = Tc;
    ep.N = V;
    ep.s = s;
    const GemmShape sh = make_shape(Tc, V, d, kLseBN, 1, band_for(pair), pair ? kPairBM : kBM);
    if (pair)
        return run_gemm_pair<kLseBN, false, false, kPairStages, 1, EpiError>(maps, ep, sh, status,
                                                                             st);
    return run_gemm<kLseBN, false, false, kLseStages, 1, EpiError>(maps, ep, sh, status, st);
}

cudaError_t launch_anchor_prob_bf16(const void* yhat, const void* W_U, const int32_t* y,
                                    const float* anchor, int T, int d, int V, float* su, float* sx,
                                    float* qz, int part_ld, void* P, unsigned* status,
                                    cudaStream_t st) {
    const bool pair = use_pair();
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], yhat, T, d, kBM) ||
        !map_kmajor(&maps.b[0], W_U, V, d, pair ? kLseBN / 2 : kLseBN))
        return cudaErrorInvalidValue;
    EpiAnchorProb::Params ep;
    if (!map_out_bf16(&ep.pmap, P, T, V)) return cudaErrorInvalidValue;
    ep.su = su;
    ep.sx = sx;
    ep.qz = qz;
    ep.part_ld = part_ld;
    ep.y = y;
    ep.anchor = anchor;
    ep.M = T;
    ep.N = V;
    const GemmShape sh = make_shape(T, V, d, kLseBN, 1, band_for(pair), pair ? kPairBM : kBM);
    if (pair)
        return run_gemm_pair<kLseBN, false, false, kPairStages, 1, EpiAnchorProb>(maps, ep, sh,
                                                                                  status, st);
    return run_gemm<kLseBN, false, false, kLseStages, 1, EpiAnchorProb>(maps, ep, sh, status, st);
}

// The fixup passes: the same GEMM as the logits pass on the gathered rows outside the
// anchor window.  Always the pair kernel (the only one that reads its row count on the
// device): the recomputed rows are identical whichever kernel variant the other GEMMs use.
cudaError_t launch_fixup_lse_bf16(const void* yfix, const void* W_U, const int* fix,
                                  const int* fix_count, int Tc, int d, int V, float2* part,
                                  int part_ld, unsigned* status, cudaStream_t st) {
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], yfix, Tc, d, kBM) || !map_kmajor(&maps.b[0], W_U, V, d, kLseBN / 2))
        return cudaErrorInvalidValue;
    EpiFixLse::Params ep;
    ep.part = part;
    ep.part_ld = part_ld;
    ep.fix = fix;
    ep.count = fix_count;
    ep.N = V;
    GemmShape sh = make_shape(Tc, V, d, kLseBN, 1, band_for(true), kPairBM);
    sh.m_dev = fix_count;
    return run_gemm_pair<kLseBN, false, false, kPairStages, 1, EpiFixLse>(maps, ep, sh, status, st);
}

cudaError_t launch_fixup_logits_bf16(const void* yfix, const void* W_U, const int* fix,
                                     const int* fix_count, const int32_t* y, const float* lse,
                                     int Tc, int d, int V, void* P, float* sx, float* qz,
                                     int n_tiles, unsigned* status, cudaStream_t st) {
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], yfix, Tc, d, kBM) || !map_kmajor(&maps.b[0], W_U, V, d, kLseBN / 2))
        return cudaErrorInvalidValue;
    EpiFixProb::Params ep;
    ep.P = static_cast<__nv_bfloat16*>(P);
    ep.sx = sx;
    ep.qz = qz;
    ep.fix = fix;
    ep.count = fix_count;
    ep.y = y;
    ep.lse = lse;
    ep.n_tiles = n_tiles;
    ep.N = V;
    GemmShape sh = make_shape(Tc, V, d, kLseBN, 1, band_for(true), kPairBM);
    sh.m_dev = fix_count;
    return run_gemm_pair<kLseBN, false, false, kPairStages, 1, EpiFixProb>(maps, ep, sh, status, st);
}

constexpr int kProjBN = 256;
constexpr int kProjStages = 4;

cudaError_t launch_proj_vjp_bf16(const void* P, const void* W_U, const int32_t* y,
                                 const float* alpha, const float* beta, const float* cv,
                                 const float* rho, const void* h, const void* w, float min_rms,
                                 int Tc, int d, int V, void* g_tilde, float* sk_scratch,
                                 unsigned* status, cudaStream_t st) {
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], P, Tc, V, kBM) || !map_mnmajor(&maps.b[0], W_U, V, d))
        return cudaErrorInvalidValue;
    EpiProjVjp::Params ep;
    if (!map_out_bf16(&ep.omap, g_tilde, Tc, d)) return cudaErrorInvalidValue;
    VjpArgs va;
    va.alpha = ep.alpha = alpha;
    va.beta = ep.beta = beta;
    va.cv = ep.cv = cv;
    va.rho = ep.rho = rho;
    va.y = ep.y = y;
    va.W_U = ep.W_U = static_cast<const __nv_bfloat16*>(W_U);
    va.h = ep.h = static_cast<const __nv_bfloat16*>(h);
    va.w = ep.w = static_cast<const __nv_bfloat16*>(w);
    va.min_rms = ep.min_rms = min_rms;
    va.inv_d = ep.inv_d = 1.0f / static_cast<float>(d);
    ep.M = Tc;
    ep.N = d;
    if (wide_proj()) {
        ep.tile_n = kWideBN;
        const GemmShape sh = make_shape(Tc, d, V, kWideBN, 1, band_for(true), kPairBM);
        SkPlan plan;
        cudaError_t e = run_gemm_pair<kWideBN, false, true, kWideStages, 1, EpiProjVjp>(
            maps, ep, sh, status, st, sk_scratch, &plan);
        if (e != cudaSuccess) return e;
        return launch_sk_fixup_vjp<kWideBN>(plan, sh, sk_scratch, g_tilde, va, st);
    }
    ep.tile_n = kProjBN;
    if (use_pair())
        return run_gemm_pair<kProjBN, false, true, kPairStages, 1, EpiProjVjp>(
            maps, ep, make_shape(Tc, d, V, kProjBN, 1, band_for(true), kPairBM), status, st);
    return run_gemm<kProjBN, false, true, kProjStages, 1, EpiProjVjp>(
        maps, ep, make_shape(Tc, d, V, kProjBN, 1, band_for(false)), status, st);
}

cudaError_t launch_proj_bf16(const void* E, const void* W_U, int Tc, int d, int V, float* g,
                             float* sk_scratch, unsigned* status, cudaStream_t st) {
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], E, Tc, V, kBM) || !map_mnmajor(&maps.b[0], W_U, V, d))
        return cudaErrorInvalidValue;
    EpiStoreF32::Params ep;
    if (!map_out_f32(&ep.Cmap, g, Tc, d)) return cudaErrorInvalidValue;
    ep.M = Tc;
    ep.N = d;
    if (wide_proj()) {
        const GemmShape sh = make_shape(Tc, d, V, kWideBN, 1, band_for(true), kPairBM);
        SkPlan plan;
        cudaError_t e = run_gemm_pair<kWideBN, false, true, kWideStages, 1, EpiStoreF32>(
            maps, ep, sh, status, st, sk_scratch, &plan);
        if (e != cudaSuccess) return e;
        return launch_sk_fixup<kWideBN>(plan, sh, sk_scratch, g, st);
    }
    if (use_pair())
        return run_gemm_pair<kProjBN, false, true, kPairStages, 1, EpiStoreF32>(
            maps, ep, make_shape(Tc, d, V, kProjBN, 1, band_for(true), kPairBM), status, st);
    return run_gemm<kProjBN, false, true, kProjStages, 1, EpiStoreF32>(
        maps, ep, make_shape(Tc, d, V, kProjBN, 1, band_for(false)), status, st);
}

constexpr int kUpdBN = 256;
constexpr int kUpdStages = 4;

cudaError_t launch_update_bf16(int n, int T, int d, int d_ff, const void* const* g,
                               const void* const* A, float lr, float* const* W_master,
                               void* const* W_out, void* const* G_out, unsigned* status,
                               cudaStream_t st) {
    if (n < 1 || n > kMaxGroups) return cudaErrorInvalidValue;
    static GemmMaps<kMaxGroups> maps;  // host staging; copied into the launch parameters
    static EpiUpdate::Params ep;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (int l = 0; l < n; ++l) {
        if (l > 0 && g[l] == g[0])
            maps.a[l] = maps.a[0];
        else if (!map_mnmajor(&maps.a[l], g[l], T, d))
            return cudaErrorInvalidValue;
        if (!map_mnmajor(&maps.b[l], A[l], T, d_ff)) return cudaErrorInvalidValue;
        ep.W_master[l] = W_master ? W_master[l] : nullptr;
        ep.W_out[l] = W_out ? static_cast<__nv_bfloat16*>(W_out[l]) : nullptr;
        ep.G_out[l] = G_out ? static_cast<__nv_bfloat16*>(G_out[l]) : nullptr;
    }
    for (int l = n; l < kMaxGroups; ++l) {
        maps.a[l] = maps.a[0];
        maps.b[l] = maps.b[0];
        ep.W_master[l] = nullptr;
        ep.W_out[l] = nullptr;
        ep.G_out[l] = nullptr;
    }
    ep.ld = d_ff;
    ep.M = d;
    ep.N = d_ff;
    ep.neg_lr = -lr;
    if (use_pair())
        return run_gemm_pair<kUpdBN, true, true, kPairStages, kMaxGroups, EpiUpdate>(
            maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(true), kPairBM), status, st);
    return run_gemm<kUpdBN, true, true, kUpdStages, kMaxGroups, EpiUpdate>(
        maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(false)), status, st);
}

cudaError_t launch_grad_bf16(int n, int T, int d, int d_ff, const void* const* g,
                             const void* const* A, float* const* G_out, unsigned* status,
                             cudaStream_t st) {
    if (n < 1 || n > kMaxGroups) return cudaErrorInvalidValue;
    static GemmMaps<kMaxGroups> maps;
    static EpiStoreGroupF32::Params ep;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (int l = 0; l < n; ++l) {
        if (l > 0 && g[l] == g[0])
            maps.a[l] = maps.a[0];
        else if (!map_mnmajor(&maps.a[l], g[l], T, d))
            return cudaErrorInvalidValue;
        if (!map_mnmajor(&maps.b[l], A[l], T, d_ff)) return cudaErrorInvalidValue;
        ep.G[l] = G_out[l];
    }
    for (int l = n; l < kMaxGroups; ++l) {
        maps.a[l] = maps.a[0];
        maps.b[l] = maps.b[0];
        ep.G[l] = G_out[0];
    }
    ep.ld = d_ff;
    ep.M = d;
    ep.N = d_ff;
    if (use_pair())
        return run_gemm_pair<kUpdBN, true, true, kPairStages, kMaxGroups, EpiStoreGroupF32>(
            maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(true), kPairBM), status, st);
    return run_gemm<kUpdBN, true, true, kUpdStages, kMaxGroups, EpiStoreGroupF32>(
        maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(false)), status, st);
}

cudaError_t launch_opt_step_bf16(int n, int T, int d, int d_ff, const void* const* g,
                                 const void* const* A, const OptimParams& op,
                                 float* const* W_master, float* const* s1, float* const* s2,
                                 float* const* D, float* part, unsigned* status, cudaStream_t st) {
    if (n < 1 || n > kMaxGroups) return cudaErrorInvalidValue;
    static GemmMaps<kMaxGroups> maps;
    static EpiOptStep::Params ep;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (int l = 0; l < kMaxGroups; ++l) {
        const int k = l < n ? l : 0;
        if (l < n) {
            if (l > 0 && g[l] == g[0])
                maps.a[l] = maps.a[0];
            else if (!map_mnmajor(&maps.a[l], g[l], T, d))
                return cudaErrorInvalidValue;
            if (!map_mnmajor(&maps.b[l], A[l], T, d_ff)) return cudaErrorInvalidValue;
        } else {
            maps.a[l] = maps.a[0];
            maps.b[l] = maps.b[0];
        }
        ep.W_master[l] = W_master[k];
        ep.s1[l] = s1 ? s1[k] : nullptr;
        ep.s2[l] = s2 ? s2[k] : nullptr;
        ep.D[l] = D ? D[k] : nullptr;
    }
    ep.part = part;
    ep.op = op;
    ep.ld = d_ff;
    ep.M = d;
    ep.N = d_ff;
    ep.m256 = (d + 255) / 256;
    ep.n_blocks = (d_ff + kUpdBN - 1) / kUpdBN;
    if (use_pair())
        return run_gemm_pair<kUpdBN, true, true, kPairStages, kMaxGroups, EpiOptStep>(
            maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(true), kPairBM), status, st);
    return run_gemm<kUpdBN, true, true, kUpdStages, kMaxGroups, EpiOptStep>(
        maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(false)), status, st);
}

size_t opt_step_partial_bytes(int n_layers, int d, int d_ff) {
    return static_cast<size_t>(n_layers) * ((d + 255) / 256) * ((d_ff + kUpdBN - 1) / kUpdBN) * 8 *
           2 * sizeof(float);
}

// Second pass of the fused cosine: one block per layer adds the layer's slot triples in a
// fixed order (thread-strided fp64 sums, a fixed butterfly per warp, then the warps' sums
// in warp order) and writes <G, Y>, ||G||^2, ||Y||^2 and the cosine.
constexpr int kCosFinalThreads = 256;

__device__ __forceinline__ double warp_sum_f64(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__global__ void __launch_bounds__(kCosFinalThreads)
    grad_cosine_final_kernel(const float* __restrict__ part, int slots, double* __restrict__ out) {
    const int layer = blockIdx.x;
    const float* p = part + static_cast<size_t>(layer) * slots * 3;
    double gy = 0.0, gg = 0.0, yy = 0.0;
#pragma unroll 4
    for (int i = threadIdx.x; i < slots; i += kCosFinalThreads) {
        gy += p[3 * i];
        gg += p[3 * i + 1];
        yy += p[3 * i + 2];
    }
    gy = warp_sum_f64(gy);
    gg = warp_sum_f64(gg);
    yy = warp_sum_f64(yy);
    __shared__ double sh[3][kCosFinalThreads / 32];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sh[0][wid] = gy;
        sh[1][wid] = gg;
        sh[2][wid] = yy;
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    gy = gg = yy = 0.0;
    for (int k = 0; k < kCosFinalThreads / 32; ++k) {
        gy += sh[0][k];
        gg += sh[1][k];
        yy += sh[2][k];
    }
    double* o = out + 4 * layer;
    o[0] = gy;
    o[1] = gg;
    o[2] = yy;
    o[3] = (gg > 0.0 && yy > 0.0) ? gy / (sqrt(gg) * sqrt(yy)) : 0.0;
}

size_t grad_cosine_partial_bytes(int n, int d, int d_ff) {
    const size_t m256 = (static_cast<size_t>(d) + 255) / 256;
    const size_t nb = (static_cast<size_t>(d_ff) + kUpdBN - 1) / kUpdBN;
    return static_cast<size_t>(n) * m256 * nb * 8 * 3 * sizeof(float);
}

cudaError_t launch_grad_cosine_bf16(int n, int T, int d, int d_ff, const void* const* g,
                                    const void* const* A, const void* const* Y,
                                    void* const* G_out, float* part, double* out,
                                    unsigned* status, cudaStream_t st) {
    if (n < 1 || n > kMaxGroups) return cudaErrorInvalidValue;
    static GemmMaps<kMaxGroups> maps;
    static EpiGradCos::Params ep;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (int l = 0; l < n; ++l) {
        if (l > 0 && g[l] == g[0])
            maps.a[l] = maps.a[0];
        else if (!map_mnmajor(&maps.a[l], g[l], T, d))
            return cudaErrorInvalidValue;
        if (!map_mnmajor(&maps.b[l], A[l], T, d_ff)) return cudaErrorInvalidValue;
        ep.G_out[l] = static_cast<__nv_bfloat16*>(G_out[l]);
        ep.Y[l] = static_cast<const __nv_bfloat16*>(Y[l]);
    }
    for (int l = n; l < kMaxGroups; ++l) {
        maps.a[l] = maps.a[0];
        maps.b[l] = maps.b[0];
        ep.G_out[l] = ep.G_out[0];
        ep.Y[l] = ep.Y[0];
    }
    ep.part = part;
    ep.ld = d_ff;
    ep.M = d;
    ep.N = d_ff;
    ep.m256 = (d + 255) / 256;
    ep.n_blocks = (d_ff + kUpdBN - 1) / kUpdBN;
    static_assert(EpiGradCos::kTileN == kUpdBN, "the cosine epilogue prefetches 256-column tiles");
    // every slot is written by a tile (pair kernel), but single-CTA 128-row tiles leave
    // the upper half of a last, short 256-row block unwritten: start from zeros
    cudaError_t e = cudaMemsetAsync(part, 0, grad_cosine_partial_bytes(n, d, d_ff), st);
    if (e != cudaSuccess) return e;
    if (use_pair())
        e = run_gemm_pair<kUpdBN, true, true, kPairStages, kMaxGroups, EpiGradCos>(
            maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(true), kPairBM), status, st);
    else
        e = run_gemm<kUpdBN, true, true, kUpdStages, kMaxGroups, EpiGradCos>(
            maps, ep, make_shape(d, d_ff, T, kUpdBN, n, band_for(false)), status, st);
    if (e != cudaSuccess) return e;
    grad_cosine_final_kernel<<<n, kCosFinalThreads, 0, st>>>(part, ep.m256 * ep.n_blocks * 8, out),
        ::fpo::note_launch();
    return cudaGetLastError();
}

cudaError_t launch_swiglu_bf16(int T, int d, int d_ff, const void* g, const void* W3,
                               const void* a, const void* b, void* dA, void* dB, unsigned* status,
                               cudaStream_t st) {
    GemmMaps<1> maps;
    if (!map_kmajor(&maps.a[0], g, T, d, kBM) || !map_mnmajor(&maps.b[0], W3, d, d_ff))
        return cudaErrorInvalidValue;
    static_assert(EpiSwiglu::kTileN == 256, "the SwiGLU epilogue prefetches 256-column tiles");
    EpiSwiglu::Params ep;
    if (!map_out_bf16(&ep.dAmap, dA, T, d_ff) || !map_out_bf16(&ep.dBmap, dB, T, d_ff))
        return cudaErrorInvalidValue;
    ep.a = static_cast<const __nv_bfloat16*>(a);
    ep.b = static_cast<const __nv_bfloat16*>(b);
    ep.ld = d_ff;
    ep.M = T;
    ep.N = d_ff;
    if (use_pair())
        return run_gemm_pair<256, false, true, kPairStages, 1, EpiSwiglu>(
            maps, ep, make_shape(T, d_ff, d, 256, 1, band_for(true), kPairBM), status, st);
    return run_gemm<256, false, true, 4, 1, EpiSwiglu>(
        maps, ep, make_shape(T, d_ff, d, 256, 1, band_for(false)), status, st);
}

cudaError_t launch_test_gemm_bf16(int M, int N, int K, bool a_mn, bool b_mn, const void* A,
                                  const void* B, float* C, unsigned* status, cudaStream_t st) {
    const bool pair = use_pair();
    GemmMaps<1> maps;
    bool ok = a_mn ? map_mnmajor(&maps.a[0], A, K, M) : map_kmajor(&maps.a[0], A, M, K, kBM);
    ok = ok && (b_mn ? map_mnmajor(&maps.b[0], B, K, N)
                     : map_kmajor(&maps.b[0], B, N, K, pair ? 128 : 256));
    if (!ok) return cudaErrorInvalidValue;
    EpiStoreF32::Params ep;
    if (!map_out_f32(&ep.Cmap, C, M, N)) return cudaErrorInvalidValue;
    ep.M = M;
    ep.N = N;
    if (wide_proj()) {  // every layout on 256 x 512 pair tiles
        const GemmShape sh = make_shape(M, N, K, kWideBN, 1, band_for(true), kPairBM);
        if (!a_mn && !b_mn)
            return run_gemm_pair<kWideBN, false, false, kWideStages, 1, EpiStoreF32>(maps, ep, sh,
                                                                                    status, st);
        if (!a_mn && b_mn)
            return run_gemm_pair<kWideBN, false, true, kWideStages, 1, EpiStoreF32>(maps, ep, sh,
                                                                                   status, st);
        if (a_mn && b_mn)
            return run_gemm_pair<kWideBN, true, true, kWideStages, 1, EpiStoreF32>(maps, ep, sh,
                                                                                  status, st);
        return cudaErrorInvalidValue;
    }
    if (pair) {
        const GemmShape sh = make_shape(M, N, K, 256, 1, band_for(true), kPairBM);
        if (!a_mn && !b_mn)
            return run_gemm_pair<256, false, false, kPairStages, 1, EpiStoreF32>(maps, ep, sh, status, st);
        if (!a_mn && b_mn)
            return run_gemm_pair<256, false, true, kPairStages, 1, EpiStoreF32>(maps, ep, sh, status, st);
        if (a_mn && b_mn)
            return run_gemm_pair<256, true, true, kPairStages, 1, EpiStoreF32>(maps, ep, sh, status, st);
        return cudaErrorInvalidValue;
    }
    const GemmShape sh = make_shape(M, N, K, 256, 1, band_for(false));
    if (!a_mn && !b_mn) return run_gemm<256, false, false, 4, 1, EpiStoreF32>(maps, ep, sh, status, st);
    if (!a_mn && b_mn) return run_gemm<256, false, true, 4, 1, EpiStoreF32>(maps, ep, sh, status, st);
    if (a_mn && b_mn) return run_gemm<256, true, true, 4, 1, EpiStoreF32>(maps, ep, sh, status, st);
    return cudaErrorInvalidValue;
}

}  // namespace fpo
