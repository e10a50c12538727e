// tc_gemm.cuh -- persistent tcgen05 GEMM core with pluggable epilogues.
//
//   C[g][m, n] = sum_k A(m, k) * B[g](n, k)      (bf16 inputs, fp32 accumulate)
//
// One CTA per SM (persistent over output tiles), 192 threads:
//   warp 0      TMA producer: streams A/B k-blocks into a STAGES-deep ring of
//               128-byte-swizzled shared-memory buffers (mbarrier full/empty).
//   warp 1      allocates TMEM; lane 0 issues tcgen05.mma (128 x BN x 16) and
//               commits stage releases / accumulator-ready signals.
//   warps 2..5  epilogue: tcgen05.ld of the fp32 accumulator (one row per
//               thread), hand the values to the Epilogue functor.
// The accumulator is double-buffered in TMEM (2 x BN columns) so the epilogue
// of tile i overlaps the mainloop of tile i+1.
//
// Operands may be K-major (K contiguous) or MN-major (M/N contiguous); both
// are loaded by the TMA engine with the 128-byte swizzle and described to the
// tensor core by the matching shared-memory descriptor.  Every wait is bounded
// (WaitGuard); on a timeout all roles stop issuing, in-flight copies and MMAs
// are drained with a second wait of a fixed, generous limit (kDrainLimitNs), TMEM
// is freed and the kernel returns with the timeout bit set in the status word.
#pragma once

#include "ptx.cuh"

namespace fpo {

constexpr int kBM = 128;       // UMMA M (one TMEM lane per output row)
constexpr int kBK = 64;        // k-block: 64 bf16 = one 128-byte swizzle row
constexpr int kUmmaK = 16;     // K of one tcgen05.mma.kind::f16
constexpr int kGemmThreads = 192;
constexpr int kMaxGroups = 64;
// Limit of the teardown waits for copies and MMAs already issued (they complete in
// microseconds); fixed, so that a short wait limit cannot cut them off.
constexpr uint64_t kDrainLimitNs = 1000000000ull;

struct GemmShape {
    int M, N, K;
    int m_blocks, n_blocks, k_blocks;
    int groups;        // independent problems with equal shapes (target layers)
    int band;          // rasterisation band height in m-blocks (L2 reuse)
    long long tiles;   // groups * m_blocks * n_blocks
    // Split-K tail (pair kernel only): the last tail_tiles tiles (less than one wave)
    // are each split into tail_split equal k-block ranges, and every range leaves its
    // fp32 sums in sk_scratch ([unit][256][BN]) for a fixup kernel.  0 = whole tiles.
    long long tail_tiles;
    int tail_split;
    float* sk_scratch;
    // Pair kernel only: when set, the number of rows of A is read here on the device at
    // kernel start (at most M; the tensor maps cover M rows) and the tiles beyond it are
    // dropped; with no rows the kernel returns before it sets anything up.
    const int* m_dev;
};

template <int MAXG>
struct GemmMaps {
    CUtensorMap a[MAXG];    // one per group (copies of one map when the groups share A)
    CUtensorMap b[MAXG];    // one per group
};

// Output staging for TMA stores: per epilogue warp two 4 KB buffers, each a
// 32-row x 128-byte tile in the 128-byte-swizzled layout (1024-byte aligned).
constexpr int kOutBufBytes = 4096;
constexpr int kOutBytesPerWarp = 2 * kOutBufBytes;

template <int BN, int STAGES>
struct GemmSmem {
    static constexpr int kABytes = kBM * kBK * 2;
    static constexpr int kBBytes = BN * kBK * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kOutOffset = STAGES * kStageBytes;
    static constexpr int kBarOffset = kOutOffset + 4 * kOutBytesPerWarp;
    // full[S], empty[S], tmem_full[2], tmem_empty[2], drain[1]
    static constexpr int kNumBars = 2 * STAGES + 5;
    static constexpr int kMiscOffset = kBarOffset + kNumBars * 8;
    static constexpr int kBytes = kMiscOffset + 16 + 1024;  // + alignment slack
};

__device__ __forceinline__ void tile_coords(long long t, const GemmShape& sh, int& g, int& mb,
                                            int& nb) {
    const long long per = static_cast<long long>(sh.m_blocks) * sh.n_blocks;
    g = static_cast<int>(t / per);
    const int local = static_cast<int>(t - static_cast<long long>(g) * per);
    const int per_band = sh.band * sh.n_blocks;
    const int band = local / per_band;
    const int first_m = band * sh.band;
    const int h = min(sh.m_blocks - first_m, sh.band);
    const int r = local - band * per_band;
    mb = first_m + r % h;
    nb = r / h;
}

// Load one operand k-block.  K-major: a single box {64 (K), ROWS}.  MN-major:
// ROWS/64 boxes {64 (M or N), 64 (K)}, each 8 KB, stacked along M/N.
template <bool MN, int ROWS>
__device__ __forceinline__ void load_operand(const CUtensorMap* map, uint32_t dst, uint32_t bar,
                                             int row0, int k0) {
    if constexpr (!MN) {
        tma_load_2d(map, dst, bar, k0, row0);
    } else {
#pragma unroll
        for (int i = 0; i < ROWS / 64; ++i) tma_load_2d(map, dst + i * (64 * kBK * 2), bar, row0 + 64 * i, k0);
    }
}

// Descriptor of the kk-th K=16 slice of an operand k-block.
//  K-major SW128: rows of 128 B (64 K-elements), 8-row groups 1024 B apart
//                 (SBO); the K slice starts 32 B further along the row.
//  MN-major SW128: 64-element MN chunks of 64 K-rows (8 KB, LBO apart), 8-row
//                 K groups 1024 B apart (SBO); the K slice starts 16 rows
//                 (2048 B) further down.
template <bool MN>
__device__ __forceinline__ uint64_t operand_desc(uint32_t base, int kk) {
    if constexpr (!MN)
        return smem_desc_sw128(base + kk * (kUmmaK * 2), 16, 1024);
    else
        return smem_desc_sw128(base + kk * (kUmmaK * 128), 64 * kBK * 2, 1024);
}

// Per-warp output context of the epilogue: the warp's staging buffers and the
// count of TMA stores it issued (which buffer is next).  All decisions that
// touch it are warp-uniform.
struct EpiIO {
    uint32_t out;     // shared address of this warp's two staging buffers
    int lane;
    int row0;         // absolute output row of lane 0 of this warp
    uint32_t count;   // stores issued so far
};

// Next staging buffer, once the store that last used it has read it.
__device__ __forceinline__ uint32_t out_acquire(const EpiIO& io) {
    if (io.lane == 0) bulk_wait_group_read<1>();
    __syncwarp();
    return io.out + (io.count & 1u) * kOutBufBytes;
}

// Each thread writes its 128-byte row r (32 words) of a staging buffer: 16-byte
// piece c goes to position c ^ (r mod 8), the 128-byte swizzle the TMA store
// undoes; 8 consecutive rows hit 8 different bank groups.
__device__ __forceinline__ void out_stage_row(uint32_t buf, int r, const uint32_t (&w)[32]) {
    const uint32_t row = buf + static_cast<uint32_t>(r) * 128u;
#pragma unroll
    for (int c = 0; c < 8; ++c)
        st_shared_v4(row + ((static_cast<uint32_t>(c) ^ (static_cast<uint32_t>(r) & 7u)) << 4),
                     w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
}

// Write 16 words (64 bytes) of row r into half `h` (pieces 4h..4h+3) of a
// staging buffer, same swizzle as out_stage_row.
__device__ __forceinline__ void out_stage_half(uint32_t buf, int r, int h, const uint32_t (&w)[16]) {
    const uint32_t row = buf + static_cast<uint32_t>(r) * 128u;
#pragma unroll
    for (int c = 0; c < 4; ++c)
        st_shared_v4(row + (((static_cast<uint32_t>(4 * h + c)) ^ (static_cast<uint32_t>(r) & 7u)) << 4),
                     w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
}

// Store a filled staging buffer to (x, y) of `map` (rows/columns outside the
// tensor are clipped by the TMA engine).
__device__ __forceinline__ void out_commit(EpiIO& io, const CUtensorMap* map, uint32_t buf, int x,
                                           int y) {
    fence_proxy_async_smem();
    __syncwarp();
    if (io.lane == 0) {
        tma_store_2d(map, buf, x, y);
        bulk_commit_group();
    }
    ++io.count;
}

template <int BN, bool A_MN, bool B_MN, int STAGES, int MAXG, class Epi>
__global__ void __launch_bounds__(kGemmThreads, 1)
    tc_gemm_kernel(const __grid_constant__ GemmMaps<MAXG> maps,
                   const __grid_constant__ typename Epi::Params ep, const GemmShape sh,
                   unsigned int* status, unsigned long long wait_limit_ns) {
    using L = GemmSmem<BN, STAGES>;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kBM, BN, A_MN, B_MN);
    constexpr int kTmemCols = 2 * BN;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    const uint32_t sbase = raw + pad;

    const uint32_t bar0 = sbase + L::kBarOffset;
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + a); };
    auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * STAGES + 2 + a); };
    const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(smem + L::kMiscOffset);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kMiscOffset + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull_bar(a), 1);
            mbar_init(tempty_bar(a), 4);
        }
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&maps.a[0]);
    }
    if (warp == 1) {
        tmem_alloc<kTmemCols>(smem_u32(tmem_holder));
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    const WaitGuard guard{abort_flag, status, wait_limit_ns};

    if (warp == 0) {
        // ------------------------------------------------------- TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0;       // stages with a copy issued
            uint32_t issued_parity = 0;     // parity of that copy's phase
            bool ok = true;
            for (long long t = blockIdx.x; t < sh.tiles && ok; t += gridDim.x) {
                int g, mb, nb;
                tile_coords(t, sh, g, mb, nb);
                const CUtensorMap* amap = &maps.a[MAXG == 1 ? 0 : g];
                const CUtensorMap* bmap = &maps.b[MAXG == 1 ? 0 : g];
                for (int kb = 0; kb < sh.k_blocks; ++kb) {
                    if (!mbar_wait(empty_bar(stage), phase ^ 1u, guard)) { ok = false; break; }
                    const uint32_t sa = sbase + stage * L::kStageBytes;
                    const uint32_t sb = sa + L::kABytes;
                    mbar_arrive_expect_tx(full_bar(stage), L::kStageBytes);
                    load_operand<A_MN, kBM>(amap, sa, full_bar(stage), mb * kBM, kb * kBK);
                    load_operand<B_MN, BN>(bmap, sb, full_bar(stage), nb * BN, kb * kBK);
                    issued_mask |= 1u << stage;
                    issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
            }
            // Do not leave copies landing in shared memory after exit: the last copy of
            // every stage is awaited (at once when it was consumed), also when another
            // role gave up first.
            for (int s = 0; s < STAGES; ++s)
                if (issued_mask & (1u << s))
                    mbar_wait_drain(full_bar(s), (issued_parity >> s) & 1u, kDrainLimitNs);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true, issued_any = false;
            for (long long t = blockIdx.x; t < sh.tiles && ok; t += gridDim.x) {
                if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, guard)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
                for (int kb = 0; kb < sh.k_blocks; ++kb) {
                    if (!mbar_wait(full_bar(stage), phase, guard)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t sa = sbase + stage * L::kStageBytes;
                    const uint32_t sb = sa + L::kABytes;
#pragma unroll
                    for (int kk = 0; kk < kBK / kUmmaK; ++kk) {
                        tc_mma_bf16(d_tmem, operand_desc<A_MN>(sa, kk), operand_desc<B_MN>(sb, kk),
                                    kIdesc, (kb | kk) != 0 ? 1u : 0u);
                    }
                    issued_any = true;
                    tc_commit(empty_bar(stage));
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                tc_commit(tfull_bar(acc));
                if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            }
            if (issued_any) {
                // Wait for the MMAs already issued before TMEM and smem go away (also
                // when only the epilogue gave up).
                tc_commit(drain_bar);
                mbar_wait_drain(drain_bar, 0, kDrainLimitNs);
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------- epilogue
        const int q = warp & 3;  // TMEM lane quarter this warp may access
        const int r_in_tile = q * 32 + lane;
        EpiIO io{sbase + L::kOutOffset + static_cast<uint32_t>((warp - 2) * kOutBytesPerWarp), lane,
                 0, 0u};
        int acc = 0;
        uint32_t acc_phase = 0;
        for (long long t = blockIdx.x; t < sh.tiles; t += gridDim.x) {
            int g, mb, nb;
            tile_coords(t, sh, g, mb, nb);
            if (!mbar_wait(tfull_bar(acc), acc_phase, guard)) break;
            tc_fence_after();
            const int row = mb * kBM + r_in_tile;
            const int n0 = nb * BN;
            io.row0 = mb * kBM + q * 32;
            Epi epi(ep, g, row, n0);
            const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                   static_cast<uint32_t>(acc * BN);
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                float v[32];
                tmem_ld_32x32b_x32(t_row + c * 32, v);
                epi.chunk(ep, v, n0 + c * 32, c * 32, io);
            }
            epi.finish(ep, nb);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty_bar(acc));
            if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
        }
        if (lane == 0) bulk_wait_group_all();  // stores done before shared memory goes away
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc<kTmemCols>(tmem_base);
    }
}

}  // namespace fpo
