// tc_gemm_pair.cuh -- CTA-pair variant of the persistent tcgen05 GEMM.
//
// A cluster of two CTAs (on two SMs) computes one 256 x BN output tile with
// tcgen05.mma.cta_group::2: CTA r holds rows [128 r, 128 r + 128) of the A
// tile and columns [BN/2 r, BN/2 (r + 1)) of the B tile in its own shared
// memory, and its TMEM receives output rows [128 r, 128 r + 128).  Per SM a
// 64-deep k-block is A 16 KB + B 16 KB (instead of A 16 KB + B 32 KB), so each
// SM streams a third less operand data per FLOP.
//
// A pipeline stage of the 256-column tiles holds two consecutive 64-deep k-blocks
// (64 KB per CTA, three stages), each with its own full barrier, and is freed by one
// commit: the MMA thread issues eight N = 256 MMAs (1024 tensor cycles) per commit and
// starts the first four as soon as the stage's first half has landed.  Measured with
// clock counters in the MMA thread, one wait + fence + four MMAs + commit per 32 KB
// stage took ~550 cycles for 512 cycles of tensor work, at the same rate with the
// operands loaded only once per launch: the issuing thread, not the operand supply,
// set the pace.  With eight MMAs per commit the loop keeps pace with the tensor pipe
// (512 cycles per k-block without copies).  The 512-column tiles issue eight MMAs per
// 64-deep k-block already and keep one k-block (48 KB) per stage.  Six k-blocks in
// flight is the depth that measured best in the power-capped step: four cost about a
// quarter of the per-clock rate, six one-k-block stages (a commit per four MMAs) 3-7%,
// and a seventh k-block (a ring of seven 32 KB slots committed in pairs) raised the
// per-clock rates 1-2% but lowered the clock more.
//
//   both CTAs, warp 0   TMA loads of the CTA's halves; completion is counted
//                       on the LEADER's (rank 0) full barrier
//   leader, warp 1      issues the pair MMAs and commits to the empty /
//                       accumulator-ready barriers of BOTH CTAs (multicast)
//   both CTAs, warps 2-5  epilogue on the CTA's 128 rows; arrive on the
//                       leader's accumulator-empty barrier (8 arrivals)
// TMEM (512 columns) is allocated collectively by warp 1 of both CTAs.
//
// BN is 256 (two accumulator buffers of 256 columns: the epilogue of one tile
// overlaps the mainloop of the next) or 512 (two N=256 MMAs per K slice into
// one 512-column accumulator: a quarter less operand traffic per FLOP, but the
// next tile waits for the epilogue; for GEMMs with a long K loop).
// All waits are bounded as in the single-CTA kernel.  Teardown: the pair meets at
// a cluster barrier, the leader waits (with a separate, fixed limit) for every
// operand copy either CTA issued into the last ring positions, which its full
// barriers count, and the pair meets again before TMEM is freed and before either
// CTA exits (pair_drain_copies below).
#pragma once

#include "tc_gemm.cuh"

namespace fpo {

constexpr int kPairBM = 256;  // output rows of one pair tile

// 64-deep k-blocks per pipeline stage of a BN-column pair tile.
template <int BN, bool A_MN, bool B_MN>
constexpr int pair_ksub() {
    return BN == 256 ? 2 : 1;
}

template <int BN, int STAGES, int KSUB>
struct GemmPairSmem {
    static constexpr int kSub = KSUB;
    static constexpr int kABytes = 128 * kBK * 2;         // one 64-deep k-block of A
    static constexpr int kBBytes = (BN / 2) * kBK * 2;    // one 64-deep k-block of B
    static constexpr int kStageBytes = kSub * (kABytes + kBBytes);  // A blocks, then B blocks
    static constexpr int kOutOffset = STAGES * kStageBytes;
    static constexpr int kBarOffset = kOutOffset + 4 * kOutBytesPerWarp;
    static constexpr int kNumBars = STAGES * KSUB + STAGES + 5;
    static constexpr int kMiscOffset = kBarOffset + kNumBars * 8;
    static constexpr int kBytes = kMiscOffset + 16 + 1024;
};

// Misc words of the pair kernel's shared memory: TMEM base address, abort flag,
// and the number of k-blocks this CTA's producer issued.
constexpr int kMiscTmem = 0, kMiscAbort = 4, kMiscIssued = 8;

__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// mbar_wait with cluster-scope acquire (the barriers of the pair kernel are
// arrived on by the other CTA too).
__device__ __forceinline__ bool mbar_wait_cl(uint32_t bar, uint32_t parity, const WaitGuard& g) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait_cluster(bar, parity)) return true;
        if (*g.abort_flag) return false;
        if (global_timer_ns() - t0 > g.limit_ns) {
            *g.abort_flag = 1;
            if (g.status) atomicOr(g.status, kDevTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ bool mbar_test_wait_cluster(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// mbar_wait_cl for the MMA thread's stage waits: it polls with test_wait, which never
// suspends the thread, so the next MMAs issue as soon as the stage lands (measured: the
// layer update 1% faster than with try_wait, the other GEMMs unchanged).  The limit and
// the abort flag are checked every 32 polls.
__device__ __forceinline__ bool mbar_wait_cl_poll(uint32_t bar, uint32_t parity, const WaitGuard& g) {
    if (mbar_test_wait_cluster(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_test_wait_cluster(bar, parity)) return true;
        if ((i & 31u) == 0) {
            if (*g.abort_flag) return false;
            if (global_timer_ns() - t0 > g.limit_ns) {
                *g.abort_flag = 1;
                if (g.status) atomicOr(g.status, kDevTimeout);
                return false;
            }
        }
    }
}

__device__ __forceinline__ bool mbar_wait_cl_drain(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait_cluster(bar, parity))
        if (global_timer_ns() - t0 > limit_ns) return false;
    return true;
}

// The work of one pair cluster as a sequence of segments (tile, k-blocks [kb0, kb1)).
// Tiles [0, tiles - tail_tiles) are whole and dealt round robin (cluster c takes c,
// c + C, ...: concurrent tiles are neighbours in the rasterisation and stream the same
// k-blocks, sharing operands in L2).  The tail_tiles = R tiles of the last, partial
// wave are each split into S = tail_split equal k-block ranges; the R S units, ordered
// by range then tile (so concurrent units stream the same k-blocks), are dealt round
// robin too, and unit u leaves its sums in slot u.  part = -1 marks a whole tile.
// Every role of every CTA walks the same sequence.
struct SegCursor {
    long long C, t, u;

    __device__ __forceinline__ SegCursor(const GemmShape&, long long c, long long C_)
        : C(C_), t(c), u(c) {}

    __device__ __forceinline__ bool next(const GemmShape& sh, long long& tile, int& kb0, int& kb1,
                                         int& part, int& slot) {
        const long long dp = sh.tiles - sh.tail_tiles;
        if (t < dp) {
            tile = t;
            kb0 = 0;
            kb1 = sh.k_blocks;
            part = -1;
            slot = -1;
            t += C;
            return true;
        }
        const long long R = sh.tail_tiles, S = sh.tail_split;
        if (u >= R * S) return false;
        const long long q = u / R;
        tile = dp + (u - q * R);
        kb0 = static_cast<int>((q * sh.k_blocks) / S);
        kb1 = static_cast<int>(((q + 1) * sh.k_blocks) / S);
        part = static_cast<int>(q);
        slot = static_cast<int>(u);
        u += C;
        return true;
    }
};

// One CTA's half of an operand k-block, counted on the leader's barrier.
template <bool MN, int ROWS>
__device__ __forceinline__ void load_operand_pair(const CUtensorMap* map, uint32_t dst,
                                                  uint32_t bar_leader, int row0, int k0) {
    if constexpr (!MN) {
        tma_load_2d_pair(map, dst, bar_leader, k0, row0);
    } else {
#pragma unroll
        for (int i = 0; i < ROWS / 64; ++i)
            tma_load_2d_pair(map, dst + i * (64 * kBK * 2), bar_leader, row0 + 64 * i, k0);
    }
}

// Teardown of the pair (leader's producer thread, after both producers have stopped
// and published their issued stage counts n_self and n_peer): every copy either CTA
// issued must have landed before the CTAs exit.  The stage with index i sits in ring
// slot i % STAGES, phase parity (i / STAGES) & 1; each of its KSUB 64-deep k-blocks has
// a leader full barrier that counts both CTAs' halves (2 x half_bytes, armed by the
// leader's expect_tx), and a producer issues all KSUB k-blocks of a stage together.
// Every stage below max(n_self, n_peer) - STAGES was consumed by MMAs, so all its
// copies landed; for the last STAGES indices each barrier is still in that stage's
// phase (or completed it), and the side that did not issue the stage is accounted for
// here: a missing peer half by completing its bytes, a missing leader expect_tx by
// arming the barrier for the peer's half only.  Each such phase is then awaited with
// the fixed drain limit.
template <int STAGES, int KSUB>
__device__ __forceinline__ void pair_drain_copies(uint32_t bar0, long long n_self, long long n_peer,
                                                  uint32_t half_bytes) {
    const long long hi = n_self > n_peer ? n_self : n_peer;
    for (long long i = hi - STAGES > 0 ? hi - STAGES : 0; i < hi; ++i) {
        const uint32_t parity = static_cast<uint32_t>((i / STAGES) & 1);
        const bool mine = i < n_self, peer = i < n_peer;
        for (int j = 0; j < KSUB; ++j) {
            const uint32_t bar = bar0 + 8u * static_cast<uint32_t>((i % STAGES) * KSUB + j);
            if (mine && !peer) mbar_complete_tx(bar, half_bytes);
            if (!mine && peer) mbar_arrive_expect_tx(bar, half_bytes);
            mbar_wait_cl_drain(bar, parity, kDrainLimitNs);
        }
    }
}

template <int BN, bool A_MN, bool B_MN, int STAGES, int MAXG, class Epi>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    tc_gemm_pair_kernel(const __grid_constant__ GemmMaps<MAXG> maps,
                        const __grid_constant__ typename Epi::Params ep, const GemmShape sh_in,
                        unsigned int* status, unsigned long long wait_limit_ns) {
    static_assert(BN == 256 || BN == 512, "pair tiles are 256 or 512 columns wide");
    using L = GemmPairSmem<BN, STAGES, pair_ksub<BN, A_MN, B_MN>()>;
    constexpr int kSub = L::kSub;                  // 64-deep k-blocks per stage
    constexpr int kNSub = BN / 256;                // N = 256 MMAs per K slice
    constexpr int kAccBufs = kNSub == 1 ? 2 : 1;   // accumulator buffers in TMEM
    constexpr int kBSub = 128;                     // B columns per CTA per N = 256 MMA
    constexpr uint32_t kBSubBytes = kBSub * kBK * 2;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kPairBM, 256, A_MN, B_MN);
    constexpr int kTmemCols = kAccBufs * BN;       // 512 either way
    constexpr uint16_t kBoth = 0x3;                // both CTAs of the pair

    GemmShape sh = sh_in;
    // from here on a "k-block" is one stage: kSub 64-deep k-blocks (the last one may
    // reach past K; its loads read zeros there)
    sh.k_blocks = (sh.k_blocks + kSub - 1) / kSub;
    if (sh.m_dev) {  // rows counted on the device (every thread reads the same value)
        const int m = min(*sh.m_dev, sh.M);
        if (m <= 0) return;
        sh.M = m;
        sh.m_blocks = (m + kPairBM - 1) / kPairBM;
        sh.tiles = static_cast<long long>(sh.groups) * sh.m_blocks * sh.n_blocks;
        sh.tail_tiles = 0;
    }

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    const uint32_t sbase = raw + pad;

    const uint32_t rank = cluster_ctarank();  // position in the CTA pair
    const bool leader = rank == 0;            // the leader issues the pair's MMAs
    const long long cluster = blockIdx.x / 2;
    const long long n_clusters = gridDim.x / 2;

    const uint32_t bar0 = sbase + L::kBarOffset;
    constexpr int kFull = STAGES * kSub;  // one full barrier per 64-deep k-block
    auto full_bar = [&](int s, int j) { return bar0 + 8u * (s * kSub + j); };
    auto empty_bar = [&](int s) { return bar0 + 8u * (kFull + s); };
    auto tfull_bar = [&](int a) { return bar0 + 8u * (kFull + STAGES + a); };
    auto tempty_bar = [&](int a) { return bar0 + 8u * (kFull + STAGES + 2 + a); };
    const uint32_t drain_bar = bar0 + 8u * (kFull + STAGES + 4);
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(smem + L::kMiscOffset + kMiscTmem);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kMiscOffset + kMiscAbort);
    uint32_t* issued_word = reinterpret_cast<uint32_t*>(smem + L::kMiscOffset + kMiscIssued);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            for (int j = 0; j < kSub; ++j)
                mbar_init(full_bar(s, j), 1);  // leader's: one expect_tx arrival, both CTAs' bytes
            mbar_init(empty_bar(s), 1);  // one multicast commit from the leader
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull_bar(a), 1);
            mbar_init(tempty_bar(a), 8);  // leader's: 4 epilogue warps x 2 CTAs
        }
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        *issued_word = 0;
        fence_mbar_init();
        tma_prefetch_desc(&maps.a[0]);
    }
    if (warp == 1) {
        tmem_alloc_pair<kTmemCols>(smem_u32(tmem_holder));
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // barrier initialisation and TMEM allocation visible to the pair
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    const WaitGuard guard{abort_flag, status, wait_limit_ns};

    if (warp == 0) {
        // ------------------------------------------------------- TMA producer (both CTAs)
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued = 0;  // k-blocks issued: k-block i used stage i % STAGES
            bool ok = true;
            SegCursor seg(sh, cluster, n_clusters);
            long long t;
            int kb0, kb1, part, slot;
            while (ok && seg.next(sh, t, kb0, kb1, part, slot)) {
                int g, mp, nb;
                tile_coords(t, sh, g, mp, nb);
                const CUtensorMap* amap = &maps.a[MAXG == 1 ? 0 : g];
                const CUtensorMap* bmap = &maps.b[MAXG == 1 ? 0 : g];
                const int a_row = mp * kPairBM + 128 * static_cast<int>(rank);
                const int b_row = nb * BN + kBSub * static_cast<int>(rank);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait_cl(empty_bar(stage), phase ^ 1u, guard)) { ok = false; break; }
                    const uint32_t sa = sbase + stage * L::kStageBytes;
                    const uint32_t sb = sa + kSub * L::kABytes;
#pragma unroll
                    for (int j = 0; j < kSub; ++j) {
                        const uint32_t fb = mapa_shared(full_bar(stage, j), 0);
                        if (leader)
                            mbar_arrive_expect_tx(full_bar(stage, j), 2 * (L::kStageBytes / kSub));
                        const int k0 = (kb * kSub + j) * kBK;
                        load_operand_pair<A_MN, 128>(amap, sa + j * L::kABytes, fb, a_row, k0);
#pragma unroll
                        for (int h = 0; h < kNSub; ++h)
                            load_operand_pair<B_MN, kBSub>(
                                bmap, sb + j * L::kBBytes + h * kBSubBytes, fb, b_row + 256 * h, k0);
                    }
                    ++issued;
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
            }
            *issued_word = issued;  // read by the leader at teardown
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------- pair MMA (leader only)
        if (leader && lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true, issued_any = false;
            SegCursor seg(sh, cluster, n_clusters);
            long long t;
            int kb0, kb1, part, slot;
            while (ok && seg.next(sh, t, kb0, kb1, part, slot)) {
                if (!mbar_wait_cl(tempty_bar(acc), acc_phase ^ 1u, guard)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    const uint32_t sa = sbase + stage * L::kStageBytes;
                    const uint32_t sb = sa + kSub * L::kABytes;
#pragma unroll
                    for (int j = 0; j < kSub; ++j) {
                        if (!mbar_wait_cl_poll(full_bar(stage, j), phase, guard)) { ok = false; break; }
                        tc_fence_after();
#pragma unroll
                        for (int kk = 0; kk < kBK / kUmmaK; ++kk)
#pragma unroll
                            for (int h = 0; h < kNSub; ++h)
                                tc_mma_bf16_pair(
                                    d_tmem + 256u * h, operand_desc<A_MN>(sa + j * L::kABytes, kk),
                                    operand_desc<B_MN>(sb + j * L::kBBytes + h * kBSubBytes, kk),
                                    kIdesc, (kb != kb0 || j != 0 || kk != 0) ? 1u : 0u);
                        issued_any = true;
                    }
                    if (!ok) break;
                    // the stage is free in both CTAs once the MMAs reading it completed
                    tc_commit_pair_multicast(empty_bar(stage), kBoth);
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                tc_commit_pair_multicast(tfull_bar(acc), kBoth);
                if (++acc == kAccBufs) { acc = 0; acc_phase ^= 1u; }
            }
            if (issued_any) {
                // every MMA issued, which reads both CTAs' stages and writes their TMEM,
                // completes before teardown (also when only the epilogue gave up)
                tc_commit_pair_multicast(drain_bar, 0x1);
                mbar_wait_cl_drain(drain_bar, 0, kDrainLimitNs);
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------- epilogue (both CTAs)
        const int q = warp & 3;
        const int r_in_tile = 128 * static_cast<int>(rank) + q * 32 + lane;
        EpiIO io{sbase + L::kOutOffset + static_cast<uint32_t>((warp - 2) * kOutBytesPerWarp), lane,
                 0, 0u};
        int acc = 0;
        uint32_t acc_phase = 0;
        SegCursor seg(sh, cluster, n_clusters);
        long long t;
        int kb0, kb1, part, slot;
        while (seg.next(sh, t, kb0, kb1, part, slot)) {
            int g, mp, nb;
            tile_coords(t, sh, g, mp, nb);
            if (!mbar_wait_cl(tfull_bar(acc), acc_phase, guard)) break;
            tc_fence_after();
            const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                   static_cast<uint32_t>(acc * BN);
            if (part < 0) {
                const int tile_row0 = mp * kPairBM;
                const int row = tile_row0 + r_in_tile;
                const int n0 = nb * BN;
                io.row0 = tile_row0 + 128 * static_cast<int>(rank) + q * 32;
                Epi epi(ep, g, row, n0);
#pragma unroll 1
                for (int c = 0; c < BN / 32; ++c) {
                    float v[32];
                    tmem_ld_32x32b_x32(t_row + c * 32, v);
                    epi.chunk(ep, v, n0 + c * 32, c * 32, io);
                }
                epi.finish(ep, nb);
            } else {
                // one k range of a split tile: its raw fp32 sums, row r_in_tile, to its slot
                float* dst = sh.sk_scratch + (static_cast<size_t>(slot) * kPairBM + r_in_tile) * BN;
#pragma unroll 1
                for (int c = 0; c < BN / 32; ++c) {
                    float v[32];
                    tmem_ld_32x32b_x32(t_row + c * 32, v);
                    float4* d4 = reinterpret_cast<float4*>(dst + c * 32);
#pragma unroll
                    for (int q4 = 0; q4 < 8; ++q4)
                        d4[q4] = make_float4(v[4 * q4], v[4 * q4 + 1], v[4 * q4 + 2], v[4 * q4 + 3]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (leader)
                    mbar_arrive(tempty_bar(acc));
                else
                    mbar_arrive_cluster(mapa_shared(tempty_bar(acc), 0));
            }
            if (++acc == kAccBufs) { acc = 0; acc_phase ^= 1u; }
        }
        if (lane == 0) bulk_wait_group_all();
        __syncwarp();
    }

    // Teardown.  Every role has stopped; both producers have published their issued
    // k-block counts.  After the first pair barrier the leader waits for each copy of
    // either CTA that no MMA consumed (pair_drain_copies: a no-op wait on completed
    // phases when nothing gave up); the second barrier keeps both CTAs, and their
    // shared memory and TMEM, alive until then.
    tc_fence_before();
    __syncthreads();
    cluster_sync();
    if (leader && threadIdx.x == 0)
        pair_drain_copies<STAGES, kSub>(bar0, *issued_word,
                                        ld_shared_cluster_u32(mapa_shared(smem_u32(issued_word), 1)),
                                        L::kStageBytes / kSub);
    __syncthreads();
    cluster_sync();  // no CTA frees TMEM or exits while another may still touch it
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair<kTmemCols>(tmem_base);
    }
}

}  // namespace fpo
