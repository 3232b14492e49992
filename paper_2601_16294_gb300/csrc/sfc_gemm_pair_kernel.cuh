// sfc_gemm_pair_kernel.cuh -- the SFC / SFC-CA GEMM on 2-SM CTA pairs.
//
// Same task space, item order, accumulation chunks and epilogue as
// sfc_gemm_kernel, but each worker is a cluster of two CTAs on two SMs that
// computes a 256 x BN output tile with tcgen05.mma.cta_group::2 (UMMA M = 256):
//
//   - CTA r of the pair loads rows [128 r, 128 r + 128) of the A slab and
//     columns [r BN/2, (r+1) BN/2) of the B slab into its own shared memory;
//     both CTAs' TMA copies complete on the leader CTA's "full" barrier;
//   - the leader's MMA warp issues the pair MMAs.  Each SM's tensor core uses
//     its own A half and both B halves, so a 256 x BN tile costs each SM
//     128 x 64 + 64 x BN/2 bf16 of shared-memory and L2 traffic per slab,
//     against 128 x 64 + 64 x BN for a 128 x BN tile on one SM;
//   - MMA completion (tcgen05.commit ... multicast) frees the ring stage in
//     both CTAs and publishes the accumulator chunk to both epilogues;
//   - CTA r's tensor memory holds rows [128 r, 128 r + 128) of the tile; its
//     epilogue warps drain them and arrive on the leader's accumulator-empty
//     barrier.
//
// Every TMA load writes the shared memory of the CTA that issues it (no
// multicast loads); only the MMA completion signals (tcgen05.commit) are
// multicast, as mbarrier arrivals within the pair.
//
// Waits are bounded as in the single-SM kernel.  The pair meets at a cluster
// barrier after set-up (barriers initialised before any remote signal) and
// before exit (no CTA leaves while its peer may still signal it); then both
// CTAs free their tensor memory.
#pragma once

#include "sfc_gemm_kernel.cuh"

namespace sfc {

constexpr int kPairBM = 256;  // output tile rows of a pair (128 per CTA)

template <int BN>
struct PairStage {
    static constexpr int kHalfN = BN / 2;
    static constexpr int kABytes = 128 * 128;     // 128 rows of 128 bytes
    static constexpr int kBBytes = kHalfN * 128;  // this CTA's half of the B slab
    static constexpr int kBytes = kABytes + kBBytes;
    static_assert(kABytes % 1024 == 0 && kBBytes % 1024 == 0, "swizzle atoms need 1 KB alignment");
};

template <int BN, int STAGES, typename OutT, bool F8>
__global__ void __launch_bounds__(block_threads(BN), 1)
sfc_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                     const __grid_constant__ CUtensorMap tmap_c, const GemmParams p) {
    static_assert(BN == 128 || BN == 256, "pair tiles are 256 x 128 or 256 x 256");
    using I = InKind<F8>;
    using S = PairStage<BN>;
    constexpr int kEpiWarps = BN / 32;
    using L = RingLayout<S::kBytes, STAGES, kEpiWarps>;
    constexpr int kHalfN = S::kHalfN;

    constexpr uint32_t kTmemCols = 2 * BN;
    constexpr int kCtas = 2;
    constexpr int kItemRows = kPairBM;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);
    const uint32_t ring = base;
    const Barriers B{base + L::kBarOffset, STAGES};
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kMiscOffset);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kMiscOffset + 4);

    const int warp = threadIdx.x / 32;
    const int lane = threadIdx.x % 32;
    const uint32_t rank = ptx::cluster_ctarank();
    const uint32_t r = rank;                    // position in the pair
    const uint32_t pair_leader = 0;             // the pair's MMA-issuing CTA
    const bool leader = (r == 0);
    const uint16_t pair_mask = 0x3;             // both CTAs of the pair
    ItemSource src;
    worker_items(p, blockIdx.x / kCtas, gridDim.x / kCtas, src.first, src.end, src.step);
    src.worker = blockIdx.x / kCtas;
    src.workers = gridDim.x / kCtas;
    src.dynamic = p.dynamic;
    src.q_full0 = B.q_full(0);
    src.q_empty0 = ptx::map_to_cta(B.q_empty(0), 0);
    src.q_entry = reinterpret_cast<volatile int*>(smem + L::kQueueOffset);
    // CTA 0's scheduler deals the cluster's items.  The first needs no memory
    // at all and no message: the scheduler warp of each CTA decodes it into its
    // own queue's slot 0 while the other warps set up.
    const bool sched_thread = (rank == 0 && warp == scheduler_warp(BN) && lane == 0);
    int item0 = -1;
    if (warp == scheduler_warp(BN) && lane == 0) {
        item0 = sched_next(src, 0, p);
        sched_local_first(src, sched_entry(item0, p));
    }

    if (threadIdx.x == 0) {
        ptx::pdl_launch_dependents();
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(B.full(s), 1);   // the pair leader's producer arrives once (+ tx bytes)
            ptx::mbar_init(B.empty(s), 1);  // one multicast commit of the pair's MMAs
        }
        for (int a = 0; a < 2; ++a) {
            ptx::mbar_init(B.acc_full(a), 1);               // one multicast commit per chunk
            ptx::mbar_init(B.acc_empty(a), 2 * kEpiWarps);  // epilogue warps of the pair (leader's copy used)
        }
        ptx::mbar_init(B.drain(), 1);
        ptx::mbar_init(B.never(), 1);
        for (int q = 0; q < kQueue; ++q) {
            ptx::mbar_init(B.q_full(q), 1);  // the cluster's scheduler (in CTA 0) publishes
            // (CTA 0's copy is used) every consuming role of the pair has read: both producers,
            // the leader's MMA warp and all epilogue warps
            ptx::mbar_init(B.q_empty(q), kCtas + 1 + kCtas * kEpiWarps);
        }
        ptx::mbar_init(B.q_taken(), 1);  // CTA 0's producer took an item (CTA 0's copy is used)
        *abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        ptx::tma_prefetch_desc(&tmap_a);
        ptx::tma_prefetch_desc(&tmap_b);
        if (p.tma_store) ptx::tma_prefetch_desc(&tmap_c);
    }
    if (warp == 1) {
        ptx::tmem_alloc_pair(ptx::smem_addr(tmem_slot), kTmemCols);
        ptx::tmem_relinquish_pair();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // every CTA's barriers are initialised before anyone signals them
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (sched_thread) sched_mark_first(src, kCtas);
    ptx::pdl_wait();  // on-chip set-up above overlaps the previous kernel; global memory only after it

    if (warp == 0) {
        // ----------------------------------------------- TMA producer (every CTA)
        if (lane == 0) {
            int64_t issued = 0;
            bool ok = produce<STAGES>(src, p, B, abort_flag, /*signal_taken=*/rank == 0, issued,
                                      [&](const WorkItem& w, int kt, int stage) {
                const int32_t a_row = w.tm * kItemRows + static_cast<int32_t>(r * 128);
                const int32_t b_col = w.tn * BN + static_cast<int32_t>(r) * kHalfN;
                if (leader) ptx::mbar_arrive_expect_tx(B.full(stage), 2 * S::kBytes);
                const uint32_t leader_full = ptx::map_to_cta(B.full(stage), pair_leader);
                const uint32_t sa = ring + stage * S::kBytes;
                const uint32_t sb = sa + S::kABytes;
                ptx::tma_load_2d_pair(sa, &tmap_a, leader_full, kt * I::kSlabK, a_row);
                if (p.b_kmajor) {
                    // this CTA's half of the B^T rows (N) x one slab of k, K-major like A
                    ptx::tma_load_2d_pair(sb, &tmap_b, leader_full, kt * I::kSlabK, b_col);
                } else {
                    // N-major boxes of 128-byte rows (the host keeps 8-bit inputs with BN/2 >= 128 here)
#pragma unroll
                    for (int jb = 0; jb < kHalfN / I::kBCols; ++jb)
                        ptx::tma_load_2d_pair(sb + jb * I::kBBoxBytes, &tmap_b, leader_full, b_col + jb * I::kBCols,
                                              kt * I::kSlabK);
                }
            });
            // Tail: on success wait until the last STAGES issues are released
            // (no commit may land after exit).  After a failure a pair leader waits
            // (bounded) on its full barriers, which count all its pair's bytes;
            // the other CTA cannot observe them and waits a fixed 2 ms, far beyond
            // the latency of a tile load.
            const int64_t n0 = issued > STAGES ? issued - STAGES : 0;
            for (int64_t n = n0; n < issued && ok; ++n)
                ok = wait_bounded(B.empty(static_cast<int>(n % STAGES)), static_cast<uint32_t>((n / STAGES) & 1),
                                  abort_flag, p.timeout_ns, kWaitProducerEmpty);
            if (!ok) {
                if (leader) {
                    for (int64_t n = n0; n < issued; ++n)
                        wait_bounded(B.full(static_cast<int>(n % STAGES)), static_cast<uint32_t>((n / STAGES) & 1),
                                     abort_flag, p.timeout_ns, kWaitDrain, /*honour_abort=*/false);
                } else {
                    const uint64_t t0 = ptx::global_timer_ns();
                    while (ptx::global_timer_ns() - t0 < 2000000ull) {
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------ MMA issuer (each pair's leader)
        if (lane == 0 && leader) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            const bool bk = p.b_kmajor != 0;
            const uint32_t idesc = ptx::idesc_f32(kPairBM, BN, /*A K-major*/ 0, bk ? 0u : 1u, p.ab_fmt);
            if (p.debug_never) ok = wait_bounded(B.never(), 0, abort_flag, p.timeout_ns, kWaitDebugNever);
            for (int j = 0; ok; ++j) {
                WorkItem w;
                const int64_t it = src_take<true>(src, j, p, abort_flag, w);
                if (it < 0) {
                    ok = (it == -1);
                    break;
                }
                const int nch = num_chunks(w, p.kc);
                ChunkWalk cw(w, nch);
                for (int ck = 0; ok && ck < nch; ++ck) {
                    const int kb = cw.begin, ke = cw.next();
                    if (!wait_bounded(B.acc_empty(acc), acc_phase ^ 1u, abort_flag, p.timeout_ns, kWaitMmaAccEmpty)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
                    for (int q = kb; q < ke; ++q) {
                        if (!wait_bounded(B.full(stage), phase, abort_flag, p.timeout_ns, kWaitMmaFull)) {
                            ok = false;
                            break;
                        }
                        ptx::tc_fence_after();
                        const uint32_t sa = ring + stage * S::kBytes;
                        const uint32_t sb = sa + S::kABytes;
                        // A half: K-major, 128-byte rows, 8-row atoms 1 KB apart; 32 B per instruction.
                        // B half N-major: 128-byte-wide boxes one box apart, kMmaK rows per
                        // instruction; K-major: as A.  Later instructions step the start-address
                        // field (16-byte units, bits 0-13; the ring lies below 256 KB: no carry).
                        const uint64_t adesc = ptx::smem_desc_sw128(sa, 16, 1024);
                        const uint64_t bdesc = bk ? ptx::smem_desc_sw128(sb, 16, 1024)
                                                  : ptx::smem_desc_sw128(sb, I::kBBoxBytes, 1024);
                        const uint32_t bstep = bk ? 2u : (I::kMmaK * 128) / 16;
#pragma unroll
                        for (int kk = 0; kk < I::kSlabK / I::kMmaK; ++kk)
                            ptx::tc_mma_pair<F8>(d_tmem, adesc + 2u * kk, bdesc + bstep * kk, idesc,
                                                 (q > kb || kk > 0) ? 1u : 0u);
                        // the stage is free in both CTAs once these MMAs have read it
                        ptx::tc_commit_pair_multicast(B.empty(stage), pair_mask);
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (!ok) break;
                    ptx::tc_commit_pair_multicast(B.acc_full(acc), pair_mask);
                    if (++acc == 2) {
                        acc = 0;
                        acc_phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                ptx::tc_commit_pair(B.drain());
                wait_bounded(B.drain(), 0, abort_flag, p.timeout_ns, kWaitDrain, /*honour_abort=*/false);
            }
        }
    } else if (warp < scheduler_warp(BN)) {
        run_epilogue<BN, OutT, true>(p, B, tmem_base, abort_flag, src, kItemRows,
                                     static_cast<int>(r * 128), warp, lane, &tmap_c,
                                     smem + L::kStagingOffset, pair_leader);
    } else if (sched_thread) {
        // -------------------------------------------------------- scheduler
        run_scheduler(src, item0, p, B, abort_flag, kCtas);
    }

    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // no CTA leaves while another CTA of the cluster may still signal it
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc_pair(tmem_base, kTmemCols);
}

}  // namespace sfc
