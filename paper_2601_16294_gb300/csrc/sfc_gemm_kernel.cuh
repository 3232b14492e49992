// sfc_gemm_kernel.cuh -- persistent SFC / SFC-CA GEMM kernel for sm_103a.
//
// One thread block per SM walks its share of the task space of Listing 1
// (Mt*Nt*K_layers items: item i -> K layer i / (Mt*Nt), curve position
// i % (Mt*Nt) -> output tile).  For each item it contracts the layer's K range
// of one 128 x BN output tile (the paper's batch-reduce GEMM over K blocks,
// Sec. II-A; C is zeroed at the first K block, Listing 1) on the tcgen05
// tensor cores:
//
//   warp 0      TMA producer: loads 128x64 A and 64xBN B slabs (bf16, 128-byte
//               swizzle) into a STAGES-deep shared-memory ring, completion on
//               the stage's "full" mbarrier;
//   warp 1      MMA issuer: 4 x tcgen05.mma (128 x BN x 16) per slab into one
//               of two tensor-memory accumulators; tcgen05.commit frees the
//               ring stage and, after the last slab, publishes the accumulator;
//   warps 2..5  epilogue: tcgen05.ld the accumulator (warp w reads TMEM lanes
//               32*(w%4)...), convert, store the tile (masked at the M/N edges),
//               then hand the accumulator back.  Two accumulators let the
//               epilogue of one tile overlap the main loop of the next.
//
// With K_layers > 1 the epilogue writes the layer's fp32 partial tile to the
// workspace copy of C for that layer; ca_reduce_kernel sums the copies.
//
// Every mbarrier wait is bounded (globaltimer).  A wait that runs out sets the
// device error word and a block-wide abort flag; all roles then leave their
// loops, the producer waits (bounded) for its in-flight TMA copies, the MMA
// warp for its in-flight MMAs, and tensor memory is freed before returning.
#pragma once

#include <cuda_bf16.h>
#include <cstdint>

#include "ptx.cuh"
#include "sfc_curve.cuh"

namespace sfc {

constexpr int kBM = 128;            // output tile rows (UMMA M)
constexpr int kBK = 64;             // K slab: 64 bf16 = one 128-byte swizzle row
constexpr int kUmmaK = 16;          // K per tcgen05.mma for 16-bit inputs
constexpr int kThreads = 192;       // 6 warps
constexpr int kBBox = 64;           // B is loaded in 64-column boxes (128 bytes)

// device error word: bit 0 = a bounded wait gave up; bits 8.. = which wait
__device__ unsigned int g_sfc_status = 0;

enum WaitSite : unsigned int {
    kWaitProducerEmpty = 1u << 8,
    kWaitMmaFull = 1u << 9,
    kWaitMmaAccEmpty = 1u << 10,
    kWaitEpiAccFull = 1u << 11,
    kWaitDebugNever = 1u << 12,
    kWaitDrain = 1u << 13,
};

struct GemmParams {
    int64_t M, N;
    int Mt, Nt, Kt;
    int ca_c;
    int64_t num_items;     // Mt * Nt * ca_c
    void* out;             // C when ca_c == 1, else the fp32 workspace
    int64_t ldo;           // row stride of `out` in elements
    int64_t layer_stride;  // elements between K-layer copies in `out`
    int order;             // 0 = generalized Hilbert, 1 = raster
    int assign;            // 0 = contiguous segments, 1 = strided waves
    int vec_store;         // 1 if 16-byte vector stores are aligned
    int debug_never;       // test hook: MMA warp waits on a barrier nobody arrives at
    uint64_t timeout_ns;   // bound for every mbarrier wait
};

template <int BN, int STAGES>
struct SmemLayout {
    static constexpr int kABytes = kBM * kBK * 2;
    static constexpr int kBBytes = BN * kBK * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kRingBytes = kStageBytes * STAGES;
    static constexpr int kNumBars = 2 * STAGES + 6;  // full, empty, acc full x2, acc empty x2, drain, never
    static constexpr int kBarOffset = kRingBytes;
    static constexpr int kMiscOffset = kBarOffset + kNumBars * 8;
    static constexpr int kBytes = kMiscOffset + 16;
    static constexpr int kDynamicBytes = kBytes + 1024;  // slack to align the ring to 1024 B
    static_assert(kABytes % 1024 == 0 && kBBytes % 1024 == 0, "swizzle atoms need 1 KB alignment");
};

struct WorkItem {
    int tm, tn, k0, k1, layer;
};

__device__ __forceinline__ WorkItem decode_item(int64_t i, const GemmParams& p) {
    const int64_t grid = static_cast<int64_t>(p.Mt) * p.Nt;
    const int layer = static_cast<int>(i / grid);
    const int64_t s = i - static_cast<int64_t>(layer) * grid;
    const TileCoord t = (p.order == 0) ? curve_decode(s, p.Mt, p.Nt) : raster_decode(s, p.Nt);
    WorkItem w;
    w.tm = t.tm;
    w.tn = t.tn;
    w.layer = layer;
    w.k0 = static_cast<int>((static_cast<int64_t>(layer) * p.Kt) / p.ca_c);
    w.k1 = static_cast<int>((static_cast<int64_t>(layer + 1) * p.Kt) / p.ca_c);
    return w;
}

// Items of this block: [first, end) with stride `step`.
__device__ __forceinline__ void block_items(const GemmParams& p, int64_t& first, int64_t& end,
                                            int64_t& step) {
    const int64_t P = gridDim.x, b = blockIdx.x;
    if (p.assign == 0) {
        first = b * p.num_items / P;
        end = (b + 1) * p.num_items / P;
        step = 1;
    } else {
        first = b;
        end = p.num_items;
        step = P;
    }
}

// Bounded wait for phase `parity` of `bar`.  Gives up (returns false) when the
// block-wide abort flag is raised, or after `limit_ns`, raising it itself.
__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             uint64_t limit_ns, unsigned int site,
                                             bool honour_abort = true) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::global_timer_ns();
    for (;;) {
        if (ptx::mbar_try_wait(bar, parity)) return true;
        if (honour_abort && *abort_flag) return false;
        if (ptx::global_timer_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            atomicOr(&g_sfc_status, 1u | site);
            return false;
        }
    }
}

template <typename OutT>
__device__ __forceinline__ OutT cvt_out(float v);
template <>
__device__ __forceinline__ float cvt_out<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 cvt_out<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// Store 32 consecutive accumulator columns of one row.
template <typename OutT>
__device__ __forceinline__ void store_chunk(OutT* row_ptr, int64_t col0, int64_t N, const uint32_t (&r)[32],
                                            bool vec) {
    if (vec && col0 + 32 <= N) {
        if constexpr (sizeof(OutT) == 4) {
            float4* dst = reinterpret_cast<float4*>(row_ptr + col0);
#pragma unroll
            for (int j = 0; j < 8; ++j)
                dst[j] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                     __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
        } else {
            uint4* dst = reinterpret_cast<uint4*>(row_ptr + col0);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                uint32_t w[4];
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    __nv_bfloat162 v = __floats2bfloat162_rn(__uint_as_float(r[8 * j + 2 * h]),
                                                             __uint_as_float(r[8 * j + 2 * h + 1]));
                    w[h] = *reinterpret_cast<uint32_t*>(&v);
                }
                dst[j] = make_uint4(w[0], w[1], w[2], w[3]);
            }
        }
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (col0 + j < N) row_ptr[col0 + j] = cvt_out<OutT>(__uint_as_float(r[j]));
    }
}

template <int BN, int STAGES, typename OutT>
__global__ void __launch_bounds__(kThreads, 1)
sfc_gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                const GemmParams p) {
    using L = SmemLayout<BN, STAGES>;
    static_assert(BN % kBBox == 0 && BN >= 64 && BN <= 256, "BN must be 64..256 in steps of 64");
    static_assert(2 * BN <= 512, "two accumulators must fit in 512 TMEM columns");
    constexpr uint32_t kIdesc = ptx::idesc_bf16_f32(kBM, BN, /*A K-major*/ 0, /*B MN-major*/ 1);
    constexpr uint32_t kTmemCols = 2 * BN;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);
    const uint32_t ring = base;
    const uint32_t bars = base + L::kBarOffset;
    const uint32_t drain_bar = bars + 8 * (2 * STAGES + 4);
    const uint32_t never_bar = bars + 8 * (2 * STAGES + 5);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kMiscOffset);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kMiscOffset + 4);
    auto full_bar = [&](int s) { return bars + 8u * s; };
    auto empty_bar = [&](int s) { return bars + 8u * (STAGES + s); };
    auto accf_bar = [&](int a) { return bars + 8u * (2 * STAGES + a); };
    auto acce_bar = [&](int a) { return bars + 8u * (2 * STAGES + 2 + a); };

    const int warp = threadIdx.x / 32;
    const int lane = threadIdx.x % 32;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(full_bar(s), 1);
            ptx::mbar_init(empty_bar(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            ptx::mbar_init(accf_bar(a), 1);
            ptx::mbar_init(acce_bar(a), 4);  // one arrive per epilogue warp
        }
        ptx::mbar_init(drain_bar, 1);
        ptx::mbar_init(never_bar, 1);
        *abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        ptx::tma_prefetch_desc(&tmap_a);
        ptx::tma_prefetch_desc(&tmap_b);
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_addr(tmem_slot), kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    int64_t first, end, step;
    block_items(p, first, end, step);

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int64_t issued = 0;
            bool ok = true;
            for (int64_t it = first; ok && it < end; it += step) {
                const WorkItem w = decode_item(it, p);
                for (int kt = w.k0; kt < w.k1; ++kt) {
                    if (!wait_bounded(empty_bar(stage), phase ^ 1u, abort_flag, p.timeout_ns,
                                      kWaitProducerEmpty)) {
                        ok = false;
                        break;
                    }
                    ptx::mbar_arrive_expect_tx(full_bar(stage), L::kStageBytes);
                    const uint32_t sa = ring + stage * L::kStageBytes;
                    const uint32_t sb = sa + L::kABytes;
                    ptx::tma_load_2d(sa, &tmap_a, full_bar(stage), kt * kBK, w.tm * kBM);
#pragma unroll
                    for (int j = 0; j < BN / kBBox; ++j)
                        ptx::tma_load_2d(sb + j * (kBBox * kBK * 2), &tmap_b, full_bar(stage),
                                         w.tn * BN + j * kBBox, kt * kBK);
                    ++issued;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            // Tail: the last STAGES issues.  On success wait until the MMA warp's
            // commits have released them (no arrive may land after exit); after a
            // failure wait (bounded) for the copies still in flight into the ring.
            const int64_t n0 = issued > STAGES ? issued - STAGES : 0;
            for (int64_t n = n0; n < issued; ++n) {
                const int slot = static_cast<int>(n % STAGES);
                const uint32_t par = static_cast<uint32_t>((n / STAGES) & 1);
                if (ok)
                    ok = wait_bounded(empty_bar(slot), par, abort_flag, p.timeout_ns, kWaitProducerEmpty);
                if (!ok)
                    wait_bounded(full_bar(slot), par, abort_flag, p.timeout_ns, kWaitDrain,
                                 /*honour_abort=*/false);
            }
        }
    } else if (warp == 1) {
        // -------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            if (p.debug_never)
                ok = wait_bounded(never_bar, 0, abort_flag, p.timeout_ns, kWaitDebugNever);
            for (int64_t it = first; ok && it < end; it += step) {
                const WorkItem w = decode_item(it, p);
                if (!wait_bounded(acce_bar(acc), acc_phase ^ 1u, abort_flag, p.timeout_ns,
                                  kWaitMmaAccEmpty)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
                for (int kt = w.k0; kt < w.k1; ++kt) {
                    if (!wait_bounded(full_bar(stage), phase, abort_flag, p.timeout_ns, kWaitMmaFull)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t sa = ring + stage * L::kStageBytes;
                    const uint32_t sb = sa + L::kABytes;
#pragma unroll
                    for (int kk = 0; kk < kBK / kUmmaK; ++kk) {
                        // A: K-major, 128-byte rows, 8-row atoms 1024 B apart; step 32 B per K=16
                        const uint64_t adesc = ptx::smem_desc_sw128(sa + kk * (kUmmaK * 2), 16, 1024);
                        // B: MN-major, 64-column boxes 8 KB apart, 8-row atoms 1024 B apart;
                        // step 16 rows (2 KB) per K=16
                        const uint64_t bdesc =
                            ptx::smem_desc_sw128(sb + kk * (kUmmaK * 128), kBBox * kBK * 2, 1024);
                        ptx::tc_mma_f16(d_tmem, adesc, bdesc, kIdesc, (kt > w.k0 || kk > 0) ? 1u : 0u);
                    }
                    ptx::tc_commit(empty_bar(stage));  // frees the stage once these MMAs finish
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                ptx::tc_commit(accf_bar(acc));  // accumulator ready for the epilogue
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
            if (!ok) {
                // wait (bounded) until every MMA issued so far has finished
                ptx::tc_commit(drain_bar);
                wait_bounded(drain_bar, 0, abort_flag, p.timeout_ns, kWaitDrain, /*honour_abort=*/false);
            }
        }
    } else {
        // ---------------------------------------------------------- epilogue
        const int quarter = warp & 3;  // TMEM lanes 32*quarter .. +31
        int acc = 0;
        uint32_t acc_phase = 0;
        OutT* out = static_cast<OutT*>(p.out);
        for (int64_t it = first; it < end; it += step) {
            const WorkItem w = decode_item(it, p);
            // lane 0 waits, the warp follows its verdict (tcgen05.ld needs the whole warp)
            int ready = 1;
            if (lane == 0)
                ready = wait_bounded(accf_bar(acc), acc_phase, abort_flag, p.timeout_ns, kWaitEpiAccFull);
            ready = __shfl_sync(0xffffffffu, ready, 0);
            if (!ready) break;
            ptx::tc_fence_after();
            const int64_t row = static_cast<int64_t>(w.tm) * kBM + quarter * 32 + lane;
            OutT* row_ptr = out + static_cast<int64_t>(w.layer) * p.layer_stride + row * p.ldo;
            const uint32_t taddr =
                tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(acc * BN);
            const int64_t col_base = static_cast<int64_t>(w.tn) * BN;
#pragma unroll 1
            for (int ch = 0; ch < BN / 32; ++ch) {
                uint32_t r[32];
                ptx::tmem_ld_32x32b_x32(taddr + ch * 32, r);
                ptx::tmem_ld_wait();
                if (row < p.M) store_chunk<OutT>(row_ptr, col_base + ch * 32, p.N, r, p.vec_store != 0);
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(acce_bar(acc));
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem_base, kTmemCols);
}

// C = cvt(sum_{l=0}^{c-1} P_l), summed in layer order, 4 columns per thread.
// P_l rows are `ldw` floats apart (ldw % 4 == 0), layers `layer_stride` apart.
template <typename OutT>
__global__ void __launch_bounds__(256)
ca_reduce_kernel(const float* __restrict__ ws, int64_t ldw, int64_t layer_stride, int c, int64_t M,
                 int64_t N, OutT* __restrict__ C, int64_t ldc, int vec_store) {
    const int64_t n4 = (N + 3) / 4;
    const int64_t total = M * n4;
    for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t i = idx / n4;
        const int64_t j = (idx - i * n4) * 4;
        const float* src = ws + i * ldw + j;
        float4 acc = __ldcs(reinterpret_cast<const float4*>(src));
        for (int l = 1; l < c; ++l) {
            const float4 v = __ldcs(reinterpret_cast<const float4*>(src + l * layer_stride));
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
        OutT* dst = C + i * ldc + j;
        if (vec_store && j + 4 <= N) {
            if constexpr (sizeof(OutT) == 4) {
                *reinterpret_cast<float4*>(dst) = acc;
            } else {
                __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
                __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
                uint2 u;
                u.x = *reinterpret_cast<uint32_t*>(&lo);
                u.y = *reinterpret_cast<uint32_t*>(&hi);
                *reinterpret_cast<uint2*>(dst) = u;
            }
        } else {
            const float v[4] = {acc.x, acc.y, acc.z, acc.w};
            for (int h = 0; h < 4 && j + h < N; ++h) dst[h] = cvt_out<OutT>(v[h]);
        }
    }
}

// out[s] = tm * Nt + tn for every curve position s, with the kernel's decoder.
__global__ void tile_order_kernel(int Mt, int Nt, int32_t* __restrict__ out) {
    const int64_t n = static_cast<int64_t>(Mt) * Nt;
    for (int64_t s = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; s < n;
         s += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const TileCoord t = curve_decode(s, Mt, Nt);
        out[s] = t.tm * Nt + t.tn;
    }
}

}  // namespace sfc
