// sfc_gemm_kernel.cuh -- persistent SFC / SFC-CA GEMM kernels for sm_103a.
//
// A block (or a 2-SM pair of blocks) resident on each SM walks its share of
// the task space of Listing 1: Mt*Nt*K_layers items, item i -> K layer
// i / (Mt*Nt), curve position i % (Mt*Nt) -> output tile.  For each item it
// contracts the layer's K range of one output tile (the paper's batch-reduce
// GEMM over K blocks, Sec. II-A; C is zeroed at the first K block, Listing 1)
// on the tcgen05 tensor cores:
//
//   warp 0        TMA producer: 64-wide K slabs of A and B (bf16, 128-byte
//                 swizzle) into a STAGES-deep shared-memory ring;
//   warp 1        MMA issuer: tcgen05.mma (K = 16 each) into one of two
//                 tensor-memory accumulators; tcgen05.commit frees ring stages
//                 and publishes finished accumulators;
//   warps 2..     epilogue: tcgen05.ld the accumulator (warp w reads TMEM lanes
//                 32*(w%4)..), add it into fp32 running sums held in registers,
//                 and after the item's last chunk convert and store the tile
//                 (masked at the M/N edges);
//   last warp     scheduler: deals the worker's items (curve positions) and
//                 decodes each into its tile before any other role needs it.
//
// Accumulation chains.  The tensor core's fp32 accumulation drops low-order
// bits on every accumulate, so the error of one long chain grows linearly with
// K.  Each item's K range is therefore cut into chunks of at most p.kc slabs;
// every chunk restarts the tensor-memory accumulator and the epilogue adds the
// chunk's result into its register running sum with round-to-nearest fp32
// adds.  Two accumulators let chunk j+1 run on the tensor core while the
// epilogue drains chunk j, and the last chunk of a tile overlap the next tile.
//
// With K_layers > 1 the epilogue writes the layer's fp32 partial tile to that
// layer's workspace copy of C; ca_reduce_kernel sums the copies in layer order.
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

constexpr int kBM = 128;          // output tile rows per CTA (UMMA M of one CTA)
constexpr int kBK = 64;           // K slab of bf16 inputs: 64 values = one 128-byte swizzle row
constexpr int kEpiCols = 128;     // accumulator columns each epilogue thread owns

// Per input kind (bf16, or 8-bit floats with F8): the K values of one
// 128-byte shared-memory row (a slab), of one tcgen05.mma, and the columns of
// an N-major B box (also 128 bytes).  Every stage row is 128 bytes either way.
template <bool F8>
struct InKind {
    static constexpr int kSlabK = F8 ? 128 : 64;
    static constexpr int kMmaK = F8 ? 32 : 16;
    static constexpr int kBCols = F8 ? 128 : 64;
    static constexpr int kBBoxBytes = kSlabK * 128;  // one N-major box: slab rows x 128 bytes
};

// Threads of a block: producer warp, MMA warp, BN/32 epilogue warps
// (4 warps per 128 columns: one warp per TMEM lane quarter), scheduler warp.
__host__ __device__ constexpr int block_threads(int bn) { return 96 + 32 * (bn / 32); }
__host__ __device__ constexpr int scheduler_warp(int bn) { return 2 + bn / 32; }

// device error word: bit 0 = a bounded wait gave up; bits 8.. = which wait
__device__ unsigned int g_sfc_status = 0;

enum WaitSite : unsigned int {
    kWaitProducerEmpty = 1u << 8,
    kWaitMmaFull = 1u << 9,
    kWaitMmaAccEmpty = 1u << 10,
    kWaitEpiAccFull = 1u << 11,
    kWaitDebugNever = 1u << 12,
    kWaitDrain = 1u << 13,
    kWaitQueueFull = 1u << 14,
    kWaitQueueEmpty = 1u << 15,
};

// Item dealing.  One scheduler thread per worker decodes the worker's items
// (curve position -> tile, K layer) and hands them to every role of every CTA
// of the worker through a small queue in shared memory.  Static dealing gives
// worker w the items first + j * step; dynamic dealing gives it item w first
// (so no block waits on a counter to start) and then workers + the next value
// of the launch's ticket counter, i.e. curve positions are taken in order as
// workers free up.  The counter ({next ticket, schedulers done}, two 64-bit
// words) is memory of the call that launched the kernel, so no other launch
// can share it.  Each word carries the launch's epoch (a 32-bit tag the host
// gives every call) above a 32-bit count: a word whose tag is not the epoch is
// read as a count of zero, so the memory needs no clearing before a launch,
// also when it is fresh graph memory whose contents are unknown.  The last
// scheduler to finish sets both words to zero (also after a wait gave up), so
// that a replay of a captured launch, which keeps its epoch, starts from zero.
constexpr int kQueue = 4;

// At a launch's start (after the wait for the previous grid): tag the word with
// this epoch and a count of zero unless it carries the epoch already, so that
// the first tickets find their tag and take one atomic add.  One attempt: a
// failed swap means another worker changed the word first.
__device__ __forceinline__ void epoch_claim(unsigned long long* word, unsigned int epoch) {
    const unsigned long long tag = static_cast<unsigned long long>(epoch) << 32;
    const unsigned long long cur = atomicOr(word, 0ull);
    if ((cur & 0xffffffff00000000ull) != tag) atomicCAS(word, cur, tag);
}

// Next value of an epoch-tagged counter (see above); 32-bit counts.  The
// common case is one atomic add.  An add that finds another tag is void: the
// word is then set to "this epoch, one ticket taken" by a compare-and-swap,
// whose winner holds ticket 0 (every other taker retries and, once the tag is
// this epoch's, adds again), so every ticket of the epoch is handed out once.
__device__ __forceinline__ unsigned int epoch_ticket(unsigned long long* word, unsigned int epoch) {
    constexpr unsigned long long kTagMask = 0xffffffff00000000ull;
    const unsigned long long tag = static_cast<unsigned long long>(epoch) << 32;
    unsigned long long old = atomicAdd(word, 1ull);
    while ((old & kTagMask) != tag) {
        const unsigned long long cur = atomicOr(word, 0ull);  // an atomic read of the word
        if ((cur & kTagMask) == tag) {
            old = atomicAdd(word, 1ull);
        } else if (atomicCAS(word, cur, tag | 1ull) == cur) {
            return 0u;
        }
    }
    return static_cast<unsigned int>(old);
}

struct GemmParams {
    int64_t M, N;
    int Mt, Nt, Kt;        // tile grid and number of 64-wide K slabs
    int ca_c;              // K layers
    int grid_tiles;        // Mt * Nt
    int kq, kr;            // Kt / ca_c and Kt % ca_c (layer l starts at l*kq + l*kr/ca_c)
    int kc;                // max slabs per tensor-memory accumulation chain
    int64_t num_items;     // Mt * Nt * ca_c
    void* out;             // C when ca_c == 1, else the fp32 workspace
    int64_t ldo;           // row stride of `out` in elements
    int64_t layer_stride;  // elements between K-layer copies in `out`
    int order;             // 0 = generalized Hilbert, 1 = raster
    int assign;            // static deal: 0 = contiguous segments, 1 = strided waves
    int dynamic;           // 1: workers take the next curve position from a shared counter
    unsigned long long* ticket;  // dynamic dealing: this launch's counter words {next, done}
    unsigned int epoch;          // the call's tag for its counter words (never 0)
    int vec_store;         // 1 if 16-byte vector stores are aligned
    int tma_store;         // 1: stores go through smem staging and the output tensor map
    int debug_never;       // test hook: MMA warp waits on a barrier nobody arrives at
    uint64_t timeout_ns;   // bound for every mbarrier wait
    int b_kmajor;          // 1: B is given as N x K row-major (B transposed), loaded K-major
    float beta;            // C = A B + beta C_in + bias (ca_c == 1: applied by the epilogue)
    const void* c_in;      // C_in (the output array, read before it is written) when beta != 0
    int64_t ldc_in;        // its row stride in elements
    int64_t c_in_layer_stride;  // != 0: C_in is `out` itself, K-layer copy by copy (beta applied per layer)
    const float* bias;     // N fp32 values or null
    int ab_fmt;            // A/B format code of the instruction descriptor (bf16: 1; e4m3: 0, e5m2: 1)
    int kbf, pass;         // k_block_factor > 1: this launch contracts K block `pass` of every layer
    int accumulate;        // 1: the TMA stores add into `out` (fp32, in L2) instead of overwriting it
};

struct WorkItem {
    int tm, tn, k0, k1, layer;
};

// Slab index of the q-th slab this item processes (K slabs in increasing order).
__device__ __forceinline__ int slab_at(const WorkItem& w, int q) { return w.k0 + q; }

// First K slab of layer l: floor(l * Kt / c) = l * (Kt / c) + floor(l * (Kt % c) / c),
// in 32-bit arithmetic (c <= 4096 keeps l * (Kt % c) below 2^24).
__device__ __forceinline__ int layer_k0(int l, const GemmParams& p) { return l * p.kq + (l * p.kr) / p.ca_c; }

// With k_block_factor > 1 (the outer K-block loop of Listing 1) a launch
// contracts block `pass` of each layer's slabs: [k0 + floor(pass * len / kbf),
// k0 + floor((pass + 1) * len / kbf)).  kbf <= 64 and len < 2^25 keep the
// products in 32 bits.
__device__ __forceinline__ void narrow_to_pass(WorkItem& w, const GemmParams& p) {
    if (p.kbf > 1) {
        const unsigned len = static_cast<unsigned>(w.k1 - w.k0), kbf = static_cast<unsigned>(p.kbf);
        const unsigned pass = static_cast<unsigned>(p.pass);
        const int base = w.k0;
        w.k0 = base + static_cast<int>(pass * len / kbf);
        w.k1 = base + static_cast<int>((pass + 1u) * len / kbf);
    }
}

// Item index i < 2^31 (validated on the host) -> tile, K layer and K range.
__device__ __forceinline__ WorkItem decode_item(int64_t i64, const GemmParams& p) {
    const int i = static_cast<int>(i64);
    const int layer = (p.ca_c == 1) ? 0 : i / p.grid_tiles;
    const int s = i - layer * p.grid_tiles;
    const TileCoord t = (p.order == 0) ? curve_decode(s, p.Mt, p.Nt) : raster_decode(s, p.Nt);
    WorkItem w;
    w.tm = t.tm;
    w.tn = t.tn;
    w.layer = layer;
    w.k0 = layer_k0(layer, p);
    w.k1 = layer_k0(layer + 1, p);
    narrow_to_pass(w, p);
    return w;
}

// Chunks of an item's K range: n = ceil(len / kc), boundaries balanced.
__device__ __forceinline__ int num_chunks(const WorkItem& w, int kc) {
    const int len = w.k1 - w.k0;
    return len <= kc ? 1 : (len + kc - 1) / kc;
}
// Position (0-based, in processing order) where chunk j of n starts.
// Chunk j of n starts at position floor(j * len / n) of the item's K range;
// the walk steps through j = 0, 1, ..., n with one 32-bit division per item
// (the MMA issuer does this between its MMAs).
struct ChunkWalk {
    int q, r, n, begin, rem;
    __device__ __forceinline__ ChunkWalk(const WorkItem& w, int n_) : n(n_), begin(0), rem(0) {
        const int len = w.k1 - w.k0;
        q = (n_ == 1) ? len : len / n_;
        r = len - q * n_;
    }
    // end of the current chunk = begin of the next; advances
    __device__ __forceinline__ int next() {
        rem += r;
        begin += q;
        if (rem >= n) {
            rem -= n;
            ++begin;
        }
        return begin;
    }
};

// Items of worker `worker` out of `workers`: [first, end) with stride `step`.
__device__ __forceinline__ void worker_items(const GemmParams& p, int64_t worker, int64_t workers,
                                             int64_t& first, int64_t& end, int64_t& step) {
    if (p.assign == 0) {
        first = worker * p.num_items / workers;
        end = (worker + 1) * p.num_items / workers;
        step = 1;
    } else {
        first = worker;
        end = p.num_items;
        step = workers;
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

// wait_bounded for roles that wait long and can answer late (the epilogue,
// the scheduler): sleeps between polls, so that idle warps neither take issue
// slots from the producer and MMA warps nor burn power spinning.
__device__ __forceinline__ bool wait_bounded_idle(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                                  uint64_t limit_ns, unsigned int site, unsigned int sleep_ns) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::global_timer_ns();
    for (;;) {
        __nanosleep(sleep_ns);
        if (ptx::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
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

// beta * C_in + bias for columns [col0, col0 + n) of one row of K layer
// `layer`, added into v (fp32, before rounding to the output type).  Columns
// >= N are left alone.
template <typename OutT, int n>
__device__ __forceinline__ void apply_affine(const GemmParams& p, int64_t row, int64_t col0, int layer, float* v) {
    if (p.beta != 0.0f && row < p.M) {
        const OutT* src = static_cast<const OutT*>(p.c_in) + layer * p.c_in_layer_stride + row * p.ldc_in + col0;
#pragma unroll
        for (int j = 0; j < n; ++j)
            if (col0 + j < p.N) v[j] = __fmaf_rn(p.beta, static_cast<float>(src[j]), v[j]);
    }
    if (p.bias) {
#pragma unroll
        for (int j = 0; j < n; ++j)
            if (col0 + j < p.N) v[j] = __fadd_rn(v[j], __ldg(p.bias + col0 + j));
    }
}

// Per-block barrier set and smem layout shared by both kernels.
struct Barriers {
    uint32_t bars;
    int stages;
    __device__ __forceinline__ uint32_t full(int s) const { return bars + 8u * s; }
    __device__ __forceinline__ uint32_t empty(int s) const { return bars + 8u * (stages + s); }
    __device__ __forceinline__ uint32_t acc_full(int a) const { return bars + 8u * (2 * stages + a); }
    __device__ __forceinline__ uint32_t acc_empty(int a) const { return bars + 8u * (2 * stages + 2 + a); }
    __device__ __forceinline__ uint32_t drain() const { return bars + 8u * (2 * stages + 4); }
    __device__ __forceinline__ uint32_t never() const { return bars + 8u * (2 * stages + 5); }
    __device__ __forceinline__ uint32_t q_full(int q) const { return bars + 8u * (2 * stages + 6 + q); }
    __device__ __forceinline__ uint32_t q_empty(int q) const { return bars + 8u * (2 * stages + 6 + kQueue + q); }
    __device__ __forceinline__ uint32_t q_taken() const { return bars + 8u * (2 * stages + 6 + 2 * kQueue); }
};

// Epilogue staging: one 4 KB buffer per epilogue warp (two output boxes).
constexpr int kStageBufBytes = 4096;

template <int STAGE_BYTES, int STAGES, int EPI_WARPS>
struct RingLayout {
    static constexpr int kRingBytes = STAGE_BYTES * STAGES;
    static constexpr int kStagingOffset = kRingBytes;
    static constexpr int kStagingBytes = EPI_WARPS * kStageBufBytes;
    static constexpr int kQueueOffset = kRingBytes + kStagingBytes;  // kQueue entries of 16 bytes
    static constexpr int kNumBars = 2 * STAGES + 7 + 2 * kQueue;
    static constexpr int kBarOffset = kQueueOffset + 16 * kQueue;
    static constexpr int kMiscOffset = kBarOffset + kNumBars * 8;
    static constexpr int kBytes = kMiscOffset + 16;
    static constexpr int kDynamicBytes = kBytes + 1024;  // slack to align the ring to 1024 B
};

// A worker's item source: the scheduler's deal parameters and the queue.
// Queue entry q (16 bytes): item index (-1: no more items), tm, tn, K layer.
struct ItemSource {
    int64_t first, end, step;  // static deal: first + j * step while < end
    int64_t worker, workers;   // this worker and the launch's worker count
    int dynamic;
    uint32_t q_full0;          // this CTA's q_full[0]
    uint32_t q_empty0;         // the scheduler CTA's q_empty[0] (cluster address)
    volatile int* q_entry;     // this CTA's queue
};

// Item j of a consuming role: fills w (tile, K layer and range; K order from
// j) and returns the item index >= 0, or -1 when there are no more, -2 when a
// bounded wait gave up.  Item 0 needs no wait (`first_local`, for the roles on
// the start-up path: producer and MMA issuer): every CTA decodes it into its
// own slot 0 during set-up (sched_local_first), before the block barrier.  The
// epilogue waits for the slot's first phase as for any other item (it needs
// item 0 only microseconds later, and the branch would cost it registers).
template <bool kFirstLocal = false>
__device__ __forceinline__ int64_t src_take(const ItemSource& S, int j, const GemmParams& p, volatile int* abort_flag,
                                            WorkItem& w) {
    const int q = j % kQueue;
    if ((!kFirstLocal || j > 0) &&
        !wait_bounded(S.q_full0 + 8u * q, static_cast<uint32_t>((j / kQueue) & 1), abort_flag, p.timeout_ns,
                      kWaitQueueFull))
        return -2;
    const int item = S.q_entry[4 * q];
    w.tm = S.q_entry[4 * q + 1];
    w.tn = S.q_entry[4 * q + 2];
    w.layer = S.q_entry[4 * q + 3];
    ptx::mbar_arrive_remote(S.q_empty0 + 8u * q);  // slot free once every consumer has read it
    w.k0 = (p.ca_c == 1) ? 0 : layer_k0(w.layer, p);
    w.k1 = (p.ca_c == 1) ? p.Kt : layer_k0(w.layer + 1, p);
    narrow_to_pass(w, p);
    return item;
}

// Scheduler: the queue entry of an item (decoded tile and K layer).
struct QueueEntry {
    int e[4];
};
__device__ __forceinline__ QueueEntry sched_entry(int item, const GemmParams& p) {
    QueueEntry x{{item, 0, 0, 0}};
    if (item >= 0) {
        const WorkItem w = decode_item(item, p);
        x.e[1] = w.tm;
        x.e[2] = w.tn;
        x.e[3] = w.layer;
    }
    return x;
}

// Scheduler: publish entry x as item j, to slot j % kQueue of this CTA's queue
// and of the other n_ctas - 1 CTAs of the cluster (the slot is free).
__device__ __forceinline__ void sched_send(const ItemSource& S, int j, const QueueEntry& x, int n_ctas) {
    const int q = j % kQueue;
    const int(&e)[4] = x.e;
#pragma unroll
    for (int k = 0; k < 4; ++k) S.q_entry[4 * q + k] = e[k];
    ptx::mbar_arrive(S.q_full0 + 8u * q);
    // the peers get the entry by st.async, counted as 16 bytes by their q_full
    const uint32_t mine = ptx::smem_addr(const_cast<int*>(S.q_entry) + 4 * q);
    for (int r = 1; r < n_ctas; ++r) {
        const uint32_t rbar = ptx::map_to_cta(S.q_full0 + 8u * q, r);
        ptx::mbar_expect_tx_remote(rbar, 16);
        ptx::st_async_v4(ptx::map_to_cta(mine, r), e, rbar);
    }
}

// Set-up of every CTA of a worker: its first item (the same in each CTA: the
// worker's first position of the deal, which takes no ticket) written into
// slot 0 of the CTA's own queue, so that no role waits for the scheduler's
// message to start.  Called by one thread before the set-up's block barrier.
__device__ __forceinline__ void sched_local_first(const ItemSource& S, const QueueEntry& x) {
#pragma unroll
    for (int k = 0; k < 4; ++k) S.q_entry[k] = x.e[k];
}

// Scheduler: item 0 is already in every CTA's slot 0; complete phase 0 of
// each CTA's q_full[0] all the same (no data), so that the slot's later uses
// line up with their phases.  After the cluster barrier of the set-up.
__device__ __forceinline__ void sched_mark_first(const ItemSource& S, int n_ctas) {
    ptx::mbar_arrive(S.q_full0);
    for (int r = 1; r < n_ctas; ++r) ptx::mbar_arrive_remote(ptx::map_to_cta(S.q_full0, r));
}

// Item j of the worker's deal (j >= 1 for dynamic dealing takes a ticket).
__device__ __forceinline__ int sched_next(const ItemSource& S, int j, const GemmParams& p) {
    int64_t pos;
    if (S.dynamic)
        pos = (j == 0) ? S.worker : S.workers + static_cast<int64_t>(epoch_ticket(&p.ticket[0], p.epoch));
    else
        pos = S.first + j * S.step;
    const int64_t end = S.dynamic ? p.num_items : S.end;
    return pos < end ? static_cast<int>(pos) : -1;
}

// Scheduler loop, items 1.. (item 0 is published during set-up).  Item j is
// published once the worker's producer has taken item j - 1, so tickets are
// taken one item ahead of need: late enough that dynamic dealing still
// balances the last wave, early enough that the counter's round trip and the
// decode are off every other role's path.  Returns false when a bounded wait
// gave up.
__device__ __forceinline__ bool run_scheduler(const ItemSource& S, int item0, const GemmParams& p, const Barriers& B,
                                              volatile int* abort_flag, int n_ctas) {
    bool ok = true;
    if (S.dynamic) {
        epoch_claim(&p.ticket[0], p.epoch);
        epoch_claim(&p.ticket[1], p.epoch);
    }
    for (int j = 1; ok && item0 >= 0; ++j) {
        if (!wait_bounded_idle(B.q_taken(), static_cast<uint32_t>((j - 1) & 1), abort_flag, p.timeout_ns,
                               kWaitQueueEmpty, 256) ||
            !wait_bounded_idle(S.q_empty0 + 8u * (j % kQueue), static_cast<uint32_t>(((j / kQueue) & 1) ^ 1),
                               abort_flag, p.timeout_ns, kWaitQueueEmpty, 256)) {
            ok = false;
            break;
        }
        const int item = sched_next(S, j, p);
        sched_send(S, j, sched_entry(item, p), n_ctas);
        if (item < 0) break;
    }
    if (S.dynamic) {
        // the last scheduler of the launch returns the counter to zero
        __threadfence();
        const unsigned int before = epoch_ticket(&p.ticket[1], p.epoch);
        if (static_cast<int64_t>(before) == S.workers - 1) {
            p.ticket[0] = 0ull;
            p.ticket[1] = 0ull;
            __threadfence();
        }
    }
    return ok;
}

// Producer loop shared by the kernels: takes the worker's items from the
// queue and, for each K slab, waits for a free ring stage and calls
// issue(w, kt, stage).  `signal_taken`: this is the producer the scheduler
// paces itself on.  Returns false when a bounded wait gave up; `issued`
// counts the stages filled.
template <int STAGES, typename IssueFn>
__device__ __forceinline__ bool produce(const ItemSource& src, const GemmParams& p, const Barriers& B,
                                        volatile int* abort_flag, bool signal_taken, int64_t& issued,
                                        IssueFn&& issue) {
    int stage = 0;
    uint32_t phase = 0;
    for (int j = 0;; ++j) {
        WorkItem w;
        const int64_t it = src_take<true>(src, j, p, abort_flag, w);
        if (it < 0) return it == -1;
        if (signal_taken) ptx::mbar_arrive(B.q_taken());
        const int nq = w.k1 - w.k0;
        for (int q = 0; q < nq; ++q) {
            if (!wait_bounded(B.empty(stage), phase ^ 1u, abort_flag, p.timeout_ns, kWaitProducerEmpty))
                return false;
            issue(w, slab_at(w, q), stage);
            ++issued;
            if (++stage == STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
    }
}

// Output staging boxes are 32 rows x 64 bytes: 32 bf16 or 16 fp32 columns,
// in the layout of a 64-byte swizzled TMA box (16-byte unit j of row r sits at
// unit j ^ ((r >> 1) & 3)).  Each epilogue warp owns a 4 KB buffer holding two
// boxes, so one box is filled while the TMA still reads the other.
constexpr int kBoxBytes = 2048;
template <typename OutT>
__host__ __device__ constexpr int box_cols() { return 64 / static_cast<int>(sizeof(OutT)); }

// Write this lane's row of one box (box_cols<OutT>() values from v).
template <typename OutT>
__device__ __forceinline__ void stage_row(uint8_t* box, int lane, const float* v) {
    uint8_t* row = box + lane * 64;
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        uint4 u;
        if constexpr (sizeof(OutT) == 4) {
            u = make_uint4(__float_as_uint(v[4 * j]), __float_as_uint(v[4 * j + 1]), __float_as_uint(v[4 * j + 2]),
                           __float_as_uint(v[4 * j + 3]));
        } else {
            uint32_t w[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                __nv_bfloat162 b = __floats2bfloat162_rn(v[8 * j + 2 * h], v[8 * j + 2 * h + 1]);
                w[h] = *reinterpret_cast<uint32_t*>(&b);
            }
            u = make_uint4(w[0], w[1], w[2], w[3]);
        }
        *reinterpret_cast<uint4*>(row + ((j ^ sw) * 16)) = u;
    }
}

// -------------------------------------------------------------------------
// Epilogue of one block: drain chunks, promote, store.  `rows_base` is the
// first output row this block's TMEM lanes map to for tile row tm.
// -------------------------------------------------------------------------
template <int BN, typename OutT, bool PAIR>
__device__ __forceinline__ void run_epilogue(const GemmParams& p, const Barriers& B, uint32_t tmem_base,
                                             volatile int* abort_flag, const ItemSource& src,
                                             int tile_rows, int row_offset, int warp, int lane,
                                             const CUtensorMap* tmap_c, uint8_t* staging, uint32_t pair_leader = 0) {
    const int ew = warp - 2;                 // epilogue warp index
    const int quarter = warp & 3;            // TMEM lane quarter this warp may access
    const int half = ew / 4;                 // which 128-column half of the tile
    int acc = 0;
    uint32_t acc_phase = 0;
    OutT* out = static_cast<OutT*>(p.out);
    const uint32_t acce_target = PAIR ? ptx::map_to_cta(B.acc_empty(0), pair_leader) : B.acc_empty(0);
    float run[kEpiCols];
    // beta C_in + bias in this epilogue only without K layers (else the reduction applies
    // it), or when a later K block adds into the layer copies (k_block_factor > 1)
    const bool affine = (p.ca_c == 1 || p.c_in_layer_stride != 0) && (p.beta != 0.0f || p.bias != nullptr);
    for (int j = 0;; ++j) {
        // lane 0 takes the item, the warp follows (tcgen05.ld needs the whole warp)
        int64_t it = 0;
        WorkItem w{};
        if (lane == 0) it = src_take(src, j, p, abort_flag, w);
        it = __shfl_sync(0xffffffffu, it, 0);
        if (it < 0) break;
        w.tm = __shfl_sync(0xffffffffu, w.tm, 0);
        w.tn = __shfl_sync(0xffffffffu, w.tn, 0);
        w.layer = __shfl_sync(0xffffffffu, w.layer, 0);
        w.k0 = __shfl_sync(0xffffffffu, w.k0, 0);
        w.k1 = __shfl_sync(0xffffffffu, w.k1, 0);
        const int nch = num_chunks(w, p.kc);
        bool ok = true;
        for (int ck = 0; ck < nch; ++ck) {
            int ready = 1;
            if (lane == 0)  // no sleeps: try_wait suspends the thread until the phase completes
                ready = wait_bounded(B.acc_full(acc), acc_phase, abort_flag, p.timeout_ns, kWaitEpiAccFull);
            ready = __shfl_sync(0xffffffffu, ready, 0);
            if (!ready) {
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                   static_cast<uint32_t>(acc * BN + half * kEpiCols);
            if (ck == 0) {
                // the chain's first chunk becomes the running sum as loaded
#pragma unroll
                for (int g = 0; g < kEpiCols / 32; ++g) {
                    uint32_t r[32];
                    ptx::tmem_ld_32x32b_x32(taddr + g * 32, r);
                    ptx::tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j) run[g * 32 + j] = __uint_as_float(r[j]);
                }
            } else {
                // later chunks are added in 16-column pieces (fewer registers live beside run[])
#pragma unroll
                for (int g = 0; g < kEpiCols / 16; ++g) {
                    uint32_t r[16];
                    ptx::tmem_ld_32x32b_x16(taddr + g * 16, r);
                    ptx::tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 16; ++j) run[g * 16 + j] = __fadd_rn(run[g * 16 + j], __uint_as_float(r[j]));
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                // the accumulator-empty barriers are 8 bytes apart
                if (PAIR) ptx::mbar_arrive_remote(acce_target + 8u * acc);
                else ptx::mbar_arrive(B.acc_empty(acc));
            }
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if (!ok) break;
        const int64_t warp_row = static_cast<int64_t>(w.tm) * tile_rows + row_offset + quarter * 32;
        const int64_t col_base = static_cast<int64_t>(w.tn) * BN + half * kEpiCols;
        if (p.tma_store) {
            // stage 32-row boxes and let the TMA write them (edges clipped by the map);
            // the two boxes of the buffer alternate
            constexpr int kCols = box_cols<OutT>();
            // the two boxes of the warp's buffer are staged together, then one proxy fence,
            // one warp sync and one bulk group store both (a round per pair of boxes, not per box)
            uint8_t* buf = staging + ew * kStageBufBytes;
#pragma unroll
            for (int g = 0; g < kEpiCols / kCols; g += 2) {
                if (col_base + g * kCols >= p.N) break;  // warp-uniform
                const bool has1 = col_base + (g + 1) * kCols < p.N;
                if (affine) {
                    apply_affine<OutT, kCols>(p, warp_row + lane, col_base + g * kCols, w.layer, run + g * kCols);
                    if (has1)
                        apply_affine<OutT, kCols>(p, warp_row + lane, col_base + (g + 1) * kCols, w.layer,
                                                  run + (g + 1) * kCols);
                }
                if (lane == 0) ptx::bulk_wait_read_all();  // the previous pair's stores have read the buffer
                __syncwarp();
                stage_row<OutT>(buf, lane, run + g * kCols);
                if (has1) stage_row<OutT>(buf + kBoxBytes, lane, run + (g + 1) * kCols);
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        if (h == 1 && !has1) break;
                        const uint32_t box_addr = ptx::smem_addr(buf + h * kBoxBytes);
                        const int32_t x = static_cast<int32_t>(col_base + (g + h) * kCols);
                        const int32_t y = static_cast<int32_t>(warp_row);
                        if (p.ca_c > 1) {
                            if (p.accumulate) ptx::tma_reduce_add_3d(tmap_c, box_addr, x, y, w.layer);
                            else ptx::tma_store_3d(tmap_c, box_addr, x, y, w.layer);
                        } else {
                            if (p.accumulate) ptx::tma_reduce_add_2d(tmap_c, box_addr, x, y);
                            else ptx::tma_store_2d(tmap_c, box_addr, x, y);
                        }
                    }
                    ptx::bulk_commit();
                }
            }
        } else {
            // C rows the TMA cannot store (C's base or row stride not a multiple of 16 bytes): each
            // 32-row box is staged in the warp's buffer as for the TMA, then read back so that one
            // warp store covers consecutive columns of one row (of two rows for fp32), not one
            // value in each of 32 rows
            constexpr int kCols = box_cols<OutT>();    // 32 bf16 or 16 fp32 columns: 64 bytes per row
            constexpr int kRowsPerStore = 32 / kCols;  // rows one warp store covers
            uint8_t* box = staging + ew * kStageBufBytes;
            OutT* base = out + static_cast<int64_t>(w.layer) * p.layer_stride;
            const int c = lane % kCols;                // this lane's column within the box
            const int cbyte = c * static_cast<int>(sizeof(OutT));
#pragma unroll
            for (int g = 0; g < kEpiCols / kCols; ++g) {  // unrolled: run[] stays in registers
                const int64_t col0 = col_base + g * kCols;
                if (col0 >= p.N) break;  // warp-uniform
                if (affine) apply_affine<OutT, kCols>(p, warp_row + lane, col0, w.layer, run + g * kCols);
                __syncwarp();  // the previous box has been read back by every lane
                stage_row<OutT>(box, lane, run + g * kCols);
                __syncwarp();
                const int64_t col = col0 + c;
#pragma unroll 4
                for (int r0 = 0; r0 < 32; r0 += kRowsPerStore) {
                    const int r = r0 + lane / kCols;
                    const int64_t row = warp_row + r;
                    const int off = r * 64 + (((cbyte >> 4) ^ ((r >> 1) & 3)) << 4) + (cbyte & 15);
                    if (row < p.M && col < p.N) base[row * p.ldo + col] = *reinterpret_cast<const OutT*>(box + off);
                }
            }
        }
    }
    // the staging buffer must not be released while the TMA still reads it
    if (p.tma_store && lane == 0) ptx::bulk_wait_read_all();
}

// -------------------------------------------------------------------------
// Single-SM kernel: 128 x BN tiles, UMMA 128 x BN x 16.
// -------------------------------------------------------------------------
template <int BN, int STAGES, typename OutT, bool F8>
__global__ void __launch_bounds__(block_threads(BN), 1)
sfc_gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                const __grid_constant__ CUtensorMap tmap_c, const GemmParams p) {
    static_assert(BN == 128 || BN == 256, "tiles are 128 x 128 or 128 x 256");
    using I = InKind<F8>;
    constexpr int kABytes = kBM * 128;  // 128-byte rows
    constexpr int kBBytes = BN * 128;
    constexpr int kStageBytes = kABytes + kBBytes;
    constexpr int kEpiWarps = BN / 32;
    using L = RingLayout<kStageBytes, STAGES, kEpiWarps>;
    constexpr uint32_t kTmemCols = 2 * BN;

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

    ItemSource src;
    worker_items(p, blockIdx.x, gridDim.x, src.first, src.end, src.step);
    src.worker = blockIdx.x;
    src.workers = gridDim.x;
    src.dynamic = p.dynamic;
    src.q_full0 = B.q_full(0);
    src.q_empty0 = B.q_empty(0);
    src.q_entry = reinterpret_cast<volatile int*>(smem + L::kQueueOffset);
    // the first item needs no memory at all: the scheduler thread decodes it into the
    // queue's slot 0 while the other warps set up (every role reads it after the barrier)
    const bool sched_thread = (warp == scheduler_warp(BN) && lane == 0);
    int item0 = -1;
    if (sched_thread) {
        item0 = sched_next(src, 0, p);
        sched_local_first(src, sched_entry(item0, p));
    }

    if (threadIdx.x == 0) {
        ptx::pdl_launch_dependents();
        for (int s = 0; s < STAGES; ++s) {
            ptx::mbar_init(B.full(s), 1);
            ptx::mbar_init(B.empty(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            ptx::mbar_init(B.acc_full(a), 1);
            ptx::mbar_init(B.acc_empty(a), kEpiWarps);  // one arrive per epilogue warp
        }
        ptx::mbar_init(B.drain(), 1);
        ptx::mbar_init(B.never(), 1);
        for (int q = 0; q < kQueue; ++q) {
            ptx::mbar_init(B.q_full(q), 1);               // the scheduler publishes
            ptx::mbar_init(B.q_empty(q), 2 + kEpiWarps);  // producer, MMA warp and epilogue warps have read
        }
        ptx::mbar_init(B.q_taken(), 1);  // the producer took an item
        *abort_flag = 0;
        ptx::fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        ptx::tma_prefetch_desc(&tmap_a);
        ptx::tma_prefetch_desc(&tmap_b);
        if (p.tma_store) ptx::tma_prefetch_desc(&tmap_c);
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_addr(tmem_slot), kTmemCols);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    if (sched_thread) sched_mark_first(src, 1);
    ptx::pdl_wait();  // on-chip set-up above overlaps the previous kernel; global memory only after it

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            int64_t issued = 0;
            bool ok = produce<STAGES>(src, p, B, abort_flag, /*signal_taken=*/true, issued,
                                      [&](const WorkItem& w, int kt, int stage) {
                ptx::mbar_arrive_expect_tx(B.full(stage), kStageBytes);
                const uint32_t sa = ring + stage * kStageBytes;
                const uint32_t sb = sa + kABytes;
                ptx::tma_load_2d(sa, &tmap_a, B.full(stage), kt * I::kSlabK, w.tm * kBM);
                if (p.b_kmajor) {
                    // B^T rows (N) x one slab of k, K-major like A
                    ptx::tma_load_2d(sb, &tmap_b, B.full(stage), kt * I::kSlabK, w.tn * BN);
                } else {
#pragma unroll
                    for (int jb = 0; jb < BN / I::kBCols; ++jb)
                        ptx::tma_load_2d(sb + jb * I::kBBoxBytes, &tmap_b, B.full(stage), w.tn * BN + jb * I::kBCols,
                                         kt * I::kSlabK);
                }
            });
            // Tail: the last STAGES issues.  On success wait until the MMA warp's
            // commits have released them (no arrive may land after exit); after a
            // failure wait (bounded) for the copies still in flight into the ring.
            const int64_t n0 = issued > STAGES ? issued - STAGES : 0;
            for (int64_t n = n0; n < issued; ++n) {
                const int slot = static_cast<int>(n % STAGES);
                const uint32_t par = static_cast<uint32_t>((n / STAGES) & 1);
                if (ok) ok = wait_bounded(B.empty(slot), par, abort_flag, p.timeout_ns, kWaitProducerEmpty);
                if (!ok)
                    wait_bounded(B.full(slot), par, abort_flag, p.timeout_ns, kWaitDrain, /*honour_abort=*/false);
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
            const uint32_t idesc = ptx::idesc_f32(kBM, BN, /*A K-major*/ 0, p.b_kmajor ? 0u : 1u, p.ab_fmt);
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
                        const uint32_t sa = ring + stage * kStageBytes;
                        const uint32_t sb = sa + kABytes;
                        // A: K-major, 128-byte rows, 8-row atoms 1024 B apart; 32 B per instruction.
                        // B N-major: 128-byte-wide boxes one box apart, 8-row atoms 1 KB apart, kMmaK
                        // rows per instruction; B K-major: as A.  Later instructions of the slab step
                        // the start-address field (16-byte units, bits 0-13; the ring lies below
                        // 256 KB, so the field never carries).
                        const uint64_t adesc = ptx::smem_desc_sw128(sa, 16, 1024);
                        const uint64_t bdesc = p.b_kmajor ? ptx::smem_desc_sw128(sb, 16, 1024)
                                                          : ptx::smem_desc_sw128(sb, I::kBBoxBytes, 1024);
                        const uint32_t bstep = p.b_kmajor ? 2u : (I::kMmaK * 128) / 16;
#pragma unroll
                        for (int kk = 0; kk < I::kSlabK / I::kMmaK; ++kk)
                            ptx::tc_mma<F8>(d_tmem, adesc + 2u * kk, bdesc + bstep * kk, idesc,
                                            (q > kb || kk > 0) ? 1u : 0u);
                        ptx::tc_commit(B.empty(stage));  // frees the stage once these MMAs finish
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (!ok) break;
                    ptx::tc_commit(B.acc_full(acc));  // chunk ready for the epilogue
                    if (++acc == 2) {
                        acc = 0;
                        acc_phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                // wait (bounded) until every MMA issued so far has finished
                ptx::tc_commit(B.drain());
                wait_bounded(B.drain(), 0, abort_flag, p.timeout_ns, kWaitDrain, /*honour_abort=*/false);
            }
        }
    } else if (warp < scheduler_warp(BN)) {
        run_epilogue<BN, OutT, false>(p, B, tmem_base, abort_flag, src, kBM, 0, warp, lane, &tmap_c,
                                      smem + L::kStagingOffset);
    } else if (sched_thread) {
        // -------------------------------------------------------- scheduler
        run_scheduler(src, item0, p, B, abort_flag, 1);
    }

    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    if (warp == 1) ptx::tmem_dealloc(tmem_base, kTmemCols);
}

// C = cvt(sum_{l=0}^{c-1} P_l), summed in layer order, 4 columns per thread.
// P_l rows are `ldw` floats apart (ldw % 4 == 0), layers `layer_stride` apart.
// Then, if asked, C = that + beta * C_in + bias (C_in is C read first).
template <typename OutT>
__global__ void __launch_bounds__(256)
ca_reduce_kernel(const float* __restrict__ ws, int64_t ldw, int64_t layer_stride, int c, int64_t M,
                 int64_t N, OutT* __restrict__ C, int64_t ldc, int vec_store, float beta,
                 const float* __restrict__ bias) {
    ptx::pdl_launch_dependents();
    ptx::pdl_wait();  // the partials come from the GEMM kernel just before
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
        if (beta != 0.0f || bias) {
            float v[4] = {acc.x, acc.y, acc.z, acc.w};
            for (int h = 0; h < 4 && j + h < N; ++h) {
                if (beta != 0.0f) v[h] = __fmaf_rn(beta, static_cast<float>(dst[h]), v[h]);
                if (bias) v[h] = __fadd_rn(v[h], bias[j + h]);
            }
            acc = make_float4(v[0], v[1], v[2], v[3]);
        }
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

// Row-major copy of a rows x cols matrix of `elem`-byte values (2 or 1) into a
// buffer whose rows are 16-byte aligned (row stride ld_dst), for inputs whose
// own rows or base are not: the tile loads need 16-byte-aligned rows.
__global__ void __launch_bounds__(256)
pack_rows_kernel(const uint8_t* __restrict__ src, int64_t ld_src, int64_t rows, int64_t cols, int elem,
                 uint8_t* __restrict__ dst, int64_t ld_dst) {
    const int64_t total = rows * cols;
    for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t r = idx / cols;
        const int64_t c = idx - r * cols;
        if (elem == 2)
            reinterpret_cast<uint16_t*>(dst)[r * ld_dst + c] = reinterpret_cast<const uint16_t*>(src)[r * ld_src + c];
        else
            dst[r * ld_dst + c] = src[r * ld_src + c];
    }
}

// Clears `bits` of the device error word (after the host has read them).
__global__ void status_clear_kernel(unsigned int bits) { atomicAnd(&g_sfc_status, ~bits); }

// out[s] = tm * Nt + tn for every curve position s, with the kernels' decoder.
__global__ void tile_order_kernel(int Mt, int Nt, int32_t* __restrict__ out) {
    const int64_t n = static_cast<int64_t>(Mt) * Nt;
    for (int64_t s = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; s < n;
         s += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const TileCoord t = curve_decode(static_cast<int>(s), Mt, Nt);
        out[s] = t.tm * Nt + t.tn;
    }
}

}  // namespace sfc
