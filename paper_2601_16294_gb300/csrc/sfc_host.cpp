// sfc_host.cpp -- the host-buffer entry point (sfc_gemm_host): C = A * B with
// A, B and C in host memory, the host<->device copies pipelined against the
// tile contraction.
//
// A is cut into row panels and B into column panels.  The uploads follow a
// staircase: after the first panel of each, the next upload is the panel that
// keeps the rows and columns covered so far closest to equal, and each upload
// is followed by the GEMM of the strip of C it completes (the new rows against
// every column present, or the new columns against every row present).  The
// GEMMs thus start after two panels instead of a whole operand, and C's
// strips go back while later strips compute.  This is the idea of the curve
// order one level up: the output is grown so that what is already resident
// (here in device memory, behind the host link) is reused as much as possible
// per byte moved.  Panel edges fall on multiples of the largest output tile,
// so every output tile is contracted exactly as a single sfc_gemm_ex2 call
// over the whole problem with the same tile and layer count would contract it:
// the results are bit-identical.
//
// Streams: uploads run on a library stream `up`, GEMMs on `comp`, downloads
// on `down`, ordered by events; the caller's stream only waits for the call's
// last download.  The GEMMs read and write staging memory alone, so they need
// no order against the caller's earlier work, and the next call's GEMMs do not
// wait for this call's downloads: consecutive calls overlap their GEMMs, their
// uploads and their downloads.  Device memory comes from staging slots owned
// by the library: a slot holds one call's device copies of A, B and C and is
// reused once the event recorded after that call's last download has
// completed.  sfc_release frees the slots.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>
#include <vector>

#include "sfc_gemm.h"
#include "sfc_internal.h"

#define SFC_API extern "C" __attribute__((visibility("default")))

namespace sfc_host {
namespace {

constexpr int kMaxDevices = 64;
constexpr int64_t kMaxPanels = 64;
constexpr int64_t kPanelRowsM = 512;    // a multiple of the rows of every output tile (256 at most)
constexpr int64_t kPanelColsN = 256;    // columns of the widest output tile
constexpr int64_t kAutoPanelSpan = 2048;  // automatic panels: about this many rows or columns each
constexpr int64_t kAutoMaxPanels = 8;  // panels of the automatic span before the span grows
// Pitched host<->device copies run below the link's rate for short rows
// (measured on GB300: 2 KB rows 128 GB/s, 4 KB 175, 8 KB 188, 16 KB and up 211).
constexpr int64_t kMinPitchedRowBytes = 8192;

int fail(cudaError_t e) { return sfc::cuda_fail(e); }

struct Slot {
    void* base = nullptr;
    size_t bytes = 0;
    cudaEvent_t done = nullptr;  // recorded after the call's last download
    bool recorded = false;
    bool taken = false;          // reserved by a call that is still enqueueing
};

struct Pipe {
    std::mutex mu;
    bool ready = false;
    cudaStream_t up = nullptr, comp = nullptr, down = nullptr;
    std::vector<Slot> slots;
    size_t held = 0, cap = 0;
};

Pipe g_pipe[kMaxDevices];

int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// Per-device streams and the staging budget (half the memory free at first use).
int pipe_setup(Pipe& p) {
    if (p.ready) return SFC_OK;
    cudaError_t e = cudaStreamCreateWithFlags(&p.up, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p.comp, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&p.down, cudaStreamNonBlocking);
    size_t free_b = 0, total_b = 0;
    if (e == cudaSuccess) e = cudaMemGetInfo(&free_b, &total_b);
    if (e != cudaSuccess) return fail(e);
    p.cap = free_b / 2;
    p.ready = true;
    return SFC_OK;
}

bool slot_idle(Slot& s, cudaError_t* err) {
    *err = cudaSuccess;
    if (s.taken) return false;
    if (!s.recorded) return true;
    cudaError_t q = cudaEventQuery(s.done);
    if (q == cudaSuccess) return true;
    if (q != cudaErrorNotReady) *err = q;
    return false;
}

int free_slot(Pipe& p, size_t i) {
    Slot& s = p.slots[i];
    cudaError_t e = cudaSuccess;
    if (s.recorded) e = cudaEventSynchronize(s.done);
    if (e == cudaSuccess && s.base) e = cudaFree(s.base);
    if (e == cudaSuccess && s.done) e = cudaEventDestroy(s.done);
    if (e != cudaSuccess) return fail(e);
    p.held -= s.bytes;
    p.slots.erase(p.slots.begin() + static_cast<std::ptrdiff_t>(i));
    return SFC_OK;
}

// Reserve a slot of at least `need` bytes: the smallest idle one that fits;
// else a new one within the budget; else (rare) wait for the slots in use,
// free them all and allocate exactly.  Caller holds p.mu.
int acquire(Pipe& p, size_t need, size_t* out) {
    size_t best = p.slots.size();
    for (size_t i = 0; i < p.slots.size(); ++i) {
        cudaError_t err;
        if (!slot_idle(p.slots[i], &err)) {
            if (err != cudaSuccess) return fail(err);
            continue;
        }
        if (p.slots[i].bytes >= need && (best == p.slots.size() || p.slots[i].bytes < p.slots[best].bytes)) best = i;
    }
    if (best == p.slots.size()) {
        if (p.held + need > p.cap) {
            for (size_t i = p.slots.size(); i-- > 0;) {
                if (p.slots[i].taken) continue;
                int rc = free_slot(p, i);
                if (rc != SFC_OK) return rc;
            }
        }
        Slot s;
        s.bytes = need;
        cudaError_t e = cudaMalloc(&s.base, need);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&s.done, cudaEventDisableTiming);
        if (e != cudaSuccess) {
            if (s.base) cudaFree(s.base);
            return fail(e);
        }
        p.slots.push_back(s);
        p.held += need;
        best = p.slots.size() - 1;
    }
    p.slots[best].taken = true;
    *out = best;
    return SFC_OK;
}

// Output rows [r0, r1) x columns [c0, c1) computed by one GEMM.
struct Region {
    int64_t r0, r1, c0, c1;
};

// Panel edges [0, e_1, ..., extent] along a dimension, every inner edge a
// multiple of `unit`.  `panels` > 0: that many equal panels (at most
// kMaxPanels, at most one per unit).  0: panels of about `auto_span` elements
// (more when that would make over kAutoMaxPanels of them); with `ramp`, the
// first two and the last two are a quarter and a half of that, so that the
// first GEMM starts after little data has arrived and the last leaves little
// to do after the final upload (not for pitched copies, whose short rows
// would slow the link down).
std::vector<int64_t> panel_edges(int64_t extent, int64_t unit, int panels, int64_t auto_span, bool ramp_ok) {
    const int64_t units = (extent + unit - 1) / unit;
    std::vector<int64_t> sizes;  // in units
    if (panels > 0) {
        int64_t np = panels;
        if (np > kMaxPanels) np = kMaxPanels;
        if (np > units) np = units;
        const int64_t per = (units + np - 1) / np;
        for (int64_t done = 0; done < units; done += per) sizes.push_back(per < units - done ? per : units - done);
    } else {
        int64_t mid = auto_span / unit;
        if (mid < 1) mid = 1;
        const int64_t spread = (units + kAutoMaxPanels - 1) / kAutoMaxPanels;
        if (mid < spread) mid = spread;
        const int64_t q = mid / 4 > 0 ? mid / 4 : 1, h = mid / 2 > 0 ? mid / 2 : 1;
        int64_t rest = units;
        const bool ramp = ramp_ok && units > 2 * (q + h) + 2 * mid;
        if (ramp) {
            sizes.push_back(q);
            sizes.push_back(h);
            rest -= 2 * (q + h);
        }
        while (rest > 0) {
            const int64_t sz = mid < rest ? mid : rest;
            sizes.push_back(sz);
            rest -= sz;
        }
        if (ramp) {
            sizes.push_back(h);
            sizes.push_back(q);
        }
    }
    std::vector<int64_t> edges{0};
    int64_t at = 0;
    for (int64_t sz : sizes) {
        at += sz;
        edges.push_back(at * unit < extent ? at * unit : extent);
    }
    return edges;
}

// Row-major copy of `rows` rows of `width` bytes between pitched buffers.
cudaError_t copy_rows(void* dst, int64_t dpitch, const void* src, int64_t spitch, int64_t width, int64_t rows,
                      cudaMemcpyKind kind, cudaStream_t s) {
    if (dpitch == width && spitch == width)
        return cudaMemcpyAsync(dst, src, static_cast<size_t>(width * rows), kind, s);
    return cudaMemcpy2DAsync(dst, static_cast<size_t>(dpitch), src, static_cast<size_t>(spitch),
                             static_cast<size_t>(width), static_cast<size_t>(rows), kind, s);
}

struct Events {
    std::vector<cudaEvent_t> ev;
    ~Events() {
        for (cudaEvent_t e : ev) cudaEventDestroy(e);  // released by the driver once completed
    }
    cudaError_t make(cudaEvent_t* e) {
        cudaError_t r = cudaEventCreateWithFlags(e, cudaEventDisableTiming);
        if (r == cudaSuccess) ev.push_back(*e);
        return r;
    }
};

// s waits for the work enqueued on `on` so far.
cudaError_t join(cudaStream_t s, cudaStream_t on, Events& evs) {
    cudaEvent_t e;
    cudaError_t r = evs.make(&e);
    if (r == cudaSuccess) r = cudaEventRecord(e, on);
    if (r == cudaSuccess) r = cudaStreamWaitEvent(s, e, 0);
    return r;
}

}  // namespace
}  // namespace sfc_host

using namespace sfc_host;

SFC_API int sfc_gemm_host(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda,
                          int64_t ldb, int64_t ldc, int ab_dtype, int b_layout, int ca_c, sfc_dtype_t c_dtype,
                          sfc_tile_t tile, int panels, void* stream) {
    // argument checks that need no device come first
    if (M <= 0 || N <= 0 || K <= 0 || !A || !B || !C) return SFC_ERR_INVALID_ARG;
    if (ab_dtype != SFC_AB_BF16 && ab_dtype != SFC_AB_E4M3 && ab_dtype != SFC_AB_E5M2) return SFC_ERR_INVALID_ARG;
    if (b_layout != SFC_B_KN && b_layout != SFC_B_NK) return SFC_ERR_INVALID_ARG;
    if (c_dtype != SFC_F32 && c_dtype != SFC_BF16) return SFC_ERR_INVALID_ARG;
    const bool b_nk = (b_layout == SFC_B_NK);
    if (lda < K || ldb < (b_nk ? K : N) || ldc < N || panels < 0) return SFC_ERR_INVALID_ARG;
    const int64_t eb = (ab_dtype == SFC_AB_BF16) ? 2 : 1;
    const int64_t ob = (c_dtype == SFC_F32) ? 4 : 2;
    const uintptr_t ea = static_cast<uintptr_t>(eb) - 1u, oa = static_cast<uintptr_t>(ob) - 1u;
    if ((reinterpret_cast<uintptr_t>(A) & ea) || (reinterpret_cast<uintptr_t>(B) & ea) ||
        (reinterpret_cast<uintptr_t>(C) & oa))
        return SFC_ERR_UNALIGNED;

    // one plan for the whole problem (validates sizes, ca_c and tile), used by every panel
    int tile_used = 0, c_used = 0;
    int rc = sfc_gemm_plan(M, N, K, ca_c, c_dtype, tile, ab_dtype, b_layout, &tile_used, &c_used);
    if (rc != SFC_OK) return rc;

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(e);
    if (dev < 0 || dev >= kMaxDevices) return SFC_ERR_UNSUPPORTED;
    Pipe& p = g_pipe[dev];
    cudaStream_t s = static_cast<cudaStream_t>(stream);

    // device copies with 16-byte rows
    const int64_t lda_d = round_up(K * eb, 16) / eb;
    const int64_t b_rows = b_nk ? N : K, b_cols = b_nk ? K : N;
    const int64_t ldb_d = round_up(b_cols * eb, 16) / eb;
    const int64_t ldc_d = round_up(N * ob, 16) / ob;
    const size_t a_bytes = static_cast<size_t>(round_up(M * lda_d * eb, 256));
    const size_t b_bytes = static_cast<size_t>(round_up(b_rows * ldb_d * eb, 256));
    const size_t c_bytes = static_cast<size_t>(round_up(M * ldc_d * ob, 256));

    // row panels of A (multiples of 512 rows) and column panels of B (multiples of 256 columns)
    // a column panel of an N-major B is a pitched copy: keep its rows at least 8 KB long
    const int64_t col_span = b_nk ? kAutoPanelSpan : (kMinPitchedRowBytes / eb > kAutoPanelSpan
                                                         ? kMinPitchedRowBytes / eb : kAutoPanelSpan);
    // row panels of A (and of a K-major B) copy rows of K values: ramp them when those rows are
    // contiguous or long
    const bool k_rows_fast = K * eb >= kMinPitchedRowBytes;
    const std::vector<int64_t> em =
        panel_edges(M, kPanelRowsM, panels, kAutoPanelSpan, k_rows_fast || (lda == K && lda_d == K));
    const std::vector<int64_t> en =
        panel_edges(N, kPanelColsN, panels, col_span, b_nk && (k_rows_fast || (ldb == K && ldb_d == K)));
    const int64_t pm = static_cast<int64_t>(em.size()) - 1, pn = static_cast<int64_t>(en.size()) - 1;
    auto row_end = [&](int64_t i) { return em[static_cast<size_t>(i)]; };
    auto col_end = [&](int64_t j) { return en[static_cast<size_t>(j)]; };

    std::lock_guard<std::mutex> lock(p.mu);
    rc = pipe_setup(p);
    if (rc != SFC_OK) return rc;
    size_t si = 0;
    rc = acquire(p, a_bytes + b_bytes + c_bytes, &si);
    if (rc != SFC_OK) return rc;
    char* base = static_cast<char*>(p.slots[si].base);
    char* Ad = base;
    char* Bd = base + a_bytes;
    char* Cd = base + a_bytes + b_bytes;
    const char* Ah = static_cast<const char*>(A);
    const char* Bh = static_cast<const char*>(B);
    char* Ch = static_cast<char*>(C);

    auto upload_a = [&](int64_t i) {
        const int64_t r0 = row_end(i), r1 = row_end(i + 1);
        return copy_rows(Ad + r0 * lda_d * eb, lda_d * eb, Ah + r0 * lda * eb, lda * eb, K * eb, r1 - r0,
                         cudaMemcpyHostToDevice, p.up);
    };
    auto upload_b = [&](int64_t j) {
        const int64_t c0 = col_end(j), c1 = col_end(j + 1);
        if (b_nk)
            return copy_rows(Bd + c0 * ldb_d * eb, ldb_d * eb, Bh + c0 * ldb * eb, ldb * eb, K * eb, c1 - c0,
                             cudaMemcpyHostToDevice, p.up);
        return copy_rows(Bd + c0 * eb, ldb_d * eb, Bh + c0 * eb, ldb * eb, (c1 - c0) * eb, K,
                         cudaMemcpyHostToDevice, p.up);
    };

    Events evs;
    std::vector<Region> regions;
    std::vector<cudaEvent_t> computed;
    // GEMM of the block of C that the panels uploaded so far newly cover
    auto compute = [&](Region g) -> cudaError_t {
        cudaError_t r = join(p.comp, p.up, evs);
        if (r != cudaSuccess) return r;
        const char* a = Ad + g.r0 * lda_d * eb;
        const char* b = b_nk ? Bd + g.c0 * ldb_d * eb : Bd + g.c0 * eb;
        char* c = Cd + g.r0 * ldc_d * ob + g.c0 * ob;
        rc = sfc_gemm_ex2(g.r1 - g.r0, g.c1 - g.c0, K, a, b, c, lda_d, ldb_d, ldc_d, ab_dtype, b_layout, 0.0f,
                          nullptr, c_used, c_dtype, SFC_ORDER_SFC, SFC_ASSIGN_AUTO,
                          static_cast<sfc_tile_t>(tile_used), nullptr, 0, p.comp);
        if (rc != SFC_OK) return cudaSuccess;
        cudaEvent_t done;
        r = evs.make(&done);
        if (r == cudaSuccess) r = cudaEventRecord(done, p.comp);
        if (r == cudaSuccess) {
            regions.push_back(g);
            computed.push_back(done);
        }
        return r;
    };

    // Staircase walk: after the first row and column panel, upload whichever
    // panel keeps the covered rows and columns closest to equal (most output
    // per uploaded byte), and compute the strip of C it completes.
    e = upload_a(0);
    if (e == cudaSuccess) e = upload_b(0);
    if (e == cudaSuccess) e = compute(Region{0, row_end(1), 0, col_end(1)});
    int64_t a = 1, b = 1;
    while (e == cudaSuccess && rc == SFC_OK && (a < pm || b < pn)) {
        const bool take_a = b >= pn || (a < pm && row_end(a) <= col_end(b));
        if (take_a) {
            e = upload_a(a);
            if (e == cudaSuccess) e = compute(Region{row_end(a), row_end(a + 1), 0, col_end(b)});
            ++a;
        } else {
            e = upload_b(b);
            if (e == cudaSuccess) e = compute(Region{0, row_end(a), col_end(b), col_end(b + 1)});
            ++b;
        }
    }
    // downloads are enqueued after every GEMM, so a blocking copy into pageable memory cannot hold one back
    for (size_t i = 0; i < computed.size() && e == cudaSuccess; ++i) {
        const Region& g = regions[i];
        e = cudaStreamWaitEvent(p.down, computed[i], 0);
        if (e == cudaSuccess)
            e = copy_rows(Ch + g.r0 * ldc * ob + g.c0 * ob, ldc * ob, Cd + g.r0 * ldc_d * ob + g.c0 * ob, ldc_d * ob,
                          (g.c1 - g.c0) * ob, g.r1 - g.r0, cudaMemcpyDeviceToHost, p.down);
    }
    // the slot is free, and the caller's stream may go on, after everything
    // this call enqueued (downloads wait for their GEMMs, GEMMs for their
    // uploads; the joins also cover a call that stopped early)
    cudaError_t j = join(p.down, p.up, evs);
    if (j == cudaSuccess) j = join(p.down, p.comp, evs);
    if (j == cudaSuccess) j = cudaEventRecord(p.slots[si].done, p.down);
    if (j == cudaSuccess) j = cudaStreamWaitEvent(s, p.slots[si].done, 0);
    Slot& slot = p.slots[si];
    slot.taken = false;
    if (j == cudaSuccess) {
        slot.recorded = true;
    } else {
        // nothing orders the slot's reuse: drain the device before it can be taken again
        cudaDeviceSynchronize();
        slot.recorded = false;
    }
    if (rc != SFC_OK) return rc;
    if (e != cudaSuccess) return fail(e);
    if (j != cudaSuccess) return fail(j);
    return SFC_OK;
}

namespace sfc {

int host_release_staging() {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(e);
    if (dev < 0 || dev >= kMaxDevices) return SFC_ERR_UNSUPPORTED;
    Pipe& p = g_pipe[dev];
    std::lock_guard<std::mutex> lock(p.mu);
    for (size_t i = p.slots.size(); i-- > 0;) {
        if (p.slots[i].taken) continue;
        int rc = free_slot(p, i);
        if (rc != SFC_OK) return rc;
    }
    return SFC_OK;
}

}  // namespace sfc
