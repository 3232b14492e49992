// sfc_host.cpp -- the host-buffer entry point (sfc_gemm_host): C = A * B with
// A, B and C in host memory, the host<->device copies pipelined against the
// tile contraction.
//
// The output is cut into panels along the dimension of the larger operand
// (rows of C when A is at least as large as B, else columns).  The smaller
// operand is uploaded whole, then each panel's slice of the larger one; the
// GEMM of panel p starts as soon as its slice has arrived and its slice of C
// is copied back while panel p + 1 computes.  Panel edges fall on multiples
// of the largest output tile, so every output tile is contracted exactly as a
// single sfc_gemm_ex2 call over the whole problem with the same tile and layer
// count would contract it: the results are bit-identical.
//
// Streams: uploads run on a library stream `up`, downloads on `down`, the
// GEMMs on the caller's stream, ordered by events.  Device memory comes from
// staging slots owned by the library: a slot holds one call's device copies of
// A, B and C and is reused once the event recorded at the end of that call has
// completed, so calls issued back to back overlap (the next call's uploads
// proceed while this call computes).  sfc_release frees the slots.
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
constexpr int kMaxPanels = 64;
constexpr int64_t kPanelRowsM = 512;    // rows of the largest output tile (two stacked 2-SM pairs)
constexpr int64_t kPanelColsN = 256;    // columns of the widest output tile
constexpr int64_t kAutoPanelSpan = 2048;  // automatic panels: about this many rows or columns each
constexpr int kAutoMaxPanels = 8;

int fail(cudaError_t e) { return sfc::cuda_fail(e); }

struct Slot {
    void* base = nullptr;
    size_t bytes = 0;
    cudaEvent_t done = nullptr;  // recorded on the caller's stream after the call's last use
    bool recorded = false;
    bool taken = false;          // reserved by a call that is still enqueueing
};

struct Pipe {
    std::mutex mu;
    bool ready = false;
    cudaStream_t up = nullptr, down = nullptr;
    std::vector<Slot> slots;
    size_t held = 0, cap = 0;
};

Pipe g_pipe[kMaxDevices];

int64_t round_up(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// Per-device streams and the staging budget (half the memory free at first use).
int pipe_setup(Pipe& p) {
    if (p.ready) return SFC_OK;
    cudaError_t e = cudaStreamCreateWithFlags(&p.up, cudaStreamNonBlocking);
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

    // panels along M when A is at least as large as B, else along N
    const bool by_rows = M >= N;
    const int64_t extent = by_rows ? M : N, unit = by_rows ? kPanelRowsM : kPanelColsN;
    const int64_t units = (extent + unit - 1) / unit;
    int64_t np = panels;
    if (np == 0) {
        np = (extent + kAutoPanelSpan - 1) / kAutoPanelSpan;
        if (np > kAutoMaxPanels) np = kAutoMaxPanels;
    }
    if (np > units) np = units;
    if (np > kMaxPanels) np = kMaxPanels;
    if (np < 1) np = 1;
    const int64_t per = (units + np - 1) / np * unit;  // panel span, a multiple of the tile
    np = (extent + per - 1) / per;

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

    Events evs;
    std::vector<cudaEvent_t> computed;
    // the operand every panel needs goes up first
    if (by_rows)
        e = copy_rows(Bd, ldb_d * eb, Bh, ldb * eb, b_cols * eb, b_rows, cudaMemcpyHostToDevice, p.up);
    else
        e = copy_rows(Ad, lda_d * eb, Ah, lda * eb, K * eb, M, cudaMemcpyHostToDevice, p.up);
    for (int64_t i = 0; i < np && e == cudaSuccess && rc == SFC_OK; ++i) {
        const int64_t lo = i * per, hi = (lo + per < extent) ? lo + per : extent;
        const void *a = Ad, *b = Bd;
        void* c = Cd;
        int64_t m = M, n = N;
        if (by_rows) {
            e = copy_rows(Ad + lo * lda_d * eb, lda_d * eb, Ah + lo * lda * eb, lda * eb, K * eb, hi - lo,
                          cudaMemcpyHostToDevice, p.up);
            a = Ad + lo * lda_d * eb;
            c = Cd + lo * ldc_d * ob;
            m = hi - lo;
        } else if (b_nk) {
            e = copy_rows(Bd + lo * ldb_d * eb, ldb_d * eb, Bh + lo * ldb * eb, ldb * eb, K * eb, hi - lo,
                          cudaMemcpyHostToDevice, p.up);
            b = Bd + lo * ldb_d * eb;
            c = Cd + lo * ob;
            n = hi - lo;
        } else {
            e = copy_rows(Bd + lo * eb, ldb_d * eb, Bh + lo * eb, ldb * eb, (hi - lo) * eb, K,
                          cudaMemcpyHostToDevice, p.up);
            b = Bd + lo * eb;
            c = Cd + lo * ob;
            n = hi - lo;
        }
        if (e == cudaSuccess) e = join(s, p.up, evs);
        if (e != cudaSuccess) break;
        rc = sfc_gemm_ex2(m, n, K, a, b, c, lda_d, ldb_d, ldc_d, ab_dtype, b_layout, 0.0f, nullptr, c_used,
                          c_dtype, SFC_ORDER_SFC, SFC_ASSIGN_AUTO, static_cast<sfc_tile_t>(tile_used), nullptr, 0,
                          stream);
        if (rc != SFC_OK) break;
        cudaEvent_t done;
        e = evs.make(&done);
        if (e == cudaSuccess) e = cudaEventRecord(done, s);
        if (e == cudaSuccess) computed.push_back(done);
    }
    // downloads are enqueued after every GEMM, so a blocking copy into pageable memory cannot hold one back
    for (size_t i = 0; i < computed.size() && e == cudaSuccess; ++i) {
        const int64_t lo = static_cast<int64_t>(i) * per, hi = (lo + per < extent) ? lo + per : extent;
        e = cudaStreamWaitEvent(p.down, computed[i], 0);
        if (e != cudaSuccess) break;
        if (by_rows)
            e = copy_rows(Ch + lo * ldc * ob, ldc * ob, Cd + lo * ldc_d * ob, ldc_d * ob, N * ob, hi - lo,
                          cudaMemcpyDeviceToHost, p.down);
        else
            e = copy_rows(Ch + lo * ob, ldc * ob, Cd + lo * ob, ldc_d * ob, (hi - lo) * ob, M,
                          cudaMemcpyDeviceToHost, p.down);
    }
    // the caller's stream ends after everything this call enqueued; the slot is free after that
    cudaError_t j = join(s, p.up, evs);
    if (j == cudaSuccess) j = join(s, p.down, evs);
    if (j == cudaSuccess) j = cudaEventRecord(p.slots[si].done, s);
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
