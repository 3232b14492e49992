// sfc_gemm.cu -- host side of the SFC GEMM library: argument validation, TMA
// descriptors, launch configuration and the exported C ABI (include/sfc_gemm.h).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>
#include <vector>

#include "sfc_gemm.h"
#include "sfc_gemm_kernel.cuh"
#include "sfc_gemm_pair_kernel.cuh"
#include "sfc_internal.h"

#define SFC_API extern "C" __attribute__((visibility("default")))

namespace sfc {

thread_local int t_last_cuda_error = 0;

int cuda_fail(cudaError_t e) {
    t_last_cuda_error = static_cast<int>(e);
    // the runtime also keeps the error as the thread's last error; the status code reports it, so
    // clear it (a non-sticky error left there would read as the failure of a later, good launch)
    (void)cudaGetLastError();
    return SFC_ERR_CUDA;
}

// Launches check the error cudaLaunchKernelEx returns, never cudaGetLastError (which could hold
// an earlier, unrelated failure of the caller's).
template <typename... Params, typename... Args>
cudaError_t launch_plain(void (*kernel)(Params...), unsigned grid, unsigned block, cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(block, 1, 1);
    cfg.stream = s;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

namespace {

constexpr int kMaxDevices = 64;
constexpr int kMaxLayers = 4096;  // keeps the kernels' layer arithmetic in 32 bits
constexpr int kMaxKBlocks = 64;   // k_block_factor bound (keeps the kernels' pass arithmetic in 32 bits)
constexpr uint64_t kDefaultTimeoutNs = 2000000000ull;  // 2 s per wait

constexpr size_t kTicketBytes = 256;  // one call's ticket allocation (two 64-bit counter words used)
constexpr double kSlabClockGhz = 1.9;     // SM clock the time model's slab times assume
constexpr double kHbmBytesPerNs = 6700.0; // attainable DRAM bandwidth of GB300 (a copy's, GB/s)

// ---------------------------------------------------------- per-device state

// Kernel variants.  Stage counts fill ~192 KB of shared memory per block.
enum Variant { kSingle128 = 0, kSingle256 = 1, kPair128 = 2, kPair256 = 3, kNumVariants = 4 };
constexpr int kStagesSingle256 = 4;  // 48 KB stages
constexpr int kStagesSingle128 = 6;  // 32 KB stages
constexpr int kStagesPair256 = 6;    // 32 KB stages per CTA
constexpr int kStagesPair128 = 8;    // 24 KB stages per CTA
constexpr int kDefaultChunkSlabs = 64;  // 4096 values of k per tensor-memory accumulation chain

constexpr int variant_bn(int v) { return (v == kSingle128 || v == kPair128) ? 128 : 256; }
constexpr bool variant_pair(int v) { return v == kPair128 || v == kPair256; }
constexpr int variant_cluster(int v) { return variant_pair(v) ? 2 : 1; }
constexpr int variant_bm(int v) { return variant_pair(v) ? 256 : 128; }

template <int BN, int STAGES>
constexpr int single_smem() { return RingLayout<(kBM + BN) * 128, STAGES, BN / 32>::kDynamicBytes; }
template <int BN, int STAGES>
constexpr int pair_smem() { return RingLayout<PairStage<BN>::kBytes, STAGES, BN / 32>::kDynamicBytes; }

// Kernel of each variant for one output type and input kind (F8: 8-bit float inputs).
template <typename OutT, bool F8>
struct Kernels {
    using Fn = void (*)(CUtensorMap, CUtensorMap, CUtensorMap, GemmParams);
    static constexpr Fn single128 = sfc_gemm_kernel<128, kStagesSingle128, OutT, F8>;
    static constexpr Fn single256 = sfc_gemm_kernel<256, kStagesSingle256, OutT, F8>;
    static constexpr Fn pair128 = sfc_gemm_pair_kernel<128, kStagesPair128, OutT, F8>;
    static constexpr Fn pair256 = sfc_gemm_pair_kernel<256, kStagesPair256, OutT, F8>;
    static Fn get(int v) {
        switch (v) {
            case kSingle128: return single128;
            case kSingle256: return single256;
            case kPair128: return pair128;
            default: return pair256;
        }
    }
};

constexpr int variant_smem(int v) {
    return v == kSingle128   ? single_smem<128, kStagesSingle128>()
           : v == kSingle256 ? single_smem<256, kStagesSingle256>()
           : v == kPair128   ? pair_smem<128, kStagesPair128>()
                             : pair_smem<256, kStagesPair256>();
}

// attr must hold two entries.  With `pdl` the kernel may begin launching
// while the previous kernel in the stream finishes (programmatic dependent
// launch); the kernels wait for it before touching global memory.
cudaLaunchConfig_t launch_config(int v, int grid, cudaStream_t s, cudaLaunchAttribute* attr, bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(block_threads(variant_bn(v)), 1, 1);
    cfg.dynamicSmemBytes = variant_smem(v);
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 0;
    if (variant_cluster(v) > 1) {
        attr[cfg.numAttrs].id = cudaLaunchAttributeClusterDimension;
        attr[cfg.numAttrs].val.clusterDim.x = variant_cluster(v);
        attr[cfg.numAttrs].val.clusterDim.y = 1;
        attr[cfg.numAttrs].val.clusterDim.z = 1;
        ++cfg.numAttrs;
    }
    if (pdl) {
        attr[cfg.numAttrs].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[cfg.numAttrs].val.programmaticStreamSerializationAllowed = 1;
        ++cfg.numAttrs;
    }
    return cfg;
}

// What the time model needs to know of a device (sfc_gemm_plan_desc takes it from the caller).
struct Machine {
    int workers[kNumVariants] = {0, 0, 0, 0};  // co-resident workers (blocks or clusters) per variant
    double hbm_bytes_per_ns = 0.0;               // attainable DRAM bandwidth (bytes per ns = GB/s)
    double sm_ghz = 0.0;                         // SM clock the tensor-core rate is taken at
};

struct DeviceInfo {
    std::once_flag once;
    int status = SFC_ERR_UNSUPPORTED;
    int num_sms = 0;
    int workers[kNumVariants] = {0, 0, 0, 0};  // co-resident workers (blocks or clusters) per variant
    Machine machine;
    // the library's stream-ordered pool (layer workspaces, repacked operands): it keeps
    // freed memory for reuse, so a call after a synchronisation does not map new pages
    cudaMemPool_t pool = nullptr;
    // ticket counters of the calls (dynamic dealing), from a pool of their own; their
    // words are tagged with the call's epoch, so they need no clearing
    cudaMemPool_t ticket_pool = nullptr;
};
DeviceInfo g_devices[kMaxDevices];

int current_device(int* dev) {
    cudaError_t e = cudaGetDevice(dev);
    if (e != cudaSuccess) return cuda_fail(e);
    if (*dev < 0 || *dev >= kMaxDevices) return SFC_ERR_UNSUPPORTED;
    return SFC_OK;
}

template <typename OutT, bool F8>
cudaError_t set_attrs() {
    for (int v = 0; v < kNumVariants; ++v) {
        cudaError_t e = cudaFuncSetAttribute(Kernels<OutT, F8>::get(v),
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, variant_smem(v));
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// One-time set-up of the current device: check it is an sm_103 part, read its
// SM count, raise the shared-memory limit of every kernel instantiation, and
// find how many 2-SM pairs can be resident at once (clusters must fit in one
// GPC, so this can be fewer than half the SMs).
int device_setup(DeviceInfo** info) {
    int dev;
    int rc = current_device(&dev);
    if (rc != SFC_OK) return rc;
    DeviceInfo& d = g_devices[dev];
    std::call_once(d.once, [&]() {
        cudaDeviceProp prop;
        cudaError_t e = cudaGetDeviceProperties(&prop, dev);
        if (e != cudaSuccess) { d.status = cuda_fail(e); return; }
        if (prop.major != 10 || prop.minor != 3) { d.status = SFC_ERR_UNSUPPORTED; return; }
        d.num_sms = prop.multiProcessorCount;
        e = set_attrs<float, false>();
        if (e == cudaSuccess) e = set_attrs<__nv_bfloat16, false>();
        if (e == cudaSuccess) e = set_attrs<float, true>();
        if (e == cudaSuccess) e = set_attrs<__nv_bfloat16, true>();
        if (e != cudaSuccess) { d.status = cuda_fail(e); return; }
        cudaMemPoolProps props;
        std::memset(&props, 0, sizeof(props));
        props.allocType = cudaMemAllocationTypePinned;
        props.handleTypes = cudaMemHandleTypeNone;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        e = cudaMemPoolCreate(&d.pool, &props);
        uint64_t keep = UINT64_MAX;  // released only by sfc_release
        if (e == cudaSuccess) e = cudaMemPoolSetAttribute(d.pool, cudaMemPoolAttrReleaseThreshold, &keep);
        if (e == cudaSuccess) e = cudaMemPoolCreate(&d.ticket_pool, &props);
        if (e == cudaSuccess) e = cudaMemPoolSetAttribute(d.ticket_pool, cudaMemPoolAttrReleaseThreshold, &keep);
        if (e != cudaSuccess) { d.status = cuda_fail(e); return; }
        for (int v = 0; v < kNumVariants; ++v) {
            if (!variant_pair(v)) {
                d.workers[v] = d.num_sms;
                continue;
            }
            cudaLaunchAttribute attr[2];
            cudaLaunchConfig_t cfg = launch_config(v, d.num_sms, nullptr, attr, false);
            int clusters = 0;
            e = cudaOccupancyMaxActiveClusters(&clusters, Kernels<float, false>::get(v), &cfg);
            if (e != cudaSuccess) { d.status = cuda_fail(e); return; }
            d.workers[v] = clusters;
        }
        for (int v = 0; v < kNumVariants; ++v) d.machine.workers[v] = d.workers[v];
        d.machine.hbm_bytes_per_ns = kHbmBytesPerNs;
        d.machine.sm_ghz = kSlabClockGhz;
        d.status = SFC_OK;
    });
    if (d.status == SFC_OK) *info = &d;
    return d.status;
}

// ------------------------------------------------------------ TMA descriptors

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

int get_encoder(PFN_cuTensorMapEncodeTiled_v12000* fn) {
    std::call_once(g_encode_once, []() {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                                         cudaEnableDefault, &q);
        if (e == cudaSuccess && q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    *fn = g_encode;
    return g_encode ? SFC_OK : SFC_ERR_UNSUPPORTED;
}

// Row-major input matrix (bf16, or 8-bit floats with elem_bytes 1) rows x cols
// with row stride ld (elements), boxes of box_rows x box_cols with 128-byte
// swizzle; out-of-range elements read as 0.
int make_in_map(CUtensorMap* map, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int elem_bytes,
                uint32_t box_rows, uint32_t box_cols) {
    PFN_cuTensorMapEncodeTiled_v12000 encode;
    int rc = get_encoder(&encode);
    if (rc != SFC_OK) return rc;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * elem_bytes};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    const CUtensorMapDataType dt = elem_bytes == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    CUresult r = encode(map, dt, 2, const_cast<void*>(ptr), dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        t_last_cuda_error = static_cast<int>(r);
        return SFC_ERR_CUDA;
    }
    return SFC_OK;
}

// Output map for the staged TMA-store epilogue: 32 x 32 element boxes, swizzled
// to match the staging layout (64-byte rows for bf16, 128-byte rows for fp32).
// layers > 1: a 3-D map (columns, rows, layer) over the workspace copies, so a
// box at the M edge of one layer is clipped instead of spilling into the next.
int make_out_map(CUtensorMap* map, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int elem_bytes,
                 int layers) {
    PFN_cuTensorMapEncodeTiled_v12000 encode;
    int rc = get_encoder(&encode);
    if (rc != SFC_OK) return rc;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows),
                          static_cast<cuuint64_t>(layers)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(ld) * elem_bytes,
                             static_cast<cuuint64_t>(ld) * elem_bytes * static_cast<cuuint64_t>(rows)};
    // boxes of 32 rows x 64 bytes (32 bf16 or 16 fp32 columns), 64-byte swizzle
    cuuint32_t box[3] = {static_cast<cuuint32_t>(64 / elem_bytes), 32, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    const CUtensorMapDataType dt = elem_bytes == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const CUtensorMapSwizzle sw = CU_TENSOR_MAP_SWIZZLE_64B;
    CUresult r = encode(map, dt, layers > 1 ? 3 : 2, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        t_last_cuda_error = static_cast<int>(r);
        return SFC_ERR_CUDA;
    }
    return SFC_OK;
}

// ------------------------------------------------------------------ planning

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// row stride (elements) of the fp32 layer copies of C
int64_t ws_ld(int64_t N) { return (N + 3) / 4 * 4; }

// Planning a call: the tile variant and, when the caller asks for it
// (ca_c = 0), the number of K layers, from a time model in the spirit of the
// paper's fine-grained roofline (Sec. III-B, Eqs. 1-4: a BRGEMM takes
// max(G gamma, beta (S_A + S_B))), written for the GPU's two levels:
//   - on a worker, a slab (the BRGEMM step: 128 x bn x 64 per SM) takes the
//     longer of its MMA time and its operand intake from L2; both are folded
//     into the variant's measured efficiency kEff (one-SM tiles are intake
//     bound, 2-SM 256-wide tiles are not), so the launch's tensor time is
//     waves x (slabs of the longest layer) x slab time, waves = ceil(items /
//     workers);
//   - against DRAM, the launch reads A and B at least once (the curve order
//     keeps the panels of the tiles in flight in L2) and writes C, or for c > 1
//     the c fp32 partial copies of C: the launch takes at least those bytes /
//     DRAM bandwidth, and the longer of the two times is the GEMM's;
//   - for c > 1 the reduction adds its launch and its own DRAM traffic (the c
//     copies read back, C written).
// The tile and layer count with the least time win (ties keep fewer layers).
constexpr double kReduceLaunchNs = 3000.0;   // reduction kernel launch and ramp
// relative tensor-pipe efficiency measured on GB300, back to back at 8192 x
// 8192 x 4096 and 6144^2 x 4096 (256-wide tiles feed the tensor core with fewer
// shared-memory bytes per flop)
constexpr double kEff[kNumVariants] = {0.60, 0.82, 0.62, 0.95};

// Layers ca_c = 0 may choose: enough to give about 320 items of 128 x 128,
// never more than 64 or the number of K slabs (host-only, so the workspace
// bound below needs no device).
// K values per 128-byte slab row: 64 bf16, 128 8-bit floats.
constexpr int slab_k(int ab) { return ab == SFC_AB_BF16 ? kBK : 2 * kBK; }
constexpr int in_bytes(int ab) { return ab == SFC_AB_BF16 ? 2 : 1; }

int64_t auto_layer_cap(int64_t M, int64_t N, int64_t K, int ab = SFC_AB_BF16) {
    const int64_t tiles = ceil_div(M, kBM) * ceil_div(N, 128);
    int64_t cap = ceil_div(320, tiles);
    const int64_t Kt = ceil_div(K, slab_k(ab));
    if (cap > Kt) cap = Kt;
    if (cap > 64) cap = 64;
    return cap < 1 ? 1 : cap;
}

// The model's tensor time and DRAM time of the GEMM launch (the reduction not included).
void gemm_times(int64_t M, int64_t N, int64_t K, int c, int v, const Machine& m, int out_bytes, int ab,
                double* t_tensor_out, double* t_dram_out) {
    const int64_t items = ceil_div(M, variant_bm(v)) * ceil_div(N, variant_bn(v)) * c;
    const int64_t waves = ceil_div(items, m.workers[v]);
    const int64_t slabs = ceil_div(ceil_div(K, slab_k(ab)), c);
    const double slab_ns = 128.0 * variant_bn(v) * kBK * 2.0 / (8192.0 * kEff[v]) / m.sm_ghz;
    *t_tensor_out = static_cast<double>(waves) * static_cast<double>(slabs) * slab_ns;
    const double ab_bytes = in_bytes(ab) * (static_cast<double>(M) * K + static_cast<double>(K) * N);
    const double out_gemm = (c > 1) ? 4.0 * c * static_cast<double>(M) * static_cast<double>(ws_ld(N))
                                    : out_bytes * static_cast<double>(M) * static_cast<double>(N);
    *t_dram_out = (ab_bytes + out_gemm) / m.hbm_bytes_per_ns;
}

double plan_cost(int64_t M, int64_t N, int64_t K, int c, int v, const Machine& m, int out_bytes, int ab) {
    double t_tensor = 0.0, t_dram = 0.0;
    gemm_times(M, N, K, c, v, m, out_bytes, ab, &t_tensor, &t_dram);
    double t = t_tensor > t_dram ? t_tensor : t_dram;
    if (c > 1) {
        t += kReduceLaunchNs + (4.0 * c + out_bytes) * static_cast<double>(M) * static_cast<double>(N) /
                                   m.hbm_bytes_per_ns;
    }
    return t;
}

struct Plan {
    int v;
    int c;
};

// ca_c >= 1: the variant for it; ca_c = 0: the best (variant, c) with c up to
// max_c.  A requested tile fixes the variant (falling back to one SM when
// pairs cannot be co-scheduled).
// Variants that can serve a call: 8-bit N-major B needs 128-byte (128-column)
// boxes per CTA, which the 256 x 128 pair tile (64 columns per CTA) does not have.
bool variant_allowed(int v, bool b_kmajor, int ab) {
    if (v == kPair128 && ab != SFC_AB_BF16 && !b_kmajor) return false;
    return true;
}

Plan make_plan(int64_t M, int64_t N, int64_t K, int ca_c, int max_c, const Machine& d, sfc_tile_t tile,
               int out_bytes, bool b_kmajor = false, int ab = SFC_AB_BF16, double* t_out = nullptr) {
    int fixed = -1;
    if (tile == SFC_TILE_PAIR_N128 && !variant_allowed(kPair128, b_kmajor, ab)) tile = SFC_TILE_N128;
    switch (tile) {
        case SFC_TILE_N128: fixed = kSingle128; break;
        case SFC_TILE_N256: fixed = kSingle256; break;
        case SFC_TILE_PAIR_N128: fixed = d.workers[kPair128] > 0 ? kPair128 : kSingle128; break;
        case SFC_TILE_PAIR_N256: fixed = d.workers[kPair256] > 0 ? kPair256 : kSingle256; break;
        default: break;
    }
    Plan best{fixed >= 0 ? fixed : kSingle128, ca_c > 0 ? ca_c : 1};
    double best_t = -1.0;
    const int c_lo = ca_c > 0 ? ca_c : 1, c_hi = ca_c > 0 ? ca_c : max_c;
    for (int v = 0; v < kNumVariants; ++v) {
        if (d.workers[v] <= 0 || (fixed >= 0 && v != fixed) || !variant_allowed(v, b_kmajor, ab)) continue;
        for (int c = c_lo; c <= c_hi; ++c) {
            const double t = plan_cost(M, N, K, c, v, d, out_bytes, ab);
            if (best_t < 0.0 || t < best_t) {  // ties keep fewer layers, then the earlier variant
                best = Plan{v, c};
                best_t = t;
            }
        }
    }
    if (t_out) *t_out = best_t;
    return best;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int validate(int64_t M, int64_t N, int64_t K, const void* A, const void* B, const void* C, int64_t lda,
             int64_t ldb, int64_t ldc, int ca_c, int c_dtype, int order, int assign, int tile,
             int b_layout = SFC_B_KN, int ab = SFC_AB_BF16) {
    if (M <= 0 || N <= 0 || K <= 0 || !A || !B || !C) return SFC_ERR_INVALID_ARG;
    if (b_layout != SFC_B_KN && b_layout != SFC_B_NK) return SFC_ERR_INVALID_ARG;
    if (ab != SFC_AB_BF16 && ab != SFC_AB_E4M3 && ab != SFC_AB_E5M2) return SFC_ERR_INVALID_ARG;
    if (lda < K || ldb < (b_layout == SFC_B_NK ? K : N) || ldc < N) return SFC_ERR_INVALID_ARG;
    if (c_dtype != SFC_F32 && c_dtype != SFC_BF16) return SFC_ERR_INVALID_ARG;
    if (order != SFC_ORDER_SFC && order != SFC_ORDER_RASTER) return SFC_ERR_INVALID_ARG;
    if (assign != SFC_ASSIGN_SEGMENT && assign != SFC_ASSIGN_WAVE && assign != SFC_ASSIGN_AUTO &&
        assign != SFC_ASSIGN_WAVE_STATIC)
        return SFC_ERR_INVALID_ARG;
    if (tile != SFC_TILE_AUTO && tile != SFC_TILE_N128 && tile != SFC_TILE_N256 && tile != SFC_TILE_PAIR_N128 &&
        tile != SFC_TILE_PAIR_N256)
        return SFC_ERR_INVALID_ARG;
    // TMA coordinates and tile indices are 32-bit
    if (M > (int64_t(1) << 31) - kBM || N > (int64_t(1) << 31) - 256 || K > (int64_t(1) << 31) - slab_k(ab))
        return SFC_ERR_INVALID_ARG;
    const int64_t Kt = ceil_div(K, slab_k(ab));
    if (ca_c < 0 || ca_c > Kt || ca_c > kMaxLayers) return SFC_ERR_INVALID_ARG;  // 0: chosen per call
    const int64_t layers = ca_c > 0 ? ca_c : auto_layer_cap(M, N, K, ab);
    if (ceil_div(M, kBM) * ceil_div(N, 128) * layers > (int64_t(1) << 31) - 1) return SFC_ERR_INVALID_ARG;
    // elements must be naturally aligned; rows that are not 16-byte aligned are
    // repacked before the tile loads (run_gemm)
    const uintptr_t ea = static_cast<uintptr_t>(in_bytes(ab)) - 1u;
    if ((reinterpret_cast<uintptr_t>(A) & ea) || (reinterpret_cast<uintptr_t>(B) & ea)) return SFC_ERR_UNALIGNED;
    if (lda >= (int64_t(1) << 39) || ldb >= (int64_t(1) << 39)) return SFC_ERR_INVALID_ARG;
    return SFC_OK;
}

// fp32 workspace of a call: one copy of C per K layer when there is more than
// one layer, and one copy when K blocks are summed for a bf16 C (an fp32 C
// sums them in place).
size_t workspace_bytes_for(int64_t M, int64_t N, int c, int kbf, int c_dtype) {
    const int copies = (c > 1) ? c : ((kbf > 1 && c_dtype != SFC_F32) ? 1 : 0);
    return static_cast<size_t>(copies) * static_cast<size_t>(M) * static_cast<size_t>(ws_ld(N)) * 4u;
}

template <typename OutT>
cudaError_t launch_gemm(int v, bool f8, const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc,
                        const GemmParams& p, int grid, cudaStream_t s) {
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = launch_config(v, grid, s, attr, true);
    cudaError_t e = cudaLaunchKernelEx(&cfg, f8 ? Kernels<OutT, true>::get(v) : Kernels<OutT, false>::get(v), ta, tb,
                                       tc, p);
    return e;
}

// ------------------------------------------------------------ tuning table
// Shapes measured by sfc_gemm_tune (the paper's a-priori autotuning of a
// shape, Sec. III-C): per layer count the fastest tile, and the fastest
// (tile, layers, K blocks) overall.  Calls with tile = AUTO (and one K block)
// use them; everything else uses the time model.
constexpr int kTuneMaxLayers = 64;

struct TuneKey {
    int64_t M, N, K;
    int ab, b_layout, c_dtype;
    bool operator<(const TuneKey& o) const {
        return std::tie(M, N, K, ab, b_layout, c_dtype) < std::tie(o.M, o.N, o.K, o.ab, o.b_layout, o.c_dtype);
    }
};

struct TuneEntry {
    int tile_for_c[kTuneMaxLayers + 1];  // SFC_TILE_* per layer count, 0 = not measured
    int tile, c, kbf;                    // fastest overall
};

struct TuneTable {
    std::mutex mu;
    std::map<TuneKey, TuneEntry> map;
};
TuneTable g_tune[kMaxDevices];
std::atomic<int> g_tune_lookup{1};  // 1: exact shape only; 2: else the nearest tuned shape (Sec. III-C, third way)

constexpr int kTileOf[kNumVariants] = {SFC_TILE_N128, SFC_TILE_N256, SFC_TILE_PAIR_N128, SFC_TILE_PAIR_N256};

// Tuned (tile, layers) for a call that lets the library choose the tile:
// with ca_c > 0 the fastest tile for that layer count, with ca_c = 0 the
// fastest pair.  False when the shape was not tuned (or not at that count).
bool tuned_choice(int64_t M, int64_t N, int64_t K, int ab, int b_layout, int c_dtype, int ca_c, int* tile,
                  int* layers) {
    int dev;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
    TuneTable& t = g_tune[dev];
    std::lock_guard<std::mutex> lock(t.mu);
    if (t.map.empty()) return false;
    auto it = t.map.find(TuneKey{M, N, K, ab, b_layout, c_dtype});
    if (it == t.map.end() && g_tune_lookup.load(std::memory_order_relaxed) == 2) {
        // nearest tuned shape of the same types and layout, by distance in log M, log N, log K;
        // it must have been measured at the asked layer count, and its layer count must fit K
        const int64_t Kt = ceil_div(K, slab_k(ab));
        double best = -1.0;
        for (auto cand = t.map.begin(); cand != t.map.end(); ++cand) {
            const TuneKey& k = cand->first;
            if (k.ab != ab || k.b_layout != b_layout || k.c_dtype != c_dtype) continue;
            if (ca_c > 0 ? (ca_c > kTuneMaxLayers || cand->second.tile_for_c[ca_c] == 0) : cand->second.c > Kt)
                continue;
            const double dm = std::log(double(M) / k.M), dn = std::log(double(N) / k.N), dk = std::log(double(K) / k.K);
            const double d = dm * dm + dn * dn + dk * dk;
            if (best < 0.0 || d < best) {
                best = d;
                it = cand;
            }
        }
    }
    if (it == t.map.end()) return false;
    const TuneEntry& e = it->second;
    if (ca_c == 0) {
        *tile = e.tile;
        *layers = e.c;
        return true;
    }
    if (ca_c > kTuneMaxLayers || e.tile_for_c[ca_c] == 0) return false;
    *tile = e.tile_for_c[ca_c];
    *layers = ca_c;
    return true;
}

// Operands whose rows (or base) are not 16-byte aligned are copied into
// padded pool buffers (packed[0] for A, packed[1] for B), and the pointer and
// row stride are redirected to the copy.
int pack_operands(const DeviceInfo* dev, int ab, int b_layout, int64_t M, int64_t N, int64_t K, const void** A,
                  int64_t* lda, const void** B, int64_t* ldb, void* packed[2], cudaStream_t stream) {
    const int eb = in_bytes(ab);
    const int64_t row_align = 16 / eb;
    const int64_t b_rows = (b_layout == SFC_B_NK) ? N : K, b_cols = (b_layout == SFC_B_NK) ? K : N;
    for (int which = 0; which < 2; ++which) {
        const void** ptr = which == 0 ? A : B;
        int64_t* ld = which == 0 ? lda : ldb;
        if (aligned16(*ptr) && (*ld % row_align) == 0) continue;
        const int64_t rows = which == 0 ? M : b_rows, cols = which == 0 ? K : b_cols;
        const int64_t ld_dst = (cols + row_align - 1) / row_align * row_align;
        cudaError_t e = cudaMallocFromPoolAsync(&packed[which], static_cast<size_t>(rows * ld_dst * eb), dev->pool,
                                                stream);
        if (e != cudaSuccess) return cuda_fail(e);
        int64_t blocks = ceil_div(rows * cols, 256);
        if (blocks > static_cast<int64_t>(dev->num_sms) * 16) blocks = static_cast<int64_t>(dev->num_sms) * 16;
        e = launch_plain(pack_rows_kernel, static_cast<unsigned>(blocks), 256, stream,
                         static_cast<const uint8_t*>(*ptr), *ld, rows, cols, eb, static_cast<uint8_t*>(packed[which]),
                         ld_dst);
        if (e != cudaSuccess) return cuda_fail(e);
        *ptr = packed[which];
        *ld = ld_dst;
    }
    return SFC_OK;
}

void free_packed(void* packed[2], cudaStream_t stream) {
    for (int i = 0; i < 2; ++i)
        if (packed[i]) cudaFreeAsync(packed[i], stream);  // stream-ordered: after the kernels that read them
}

// The ticket counter of one call's kernels (dynamic dealing), in memory the
// call owns: stream-ordered from the ticket pool, freed after the call's last
// kernel, so launches in flight at the same time -- on other streams, or
// replays of captured graphs -- never share a counter.  Its words carry the
// call's epoch (next_epoch), so whatever the memory held before reads as a
// count of zero: no clearing is issued on the stream (a memset between two
// GEMM launches would also break their programmatic dependent launch).
int take_ticket(DeviceInfo* dev, cudaStream_t stream, unsigned long long** out) {
    void* ptr = nullptr;
    cudaError_t e = cudaMallocFromPoolAsync(&ptr, kTicketBytes, dev->ticket_pool, stream);
    if (e != cudaSuccess) return cuda_fail(e);
    *out = static_cast<unsigned long long*>(ptr);
    return SFC_OK;
}

// A tag no earlier call of this process used (never 0, so zeroed memory never matches).
std::atomic<unsigned int> g_epoch{0};
unsigned int next_epoch() {
    unsigned int e = g_epoch.fetch_add(1u, std::memory_order_relaxed) + 1u;
    while (e == 0u) e = g_epoch.fetch_add(1u, std::memory_order_relaxed) + 1u;
    return e;
}

// C = cvt(sum over layers of the fp32 copies in ws [+ beta * C + bias]), Listing 1's final reduction.
cudaError_t launch_reduce(const DeviceInfo* dev, const float* ws, int64_t ldo, int64_t layer_stride, int layers,
                          int64_t M, int64_t N, void* C, int64_t ldc, int c_dtype, float beta, const float* bias,
                          cudaStream_t stream) {
    const int64_t work = M * ((N + 3) / 4);
    int64_t blocks = ceil_div(work, 256);
    const int64_t cap = static_cast<int64_t>(dev->num_sms) * 8;
    if (blocks > cap) blocks = cap;
    const int vec = (c_dtype == SFC_F32) ? (aligned16(C) && (ldc % 4) == 0)
                                         : (((reinterpret_cast<uintptr_t>(C) & 7u) == 0) && (ldc % 4) == 0);
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(blocks), 1, 1);
    cfg.blockDim = dim3(256, 1, 1);
    cfg.stream = stream;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    cudaError_t e;
    if (c_dtype == SFC_F32)
        e = cudaLaunchKernelEx(&cfg, ca_reduce_kernel<float>, ws, ldo, layer_stride, layers, M, N,
                               static_cast<float*>(C), ldc, vec, beta, bias);
    else
        e = cudaLaunchKernelEx(&cfg, ca_reduce_kernel<__nv_bfloat16>, ws, ldo, layer_stride, layers, M, N,
                               static_cast<__nv_bfloat16*>(C), ldc, vec, beta, bias);
    return e;
}

int run_gemm(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda, int64_t ldb,
             int64_t ldc, int ca_c, int c_dtype, int order, int assign, int tile, void* workspace,
             size_t workspace_bytes, cudaStream_t stream, int debug_never, uint64_t timeout_ns,
             int b_layout = SFC_B_KN, float beta = 0.0f, const float* bias = nullptr, int ab = SFC_AB_BF16,
             bool allow_pack = true, int kbf = 1, unsigned long long* fixed_ticket = nullptr) {
    int rc = validate(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, order, assign, tile, b_layout, ab);
    if (rc != SFC_OK) return rc;
    // K blocks per layer (Listing 1's k_block_factor): every layer needs at least kbf slabs
    if (kbf < 1 || kbf > kMaxKBlocks) return SFC_ERR_INVALID_ARG;
    const int64_t Kt_all = ceil_div(K, slab_k(ab));
    if (kbf > Kt_all || (ca_c > 0 && Kt_all / ca_c < kbf)) return SFC_ERR_INVALID_ARG;
    const bool f8 = (ab != SFC_AB_BF16);
    const int sk = slab_k(ab), eb = in_bytes(ab);
    // operands whose rows (or base) are not 16-byte aligned are repacked into pool memory
    const int64_t row_align = 16 / eb;
    const bool pack_a = !aligned16(A) || (lda % row_align) != 0;
    const bool pack_b = !aligned16(B) || (ldb % row_align) != 0;
    if ((pack_a || pack_b) && !allow_pack) return SFC_ERR_UNALIGNED;
    if (bias && (reinterpret_cast<uintptr_t>(bias) & 3u) != 0) return SFC_ERR_UNALIGNED;
    const bool b_kmajor = (b_layout == SFC_B_NK);
    if (ca_c > 0 && workspace && workspace_bytes < workspace_bytes_for(M, N, ca_c, kbf, c_dtype))
        return SFC_ERR_WORKSPACE;
    if (workspace && !aligned16(workspace)) return SFC_ERR_UNALIGNED;

    DeviceInfo* dev = nullptr;
    rc = device_setup(&dev);
    if (rc != SFC_OK) return rc;

    // a tuned shape: its measured tile (and, for ca_c = 0, layer count) replace the time model's
    if (tile == SFC_TILE_AUTO && kbf == 1) {
        int t_tile = 0, t_c = 0;
        if (tuned_choice(M, N, K, ab, b_layout, c_dtype, ca_c, &t_tile, &t_c) &&
            (ca_c > 0 || !workspace || workspace_bytes >= workspace_bytes_for(M, N, t_c, 1, c_dtype))) {
            tile = t_tile;
            ca_c = t_c;
        }
    }

    // ca_c = 0: the planner's layer count, within the caller's workspace if one is given
    int max_c = static_cast<int>(auto_layer_cap(M, N, K, ab));
    if (max_c > Kt_all / kbf) max_c = static_cast<int>(Kt_all / kbf);
    while (ca_c == 0 && workspace && max_c > 1 && workspace_bytes < workspace_bytes_for(M, N, max_c, kbf, c_dtype))
        --max_c;
    const Plan plan = make_plan(M, N, K, ca_c, max_c, dev->machine, static_cast<sfc_tile_t>(tile), c_dtype == SFC_F32 ? 4 : 2,
                                b_kmajor, ab);
    const int v = plan.v;
    ca_c = plan.c;
    const size_t ws_need = workspace_bytes_for(M, N, ca_c, kbf, c_dtype);
    const int bn = variant_bn(v);
    const int bm = variant_bm(v);
    void* packed[2] = {nullptr, nullptr};
    auto release_packed = [&]() { free_packed(packed, stream); };
    rc = pack_operands(dev, ab, b_layout, M, N, K, &A, &lda, &B, &ldb, packed, stream);
    if (rc != SFC_OK) {
        release_packed();
        return rc;
    }
    CUtensorMap ta, tb;
    rc = make_in_map(&ta, A, M, K, lda, eb, kBM, sk);  // each CTA loads 128 rows of A, one slab of k
    if (rc == SFC_OK) {
        if (b_kmajor) {
            // B given as N x K: boxes of (this CTA's share of the tile's N rows) x one slab of k, like A
            rc = make_in_map(&tb, B, N, K, ldb, eb, variant_pair(v) ? bn / 2 : bn, sk);
        } else {
            // N-major B boxes: one slab of k rows x 128 bytes of columns
            rc = make_in_map(&tb, B, K, N, ldb, eb, sk, 128 / eb);
        }
    }
    if (rc != SFC_OK) {
        release_packed();
        return rc;
    }

    GemmParams p;
    p.M = M;
    p.N = N;
    p.Mt = static_cast<int>(ceil_div(M, bm));
    p.Nt = static_cast<int>(ceil_div(N, bn));
    p.Kt = static_cast<int>(ceil_div(K, sk));
    p.ca_c = ca_c;
    p.grid_tiles = p.Mt * p.Nt;
    p.kq = p.Kt / ca_c;
    p.kr = p.Kt % ca_c;
    p.kc = kDefaultChunkSlabs;
    p.num_items = static_cast<int64_t>(p.Mt) * p.Nt * ca_c;
    p.order = order;
    p.assign = (assign == SFC_ASSIGN_SEGMENT) ? 0 : 1;
    // dynamic dealing of curve positions for WAVE / AUTO; the static deals stay for comparison
    p.dynamic = (assign == SFC_ASSIGN_WAVE || assign == SFC_ASSIGN_AUTO) ? 1 : 0;
    p.ticket = nullptr;
    p.epoch = next_epoch();
    p.debug_never = debug_never;
    p.timeout_ns = timeout_ns;
    p.b_kmajor = b_kmajor ? 1 : 0;
    p.beta = beta;
    p.c_in = C;
    p.ldc_in = ldc;
    p.c_in_layer_stride = 0;
    p.bias = bias;
    p.ab_fmt = (ab == SFC_AB_E4M3) ? 0 : 1;  // bf16 (kind::f16) and e5m2 (kind::f8f6f4) are both code 1
    p.kbf = 1;
    p.pass = 0;
    p.accumulate = 0;
    const int64_t workers = dev->workers[v];
    const int64_t used = p.num_items < workers ? p.num_items : workers;
    const int grid = static_cast<int>(variant_cluster(v) * used);
    // one item per worker: dynamic dealing would hand worker w item w and nothing else, which is
    // the static wave deal (the same items, the same bits) without a counter
    if (p.dynamic && p.num_items <= workers) p.dynamic = 0;

    void* ws = workspace;
    bool pooled = false;
    if (ws_need > 0 && !ws) {
        cudaError_t e = cudaMallocFromPoolAsync(&ws, ws_need, dev->pool, stream);
        if (e != cudaSuccess) {
            release_packed();
            return cuda_fail(e);
        }
        pooled = true;
    }
    // dynamic dealing: the call's own ticket counter (the K-block passes share it: each kernel
    // leaves it zero, and a pass touches it only after the previous pass has finished)
    bool own_ticket = false;
    if (p.dynamic) {
        if (fixed_ticket) {
            p.ticket = fixed_ticket;
        } else {
            rc = take_ticket(dev, stream, &p.ticket);
            if (rc != SFC_OK) {
                if (pooled) cudaFreeAsync(ws, stream);
                release_packed();
                return rc;
            }
            own_ticket = true;
        }
    }

    cudaError_t e = cudaSuccess;
    CUtensorMap tc;
    std::memset(&tc, 0, sizeof(tc));
    if (ws_need == 0) {
        // one pass straight into C, or K blocks added into an fp32 C in place
        p.out = C;
        p.ldo = ldc;
        p.layer_stride = 0;
        const int esz = (c_dtype == SFC_F32) ? 4 : 2;
        p.vec_store = aligned16(C) && ((ldc * esz) % 16 == 0);
        p.tma_store = p.vec_store && make_out_map(&tc, C, M, N, ldc, esz, 1) == SFC_OK;
        if (beta == 1.0f && !bias && c_dtype == SFC_F32 && p.tma_store) {
            // C += A B: the stores add into C in L2 (the same rounding as reading C and adding)
            p.accumulate = 1;
            p.beta = 0.0f;
        }
        for (int pass = 0; pass < kbf && e == cudaSuccess; ++pass) {
            if (pass > 0) {
                // C holds the earlier K blocks' sum (and beta C + bias): the stores add into it
                // (TMA reduction in L2), or, for rows the TMA cannot store, the epilogue reads it
                p.accumulate = p.tma_store;
                p.beta = p.tma_store ? 0.0f : 1.0f;
                p.bias = nullptr;
            }
            p.kbf = kbf;
            p.pass = pass;
            e = (c_dtype == SFC_F32) ? launch_gemm<float>(v, f8, ta, tb, tc, p, grid, stream)
                                     : launch_gemm<__nv_bfloat16>(v, f8, ta, tb, tc, p, grid, stream);
        }
    } else {
        // fp32 copies of C, one per K layer (K blocks added in place), then the reduction
        p.out = ws;
        p.ldo = ws_ld(N);
        p.layer_stride = M * p.ldo;
        p.vec_store = 1;
        p.tma_store = make_out_map(&tc, ws, M, N, p.ldo, 4, ca_c) == SFC_OK;
        p.beta = 0.0f;
        p.bias = nullptr;
        for (int pass = 0; pass < kbf && e == cudaSuccess; ++pass) {
            if (pass > 0) {
                p.accumulate = p.tma_store;
                p.beta = p.tma_store ? 0.0f : 1.0f;
                p.c_in = ws;
                p.ldc_in = p.ldo;
                p.c_in_layer_stride = p.layer_stride;
            }
            p.kbf = kbf;
            p.pass = pass;
            e = launch_gemm<float>(v, f8, ta, tb, tc, p, grid, stream);
        }
        if (e == cudaSuccess)
            e = launch_reduce(dev, static_cast<const float*>(ws), p.ldo, p.layer_stride, ca_c, M, N, C, ldc, c_dtype,
                              beta, bias, stream);
    }
    if (pooled) {
        cudaError_t f = cudaFreeAsync(ws, stream);
        if (e == cudaSuccess) e = f;
    }
    if (own_ticket) {
        cudaError_t f = cudaFreeAsync(p.ticket, stream);
        if (e == cudaSuccess) e = f;
    }
    release_packed();  // stream-ordered: after the kernels that read the packed copies
    if (e != cudaSuccess) return cuda_fail(e);
    return SFC_OK;
}

}  // namespace
}  // namespace sfc

using namespace sfc;

SFC_API int sfc_tile_order(int Mt, int Nt, int32_t* out_idx) {
    if (Mt < 1 || Nt < 1 || !out_idx) return SFC_ERR_INVALID_ARG;
    const int64_t n = static_cast<int64_t>(Mt) * Nt;
    if (n > INT32_MAX) return SFC_ERR_INVALID_ARG;
    for (int64_t s = 0; s < n; ++s) {
        const TileCoord t = curve_decode(static_cast<int>(s), Mt, Nt);
        out_idx[s] = t.tm * Nt + t.tn;
    }
    return SFC_OK;
}

SFC_API int sfc_tile_order_device(int Mt, int Nt, int32_t* out_idx_dev, void* stream) {
    if (Mt < 1 || Nt < 1 || !out_idx_dev) return SFC_ERR_INVALID_ARG;
    const int64_t n = static_cast<int64_t>(Mt) * Nt;
    if (n > INT32_MAX) return SFC_ERR_INVALID_ARG;
    DeviceInfo* dev = nullptr;
    int rc = device_setup(&dev);
    if (rc != SFC_OK) return rc;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 65535) blocks = 65535;
    cudaError_t e = launch_plain(tile_order_kernel, static_cast<unsigned>(blocks), 256,
                                 static_cast<cudaStream_t>(stream), Mt, Nt, out_idx_dev);
    return e == cudaSuccess ? SFC_OK : cuda_fail(e);
}

SFC_API size_t sfc_gemm_workspace_size(int64_t M, int64_t N, int64_t K, int ca_c) {
    if (M <= 0 || N <= 0 || K <= 0 || ca_c < 0) return 0;
    const int64_t layers = ca_c > 0 ? ca_c : auto_layer_cap(M, N, K);  // 0: the most the planner may choose
    if (layers == 1) return 0;
    return static_cast<size_t>(layers) * static_cast<size_t>(M) * static_cast<size_t>(ws_ld(N)) * 4u;
}

SFC_API int sfc_gemm_plan(int64_t M, int64_t N, int64_t K, int ca_c, int c_dtype, int tile, int ab_dtype,
                          int b_layout, int* out_tile, int* out_ca_c) {
    if (!out_tile || !out_ca_c) return SFC_ERR_INVALID_ARG;
    const int64_t kp = K + (16 - K % 16) % 16, np = N + (16 - N % 16) % 16;  // strides that pass the checks
    int rc = validate(M, N, K, reinterpret_cast<const void*>(16), reinterpret_cast<const void*>(16),
                      reinterpret_cast<const void*>(16), kp, b_layout == SFC_B_NK ? kp : np, N, ca_c, c_dtype,
                      SFC_ORDER_SFC, SFC_ASSIGN_AUTO, tile, b_layout, ab_dtype);
    if (rc != SFC_OK) return rc;
    DeviceInfo* dev = nullptr;
    rc = device_setup(&dev);
    if (rc != SFC_OK) return rc;
    if (tile == SFC_TILE_AUTO) {
        int t_tile = 0, t_c = 0;
        if (tuned_choice(M, N, K, ab_dtype, b_layout, c_dtype, ca_c, &t_tile, &t_c)) {
            tile = t_tile;
            ca_c = t_c;
        }
    }
    const Plan plan = make_plan(M, N, K, ca_c, static_cast<int>(auto_layer_cap(M, N, K, ab_dtype)), dev->machine,
                                static_cast<sfc_tile_t>(tile), c_dtype == SFC_F32 ? 4 : 2, b_layout == SFC_B_NK,
                                ab_dtype);
    *out_tile = kTileOf[plan.v];
    *out_ca_c = plan.c;
    return SFC_OK;
}

SFC_API int sfc_gemm_plan_desc(const sfc_device_desc_t* desc, int64_t M, int64_t N, int64_t K, int ca_c,
                               int c_dtype, int ab_dtype, int b_layout, int* out_tile, int* out_ca_c,
                               double* out_ns) {
    if (!desc || !out_tile || !out_ca_c || !out_ns) return SFC_ERR_INVALID_ARG;
    if (desc->num_sms < 1 || desc->pair_workers < 0 || 2 * desc->pair_workers > desc->num_sms ||
        !(desc->hbm_gbs > 0.0) || !(desc->sm_ghz > 0.0))
        return SFC_ERR_INVALID_ARG;
    const int64_t kp = K + (16 - K % 16) % 16, np = N + (16 - N % 16) % 16;  // strides that pass the checks
    int rc = validate(M, N, K, reinterpret_cast<const void*>(16), reinterpret_cast<const void*>(16),
                      reinterpret_cast<const void*>(16), kp, b_layout == SFC_B_NK ? kp : np, N, ca_c, c_dtype,
                      SFC_ORDER_SFC, SFC_ASSIGN_AUTO, SFC_TILE_AUTO, b_layout, ab_dtype);
    if (rc != SFC_OK) return rc;
    Machine m;
    for (int v = 0; v < kNumVariants; ++v) m.workers[v] = variant_pair(v) ? desc->pair_workers : desc->num_sms;
    m.hbm_bytes_per_ns = desc->hbm_gbs;
    m.sm_ghz = desc->sm_ghz;
    double t = 0.0;
    const Plan plan = make_plan(M, N, K, ca_c, static_cast<int>(auto_layer_cap(M, N, K, ab_dtype)), m, SFC_TILE_AUTO,
                                c_dtype == SFC_F32 ? 4 : 2, b_layout == SFC_B_NK, ab_dtype, &t);
    *out_tile = kTileOf[plan.v];
    *out_ca_c = plan.c;
    *out_ns = t;
    return SFC_OK;
}

SFC_API int sfc_release(void) {
    // The library holds device memory between calls in two places: the staging
    // slots of sfc_gemm_host, and what its stream-ordered pool keeps after
    // K-layer workspaces and repacked operands were freed.
    DeviceInfo* dev = nullptr;
    int rc = device_setup(&dev);
    if (rc != SFC_OK) return rc;
    rc = host_release_staging();
    if (rc != SFC_OK) return rc;
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemPoolTrimTo(dev->pool, 0);
    if (e == cudaSuccess) e = cudaMemPoolTrimTo(dev->ticket_pool, 0);
    return e == cudaSuccess ? SFC_OK : cuda_fail(e);
}

SFC_API int sfc_gemm(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda,
                     int64_t ldb, int64_t ldc, int ca_c, void* stream) {
    return run_gemm(M, N, K, A, B, C, lda, ldb, ldc, ca_c, SFC_F32, SFC_ORDER_SFC, SFC_ASSIGN_AUTO,
                    SFC_TILE_AUTO, nullptr, 0, static_cast<cudaStream_t>(stream), 0, kDefaultTimeoutNs);
}

SFC_API int sfc_gemm_ex(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda,
                        int64_t ldb, int64_t ldc, int ca_c, sfc_dtype_t c_dtype, sfc_order_t order,
                        sfc_assign_t assign, sfc_tile_t tile, void* workspace, size_t workspace_bytes,
                        void* stream) {
    return run_gemm(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, order, assign, tile, workspace,
                    workspace_bytes, static_cast<cudaStream_t>(stream), 0, kDefaultTimeoutNs);
}

SFC_API int sfc_gemm_ex2(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda,
                         int64_t ldb, int64_t ldc, int ab_dtype, int b_layout, float beta, const float* bias,
                         int ca_c, sfc_dtype_t c_dtype, sfc_order_t order, sfc_assign_t assign, sfc_tile_t tile,
                         void* workspace, size_t workspace_bytes, void* stream) {
    return run_gemm(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, order, assign, tile, workspace,
                    workspace_bytes, static_cast<cudaStream_t>(stream), 0, kDefaultTimeoutNs, b_layout, beta, bias,
                    ab_dtype);
}

SFC_API int sfc_gemm_ex3(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda,
                         int64_t ldb, int64_t ldc, int ab_dtype, int b_layout, float beta, const float* bias,
                         int ca_c, int k_block_factor, sfc_dtype_t c_dtype, sfc_order_t order, sfc_assign_t assign,
                         sfc_tile_t tile, void* workspace, size_t workspace_bytes, void* stream) {
    return run_gemm(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, order, assign, tile, workspace,
                    workspace_bytes, static_cast<cudaStream_t>(stream), 0, kDefaultTimeoutNs, b_layout, beta, bias,
                    ab_dtype, true, k_block_factor);
}

SFC_API size_t sfc_gemm_workspace_size2(int64_t M, int64_t N, int64_t K, int ca_c, int k_block_factor,
                                        sfc_dtype_t c_dtype) {
    if (M <= 0 || N <= 0 || K <= 0 || ca_c < 0 || k_block_factor < 1 || k_block_factor > kMaxKBlocks) return 0;
    if (c_dtype != SFC_F32 && c_dtype != SFC_BF16) return 0;
    int64_t layers = ca_c;
    if (layers == 0) {  // the most the planner may choose
        layers = auto_layer_cap(M, N, K);
        const int64_t per = ceil_div(K, kBK) / k_block_factor;
        if (layers > per) layers = per;
        if (layers < 1) layers = 1;
    }
    return workspace_bytes_for(M, N, static_cast<int>(layers), k_block_factor, c_dtype);
}

SFC_API int sfc_gemm_tune(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda,
                          int64_t ldb, int64_t ldc, int ab_dtype, int b_layout, sfc_dtype_t c_dtype, int max_layers,
                          int max_kbf, void* stream, int* out_tile, int* out_ca_c, int* out_kbf) {
    if (!out_tile || !out_ca_c || !out_kbf) return SFC_ERR_INVALID_ARG;
    if (max_layers < 1 || max_layers > kTuneMaxLayers || max_kbf < 1 || max_kbf > kMaxKBlocks)
        return SFC_ERR_INVALID_ARG;
    int rc = validate(M, N, K, A, B, C, lda, ldb, ldc, 1, c_dtype, SFC_ORDER_SFC, SFC_ASSIGN_AUTO, SFC_TILE_AUTO,
                      b_layout, ab_dtype);
    if (rc != SFC_OK) return rc;
    DeviceInfo* dev = nullptr;
    rc = device_setup(&dev);
    if (rc != SFC_OK) return rc;
    int devi = 0;
    rc = current_device(&devi);
    if (rc != SFC_OK) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaStreamCaptureStatus capturing = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(s, &capturing);
    if (e != cudaSuccess) return cuda_fail(e);
    if (capturing != cudaStreamCaptureStatusNone) return SFC_ERR_UNSUPPORTED;  // it times on the host

    const int64_t Kt = ceil_div(K, slab_k(ab_dtype));
    const bool b_kmajor = (b_layout == SFC_B_NK);
    // layer counts 1, 2, 4, ... and the time model's own choice
    std::vector<int> counts;
    for (int c = 1; c <= max_layers && c <= Kt; c *= 2) counts.push_back(c);
    const Plan model = make_plan(M, N, K, 0, static_cast<int>(auto_layer_cap(M, N, K, ab_dtype)), dev->machine,
                                 SFC_TILE_AUTO, c_dtype == SFC_F32 ? 4 : 2, b_kmajor, ab_dtype);
    if (model.c <= max_layers && std::find(counts.begin(), counts.end(), model.c) == counts.end())
        counts.push_back(model.c);

    cudaEvent_t e0 = nullptr, e1 = nullptr;
    e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    if (e != cudaSuccess) {
        if (e0) cudaEventDestroy(e0);
        return cuda_fail(e);
    }
    auto call = [&](int c, int tile, int kbf) {
        return run_gemm(M, N, K, A, B, C, lda, ldb, ldc, c, c_dtype, SFC_ORDER_SFC, SFC_ASSIGN_AUTO, tile, nullptr,
                        0, s, 0, kDefaultTimeoutNs, b_layout, 0.0f, nullptr, ab_dtype, true, kbf);
    };
    // one call to warm up, then the mean of kReps
    constexpr int kReps = 5;
    auto measure = [&](int c, int tile, int kbf, float* us) {
        int r = call(c, tile, kbf);
        cudaError_t ce = cudaSuccess;
        if (r == SFC_OK) ce = cudaEventRecord(e0, s);
        for (int i = 0; i < kReps && r == SFC_OK && ce == cudaSuccess; ++i) r = call(c, tile, kbf);
        if (r == SFC_OK && ce == cudaSuccess) ce = cudaEventRecord(e1, s);
        if (r == SFC_OK && ce == cudaSuccess) ce = cudaEventSynchronize(e1);
        float ms = 0.0f;
        if (r == SFC_OK && ce == cudaSuccess) ce = cudaEventElapsedTime(&ms, e0, e1);
        if (r == SFC_OK && ce != cudaSuccess) r = cuda_fail(ce);
        *us = ms * 1000.0f / static_cast<float>(kReps);
        return r;
    };
    // A measured alternative replaces the time model's choice only when it is clearly faster:
    // candidates within timing noise of each other keep the model's (steadier) pick.
    constexpr float kMargin = 0.97f;

    TuneEntry entry;
    std::memset(&entry, 0, sizeof(entry));
    float best = -1.0f;            // the fastest configuration so far
    float model_us = -1.0f;        // the time model's layer count, with its measured tile
    for (int c : counts) {
        const int model_v = make_plan(M, N, K, c, c, dev->machine, SFC_TILE_AUTO, c_dtype == SFC_F32 ? 4 : 2, b_kmajor,
                                      ab_dtype).v;
        float t[kNumVariants];
        for (int v = 0; v < kNumVariants; ++v) t[v] = -1.0f;
        for (int v = 0; v < kNumVariants && rc == SFC_OK; ++v) {
            if (dev->workers[v] <= 0 || !variant_allowed(v, b_kmajor, ab_dtype)) continue;
            rc = measure(c, kTileOf[v], 1, &t[v]);
        }
        if (rc != SFC_OK) break;
        int pick = (t[model_v] >= 0.0f) ? model_v : -1;
        for (int v = 0; v < kNumVariants; ++v) {
            if (t[v] < 0.0f) continue;
            if (pick < 0 || t[v] < t[pick] * kMargin) pick = v;
        }
        entry.tile_for_c[c] = kTileOf[pick];
        if (c == model.c) model_us = t[pick];
        if (best < 0.0f || t[pick] < best) {
            best = t[pick];
            entry.tile = kTileOf[pick];
            entry.c = c;
            entry.kbf = 1;
        }
    }
    // the model's layer count stays unless another is clearly faster
    if (rc == SFC_OK && model_us >= 0.0f && best > model_us * kMargin && entry.tile_for_c[model.c] != 0) {
        best = model_us;
        entry.tile = entry.tile_for_c[model.c];
        entry.c = model.c;
    }
    // K blocks on the chosen (tile, layers), taken only when clearly faster
    const int base_kbf_c = entry.c;
    for (int kbf = 2; rc == SFC_OK && kbf <= max_kbf && Kt / base_kbf_c >= kbf; kbf *= 2) {
        float us = 0.0f;
        rc = measure(entry.c, entry.tile, kbf, &us);
        if (rc == SFC_OK && us < best * kMargin) {
            best = us;
            entry.kbf = kbf;
        }
    }
    if (rc == SFC_OK) rc = call(entry.c, entry.tile, entry.kbf);  // C holds the chosen configuration's result
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (rc != SFC_OK) return rc;
    {
        TuneTable& t = g_tune[devi];
        std::lock_guard<std::mutex> lock(t.mu);
        t.map[TuneKey{M, N, K, ab_dtype, b_layout, c_dtype}] = entry;
    }
    *out_tile = entry.tile;
    *out_ca_c = entry.c;
    *out_kbf = entry.kbf;
    return SFC_OK;
}

SFC_API int sfc_gemm_tune_lookup(int mode) {
    if (mode != 1 && mode != 2) return SFC_ERR_INVALID_ARG;
    g_tune_lookup.store(mode, std::memory_order_relaxed);
    return SFC_OK;
}

SFC_API int sfc_gemm_tune_forget(void) {
    int dev;
    int rc = current_device(&dev);
    if (rc != SFC_OK) return rc;
    TuneTable& t = g_tune[dev];
    std::lock_guard<std::mutex> lock(t.mu);
    t.map.clear();
    return SFC_OK;
}

SFC_API int sfc_get_device_status(void* stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e);
    unsigned int word = 0;
    e = cudaMemcpyFromSymbol(&word, g_sfc_status, sizeof(word));
    if (e != cudaSuccess) return cuda_fail(e);
    if (word == 0) return SFC_OK;
    // clear the bits that were read (atomically: a kernel on another stream may be setting others)
    e = launch_plain(status_clear_kernel, 1, 1, s, word);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e);
    return SFC_ERR_TIMEOUT;
}

SFC_API int sfc_last_cuda_error(void) { return t_last_cuda_error; }

SFC_API int sfc_num_workers(void) {
    DeviceInfo* dev = nullptr;
    int rc = device_setup(&dev);
    return rc == SFC_OK ? dev->num_sms : rc;
}

SFC_API int sfc_debug_force_timeout(const void* A, const void* B, void* C, int limit_ms, void* stream) {
    if (limit_ms < 1 || limit_ms > 1000) return SFC_ERR_INVALID_ARG;
    return run_gemm(128, 128, 64, A, B, C, 64, 128, 128, 1, SFC_F32, SFC_ORDER_SFC, SFC_ASSIGN_WAVE,
                    SFC_TILE_N128, nullptr, 0, static_cast<cudaStream_t>(stream), 1,
                    static_cast<uint64_t>(limit_ms) * 1000000ull);
}

// ---------------------------------------------------------------------------
// Allocation-free entry point.  The fp32 partial copies of C live in a fixed
// device array of this module instead of caller or pool memory, and so does
// the call's ticket counter (after the partials).  Host code must not pass
// the array's name to a kernel (on the host it is only a stand-in symbol), so
// its device address is looked up once per device.
// ---------------------------------------------------------------------------
namespace sfc {
namespace {

// the ticket counter's words are tagged with each call's epoch, so the area needs no clearing
static __device__ __align__(256) unsigned char g_noalloc_scratch[SFC_NOALLOC_SCRATCH_BYTES + kTicketBytes];

struct NoAllocScratch {
    std::mutex mu;
    bool found = false;  // set only once a lookup has succeeded; a failed one is retried next call
    void* ptr = nullptr;
};
NoAllocScratch g_noalloc[kMaxDevices];

int noalloc_scratch(void** ptr) {
    int dev;
    int rc = current_device(&dev);
    if (rc != SFC_OK) return rc;
    NoAllocScratch& s = g_noalloc[dev];
    std::lock_guard<std::mutex> lock(s.mu);
    if (!s.found) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return cuda_fail(e);
        s.ptr = p;
        s.found = true;
    }
    *ptr = s.ptr;
    return SFC_OK;
}

}  // namespace
}  // namespace sfc

SFC_API int sfc_gemm_noalloc(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C,
                             int64_t lda, int64_t ldb, int64_t ldc, int ca_c, sfc_dtype_t c_dtype,
                             void* stream) {
    void* scratch = nullptr;
    int rc = noalloc_scratch(&scratch);
    if (rc != SFC_OK) return rc;
    // ca_c > 0 whose partials exceed the scratch area: SFC_ERR_WORKSPACE from run_gemm;
    // ca_c = 0: the library's layer count is limited to what fits
    unsigned long long* ticket = reinterpret_cast<unsigned long long*>(static_cast<unsigned char*>(scratch) +
                                                                       SFC_NOALLOC_SCRATCH_BYTES);
    return run_gemm(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, SFC_ORDER_SFC, SFC_ASSIGN_AUTO, SFC_TILE_AUTO,
                    scratch, SFC_NOALLOC_SCRATCH_BYTES, static_cast<cudaStream_t>(stream), 0, kDefaultTimeoutNs,
                    SFC_B_KN, 0.0f, nullptr, SFC_AB_BF16, /*allow_pack=*/false, /*kbf=*/1, ticket);
}

SFC_API int sfc_debug_pool_used_high(size_t* used_high_bytes, int reset) {
    if (!used_high_bytes || (reset != 0 && reset != 1)) return SFC_ERR_INVALID_ARG;
    DeviceInfo* dev = nullptr;
    int rc = device_setup(&dev);
    if (rc != SFC_OK) return rc;
    size_t total = 0;
    for (cudaMemPool_t pool : {dev->pool, dev->ticket_pool}) {
        cuuint64_t v = 0;
        cudaError_t e = cudaMemPoolGetAttribute(pool, cudaMemPoolAttrUsedMemHigh, &v);
        if (e != cudaSuccess) return cuda_fail(e);
        total += static_cast<size_t>(v);
        if (reset) {
            cuuint64_t zero = 0;
            e = cudaMemPoolSetAttribute(pool, cudaMemPoolAttrUsedMemHigh, &zero);
            if (e != cudaSuccess) return cuda_fail(e);
        }
    }
    *used_high_bytes = total;
    return SFC_OK;
}
