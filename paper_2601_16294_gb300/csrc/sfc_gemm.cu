// sfc_gemm.cu -- host side of the SFC GEMM library: argument validation, TMA
// descriptors, launch configuration and the exported C ABI (include/sfc_gemm.h).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "sfc_gemm.h"
#include "sfc_gemm_kernel.cuh"

#define SFC_API extern "C" __attribute__((visibility("default")))

namespace sfc {
namespace {

constexpr int kMaxDevices = 64;
constexpr uint64_t kDefaultTimeoutNs = 2000000000ull;  // 2 s per wait

thread_local int t_last_cuda_error = 0;

int cuda_fail(cudaError_t e) {
    t_last_cuda_error = static_cast<int>(e);
    return SFC_ERR_CUDA;
}

// ---------------------------------------------------------- per-device state

struct DeviceInfo {
    std::once_flag once;
    int status = SFC_ERR_UNSUPPORTED;
    int num_sms = 0;
};
DeviceInfo g_devices[kMaxDevices];

int current_device(int* dev) {
    cudaError_t e = cudaGetDevice(dev);
    if (e != cudaSuccess) return cuda_fail(e);
    if (*dev < 0 || *dev >= kMaxDevices) return SFC_ERR_UNSUPPORTED;
    return SFC_OK;
}

template <int BN, int STAGES, typename OutT>
cudaError_t set_smem_attr() {
    return cudaFuncSetAttribute(sfc_gemm_kernel<BN, STAGES, OutT>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SmemLayout<BN, STAGES>::kDynamicBytes);
}

constexpr int kStages256 = 4;  // 4 x 48 KB ring
constexpr int kStages128 = 6;  // 6 x 32 KB ring

// One-time set-up of the current device: check it is an sm_103 part, read its
// SM count, raise the shared-memory limit of every kernel instantiation.
int device_setup(int* num_sms) {
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
        cudaError_t errs[] = {
            set_smem_attr<256, kStages256, float>(), set_smem_attr<256, kStages256, __nv_bfloat16>(),
            set_smem_attr<128, kStages128, float>(), set_smem_attr<128, kStages128, __nv_bfloat16>(),
        };
        for (cudaError_t x : errs)
            if (x != cudaSuccess) { d.status = cuda_fail(x); return; }
        d.status = SFC_OK;
    });
    if (d.status == SFC_OK) *num_sms = d.num_sms;
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

// Row-major bf16 matrix rows x cols with row stride ld (elements), boxes of
// box_rows x box_cols with 128-byte swizzle; out-of-range elements read as 0.
int make_bf16_map(CUtensorMap* map, const void* ptr, int64_t rows, int64_t cols, int64_t ld,
                  uint32_t box_rows, uint32_t box_cols) {
    PFN_cuTensorMapEncodeTiled_v12000 encode;
    int rc = get_encoder(&encode);
    if (rc != SFC_OK) return rc;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        t_last_cuda_error = static_cast<int>(r);
        return SFC_ERR_CUDA;
    }
    return SFC_OK;
}

// ------------------------------------------------------------------ planning

struct Plan {
    int64_t M, N, K;
    int Mt, Nt, Kt, bn, ca_c, grid;
    int64_t items;
};

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

int pick_bn(int64_t M, int64_t N, int ca_c, int num_sms, sfc_tile_t tile) {
    if (tile == SFC_TILE_N128) return 128;
    if (tile == SFC_TILE_N256) return 256;
    // wide tiles halve the shared-memory traffic per flop; use them when they
    // still give every SM at least one item
    const int64_t items256 = ceil_div(M, kBM) * ceil_div(N, 256) * ca_c;
    return items256 >= num_sms ? 256 : 128;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int validate(int64_t M, int64_t N, int64_t K, const void* A, const void* B, const void* C, int64_t lda,
             int64_t ldb, int64_t ldc, int ca_c, int c_dtype, int order, int assign, int tile) {
    if (M <= 0 || N <= 0 || K <= 0 || !A || !B || !C) return SFC_ERR_INVALID_ARG;
    if (lda < K || ldb < N || ldc < N) return SFC_ERR_INVALID_ARG;
    if (c_dtype != SFC_F32 && c_dtype != SFC_BF16) return SFC_ERR_INVALID_ARG;
    if (order != SFC_ORDER_SFC && order != SFC_ORDER_RASTER) return SFC_ERR_INVALID_ARG;
    if (assign != SFC_ASSIGN_SEGMENT && assign != SFC_ASSIGN_WAVE && assign != SFC_ASSIGN_AUTO)
        return SFC_ERR_INVALID_ARG;
    if (tile != SFC_TILE_AUTO && tile != SFC_TILE_N128 && tile != SFC_TILE_N256) return SFC_ERR_INVALID_ARG;
    // TMA coordinates and tile indices are 32-bit
    if (M > (int64_t(1) << 31) - kBM || N > (int64_t(1) << 31) - 256 || K > (int64_t(1) << 31) - kBK)
        return SFC_ERR_INVALID_ARG;
    const int64_t Kt = ceil_div(K, kBK);
    if (ca_c < 1 || ca_c > Kt) return SFC_ERR_INVALID_ARG;
    if (ceil_div(M, kBM) * ceil_div(N, 128) * ca_c > (int64_t(1) << 31) - 1) return SFC_ERR_INVALID_ARG;
    if (!aligned16(A) || !aligned16(B) || (lda % 8) != 0 || (ldb % 8) != 0) return SFC_ERR_UNALIGNED;
    if (lda >= (int64_t(1) << 39) || ldb >= (int64_t(1) << 39)) return SFC_ERR_INVALID_ARG;
    return SFC_OK;
}

int64_t ws_ld(int64_t N) { return (N + 3) / 4 * 4; }

template <int BN, int STAGES, typename OutT>
cudaError_t launch_gemm(const CUtensorMap& ta, const CUtensorMap& tb, const GemmParams& p, int grid,
                        cudaStream_t s) {
    sfc_gemm_kernel<BN, STAGES, OutT>
        <<<grid, kThreads, SmemLayout<BN, STAGES>::kDynamicBytes, s>>>(ta, tb, p);
    return cudaGetLastError();
}

template <typename OutT>
cudaError_t dispatch_bn(int bn, const CUtensorMap& ta, const CUtensorMap& tb, const GemmParams& p, int grid,
                        cudaStream_t s) {
    if (bn == 256) return launch_gemm<256, kStages256, OutT>(ta, tb, p, grid, s);
    return launch_gemm<128, kStages128, OutT>(ta, tb, p, grid, s);
}

int run_gemm(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C, int64_t lda, int64_t ldb,
             int64_t ldc, int ca_c, int c_dtype, int order, int assign, int tile, void* workspace,
             size_t workspace_bytes, cudaStream_t stream, int debug_never, uint64_t timeout_ns) {
    int rc = validate(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, order, assign, tile);
    if (rc != SFC_OK) return rc;
    const size_t ws_need = sfc_gemm_workspace_size(M, N, K, ca_c);
    if (workspace && workspace_bytes < ws_need) return SFC_ERR_WORKSPACE;
    if (workspace && !aligned16(workspace)) return SFC_ERR_UNALIGNED;

    int num_sms = 0;
    rc = device_setup(&num_sms);
    if (rc != SFC_OK) return rc;

    const int bn = pick_bn(M, N, ca_c, num_sms, static_cast<sfc_tile_t>(tile));
    CUtensorMap ta, tb;
    rc = make_bf16_map(&ta, A, M, K, lda, kBM, kBK);
    if (rc != SFC_OK) return rc;
    rc = make_bf16_map(&tb, B, K, N, ldb, kBK, kBBox);
    if (rc != SFC_OK) return rc;

    GemmParams p;
    p.M = M;
    p.N = N;
    p.Mt = static_cast<int>(ceil_div(M, kBM));
    p.Nt = static_cast<int>(ceil_div(N, bn));
    p.Kt = static_cast<int>(ceil_div(K, kBK));
    p.ca_c = ca_c;
    p.num_items = static_cast<int64_t>(p.Mt) * p.Nt * ca_c;
    p.order = order;
    p.assign = (assign == SFC_ASSIGN_SEGMENT) ? 0 : 1;
    p.debug_never = debug_never;
    p.timeout_ns = timeout_ns;
    const int grid = static_cast<int>(p.num_items < num_sms ? p.num_items : num_sms);

    void* ws = workspace;
    bool pooled = false;
    if (ca_c > 1 && !ws) {
        cudaError_t e = cudaMallocAsync(&ws, ws_need, stream);
        if (e != cudaSuccess) return cuda_fail(e);
        pooled = true;
    }

    cudaError_t e;
    if (ca_c == 1) {
        p.out = C;
        p.ldo = ldc;
        p.layer_stride = 0;
        const size_t esz = (c_dtype == SFC_F32) ? 4 : 2;
        p.vec_store = aligned16(C) && ((ldc * esz) % 16 == 0);
        e = (c_dtype == SFC_F32) ? dispatch_bn<float>(bn, ta, tb, p, grid, stream)
                                 : dispatch_bn<__nv_bfloat16>(bn, ta, tb, p, grid, stream);
    } else {
        p.out = ws;
        p.ldo = ws_ld(N);
        p.layer_stride = M * p.ldo;
        p.vec_store = 1;
        e = dispatch_bn<float>(bn, ta, tb, p, grid, stream);
        if (e == cudaSuccess) {
            const int64_t work = M * ((N + 3) / 4);
            int64_t blocks = ceil_div(work, 256);
            const int64_t cap = static_cast<int64_t>(num_sms) * 8;
            if (blocks > cap) blocks = cap;
            const int vec = (c_dtype == SFC_F32) ? (aligned16(C) && (ldc % 4) == 0)
                                                 : (((reinterpret_cast<uintptr_t>(C) & 7u) == 0) && (ldc % 4) == 0);
            if (c_dtype == SFC_F32)
                ca_reduce_kernel<float><<<static_cast<int>(blocks), 256, 0, stream>>>(
                    static_cast<const float*>(ws), p.ldo, p.layer_stride, ca_c, M, N, static_cast<float*>(C),
                    ldc, vec);
            else
                ca_reduce_kernel<__nv_bfloat16><<<static_cast<int>(blocks), 256, 0, stream>>>(
                    static_cast<const float*>(ws), p.ldo, p.layer_stride, ca_c, M, N,
                    static_cast<__nv_bfloat16*>(C), ldc, vec);
            e = cudaGetLastError();
        }
    }
    if (pooled) {
        cudaError_t f = cudaFreeAsync(ws, stream);
        if (e == cudaSuccess) e = f;
    }
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
        const TileCoord t = curve_decode(s, Mt, Nt);
        out_idx[s] = t.tm * Nt + t.tn;
    }
    return SFC_OK;
}

SFC_API int sfc_tile_order_device(int Mt, int Nt, int32_t* out_idx_dev, void* stream) {
    if (Mt < 1 || Nt < 1 || !out_idx_dev) return SFC_ERR_INVALID_ARG;
    const int64_t n = static_cast<int64_t>(Mt) * Nt;
    if (n > INT32_MAX) return SFC_ERR_INVALID_ARG;
    int num_sms = 0;
    int rc = device_setup(&num_sms);
    if (rc != SFC_OK) return rc;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 65535) blocks = 65535;
    tile_order_kernel<<<static_cast<int>(blocks), 256, 0, static_cast<cudaStream_t>(stream)>>>(Mt, Nt,
                                                                                              out_idx_dev);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? SFC_OK : cuda_fail(e);
}

SFC_API size_t sfc_gemm_workspace_size(int64_t M, int64_t N, int64_t K, int ca_c) {
    if (M <= 0 || N <= 0 || K <= 0 || ca_c < 1) return 0;
    if (ca_c == 1) return 0;
    return static_cast<size_t>(ca_c) * static_cast<size_t>(M) * static_cast<size_t>(ws_ld(N)) * 4u;
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

SFC_API int sfc_get_device_status(void* stream) {
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e);
    unsigned int word = 0;
    e = cudaMemcpyFromSymbol(&word, g_sfc_status, sizeof(word));
    if (e != cudaSuccess) return cuda_fail(e);
    if (word == 0) return SFC_OK;
    const unsigned int zero = 0;
    e = cudaMemcpyToSymbol(g_sfc_status, &zero, sizeof(zero));
    if (e != cudaSuccess) return cuda_fail(e);
    return SFC_ERR_TIMEOUT;
}

SFC_API int sfc_last_cuda_error(void) { return t_last_cuda_error; }

SFC_API int sfc_num_workers(void) {
    int n = 0;
    int rc = device_setup(&n);
    return rc == SFC_OK ? n : rc;
}

SFC_API int sfc_debug_force_timeout(const void* A, const void* B, void* C, int limit_ms, void* stream) {
    if (limit_ms < 1 || limit_ms > 1000) return SFC_ERR_INVALID_ARG;
    return run_gemm(128, 128, 64, A, B, C, 64, 128, 128, 1, SFC_F32, SFC_ORDER_SFC, SFC_ASSIGN_WAVE,
                    SFC_TILE_N128, nullptr, 0, static_cast<cudaStream_t>(stream), 1,
                    static_cast<uint64_t>(limit_ms) * 1000000ull);
}

// ---------------------------------------------------------------------------
// Allocation-free entry point.  The fp32 partial copies of C live in a fixed
// device array of this module instead of caller or pool memory; host code
// must not pass the array's name to a kernel (on the host it is only a
// stand-in symbol), so its device address is looked up once per device.
// ---------------------------------------------------------------------------
namespace sfc {
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[SFC_NOALLOC_SCRATCH_BYTES];

struct NoAllocScratch {
    std::once_flag once;
    int status = SFC_ERR_CUDA;
    void* ptr = nullptr;
};
NoAllocScratch g_noalloc[kMaxDevices];

int noalloc_scratch(void** ptr) {
    int dev;
    int rc = current_device(&dev);
    if (rc != SFC_OK) return rc;
    NoAllocScratch& s = g_noalloc[dev];
    std::call_once(s.once, [&]() {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) { s.status = cuda_fail(e); return; }
        s.ptr = p;
        s.status = SFC_OK;
    });
    if (s.status == SFC_OK) *ptr = s.ptr;
    return s.status;
}

}  // namespace
}  // namespace sfc

SFC_API int sfc_gemm_noalloc(int64_t M, int64_t N, int64_t K, const void* A, const void* B, void* C,
                             int64_t lda, int64_t ldb, int64_t ldc, int ca_c, sfc_dtype_t c_dtype,
                             void* stream) {
    if (sfc_gemm_workspace_size(M, N, K, ca_c) > SFC_NOALLOC_SCRATCH_BYTES) return SFC_ERR_WORKSPACE;
    void* scratch = nullptr;
    int rc = noalloc_scratch(&scratch);
    if (rc != SFC_OK) return rc;
    return sfc_gemm_ex(M, N, K, A, B, C, lda, ldb, ldc, ca_c, c_dtype, SFC_ORDER_SFC, SFC_ASSIGN_AUTO,
                       SFC_TILE_AUTO, scratch, SFC_NOALLOC_SCRATCH_BYTES, stream);
}

