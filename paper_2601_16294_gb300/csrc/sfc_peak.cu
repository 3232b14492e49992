// sfc_peak.cu -- the tensor cores' attainable rate on this device: back-to-back
// tcgen05.mma from operands resident in shared memory, no loads, no epilogue.
//
// This is the per-SM constant of the paper's roofline (the compute term of its
// performance model, Sec. III-B), measured rather than taken from a data
// sheet: FLOP per clock per SM at whatever clock the part runs.  Each 2-CTA
// cluster issues the same instruction the GEMM's pair tiles issue (256 x 256 x
// 16, bf16 in, fp32 in tensor memory, A K-major and B N-major with 128-byte
// swizzle) `iters` x 4 times on one zero-filled stage, and times the issue
// loop with clock64 from the first instruction to the commit's arrival.
#include <cuda_runtime.h>

#include <cstdint>
#include <vector>

#include "ptx.cuh"
#include "sfc_gemm.h"
#include "sfc_internal.h"

#define SFC_API extern "C" __attribute__((visibility("default")))

namespace sfc {
namespace {

constexpr int kPeakThreads = 128;
constexpr uint32_t kPeakABytes = 128 * 128;  // this CTA's 128 rows of A: 64 values of k, 128-byte rows
constexpr uint32_t kPeakBBytes = 128 * 128;  // this CTA's 128 columns of B: two 64-column boxes of 64 k rows
constexpr uint32_t kPeakBoxBytes = 64 * 128;
// operands, barrier and 1 KB of alignment slack need 34 KB; asking for more
// than half an SM's shared memory keeps one CTA per SM, so one pair owns the
// two SMs' tensor cores
constexpr uint32_t kPeakSmem = 140 * 1024;
constexpr int kPeakMaxIters = 1 << 20;

__device__ unsigned int g_peak_status;

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPeakThreads, 1)
    mma_peak_kernel(int iters, uint64_t timeout_ns, unsigned long long* cycles) {
    extern __shared__ uint8_t raw[];
    uint8_t* smem = raw + ((1024u - (ptx::smem_addr(raw) & 1023u)) & 1023u);  // swizzle atoms need 1 KB
    const uint32_t sa = ptx::smem_addr(smem), sb = sa + kPeakABytes;
    const uint32_t tmem_slot = sb + kPeakBBytes;
    const uint32_t done = tmem_slot + 16;
    const uint32_t rank = ptx::cluster_ctarank();
    const int warp = threadIdx.x / 32;

    // operand values do not matter: zeros keep the arithmetic finite
    uint4* z = reinterpret_cast<uint4*>(smem);
    for (uint32_t i = threadIdx.x; i < (kPeakABytes + kPeakBBytes) / 16; i += blockDim.x) z[i] = make_uint4(0, 0, 0, 0);
    ptx::fence_proxy_async_smem();  // the tensor cores (async proxy) read what the threads wrote
    if (threadIdx.x == 0) {
        ptx::mbar_init(done, 1);
        ptx::fence_barrier_init();
    }
    if (warp == 0) {
        ptx::tmem_alloc_pair(tmem_slot, 256);
        ptx::tmem_relinquish_pair();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();  // both CTAs' operands and barriers are ready
    ptx::tc_fence_after();
    const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(smem + kPeakABytes + kPeakBBytes);

    if (threadIdx.x == 0) {
        unsigned long long t0 = 0;
        if (rank == 0) {
            const uint32_t idesc = ptx::idesc_f32(256, 256, /*A K-major*/ 0, /*B N-major*/ 1, /*bf16*/ 1);
            const uint64_t adesc = ptx::smem_desc_sw128(sa, 16, 1024);
            const uint64_t bdesc = ptx::smem_desc_sw128(sb, kPeakBoxBytes, 1024);
            const uint32_t bstep = (16 * 128) / 16;  // 16 rows of k per instruction
            t0 = clock64();
            for (int i = 0; i < iters; ++i)
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    ptx::tc_mma_f16_pair(tmem, adesc + 2u * kk, bdesc + bstep * kk, idesc, (i | kk) ? 1u : 0u);
            ptx::tc_commit_pair_multicast(done, 0x3);  // arrives in both CTAs of the pair
        }
        // both CTAs wait (bounded) for the MMAs before freeing their tensor memory
        bool ok = ptx::mbar_try_wait(done, 0);
        const uint64_t w0 = ptx::global_timer_ns();
        while (!ok) {
            ok = ptx::mbar_try_wait(done, 0);
            if (!ok && ptx::global_timer_ns() - w0 > timeout_ns) break;
        }
        if (!ok) atomicOr(&g_peak_status, 1u);
        if (rank == 0) cycles[blockIdx.x / 2] = ok ? clock64() - t0 : 0ull;
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::cluster_sync();
    ptx::tc_fence_after();
    if (warp == 0) ptx::tmem_dealloc_pair(tmem, 256);
}

}  // namespace
}  // namespace sfc

using namespace sfc;

SFC_API int sfc_mma_peak(int iters, double* flop_per_clk_per_sm, double* tflops, void* stream) {
    if (iters < 1 || iters > kPeakMaxIters || !flop_per_clk_per_sm || !tflops) return SFC_ERR_INVALID_ARG;
    int dev = 0;
    cudaDeviceProp prop;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaGetDeviceProperties(&prop, dev);
    if (e != cudaSuccess) return cuda_fail(e);
    if (prop.major != 10 || prop.minor != 3) return SFC_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // every pair of SMs the hardware can co-schedule
    int clusters = 0;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 2;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.blockDim = dim3(kPeakThreads, 1, 1);
    cfg.dynamicSmemBytes = kPeakSmem;
    cfg.stream = s;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(prop.multiProcessorCount), 1, 1);
    e = cudaFuncSetAttribute(mma_peak_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kPeakSmem));
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveClusters(&clusters, mma_peak_kernel, &cfg);
    if (e != cudaSuccess) return cuda_fail(e);
    if (clusters < 1) return SFC_ERR_UNSUPPORTED;
    cfg.gridDim = dim3(static_cast<unsigned>(2 * clusters), 1, 1);
    cfg.numAttrs = 0;  // the kernel declares its cluster shape
    unsigned long long* d_cycles = nullptr;
    e = cudaMallocAsync(reinterpret_cast<void**>(&d_cycles), sizeof(unsigned long long) * clusters, s);
    if (e != cudaSuccess) return cuda_fail(e);
    const unsigned int zero = 0;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    e = cudaMemcpyToSymbolAsync(g_peak_status, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    // one launch to warm up, then the timed one
    for (int rep = 0; rep < 2 && e == cudaSuccess; ++rep) {
        if (rep == 1) e = cudaEventRecord(e0, s);
        if (e == cudaSuccess)
            e = cudaLaunchKernelEx(&cfg, mma_peak_kernel, iters, static_cast<uint64_t>(2000000000ull), d_cycles);
    }
    if (e == cudaSuccess) e = cudaEventRecord(e1, s);
    std::vector<unsigned long long> cyc(static_cast<size_t>(clusters), 0ull);
    unsigned int status = 0;
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(cyc.data(), d_cycles, sizeof(unsigned long long) * clusters, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess)
        e = cudaMemcpyFromSymbolAsync(&status, g_peak_status, sizeof(status), 0, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    float ms = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    cudaFreeAsync(d_cycles, s);
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    if (e != cudaSuccess) return cuda_fail(e);
    if (status != 0) return SFC_ERR_TIMEOUT;
    unsigned long long worst = 0;
    for (unsigned long long c : cyc) worst = c > worst ? c : worst;
    if (worst == 0 || ms <= 0.0f) return SFC_ERR_CUDA;
    const double flop_per_cluster = 2.0 * 256.0 * 256.0 * 16.0 * 4.0 * static_cast<double>(iters);
    *flop_per_clk_per_sm = flop_per_cluster / 2.0 / static_cast<double>(worst);
    *tflops = flop_per_cluster * clusters / (ms * 1e-3) / 1e12;
    return SFC_OK;
}
