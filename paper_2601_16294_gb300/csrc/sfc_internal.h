// sfc_internal.h -- functions shared by the library's translation units; not
// part of the C ABI (the library is built with hidden visibility).
#pragma once

#include <cuda_runtime.h>

namespace sfc {

// Records `e` as the calling thread's last CUDA error (sfc_last_cuda_error)
// and returns SFC_ERR_CUDA.  Defined in sfc_gemm.cu.
int cuda_fail(cudaError_t e);

// Frees the staging memory of sfc_gemm_host on the current device after the
// calls that use it have completed.  Defined in sfc_host.cpp.
int host_release_staging();

}  // namespace sfc
