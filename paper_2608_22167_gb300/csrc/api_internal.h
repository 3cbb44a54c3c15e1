// Host-side pieces shared by the translation units of the C ABI (api.cu,
// api_noalloc.cu): the dimension checks every forward entry point applies,
// and the recording of the failed CUDA call behind an MCPU_ERR_CUDA (read
// back with mcpu_last_cuda_error).
#pragma once

#include <cuda_runtime.h>

#include "../../include/mcpu.h"

namespace mcpu {

// MCPU_OK, or the error for dims the kernels cannot serve: null, negative
// or inconsistent sizes (MCPU_ERR_INVALID_ARG); head_dim != 64,
// page_size != 16, H_q / H_kv outside {1, 2, 4, 8}, more than 2048 rows, or
// pools / tables too large for 32-bit TMA row coordinates
// (MCPU_ERR_UNSUPPORTED).
mcpu_status check_dims(const mcpu_dims* d);

// Records e as the calling thread's last failed CUDA call; MCPU_ERR_CUDA.
mcpu_status cuda_fail(cudaError_t e);

// MCPU_OK for cudaSuccess, else cuda_fail(e).
mcpu_status from_cuda(cudaError_t e);

}  // namespace mcpu
