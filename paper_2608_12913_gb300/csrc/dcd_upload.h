// dcd_upload.h -- launcher of the q staging kernel (dcd_upload.cu), for the C ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dcd {

// Copies, on `stream`, the rows of q a sampled call reads (rows of sequences with a positive
// temperature whose node has a child) from `src_dev_view` -- the device mapping of page-locked
// host memory -- into `dst`; both [B*N, ldq] fp32.  parents [B, N] and temperature [B] are device
// arrays.
cudaError_t launch_upload_q_rows(int32_t B, int32_t N, int64_t V, int64_t ldq, const float* src_dev_view, float* dst,
                                 const int32_t* parents, const float* temperature, cudaStream_t stream);

}  // namespace dcd
