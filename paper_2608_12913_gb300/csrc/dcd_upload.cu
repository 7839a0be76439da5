// dcd_upload.cu -- host-to-device staging of the draft distributions q for a sampled call.
//
// A sampled verification reads q only in the rows of sequences with a positive temperature whose
// node has at least one child: the sibling test reads q at the children's tokens, and a residual
// pass reads the whole row (Algorithm 1); a leaf draws its terminal token from pi_CD alone.
// upload_q_rows_kernel copies exactly those rows from page-locked host memory, read by the SMs
// through its device mapping, in one launch: one CTA per row in turn, 16-byte loads where the
// row allows them.

#include <cuda_runtime.h>
#include <stdint.h>

#include "dcd.h"
#include "dcd_upload.h"

namespace dcd {
namespace {

constexpr int kUploadThreads = 512;

__global__ void __launch_bounds__(kUploadThreads) upload_q_rows_kernel(int32_t B, int32_t N, int64_t V, int64_t ldq,
                                                                       const float* __restrict__ src,
                                                                       float* __restrict__ dst,
                                                                       const int32_t* __restrict__ parents,
                                                                       const float* __restrict__ temperature,
                                                                       int vec) {
  const int64_t R = static_cast<int64_t>(B) * N;
  for (int64_t g = blockIdx.x; g < R; g += gridDim.x) {
    const int b = static_cast<int>(g / N), n = static_cast<int>(g % N);
    if (!(temperature[b] > 0.f)) continue;  // CTA-uniform
    // does node n have a child?  (children come after their parent in the tree order)
    const int32_t* par = parents + static_cast<int64_t>(b) * N;
    int found = 0;
    for (int c = n + 1 + static_cast<int>(threadIdx.x); c < N; c += kUploadThreads) found |= par[c] == n;
    if (!__syncthreads_or(found)) continue;
    const float* s = src + g * ldq;
    float* d = dst + g * ldq;
    if (vec) {
      const int64_t n4 = V / 4;
      const float4* s4 = reinterpret_cast<const float4*>(s);
      float4* d4 = reinterpret_cast<float4*>(d);
      for (int64_t i = threadIdx.x; i < n4; i += kUploadThreads) d4[i] = s4[i];
      for (int64_t i = n4 * 4 + threadIdx.x; i < V; i += kUploadThreads) d[i] = s[i];
    } else {
      for (int64_t i = threadIdx.x; i < V; i += kUploadThreads) d[i] = s[i];
    }
  }
}

}  // namespace

cudaError_t launch_upload_q_rows(int32_t B, int32_t N, int64_t V, int64_t ldq, const float* src_dev_view, float* dst,
                                 const int32_t* parents, const float* temperature, cudaStream_t stream) {
  const int64_t R = static_cast<int64_t>(B) * N;
  if (R == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int64_t grid = R < 4ll * sms ? R : 4ll * sms;
  const int vec = (reinterpret_cast<uintptr_t>(src_dev_view) % 16 == 0 && reinterpret_cast<uintptr_t>(dst) % 16 == 0 &&
                   ldq % 4 == 0)
                      ? 1
                      : 0;
  upload_q_rows_kernel<<<static_cast<unsigned>(grid), kUploadThreads, 0, stream>>>(B, N, V, ldq, src_dev_view, dst,
                                                                                   parents, temperature, vec);
  return cudaGetLastError();
}

}  // namespace dcd
