// dcd_static.cu -- dcd_verify_sample_noalloc: the sampled/greedy verification with its scratch
// in a fixed device array compiled into the library, for callers that cannot allocate.
//
// Who needs this: code that runs where device allocation is not allowed or not safe, such as a
// plugin inside an inference engine whose device memory is entirely reserved and handed out by
// the engine's own allocator, or a hook that must not call cudaMalloc/cudaFree because those
// calls may synchronise the device or fail under a fixed memory budget.  Such a caller still
// owns and passes every input and output buffer; only the scratch (the per-row records and the
// device error word) moves into the array below.
//
// The array is a file-scope __device__ object, so every GPU that loads the library holds it
// (DCD_STATIC_SCRATCH_BYTES) until the process exits.  Its host-side name is only a handle:
// host code must not pass it to a kernel, so its device address is looked up once per device
// with cudaGetSymbolAddress, with that device current, and cached.

#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "dcd.h"

static __device__ __align__(256) unsigned char g_dcd_static_scratch[DCD_STATIC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up on first use).
int scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return DCD_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_dcd_static_scratch) != cudaSuccess || !p) return DCD_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return DCD_OK;
}

}  // namespace

extern "C" int dcd_verify_sample_noalloc(const dcd_shape* shape, const void* z_exp, const void* z_ama,
                                         const float* q, const int32_t* tokens, const int32_t* parents,
                                         const float* alpha, const float* beta, const float* temperature,
                                         uint64_t seed, uint64_t offset, int32_t* accept_len, int32_t* accept_path,
                                         int32_t* bonus, float* cd_logprob, int32_t* cd_argmax, float* cd_lse,
                                         float* residual, dcd_stream_t stream) {
  const size_t need = dcd_workspace_bytes(shape);
  if (need == 0) return DCD_ERR_INVALID_ARG;
  if (need > DCD_STATIC_SCRATCH_BYTES) return DCD_ERR_UNSUPPORTED;  // B*N above the fixed capacity
  void* scratch = nullptr;
  const int rc = scratch_address(&scratch);
  if (rc != DCD_OK) return rc;
  // Every call zeroes the error word and the work counter with a stream-ordered memset before
  // its kernels run, and rewrites every row record, so nothing left by an earlier call leaks in.
  return dcd_verify_sample(shape, z_exp, z_ama, q, tokens, parents, alpha, beta, temperature, seed, offset,
                           accept_len, accept_path, bonus, cd_logprob, cd_argmax, cd_lse, residual, scratch,
                           DCD_STATIC_SCRATCH_BYTES, stream);
}
