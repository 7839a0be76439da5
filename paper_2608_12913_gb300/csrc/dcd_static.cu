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
// host code must not pass it to a kernel, so its device address is looked up with
// cudaGetSymbolAddress, with the device current, and cached.  The cache is keyed on the device
// and on the unique id of the context current on it: after cudaDeviceReset (or anything else
// that creates a new context) the module is loaded again and the array may move, so a new
// context triggers a new lookup instead of reusing a dead address.

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdint.h>

#include <mutex>

#include "dcd.h"

static __device__ __align__(256) unsigned char g_dcd_static_scratch[DCD_STATIC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
struct ScratchCache {
  unsigned long long ctx_id;  // context the address belongs to (0: none yet)
  void* addr;
};
ScratchCache g_cache[kMaxDevices] = {};

// Driver entry points for the current context and its process-unique id, looked up once through
// the runtime (no link against the driver library).
struct CtxFns {
  PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  PFN_cuCtxGetId_v12000 get_id = nullptr;
};

const CtxFns& ctx_fns() {
  static std::once_flag once;
  static CtxFns f;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
  });
  return f;
}

// Id of the context current on this thread, 0 if there is none yet.
int current_ctx_id(unsigned long long* id) {
  const CtxFns& f = ctx_fns();
  if (!f.get_current || !f.get_id) return DCD_ERR_CUDA;
  CUcontext ctx = nullptr;
  if (f.get_current(&ctx) != CUDA_SUCCESS) return DCD_ERR_CUDA;
  *id = 0;
  if (ctx && f.get_id(ctx, id) != CUDA_SUCCESS) return DCD_ERR_CUDA;
  return DCD_OK;
}

// Device address of the scratch array in the current device's current context (looked up on the
// first use in each context).
int scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return DCD_ERR_CUDA;
  unsigned long long id = 0;
  int rc = current_ctx_id(&id);
  if (rc != DCD_OK) return rc;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (id == 0 || g_cache[dev].ctx_id != id || !g_cache[dev].addr) {
    void* p = nullptr;
    // also makes the device's primary context current when no context was yet
    if (cudaGetSymbolAddress(&p, g_dcd_static_scratch) != cudaSuccess || !p) return DCD_ERR_CUDA;
    if (id == 0) {
      rc = current_ctx_id(&id);
      if (rc != DCD_OK || id == 0) return DCD_ERR_CUDA;
    }
    g_cache[dev].ctx_id = id;
    g_cache[dev].addr = p;
  }
  *out = g_cache[dev].addr;
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
