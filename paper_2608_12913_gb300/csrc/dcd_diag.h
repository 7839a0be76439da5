// dcd_diag.h -- internal declarations of the per-row diagnostics (dcd_diag.cu).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace dcd {

// Statistics of one chunk of one row's vocabulary (see dcd_diag.cu for their definitions).
struct alignas(16) DiagPart {
  float mp, sp, mq, sq, tq, a, e1, ez, h, tp, pad[2];
};
constexpr int kDiagCols = 8;  // diagnostics per row
constexpr int kDiagMinChunk = 2048;   // tokens per CTA of the streaming pass: at least ...
constexpr int kDiagMaxChunk = 16384;  // ... and at most
// Tokens per chunk for R rows of V tokens on a GPU with `sms` SMs (a multiple of kDiagMinChunk).
int diag_chunk(int64_t R, int64_t V, int sms);
inline size_t diag_workspace_bytes(int64_t R, int64_t V) {
  const size_t raw = static_cast<size_t>(R) * static_cast<size_t>((V + kDiagMinChunk - 1) / kDiagMinChunk) *
                     sizeof(DiagPart);
  return (raw + 255) & ~static_cast<size_t>(255);
}

struct DiagArgs {
  int64_t R, V, ld, ldq;
  int N;                 // nodes per sequence (row r belongs to sequence r / N)
  int dtype;
  const void* z_exp;
  const void* z_ama;
  const float* q;        // may be null
  const int32_t* xstar;  // may be null
  const float* cd_lse;   // [R] from a verification call, or null
  const float* alpha;    // [B], or null
  const float* beta;     // [B], or null (beta = 0)
  const float* temp;     // [B], or null (greedy)
  float* out;            // [R, kDiagCols]
  DiagPart* part;        // workspace
  cudaStream_t stream;
  void* start;  // optional cudaEvent_t pair around the streaming pass (timing)
  void* stop;
};
cudaError_t launch_diagnostics(const DiagArgs& d);

}  // namespace dcd
