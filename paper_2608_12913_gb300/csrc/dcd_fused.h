// dcd_fused.h -- internal declarations of the greedy step fused with the two LM heads
// (dcd_fused.cu).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace dcd {

struct FusedArgs {
  int32_t B, N;
  int64_t V;
  int32_t H_exp, H_ama;
  const void* h_exp;  // bf16 [B*N, H_exp]
  const void* w_exp;  // bf16 [V, H_exp]
  const void* h_ama;  // bf16 [B*N, H_ama]
  const void* w_ama;  // bf16 [V, H_ama]
  const int32_t* tokens;
  const int32_t* parents;
  const float* alpha;
  const float* beta;  // fp32 [B] or null (beta = 0: one sweep); else two sweeps (max z_p first)
  int32_t* accept_len;
  int32_t* accept_path;
  int32_t* bonus;
  float* cd_logprob;
  int32_t* cd_argmax;
  float* cd_lse;
  void* workspace;
  cudaEvent_t gemm_start, gemm_stop;  // optional: recorded around the GEMM launch (timing)
};

// Workspace of the fused step: [WsHeader][child nodes][child tokens][child scores][row status]
// [RowRecord x R][tile statistics x R x ceil(V / 256)][row max of z_p x R] (byte offsets).
struct FusedLayout {
  size_t kid_node, kid_tok, kid_u, row_status, rec, part, zmax, total;
};
FusedLayout fused_layout(int64_t rows, int64_t V);

// Launches the fused step; *status is set to a DCD_ERR_* code for requests the launch cannot
// describe (tensor maps), with cudaSuccess returned.
cudaError_t launch_fused(const FusedArgs& f, cudaStream_t stream, int* status);

}  // namespace dcd
