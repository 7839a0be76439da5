// dcd_internal.h -- declarations shared by the library's CUDA translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dcd {

// Workspace layout: a 256-byte header (word 0 = device error bits, word 1 = the row
// kernel's work counter, both zeroed at the start of every call), then one RowRecord per
// row g = b * N + n.
constexpr size_t kWorkspaceHeader = 256;

struct RowRecord {
  int32_t acc_child;   // accepted child node id, -1 if none
  int32_t term_token;  // terminal token of this node when acc_child < 0, else -1
  uint32_t status;     // DCD_DEVERR_* bits raised while scoring this row
  int32_t reserved;
};
static_assert(sizeof(RowRecord) == 16, "RowRecord layout");

struct ScoreArgs {
  const void* zp;
  const void* zq;
  const float* q;  // may be null (all-greedy call)
  int64_t ld, ldq, V;
  const int32_t* tokens;
  const int32_t* parents;
  const float* alpha;
  const float* beta;  // may be null
  const float* temp;  // may be null (all greedy)
  int32_t B, N;
  int32_t dtype;  // DCD_F32 / DCD_BF16
  uint64_t seed, offset;
  float* cd_logprob;  // may be null
  int32_t* cd_argmax; // may be null
  float* cd_lse;      // may be null
  RowRecord* rec;
  uint32_t* err;
  int32_t force_stages;   // 0 = automatic, else the ring depth to use (tests / tuning)
  int32_t force_plain;    // 1 = plain loads instead of bulk async copies
};

cudaError_t launch_score_rows(const ScoreArgs& a, cudaStream_t stream);

cudaError_t launch_tree_walk(int32_t B, int32_t N, const RowRecord* rec, uint32_t* err, int32_t* accept_len,
                             int32_t* accept_path, int32_t* bonus, cudaStream_t stream);

cudaError_t launch_terminal_residual(const ScoreArgs& a, const int32_t* accept_len, const int32_t* accept_path,
                                     const int32_t* bonus, float* residual, cudaStream_t stream);

// Launch geometry the row kernel would use for a call (exposed for diagnostics).
struct RowGeometry {
  int stages;        // ring depth per CTA
  int stage_tokens;  // vocabulary tokens per ring stage
  size_t smem;       // dynamic shared memory per CTA
  int ctas_per_sm;   // resident CTAs per SM
  int bulk;          // 1 when rows are staged with bulk asynchronous copies
};
RowGeometry row_geometry(const ScoreArgs& a);

}  // namespace dcd
