// dcd_small.h -- the one-launch greedy verification of small calls (dcd_small.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "dcd_internal.h"

namespace dcd {

constexpr int64_t kSmallMaxRows = 512;  // rows (B * N) up to which a greedy call takes one launch
constexpr int kSmallMaxNodes = 256;     // nodes per sequence up to which it does

// Whether a greedy verification call (a.q null) takes the one-launch path.
bool greedy_small_ok(const ScoreArgs& a);

// The whole greedy verification of a small call: rows and tree walk in one kernel (after a
// memset of the workspace counters).  Uses the workspace header, part counters, row records and
// part statistics of the common layout.
cudaError_t launch_greedy_small(const ScoreArgs& a, int32_t* accept_len, int32_t* accept_path, int32_t* bonus,
                                cudaStream_t stream);

}  // namespace dcd
