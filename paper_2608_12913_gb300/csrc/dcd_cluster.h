// dcd_cluster.h -- the cluster-per-row verification kernel (dcd_cluster.cu).
#pragma once

#include <cuda_runtime.h>

#include "dcd_internal.h"

namespace dcd {

// True when the call can take the cluster-per-row kernel: siblings drawn i.i.d., 16-byte aligned
// rows and a vocabulary whose slices fit the kernel's shared memory.
bool cluster_rows_ok(const ScoreArgs& a);

// The per-row step of dcd_score_rows on the cluster-per-row kernel: the call's records (read by
// the tree walk) and its Eq. 1 outputs.
cudaError_t launch_cluster_rows(const ScoreArgs& a, cudaStream_t stream);

}  // namespace dcd
