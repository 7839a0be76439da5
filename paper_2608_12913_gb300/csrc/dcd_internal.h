// dcd_internal.h -- declarations shared by the library's CUDA translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dcd {

// Workspace layout, all in the caller's buffer:
//   [WsHeader, 256 B][part counter x R, padded to 16 B][Job x R][RowRecord x R]
//   [RowPart x kMaxParts x R][slot x R]
// The header and the part counters are zeroed at the start of every call; the rest is written
// before it is read.  R = B * N rows; a row streamed in parts leaves one RowPart
// per part; a slot (SlotHead + one PiecePart per residual piece) holds the chain state of a row
// whose first sibling was rejected.
constexpr size_t kWorkspaceHeader = 256;
#ifndef DCD_MAX_PARTS
#define DCD_MAX_PARTS 4
#endif
constexpr int kMaxParts = DCD_MAX_PARTS;  // parts a row may be split into

inline size_t part_counter_bytes(size_t rows) { return (rows * 4 + 15) & ~static_cast<size_t>(15); }

struct WsHeader {
  uint32_t err;        // DCD_DEVERR_* bits of the call (read by dcd_get_device_error)
  uint32_t work;       // rows claimed by the streaming kernel
  uint32_t job_alloc;       // residual passes created
  uint32_t jobs_published;  // passes published, in creation order
  uint32_t nslots;          // rows handed to residual passes
  uint32_t rows_done;       // rows whose record is written
  uint32_t job_head;        // passes before it have every piece claimed
  uint32_t reserved[57];
};
static_assert(sizeof(WsHeader) == kWorkspaceHeader, "WsHeader layout");

struct Job {             // one residual pass of one row, with what streaming it needs
  int32_t slot;          // the row's slot
  int32_t J;             // the pass (rejections so far, >= 1)
  uint32_t next_piece;   // pieces claimed
  uint32_t done;         // pieces finished
  int32_t g, m;          // row, children of its node
  uint32_t status;       // DCD_DEVERR_* bits of the row so far
  int32_t pad0;
  float M, S, Mp;        // the row's max, normaliser and expert max
  float c;               // c_J of the residual this pass sums
  float alpha, beta, T;  // the sequence's parameters
  int32_t pad1;
};
static_assert(sizeof(Job) == 64, "Job layout");

struct RowRecord {
  int32_t acc_child;   // accepted child node id, -1 if none
  int32_t term_token;  // terminal token of this node when acc_child < 0, else -1
  uint32_t status;     // DCD_DEVERR_* bits raised while scoring this row
  int32_t reserved;
};
static_assert(sizeof(RowRecord) == 16, "RowRecord layout");

struct RowPart {    // one part's statistics of a row streamed in parts
  float M, S;        // max of u over the part and sum of 2^(u - M)
  int32_t arg;       // argmax (lowest token on ties)
  float key;         // best terminal-race block key of the part (log2 mass without the row max)
  int32_t blk;       // its block, INT_MAX if none
  int32_t timed_out;
  int32_t pad[2];
};
static_assert(sizeof(RowPart) == 32, "RowPart layout");

struct SlotHead {  // chain state of a handed-over row
  int32_t g, m;    // row, children of its node
  float M, S, Mp;  // max CD score, normaliser sum 2^((s' - M) k2), expert max
  float c, D;      // c and mass of the current residual r = max(0, pi - c q) / D (as of the last pass)
  int32_t degen;   // a pass found no residual mass
  uint32_t status;
  float Z;         // distinct siblings: mass of q not yet removed
  int32_t nrem;    // distinct siblings: tokens removed (first occurrences), listed after the parts
  int32_t pad[5];
};
static_assert(sizeof(SlotHead) == 64, "SlotHead layout");

// Distinct siblings: a removed token and its frozen residual mass max(0, pi - c q) at the c in
// effect when it was removed (the residual does not change there afterwards: its proposal is 0).
struct Removed {
  int32_t tok;
  float fz;
};
constexpr int kMaxRemoved = 32;

struct PiecePart {  // one piece's share of a residual pass
  float z;          // sum of max(0, pi - c_J q) over the piece
  float key;        // best race key of the piece's blocks (last pass only)
  int32_t blk;      // its block
  float qs;         // sum of q over the piece (first pass, distinct siblings only)
};
static_assert(sizeof(PiecePart) == 16, "PiecePart layout");

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
  WsHeader* hdr;
  Job* jobs;
  uint32_t* pdone;  // per row: parts finished
  RowRecord* rec;
  RowPart* parts;   // per row: kMaxParts part statistics
  unsigned char* slots;
  int32_t distinct;       // 1: siblings drawn without replacement (DCD_SIBLINGS_DISTINCT)
  int32_t force_stages;   // 0 = automatic, else the ring depth to use (tests / tuning)
  int32_t force_plain;    // 1 = plain loads instead of bulk async copies
  int64_t poll_cycles;    // limit of a producer's poll for residual passes once its rows are
                          // done (0 = the default bounded wait; tests shorten it)
};

// Residual pieces per pass and slot bytes per row for a vocabulary of V tokens in a call of
// `rows` rows (small calls use smaller pieces).
int residual_pieces(int64_t V, int dtype, int64_t rows);
size_t slot_bytes(int64_t V, int dtype, int64_t rows);

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
