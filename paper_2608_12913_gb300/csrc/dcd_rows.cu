// dcd_rows.cu -- the streaming kernels of the CD verification step on sm_103a.
//
// launch_score_rows runs cluster_rows_kernel (dcd_cluster.cu) whenever its geometry fits (rows
// 16 bytes aligned, no forced ring depth, plain loads or poll limit), for either sibling rule;
// score_rows_kernel below serves the forced geometries and unaligned rows.
//
// score_rows_kernel: a persistent, cooperatively launched grid (a few CTAs per SM).  Each CTA
// is warp-specialised: one producer warp claims work and streams it into a ring of 32 KB
// shared-memory stages with bulk asynchronous copies (one "full" mbarrier per stage, completed
// by the copies' byte count; one "empty" mbarrier per stage, on which the eight consumer warps
// release it); the eight consumer warps compute.  The producer runs ahead across work items:
// while the consumers finish one item (its last stages and its epilogue), the next item is
// already claimed, described to them through a small descriptor queue, and streaming in.
// Work comes in two kinds.
//
//  * Rows.  Whole tree-node rows g = b * N + n, claimed from a counter in node-major order
//    (every sequence's node 0, then every node 1, ...), so internal nodes -- the rows that may
//    start residual work -- come first and leaves last.  The "stats" pass computes the CD
//    score s' = (1 + alpha) z_p - alpha z_q (Eq. 1; the two log-softmax shifts are constant
//    per row and cancel in the normaliser) on the plausibility set P_beta of Sec. 2.1, in the
//    scaled unit u = k2 s' (k2 = log2(e) / T, so pi_CD,T ~ 2^u).  A warp takes a contiguous
//    eighth of each stage; every lane keeps an online max of u, a sum of 2^(u - max) rescaled
//    when its max grows, and its argmax, combined over the consumers at the end of the row.
//    With beta > 0 a "max" pass over z_p comes first.  Sampled rows also keep each warp's
//    share of the row's mass, from which a leaf gets the mass of every 1024-token block for
//    its terminal race.  The greedy rule, the first sibling test of the sampled rule and the
//    leaf race then finish the row.
//
//  * Residual pieces.  After a rejected sibling, Algorithm 1 (generalised to sibling lists)
//    needs the next residual over the whole vocabulary.  With c_0 = 0, D_0 = 1 the j-th
//    residual is r_j = max(0, pi - c_j q) / D_j, where c_j = c_{j-1} + D_{j-1} and D_j =
//    sum_x max(0, pi(x) - c_j q(x)) (induction on j from r_j = normalise(max(0, r_{j-1} -
//    q))), so a pass needs only two scalars from the one before.  A row that needs a pass is
//    handed to a job list; the pass is split into pieces of four ring stages (16384 tokens for
//    bf16 logits; two stages in a call of at most 256 rows) that any CTA's producer claims
//    before taking a new row.  Each piece writes its partial sum (and, in the pass after the
//    last sibling, its best race key) to its own slot; the CTA that finishes a pass's last piece
//    (an atomic ticket, no waiting) sums the slots in a fixed order while it lists the node's
//    children, tests the next sibling, and either queues the next pass or runs the terminal
//    race.  A producer with no row left polls for pieces until every row's record
//    is written (bounded; all CTAs are co-resident under a cooperative launch), so the passes
//    of late chains still spread over the GPU.
//
//  A node without an accepted child draws its terminal token by a two-level exponential
//  race: a 1024-token block by its mass, then a token of that block (four tokens a thread,
//  re-read directly).
// tree_walk_kernel: one warp per sequence follows the accepted children.
// terminal_residual_kernel: one block per sequence rebuilds the distribution its bonus
//   token was drawn from (test output only).

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <mutex>

#include "dcd.h"
#include "dcd_cluster.h"
#include "dcd_device.cuh"
#include "dcd_internal.h"

namespace dcd {
namespace {

using namespace dev;

#ifndef DCD_STAGE_KIB
#define DCD_STAGE_KIB 32
#endif
constexpr int kStageBytes = DCD_STAGE_KIB * 1024;  // bytes per ring stage
constexpr int kMaxStages = 8;
#ifndef DCD_PIECE_STAGES
#define DCD_PIECE_STAGES 4
#endif
#ifndef DCD_PARTS_BELOW
#define DCD_PARTS_BELOW 2
#endif
constexpr int kPieceStages = DCD_PIECE_STAGES;     // ring stages per residual piece (at most)
#ifndef DCD_SMALL_PIECE_ROWS
#define DCD_SMALL_PIECE_ROWS 256
#endif
#ifndef DCD_SMALL_PIECE_STAGES
#define DCD_SMALL_PIECE_STAGES 2
#endif
// A call with at most kSmallPieceRows rows splits residual passes into pieces of
// kSmallPieceStages stages: its chains of passes are on the critical path, and smaller pieces
// spread each pass over more CTAs (measured: 4% faster at 120 rows, neutral at 480; one-stage
// pieces were slower at 480 rows).
constexpr int64_t kSmallPieceRows = DCD_SMALL_PIECE_ROWS;
constexpr int kSmallPieceStages = DCD_SMALL_PIECE_STAGES;
// Rows are streamed in parts only when the batch has at most this many rows per resident CTA:
// then whole rows would leave most CTAs idle for part of the step; with more rows than that,
// dynamic claiming of whole rows balances better than parts (measured).
constexpr int kPartsBelow = DCD_PARTS_BELOW;
#ifndef DCD_TAIL_ROWS
#define DCD_TAIL_ROWS 0
#endif
// In a larger batch, the last kTailRows rows (in claim order) are streamed in parts (0: none).
constexpr int64_t kTailRows = DCD_TAIL_ROWS;
constexpr int kDesc = 4;                           // work descriptors in flight per CTA
#ifndef DCD_ROW_WARPS
#define DCD_ROW_WARPS 8
#endif
#ifndef DCD_MIN_CTAS
#define DCD_MIN_CTAS 3
#endif
#ifndef DCD_RING_STAGES
#define DCD_RING_STAGES 2
#endif
constexpr int kRowWarps = DCD_ROW_WARPS;           // consumer warps per CTA
constexpr int kRowThreads = kRowWarps * 32;
constexpr int kCtaThreads = kRowThreads + 32;      // the consumer warps and one producer warp
constexpr int kMinCtasPerSm = DCD_MIN_CTAS;
constexpr int kRingStages = DCD_RING_STAGES;       // default ring depth
static_assert(kRowWarps == 8 || kRowWarps == 12 || kRowWarps == 16, "consumer warps");
using RowSync = SyncConsumersN<kRowThreads>;
constexpr size_t kSmemMax = 227 * 1024;
constexpr size_t kSmemPerSm = 228 * 1024;
constexpr float kLn2 = 0.69314718055994531f;

enum WorkKind { kWorkNone = 0, kWorkRow = 1, kWorkPiece = 2, kWorkPart = 3 };

// ------------------------------------------------------------------------------------------
struct SParams {
  ScoreArgs a;
  int32_t nst;           // ring depth (stages of kStageBytes)
  int32_t tok_a;         // tokens per stage in row passes (z_p, then z_q)
  int32_t tok_r;         // tokens per stage in residual pieces (z_p, z_q, then q)
  int32_t npieces;       // pieces per residual pass
  int32_t piece_stages;  // ring stages per residual piece
  int32_t bulk;          // 1: bulk asynchronous copies, 0: plain loads
  int32_t nblk;          // race blocks per row, ceil(V / 1024)
  int32_t nchunk;        // warp chunks per row in the stats pass, ceil(V / (tok_a / 8))
  int32_t meta_offset;   // byte offsets into dynamic shared memory
  int32_t chunk_offset;
  int32_t stage_offset;
  int32_t slot_bytes;
  int32_t r_whole;       // row items streamed whole; the rows after them are streamed in parts
  int32_t parts;         // parts of such a row (stages of the stats pass split in runs of spp)
  int32_t spp;           // stats-pass stages per part
  int32_t items;         // row items: r_whole + (R - r_whole) * parts
  int32_t keep_internal; // small batch: keep sampled internal rows and pieces in L2 (evict-last)
  long long poll_cycles; // bound of the end-of-work poll for residual passes
  WsHeader* hdr;         // counters, zeroed before the launch
  Job* jobs;             // residual passes (zeroed before the launch)
  unsigned char* slots;  // per handed-over row: SlotHead + npieces PieceParts
};

// A work item as the producer hands it to the consumers.
struct WorkDesc {
  int32_t kind;        // WorkKind
  int32_t g;           // row
  int32_t job, piece;  // residual piece: job index and piece index; row part: part index
  int32_t J;           // residual pass (rejections so far)
  int32_t slot;        // slot of the handed-over row
  int32_t m;           // children of the row's node
  uint32_t status;     // DCD_DEVERR_* bits carried by the slot
  float alpha, beta, T;
  float M, S, Mp, c;   // pieces: the row's max, normaliser, expert max and c_J
  int32_t pad;
};
static_assert(sizeof(WorkDesc) == 64, "WorkDesc layout");

// Consumer state shared by the eight consumer warps (written by one thread, read after a
// consumer barrier).
struct RowShared {
  int32_t m;        // children of the row's node
  uint32_t status;  // DCD_DEVERR_* bits
  int32_t accept;   // outcome of a sibling test
  int32_t term;     // winning race block of a completed pass
  int32_t last;     // this CTA finished a pass's last piece
  int32_t degen;    // a pass found no residual mass left
  float c, D;
  // Distinct siblings: a chain's removed tokens, their frozen masses, and pi and q at them (then
  // at siblings J - 1 and J), read by two warps in parallel before a pass's sibling step
  int32_t rn;
  int32_t rtok[kMaxRemoved + 2];
  float rfz[kMaxRemoved + 2];
  float rpit[kMaxRemoved + 2];
  float rq[kMaxRemoved + 2];
};
static_assert(kMaxRemoved <= 32, "one lane a removed token");

template <typename TIn>
struct Stage {
  TIn* zp;
  TIn* zq;
  float* q;
};

// A stage holds `tok` tokens of z_p, then of z_q, then (residual pieces) of q.
template <typename TIn>
__device__ __forceinline__ Stage<TIn> stage_at(unsigned char* base, int s, int tok) {
  Stage<TIn> st;
  st.zp = reinterpret_cast<TIn*>(base + static_cast<size_t>(s) * kStageBytes);
  st.zq = st.zp + tok;
  st.q = reinterpret_cast<float*>(st.zq + tok);
  return st;
}

__device__ __forceinline__ uint32_t ld_volatile(const uint32_t* p) {
  return *reinterpret_cast<const volatile uint32_t*>(p);
}

__device__ __forceinline__ SlotHead* slot_head(const SParams& sp, int s) {
  return reinterpret_cast<SlotHead*>(sp.slots + static_cast<size_t>(s) * sp.slot_bytes);
}

__device__ __forceinline__ PiecePart* slot_parts(const SParams& sp, int s) {
  return reinterpret_cast<PiecePart*>(sp.slots + static_cast<size_t>(s) * sp.slot_bytes + sizeof(SlotHead));
}

// Distinct siblings: the removed tokens of a chain, after its pieces' parts.
__device__ __forceinline__ Removed* slot_removed(const SParams& sp, int s) {
  return reinterpret_cast<Removed*>(sp.slots + static_cast<size_t>(s) * sp.slot_bytes + sizeof(SlotHead) +
                                    static_cast<size_t>(sp.npieces) * sizeof(PiecePart));
}

__device__ __forceinline__ int find_removed(const Removed* rem, int nrem, int t) {
  for (int i = 0; i < nrem; ++i)
    if (rem[i].tok == t) return i;
  return -1;
}

// Publishes residual pass `job` (its counters are reset here; one consumer thread).  Passes are
// published in creation order, so the passes with unclaimed pieces are the window [job_head,
// jobs_published); the wait for the previous creator spans a few stores and is bounded.
__device__ __forceinline__ void create_job(const SParams& sp, Job job) {
  const uint32_t k = atomicAdd(&sp.hdr->job_alloc, 1u);
  job.next_piece = 0u;
  job.done = 0u;
  job.pad0 = job.pad1 = 0;
  sp.jobs[k] = job;
  __threadfence();
  const long long t0 = clock64();
  while (ld_volatile(&sp.hdr->jobs_published) != k) {
    if (clock64() - t0 > kWaitCycles) {
      atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
      break;
    }
  }
  *reinterpret_cast<volatile uint32_t*>(&sp.hdr->jobs_published) = k + 1u;
}

// A published pass record, read past the non-coherent L1.
__device__ __forceinline__ Job load_job(const Job* j) {
  Job r;
  const int4* src = reinterpret_cast<const int4*>(j);
  int4* dst = reinterpret_cast<int4*>(&r);
#pragma unroll
  for (int i = 0; i < 4; ++i) dst[i] = __ldcg(src + i);
  return r;
}

// Lists the children of node n (ascending id) into kids / ktok with the calling warp; returns
// their count in every lane.
__device__ __forceinline__ int list_children(const ScoreArgs& p, int b, int n, int* kids, int* ktok) {
  const int lane = threadIdx.x & 31;
  const int32_t* parr = p.parents + static_cast<int64_t>(b) * p.N;
  const int32_t* tokr = p.tokens + static_cast<int64_t>(b) * p.N;
  int count = 0;
  for (int base = n + 1; base < p.N; base += 32) {
    const int c = base + lane;
    const bool is = c < p.N && parr[c] == n;
    const unsigned msk = __ballot_sync(~0u, is);
    if (is) {
      const int pos = count + __popc(msk & ((1u << lane) - 1u));
      kids[pos] = c;
      ktok[pos] = tokr[c];
    }
    count += __popc(msk);
  }
  __syncwarp();
  return count;
}

// The scaled CD score u = c1k z_p - ak z_q of 8 tokens of a stage; tokens past `clen` or
// outside P_beta get -inf.  A whole 256-token group of an unmasked row skips the per-token
// predicates and uses packed fp32x2 arithmetic (the same roundings as the scalar path).
template <typename TIn>
__device__ __forceinline__ void scores8(const TIn* zp_s, const TIn* zq_s, int i0, int sb, int clen, bool masked,
                                        float c1k, float ak, float Mp, float logb, float u[8]) {
  if (!masked && sb + kSub <= clen) {
    const float2 c1k2 = make_float2(c1k, c1k), nak2 = make_float2(-ak, -ak);
    float2 zp2[4], zq2[4];
    ld8x2(zp_s + i0, zp2);
    ld8x2(zq_s + i0, zq2);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 s2 = __ffma2_rn(zp2[k], c1k2, __fmul2_rn(zq2[k], nak2));
      u[2 * k] = s2.x;
      u[2 * k + 1] = s2.y;
    }
  } else {
    float zp[8], zq[8];
    ld8(zp_s + i0, zp);
    ld8(zq_s + i0, zq);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const bool in = (i0 + e < clen) && (!masked || (zp[e] - Mp >= logb));
      u[e] = in ? fmaf(c1k, zp[e], -ak * zq[e]) : -INFINITY;
    }
  }
}

// The sibling test of child `node` (token t): accept iff u <= r(t) / q(t) with
// r = max(0, pi - c q) / D, or r = q once a pass found no residual mass (`degen`); pi(t) =
// 2^(u(t) - M) / S.  One thread.
template <typename TIn>
__device__ bool sibling_test(const ScoreArgs& p, int b, int node, int t, const TIn* zp_row, const TIn* zq_row,
                             const float* q_row, float c1k, float ak, bool masked, float Mp, float logb, float M,
                             float invS, float c, float D, bool degen) {
  const bool ok = t >= 0 && t < p.V;
  const float z = ok ? ld1(zp_row, t) : 0.f;
  const float zz = ok ? ld1(zq_row, t) : 0.f;
  const float qt = ok ? q_row[t] : 0.f;
  const bool in = ok && (!masked || (z - Mp >= logb));
  const float pit = in ? ex2(fmaf(c1k, z, -ak * zz) - M) * invS : 0.f;
  const float rt = degen ? qt : fmaxf(pit - c * qt, 0.f) / D;
  const float ratio = qt > 0.f ? rt / qt : (rt > 0.f ? INFINITY : 0.f);
  const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * p.N + node);
  const float u = u01(philox_block(p.seed, p.offset, G, 0u).x);
  return u <= ratio;
}

// Second level of the terminal race: the token x of race block `kstar` with the largest
// log2 r(x) - log2(-log2 u_x), four tokens a consumer thread (one Philox call, counter
// 1 + x / 4).  `mass(x)` returns r(x) up to a common factor.  Every consumer thread calls it
// and gets the token (INT_MAX when no block had mass).
template <typename MassFn>
__device__ int token_race(const ScoreArgs& p, int64_t g, int kstar, MassFn mass, float* redf, int* redi) {
  float tk = -INFINITY;
  int tx = INT_MAX;
  if (kstar != INT_MAX && threadIdx.x < kRaceBlock / 4) {
    const int64_t x = static_cast<int64_t>(kstar) * kRaceBlock + threadIdx.x * 4;
    if (x < p.V) {
      const uint4 w =
          philox_block(p.seed, p.offset, static_cast<uint32_t>(g), 1u + static_cast<uint32_t>(x >> 2));
      const uint32_t words[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (x + e < p.V) {
          const float v = mass(x + e);
          if (v > 0.f) {
            const float key = race_key(lg2(v), words[e]);
            if (key > tk) {
              tk = key;
              tx = static_cast<int>(x + e);
            }
          }
        }
      }
    }
  }
  block_argmax(tk, tx, redf, redi, RowSync());
  return tx;
}

// First level of the race for one block: its key from log2 of its mass.
__device__ __forceinline__ float block_key(const ScoreArgs& p, int64_t g, int k, float log2_mass) {
  const uint4 w =
      philox_block(p.seed, p.offset, static_cast<uint32_t>(g), 0x80000000u | (static_cast<uint32_t>(k) >> 2));
  return race_key(log2_mass, word_of(w, k & 3));
}

__device__ __forceinline__ void warp_release(uint64_t* bar) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

// ------------------------------------------------------------------------------------------
// kDistinct: siblings drawn without replacement (a separate instantiation, so that the i.i.d.
// rule's code and registers are untouched by the distinct rule's bookkeeping).
template <typename TIn, bool kDistinct>
__global__ void __launch_bounds__(kCtaThreads, kMinCtasPerSm) score_rows_kernel(const __grid_constant__ SParams sp) {
  const ScoreArgs& p = sp.a;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int N = p.N;
  const int64_t V = p.V;
  const int R = p.B * N;
  const int nch_a = static_cast<int>((V + sp.tok_a - 1) / sp.tok_a);  // stages of a max / stats pass
  const RowSync csync;

  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);  // [kMaxStages] stage filled
  uint64_t* empty = full + kMaxStages;                 // [kMaxStages] stage released by the consumers
  uint64_t* dfull = empty + kMaxStages;                // [kDesc] descriptor written
  uint64_t* dempty = dfull + kDesc;                    // [kDesc] descriptor released
  float* redf = reinterpret_cast<float*>(dempty + kDesc);  // [32]
  int* redi = reinterpret_cast<int*>(redf + 32);           // [32]
  WorkDesc* desc = reinterpret_cast<WorkDesc*>(redi + 32); // [kDesc]
  RowShared* rs = reinterpret_cast<RowShared*>(smem + sp.meta_offset);
  int* kids = reinterpret_cast<int*>(rs + 1);                    // [N] children, ascending id
  int* ktok = kids + N;                                          // [N] their tokens
  float* czp = reinterpret_cast<float*>(ktok + N);               // [N] z_p at those tokens
  float* czq = czp + N;                                          // [N] z_q at those tokens
  float* cq = czq + N;                                           // [N] q at those tokens
  float* cref = reinterpret_cast<float*>(smem + sp.chunk_offset);  // [nchunk] warp chunk reference
  float* csum = cref + sp.nchunk;                                // [nchunk] chunk sum of 2^(u - ref)
  unsigned char* ring = smem + sp.stage_offset;

  if (tid == 0) {
    for (int s = 0; s < sp.nst; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kRowWarps);
    }
    for (int d = 0; d < kDesc; ++d) {
      mbar_init(&dfull[d], 1);
      mbar_init(&dempty[d], 1);
    }
    fence_mbar_init();
  }
  __syncthreads();  // the last CTA-wide barrier: from here on the two roles synchronise by mbarriers

  if (warp == kRowWarps) {
    // ===================================== producer warp
    const uint64_t pol_last = l2_policy_evict_last();
    const uint64_t pol_normal = l2_policy_evict_normal();
    const uint64_t pol_first = l2_policy_evict_first();
    uint32_t issued = 0;  // ring items issued

    // The next row item and what streaming it needs are fetched while the current item streams,
    // so switching items costs no dependent round trip; `nr` is claimed one ahead.
    struct RowMeta {
      int item, g, part, m;
      float alpha, beta, T;
    };
    auto load_meta = [&](int item) -> RowMeta {  // the whole warp, `item` uniform
      RowMeta mt;
      mt.item = item;
      mt.g = -1;
      mt.part = -1;
      mt.m = 0;
      mt.alpha = mt.beta = mt.T = 0.f;
      if (item >= sp.items) return mt;
      int r = item;  // row items: whole rows in node-major order, then parts of the last rows
      if (item >= sp.r_whole) {
        r = sp.r_whole + (item - sp.r_whole) / sp.parts;
        mt.part = (item - sp.r_whole) % sp.parts;
      }
      const int b = r % p.B, n = r / p.B;
      mt.g = b * N + n;
      mt.alpha = p.alpha[b];
      mt.beta = p.beta ? p.beta[b] : 0.f;
      mt.T = p.temp ? p.temp[b] : 0.f;
      const int32_t* parr = p.parents + static_cast<int64_t>(b) * N;  // children of node n
      for (int base = n + 1; base < N; base += 32) {
        const int c = base + lane;
        mt.m += __popc(__ballot_sync(~0u, c < N && parr[c] == n));
      }
      return mt;
    };
    int nr = 0;  // lane 0: the next row item (its claim returns while the current item streams)
    if (lane == 0) nr = static_cast<int>(atomicAdd(&sp.hdr->work, 1u));
    RowMeta meta;
    bool meta_stale = true;  // `meta` was used; the next one is fetched after the next issue
    auto refresh_meta = [&]() {  // the whole warp
      nr = __shfl_sync(~0u, nr, 0);
      meta = load_meta(nr);
      meta_stale = false;
    };
    refresh_meta();
    uint32_t pub_seen = 0u, head_seen = 0u;  // job-list state read before the last issue (lane 0)

    for (uint32_t w = 0;; ++w) {
      // ---- claim: a residual piece if one is available, else the next row item; with no row
      // item left, poll (bounded) for pieces until every row's record is written.  The last row
      // items are parts of rows, so the rows still streaming at the end are spread over more CTAs.
      int kind = kWorkNone;
      WorkDesc D;
      int nitems = 0, tok = sp.tok_a, nmax = 0;  // items; tokens per item; leading max-pass items
      bool with_q = false;
      uint64_t pol = pol_first;
      int64_t x_lo = 0;
      for (bool skip = true; skip;) {
        skip = false;
        if (meta_stale) refresh_meta();  // after a skipped part
        int item = 0, piece = 0;
        kind = kWorkNone;
        Job job_rec;  // lane 0: the claimed pass
        {
          const uint32_t np_u = static_cast<uint32_t>(sp.npieces);
          const long long t0 = clock64();
          for (int poll = 0;; ++poll) {
            uint32_t pub = 0u, k0 = 0u;
            if (lane == 0) {
              pub = poll ? ld_volatile(&sp.hdr->jobs_published) : pub_seen;
              k0 = poll ? ld_volatile(&sp.hdr->job_head) : head_seen;
            }
            pub = __shfl_sync(~0u, pub, 0);
            k0 = __shfl_sync(~0u, k0, 0);
            // a piece of the oldest published pass that still has one: the lanes look at 32
            // passes at once and only a pass seen open is claimed from (one atomic), so a stale
            // view of the list costs one round of loads, not an atomic per drained pass.  Every
            // pass before the claimed one was seen drained, so whoever claims the last piece of a
            // pass may move the head past it.
            for (; k0 < pub && kind == kWorkNone; k0 += 32u) {
              const uint32_t k = k0 + static_cast<uint32_t>(lane);
              const bool open = k < pub && ld_volatile(&sp.jobs[k].next_piece) < np_u;
              for (unsigned avail = __ballot_sync(~0u, open); avail != 0u; avail &= avail - 1u) {
                const uint32_t kc = k0 + static_cast<uint32_t>(__ffs(avail) - 1);
                uint32_t pc = 0u;
                if (lane == 0) pc = atomicAdd(&sp.jobs[kc].next_piece, 1u);
                pc = __shfl_sync(~0u, pc, 0);
                if (pc < np_u) {
                  kind = kWorkPiece;
                  item = static_cast<int>(kc);
                  piece = static_cast<int>(pc);
                  if (lane == 0) {
                    if (pc + 1u == np_u) atomicMax(&sp.hdr->job_head, kc + 1u);
                    __threadfence();  // the record was written before the pass was published
                    job_rec = load_job(&sp.jobs[kc]);
                  }
                  break;
                }
              }
            }
            if (kind != kWorkNone) break;
            if (meta.g >= 0) {
              kind = kWorkRow;
              if (lane == 0) nr = static_cast<int>(atomicAdd(&sp.hdr->work, 1u));  // read after the next issue
              break;
            }
            int stop = 0;
            if (lane == 0) {
              if (poll && ld_volatile(&sp.hdr->rows_done) >= static_cast<uint32_t>(R)) {
                stop = 1;
              } else if (clock64() - t0 > sp.poll_cycles) {
                atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
                stop = 1;
              }
            }
            if (__shfl_sync(~0u, stop, 0)) break;
            if (poll) __nanosleep(256);
          }
        }
        kind = __shfl_sync(~0u, kind, 0);
        item = __shfl_sync(~0u, item, 0);
        piece = __shfl_sync(~0u, piece, 0);

        D.kind = kind;
        D.g = 0;
        D.job = item;
        D.piece = piece;
        D.J = 0;
        D.slot = 0;
        D.m = 0;
        D.status = 0u;
        D.alpha = D.beta = D.T = 0.f;
        D.M = D.S = D.Mp = D.c = 0.f;
        D.pad = 0;
        nitems = 0;
        tok = sp.tok_a;
        nmax = 0;
        with_q = false;
        pol = pol_first;
        x_lo = 0;
        if (kind == kWorkRow) {
          meta_stale = true;
          D.g = meta.g;
          D.m = meta.m;
          D.alpha = meta.alpha;
          D.beta = meta.beta;
          D.T = meta.T;
          const bool masked = D.beta > 0.f;
          const bool sampled = D.T > 0.f && p.q != nullptr;
          // In a small batch a sampled internal row keeps its logits in L2 for residual passes,
          // which are then on the critical path.  In a large batch only about a quarter of those
          // rows take a pass, and keeping them all crowds L2: every row is streamed evict-first
          // (measured both ways).
          pol = (sampled && meta.m > 0 && sp.keep_internal) ? pol_last : pol_first;
          if (meta.part >= 0 && !masked) {
            D.kind = kWorkPart;
            D.piece = meta.part;
            x_lo = static_cast<int64_t>(meta.part) * sp.spp * sp.tok_a;
            nitems = nch_a - meta.part * sp.spp < sp.spp ? nch_a - meta.part * sp.spp : sp.spp;
          } else if (meta.part > 0) {
            skip = true;  // a beta > 0 row needs its expert max first: its part 0 streams it whole
          } else {
            nmax = masked ? nch_a : 0;
            nitems = nmax + nch_a;
          }
        } else if (kind == kWorkPiece) {
          if (lane == 0) {
            D.slot = job_rec.slot;
            D.J = job_rec.J;
            D.g = job_rec.g;
            D.m = job_rec.m;
            D.M = job_rec.M;
            D.S = job_rec.S;
            D.Mp = job_rec.Mp;
            D.c = job_rec.c;
            D.status = job_rec.status;
            D.alpha = job_rec.alpha;
            D.beta = job_rec.beta;
            D.T = job_rec.T;
          }
          D.g = __shfl_sync(~0u, D.g, 0);
          D.J = __shfl_sync(~0u, D.J, 0);
          D.m = __shfl_sync(~0u, D.m, 0);
          tok = sp.tok_r;
          x_lo = static_cast<int64_t>(piece) * sp.piece_stages * sp.tok_r;
          const int64_t rem = (V - x_lo + sp.tok_r - 1) / sp.tok_r;
          nitems = static_cast<int>(rem < sp.piece_stages ? rem : sp.piece_stages);
          with_q = true;
          // a later pass re-reads the piece; the pass after the last sibling is the last read
          pol = D.J < D.m ? (sp.keep_internal ? pol_last : pol_normal) : pol_first;
        }
      }
      // ---- publish the descriptor
      if (lane == 0) {
        const int d = static_cast<int>(w % kDesc);
        if (!mbar_wait_bounded(&dempty[d], ((w / kDesc) & 1u) ^ 1u)) atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
        desc[d] = D;
        mbar_arrive(&dfull[d]);
      }
      if (kind == kWorkNone) break;

      // ---- stream the item's stages
      const int64_t g = D.g;
      const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
      const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;
      const float* q_row = with_q ? p.q + g * p.ldq : nullptr;
      for (int L = 0; L < nitems; ++L, ++issued) {
        const int s = static_cast<int>(issued % static_cast<uint32_t>(sp.nst));
        const uint32_t phase = ((issued / static_cast<uint32_t>(sp.nst)) & 1u) ^ 1u;
        const bool maxpass = L < nmax;
        const int64_t x0 = x_lo + static_cast<int64_t>(maxpass ? L : L - nmax) * tok;
        const int clen = static_cast<int>((V - x0) < tok ? (V - x0) : tok);
        const Stage<TIn> st = stage_at<TIn>(ring, s, tok);
        if (lane == 0 && L == nitems - 1) {  // read for the next claim while the stage drains
          pub_seen = ld_volatile(&sp.hdr->jobs_published);
          head_seen = ld_volatile(&sp.hdr->job_head);
        }
        if (lane == 0 && !mbar_wait_bounded(&empty[s], phase)) atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
        __syncwarp();
        if (!sp.bulk) {
          // plain loads (rows whose start or stride is not 16-byte aligned)
          for (int i = lane; i < clen; i += 32) {
            st.zp[i] = zp_row[x0 + i];
            if (!maxpass) st.zq[i] = zq_row[x0 + i];
            if (with_q) st.q[i] = q_row[x0 + i];
          }
          __threadfence_block();
          __syncwarp();
          if (lane == 0) mbar_arrive(&full[s]);
        } else if (lane == 0) {
          // bulk copies of the 16-byte multiple; the ragged remainder is stored first
          const int zfirst = ((clen * static_cast<int>(sizeof(TIn))) & ~15) / static_cast<int>(sizeof(TIn));
          const int qfirst = ((clen * 4) & ~15) / 4;
          for (int i = zfirst; i < clen; ++i) {
            st.zp[i] = zp_row[x0 + i];
            if (!maxpass) st.zq[i] = zq_row[x0 + i];
          }
          if (with_q)
            for (int i = qfirst; i < clen; ++i) st.q[i] = q_row[x0 + i];
          const uint32_t zb = static_cast<uint32_t>(zfirst) * static_cast<uint32_t>(sizeof(TIn));
          const uint32_t qb = with_q ? static_cast<uint32_t>(qfirst) * 4u : 0u;
          const uint64_t pl = maxpass ? pol_last : pol;  // the stats pass re-reads the max pass
          mbar_arrive_expect_tx(&full[s], (maxpass ? zb : 2u * zb) + qb);
          if (zb) {
            bulk_g2s(st.zp, zp_row + x0, zb, &full[s], pl);
            if (!maxpass) bulk_g2s(st.zq, zq_row + x0, zb, &full[s], pl);
          }
          if (qb) bulk_g2s(st.q, q_row + x0, qb, &full[s], pl);
        }
        if (L == 0 && meta_stale) refresh_meta();  // the next row item's metadata, while this item streams
      }
    }
    return;
  }

  // ===================================== consumer warps
  uint32_t seq = 0;  // ring items consumed (identical in every consumer thread)
  bool timed_out = false;
  auto wait_full = [&](uint32_t sq) {
    if (!mbar_wait_bounded(&full[sq % static_cast<uint32_t>(sp.nst)], (sq / static_cast<uint32_t>(sp.nst)) & 1u))
      timed_out = true;
  };

  for (uint32_t w = 0;; ++w) {
    const int d = static_cast<int>(w % kDesc);
    if (!mbar_wait_bounded(&dfull[d], (w / kDesc) & 1u)) {
      if (tid == 0) atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
      break;
    }
    const WorkDesc D = desc[d];
    if (D.kind == kWorkNone) break;
    timed_out = false;

    const int64_t g = D.g;
    const int b = static_cast<int>(g / N), n = static_cast<int>(g % N);
    const float alpha = D.alpha, beta = D.beta, T = D.T;
    const bool masked = beta > 0.f;
    const float k2 = kLog2e * (T > 0.f ? 1.f / T : 1.f);  // exp(x / T) = 2^(x * k2)
    // scores are kept in the scaled unit u = k2 s' = c1k z_p - ak z_q, so pi_CD,T ~ 2^u
    const float c1k = (1.f + alpha) * k2, ak = alpha * k2;
    const float logb = masked ? logf(beta) : -INFINITY;
    const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
    const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;

    if (D.kind == kWorkPiece) {
      // ================= one piece of residual pass J of a handed-over row
      const int J = D.J, m = D.m, piece = D.piece;
      const float M = D.M, invS = 1.f / D.S, Mp = D.Mp, cJ = D.c;
      const bool race = J == m;  // the pass after the last sibling also ranks race blocks
      const float* q_row = p.q + g * p.ldq;
      // a warp takes tok_r / 8 consecutive tokens of each stage (a chunk); `wpb` chunks make a
      // race block
      const int tpw = sp.tok_r / kRowWarps, wpb = kRaceBlock / tpw;
      const int64_t piece_lo = static_cast<int64_t>(piece) * sp.piece_stages * sp.tok_r;
      const int64_t rem = (V - piece_lo + sp.tok_r - 1) / sp.tok_r;
      const int nst_piece = static_cast<int>(rem < sp.piece_stages ? rem : sp.piece_stages);
      // distinct siblings: the first pass also sums q, whose actual mass (the drafter's q may be
      // truncated or rounded away from 1) normalises the proposal once a token is removed
      const bool sum_q = kDistinct && J == 1;
      float zl = 0.f, ql = 0.f;
      for (int L = 0; L < nst_piece; ++L, ++seq) {
        const Stage<TIn> st = stage_at<TIn>(ring, static_cast<int>(seq % static_cast<uint32_t>(sp.nst)), sp.tok_r);
        const int64_t x0 = piece_lo + static_cast<int64_t>(L) * sp.tok_r;
        const int clen = static_cast<int>((V - x0) < sp.tok_r ? (V - x0) : sp.tok_r);
        wait_full(seq);
        float part = 0.f;
        for (int sb = warp * tpw; sb < (warp + 1) * tpw && sb < clen; sb += kSub) {  // warp-uniform
          const int i0 = sb + lane * 8;
          float u[8], qv[8];
          scores8(st.zp, st.zq, i0, sb, clen, masked, c1k, ak, Mp, logb, u);
          ld8(st.q + i0, qv);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            part += (i0 + e < clen) ? fmaxf(ex2(u[e] - M) * invS - cJ * qv[e], 0.f) : 0.f;
          if (sum_q) {
#pragma unroll
            for (int e = 0; e < 8; ++e) ql += (i0 + e < clen) ? qv[e] : 0.f;
          }
        }
        zl += part;
        if (race) {
          const float ws = warp_sum(part);
          if (lane == 0) csum[L * kRowWarps + warp] = ws;
        }
        warp_release(&empty[seq % static_cast<uint32_t>(sp.nst)]);
      }
      const float zsum = block_sum(zl, redf, csync);  // its barriers also publish csum
      const float qsum = sum_q ? block_sum(ql, redf, csync) : 0.f;
      // race keys of the piece's blocks (the pass after the last sibling)
      float bk = -INFINITY;
      int bb = INT_MAX;
      if (race && tid < nst_piece * (sp.tok_r / kRaceBlock) &&
          piece_lo + static_cast<int64_t>(tid) * kRaceBlock < V) {
        float mass = 0.f;
        for (int i = 0; i < wpb; ++i) mass += csum[tid * wpb + i];
        const int kabs = static_cast<int>(piece_lo / kRaceBlock) + tid;
        if (kDistinct) {
          // removed siblings' tokens in this block carry their frozen mass, not the streamed one
          const SlotHead* sh = slot_head(sp, D.slot);
          const Removed* rem = slot_removed(sp, D.slot);
          const int nrem = sh->nrem;
          for (int i = 0; i < nrem; ++i) {
            const int t = rem[i].tok;
            if (t / kRaceBlock != kabs) continue;
            const float z = ld1(zp_row, t);
            const bool in = !masked || (z - Mp >= logb);
            const float pit = in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, t)) - M) * invS : 0.f;
            mass += rem[i].fz - fmaxf(pit - cJ * q_row[t], 0.f);
          }
        }
        if (mass > 0.f) {
          bk = block_key(p, g, kabs, lg2(mass));
          bb = kabs;
        }
      }
      if (race) block_argmax(bk, bb, redf, redi, csync);  // CTA-uniform; other passes rank no blocks
      if (tid == 0) {
        PiecePart pp;
        pp.z = zsum;
        pp.key = bk;
        pp.blk = bb;
        pp.qs = qsum;
        // a wait that gave up fails the call (the tree walk reads the error word)
        if (timed_out) atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
        slot_parts(sp, D.slot)[piece] = pp;
        const uint32_t t = atomic_add_acq_rel(&sp.jobs[D.job].done, 1u);
        rs->last = t + 1u == static_cast<uint32_t>(sp.npieces) ? 1 : 0;
      }
      csync();
      if (rs->last) {
        // ================= the pass is complete: next sibling test, next pass or terminal race
        // pi at token t (0 outside P_beta) and q there, as every sibling step computes them
        auto value_at = [&](int t, float& pit, float& qt) {
          const float z = ld1(zp_row, t);
          const bool in = !masked || (z - Mp >= logb);
          pit = in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, t)) - M) * invS : 0.f;
          qt = q_row[t];
        };
        if (warp == 0) {
          const int cnt = list_children(p, b, n, kids, ktok);
          if (kDistinct && lane < 2) {  // the values at siblings J - 1 (removed now) and J (tested next)
            const int j = J - 1 + lane;
            const int t = j < cnt ? ktok[j] : -1;
            const bool ok = t >= 0 && t < V;
            rs->rtok[kMaxRemoved + lane] = ok ? t : -1;
            if (ok) value_at(t, rs->rpit[kMaxRemoved + lane], rs->rq[kMaxRemoved + lane]);
          }
        }
        if (kDistinct && warp == 2) {  // the removed tokens so far and the values at them
          const int nr = slot_head(sp, D.slot)->nrem;
          if (lane < nr) {
            const Removed r = slot_removed(sp, D.slot)[lane];
            rs->rtok[lane] = r.tok;
            rs->rfz[lane] = r.fz;
            value_at(r.tok, rs->rpit[lane], rs->rq[lane]);
          }
          if (lane == 0) rs->rn = nr;
        }
        if (warp == 1 && lane == 0) {
          // the pieces' partial sums and race keys, read while warp 0 lists the children
          const PiecePart* parts = slot_parts(sp, D.slot);
          float DJ = 0.f, K = -INFINITY, QS = 0.f;
          int kstar = INT_MAX;
          uint32_t st2 = D.status;
          for (int k = 0; k < sp.npieces; ++k) {  // a fixed order
            DJ += parts[k].z;
            QS += parts[k].qs;
            argmax_merge(K, kstar, parts[k].key, parts[k].blk);
          }
          rs->D = DJ;
          rs->c = QS;  // (consumer scratch: the mass of q, first pass of distinct siblings)
          rs->term = kstar;
          rs->status = st2;
        }
        csync();
        if (tid == 0) {
          SlotHead* sh = slot_head(sp, D.slot);
          const float DJ = rs->D;
          const int kstar = rs->term;
          uint32_t st2 = rs->status;
          bool degen = sh->degen != 0;
          float c = sh->c, Dn = sh->D;
          int acc = -1;
          bool queued = false, ranked = J == m;
          if (kDistinct) {
            // Siblings without replacement.  With the tokens removed so far frozen at their
            // mass fz, the residual after this pass is max(0, pi - c_J q) elsewhere: its mass is
            // the streamed sum corrected at the removed tokens.  A pass without mass keeps the
            // residual it started from.  Then sibling J's token is removed from the proposal
            // (frozen at the current residual) and the next siblings are tested against r with
            // the proposal q / Z without the removed tokens.
            Removed* rem = slot_removed(sp, D.slot);
            int nrem = rs->rn;
            // the proposal's mass: q's own before the first removal (then less the removed q)
            float Z = J == 1 ? rs->c : sh->Z;
            // the values read before the barrier; a token not among them is loaded here
            auto value_of = [&](int t, float& pit, float& qt) {
              for (int i = 0; i < nrem; ++i)
                if (rs->rtok[i] == t) {
                  pit = rs->rpit[i];
                  qt = rs->rq[i];
                  return;
                }
              for (int i = kMaxRemoved; i < kMaxRemoved + 2; ++i)
                if (rs->rtok[i] == t) {
                  pit = rs->rpit[i];
                  qt = rs->rq[i];
                  return;
                }
              value_at(t, pit, qt);
            };
            auto removed_index = [&](int t) {
              for (int i = 0; i < nrem; ++i)
                if (rs->rtok[i] == t) return i;
              return -1;
            };
            float EJ = DJ;
            for (int i = 0; i < nrem; ++i) EJ += rs->rfz[i] - fmaxf(rs->rpit[i] - cJ * rs->rq[i], 0.f);
            if (EJ > 0.f) {
              c = cJ;
              Dn = EJ;
            } else {
              ranked = false;  // the pieces ranked blocks of a residual that is not used
            }
            auto remove = [&](int t) {
              if (t < 0 || t >= V || removed_index(t) >= 0) return;
              if (nrem >= kMaxRemoved) {
                st2 |= DCD_DEVERR_UNSUPPORTED;
                return;
              }
              float pit, qt;
              value_of(t, pit, qt);
              const float fz = fmaxf(pit - c * qt, 0.f);
              rem[nrem].tok = t;
              rem[nrem].fz = fz;
              rs->rtok[nrem] = t;
              rs->rfz[nrem] = fz;
              rs->rpit[nrem] = pit;
              rs->rq[nrem] = qt;
              ++nrem;
              Z -= qt;
            };
            remove(ktok[J - 1]);
            for (int j = J; j < m; ++j) {
              const int t = ktok[j];
              float ratio = 0.f;
              if (t >= 0 && t < V) {
                const int ri = removed_index(t);
                if (ri >= 0) {
                  ratio = rs->rfz[ri] > 0.f ? INFINITY : 0.f;  // its proposal is 0
                } else {
                  float pit, qt;
                  value_of(t, pit, qt);
                  const float rho = fmaxf(pit - c * qt, 0.f);
                  const float qp = Z > 0.f ? qt / Z : 0.f;
                  ratio = qp > 0.f ? (rho / Dn) / qp : (rho > 0.f ? INFINITY : 0.f);
                }
              }
              const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * N + kids[j]);
              if (u01(philox_block(p.seed, p.offset, G, 0u).x) <= ratio) {
                acc = kids[j];
                break;
              }
              if (Z > 0.f) {
                sh->c = c;
                sh->D = Dn;
                sh->Z = Z;
                sh->nrem = nrem;
                sh->status = st2;
                Job nj;
                nj.slot = D.slot;
                nj.J = j + 1;
                nj.g = static_cast<int32_t>(g);
                nj.m = m;
                nj.status = st2;
                nj.M = M;
                nj.S = D.S;
                nj.Mp = Mp;
                nj.c = c + Dn / Z;  // the next residual: max(0, r - q / Z) off the removed tokens
                nj.alpha = alpha;
                nj.beta = beta;
                nj.T = T;
                create_job(sp, nj);
                queued = true;
                break;
              }
              // every token of q is removed: the proposal is 0 and the residual stays
              ranked = false;
              remove(t);
            }
            if (!queued) {
              sh->nrem = nrem;  // the final race reads the removed tokens
              sh->Z = Z;
            }
          } else {
          if (DJ > 0.f) {
            c = cJ;
            Dn = DJ;
          } else {
            degen = true;  // r_{J-1} == q in exact arithmetic: r_J is taken as q from here on
          }
          // test the remaining siblings; after a pass without residual mass no pass is needed
          for (int j = J; j < m; ++j) {
            if (sibling_test<TIn>(p, b, kids[j], ktok[j], zp_row, zq_row, q_row, c1k, ak, masked, Mp, logb, M, invS,
                                  c, Dn, degen)) {
              acc = kids[j];
              break;
            }
            if (!degen) {
              sh->c = c;
              sh->D = Dn;
              sh->degen = 0;
              sh->status = st2;
              Job nj;
              nj.slot = D.slot;
              nj.J = j + 1;
              nj.g = static_cast<int32_t>(g);
              nj.m = m;
              nj.status = st2;
              nj.M = M;
              nj.S = D.S;
              nj.Mp = Mp;
              nj.c = c + Dn;  // c_{J+1} = c_J + D_J
              nj.alpha = alpha;
              nj.beta = beta;
              nj.T = T;
              create_job(sp, nj);
              queued = true;
              break;
            }
          }
          }
          rs->accept = queued ? -2 : acc;
          rs->term = ranked ? kstar : INT_MAX - 1;  // the winning block when this pass ranked r_m
          rs->status = st2;
          rs->c = c;
          rs->D = Dn;
          rs->degen = degen ? 1 : 0;
        }
        csync();
        const int acc = rs->accept;
        if (acc != -2) {
          int term = -1;
          if (acc < 0) {
            // every sibling rejected: terminal draw from r_m, or from q after a pass without mass
            const bool degen = rs->degen != 0;
            const float c = rs->c, Dn = rs->D;
            int kstar = rs->term;
            const Removed* rem = slot_removed(sp, D.slot);
            const int nrem = kDistinct ? slot_head(sp, D.slot)->nrem : 0;
            auto rho_at = [&](int64_t x) -> float {  // the final residual's unnormalised mass
              if (kDistinct) {
                const int ri = find_removed(rem, nrem, static_cast<int>(x));
                if (ri >= 0) return rem[ri].fz;
              }
              const float z = ld1(zp_row, x);
              const bool in = !masked || (z - Mp >= logb);
              const float pit = in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, x)) - M) * invS : 0.f;
              return fmaxf(pit - c * q_row[x], 0.f);
            };
            if (kDistinct && kstar == INT_MAX - 1) {
              // block masses of the final residual, computed by this CTA alone (rare: the last
              // pass found no mass, or q was used up)
              float bk2 = -INFINITY;
              int bb2 = INT_MAX;
              for (int kb = warp; kb < sp.nblk; kb += kRowWarps) {
                float part = 0.f;
                for (int64_t x = static_cast<int64_t>(kb) * kRaceBlock + lane; x < V && x < (kb + 1) * kRaceBlock;
                     x += 32)
                  part += rho_at(x);
                const float mass = warp_sum(part);
                if (lane == 0 && mass > 0.f) {
                  const float key = block_key(p, g, kb, lg2(mass));
                  if (key > bk2) {
                    bk2 = key;
                    bb2 = kb;
                  }
                }
              }
              block_argmax(bk2, bb2, redf, redi, csync);
              kstar = bb2;
            } else if (degen) {
              // block masses of q, computed by this CTA alone (rare: a residual without mass)
              float bk2 = -INFINITY;
              int bb2 = INT_MAX;
              for (int kb = warp; kb < sp.nblk; kb += kRowWarps) {
                float part = 0.f;
                for (int64_t x = static_cast<int64_t>(kb) * kRaceBlock + lane; x < V && x < (kb + 1) * kRaceBlock;
                     x += 32)
                  part += q_row[x];
                const float mass = warp_sum(part);
                if (lane == 0 && mass > 0.f) {
                  const float key = block_key(p, g, kb, lg2(mass));
                  if (key > bk2) {
                    bk2 = key;
                    bb2 = kb;
                  }
                }
              }
              block_argmax(bk2, bb2, redf, redi, csync);
              kstar = bb2;
            }
            term = token_race(
                p, g, kstar,
                [&](int64_t x) -> float {
                  if (degen && !kDistinct) return q_row[x];
                  return rho_at(x) / Dn;
                },
                redf, redi);
          }
          if (tid == 0) {
            RowRecord r;
            r.acc_child = acc;
            r.term_token = acc < 0 ? term : -1;
            r.status = rs->status;
            r.reserved = 0;
            p.rec[g] = r;
            atomicAdd(&sp.hdr->rows_done, 1u);  // only counts: records are read after the kernel
          }
        }
      }
      csync();  // consumer state in shared memory is rewritten by the next work
      if (tid == 0) mbar_arrive(&dempty[d]);
      continue;
    }

    // ================= a row, or a part of one
    const bool is_part = D.kind == kWorkPart;
    const bool sampled = T > 0.f && p.q != nullptr;
    const bool leaf_race = sampled && D.m == 0;  // a sampled leaf draws its terminal token here
    const float* q_row = sampled ? p.q + g * p.ldq : nullptr;
    const int L0 = is_part ? D.piece * sp.spp : 0;  // the stats pass's stages [L0, L0 + nL)
    const int nL = is_part ? (nch_a - L0 < sp.spp ? nch_a - L0 : sp.spp) : nch_a;

    // a whole row: warp 1 lists the children of node n, checks the row and loads the values at
    // the children's tokens while the stats pass streams; they are consumed after it
    float pzp = 0.f, pzq = 0.f, pq = 0.f;
    auto check_row = [&](int count) {  // lane 0 of the listing warp
      uint32_t st = 0u;
      const int pp = p.parents[static_cast<int64_t>(b) * N + n];
      if (n == 0 ? pp != -1 : (pp < 0 || pp >= n)) st |= DCD_DEVERR_BAD_PARENT;
      if (n > 0) {
        const int t = p.tokens[static_cast<int64_t>(b) * N + n];
        if (t < 0 || t >= V) st |= DCD_DEVERR_BAD_TOKEN;
      }
      if (!(alpha >= 0.f && alpha <= 3.0e38f) || !(beta >= 0.f && beta <= 1.f) || !(T >= 0.f && T <= 3.0e38f))
        st |= DCD_DEVERR_BAD_PARAM;
      rs->m = count;
      rs->status = st;
    };
    if (!is_part && warp == 1) {
      const int count = list_children(p, b, n, kids, ktok);
      if (lane < count) {
        const int t = ktok[lane];
        if (t >= 0 && t < V) {
          pzp = ld1(zp_row, t);
          pzq = ld1(zq_row, t);
          if (sampled) pq = q_row[t];
        }
      }
      if (lane == 0) check_row(count);
    }

    // ---- pass A (beta > 0, whole rows): the expert max, for P_beta = {x : z_p(x) - max z_p >=
    // log beta}
    float Mp = 0.f;
    if (masked) {
      float lm = -INFINITY;
      for (int L = 0; L < nch_a; ++L, ++seq) {
        const Stage<TIn> st = stage_at<TIn>(ring, static_cast<int>(seq % static_cast<uint32_t>(sp.nst)), sp.tok_a);
        const int64_t x0 = static_cast<int64_t>(L) * sp.tok_a;
        const int clen = static_cast<int>((V - x0) < sp.tok_a ? (V - x0) : sp.tok_a);
        wait_full(seq);
        for (int i0 = tid * 8; i0 < clen; i0 += kRowThreads * 8) {
          float zp[8];
          ld8(st.zp + i0, zp);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            if (i0 + e < clen) lm = fmaxf(lm, zp[e]);
        }
        warp_release(&empty[seq % static_cast<uint32_t>(sp.nst)]);
      }
      Mp = block_max(lm, redf, csync);
    }

    // ---- pass B: per lane an online max of u on P_beta, the sum of 2^(u - max) rescaled when
    // the max grows, and the argmax.  A warp takes tok_a / 8 consecutive tokens (a chunk) of each
    // stage; for a sampled leaf it also records the chunk's mass relative to a chunk reference.
    const int tpw = sp.tok_a / kRowWarps, wpb = kRaceBlock / tpw;
    float lmax = -INFINITY, lsum = 0.f;
    int larg = INT_MAX;
    for (int L = L0; L < L0 + nL; ++L, ++seq) {
      const Stage<TIn> st = stage_at<TIn>(ring, static_cast<int>(seq % static_cast<uint32_t>(sp.nst)), sp.tok_a);
      const int64_t x0 = static_cast<int64_t>(L) * sp.tok_a;
      const int clen = static_cast<int>((V - x0) < sp.tok_a ? (V - x0) : sp.tok_a);
      wait_full(seq);
      float bpart = 0.f;  // this lane's share of the chunk's mass, relative to lmax
      for (int sb = warp * tpw; sb < (warp + 1) * tpw && sb < clen; sb += kSub) {  // warp-uniform
        const int i0 = sb + lane * 8;
        float u[8];
        scores8(st.zp, st.zq, i0, sb, clen, masked, c1k, ak, Mp, logb, u);
        const float gm = max8(u);
        if (gm > lmax) {
          const float f = ex2(lmax - gm);  // 0 while lmax is -inf
          lsum *= f;
          bpart *= f;
          lmax = gm;
#pragma unroll
          for (int e = 7; e >= 0; --e)
            if (u[e] == gm) larg = static_cast<int>(x0) + i0 + e;
        }
        if (lmax > -INFINITY) {
          const float2 nm2 = make_float2(-lmax, -lmax);
          float2 acc2 = make_float2(0.f, 0.f);
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float2 dd = __fadd2_rn(make_float2(u[2 * k], u[2 * k + 1]), nm2);
            acc2 = __fadd2_rn(acc2, make_float2(ex2(dd.x), ex2(dd.y)));
          }
          const float a = acc2.x + acc2.y;
          lsum += a;
          bpart += a;
        }
      }
      if (leaf_race) {
        const float ref = warp_max(lmax);
        const float ws = warp_sum(lmax > -INFINITY ? bpart * ex2(lmax - ref) : 0.f);
        if (lane == 0 && x0 + static_cast<int64_t>(warp) * tpw < V) {
          const int ch = static_cast<int>(x0 / tpw) + warp;
          cref[ch] = ref;
          csum[ch] = ws;
        }
      }
      warp_release(&empty[seq % static_cast<uint32_t>(sp.nst)]);
    }
    // statistics of the streamed range (the reduction's barriers also publish the chunk masses
    // and warp 1's child list): M = max u, S = sum 2^(u - M), argmax
    float M = lmax, S = lsum;
    int arg = larg;
    block_stats(M, S, arg, redf, redi, csync);

    // First level of a leaf's terminal race over the blocks of the streamed range: the key of a
    // block is log2 of its mass 2^ref * (rescaled chunk sum) against its uniform; the row max is
    // left out (a common shift), so parts of a row rank their blocks on one scale.
    auto best_block = [&](float& bk, int& bb) {
      const int nch_row = static_cast<int>((V + tpw - 1) / tpw);  // chunks a row has
      const int k_lo = static_cast<int>(static_cast<int64_t>(L0) * sp.tok_a / kRaceBlock);
      int k_hi = static_cast<int>(static_cast<int64_t>(L0 + nL) * sp.tok_a / kRaceBlock);
      if (k_hi > sp.nblk) k_hi = sp.nblk;
      bk = -INFINITY;
      bb = INT_MAX;
      for (int k = k_lo + tid; k < k_hi; k += kRowThreads) {
        float ref = -INFINITY, sum = 0.f;
        for (int i = 0; i < wpb && k * wpb + i < nch_row; ++i) ref = fmaxf(ref, cref[k * wpb + i]);
        if (ref > -INFINITY)
          for (int i = 0; i < wpb && k * wpb + i < nch_row; ++i) {
            const float r = cref[k * wpb + i];
            if (r > -INFINITY) sum += csum[k * wpb + i] * ex2(r - ref);
          }
        if (ref > -INFINITY && sum > 0.f) {
          const float key = block_key(p, g, k, lg2(sum) + ref);
          if (key > bk) {
            bk = key;
            bb = k;
          }
        }
      }
      block_argmax(bk, bb, redf, redi, csync);
    };

    uint32_t status;
    int m, kstar = INT_MAX;
    if (is_part) {
      // ---- a part: publish its statistics; the CTA that finishes a row's last part combines
      // them and finishes the row
      float bk = -INFINITY;
      int bb = INT_MAX;
      if (leaf_race) best_block(bk, bb);
      if (tid == 0) {
        RowPart rp;
        rp.M = M;
        rp.S = S;
        rp.arg = arg;
        rp.key = bk;
        rp.blk = bb;
        rp.timed_out = timed_out ? 1 : 0;
        rp.pad[0] = rp.pad[1] = 0;
        p.parts[g * kMaxParts + D.piece] = rp;
        const uint32_t t = atomic_add_acq_rel(&p.pdone[g], 1u);
        rs->last = t + 1u == static_cast<uint32_t>(sp.parts) ? 1 : 0;
      }
      csync();
      if (!rs->last) {
        if (tid == 0) mbar_arrive(&dempty[d]);
        continue;  // no consumer state of this part is read again
      }
      if (tid == 0) {
        float cM = -INFINITY, cS = 0.f, K = -INFINITY;
        int carg = INT_MAX, kb = INT_MAX, tmo = 0;
        for (int k = 0; k < sp.parts; ++k) {  // a fixed order: the result does not depend on timing
          const RowPart rp = p.parts[g * kMaxParts + k];
          const float nM = fmaxf(cM, rp.M);
          cS = (cM > -INFINITY ? cS * ex2(cM - nM) : 0.f) + (rp.M > -INFINITY ? rp.S * ex2(rp.M - nM) : 0.f);
          if (rp.M > cM || (rp.M == cM && rp.arg < carg)) carg = rp.arg;
          cM = nM;
          argmax_merge(K, kb, rp.key, rp.blk);
          tmo |= rp.timed_out;
        }
        rs->c = cM;  // (consumer scratch: the combined statistics)
        rs->D = cS;
        rs->accept = carg;
        rs->term = kb;
        rs->degen = tmo;
      }
      if (warp == 1) {
        const int count = list_children(p, b, n, kids, ktok);
        if (lane == 0) check_row(count);
      }
      csync();
      M = rs->c;
      S = rs->D;
      arg = rs->accept;
      kstar = rs->term;
      m = rs->m;
      status = rs->status | (rs->degen ? DCD_DEVERR_TIMEOUT : 0u);
      for (int k = tid; k < m; k += kRowThreads) {
        const int t = ktok[k];
        const bool ok = t >= 0 && t < V;
        czp[k] = ok ? ld1(zp_row, t) : 0.f;
        czq[k] = ok ? ld1(zq_row, t) : 0.f;
        cq[k] = (ok && sampled) ? q_row[t] : 0.f;
      }
      csync();
    } else {
      m = rs->m;
      if (warp == 1 && lane < m) {
        czp[lane] = pzp;
        czq[lane] = pzq;
        cq[lane] = pq;
      }
      for (int k = 32 + tid; k < m; k += kRowThreads) {  // nodes with more children than a warp has lanes
        const int t = ktok[k];
        const bool ok = t >= 0 && t < V;
        czp[k] = ok ? ld1(zp_row, t) : 0.f;
        czq[k] = ok ? ld1(zq_row, t) : 0.f;
        cq[k] = (ok && sampled) ? q_row[t] : 0.f;
      }
      status = rs->status | (timed_out ? DCD_DEVERR_TIMEOUT : 0u);
      float bk = -INFINITY;
      if (leaf_race) best_block(bk, kstar);  // its barriers also publish czp / czq / cq
      else csync();
    }
    if (!(M > -INFINITY && M < INFINITY) || !(S > 0.f && S < INFINITY)) status |= DCD_DEVERR_NONFINITE;
    if (sampled && kDistinct && m > kMaxRemoved) status |= DCD_DEVERR_UNSUPPORTED;
    // log sum exp(s' / T) over P_beta = M ln 2 + ln S
    const float logS = logf(S);
    const float invS = 1.f / S;

    // ---- outputs of the Eq. 1 target
    if (tid == 0) {
      if (p.cd_argmax) p.cd_argmax[g] = arg;
      if (p.cd_lse) p.cd_lse[g] = M * kLn2 + logS;
      if (n == 0 && p.cd_logprob) p.cd_logprob[g] = 0.f;
    }
    if (p.cd_logprob) {
      for (int k = tid; k < m; k += kRowThreads) {
        const bool in = !masked || (czp[k] - Mp >= logb);
        p.cd_logprob[static_cast<int64_t>(b) * N + kids[k]] =
            in ? (fmaf(c1k, czp[k], -ak * czq[k]) - M) * kLn2 - logS : -INFINITY;
      }
    }

    int acc = -1, term = -1;
    bool handed_over = false;
    if (!sampled) {
      // ---- greedy rule: the first child whose token is the argmax
      for (int k = 0; k < m; ++k)
        if (ktok[k] == arg) {
          acc = kids[k];
          break;
        }
      if (acc < 0) term = arg;
    } else if (m > 0) {
      // ---- sampled rule, first sibling: accept child 0 iff u <= pi_CD,T(t) / q(t); a rejection
      // queues the first residual pass (the row's record is written when its chain ends)
      if (tid == 0) {
        const bool in = !masked || (czp[0] - Mp >= logb);
        const float rt = in ? ex2(fmaf(c1k, czp[0], -ak * czq[0]) - M) * invS : 0.f;
        const float qt = cq[0];
        const float ratio = qt > 0.f ? rt / qt : (rt > 0.f ? INFINITY : 0.f);
        const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * N + kids[0]);
        const float u = u01(philox_block(p.seed, p.offset, G, 0u).x);
        int accept = u <= ratio ? 1 : 0;
        if (!accept && !(status & (DCD_DEVERR_BAD_PARENT | DCD_DEVERR_BAD_TOKEN | DCD_DEVERR_BAD_PARAM |
                                   DCD_DEVERR_NONFINITE | DCD_DEVERR_UNSUPPORTED))) {
          const int s = static_cast<int>(atomicAdd(&sp.hdr->nslots, 1u));
          SlotHead* sh = slot_head(sp, s);
          sh->g = static_cast<int32_t>(g);
          sh->m = m;
          sh->M = M;
          sh->S = S;
          sh->Mp = Mp;
          sh->c = 0.f;  // r_0 = pi: c_0 = 0, D_0 = 1
          sh->D = 1.f;
          sh->degen = 0;
          sh->status = status;
          sh->Z = 1.f;  // distinct siblings: nothing removed yet
          sh->nrem = 0;
          Job nj;
          nj.slot = s;
          nj.J = 1;
          nj.g = static_cast<int32_t>(g);
          nj.m = m;
          nj.status = status;
          nj.M = M;
          nj.S = S;
          nj.Mp = Mp;
          nj.c = 1.f;  // c_1 = c_0 + D_0
          nj.alpha = alpha;
          nj.beta = beta;
          nj.T = T;
          create_job(sp, nj);
          accept = -1;
        }
        rs->accept = accept;
      }
      csync();
      if (rs->accept == 1) acc = kids[0];
      if (rs->accept == -1) handed_over = true;
    } else {
      // ---- sampled leaf: the terminal token is drawn from pi_CD,T by the two-level race: the
      // block kstar won by its mass, then a token of that block
      term = token_race(
          p, g, kstar,
          [&](int64_t x) -> float {
            const float z = ld1(zp_row, x);
            const bool in = !masked || (z - Mp >= logb);
            return in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, x)) - M) : 0.f;
          },
          redf, redi);
    }
    if (tid == 0 && !handed_over) {
      RowRecord r;
      r.acc_child = acc;
      r.term_token = acc < 0 ? term : -1;
      r.status = status;
      r.reserved = 0;
      p.rec[g] = r;
      atomicAdd(&sp.hdr->rows_done, 1u);  // only counts: records and outputs are read after the kernel
    }
    csync();  // consumer state in shared memory is rewritten by the next work
    if (tid == 0) mbar_arrive(&dempty[d]);
  }
}

// ------------------------------------------------------------------------------------------
// One warp per sequence: the N records are read at once into shared memory, then lane 0 follows
// the accepted children from the root and the warp writes the path.  Launched as a programmatic
// dependent of the row kernel: it waits for that grid's completion (and its memory) first.
constexpr int kWalkWarps = 4;

__global__ void __launch_bounds__(kWalkWarps * 32) tree_walk_kernel(int32_t B, int32_t N,
                                                                    const RowRecord* __restrict__ rec, uint32_t* err,
                                                                    int32_t* accept_len, int32_t* accept_path,
                                                                    int32_t* bonus) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  extern __shared__ int walk_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.x * kWalkWarps + warp;
  if (b >= B) return;
  int* wacc = walk_smem + warp * 3 * N;
  int* wterm = wacc + N;
  int* wpath = wterm + N;
  const RowRecord* r = rec + static_cast<int64_t>(b) * N;
  uint32_t st = 0u;
  for (int i = lane; i < N; i += 32) {
    const RowRecord v = r[i];
    wacc[i] = v.acc_child;
    wterm[i] = v.term_token;
    st |= v.status;
  }
  st = __reduce_or_sync(~0u, st);
  // A bounded wait that gave up anywhere in the call may have left rows without a fresh record
  // (a record of an earlier call in the same workspace would look valid), so a timeout recorded
  // in the call's error word fails every sequence.
  st |= ld_volatile(err) & DCD_DEVERR_TIMEOUT;
  __syncwarp();
  int32_t* path = accept_path + static_cast<int64_t>(b) * N;
  if (st) {
    if (lane == 0) {
      atomicOr(err, st);
      accept_len[b] = 0;
      bonus[b] = -1;
    }
    for (int i = lane; i < N; i += 32) path[i] = i == 0 ? 0 : -1;
    return;
  }
  int len = 0;
  if (lane == 0) {
    int cur = 0;
    wpath[0] = 0;
    while (len < N - 1) {
      const int a = wacc[cur];
      if (a <= cur || a >= N) break;
      cur = a;
      wpath[++len] = cur;
    }
    accept_len[b] = len;
    bonus[b] = wterm[cur];
  }
  len = __shfl_sync(~0u, len, 0);
  __syncwarp();
  for (int i = lane; i < N; i += 32) path[i] = i <= len ? wpath[i] : -1;
}

// ------------------------------------------------------------------------------------------
// Terminal residual (test output): one block per sequence, plain passes over global memory,
// the output row doubling as the working buffer.
template <typename TIn>
__global__ void __launch_bounds__(kThreads) terminal_residual_kernel(const ScoreArgs p, const int32_t* accept_len,
                                                                     const int32_t* accept_path,
                                                                     const int32_t* bonus, float* residual) {
  __shared__ float redf[32];
  const int b = blockIdx.x;
  const int64_t V = p.V;
  float* out = residual + static_cast<int64_t>(b) * V;
  const float T = p.temp ? p.temp[b] : 0.f;
  const int bon = bonus[b];
  if (!(T > 0.f) || bon < 0 || p.q == nullptr) {
    for (int64_t x = threadIdx.x; x < V; x += kThreads) out[x] = (x == bon) ? 1.f : 0.f;
    return;
  }
  const int N = p.N;
  const int cur = accept_path[static_cast<int64_t>(b) * N + accept_len[b]];
  const int64_t g = static_cast<int64_t>(b) * N + cur;
  const TIn* zp = static_cast<const TIn*>(p.zp) + g * p.ld;
  const TIn* zq = static_cast<const TIn*>(p.zq) + g * p.ld;
  const float* q = p.q + g * p.ldq;
  const float alpha = p.alpha[b];
  const float beta = p.beta ? p.beta[b] : 0.f;
  const bool masked = beta > 0.f;
  const float logb = masked ? logf(beta) : -INFINITY;
  const float c1 = 1.f + alpha, invT = 1.f / T;
  float Mp = 0.f;
  if (masked) {
    float v = -INFINITY;
    for (int64_t x = threadIdx.x; x < V; x += kThreads) v = fmaxf(v, ld1(zp, x));
    Mp = block_max(v, redf);
  }
  float M = -INFINITY;
  for (int64_t x = threadIdx.x; x < V; x += kThreads) {
    const float z = ld1(zp, x);
    if (!masked || z - Mp >= logb) M = fmaxf(M, fmaf(c1, z, -alpha * ld1(zq, x)));
  }
  M = block_max(M, redf);
  float s = 0.f;
  for (int64_t x = threadIdx.x; x < V; x += kThreads) {
    const float z = ld1(zp, x);
    const float e = (!masked || z - Mp >= logb) ? expf((fmaf(c1, z, -alpha * ld1(zq, x)) - M) * invT) : 0.f;
    out[x] = e;
    s += e;
  }
  const float inv = 1.f / block_sum(s, redf);
  for (int64_t x = threadIdx.x; x < V; x += kThreads) out[x] *= inv;
  __syncthreads();
  // every child of the terminal node was rejected, in ascending node id
  __shared__ int removed[kMaxRemoved];
  __shared__ float zrem;
  int nrem = 0;
  float qtot = 0.f;  // the mass of q (the drafter's q need not sum to 1)
  if (p.distinct) {
    for (int64_t x = threadIdx.x; x < V; x += kThreads) qtot += q[x];
    qtot = block_sum(qtot, redf);
  }
  if (threadIdx.x == 0) zrem = qtot;
  __syncthreads();
  for (int c = cur + 1; c < N; ++c) {
    if (p.parents[static_cast<int64_t>(b) * N + c] != cur) continue;
    // the proposal of this sibling: q, or (distinct siblings, once a token is removed) q without
    // the removed tokens over their remaining mass Z
    const float Z = zrem;
    auto prop = [&](int64_t x) -> float {
      if (!p.distinct || nrem == 0) return q[x];
      for (int i = 0; i < nrem; ++i)
        if (removed[i] == x) return 0.f;
      return Z > 0.f ? q[x] / Z : 0.f;
    };
    float z = 0.f;
    for (int64_t x = threadIdx.x; x < V; x += kThreads) z += fmaxf(out[x] - prop(x), 0.f);
    z = block_sum(z, redf);
    if (z > 0.f) {
      const float iz = 1.f / z;
      for (int64_t x = threadIdx.x; x < V; x += kThreads) out[x] = fmaxf(out[x] - prop(x), 0.f) * iz;
    } else if (!p.distinct) {
      for (int64_t x = threadIdx.x; x < V; x += kThreads) out[x] = q[x];
    }  // distinct siblings: a step without mass leaves the residual as it is
    __syncthreads();
    if (p.distinct) {
      const int t = p.tokens[static_cast<int64_t>(b) * N + c];
      bool seen = t < 0 || t >= V;
      for (int i = 0; i < nrem; ++i) seen = seen || removed[i] == t;
      if (!seen && nrem < kMaxRemoved) {
        if (threadIdx.x == 0) {
          removed[nrem] = t;
          zrem = Z - q[t];
        }
        ++nrem;
      }
      __syncthreads();
    }
  }
}

// ------------------------------------------------------------------------------------------
struct DeviceInfo {
  int sms = 0;
  cudaError_t err = cudaSuccess;
};

template <typename TIn>
cudaError_t prepare_kernel(int* sms) {
  static std::once_flag once[64];
  static DeviceInfo info[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::call_once(once[dev], [&] {
    DeviceInfo d;
    d.err = cudaFuncSetAttribute(score_rows_kernel<TIn, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmemMax));
    if (d.err == cudaSuccess)
      d.err = cudaFuncSetAttribute(score_rows_kernel<TIn, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(kSmemMax));
    if (d.err == cudaSuccess) d.err = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
    info[dev] = d;
  });
  *sms = info[dev].sms;
  return info[dev].err;
}

struct Layout {
  int meta_offset, chunk_offset, stage_offset;
  size_t total;
};

// Dynamic shared memory: mbarriers, reduction scratch and descriptors; consumer state and the
// child lists; chunk masses; the ring.
Layout layout_for(int N, int nchunk, int nst) {
  Layout l;
  const size_t fixed = 8 * (2 * kMaxStages + 2 * kDesc) + 64 * 4 + sizeof(WorkDesc) * kDesc;
  l.meta_offset = static_cast<int>((fixed + 15) & ~static_cast<size_t>(15));
  const size_t meta_end = static_cast<size_t>(l.meta_offset) + sizeof(RowShared) + static_cast<size_t>(N) * 4 * 5;
  l.chunk_offset = static_cast<int>((meta_end + 15) & ~static_cast<size_t>(15));
  const size_t chunk_end = static_cast<size_t>(l.chunk_offset) + static_cast<size_t>(nchunk) * 4 * 2;
  l.stage_offset = static_cast<int>((chunk_end + 127) & ~static_cast<size_t>(127));
  l.total = static_cast<size_t>(l.stage_offset) + static_cast<size_t>(nst) * kStageBytes;
  return l;
}

// Tokens per stage: every consumer warp takes tpw consecutive tokens of a stage, with tpw a
// multiple of the 256-token group that divides a race block (256, 512 or 1024 tokens), so whole
// warp chunks make a race block.  z_p and z_q fill a stage in row passes; z_p, z_q and q share it
// in residual pieces.
int split_tokens(int cap) {
  for (int tpw = kRaceBlock; tpw >= kSub; tpw /= 2)
    if (kRowWarps * tpw <= cap) return kRowWarps * tpw;
  return 0;
}
int tokens_a(int es) { return split_tokens(kStageBytes / (2 * es)); }
int tokens_r(int es) { return split_tokens(kStageBytes / (2 * es + 4)); }

// A warp takes tok / kRowWarps tokens of a stage in groups of 256, whole chunks make a race
// block, and a piece's race blocks fit the consumer threads.
bool stage_split_ok(int tok) {
  const int tpw = tok / kRowWarps;
  return tok > 0 && tok % (kRowWarps * kSub) == 0 && tpw <= kRaceBlock && kRaceBlock % tpw == 0 &&
         kPieceStages * (tok / kRaceBlock) <= kRowThreads;
}

int chunks_per_row(int64_t V, int es) {
  const int tpw = tokens_a(es) / kRowWarps;
  const int64_t rows_chunks = (V + tpw - 1) / tpw;
  const int piece_chunks = kPieceStages * kRowWarps;  // csum slots a residual piece uses
  return static_cast<int>(rows_chunks > piece_chunks ? rows_chunks : piece_chunks);
}

}  // namespace

int piece_stages_for(int64_t rows) { return rows <= kSmallPieceRows ? kSmallPieceStages : kPieceStages; }

int residual_pieces(int64_t V, int dtype, int64_t rows) {
  const int es = dtype == DCD_BF16 ? 2 : 4;
  const int64_t tok = static_cast<int64_t>(tokens_r(es)) * piece_stages_for(rows);
  return static_cast<int>((V + tok - 1) / tok);
}

size_t slot_bytes(int64_t V, int dtype, int64_t rows) {
  return sizeof(SlotHead) + static_cast<size_t>(residual_pieces(V, dtype, rows)) * sizeof(PiecePart) +
         kMaxRemoved * sizeof(Removed);
}

RowGeometry row_geometry(const ScoreArgs& a) {
  RowGeometry geo{};
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  // the default ring depth, or fewer stages (at least two) where a large tree or vocabulary
  // leaves no room for it
  int nst = a.force_stages > 0 ? a.force_stages : kRingStages;
  Layout l = layout_for(a.N, chunks_per_row(a.V, es), nst);
  while (a.force_stages <= 0 && nst > 2 && l.total > kSmemMax) l = layout_for(a.N, chunks_per_row(a.V, es), --nst);
  const int per_sm = static_cast<int>(kSmemPerSm / (l.total + 1024));
  geo.stages = nst;
  geo.stage_tokens = tokens_a(es);
  geo.smem = l.total;
  geo.ctas_per_sm = per_sm > 4 ? 4 : per_sm;
  auto al16 = [](const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
  geo.bulk = !a.force_plain && al16(a.zp) && al16(a.zq) && (a.ld * es) % 16 == 0 &&
             (!a.q || (al16(a.q) && (a.ldq * 4) % 16 == 0));
  return geo;
}

#ifndef DCD_USE_CLUSTER
#define DCD_USE_CLUSTER 1
#endif

cudaError_t launch_score_rows(const ScoreArgs& a, cudaStream_t stream) {
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  if (R == 0) return cudaSuccess;
  if (DCD_USE_CLUSTER && cluster_rows_ok(a)) return launch_cluster_rows(a, stream);
  const RowGeometry geo = row_geometry(a);
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  if (geo.smem > kSmemMax || geo.stages < 1 || geo.stages > kMaxStages || geo.ctas_per_sm < 1 ||
      !stage_split_ok(tokens_a(es)) || !stage_split_ok(tokens_r(es)))
    return cudaErrorInvalidConfiguration;
  int sms = 0;
  cudaError_t e = a.dtype == DCD_BF16 ? prepare_kernel<__nv_bfloat16>(&sms) : prepare_kernel<float>(&sms);
  if (e != cudaSuccess) return e;
  SParams sp;
  sp.a = a;
  sp.nst = geo.stages;
  sp.tok_a = tokens_a(es);
  sp.tok_r = tokens_r(es);
  sp.npieces = residual_pieces(a.V, a.dtype, R);
  sp.piece_stages = piece_stages_for(R);
  sp.bulk = geo.bulk;
  sp.nblk = static_cast<int>((a.V + kRaceBlock - 1) / kRaceBlock);
  sp.nchunk = chunks_per_row(a.V, es);
  const Layout l = layout_for(a.N, sp.nchunk, sp.nst);
  sp.meta_offset = l.meta_offset;
  sp.chunk_offset = l.chunk_offset;
  sp.stage_offset = l.stage_offset;
  sp.slot_bytes = static_cast<int32_t>(slot_bytes(a.V, a.dtype, R));
  sp.poll_cycles = a.poll_cycles > 0 ? a.poll_cycles : kWaitCycles;
  sp.hdr = a.hdr;
  sp.jobs = a.jobs;
  sp.slots = a.slots;
  // the header counters and the part counters start every call at zero
  e = cudaMemsetAsync(a.hdr, 0, kWorkspaceHeader + part_counter_bytes(static_cast<size_t>(R)), stream);
  if (e != cudaSuccess) return e;
  // a CTA may wait for work queued by another, so all CTAs must be resident at once: the grid is
  // the resident capacity (capped at the row count) and the launch is cooperative
  int per_sm = 0;
  const void* fn = a.dtype == DCD_BF16
                       ? (a.distinct ? reinterpret_cast<const void*>(score_rows_kernel<__nv_bfloat16, true>)
                                     : reinterpret_cast<const void*>(score_rows_kernel<__nv_bfloat16, false>))
                       : (a.distinct ? reinterpret_cast<const void*>(score_rows_kernel<float, true>)
                                     : reinterpret_cast<const void*>(score_rows_kernel<float, false>));
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kCtaThreads, geo.smem);
  if (e != cudaSuccess) return e;
  if (per_sm > geo.ctas_per_sm) per_sm = geo.ctas_per_sm;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  const int64_t resident = static_cast<int64_t>(sms) * per_sm;
  // A small batch (at most kPartsBelow rows per resident CTA) is streamed in parts of spp stages
  // each, so that its rows spread over more CTAs.
  const int nch_a = static_cast<int>((a.V + sp.tok_a - 1) / sp.tok_a);
  const int want = nch_a < kMaxParts ? nch_a : kMaxParts;
  sp.spp = (nch_a + want - 1) / want;
  sp.parts = (nch_a + sp.spp - 1) / sp.spp;
  int64_t tail = (sp.parts > 1 && R <= kPartsBelow * resident) ? R : 0;
  if (sp.parts > 1 && tail == 0) tail = R < kTailRows ? R : kTailRows;
  sp.r_whole = static_cast<int32_t>(R - tail);
  sp.keep_internal = R <= kPartsBelow * resident ? 1 : 0;
  sp.items = static_cast<int32_t>(sp.r_whole + tail * sp.parts);
  int64_t grid = resident;
  if (grid > sp.items) grid = sp.items;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kCtaThreads);
  cfg.dynamicSmemBytes = geo.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (a.dtype == DCD_BF16)
    return a.distinct ? cudaLaunchKernelEx(&cfg, score_rows_kernel<__nv_bfloat16, true>, sp)
                      : cudaLaunchKernelEx(&cfg, score_rows_kernel<__nv_bfloat16, false>, sp);
  return a.distinct ? cudaLaunchKernelEx(&cfg, score_rows_kernel<float, true>, sp)
                    : cudaLaunchKernelEx(&cfg, score_rows_kernel<float, false>, sp);
}

cudaError_t launch_tree_walk(int32_t B, int32_t N, const RowRecord* rec, uint32_t* err, int32_t* accept_len,
                             int32_t* accept_path, int32_t* bonus, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const size_t smem = static_cast<size_t>(kWalkWarps) * 3 * N * sizeof(int);  // <= 48 KB for N <= 1024
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>((B + kWalkWarps - 1) / kWalkWarps));
  cfg.blockDim = dim3(kWalkWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  // launched while the previous kernel in the stream finishes; the kernel waits for it first
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, tree_walk_kernel, B, N, rec, err, accept_len, accept_path, bonus);
}

cudaError_t launch_terminal_residual(const ScoreArgs& a, const int32_t* accept_len, const int32_t* accept_path,
                                     const int32_t* bonus, float* residual, cudaStream_t stream) {
  if (a.B == 0) return cudaSuccess;
  if (a.dtype == DCD_BF16)
    terminal_residual_kernel<__nv_bfloat16><<<a.B, kThreads, 0, stream>>>(a, accept_len, accept_path, bonus, residual);
  else
    terminal_residual_kernel<float><<<a.B, kThreads, 0, stream>>>(a, accept_len, accept_path, bonus, residual);
  return cudaGetLastError();
}

}  // namespace dcd
