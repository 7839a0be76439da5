// dcd_rows.cu -- the streaming kernels of the CD verification step on sm_103a.
//
// score_rows_kernel: a persistent, cooperatively launched grid (a few CTAs per SM) with two
// kinds of work.
//
//  * Rows.  A CTA claims whole tree-node rows g = b * N + n from a work counter, in
//    node-major order (every sequence's node 0, then every node 1, ...), so internal
//    nodes -- the rows that may start residual work -- come first and leaves last.  A
//    row is streamed through a ring of 32 KB shared-memory stages filled by bulk
//    asynchronous copies that complete on one mbarrier per stage; thread 0 refills a
//    stage as soon as the block has consumed it.  The "stats" pass computes the CD score
//    s' = (1 + alpha) z_p - alpha z_q (Eq. 1; the two log-softmax shifts are constant per
//    row and cancel in the normaliser) on the plausibility set P_beta of Sec. 2.1, in the
//    scaled unit u = k2 s' (k2 = log2(e) / T, so pi_CD,T ~ 2^u).  A warp takes a
//    contiguous eighth of each stage; every lane keeps an online max of u, a sum of
//    2^(u - max) rescaled when its max grows, and its argmax, combined over the block at the
//    end of the row.  With beta > 0 a "max" pass over z_p comes first.  Sampled rows also
//    get, from the same exponentials, each 1024-token block's mass of pi_CD for a terminal
//    race.  The greedy rule, the first sibling test of the sampled rule and the leaf race
//    then finish the row.
//
//  * Residual pieces.  After a rejected sibling, Algorithm 1 (generalised to sibling
//    lists) needs the next residual over the whole vocabulary.  With c_0 = 0, D_0 = 1 the
//    j-th residual is r_j = max(0, pi - c_j q) / D_j, where c_j = c_{j-1} + D_{j-1} and
//    D_j = sum_x max(0, pi(x) - c_j q(x)) (induction on j from r_j = normalise(max(0,
//    r_{j-1} - q))), so a pass needs only two scalars from the one before.  A row that
//    needs a pass is handed to a job list; the pass is split into pieces of four ring
//    stages (16384 tokens for bf16 logits) that any CTA claims before taking a new row.
//    Each piece writes its partial sum (and, in the pass after the last sibling, its best
//    race key) to its own slot; the CTA that finishes a pass's last piece (an atomic
//    ticket, no waiting) sums the slots in a fixed order, tests the next sibling, and
//    either queues the next pass or runs the terminal race.  A CTA with no row left polls
//    for pieces until every row's record is written (bounded; all CTAs are co-resident
//    under a cooperative launch), so the passes of late chains still spread over the GPU.
//
//  A node without an accepted child draws its terminal token by a two-level exponential
//  race: a 1024-token block by its mass, then a token of that block (four tokens a thread,
//  re-read directly).
// tree_walk_kernel: one thread per sequence follows the accepted children.
// terminal_residual_kernel: one block per sequence rebuilds the distribution its bonus
//   token was drawn from (test output only).

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <mutex>

#include "dcd.h"
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
constexpr int kPieceStages = 4;                    // ring stages per residual piece
constexpr size_t kSmemMax = 227 * 1024;
constexpr size_t kSmemPerSm = 228 * 1024;
constexpr float kLn2 = 0.69314718055994531f;

enum PassKind { kPassMax = 0, kPassStats = 1 };
enum WorkKind { kWorkNone = 0, kWorkRow = 1, kWorkPiece = 2 };

// ------------------------------------------------------------------------------------------
struct SParams {
  ScoreArgs a;
  int32_t nst;           // ring depth (stages of kStageBytes)
  int32_t tok_a;         // tokens per stage in row passes (z_p, then z_q)
  int32_t tok_r;         // tokens per stage in residual pieces (z_p, z_q, then q)
  int32_t npieces;       // pieces per residual pass
  int32_t bulk;          // 1: bulk asynchronous copies, 0: plain loads
  int32_t nblk;          // race blocks per row, ceil(V / 1024)
  int32_t meta_offset;   // byte offsets into dynamic shared memory
  int32_t blk_offset;
  int32_t stage_offset;
  int32_t slot_bytes;
  WsHeader* hdr;         // counters, zeroed before the launch
  Job* jobs;             // residual passes (zeroed before the launch)
  unsigned char* slots;  // per handed-over row: SlotHead + npieces PieceParts
};

// Row / piece state shared by the block (written by one thread, read after a barrier).
struct RowShared {
  int32_t next;      // the next claimed row item
  int32_t kind;      // WorkKind of the current work
  int32_t item;      // row item or job index
  int32_t piece;     // piece index
  int32_t m;         // children of the row's node
  uint32_t status;   // DCD_DEVERR_* bits
  int32_t accept;    // outcome of a sibling test
  int32_t term;      // winning race block of a completed pass
  int32_t last;      // this CTA finished a pass's last piece
  int32_t degen;     // a pass found no residual mass left
  int32_t slot;      // slot of the handed-over row
  int32_t J;         // residual pass index (rejections so far)
  int32_t g;         // row of the piece
  float M, S, Mp, c, D;
  int32_t pad[2];
  float wref[2][kWarps];  // per-warp shares of race-block masses, double-buffered by stage
  float wsum[2][kWarps];
};

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
__device__ __forceinline__ int32_t ld_volatile(const int32_t* p) {
  return *reinterpret_cast<const volatile int32_t*>(p);
}

__device__ __forceinline__ SlotHead* slot_head(const SParams& sp, int s) {
  return reinterpret_cast<SlotHead*>(sp.slots + static_cast<size_t>(s) * sp.slot_bytes);
}

__device__ __forceinline__ PiecePart* slot_parts(const SParams& sp, int s) {
  return reinterpret_cast<PiecePart*>(sp.slots + static_cast<size_t>(s) * sp.slot_bytes + sizeof(SlotHead));
}

// Publishes residual pass J of slot s (thread 0 of the creating CTA).
__device__ __forceinline__ void create_job(const SParams& sp, int s, int J) {
  const uint32_t k = atomicAdd(&sp.hdr->job_alloc, 1u);
  Job* job = &sp.jobs[k];
  job->slot = s;
  job->next_piece = 0u;
  job->done = 0u;
  __threadfence();
  *reinterpret_cast<volatile int32_t*>(&job->J) = J;
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
// log2 r(x) - log2(-log2 u_x), four tokens a thread (one Philox call, counter 1 + x / 4).
// `mass(x)` returns r(x) up to a common factor.  Every thread of the block calls it and gets
// the token (INT_MAX when no block had mass).
template <typename MassFn>
__device__ int token_race(const ScoreArgs& p, int64_t g, int kstar, MassFn mass, float* redf, int* redi) {
  float tk = -INFINITY;
  int tx = INT_MAX;
  if (kstar != INT_MAX) {
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
  block_argmax(tk, tx, redf, redi);
  return tx;
}

// First level of the race for one block: its key from log2 of its mass.
__device__ __forceinline__ float block_key(const ScoreArgs& p, int64_t g, int k, float log2_mass) {
  const uint4 w = philox_block(p.seed, p.offset, static_cast<uint32_t>(g), 0x80000000u | (static_cast<uint32_t>(k) >> 2));
  return race_key(log2_mass, word_of(w, k & 3));
}

// ------------------------------------------------------------------------------------------
template <typename TIn>
__global__ void __launch_bounds__(kThreads, 3) score_rows_kernel(const __grid_constant__ SParams sp) {
  const ScoreArgs& p = sp.a;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int N = p.N;
  const int64_t V = p.V;
  const int R = p.B * N;
  const int nch_a = static_cast<int>((V + sp.tok_a - 1) / sp.tok_a);  // chunks of a max / stats pass

  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);             // [kMaxStages]
  float* redf = reinterpret_cast<float*>(smem + 8 * kMaxStages);  // [32]
  int* redi = reinterpret_cast<int*>(redf + 32);                  // [32]
  RowShared* rs = reinterpret_cast<RowShared*>(smem + sp.meta_offset);
  int* kids = reinterpret_cast<int*>(rs + 1);                     // [N] children, ascending id
  int* ktok = kids + N;                                           // [N] their tokens
  float* czp = reinterpret_cast<float*>(ktok + N);                // [N] z_p at those tokens
  float* czq = czp + N;                                           // [N] z_q at those tokens
  float* cq = czq + N;                                            // [N] q at those tokens
  float* bmax = reinterpret_cast<float*>(smem + sp.blk_offset);   // [nblk] block reference of u
  float* bsum = bmax + sp.nblk;                                   // [nblk] block sum of 2^(u - ref)
  unsigned char* ring = smem + sp.stage_offset;

  if (tid == 0) {
    for (int s = 0; s < sp.nst; ++s) mbar_init(&full[s], 1);
    fence_mbar_init();
    rs->next = static_cast<int32_t>(atomicAdd(&sp.hdr->work, 1u));
  }
  __syncthreads();
  const uint64_t pol_last = l2_policy_evict_last();
  const uint64_t pol_first = l2_policy_evict_first();
  uint32_t seq = 0;  // ring items consumed by this CTA so far (identical in every thread)

  // Waits for ring item `sq`, then fills a ragged or unaligned remainder with plain loads.
  auto wait_stage = [&](uint32_t sq, const Stage<TIn>& st, const TIn* zp_row, const TIn* zq_row,
                        const float* q_row, int64_t x0, int clen, bool with_zq, bool with_q, bool& timed_out) {
    const int s = static_cast<int>(sq % static_cast<uint32_t>(sp.nst));
    const uint32_t parity = (sq / static_cast<uint32_t>(sp.nst)) & 1u;
    if (!mbar_wait_bounded(&full[s], parity)) timed_out = true;
    const int zfirst =
        sp.bulk ? ((clen * static_cast<int>(sizeof(TIn))) & ~15) / static_cast<int>(sizeof(TIn)) : 0;
    const int qfirst = sp.bulk ? ((clen * 4) & ~15) / 4 : 0;
    if (zfirst < clen || (with_q && qfirst < clen)) {
      for (int i = zfirst + tid; i < clen; i += kThreads) {
        st.zp[i] = zp_row[x0 + i];
        if (with_zq) st.zq[i] = zq_row[x0 + i];
      }
      if (with_q)
        for (int i = qfirst + tid; i < clen; i += kThreads) st.q[i] = q_row[x0 + i];
      __syncthreads();
    }
  };

  for (;;) {
    // ---- next work: a residual piece if one can be claimed, else the next row.  With no row
    // left, a CTA stays (all CTAs are co-resident: cooperative launch) until every row's record
    // is written, to take pieces of passes other CTAs queue; the wait is bounded.
    if (tid == 0) {
      int kind = kWorkNone, job = -1, piece = 0;
      const long long t0 = clock64();
      for (;;) {
        const uint32_t alloc = ld_volatile(&sp.hdr->job_alloc);
        for (uint32_t k = ld_volatile(&sp.hdr->job_head); k < alloc; ++k) {
          if (ld_volatile(&sp.jobs[k].J) == 0) break;  // not yet published
          const uint32_t pc = atomicAdd(&sp.jobs[k].next_piece, 1u);
          if (pc < static_cast<uint32_t>(sp.npieces)) {
            job = static_cast<int>(k);
            piece = static_cast<int>(pc);
            break;
          }
          atomicMax(&sp.hdr->job_head, k + 1u);
        }
        if (job >= 0) {
          kind = kWorkPiece;
          rs->item = job;
          rs->piece = piece;
          break;
        }
        if (rs->next < R) {
          kind = kWorkRow;
          rs->item = rs->next;
          rs->next = static_cast<int32_t>(atomicAdd(&sp.hdr->work, 1u));
          break;
        }
        if (ld_volatile(&sp.hdr->rows_done) >= static_cast<uint32_t>(R)) break;
        if (clock64() - t0 > kWaitCycles) {
          atomicOr(&sp.hdr->err, DCD_DEVERR_TIMEOUT);
          break;
        }
        __nanosleep(256);
      }
      rs->kind = kind;
    }
    __syncthreads();
    const int kind = rs->kind;
    if (kind == kWorkNone) break;

    if (kind == kWorkPiece) {
      // ================= one piece of residual pass J of a handed-over row
      if (tid == 0) {
        __threadfence();  // the job and its slot were written before J was published
        const Job* job = &sp.jobs[rs->item];
        const int s = ld_volatile(&job->slot);
        const SlotHead* sh = slot_head(sp, s);
        rs->slot = s;
        rs->J = ld_volatile(&job->J);
        rs->g = sh->g;
        rs->m = sh->m;
        rs->M = sh->M;
        rs->S = sh->S;
        rs->Mp = sh->Mp;
        rs->c = sh->c + sh->D;  // c_J = c_{J-1} + D_{J-1}
        rs->status = sh->status;
      }
      __syncthreads();
      const int64_t g = rs->g;
      const int J = rs->J, m = rs->m, piece = rs->piece;
      const int b = static_cast<int>(g / N);
      const float alpha = p.alpha[b];
      const float beta = p.beta ? p.beta[b] : 0.f;
      const float T = p.temp[b];
      const bool masked = beta > 0.f;
      const float k2 = kLog2e / T;
      const float c1k = (1.f + alpha) * k2, ak = alpha * k2;  // u = k2 s' = c1k z_p - ak z_q
      const float logb = masked ? logf(beta) : -INFINITY;
      const float M = rs->M, invS = 1.f / rs->S, Mp = rs->Mp, cJ = rs->c;
      const bool race = J == m;  // the pass after the last sibling also ranks race blocks
      const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
      const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;
      const float* q_row = p.q + g * p.ldq;
      // the piece's stages, streamed through the ring like a row; a warp takes tok_r / 8
      // consecutive tokens of each stage, so `wpb` warps cover one race block
      const int tpw = sp.tok_r / kWarps, wpb = kRaceBlock / tpw;
      const int64_t piece_lo = static_cast<int64_t>(piece) * kPieceStages * sp.tok_r;
      const int64_t rem = (V - piece_lo + sp.tok_r - 1) / sp.tok_r;
      const int nst_piece = static_cast<int>(rem < kPieceStages ? rem : kPieceStages);
      const uint32_t seq0 = seq;
      auto issue_piece = [&](int L) {  // thread 0 only
        const uint32_t sq = seq0 + static_cast<uint32_t>(L);
        const int s = static_cast<int>(sq % static_cast<uint32_t>(sp.nst));
        const Stage<TIn> st = stage_at<TIn>(ring, s, sp.tok_r);
        const int64_t x0 = piece_lo + static_cast<int64_t>(L) * sp.tok_r;
        const int clen = static_cast<int>((V - x0) < sp.tok_r ? (V - x0) : sp.tok_r);
        const uint32_t zb = sp.bulk ? static_cast<uint32_t>(clen * static_cast<int>(sizeof(TIn))) & ~15u : 0u;
        const uint32_t qb = sp.bulk ? static_cast<uint32_t>(clen * 4) & ~15u : 0u;
        mbar_arrive_expect_tx(&full[s], 2u * zb + qb);
        if (zb) {
          bulk_g2s(st.zp, zp_row + x0, zb, &full[s], pol_last);
          bulk_g2s(st.zq, zq_row + x0, zb, &full[s], pol_last);
        }
        if (qb) bulk_g2s(st.q, q_row + x0, qb, &full[s], pol_last);
      };
      if (tid == 0)
        for (int L = 0; L < nst_piece && L < sp.nst; ++L) issue_piece(L);
      bool timed_out = false;
      float zl = 0.f, bk = -INFINITY;
      int bb = INT_MAX;
      for (int L = 0; L < nst_piece; ++L) {
        const uint32_t sq = seq0 + static_cast<uint32_t>(L);
        const Stage<TIn> st = stage_at<TIn>(ring, static_cast<int>(sq % static_cast<uint32_t>(sp.nst)), sp.tok_r);
        const int64_t x0 = piece_lo + static_cast<int64_t>(L) * sp.tok_r;
        const int clen = static_cast<int>((V - x0) < sp.tok_r ? (V - x0) : sp.tok_r);
        const int par = L & 1;
        wait_stage(sq, st, zp_row, zq_row, q_row, x0, clen, true, true, timed_out);
        float part = 0.f;
        for (int sb = warp * tpw; sb < (warp + 1) * tpw && sb < clen; sb += kSub) {  // warp-uniform
          const int i0 = sb + lane * 8;
          float u[8], qv[8];
          scores8(st.zp, st.zq, i0, sb, clen, masked, c1k, ak, Mp, logb, u);
          ld8(st.q + i0, qv);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            part += (i0 + e < clen) ? fmaxf(ex2(u[e] - M) * invS - cJ * qv[e], 0.f) : 0.f;
        }
        zl += part;
        if (race) {
          const float ws = warp_sum(part);
          if (lane == 0) rs->wsum[par][warp] = ws;
        }
        __syncthreads();
        if (tid == 0 && L + sp.nst < nst_piece) issue_piece(L + sp.nst);
        // block masses of the last pass's residual (read while the next stage streams in; the
        // shares are double-buffered, so the next stage's writes go to the other half)
        if (race && tid < sp.tok_r / kRaceBlock && x0 + static_cast<int64_t>(tid) * kRaceBlock < V) {
          float mass = 0.f;
          for (int w = 0; w < wpb; ++w) mass += rs->wsum[par][tid * wpb + w];
          if (mass > 0.f) {
            const int kabs = static_cast<int>(x0 / kRaceBlock) + tid;
            const float key = block_key(p, g, kabs, lg2(mass));
            if (key > bk) {
              bk = key;
              bb = kabs;
            }
          }
        }
      }
      seq = seq0 + static_cast<uint32_t>(nst_piece);
      const float zsum = block_sum(zl, redf);
      block_argmax(bk, bb, redf, redi);
      if (tid == 0) {
        PiecePart pp;
        pp.z = zsum;
        pp.key = bk;
        pp.blk = bb;
        pp.timed_out = timed_out ? 1 : 0;
        slot_parts(sp, rs->slot)[piece] = pp;
        __threadfence();
        const uint32_t t = atomicAdd(&sp.jobs[rs->item].done, 1u);
        rs->last = t + 1u == static_cast<uint32_t>(sp.npieces) ? 1 : 0;
      }
      __syncthreads();
      if (!rs->last) continue;

      // ================= the pass is complete: next sibling test, next pass or terminal race
      const int n = static_cast<int>(g % N);
      if (warp == 0) list_children(p, b, n, kids, ktok);
      if (tid == 0) {
        __threadfence();  // every piece's part was written before its ticket
        SlotHead* sh = slot_head(sp, rs->slot);
        const PiecePart* parts = slot_parts(sp, rs->slot);
        float DJ = 0.f, K = -INFINITY;
        int kstar = INT_MAX;
        uint32_t st2 = sh->status;
        for (int k = 0; k < sp.npieces; ++k) {
          DJ += parts[k].z;
          argmax_merge(K, kstar, parts[k].key, parts[k].blk);
          if (parts[k].timed_out) st2 |= DCD_DEVERR_TIMEOUT;
        }
        bool degen = sh->degen != 0;
        float c = sh->c, D = sh->D;
        if (DJ > 0.f) {
          c = cJ;
          D = DJ;
        } else {
          degen = true;  // r_{J-1} == q in exact arithmetic: r_J is taken as q from here on
        }
        // test the remaining siblings; after a pass without residual mass no pass is needed
        int acc = -1;
        bool queued = false;
        for (int j = J; j < m; ++j) {
          if (sibling_test<TIn>(p, b, kids[j], ktok[j], zp_row, zq_row, q_row, c1k, ak, masked, Mp, logb, M, invS, c,
                                D, degen)) {
            acc = kids[j];
            break;
          }
          if (!degen) {
            sh->c = c;
            sh->D = D;
            sh->degen = 0;
            sh->status = st2;
            create_job(sp, rs->slot, j + 1);
            queued = true;
            break;
          }
        }
        rs->accept = queued ? -2 : acc;
        rs->term = kstar;  // the winning race block when this pass ranked them
        rs->status = st2;
        rs->c = c;
        rs->D = D;
        rs->degen = degen ? 1 : 0;
      }
      __syncthreads();
      if (rs->accept == -2) continue;  // the next pass is queued
      const int acc = rs->accept;
      int term = -1;
      if (acc < 0) {
        // every sibling rejected: terminal draw from r_m, or from q after a pass without mass
        const bool degen = rs->degen != 0;
        const float c = rs->c, D = rs->D;
        int kstar = rs->term;
        if (degen) {
          // block masses of q, computed by this CTA alone (rare: a residual without mass)
          float bk2 = -INFINITY;
          int bb2 = INT_MAX;
          for (int kb = warp; kb < sp.nblk; kb += kWarps) {
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
          block_argmax(bk2, bb2, redf, redi);
          kstar = bb2;
        }
        term = token_race(
            p, g, kstar,
            [&](int64_t x) -> float {
              const float qe = q_row[x];
              if (degen) return qe;
              const float z = ld1(zp_row, x);
              const bool in = !masked || (z - Mp >= logb);
              const float pit = in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, x)) - M) * invS : 0.f;
              return fmaxf(pit - c * qe, 0.f) / D;
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
        __threadfence();
        atomicAdd(&sp.hdr->rows_done, 1u);
      }
      __syncthreads();
      continue;
    }

    // ================= a row
    const int item = rs->item;
    const int b = item % p.B, n = item / p.B;  // node-major order
    const int64_t g = static_cast<int64_t>(b) * N + n;
    const float alpha = p.alpha[b];
    const float beta = p.beta ? p.beta[b] : 0.f;
    const float T = p.temp ? p.temp[b] : 0.f;
    const bool sampled = T > 0.f && p.q != nullptr;
    const bool masked = beta > 0.f;
    const float invT = T > 0.f ? 1.f / T : 1.f;
    const float k2 = kLog2e * invT;  // exp(x / T) = 2^(x * k2)
    // scores are kept in the scaled unit u = k2 s' = c1k z_p - ak z_q, so pi_CD,T ~ 2^u
    const float c1k = (1.f + alpha) * k2, ak = alpha * k2;
    const float logb = masked ? logf(beta) : -INFINITY;
    const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
    const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;
    const float* q_row = sampled ? p.q + g * p.ldq : nullptr;

    // ring items of this row: [max pass if beta > 0] [stats pass]; thread 0 keeps up to nst
    // items in flight
    const int nknown = (masked ? 2 : 1) * nch_a;
    const uint32_t seq0 = seq;
    auto pass_of = [&](int L) -> int { return (masked && L < nch_a) ? kPassMax : kPassStats; };
    auto issue = [&](int L, uint64_t pol) {  // thread 0 only
      const uint32_t sq = seq0 + static_cast<uint32_t>(L);
      const int s = static_cast<int>(sq % static_cast<uint32_t>(sp.nst));
      const int64_t x0 = static_cast<int64_t>(L % nch_a) * sp.tok_a;
      const int clen = static_cast<int>((V - x0) < sp.tok_a ? (V - x0) : sp.tok_a);
      const Stage<TIn> st = stage_at<TIn>(ring, s, sp.tok_a);
      const int kind2 = pass_of(L);
      const uint32_t zb = sp.bulk ? static_cast<uint32_t>(clen * static_cast<int>(sizeof(TIn))) & ~15u : 0u;
      mbar_arrive_expect_tx(&full[s], kind2 == kPassMax ? zb : 2u * zb);
      if (zb) {
        bulk_g2s(st.zp, zp_row + x0, zb, &full[s], pol);
        if (kind2 != kPassMax) bulk_g2s(st.zq, zq_row + x0, zb, &full[s], pol);
      }
    };

    // Thread 0 starts the row's stream at once.  A beta > 0 row keeps its max pass in L2 for
    // the stats pass, and a sampled row its logits for residual pieces until it is known to be
    // a leaf.  Warp 1 meanwhile lists the children of node n, checks the row and loads the
    // values at the children's tokens, which are consumed after the stats pass; the first
    // stage barrier publishes the child count.
    if (tid == 0) {
      const uint64_t pol0 = (masked || sampled) ? pol_last : pol_first;
      const int first = nknown < sp.nst ? nknown : sp.nst;
      for (int L = 0; L < first; ++L) issue(L, pol0);
    }
    float pzp = 0.f, pzq = 0.f, pq = 0.f;
    if (warp == 1) {
      const int count = list_children(p, b, n, kids, ktok);
      if (lane < count) {
        const int t = ktok[lane];
        if (t >= 0 && t < V) {
          pzp = ld1(zp_row, t);
          pzq = ld1(zq_row, t);
          if (sampled) pq = q_row[t];
        }
      }
      if (lane == 0) {
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
      }
    }

    int L = 0;  // next item to consume
    bool timed_out = false;
    // Consumes `count` items: waits for each stage, hands it to `body`, refills the stage once
    // the block has finished it, then runs `after` (which may read what `body` left in shared
    // memory, double-buffered by item parity).
    auto run_items = [&](int count, auto&& body, auto&& after) {
      for (int it = 0; it < count; ++it, ++L) {
        const uint32_t sq = seq0 + static_cast<uint32_t>(L);
        const int s = static_cast<int>(sq % static_cast<uint32_t>(sp.nst));
        const int64_t x0 = static_cast<int64_t>(L % nch_a) * sp.tok_a;
        const int clen = static_cast<int>((V - x0) < sp.tok_a ? (V - x0) : sp.tok_a);
        const Stage<TIn> st = stage_at<TIn>(ring, s, sp.tok_a);
        wait_stage(sq, st, zp_row, zq_row, nullptr, x0, clen, pass_of(L) != kPassMax, false, timed_out);
        body(st, x0, clen, L & 1);
        __syncthreads();
        if (tid == 0 && L + sp.nst < nknown) {
          const bool keep = (masked && L + sp.nst < nch_a) || (sampled && rs->m > 0);
          issue(L + sp.nst, keep ? pol_last : pol_first);
        }
        after(x0, clen, L & 1);
      }
    };
    auto no_after = [](int64_t, int, int) {};

    // ---- pass A (beta > 0): the expert max, for P_beta = {x : z_p(x) - max z_p >= log beta}
    float Mp = 0.f;
    if (masked) {
      float lm = -INFINITY;
      run_items(
          nch_a,
          [&](const Stage<TIn>& st, int64_t, int clen, int) {
            for (int i0 = tid * 8; i0 < clen; i0 += kThreads * 8) {
              float zp[8];
              ld8(st.zp + i0, zp);
#pragma unroll
              for (int e = 0; e < 8; ++e)
                if (i0 + e < clen) lm = fmaxf(lm, zp[e]);
            }
          },
          no_after);
      Mp = block_max(lm, redf);
    }

    // ---- pass B: per lane an online max of u on P_beta, the sum of 2^(u - max) rescaled when
    // the max grows, and the argmax.  A warp takes tok_a / 8 consecutive tokens of each stage, so
    // `wpb` warps cover one race block; for sampled rows each warp also reports its share of the
    // stage's mass, which threads 0.. combine into the block masses after the stage barrier.
    const int tpw = sp.tok_a / kWarps, wpb = kRaceBlock / tpw;
    float lmax = -INFINITY, lsum = 0.f;
    int larg = INT_MAX;
    run_items(
        nch_a,
        [&](const Stage<TIn>& st, int64_t x0, int clen, int par) {
          float bpart = 0.f;  // this lane's share of the warp's mass in this stage, relative to lmax
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
                const float2 d = __fadd2_rn(make_float2(u[2 * k], u[2 * k + 1]), nm2);
                acc2 = __fadd2_rn(acc2, make_float2(ex2(d.x), ex2(d.y)));
              }
              const float a = acc2.x + acc2.y;
              lsum += a;
              bpart += a;
            }
          }
          if (sampled) {
            const float ref = warp_max(lmax);
            const float ws = warp_sum(lmax > -INFINITY ? bpart * ex2(lmax - ref) : 0.f);
            if (lane == 0) {
              rs->wref[par][warp] = ref;
              rs->wsum[par][warp] = ws;
            }
          }
        },
        [&](int64_t x0, int clen, int par) {
          if (sampled && tid < sp.tok_a / kRaceBlock && tid * kRaceBlock < clen) {
            float ref = -INFINITY, sum = 0.f;
            for (int w = 0; w < wpb; ++w) ref = fmaxf(ref, rs->wref[par][tid * wpb + w]);
            if (ref > -INFINITY)
              for (int w = 0; w < wpb; ++w) {
                const float r = rs->wref[par][tid * wpb + w];
                if (r > -INFINITY) sum += rs->wsum[par][tid * wpb + w] * ex2(r - ref);
              }
            const int kabs = static_cast<int>(x0 / kRaceBlock) + tid;
            bmax[kabs] = ref;
            bsum[kabs] = sum;
          }
        });
    seq = seq0 + static_cast<uint32_t>(L);
    const int m = rs->m;
    if (warp == 1 && lane < m) {
      czp[lane] = pzp;
      czq[lane] = pzq;
      cq[lane] = pq;
    }
    for (int k = 32 + tid; k < m; k += kThreads) {  // nodes with more children than a warp has lanes
      const int t = ktok[k];
      const bool ok = t >= 0 && t < V;
      czp[k] = ok ? ld1(zp_row, t) : 0.f;
      czq[k] = ok ? ld1(zq_row, t) : 0.f;
      cq[k] = (ok && sampled) ? q_row[t] : 0.f;
    }
    // row statistics (the reduction's barriers also publish czp / czq / cq and the block masses):
    // M = max u, S = sum 2^(u - M), so log sum exp(s' / T) = M ln 2 + ln S
    float M = lmax, S = lsum;
    int arg = larg;
    block_stats(M, S, arg, redf, redi);
    uint32_t status = rs->status | (timed_out ? DCD_DEVERR_TIMEOUT : 0u);
    if (!(M > -INFINITY && M < INFINITY) || !(S > 0.f && S < INFINITY)) status |= DCD_DEVERR_NONFINITE;
    const float logS = logf(S);
    const float invS = 1.f / S;

    // ---- outputs of the Eq. 1 target
    if (tid == 0) {
      if (p.cd_argmax) p.cd_argmax[g] = arg;
      if (p.cd_lse) p.cd_lse[g] = M * kLn2 + logS;
      if (n == 0 && p.cd_logprob) p.cd_logprob[g] = 0.f;
    }
    if (p.cd_logprob) {
      for (int k = tid; k < m; k += kThreads) {
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
                                   DCD_DEVERR_NONFINITE))) {
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
          create_job(sp, s, 1);
          accept = -1;
        }
        rs->accept = accept;
      }
      __syncthreads();
      if (rs->accept == 1) acc = kids[0];
      if (rs->accept == -1) handed_over = true;
    } else {
      // ---- sampled leaf: the terminal token is drawn from pi_CD,T by the two-level race: a
      // 1024-token block by its mass 2^(bmax - M) bsum ...
      float bk = -INFINITY;
      int bb = INT_MAX;
      for (int k = tid; k < sp.nblk; k += kThreads) {
        if (bmax[k] > -INFINITY && bsum[k] > 0.f) {
          const float key = block_key(p, g, k, lg2(bsum[k]) + (bmax[k] - M));
          if (key > bk) {
            bk = key;
            bb = k;
          }
        }
      }
      block_argmax(bk, bb, redf, redi);
      // ... then a token of that block
      term = token_race(
          p, g, bb,
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
      __threadfence();
      atomicAdd(&sp.hdr->rows_done, 1u);
    }
    __syncthreads();  // row state in shared memory is rewritten by the next work
  }
}

// ------------------------------------------------------------------------------------------
__global__ void tree_walk_kernel(int32_t B, int32_t N, const RowRecord* __restrict__ rec, uint32_t* err,
                                 int32_t* accept_len, int32_t* accept_path, int32_t* bonus) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const RowRecord* r = rec + static_cast<int64_t>(b) * N;
  int32_t* path = accept_path + static_cast<int64_t>(b) * N;
  uint32_t st = 0u;
  for (int i = 0; i < N; ++i) st |= r[i].status;
  int cur = 0, len = 0;
  path[0] = 0;
  if (st) {
    atomicOr(err, st);
    for (int i = 1; i < N; ++i) path[i] = -1;
    accept_len[b] = 0;
    bonus[b] = -1;
    return;
  }
  while (len < N - 1) {
    const int a = r[cur].acc_child;
    if (a <= cur || a >= N) break;
    cur = a;
    path[++len] = cur;
  }
  for (int i = len + 1; i < N; ++i) path[i] = -1;
  accept_len[b] = len;
  bonus[b] = r[cur].term_token;
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
  for (int c = cur + 1; c < N; ++c) {
    if (p.parents[static_cast<int64_t>(b) * N + c] != cur) continue;
    float z = 0.f;
    for (int64_t x = threadIdx.x; x < V; x += kThreads) {
      const float nv = fmaxf(out[x] - q[x], 0.f);
      out[x] = nv;
      z += nv;
    }
    z = block_sum(z, redf);
    if (z > 0.f) {
      const float iz = 1.f / z;
      for (int64_t x = threadIdx.x; x < V; x += kThreads) out[x] *= iz;
    } else {
      for (int64_t x = threadIdx.x; x < V; x += kThreads) out[x] = q[x];
    }
    __syncthreads();
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
    d.err = cudaFuncSetAttribute(score_rows_kernel<TIn>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kSmemMax));
    if (d.err == cudaSuccess) d.err = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
    info[dev] = d;
  });
  *sms = info[dev].sms;
  return info[dev].err;
}

struct Layout {
  int meta_offset, blk_offset, stage_offset;
  size_t total;
};

Layout layout_for(int N, int nblk, int nst) {
  Layout l;
  l.meta_offset = 8 * kMaxStages + 64 * 4;
  const size_t meta_end = static_cast<size_t>(l.meta_offset) + sizeof(RowShared) + static_cast<size_t>(N) * 4 * 5;
  l.blk_offset = static_cast<int>((meta_end + 15) & ~static_cast<size_t>(15));
  const size_t blk_end = static_cast<size_t>(l.blk_offset) + static_cast<size_t>(nblk) * 4 * 2;
  l.stage_offset = static_cast<int>((blk_end + 127) & ~static_cast<size_t>(127));
  l.total = static_cast<size_t>(l.stage_offset) + static_cast<size_t>(nst) * kStageBytes;
  return l;
}

// Tokens per stage, in whole race blocks: z_p and z_q fill a stage in row passes; z_p, z_q and
// q share it in residual pieces.
int tokens_a(int es) { return kStageBytes / (2 * es) / kRaceBlock * kRaceBlock; }
int tokens_r(int es) { return kStageBytes / (2 * es + 4) / kRaceBlock * kRaceBlock; }

// A warp takes tok / 8 tokens of a stage in groups of 256, and whole warps cover a race block.
bool stage_split_ok(int tok) {
  const int tpw = tok / kWarps;
  return tok > 0 && tok % (kWarps * kSub) == 0 && tpw <= kRaceBlock && kRaceBlock % tpw == 0 &&
         tok / kRaceBlock <= kThreads;
}

}  // namespace

int residual_pieces(int64_t V, int dtype) {
  const int es = dtype == DCD_BF16 ? 2 : 4;
  const int64_t tok = static_cast<int64_t>(tokens_r(es)) * kPieceStages;
  return static_cast<int>((V + tok - 1) / tok);
}

size_t slot_bytes(int64_t V, int dtype) {
  return sizeof(SlotHead) + static_cast<size_t>(residual_pieces(V, dtype)) * sizeof(PiecePart);
}

RowGeometry row_geometry(const ScoreArgs& a) {
  RowGeometry geo{};
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  const int nblk = static_cast<int>((a.V + kRaceBlock - 1) / kRaceBlock);
  const int nst = a.force_stages > 0 ? a.force_stages : 2;
  const Layout l = layout_for(a.N, nblk, nst);
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

cudaError_t launch_score_rows(const ScoreArgs& a, cudaStream_t stream) {
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  if (R == 0) return cudaSuccess;
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
  sp.npieces = residual_pieces(a.V, a.dtype);
  sp.bulk = geo.bulk;
  sp.nblk = static_cast<int>((a.V + kRaceBlock - 1) / kRaceBlock);
  const Layout l = layout_for(a.N, sp.nblk, sp.nst);
  sp.meta_offset = l.meta_offset;
  sp.blk_offset = l.blk_offset;
  sp.stage_offset = l.stage_offset;
  sp.slot_bytes = static_cast<int32_t>(slot_bytes(a.V, a.dtype));
  sp.hdr = a.hdr;
  sp.jobs = a.jobs;
  sp.slots = a.slots;
  // the header counters and the job list start every call at zero
  e = cudaMemsetAsync(a.hdr, 0, kWorkspaceHeader + static_cast<size_t>(R) * sizeof(Job), stream);
  if (e != cudaSuccess) return e;
  // a CTA may wait for work queued by another, so all CTAs must be resident at once: the grid is
  // the resident capacity (capped at the row count) and the launch is cooperative
  int per_sm = 0;
  e = a.dtype == DCD_BF16
          ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_rows_kernel<__nv_bfloat16>, kThreads, geo.smem)
          : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_rows_kernel<float>, kThreads, geo.smem);
  if (e != cudaSuccess) return e;
  if (per_sm > geo.ctas_per_sm) per_sm = geo.ctas_per_sm;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  int64_t grid = static_cast<int64_t>(sms) * per_sm;
  if (grid > R) grid = R;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = geo.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (a.dtype == DCD_BF16) return cudaLaunchKernelEx(&cfg, score_rows_kernel<__nv_bfloat16>, sp);
  return cudaLaunchKernelEx(&cfg, score_rows_kernel<float>, sp);
}

cudaError_t launch_tree_walk(int32_t B, int32_t N, const RowRecord* rec, uint32_t* err, int32_t* accept_len,
                             int32_t* accept_path, int32_t* bonus, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const int threads = 128;
  tree_walk_kernel<<<(B + threads - 1) / threads, threads, 0, stream>>>(B, N, rec, err, accept_len, accept_path,
                                                                        bonus);
  return cudaGetLastError();
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
