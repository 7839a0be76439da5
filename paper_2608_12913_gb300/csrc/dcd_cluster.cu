// dcd_cluster.cu -- the CD verification step with one thread-block cluster per tree-node row.
//
// cluster_rows_kernel: a row g = b * N + n is verified by a cluster of C CTAs (C = 1, 2, 4 or
// 8, chosen per call so that the grid has several waves).  CTA s of the cluster owns a slice of
// the vocabulary, whole ring stages of the statistics pass, so that slices are whole blocks of
// the terminal race.  Each CTA is warp-specialised like the persistent row kernel: a producer
// warp streams its slice with bulk asynchronous copies into a ring of 32 KB shared-memory stages
// (full / empty mbarriers), and eight consumer warps score it.
//
//  * Statistics.  The consumers compute the CD score of Eq. 1 on the plausibility set P_beta of
//    Sec. 2.1 in the scaled unit u = k2 s' (k2 = log2(e) / T), keep per lane an online max,
//    a rescaled sum of 2^(u - max) and the argmax, and reduce them over the CTA.  The C slices'
//    statistics are then exchanged through distributed shared memory: every CTA pushes its share
//    into every CTA of the cluster (remote stores, then a remote mbarrier arrive with release
//    semantics at cluster scope) and waits on its own mbarrier, so every CTA combines the same C
//    values in the same order and takes the same decisions.  With beta > 0 an exchange of the
//    slices' expert maxima comes first.
//  * Greedy rule, first sibling test, leaf race: as in Algorithm 1 (T -> 0 limit, or the first
//    sibling with r_0 = pi); a sampled leaf draws its terminal token by the two-level exponential
//    race, the block by its mass over the exchange, the token by the CTA that owns the block.
//  * Residual chain.  After a rejected sibling the next residual r_J = max(0, pi - c_J q) / D_J
//    (c_1 = 1, c_{J+1} = c_J + D_J) needs D_J over the whole vocabulary: the consumers tell their
//    producer to stream the slice again with q, sum max(0, pi - c_J q), and exchange the sums;
//    every CTA then tests the next sibling.  The pass after the last sibling also ranks its race
//    blocks, and the CTA that owns the winning block draws the terminal token.
//  * Siblings without replacement (DCD_SIBLINGS_DISTINCT, a template parameter): each CTA keeps
//    the same list of removed tokens, the first pass also sums q (the proposal's actual mass),
//    and the exchanged sums and the owning CTA's race blocks are corrected at the removed
//    tokens, whose residual mass stays frozen; the next residual is max(0, pi - c q) with
//    c_{J+1} = c_J + D_J / Z off them.
//
// No CTA waits for a CTA of another cluster, and the CTAs of a cluster are co-scheduled, so the
// grid needs no co-residency.  Every wait is bounded and sets DCD_DEVERR_TIMEOUT when it gives
// up.  The records are read by tree_walk_kernel (dcd_rows.cu).

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <cfloat>
#include <climits>
#include <mutex>

#include "dcd.h"
#include "dcd_cluster.h"
#include "dcd_device.cuh"
#include "dcd_internal.h"

namespace dcd {
namespace {

using namespace dev;

constexpr int kCStage = 32 * 1024;         // bytes per ring stage
constexpr int kCWarps = 8;                 // consumer warps
constexpr int kCThreads = kCWarps * 32;
constexpr int kCCtaThreads = kCThreads + 32;
constexpr int kCMaxStages = 4;
constexpr int kCMaxCluster = 8;
#ifndef DCD_CLUSTER_CTAS_PER_SM
#define DCD_CLUSTER_CTAS_PER_SM 3
#endif
#ifndef DCD_CLUSTER_RING
#define DCD_CLUSTER_RING 2
#endif
#ifndef DCD_CLUSTER_MAX
#define DCD_CLUSTER_MAX 8
#endif
#ifndef DCD_CLUSTER_C
#define DCD_CLUSTER_C 0
#endif
constexpr int kCMinCtas = DCD_CLUSTER_CTAS_PER_SM;
constexpr int kCRing = DCD_CLUSTER_RING;
constexpr int kCMax = DCD_CLUSTER_MAX;
constexpr int kCFixed = DCD_CLUSTER_C;     // nonzero: this cluster size whenever it fits
// how a CTA takes a row: whole, its slice of a row split over the cluster, or one of P parts
enum RowMode { kWhole = 0, kSplit = 1, kPart = 2 };
constexpr int kMail = 4;                   // row messages in flight from a cluster's first CTA
constexpr int kCDesc = 2;                  // rows handed to the consumers ahead
constexpr int kSeqListMax = 1024;
#ifndef DCD_CLUSTER_HOLD_MAX
#define DCD_CLUSTER_HOLD_MAX 2
#endif
// A cluster claims its next sampled row one ahead of a node with at most kHoldMax children (a
// rejection there starts a chain of at most kHoldMax passes, which the row claimed ahead waits
// out); after a wider node it claims once the first sibling is decided or the chain settled.
constexpr int kHoldMax = DCD_CLUSTER_HOLD_MAX;
#ifndef DCD_CLUSTER_SUSPEND_NS
#define DCD_CLUSTER_SUSPEND_NS 20000
#endif
constexpr uint32_t kSuspendNs = DCD_CLUSTER_SUSPEND_NS;  // try_wait suspend-time hint, 0: none
#ifndef DCD_CLUSTER_HALF_ROWS
#define DCD_CLUSTER_HALF_ROWS -1
#endif
#ifndef DCD_CLUSTER_QUARTER_ROWS
#define DCD_CLUSTER_QUARTER_ROWS 0
#endif
// The greedy rows of phase 2 go out whole, then (the last kHalfRows + kQuarterRows) as two, then
// (the last kQuarterRows) as four part units each, so that the step's last units are short; a
// row's parts combine through the workspace (a ticket per row).  kHalfRows < 0: a quarter as
// many rows as the grid has CTAs in halves (measured on 456 CTAs: 114-152 rows best; none, or a
// whole wave of 456, about 1.5 % slower; all rows in halves or quarters slower still).
constexpr int kHalfRows = DCD_CLUSTER_HALF_ROWS;
constexpr int kQuarterRows = DCD_CLUSTER_QUARTER_ROWS;
static_assert(kMaxParts >= 4, "part records");          // sequences up to which the row order lists them in shared memory
static_assert(kCMax >= 1 && kCMax <= kCMaxCluster, "cluster size");
constexpr float kLn2c = 0.69314718055994531f;
#ifdef DCD_CLUSTER_DEBUG
// debug builds record which bounded wait gave up (a bit per site in the header's first spare word)
// and a timeline of the rows (records of 8 words in the workspace's slot area)
#define CL_SITE(n) atomicOr(&p.hdr->reserved[0], 1u << (n))
__device__ __forceinline__ unsigned long long gtimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
#define CL_T(var) const unsigned long long var = gtimer()
#define CL_ACC(acc, t0) (acc += gtimer() - (t0))
#define CL_REC(g, split, t0, t1, npass, m)                                                           \
  do {                                                                                              \
    const uint32_t ei = atomicAdd(&p.hdr->reserved[2], 1u);                                         \
    if (ei < 8192u) {                                                                               \
      uint32_t* r = reinterpret_cast<uint32_t*>(p.slots) + 16u * ei;                                \
      r[8] = static_cast<uint32_t>(w_full);                                                         \
      r[9] = static_cast<uint32_t>(w_xchg);                                                         \
      r[10] = static_cast<uint32_t>(w_desc);                                                        \
      const unsigned long long t2 = gtimer();                                                        \
      r[0] = blockIdx.x;                                                                            \
      r[1] = static_cast<uint32_t>(g);                                                              \
      r[11] = static_cast<uint32_t>(split);                                                         \
      r[2] = static_cast<uint32_t>(t0);                                                             \
      r[3] = static_cast<uint32_t>(t0 >> 32);                                                       \
      r[4] = static_cast<uint32_t>(t1 - t0);                                                        \
      r[5] = static_cast<uint32_t>(t2 - t0);                                                        \
      r[6] = static_cast<uint32_t>(npass);                                                          \
      r[7] = static_cast<uint32_t>(m);                                                              \
    }                                                                                               \
  } while (0)
#else
#define CL_SITE(n) ((void)0)
#define CL_T(var) \
  const unsigned long long var = 0;  \
  (void)var
#define CL_ACC(acc, t0) ((void)0)
#define CL_REC(g, split, t0, t1, npass, m) ((void)0)
#endif
using CSync = SyncConsumersN<kCThreads>;

// One CTA's share of an exchange (32 bytes, pushed as two 16-byte stores).
struct alignas(16) XPart {
  float a, b;       // statistics: max u and rescaled sum; residual pass: partial mass; max pass: max z_p
  int32_t i;        // statistics: argmax
  float key;        // best race key of the slice's blocks
  int32_t blk;      // its block (INT_MAX: none)
  uint32_t status;  // DCD_DEVERR_* bits
  int32_t pad[2];
};
static_assert(sizeof(XPart) == 32, "XPart layout");

struct CParams {
  ScoreArgs a;
  int32_t C;             // CTAs per cluster: slices per row
  int32_t tok_a, tok_r;  // tokens per stage: statistics (z_p, z_q) and residual passes (z_p, z_q, q)
  int32_t spc;           // statistics stages per slice
  int32_t nchunk;        // chunk-mass slots
  int32_t meta_offset, chunk_offset, stage_offset;
  int32_t seq_offset;    // shared-memory offset of the sequence list (sampled first), 0: none
};

// Consumer state shared by the consumer warps (written by one thread, read after a barrier).
struct CShared {
  int32_t m;         // children of the row's node
  uint32_t status;   // DCD_DEVERR_* bits of the row
  int32_t decision;  // outcome of thread 0's sibling steps
  int32_t term;      // winning race block
  int32_t J;         // next residual pass
  float c, D;        // current residual max(0, pi - c q) / D
  float cJ;          // c of the next pass
  int32_t degen;     // a pass found no residual mass: r = q from here on
  // Distinct siblings: the proposal's mass Z (q's own, less the removed tokens' q), and the
  // removed tokens with their frozen residual masses and pi and q at them (every CTA of a
  // cluster keeps the same copy, written by its thread 0 from the same values)
  float Z;
  int32_t nrem;
  int32_t pad;
  int32_t rtok[kMaxRemoved];
  float rfz[kMaxRemoved];
  float rpit[kMaxRemoved];
  float rq[kMaxRemoved];
};

struct Cmd {
  int32_t kind;  // 1: stream the slice for a residual pass (hint: 1 = a later pass re-reads it), 0: stop
  int32_t keep;
  int32_t pad[2];
};

template <typename TIn>
struct CStage {
  TIn* zp;
  TIn* zq;
  float* q;
};

template <typename TIn>
__device__ __forceinline__ CStage<TIn> cstage(unsigned char* base, int s, int tok) {
  CStage<TIn> st;
  st.zp = reinterpret_cast<TIn*>(base + static_cast<size_t>(s) * kCStage);
  st.zq = st.zp + tok;
  st.q = reinterpret_cast<float*>(st.zq + tok);
  return st;
}

// ---- cluster PTX: rank, barrier, remote shared-memory addresses, stores and arrivals
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Before exit: no CTA of the cluster leaves while another may still access its shared memory
// (the threads of a CTA arrive at different times, so the barrier is not .aligned).
__device__ __forceinline__ void cluster_sync_end() {
  asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

__device__ __forceinline__ uint32_t map_rank(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(p)), "r"(rank));
  return r;
}

__device__ __forceinline__ void st_cluster_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared::cluster.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

__device__ __forceinline__ void arrive_cluster(uint32_t bar_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_addr) : "memory");
}

__device__ __forceinline__ bool try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  if (kSuspendNs == 0)
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.b32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
  else
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.b32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity), "r"(kSuspendNs)
        : "memory");
  return done != 0;
}

__device__ __forceinline__ bool wait_cluster_bounded(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!try_wait_cluster(bar, parity))
    if (clock64() - t0 > kWaitCycles) return false;
  return true;
}

// A CTA-scope wait whose try_wait may suspend the thread for up to kSuspendNs (it resumes when
// the phase completes), so that a waiting warp does not take issue slots from the computing ones;
// bounded like mbar_wait_bounded.
__device__ __forceinline__ bool cwait_bounded(uint64_t* bar, uint32_t parity) {
  if (kSuspendNs == 0) return mbar_wait_bounded(bar, parity);
  const long long t0 = clock64();
  for (;;) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.b32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity), "r"(kSuspendNs)
        : "memory");
    if (done) return true;
    if (clock64() - t0 > kWaitCycles) return false;
  }
}

// Lists the children of node n (ascending id) with the calling warp; returns their count.
__device__ __forceinline__ int clist_children(const ScoreArgs& p, int b, int n, int* kids, int* ktok) {
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

// The scaled CD score u = c1k z_p - ak z_q of 8 staged tokens; tokens past `clen` or outside
// P_beta get -inf.  A whole 256-token group of an unmasked row uses packed fp32x2 arithmetic
// (the same roundings as the scalar path).
template <typename TIn>
__device__ __forceinline__ void cscores8(const TIn* zp_s, const TIn* zq_s, int i0, int sb, int clen, bool masked,
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

// Second level of the terminal race over block `kstar`: the token x with the largest
// log2 r(x) - log2(-log2 u_x), four tokens a consumer thread (Philox counter 1 + x / 4);
// `mass(x)` returns r(x) up to a common factor.  Every consumer thread gets the token.
template <typename MassFn>
__device__ int ctoken_race(const ScoreArgs& p, int64_t g, int kstar, MassFn mass, float* redf, int* redi) {
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
  block_argmax(tk, tx, redf, redi, CSync());
  return tx;
}

// First level of the race: the key of block k from log2 of its mass.
__device__ __forceinline__ float cblock_key(const ScoreArgs& p, int64_t g, int k, float log2_mass) {
  const uint4 w =
      philox_block(p.seed, p.offset, static_cast<uint32_t>(g), 0x80000000u | (static_cast<uint32_t>(k) >> 2));
  return race_key(log2_mass, word_of(w, k & 3));
}

template <typename TIn, bool kDistinct>
__global__ void __launch_bounds__(kCCtaThreads, kCMinCtas) cluster_rows_kernel(const __grid_constant__ CParams cp) {
  const ScoreArgs& p = cp.a;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int C = cp.C;
  const uint32_t rank = cluster_rank();
  const int N = p.N;
  const int64_t V = p.V;
  const int R = p.B * N;
  const int nch_a = static_cast<int>((V + cp.tok_a - 1) / cp.tok_a);
  const int st_lo = static_cast<int>(rank) * cp.spc;
  const int st_hi = st_lo + cp.spc < nch_a ? st_lo + cp.spc : nch_a;
  // this CTA's slice of a row split over the cluster; a whole row spans [0, V)
  const int64_t sl_lo = static_cast<int64_t>(st_lo) * cp.tok_a;
  const int64_t sl_hi =
      st_hi > st_lo ? (static_cast<int64_t>(st_hi) * cp.tok_a < V ? static_cast<int64_t>(st_hi) * cp.tok_a : V) : sl_lo;

  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);  // [kCMaxStages] stage filled
  uint64_t* empty = full + kCMaxStages;                // [kCMaxStages] stage released
  uint64_t* xbar = empty + kCMaxStages;                // [2] exchange buffer filled
  uint64_t* cmdbar = xbar + 2;                         // [1] command posted
  uint64_t* mfull = cmdbar + 1;                        // [kMail] row message received
  uint64_t* mempty = mfull + kMail;                    // [kMail] (rank 0) message slot read by the peers
  uint64_t* dfull = mempty + kMail;                    // [kCDesc] row handed to the consumers
  uint64_t* dempty = dfull + kCDesc;                   // [kCDesc] row descriptor read
  float* redf = reinterpret_cast<float*>(dempty + kCDesc + 1);  // [64]
  int* redi = reinterpret_cast<int*>(redf + 64);               // [32]
  XPart* xpart = reinterpret_cast<XPart*>(redi + 32);          // [2][kCMaxCluster]
  Cmd* cmd = reinterpret_cast<Cmd*>(xpart + 2 * kCMaxCluster);
  int* mail = reinterpret_cast<int*>(cmd + 1);  // [kMail]
  int* desc = mail + kMail;                     // [kCDesc][8] row, mode, flags, alpha, beta, T
  CShared* sh = reinterpret_cast<CShared*>(smem + cp.meta_offset);
  int* seqs = cp.seq_offset > 0 ? reinterpret_cast<int*>(smem + cp.seq_offset) : nullptr;  // [B]
  int* kids = reinterpret_cast<int*>(sh + 1);  // [N]
  int* ktok = kids + N;                        // [N]
  float* czp = reinterpret_cast<float*>(ktok + N);
  float* czq = czp + N;
  float* cq = czq + N;
  float* cref = reinterpret_cast<float*>(smem + cp.chunk_offset);  // [nchunk]
  float* csum = cref + cp.nchunk;                                  // [nchunk]
  unsigned char* ring = smem + cp.stage_offset;

  if (tid == 0) {
    for (int s = 0; s < kCRing; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCWarps);
    }
    mbar_init(&xbar[0], static_cast<uint32_t>(C));
    mbar_init(&xbar[1], static_cast<uint32_t>(C));
    mbar_init(cmdbar, 1);
    for (int d = 0; d < kMail; ++d) {
      mbar_init(&mfull[d], 1);
      mbar_init(&mempty[d], static_cast<uint32_t>(C > 1 ? C - 1 : 1));
    }
    for (int d = 0; d < kCDesc; ++d) {
      mbar_init(&dfull[d], 1);
      mbar_init(&dempty[d], 1);
    }
    fence_mbar_init();
  }
  // The producer warp lists the sampled sequences, then the greedy ones.  Phase 1 takes the sampled
  // sequences' rows, split over the cluster: their residual chains then run on C CTAs, and start
  // early.  Phase 2 takes the greedy sequences' rows, each whole on one CTA.  Without a list (a
  // very large batch) every row is taken whole in phase 2, in node-major order.
  int nS = 0;
  if (warp == kCWarps && seqs) {
    for (int pass = 0; pass < 2; ++pass) {
      int cnt = pass == 0 ? 0 : nS;
      for (int base = 0; base < p.B; base += 32) {
        const int bb = base + lane;
        const bool smp = bb < p.B && p.temp && p.q && p.temp[bb] > 0.f;
        const bool take = bb < p.B && (pass == 0 ? smp : !smp);
        const unsigned msk = __ballot_sync(~0u, take);
        if (take) seqs[cnt + __popc(msk & ((1u << lane) - 1u))] = bb;
        cnt += __popc(msk);
      }
      if (pass == 0) nS = cnt;
    }
    __syncwarp();
  }
  __syncthreads();
  cluster_sync_all();  // every CTA's barriers are initialised before any remote arrival

  if (warp == kCWarps) {
    // ===================================== producer warp (lane 0 issues the copies)
    const uint64_t pol_first = l2_policy_evict_first();
    const uint64_t pol_normal = l2_policy_evict_normal();
    const uint64_t pol_last = l2_policy_evict_last();
    const int nA = nS * N;  // phase-1 rows
    // the row of claim index i of phase 1 (sampled sequences) or of phase 2 (the others)
    auto row1 = [&](int i) { return seqs[i % nS] * N + i / nS; };
    auto row2 = [&](int i) {
      const int ng = p.B - nS;
      return seqs ? seqs[nS + i % ng] * N + i / ng : (i % p.B) * N + i / p.B;
    };
    uint32_t issued = 0, ncmd = 0, kd = 0;  // ring stages issued, commands read, descriptors handed
    // kind 0: z_p only (expert max), 1: z_p and z_q, 2: z_p, z_q and q; `first` runs at the first
    // stage (rank 0 announces the cluster's next row there, while this one streams)
    auto stream = [&](int g, int64_t lo, int64_t hi, int tok, int kind, uint64_t pol, auto first) {
      const TIn* zp_row = static_cast<const TIn*>(p.zp) + static_cast<int64_t>(g) * p.ld;
      const TIn* zq_row = static_cast<const TIn*>(p.zq) + static_cast<int64_t>(g) * p.ld;
      const float* q_row = kind == 2 ? p.q + static_cast<int64_t>(g) * p.ldq : nullptr;
      for (int64_t x0 = lo; x0 < hi; x0 += tok, ++issued) {
        const int s = static_cast<int>(issued % static_cast<uint32_t>(kCRing));
        const uint32_t phase = ((issued / static_cast<uint32_t>(kCRing)) & 1u) ^ 1u;
        const int clen = static_cast<int>((hi - x0) < tok ? (hi - x0) : tok);
        const CStage<TIn> st = cstage<TIn>(ring, s, tok);
        if (!cwait_bounded(&empty[s], phase)) {
          atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
          CL_SITE(0);
        }
        // bulk copies of the 16-byte multiple; the ragged remainder is stored first
        const int zfirst = ((clen * static_cast<int>(sizeof(TIn))) & ~15) / static_cast<int>(sizeof(TIn));
        const int qfirst = ((clen * 4) & ~15) / 4;
        for (int i = zfirst; i < clen; ++i) {
          st.zp[i] = zp_row[x0 + i];
          if (kind > 0) st.zq[i] = zq_row[x0 + i];
        }
        if (kind == 2)
          for (int i = qfirst; i < clen; ++i) st.q[i] = q_row[x0 + i];
        const uint32_t zb = static_cast<uint32_t>(zfirst) * static_cast<uint32_t>(sizeof(TIn));
        const uint32_t qb = kind == 2 ? static_cast<uint32_t>(qfirst) * 4u : 0u;
        mbar_arrive_expect_tx(&full[s], (kind == 0 ? zb : 2u * zb) + qb);
        if (zb) {
          bulk_g2s(st.zp, zp_row + x0, zb, &full[s], pol);
          if (kind > 0) bulk_g2s(st.zq, zq_row + x0, zb, &full[s], pol);
        }
        if (qb) bulk_g2s(st.q, q_row + x0, qb, &full[s], pol);
        if (x0 == lo) first();
      }
    };
    // The row's parameters travel with its descriptor, so the consumers start on its stages with
    // no dependent global load.  flags: 1 sampled, 2 node with a child, 4 beta > 0.
    struct Meta {
      int g, mode, flags;
      float alpha, beta, T;
    };
    auto meta_of = [&](int g, int mode) -> Meta {  // the whole warp
      Meta mt{g, mode, 0, 0.f, 0.f, 0.f};
      if (g < 0) return mt;
      const int b = g / N, n = g % N;
      mt.alpha = p.alpha[b];
      mt.beta = p.beta ? p.beta[b] : 0.f;
      mt.T = p.temp ? p.temp[b] : 0.f;
      int nkids = 0;
      for (int base = n + 1; base < N; base += 32) {
        const int c = base + lane;
        nkids += __popc(__ballot_sync(~0u, c < N && p.parents[static_cast<int64_t>(b) * N + c] == n));
      }
      mt.flags = ((mt.T > 0.f && p.q != nullptr) ? 1 : 0) | (nkids > 0 ? 2 : 0) | (mt.beta > 0.f ? 4 : 0) |
                 ((nkids > kHoldMax ? 1 : 0) << 3);
      return mt;
    };
    auto hand = [&](const Meta& mt) {  // lane 0: the next row descriptor for the consumers
      const int d = static_cast<int>(kd % kCDesc);
      if (!cwait_bounded(&dempty[d], ((kd / kCDesc) & 1u) ^ 1u)) {
        atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
        CL_SITE(3);
      }
      int* dd = desc + 8 * d;
      dd[0] = mt.g;
      dd[1] = mt.mode;
      dd[2] = mt.flags;
      dd[3] = __float_as_int(mt.alpha);
      dd[4] = __float_as_int(mt.beta);
      dd[5] = __float_as_int(mt.T);
      mbar_arrive(&dfull[d]);
      ++kd;
    };
    auto nop = [] {};

    // ---- phase 1: the sampled sequences' rows, each split over the cluster.  The cluster's first
    // CTA claims them and sends each to the others as message k: one row ahead of a node with at
    // most kHoldMax children, else once the node's first sibling is accepted or its chain is
    // settled (a row claimed ahead of a long chain would wait for it, and finish last).
    int next_i = 0, g_next = -1;
    auto send = [&](uint32_t k, int gr) {  // rank 0, lane 0
      const int d = static_cast<int>(k % kMail);
      if (C > 1 && k >= static_cast<uint32_t>(kMail) && !wait_cluster_bounded(&mempty[d], ((k / kMail) - 1u) & 1u)) {
        atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
        CL_SITE(1);
      }
      for (int t = 1; t < C; ++t) {
        asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(map_rank(&mail[d], static_cast<uint32_t>(t))), "r"(gr)
                     : "memory");
        arrive_cluster(map_rank(&mfull[d], static_cast<uint32_t>(t)));
      }
    };
    // the first row of cluster c is claim index c, which every CTA of the cluster computes itself;
    // later claims come from the counter, after the ncl static ones.  Message j carries the row of
    // iteration j + 1.
    const int ncl = static_cast<int>(gridDim.x) / C;
    auto claim = [&]() { return ncl + static_cast<int>(atomicAdd(&p.hdr->work, 1u)); };
    {
      const int i0 = static_cast<int>(blockIdx.x) / C;
      next_i = i0;
      g_next = i0 < nA ? row1(i0) : -1;
    }
    bool stop = false;
    for (uint32_t k = 0; !stop; ++k) {
      int g = -1;
      if (lane == 0) {
        if (rank == 0 || k == 0) {
          g = g_next;
        } else {
          const uint32_t j = k - 1u;  // message index
          const int d = static_cast<int>(j % kMail);
          if (!wait_cluster_bounded(&mfull[d], (j / kMail) & 1u)) {
            atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
            CL_SITE(2);
            g = -1;
          } else {
            g = *reinterpret_cast<volatile int*>(&mail[d]);
            if (g >= 0) arrive_cluster(map_rank(&mempty[d], 0u));  // the last message is not acknowledged
          }
        }
      }
      g = __shfl_sync(~0u, g, 0);
      if (g < 0) break;
      const Meta mt = meta_of(g, kSplit);
      const bool masked = (mt.flags & 4) != 0;
      const bool has_child = (mt.flags & 2) != 0;  // a sampled node with a child may start a residual chain
      const bool wide = (mt.flags & 8) != 0;       // more than kHoldMax children
      if (lane == 0) {
        bool sent = false;
        if (rank == 0 && !wide) next_i = claim();  // one row ahead
        hand(mt);
        if (masked) stream(g, sl_lo, sl_hi, cp.tok_a, 0, pol_last, nop);  // the statistics pass re-reads it
        // the slice of a node with a child stays in L2 for the residual pass that may follow
        stream(g, sl_lo, sl_hi, cp.tok_a, 1, has_child ? pol_normal : pol_first, [&] {
          if (rank == 0 && !wide) {
            g_next = next_i < nA ? row1(next_i) : -1;
            send(k, g_next);
            sent = true;
          }
        });
        for (; has_child; ++ncmd) {
          if (!cwait_bounded(cmdbar, ncmd & 1u)) {
            atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
            CL_SITE(4);
            stop = true;
            break;
          }
          const int kind = *reinterpret_cast<volatile int32_t*>(&cmd->kind);
          const int keep = *reinterpret_cast<volatile int32_t*>(&cmd->keep);
          if (kind == 0) {
            ++ncmd;
            break;
          }
          stream(g, sl_lo, sl_hi, cp.tok_r, 2, keep ? pol_normal : pol_first, nop);
        }
        if (rank == 0 && !sent) {  // a wide node's first sibling decided or its chain settled
          next_i = stop ? nA : claim();
          g_next = next_i < nA ? row1(next_i) : -1;
          send(k, g_next);
        }
      }
      stop = __shfl_sync(~0u, stop ? 1 : 0, 0) != 0;
    }
    // ---- phase 2: every other row, whole or (the last nH) as two half-row units, claimed by each
    // CTA on its own (one ahead)
    const int nB = R - nA;
    // rows in parts (greedy rows when listed): the last nQ in quarters, the nH before them in halves
    const int nQ = seqs ? (nB < kQuarterRows ? nB : kQuarterRows) : 0;
    const int want_h = kHalfRows < 0 ? static_cast<int>(gridDim.x) / 4 : kHalfRows;
    const int nH = seqs ? (nB - nQ < want_h ? nB - nQ : want_h) : 0;
    const int nW = nB - nH - nQ;
    const int units = nW + 2 * nH + 4 * nQ;
    const int nch_a = static_cast<int>((V + cp.tok_a - 1) / cp.tok_a);
    int i2 = 0;
    if (lane == 0 && !stop) i2 = static_cast<int>(atomicAdd(&p.hdr->job_alloc, 1u));
    while (!stop) {
      int g = -1, mode = kWhole;
      if (lane == 0) {
        for (;;) {
          if (i2 >= units) {
            g = -1;
            break;
          }
          int r2 = i2, P = 1, part = 0;
          if (i2 >= nW + 2 * nH) {
            r2 = nW + nH + (i2 - nW - 2 * nH) / 4;
            P = 4;
            part = (i2 - nW - 2 * nH) & 3;
          } else if (i2 >= nW) {
            r2 = nW + (i2 - nW) / 2;
            P = 2;
            part = (i2 - nW) & 1;
          }
          g = row2(r2);
          // a row with beta > 0 needs its expert max over the whole row: its first unit takes it
          // whole; so does a row with fewer stages than parts
          const bool whole = P == 1 || (p.beta && p.beta[g / N] > 0.f) || nch_a < P;
          if (whole && part > 0) {
            i2 = static_cast<int>(atomicAdd(&p.hdr->job_alloc, 1u));
            continue;
          }
          mode = whole ? kWhole : (kPart | (P << 4) | (part << 8));
          break;
        }
        if (g >= 0) i2 = static_cast<int>(atomicAdd(&p.hdr->job_alloc, 1u));
      }
      g = __shfl_sync(~0u, g, 0);
      mode = __shfl_sync(~0u, mode, 0);
      const Meta mt = meta_of(g, mode);
      if (lane == 0) hand(mt);
      if (g < 0) break;
      int64_t lo = 0, hi = V;
      if ((mode & 15) == kPart) {
        const int P = (mode >> 4) & 15, part = mode >> 8, spp = (nch_a + P - 1) / P;
        lo = static_cast<int64_t>(part) * spp * cp.tok_a;
        hi = static_cast<int64_t>(part + 1) * spp * cp.tok_a < V ? static_cast<int64_t>(part + 1) * spp * cp.tok_a : V;
      }
      const bool masked = (mt.flags & 4) != 0;
      // a whole row of a sampled sequence (a batch without the sequence list) may start a chain
      const bool sampled = (mt.flags & 1) != 0;
      const bool has_child = (mt.flags & 2) != 0;
      if (lane == 0) {
        if (masked) stream(g, 0, V, cp.tok_a, 0, pol_last, nop);
        stream(g, lo, hi, cp.tok_a, 1, sampled && has_child ? pol_normal : pol_first, nop);
        for (; sampled && has_child; ++ncmd) {
          if (!cwait_bounded(cmdbar, ncmd & 1u)) {
            atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
            CL_SITE(4);
            stop = true;
            break;
          }
          const int kind = *reinterpret_cast<volatile int32_t*>(&cmd->kind);
          const int keep = *reinterpret_cast<volatile int32_t*>(&cmd->keep);
          if (kind == 0) {
            ++ncmd;
            break;
          }
          stream(g, 0, V, cp.tok_r, 2, keep ? pol_normal : pol_first, nop);
        }
      }
      stop = __shfl_sync(~0u, stop ? 1 : 0, 0) != 0;
    }
    if (lane == 0 && stop) hand(Meta{-1, kWhole, 0, 0.f, 0.f, 0.f});
    __syncwarp();
    cluster_sync_end();
    return;
  }

  // ===================================== consumer warps
  const CSync csync;
  uint32_t seq = 0;  // ring stages consumed
  uint32_t xk = 0;   // exchanges done (the same count in every CTA of the cluster)
  bool timed_out = false;
  unsigned long long w_full = 0, w_xchg = 0, w_desc = 0;  // debug builds: time spent waiting
  (void)w_full;
  (void)w_xchg;
  (void)w_desc;
  auto wait_full = [&](uint32_t sq) {
    CL_T(tw);
    if (!cwait_bounded(&full[sq % static_cast<uint32_t>(kCRing)], (sq / static_cast<uint32_t>(kCRing)) & 1u)) {
      timed_out = true;
      CL_SITE(5);
    }
    CL_ACC(w_full, tw);
  };
  auto release = [&](uint32_t sq) {
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[sq % static_cast<uint32_t>(kCRing)]);
  };
  // Exchange: thread 0 pushes this CTA's share into slot `rank` of buffer xk & 1 in every CTA of
  // the cluster and arrives there; every consumer thread then waits until its own buffer holds
  // all C shares.  Buffers alternate, and a CTA pushes into a buffer again only after every CTA
  // has arrived for the exchange in between, which each does only after a consumer barrier that
  // follows its reads of the buffer.
  auto exchange = [&](const XPart& mine) -> const XPart* {
    const int buf = static_cast<int>(xk & 1u);
    XPart* slots = xpart + buf * kCMaxCluster;
    if (tid < C) {  // thread t pushes to CTA t
      const uint4* w = reinterpret_cast<const uint4*>(&mine);
      const uint32_t dst = map_rank(&slots[rank], static_cast<uint32_t>(tid));
      st_cluster_v4(dst, w[0]);
      st_cluster_v4(dst + 16u, w[1]);
      arrive_cluster(map_rank(&xbar[buf], static_cast<uint32_t>(tid)));
    }
    CL_T(tx);
    const bool xok = wait_cluster_bounded(&xbar[buf], (xk >> 1) & 1u);
    CL_ACC(w_xchg, tx);
    if (!xok) {
      timed_out = true;
      if (tid == 0) atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
      CL_SITE(6);
    }
    ++xk;
    return slots;
  };
  auto post = [&](int kind, int keep) {  // thread 0: the producer's next command
    cmd->kind = kind;
    cmd->keep = keep;
    mbar_arrive(cmdbar);
  };

  for (uint32_t k = 0;; ++k) {
    const int dd = static_cast<int>(k % kCDesc);
    CL_T(td);
    const bool dok = cwait_bounded(&dfull[dd], (k / kCDesc) & 1u);
    CL_ACC(w_desc, td);
    if (!dok) {
      if (tid == 0) atomicOr(&p.hdr->err, DCD_DEVERR_TIMEOUT);
      CL_SITE(7);
      break;
    }
    const int* dsc = desc + 8 * dd;
    const int gi = dsc[0];
    const int mode = dsc[1];
    const int flags = dsc[2];
    const float alpha = __int_as_float(dsc[3]);
    const float beta = __int_as_float(dsc[4]);
    const float T = __int_as_float(dsc[5]);
    const bool split = mode == kSplit;
    const bool halfrow = (mode & 15) == kPart;  // one of P parts of a row
    const int nparts_row = halfrow ? (mode >> 4) & 15 : 1, mypart = halfrow ? mode >> 8 : 0;
    csync();  // every consumer has read the descriptor
    if (tid == 0) mbar_arrive(&dempty[dd]);
    if (gi < 0) break;
    const int64_t g = gi;
    const int b = gi / N, n = gi % N;
    const bool masked = (flags & 4) != 0;
    const bool sampled = (flags & 1) != 0;
    const bool has_child = (flags & 2) != 0;
    const float k2 = kLog2e * (T > 0.f ? 1.f / T : 1.f);  // exp(x / T) = 2^(x * k2)
    const float c1k = (1.f + alpha) * k2, ak = alpha * k2;
    const float logb = masked ? logf(beta) : -INFINITY;
    const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
    const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;
    const float* q_row = sampled ? p.q + g * p.ldq : nullptr;
    // a row split over the cluster: this CTA's slice, statistics exchanged; a whole row: [0, V);
    // part q of P: whole stages [q spp, (q + 1) spp), combined through the workspace
    int64_t x_lo = split ? sl_lo : 0, x_hi = split ? sl_hi : V;
    if (halfrow) {
      const int spp = (static_cast<int>((V + cp.tok_a - 1) / cp.tok_a) + nparts_row - 1) / nparts_row;
      x_lo = static_cast<int64_t>(mypart) * spp * cp.tok_a;
      const int64_t e = static_cast<int64_t>(mypart + 1) * spp * cp.tok_a;
      x_hi = e < V ? e : V;
    }
    bool leader = !split || rank == 0;  // writes the row's outputs
    timed_out = false;
    CL_T(t_row0);
    unsigned long long t_dec = 0;
    int npass = 0;
    {
      // ---- warp 1 lists the children, checks the row and loads the values at the children's
      // tokens while the statistics pass streams
      if (warp == 1) {
        const int count = clist_children(p, b, n, kids, ktok);
        for (int kk = lane; kk < count; kk += 32) {
          const int t = ktok[kk];
          const bool ok = t >= 0 && t < V;
          czp[kk] = ok ? ld1(zp_row, t) : 0.f;
          czq[kk] = ok ? ld1(zq_row, t) : 0.f;
          cq[kk] = (ok && sampled) ? q_row[t] : 0.f;
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
          sh->m = count;
          sh->status = st;
        }
      }

      // ---- beta > 0: the expert max over the row, for P_beta = {x : z_p(x) - max z_p >= log beta}
      float Mp = 0.f;
      if (masked) {
        float lm = -INFINITY;
        for (int64_t x0 = x_lo; x0 < x_hi; x0 += cp.tok_a, ++seq) {
          const CStage<TIn> st = cstage<TIn>(ring, static_cast<int>(seq % static_cast<uint32_t>(kCRing)), cp.tok_a);
          const int clen = static_cast<int>((x_hi - x0) < cp.tok_a ? (x_hi - x0) : cp.tok_a);
          wait_full(seq);
          for (int i0 = tid * 8; i0 < clen; i0 += kCThreads * 8) {
            float zp[8];
            ld8(st.zp + i0, zp);
#pragma unroll
            for (int e = 0; e < 8; ++e)
              if (i0 + e < clen) lm = fmaxf(lm, zp[e]);
          }
          release(seq);
        }
        lm = block_max(lm, redf, csync);
        Mp = lm;
        if (split) {
          XPart mine{};
          mine.a = lm;
          mine.blk = INT_MAX;
          const XPart* all = exchange(mine);
          Mp = -INFINITY;
          for (int t = 0; t < C; ++t) Mp = fmaxf(Mp, all[t].a);
        }
      }

      // ---- statistics pass over the slice: per lane an online max of u on P_beta, the sum of
      // 2^(u - max) rescaled when the max grows, and the argmax; a sampled leaf also records the
      // mass of each warp chunk relative to a chunk reference
      const int tpw = cp.tok_a / kCWarps, wpb = kRaceBlock / tpw;
      // the running max starts finite (no score is that low), so that 2^(u - max) needs no test
      // for an empty max; it is -inf again below if no score was finite
      float lmax = -FLT_MAX, lsum = 0.f;
      int larg = INT_MAX;
      const bool rec_chunks = sampled && !has_child;  // a sampled leaf's race needs the chunk masses
      const float2 c1k2 = make_float2(c1k, c1k), nak2 = make_float2(-ak, -ak);
      int L = 0;  // stage of the slice
      for (int64_t x0 = x_lo; x0 < x_hi; x0 += cp.tok_a, ++seq, ++L) {
        const CStage<TIn> st = cstage<TIn>(ring, static_cast<int>(seq % static_cast<uint32_t>(kCRing)), cp.tok_a);
        const int clen = static_cast<int>((x_hi - x0) < cp.tok_a ? (x_hi - x0) : cp.tok_a);
        const int sb_end = (warp + 1) * tpw < clen ? (warp + 1) * tpw : clen;
        wait_full(seq);
        float2 acc2 = make_float2(0.f, 0.f);  // this stage's sum of 2^(u - lmax), in lane pairs
        // a stage-wide step: the max, the rescale when it grows (with the argmax), the sum
        auto step = [&](const float (&u)[8], int i0) {
          const float gm = max8(u);
          if (gm > lmax) {
            const float f = ex2(lmax - gm);  // 0 while lmax is the start value
            lsum *= f;
            acc2 = __fmul2_rn(acc2, make_float2(f, f));
            lmax = gm;
#pragma unroll
            for (int e = 7; e >= 0; --e)
              if (u[e] == gm) larg = static_cast<int>(x0) + i0 + e;
          }
          const float2 nm2 = make_float2(-lmax, -lmax);
          float2 e2[4];
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const float2 d2 = __fadd2_rn(make_float2(u[2 * kk], u[2 * kk + 1]), nm2);
            e2[kk] = make_float2(ex2(d2.x), ex2(d2.y));
          }
          acc2 = __fadd2_rn(acc2, __fadd2_rn(__fadd2_rn(e2[0], e2[1]), __fadd2_rn(e2[2], e2[3])));
        };
        int sb = warp * tpw;
        if (!masked) {
          for (; sb + kSub <= sb_end; sb += kSub) {  // whole sub-blocks (warp-uniform)
            const int i0 = sb + lane * 8;
            float2 zp2[4], zq2[4];
            ld8x2(st.zp + i0, zp2);
            ld8x2(st.zq + i0, zq2);
            float u[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float2 s2 = __ffma2_rn(zp2[k], c1k2, __fmul2_rn(zq2[k], nak2));
              u[2 * k] = s2.x;
              u[2 * k + 1] = s2.y;
            }
            step(u, i0);
          }
        }
        for (; sb < sb_end; sb += kSub) {  // the plausibility mask, or the stage's ragged end
          const int i0 = sb + lane * 8;
          float u[8];
          cscores8(st.zp, st.zq, i0, sb, clen, masked, c1k, ak, Mp, logb, u);
          step(u, i0);
        }
        const float bpart = acc2.x + acc2.y;
        lsum += bpart;
        if (rec_chunks) {
          const float ref = warp_max(lmax);
          const float ws = warp_sum(bpart * ex2(lmax - ref));
          if (lane == 0 && x0 + static_cast<int64_t>(warp) * tpw < x_hi) {
            const int ch = L * kCWarps + warp;  // (x0 - x_lo) / tpw + warp
            cref[ch] = ref > -FLT_MAX ? ref : -INFINITY;
            csum[ch] = ws;
          }
        }
        release(seq);
      }
      if (lmax == -FLT_MAX) lmax = -INFINITY;  // no finite score
      float M = lmax, S = lsum;
      int arg = larg;
      block_stats(M, S, arg, redf, redi, csync);  // its barriers also publish warp 1's child list
      const int m = sh->m;
      if (halfrow) {
        // a part of a (greedy) row: publish its statistics; the CTA that finishes the last part
        // combines them in part order and finishes the row
        if (tid == 0) {
          const int part = mypart;
          RowPart rp;
          rp.M = M;
          rp.S = S;
          rp.arg = arg;
          rp.key = -INFINITY;
          rp.blk = INT_MAX;
          rp.timed_out = timed_out ? 1 : 0;
          rp.pad[0] = rp.pad[1] = 0;
          p.parts[g * kMaxParts + part] = rp;
          const uint32_t t = atomic_add_acq_rel(&p.pdone[g], 1u);
          const bool last = t + 1u == static_cast<uint32_t>(nparts_row);
          sh->decision = last ? 1 : 0;
          if (last) {
            float cM = -INFINITY, cS = 0.f;
            int carg = INT_MAX, tmo = 0;
            for (int q = 0; q < nparts_row; ++q) {  // part order: the result does not depend on timing
              const RowPart o = q == part ? rp : p.parts[g * kMaxParts + q];
              stats_merge(cM, cS, carg, o.M, o.S, o.arg);
              tmo |= o.timed_out;
            }
            sh->c = cM;  // (scratch: the combined statistics)
            sh->D = cS;
            sh->term = carg;
            sh->degen = tmo;
          }
        }
        csync();
        if (sh->decision == 0) goto row_done;  // another part finishes the row
        M = sh->c;
        S = sh->D;
        arg = sh->term;
        timed_out = timed_out || sh->degen != 0;
      }

      // first level of a leaf's race over the slice's blocks: log2 of a block's mass is
      // log2(sum of its chunks' 2^ref-scaled sums) + max ref (the row max is a common shift)
      float bk = -INFINITY;
      int bb = INT_MAX;
      if (rec_chunks) {
        const int nch_sl = static_cast<int>((x_hi - x_lo + tpw - 1) / tpw);
        const int k_lo = static_cast<int>(x_lo / kRaceBlock);
        const int k_hi = static_cast<int>((x_hi + kRaceBlock - 1) / kRaceBlock);
        for (int kb = k_lo + tid; kb < k_hi; kb += kCThreads) {
          const int c0 = (kb - k_lo) * wpb;
          float ref = -INFINITY, sum = 0.f;
          for (int i = 0; i < wpb && c0 + i < nch_sl; ++i) ref = fmaxf(ref, cref[c0 + i]);
          if (ref > -INFINITY)
            for (int i = 0; i < wpb && c0 + i < nch_sl; ++i) {
              const float rr = cref[c0 + i];
              if (rr > -INFINITY) sum += csum[c0 + i] * ex2(rr - ref);
            }
          if (ref > -INFINITY && sum > 0.f) {
            const float key = cblock_key(p, g, kb, lg2(sum) + ref);
            if (key > bk) {
              bk = key;
              bb = kb;
            }
          }
        }
        block_argmax(bk, bb, redf, redi, csync);
      }

      // ---- exchange of the slices' statistics; every CTA combines them in rank order
      if (split) {
        XPart mine{};
        mine.a = M;
        mine.b = S;
        mine.i = arg;
        mine.key = bk;
        mine.blk = bb;
        mine.status = timed_out ? DCD_DEVERR_TIMEOUT : 0u;
        const XPart* all = exchange(mine);
        M = -INFINITY;
        S = 0.f;
        arg = INT_MAX;
        float K = -INFINITY;
        int kb = INT_MAX;
        uint32_t xs = 0u;
        for (int t = 0; t < C; ++t) {
          const XPart pt = all[t];
          stats_merge(M, S, arg, pt.a, pt.b, pt.i);
          argmax_merge(K, kb, pt.key, pt.blk);
          xs |= pt.status;
        }
        bk = K;
        bb = kb;
        timed_out = timed_out || xs != 0u;
      }
      {
        CL_T(t_now);
        t_dec = t_now;
      }
      uint32_t status = sh->status | (timed_out ? DCD_DEVERR_TIMEOUT : 0u);
      if (!(M > -INFINITY && M < INFINITY) || !(S > 0.f && S < INFINITY)) status |= DCD_DEVERR_NONFINITE;
      if (kDistinct && sampled && m > kMaxRemoved) status |= DCD_DEVERR_UNSUPPORTED;
      const float logS = logf(S);
      const float invS = 1.f / S;

      // ---- outputs of the Eq. 1 target (the cluster's first CTA for a split row)
      if (leader) {
        if (tid == 0) {
          if (p.cd_argmax) p.cd_argmax[g] = arg;
          if (p.cd_lse) p.cd_lse[g] = M * kLn2c + logS;
          if (n == 0 && p.cd_logprob) p.cd_logprob[g] = 0.f;
        }
        if (p.cd_logprob)
          for (int kk = tid; kk < m; kk += kCThreads) {
            const bool in = !masked || (czp[kk] - Mp >= logb);
            p.cd_logprob[static_cast<int64_t>(b) * N + kids[kk]] =
                in ? (fmaf(c1k, czp[kk], -ak * czq[kk]) - M) * kLn2c - logS : -INFINITY;
          }
      }
      auto write_record = [&](int acc, int term, uint32_t st) {  // one thread
        RowRecord rr;
        rr.acc_child = acc;
        rr.term_token = acc < 0 ? term : -1;
        rr.status = st;
        rr.reserved = 0;
        p.rec[g] = rr;
      };
      auto owns = [&](int kblk) -> bool {  // this CTA holds race block kblk (or none was drawn)
        if (!split) return true;
        if (kblk == INT_MAX) return rank == 0;
        return rank ==
               static_cast<uint32_t>(static_cast<int64_t>(kblk) * kRaceBlock /
                                     (static_cast<int64_t>(cp.spc) * cp.tok_a));
      };

      if (!sampled) {
        // ---- greedy rule: the first child whose token is the argmax, else the argmax is the bonus
        if (leader && tid == 0) {
          int acc = -1;
          for (int kk = 0; kk < m; ++kk)
            if (ktok[kk] == arg) {
              acc = kids[kk];
              break;
            }
          write_record(acc, acc < 0 ? arg : -1, status);
        }
      } else if (m == 0) {
        // ---- sampled leaf: the terminal token from pi_CD,T by the two-level race
        if (owns(bb)) {
          const int term = ctoken_race(
              p, g, bb,
              [&](int64_t x) -> float {
                const float z = ld1(zp_row, x);
                const bool in = !masked || (z - Mp >= logb);
                return in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, x)) - M) : 0.f;
              },
              redf, redi);
          if (tid == 0) write_record(-1, term, status);
        }
      } else {
        // ---- sampled rule, first sibling: accept child 0 iff u <= pi_CD,T(t) / q(t) (every CTA of
        // the cluster takes the same decision from the same values)
        const uint32_t fatal = DCD_DEVERR_BAD_PARENT | DCD_DEVERR_BAD_TOKEN | DCD_DEVERR_BAD_PARAM |
                               DCD_DEVERR_NONFINITE | DCD_DEVERR_UNSUPPORTED;
        if (tid == 0) {
          const bool in = !masked || (czp[0] - Mp >= logb);
          const float rt = in ? ex2(fmaf(c1k, czp[0], -ak * czq[0]) - M) * invS : 0.f;
          const float qt = cq[0];
          const float ratio = qt > 0.f ? rt / qt : (rt > 0.f ? INFINITY : 0.f);
          const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * N + kids[0]);
          const float u = u01(philox_block(p.seed, p.offset, G, 0u).x);
          const bool accept = u <= ratio || (status & fatal) != 0u;
          sh->decision = accept ? 1 : 0;
          if (accept && leader) write_record(u <= ratio ? kids[0] : -1, -1, status);
          if (accept) {
            post(0, 0);
          } else {
            post(1, m > 1 ? 1 : 0);  // the first residual pass
            if (leader) atomicAdd(&p.hdr->nslots, 1u);  // rows that took residual passes (a count only)
          }
          sh->J = 1;
          sh->cJ = 1.f;  // c_1 = c_0 + D_0 with r_0 = pi (c_0 = 0, D_0 = 1)
          sh->c = 0.f;
          sh->D = 1.f;
          sh->degen = 0;
          sh->Z = 1.f;  // distinct siblings: nothing removed yet
          sh->nrem = 0;
        }
        csync();
        if (sh->decision != 1) {
          // ---- the residual chain
          const int tpw_r = cp.tok_r / kCWarps, wpb_r = kRaceBlock / tpw_r;
          for (;;) {
            const int J = sh->J;
            const float cJ = sh->cJ;
            const bool race = J == m;  // the pass after the last sibling also ranks race blocks
            // distinct siblings: the first pass also sums q, whose actual mass (the drafter's q
            // may be truncated or rounded away from 1) normalises the proposal once a token is
            // removed
            const bool sum_q = kDistinct && J == 1;
            ++npass;
            float part = 0.f, ql = 0.f;
            int L = 0;
            // r(x) S = max(2^(u - M) - c_J S q(x), 0): the factor 1 / S is applied to the sums
            const float2 nM2 = make_float2(-M, -M), ncs2 = make_float2(-cJ * S, -cJ * S);
            const float2 c1k2 = make_float2(c1k, c1k), nak2 = make_float2(-ak, -ak);
            for (int64_t x0 = x_lo; x0 < x_hi; x0 += cp.tok_r, ++seq, ++L) {
              const CStage<TIn> st =
                  cstage<TIn>(ring, static_cast<int>(seq % static_cast<uint32_t>(kCRing)), cp.tok_r);
              const int clen = static_cast<int>((x_hi - x0) < cp.tok_r ? (x_hi - x0) : cp.tok_r);
              const int sb_end = (warp + 1) * tpw_r < clen ? (warp + 1) * tpw_r : clen;
              wait_full(seq);
              float2 sp2 = make_float2(0.f, 0.f), ql2 = make_float2(0.f, 0.f);
              auto rstep = [&](const float (&u)[8], const float2 (&q2)[4]) {
                float2 t2[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const float2 d2 = __fadd2_rn(make_float2(u[2 * k], u[2 * k + 1]), nM2);
                  const float2 r2 = __ffma2_rn(q2[k], ncs2, make_float2(ex2(d2.x), ex2(d2.y)));
                  t2[k] = make_float2(fmaxf(r2.x, 0.f), fmaxf(r2.y, 0.f));
                }
                sp2 = __fadd2_rn(sp2, __fadd2_rn(__fadd2_rn(t2[0], t2[1]), __fadd2_rn(t2[2], t2[3])));
                if (sum_q) ql2 = __fadd2_rn(ql2, __fadd2_rn(__fadd2_rn(q2[0], q2[1]), __fadd2_rn(q2[2], q2[3])));
              };
              int sb = warp * tpw_r;
              if (!masked) {
                for (; sb + kSub <= sb_end; sb += kSub) {  // whole sub-blocks (warp-uniform)
                  const int i0 = sb + lane * 8;
                  float2 zp2[4], zq2[4];
                  ld8x2(st.zp + i0, zp2);
                  ld8x2(st.zq + i0, zq2);
                  float u[8];
#pragma unroll
                  for (int k = 0; k < 4; ++k) {
                    const float2 s2 = __ffma2_rn(zp2[k], c1k2, __fmul2_rn(zq2[k], nak2));
                    u[2 * k] = s2.x;
                    u[2 * k + 1] = s2.y;
                  }
                  float2 q2[4];
                  ld8x2(st.q + i0, q2);
                  rstep(u, q2);
                }
              }
              for (; sb < sb_end; sb += kSub) {  // the plausibility mask, or the stage's ragged end
                const int i0 = sb + lane * 8;
                float u[8], qv[8];
                cscores8(st.zp, st.zq, i0, sb, clen, masked, c1k, ak, Mp, logb, u);  // -inf past the end
                ld8(st.q + i0, qv);
                float2 q2[4];
#pragma unroll
                for (int k = 0; k < 4; ++k)  // q past the end is whatever the stage held before
                  q2[k] = make_float2(i0 + 2 * k < clen ? qv[2 * k] : 0.f, i0 + 2 * k + 1 < clen ? qv[2 * k + 1] : 0.f);
                rstep(u, q2);
              }
              const float sp = (sp2.x + sp2.y) * invS;
              ql += ql2.x + ql2.y;
              part += sp;
              if (race) {
                const float ws = warp_sum(sp);
                if (lane == 0) csum[L * kCWarps + warp] = ws;
              }
              release(seq);
            }
            const float zsum = block_sum(part, redf, csync);  // its barriers also publish csum
            const float qsum = sum_q ? block_sum(ql, redf, csync) : 0.f;
            float rk = -INFINITY;
            int rb = INT_MAX;
            if (race) {
              const int nch_sl = static_cast<int>((x_hi - x_lo + tpw_r - 1) / tpw_r);
              const int k_lo = static_cast<int>(x_lo / kRaceBlock);
              const int k_hi = static_cast<int>((x_hi + kRaceBlock - 1) / kRaceBlock);
              for (int kb = k_lo + tid; kb < k_hi; kb += kCThreads) {
                float mass = 0.f;
                for (int i = 0; i < wpb_r && (kb - k_lo) * wpb_r + i < nch_sl; ++i)
                  mass += csum[(kb - k_lo) * wpb_r + i];
                if (kDistinct) {
                  // removed siblings' tokens in this block carry their frozen mass, not the
                  // streamed one
                  const int nrem = sh->nrem;
                  for (int i = 0; i < nrem; ++i)
                    if (sh->rtok[i] / kRaceBlock == kb)
                      mass += sh->rfz[i] - fmaxf(sh->rpit[i] - cJ * sh->rq[i], 0.f);
                }
                if (mass > 0.f) {
                  const float key = cblock_key(p, g, kb, lg2(mass));
                  if (key > rk) {
                    rk = key;
                    rb = kb;
                  }
                }
              }
              block_argmax(rk, rb, redf, redi, csync);
            }
            const XPart* all = nullptr;
            if (split) {
              XPart mine{};
              mine.a = zsum;
              mine.b = qsum;
              mine.key = rk;
              mine.blk = rb;
              mine.status = timed_out ? DCD_DEVERR_TIMEOUT : 0u;
              all = exchange(mine);
            }
            if (tid == 0) {
              float DJ = zsum, K = rk, QS = qsum;
              int kstar = rb;
              uint32_t st2 = status | (timed_out ? DCD_DEVERR_TIMEOUT : 0u);
              if (split) {
                DJ = 0.f;
                QS = 0.f;
                K = -INFINITY;
                kstar = INT_MAX;
                for (int t = 0; t < C; ++t) {  // a fixed order
                  DJ += all[t].a;
                  QS += all[t].b;
                  argmax_merge(K, kstar, all[t].key, all[t].blk);
                  st2 |= all[t].status;
                }
              }
              float c = sh->c, Dn = sh->D;
              bool degen = sh->degen != 0;
              int acc = -1;
              bool queued = false, ranked = J == m;
              if constexpr (kDistinct) {
                // Siblings without replacement.  With the tokens removed so far frozen at their
                // mass fz, the residual after this pass is max(0, pi - c_J q) elsewhere: its
                // mass is the streamed sum corrected at the removed tokens.  A pass without mass
                // keeps the residual it started from.  Then sibling J's token is removed from
                // the proposal (frozen at the current residual) and the next siblings are tested
                // against r with the proposal q / Z without the removed tokens.
                int nrem = sh->nrem;
                float Z = J == 1 ? QS : sh->Z;  // q's own mass before the first removal
                auto value_at = [&](int j, float& pit, float& qt) {  // at sibling j's (valid) token
                  const bool in = !masked || (czp[j] - Mp >= logb);
                  pit = in ? ex2(fmaf(c1k, czp[j], -ak * czq[j]) - M) * invS : 0.f;
                  qt = cq[j];
                };
                auto removed_index = [&](int t) {
                  for (int i = 0; i < nrem; ++i)
                    if (sh->rtok[i] == t) return i;
                  return -1;
                };
                float EJ = DJ;
                for (int i = 0; i < nrem; ++i) EJ += sh->rfz[i] - fmaxf(sh->rpit[i] - cJ * sh->rq[i], 0.f);
                if (EJ > 0.f) {
                  c = cJ;
                  Dn = EJ;
                } else {
                  ranked = false;  // the pass ranked blocks of a residual that is not used
                }
                auto remove = [&](int j) {  // sibling j's token
                  const int t = ktok[j];
                  if (t < 0 || t >= V || removed_index(t) >= 0) return;
                  if (nrem >= kMaxRemoved) {
                    st2 |= DCD_DEVERR_UNSUPPORTED;
                    return;
                  }
                  float pit, qt;
                  value_at(j, pit, qt);
                  sh->rtok[nrem] = t;
                  sh->rfz[nrem] = fmaxf(pit - c * qt, 0.f);
                  sh->rpit[nrem] = pit;
                  sh->rq[nrem] = qt;
                  ++nrem;
                  Z -= qt;
                };
                remove(J - 1);
                for (int j = J; j < m; ++j) {
                  const int t = ktok[j];
                  float ratio = 0.f;
                  if (t >= 0 && t < V) {
                    const int ri = removed_index(t);
                    if (ri >= 0) {
                      ratio = sh->rfz[ri] > 0.f ? INFINITY : 0.f;  // its proposal is 0
                    } else {
                      float pit, qt;
                      value_at(j, pit, qt);
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
                    sh->J = j + 1;
                    sh->cJ = c + Dn / Z;  // the next residual: max(0, r - q / Z) off the removed tokens
                    queued = true;
                    break;
                  }
                  // every token of q is removed: the proposal is 0 and the residual stays
                  ranked = false;
                  remove(j);
                }
                sh->nrem = nrem;
                sh->Z = Z;
              } else {
              if (DJ > 0.f) {
                c = cJ;
                Dn = DJ;
              } else {
                degen = true;  // r_{J-1} == q in exact arithmetic: r_J is taken as q from here on
              }
              // test the remaining siblings; after a pass without residual mass no pass is needed
              for (int j = J; j < m; ++j) {
                // the values at the children's tokens were loaded into shared memory with the row
                const int t = ktok[j];
                const bool ok = t >= 0 && t < V;
                const float z = czp[j];
                const float qt = cq[j];
                const bool in = ok && (!masked || (z - Mp >= logb));
                const float pit = in ? ex2(fmaf(c1k, z, -ak * czq[j]) - M) * invS : 0.f;
                const float rt = degen ? qt : fmaxf(pit - c * qt, 0.f) / Dn;
                const float ratio = qt > 0.f ? rt / qt : (rt > 0.f ? INFINITY : 0.f);
                const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * N + kids[j]);
                if (u01(philox_block(p.seed, p.offset, G, 0u).x) <= ratio) {
                  acc = kids[j];
                  break;
                }
                if (!degen) {
                  sh->J = j + 1;
                  sh->cJ = c + Dn;  // c_{J+1} = c_J + D_J
                  queued = true;
                  break;
                }
              }
              }
              sh->c = c;
              sh->D = Dn;
              sh->degen = degen ? 1 : 0;
              sh->status = st2;
              sh->term = (ranked && !degen) ? kstar : INT_MAX - 1;  // the winning block when this pass ranked r_m
              sh->decision = queued ? 2 : (acc >= 0 ? 1 : 0);
              if (queued) {
                post(1, sh->J < m ? 1 : 0);
              } else {
                post(0, 0);
                if (acc >= 0 && leader) write_record(acc, -1, st2);
              }
            }
            csync();
            const int dec = sh->decision;
            if (dec == 2) continue;
            if (dec == 1) break;
            // ---- every sibling rejected: the terminal token from r_m, or from q after a pass
            // without mass
            const bool degen = sh->degen != 0;
            const float c = sh->c, Dn = sh->D;
            const uint32_t st2 = sh->status;
            const int nrem = kDistinct ? sh->nrem : 0;
            int kstar = sh->term;
            auto rho_at = [&](int64_t x) -> float {  // the final residual's unnormalised mass
              if (kDistinct)
                for (int i = 0; i < nrem; ++i)
                  if (sh->rtok[i] == x) return sh->rfz[i];
              const float z = ld1(zp_row, x);
              const bool in = !masked || (z - Mp >= logb);
              const float pit = in ? ex2(fmaf(c1k, z, -ak * ld1(zq_row, x)) - M) * invS : 0.f;
              return fmaxf(pit - c * q_row[x], 0.f);
            };
            if (kstar == INT_MAX - 1) {
              // block masses over the slices of q (a residual without mass), or (distinct
              // siblings) of the final residual when the last pass did not rank it (rare: the
              // last pass found no mass, or q was used up)
              float qk = -INFINITY;
              int qb = INT_MAX;
              const int k_lo = static_cast<int>(x_lo / kRaceBlock);
              const int k_hi = static_cast<int>((x_hi + kRaceBlock - 1) / kRaceBlock);
              for (int kb = k_lo + warp; kb < k_hi; kb += kCWarps) {
                float s2 = 0.f;
                for (int64_t x = static_cast<int64_t>(kb) * kRaceBlock + lane; x < x_hi && x < (kb + 1) * kRaceBlock;
                     x += 32)
                  s2 += kDistinct ? rho_at(x) : q_row[x];
                const float mass = warp_sum(s2);
                if (lane == 0 && mass > 0.f) {
                  const float key = cblock_key(p, g, kb, lg2(mass));
                  if (key > qk) {
                    qk = key;
                    qb = kb;
                  }
                }
              }
              block_argmax(qk, qb, redf, redi, csync);
              kstar = qb;
              if (split) {
                XPart mine2{};
                mine2.key = qk;
                mine2.blk = qb;
                const XPart* all2 = exchange(mine2);
                float K = -INFINITY;
                kstar = INT_MAX;
                for (int t = 0; t < C; ++t) argmax_merge(K, kstar, all2[t].key, all2[t].blk);
              }
            }
            if (owns(kstar)) {
              const int term = ctoken_race(
                  p, g, kstar,
                  [&](int64_t x) -> float {
                    if (degen && !kDistinct) return q_row[x];
                    return rho_at(x) / Dn;
                  },
                  redf, redi);
              if (tid == 0) write_record(-1, term, st2);
            }
            break;
          }
        }
      }
    }
  row_done:
    csync();  // the row's shared state (children, chunk masses) is rewritten by the next row
    if (tid == 0) CL_REC(gi, mode, t_row0, t_dec, npass, sh->m);
    w_full = w_xchg = w_desc = 0;
    (void)t_dec;
    (void)npass;
  }
  cluster_sync_end();
}

struct CDeviceInfo {
  int sms = 0;
  cudaError_t err = cudaSuccess;
};

template <typename TIn, bool kDistinct>
cudaError_t prepare_cluster_kernel(int* sms) {
  static std::once_flag once[64];
  static CDeviceInfo info[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::call_once(once[dev], [&] {
    CDeviceInfo d;
    d.err = cudaFuncSetAttribute(cluster_rows_kernel<TIn, kDistinct>, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    if (d.err == cudaSuccess) d.err = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev);
    info[dev] = d;
  });
  *sms = info[dev].sms;
  return info[dev].err;
}

int ctok_split(int cap) {
  for (int tpw = kRaceBlock; tpw >= kSub; tpw /= 2)
    if (kCWarps * tpw <= cap) return kCWarps * tpw;
  return 0;
}

struct CLayout {
  int meta_offset, chunk_offset, seq_offset, stage_offset;
  size_t total;
};

CLayout clayout(int N, int nchunk, int nst, int nseq) {
  CLayout l;
  const size_t fixed = 8 * (2 * kCMaxStages + 3 + 2 * kMail + 2 * kCDesc + 1) + 96 * 4 +
                       sizeof(XPart) * 2 * kCMaxCluster + sizeof(Cmd) + 4 * (kMail + 8 * kCDesc);
  l.meta_offset = static_cast<int>((fixed + 15) & ~static_cast<size_t>(15));
  const size_t meta_end = static_cast<size_t>(l.meta_offset) + sizeof(CShared) + static_cast<size_t>(N) * 4 * 5;
  l.chunk_offset = static_cast<int>((meta_end + 15) & ~static_cast<size_t>(15));
  const size_t chunk_end = static_cast<size_t>(l.chunk_offset) + static_cast<size_t>(nchunk) * 4 * 2;
  l.seq_offset = nseq > 0 ? static_cast<int>((chunk_end + 15) & ~static_cast<size_t>(15)) : 0;
  const size_t seq_end = nseq > 0 ? static_cast<size_t>(l.seq_offset) + static_cast<size_t>(nseq) * 4 : chunk_end;
  l.stage_offset = static_cast<int>((seq_end + 127) & ~static_cast<size_t>(127));
  l.total = static_cast<size_t>(l.stage_offset) + static_cast<size_t>(nst) * kCStage;
  return l;
}

// The cluster geometry of a call: CTAs per cluster, tokens per stage, slices, shared memory.
bool cluster_geometry(const ScoreArgs& a, int sms, CParams* cp, size_t* smem) {
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  const int tok_a = ctok_split(kCStage / (2 * es));
  const int tok_r = ctok_split(kCStage / (2 * es + 4));
  if (tok_a == 0 || tok_r == 0 || tok_a % tok_r != 0 || tok_a % kRaceBlock != 0) return false;
  if (kCRing > kCMaxStages || kCRing < 2) return false;
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  const int nch_a = static_cast<int>((a.V + tok_a - 1) / tok_a);
  const int64_t slots = static_cast<int64_t>(sms) * kCMinCtas;
  // CTAs per cluster: a row of a sampled sequence is split over C CTAs, so its residual chain
  // runs on C of them.  A smaller sampled call gets larger clusters (measured on 152 SMs: 2 at
  // 1920 rows, 4 at 480, 8 at 60); a greedy call takes every row whole (C = 1).
  const bool sampled_call = a.temp != nullptr && a.q != nullptr;
  const int want = kCFixed > 0 ? kCFixed : (!sampled_call ? 1 : (R >= 2 * slots ? 2 : (R >= slots / 2 ? 4 : 8)));
  int C = 1;
  while (C < want && C < kCMax && C * 2 <= nch_a) C *= 2;
  const int spc = (nch_a + C - 1) / C;
  // chunk slots: statistics and residual-pass chunks of a whole row (a slice needs fewer)
  const int64_t ch_a = (a.V + tok_a / kCWarps - 1) / (tok_a / kCWarps);
  const int64_t ch_r = (a.V + tok_r - 1) / tok_r * kCWarps;
  const int64_t nchunk = ch_a > ch_r ? ch_a : ch_r;
  if (nchunk > (1 << 20)) return false;
  const int nseq = a.B <= kSeqListMax ? a.B : 0;
  const CLayout l = clayout(a.N, static_cast<int>(nchunk), kCRing, nseq);
  if (l.total > 227 * 1024) return false;
  cp->a = a;
  cp->C = C;
  cp->tok_a = tok_a;
  cp->tok_r = tok_r;
  cp->spc = spc;
  cp->nchunk = static_cast<int32_t>(nchunk);
  cp->meta_offset = l.meta_offset;
  cp->chunk_offset = l.chunk_offset;
  cp->stage_offset = l.stage_offset;
  cp->seq_offset = l.seq_offset;
  *smem = l.total;
  return true;
}

// Resident clusters of the kernel for a launch shape, cached (the occupancy query is not free).
cudaError_t resident_clusters(const void* fn, const cudaLaunchConfig_t& cfg, int variant, int C, size_t smem, int* ncl) {
  struct Entry {
    int dev, variant, C;  // variant: element type and sibling rule
    size_t smem;
    int ncl;
  };
  static std::mutex mu;
  static Entry cache[64];
  static int n = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  {
    std::lock_guard<std::mutex> lk(mu);
    for (int i = 0; i < n; ++i)
      if (cache[i].dev == dev && cache[i].variant == variant && cache[i].C == C && cache[i].smem == smem) {
        *ncl = cache[i].ncl;
        return cudaSuccess;
      }
  }
  e = cudaOccupancyMaxActiveClusters(ncl, fn, &cfg);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  if (n < 64) cache[n++] = Entry{dev, variant, C, smem, *ncl};
  return cudaSuccess;
}

}  // namespace

bool cluster_rows_ok(const ScoreArgs& a) {
  if (a.force_stages || a.force_plain || a.poll_cycles) return false;
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  auto al16 = [](const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
  if (!al16(a.zp) || !al16(a.zq) || (a.ld * es) % 16 != 0) return false;
  if (a.q && (!al16(a.q) || (a.ldq * 4) % 16 != 0)) return false;
  CParams cp;
  size_t smem = 0;
  return cluster_geometry(a, 152, &cp, &smem);
}

cudaError_t launch_cluster_rows(const ScoreArgs& a, cudaStream_t stream) {
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  if (R == 0) return cudaSuccess;
  int sms = 0;
  const bool bf = a.dtype == DCD_BF16;
  cudaError_t e = bf ? (a.distinct ? prepare_cluster_kernel<__nv_bfloat16, true>(&sms)
                                   : prepare_cluster_kernel<__nv_bfloat16, false>(&sms))
                     : (a.distinct ? prepare_cluster_kernel<float, true>(&sms) : prepare_cluster_kernel<float, false>(&sms));
  if (e != cudaSuccess) return e;
  CParams cp;
  size_t smem = 0;
  if (!cluster_geometry(a, sms, &cp, &smem)) return cudaErrorInvalidConfiguration;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kCCtaThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(cp.C);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const void* fn = bf ? (a.distinct ? reinterpret_cast<const void*>(cluster_rows_kernel<__nv_bfloat16, true>)
                                    : reinterpret_cast<const void*>(cluster_rows_kernel<__nv_bfloat16, false>))
                      : (a.distinct ? reinterpret_cast<const void*>(cluster_rows_kernel<float, true>)
                                    : reinterpret_cast<const void*>(cluster_rows_kernel<float, false>));
  // a persistent grid: as many clusters as can be resident at once (each claims rows until none
  // is left; no CTA waits for another cluster, so fewer resident clusters only take longer); the
  // count is queried once per device, kernel variant, cluster size and shared-memory size
  cfg.gridDim = dim3(static_cast<unsigned>(cp.C));
  int ncl = 0;
  e = resident_clusters(fn, cfg, a.dtype * 2 + (a.distinct ? 1 : 0), cp.C, smem, &ncl);
  if (e != cudaSuccess) return e;
  if (ncl < 1) return cudaErrorInvalidConfiguration;
  if (ncl > R) ncl = static_cast<int>(R);
  cfg.gridDim = dim3(static_cast<unsigned>(ncl * cp.C));
  // the error word, the row counters and the half-row tickets start every call at zero
  e = cudaMemsetAsync(a.hdr, 0, kWorkspaceHeader + part_counter_bytes(static_cast<size_t>(R)), stream);
  if (e != cudaSuccess) return e;
  if (bf)
    return a.distinct ? cudaLaunchKernelEx(&cfg, cluster_rows_kernel<__nv_bfloat16, true>, cp)
                      : cudaLaunchKernelEx(&cfg, cluster_rows_kernel<__nv_bfloat16, false>, cp);
  return a.distinct ? cudaLaunchKernelEx(&cfg, cluster_rows_kernel<float, true>, cp)
                    : cudaLaunchKernelEx(&cfg, cluster_rows_kernel<float, false>, cp);
}

}  // namespace dcd
