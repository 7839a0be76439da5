// dcd_fused.cu -- the greedy CD verification step fused with the two LM heads: the logits
// z_p = h_exp W_exp^T and z_q = h_ama W_ama^T are never written to memory.
//
// fused_lmhead_kernel: a persistent grid, one CTA per SM.  An output tile is 128 rows x 256
// vocabulary tokens; its two accumulators, z_p and z_q, live in tensor memory (2 x 256 fp32
// columns x 128 lanes: the whole of it).  Per CTA:
//   warp 0  -- TMA producer: for every K block of 64 it loads the 128 x 64 bf16 tile of h and the
//              256 x 64 bf16 tile of W (128-byte swizzle) into a 4-stage shared-memory ring,
//              first the amateur's K blocks, then the expert's;
//   warp 1  -- allocates tensor memory, and its lane 0 issues tcgen05.mma (M = 128, N = 256,
//              K = 16; bf16 in, fp32 accumulate) into z_q then z_p, committing each stage back to
//              the producer and each finished tile to the epilogue;
//   warps 2-5 -- epilogue: each thread owns one row of the tile (one TMEM lane).  Phase 1 reads
//              both accumulators 64 columns at a time, forms the scaled CD score u = log2(e)
//              ((1 + alpha) z_p - alpha z_q) (Eq. 1 at T = 1; the log-softmax shifts cancel) on
//              P_beta, keeps the score at each child token of the tile, and stores u over z_p;
//              the z_q columns then go back to the MMA warp, which starts the next tile's amateur
//              blocks.  Phase 2 reduces u to the tile's max, sum of 2^(u - max) and argmax while
//              those MMAs run, then hands back the z_p columns.  Tiles are visited in groups of
//              row tiles (about 40 MB of h each), vocabulary-block major within a group, so the
//              group's row tiles read each block of W while it is in L2, and the group's h (read
//              once per vocabulary block) stays in L2 with an evict-last policy.
//   With a plausibility mask (beta > 0, Sec. 2.1) the kernel runs twice: a first sweep over the
//   expert's K blocks only keeps each tile's max of z_p, fused_rowmax_kernel reduces them per
//   row, and the full sweep then scores only tokens with z_p - max z_p >= log beta.
// fused_children_kernel: per row, the children of its node (ascending id, at most 8) and the
//   row's input checks.
// fused_combine_kernel: one warp per row merges the tiles' statistics in order, writes
//   cd_argmax / cd_lse / cd_logprob, applies the greedy rule and leaves the row record for the
//   tree walk.

#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <mutex>

#include "dcd.h"
#include "dcd_device.cuh"
#include "dcd_fused.h"
#include "dcd_internal.h"
#include "dcd_tc.cuh"

namespace dcd {
namespace {

using namespace dev;

constexpr int kBM = 128;  // rows per tile (TMEM lanes)
constexpr int kBN = 256;  // vocabulary tokens per tile (TMEM columns per accumulator)
constexpr int kBK = 64;   // K per stage: one 128-byte swizzle row of bf16
constexpr int kGStages = 4;
constexpr int kABytes = kBM * kBK * 2;
constexpr int kBBytes = kBN * kBK * 2;
constexpr int kGStageBytes = kABytes + kBBytes;
constexpr int kGemmThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr int kMaxKids = 8;
constexpr size_t kGemmSmem = 1024 + static_cast<size_t>(kGStages) * kGStageBytes + 256;  // + barriers, flags
constexpr float kLn2f = 0.69314718055994531f;
constexpr int64_t kGroupHBytes = 40ll << 20;  // hidden-state bytes a group of row tiles keeps in L2

struct FusedParams {
  CUtensorMap tm_hp, tm_wp, tm_hq, tm_wq;
  int32_t R, V, N, nkp, nkq, nmt, nvt, ntiles;
  int32_t group;           // row tiles per group of the tile order
  int32_t sweep;           // 0: both models, the tile statistics of u; 1: the expert only, tile max of z_p
  const float* alpha;
  const float* beta;       // [B] or null (no plausibility mask)
  const float* zmax;       // [R] row max of z_p (sweep 0 with beta)
  const int32_t* kid_tok;  // [R][kMaxKids], -1 past the last child
  float* kid_u;            // [R][kMaxKids] scaled score at each child's token
  float4* part;            // [R][nvt] tile statistics {max u, sum 2^(u - max), argmax, -}
  uint32_t* err;
};

// Tile t -> (row tile i, vocabulary tile j).  Row tiles are visited in groups of `group`:
// within a group vocabulary-block major, so the group's row tiles read each block of W while it
// is in L2, and only the group's hidden states need to stay in L2 (W is read once per group).
__device__ __forceinline__ void tile_coords(int tile, int nmt, int nvt, int group, int& i, int& j) {
  const int G = (group > 0 && group < nmt) ? group : nmt;
  const int full = nmt / G;  // groups of G row tiles; the rest form a last, smaller group
  const int per = G * nvt;
  if (tile < full * per) {
    const int g = tile / per, r = tile - g * per;
    j = r / G;
    i = g * G + (r - j * G);
  } else {
    const int r = tile - full * per, gl = nmt - full * G;
    j = r / gl;
    i = full * G + (r - j * gl);
  }
}

// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kGemmThreads, 1) fused_lmhead_kernel(const __grid_constant__ FusedParams P) {
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                         ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kGStages * kGStageBytes);
  uint64_t* empty = full + kGStages;
  uint64_t* tfull = empty + kGStages;  // accumulators of a tile complete
  uint64_t* qfree = tfull + 1;         // the z_q columns read by the epilogue (u is in the z_p columns)
  uint64_t* pfree = qfree + 1;         // the z_p columns (holding u) read by the epilogue
  uint64_t* drained = pfree + 1;       // every MMA issued has completed (before tensor memory is freed)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drained + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = P.sweep == 1 ? P.nkp : P.nkp + P.nkq;  // the max sweep runs the expert's K blocks only
  const int qblocks = P.sweep == 1 ? 0 : P.nkq;          // K blocks of the amateur, issued first
  // A bounded wait that gives up records the error and makes every role of the CTA leave its
  // loop, so a failure costs one wait limit, not one per remaining stage.
  auto wait_or_abort = [&](uint64_t* bar, uint32_t parity) -> bool {
    if (mbar_wait_bounded(bar, parity)) return true;
    atomicOr(P.err, DCD_DEVERR_TIMEOUT);
    *abort_flag = 1;
    return false;
  };

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(tfull, 1);
    mbar_init(qfree, 4);
    mbar_init(pfree, 4);
    mbar_init(drained, 1);
    fence_mbar_init();
    tc::prefetch_tensormap(&P.tm_hp);
    tc::prefetch_tensormap(&P.tm_wp);
    tc::prefetch_tensormap(&P.tm_hq);
    tc::prefetch_tensormap(&P.tm_wq);
  }
  if (warp == 1) tc::tmem_alloc(tmem_slot, kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer
    if (lane == 0) {
      const uint64_t pol_h = l2_policy_evict_last();  // h is re-read for every vocabulary block
      uint32_t it = 0;
      for (int tile = blockIdx.x; tile < P.ntiles && !*abort_flag; tile += gridDim.x) {
        int i, j;
        tile_coords(tile, P.nmt, P.nvt, P.group, i, j);
        for (int kb = 0; kb < nk; ++kb) {
          const int s = static_cast<int>(it % kGStages);
          if (!wait_or_abort(&empty[s], ((it / kGStages) & 1u) ^ 1u)) break;
          ++it;
          unsigned char* a = smem + s * kGStageBytes;
          unsigned char* b = a + kABytes;
          mbar_arrive_expect_tx(&full[s], kGStageBytes);
          if (kb < qblocks) {  // the amateur's K blocks first
            tc::tma_load_2d(a, &P.tm_hq, kb * kBK, i * kBM, &full[s], pol_h);
            tc::tma_load_2d(b, &P.tm_wq, kb * kBK, j * kBN, &full[s]);
          } else {
            tc::tma_load_2d(a, &P.tm_hp, (kb - qblocks) * kBK, i * kBM, &full[s], pol_h);
            tc::tma_load_2d(b, &P.tm_wp, (kb - qblocks) * kBK, j * kBN, &full[s]);
          }
        }
      }
      // every copy this CTA issued (`it` fills) has landed before it exits (the MMA warp waited
      // for them, unless a bounded wait gave up)
      for (int s = 0; s < kGStages && static_cast<uint32_t>(s) < it; ++s) {
        const uint32_t last = it - 1 - ((it - 1 - s) % kGStages);  // last iteration that used stage s
        mbar_wait_bounded(&full[s], (last / kGStages) & 1u);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16_f32(kBM, kBN);
      uint32_t it = 0, tcount = 0;
      for (int tile = blockIdx.x; tile < P.ntiles && !*abort_flag; tile += gridDim.x, ++tcount) {
        // The amateur's blocks go to the z_q columns as soon as the epilogue has read the last
        // tile's z_q (it keeps that tile's scores u in the z_p columns); the expert's blocks wait
        // until it has read those too.  The epilogue's reductions overlap the amateur's MMAs.
        bool ok = true;
        for (int kb = 0; kb < nk; ++kb, ++it) {
          if (kb == 0 && qblocks > 0) {
            if (!wait_or_abort(qfree, (tcount & 1u) ^ 1u)) { ok = false; break; }
            tc::fence_after_sync();
          }
          if (kb == qblocks) {
            if (!wait_or_abort(pfree, (tcount & 1u) ^ 1u)) { ok = false; break; }
            tc::fence_after_sync();
          }
          const int s = static_cast<int>(it % kGStages);
          if (!wait_or_abort(&full[s], (it / kGStages) & 1u)) { ok = false; break; }
          tc::fence_after_sync();
          const unsigned char* a = smem + s * kGStageBytes;
          const uint64_t ad = tc::sw128_kmajor_desc(a), bd = tc::sw128_kmajor_desc(a + kABytes);
          const uint32_t d = tmem + (kb < qblocks ? static_cast<uint32_t>(kBN) : 0u);
          const bool first = kb == 0 || kb == qblocks;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)  // K = 16 per MMA: 32 bytes along the swizzled row
            tc::mma_bf16(d, ad + 2 * k, bd + 2 * k, idesc, !(first && k == 0));
          tc::mma_commit(&empty[s]);
        }
        if (!ok || *abort_flag) break;
        tc::mma_commit(tfull);
      }
      tc::mma_commit(drained);
      mbar_wait_bounded(drained, 0u);
    }
  } else {
    // ---------------- epilogue: warps 2..5, TMEM lanes 32 * (warp % 4) ..
    const int quarter = warp & 3;
    uint32_t tcount = 0;
    for (int tile = blockIdx.x; tile < P.ntiles; tile += gridDim.x, ++tcount) {
      if (__any_sync(~0u, *abort_flag != 0)) break;  // warp-uniform, before the warp-wide loads
      int i, j;
      tile_coords(tile, P.nmt, P.nvt, P.group, i, j);
      const int r = i * kBM + quarter * 32 + lane;
      const bool valid = r < P.R;
      float c1k = 0.f, ak = 0.f, Mp = 0.f, logb = -INFINITY;
      int kt[kMaxKids];
#pragma unroll
      for (int k = 0; k < kMaxKids; ++k) kt[k] = -1;
      if (valid && P.sweep == 0) {
        const float alpha = P.alpha[r / P.N];
        c1k = (1.f + alpha) * kLog2e;
        ak = alpha * kLog2e;
        if (P.beta) {
          const float be = P.beta[r / P.N];
          if (be > 0.f) {  // P_beta = {x : z_p(x) - max z_p >= log beta}
            logb = logf(be);
            Mp = P.zmax[r];
          }
        }
        const int4 k0 = reinterpret_cast<const int4*>(P.kid_tok)[2 * r];
        const int4 k1 = reinterpret_cast<const int4*>(P.kid_tok)[2 * r + 1];
        kt[0] = k0.x; kt[1] = k0.y; kt[2] = k0.z; kt[3] = k0.w;
        kt[4] = k1.x; kt[5] = k1.y; kt[6] = k1.z; kt[7] = k1.w;
      }
      const bool ok = mbar_wait_bounded(tfull, tcount & 1u);
      if (__any_sync(~0u, !ok)) {
        if (lane == 0) {
          atomicOr(P.err, DCD_DEVERR_TIMEOUT);
          *abort_flag = 1;
        }
        break;
      }
      tc::fence_after_sync();
      const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
      if (P.sweep == 1) {
        // the max sweep: this tile's max of z_p over the vocabulary
        float mz = -INFINITY;
#pragma unroll 1
        for (int c = 0; c < kBN / 64; ++c) {
          float za[32], zb[32];
          tc::tmem_ld32x2(trow + c * 64, trow + c * 64 + 32, za, zb);
          const int col0 = j * kBN + c * 64;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            if (col0 + e < P.V) mz = fmaxf(mz, za[e]);
            if (col0 + 32 + e < P.V) mz = fmaxf(mz, zb[e]);
          }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(qfree);
          mbar_arrive(pfree);
        }
        if (valid) __stcs(&P.part[static_cast<int64_t>(r) * P.nvt + j], make_float4(mz, 0.f, 0.f, 0.f));
        continue;
      }
      const bool masked = logb > -INFINITY;
      // phase 1: u = log2(e) ((1 + alpha) z_p - alpha z_q) on P_beta, written over z_p; the scores at
      // the children's tokens; then the z_q columns go back to the MMA warp
#pragma unroll 1
      for (int c = 0; c < kBN / 64; ++c) {
        float zp[64], zq[64];
        tc::tmem_ld64x2(trow + c * 64, trow + kBN + c * 64, zp, zq);
        const int col0 = j * kBN + c * 64;
#pragma unroll
        for (int e = 0; e < 64; ++e)  // u in place of z_p
          zp[e] = (col0 + e < P.V && (!masked || zp[e] - Mp >= logb)) ? fmaf(c1k, zp[e], -ak * zq[e]) : -INFINITY;
#pragma unroll
        for (int k = 0; k < kMaxKids; ++k) {
          const unsigned d = static_cast<unsigned>(kt[k] - col0);
          if (d < 64u) {  // rare: this child's token is in the chunk
            float v = 0.f;
#pragma unroll
            for (int e = 0; e < 64; ++e) v = (d == static_cast<unsigned>(e)) ? zp[e] : v;
            P.kid_u[r * kMaxKids + k] = v;
          }
        }
        tc::tmem_st64(trow + c * 64, zp);
      }
      tc::tmem_st_wait();
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(qfree);
      // phase 2 (while the next tile's amateur MMAs run): the tile's max of u, sum of 2^(u - max)
      // and argmax, from the z_p columns
      float m = -INFINITY, ssum = 0.f;
      int arg = INT_MAX;
#pragma unroll 1
      for (int c = 0; c < kBN / 64; ++c) {
        float u[64];
        tc::tmem_ld32x2(trow + c * 64, trow + c * 64 + 32, u, u + 32);
        const int col0 = j * kBN + c * 64;
        float cm = -INFINITY;
#pragma unroll
        for (int e = 0; e < 64; ++e) cm = fmaxf(cm, u[e]);
        if (cm > m) {
          ssum = m > -INFINITY ? ssum * ex2(m - cm) : 0.f;
          m = cm;
#pragma unroll
          for (int e = 63; e >= 0; --e)
            if (u[e] == cm) arg = col0 + e;
        }
        if (m > -INFINITY) {
          float acc = 0.f;
#pragma unroll
          for (int e = 0; e < 64; ++e) acc += ex2(u[e] - m);
          ssum += acc;
        }
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(pfree);
      // streaming store: read once by the combine kernel, it should not displace h in L2
      if (valid) __stcs(&P.part[static_cast<int64_t>(r) * P.nvt + j], make_float4(m, ssum, __int_as_float(arg), 0.f));
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------------------------------
// Per row: the children of its node in ascending id (at most kMaxKids) and the row's checks.
__global__ void fused_children_kernel(int32_t B, int32_t N, int32_t V, const int32_t* __restrict__ tokens,
                                      const int32_t* __restrict__ parents, const float* __restrict__ alpha,
                                      const float* __restrict__ beta, int32_t* kid_node, int32_t* kid_tok,
                                      uint32_t* row_status) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= B * N) return;
  const int b = r / N, n = r % N;
  const int32_t* par = parents + static_cast<int64_t>(b) * N;
  const int32_t* tok = tokens + static_cast<int64_t>(b) * N;
  uint32_t st = 0u;
  const int pp = par[n];
  if (n == 0 ? pp != -1 : (pp < 0 || pp >= n)) st |= DCD_DEVERR_BAD_PARENT;
  if (n > 0 && (tok[n] < 0 || tok[n] >= V)) st |= DCD_DEVERR_BAD_TOKEN;
  const float a = alpha[b];
  if (!(a >= 0.f && a <= 3.0e38f)) st |= DCD_DEVERR_BAD_PARAM;
  if (beta && !(beta[b] >= 0.f && beta[b] <= 1.f)) st |= DCD_DEVERR_BAD_PARAM;
  int count = 0;
  for (int c = n + 1; c < N; ++c) {
    if (par[c] != n) continue;
    if (count < kMaxKids) {
      kid_node[r * kMaxKids + count] = c;
      kid_tok[r * kMaxKids + count] = tok[c];
    }
    ++count;
  }
  if (count > kMaxKids) st |= DCD_DEVERR_UNSUPPORTED;
  for (int k = count; k < kMaxKids; ++k) {
    kid_node[r * kMaxKids + k] = -1;
    kid_tok[r * kMaxKids + k] = -1;
  }
  row_status[r] = st;
}

// One warp per row: the row's max of z_p over its tiles' maxima (the max sweep's result).
__global__ void fused_rowmax_kernel(int32_t R, int32_t nvt, const float4* __restrict__ part, float* zmax) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= R) return;
  float m = -INFINITY;
  for (int j = lane; j < nvt; j += 32) m = fmaxf(m, part[static_cast<int64_t>(r) * nvt + j].x);
  m = warp_max(m);
  if (lane == 0) zmax[r] = m;
}

// ------------------------------------------------------------------------------------------
struct CombineArgs {
  int32_t B, N, nvt;
  const float4* part;
  const int32_t* kid_node;
  const int32_t* kid_tok;
  const float* kid_u;
  const uint32_t* row_status;
  float* cd_logprob;
  int32_t* cd_argmax;
  float* cd_lse;
  RowRecord* rec;
};

// One warp per row: merge the tiles' statistics in tile order, then the Eq. 1 outputs and the
// greedy rule (the first child whose token is the argmax).
__global__ void fused_combine_kernel(const CombineArgs C) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= C.B * C.N) return;
  auto merge = [](float& m1, float& s1, int& a1, float m2, float s2, int a2) {
    const float M = fmaxf(m1, m2);
    const float t1 = m1 > -INFINITY ? s1 * ex2(m1 - M) : 0.f;
    const float t2 = m2 > -INFINITY ? s2 * ex2(m2 - M) : 0.f;
    if (m2 > m1 || (m2 == m1 && a2 < a1)) a1 = a2;
    m1 = M;
    s1 = t1 + t2;
  };
  float m = -INFINITY, s = 0.f;
  int arg = INT_MAX;
  const float4* pr = C.part + static_cast<int64_t>(r) * C.nvt;
  for (int j = lane; j < C.nvt; j += 32) {
    const float4 v = pr[j];
    merge(m, s, arg, v.x, v.y, __float_as_int(v.z));
  }
#pragma unroll
  for (int o = 16; o; o >>= 1)
    merge(m, s, arg, __shfl_xor_sync(~0u, m, o), __shfl_xor_sync(~0u, s, o), __shfl_xor_sync(~0u, arg, o));
  if (lane != 0) return;
  const int b = r / C.N, n = r % C.N;
  uint32_t status = C.row_status[r];
  if (!(m > -INFINITY && m < INFINITY) || !(s > 0.f && s < INFINITY)) status |= DCD_DEVERR_NONFINITE;
  const float logS = logf(s);
  if (C.cd_argmax) C.cd_argmax[r] = arg;
  if (C.cd_lse) C.cd_lse[r] = m * kLn2f + logS;
  if (C.cd_logprob && n == 0) C.cd_logprob[r] = 0.f;
  int acc = -1;
  for (int k = 0; k < kMaxKids; ++k) {
    const int node = C.kid_node[r * kMaxKids + k];
    if (node < 0) break;
    if (C.cd_logprob) C.cd_logprob[static_cast<int64_t>(b) * C.N + node] = (C.kid_u[r * kMaxKids + k] - m) * kLn2f - logS;
    if (acc < 0 && C.kid_tok[r * kMaxKids + k] == arg) acc = node;
  }
  RowRecord rr;
  rr.acc_child = acc;
  rr.term_token = acc < 0 ? arg : -1;
  rr.status = status;
  rr.reserved = 0;
  C.rec[r] = rr;
}

// ------------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// A [rows, K] row-major bf16 matrix as TMA boxes of 64 x box_rows, 128-byte swizzle, zero fill
// outside the matrix.
bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t K, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

}  // namespace

FusedLayout fused_layout(int64_t rows, int64_t V) {
  FusedLayout l;
  const int64_t nvt = (V + kBN - 1) / kBN;
  size_t off = kWorkspaceHeader;
  l.kid_node = off;
  off += static_cast<size_t>(rows) * kMaxKids * 4;
  l.kid_tok = off;
  off += static_cast<size_t>(rows) * kMaxKids * 4;
  l.kid_u = off;
  off += static_cast<size_t>(rows) * kMaxKids * 4;
  l.row_status = off;
  off += (static_cast<size_t>(rows) * 4 + 15) & ~static_cast<size_t>(15);
  l.rec = off;
  off += static_cast<size_t>(rows) * sizeof(RowRecord);
  l.part = off;
  off += static_cast<size_t>(rows) * static_cast<size_t>(nvt) * 16;
  l.zmax = off;
  off += (static_cast<size_t>(rows) * 4 + 15) & ~static_cast<size_t>(15);
  l.total = (off + 255) & ~static_cast<size_t>(255);
  return l;
}

cudaError_t launch_fused(const FusedArgs& f, cudaStream_t stream, int* status) {
  *status = DCD_OK;
  const int64_t R = static_cast<int64_t>(f.B) * f.N;
  if (R == 0) return cudaSuccess;
  const FusedLayout l = fused_layout(R, f.V);
  unsigned char* ws = static_cast<unsigned char*>(f.workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(ws);
  int32_t* kid_node = reinterpret_cast<int32_t*>(ws + l.kid_node);
  int32_t* kid_tok = reinterpret_cast<int32_t*>(ws + l.kid_tok);
  float* kid_u = reinterpret_cast<float*>(ws + l.kid_u);
  uint32_t* row_status = reinterpret_cast<uint32_t*>(ws + l.row_status);
  RowRecord* rec = reinterpret_cast<RowRecord*>(ws + l.rec);
  float4* part = reinterpret_cast<float4*>(ws + l.part);
  float* zmax = reinterpret_cast<float*>(ws + l.zmax);

  FusedParams P;
  if (!make_map(&P.tm_hp, f.h_exp, R, f.H_exp, kBM) || !make_map(&P.tm_wp, f.w_exp, f.V, f.H_exp, kBN) ||
      !make_map(&P.tm_hq, f.h_ama, R, f.H_ama, kBM) || !make_map(&P.tm_wq, f.w_ama, f.V, f.H_ama, kBN)) {
    *status = DCD_ERR_UNSUPPORTED;
    return cudaSuccess;
  }
  P.R = static_cast<int32_t>(R);
  P.V = static_cast<int32_t>(f.V);
  P.N = f.N;
  P.nkp = (f.H_exp + kBK - 1) / kBK;
  P.nkq = (f.H_ama + kBK - 1) / kBK;
  P.nmt = static_cast<int32_t>((R + kBM - 1) / kBM);
  P.nvt = static_cast<int32_t>((f.V + kBN - 1) / kBN);
  P.ntiles = P.nmt * P.nvt;
  // A group of row tiles keeps about kGroupHBytes of hidden states live in L2 (measured at the
  // full workload: groups of 15 row tiles, 39 MB, 2.6% faster than all 30 at once, whose 79 MB of h
  // missed L2 a quarter of the time next to the weight blocks in flight).
  {
    const int64_t per_tile = static_cast<int64_t>(kBM) * (static_cast<int64_t>(f.H_exp) + f.H_ama) * 2;
    int64_t g = kGroupHBytes / (per_tile > 0 ? per_tile : 1);
    P.group = static_cast<int32_t>(g < 1 ? 1 : (g > P.nmt ? P.nmt : g));
  }
  P.sweep = 0;
  P.alpha = f.alpha;
  P.beta = f.beta;
  P.zmax = zmax;
  P.kid_tok = kid_tok;
  P.kid_u = kid_u;
  P.part = part;
  P.err = &hdr->err;

  cudaError_t e = cudaMemsetAsync(hdr, 0, kWorkspaceHeader, stream);
  if (e != cudaSuccess) return e;
  fused_children_kernel<<<static_cast<unsigned>((R + 127) / 128), 128, 0, stream>>>(
      f.B, f.N, static_cast<int32_t>(f.V), f.tokens, f.parents, f.alpha, f.beta, kid_node, kid_tok, row_status);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;

  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(fused_lmhead_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(kGemmSmem));
  });
  if (attr_err != cudaSuccess) return attr_err;
  int grid = sm_count();
  if (grid <= 0) return cudaErrorInvalidDevice;
  if (grid > P.ntiles) grid = P.ntiles;
  if (f.gemm_start) {
    e = cudaEventRecord(f.gemm_start, stream);
    if (e != cudaSuccess) return e;
  }
  if (f.beta) {
    // with a plausibility mask: first the expert's logits alone for each row's max of z_p (the
    // same MMAs in the same order as below, so the second sweep sees bit-identical z_p)
    FusedParams P1 = P;
    P1.sweep = 1;
    fused_lmhead_kernel<<<grid, kGemmThreads, kGemmSmem, stream>>>(P1);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    fused_rowmax_kernel<<<static_cast<unsigned>((R + 7) / 8), 256, 0, stream>>>(P.R, P.nvt, part, zmax);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  fused_lmhead_kernel<<<grid, kGemmThreads, kGemmSmem, stream>>>(P);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (f.gemm_stop) {
    e = cudaEventRecord(f.gemm_stop, stream);
    if (e != cudaSuccess) return e;
  }

  CombineArgs C;
  C.B = f.B;
  C.N = f.N;
  C.nvt = P.nvt;
  C.part = part;
  C.kid_node = kid_node;
  C.kid_tok = kid_tok;
  C.kid_u = kid_u;
  C.row_status = row_status;
  C.cd_logprob = f.cd_logprob;
  C.cd_argmax = f.cd_argmax;
  C.cd_lse = f.cd_lse;
  C.rec = rec;
  fused_combine_kernel<<<static_cast<unsigned>((R + 7) / 8), 256, 0, stream>>>(C);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_tree_walk(f.B, f.N, rec, &hdr->err, f.accept_len, f.accept_path, f.bonus, stream);
}

}  // namespace dcd
