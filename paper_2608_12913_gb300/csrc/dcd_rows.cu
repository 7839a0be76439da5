// dcd_rows.cu -- the streaming kernels of the CD verification step on sm_103a.
//
// score_rows_kernel: a persistent grid (a few CTAs per SM).  Each CTA claims whole
//   tree-node rows g = b * N + n from a work counter, in node-major order (every
//   sequence's node 0, then every node 1, ...), so internal nodes -- the rows that
//   may need extra passes -- come first and leaves last.  A row is streamed through
//   a ring of 32 KB shared-memory stages filled by bulk
//   asynchronous copies that complete on one mbarrier per stage; thread 0 refills a
//   stage as soon as the block has consumed it, so a ring's worth of the row is
//   always in flight.
//   The "stats" pass computes the CD score s' = (1 + alpha) z_p - alpha z_q (Eq. 1;
//   the two log-softmax shifts are constant per row and cancel in the normaliser)
//   on the plausibility set P_beta of Sec. 2.1; every lane keeps an online max, a
//   sum of 2^((s' - max) k2) (k2 = log2(e) / T) rescaled when its max grows, and
//   its argmax, reduced over the block at the end of the row.  Rows whose terminal
//   draw races over pi_CD itself (sampled leaves) also keep, per 256-token block,
//   the block max and sum, i.e. the block masses of pi_CD.  With beta > 0 a "max"
//   pass over z_p comes first.  Sampled rows then test their children in ascending node id (Algorithm 1
//   on sibling lists); each rejection streams the row once more (z_p, z_q and q) to
//   get the next residual's mass Z_j, recomputing r_j(x) = max(0, r_{j-1}(x) - q(x))
//   / Z_j token by token from pi_CD(x), q(x) and the earlier Z's, so nothing per
//   token is stored between passes.  Rows that take more than one pass are read with
//   an L2 evict-last policy, so their later passes hit L2 and HBM is read once.  A
//   node without an accepted child draws its terminal token by a two-level
//   exponential race: a 256-token block by its mass, then a token of that block,
//   whose 256 values are re-read directly.
// tree_walk_kernel: one thread per sequence follows the accepted children.
// terminal_residual_kernel: one block per sequence rebuilds the distribution its
//   bonus token was drawn from (test output only).

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <mutex>

#include "dcd.h"
#include "dcd_internal.h"

namespace dcd {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kStageBytes = 32 * 1024;            // bytes per ring stage
constexpr int kRaceBlock = 256;                   // tokens per block of the two-level terminal race
constexpr int kMaxStages = 8;
constexpr size_t kSmemMax = 227 * 1024;
constexpr size_t kSmemPerSm = 228 * 1024;
constexpr long long kWaitCycles = 4000000000ll;  // about two seconds at the boost clock
constexpr float kLog2e = 1.4426950408889634f;

enum PassKind { kPassMax = 0, kPassStats = 1, kPassRes = 2 };

// ------------------------------------------------------------------------------------------
// PTX wrappers: mbarrier, L2 cache policies and bulk asynchronous global->shared copies.
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(smem_addr(bar)),
      "r"(bytes)
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.b32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// Bounded wait: gives up after kWaitCycles and reports false.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  const long long start = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - start > kWaitCycles) return false;
  }
  return true;
}

__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
      "%4;" ::"r"(smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// ------------------------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32->64 products
// with the published multipliers, the key advanced by the published Weyl increments.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

__device__ __forceinline__ uint4 philox_block(uint64_t seed, uint64_t off, uint32_t c0, uint32_t c1) {
  return philox4x32_10(make_uint4(c0, c1, static_cast<uint32_t>(off), static_cast<uint32_t>(off >> 32)),
                       static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32));
}

__device__ __forceinline__ uint32_t word_of(const uint4& w, int i) {
  return i == 0 ? w.x : i == 1 ? w.y : i == 2 ? w.z : w.w;
}

// 32-bit word -> uniform in (0, 1): ((w >> 9) + 1/2) 2^-23, exact in fp32.
__device__ __forceinline__ float u01(uint32_t w) {
  return (__uint2float_rn(w >> 9) + 0.5f) * 1.1920928955078125e-07f;
}

// Race key in log2 units: log2 r - log2(-log2 u) orders tokens exactly as ln r - ln(-ln u)
// (the two differ by a positive factor and a constant).
__device__ __forceinline__ float race_key(float log2_mass, uint32_t word) {
  return log2_mass - lg2(-lg2(u01(word)));
}

// ------------------------------------------------------------------------------------------
// Element access: 8 consecutive tokens as fp32 (16 B of bf16 or 32 B of fp32).
__device__ __forceinline__ void ld8(const float* p, float v[8]) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ void ld8(const __nv_bfloat16* p, float v[8]) {
  const uint4 a = *reinterpret_cast<const uint4*>(p);
  v[0] = __uint_as_float(a.x << 16); v[1] = __uint_as_float(a.x & 0xffff0000u);
  v[2] = __uint_as_float(a.y << 16); v[3] = __uint_as_float(a.y & 0xffff0000u);
  v[4] = __uint_as_float(a.z << 16); v[5] = __uint_as_float(a.z & 0xffff0000u);
  v[6] = __uint_as_float(a.w << 16); v[7] = __uint_as_float(a.w & 0xffff0000u);
}

__device__ __forceinline__ float ld1(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float ld1(const __nv_bfloat16* p, int64_t i) { return __bfloat162float(p[i]); }

// ------------------------------------------------------------------------------------------
// Reductions.
__device__ __forceinline__ void argmax_merge(float& v, int& i, float v2, int i2) {
  if (v2 > v || (v2 == v && i2 < i)) {
    v = v2;
    i = i2;
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(~0u, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(~0u, v, o));
  return v;
}

__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int o = 16; o; o >>= 1) argmax_merge(v, i, __shfl_xor_sync(~0u, v, o), __shfl_xor_sync(~0u, i, o));
}

// Block reductions: every thread gets the result; the scratch is free again on return.
__device__ __forceinline__ void block_argmax(float& v, int& i, float* redf, int* redi) {
  warp_argmax(v, i);
  if ((threadIdx.x & 31) == 0) {
    redf[threadIdx.x >> 5] = v;
    redi[threadIdx.x >> 5] = i;
  }
  __syncthreads();
  v = redf[0];
  i = redi[0];
#pragma unroll
  for (int w = 1; w < kWarps; ++w) argmax_merge(v, i, redf[w], redi[w]);
  __syncthreads();
}

__device__ __forceinline__ float block_sum(float v, float* redf) {
  v = warp_sum(v);
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = v;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) s += redf[w];
  __syncthreads();
  return s;
}

__device__ __forceinline__ float block_max(float v, float* redf) {
  v = warp_max(v);
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = v;
  __syncthreads();
  float s = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) s = fmaxf(s, redf[w]);
  __syncthreads();
  return s;
}

// ------------------------------------------------------------------------------------------
struct SParams {
  ScoreArgs a;
  int32_t nst;           // ring depth (stages of kStageBytes)
  int32_t tok_a;         // tokens per stage in the max and stats passes (z_p, z_q)
  int32_t tok_r;         // tokens per stage in residual passes (z_p, z_q, q)
  int32_t bulk;          // 1: bulk asynchronous copies, 0: plain loads
  int32_t nblk;          // race blocks per row, ceil(V / 256)
  int32_t meta_offset;   // byte offsets into dynamic shared memory
  int32_t blk_offset;
  int32_t stage_offset;
  uint32_t* work;        // row counter, zeroed before the launch
};

// Row state shared by the block (written by one thread, read after a barrier).
struct RowShared {
  int32_t next;      // the next claimed work item
  int32_t m;         // children of the row's node
  uint32_t status;   // DCD_DEVERR_* bits
  int32_t accept;    // outcome of the current sibling test
  int32_t term;      // terminal token
  int32_t pad[3];
};

template <typename TIn>
struct Stage {
  TIn* zp;
  TIn* zq;
  float* q;
};

// A stage holds `tok` tokens of z_p, then of z_q, then (residual passes) of q.
template <typename TIn>
__device__ __forceinline__ Stage<TIn> stage_at(unsigned char* base, int s, int tok) {
  Stage<TIn> st;
  st.zp = reinterpret_cast<TIn*>(base + static_cast<size_t>(s) * kStageBytes);
  st.zq = st.zp + tok;
  st.q = reinterpret_cast<float*>(st.zq + tok);
  return st;
}

// ------------------------------------------------------------------------------------------
template <typename TIn>
__global__ void __launch_bounds__(kThreads) score_rows_kernel(const __grid_constant__ SParams sp) {
  const ScoreArgs& p = sp.a;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int N = p.N;
  const int64_t V = p.V;
  const int R = p.B * N;
  const int nch_a = static_cast<int>((V + sp.tok_a - 1) / sp.tok_a);  // chunks of a max / stats pass
  const int nch_r = static_cast<int>((V + sp.tok_r - 1) / sp.tok_r);  // chunks of a residual pass

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
  float* invZ = cq + N;                                           // [N] 1/Z_j (0 marks Z_j = 0)
  float* bmax = reinterpret_cast<float*>(smem + sp.blk_offset);   // [nblk] block max of s'
  float* bsum = bmax + sp.nblk;                                   // [nblk] block sums
  float* bres = bsum + sp.nblk;                                   // [nblk] final residual block masses
  float* bq = bres + sp.nblk;                                     // [nblk] block masses of q
  unsigned char* ring = smem + sp.stage_offset;

  if (tid == 0) {
    for (int s = 0; s < sp.nst; ++s) mbar_init(&full[s], 1);
    fence_mbar_init();
    rs->next = static_cast<int32_t>(atomicAdd(sp.work, 1u));
  }
  __syncthreads();
  const uint64_t pol_last = l2_policy_evict_last();
  const uint64_t pol_first = l2_policy_evict_first();
  uint32_t seq = 0;  // ring items consumed by this CTA so far (identical in every thread)

  for (;;) {
    const int item = rs->next;
    __syncthreads();  // every thread has read the claim before thread 0 replaces it
    if (item >= R) break;
    if (tid == 0) rs->next = static_cast<int32_t>(atomicAdd(sp.work, 1u));  // used by the next row
    const int b = item % p.B, n = item / p.B;  // node-major order
    const int64_t g = static_cast<int64_t>(b) * N + n;
    const float alpha = p.alpha[b];
    const float beta = p.beta ? p.beta[b] : 0.f;
    const float T = p.temp ? p.temp[b] : 0.f;
    const bool sampled = T > 0.f && p.q != nullptr;
    const bool masked = beta > 0.f;
    const float invT = T > 0.f ? 1.f / T : 1.f;
    const float k2 = kLog2e * invT;  // exp(x / T) = 2^(x * k2)
    const float c1 = 1.f + alpha;
    const float logb = masked ? logf(beta) : -INFINITY;
    const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
    const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;
    const float* q_row = sampled ? p.q + g * p.ldq : nullptr;

    // ---- ring items of this row: [max pass if beta > 0] [stats pass] [a residual pass per
    // rejected child]; thread 0 keeps up to nst items in flight, never past `limit`
    const int nknown = (masked ? 2 : 1) * nch_a;
    const uint32_t seq0 = seq;
    auto pass_of = [&](int L) -> int {
      if (L < nknown) return (masked && L < nch_a) ? kPassMax : kPassStats;
      return kPassRes;
    };
    // token range and stage layout of item L
    auto chunk_of = [&](int L, int64_t& x0, int& clen, int& tok) {
      const bool res = L >= nknown;
      tok = res ? sp.tok_r : sp.tok_a;
      const int c = res ? (L - nknown) % nch_r : L % nch_a;
      x0 = static_cast<int64_t>(c) * tok;
      clen = static_cast<int>((V - x0) < tok ? (V - x0) : tok);
    };
    auto issue = [&](int L, uint64_t pol) {  // thread 0 only
      const uint32_t sq = seq0 + static_cast<uint32_t>(L);
      const int s = static_cast<int>(sq % static_cast<uint32_t>(sp.nst));
      int64_t x0;
      int clen, tok;
      chunk_of(L, x0, clen, tok);
      const Stage<TIn> st = stage_at<TIn>(ring, s, tok);
      const int kind = pass_of(L);
      uint32_t zb = 0, qb = 0;
      if (sp.bulk) {
        zb = static_cast<uint32_t>(clen * static_cast<int>(sizeof(TIn))) & ~15u;
        qb = kind == kPassRes ? static_cast<uint32_t>(clen * 4) & ~15u : 0u;
      }
      mbar_arrive_expect_tx(&full[s], (kind == kPassMax ? zb : 2u * zb) + qb);
      if (zb) {
        bulk_g2s(st.zp, zp_row + x0, zb, &full[s], pol);
        if (kind != kPassMax) bulk_g2s(st.zq, zq_row + x0, zb, &full[s], pol);
      }
      if (qb) bulk_g2s(st.q, q_row + x0, qb, &full[s], pol);
    };

    // thread 0 starts the row's stream at once (rows that may take more than one pass are
    // kept in L2); warp 1 meanwhile finds the children of node n and checks this row's node
    uint64_t pol = (masked || sampled) ? pol_last : pol_first;
    if (tid == 0) {
      const int first = nknown < sp.nst ? nknown : sp.nst;
      for (int L = 0; L < first; ++L) issue(L, pol);
    }
    if (warp == 1) {
      const int32_t* par = p.parents + static_cast<int64_t>(b) * N;
      const int32_t* tok = p.tokens + static_cast<int64_t>(b) * N;
      int count = 0;
      for (int base = n + 1; base < N; base += 32) {
        const int c = base + lane;
        const bool is = c < N && par[c] == n;
        const unsigned msk = __ballot_sync(~0u, is);
        if (is) {
          const int pos = count + __popc(msk & ((1u << lane) - 1u));
          kids[pos] = c;
          ktok[pos] = tok[c];
        }
        count += __popc(msk);
      }
      if (lane == 0) {
        uint32_t st = 0u;
        const int pp = par[n];
        if (n == 0 ? pp != -1 : (pp < 0 || pp >= n)) st |= DCD_DEVERR_BAD_PARENT;
        if (n > 0) {
          const int t = tok[n];
          if (t < 0 || t >= V) st |= DCD_DEVERR_BAD_TOKEN;
        }
        if (!(alpha >= 0.f && alpha <= 3.0e38f) || !(beta >= 0.f && beta <= 1.f) || !(T >= 0.f && T <= 3.0e38f))
          st |= DCD_DEVERR_BAD_PARAM;
        rs->m = count;
        rs->status = st;
      }
    }
    __syncthreads();
    const int m = rs->m;
    pol = (masked || (sampled && m > 0)) ? pol_last : pol_first;
    // values at the children's tokens: the loads are issued now and consumed after the stats pass
    float pzp = 0.f, pzq = 0.f, pq = 0.f;
    if (tid < m) {
      const int t = ktok[tid];
      if (t >= 0 && t < V) {
        pzp = ld1(zp_row, t);
        pzq = ld1(zq_row, t);
        if (sampled) pq = q_row[t];
      }
    }

    int limit = nknown;  // items planned so far
    int L = 0;           // next item to consume
    bool timed_out = false;

    // Consumes `count` items: waits for each stage, fills a ragged or unaligned remainder with
    // plain loads, hands the stage to `body`, releases the stage and refills it.
    auto run_items = [&](int count, auto&& body) {
      for (int it = 0; it < count; ++it, ++L) {
        const uint32_t sq = seq0 + static_cast<uint32_t>(L);
        const int s = static_cast<int>(sq % static_cast<uint32_t>(sp.nst));
        const uint32_t parity = (sq / static_cast<uint32_t>(sp.nst)) & 1u;
        int64_t x0;
        int clen, tok;
        chunk_of(L, x0, clen, tok);
        const Stage<TIn> st = stage_at<TIn>(ring, s, tok);
        const int kind = pass_of(L);
        if (!mbar_wait_bounded(&full[s], parity)) timed_out = true;
        const int zfirst =
            sp.bulk ? ((clen * static_cast<int>(sizeof(TIn))) & ~15) / static_cast<int>(sizeof(TIn)) : 0;
        const int qfirst = sp.bulk ? ((clen * 4) & ~15) / 4 : 0;
        if (zfirst < clen || (kind == kPassRes && qfirst < clen)) {
          for (int i = zfirst + tid; i < clen; i += kThreads) {
            st.zp[i] = zp_row[x0 + i];
            if (kind != kPassMax) st.zq[i] = zq_row[x0 + i];
          }
          if (kind == kPassRes)
            for (int i = qfirst + tid; i < clen; i += kThreads) st.q[i] = q_row[x0 + i];
          __syncthreads();
        }
        body(st, x0, clen);
        __syncthreads();
        if (tid == 0 && L + sp.nst < limit) issue(L + sp.nst, pol);
      }
    };

    // ---- pass A (beta > 0): the expert max, for P_beta = {x : z_p(x) - max z_p >= log beta}
    float Mp = 0.f;
    if (masked) {
      float lm = -INFINITY;
      run_items(nch_a, [&](const Stage<TIn>& st, int64_t, int clen) {
        for (int i0 = tid * 8; i0 < clen; i0 += kThreads * 8) {
          float zp[8];
          ld8(st.zp + i0, zp);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            if (i0 + e < clen) lm = fmaxf(lm, zp[e]);
        }
      });
      Mp = block_max(lm, redf);
    }

    // ---- pass B: the CD score s' on P_beta.  Each lane keeps an online max, a sum of
    // 2^((s' - max) k2) rescaled whenever its max grows, and its argmax.  Rows that end in a
    // race over pi_CD itself (sampled leaves) also record, per 256-token block (one warp, 8
    // tokens a lane), the block's max and its sum relative to that max.
    const bool leaf_race = sampled && m == 0;
    float lmax = -INFINITY, lsum = 0.f;
    int larg = INT_MAX;
    run_items(nch_a, [&](const Stage<TIn>& st, int64_t x0, int clen) {
      for (int kb = warp; kb * kRaceBlock < sp.tok_a; kb += kWarps) {
        if (kb * kRaceBlock >= clen) break;  // warp-uniform
        const int i0 = kb * kRaceBlock + lane * 8;
        float zp[8], zq[8], sv[8];
        ld8(st.zp + i0, zp);
        ld8(st.zq + i0, zq);
        float gm = -INFINITY;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const bool in = (i0 + e < clen) && (!masked || (zp[e] - Mp >= logb));
          sv[e] = in ? fmaf(c1, zp[e], -alpha * zq[e]) : -INFINITY;
          gm = fmaxf(gm, sv[e]);
        }
        if (gm > lmax) {
          lsum *= ex2((lmax - gm) * k2);  // 0 while lmax is -inf
          lmax = gm;
#pragma unroll
          for (int e = 7; e >= 0; --e)
            if (sv[e] == gm) larg = static_cast<int>(x0) + i0 + e;
        }
        if (lmax > -INFINITY) {
          const float mk = lmax * k2;
          float s0 = 0.f, s1 = 0.f;
#pragma unroll
          for (int e = 0; e < 8; e += 2) {
            s0 += ex2(fmaf(sv[e], k2, -mk));
            s1 += ex2(fmaf(sv[e + 1], k2, -mk));
          }
          lsum += s0 + s1;
        }
        if (leaf_race) {
          const float bm = warp_max(gm);
          float part = 0.f;
          if (bm > -INFINITY) {
            const float mk = bm * k2;
#pragma unroll
            for (int e = 0; e < 8; ++e) part += ex2(fmaf(sv[e], k2, -mk));
          }
          const float bs = warp_sum(part);
          if (lane == 0) {
            const int kabs = static_cast<int>(x0 / kRaceBlock) + kb;
            bmax[kabs] = bm;
            bsum[kabs] = bs;
          }
        }
      }
    });
    if (tid < m) {
      czp[tid] = pzp;
      czq[tid] = pzq;
      cq[tid] = pq;
    }
    for (int k = kThreads + tid; k < m; k += kThreads) {  // rows with more children than threads
      const int t = ktok[k];
      const bool ok = t >= 0 && t < V;
      czp[k] = ok ? ld1(zp_row, t) : 0.f;
      czq[k] = ok ? ld1(zq_row, t) : 0.f;
      cq[k] = (ok && sampled) ? q_row[t] : 0.f;
    }
    // row statistics from the lanes' (max, sum, argmax) (the reductions below also publish
    // czp/czq/cq)
    const float M = block_max(lmax, redf);
    const float S = block_sum(lmax > -INFINITY ? lsum * ex2((lmax - M) * k2) : 0.f, redf);
    float lbest = lmax;
    block_argmax(lbest, larg, redf, redi);
    const int arg = larg;
    uint32_t status = rs->status;
    if (!(M > -INFINITY && M < INFINITY) || !(S > 0.f && S < INFINITY)) status |= DCD_DEVERR_NONFINITE;
    const float logS = logf(S);
    const float invS = 1.f / S;
    const float Mk2 = M * k2;

    // ---- outputs of the Eq. 1 target
    if (tid == 0) {
      if (p.cd_argmax) p.cd_argmax[g] = arg;
      if (p.cd_lse) p.cd_lse[g] = M * invT + logS;
      if (n == 0 && p.cd_logprob) p.cd_logprob[g] = 0.f;
    }
    if (p.cd_logprob) {
      for (int k = tid; k < m; k += kThreads) {
        const bool in = !masked || (czp[k] - Mp >= logb);
        p.cd_logprob[static_cast<int64_t>(b) * N + kids[k]] =
            in ? (fmaf(c1, czp[k], -alpha * czq[k]) - M) * invT - logS : -INFINITY;
      }
    }

    int acc = -1, term = -1;
    if (!sampled) {
      // ---- greedy rule: the first child whose token is the argmax
      for (int k = 0; k < m; ++k)
        if (ktok[k] == arg) {
          acc = kids[k];
          break;
        }
      if (acc < 0) term = arg;
    } else {
      // ---- sampled rule: test the children in order; each rejection streams one residual pass.
      // r_j(x) = max(0, r_{j-1}(x) - q(x)) / Z_j with r_0 = pi_CD,T; invZ[j] = 0 marks Z_j = 0,
      // where r_{j-1} equals q exactly and r_j is taken as q.
      auto residual_at = [&](float s, bool in, float qv, int levels) -> float {
        float r = in ? ex2(fmaf(s, k2, -Mk2)) * invS : 0.f;
        for (int i = 1; i <= levels; ++i) {
          const float iz = invZ[i];
          r = iz > 0.f ? fmaxf(r - qv, 0.f) * iz : qv;
        }
        return r;
      };
      for (int j = 0; j < m; ++j) {
        if (tid == 0) {
          const bool in = !masked || (czp[j] - Mp >= logb);
          const float rt = residual_at(fmaf(c1, czp[j], -alpha * czq[j]), in, cq[j], j);
          const float qt = cq[j];
          const float ratio = qt > 0.f ? rt / qt : (rt > 0.f ? INFINITY : 0.f);
          const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * N + kids[j]);
          const float u = u01(philox_block(p.seed, p.offset, G, 0u).x);
          rs->accept = u <= ratio;
        }
        __syncthreads();
        if (rs->accept) {
          acc = kids[j];
          break;
        }
        // rejected: one more pass gives Z_{j+1}; after the last child it also keeps the block
        // masses of the final residual and of q for the terminal race
        const bool last = j + 1 == m;
        const int first = limit;
        limit += nch_r;
        if (tid == 0)
          for (int Li = first; Li < limit && Li < first + sp.nst; ++Li) issue(Li, pol);
        float zl = 0.f;
        run_items(nch_r, [&](const Stage<TIn>& st, int64_t x0, int clen) {
          for (int kb = warp; kb * kRaceBlock < sp.tok_r; kb += kWarps) {
            if (kb * kRaceBlock >= clen) break;  // warp-uniform
            const int i0 = kb * kRaceBlock + lane * 8;
            float zp[8], zq[8], qv[8];
            ld8(st.zp + i0, zp);
            ld8(st.zq + i0, zq);
            ld8(st.q + i0, qv);
            float part = 0.f, partq = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const bool valid = i0 + e < clen;
              const float qe = valid ? qv[e] : 0.f;
              const bool in = valid && (!masked || (zp[e] - Mp >= logb));
              const float r = residual_at(fmaf(c1, zp[e], -alpha * zq[e]), in, qe, j);
              part += valid ? fmaxf(r - qe, 0.f) : 0.f;
              partq += qe;
            }
            zl += part;
            if (last) {
              const float br = warp_sum(part);
              const float bqq = warp_sum(partq);
              if (lane == 0) {
                const int kabs = static_cast<int>(x0 / kRaceBlock) + kb;
                bres[kabs] = br;
                bq[kabs] = bqq;
              }
            }
          }
        });
        const float Z = block_sum(zl, redf);
        if (tid == 0) invZ[j + 1] = Z > 0.f ? 1.f / Z : 0.f;
        __syncthreads();
      }
      if (acc < 0) {
        // ---- terminal draw, two-level exponential race: a 256-token block by its mass ...
        const bool leaf = m == 0;
        const bool degen = !leaf && !(invZ[m] > 0.f);
        float bk = -INFINITY;
        int bb = INT_MAX;
        for (int k = tid; k < sp.nblk; k += kThreads) {
          float lm = -INFINITY;
          if (leaf) {
            if (bmax[k] > -INFINITY && bsum[k] > 0.f) lm = lg2(bsum[k]) + (bmax[k] - M) * k2;
          } else {
            const float Rk = degen ? bq[k] : bres[k];
            if (Rk > 0.f) lm = lg2(Rk);
          }
          if (lm > -INFINITY) {
            const uint4 w = philox_block(p.seed, p.offset, static_cast<uint32_t>(g),
                                         0x80000000u | (static_cast<uint32_t>(k) >> 2));
            const float key = race_key(lm, word_of(w, k & 3));
            if (key > bk) {
              bk = key;
              bb = k;
            }
          }
        }
        block_argmax(bk, bb, redf, redi);
        // ... then a token of that block (warp 0 re-reads the block's 256 tokens)
        if (warp == 0) {
          float tk = -INFINITY;
          int tx = INT_MAX;
          if (bb != INT_MAX) {
            const int64_t xb = static_cast<int64_t>(bb) * kRaceBlock + lane * 8;
            const uint4 wa = philox_block(p.seed, p.offset, static_cast<uint32_t>(g),
                                          1u + static_cast<uint32_t>(xb >> 2));
            const uint4 wb = philox_block(p.seed, p.offset, static_cast<uint32_t>(g),
                                          2u + static_cast<uint32_t>(xb >> 2));
            const uint32_t w[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int64_t x = xb + e;
              if (x < V) {
                const float z = ld1(zp_row, x);
                const bool in = !masked || (z - Mp >= logb);
                const float s = fmaf(c1, z, -alpha * ld1(zq_row, x));
                float v;
                if (leaf) {
                  v = in ? ex2(fmaf(s, k2, -Mk2)) : 0.f;
                } else {
                  const float qe = q_row[x];
                  v = degen ? qe : fmaxf(residual_at(s, in, qe, m - 1) - qe, 0.f);
                }
                if (v > 0.f) {
                  const float key = race_key(lg2(v), w[e]);
                  if (key > tk) {
                    tk = key;
                    tx = static_cast<int>(x);
                  }
                }
              }
            }
          }
          warp_argmax(tk, tx);
          if (lane == 0) rs->term = tx;
        }
        __syncthreads();
        term = rs->term;
      }
    }
    if (tid == 0) {
      RowRecord r;
      r.acc_child = acc;
      r.term_token = acc < 0 ? term : -1;
      r.status = status | (timed_out ? DCD_DEVERR_TIMEOUT : 0u);
      r.reserved = 0;
      p.rec[g] = r;
    }
    seq = seq0 + static_cast<uint32_t>(L);
    __syncthreads();  // row state in shared memory is rewritten by the next row
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

Layout layout_for(int N, int nblk, int nst, int stage_bytes) {
  Layout l;
  l.meta_offset = 8 * kMaxStages + 64 * 4;
  const size_t meta_end = static_cast<size_t>(l.meta_offset) + sizeof(RowShared) + static_cast<size_t>(N) * 4 * 6;
  l.blk_offset = static_cast<int>((meta_end + 15) & ~static_cast<size_t>(15));
  const size_t blk_end = static_cast<size_t>(l.blk_offset) + static_cast<size_t>(nblk) * 4 * 4;
  l.stage_offset = static_cast<int>((blk_end + 127) & ~static_cast<size_t>(127));
  l.total = static_cast<size_t>(l.stage_offset) + static_cast<size_t>(nst) * stage_bytes;
  return l;
}

// Tokens per stage: z_p and z_q fill a stage in the max / stats passes; z_p, z_q and q share
// it in residual passes (whole race blocks of 256 tokens either way).
int tokens_a(int es) { return kStageBytes / (2 * es); }
int tokens_r(int es) { return kStageBytes / (2 * es + 4) / kRaceBlock * kRaceBlock; }

}  // namespace

RowGeometry row_geometry(const ScoreArgs& a) {
  RowGeometry geo{};
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  const int nblk = static_cast<int>((a.V + kRaceBlock - 1) / kRaceBlock);
  int nst = a.force_stages;
  if (nst <= 0) {
    // the deepest ring (up to 3 stages) that still lets two CTAs share an SM
    nst = 2;
    for (int s = 3; s >= 2; --s)
      if (2 * (layout_for(a.N, nblk, s, kStageBytes).total + 1024) <= kSmemPerSm) {
        nst = s;
        break;
      }
  }
  const Layout l = layout_for(a.N, nblk, nst, kStageBytes);
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
  if (geo.smem > kSmemMax || geo.stages < 1 || geo.stages > kMaxStages || geo.ctas_per_sm < 1)
    return cudaErrorInvalidConfiguration;
  int sms = 0;
  cudaError_t e = a.dtype == DCD_BF16 ? prepare_kernel<__nv_bfloat16>(&sms) : prepare_kernel<float>(&sms);
  if (e != cudaSuccess) return e;
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  SParams sp;
  sp.a = a;
  sp.nst = geo.stages;
  sp.tok_a = tokens_a(es);
  sp.tok_r = tokens_r(es);
  sp.bulk = geo.bulk;
  sp.nblk = static_cast<int>((a.V + kRaceBlock - 1) / kRaceBlock);
  const Layout l = layout_for(a.N, sp.nblk, sp.nst, kStageBytes);
  sp.meta_offset = l.meta_offset;
  sp.blk_offset = l.blk_offset;
  sp.stage_offset = l.stage_offset;
  sp.work = a.err + 1;  // header word 1
  // the device error word and the work counter start every call at zero
  e = cudaMemsetAsync(a.err, 0, 2 * sizeof(uint32_t), stream);
  if (e != cudaSuccess) return e;
  int64_t grid = static_cast<int64_t>(sms) * geo.ctas_per_sm;
  if (grid > R) grid = R;
  if (grid < 1) grid = 1;
  if (a.dtype == DCD_BF16)
    score_rows_kernel<__nv_bfloat16><<<static_cast<unsigned>(grid), kThreads, geo.smem, stream>>>(sp);
  else
    score_rows_kernel<float><<<static_cast<unsigned>(grid), kThreads, geo.smem, stream>>>(sp);
  return cudaGetLastError();
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
