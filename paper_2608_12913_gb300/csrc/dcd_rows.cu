// dcd_rows.cu -- the streaming kernels of the CD verification step on sm_103a.
//
// score_rows_kernel: one thread-block cluster per tree-node row g = b * N + n.  The
//   row's vocabulary is split into `cluster` contiguous slices (whole blocks of 256
//   tokens); each CTA stages its slice of z_p, z_q (and q for sampled non-leaf rows)
//   in shared memory with bulk asynchronous copies, so HBM is read exactly once per
//   row however many passes the row needs.  Passes over shared memory compute, in
//   order: the expert max (only when beta > 0, for the plausibility set of Sec. 2.1),
//   the CD score s' = (1 + alpha) z_p - alpha z_q with its max and argmax (Eq. 1; the
//   two log-softmax shifts are constant per row and cancel in the normaliser), stored
//   in place; the normaliser sum exp((s' - max) / T); then for sampled rows the
//   sibling-rejection chain of Algorithm 1 (one residual pass per rejected child,
//   r_j = max(0, r_{j-1} - q) / Z_j, in place) and the terminal draw, a two-level
//   exponential race (a 256-token block by its mass, then a token of that block).
//   Per-CTA partials are combined across the cluster through distributed shared
//   memory; every CTA combines them in the same order, so all CTAs take identical
//   decisions and run the same number of cluster barriers.
// tree_walk_kernel: one thread per sequence follows the accepted children.
// terminal_residual_kernel: one block per sequence rebuilds the distribution its
//   bonus token was drawn from (test output only).

#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>
#include <mutex>

#include "dcd.h"
#include "dcd_internal.h"

namespace cg = cooperative_groups;

namespace dcd {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxCluster = 16;
constexpr size_t kSmemBudget = 64 * 1024 + 1024;  // data bytes per CTA the automatic geometry aims for
constexpr size_t kSmemMax = 227 * 1024;
constexpr long long kWaitCycles = 4000000000ll;  // about two seconds at the boost clock
constexpr int kRaceBlock = 256;                  // tokens per block of the two-level terminal race
constexpr float kLog2e = 1.4426950408889634f;

// ------------------------------------------------------------------------------------------
// PTX wrappers: mbarrier and bulk asynchronous global->shared copies.
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

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(smem_addr(bar))
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

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
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

// 32-bit word -> uniform in (0, 1): ((w >> 9) + 1/2) 2^-23, exact in fp32.
__device__ __forceinline__ float u01(uint32_t w) {
  return (__uint2float_rn(w >> 9) + 0.5f) * 1.1920928955078125e-07f;
}

__device__ __forceinline__ float accept_uniform(uint64_t seed, uint64_t off, uint32_t G) {
  const uint4 w = philox4x32_10(make_uint4(G, 0u, (uint32_t)off, (uint32_t)(off >> 32)), (uint32_t)seed,
                                (uint32_t)(seed >> 32));
  return u01(w.x);
}

// ------------------------------------------------------------------------------------------
// Shared-memory element access.  Slices are read 8 tokens at a time (16 B of bf16 or 32 B of
// fp32).  Sampled rows overwrite their logits in place with fp32 values: for fp32 input the
// value takes the z_p slot; for bf16 input its low half goes to the z_p slot and its high
// half to the z_q slot of the same token, so no token's slots are shared with another's.
__device__ __forceinline__ void lds8(const float* p, float v[8]) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ void lds8(const __nv_bfloat16* p, float v[8]) {
  const uint4 a = *reinterpret_cast<const uint4*>(p);
  v[0] = __uint_as_float(a.x << 16); v[1] = __uint_as_float(a.x & 0xffff0000u);
  v[2] = __uint_as_float(a.y << 16); v[3] = __uint_as_float(a.y & 0xffff0000u);
  v[4] = __uint_as_float(a.z << 16); v[5] = __uint_as_float(a.z & 0xffff0000u);
  v[6] = __uint_as_float(a.w << 16); v[7] = __uint_as_float(a.w & 0xffff0000u);
}

__device__ __forceinline__ void st8_value(float* zp, float* /*zq*/, int i0, const float v[8]) {
  reinterpret_cast<float4*>(zp + i0)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(zp + i0)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

__device__ __forceinline__ void st8_value(__nv_bfloat16* zp, __nv_bfloat16* zq, int i0, const float v[8]) {
  uint32_t w[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) w[e] = __float_as_uint(v[e]);
  *reinterpret_cast<uint4*>(zp + i0) = make_uint4(__byte_perm(w[0], w[1], 0x5410), __byte_perm(w[2], w[3], 0x5410),
                                                 __byte_perm(w[4], w[5], 0x5410), __byte_perm(w[6], w[7], 0x5410));
  *reinterpret_cast<uint4*>(zq + i0) = make_uint4(__byte_perm(w[0], w[1], 0x7632), __byte_perm(w[2], w[3], 0x7632),
                                                 __byte_perm(w[4], w[5], 0x7632), __byte_perm(w[6], w[7], 0x7632));
}

__device__ __forceinline__ void ld8_value(const float* zp, const float* /*zq*/, int i0, float v[8]) {
  lds8(zp + i0, v);
}

__device__ __forceinline__ void ld8_value(const __nv_bfloat16* zp, const __nv_bfloat16* zq, int i0, float v[8]) {
  const uint4 lo = *reinterpret_cast<const uint4*>(zp + i0);
  const uint4 hi = *reinterpret_cast<const uint4*>(zq + i0);
  const uint32_t l[4] = {lo.x, lo.y, lo.z, lo.w}, h[4] = {hi.x, hi.y, hi.z, hi.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    v[2 * k] = __uint_as_float(__byte_perm(l[k], h[k], 0x5410));
    v[2 * k + 1] = __uint_as_float(__byte_perm(l[k], h[k], 0x7632));
  }
}

__device__ __forceinline__ float ld1_value(const float* zp, const float* /*zq*/, int i) { return zp[i]; }

__device__ __forceinline__ float ld1_value(const __nv_bfloat16* zp, const __nv_bfloat16* zq, int i) {
  const uint32_t lo = reinterpret_cast<const uint16_t*>(zp)[i];
  const uint32_t hi = reinterpret_cast<const uint16_t*>(zq)[i];
  return __uint_as_float((hi << 16) | lo);
}

// ------------------------------------------------------------------------------------------
// Block reductions (every thread gets the result).
__device__ __forceinline__ void argmax_merge(float& v, int& i, float v2, int i2) {
  if (v2 > v || (v2 == v && i2 < i)) {
    v = v2;
    i = i2;
  }
}

__device__ __forceinline__ void block_argmax(float& v, int& i, float* redf, int* redi) {
#pragma unroll
  for (int o = 16; o; o >>= 1) argmax_merge(v, i, __shfl_xor_sync(~0u, v, o), __shfl_xor_sync(~0u, i, o));
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
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(~0u, v, o);
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = v;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) s += redf[w];
  __syncthreads();
  return s;
}

__device__ __forceinline__ float block_max(float v, float* redf) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(~0u, v, o));
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = v;
  __syncthreads();
  float s = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) s = fmaxf(s, redf[w]);
  __syncthreads();
  return s;
}

// ------------------------------------------------------------------------------------------
// Cluster exchange: each CTA publishes one Partial; after the cluster barrier every CTA
// gathers all of them from distributed shared memory.  Partial slots alternate between two
// buffers: a CTA rewrites a buffer only after the next barrier, which its peers pass only
// once they have finished reading it.
struct Partial {
  float m;          // max (score or race key)
  float s;          // sum
  int32_t arg;      // token id attaining m
  float cap_r;      // value captured at the next candidate token (owner CTA only)
  float cap_q;      // q at that token (owner CTA only)
  int32_t cap_own;  // 1 in the CTA whose slice holds the candidate token
  uint32_t status;  // DCD_DEVERR_* bits
  int32_t pad;
};

__device__ __forceinline__ Partial neutral_partial() {
  Partial p;
  p.m = -INFINITY;
  p.s = 0.f;
  p.arg = INT_MAX;
  p.cap_r = 0.f;
  p.cap_q = 0.f;
  p.cap_own = 0;
  p.status = 0u;
  p.pad = 0;
  return p;
}

__device__ __forceinline__ void cluster_exchange(cg::cluster_group& cl, Partial* part, Partial* gath, int& stage,
                                                 const Partial& mine, int C) {
  Partial* slot = &part[stage & 1];
  ++stage;
  if (threadIdx.x == 0) *slot = mine;
  cl.sync();
  if (threadIdx.x < C) gath[threadIdx.x] = *cl.map_shared_rank(slot, threadIdx.x);
  __syncthreads();
}

struct KParams {
  ScoreArgs a;
  int32_t cluster;
  int32_t chunk;   // tokens per CTA (multiple of kRaceBlock)
  int32_t bulk;    // 1: bulk asynchronous copies, 0: plain loads
  int32_t data_offset;
};

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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(~0u, v, o);
  return v;
}

// log2 of a Gumbel-race divisor: key = log2 r - log2(-log2 u) orders tokens exactly as
// ln r - ln(-ln u) does (the two differ by a positive factor and a constant).
__device__ __forceinline__ float race_key(float log2_mass, uint32_t word) {
  return log2_mass - lg2(-lg2(u01(word)));
}

__device__ __forceinline__ uint32_t philox_word(uint64_t seed, uint64_t off, uint32_t c0, uint32_t c1, int word) {
  const uint4 w = philox4x32_10(make_uint4(c0, c1, (uint32_t)off, (uint32_t)(off >> 32)), (uint32_t)seed,
                                (uint32_t)(seed >> 32));
  return word == 0 ? w.x : word == 1 ? w.y : word == 2 ? w.z : w.w;
}

// ------------------------------------------------------------------------------------------
template <typename TIn>
__global__ void __launch_bounds__(kThreads) score_rows_kernel(const __grid_constant__ KParams kp) {
  const ScoreArgs& p = kp.a;
  cg::cluster_group cl = cg::this_cluster();
  const int C = kp.cluster;
  const int rank = static_cast<int>(cl.block_rank());
  const int64_t g = static_cast<int64_t>(blockIdx.x) / C;
  const int N = p.N;
  const int b = static_cast<int>(g / N), n = static_cast<int>(g % N);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem);
  Partial* part = reinterpret_cast<Partial*>(smem + 16);
  Partial* gath = part + 2;
  float* redf = reinterpret_cast<float*>(gath + kMaxCluster);
  int* redi = reinterpret_cast<int*>(redf + 32);
  int* meta = redi + 32;  // [0] child count, [1] status bits
  int* kids = meta + 8;
  int* ktok = kids + N;
  float* ksv = reinterpret_cast<float*>(ktok + N);
  float* blk = ksv + N;  // per 256-token block masses of this slice
  TIn* zp_s = reinterpret_cast<TIn*>(smem + kp.data_offset);
  TIn* zq_s = zp_s + kp.chunk;
  float* q_s = reinterpret_cast<float*>(zq_s + kp.chunk);

  const int64_t lo = static_cast<int64_t>(rank) * kp.chunk;
  const int64_t hi = lo + kp.chunk < p.V ? lo + kp.chunk : p.V;
  const int len = hi > lo ? static_cast<int>(hi - lo) : 0;
  const TIn* zp_g = static_cast<const TIn*>(p.zp) + g * p.ld + lo;
  const TIn* zq_g = static_cast<const TIn*>(p.zq) + g * p.ld + lo;

  const float alpha = p.alpha[b];
  const float beta = p.beta ? p.beta[b] : 0.f;
  const float T = p.temp ? p.temp[b] : 0.f;
  const bool sampled = T > 0.f;
  const float invT = sampled ? 1.f / T : 1.f;
  const float k2 = kLog2e * invT;  // exp(x / T) = 2^(x * k2)

  if (g == 0 && rank == 0 && tid == 0) *p.err = 0u;

  // ---- stage the slice: bulk copies of z_p / z_q first, q once the children are known
  const uint32_t zbulk = kp.bulk ? static_cast<uint32_t>((len * static_cast<int>(sizeof(TIn))) & ~15) : 0u;
  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    if (zbulk) {
      mbar_expect_tx(bar, 2u * zbulk);
      bulk_g2s(zp_s, zp_g, zbulk, bar);
      bulk_g2s(zq_s, zq_g, zbulk, bar);
    }
  }
  if (warp == 0) {
    // children of node n in ascending id, and the checks of this row's own node
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
        if (t < 0 || t >= p.V) st |= DCD_DEVERR_BAD_TOKEN;
      }
      if (!(alpha >= 0.f && alpha <= 3.0e38f) || !(beta >= 0.f && beta <= 1.f) || !(T >= 0.f && T <= 3.0e38f))
        st |= DCD_DEVERR_BAD_PARAM;
      meta[0] = count;
      meta[1] = static_cast<int>(st);
    }
  }
  __syncthreads();
  const int m = meta[0];
  const bool need_q = sampled && m > 0 && p.q != nullptr;
  const float* q_g = need_q ? p.q + g * p.ldq + lo : nullptr;
  const uint32_t qbulk = (kp.bulk && need_q) ? static_cast<uint32_t>((len * 4) & ~15) : 0u;
  if (tid == 0) {
    if (qbulk) {
      mbar_expect_tx(bar, qbulk);
      bulk_g2s(q_s, q_g, qbulk, bar);
    }
    mbar_arrive(bar);
  }
  {  // plain loads: the whole slice without bulk copies, else only the ragged tail
    const int zfirst = static_cast<int>(zbulk / sizeof(TIn));
    for (int i = zfirst + tid; i < len; i += kThreads) {
      zp_s[i] = zp_g[i];
      zq_s[i] = zq_g[i];
    }
    if (need_q) {
      const int qfirst = static_cast<int>(qbulk / 4);
      for (int i = qfirst + tid; i < len; i += kThreads) q_s[i] = q_g[i];
    }
  }
  if (!mbar_wait_bounded(bar, 0)) {
    atomicOr(reinterpret_cast<unsigned*>(&meta[1]), DCD_DEVERR_TIMEOUT);
    mbar_wait_bounded(bar, 0);  // give copies still in flight a second bounded chance
  }
  __syncthreads();

  // Loops run over 8-token groups; a warp's 32 groups are one 256-token race block, and the
  // group count is rounded up to whole warps so every branch on `grp < ngw` is warp-uniform.
  const int ngw = (((len + 7) >> 3) + 31) & ~31;
  const bool masked = beta > 0.f;
  const float logb = masked ? logf(beta) : -INFINITY;
  const float c1 = 1.f + alpha;
  int stage = 0;
  Partial mine = neutral_partial();
  uint32_t status = 0u;

  // ---- pass A (beta > 0): the expert max, for P_beta = {x : z_p(x) - max z_p >= log beta}
  float Mp = 0.f;
  if (masked) {
    float lm = -INFINITY;
    for (int base = 0; base < ngw; base += kThreads) {
      const int grp = base + tid;
      if (grp >= ngw) continue;
      const int i0 = grp << 3;
      float zp[8];
      lds8(zp_s + i0, zp);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        if (i0 + e < len) lm = fmaxf(lm, zp[e]);
    }
    lm = block_max(lm, redf);
    mine.m = lm;
    cluster_exchange(cl, part, gath, stage, mine, C);
    Mp = -INFINITY;
    for (int k = 0; k < C; ++k) Mp = fmaxf(Mp, gath[k].m);
  }

  // ---- pass B: CD score s' = (1 + alpha) z_p - alpha z_q on P_beta (-inf elsewhere), its max and
  // argmax; s' overwrites the slice in place as fp32
  float best = -INFINITY;
  int barg = INT_MAX;
  for (int base = 0; base < ngw; base += kThreads) {
    const int grp = base + tid;
    if (grp >= ngw) continue;
    const int i0 = grp << 3;
    float zp[8], zq[8], sv[8];
    lds8(zp_s + i0, zp);
    lds8(zq_s + i0, zq);
    float gm = -INFINITY;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const bool in = (i0 + e < len) && (!masked || (zp[e] - Mp >= logb));
      sv[e] = in ? fmaf(c1, zp[e], -alpha * zq[e]) : -INFINITY;
      gm = fmaxf(gm, sv[e]);
    }
    if (gm > best) {
      best = gm;
#pragma unroll
      for (int e = 7; e >= 0; --e)
        if (sv[e] == gm) barg = static_cast<int>(lo) + i0 + e;
    }
    st8_value(zp_s, zq_s, i0, sv);
  }
  block_argmax(best, barg, redf, redi);  // ends with __syncthreads: every s' is stored
  const float m_cta = best;
  // children's scores, read by the CTA whose slice holds the token
  for (int k = tid; k < m; k += kThreads) {
    const int t = ktok[k];
    if (t >= lo && t < hi) ksv[k] = ld1_value(zp_s, zq_s, t - static_cast<int>(lo));
  }
  __syncthreads();  // the captures above finish before pass C rewrites the slice

  // ---- pass C: normaliser sum 2^((s' - m_cta) k2); sampled rows keep e(x) in place, and leaf rows
  // (whose terminal draw races over pi_CD itself) keep the 256-token block masses
  const bool leaf_race = sampled && m == 0;
  float ssum = 0.f;
  if (m_cta > -INFINITY) {
    const float mk2 = m_cta * k2;
    for (int base = 0; base < ngw; base += kThreads) {
      const int grp = base + tid;
      if (grp >= ngw) continue;
      const int i0 = grp << 3;
      float sv[8];
      ld8_value(zp_s, zq_s, i0, sv);
      float part = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        sv[e] = ex2(fmaf(sv[e], k2, -mk2));
        part += sv[e];
      }
      ssum += part;
      if (sampled) st8_value(zp_s, zq_s, i0, sv);
      if (leaf_race) {
        const float bs = warp_sum(part);
        if (lane == 0) blk[grp >> 5] = bs;
      }
    }
  } else if (sampled) {
    const float zero[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int grp = tid; grp < ngw; grp += kThreads) st8_value(zp_s, zq_s, grp << 3, zero);
    for (int t = tid; t < (ngw >> 5); t += kThreads) blk[t] = 0.f;
  }
  const float s_cta = block_sum(ssum, redf);  // ends with __syncthreads

  mine = neutral_partial();
  mine.m = m_cta;
  mine.s = s_cta;
  mine.arg = barg;
  if (sampled && m > 0 && tid == 0) {
    const int t = ktok[0];
    if (t >= lo && t < hi) {
      mine.cap_own = 1;
      mine.cap_r = ld1_value(zp_s, zq_s, t - static_cast<int>(lo));
      mine.cap_q = q_s[t - static_cast<int>(lo)];
    }
  }
  if (tid == 0) mine.status = static_cast<uint32_t>(meta[1]);
  cluster_exchange(cl, part, gath, stage, mine, C);

  float M = -INFINITY;
  for (int k = 0; k < C; ++k) M = fmaxf(M, gath[k].m);
  int arg = INT_MAX;
  float S = 0.f;
  float rt = 0.f, qt = 0.f;
  for (int k = 0; k < C; ++k) {
    status |= gath[k].status;
    if (gath[k].m == M && arg == INT_MAX) arg = gath[k].arg;
    if (gath[k].m > -INFINITY) S += gath[k].s * exp2f((gath[k].m - M) * k2);
  }
  if (!(M > -INFINITY && M < INFINITY) || !(S > 0.f && S < INFINITY)) status |= DCD_DEVERR_NONFINITE;
  for (int k = 0; k < C; ++k)
    if (gath[k].cap_own) {
      rt = gath[k].cap_r * (exp2f((gath[k].m - M) * k2) / S);
      qt = gath[k].cap_q;
    }
  const float logS = logf(S);

  // ---- outputs of the Eq. 1 target
  if (rank == 0 && tid == 0) {
    if (p.cd_argmax) p.cd_argmax[g] = arg;
    if (p.cd_lse) p.cd_lse[g] = M * invT + logS;
    if (n == 0 && p.cd_logprob) p.cd_logprob[g] = 0.f;
  }
  if (p.cd_logprob) {
    for (int k = tid; k < m; k += kThreads) {
      const int t = ktok[k];
      if (t >= lo && t < hi)
        p.cd_logprob[static_cast<int64_t>(b) * N + kids[k]] =
            ksv[k] > -INFINITY ? (ksv[k] - M) * invT - logS : -INFINITY;
    }
  }

  int acc = -1, term = -1;
  if (!sampled) {
    // ---- greedy rule
    for (int k = 0; k < m; ++k)
      if (ktok[k] == arg) {
        acc = kids[k];
        break;
      }
    if (acc < 0) term = arg;
  } else {
    // ---- sampled rule: sibling-rejection chain over the slice, then the terminal race if needed
    const float scale_me = m_cta > -INFINITY ? exp2f((m_cta - M) * k2) / S : 0.f;
    float invZ = 0.f;
    bool degen = false;
    for (int j = 0; j < m; ++j) {
      const uint32_t G = static_cast<uint32_t>(static_cast<int64_t>(b) * N + kids[j]);
      const float u = accept_uniform(p.seed, p.offset, G);
      const float ratio = qt > 0.f ? rt / qt : (rt > 0.f ? INFINITY : 0.f);
      if (u <= ratio) {
        acc = kids[j];
        break;
      }
      // rejected: r_{j+1} = max(0, r_j - q) / Z, written over the slice; the last residual also
      // records its block masses for the terminal race
      const bool last = j == m - 1;
      float zsum = 0.f;
      for (int base = 0; base < ngw; base += kThreads) {
        const int grp = base + tid;
        if (grp >= ngw) continue;
        const int i0 = grp << 3;
        float r[8], qv[8];
        ld8_value(zp_s, zq_s, i0, r);
        lds8(q_s + i0, qv);
        float part = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float prev = j == 0 ? r[e] * scale_me : (degen ? qv[e] : r[e] * invZ);
          const float nv = (i0 + e < len) ? fmaxf(prev - qv[e], 0.f) : 0.f;
          r[e] = nv;
          part += nv;
        }
        st8_value(zp_s, zq_s, i0, r);
        zsum += part;
        if (last) {
          const float bs = warp_sum(part);
          if (lane == 0) blk[grp >> 5] = bs;
        }
      }
      zsum = block_sum(zsum, redf);
      mine = neutral_partial();
      mine.s = zsum;
      if (tid == 0 && j + 1 < m) {
        const int t = ktok[j + 1];
        if (t >= lo && t < hi) {
          mine.cap_own = 1;
          mine.cap_r = ld1_value(zp_s, zq_s, t - static_cast<int>(lo));
          mine.cap_q = q_s[t - static_cast<int>(lo)];
        }
      }
      cluster_exchange(cl, part, gath, stage, mine, C);
      float Z = 0.f, cr = 0.f, cq = 0.f;
      for (int k = 0; k < C; ++k) {
        Z += gath[k].s;
        if (gath[k].cap_own) {
          cr = gath[k].cap_r;
          cq = gath[k].cap_q;
        }
      }
      if (Z > 0.f) {
        degen = false;
        invZ = 1.f / Z;
        rt = cr * invZ;
      } else {
        degen = true;  // r_j == q in exact arithmetic when nothing is left
        rt = cq;
      }
      qt = cq;
    }
    if (acc < 0) {
      // ---- terminal draw: two-level exponential race (block of 256 tokens, then a token)
      if (degen) {  // the residual is q itself: its block masses
        for (int base = 0; base < ngw; base += kThreads) {
          const int grp = base + tid;
          if (grp >= ngw) continue;
          const int i0 = grp << 3;
          float qv[8];
          lds8(q_s + i0, qv);
          float part = 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) part += (i0 + e < len) ? qv[e] : 0.f;
          const float bs = warp_sum(part);
          if (lane == 0) blk[grp >> 5] = bs;
        }
        __syncthreads();
      }
      // leaf rows hold e(x) relative to this CTA's max; bring block masses to the common scale
      const float offset2 = leaf_race ? (m_cta - M) * k2 : 0.f;
      const int nblk = (len + kRaceBlock - 1) / kRaceBlock;
      const int kbase = static_cast<int>(lo / kRaceBlock);
      float bk = -INFINITY;
      int bb = INT_MAX;
      for (int t = tid; t < nblk; t += kThreads) {
        const float R = blk[t];
        if (R > 0.f) {
          const uint32_t kabs = static_cast<uint32_t>(kbase + t);
          const float key = race_key(lg2(R) + offset2,
                                     philox_word(p.seed, p.offset, static_cast<uint32_t>(g),
                                                 0x80000000u | (kabs >> 2), static_cast<int>(kabs & 3)));
          if (key > bk) {
            bk = key;
            bb = static_cast<int>(kabs);
          }
        }
      }
      block_argmax(bk, bb, redf, redi);
      mine = neutral_partial();
      mine.m = bk;
      mine.arg = bb;
      cluster_exchange(cl, part, gath, stage, mine, C);
      float K = -INFINITY;
      int kstar = INT_MAX;
      for (int k = 0; k < C; ++k) argmax_merge(K, kstar, gath[k].m, gath[k].arg);
      // token race inside block kstar, by the CTA whose slice holds it (one warp, 8 tokens a lane)
      mine = neutral_partial();
      const int64_t x_first = static_cast<int64_t>(kstar) * kRaceBlock;
      if (kstar != INT_MAX && x_first >= lo && x_first < hi && warp == 0) {
        const int i0 = static_cast<int>(x_first - lo) + lane * 8;
        float r[8], qv[8];
        ld8_value(zp_s, zq_s, i0, r);
        if (degen) lds8(q_s + i0, qv);
        const uint32_t x0 = static_cast<uint32_t>(x_first) + static_cast<uint32_t>(lane * 8);
        const uint32_t o0 = static_cast<uint32_t>(p.offset), o1 = static_cast<uint32_t>(p.offset >> 32);
        const uint32_t s0 = static_cast<uint32_t>(p.seed), s1 = static_cast<uint32_t>(p.seed >> 32);
        const uint4 wa = philox4x32_10(make_uint4(static_cast<uint32_t>(g), 1u + (x0 >> 2), o0, o1), s0, s1);
        const uint4 wb = philox4x32_10(make_uint4(static_cast<uint32_t>(g), 2u + (x0 >> 2), o0, o1), s0, s1);
        const uint32_t w[8] = {wa.x, wa.y, wa.z, wa.w, wb.x, wb.y, wb.z, wb.w};
        float tk = -INFINITY;
        int tx = INT_MAX;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float v = degen ? qv[e] : r[e];
          if (i0 + e < len && v > 0.f) {
            const float key = race_key(lg2(v), w[e]);
            if (key > tk) {
              tk = key;
              tx = static_cast<int>(x0) + e;
            }
          }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) argmax_merge(tk, tx, __shfl_xor_sync(~0u, tk, o), __shfl_xor_sync(~0u, tx, o));
        if (lane == 0) {
          mine.m = tk;
          mine.arg = tx;
          mine.cap_own = 1;
        }
      }
      cluster_exchange(cl, part, gath, stage, mine, C);
      for (int k = 0; k < C; ++k)
        if (gath[k].cap_own) term = gath[k].arg;
    }
  }

  if (rank == 0 && tid == 0) {
    RowRecord r;
    r.acc_child = acc;
    r.term_token = acc < 0 ? term : -1;
    r.status = status;
    r.reserved = 0;
    p.rec[g] = r;
  }
  cl.sync();  // no CTA leaves while a peer may still read its partial slots
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
  auto ld = [](const TIn* a, int64_t i) -> float {
    if constexpr (sizeof(TIn) == 2) {
      return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(a)[i]);
    } else {
      return static_cast<float>(reinterpret_cast<const float*>(a)[i]);
    }
  };
  float Mp = 0.f;
  if (masked) {
    float v = -INFINITY;
    for (int64_t x = threadIdx.x; x < V; x += kThreads) v = fmaxf(v, ld(zp, x));
    Mp = block_max(v, redf);
  }
  float M = -INFINITY;
  for (int64_t x = threadIdx.x; x < V; x += kThreads) {
    const float z = ld(zp, x);
    if (!masked || z - Mp >= logb) M = fmaxf(M, fmaf(c1, z, -alpha * ld(zq, x)));
  }
  M = block_max(M, redf);
  float s = 0.f;
  for (int64_t x = threadIdx.x; x < V; x += kThreads) {
    const float z = ld(zp, x);
    const float e = (!masked || z - Mp >= logb) ? expf((fmaf(c1, z, -alpha * ld(zq, x)) - M) * invT) : 0.f;
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
template <typename TIn>
cudaError_t prepare_kernel_attributes() {
  static std::once_flag once[64];
  static cudaError_t result[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::call_once(once[dev], [&] {
    cudaError_t r = cudaFuncSetAttribute(score_rows_kernel<TIn>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kSmemMax));
    if (r == cudaSuccess) r = cudaFuncSetAttribute(score_rows_kernel<TIn>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    result[dev] = r;
  });
  return result[dev];
}

size_t header_bytes(int N, int64_t chunk) {
  const size_t h = 16 + 2 * sizeof(Partial) + kMaxCluster * sizeof(Partial) + 64 * sizeof(float) + 8 * sizeof(int) +
                   static_cast<size_t>(N) * 12 + static_cast<size_t>(chunk / kRaceBlock) * sizeof(float);
  return (h + 127) & ~static_cast<size_t>(127);
}

}  // namespace

RowGeometry row_geometry(const ScoreArgs& a) {
  RowGeometry geo{};
  const size_t es = a.dtype == DCD_BF16 ? 2 : 4;
  const size_t bpe = 2 * es + (a.q ? 4 : 0);
  auto chunk_for = [&](int c) {  // slices hold whole 256-token race blocks
    const int64_t per = (a.V + c - 1) / c;
    return (per + kRaceBlock - 1) / kRaceBlock * kRaceBlock;
  };
  int C = a.force_cluster;
  if (C <= 0) {
    C = kMaxCluster;
    for (int c = 1; c <= kMaxCluster; c *= 2)
      if (static_cast<size_t>(chunk_for(c)) * bpe <= kSmemBudget) {
        C = c;
        break;
      }
  }
  geo.cluster = C;
  geo.chunk = chunk_for(C);
  geo.smem = header_bytes(a.N, geo.chunk) + static_cast<size_t>(geo.chunk) * bpe;
  auto al16 = [](const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
  geo.bulk = !a.force_plain && al16(a.zp) && al16(a.zq) && (a.ld * static_cast<int64_t>(es)) % 16 == 0 &&
             (!a.q || (al16(a.q) && (a.ldq * 4) % 16 == 0));
  return geo;
}

cudaError_t launch_score_rows(const ScoreArgs& a, cudaStream_t stream) {
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  if (R == 0) return cudaSuccess;
  const RowGeometry geo = row_geometry(a);
  if (geo.smem > kSmemMax || geo.cluster < 1 || geo.cluster > kMaxCluster ||
      (geo.cluster & (geo.cluster - 1)) != 0 || R * geo.cluster > INT_MAX)
    return cudaErrorInvalidConfiguration;
  KParams kp;
  kp.a = a;
  kp.cluster = geo.cluster;
  kp.chunk = static_cast<int32_t>(geo.chunk);
  kp.bulk = geo.bulk;
  kp.data_offset = static_cast<int32_t>(header_bytes(a.N, geo.chunk));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(R * geo.cluster));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = geo.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = geo.cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e;
  if (a.dtype == DCD_BF16) {
    e = prepare_kernel_attributes<__nv_bfloat16>();
    if (e != cudaSuccess) return e;
    e = cudaLaunchKernelEx(&cfg, score_rows_kernel<__nv_bfloat16>, kp);
  } else {
    e = prepare_kernel_attributes<float>();
    if (e != cudaSuccess) return e;
    e = cudaLaunchKernelEx(&cfg, score_rows_kernel<float>, kp);
  }
  return e;
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
