// dcd_device.cuh -- device helpers shared by the library's CUDA kernels (not by the oracle):
// PTX wrappers for mbarriers, L2 cache policies and bulk asynchronous copies; fast exp2/log2;
// Philox4x32-10; shared-memory element access; warp and block reductions.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <climits>

namespace dcd {
namespace dev {

constexpr int kThreads = 256;  // compute threads per CTA of every row kernel (the consumers of a
                               // warp-specialised CTA)
constexpr int kWarps = kThreads / 32;
constexpr int kRaceBlock = 1024;                  // tokens per block of the two-level terminal race
constexpr int kSub = 256;                         // tokens a warp handles at once (8 a lane)
#ifndef DCD_WAIT_CYCLES
#define DCD_WAIT_CYCLES 4000000000ll
#endif
constexpr long long kWaitCycles = DCD_WAIT_CYCLES;  // bounded waits: about two seconds at the boost clock
constexpr float kLog2e = 1.4426950408889634f;

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

__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ uint64_t l2_policy_evict_normal() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
      "%4;" ::"r"(smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

// Ticket counter: an atomic add with acquire-release semantics at GPU scope, so that writes made
// before it are visible to whoever draws a later ticket, and that one sees them after its own.
__device__ __forceinline__ uint32_t atomic_add_acq_rel(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
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

// The same 8 tokens as four fp32 pairs (operands of the packed fp32x2 instructions).
__device__ __forceinline__ void ld8x2(const float* p, float2 v[4]) {
  const float4 a = reinterpret_cast<const float4*>(p)[0];
  const float4 b = reinterpret_cast<const float4*>(p)[1];
  v[0] = make_float2(a.x, a.y);
  v[1] = make_float2(a.z, a.w);
  v[2] = make_float2(b.x, b.y);
  v[3] = make_float2(b.z, b.w);
}

__device__ __forceinline__ void ld8x2(const __nv_bfloat16* p, float2 v[4]) {
  const uint4 a = *reinterpret_cast<const uint4*>(p);
  v[0] = make_float2(__uint_as_float(a.x << 16), __uint_as_float(a.x & 0xffff0000u));
  v[1] = make_float2(__uint_as_float(a.y << 16), __uint_as_float(a.y & 0xffff0000u));
  v[2] = make_float2(__uint_as_float(a.z << 16), __uint_as_float(a.z & 0xffff0000u));
  v[3] = make_float2(__uint_as_float(a.w << 16), __uint_as_float(a.w & 0xffff0000u));
}

// max(a, b, c) in one instruction (NaN operands are ignored, as by fmaxf).
__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

__device__ __forceinline__ float max8(const float u[8]) {
  return fmaxf(max3(max3(u[0], u[1], u[2]), u[3], u[4]), max3(u[5], u[6], u[7]));
}

__device__ __forceinline__ float ld1(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float ld1(const __nv_bfloat16* p, int64_t i) { return __bfloat162float(p[i]); }

// ------------------------------------------------------------------------------------------
// Reductions.  A block reduction synchronises the threads that take part in it: the whole CTA
// (SyncCta), or the kThreads consumer threads of a warp-specialised CTA, whose producer warp
// does not take part (SyncConsumers, named barrier 1).
struct SyncCta {
  __device__ __forceinline__ void operator()() const { __syncthreads(); }
};
template <int NT>
struct SyncConsumersN {
  __device__ __forceinline__ void operator()() const {
    asm volatile("bar.sync 1, %0;" ::"n"(NT) : "memory");
  }
};
using SyncConsumers = SyncConsumersN<kThreads>;

// Warps taking part in a block reduction: the whole CTA's kWarps, or a SyncConsumersN group's.
template <typename Sync>
struct SyncWarps {
  static constexpr int value = kWarps;
};
template <int NT>
struct SyncWarps<SyncConsumersN<NT>> {
  static constexpr int value = NT / 32;
};

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
template <typename Sync = SyncCta>
__device__ __forceinline__ void block_argmax(float& v, int& i, float* redf, int* redi, Sync sync = Sync()) {
  warp_argmax(v, i);
  if ((threadIdx.x & 31) == 0) {
    redf[threadIdx.x >> 5] = v;
    redi[threadIdx.x >> 5] = i;
  }
  sync();
  v = redf[0];
  i = redi[0];
#pragma unroll
  for (int w = 1; w < SyncWarps<Sync>::value; ++w) argmax_merge(v, i, redf[w], redi[w]);
  sync();
}

template <typename Sync = SyncCta>
__device__ __forceinline__ float block_sum(float v, float* redf, Sync sync = Sync()) {
  v = warp_sum(v);
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = v;
  sync();
  float s = 0.f;
#pragma unroll
  for (int w = 0; w < SyncWarps<Sync>::value; ++w) s += redf[w];
  sync();
  return s;
}

// Merges (max m, sum s of 2^(x - m), argmax) of two ranges in log2 units (ties to the lower index).
__device__ __forceinline__ void stats_merge(float& m1, float& s1, int& a1, float m2, float s2, int a2) {
  const float M = fmaxf(m1, m2);
  const float t1 = m1 > -INFINITY ? s1 * ex2(m1 - M) : 0.f;
  const float t2 = m2 > -INFINITY ? s2 * ex2(m2 - M) : 0.f;
  if (m2 > m1 || (m2 == m1 && a2 < a1)) a1 = a2;
  m1 = M;
  s1 = t1 + t2;
}

// The same over the 32 lanes of a warp: every lane gets the warp's max, rescaled sum and argmax.
__device__ __forceinline__ void warp_stats(float& m, float& s, int& arg) {
#pragma unroll
  for (int o = 16; o; o >>= 1)
    stats_merge(m, s, arg, __shfl_xor_sync(~0u, m, o), __shfl_xor_sync(~0u, s, o), __shfl_xor_sync(~0u, arg, o));
}

// Combines per-thread (max m, sum s of 2^(x - m), argmax) over the block in log2 units: every
// thread gets the block max, the sum rescaled to it, and the argmax (ties to the lowest index).
template <typename Sync = SyncCta>
__device__ __forceinline__ void block_stats(float& m, float& s, int& arg, float* redf, int* redi, Sync sync = Sync()) {
  auto merge = [](float& m1, float& s1, int& a1, float m2, float s2, int a2) {
    const float M = fmaxf(m1, m2);
    const float t1 = m1 > -INFINITY ? s1 * ex2(m1 - M) : 0.f;
    const float t2 = m2 > -INFINITY ? s2 * ex2(m2 - M) : 0.f;
    if (m2 > m1 || (m2 == m1 && a2 < a1)) a1 = a2;
    m1 = M;
    s1 = t1 + t2;
  };
#pragma unroll
  for (int o = 16; o; o >>= 1)
    merge(m, s, arg, __shfl_xor_sync(~0u, m, o), __shfl_xor_sync(~0u, s, o), __shfl_xor_sync(~0u, arg, o));
  constexpr int NW = SyncWarps<Sync>::value;  // redf holds 2 * NW values (at least 32 floats)
  static_assert(2 * NW <= 64, "reduction scratch");
  if ((threadIdx.x & 31) == 0) {
    redf[threadIdx.x >> 5] = m;
    redf[NW + (threadIdx.x >> 5)] = s;
    redi[threadIdx.x >> 5] = arg;
  }
  sync();
  m = redf[0];
  s = redf[NW];
  arg = redi[0];
#pragma unroll
  for (int w = 1; w < NW; ++w) merge(m, s, arg, redf[w], redf[NW + w], redi[w]);
  sync();
}

template <typename Sync = SyncCta>
__device__ __forceinline__ float block_max(float v, float* redf, Sync sync = Sync()) {
  v = warp_max(v);
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = v;
  sync();
  float s = -INFINITY;
#pragma unroll
  for (int w = 0; w < SyncWarps<Sync>::value; ++w) s = fmaxf(s, redf[w]);
  sync();
  return s;
}


// ------------------------------------------------------------------------------------------
// In-place fp32 values over a staged (z_p, z_q) slice: for fp32 input a token's value takes its
// z_p slot; for bf16 input its low half goes to the token's z_p slot and its high half to its z_q
// slot, so no token's slots are shared with another's.
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

__device__ __forceinline__ void ld8_value(const float* zp, const float* /*zq*/, int i0, float v[8]) { ld8(zp + i0, v); }

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

}  // namespace dev
}  // namespace dcd
