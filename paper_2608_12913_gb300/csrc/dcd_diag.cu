// dcd_diag.cu -- per-row diagnostics of contrastive verification (the signal / proposal-error
// quantities of Sec. 3.1 and the alignment-gap estimator of App. C), one streaming pass over the
// expert's and amateur's logits and, when given, the drafter's distribution q.
//
// For a row with logits z_p, z_q and reference values r_p = z_p(0), r_q = z_q(0) the pass keeps,
// per thread and then per chunk of the vocabulary:
//   m_p, s_p = sum exp(z_p - m_p), t_p = sum exp(z_p - m_p) d   (online max / rescaled sums)
//   m_q, s_q = sum exp(z_q - m_q), t_q = sum exp(z_q - m_q) d,   d = (z_p - r_p) - (z_q - r_q)
//   with q:  a = sum q d,  e1 = sum q,  ez = sum q (z_p - r_p),  h = sum_{q > 0} q log2 q
// and a per-row combine turns them into
//   lse_p, lse_q; signal = |(z_p(x*) - lse_p) - (z_q(x*) - lse_q)|;
//   e_q = E_{pi_q}[log pi_p - log pi_q] = t_q / s_q - (L_p - L_q),
//   kl_pq = D_KL(pi_p || pi_q)          = t_p / s_p - (L_p - L_q),
//   e_e = E_q[log pi_p - log pi_q]      = a - (L_p - L_q) e1,
//   kl  = D_KL(q || pi_p)               = h ln 2 - ez + L_p e1,        L_p = lse_p - r_p, L_q = lse_q - r_q.
// and, given the CD normaliser cd_lse = log sum exp((1 + alpha) z_p - alpha z_q) of a verification
// call with beta = 0 and T = 1, the decomposition lemma of App. B gives
//   kl_pcd = D_KL(pi_p || pi_CD) = log Z_CD - alpha kl_pq,  log Z_CD = cd_lse - (1 + alpha) lse_p + alpha lse_q.
// Shifting by r_p, r_q keeps every linear term at the scale of the logit spread rather than of
// the logits' absolute offset, so fp32 accumulation loses little to cancellation.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

#include "dcd.h"
#include "dcd_device.cuh"
#include "dcd_diag.h"
#include "dcd_internal.h"

namespace dcd {
namespace {

constexpr int kDiagThreads = 256;
constexpr int kDiagWarps = kDiagThreads / 32;
constexpr int kDiagStep = 8 * kDiagThreads;  // tokens one pass of the CTA covers (8 a thread)
constexpr int kDiagCtasPerSm = 4;          // resident CTAs per SM (64 registers a thread)
constexpr float kLn2 = 0.6931471805599453f;

struct Acc {
  float mp, sp, mq, sq, tq, a, e1, ez, h, tp;
};

// Adds tokens with values p[k], z[k] (and q values e[k]) to the accumulator.
template <int K, bool kQ>
__device__ __forceinline__ void accumulate(Acc& c, const float* p, const float* z, const float* e, float rp,
                                           float rq) {
  float lp = p[0], lq = z[0];
#pragma unroll
  for (int k = 1; k < K; ++k) {
    lp = fmaxf(lp, p[k]);
    lq = fmaxf(lq, z[k]);
  }
  if (lp > c.mp) {
    const float f = dev::ex2((c.mp - lp) * dev::kLog2e);
    c.sp *= f;
    c.tp *= f;
    c.mp = lp;
  }
  if (lq > c.mq) {
    const float f = dev::ex2((c.mq - lq) * dev::kLog2e);
    c.sq *= f;
    c.tq *= f;
    c.mq = lq;
  }
  const float mpl = c.mp * dev::kLog2e, mql = c.mq * dev::kLog2e;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    const float pr = p[k] - rp;
    const float d = pr - (z[k] - rq);
    const float wp = dev::ex2(fmaf(p[k], dev::kLog2e, -mpl));
    c.sp += wp;
    c.tp = fmaf(wp, d, c.tp);
    const float w = dev::ex2(fmaf(z[k], dev::kLog2e, -mql));
    c.sq += w;
    c.tq = fmaf(w, d, c.tq);
    if (kQ) {
      const float ek = e[k];
      c.a = fmaf(ek, d, c.a);
      c.e1 += ek;
      c.ez = fmaf(ek, pr, c.ez);
      c.h += ek > 0.f ? ek * dev::lg2(ek) : 0.f;
    }
  }
}

__device__ __forceinline__ void merge(Acc& c, const Acc& o) {
  const float mp = fmaxf(c.mp, o.mp), mq = fmaxf(c.mq, o.mq);
  const float fp = c.mp == mp ? 1.f : dev::ex2((c.mp - mp) * dev::kLog2e);
  const float gp = o.mp == mp ? 1.f : dev::ex2((o.mp - mp) * dev::kLog2e);
  c.sp = c.sp * fp + o.sp * gp;
  c.tp = c.tp * fp + o.tp * gp;
  c.mp = mp;
  const float fq = c.mq == mq ? 1.f : dev::ex2((c.mq - mq) * dev::kLog2e);
  const float gq = o.mq == mq ? 1.f : dev::ex2((o.mq - mq) * dev::kLog2e);
  c.sq = c.sq * fq + o.sq * gq;
  c.tq = c.tq * fq + o.tq * gq;
  c.mq = mq;
  c.a += o.a;
  c.e1 += o.e1;
  c.ez += o.ez;
  c.h += o.h;
}

__device__ __forceinline__ Acc shfl_down(const Acc& c, int off) {
  Acc o;
  o.mp = __shfl_down_sync(0xffffffffu, c.mp, off);
  o.sp = __shfl_down_sync(0xffffffffu, c.sp, off);
  o.mq = __shfl_down_sync(0xffffffffu, c.mq, off);
  o.sq = __shfl_down_sync(0xffffffffu, c.sq, off);
  o.tq = __shfl_down_sync(0xffffffffu, c.tq, off);
  o.a = __shfl_down_sync(0xffffffffu, c.a, off);
  o.e1 = __shfl_down_sync(0xffffffffu, c.e1, off);
  o.ez = __shfl_down_sync(0xffffffffu, c.ez, off);
  o.h = __shfl_down_sync(0xffffffffu, c.h, off);
  o.tp = __shfl_down_sync(0xffffffffu, c.tp, off);
  return o;
}

// 16-byte streaming loads of 8 tokens: read once, so marked evict-first in L1 and L2.
__device__ __forceinline__ void ld8_stream(const __nv_bfloat16* p, float v[8]) {
  const uint4 a = __ldcs(reinterpret_cast<const uint4*>(p));
  v[0] = __uint_as_float(a.x << 16); v[1] = __uint_as_float(a.x & 0xffff0000u);
  v[2] = __uint_as_float(a.y << 16); v[3] = __uint_as_float(a.y & 0xffff0000u);
  v[4] = __uint_as_float(a.z << 16); v[5] = __uint_as_float(a.z & 0xffff0000u);
  v[6] = __uint_as_float(a.w << 16); v[7] = __uint_as_float(a.w & 0xffff0000u);
}

__device__ __forceinline__ void ld8_stream(const float* p, float v[8]) {
  const float4 a = __ldcs(reinterpret_cast<const float4*>(p));
  const float4 b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// One CTA per (chunk, row): grid (chunks per row, min(rows, 65535)), rows strided by gridDim.y.
// kVec: 16-byte loads (every row start 16-byte aligned); else one token per thread per step.
template <typename TIn, bool kVec, bool kQ>
__global__ void __launch_bounds__(kDiagThreads, kDiagCtasPerSm) diag_partial_kernel(const TIn* __restrict__ zp,
                                                                   const TIn* __restrict__ zq,
                                                                   const float* __restrict__ q, int64_t R,
                                                                   int64_t V, int64_t ld, int64_t ldq, int chunk,
                                                                   DiagPart* __restrict__ part) {
  __shared__ Acc red[kDiagWarps];
  const int tid = threadIdx.x;
  const int64_t lo = static_cast<int64_t>(blockIdx.x) * chunk;
  const int64_t hi = lo + chunk < V ? lo + chunk : V;
  for (int64_t row = blockIdx.y; row < R; row += gridDim.y) {
    const TIn* p = zp + row * ld;
    const TIn* z = zq + row * ld;
    const float* e = kQ ? q + row * ldq : nullptr;
    const float rp = dev::ld1(p, 0), rq = dev::ld1(z, 0);
    Acc c = {-INFINITY, 0.f, -INFINITY, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    int64_t i = lo;
    if (kVec) {
      const int64_t hv = lo + ((hi - lo) & ~static_cast<int64_t>(7));
      constexpr int U = kQ ? 1 : 2;  // 64 B of loads in flight per thread either way
      for (i = lo + 8 * tid; i < hv; i += U * kDiagStep) {
        float pv[U][8], zv[U][8], ev[U][8];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (u == 0 || i + u * kDiagStep < hv) {
            ld8_stream(p + i + u * kDiagStep, pv[u]);
            ld8_stream(z + i + u * kDiagStep, zv[u]);
            if (kQ) ld8_stream(e + i + u * kDiagStep, ev[u]);
          }
        }
#pragma unroll
        for (int u = 0; u < U; ++u)
          if (u == 0 || i + u * kDiagStep < hv) accumulate<8, kQ>(c, pv[u], zv[u], ev[u], rp, rq);
      }
      i = hv + tid;  // ragged end of the row (fewer than 8 tokens)
    } else {
      i = lo + tid;
    }
    for (; i < hi; i += kDiagThreads) {
      const float pv = dev::ld1(p, i), zv = dev::ld1(z, i);
      const float ev = kQ ? e[i] : 0.f;
      accumulate<1, kQ>(c, &pv, &zv, &ev, rp, rq);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) merge(c, shfl_down(c, off));
    if ((tid & 31) == 0) red[tid >> 5] = c;
    __syncthreads();
    if (tid == 0) {
      Acc t = red[0];
      for (int w = 1; w < kDiagWarps; ++w) merge(t, red[w]);
      DiagPart o;
      o.mp = t.mp; o.sp = t.sp; o.mq = t.mq; o.sq = t.sq; o.tq = t.tq;
      o.a = t.a; o.e1 = t.e1; o.ez = t.ez; o.h = t.h; o.tp = t.tp;
      o.pad[0] = o.pad[1] = 0.f;
      part[row * gridDim.x + blockIdx.x] = o;
    }
    __syncthreads();
  }
}

// One warp per row: lanes merge the row's chunk partials (the same rescaled fp32 merge as the
// streaming pass), then lane 0 forms the diagnostics in fp32 (fp64 is avoided: its rate on this GPU
// is a small fraction of fp32's, and two fp64 logarithms a row cost more than the merge).
constexpr int kCombineWarps = 8;

struct CombineArgs {
  const int32_t* xstar;
  const float* cd_lse;
  const float* alpha;
  const float* beta;
  const float* temp;
  bool has_q;
  int64_t R, V, ld;
  int N, nchunk;
  const DiagPart* part;
  float* out;
};

template <typename TIn>
__global__ void __launch_bounds__(32 * kCombineWarps) diag_combine_kernel(const TIn* __restrict__ zp,
                                                                          const TIn* __restrict__ zq,
                                                                          const CombineArgs a) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int lane = threadIdx.x & 31;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * kCombineWarps + (threadIdx.x >> 5);
  if (row >= a.R) return;
  const DiagPart* pp = a.part + row * a.nchunk;
  const TIn* p = zp + row * a.ld;
  const TIn* z = zq + row * a.ld;
  // lanes 0-3 fetch the logits the outputs need (r_p, r_q, z_p(x*), z_q(x*)) while the partials
  // load; lanes 4-7 the lemma's inputs (cd_lse, alpha, beta, T)
  const int32_t x = a.xstar ? a.xstar[row] : -1;
  const bool x_ok = x >= 0 && x < a.V;
  const int64_t b = row / a.N;
  const bool want_cd = a.cd_lse && a.alpha;
  float lv = 0.f;
  if (lane < 2) lv = dev::ld1(lane == 0 ? p : z, 0);
  else if (lane < 4 && x_ok) lv = dev::ld1(lane == 2 ? p : z, x);
  else if (lane == 4 && want_cd) lv = a.cd_lse[row];
  else if (lane == 5 && want_cd) lv = a.alpha[b];
  else if (lane == 6 && want_cd && a.beta) lv = a.beta[b];
  else if (lane == 7 && want_cd && a.temp) lv = a.temp[b];
  Acc c = {-INFINITY, 0.f, -INFINITY, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int k = lane; k < a.nchunk; k += 32) {
    const DiagPart& d = pp[k];
    const Acc o = {d.mp, d.sp, d.mq, d.sq, d.tq, d.a, d.e1, d.ez, d.h, d.tp};
    merge(c, o);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) merge(c, shfl_down(c, off));
  const float rp = __shfl_sync(0xffffffffu, lv, 0), rq = __shfl_sync(0xffffffffu, lv, 1);
  const float px = __shfl_sync(0xffffffffu, lv, 2), qx = __shfl_sync(0xffffffffu, lv, 3);
  const float cdl = __shfl_sync(0xffffffffu, lv, 4), al = __shfl_sync(0xffffffffu, lv, 5);
  const float be = __shfl_sync(0xffffffffu, lv, 6), tt = __shfl_sync(0xffffffffu, lv, 7);
  if (lane != 0) return;
  const float ls_p = logf(c.sp), ls_q = logf(c.sq);  // lse = m + ls
  // L_p = lse_p - r_p, with m - r the difference of two stored logits (exact for bf16 inputs)
  const float Lp = (c.mp - rp) + ls_p, Lq = (c.mq - rq) + ls_q;
  const float signal = x_ok ? fabsf(((px - c.mp) - ls_p) - ((qx - c.mq) - ls_q)) : NAN;
  const float lse_p = c.mp + ls_p, lse_q = c.mq + ls_q;
  const float kl_pq = c.tp / c.sp - (Lp - Lq);
  // the lemma holds for the untruncated target at T = 1 (greedy sequences report cd_lse at T = 1)
  const bool lemma = want_cd && be == 0.f && (tt == 0.f || tt == 1.f) && al >= 0.f;
  float* o = a.out + row * kDiagCols;
  o[0] = lse_p;
  o[1] = lse_q;
  o[2] = signal;
  o[3] = c.tq / c.sq - (Lp - Lq);
  o[4] = a.has_q ? fmaf(-(Lp - Lq), c.e1, c.a) : NAN;
  o[5] = a.has_q ? fmaf(Lp, c.e1, fmaf(c.h, kLn2, -c.ez)) : NAN;
  o[6] = kl_pq;
  o[7] = lemma ? (cdl - (1.f + al) * lse_p + al * lse_q) - al * kl_pq : NAN;
}

template <typename TIn, bool kVec, bool kQ>
cudaError_t launch_partial(const DiagArgs& d, int chunk, int nchunk) {
  const dim3 grid(static_cast<unsigned>(nchunk), static_cast<unsigned>(std::min<int64_t>(d.R, 65535)));
  diag_partial_kernel<TIn, kVec, kQ><<<grid, kDiagThreads, 0, d.stream>>>(
      static_cast<const TIn*>(d.z_exp), static_cast<const TIn*>(d.z_ama), d.q, d.R, d.V, d.ld, d.ldq, chunk, d.part);
  return cudaGetLastError();
}

template <typename TIn>
cudaError_t launch_typed(const DiagArgs& d) {
  int dev_id = 0, sms = 152;
  if (cudaGetDevice(&dev_id) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev_id);
  const int chunk = diag_chunk(d.R, d.V, sms);
  const int nchunk = static_cast<int>((d.V + chunk - 1) / chunk);
  const auto aligned = [](const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
  const bool vec = aligned(d.z_exp) && aligned(d.z_ama) && (d.ld * static_cast<int64_t>(sizeof(TIn))) % 16 == 0 &&
                   (!d.q || (aligned(d.q) && d.ldq % 4 == 0));
  cudaError_t e;
  if (vec)
    e = d.q ? launch_partial<TIn, true, true>(d, chunk, nchunk) : launch_partial<TIn, true, false>(d, chunk, nchunk);
  else
    e = d.q ? launch_partial<TIn, false, true>(d, chunk, nchunk) : launch_partial<TIn, false, false>(d, chunk, nchunk);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>((d.R + kCombineWarps - 1) / kCombineWarps));
  cfg.blockDim = dim3(32 * kCombineWarps);
  cfg.stream = d.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (d.stop && (e = cudaEventRecord(static_cast<cudaEvent_t>(d.stop), d.stream)) != cudaSuccess) return e;
  CombineArgs ca;
  ca.xstar = d.xstar;
  ca.cd_lse = d.cd_lse;
  ca.alpha = d.alpha;
  ca.beta = d.beta;
  ca.temp = d.temp;
  ca.has_q = d.q != nullptr;
  ca.R = d.R;
  ca.V = d.V;
  ca.ld = d.ld;
  ca.N = d.N;
  ca.nchunk = nchunk;
  ca.part = d.part;
  ca.out = d.out;
  return cudaLaunchKernelEx(&cfg, diag_combine_kernel<TIn>, static_cast<const TIn*>(d.z_exp),
                            static_cast<const TIn*>(d.z_ama), ca);
}

}  // namespace

int diag_chunk(int64_t R, int64_t V, int sms) {
  // enough CTAs for about four waves of resident CTAs, in whole passes of the CTA
  const int64_t want = static_cast<int64_t>(4) * kDiagCtasPerSm * std::max(sms, 1);
  int64_t per = (V * R + want - 1) / want;
  per = (per + kDiagStep - 1) / kDiagStep * kDiagStep;
  return static_cast<int>(std::min<int64_t>(std::max<int64_t>(per, kDiagMinChunk), kDiagMaxChunk));
}

cudaError_t launch_diagnostics(const DiagArgs& d) {
  if (d.R == 0) return cudaSuccess;
  if (d.start) {
    const cudaError_t e = cudaEventRecord(static_cast<cudaEvent_t>(d.start), d.stream);
    if (e != cudaSuccess) return e;
  }
  return d.dtype == DCD_BF16 ? launch_typed<__nv_bfloat16>(d) : launch_typed<float>(d);
}

}  // namespace dcd
