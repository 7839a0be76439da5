// dcd_small.cu -- greedy verification of a small call in one launch (chains and small trees:
// the latency case of single-request decoding).
//
// greedy_small_kernel: one CTA per (part, row).  The eight warps read their part of z_p and z_q
// directly with 16-byte loads (128 B in flight a thread for bf16) and keep per lane an online
// max of the scaled CD score u = k2 ((1 + alpha) z_p - alpha z_q) on P_beta (Eq. 1, Sec. 2.1), the
// rescaled sum of 2^(u - max) and the argmax; a row with beta > 0 is read whole by its part-0 CTA
// (a max pass over z_p first).  Each CTA publishes its part's statistics and takes the row's
// acquire-release ticket; the CTA with the row's last ticket combines the parts in a fixed order
// and finishes the row (the outputs of Eq. 1 and the greedy rule: the first child whose token is
// the argmax, else the argmax as the terminal token).  It then takes the call's row ticket; the
// CTA that finishes the last row walks every sequence's tree (the T -> 0 limit of Algorithm 1).
// Nothing waits on another CTA, so the grid needs no co-residency.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <climits>

#include "dcd.h"
#include "dcd_device.cuh"
#include "dcd_internal.h"
#include "dcd_small.h"

namespace dcd {
namespace {

using namespace dev;

constexpr int kSmallThreads = kThreads;
constexpr int kStep = 8 * kSmallThreads;  // tokens one step of the CTA covers
constexpr float kLn2f = 0.69314718055994531f;

// 8 fp32 tokens read once (evict-first).
__device__ __forceinline__ void ld8_first(const float* p, float v[8]) {
  const float4 a = __ldcs(reinterpret_cast<const float4*>(p));
  const float4 b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

template <typename TIn, bool kVec>
__global__ void __launch_bounds__(kSmallThreads, 4) greedy_small_kernel(const ScoreArgs p, int pchunk, int pparts,
                                                                        int32_t* accept_len, int32_t* accept_path,
                                                                        int32_t* bonus) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int N = p.N;
  const int64_t V = p.V;
  const int R = p.B * N;
  constexpr int kU = sizeof(TIn) == 2 ? 4 : 2;  // 8-token groups in flight a thread: 128 B of loads

  __shared__ float redf[32];
  __shared__ int redi[32];
  __shared__ int sh_last, sh_m, sh_walk;
  __shared__ uint32_t sh_status;
  __shared__ float sh_M, sh_S;
  __shared__ int sh_arg;
  extern __shared__ __align__(16) int small_smem[];

  const int part = blockIdx.x;
  const int64_t g = blockIdx.y;
  const int b = static_cast<int>(g / N), n = static_cast<int>(g % N);
  const float alpha = p.alpha[b];
  const float beta = p.beta ? p.beta[b] : 0.f;
  const bool masked = beta > 0.f;
  if (masked && part > 0) return;  // the part-0 CTA reads a masked row whole
  const int nparts = masked ? 1 : pparts;
  const float c1k = (1.f + alpha) * kLog2e, ak = alpha * kLog2e;  // u in units of log2
  const float logb = masked ? logf(beta) : -INFINITY;
  const TIn* zp_row = static_cast<const TIn*>(p.zp) + g * p.ld;
  const TIn* zq_row = static_cast<const TIn*>(p.zq) + g * p.ld;
  const int64_t lo = masked ? 0 : static_cast<int64_t>(part) * pchunk;
  const int64_t hi = masked ? V : (lo + pchunk < V ? lo + pchunk : V);

  // ---- max pass (beta > 0): the expert max for P_beta = {x : z_p(x) - max z_p >= log beta}
  float Mp = 0.f;
  if (masked) {
    float lm = -INFINITY;
    for (int64_t x = lo + tid * 8; x < hi; x += kStep) {
      if (kVec && x + 8 <= hi) {
        float z[8];
        ld8(zp_row + x, z);
        lm = fmaxf(lm, max8(z));
      } else {
        for (int e = 0; e < 8 && x + e < hi; ++e) lm = fmaxf(lm, ld1(zp_row, x + e));
      }
    }
    Mp = block_max(lm, redf);
  }

  // ---- stats pass: per lane the online max of u, the rescaled sum of 2^(u - max), the argmax
  float lmax = -INFINITY, lsum = 0.f;
  int larg = INT_MAX;
  auto add8 = [&](const float u[8], int64_t x0) {
    const float gm = max8(u);
    if (gm > lmax) {
      lsum *= ex2(lmax - gm);  // 0 while lmax is -inf
      lmax = gm;
#pragma unroll
      for (int e = 7; e >= 0; --e)
        if (u[e] == gm) larg = static_cast<int>(x0) + e;
    }
    if (lmax > -INFINITY) {
      float a = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) a += ex2(u[e] - lmax);
      lsum += a;
    }
  };
  for (int64_t x0 = lo + tid * 8; x0 < hi; x0 += kU * kStep) {
    if (kVec && !masked && x0 + (kU - 1) * kStep + 8 <= hi) {
      if constexpr (sizeof(TIn) == 2) {
        // the loads first (kept packed), then the arithmetic
        uint4 rp[kU], rq[kU];
#pragma unroll
        for (int h = 0; h < kU; ++h) {
          rp[h] = __ldcs(reinterpret_cast<const uint4*>(zp_row + x0 + h * kStep));
          rq[h] = __ldcs(reinterpret_cast<const uint4*>(zq_row + x0 + h * kStep));
        }
#pragma unroll
        for (int h = 0; h < kU; ++h) {
          const uint32_t pw[4] = {rp[h].x, rp[h].y, rp[h].z, rp[h].w};
          const uint32_t qw[4] = {rq[h].x, rq[h].y, rq[h].z, rq[h].w};
          float u[8];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            u[2 * e] = fmaf(c1k, __uint_as_float(pw[e] << 16), -ak * __uint_as_float(qw[e] << 16));
            u[2 * e + 1] =
                fmaf(c1k, __uint_as_float(pw[e] & 0xffff0000u), -ak * __uint_as_float(qw[e] & 0xffff0000u));
          }
          add8(u, x0 + h * kStep);
        }
      } else {
        float zp[kU][8], zq[kU][8];
#pragma unroll
        for (int h = 0; h < kU; ++h) {
          ld8_first(zp_row + x0 + h * kStep, zp[h]);
          ld8_first(zq_row + x0 + h * kStep, zq[h]);
        }
#pragma unroll
        for (int h = 0; h < kU; ++h) {
          float u[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) u[e] = fmaf(c1k, zp[h][e], -ak * zq[h][e]);
          add8(u, x0 + h * kStep);
        }
      }
    } else {
      for (int h = 0; h < kU; ++h) {
        const int64_t x = x0 + h * kStep;
        if (x >= hi) break;
        float zp[8], zq[8], u[8];
        if (kVec && x + 8 <= hi) {
          ld8(zp_row + x, zp);
          ld8(zq_row + x, zq);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const bool ok = x + e < hi;
            zp[e] = ok ? ld1(zp_row, x + e) : 0.f;
            zq[e] = ok ? ld1(zq_row, x + e) : 0.f;
          }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const bool in = (x + e < hi) && (!masked || (zp[e] - Mp >= logb));
          u[e] = in ? fmaf(c1k, zp[e], -ak * zq[e]) : -INFINITY;
        }
        add8(u, x);
      }
    }
  }
  float M = lmax, S = lsum;
  int arg = larg;
  block_stats(M, S, arg, redf, redi);

  // ---- publish the part; the CTA with the row's last ticket finishes the row
  if (tid == 0) {
    int last = 1;
    if (nparts > 1) {
      RowPart rp;
      rp.M = M;
      rp.S = S;
      rp.arg = arg;
      rp.key = -INFINITY;
      rp.blk = INT_MAX;
      rp.timed_out = 0;
      rp.pad[0] = rp.pad[1] = 0;
      p.parts[g * kMaxParts + part] = rp;
      const uint32_t t = atomic_add_acq_rel(&p.pdone[g], 1u);
      last = t + 1u == static_cast<uint32_t>(nparts) ? 1 : 0;
      if (last) {
        float cM = -INFINITY, cS = 0.f;
        int carg = INT_MAX;
        for (int k = 0; k < nparts; ++k) {  // a fixed order: the result does not depend on timing
          const RowPart* src = &p.parts[g * kMaxParts + k];
          const float pM = __ldcg(&src->M), pS = __ldcg(&src->S);
          const int parg = __ldcg(&src->arg);
          const float nM = fmaxf(cM, pM);
          cS = (cM > -INFINITY ? cS * ex2(cM - nM) : 0.f) + (pM > -INFINITY ? pS * ex2(pM - nM) : 0.f);
          if (pM > cM || (pM == cM && parg < carg)) carg = parg;
          cM = nM;
        }
        M = cM;
        S = cS;
        arg = carg;
      }
    }
    sh_last = last;
    sh_M = M;
    sh_S = S;
    sh_arg = arg;
  }
  __syncthreads();
  if (!sh_last) return;
  M = sh_M;
  S = sh_S;
  arg = sh_arg;

  // ---- finish the row: children and checks, then the greedy rule
  int* kids = small_smem;  // [N] children, ascending id
  int* ktok = kids + N;    // [N] their tokens
  if (warp == 0) {
    const int32_t* parr = p.parents + static_cast<int64_t>(b) * N;
    const int32_t* tokr = p.tokens + static_cast<int64_t>(b) * N;
    int count = 0;
    for (int base = n + 1; base < N; base += 32) {
      const int c = base + lane;
      const bool is = c < N && parr[c] == n;
      const unsigned msk = __ballot_sync(~0u, is);
      if (is) {
        const int pos = count + __popc(msk & ((1u << lane) - 1u));
        kids[pos] = c;
        ktok[pos] = tokr[c];
      }
      count += __popc(msk);
    }
    if (lane == 0) {
      uint32_t st = 0u;
      const int pp = parr[n];
      if (n == 0 ? pp != -1 : (pp < 0 || pp >= n)) st |= DCD_DEVERR_BAD_PARENT;
      if (n > 0) {
        const int t = tokr[n];
        if (t < 0 || t >= V) st |= DCD_DEVERR_BAD_TOKEN;
      }
      if (!(alpha >= 0.f && alpha <= 3.0e38f) || !(beta >= 0.f && beta <= 1.f)) st |= DCD_DEVERR_BAD_PARAM;
      if (!(M > -INFINITY && M < INFINITY) || !(S > 0.f && S < INFINITY)) st |= DCD_DEVERR_NONFINITE;
      sh_m = count;
      sh_status = st;
    }
  }
  __syncthreads();
  const int m = sh_m;
  const float logS = logf(S);
  if (tid == 0) {
    if (p.cd_argmax) p.cd_argmax[g] = arg;
    if (p.cd_lse) p.cd_lse[g] = M * kLn2f + logS;
    if (n == 0 && p.cd_logprob) p.cd_logprob[g] = 0.f;
  }
  if (p.cd_logprob) {
    for (int k = tid; k < m; k += kSmallThreads) {
      const int t = ktok[k];
      float v = -INFINITY;
      if (t >= 0 && t < V) {
        const float z = ld1(zp_row, t), zz = ld1(zq_row, t);
        if (!masked || (z - Mp >= logb)) v = (fmaf(c1k, z, -ak * zz) - M) * kLn2f - logS;
      }
      p.cd_logprob[static_cast<int64_t>(b) * N + kids[k]] = v;
    }
  }
  if (tid == 0) {
    int acc = -1;
    for (int k = 0; k < m; ++k)
      if (ktok[k] == arg) {
        acc = kids[k];
        break;
      }
    RowRecord r;
    r.acc_child = acc;
    r.term_token = acc < 0 ? arg : -1;
    r.status = sh_status;
    r.reserved = 0;
    p.rec[g] = r;
    const uint32_t t = atomic_add_acq_rel(&p.hdr->rows_done, 1u);
    sh_walk = t + 1u == static_cast<uint32_t>(R) ? 1 : 0;
  }
  __syncthreads();
  if (!sh_walk) return;

  // ---- the last row is done: walk every sequence (a warp each) from the records
  for (int sb = warp; sb < p.B; sb += kWarps) {
    int* wacc = small_smem + warp * 2 * N;
    int* wterm = wacc + N;
    const RowRecord* r = p.rec + static_cast<int64_t>(sb) * N;
    uint32_t st = 0u;
    for (int i = lane; i < N; i += 32) {
      wacc[i] = __ldcg(&r[i].acc_child);
      wterm[i] = __ldcg(&r[i].term_token);
      st |= static_cast<uint32_t>(__ldcg(reinterpret_cast<const int*>(&r[i].status)));
    }
    st = __reduce_or_sync(~0u, st);
    __syncwarp();
    int32_t* path = accept_path + static_cast<int64_t>(sb) * N;
    if (st) {
      if (lane == 0) {
        atomicOr(&p.hdr->err, st);
        accept_len[sb] = 0;
        bonus[sb] = -1;
      }
      for (int i = lane; i < N; i += 32) path[i] = i == 0 ? 0 : -1;
      continue;
    }
    // lane 0 follows the accepted children; the path is written as it is found
    int len = 0, cur = 0;
    if (lane == 0) {
      path[0] = 0;
      while (len < N - 1) {
        const int a = wacc[cur];
        if (a <= cur || a >= N) break;
        cur = a;
        path[++len] = cur;
      }
      accept_len[sb] = len;
      bonus[sb] = wterm[cur];
    }
    len = __shfl_sync(~0u, len, 0);
    for (int i = len + 1 + lane; i < N; i += 32) path[i] = -1;
    __syncwarp();
  }
}

}  // namespace

bool greedy_small_ok(const ScoreArgs& a) {
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  return a.q == nullptr && R > 0 && R <= kSmallMaxRows && a.N <= kSmallMaxNodes;
}

cudaError_t launch_greedy_small(const ScoreArgs& a, int32_t* accept_len, int32_t* accept_path, int32_t* bonus,
                                cudaStream_t stream) {
  const int64_t R = static_cast<int64_t>(a.B) * a.N;
  if (R == 0) return cudaSuccess;
  // parts of kStep-token multiples, at most kMaxParts a row
  const int64_t per = (a.V + kMaxParts - 1) / kMaxParts;
  const int64_t chunk = (per + kStep - 1) / kStep * kStep;
  const int pparts = static_cast<int>((a.V + chunk - 1) / chunk);
  cudaError_t e = cudaMemsetAsync(a.hdr, 0, kWorkspaceHeader + part_counter_bytes(static_cast<size_t>(R)), stream);
  if (e != cudaSuccess) return e;
  const int es = a.dtype == DCD_BF16 ? 2 : 4;
  auto al16 = [](const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
  const bool vec = !a.force_plain && al16(a.zp) && al16(a.zq) && (a.ld * es) % 16 == 0;
  const dim3 grid(static_cast<unsigned>(pparts), static_cast<unsigned>(R));
  // the child lists, then the walk's two arrays per warp
  const size_t smem = static_cast<size_t>(a.N) * 4 * (2 * kWarps > 2 ? 2 * kWarps : 2);
  if (a.dtype == DCD_BF16) {
    if (vec)
      greedy_small_kernel<__nv_bfloat16, true><<<grid, kSmallThreads, smem, stream>>>(
          a, static_cast<int>(chunk), pparts, accept_len, accept_path, bonus);
    else
      greedy_small_kernel<__nv_bfloat16, false><<<grid, kSmallThreads, smem, stream>>>(
          a, static_cast<int>(chunk), pparts, accept_len, accept_path, bonus);
  } else {
    if (vec)
      greedy_small_kernel<float, true><<<grid, kSmallThreads, smem, stream>>>(a, static_cast<int>(chunk), pparts,
                                                                             accept_len, accept_path, bonus);
    else
      greedy_small_kernel<float, false><<<grid, kSmallThreads, smem, stream>>>(a, static_cast<int>(chunk), pparts,
                                                                              accept_len, accept_path, bonus);
  }
  return cudaGetLastError();
}

}  // namespace dcd
