// dcd_api.cu -- the C ABI of include/dcd.h: argument checks, workspace layout and the
// stream-ordered launches of the verification step.

#include <cuda_runtime.h>
#include <stdint.h>

#include <climits>

#include "dcd.h"
#include "dcd_diag.h"
#include "dcd_fused.h"
#include "dcd_internal.h"
#include "dcd_upload.h"
#include "dcd_small.h"

namespace {

constexpr int kVersion = 10100;  // 1.1.0

bool shape_ok(const dcd_shape* s, bool need_q) {
  if (!s) return false;
  if (s->B < 0 || s->N < 1 || s->V < 1 || s->V > INT_MAX || (s->flags & ~DCD_SIBLINGS_DISTINCT) != 0) return false;
  if (s->logits_dtype != DCD_F32 && s->logits_dtype != DCD_BF16) return false;
  if (s->ld_logits < s->V) return false;
  if (need_q && s->ld_q < s->V) return false;
  if (static_cast<int64_t>(s->B) * s->N > INT_MAX / 16) return false;
  return true;
}

size_t workspace_bytes_for(const dcd_shape* s) {
  const size_t rows = static_cast<size_t>(s->B) * static_cast<size_t>(s->N);
  const size_t raw = dcd::kWorkspaceHeader + dcd::part_counter_bytes(rows) +
                     rows * (sizeof(dcd::Job) + sizeof(dcd::RowRecord) + dcd::kMaxParts * sizeof(dcd::RowPart) +
                             dcd::slot_bytes(s->V, s->logits_dtype, static_cast<int64_t>(rows)));
  return (raw + 255) & ~static_cast<size_t>(255);
}

int check_workspace(const dcd_shape* s, const void* ws, size_t bytes) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return DCD_ERR_WORKSPACE;
  if (bytes < workspace_bytes_for(s)) return DCD_ERR_WORKSPACE;
  return DCD_OK;
}

struct WsView {
  dcd::WsHeader* hdr;
  dcd::Job* jobs;
  uint32_t* pdone;
  dcd::RowRecord* rec;
  dcd::RowPart* parts;
  unsigned char* slots;
};

WsView view(void* ws, const dcd_shape* s) {
  const size_t rows = static_cast<size_t>(s->B) * static_cast<size_t>(s->N);
  char* p = static_cast<char*>(ws);
  WsView v;
  v.hdr = reinterpret_cast<dcd::WsHeader*>(p);
  p += dcd::kWorkspaceHeader;
  v.pdone = reinterpret_cast<uint32_t*>(p);
  p += dcd::part_counter_bytes(rows);
  v.jobs = reinterpret_cast<dcd::Job*>(p);
  p += rows * sizeof(dcd::Job);
  v.rec = reinterpret_cast<dcd::RowRecord*>(p);
  p += rows * sizeof(dcd::RowRecord);
  v.parts = reinterpret_cast<dcd::RowPart*>(p);
  p += rows * dcd::kMaxParts * sizeof(dcd::RowPart);
  v.slots = reinterpret_cast<unsigned char*>(p);
  return v;
}

int cuda_status(cudaError_t e) { return e == cudaSuccess ? DCD_OK : DCD_ERR_CUDA; }

dcd::ScoreArgs make_args(const dcd_shape* s, const void* z_exp, const void* z_ama, const float* q,
                         const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                         const float* temperature, uint64_t seed, uint64_t offset, float* cd_logprob,
                         int32_t* cd_argmax, float* cd_lse, void* ws) {
  dcd::ScoreArgs a{};
  a.zp = z_exp;
  a.zq = z_ama;
  a.q = q;
  a.ld = s->ld_logits;
  a.ldq = q ? s->ld_q : 0;
  a.V = s->V;
  a.tokens = tokens;
  a.parents = parents;
  a.alpha = alpha;
  a.beta = beta;
  a.temp = temperature;
  a.B = s->B;
  a.N = s->N;
  a.dtype = s->logits_dtype;
  a.seed = seed;
  a.offset = offset;
  a.cd_logprob = cd_logprob;
  a.cd_argmax = cd_argmax;
  a.cd_lse = cd_lse;
  const WsView v = view(ws, s);
  a.hdr = v.hdr;
  a.jobs = v.jobs;
  a.pdone = v.pdone;
  a.rec = v.rec;
  a.parts = v.parts;
  a.slots = v.slots;
  a.force_stages = 0;
  a.force_plain = 0;
  a.distinct = (s->flags & DCD_SIBLINGS_DISTINCT) ? 1 : 0;
  return a;
}

int score_rows_impl(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                    const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                    const float* temperature, uint64_t seed, uint64_t offset, float* cd_logprob, int32_t* cd_argmax,
                    float* cd_lse, void* workspace, size_t workspace_bytes, cudaStream_t stream, int force_stages,
                    int force_plain, int64_t poll_cycles) {
  const bool sampled_call = temperature != nullptr;
  if (!shape_ok(shape, sampled_call)) return DCD_ERR_INVALID_ARG;
  if (shape->N > DCD_MAX_NODES) return DCD_ERR_UNSUPPORTED;
  if (sampled_call && !q) return DCD_ERR_INVALID_ARG;
  if (!sampled_call && q) return DCD_ERR_INVALID_ARG;
  if (shape->B == 0) return DCD_OK;
  if (!z_exp || !z_ama || !tokens || !parents || !alpha) return DCD_ERR_INVALID_ARG;
  const int ws = check_workspace(shape, workspace, workspace_bytes);
  if (ws != DCD_OK) return ws;
  dcd::ScoreArgs a = make_args(shape, z_exp, z_ama, q, tokens, parents, alpha, beta, temperature, seed, offset,
                               cd_logprob, cd_argmax, cd_lse, workspace);
  a.force_stages = force_stages;
  a.force_plain = force_plain;
  a.poll_cycles = poll_cycles;
  const dcd::RowGeometry geo = dcd::row_geometry(a);
  if (geo.smem > 227 * 1024 || geo.ctas_per_sm < 1) return DCD_ERR_UNSUPPORTED;
  return cuda_status(dcd::launch_score_rows(a, stream));
}

}  // namespace

extern "C" {

size_t dcd_workspace_bytes(const dcd_shape* shape) {
  if (!shape_ok(shape, false)) return 0;
  return workspace_bytes_for(shape);
}

int dcd_score_rows(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                   const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                   const float* temperature, uint64_t seed, uint64_t offset, float* cd_logprob, int32_t* cd_argmax,
                   float* cd_lse, void* workspace, size_t workspace_bytes, dcd_stream_t stream) {
  return score_rows_impl(shape, z_exp, z_ama, q, tokens, parents, alpha, beta, temperature, seed, offset, cd_logprob,
                         cd_argmax, cd_lse, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream), 0, 0, 0);
}

int dcd_tree_walk(const dcd_shape* shape, int32_t* accept_len, int32_t* accept_path, int32_t* bonus,
                  void* workspace, size_t workspace_bytes, dcd_stream_t stream) {
  if (!shape_ok(shape, false)) return DCD_ERR_INVALID_ARG;
  if (shape->N > DCD_MAX_NODES) return DCD_ERR_UNSUPPORTED;
  if (shape->B == 0) return DCD_OK;
  if (!accept_len || !accept_path || !bonus) return DCD_ERR_INVALID_ARG;
  const int ws = check_workspace(shape, workspace, workspace_bytes);
  if (ws != DCD_OK) return ws;
  const WsView v = view(workspace, shape);
  return cuda_status(dcd::launch_tree_walk(shape->B, shape->N, v.rec, &v.hdr->err, accept_len, accept_path, bonus,
                                           reinterpret_cast<cudaStream_t>(stream)));
}

int dcd_verify_greedy(const dcd_shape* shape, const void* z_exp, const void* z_ama, const int32_t* tokens,
                      const int32_t* parents, const float* alpha, const float* beta, int32_t* accept_len,
                      int32_t* accept_path, int32_t* bonus, float* cd_logprob, int32_t* cd_argmax, float* cd_lse,
                      void* workspace, size_t workspace_bytes, dcd_stream_t stream) {
  if (!shape_ok(shape, false)) return DCD_ERR_INVALID_ARG;
  if (shape->B > 0 && (!accept_len || !accept_path || !bonus)) return DCD_ERR_INVALID_ARG;
  if (shape->N > DCD_MAX_NODES) return DCD_ERR_UNSUPPORTED;
  if (shape->B > 0 && shape->N <= dcd::kSmallMaxNodes &&
      static_cast<int64_t>(shape->B) * shape->N <= dcd::kSmallMaxRows) {
    // a small call: rows and tree walk in one launch
    if (!z_exp || !z_ama || !tokens || !parents || !alpha) return DCD_ERR_INVALID_ARG;
    const int ws = check_workspace(shape, workspace, workspace_bytes);
    if (ws != DCD_OK) return ws;
    const dcd::ScoreArgs a = make_args(shape, z_exp, z_ama, nullptr, tokens, parents, alpha, beta, nullptr, 0, 0,
                                       cd_logprob, cd_argmax, cd_lse, workspace);
    if (dcd::greedy_small_ok(a))
      return cuda_status(dcd::launch_greedy_small(a, accept_len, accept_path, bonus,
                                                  reinterpret_cast<cudaStream_t>(stream)));
  }
  int rc = dcd_score_rows(shape, z_exp, z_ama, nullptr, tokens, parents, alpha, beta, nullptr, 0, 0, cd_logprob,
                          cd_argmax, cd_lse, workspace, workspace_bytes, stream);
  if (rc != DCD_OK) return rc;
  return dcd_tree_walk(shape, accept_len, accept_path, bonus, workspace, workspace_bytes, stream);
}

int dcd_verify_sample(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                      const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                      const float* temperature, uint64_t seed, uint64_t offset, int32_t* accept_len,
                      int32_t* accept_path, int32_t* bonus, float* cd_logprob, int32_t* cd_argmax, float* cd_lse,
                      float* residual, void* workspace, size_t workspace_bytes, dcd_stream_t stream) {
  if (!shape_ok(shape, true)) return DCD_ERR_INVALID_ARG;
  if (!temperature || !q) return DCD_ERR_INVALID_ARG;
  if (shape->B > 0 && (!accept_len || !accept_path || !bonus)) return DCD_ERR_INVALID_ARG;
  int rc = dcd_score_rows(shape, z_exp, z_ama, q, tokens, parents, alpha, beta, temperature, seed, offset,
                          cd_logprob, cd_argmax, cd_lse, workspace, workspace_bytes, stream);
  if (rc != DCD_OK) return rc;
  rc = dcd_tree_walk(shape, accept_len, accept_path, bonus, workspace, workspace_bytes, stream);
  if (rc != DCD_OK || !residual || shape->B == 0) return rc;
  dcd::ScoreArgs a = make_args(shape, z_exp, z_ama, q, tokens, parents, alpha, beta, temperature, seed, offset,
                               cd_logprob, cd_argmax, cd_lse, workspace);
  return cuda_status(dcd::launch_terminal_residual(a, accept_len, accept_path, bonus, residual,
                                                   reinterpret_cast<cudaStream_t>(stream)));
}

int dcd_upload_q_rows(const dcd_shape* shape, const float* q_host, float* q_dev, const int32_t* parents,
                      const float* temperature, dcd_stream_t stream) {
  if (!shape_ok(shape, true)) return DCD_ERR_INVALID_ARG;
  if (shape->B == 0) return DCD_OK;
  if (!q_host || !q_dev || !parents || !temperature) return DCD_ERR_INVALID_ARG;
  // the first and the last element read must be page-locked host memory mapped into the device
  const int64_t R = static_cast<int64_t>(shape->B) * shape->N;
  const float* last = q_host + (R - 1) * shape->ld_q + (shape->V - 1);
  cudaPointerAttributes a0, a1;
  if (cudaPointerGetAttributes(&a0, q_host) != cudaSuccess || cudaPointerGetAttributes(&a1, last) != cudaSuccess) {
    (void)cudaGetLastError();
    return DCD_ERR_INVALID_ARG;
  }
  if (a0.type != cudaMemoryTypeHost || a1.type != cudaMemoryTypeHost || !a0.devicePointer || !a1.devicePointer)
    return DCD_ERR_INVALID_ARG;
  return cuda_status(dcd::launch_upload_q_rows(shape->B, shape->N, shape->V, shape->ld_q,
                                               static_cast<const float*>(a0.devicePointer), q_dev, parents,
                                               temperature, reinterpret_cast<cudaStream_t>(stream)));
}

size_t dcd_fused_workspace_bytes(const dcd_shape* s) {
  if (!s || s->B < 0 || s->N < 1 || s->V < 1 || s->V > INT_MAX || s->flags != 0) return 0;
  if (s->logits_dtype != DCD_BF16) return 0;
  if (static_cast<int64_t>(s->B) * s->N > INT_MAX / 16) return 0;
  return dcd::fused_layout(static_cast<int64_t>(s->B) * s->N, s->V).total;
}

int dcd_verify_fused_lmhead(const dcd_shape* shape, const void* h_exp, int32_t H_exp, const void* w_exp,
                            const void* h_ama, int32_t H_ama, const void* w_ama, const int32_t* tokens,
                            const int32_t* parents, const float* alpha, int32_t* accept_len,
                            int32_t* accept_path, int32_t* bonus, float* cd_logprob, int32_t* cd_argmax,
                            float* cd_lse, void* workspace, size_t workspace_bytes, dcd_stream_t stream) {
  return dcd_verify_fused_lmhead_ex(shape, h_exp, H_exp, w_exp, h_ama, H_ama, w_ama, tokens, parents, alpha,
                                    nullptr, accept_len, accept_path, bonus, cd_logprob, cd_argmax, cd_lse,
                                    workspace, workspace_bytes, stream, nullptr, nullptr);
}

int dcd_verify_fused_lmhead_ex(const dcd_shape* shape, const void* h_exp, int32_t H_exp, const void* w_exp,
                               const void* h_ama, int32_t H_ama, const void* w_ama, const int32_t* tokens,
                               const int32_t* parents, const float* alpha, const float* beta,
                               int32_t* accept_len, int32_t* accept_path, int32_t* bonus, float* cd_logprob,
                               int32_t* cd_argmax, float* cd_lse, void* workspace, size_t workspace_bytes,
                               dcd_stream_t stream, void* gemm_start, void* gemm_stop) {
  const size_t need = dcd_fused_workspace_bytes(shape);
  if (need == 0) return DCD_ERR_INVALID_ARG;
  if (shape->N > DCD_MAX_NODES) return DCD_ERR_UNSUPPORTED;
  if (shape->B == 0) return DCD_OK;
  auto al16 = [](const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(h_exp) || !al16(w_exp) || !al16(h_ama) || !al16(w_ama)) return DCD_ERR_INVALID_ARG;
  if (H_exp < 1 || H_ama < 1 || H_exp % 8 != 0 || H_ama % 8 != 0) return DCD_ERR_INVALID_ARG;
  if (!tokens || !parents || !alpha || !accept_len || !accept_path || !bonus) return DCD_ERR_INVALID_ARG;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 || workspace_bytes < need)
    return DCD_ERR_WORKSPACE;
  dcd::FusedArgs f;
  f.B = shape->B;
  f.N = shape->N;
  f.V = shape->V;
  f.H_exp = H_exp;
  f.H_ama = H_ama;
  f.h_exp = h_exp;
  f.w_exp = w_exp;
  f.h_ama = h_ama;
  f.w_ama = w_ama;
  f.tokens = tokens;
  f.parents = parents;
  f.alpha = alpha;
  f.beta = beta;
  f.accept_len = accept_len;
  f.accept_path = accept_path;
  f.bonus = bonus;
  f.cd_logprob = cd_logprob;
  f.cd_argmax = cd_argmax;
  f.cd_lse = cd_lse;
  f.workspace = workspace;
  f.gemm_start = static_cast<cudaEvent_t>(gemm_start);
  f.gemm_stop = static_cast<cudaEvent_t>(gemm_stop);
  int status = DCD_OK;
  const cudaError_t e = dcd::launch_fused(f, stream, &status);
  if (status != DCD_OK) return status;
  return cuda_status(e);
}

size_t dcd_diagnostics_workspace_bytes(const dcd_shape* shape) {
  if (!shape_ok(shape, false)) return 0;
  const size_t b = dcd::diag_workspace_bytes(static_cast<int64_t>(shape->B) * shape->N, shape->V);
  return b ? b : 256;
}

int dcd_row_diagnostics_ex(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                           const int32_t* xstar, const float* cd_lse, const float* alpha, const float* beta,
                           const float* temperature, float* diag, void* workspace, size_t workspace_bytes,
                           dcd_stream_t stream, void* pass_start, void* pass_stop) {
  if (!shape_ok(shape, q != nullptr) || shape->flags != 0) return DCD_ERR_INVALID_ARG;
  const int64_t R = static_cast<int64_t>(shape->B) * shape->N;
  if (R > 0 && (!z_exp || !z_ama || !diag)) return DCD_ERR_INVALID_ARG;
  if ((cd_lse != nullptr) != (alpha != nullptr)) return DCD_ERR_INVALID_ARG;  // the lemma needs both
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 ||
      workspace_bytes < dcd_diagnostics_workspace_bytes(shape))
    return DCD_ERR_WORKSPACE;
  dcd::DiagArgs d;
  d.R = R;
  d.V = shape->V;
  d.ld = shape->ld_logits;
  d.ldq = shape->ld_q;
  d.N = shape->N;
  d.dtype = shape->logits_dtype;
  d.z_exp = z_exp;
  d.z_ama = z_ama;
  d.q = q;
  d.xstar = xstar;
  d.cd_lse = cd_lse;
  d.alpha = alpha;
  d.beta = beta;
  d.temp = temperature;
  d.out = diag;
  d.part = static_cast<dcd::DiagPart*>(workspace);
  d.stream = stream;
  d.start = pass_start;
  d.stop = pass_stop;
  return cuda_status(dcd::launch_diagnostics(d));
}

int dcd_row_diagnostics(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                        const int32_t* xstar, const float* cd_lse, const float* alpha, const float* beta,
                        const float* temperature, float* diag, void* workspace, size_t workspace_bytes,
                        dcd_stream_t stream) {
  return dcd_row_diagnostics_ex(shape, z_exp, z_ama, q, xstar, cd_lse, alpha, beta, temperature, diag, workspace,
                                workspace_bytes, stream, nullptr, nullptr);
}

int dcd_get_device_error(const void* workspace, dcd_stream_t stream, uint32_t* bits) {
  if (!workspace || !bits) return DCD_ERR_INVALID_ARG;
  uint32_t host = 0;
  cudaError_t e = cudaMemcpyAsync(&host, workspace, sizeof host, cudaMemcpyDeviceToHost,
                                  reinterpret_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return DCD_ERR_CUDA;
  *bits = host;
  return host ? DCD_ERR_DEVICE_INPUT : DCD_OK;
}

const char* dcd_status_string(int status) {
  switch (status) {
    case DCD_OK: return "ok";
    case DCD_ERR_INVALID_ARG: return "invalid argument";
    case DCD_ERR_BAD_TREE: return "malformed draft tree";
    case DCD_ERR_UNSUPPORTED: return "unsupported request";
    case DCD_ERR_CUDA: return "CUDA error";
    case DCD_ERR_TIMEOUT: return "device wait timed out";
    case DCD_ERR_DEVICE_INPUT: return "device-side input error";
    case DCD_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    default: return "unknown status";
  }
}

int dcd_version(void) { return kVersion; }

// Test and tuning hook: dcd_score_rows with a forced ring depth and/or plain loads.
int dcd_score_rows_ex(const dcd_shape* shape, const void* z_exp, const void* z_ama, const float* q,
                      const int32_t* tokens, const int32_t* parents, const float* alpha, const float* beta,
                      const float* temperature, uint64_t seed, uint64_t offset, float* cd_logprob,
                      int32_t* cd_argmax, float* cd_lse, void* workspace, size_t workspace_bytes, dcd_stream_t stream,
                      int stages, int plain_loads, int64_t poll_limit_cycles) {
  if (stages != 0 && (stages < 2 || stages > 8)) return DCD_ERR_INVALID_ARG;
  if (poll_limit_cycles < 0) return DCD_ERR_INVALID_ARG;
  return score_rows_impl(shape, z_exp, z_ama, q, tokens, parents, alpha, beta, temperature, seed, offset, cd_logprob,
                         cd_argmax, cd_lse, workspace, workspace_bytes, reinterpret_cast<cudaStream_t>(stream),
                         stages, plain_loads, poll_limit_cycles);
}

}  // extern "C"
