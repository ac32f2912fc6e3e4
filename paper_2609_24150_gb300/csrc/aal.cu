// C ABI of libaal (include/aal.h): argument checks, workspace layout, launches.
#include <math.h>
#include <string.h>

#include <atomic>

#include "aal_internal.cuh"
#include "../../include/aal_debug.h"

using namespace aal;

namespace {

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
// target logits start on 16 bytes; target token ids (mode AAL_IDS) on 4
size_t target_align(int32_t mode) { return (mode & AAL_IDS) ? 4 : 16; }

// Failure-detection test hooks (include/aal_debug.h).
std::atomic<uint64_t> g_wait_limit_ns{0};
std::atomic<int64_t> g_skip_chunk{-1};
std::atomic<int64_t> g_fused_min_row_bytes{AAL_FUSED_MIN_ROW_BYTES_DEFAULT};

aal_status check_shape(int64_t N, int64_t K, int64_t V, int32_t dtype) {
  if (N < 0 || K < 1 || V < 1) return AAL_ERR_INVALID_ARG;
  if (K > AAL_MAX_K) return AAL_ERR_UNSUPPORTED;
  if (V > 0x7fffffff) return AAL_ERR_UNSUPPORTED;  // token ids are int32
  if (dtype != AAL_F32 && dtype != AAL_BF16) return AAL_ERR_INVALID_ARG;
  if (N > 0 && N > INT64_MAX / (K * V * 4)) return AAL_ERR_INVALID_ARG;  // element count overflow
  return AAL_OK;
}

aal_status check_problem(const aal_problem* p) {
  if (p == nullptr) return AAL_ERR_INVALID_ARG;
  aal_status st = check_shape(p->N, p->K, p->V, p->dtype);
  if (st != AAL_OK) return st;
  if (p->mode < 1 || p->mode > (AAL_BOTH | AAL_KL | AAL_GRPO | AAL_TV | AAL_IDS)) return AAL_ERR_INVALID_ARG;
  if ((p->mode & AAL_IDS) && ((p->mode & (AAL_SAMPLING | AAL_KL | AAL_TV)) || !(p->mode & (AAL_GREEDY | AAL_GRPO))))
    return AAL_ERR_INVALID_ARG;  // token ids define x* only: the greedy and GRPO terms
  if ((p->mode & (AAL_SAMPLING | AAL_TV)) && !(isfinite(p->temperature) && p->temperature > 0.f))
    return AAL_ERR_INVALID_ARG;
  if (!isfinite(p->w_greedy) || !isfinite(p->w_sampling) || !isfinite(p->w_kl) || !isfinite(p->w_tv))
    return AAL_ERR_INVALID_ARG;
  if (p->global_counts != 0 && p->global_counts != 1) return AAL_ERR_INVALID_ARG;
  if (p->global_counts == 1 && !(p->n_windows_global >= 0 && p->n_windows_global <= INT32_MAX &&
                                 p->n_positions_global >= 0 && p->n_positions_global <= INT32_MAX))
    return AAL_ERR_INVALID_ARG;
  return AAL_OK;
}

aal_status check_reward(const aal_reward_problem* p) {
  if (p == nullptr) return AAL_ERR_INVALID_ARG;
  aal_status st = check_shape(p->N, p->K, p->V, p->dtype);
  if (st != AAL_OK) return st;
  if (p->mode != AAL_GREEDY && p->mode != AAL_SAMPLING && p->mode != (AAL_SAMPLING | AAL_SAMPLED_DRAFT))
    return AAL_ERR_INVALID_ARG;
  if ((p->mode & AAL_SAMPLING) && !(isfinite(p->temperature) && p->temperature > 0.f)) return AAL_ERR_INVALID_ARG;
  if (p->windows_per_rollout < 1 || p->rollouts_per_group < 1) return AAL_ERR_INVALID_ARG;
  if (p->windows_per_rollout > INT64_MAX / p->rollouts_per_group) return AAL_ERR_INVALID_ARG;
  if (p->N % (p->windows_per_rollout * p->rollouts_per_group) != 0) return AAL_ERR_INVALID_ARG;
  if (!(isfinite(p->adv_clip) && p->adv_clip > 0.f)) return AAL_ERR_INVALID_ARG;
  if (p->row_offset < 0) return AAL_ERR_INVALID_ARG;
  return AAL_OK;
}

aal_status check_seq(const aal_seq_problem* p) {
  if (p == nullptr) return AAL_ERR_INVALID_ARG;
  if (p->B < 0 || p->seq_len < 0) return AAL_ERR_INVALID_ARG;
  if (p->full_windows != 0 && p->full_windows != 1) return AAL_ERR_INVALID_ARG;
  if (p->seq_len > 0 && p->B > INT64_MAX / p->seq_len) return AAL_ERR_INVALID_ARG;
  // the checks of a windowed problem with one window per position (R * K * V elements bound
  // the per-depth partials too)
  const aal_problem q{p->B * p->seq_len, p->K,          p->V,          p->dtype,
                      p->mode,           p->temperature, p->w_greedy, p->w_sampling,
                      p->w_kl,           p->w_tv,       p->global_counts,
                      p->global_counts == 1 ? p->n_windows_global : 0,
                      p->global_counts == 1 ? p->n_positions_global : 0};
  return check_problem(&q);
}

aal_status check_grpo(const aal_grpo_problem* p) {
  if (p == nullptr) return AAL_ERR_INVALID_ARG;
  aal_status st = check_shape(p->N, p->K, p->V, p->dtype);
  if (st != AAL_OK) return st;
  if (p->reserved != 0) return AAL_ERR_INVALID_ARG;
  if (p->windows_per_rollout < 1 || p->rollouts_per_group < 1) return AAL_ERR_INVALID_ARG;
  if (p->windows_per_rollout > INT64_MAX / p->rollouts_per_group) return AAL_ERR_INVALID_ARG;
  if (p->N % (p->windows_per_rollout * p->rollouts_per_group) != 0) return AAL_ERR_INVALID_ARG;
  if (!(isfinite(p->adv_clip) && p->adv_clip > 0.f)) return AAL_ERR_INVALID_ARG;
  if (!(p->eps_clip >= 0.f && p->eps_clip < 1.f)) return AAL_ERR_INVALID_ARG;
  if (!(isfinite(p->rho_min) && isfinite(p->rho_max) && p->rho_min >= 0.f && p->rho_min <= p->rho_max))
    return AAL_ERR_INVALID_ARG;
  if (!(isfinite(p->log_rho_clip) && p->log_rho_clip > 0.f)) return AAL_ERR_INVALID_ARG;
  if (!isfinite(p->w_grpo)) return AAL_ERR_INVALID_ARG;
  return AAL_OK;
}

aal_status cuda_status(cudaError_t e) { return e == cudaSuccess ? AAL_OK : AAL_ERR_CUDA; }

// The statistics pass over z_p and z_q for the mode's terms (takes the test hook's chunk).
RowStatsArgs stats_args(const void* draft, const void* target, int64_t R, int64_t V, int32_t mode,
                        float temperature, const LossWs& ws) {
  const bool greedy = (mode & AAL_GREEDY) != 0;
  const bool sampling = (mode & (AAL_SAMPLING | AAL_TV)) != 0;  // both need a^sample
  const bool kl = (mode & AAL_KL) != 0;
  const bool grpo = (mode & AAL_GRPO) != 0;  // log pi_theta(y) needs the T = 1 normaliser
  RowStatsArgs ra;
  ra.zq = draft;
  ra.zp = target;
  ra.R = R;
  ra.V = V;
  ra.sT = sampling ? kLog2e / temperature : 0.f;
  ra.need_p = sampling;
  ra.need_q = sampling;
  ra.need_q1 = (greedy || kl || grpo) && !(sampling && temperature == 1.0f);
  ra.overlap = sampling;
  ra.need_kl = kl;
  ra.skip_chunk = debug_take_skip_chunk();
  ra.ws = ws;
  return ra;
}

// The draft's statistics pass with x* as token ids (`target` holds them; takes the test hook's
// chunk).
Stream1Args ids_args(const void* draft, const void* target, int64_t R, int64_t V, const LossWs& ws) {
  Stream1Args a;
  a.z = draft;
  a.R = R;
  a.V = V;
  a.lws = ws;
  a.ids = static_cast<const int32_t*>(target);
  a.acc = nullptr;
  a.acc_ref = nullptr;
  a.lpr = nullptr;
  a.hdr = ws.hdr;
  a.skip_chunk = debug_take_skip_chunk();
  return a;
}

// Per-row statistics of R logit rows (pass over z_p and z_q, or over z_q alone when `target`
// holds token ids), shared by both layouts.
cudaError_t launch_stats(const void* draft, const void* target, int64_t R, int64_t V, int32_t dtype,
                         int32_t mode, float temperature, const LossWs& ws, cudaStream_t s, int* cluster) {
  if (mode & AAL_IDS) {
    *cluster = 1;
    return launch_one_tensor(ids_args(draft, target, R, V, ws), dtype == AAL_BF16, true, s);
  }
  *cluster = 1;
  return launch_rowstats(stats_args(draft, target, R, V, mode, temperature, ws), dtype == AAL_BF16, s, cluster);
}

// The gradient pass for the mode's terms.
BackwardArgs grad_args(const void* draft, const void* target, const uint8_t* mask, int64_t R, int64_t V,
                       int32_t mode, float temperature, float w_greedy, float w_kl, float dloss, const LossWs& ws,
                       void* grad) {
  const bool greedy = (mode & AAL_GREEDY) != 0;
  const bool sampling = (mode & (AAL_SAMPLING | AAL_TV)) != 0;
  const bool kl = (mode & AAL_KL) != 0;
  const bool grpo = (mode & AAL_GRPO) != 0;
  BackwardArgs ba;
  ba.zq = draft;
  ba.zp = target;
  ba.grad = grad;
  ba.R = R;
  ba.V = V;
  ba.K = 1;
  ba.sT = sampling ? kLog2e / temperature : 0.f;
  ba.invT = sampling ? 1.0f / temperature : 0.f;
  ba.dloss = dloss;
  ba.w_greedy = greedy ? w_greedy : 0.f;
  ba.w_sampling = sampling ? 1.f : 0.f;  // the window kernels fold w_s and w_tv into dE^s/da
  ba.w_kl = kl ? w_kl : 0.f;
  ba.grpo = grpo;
  ba.mask = mask;
  ba.q1_is_qT = (greedy || kl || grpo) && sampling && temperature == 1.0f;
  ba.ws = ws;
  return ba;
}

// Gradient rows from the statistics and dE/da in the workspace, shared by both layouts.
cudaError_t launch_grad(const void* draft, const void* target, const uint8_t* mask, int64_t R, int64_t V,
                        int32_t dtype, int32_t mode, float temperature, float w_greedy, float w_sampling,
                        float w_kl, float dloss, const LossWs& ws, void* grad, cudaStream_t s) {
  (void)w_sampling;  // folded into dE^s/da by the window kernels
  return launch_backward(grad_args(draft, target, mask, R, V, mode, temperature, w_greedy, w_kl, dloss, ws, grad),
                         dtype == AAL_BF16, s);
}

// The window terms of an [N][K] problem.
WindowArgs window_args(const aal_problem* prob, const uint8_t* mask, int cluster, float* loss, float* eal,
                       const LossWs& ws, int64_t nwblk) {
  WindowArgs wa;
  wa.mask = mask;
  wa.N = prob->N;
  wa.K = (int32_t)prob->K;
  wa.cluster = cluster;
  wa.greedy = (prob->mode & AAL_GREEDY) != 0;
  wa.sampling = (prob->mode & AAL_SAMPLING) != 0;
  wa.kl = (prob->mode & AAL_KL) != 0;
  wa.tv = (prob->mode & AAL_TV) != 0;
  wa.w_greedy = prob->w_greedy;
  wa.w_sampling = prob->w_sampling;
  wa.w_kl = prob->w_kl;
  wa.w_tv = prob->w_tv;
  wa.loss = loss;
  wa.eal = eal;
  wa.ws = ws;
  wa.nwblk = nwblk;
  wa.nvalid_g = prob->global_counts == 1 ? (int32_t)prob->n_windows_global : -1;
  wa.npos_g = prob->global_counts == 1 ? (int32_t)prob->n_positions_global : -1;
  return wa;
}

// The window terms of a sequence problem.
SeqWindowArgs seq_window_args(const aal_seq_problem* prob, const uint8_t* mask, int cluster, float* loss,
                              float* eal, void* workspace, const SeqLayout& L) {
  char* base = static_cast<char*>(workspace);
  SeqWindowArgs wa;
  wa.mask = mask;
  wa.B = prob->B;
  wa.T = prob->seq_len;
  wa.K = (int32_t)prob->K;
  wa.full_windows = prob->full_windows != 0;
  wa.cluster = cluster;
  wa.greedy = (prob->mode & AAL_GREEDY) != 0;
  wa.sampling = (prob->mode & AAL_SAMPLING) != 0;
  wa.kl = (prob->mode & AAL_KL) != 0;
  wa.tv = (prob->mode & AAL_TV) != 0;
  wa.w_greedy = prob->w_greedy;
  wa.w_sampling = prob->w_sampling;
  wa.w_kl = prob->w_kl;
  wa.w_tv = prob->w_tv;
  wa.loss = loss;
  wa.eal = eal;
  wa.pg = reinterpret_cast<float*>(base + L.pg);
  wa.ps = reinterpret_cast<float*>(base + L.ps);
  wa.ws = loss_ws(workspace, L.base);
  wa.nwblk = L.base.nwblk;
  wa.nvalid_g = prob->global_counts == 1 ? (int32_t)prob->n_windows_global : -1;
  wa.npos_g = prob->global_counts == 1 ? (int32_t)prob->n_positions_global : -1;
  return wa;
}

// The window flags and weights the fused kernels' sequence exchange reads (win.N and win.mask
// are not used in the sequence layout).
WindowArgs seq_fused_win(const SeqWindowArgs& wa, int64_t R) {
  WindowArgs w{};
  w.N = R;
  w.K = wa.K;
  w.greedy = wa.greedy;
  w.sampling = wa.sampling;
  w.kl = wa.kl;
  w.tv = wa.tv;
  w.w_greedy = wa.w_greedy;
  w.w_sampling = wa.w_sampling;
  w.w_kl = wa.w_kl;
  w.w_tv = wa.w_tv;
  return w;
}

}  // namespace

namespace aal {
uint64_t debug_wait_limit_ns() { return g_wait_limit_ns.load(); }
int64_t fused_min_row_bytes() { return g_fused_min_row_bytes.load(); }
int64_t debug_take_skip_chunk() { return g_skip_chunk.exchange(-1); }
}  // namespace aal

extern "C" {

int32_t aal_abi_version(void) { return 10700; }

void aal_debug_fail_next_forward(int64_t chunk, uint64_t wait_limit_ns) {
  g_wait_limit_ns.store(wait_limit_ns);
  g_skip_chunk.store(chunk);
}

void aal_debug_fused_min_row_bytes(int64_t bytes) {
  g_fused_min_row_bytes.store(bytes < 0 ? (int64_t)AAL_FUSED_MIN_ROW_BYTES_DEFAULT : bytes);
}

int64_t aal_debug_solo_windows(int64_t N, int32_t K, int32_t G, int32_t S) {
  return aal::solo_windows_each(N, K, G, S);
}

const char* aal_status_string(aal_status s) {
  switch (s) {
    case AAL_OK: return "AAL_OK";
    case AAL_ERR_INVALID_ARG: return "AAL_ERR_INVALID_ARG: a NULL, misaligned or out-of-range argument";
    case AAL_ERR_UNSUPPORTED: return "AAL_ERR_UNSUPPORTED: valid request this build does not handle";
    case AAL_ERR_WORKSPACE: return "AAL_ERR_WORKSPACE: workspace missing or too small";
    case AAL_ERR_CUDA: return "AAL_ERR_CUDA: a CUDA call or kernel launch failed";
    case AAL_ERR_TIMEOUT: return "AAL_ERR_TIMEOUT: a device-side bounded wait ran out";
  }
  return "unknown aal_status";
}

aal_status aal_workspace_size(const aal_problem* prob, size_t* bytes) {
  aal_status st = check_problem(prob);
  if (st != AAL_OK) return st;
  if (bytes == nullptr) return AAL_ERR_INVALID_ARG;
  *bytes = loss_layout(prob->N, prob->K).total;
  return AAL_OK;
}

aal_status aal_reward_workspace_size(const aal_reward_problem* prob, size_t* bytes) {
  aal_status st = check_reward(prob);
  if (st != AAL_OK) return st;
  if (bytes == nullptr) return AAL_ERR_INVALID_ARG;
  *bytes = reward_layout(prob->N, prob->K).total;
  return AAL_OK;
}

aal_status aal_loss_fwd(const aal_problem* prob, const void* draft, const void* target,
                        const uint8_t* mask, void* workspace, size_t workspace_bytes, float* loss,
                        float* eal, void* stream) {
  aal_status st = check_problem(prob);
  if (st != AAL_OK) return st;
  if (loss == nullptr || !aligned(loss, 4) || (eal != nullptr && !aligned(eal, 4))) return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (prob->N == 0) return cuda_status(cudaMemsetAsync(loss, 0, sizeof(float), s));
  if (draft == nullptr || target == nullptr || !aligned(draft, 16) || !aligned(target, target_align(prob->mode)))
    return AAL_ERR_INVALID_ARG;
  const LossLayout L = loss_layout(prob->N, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;

  LossWs ws = loss_ws(workspace, L);
  cudaError_t e = cudaMemsetAsync(ws.hdr, 0, sizeof(WsHeader), s);
  if (e != cudaSuccess) return AAL_ERR_CUDA;
  if (prob->mode & AAL_GRPO) {  // no GRPO term until aal_grpo_from_loss writes one
    e = cudaMemsetAsync(ws.cgr, 0, (size_t)L.R * sizeof(float), s);
    if (e != cudaSuccess) return AAL_ERR_CUDA;
  }
  int cluster = 1;
  e = launch_stats(draft, target, L.R, prob->V, prob->dtype, prob->mode, prob->temperature, ws, s, &cluster);
  if (e != cudaSuccess) return AAL_ERR_CUDA;
  return cuda_status(launch_window(window_args(prob, mask, cluster, loss, eal, ws, L.nwblk), s));
}

aal_status aal_loss_bwd(const aal_problem* prob, const void* draft, const void* target,
                        const uint8_t* mask, const void* workspace, size_t workspace_bytes, float dloss,
                        void* grad_draft, void* stream) {
  // the forward folded the mask into dE/da (zero outside each window's valid prefix); the
  // anchor's rows are the valid positions themselves
  aal_status st = check_problem(prob);
  if (st != AAL_OK) return st;
  if (!isfinite(dloss)) return AAL_ERR_INVALID_ARG;
  if (prob->N == 0) return AAL_OK;
  if (draft == nullptr || target == nullptr || grad_draft == nullptr || !aligned(draft, 16) ||
      !aligned(target, target_align(prob->mode)) || !aligned(grad_draft, 16))
    return AAL_ERR_INVALID_ARG;
  const LossLayout L = loss_layout(prob->N, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  return cuda_status(launch_grad(draft, target, mask, L.R, prob->V, prob->dtype, prob->mode,
                                 prob->temperature, prob->w_greedy, prob->w_sampling, prob->w_kl, dloss,
                                 loss_ws(const_cast<void*>(workspace), L), grad_draft,
                                 static_cast<cudaStream_t>(stream)));
}

aal_status aal_loss_fwd_bwd(const aal_problem* prob, const void* draft, const void* target,
                            const uint8_t* mask, void* workspace, size_t workspace_bytes, float dloss,
                            float* loss, float* eal, void* grad_draft, void* stream) {
  aal_status st = check_problem(prob);
  if (st != AAL_OK) return st;
  if (prob->mode & AAL_GRPO) return AAL_ERR_UNSUPPORTED;  // its coefficients come between the two
  if (!isfinite(dloss)) return AAL_ERR_INVALID_ARG;
  if (loss == nullptr || !aligned(loss, 4) || (eal != nullptr && !aligned(eal, 4))) return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (prob->N == 0) return cuda_status(cudaMemsetAsync(loss, 0, sizeof(float), s));
  if (draft == nullptr || target == nullptr || grad_draft == nullptr || !aligned(draft, 16) ||
      !aligned(target, target_align(prob->mode)) || !aligned(grad_draft, 16))
    return AAL_ERR_INVALID_ARG;
  const LossLayout L = loss_layout(prob->N, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;

  // the fused kernels: bf16 rows of 16-byte multiples; with token ids, the draft alone
  const bool ids = (prob->mode & AAL_IDS) != 0;
  const bool rows16 = prob->dtype == AAL_BF16 && (prob->V * 2) % 16 == 0 &&
                      prob->V * 2 >= g_fused_min_row_bytes.load();
  const bool fusable = rows16 && !ids;
  if (rows16 && ids) {
    LossWs ws = loss_ws(workspace, L);
    if (cudaMemsetAsync(ws.hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;
    if (cudaMemsetAsync(ws.mbox, 0xff, (size_t)L.R * 8, s) != cudaSuccess) return AAL_ERR_CUDA;  // kMboxEmpty
    FusedIdsArgs f;
    f.win = window_args(prob, mask, 1, loss, eal, ws, L.nwblk);
    if (launch_count_valid(mask, prob->N, (int32_t)prob->K, f.win.nvalid_g, f.win.npos_g, ws.hdr, s) != cudaSuccess)
      return AAL_ERR_CUDA;
    f.st = ids_args(draft, target, L.R, prob->V, ws);
    f.bw = grad_args(draft, target, mask, L.R, prob->V, prob->mode, prob->temperature, prob->w_greedy,
                     prob->w_kl, dloss, ws, grad_draft);
    f.groups = 0;
    const uint64_t limit = debug_wait_limit_ns();
    bool launched = false;
    if (launch_fused_ids(f, s, limit ? limit : kWaitLimitNs, &launched) != cudaSuccess) return AAL_ERR_CUDA;
    if (launched) return cuda_status(launch_window(f.win, s));
  }
  if (fusable) {
    LossWs ws = loss_ws(workspace, L);
    if (cudaMemsetAsync(ws.hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;
    if (cudaMemsetAsync(ws.mbox, 0xff, (size_t)L.R * 8, s) != cudaSuccess) return AAL_ERR_CUDA;  // kMboxEmpty
    FusedArgs f;
    f.win = window_args(prob, mask, 1, loss, eal, ws, L.nwblk);
    if (launch_count_valid(mask, prob->N, (int32_t)prob->K, f.win.nvalid_g, f.win.npos_g, ws.hdr, s) != cudaSuccess)
      return AAL_ERR_CUDA;
    f.st = stats_args(draft, target, L.R, prob->V, prob->mode, prob->temperature, ws);
    f.bw = grad_args(draft, target, mask, L.R, prob->V, prob->mode, prob->temperature, prob->w_greedy,
                     prob->w_kl, dloss, ws, grad_draft);
    f.groups = 0;
    const uint64_t limit = debug_wait_limit_ns();
    bool launched = false;
    if (launch_fused(f, s, limit ? limit : kWaitLimitNs, &launched) != cudaSuccess) return AAL_ERR_CUDA;
    // the loss from the statistics the fused kernel wrote, as aal_loss_fwd forms it
    if (launched) return cuda_status(launch_window(f.win, s));
  }
  st = aal_loss_fwd(prob, draft, target, mask, workspace, workspace_bytes, loss, eal, stream);
  if (st != AAL_OK) return st;
  return aal_loss_bwd(prob, draft, target, mask, workspace, workspace_bytes, dloss, grad_draft, stream);
}

aal_status aal_seq_workspace_size(const aal_seq_problem* prob, size_t* bytes) {
  aal_status st = check_seq(prob);
  if (st != AAL_OK) return st;
  if (bytes == nullptr) return AAL_ERR_INVALID_ARG;
  *bytes = seq_layout(prob->B, prob->seq_len, prob->K).total;
  return AAL_OK;
}

aal_status aal_seq_loss_fwd(const aal_seq_problem* prob, const void* draft, const void* target,
                            const uint8_t* mask, void* workspace, size_t workspace_bytes, float* loss,
                            float* eal, void* stream) {
  aal_status st = check_seq(prob);
  if (st != AAL_OK) return st;
  if (loss == nullptr || !aligned(loss, 4) || (eal != nullptr && !aligned(eal, 4))) return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t R = prob->B * prob->seq_len;
  if (R == 0) return cuda_status(cudaMemsetAsync(loss, 0, sizeof(float), s));
  if (draft == nullptr || target == nullptr || !aligned(draft, 16) || !aligned(target, target_align(prob->mode)))
    return AAL_ERR_INVALID_ARG;
  const SeqLayout L = seq_layout(prob->B, prob->seq_len, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;

  LossWs ws = loss_ws(workspace, L.base);
  cudaError_t e = cudaMemsetAsync(ws.hdr, 0, sizeof(WsHeader), s);
  if (e != cudaSuccess) return AAL_ERR_CUDA;
  if (prob->mode & AAL_GRPO) {  // no GRPO term until aal_seq_grpo_from_loss writes one
    e = cudaMemsetAsync(ws.cgr, 0, (size_t)R * sizeof(float), s);
    if (e != cudaSuccess) return AAL_ERR_CUDA;
  }
  int cluster = 1;
  e = launch_stats(draft, target, R, prob->V, prob->dtype, prob->mode, prob->temperature, ws, s, &cluster);
  if (e != cudaSuccess) return AAL_ERR_CUDA;

  return cuda_status(launch_seq_window(seq_window_args(prob, mask, cluster, loss, eal, workspace, L), s));
}

aal_status aal_seq_loss_bwd(const aal_seq_problem* prob, const void* draft, const void* target,
                            const uint8_t* mask, const void* workspace, size_t workspace_bytes, float dloss,
                            void* grad_draft, void* stream) {
  // dE/da carries the windows' masks; the anchor's rows are the valid positions
  aal_status st = check_seq(prob);
  if (st != AAL_OK) return st;
  if (!isfinite(dloss)) return AAL_ERR_INVALID_ARG;
  const int64_t R = prob->B * prob->seq_len;
  if (R == 0) return AAL_OK;
  if (draft == nullptr || target == nullptr || grad_draft == nullptr || !aligned(draft, 16) ||
      !aligned(target, target_align(prob->mode)) || !aligned(grad_draft, 16))
    return AAL_ERR_INVALID_ARG;
  const SeqLayout L = seq_layout(prob->B, prob->seq_len, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  return cuda_status(launch_grad(draft, target, mask, R, prob->V, prob->dtype, prob->mode,
                                 prob->temperature, prob->w_greedy, prob->w_sampling, prob->w_kl, dloss,
                                 loss_ws(const_cast<void*>(workspace), L.base), grad_draft,
                                 static_cast<cudaStream_t>(stream)));
}

aal_status aal_seq_loss_fwd_bwd(const aal_seq_problem* prob, const void* draft, const void* target,
                                const uint8_t* mask, void* workspace, size_t workspace_bytes, float dloss,
                                float* loss, float* eal, void* grad_draft, void* stream) {
  aal_status st = check_seq(prob);
  if (st != AAL_OK) return st;
  if (prob->mode & AAL_GRPO) return AAL_ERR_UNSUPPORTED;  // its coefficients come between the two
  if (!isfinite(dloss)) return AAL_ERR_INVALID_ARG;
  if (loss == nullptr || !aligned(loss, 4) || (eal != nullptr && !aligned(eal, 4))) return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t R = prob->B * prob->seq_len;
  if (R == 0) return cuda_status(cudaMemsetAsync(loss, 0, sizeof(float), s));
  if (draft == nullptr || target == nullptr || grad_draft == nullptr || !aligned(draft, 16) ||
      !aligned(target, target_align(prob->mode)) || !aligned(grad_draft, 16))
    return AAL_ERR_INVALID_ARG;
  const SeqLayout L = seq_layout(prob->B, prob->seq_len, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;

  // the fused kernels: bf16 rows of 16-byte multiples (both tensors as logits, or the draft with
  // token ids), and a round of rows (one per SM) that spans a window or holds every row (their
  // order is deadlock-free then)
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return AAL_ERR_CUDA;
  const bool rows16 = prob->dtype == AAL_BF16 && (prob->V * 2) % 16 == 0 &&
                      prob->V * 2 >= g_fused_min_row_bytes.load() && (sms >= prob->K || R <= sms);
  const bool ids = (prob->mode & AAL_IDS) != 0;
  if (rows16 && ids) {  // x* as token ids: the draft alone is streamed
    LossWs ws = loss_ws(workspace, L.base);
    if (cudaMemsetAsync(ws.hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;
    if (cudaMemsetAsync(ws.mbox, 0xff, (size_t)R * 8, s) != cudaSuccess) return AAL_ERR_CUDA;  // kMboxEmpty
    const SeqWindowArgs wa = seq_window_args(prob, mask, 1, loss, eal, workspace, L);
    if (launch_seq_count_valid(mask, prob->B, prob->seq_len, (int32_t)prob->K, wa.full_windows, wa.nvalid_g,
                               wa.npos_g, ws.hdr, s) != cudaSuccess)
      return AAL_ERR_CUDA;
    FusedIdsArgs f;
    f.st = ids_args(draft, target, R, prob->V, ws);
    f.bw = grad_args(draft, target, mask, R, prob->V, prob->mode, prob->temperature, prob->w_greedy, prob->w_kl,
                     dloss, ws, grad_draft);
    f.win = seq_fused_win(wa, R);
    f.groups = 0;
    f.solos = 0;
    f.n_group = 0;
    f.seq_T = prob->seq_len;
    f.seq_full = wa.full_windows ? 1 : 0;
    f.seq_mask = mask;
    const uint64_t limit = debug_wait_limit_ns();
    bool launched = false;
    if (launch_fused_ids_seq(f, s, limit ? limit : kWaitLimitNs, &launched) != cudaSuccess) return AAL_ERR_CUDA;
    if (launched) return cuda_status(launch_seq_window(wa, s));
  }
  const bool fusable = rows16 && !ids;
  if (fusable) {
    LossWs ws = loss_ws(workspace, L.base);
    if (cudaMemsetAsync(ws.hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;
    if (cudaMemsetAsync(ws.mbox, 0xff, (size_t)R * 8, s) != cudaSuccess) return AAL_ERR_CUDA;  // kMboxEmpty
    const SeqWindowArgs wa = seq_window_args(prob, mask, 1, loss, eal, workspace, L);
    if (launch_seq_count_valid(mask, prob->B, prob->seq_len, (int32_t)prob->K, wa.full_windows, wa.nvalid_g,
                               wa.npos_g, ws.hdr, s) != cudaSuccess)
      return AAL_ERR_CUDA;
    FusedArgs f;
    f.st = stats_args(draft, target, R, prob->V, prob->mode, prob->temperature, ws);
    f.bw = grad_args(draft, target, mask, R, prob->V, prob->mode, prob->temperature, prob->w_greedy, prob->w_kl,
                     dloss, ws, grad_draft);
    f.win = seq_fused_win(wa, R);
    f.groups = 0;
    f.solos = 0;
    f.n_group = 0;
    f.seq_T = prob->seq_len;
    f.seq_full = wa.full_windows ? 1 : 0;
    f.seq_mask = mask;
    const uint64_t limit = debug_wait_limit_ns();
    bool launched = false;
    if (launch_fused_seq(f, s, limit ? limit : kWaitLimitNs, &launched) != cudaSuccess) return AAL_ERR_CUDA;
    // the loss from the statistics the fused kernel wrote, and each position's dE/da, as
    // aal_seq_loss_fwd forms them (the workspace then serves aal_seq_loss_bwd as well)
    if (launched) return cuda_status(launch_seq_window(wa, s));
  }
  st = aal_seq_loss_fwd(prob, draft, target, mask, workspace, workspace_bytes, loss, eal, stream);
  if (st != AAL_OK) return st;
  return aal_seq_loss_bwd(prob, draft, target, mask, workspace, workspace_bytes, dloss, grad_draft, stream);
}

aal_status aal_grpo_workspace_size(const aal_grpo_problem* prob, size_t* bytes) {
  aal_status st = check_grpo(prob);
  if (st != AAL_OK) return st;
  if (bytes == nullptr) return AAL_ERR_INVALID_ARG;
  *bytes = grpo_layout(prob->N, prob->K, prob->windows_per_rollout).total;
  return AAL_OK;
}

aal_status aal_grpo_from_loss(const aal_grpo_problem* gprob, const aal_problem* lprob, void* loss_workspace,
                              size_t loss_workspace_bytes, const void* ref_draft, void* workspace,
                              size_t workspace_bytes, float* grpo_loss, int32_t* tau, int32_t* tau_ref,
                              float* advantage, float* log_rho, void* stream) {
  aal_status st = check_grpo(gprob);
  if (st != AAL_OK) return st;
  st = check_problem(lprob);
  if (st != AAL_OK) return st;
  if (!(lprob->mode & AAL_GRPO)) return AAL_ERR_INVALID_ARG;
  if (gprob->N != lprob->N || gprob->K != lprob->K || gprob->V != lprob->V || gprob->dtype != lprob->dtype)
    return AAL_ERR_INVALID_ARG;
  if (grpo_loss == nullptr || !aligned(grpo_loss, 4) || (tau != nullptr && !aligned(tau, 4)) ||
      (tau_ref != nullptr && !aligned(tau_ref, 4)) || (advantage != nullptr && !aligned(advantage, 4)) ||
      (log_rho != nullptr && !aligned(log_rho, 4)))
    return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (gprob->N == 0) return cuda_status(cudaMemsetAsync(grpo_loss, 0, sizeof(float), s));
  if (ref_draft == nullptr || !aligned(ref_draft, 16)) return AAL_ERR_INVALID_ARG;
  const LossLayout LL = loss_layout(lprob->N, lprob->K);
  if (loss_workspace == nullptr || !aligned(loss_workspace, 256) || loss_workspace_bytes < LL.total)
    return AAL_ERR_WORKSPACE;
  const GrpoLayout L = grpo_layout(gprob->N, gprob->K, gprob->windows_per_rollout);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  char* base = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(base + L.hdr);
  if (cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;
  const LossWs lws = loss_ws(loss_workspace, LL);

  Stream1Args ra;
  ra.z = ref_draft;
  ra.R = L.R;
  ra.V = gprob->V;
  ra.lws = lws;
  ra.ids = nullptr;
  ra.acc = reinterpret_cast<uint8_t*>(base + L.acc);
  ra.acc_ref = reinterpret_cast<uint8_t*>(base + L.acc_ref);
  ra.lpr = reinterpret_cast<float*>(base + L.lpr);
  ra.hdr = hdr;
  ra.skip_chunk = debug_take_skip_chunk();
  if (launch_one_tensor(ra, gprob->dtype == AAL_BF16, false, s) != cudaSuccess) return AAL_ERR_CUDA;

  float* adv = advantage != nullptr ? advantage : reinterpret_cast<float*>(base + L.adv);
  RewardGroupArgs ga;
  ga.acc = ra.acc;
  ga.acc_ref = ra.acc_ref;
  ga.rbuf = reinterpret_cast<float*>(base + L.rbuf);
  ga.N = gprob->N;
  ga.K = (int32_t)gprob->K;
  ga.wpr = gprob->windows_per_rollout;
  ga.rpg = gprob->rollouts_per_group;
  ga.adv_clip = gprob->adv_clip;
  ga.tau = tau != nullptr ? tau : reinterpret_cast<int32_t*>(base + L.tau);
  ga.tau_ref = tau_ref != nullptr ? tau_ref : reinterpret_cast<int32_t*>(base + L.tau_ref);
  ga.rollout_len = reinterpret_cast<float*>(base + L.rl);
  ga.advantage = adv;
  if (launch_reward_groups(ga, s) != cudaSuccess) return AAL_ERR_CUDA;

  GrpoWindowArgs wa;
  wa.lws = lws;
  wa.lpr = ra.lpr;
  wa.starts = nullptr;
  wa.RP = 0;
  wa.cw = nullptr;
  wa.adv = adv;
  wa.N = gprob->N;
  wa.K = (int32_t)gprob->K;
  wa.wpr = gprob->windows_per_rollout;
  wa.eps_clip = gprob->eps_clip;
  wa.rho_min = gprob->rho_min;
  wa.rho_max = gprob->rho_max;
  wa.log_rho_clip = gprob->log_rho_clip;
  wa.w_grpo = gprob->w_grpo;
  wa.log_rho = log_rho;
  wa.part = reinterpret_cast<double*>(base + L.part);
  wa.nblk = L.nblk;
  wa.hdr = hdr;
  wa.loss = grpo_loss;
  return cuda_status(launch_grpo_windows(wa, s));
}

aal_status aal_seq_grpo_workspace_size(const aal_grpo_problem* gprob, const aal_seq_problem* sprob, size_t* bytes) {
  aal_status st = check_grpo(gprob);
  if (st != AAL_OK) return st;
  st = check_seq(sprob);
  if (st != AAL_OK) return st;
  if (bytes == nullptr) return AAL_ERR_INVALID_ARG;
  *bytes = seq_grpo_layout(gprob->N, gprob->K, gprob->windows_per_rollout, sprob->B * sprob->seq_len).total;
  return AAL_OK;
}

aal_status aal_seq_grpo_from_loss(const aal_grpo_problem* gprob, const aal_seq_problem* sprob, void* loss_workspace,
                                  size_t loss_workspace_bytes, const void* ref_draft, const int32_t* starts,
                                  void* workspace, size_t workspace_bytes, float* grpo_loss, int32_t* tau,
                                  int32_t* tau_ref, float* advantage, float* log_rho, void* stream) {
  aal_status st = check_grpo(gprob);
  if (st != AAL_OK) return st;
  st = check_seq(sprob);
  if (st != AAL_OK) return st;
  if (!(sprob->mode & AAL_GRPO)) return AAL_ERR_INVALID_ARG;
  if (gprob->K != sprob->K || gprob->V != sprob->V || gprob->dtype != sprob->dtype) return AAL_ERR_INVALID_ARG;
  if (grpo_loss == nullptr || !aligned(grpo_loss, 4) || (tau != nullptr && !aligned(tau, 4)) ||
      (tau_ref != nullptr && !aligned(tau_ref, 4)) || (advantage != nullptr && !aligned(advantage, 4)) ||
      (log_rho != nullptr && !aligned(log_rho, 4)))
    return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t RP = sprob->B * sprob->seq_len;
  if (RP == 0) return cuda_status(cudaMemsetAsync(grpo_loss, 0, sizeof(float), s));
  if (ref_draft == nullptr || !aligned(ref_draft, 16)) return AAL_ERR_INVALID_ARG;
  if (gprob->N > 0 && (starts == nullptr || !aligned(starts, 4))) return AAL_ERR_INVALID_ARG;
  const SeqLayout SL = seq_layout(sprob->B, sprob->seq_len, sprob->K);
  if (loss_workspace == nullptr || !aligned(loss_workspace, 256) || loss_workspace_bytes < SL.total)
    return AAL_ERR_WORKSPACE;
  const SeqGrpoLayout L = seq_grpo_layout(gprob->N, gprob->K, gprob->windows_per_rollout, RP);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  char* base = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(base + L.g.hdr);
  if (cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;
  const LossWs lws = loss_ws(loss_workspace, SL.base);

  // the reference pass over every position: log pi_ref at the draft's token, both flags
  Stream1Args ra;
  ra.z = ref_draft;
  ra.R = RP;
  ra.V = gprob->V;
  ra.lws = lws;
  ra.ids = nullptr;
  ra.acc = reinterpret_cast<uint8_t*>(base + L.acc_pos);
  ra.acc_ref = reinterpret_cast<uint8_t*>(base + L.accr_pos);
  ra.lpr = reinterpret_cast<float*>(base + L.lpr_pos);
  ra.hdr = hdr;
  ra.skip_chunk = debug_take_skip_chunk();
  if (launch_one_tensor(ra, gprob->dtype == AAL_BF16, false, s) != cudaSuccess) return AAL_ERR_CUDA;

  if (gprob->N == 0) {  // no windows: no GRPO term
    if (cudaMemsetAsync(lws.cgr, 0, (size_t)RP * sizeof(float), s) != cudaSuccess) return AAL_ERR_CUDA;
    return cuda_status(cudaMemsetAsync(grpo_loss, 0, sizeof(float), s));
  }
  SeqGrpoArgs qa;
  qa.starts = starts;
  qa.N = gprob->N;
  qa.T = sprob->seq_len;
  qa.RP = RP;
  qa.K = (int32_t)gprob->K;
  qa.acc_pos = ra.acc;
  qa.accr_pos = ra.acc_ref;
  qa.acc = reinterpret_cast<uint8_t*>(base + L.g.acc);
  qa.acc_ref = reinterpret_cast<uint8_t*>(base + L.g.acc_ref);
  qa.cw = reinterpret_cast<float*>(base + L.cw);
  qa.cgr = lws.cgr;
  qa.hdr = hdr;
  if (launch_seq_grpo_gather(qa, s) != cudaSuccess) return AAL_ERR_CUDA;

  float* adv = advantage != nullptr ? advantage : reinterpret_cast<float*>(base + L.g.adv);
  RewardGroupArgs ga;
  ga.acc = qa.acc;
  ga.acc_ref = qa.acc_ref;
  ga.rbuf = reinterpret_cast<float*>(base + L.g.rbuf);
  ga.N = gprob->N;
  ga.K = (int32_t)gprob->K;
  ga.wpr = gprob->windows_per_rollout;
  ga.rpg = gprob->rollouts_per_group;
  ga.adv_clip = gprob->adv_clip;
  ga.tau = tau != nullptr ? tau : reinterpret_cast<int32_t*>(base + L.g.tau);
  ga.tau_ref = tau_ref != nullptr ? tau_ref : reinterpret_cast<int32_t*>(base + L.g.tau_ref);
  ga.rollout_len = reinterpret_cast<float*>(base + L.g.rl);
  ga.advantage = adv;
  if (launch_reward_groups(ga, s) != cudaSuccess) return AAL_ERR_CUDA;

  GrpoWindowArgs wa;
  wa.lws = lws;
  wa.lpr = ra.lpr;
  wa.starts = starts;
  wa.RP = RP;
  wa.cw = reinterpret_cast<float*>(base + L.cw);
  wa.adv = adv;
  wa.N = gprob->N;
  wa.K = (int32_t)gprob->K;
  wa.wpr = gprob->windows_per_rollout;
  wa.eps_clip = gprob->eps_clip;
  wa.rho_min = gprob->rho_min;
  wa.rho_max = gprob->rho_max;
  wa.log_rho_clip = gprob->log_rho_clip;
  wa.w_grpo = gprob->w_grpo;
  wa.log_rho = log_rho;
  wa.part = reinterpret_cast<double*>(base + L.g.part);
  wa.nblk = L.g.nblk;
  wa.hdr = hdr;
  wa.loss = grpo_loss;
  if (launch_grpo_windows(wa, s) != cudaSuccess) return AAL_ERR_CUDA;
  return cuda_status(launch_seq_grpo_scatter(qa, s));
}

aal_status aal_accept_reward(const aal_reward_problem* prob, const void* draft, const void* target,
                             const void* ref_draft, void* workspace, size_t workspace_bytes, int32_t* tau,
                             int32_t* tau_ref, float* rollout_len, float* advantage, void* stream) {
  aal_status st = check_reward(prob);
  if (st != AAL_OK) return st;
  if (prob->N == 0) return AAL_OK;
  if (draft == nullptr || target == nullptr || !aligned(draft, 16) || !aligned(target, 16) ||
      (ref_draft != nullptr && !aligned(ref_draft, 16)))
    return AAL_ERR_INVALID_ARG;
  if (tau == nullptr || rollout_len == nullptr || advantage == nullptr || !aligned(tau, 4) ||
      !aligned(rollout_len, 4) || !aligned(advantage, 4) || (tau_ref != nullptr && !aligned(tau_ref, 4)))
    return AAL_ERR_INVALID_ARG;
  const RewardLayout L = reward_layout(prob->N, prob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(base + L.hdr);
  if (cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;

  const bool sampling = (prob->mode & AAL_SAMPLING) != 0;
  RewardRowArgs ra;
  ra.sampled_draft = (prob->mode & AAL_SAMPLED_DRAFT) != 0;
  ra.zq = draft;
  ra.zp = target;
  ra.zr = ref_draft;
  ra.R = L.R;
  ra.V = prob->V;
  ra.K = (int32_t)prob->K;
  ra.sampling = sampling;
  ra.sT = sampling ? kLog2e / prob->temperature : 0.f;
  ra.seed = prob->seed;
  ra.row_offset = prob->row_offset;
  ra.acc = reinterpret_cast<uint8_t*>(base + L.acc);
  ra.acc_ref = reinterpret_cast<uint8_t*>(base + L.acc_ref);
  ra.hdr = hdr;
  cudaError_t e = cudaSuccess;
  if (sampling && !ra.sampled_draft && ref_draft == nullptr && prob->dtype == AAL_BF16 && (prob->V * 2) % 16 == 0) {
    // the argmax draft under sampling verification: one TMA-streamed pass over draft and target
    // (both normalisers at T and the draft's greedy token), the flag decided at each row's end
    RowStatsArgs sa{};
    sa.zq = draft;
    sa.zp = target;
    sa.R = L.R;
    sa.V = prob->V;
    sa.sT = ra.sT;
    sa.skip_chunk = -1;
    sa.ws.hdr = hdr;
    sa.acc = ra.acc;
    sa.seed = prob->seed;
    sa.row_offset = prob->row_offset;
    sa.K = (int32_t)prob->K;
    const uint64_t limit = debug_wait_limit_ns();
    // the geometry the loss forward takes for rows of this length (the same normalisers)
    e = prob->V * 2 < fused_min_row_bytes() ? launch_reward_stream_short(sa, s, limit ? limit : kWaitLimitNs)
                                            : launch_reward_stream(sa, s, limit ? limit : kWaitLimitNs);
  } else {
    e = launch_reward_rows(ra, prob->dtype == AAL_BF16, s);
  }
  if (e != cudaSuccess) return AAL_ERR_CUDA;

  RewardGroupArgs ga;
  ga.acc = ra.acc;
  ga.acc_ref = ref_draft != nullptr ? ra.acc_ref : nullptr;
  ga.rbuf = reinterpret_cast<float*>(base + L.rbuf);
  ga.N = prob->N;
  ga.K = (int32_t)prob->K;
  ga.wpr = prob->windows_per_rollout;
  ga.rpg = prob->rollouts_per_group;
  ga.adv_clip = prob->adv_clip;
  ga.tau = tau;
  ga.tau_ref = ref_draft != nullptr ? tau_ref : nullptr;
  ga.rollout_len = rollout_len;
  ga.advantage = advantage;
  return cuda_status(launch_reward_groups(ga, s));
}

aal_status aal_accept_reward_from_loss(const aal_reward_problem* rprob, const aal_problem* lprob,
                                       const void* loss_workspace, size_t loss_workspace_bytes, void* workspace,
                                       size_t workspace_bytes, int32_t* tau, float* rollout_len, float* advantage,
                                       void* stream) {
  aal_status st = check_reward(rprob);
  if (st != AAL_OK) return st;
  st = check_problem(lprob);
  if (st != AAL_OK) return st;
  if (rprob->N != lprob->N || rprob->K != lprob->K || rprob->V != lprob->V || rprob->dtype != lprob->dtype)
    return AAL_ERR_INVALID_ARG;
  // a sampled draft token needs the logits (one noise draw per vocabulary entry)
  if (rprob->mode & AAL_SAMPLED_DRAFT) return AAL_ERR_INVALID_ARG;
  const bool sampling = rprob->mode == AAL_SAMPLING;
  // the sampling acceptance needs the loss's temperature-scaled normalisers at this T
  if (sampling && (!(lprob->mode & AAL_SAMPLING) || lprob->temperature != rprob->temperature))
    return AAL_ERR_INVALID_ARG;
  if (rprob->N == 0) return AAL_OK;
  if (tau == nullptr || rollout_len == nullptr || advantage == nullptr || !aligned(tau, 4) ||
      !aligned(rollout_len, 4) || !aligned(advantage, 4))
    return AAL_ERR_INVALID_ARG;
  const LossLayout LL = loss_layout(lprob->N, lprob->K);
  if (loss_workspace == nullptr || !aligned(loss_workspace, 256) || loss_workspace_bytes < LL.total)
    return AAL_ERR_WORKSPACE;
  const RewardLayout L = reward_layout(rprob->N, rprob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(base + L.hdr);
  if (cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;

  RewardStatsArgs fa;
  fa.ws = loss_ws(const_cast<void*>(loss_workspace), LL);
  fa.R = LL.R;
  fa.K = (int32_t)rprob->K;
  fa.sampling = sampling;
  fa.sT = sampling ? kLog2e / rprob->temperature : 0.f;
  fa.seed = rprob->seed;
  fa.row_offset = rprob->row_offset;
  fa.acc = reinterpret_cast<uint8_t*>(base + L.acc);
  if (launch_reward_flags_from_stats(fa, s) != cudaSuccess) return AAL_ERR_CUDA;

  RewardGroupArgs ga;
  ga.acc = fa.acc;
  ga.acc_ref = nullptr;
  ga.rbuf = reinterpret_cast<float*>(base + L.rbuf);
  ga.N = rprob->N;
  ga.K = (int32_t)rprob->K;
  ga.wpr = rprob->windows_per_rollout;
  ga.rpg = rprob->rollouts_per_group;
  ga.adv_clip = rprob->adv_clip;
  ga.tau = tau;
  ga.tau_ref = nullptr;
  ga.rollout_len = rollout_len;
  ga.advantage = advantage;
  return cuda_status(launch_reward_groups(ga, s));
}

aal_status aal_accept_reward_sampled_from_loss(const aal_reward_problem* rprob, const aal_problem* lprob,
                                               const void* draft, const void* target, const void* loss_workspace,
                                               size_t loss_workspace_bytes, void* workspace, size_t workspace_bytes,
                                               int32_t* tau, float* rollout_len, float* advantage, void* stream) {
  aal_status st = check_reward(rprob);
  if (st != AAL_OK) return st;
  st = check_problem(lprob);
  if (st != AAL_OK) return st;
  if (rprob->N != lprob->N || rprob->K != lprob->K || rprob->V != lprob->V || rprob->dtype != lprob->dtype)
    return AAL_ERR_INVALID_ARG;
  if (rprob->mode != (AAL_SAMPLING | AAL_SAMPLED_DRAFT)) return AAL_ERR_INVALID_ARG;
  // the acceptance needs the loss's temperature-scaled normalisers at this T, from both logit tensors
  if (!(lprob->mode & AAL_SAMPLING) || (lprob->mode & AAL_IDS) || lprob->temperature != rprob->temperature)
    return AAL_ERR_INVALID_ARG;
  if (rprob->N == 0) return AAL_OK;
  if (draft == nullptr || target == nullptr || !aligned(draft, 16) || !aligned(target, 16)) return AAL_ERR_INVALID_ARG;
  if (tau == nullptr || rollout_len == nullptr || advantage == nullptr || !aligned(tau, 4) ||
      !aligned(rollout_len, 4) || !aligned(advantage, 4))
    return AAL_ERR_INVALID_ARG;
  const LossLayout LL = loss_layout(lprob->N, lprob->K);
  if (loss_workspace == nullptr || !aligned(loss_workspace, 256) || loss_workspace_bytes < LL.total)
    return AAL_ERR_WORKSPACE;
  const RewardLayout L = reward_layout(rprob->N, rprob->K);
  if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < L.total) return AAL_ERR_WORKSPACE;
  const int64_t elt = rprob->dtype == AAL_BF16 ? 2 : 4;
  if ((rprob->V * elt) % 16 != 0)  // rows that are not 16-byte multiples: the reward's own pass
    return aal_accept_reward(rprob, draft, target, nullptr, workspace, workspace_bytes, tau, nullptr, rollout_len,
                             advantage, stream);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* base = static_cast<char*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(base + L.hdr);
  if (cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s) != cudaSuccess) return AAL_ERR_CUDA;

  RewardRowArgs ra;
  ra.sampled_draft = true;
  ra.zq = draft;
  ra.zp = target;
  ra.zr = nullptr;
  ra.R = L.R;
  ra.V = rprob->V;
  ra.K = (int32_t)rprob->K;
  ra.sampling = true;
  ra.sT = kLog2e / rprob->temperature;
  ra.seed = rprob->seed;
  ra.row_offset = rprob->row_offset;
  ra.acc = reinterpret_cast<uint8_t*>(base + L.acc);
  ra.acc_ref = nullptr;
  ra.hdr = hdr;
  ra.lws = loss_ws(const_cast<void*>(loss_workspace), LL);
  if (launch_reward_sampled_stats(ra, rprob->dtype == AAL_BF16, s) != cudaSuccess) return AAL_ERR_CUDA;

  RewardGroupArgs ga;
  ga.acc = ra.acc;
  ga.acc_ref = nullptr;
  ga.rbuf = reinterpret_cast<float*>(base + L.rbuf);
  ga.N = rprob->N;
  ga.K = (int32_t)rprob->K;
  ga.wpr = rprob->windows_per_rollout;
  ga.rpg = rprob->rollouts_per_group;
  ga.adv_clip = rprob->adv_clip;
  ga.tau = tau;
  ga.tau_ref = nullptr;
  ga.rollout_len = rollout_len;
  ga.advantage = advantage;
  return cuda_status(launch_reward_groups(ga, s));
}

aal_status aal_check_device_status(void* workspace, void* stream) {
  if (workspace == nullptr || !aligned(workspace, 256)) return AAL_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return AAL_ERR_CUDA;
  uint32_t word = 0;
  WsHeader* hdr = static_cast<WsHeader*>(workspace);  // the header is at offset 0 of both layouts
  if (cudaMemcpy(&word, &hdr->status, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess) return AAL_ERR_CUDA;
  if (word == 0) return AAL_OK;
  if (cudaMemset(&hdr->status, 0, sizeof(word)) != cudaSuccess) return AAL_ERR_CUDA;
  if (word == kStatusTimeout) return AAL_ERR_TIMEOUT;
  if (word == (uint32_t)AAL_ERR_INVALID_ARG) return AAL_ERR_INVALID_ARG;  // a token id outside [0, V)
  return AAL_ERR_CUDA;
}

}  // extern "C"
