// Internal declarations of libaal: device helpers, workspace layout, launchers.
//
// Everything here is private to the library; the public surface is include/aal.h.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/aal.h"

namespace aal {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kMaxCluster = 8;          // CTAs that may share one logit row
constexpr int kMaxGroups = 1024;        // fused forward + backward: groups of K CTAs per launch
constexpr uint64_t kMboxEmpty = ~0ull;  // a mailbox word not yet written (no arithmetic result has these bits)
constexpr uint32_t kStatusTimeout = 5;  // == AAL_ERR_TIMEOUT

// ---------------------------------------------------------------------------
// Workspace layout.  Offsets are in bytes from the (256-byte aligned) base and
// are pure functions of the problem, so forward and backward agree on them.
// ---------------------------------------------------------------------------
struct WsHeader {
  uint32_t status;        // device error word (0 = ok), set by bounded waits
  uint32_t done_blocks;   // "last block finishes" counter of the window kernel
  int32_t nvalid;         // |W|, written by the forward
  int32_t cluster;        // CTAs per row used by the row-statistics kernel
  float loss;             // copy of the loss
  int32_t npos;           // valid positions (rows), the normaliser of the KL anchor
  float pad[58];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");

struct LossLayout {
  int64_t R = 0, N = 0, nwblk = 0;
  size_t hdr = 0;
  // float[R] each: the normaliser of z_p/T, z_q/T and z_q in two parts: the raw logit
  // maximum M = max_v z_v and Ls = log2 sum_v 2^((z_v - M) s) with s = log2(e)/T, so that
  // log2 p~_v = (z_v - M) s - Ls; the maximum's own term is exactly 2^0 = 1.
  size_t Mp = 0, Lsp = 0, Mq = 0, Lsq = 0, Mq1 = 0, Lsq1 = 0;
  size_t Mp1 = 0, Lsp1 = 0;         // float[R] the normaliser of z_p at T = 1 (KL anchor)
  size_t kl = 0;                    // float[R] KL(p || q) at T = 1 (KL anchor)
  size_t cgr = 0;                   // float[R] GRPO coefficient of (delta_{u,y} - q(u)), w_grpo included
  size_t ag = 0, as = 0, qlt = 0;   // float[R] a^greedy, a^sample, sum_{lq<lp} q~
  size_t dEg = 0, dEs = 0;          // float[R] dE^g/da (unweighted); w_s dE^s/da + w_tv / K_n
  size_t xstar = 0;                 // int32[R] target argmax
  size_t yhat = 0;                  // int32[R] draft argmax (the greedy draft token)
  size_t zpy = 0;                   // float[R] z_p at the draft argmax
  size_t cpart = 0;                 // float2[R][kMaxCluster] per-CTA (overlap, Qlt) partials
  size_t wpart = 0;                 // double[nwblk][kWpart] window-kernel block partials
  size_t mbox = 0;                  // uint64[R] fused forward + backward: (a^greedy, a^sample) per row
  size_t total = 0;
};

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

constexpr int kWindowThreads = 256;
constexpr int kWpart = 8;  // block partials: sum E^g, sum E^s, |W|, sum KL, |positions|

inline LossLayout loss_layout(int64_t N, int64_t K) {
  LossLayout L;
  L.N = N;
  L.R = N * K;
  L.nwblk = (N + kWindowThreads - 1) / kWindowThreads;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t R = (size_t)L.R;
  L.hdr = take(sizeof(WsHeader));
  L.Mp = take(R * 4);
  L.Lsp = take(R * 4);
  L.Mq = take(R * 4);
  L.Lsq = take(R * 4);
  L.Mq1 = take(R * 4);
  L.Lsq1 = take(R * 4);
  L.Mp1 = take(R * 4);
  L.Lsp1 = take(R * 4);
  L.kl = take(R * 4);
  L.cgr = take(R * 4);
  L.ag = take(R * 4);
  L.as = take(R * 4);
  L.qlt = take(R * 4);
  L.dEg = take(R * 4);
  L.dEs = take(R * 4);
  L.xstar = take(R * 4);
  L.yhat = take(R * 4);
  L.zpy = take(R * 4);
  L.cpart = take(R * kMaxCluster * 8);
  L.wpart = take((size_t)(L.nwblk > 0 ? L.nwblk : 1) * kWpart * 8);
  L.mbox = take(R * 8);
  L.total = off;
  return L;
}

// Sequence layout: rows are positions (R = N = B*T, one window per start position) plus the
// per-window, per-depth partials dE_t/da_{t+j}, which a gather sums into each position's dE/da.
struct SeqLayout {
  LossLayout base;
  size_t pg = 0, ps = 0;  // float[B*T][K] each (greedy, sampling)
  size_t total = 0;
};

inline SeqLayout seq_layout(int64_t B, int64_t T, int64_t K) {
  SeqLayout L;
  L.base = loss_layout(B * T, 1);
  size_t off = L.base.total;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t nk = (size_t)(B * T * K);
  L.pg = take(nk * 4);
  L.ps = take(nk * 4);
  L.total = off;
  return L;
}

struct RewardLayout {
  int64_t R = 0;
  size_t hdr = 0, acc = 0, acc_ref = 0, rbuf = 0, total = 0;
};

inline RewardLayout reward_layout(int64_t N, int64_t K) {
  RewardLayout L;
  L.R = N * K;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  L.hdr = take(sizeof(WsHeader));
  L.acc = take((size_t)L.R);
  L.acc_ref = take((size_t)L.R);
  L.rbuf = take((size_t)N * 4);
  L.total = off;
  return L;
}

// Pointers into a loss workspace.
struct LossWs {
  WsHeader* hdr;
  float *Mp, *Lsp, *Mq, *Lsq, *Mq1, *Lsq1, *Mp1, *Lsp1, *kl, *cgr, *ag, *as, *qlt, *dEg, *dEs;
  int32_t* xstar;
  int32_t* yhat;
  float* zpy;
  float2* cpart;
  double* wpart;
  uint64_t* mbox;
};

inline LossWs loss_ws(void* base, const LossLayout& L) {
  char* b = static_cast<char*>(base);
  LossWs w;
  w.hdr = reinterpret_cast<WsHeader*>(b + L.hdr);
  w.Mp = reinterpret_cast<float*>(b + L.Mp);
  w.Lsp = reinterpret_cast<float*>(b + L.Lsp);
  w.Mq = reinterpret_cast<float*>(b + L.Mq);
  w.Lsq = reinterpret_cast<float*>(b + L.Lsq);
  w.Mq1 = reinterpret_cast<float*>(b + L.Mq1);
  w.Lsq1 = reinterpret_cast<float*>(b + L.Lsq1);
  w.Mp1 = reinterpret_cast<float*>(b + L.Mp1);
  w.Lsp1 = reinterpret_cast<float*>(b + L.Lsp1);
  w.kl = reinterpret_cast<float*>(b + L.kl);
  w.cgr = reinterpret_cast<float*>(b + L.cgr);
  w.ag = reinterpret_cast<float*>(b + L.ag);
  w.as = reinterpret_cast<float*>(b + L.as);
  w.qlt = reinterpret_cast<float*>(b + L.qlt);
  w.dEg = reinterpret_cast<float*>(b + L.dEg);
  w.dEs = reinterpret_cast<float*>(b + L.dEs);
  w.xstar = reinterpret_cast<int32_t*>(b + L.xstar);
  w.yhat = reinterpret_cast<int32_t*>(b + L.yhat);
  w.zpy = reinterpret_cast<float*>(b + L.zpy);
  w.cpart = reinterpret_cast<float2*>(b + L.cpart);
  w.wpart = reinterpret_cast<double*>(b + L.wpart);
  w.mbox = reinterpret_cast<uint64_t*>(b + L.mbox);
  return w;
}

// ---------------------------------------------------------------------------
// Launch descriptions (host side fills, kernels read by value).
// ---------------------------------------------------------------------------
struct RowStatsArgs {
  const void* zq;       // draft logits  [R][V]
  const void* zp;       // target logits [R][V]
  int64_t R, V;
  float sT;             // log2(e) / T  (scale of the temperature softmaxes)
  bool need_p;          // log-sum-exp of z_p / T   (sampling term)
  bool need_q;          // log-sum-exp of z_q / T   (sampling term)
  bool need_q1;         // log-sum-exp of z_q       (greedy term, when T != 1 or no sampling)
  bool overlap;         // second phase: sum min(p~, q~) and Qlt (sampling term)
  bool need_kl;         // KL(p || q) at T = 1 and the normaliser of z_p at T = 1 (anchor)
  int64_t skip_chunk;   // failure-detection test hook: a chunk whose copy is never armed (-1: none)
  LossWs ws;
  // the streamed sampling reward (launch_reward_stream): per-row acceptance flags, the Philox key
  // and the global window index of row 0's window; ws.hdr is the reward workspace's status word
  uint8_t* acc = nullptr;
  uint64_t seed = 0;
  int64_t row_offset = 0;
  int32_t K = 1;
};

struct WindowArgs {
  const uint8_t* mask;  // [N][K] or null
  int64_t N;
  int32_t K;
  int32_t cluster;      // partials per row in ws.cpart
  bool greedy, sampling, kl, tv;
  float w_greedy, w_sampling, w_kl, w_tv;
  float* loss;          // device float[1]
  float* eal;           // device float[N][2] or null
  LossWs ws;
  int64_t nwblk;
  int32_t nvalid_g, npos_g;  // data-parallel |W| and |P| of the whole batch, or -1: this call's
};

struct SeqWindowArgs {
  const uint8_t* mask;  // [B][T] or null
  int64_t B, T;
  int32_t K;
  int32_t cluster;
  bool greedy, sampling, kl, tv;
  bool full_windows;    // W = windows with all K positions valid
  float w_greedy, w_sampling, w_kl, w_tv;
  float* loss;
  float* eal;           // [B*T][2] or null
  float* pg;            // [B*T][K]
  float* ps;
  LossWs ws;
  int64_t nwblk;
  int32_t nvalid_g, npos_g;  // data-parallel |W| and |P| of the whole batch, or -1: this call's
};

struct BackwardArgs {
  const void* zq;
  const void* zp;
  void* grad;
  int64_t R, V;
  int32_t K;
  float sT, invT;
  float dloss;
  float w_greedy, w_sampling;  // 0 for a term the mode does not select
  float w_kl;                  // 0 without the KL anchor
  bool grpo;                   // add dloss * cgr[r] (delta_{u,y_r} - q(u)) (the GRPO surrogate)
  const uint8_t* mask;         // [R] position validity (the anchor's rows), or null
  bool q1_is_qT;               // T == 1, sampling and a T = 1 term: q = q~, one exponential
  LossWs ws;
};

// The fused forward + backward of [N][K][V] windows (aal_loss_fwd_bwd): groups of K CTAs,
// CTA k of group g taking depth k of windows g, g + G, ...
struct FusedArgs {
  RowStatsArgs st;   // the statistics passes (zq, zp, R, V, sT, flags, test hook, workspace)
  BackwardArgs bw;   // the gradient pass (grad, dloss, weights, position mask, invT)
  WindowArgs win;    // the window terms (mask [N][K], N, K, which terms, w_sampling, w_tv)
  int32_t groups;    // G
  int32_t solos;     // S solo CTAs after the groups' G K, each taking whole windows
  int64_t n_group;   // windows 0 .. n_group - 1 go to the groups, the rest to the solo CTAs
  // the sequence layout (seq_T > 0): rows are the positions b*T + t of st.R = B*T, a window
  // starts at every position; win.N and win.mask are unused there, seq_mask is the [B][T] mask
  int64_t seq_T = 0;
  int32_t seq_full = 0;  // W = windows with all K positions valid
  const uint8_t* seq_mask = nullptr;
};

struct RewardRowArgs {
  const void* zq;    // draft
  const void* zp;    // target
  const void* zr;    // reference draft or null
  int64_t R, V;
  int32_t K;
  bool sampling;
  bool sampled_draft;  // the drafted token is drawn from q~ (Gumbel-max) instead of argmax z_q
  float sT;
  uint64_t seed;
  int64_t row_offset;
  uint8_t* acc;
  uint8_t* acc_ref;
  WsHeader* hdr;
  LossWs lws;        // the sampled draft from a loss forward: its normalisers of z_p/T and z_q/T
};

// Acceptance flags from the statistics a loss forward left in its workspace.
struct RewardStatsArgs {
  LossWs ws;
  int64_t R;
  int32_t K;
  bool sampling;
  float sT;
  uint64_t seed;
  int64_t row_offset;
  uint8_t* acc;
};

struct RewardGroupArgs {
  const uint8_t* acc;
  const uint8_t* acc_ref;  // null without a reference draft
  float* rbuf;             // [N] debiased rewards
  int64_t N;
  int32_t K;
  int64_t wpr, rpg;
  float adv_clip;
  int32_t* tau;
  int32_t* tau_ref;
  float* rollout_len;
  float* advantage;
};

// GRPO workspace (aal_grpo_from_loss): reward flags and buffers, log pi_ref at the draft's
// greedy tokens, and block partials of the surrogate sum.
struct GrpoLayout {
  int64_t R = 0, N = 0, nroll = 0, nblk = 0;
  size_t hdr = 0, acc = 0, acc_ref = 0, rbuf = 0, tau = 0, tau_ref = 0, rl = 0, adv = 0, lpr = 0, part = 0;
  size_t total = 0;
};

constexpr int kGrpoThreads = 256;

inline GrpoLayout grpo_layout(int64_t N, int64_t K, int64_t wpr) {
  GrpoLayout L;
  L.N = N;
  L.R = N * K;
  L.nroll = wpr > 0 ? N / wpr : 0;
  L.nblk = (N + kGrpoThreads - 1) / kGrpoThreads;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  L.hdr = take(sizeof(WsHeader));
  L.acc = take((size_t)L.R);
  L.acc_ref = take((size_t)L.R);
  L.rbuf = take((size_t)N * 4);
  L.tau = take((size_t)N * 4);
  L.tau_ref = take((size_t)N * 4);
  L.rl = take((size_t)L.nroll * 4);
  L.adv = take((size_t)L.nroll * 4);
  L.lpr = take((size_t)L.R * 4);
  L.part = take((size_t)(L.nblk > 0 ? L.nblk : 1) * 8);
  L.total = off;
  return L;
}

// One pass over the rows of a single tensor (onetensor.cu).  REF: the GRPO reference-draft
// pass, log pi_ref at the draft's greedy token y (from the loss workspace) and both
// acceptance flags.  IDS: the loss forward with x* given as token ids (only the draft read).
struct Stream1Args {
  const void* z;       // [R][V] logits: the reference draft (REF) or the draft (IDS)
  int64_t R, V;
  LossWs lws;          // REF: x*, y of the loss forward; IDS: the statistics written
  const int32_t* ids;  // IDS: [R] target token ids
  uint8_t* acc;        // REF: [R] y == x*
  uint8_t* acc_ref;    // REF: [R] argmax z_ref == x*
  float* lpr;          // REF: [R] log pi_ref(y)
  WsHeader* hdr;       // status word (bounded waits; out-of-range ids)
  int64_t skip_chunk;  // failure-detection test hook: a chunk whose copy is never armed (-1: none)
};

// The fused forward + backward with x* as token ids (aal_loss_fwd_bwd, mode AAL_GREEDY |
// AAL_IDS): only the draft is streamed; groups of K CTAs as in FusedArgs.
struct FusedIdsArgs {
  Stream1Args st;    // the draft's statistics pass (z = draft, ids, workspace, test hook)
  BackwardArgs bw;   // the gradient pass
  WindowArgs win;    // the window terms
  int32_t groups;    // G
  int32_t solos;     // S solo CTAs after the groups' G K, each taking whole windows
  int64_t n_group;   // windows 0 .. n_group - 1 go to the groups, the rest to the solo CTAs
  // the sequence layout (seq_T > 0): rows are the positions b*T + t of st.R = B*T, a window
  // starts at every position; win.N and win.mask are unused there, seq_mask is the [B][T] mask
  int64_t seq_T = 0;
  int32_t seq_full = 0;  // W = windows with all K positions valid
  const uint8_t* seq_mask = nullptr;
};

// Windows per solo CTA for the fused kernels: G groups finish a window each in one row's time,
// each of S solo CTAs one in K row times, so with m windows per solo CTA the launch ends after
// max(ceil((N - m S) / G), m K) row times.  The best m near the balance point N / (G K + S),
// or 0 (no solo CTAs) when none shortens the launch.
inline int64_t solo_windows_each(int64_t N, int64_t K, int64_t G, int64_t S) {
  if (S <= 0 || G <= 0) return 0;
  auto cost = [&](int64_t m) {
    const int64_t a = (N - m * S + G - 1) / G, b = m * K;
    return a > b ? a : b;
  };
  int64_t best = 0;
  const int64_t m0 = N / (G * K + S);
  for (int64_t m = m0; m <= m0 + 1; ++m)
    if (m > 0 && m * S <= N && cost(m) < cost(best)) best = m;
  return best;
}

// GRPO over sequences (aal_seq_grpo_from_loss): per-position flags and log pi_ref from the
// reference pass, the windows' rows gathered from them, and the windows' coefficients before
// they are added per position.
struct SeqGrpoLayout {
  GrpoLayout g;        // per-window buffers (acc, acc_ref, rewards, advantages, partials)
  int64_t RP = 0;      // positions B*T
  size_t acc_pos = 0, accr_pos = 0, lpr_pos = 0, cw = 0;
  size_t total = 0;
};

inline SeqGrpoLayout seq_grpo_layout(int64_t N, int64_t K, int64_t wpr, int64_t positions) {
  SeqGrpoLayout L;
  L.g = grpo_layout(N, K, wpr);
  L.RP = positions;
  size_t off = L.g.total;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  L.acc_pos = take((size_t)positions);
  L.accr_pos = take((size_t)positions);
  L.lpr_pos = take((size_t)positions * 4);
  L.cw = take((size_t)(N * K) * 4);
  L.total = off;
  return L;
}

struct SeqGrpoArgs {
  const int32_t* starts;  // [N] flat start position of each window (ascending)
  int64_t N, T, RP;
  int32_t K;
  const uint8_t* acc_pos;
  const uint8_t* accr_pos;
  uint8_t* acc;           // [N][K] gathered
  uint8_t* acc_ref;
  const float* cw;        // [N][K] coefficients of the window rows
  float* cgr;             // [RP] per position (loss workspace)
  WsHeader* hdr;          // status word: AAL_ERR_INVALID_ARG for a bad start
};

// Per window: log rho, the clipped surrogate, its per-row gradient coefficients.
struct GrpoWindowArgs {
  LossWs lws;          // Lsq1 (log pi_theta(y) = -ln2 Lsq1), cgr out
  const float* lpr;
  const int32_t* starts;  // null: window rows are n*K + k; else positions starts[n] + k
  int64_t RP;             // with starts: the number of positions
  float* cw;              // with starts: the window rows' coefficients ([N][K]), not lws.cgr
  const float* adv;    // [N / wpr]
  int64_t N;
  int32_t K;
  int64_t wpr;
  float eps_clip, rho_min, rho_max, log_rho_clip, w_grpo;
  float* log_rho;      // [N] or null
  double* part;        // [nblk]
  int64_t nblk;
  WsHeader* hdr;       // of the GRPO workspace (last-block counter)
  float* loss;         // [1] L_GRPO
};

// Launchers (return cudaGetLastError() of their launches).
cudaError_t launch_rowstats(const RowStatsArgs& a, bool bf16, cudaStream_t s, int* cluster_used);
cudaError_t launch_rowstats_stream(const RowStatsArgs& a, bool bf16, cudaStream_t s, uint64_t limit_ns);
// The same kernels for short rows (rowstats_short.cu): 8 consumer warps, two CTAs an SM.
cudaError_t launch_rowstats_stream_short(const RowStatsArgs& a, bool bf16, cudaStream_t s, uint64_t limit_ns);
cudaError_t launch_reward_stream_short(const RowStatsArgs& a, cudaStream_t s, uint64_t limit_ns);
// Rows shorter than this many bytes take the short-row geometry and the two calls inside
// aal_loss_fwd_bwd / aal_seq_loss_fwd_bwd (128 KB unless the test hook changed it).
int64_t fused_min_row_bytes();
// The sampling reward's acceptance flags from one streamed pass over bf16 rows of 16-byte
// multiples (a.sT = log2(e) / T, a.acc, a.seed, a.row_offset, a.K).
cudaError_t launch_reward_stream(const RowStatsArgs& a, cudaStream_t s, uint64_t limit_ns);
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // bounded waits give up after 1 s

// Failure-detection test hooks (include/aal_debug.h); both are 0 / -1 in normal use.
uint64_t debug_wait_limit_ns();
int64_t debug_take_skip_chunk();
cudaError_t launch_window(const WindowArgs& a, cudaStream_t s);
cudaError_t launch_seq_window(const SeqWindowArgs& a, cudaStream_t s);
cudaError_t launch_backward(const BackwardArgs& a, bool bf16, cudaStream_t s);
cudaError_t launch_reward_rows(const RewardRowArgs& a, bool bf16, cudaStream_t s);
cudaError_t launch_reward_groups(const RewardGroupArgs& a, cudaStream_t s);
cudaError_t launch_reward_flags_from_stats(const RewardStatsArgs& a, cudaStream_t s);
// The sampled-draft reward with the loss forward's normalisers (RewardRowArgs.lws): the draft alone
// streamed for the draws, the target read at each drawn token; 16-byte rows.
cudaError_t launch_reward_sampled_stats(const RewardRowArgs& a, bool bf16, cudaStream_t s);
cudaError_t launch_one_tensor(const Stream1Args& a, bool bf16, bool ids, cudaStream_t s);
cudaError_t launch_grpo_windows(const GrpoWindowArgs& a, cudaStream_t s);
cudaError_t launch_seq_grpo_gather(const SeqGrpoArgs& a, cudaStream_t s);
cudaError_t launch_seq_grpo_scatter(const SeqGrpoArgs& a, cudaStream_t s);
cudaError_t launch_count_valid(const uint8_t* mask, int64_t N, int32_t K, int32_t nvalid_g, int32_t npos_g,
                               WsHeader* hdr, cudaStream_t s);
// Launches the fused forward + backward when the problem's flags have an instantiation and the
// device can hold at least one group; *launched tells whether it did.
cudaError_t launch_fused(const FusedArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched);
// The same for token ids (then resolve_draft_argmax places the draft's greedy token).
cudaError_t launch_fused_ids(const FusedIdsArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched);
// The sequence layout's |W| and |positions| from the [B][T] mask, as the sequence window kernel
// counts them.
cudaError_t launch_seq_count_valid(const uint8_t* mask, int64_t B, int64_t T, int32_t K, bool full,
                                   int32_t nvalid_g, int32_t npos_g, WsHeader* hdr, cudaStream_t s);
// The fused forward + backward over the sequence layout (FusedArgs.seq_T > 0), and with token ids.
cudaError_t launch_fused_seq(const FusedArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched);
cudaError_t launch_fused_ids_seq(const FusedIdsArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched);

// ---------------------------------------------------------------------------
// Device helpers.
// ---------------------------------------------------------------------------
#ifdef __CUDACC__

// 2^x on the MUFU unit; denormal results flush to zero.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// log2(x) on the MUFU unit; denormal inputs flush to zero (callers pass normal values only).
__device__ __forceinline__ float lg2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Expected length of one window term and its partials (Sec. 3.1, Eq. eal_generic): with
// P_k = prod_{j<k} a_j, E = sum_{k=1}^{kn} P_k and dE/da_j = P_j S_j, S_{kn-1} = 1,
// S_j = 1 + a_{j+1} S_{j+1} (0 for j >= kn).  Shared by the window kernels and the fused
// forward + backward, so both give bitwise the same partials.
__device__ __forceinline__ float window_term(const float* a, int kn, float* dE) {
  // every rounding spelled out (no contraction), so that every kernel forms the same bits
  float P[AAL_MAX_K + 1];
  P[0] = 1.f;
  float E = 0.f;
#pragma unroll
  for (int j = 0; j < AAL_MAX_K; ++j) {
    if (j < kn) {
      P[j + 1] = __fmul_rn(P[j], a[j]);
      E = __fadd_rn(E, P[j + 1]);
    }
  }
  float S = 1.f;
#pragma unroll
  for (int j = AAL_MAX_K - 1; j >= 0; --j) {
    if (j < kn) {
      dE[j] = __fmul_rn(P[j], S);
      S = __fmaf_rn(a[j], S, 1.f);
    } else {
      dE[j] = 0.f;
    }
  }
  return E;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

template <typename T>
__device__ __forceinline__ float load_elem(const T* p);
template <>
__device__ __forceinline__ float load_elem<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float load_elem<uint16_t>(const uint16_t* p) {
  return __uint_as_float(((uint32_t)__ldg(p)) << 16);
}

// Streaming 16-byte load that should not linger in L1 (read once per pass).
__device__ __forceinline__ uint4 ldg_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Online log2-sum-exp state of the values z*s: M = running raw maximum of z and
// S = sum_v 2^((z_v - M) s).  The maximum's own term is exactly 1.
struct Lse {
  float M, S;
};
__device__ __forceinline__ void lse_init(Lse& a) {
  a.M = -INFINITY;
  a.S = 0.f;
}
__device__ __forceinline__ void lse_push(Lse& a, float z, float s) {
  if (z > a.M) {
    a.S = a.S * ex2((a.M - z) * s) + 1.f;  // M == -inf: ex2(-inf) = 0 and S was 0
    a.M = z;
  } else if (a.M != -INFINITY) {
    a.S += ex2((z - a.M) * s);
  }
}
__device__ __forceinline__ Lse lse_merge(Lse a, Lse b, float s) {
  Lse r;
  r.M = fmaxf(a.M, b.M);
  if (r.M == -INFINITY) {
    r.S = 0.f;
  } else {
    const float sa = (a.M == -INFINITY) ? 0.f : a.S * ex2((a.M - r.M) * s);
    const float sb = (b.M == -INFINITY) ? 0.f : b.S * ex2((b.M - r.M) * s);
    r.S = sa + sb;
  }
  return r;
}
// Ls = log2(S), accurate log (once per row).
__device__ __forceinline__ float lse_ls(Lse a) { return log2f(a.S); }
// log2 of the scaled probability of logit z: (z - M) s - Ls.
__device__ __forceinline__ float log2_prob(float z, float s, float M, float Ls) { return fmaf(z - M, s, -Ls); }

// f32(bf16 half of w) + c in one instruction (the widening happens inside the add).
__device__ __forceinline__ float bf16lo_add(uint32_t w, float c) {
  float d;
  asm("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tadd.rn.f32.bf16 %0, lo, %2;\n\t}"
      : "=f"(d)
      : "r"(w), "f"(c));
  return d;
}
__device__ __forceinline__ float bf16hi_add(uint32_t w, float c) {
  float d;
  asm("{\n\t.reg .b16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tadd.rn.f32.bf16 %0, hi, %2;\n\t}"
      : "=f"(d)
      : "r"(w), "f"(c));
  return d;
}

// Online forward KL of one row at T = 1 (the anchor): with e_v = exp(z_p,v - M) and M the
// running maximum of z_p, S = sum e_v and D = sum e_v (z_p,v - z_q,v), both rescaled when M
// moves.  Then p_v = e_v / S and KL(p || q) = D / S - (M - M_q) - ln S + ln S_q.  A target
// logit of -inf adds nothing (0 log 0 = 0).
struct KlAcc {
  float M, S, D;
};
__device__ __forceinline__ void kl_init(KlAcc& a) {
  a.M = -INFINITY;
  a.S = 0.f;
  a.D = 0.f;
}
__device__ __forceinline__ void kl_push(KlAcc& a, float p, float q) {
  if (p > a.M) {
    const float r = ex2((a.M - p) * kLog2e);  // M == -inf: r = 0, and S, D were 0
    a.S = fmaf(a.S, r, 1.f);
    a.D = fmaf(a.D, r, p - q);
    a.M = p;
  } else if (p != -INFINITY) {
    const float e = ex2((p - a.M) * kLog2e);
    a.S += e;
    a.D = fmaf(e, p - q, a.D);
  }
}
__device__ __forceinline__ KlAcc kl_merge(KlAcc a, KlAcc b) {
  KlAcc r;
  r.M = fmaxf(a.M, b.M);
  if (r.M == -INFINITY) {
    r.S = 0.f;
    r.D = 0.f;
    return r;
  }
  const float sa = (a.M == -INFINITY) ? 0.f : ex2((a.M - r.M) * kLog2e);
  const float sb = (b.M == -INFINITY) ? 0.f : ex2((b.M - r.M) * kLog2e);
  r.S = a.S * sa + b.S * sb;
  r.D = a.D * sa + b.D * sb;
  return r;
}

// Argmax with the lowest index on ties, carrying one extra value.
struct Amax {
  float v;
  int32_t i;
  float carry;
};
__device__ __forceinline__ void amax_init(Amax& a) {
  a.v = -INFINITY;
  a.i = 0x7fffffff;
  a.carry = 0.f;
}
__device__ __forceinline__ Amax amax_merge(Amax a, Amax b) {
  return (b.v > a.v || (b.v == a.v && b.i < a.i)) ? b : a;
}

__device__ __forceinline__ Lse shfl_lse(Lse a, int off) {
  Lse b;
  b.M = __shfl_xor_sync(0xffffffffu, a.M, off);
  b.S = __shfl_xor_sync(0xffffffffu, a.S, off);
  return b;
}
__device__ __forceinline__ Amax shfl_amax(Amax a, int off) {
  Amax b;
  b.v = __shfl_xor_sync(0xffffffffu, a.v, off);
  b.i = __shfl_xor_sync(0xffffffffu, a.i, off);
  b.carry = __shfl_xor_sync(0xffffffffu, a.carry, off);
  return b;
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32->64
// multiplies with a Weyl-sequence key schedule.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// The sampling reward's uniform for (seed; window n; depth k): odd multiple of 2^-24 in (0,1).
__device__ __forceinline__ float philox_uniform(uint64_t seed, uint64_t n, uint32_t k) {
  uint4 c = make_uint4((uint32_t)n, (uint32_t)(n >> 32), k, 0u);
  uint4 x = philox4x32_10(c, (uint32_t)seed, (uint32_t)(seed >> 32));
  return (float)((x.x >> 9) * 2u + 1u) * 5.9604644775390625e-08f;  // * 2^-24
}

// The four uniforms of counter (n_lo, n_hi, k, c3), mapped like philox_uniform: the Gumbel-max
// draw of the sampled-draft reward gives vocabulary element v word v mod 4 of c3 = 1 + v div 4.
__device__ __forceinline__ float4 philox_uniform4(uint64_t seed, uint64_t n, uint32_t k, uint32_t c3) {
  uint4 x = philox4x32_10(make_uint4((uint32_t)n, (uint32_t)(n >> 32), k, c3), (uint32_t)seed,
                          (uint32_t)(seed >> 32));
  constexpr float s = 5.9604644775390625e-08f;  // 2^-24
  return make_float4((float)((x.x >> 9) * 2u + 1u) * s, (float)((x.y >> 9) * 2u + 1u) * s,
                     (float)((x.z >> 9) * 2u + 1u) * s, (float)((x.w >> 9) * 2u + 1u) * s);
}

// Bounded wait support: every spin in this library gives up after this many polls.
constexpr uint32_t kSpinLimit = 1u << 26;

#endif  // __CUDACC__

}  // namespace aal
