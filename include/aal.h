/*
 * aal.h -- acceptance-aware draft-training losses on one GB300 (sm_103a).
 *
 * C ABI of libaal.so.  It computes, over full-vocabulary draft and target logits:
 *   - the expected-accepted-length loss under greedy verification (EAL) and the
 *     window total-variation loss under sampling verification (WTV), forward and
 *     backward with respect to the draft logits;
 *   - the simulated acceptance length, debiased reward and group-normalised
 *     advantage of the GRPO stage.
 * Paper: "Acceptance-Aware Draft Model Training for Speculative Decoding",
 * Sec. 2.3 (acceptance under greedy / sampling verification, Eqs. acc_greedy,
 * acc_sample), Sec. 3.1 (speculative window, Eq. eal_generic), Sec. 3.2 (Eq.
 * loss_eal), Sec. 3.3 (Eqs. rejection_rate, eal_tv, loss_tv), Sec. 3.4 (GRPO
 * reward, Eqs. debiased_reward, advantage).
 *
 * Common conventions
 *   Layout.  Logits are row-major [N windows][K depths][V vocabulary], rows
 *     contiguous, element type fp32 or bf16; depth k of window n is position
 *     t + k of the window that starts at t.  Base pointers must be 16-byte
 *     aligned (any V is accepted; rows whose byte length is not a multiple of
 *     16 take a slower path).
 *   Memory.  Every pointer is a DEVICE pointer owned by the caller, except the
 *     aal_problem / aal_reward_problem structs, which are host memory read
 *     during the call only.  The library allocates nothing and keeps no state
 *     between calls; the workspace carries the forward's results to the
 *     backward.
 *   Streams.  `stream` is a cudaStream_t (NULL = legacy default stream).  All
 *     calls are asynchronous on it; outputs are valid once the stream reaches
 *     the call.  Calls that share a workspace must be ordered on one stream.
 *     aal_loss_fwd, aal_loss_bwd, aal_loss_fwd_bwd, aal_seq_loss_fwd_bwd (cooperative
 *     launches among them) and aal_accept_reward_from_loss enqueue only kernels and
 *     asynchronous memsets on `stream`, so a step made of them can be captured in a CUDA
 *     graph and replayed; each replay gives the same bits as eager calls.
 *   Errors.  Arguments are checked before anything is launched; a failed check
 *     returns AAL_ERR_INVALID_ARG / AAL_ERR_UNSUPPORTED / AAL_ERR_WORKSPACE and
 *     launches nothing.  A launch failure returns AAL_ERR_CUDA.  Device-side
 *     errors (a bounded wait that ran out) are recorded in the workspace and
 *     reported by aal_check_device_status().  No call aborts the process.
 *   Gradients.  The target is frozen (Sec. 3.2, 3.3); only the draft gets a
 *     gradient.
 */
#ifndef AAL_H_
#define AAL_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define AAL_API __attribute__((visibility("default")))
#else
#define AAL_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  AAL_OK = 0,
  AAL_ERR_INVALID_ARG = 1,  /* a NULL, misaligned or out-of-range argument */
  AAL_ERR_UNSUPPORTED = 2,  /* valid request this build does not handle (e.g. K > 8) */
  AAL_ERR_WORKSPACE = 3,    /* workspace missing or smaller than aal_*_workspace_size() */
  AAL_ERR_CUDA = 4,         /* a CUDA runtime call or kernel launch failed */
  AAL_ERR_TIMEOUT = 5       /* a device-side bounded wait ran out (see aal_check_device_status) */
} aal_status;

typedef enum { AAL_F32 = 0, AAL_BF16 = 1 } aal_dtype;

/* Which loss terms to compute (bits).  GREEDY: L_EAL (Eq. loss_eal); SAMPLING: L_WTV
 * (Eq. loss_tv); BOTH: w_greedy * L_EAL + w_sampling * L_WTV.  KL adds w_kl * L_KL, the
 * forward-KL anchor of the combined objectives (Sec. 4.1): the mean over valid positions of
 * KL(p || q) = sum_v p(v) (log p(v) - log q(v)) at T = 1.  The greedy-regime objective of
 * Sec. 4.1, L_KL + 0.1 L_EAL, is mode AAL_KL | AAL_GREEDY with w_kl = 1, w_greedy = 0.1;
 * mode AAL_KL alone is the L_KL baseline.  AAL_GRPO makes aal_loss_bwd add the gradient of
 * the GRPO surrogate (Sec. 3.4) whose per-row coefficients aal_grpo_from_loss writes into the
 * loss workspace between the forward and the backward; aal_loss_fwd clears them, so without
 * that call the term is zero, and the loss aal_loss_fwd reports never includes it (see
 * aal_grpo_from_loss).  AAL_TV adds w_tv * L_TV, the auxiliary term of the L_KL + L_TV baseline
 * (Sec. 4.1): each window's TV(p~, q~) = 1 - a^sample averaged over its K_n valid positions, then
 * the mean over W; the baseline L_KL + 0.1 L_TV is mode AAL_KL | AAL_TV with w_tv = 0.1 (T as for
 * the sampling term).  AAL_IDS changes what `target` points to: int32 token ids, one per logit row
 * ([N][K] or [B][seq_len]), taken as x* (Sec. 3.2: for greedy target-generated data x* is the
 * ground-truth token) instead of target logits; then only the draft is read (half the forward's
 * bytes, and the greedy backward never reads the target).  It combines with AAL_GREEDY and
 * AAL_GRPO only (the other terms need p).  An id outside [0, V) records AAL_ERR_INVALID_ARG in the
 * workspace status word (aal_check_device_status) and that row's a^greedy is 0.
 * Valid modes: 1 .. 63. */
typedef enum {
  AAL_GREEDY = 1, AAL_SAMPLING = 2, AAL_BOTH = 3, AAL_KL = 4, AAL_GRPO = 8, AAL_TV = 16, AAL_IDS = 32
} aal_mode;

#define AAL_MAX_K 8

/* One loss problem (host struct).
 *   N, K, V      windows, window size gamma (1..AAL_MAX_K), vocabulary size (>= 1); N may be 0.
 *   dtype        aal_dtype of draft, target and the gradient.
 *   mode         aal_mode.
 *   temperature  T of the sampling and TV terms (Sec. 2.3: p~ ~ exp(log p / T)); must be
 *                finite and > 0 when mode includes SAMPLING or TV.  The greedy acceptance
 *                a = q(x*) (Eq. acc_greedy) always uses the unscaled draft, so T is
 *                ignored (and may be 0) for mode GREEDY.
 *   w_greedy, w_sampling, w_kl, w_tv  weights of the terms (a term the mode does not select
 *                is not computed and its weight is ignored).  Must be finite.
 *   global_counts, n_windows_global, n_positions_global   data-parallel normalisers.  With
 *                global_counts = 0 (the default; this field was "reserved, must be 0" before ABI
 *                1.6, and the two fields after it are then not read) the loss divides by this
 *                call's own |W| and |P|.  With global_counts = 1 it divides by n_windows_global
 *                (|W| of the whole data-parallel batch, Sec. 3.2's 1/|W|: the windows whose depth
 *                0 is valid, summed over the ranks) and n_positions_global (|P| of the whole
 *                batch, the KL anchor's normaliser), each in [0, 2^31 - 1].  A batch sharded by
 *                windows over ranks then needs no collective on the data path and no rescaled
 *                dloss: the loss of the whole batch is the sum of the ranks' losses, and each
 *                rank's gradient rows are those of the whole batch's loss, bit for bit.  The
 *                backward uses the forward's normalisers (kept in the workspace). */
typedef struct {
  int64_t N, K, V;
  int32_t dtype;
  int32_t mode;
  float temperature;
  float w_greedy;
  float w_sampling;
  float w_kl;
  float w_tv;
  int32_t global_counts;      /* 0 or 1 */
  int64_t n_windows_global;   /* read only when global_counts = 1 */
  int64_t n_positions_global; /* read only when global_counts = 1 */
} aal_problem;

/* Bytes of device workspace a loss problem needs (host-only, launches nothing). */
AAL_API aal_status aal_workspace_size(const aal_problem* prob, size_t* bytes);

/* Forward of the loss (Sec. 3.2 Eq. loss_eal, Sec. 3.3 Eq. loss_tv, Sec. 4.1):
 *   L = -(1/|W|) sum_n [ w_g sum_{k=1}^{K_n} prod_{j<k} a^g_{n,j}
 *                       + w_s sum_{k=1}^{K_n} prod_{j<k} a^s_{n,j} ]
 *       + w_kl (1/|P|) sum_{valid rows r} KL(p_r || q_r)     (mode bit AAL_KL; |P| = number
 *                                                            of rows with mask 1; 0 if none)
 *       + w_tv (1/|W|) sum_n (1/K_n) sum_{j<K_n} (1 - a^s_{n,j})    (mode bit AAL_TV)
 * with a^g = q(x*) (Eq. acc_greedy, x* = target argmax, lowest index on ties) and
 * a^s = sum_v min(p~, q~) = 1 - TV(p~, q~) (Eqs. acc_sample, rejection_rate).
 *   draft, target  [N][K][V] logits of the draft (z_q) and the target (z_p).
 *   mask           [N][K] uint8, nonzero = valid position, or NULL (all valid).  A
 *                  window stops at its first invalid position (K_n = number of leading
 *                  valid depths) and belongs to W iff K_n >= 1.  |W| = 0 gives L = 0.
 *   workspace      device buffer of at least aal_workspace_size() bytes, 256-byte
 *                  aligned; holds per-row statistics for aal_loss_bwd.
 *   loss           device float[1]: L.
 *   eal            device float[N][2] or NULL: per-window expected accepted lengths
 *                  (greedy, sampling); 0 for a term not computed or a window not in W. */
AAL_API aal_status aal_loss_fwd(const aal_problem* prob, const void* draft, const void* target,
                        const uint8_t* mask, void* workspace, size_t workspace_bytes,
                        float* loss, float* eal, void* stream);

/* Backward of the loss: grad_draft = dloss * dL/dz_q, [N][K][V] in the problem's dtype.
 * Must follow aal_loss_fwd on the same stream with the same problem, inputs, mask
 * and workspace.  dloss is the upstream gradient of L (a host scalar).  Rows of
 * positions outside every window's valid prefix get exact zeros.  The gradient of
 * the sampling term uses the subgradient that follows p~ at ties p~_v = q~_v. */
AAL_API aal_status aal_loss_bwd(const aal_problem* prob, const void* draft, const void* target,
                        const uint8_t* mask, const void* workspace, size_t workspace_bytes,
                        float dloss, void* grad_draft, void* stream);

/* Forward and backward in one call: the loss, eal and workspace of aal_loss_fwd and the
 * gradient of aal_loss_bwd with the same dloss, bit for bit (same arguments, layouts and
 * rules as those two calls; dloss must be known before the forward, as it is for a loss
 * that is a fixed weight times the objective).  The result equals the two calls; the
 * difference is the traffic.  With bf16 rows whose byte length is a multiple of 16, the
 * K rows of each window are streamed by K CTAs together (one cooperative launch, one CTA
 * per SM; the SMs left over take whole windows alone), and the gradient is written while
 * the rows are still in L2: the logits are read
 * from HBM once (2 V b per row, plus V b gradient written) instead of twice (the separate
 * forward's 2 V b and the backward's 3 V b).  With token ids (AAL_GREEDY | AAL_IDS) only the
 * draft is streamed the same way: V b read and V b written per row, instead of V b + 2 V b.
 * Other problems (fp32, unaligned rows) run the two calls inside this one.
 * AAL_GRPO is rejected with AAL_ERR_UNSUPPORTED: its coefficients come from
 * aal_grpo_from_loss, between the forward and the backward.  A bounded device wait that ran
 * out (a ring copy, or the group barrier between the K CTAs of a window) is reported by
 * aal_check_device_status as AAL_ERR_TIMEOUT, and then no output may be used. */
AAL_API aal_status aal_loss_fwd_bwd(const aal_problem* prob, const void* draft, const void* target,
                                    const uint8_t* mask, void* workspace, size_t workspace_bytes,
                                    float dloss, float* loss, float* eal, void* grad_draft, void* stream);

/* Sequence layout (Sec. 3.3): the draft and the target run once over whole sequences, and a
 * window of gamma = K positions starts at every position and slides by one, so each position
 * is depth j of up to K windows.  Logits are stored once per position, not once per window.
 *   B, seq_len, K, V  sequences, positions per sequence (>= 0), window size gamma
 *                     (1..AAL_MAX_K), vocabulary size (>= 1).
 *   dtype, mode, temperature, w_greedy, w_sampling, w_kl, w_tv, global_counts,
 *   n_windows_global, n_positions_global   as in aal_problem (the anchor averages over the
 *                     valid positions; a batch is sharded over ranks by whole sequences, and
 *                     n_windows_global counts the windows in W of all of them).
 *   full_windows      which windows belong to W (the paper leaves the end of a sequence open):
 *                     0 = every start position, its window truncated at the end of the
 *                     sequence or at its first invalid position (as a masked window of
 *                     aal_loss_fwd); 1 = only windows whose K positions are all valid and
 *                     inside the sequence (starts 0 .. seq_len - K of an unmasked sequence). */
typedef struct {
  int64_t B, seq_len, K, V;
  int32_t dtype;
  int32_t mode;
  float temperature;
  float w_greedy;
  float w_sampling;
  float w_kl;
  float w_tv;
  int32_t full_windows;
  int32_t global_counts;      /* 0 or 1, as in aal_problem */
  int64_t n_windows_global;   /* read only when global_counts = 1 */
  int64_t n_positions_global; /* read only when global_counts = 1 */
} aal_seq_problem;

/* Bytes of device workspace a sequence problem needs (host-only, launches nothing). */
AAL_API aal_status aal_seq_workspace_size(const aal_seq_problem* prob, size_t* bytes);

/* Forward of the loss over every sliding window of every sequence:
 *   L = -(1/|W|) sum_{b,t} [ w_g E^g_{b,t} + w_s E^s_{b,t} ],
 * where the window starting at position t of sequence b covers positions t .. t+K-1 and stops
 * at the end of the sequence or at its first invalid position (K_{b,t} = the number of leading
 * valid positions; the window is in W iff K_{b,t} >= 1, i.e. iff position t is valid, or with
 * full_windows iff K_{b,t} = K).  E and the acceptances are those of aal_loss_fwd.
 *   draft, target  [B][seq_len][V] logits (z_q, z_p), rows contiguous, 16-byte aligned bases.
 *   mask           [B][seq_len] uint8, nonzero = valid position, or NULL (all valid).
 *   workspace      at least aal_seq_workspace_size() bytes, 256-byte aligned.
 *   loss           device float[1].
 *   eal            device float[B*seq_len][2] or NULL: E^g, E^s of the window starting at each
 *                  position (0 for a term not computed or a window not in W). */
AAL_API aal_status aal_seq_loss_fwd(const aal_seq_problem* prob, const void* draft, const void* target,
                                    const uint8_t* mask, void* workspace, size_t workspace_bytes,
                                    float* loss, float* eal, void* stream);

/* Backward of the sequence loss: grad_draft [B][seq_len][V] = dloss * dL/dz_q, each position's
 * row summed over the windows that contain it (in a fixed order, so results are reproducible).
 * Must follow aal_seq_loss_fwd on the same stream with the same problem, inputs and workspace.
 * Positions in no window's valid prefix get exact zeros; ties follow aal_loss_bwd. */
AAL_API aal_status aal_seq_loss_bwd(const aal_seq_problem* prob, const void* draft, const void* target,
                                    const uint8_t* mask, const void* workspace, size_t workspace_bytes,
                                    float dloss, void* grad_draft, void* stream);

/* Forward and backward of the sequence loss in one call (Sec. 3.3: every position's row is read
 * once for all K windows that contain it): the loss, eal and workspace of aal_seq_loss_fwd and
 * the gradient of aal_seq_loss_bwd with the same dloss, bit for bit (same arguments, layouts and
 * rules as those two calls).  With bf16 rows whose byte length is a multiple of 16, one
 * cooperative launch streams the positions with one CTA per SM, consecutive positions on
 * consecutive SMs at the same time, so that a position's gradient (which needs the acceptances
 * of the K - 1 positions before and after it) is written while its rows are still in L2: 2 V b
 * read and V b written per position, instead of 2 V b (forward) + 3 V b (backward); with token
 * ids (AAL_GREEDY | AAL_IDS) the draft alone is streamed the same way, V b read and V b written.
 * Other problems (fp32, unaligned rows) run the two calls inside this one.  AAL_GRPO is
 * rejected with AAL_ERR_UNSUPPORTED (its coefficients come from aal_seq_grpo_from_loss, between
 * the forward and the backward).  A bounded device wait that ran out is reported by
 * aal_check_device_status as AAL_ERR_TIMEOUT; the outputs are then not to be used. */
AAL_API aal_status aal_seq_loss_fwd_bwd(const aal_seq_problem* prob, const void* draft, const void* target,
                                        const uint8_t* mask, void* workspace, size_t workspace_bytes,
                                        float dloss, float* loss, float* eal, void* grad_draft, void* stream);

/* The GRPO surrogate of Sec. 3.4 over the windows of a completed aal_loss_fwd.
 *   N, K, V, dtype       must equal the loss problem's (windows of K depths, no mask: every
 *                        window is verified over all K depths).
 *   windows_per_rollout, rollouts_per_group, adv_clip   grouping and C_A as in
 *                        aal_reward_problem (N a multiple of their product); the paper's
 *                        samples are single windows (windows_per_rollout = 1, groups of m).
 *   eps_clip             PPO clip epsilon, in [0, 1).
 *   rho_min, rho_max     the ratio's safety clip, 0 <= rho_min <= rho_max (finite).
 *   log_rho_clip         clip of log rho before exponentiating (> 0; the paper uses 10).
 *   w_grpo               weight of L_GRPO in the gradient the loss backward adds (finite). */
typedef struct {
  int64_t N, K, V;
  int32_t dtype;
  int32_t reserved; /* must be 0 */
  int64_t windows_per_rollout;
  int64_t rollouts_per_group;
  float adv_clip;
  float eps_clip;
  float rho_min;
  float rho_max;
  float log_rho_clip;
  float w_grpo;
} aal_grpo_problem;

AAL_API aal_status aal_grpo_workspace_size(const aal_grpo_problem* prob, size_t* bytes);

/* GRPO stage of one batch (Sec. 3.4), from the statistics of a completed aal_loss_fwd whose mode
 * includes AAL_GRPO plus one pass over the reference draft.  Per window t with the draft's greedy
 * tokens S_k = argmax z_q (recorded by the forward):
 *   tau^theta, tau^ref    leading runs of S_k = x*_k and of argmax z_ref = x*_k (greedy
 *                         verification against the target's argmax, lowest index on ties);
 *   A                     the clipped group-standardised advantage of R = tau^theta - tau^ref
 *                         (as aal_accept_reward with the reference draft);
 *   log rho_t             (1/K) sum_k [log pi_theta(S_k) - log pi_ref(S_k)] (softmax at T = 1),
 *                         clipped to [-log_rho_clip, log_rho_clip];
 *   rho_t                 exp(log rho_t) clipped to [rho_min, rho_max];
 *   L_GRPO                -(1/N) sum_t min(rho_t A_t, clip(rho_t, 1 - eps, 1 + eps) A_t), the mean
 *                         over equal groups of the groups' mean surrogates.
 * R and A carry no gradient; the trajectory is held fixed.  The call writes, into the loss
 * workspace, w_grpo times dL_GRPO/d log pi_theta(S_k) for every row, which the following
 * aal_loss_bwd (same problem, mode with AAL_GRPO) turns into c (delta_{u,S_k} - q(u)); the
 * objective whose gradient that backward writes is therefore the forward's loss plus
 * w_grpo * L_GRPO.
 *   gprob, lprob           the GRPO problem and the loss problem of the forward.
 *   loss_workspace         the forward's workspace (read, and its GRPO coefficients written).
 *   ref_draft              [N][K][V] logits of the frozen reference draft (16-byte aligned).
 *   workspace              at least aal_grpo_workspace_size(gprob) bytes, 256-byte aligned.
 *   grpo_loss              device float[1]: L_GRPO (unweighted).
 *   tau, tau_ref           device int32[N] or NULL.
 *   advantage              device float[N / windows_per_rollout] or NULL.
 *   log_rho                device float[N] (the clipped log rho) or NULL. */
AAL_API aal_status aal_grpo_from_loss(const aal_grpo_problem* gprob, const aal_problem* lprob,
                                      void* loss_workspace, size_t loss_workspace_bytes,
                                      const void* ref_draft, void* workspace, size_t workspace_bytes,
                                      float* grpo_loss, int32_t* tau, int32_t* tau_ref, float* advantage,
                                      float* log_rho, void* stream);

/* The GRPO stage over sequences (Sec. 3.4: the forward passes run once per sequence and the window
 * samples are sliced from them), after aal_seq_loss_fwd with a mode that includes AAL_GRPO.
 *   gprob      N = the number of windows; K, V, dtype equal the sequence problem's; grouping,
 *              clips and w_grpo as for aal_grpo_from_loss (N a multiple of
 *              windows_per_rollout * rollouts_per_group).
 *   starts     device int32[N]: the flat start position b * seq_len + t of each window, in
 *              ascending order, each window inside its sequence (t + K <= seq_len).  Windows may
 *              overlap.  A start that breaks this is reported as AAL_ERR_INVALID_ARG through the
 *              status word of `workspace` (aal_check_device_status) and its window reads nothing.
 *   ref_draft  [B][seq_len][V] logits of the reference draft: read once, every position.
 *   workspace  at least aal_seq_grpo_workspace_size() bytes, 256-byte aligned.
 * Outputs as for aal_grpo_from_loss (tau, tau_ref, log_rho per window).  The loss workspace
 * receives, per position, the sum over the windows that cover it of their coefficients, so the
 * following aal_seq_loss_bwd adds the gradient of w_grpo * L_GRPO to every covered position. */
AAL_API aal_status aal_seq_grpo_workspace_size(const aal_grpo_problem* gprob, const aal_seq_problem* sprob,
                                               size_t* bytes);
AAL_API aal_status aal_seq_grpo_from_loss(const aal_grpo_problem* gprob, const aal_seq_problem* sprob,
                                          void* loss_workspace, size_t loss_workspace_bytes,
                                          const void* ref_draft, const int32_t* starts, void* workspace,
                                          size_t workspace_bytes, float* grpo_loss, int32_t* tau,
                                          int32_t* tau_ref, float* advantage, float* log_rho, void* stream);

/* Reward mode flag: with AAL_SAMPLING, the drafted token is drawn from q~ instead of taken as
 * the draft's argmax (aal_reward_problem.mode = AAL_SAMPLING | AAL_SAMPLED_DRAFT). */
#define AAL_SAMPLED_DRAFT 4

/* Simulated acceptance reward of the GRPO stage (Sec. 3.4).
 *   N, K, V, dtype       as for the loss; K is the window size gamma (1..AAL_MAX_K).
 *   mode                 AAL_GREEDY: draft token S_k = argmax z_q is accepted iff it
 *                        equals x*_k = argmax z_p (simulated greedy verification).
 *                        AAL_SAMPLING: S_k is accepted iff u < min(1, p~(S_k)/q~(S_k))
 *                        (Sec. 2.3) with u = Philox4x32-10 uniform keyed by
 *                        (seed; window row_offset + n, depth k).
 *                        AAL_SAMPLING | AAL_SAMPLED_DRAFT: the same acceptance, with S_k drawn
 *                        from q~ (sampling verification's own draft token) by Gumbel-max:
 *                        S_k = argmax_v (z_q(v)/T + G_v), G_v = -ln(-ln U_v), U_v = word v mod 4
 *                        of Philox4x32-10 at counter (n_lo, n_hi, k, 1 + v div 4) mapped like u;
 *                        the reference draft uses the same G.  Its expected tau is the WTV
 *                        expected length.  (Not with aal_accept_reward_from_loss.)
 *   temperature          T for AAL_SAMPLING (finite, > 0).
 *   seed, row_offset     Philox key and the global index of window 0 (so a batch can be
 *                        streamed in pieces with the same draws).
 *   windows_per_rollout  consecutive windows forming one rollout (>= 1).
 *   rollouts_per_group   consecutive rollouts forming one advantage group (>= 1);
 *                        N must be a multiple of windows_per_rollout * rollouts_per_group.
 *   adv_clip             C_A of Eq. advantage (> 0). */
typedef struct {
  int64_t N, K, V;
  int32_t dtype;
  int32_t mode;
  float temperature;
  float adv_clip;
  uint64_t seed;
  int64_t row_offset;
  int64_t windows_per_rollout;
  int64_t rollouts_per_group;
} aal_reward_problem;

AAL_API aal_status aal_reward_workspace_size(const aal_reward_problem* prob, size_t* bytes);

/* tau^pi = sum_{k=1}^{K} prod_{j<=k} 1[S_j accepted] per window for the draft (and the
 * reference draft), R = tau^theta - tau^ref (Eq. debiased_reward; R = tau^theta when
 * ref_draft is NULL), rollout length = mean R over the rollout's windows, and
 * advantage A = clip((x - mean_g)/(std_g + 1e-6), -C_A, C_A) over each group of
 * rollouts with the population std (Eq. advantage).
 *   draft, target, ref_draft  [N][K][V] logits; ref_draft may be NULL.
 *   tau, tau_ref              device int32[N]; tau_ref may be NULL (ignored without ref).
 *   rollout_len, advantage    device float[N / windows_per_rollout]. */
AAL_API aal_status aal_accept_reward(const aal_reward_problem* prob, const void* draft,
                             const void* target, const void* ref_draft, void* workspace,
                             size_t workspace_bytes, int32_t* tau, int32_t* tau_ref,
                             float* rollout_len, float* advantage, void* stream);

/* The same reward for the draft alone (R = tau^theta), taken from the statistics that
 * aal_loss_fwd left in `loss_workspace` instead of from the logits: the forward already
 * streams z_p and z_q and records, per row, x* = argmax z_p, the draft's greedy token
 * S_k = argmax z_q (lowest index on ties), z_p(S_k) and the normalisers.  No logit is read,
 * so a training step that computes the loss and the GRPO reward over the same logits
 * (Sec. 3.4 with the surrogate of Sec. 3.2 / 3.3) reads them once for both.
 *   rprob     N, K, V, dtype must equal lprob's.  AAL_GREEDY works after any loss mode;
 *             AAL_SAMPLING needs a loss mode with the sampling term at the same temperature
 *             (the normalisers of p~ and q~ at T); otherwise AAL_ERR_INVALID_ARG.
 *   lprob, loss_workspace  the problem and workspace of a completed aal_loss_fwd (same stream).
 *   workspace  at least aal_reward_workspace_size(rprob) bytes.
 * Outputs as for aal_accept_reward (no reference draft). */
AAL_API aal_status aal_accept_reward_from_loss(const aal_reward_problem* rprob, const aal_problem* lprob,
                                               const void* loss_workspace, size_t loss_workspace_bytes,
                                               void* workspace, size_t workspace_bytes, int32_t* tau,
                                               float* rollout_len, float* advantage, void* stream);

/* The sampled-draft reward (mode AAL_SAMPLING | AAL_SAMPLED_DRAFT, no reference draft) with the
 * normalisers of p~ and q~ that aal_loss_fwd left in `loss_workspace`: the draws need every
 * vocabulary entry of the draft, so the draft is streamed once (V b a row), but not the target,
 * which is read at the drawn token only, and no log-sum-exp is formed.  The draws are those of
 * aal_accept_reward; the acceptance uses the loss forward's normalisers instead of the reward's
 * own, which may differ from them in the last bits, so a draw within rounding of its threshold
 * may be decided the other way.
 *   rprob     mode AAL_SAMPLING | AAL_SAMPLED_DRAFT; N, K, V, dtype must equal lprob's.
 *   lprob, loss_workspace  a completed aal_loss_fwd (same stream) whose mode has the sampling
 *             term at the reward's temperature (not token ids); otherwise AAL_ERR_INVALID_ARG.
 *   draft, target  the [N][K][V] logits of that forward, 16-byte aligned.
 *   workspace  at least aal_reward_workspace_size(rprob) bytes.
 * Outputs as for aal_accept_reward (no reference draft).  Rows whose byte length is not a
 * multiple of 16 run aal_accept_reward's own pass. */
AAL_API aal_status aal_accept_reward_sampled_from_loss(const aal_reward_problem* rprob, const aal_problem* lprob,
                                                       const void* draft, const void* target,
                                                       const void* loss_workspace, size_t loss_workspace_bytes,
                                                       void* workspace, size_t workspace_bytes, int32_t* tau,
                                                       float* rollout_len, float* advantage, void* stream);

/* aal_accept_reward without a workspace argument: the scratch lives in a fixed array inside
 * the library.  The paper has no counterpart; this exists for callers that cannot allocate
 * device memory -- e.g. a training loop whose device memory is all reserved up front by its
 * own caching allocator, so a raw cudaMalloc would fail or fragment that pool, or a component
 * that only receives device pointers from another one and has no allocator of its own.
 *   Limit.   N * K <= 1048576 logit rows; larger problems return AAL_ERR_UNSUPPORTED before
 *            anything is launched.  The array (6 MiB + 4 KiB) is held by every GPU that loads
 *            the library until the process exits.
 *   Set-up.  The first call on a device (with that device current) looks up the array's device
 *            address once; make that first call before any stream capture.
 *   Sharing. Every call uses the same array, which keeps the last call's contents (each call
 *            clears what must start at zero).  Calls that overlap on the GPU (different streams,
 *            or different host threads) race on it: order them.
 *   Allocation.  Calls no cudaMalloc, cudaFree or allocating routine.
 * Other arguments and results are those of aal_accept_reward. */
AAL_API aal_status aal_accept_reward_noalloc(const aal_reward_problem* prob, const void* draft,
                                             const void* target, const void* ref_draft, int32_t* tau,
                                             int32_t* tau_ref, float* rollout_len, float* advantage,
                                             void* stream);

/* Synchronises `stream`, reads the device status word of a loss, reward or GRPO workspace,
 * clears it, and returns AAL_OK or the recorded device error: AAL_ERR_TIMEOUT (a bounded wait
 * ran out) or AAL_ERR_INVALID_ARG (a target token id outside [0, V) under AAL_IDS). */
AAL_API aal_status aal_check_device_status(void* workspace, void* stream);

/* Static description of a status code; never NULL. */
AAL_API const char* aal_status_string(aal_status status);

/* Version of the ABI described by this header (major * 10000 + minor * 100 + patch). */
AAL_API int32_t aal_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* AAL_H_ */
