// Forward and backward of the window losses in one call (aal_loss_fwd_bwd), GB300 path.
//
// The separate calls stream every row three times: twice in the forward (statistics from
// HBM, overlap sums from L2) and once more from HBM in the backward, which must wait for the
// window terms of all K depths.  Here the K rows of a window are held by K CTAs at the same
// time (a group), so that the gradient pass can follow the statistics while the rows are
// still in L2: per row, pass 1 from HBM, pass 2 (sampling term only) from L2, a group barrier
// that gives every CTA its window's acceptances, and pass 3 from L2 writing the gradient.
// The logits cross HBM once per step instead of twice.
//
// * Launch: cooperative, one CTA per SM (the ring takes ~193 KB of shared memory), grid =
//   G groups x K CTAs + S solo CTAs; CTA k of group g takes depth k of windows g, g + G, ...
//   A cooperative launch has all its CTAs resident at once, so a group never waits on a CTA
//   that is not running.
// * Solo CTAs: the S = 152 - G K SMs the groups leave over (5 at K = 7) each take whole
//   windows from the end of the batch: the statistics of the window's K rows one after
//   another, the K rows' coefficients from its own acceptances (no exchange), then the K
//   gradient rows.  The host gives them as many windows as balances the two kinds
//   (solo_windows_each); their rows stay in L2 for K rows' time instead of one.
// * Window exchange: once its row's statistics are in the workspace, thread 0 of each CTA
//   publishes the row's (a^greedy, a^sample) as one 64-bit word in a per-row mailbox that the
//   call filled with an all-ones sentinel, and warp 0 polls (bounded, like the ring waits; lane
//   j the word of depth j) the K words of its window until none is the sentinel.  The value is
//   its own ready flag, so one L2 round trip brings the data.  It then forms dE^g/da and dE^s/da with the window kernels' function
//   (window_term) and the row's gradient coefficients with the backward's (row_coef), from the
//   same floats the window kernel reads later, so that the gradient equals the one of
//   aal_loss_fwd + aal_loss_bwd bit for bit.  The loss is left to the window kernel, which runs
//   after this one over the statistics written here, exactly as in aal_loss_fwd.  The anchor
//   alone needs no window term and so no wait.
// * The counts of valid windows and positions that scale the gradient are taken from the mask
//   by count_valid before the launch (the separate forward gets them from its window kernel).
// * Sequence layout (aal_seq_loss_fwd_bwd, SEQ): rows are positions and a window starts at every
//   one, so a row's gradient needs the acceptances of the K - 1 positions on each side.  All CTAs
//   walk the positions from the last one down, CTA c taking rows R-1-c, R-1-c-C, ...: a round of
//   C consecutive positions is in flight at a time, so a row's neighbours are streamed beside it
//   (those of the last K - 1 CTAs' rows below them come with the next round), and warp 0 polls
//   the 2K - 1 mailbox words around its row (seq_exchange) and forms the row's coefficients as
//   the sequence window and gather kernels and the backward do, so that the result equals
//   aal_seq_loss_fwd + aal_seq_loss_bwd bit for bit.  Deadlock-free for C >= K (go_fused_seq).
// * Failure: every wait is bounded.  A CTA that gave up keeps walking its rows without waiting
//   and still publishes a word for each, so its group does not wait on it for the whole limit;
//   the workspace status word reports AAL_ERR_TIMEOUT and the outputs are not to be used.
#include <type_traits>

#include "grad_elem.cuh"
#include "stream_core.cuh"

namespace aal {
namespace {

constexpr int kBarCoef = 3;  // named barrier: the row's gradient coefficients are in shared memory

struct FusedSmem {
  Smem s;
  RowCoef coef;
  int32_t live;  // the row's gradient has a nonzero term
  // a solo CTA's window: its rows' statistics and acceptances, then their coefficients
  RowStat solo_st[AAL_MAX_K];
  float solo_ag[AAL_MAX_K], solo_as[AAL_MAX_K];
  RowCoef solo_coef[AAL_MAX_K];
  int32_t solo_live[AAL_MAX_K];
};

constexpr size_t kFusedSmemBytes = (size_t)kSlots * kSlotBytes + sizeof(FusedSmem);

// PASSES = 2 with the sampling (or TV) term, 1 without; NEED_Q1, KL, P1 as in rowstats_stream;
// GREEDY and Q1_IS_QT as in the backward.  bf16 rows only (16-byte multiples).
// SEQ: the sequence layout (rows are positions; see fused_seq_rows below).
template <bool NEED_Q1, int PASSES, bool KL, bool GREEDY, bool Q1_IS_QT, bool P1 = false, bool SEQ = false>
__global__ void __launch_bounds__(kThreads, 1) fused_rows(FusedArgs f, int nch, uint64_t limit_ns) {
  using T = uint16_t;
  constexpr bool SAMPLING = PASSES == 2;
  constexpr int E = 8;                // bf16 elements per 16-byte vector
  constexpr int CH = kHalfSlot / 2;   // elements per chunk per tensor
  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* ring = smem;
  FusedSmem& F = *reinterpret_cast<FusedSmem*>(smem + kSlots * kSlotBytes);
  Smem& S = F.s;
  const RowStatsArgs& a = f.st;
  volatile int* abort_flag = &S.abort_flag;
  WsHeader* hdr = a.ws.hdr;
  const int V = (int)a.V;
  const int nfull = V / CH;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = f.win.K;
  const int64_t N = f.win.N;
  const int G = f.groups;
  const int64_t NG = f.n_group;        // windows 0 .. NG - 1 go to the groups, the rest to the solo CTAs
  const bool solo = !SEQ && (int)blockIdx.x >= G * K;
  // sequence layout: CTA c takes rows R-1-c, R-1-c-C, ... (C = the grid), so that the rows in
  // flight at a time are consecutive positions and a row's neighbours within K - 1 positions,
  // whose statistics its gradient waits on, are taken in the same round or an adjacent one
  const int C = gridDim.x;
  const int g = blockIdx.x / K, k = blockIdx.x % K;  // (a group's CTA)
  const int so = (int)blockIdx.x - G * K;            // (a solo CTA)

  if (threadIdx.x == 0) {
    for (int q = 0; q < kSlots; ++q) {
      mbar_init(&S.full[q], 1);
      mbar_init(&S.empty[q], kWarps);
    }
    S.abort_flag = 0;
    S.arg_index = 0x7fffffff;
    S.arg_carry = 0.f;
    S.yarg_index = 0x7fffffff;
    S.yarg_carry = 0.f;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == kWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t keep = policy_evict_last(), drop = policy_evict_first();
      RingPos pos;
      int64_t seq = 0;
      uint32_t armed = 0, last_phase = 0;
      // passes [p0, p1) of row r: the statistics passes keep the row in L2, the gradient pass
      // (pass PASSES) is its last use
      auto issue = [&](int64_t r, int p0, int p1) {
        const char* prow = static_cast<const char*>(a.zp) + r * a.V * 2;
        const char* qrow = static_cast<const char*>(a.zq) + r * a.V * 2;
        for (int pass = p0; pass < p1 && !*abort_flag; ++pass) {
          const uint64_t pol = pass < PASSES ? keep : drop;
          for (int c = 0; c < nch; ++c) {
            if (!wait_phase(&S.empty[pos.slot], pos.phase ^ 1u, abort_flag, limit_ns, hdr)) break;
            const int e0 = c * CH;
            const uint32_t bytes = (uint32_t)(min(CH, V - e0) * 2);
            if (seq != a.skip_chunk) {  // (the test hook leaves one chunk's barrier unarmed)
              mbar_expect_tx(&S.full[pos.slot], 2u * bytes);
              bulk_load(ring + pos.slot * kSlotBytes, prow + (int64_t)e0 * 2, bytes, &S.full[pos.slot], pol);
              bulk_load(ring + pos.slot * kSlotBytes + kHalfSlot, qrow + (int64_t)e0 * 2, bytes, &S.full[pos.slot],
                        pol);
              armed |= 1u << pos.slot;
              last_phase = (last_phase & ~(1u << pos.slot)) | (pos.phase << pos.slot);
            }
            pos.next();
            ++seq;
          }
        }
      };
      if (SEQ) {
        for (int64_t p = a.R - 1 - blockIdx.x; p >= 0 && !*abort_flag; p -= C) issue(p, 0, PASSES + 1);
      } else if (!solo) {
        for (int64_t n = g; n < NG && !*abort_flag; n += G) issue(n * K + k, 0, PASSES + 1);
      } else {
        // a whole window: the statistics of its K rows, then their gradients
        for (int64_t n = NG + so; n < N && !*abort_flag; n += f.solos) {
          for (int kk = 0; kk < K; ++kk) issue(n * K + kk, 0, PASSES);
          for (int kk = 0; kk < K; ++kk) issue(n * K + kk, PASSES, PASSES + 1);
        }
      }
      for (int q = 0; q < kSlots; ++q) {
        if (!(armed & (1u << q))) continue;
        const uint32_t ph = (last_phase >> q) & 1u;
        const uint64_t t0 = now_ns();
        for (uint32_t it = 0; it < kSpinLimit && !mbar_try(&S.full[q], ph, 100000); ++it)
          if (now_ns() - t0 > limit_ns) break;
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    const int t = threadIdx.x;
    RingPos pos;
    uint32_t j = 0;  // rows walked (parity of the reduction buffers)
    const float sT = PASSES == 2 ? a.sT : kLog2e;
    // the backward's scales (thread 0 forms the coefficients)
    float scale = 0.f, kscale = 0.f;
    if (t == 0) {
      const int nvalid = hdr->nvalid;
      scale = nvalid > 0 ? -f.bw.dloss / (float)nvalid : 0.f;
      const int npos = KL ? hdr->npos : 0;
      kscale = npos > 0 ? f.bw.dloss * f.bw.w_kl / (float)npos : 0.f;
    }
    const bool ov = f.win.sampling || f.win.tv;

    // The statistics passes of row r: writes its statistics to the workspace; thread 0 gets what
    // the row's coefficients need (st) and its a^sample (st_as).
    auto stats_row = [&](int64_t r, RowStat& st, float& st_as) {
      // ---- pass 1: online normalisers and argmax (HBM)
      RowPart A;
      part_init(A);
      for (int c = 0; c < nch; ++c, pos.next()) {
        if (wait_full(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr)) {
          const int e0 = c * CH;
          const uint4* P = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes);
          const uint4* Q = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes + kHalfSlot);
          if (c < nfull) {
            uint4 pv[kNV], qv[kNV];
#pragma unroll
            for (int v = 0; v < kNV; ++v) {
              pv[v] = P[t + v * kConsumers];
              qv[v] = Q[t + v * kConsumers];
            }
            phase1_bf16<kNV, NEED_Q1, KL, P1>(A, pv, qv, e0 + t * E, kConsumers * E, sT);
          } else {
            const int nvec = (V - e0) / E;
            for (int i = t; i < nvec; i += kConsumers)
              phase1_bf16<1, NEED_Q1, KL, P1>(A, P + i, Q + i, e0 + i * E, 0, sT);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
      }
      warp_part<NEED_Q1, KL, P1>(A, sT);
      if (lane == 0) S.red[j & 1][warp] = A;
      named_barrier(kBarRow, kConsumers);
      RowPart tot;
      if (lane < kWarps) tot = S.red[j & 1][lane];
      else part_init(tot);
      warp_part<NEED_Q1, KL, P1>(tot, sT);
      const float Mp = tot.pM, Lsp = log2f(tot.pS);
      const float Mq = tot.qM, Lsq = log2f(tot.qS);
      if (KL && t == 0) {
        float Mp1, Lsp1, kl;
        kl_stats<NEED_Q1, P1>(tot, Mp, Lsp, Mq, Lsq, Mp1, Lsp1, kl);
        if (!*abort_flag) {
          a.ws.Mp1[r] = Mp1;
          a.ws.Lsp1[r] = Lsp1;
          a.ws.kl[r] = kl;
        }
        st.Mp1 = Mp1;
        st.Lsp1 = Lsp1;
      }
      if (PASSES == 1) {
        if (t == 0) {
          // x* and y to the element: their vectors are read again, from L2
          const T* zp = static_cast<const T*>(a.zp) + r * a.V;
          const T* zq = static_cast<const T*>(a.zq) + r * a.V;
          const bool ok = !*abort_flag;
          int32_t xs, ys;
          float cx, cy;
          resolve_vectors<T>(zp, zq, a.V, ok ? tot.ab : -1, ok ? tot.qb : -1, &xs, &cx, &ys, &cy);
          const float ag = exp2f(log2_prob(cx, kLog2e, Mq, Lsq));
          if (ok) {
            a.ws.Mp[r] = Mp;
            a.ws.Lsp[r] = Lsp;
            a.ws.Mq[r] = Mq;
            a.ws.Lsq[r] = Lsq;
            a.ws.Mq1[r] = Mq;
            a.ws.Lsq1[r] = Lsq;
            a.ws.cpart[r * kMaxCluster] = make_float2(0.f, 0.f);
            a.ws.xstar[r] = xs;
            a.ws.yhat[r] = ys;
            a.ws.zpy[r] = cy;
            a.ws.ag[r] = ag;
          }
          st.Mq1 = Mq;
          st.Lsq1 = Lsq;
          st.ag = ag;
          st.xs = xs;
          st.ys = ys;
          // a group CTA's row: its mailbox word as soon as it is known (the exchange then only polls)
          if (!solo) ptx::st_relaxed(&a.ws.mbox[r], mbox_word(ag, 0.f));
        }
      } else {
        // ---- pass 2: overlap sums (L2)
        float smin = 0.f, sqlt = 0.f;
        float2 smin2 = make_float2(0.f, 0.f), sqlt2 = make_float2(0.f, 0.f);
        const float nCp = -(Mp + Lsp / a.sT), nCq = -(Mq + Lsq / a.sT);
        const int cstar = tot.ab == 0x7fffffff ? -1 : tot.ab / CH;
        const int istar = tot.ab == 0x7fffffff ? 0 : (tot.ab - cstar * CH) / E;
        const int tstar = istar % kConsumers;
        const int cyh = tot.qb == 0x7fffffff ? -1 : tot.qb / CH;
        const int iyh = tot.qb == 0x7fffffff ? 0 : (tot.qb - cyh * CH) / E;
        const int tyh = iyh % kConsumers;
        for (int c = 0; c < nch; ++c, pos.next()) {
          if (wait_full(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr)) {
            const int e0 = c * CH;
            const uint4* P = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes);
            const uint4* Q = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes + kHalfSlot);
            if (c == cstar && t == tstar) {
              int at;
              float carry;
              find_first<T>(P[istar], Q[istar], tot.av, &at, &carry);
              S.arg_index = tot.ab + at;
              S.arg_carry = carry;
            }
            if (c == cyh && t == tyh) {
              int at;
              float carry;
              find_first<T>(Q[iyh], P[iyh], tot.qv, &at, &carry);
              S.yarg_index = tot.qb + at;
              S.yarg_carry = carry;
            }
            if (c < nfull) {
#pragma unroll
              for (int v = 0; v < kNV; ++v) {
                const int i = t + v * kConsumers;
                phase2_bf16(smin2, sqlt2, P[i], Q[i], a.sT, nCp, nCq);
              }
            } else {
              const int nvec = (V - e0) / E;
              for (int i = t; i < nvec; i += kConsumers) phase2_bf16(smin2, sqlt2, P[i], Q[i], a.sT, nCp, nCq);
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
        }
        smin += smin2.x + smin2.y;
        sqlt += sqlt2.x + sqlt2.y;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          smin += __shfl_xor_sync(0xffffffffu, smin, off);
          sqlt += __shfl_xor_sync(0xffffffffu, sqlt, off);
        }
        if (lane == 0) S.red2[j & 1][warp] = make_float2(smin, sqlt);
        named_barrier(kBarSum, kConsumers);
        if (t == 0) {
          float2 x = S.red2[j & 1][0];
          for (int w = 1; w < kWarps; ++w) {
            x.x += S.red2[j & 1][w].x;
            x.y += S.red2[j & 1][w].y;
          }
          const float Mq1 = NEED_Q1 ? tot.q1M : Mq;
          const float Lsq1 = NEED_Q1 ? log2f(tot.q1S) : Lsq;
          const float ag = exp2f(log2_prob(S.arg_carry, kLog2e, Mq1, Lsq1));
          if (!*abort_flag) {
            a.ws.cpart[r * kMaxCluster] = x;
            a.ws.Mp[r] = Mp;
            a.ws.Lsp[r] = Lsp;
            a.ws.Mq[r] = Mq;
            a.ws.Lsq[r] = Lsq;
            a.ws.Mq1[r] = Mq1;
            a.ws.Lsq1[r] = Lsq1;
            a.ws.xstar[r] = S.arg_index;
            a.ws.ag[r] = ag;
            a.ws.yhat[r] = S.yarg_index;
            a.ws.zpy[r] = S.yarg_carry;
          }
          st.Mq = Mq;
          st.Lsq = Lsq;
          st.Mp = Mp;
          st.Lsp = Lsp;
          st.Mq1 = Mq1;
          st.Lsq1 = Lsq1;
          st.qlt = x.y;
          st_as = x.x;
          st.ag = ag;
          st.xs = S.arg_index;
          st.ys = S.yarg_index;
          if (!solo) ptx::st_relaxed(&a.ws.mbox[r], mbox_word(ag, x.x));
          S.arg_index = 0x7fffffff;
          S.arg_carry = 0.f;
          S.yarg_index = 0x7fffffff;
          S.yarg_carry = 0.f;
        }
      }
      ++j;
    };

    // Thread 0: the coefficients of depth kk of window n (row r) from the window's acceptances
    // (agv, asv; 0 beyond K and for a term the window kernel does not form), as the window
    // kernel forms its terms and the backward its coefficients.  Returns whether any is nonzero.
    // LOCAL_DONE: the row-local part of c was formed already (row_coef_local).
    auto coef_row = [&](int64_t n, int kk, int64_t r, const float* agv, const float* asv, const RowStat& st,
                        RowCoef& c, auto local_done) -> int32_t {
      const int64_t r0 = n * K;
      int kn = K;
      if (f.win.mask != nullptr) {
        kn = 0;
        while (kn < K && f.win.mask[r0 + kn] != 0) ++kn;
      }
      float dE[AAL_MAX_K];
      float dEg = 0.f, dEs = 0.f;
      if (f.win.greedy) {
        window_term(agv, kn, dE);
        dEg = dE[kk];
      }
      if (ov) {
        if (f.win.sampling) window_term(asv, kn, dE);
        const float tvc = (f.win.tv && kn > 0) ? f.win.w_tv / (float)kn : 0.f;
        dEs = __fadd_rn(f.win.sampling ? __fmul_rn(f.win.w_sampling, dE[kk]) : 0.f, kk < kn ? tvc : 0.f);
      }
      const bool with_greedy = GREEDY && f.bw.w_greedy != 0.f;
      const bool pos_valid = f.bw.mask == nullptr || f.bw.mask[r] != 0;
      return row_coef<GREEDY, SAMPLING, KL, decltype(local_done)::value>(
                 f.bw, scale, kscale, with_greedy ? dEg : 0.f, SAMPLING ? dEs : 0.f, 0.f, pos_valid, st, c)
                 ? 1
                 : 0;
    };

    // ---- pass 3: the gradient row (L2)
    auto grad_row = [&](int64_t r, const RowCoef& c, int32_t live) {
      const int64_t xv = (live && c.xs >= 0) ? c.xs / E : -1;
      const int xe = c.xs >= 0 ? c.xs % E : 0;
      uint4* out4 = reinterpret_cast<uint4*>(static_cast<T*>(f.bw.grad) + r * a.V);
      const uint4 zero4 = make_uint4(0, 0, 0, 0);
      for (int cc = 0; cc < nch; ++cc, pos.next()) {
        if (wait_full(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr)) {
          const int e0 = cc * CH;
          const int64_t vb = e0 / E;
          const uint4* P = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes);
          const uint4* Q = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes + kHalfSlot);
          if (cc < nfull) {
#pragma unroll
            for (int v = 0; v < kNV; ++v) {
              const int i = t + v * kConsumers;
              st_stream(out4 + vb + i,
                        live ? grad_vec<T, GREEDY, SAMPLING, Q1_IS_QT, KL>(c, Q[i], P[i], vb + i, xv, xe, -1, 0) : zero4);
            }
          } else {
            const int nvec = (V - e0) / E;
            for (int i = t; i < nvec; i += kConsumers)
              st_stream(out4 + vb + i,
                        live ? grad_vec<T, GREEDY, SAMPLING, Q1_IS_QT, KL>(c, Q[i], P[i], vb + i, xv, xe, -1, 0) : zero4);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
      }
    };

    if (SEQ) {
      // row r's gradient: warp 0 takes the acceptances of rows r - K + 1 .. r + K - 1 (those of
      // its sequence) and forms the row's coefficients, as the sequence window and gather
      // kernels and the backward do, then every consumer writes the row
      const bool need = f.win.greedy || ov;
      const bool with_greedy = GREEDY && f.bw.w_greedy != 0.f;
      for (int64_t r = a.R - 1 - blockIdx.x; r >= 0; r -= C) {
        RowStat st{};
        float st_as = 0.f;
        stats_row(r, st, st_as);
        if (warp == 0) {
          const int64_t lo = r - r % f.seq_T, hi = lo + f.seq_T - 1;
          float dEg = 0.f, dEs = 0.f;
          RowCoef c;
          const bool ok = seq_exchange(a.ws.mbox, f.seq_mask, r, lo, hi, K, f.seq_full != 0, f.win.greedy,
                                       f.win.sampling, f.win.tv, f.win.w_sampling, f.win.w_tv, need, lane,
                                       abort_flag, hdr, limit_ns, &dEg, &dEs,
                                       [&]() { row_coef_local<GREEDY, SAMPLING, KL>(f.bw, st, c); });
          if (lane == 0) {
            const bool pos_valid = f.bw.mask == nullptr || f.bw.mask[r] != 0;
            F.live = ok && row_coef<GREEDY, SAMPLING, KL, true>(f.bw, scale, kscale, with_greedy ? dEg : 0.f,
                                                                SAMPLING ? dEs : 0.f, 0.f, pos_valid, st, c)
                         ? 1
                         : 0;
            if (F.live) F.coef = c;
          }
        }
        named_barrier(kBarCoef, kConsumers);
        const RowCoef c = F.coef;
        grad_row(r, c, F.live);
      }
    } else if (!solo) {
      // one row of each of the group's windows: statistics, the window exchange, the gradient
      for (int64_t n = g; n < NG; n += G) {
        const int64_t r = n * K + k;
        RowStat st{};
        float st_as = 0.f;
        stats_row(r, st, st_as);
        if (warp == 0) {
          const bool need = f.win.greedy || ov;  // the anchor alone needs no window term
          float agv[AAL_MAX_K], asv[AAL_MAX_K];
          // the row's word was published with its statistics; the row-local coefficients are
          // formed while the first poll of the window's words is in flight
          RowCoef c;
          const bool ok = window_exchange(a.ws.mbox, r, n * K, K, lane, st.ag, PASSES == 2 ? st_as : 0.f, need,
                                          abort_flag, hdr, limit_ns, agv, asv, false,
                                          [&]() { row_coef_local<GREEDY, SAMPLING, KL>(f.bw, st, c); });
#pragma unroll
          for (int jj = 0; jj < AAL_MAX_K; ++jj) {  // only the terms the window kernel forms
            if (!f.win.greedy) agv[jj] = 0.f;
            if (!ov) asv[jj] = 0.f;
          }
          if (lane == 0) {
            F.live = ok ? coef_row(n, k, r, agv, asv, st, c, std::true_type()) : 0;
            if (F.live) F.coef = c;
          }
        }
        named_barrier(kBarCoef, kConsumers);
        const RowCoef c = F.coef;
        grad_row(r, c, F.live);
      }
    } else {
      // whole windows: the statistics of the K rows, their coefficients from those rows alone
      // (no exchange), then the K gradient rows
      for (int64_t n = NG + so; n < N; n += f.solos) {
        for (int kk = 0; kk < K; ++kk) {
          RowStat st{};
          float st_as = 0.f;
          stats_row(n * K + kk, st, st_as);
          if (t == 0) {
            F.solo_st[kk] = st;
            F.solo_ag[kk] = f.win.greedy ? st.ag : 0.f;
            F.solo_as[kk] = ov && PASSES == 2 ? st_as : 0.f;
          }
        }
        if (t == 0) {
          float agv[AAL_MAX_K], asv[AAL_MAX_K];
#pragma unroll
          for (int jj = 0; jj < AAL_MAX_K; ++jj) {
            agv[jj] = jj < K ? F.solo_ag[jj] : 0.f;
            asv[jj] = jj < K ? F.solo_as[jj] : 0.f;
          }
          for (int kk = 0; kk < K; ++kk) {
            RowCoef c;
            const bool ok = !*abort_flag;
            F.solo_live[kk] = ok ? coef_row(n, kk, n * K + kk, agv, asv, F.solo_st[kk], c, std::false_type()) : 0;
            if (F.solo_live[kk]) F.solo_coef[kk] = c;
          }
        }
        named_barrier(kBarCoef, kConsumers);
        for (int kk = 0; kk < K; ++kk) {
          const RowCoef c = F.solo_coef[kk];
          grad_row(n * K + kk, c, F.solo_live[kk]);
        }
      }
    }
  }
  __syncwarp();
  __syncthreads();
}

// |W| (windows whose depth 0 is valid) and |positions| (valid rows) from the [N][K] mask, one
// block; integer sums, so the order does not matter.  Data-parallel normalisers given by the
// caller (nvalid_g, npos_g >= 0) replace the counts.
__global__ void __launch_bounds__(1024) count_valid(const uint8_t* mask, int64_t N, int32_t K, int32_t nvalid_g,
                                                    int32_t npos_g, WsHeader* hdr) {
  __shared__ unsigned long long sw, sp;
  if (threadIdx.x == 0) {
    sw = 0ull;
    sp = 0ull;
  }
  __syncthreads();
  unsigned long long w = 0, p = 0;
  if (mask == nullptr) {
    if (threadIdx.x == 0) {
      w = (unsigned long long)N;
      p = (unsigned long long)(N * K);
    }
  } else {
    for (int64_t n = threadIdx.x; n < N; n += blockDim.x) w += mask[n * K] != 0;
    for (int64_t r = threadIdx.x; r < N * K; r += blockDim.x) p += mask[r] != 0;
  }
  atomicAdd(&sw, w);
  atomicAdd(&sp, p);
  __syncthreads();
  if (threadIdx.x == 0) {
    hdr->nvalid = nvalid_g >= 0 ? nvalid_g : (int32_t)sw;
    hdr->npos = npos_g >= 0 ? npos_g : (int32_t)sp;
  }
}

// The sequence layout's counts, as the sequence window kernel takes them: window n is in W when
// its leading valid run K_n (stopping at the sequence's end or its first invalid position) is
// >= 1, i.e. when position n is valid, or = K with full windows; positions count when valid.
// Without a mask these are closed forms, and data-parallel counts given by the caller
// (nvalid_g, npos_g >= 0) replace them; otherwise integer sums over the grid, added into the
// header (zeroed by the caller), so the order does not matter.
__global__ void __launch_bounds__(1024) seq_count_valid(const uint8_t* mask, int64_t B, int64_t T, int32_t K,
                                                        bool full, int32_t nvalid_g, int32_t npos_g, WsHeader* hdr) {
  if (mask == nullptr || nvalid_g >= 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      const int64_t per_seq = full ? (T >= K ? T - K + 1 : 0) : T;
      hdr->nvalid = nvalid_g >= 0 ? nvalid_g : (int32_t)(B * per_seq);
      hdr->npos = npos_g >= 0 ? npos_g : (int32_t)(B * T);
    }
    return;
  }
  __shared__ unsigned int sw, sp;
  if (threadIdx.x == 0) {
    sw = 0u;
    sp = 0u;
  }
  __syncthreads();
  unsigned int w = 0, p = 0;
  for (int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; n < B * T; n += (int64_t)gridDim.x * blockDim.x) {
    if (mask[n] == 0) continue;
    ++p;
    if (!full) {
      ++w;
    } else if (n % T + K <= T) {
      int kk = 1;
      while (kk < K && mask[n + kk] != 0) ++kk;
      w += kk == K;
    }
  }
  atomicAdd(&sw, w);
  atomicAdd(&sp, p);
  __syncthreads();
  if (threadIdx.x == 0) {
    atomicAdd(reinterpret_cast<unsigned int*>(&hdr->nvalid), sw);
    atomicAdd(reinterpret_cast<unsigned int*>(&hdr->npos), sp);
  }
}

// The sequence layout: CTA c of C (one cooperative CTA per SM) takes rows R-1-c, R-1-c-C, ...,
// each row's statistics passes (S(p)) and then its gradient pass (G(p)), which waits on S(q) for
// |q - p| <= K - 1.  Order the work by rank(S(q)) = R-1-q and rank(G(p)) = R-1-p + K - 1/2: a
// gradient pass waits only on lower ranks, and a CTA's own sequence S(p), G(p), S(p - C), ...
// rises in rank when C >= K.  So every wait points to lower-ranked work, no cycle of waits can
// form, and the launch cannot deadlock while all its CTAs are resident (a cooperative launch).
// The caller takes the fused path only when C >= K or one round holds every row.
template <bool NQ1, int P, bool KL, bool GR, bool Q, bool P1 = false>
cudaError_t go_fused_seq(const FusedArgs& f0, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  auto kern = fused_rows<NQ1, P, KL, GR, Q, P1, true>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedSmemBytes);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per_sm = 0, coop = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, kFusedSmemBytes);
  if (e != cudaSuccess) return e;
  int64_t C = (int64_t)sms * per_sm;
  if (C > f0.st.R) C = f0.st.R;
  if (!coop || C < 1) return cudaSuccess;  // *launched stays false: the caller runs the two calls
  const int elt = 2;
  const int nch = (int)((f0.st.V + kHalfSlot / elt - 1) / (kHalfSlot / elt));
  FusedArgs f = f0;
  void* args[] = {&f, (void*)&nch, &limit_ns};
  e = cudaLaunchCooperativeKernel((const void*)kern, dim3((unsigned)C), dim3(kThreads), args, kFusedSmemBytes, s);
  if (e == cudaErrorCooperativeLaunchTooLarge) {
    cudaGetLastError();
    return cudaSuccess;
  }
  if (e == cudaSuccess) *launched = true;
  return e;
}

template <bool NQ1, int P, bool KL, bool GR, bool Q, bool P1 = false>
cudaError_t go_fused(const FusedArgs& f0, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  auto kern = fused_rows<NQ1, P, KL, GR, Q, P1>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedSmemBytes);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per_sm = 0, coop = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, kFusedSmemBytes);
  if (e != cudaSuccess) return e;
  const int64_t K = f0.win.K;
  int64_t G = (int64_t)sms * per_sm / K;
  if (G > f0.win.N) G = f0.win.N;
  if (G > kMaxGroups) G = kMaxGroups;
  if (!coop || G < 1) return cudaSuccess;  // *launched stays false: the caller runs the two calls
  // the SMs left over by the groups take whole windows alone
  const int64_t S = (int64_t)sms * per_sm - G * K;
  const int64_t m = solo_windows_each(f0.win.N, K, G, S);
  FusedArgs f = f0;
  f.groups = (int32_t)G;
  f.solos = m > 0 ? (int32_t)S : 0;
  f.n_group = f0.win.N - m * f.solos;
  const int elt = 2;
  const int nch = (int)((f.st.V + kHalfSlot / elt - 1) / (kHalfSlot / elt));
  void* args[] = {&f, (void*)&nch, &limit_ns};
  e = cudaLaunchCooperativeKernel((const void*)kern, dim3((unsigned)(G * K + f.solos)), dim3(kThreads), args,
                                  kFusedSmemBytes, s);
  if (e == cudaErrorCooperativeLaunchTooLarge) {  // fewer SMs available than the device has (shared
    cudaGetLastError();                           // device): the caller runs the two calls instead
    return cudaSuccess;
  }
  if (e == cudaSuccess) *launched = true;
  return e;
}

}  // namespace

cudaError_t launch_count_valid(const uint8_t* mask, int64_t N, int32_t K, int32_t nvalid_g, int32_t npos_g,
                               WsHeader* hdr, cudaStream_t s) {
  count_valid<<<1, 1024, 0, s>>>(mask, N, K, nvalid_g, npos_g, hdr);
  return cudaGetLastError();
}

cudaError_t launch_seq_count_valid(const uint8_t* mask, int64_t B, int64_t T, int32_t K, bool full,
                                   int32_t nvalid_g, int32_t npos_g, WsHeader* hdr, cudaStream_t s) {
  int64_t blocks = 1;
  if (mask != nullptr && nvalid_g < 0) {
    blocks = (B * T + 1023) / 1024;
    if (blocks > 152) blocks = 152;
    if (blocks < 1) blocks = 1;
  }
  seq_count_valid<<<(unsigned)blocks, 1024, 0, s>>>(mask, B, T, K, full, nvalid_g, npos_g, hdr);
  return cudaGetLastError();
}

namespace {
template <bool SEQ, bool NQ1, int P, bool KL, bool GR, bool Q, bool P1 = false>
cudaError_t go(const FusedArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  if constexpr (SEQ)
    return go_fused_seq<NQ1, P, KL, GR, Q, P1>(f, s, limit_ns, launched);
  else
    return go_fused<NQ1, P, KL, GR, Q, P1>(f, s, limit_ns, launched);
}

// The instantiation for the problem's flags, or none (launched = false) for a combination
// this path does not take.
template <bool SEQ>
cudaError_t dispatch_fused(const FusedArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  *launched = false;
  const bool two = f.st.overlap, kl = f.st.need_kl, nq1 = f.st.need_q1 && two;
  const bool greedy = f.bw.w_greedy != 0.f && !f.bw.grpo;
  const bool q = f.bw.q1_is_qT && two && (greedy || kl);
  if (!two) {
    if (greedy && !kl) return go<SEQ, false, 1, false, true, false>(f, s, limit_ns, launched);
    if (!greedy && kl) return go<SEQ, false, 1, true, false, false>(f, s, limit_ns, launched);
    if (greedy && kl) return go<SEQ, false, 1, true, true, false>(f, s, limit_ns, launched);
    return cudaSuccess;
  }
  if (kl) {  // at T = 1 q = q~ (one z_q state); else z_q and z_p both kept at T = 1 beside T
    if (q && !nq1)
      return greedy ? go<SEQ, false, 2, true, true, true>(f, s, limit_ns, launched)
                    : go<SEQ, false, 2, true, false, true>(f, s, limit_ns, launched);
    if (nq1 && !q)
      return greedy ? go<SEQ, true, 2, true, true, false, true>(f, s, limit_ns, launched)
                    : go<SEQ, true, 2, true, false, false, true>(f, s, limit_ns, launched);
    return cudaSuccess;
  }
  if (!greedy && !nq1 && !q) return go<SEQ, false, 2, false, false, false>(f, s, limit_ns, launched);
  if (greedy && !nq1 && q) return go<SEQ, false, 2, false, true, true>(f, s, limit_ns, launched);
  if (greedy && nq1 && !q) return go<SEQ, true, 2, false, true, false>(f, s, limit_ns, launched);
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_fused(const FusedArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  return dispatch_fused<false>(f, s, limit_ns, launched);
}

cudaError_t launch_fused_seq(const FusedArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  return dispatch_fused<true>(f, s, limit_ns, launched);
}

}  // namespace aal
