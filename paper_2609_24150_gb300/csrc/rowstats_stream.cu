// Forward per-row statistics, GB300 path: whole rows per CTA, streamed twice through a
// shared-memory ring by the Tensor Memory Accelerator.
//
// Same outputs as the generic kernel in rowstats.cu: the normalisers (M, Ls) of z_p/T,
// z_q/T and z_q, x* = argmax z_p with a^greedy = q(x*) (Eq. acc_greedy), and the sums
// a^sample = sum_v min(p~_v, q~_v) (Eq. acc_sample) and Qlt = sum_{q~_v < p~_v} q~_v.
// a^sample needs both normalisers first, so every row is visited twice:
//
//   * One producer thread per CTA walks its rows and, for each, issues the row's chunks
//     twice into a FIFO ring of shared-memory slots with 1-D TMA bulk copies (completion
//     counted in bytes on an mbarrier per slot).  The first pass comes from HBM and is kept
//     in L2 (evict_last); the second pass, a row later at most, is served from L2 and is
//     marked evict_first.  Slots are released as soon as a chunk has been consumed, so the
//     copies run ahead of the arithmetic by the whole ring.
//   * The consumer warps fold each first-pass chunk into online max / log-sum-exp / argmax
//     state, reduce it across the CTA at the end of the row, then fold each second-pass
//     chunk into the overlap sums.  The producer keeps streaming through that reduction.
//
// Problems without the sampling term (greedy EAL, the KL anchor, the GRPO statistics) need
// neither the second pass nor a temperature: they run the same kernel with one pass at T = 1,
// where the normalisers of z_p and z_q are those of p and q themselves.  The first pass
// finds the argmaxes only to the 16-byte vector; resolve_argmax then reads those two
// vectors of each row again (64 bytes) to place x* and y exactly.  With the KL anchor the
// first pass also folds D = sum_v e_v (z_p,v - z_q,v) next to the log-sum-exp of z_p at
// T = 1; beside a sampling term at T != 1 that is a second z_p state, next to the one at T.
//
// There is no cross-CTA communication, so all 152 SMs run one CTA each.  Every wait is
// bounded (ptx::wait_phase); after a timeout every thread keeps walking the same loops
// without waiting (a consumer still folds a chunk it finds landed, into results that are
// never written), so all meet the same named barriers, the producer drains its copies,
// and the kernel returns with AAL_ERR_TIMEOUT in the workspace status word.
#include "stream_core.cuh"

namespace aal {
namespace {

using namespace ptx;
// ---------------------------------------------------------------- the kernel

// PASSES = 2: the sampling term (normalisers at T, then the overlap sums).  PASSES = 1: no
// sampling term; everything at T = 1 (sT is log2 e), argmaxes resolved by resolve_argmax.
// KL: the anchor's D next to the z_p normaliser at T = 1: the pass's own when it runs at T = 1,
// else (P1, with NEED_Q1) a second z_p state at T = 1 beside the one at T.
template <typename T, bool NEED_Q1, int PASSES, bool KL, bool P1 = false, bool REWARD = false>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) rowstats_stream(RowStatsArgs a, int nch, uint64_t limit_ns) {
  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* ring = smem;
  Smem& S = *reinterpret_cast<Smem*>(smem + kSlots * kSlotBytes);
  volatile int* abort_flag = &S.abort_flag;
  WsHeader* hdr = a.ws.hdr;
  constexpr int ES = sizeof(T);
  constexpr int E = 16 / ES;          // elements per 16-byte vector
  constexpr int CH = kHalfSlot / ES;  // elements per chunk per tensor
  const int V = (int)a.V;
  const int nfull = V / CH;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int k = 0; k < kSlots; ++k) {
      mbar_init(&S.full[k], 1);
      mbar_init(&S.empty[k], kWarps);
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
      int64_t seq = 0;                       // chunks walked, in ring order
      uint32_t armed = 0, last_phase = 0;    // per slot: a copy was issued, and its phase
      static_assert(kSlots <= 32, "slot bitmasks");
      for (int64_t r = blockIdx.x; r < a.R && !*abort_flag; r += gridDim.x) {
        const char* prow = static_cast<const char*>(a.zp) + r * a.V * ES;
        const char* qrow = static_cast<const char*>(a.zq) + r * a.V * ES;
        for (int pass = 0; pass < PASSES && !*abort_flag; ++pass) {
          const uint64_t pol = (pass == 0 && PASSES == 2) ? keep : drop;
          for (int c = 0; c < nch; ++c) {
            if (!wait_phase(&S.empty[pos.slot], pos.phase ^ 1u, abort_flag, limit_ns, hdr)) break;
            const int e0 = c * CH;
            const uint32_t bytes = (uint32_t)(min(CH, V - e0) * ES);
            if (seq != a.skip_chunk) {  // (the test hook leaves one chunk's barrier unarmed)
              mbar_expect_tx(&S.full[pos.slot], 2u * bytes);
              bulk_load(ring + pos.slot * kSlotBytes, prow + (int64_t)e0 * ES, bytes, &S.full[pos.slot], pol);
              bulk_load(ring + pos.slot * kSlotBytes + kHalfSlot, qrow + (int64_t)e0 * ES, bytes, &S.full[pos.slot],
                        pol);
              armed |= 1u << pos.slot;
              last_phase = (last_phase & ~(1u << pos.slot)) | (pos.phase << pos.slot);
            }
            pos.next();
            ++seq;
          }
        }
      }
      // drain: the last copy issued into each slot must have landed before the CTA may exit
      for (int k = 0; k < kSlots; ++k) {
        if (!(armed & (1u << k))) continue;
        const uint32_t ph = (last_phase >> k) & 1u;
        const uint64_t t0 = now_ns();
        for (uint32_t it = 0; it < kSpinLimit && !mbar_try(&S.full[k], ph, 100000); ++it)
          if (now_ns() - t0 > limit_ns) break;
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    const int t = threadIdx.x;
    RingPos pos;
    uint32_t j = 0;
    const float sT = (PASSES == 2 || REWARD) ? a.sT : kLog2e;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x, ++j) {
      // pass 1: online normalisers and argmax
      RowPart A;
      part_init(A);
      for (int c = 0; c < nch; ++c, pos.next()) {
        if (wait_full(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr)) {
          const int e0 = c * CH;
          const uint4* P = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes);
          const uint4* Q = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes + kHalfSlot);
          if (sizeof(T) == 2 && c < nfull) {
            uint4 pv[kNV], qv[kNV];
#pragma unroll
            for (int v = 0; v < kNV; ++v) {
              pv[v] = P[t + v * kConsumers];
              qv[v] = Q[t + v * kConsumers];
            }
            phase1_bf16<kNV, NEED_Q1, KL, P1>(A, pv, qv, e0 + t * E, kConsumers * E, sT);
          } else {
            const int nvec = min(CH, V - e0) / E;
            for (int i = t; i < nvec; i += kConsumers) {
              if (sizeof(T) == 2) phase1_bf16<1, NEED_Q1, KL, P1>(A, P + i, Q + i, e0 + i * E, 0, sT);
              else phase1_vec<T, NEED_Q1, KL, P1>(A, P[i], Q[i], e0 + i * E, sT);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
      }
      warp_part<NEED_Q1, KL, P1>(A, sT);
      if (lane == 0) S.red[j & 1][warp] = A;
      named_barrier(kBarRow, kConsumers);
      // every warp combines the warp partials itself (lanes >= kWarps carry the identity)
      RowPart tot;
      if (lane < kWarps) tot = S.red[j & 1][lane];
      else part_init(tot);
      warp_part<NEED_Q1, KL, P1>(tot, sT);
      const float Mp = tot.pM, Lsp = log2f(tot.pS);
      const float Mq = tot.qM, Lsq = log2f(tot.qS);
      if (KL && t == 0 && !*abort_flag) {
        float Mp1, Lsp1, kl;
        kl_stats<NEED_Q1, P1>(tot, Mp, Lsp, Mq, Lsq, Mp1, Lsp1, kl);
        a.ws.Mp1[r] = Mp1;
        a.ws.Lsp1[r] = Lsp1;
        a.ws.kl[r] = kl;
      }
      if (PASSES == 1 && REWARD) {
        if (t == 0) {
          // the sampling reward (Sec. 3.4, Eq. acc_sample): the draft's greedy token y (the first
          // maximum of z_q, placed inside its recorded vector, read again from L2) and z_p there;
          // accept iff u < min(1, p~(y) / q~(y)), with log2 q~(y) = -Ls_q since z_q peaks at y
          const T* zp = static_cast<const T*>(a.zp) + r * a.V;
          const T* zq = static_cast<const T*>(a.zq) + r * a.V;
          int32_t xs, ys;
          float cx, cy;
          resolve_vectors<T>(zp, zq, a.V, -1, *abort_flag ? -1 : tot.qb, &xs, &cx, &ys, &cy);
          const int64_t n = r / a.K;
          const uint32_t k = (uint32_t)(r - n * a.K);
          const float u = philox_uniform(a.seed, (uint64_t)(a.row_offset + n), k);
          const float d = log2_prob(cy, sT, Mp, Lsp) + Lsq;
          if (!*abort_flag) a.acc[r] = (u < exp2f(fminf(d, 0.f))) ? 1 : 0;
        }
        continue;
      }
      if (PASSES == 1) {
        if (t == 0) {
          if (!*abort_flag) {
            a.ws.Mp[r] = Mp;
            a.ws.Lsp[r] = Lsp;
            a.ws.Mq[r] = Mq;
            a.ws.Lsq[r] = Lsq;
            a.ws.Mq1[r] = Mq;
            a.ws.Lsq1[r] = Lsq;
            a.ws.cpart[r * kMaxCluster] = make_float2(0.f, 0.f);
          }
          // the first vector holding each maximum, which resolve_argmax turns into the element;
          // -1 (no vector) after an abort, so that it reads nothing
          a.ws.xstar[r] = *abort_flag ? -1 : tot.ab;
          a.ws.yhat[r] = *abort_flag ? -1 : tot.qb;
        }
        continue;
      }

      // pass 2: overlap sums
      float smin = 0.f, sqlt = 0.f;
      float2 smin2 = make_float2(0.f, 0.f), sqlt2 = make_float2(0.f, 0.f);
      // overlap pass in unscaled units: log2 p~ = (z - Cp) s with Cp = Mp + Lsp / s
      const float nCp = -(Mp + Lsp / a.sT), nCq = -(Mq + Lsq / a.sT);
      // the vector that holds the first z_p maximum: chunk cstar, vector istar, thread tstar
      const int cstar = tot.ab == 0x7fffffff ? -1 : tot.ab / CH;
      const int istar = tot.ab == 0x7fffffff ? 0 : (tot.ab - cstar * CH) / E;
      const int tstar = istar % kConsumers;
      const int cyh = tot.qb == 0x7fffffff ? -1 : tot.qb / CH;  // same for the draft argmax
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
          if (sizeof(T) == 2 && c < nfull) {
#pragma unroll
            for (int v = 0; v < kNV; ++v) {
              const int i = t + v * kConsumers;
              phase2_bf16(smin2, sqlt2, P[i], Q[i], a.sT, nCp, nCq);
            }
          } else {
            const int nvec = min(CH, V - e0) / E;
            for (int i = t; i < nvec; i += kConsumers) {
              if (sizeof(T) == 2) phase2_bf16(smin2, sqlt2, P[i], Q[i], a.sT, nCp, nCq);
              else phase2_vec<T>(smin, sqlt, P[i], Q[i], a.sT, nCp, nCq);
            }
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
      if (t == 0 && !*abort_flag) {
        float2 x = S.red2[j & 1][0];
        for (int k = 1; k < kWarps; ++k) {
          x.x += S.red2[j & 1][k].x;
          x.y += S.red2[j & 1][k].y;
        }
        const float Mq1 = NEED_Q1 ? tot.q1M : Mq;
        const float Lsq1 = NEED_Q1 ? log2f(tot.q1S) : Lsq;
        a.ws.cpart[r * kMaxCluster] = x;
        a.ws.Mp[r] = Mp;
        a.ws.Lsp[r] = Lsp;
        a.ws.Mq[r] = Mq;
        a.ws.Lsq[r] = Lsq;
        a.ws.Mq1[r] = Mq1;
        a.ws.Lsq1[r] = Lsq1;
        a.ws.xstar[r] = S.arg_index;
        a.ws.ag[r] = exp2f(log2_prob(S.arg_carry, kLog2e, Mq1, Lsq1));
        a.ws.yhat[r] = S.yarg_index;
        a.ws.zpy[r] = S.yarg_carry;
        S.arg_index = 0x7fffffff;
        S.arg_carry = 0.f;
        S.yarg_index = 0x7fffffff;
        S.yarg_carry = 0.f;
      }
      __syncwarp();
    }
  }
  __syncwarp();
  __syncthreads();
}

constexpr size_t kSmemBytes = (size_t)kSlots * kSlotBytes + sizeof(Smem);

template <typename T, bool NEED_Q1, int PASSES, bool KL, bool P1 = false, bool REWARD = false>
cudaError_t launch_T(const RowStatsArgs& a, cudaStream_t s, int nch, uint64_t limit_ns) {
  auto kern = rowstats_stream<T, NEED_Q1, PASSES, KL, P1, REWARD>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t grid = (int64_t)sms * kCtasPerSm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  kern<<<(unsigned)grid, kThreads, kSmemBytes, s>>>(a, nch, limit_ns);
  return cudaGetLastError();
}

// One thread per row: the first element equal to the row maximum inside the vector the
// one-pass kernel recorded (x* for z_p, y for z_q), the other tensor's value there, and
// a^greedy = q(x*).
template <typename T>
__global__ void __launch_bounds__(256) resolve_argmax(RowStatsArgs a) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.R) return;
  const T* zp = static_cast<const T*>(a.zp) + r * a.V;
  const T* zq = static_cast<const T*>(a.zq) + r * a.V;
  const int32_t xb = a.ws.xstar[r], yb = a.ws.yhat[r];
  int32_t xs, ys;
  float cx, cy;
  resolve_vectors<T>(zp, zq, a.V, xb, yb, &xs, &cx, &ys, &cy);
  a.ws.xstar[r] = xs;
  a.ws.yhat[r] = ys;
  a.ws.zpy[r] = cy;
  a.ws.ag[r] = exp2f(log2_prob(cx, kLog2e, a.ws.Mq1[r], a.ws.Lsq1[r]));
}

template <typename T>
cudaError_t launch_one_pass(const RowStatsArgs& a, cudaStream_t s, int nch, uint64_t limit_ns) {
  cudaError_t e = a.need_kl ? launch_T<T, false, 1, true>(a, s, nch, limit_ns)
                            : launch_T<T, false, 1, false>(a, s, nch, limit_ns);
  if (e != cudaSuccess) return e;
  if (a.R < 1) return cudaSuccess;
  resolve_argmax<T><<<(unsigned)((a.R + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_two_pass(const RowStatsArgs& a, cudaStream_t s, int nch, uint64_t limit_ns) {
  if (a.need_kl)  // at T = 1 the pass's normalisers are the anchor's; else both are kept
    return a.need_q1 ? launch_T<T, true, 2, true, true>(a, s, nch, limit_ns)
                     : launch_T<T, false, 2, true>(a, s, nch, limit_ns);
  return a.need_q1 ? launch_T<T, true, 2, false>(a, s, nch, limit_ns) : launch_T<T, false, 2, false>(a, s, nch, limit_ns);
}

}  // namespace

cudaError_t launch_rowstats_stream(const RowStatsArgs& a, bool bf16, cudaStream_t s, uint64_t limit_ns) {
  const int elt = bf16 ? 2 : 4;
  const int64_t CH = kHalfSlot / elt;
  const int nch = (int)((a.V + CH - 1) / CH);
  if (!a.overlap) return bf16 ? launch_one_pass<uint16_t>(a, s, nch, limit_ns) : launch_one_pass<float>(a, s, nch, limit_ns);
  return bf16 ? launch_two_pass<uint16_t>(a, s, nch, limit_ns) : launch_two_pass<float>(a, s, nch, limit_ns);
}

cudaError_t launch_reward_stream(const RowStatsArgs& a, cudaStream_t s, uint64_t limit_ns) {
  const int64_t CH = kHalfSlot / 2;
  const int nch = (int)((a.V + CH - 1) / CH);
  return launch_T<uint16_t, false, 1, false, false, true>(a, s, nch, limit_ns);
}

}  // namespace aal
