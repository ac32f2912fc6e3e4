// Forward per-row statistics, GB300 path: whole rows per CTA, streamed through a shared-memory
// ring by the Tensor Memory Accelerator (one producer thread issues 1-D bulk copies into a FIFO
// of slots, completion counted in bytes on an mbarrier per slot; slots are released as soon as
// a chunk has been consumed, so the copies run ahead of the arithmetic by the whole ring).
//
// Same outputs as the generic kernel in rowstats.cu: the normalisers (M, Ls) of z_p/T,
// z_q/T and z_q, x* = argmax z_p with a^greedy = q(x*) (Eq. acc_greedy), and the sums
// a^sample = sum_v min(p~_v, q~_v) (Eq. acc_sample) and Qlt = sum_{q~_v < p~_v} q~_v.
//
//   * rowstats_twopass (a sampling or TV term): a^sample needs both normalisers first, so every
//     row is streamed twice, pass 1 from HBM (kept in L2, evict_last) and pass 2 right after it
//     from L2 (evict_first).  The consumer warps fold pass 1 into online max / log-sum-exp /
//     argmax state and reduce it across the CTA, then fold pass 2 into the overlap sums; a
//     finisher warp sums those and writes the row's outputs while the consumers go on to the
//     next row.  The re-read follows the load within one row's pass 1, inside the time L2 takes
//     to turn over at full streaming rate (~18 us): orders that re-read later miss in L2.
//   * rowstats_stream (no sampling term: greedy EAL, the KL anchor, the GRPO statistics): one
//     pass at T = 1, where the normalisers of z_p and z_q are those of p and q themselves.  It
//     finds the argmaxes only to the 16-byte vector; resolve_argmax then reads those two vectors
//     of each row again (64 bytes) to place x* and y exactly.  With the KL anchor the pass also
//     folds D = sum_v e_v (z_p,v - z_q,v) next to the log-sum-exp of z_p at T = 1; beside a
//     sampling term at T != 1 that is a second z_p state, next to the one at T.  Its REWARD
//     instance runs at the reward's T and decides the sampling acceptance at each row's end.
//
// There is no cross-CTA communication, so all 152 SMs run one CTA each (two with the short-row
// geometry of rowstats_short.cu).  Every wait is
// bounded (ptx::wait_phase); after a timeout every thread keeps walking the same loops
// without waiting (a consumer still folds a chunk it finds landed, into results that are
// never written), so all meet the same barriers, the producer drains its copies, and the
// kernel returns with AAL_ERR_TIMEOUT in the workspace status word.
#include "stream_core.cuh"

namespace aal {
namespace {

// An L2 prefetch of global memory (no shared-memory destination, nothing to wait on).
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Chunks of the next row that the two-pass producer prefetches into L2 when it starts a row's
// L2 pass: its ring slots then hold that pass's chunks, so without the prefetch the next row's
// first HBM copies would be issued only a few chunks before they are needed.
constexpr int kPrefetchChunks = 2;

}  // namespace
}  // namespace aal

namespace aal {
namespace {

using namespace ptx;

// ---------------------------------------------------------------- whole-chunk steps

// Pass 1 on one ring chunk (chunk c of the row): fold both tensors' vectors into A.  Full bf16
// chunks take kNV vectors per thread on the packed path; the partial last chunk, and fp32 rows,
// walk their vectors one by one.
template <typename T, bool NEED_Q1, bool KL = false, bool P1 = false>
__device__ __forceinline__ void p1_chunk(RowPart& A, const unsigned char* slot, int c, int nfull, int V, int t,
                                         float sT) {
  constexpr int ES = sizeof(T), E = 16 / ES, CH = kHalfSlot / ES;
  const int e0 = c * CH;
  const uint4* P = reinterpret_cast<const uint4*>(slot);
  const uint4* Q = reinterpret_cast<const uint4*>(slot + kHalfSlot);
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

// What the overlap pass of a row needs from its reduced pass-1 state: the unscaled offsets
// nC = -(M + Ls / s), and where the two argmax vectors lie (cx: the chunk of x*'s vector for
// the one thread that streams it, -1 for every other thread; ix: the vector in the chunk).
struct P2Row {
  float nCp, nCq;
  float av, qv;
  int32_t ab, qb;
  int32_t cx, ix, cy, iy;
};

// A first-occurrence result of the overlap pass, written by the thread that finds it.
struct ArgSlot {
  int32_t index;
  float carry;
};

template <typename T>
__device__ __forceinline__ P2Row p2_row(const RowPart& tot, float Mp, float Lsp, float Mq, float Lsq, float sT, int V,
                                        int t) {
  constexpr int E = 16 / sizeof(T), CH = kHalfSlot / sizeof(T);
  P2Row x;
  x.nCp = -(Mp + Lsp / sT);
  x.nCq = -(Mq + Lsq / sT);
  x.av = tot.av;
  x.qv = tot.qv;
  x.ab = tot.ab;
  x.qb = tot.qb;
  // a vector start outside [0, V) (no maximum: an all -inf row, or a state read after an abort)
  // is located nowhere, so no thread indexes the ring with it
  const bool okx = tot.ab >= 0 && tot.ab < V, oky = tot.qb >= 0 && tot.qb < V;
  const int cx = okx ? tot.ab / CH : -1, ix = okx ? (tot.ab - cx * CH) / E : 0;
  const int cy = oky ? tot.qb / CH : -1, iy = oky ? (tot.qb - cy * CH) / E : 0;
  x.cx = (okx && t == ix % kConsumers) ? cx : -1;
  x.ix = ix;
  x.cy = (oky && t == iy % kConsumers) ? cy : -1;
  x.iy = iy;
  return x;
}

struct P2Acc {
  float2 smin2, sqlt2;  // bf16 path (fp32 pairs)
  float smin, sqlt;     // fp32 path
};
__device__ __forceinline__ void p2_init(P2Acc& s) {
  s.smin2 = s.sqlt2 = make_float2(0.f, 0.f);
  s.smin = s.sqlt = 0.f;
}

// Pass 2 on one ring chunk: the overlap sums, and the exact first argmax of either tensor by
// the thread that streams its vector.
template <typename T>
__device__ __forceinline__ void p2_chunk(P2Acc& s, const P2Row& x, const unsigned char* slot, int c, int nfull,
                                         int V, int t, float sT, ArgSlot* ax, ArgSlot* ay) {
  constexpr int ES = sizeof(T), E = 16 / ES, CH = kHalfSlot / ES;
  const int e0 = c * CH;
  const uint4* P = reinterpret_cast<const uint4*>(slot);
  const uint4* Q = reinterpret_cast<const uint4*>(slot + kHalfSlot);
  if (c == x.cx) {
    int at;
    float carry;
    find_first<T>(P[x.ix], Q[x.ix], x.av, &at, &carry);
    ax->index = x.ab + at;
    ax->carry = carry;
  }
  if (c == x.cy) {
    int at;
    float carry;
    find_first<T>(Q[x.iy], P[x.iy], x.qv, &at, &carry);
    ay->index = x.qb + at;
    ay->carry = carry;
  }
  if (sizeof(T) == 2 && c < nfull) {
#pragma unroll
    for (int v = 0; v < kNV; ++v) {
      const int i = t + v * kConsumers;
      phase2_bf16(s.smin2, s.sqlt2, P[i], Q[i], sT, x.nCp, x.nCq);
    }
  } else {
    const int nvec = min(CH, V - e0) / E;
    for (int i = t; i < nvec; i += kConsumers) {
      if (sizeof(T) == 2) phase2_bf16(s.smin2, s.sqlt2, P[i], Q[i], sT, x.nCp, x.nCq);
      else phase2_vec<T>(s.smin, s.sqlt, P[i], Q[i], sT, x.nCp, x.nCq);
    }
  }
}

// A thread's overlap sums reduced over its warp (every lane gets them), in the order the
// kernels have always used: the fp32 pairs folded into the scalars, then a butterfly.
__device__ __forceinline__ float2 p2_warp_sum(const P2Acc& s) {
  float smin = s.smin + (s.smin2.x + s.smin2.y);
  float sqlt = s.sqlt + (s.sqlt2.x + s.sqlt2.y);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    smin += __shfl_xor_sync(0xffffffffu, smin, off);
    sqlt += __shfl_xor_sync(0xffffffffu, sqlt, off);
  }
  return make_float2(smin, sqlt);
}

// The producer's last copy into each slot must have landed before the CTA may exit (bounded).
__device__ __forceinline__ void drain_ring(uint64_t* full, uint32_t armed, uint32_t last_phase, uint64_t limit_ns) {
  for (int q = 0; q < kSlots; ++q) {
    if (!(armed & (1u << q))) continue;
    const uint32_t ph = (last_phase >> q) & 1u;
    const uint64_t t0 = now_ns();
    for (uint32_t it = 0; it < kSpinLimit && !mbar_try(&full[q], ph, 100000); ++it)
      if (now_ns() - t0 > limit_ns) break;
  }
}

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
    static_assert(PASSES == 1, "the two-pass statistics run in rowstats_twopass");
    const float sT = REWARD ? a.sT : kLog2e;
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
      if (REWARD) {
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
    }
  }
  __syncwarp();
  __syncthreads();
}

// ---------------------------------------------------------------- two passes, finisher warp

// The two-pass statistics (a sampling or TV term), with the row ends taken off the consumers:
// per row, pass 1 (HBM) and its CTA reduction, then pass 2 (L2); each consumer warp posts its
// pass-2 sums on the mbarrier `hand` and goes on to the next row's pass 1 without waiting, and
// a finisher warp (warp kWarps + 1) forms the row's outputs and writes them to the workspace,
// then arrives on `fin`.  Before it posts row i, a warp waits for `fin` of row i - 1, so `hand`
// never runs two rows ahead of the finisher; the buffers are double, by row parity.  The pass
// order, and so the time between a row's HBM pass and its L2 re-read, is that of the
// single-warp-finish form.
constexpr int kThreads2 = kThreads + 32;  // + the finisher warp

struct Smem2 {
  uint64_t full[kSlots];
  uint64_t empty[kSlots];
  uint64_t hand;   // the consumer warps' pass-2 sums of a row are in red2[] (the finisher takes over)
  uint64_t fin;    // the finisher is done with a row's buffers
  RowPart red[2][kWarps];  // by row parity
  float2 red2[2][kWarps];
  ArgSlot ax[2], ay[2];    // x* (with z_q there) and the draft argmax (with z_p there)
  float nst[2][9];         // Mp, Lsp, Mq, Lsq, Mq1, Lsq1, Mp1, Lsp1, KL of the row
  int abort_flag;
};

template <typename T, bool NEED_Q1, bool KL, bool P1 = false>
__global__ void __launch_bounds__(kThreads2, kCtasPerSm) rowstats_twopass(RowStatsArgs a, int nch, uint64_t limit_ns) {
  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* ring = smem;
  Smem2& S = *reinterpret_cast<Smem2*>(smem + kSlots * kSlotBytes);
  volatile int* abort_flag = &S.abort_flag;
  WsHeader* hdr = a.ws.hdr;
  constexpr int ES = sizeof(T);
  constexpr int CH = kHalfSlot / ES;
  const int V = (int)a.V;
  const int nfull = V / CH;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the CTA's rows: blockIdx.x + i * gridDim.x, i < m
  const int64_t m = a.R > (int64_t)blockIdx.x ? (a.R - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  auto row = [&](int64_t i) { return (int64_t)blockIdx.x + i * gridDim.x; };

  if (threadIdx.x == 0) {
    for (int k = 0; k < kSlots; ++k) {
      mbar_init(&S.full[k], 1);
      mbar_init(&S.empty[k], kWarps);
    }
    mbar_init(&S.hand, kWarps);
    mbar_init(&S.fin, 1);
    for (int q = 0; q < 2; ++q) {
      S.ax[q] = ArgSlot{0x7fffffff, 0.f};
      S.ay[q] = ArgSlot{0x7fffffff, 0.f};
    }
    S.abort_flag = 0;
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
      for (int64_t i = 0; i < m && !*abort_flag; ++i) {
        const int64_t r = row(i);
        const char* prow = static_cast<const char*>(a.zp) + r * a.V * ES;
        const char* qrow = static_cast<const char*>(a.zq) + r * a.V * ES;
        for (int pass = 0; pass < 2 && !*abort_flag; ++pass) {
          const uint64_t pol = pass == 0 ? keep : drop;
          if (pass == 1 && i + 1 < m) {  // the next row's first chunks, into L2
            const int64_t rn = row(i + 1);
            const uint32_t pb = (uint32_t)(min((int64_t)kPrefetchChunks * CH, (int64_t)V) * ES);
            bulk_prefetch_l2(static_cast<const char*>(a.zp) + rn * a.V * ES, pb);
            bulk_prefetch_l2(static_cast<const char*>(a.zq) + rn * a.V * ES, pb);
          }
          for (int c = 0; c < nch; ++c) {
            if (!wait_phase(&S.empty[pos.slot], pos.phase ^ 1u, abort_flag, limit_ns, hdr)) break;
            const int e0 = c * CH;
            const uint32_t bytes = (uint32_t)(min(CH, V - e0) * ES);
            if (seq != a.skip_chunk) {  // (the test hook leaves one chunk's barrier unarmed)
              mbar_expect_tx(&S.full[pos.slot], 2u * bytes);
              bulk_load(ring + pos.slot * kSlotBytes, prow + (int64_t)e0 * ES, bytes, &S.full[pos.slot], pol);
              bulk_load(ring + pos.slot * kSlotBytes + kHalfSlot, qrow + (int64_t)e0 * ES, bytes,
                        &S.full[pos.slot], pol);
              armed |= 1u << pos.slot;
              last_phase = (last_phase & ~(1u << pos.slot)) | (pos.phase << pos.slot);
            }
            pos.next();
            ++seq;
          }
        }
      }
      drain_ring(S.full, armed, last_phase, limit_ns);
    }
  } else if (warp == kWarps + 1) {
    // ------------------------------------------------------------ finisher
    for (int64_t i = 0; i < m; ++i) {
      const uint32_t par = (uint32_t)(i & 1);
      wait_phase(&S.hand, par, abort_flag, limit_ns, hdr);
      if (lane == 0) {
        float2 x = S.red2[par][0];
        for (int w = 1; w < kWarps; ++w) {
          x.x += S.red2[par][w].x;
          x.y += S.red2[par][w].y;
        }
        const float* n = S.nst[par];
        const ArgSlot gx = S.ax[par], gy = S.ay[par];
        if (!*abort_flag) {
          const int64_t r = row(i);
          a.ws.cpart[r * kMaxCluster] = x;
          a.ws.Mp[r] = n[0];
          a.ws.Lsp[r] = n[1];
          a.ws.Mq[r] = n[2];
          a.ws.Lsq[r] = n[3];
          a.ws.Mq1[r] = n[4];
          a.ws.Lsq1[r] = n[5];
          if (KL) {
            a.ws.Mp1[r] = n[6];
            a.ws.Lsp1[r] = n[7];
            a.ws.kl[r] = n[8];
          }
          a.ws.xstar[r] = gx.index;
          a.ws.ag[r] = exp2f(log2_prob(gx.carry, kLog2e, n[4], n[5]));
          a.ws.yhat[r] = gy.index;
          a.ws.zpy[r] = gy.carry;
        }
        S.ax[par] = ArgSlot{0x7fffffff, 0.f};
        S.ay[par] = ArgSlot{0x7fffffff, 0.f};
        mbar_arrive(&S.fin);
      }
      __syncwarp();
    }
  } else {
    // ------------------------------------------------------------ consumers
    const int t = threadIdx.x;
    const float sT = a.sT;
    RingPos pos;
    for (int64_t i = 0; i < m; ++i) {
      const uint32_t par = (uint32_t)(i & 1);
      // pass 1: online normalisers and argmax (HBM)
      RowPart A;
      part_init(A);
      for (int c = 0; c < nch; ++c, pos.next()) {
        if (wait_full(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr))
          p1_chunk<T, NEED_Q1, KL, P1>(A, ring + pos.slot * kSlotBytes, c, nfull, V, t, sT);
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
      }
      warp_part<NEED_Q1, KL, P1>(A, sT);
      if (lane == 0) S.red[par][warp] = A;
      named_barrier(kBarRow, kConsumers);
      RowPart tot;
      if (lane < kWarps) tot = S.red[par][lane];
      else part_init(tot);
      warp_part<NEED_Q1, KL, P1>(tot, sT);
      const float Mp = tot.pM, Lsp = log2f(tot.pS);
      const float Mq = tot.qM, Lsq = log2f(tot.qS);
      const P2Row cur = p2_row<T>(tot, Mp, Lsp, Mq, Lsq, sT, V, t);
      if (t == 0) {  // (row i - 2's buffers: the finisher was waited for before row i - 1 was posted)
        float* n = S.nst[par];
        n[0] = Mp;
        n[1] = Lsp;
        n[2] = Mq;
        n[3] = Lsq;
        n[4] = NEED_Q1 ? tot.q1M : Mq;
        n[5] = NEED_Q1 ? log2f(tot.q1S) : Lsq;
        if (KL) kl_stats<NEED_Q1, P1>(tot, Mp, Lsp, Mq, Lsq, n[6], n[7], n[8]);
      }
      // pass 2: overlap sums (L2)
      P2Acc acc;
      p2_init(acc);
      for (int c = 0; c < nch; ++c, pos.next()) {
        if (wait_full(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr))
          p2_chunk<T>(acc, cur, ring + pos.slot * kSlotBytes, c, nfull, V, t, sT, &S.ax[par], &S.ay[par]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
      }
      const float2 x = p2_warp_sum(acc);
      // the finisher must be done with row i - 1 before row i is posted
      if (i >= 1) wait_phase(&S.fin, par ^ 1u, abort_flag, limit_ns, hdr);
      if (lane == 0) {
        S.red2[par][warp] = x;
        mbar_arrive(&S.hand);
      }
    }
  }
  __syncwarp();
  __syncthreads();
}

constexpr size_t kSmemBytes = (size_t)kSlots * kSlotBytes + sizeof(Smem);
constexpr size_t kSmem2Bytes = (size_t)kSlots * kSlotBytes + sizeof(Smem2);

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

template <typename T, bool NEED_Q1, bool KL, bool P1 = false>
cudaError_t launch_twopass(const RowStatsArgs& a, cudaStream_t s, int nch, uint64_t limit_ns) {
  auto kern = rowstats_twopass<T, NEED_Q1, KL, P1>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem2Bytes);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t grid = (int64_t)sms * kCtasPerSm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  kern<<<(unsigned)grid, kThreads2, kSmem2Bytes, s>>>(a, nch, limit_ns);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_two_pass(const RowStatsArgs& a, cudaStream_t s, int nch, uint64_t limit_ns) {
  if (a.need_kl)  // at T = 1 the pass's normalisers are the anchor's; else both are kept
    return a.need_q1 ? launch_twopass<T, true, true, true>(a, s, nch, limit_ns)
                     : launch_twopass<T, false, true>(a, s, nch, limit_ns);
  return a.need_q1 ? launch_twopass<T, true, false>(a, s, nch, limit_ns)
                   : launch_twopass<T, false, false>(a, s, nch, limit_ns);
}

}  // namespace

// The exported launchers; rowstats_short.cu compiles this file again for short rows, under
// other names and another ring geometry.
#ifndef AAL_ROWSTATS_STREAM_NAME
#define AAL_ROWSTATS_STREAM_NAME launch_rowstats_stream
#define AAL_REWARD_STREAM_NAME launch_reward_stream
#endif

cudaError_t AAL_ROWSTATS_STREAM_NAME(const RowStatsArgs& a, bool bf16, cudaStream_t s, uint64_t limit_ns) {
  const int elt = bf16 ? 2 : 4;
  const int64_t CH = kHalfSlot / elt;
  const int nch = (int)((a.V + CH - 1) / CH);
  if (!a.overlap) return bf16 ? launch_one_pass<uint16_t>(a, s, nch, limit_ns) : launch_one_pass<float>(a, s, nch, limit_ns);
  return bf16 ? launch_two_pass<uint16_t>(a, s, nch, limit_ns) : launch_two_pass<float>(a, s, nch, limit_ns);
}

cudaError_t AAL_REWARD_STREAM_NAME(const RowStatsArgs& a, cudaStream_t s, uint64_t limit_ns) {
  const int64_t CH = kHalfSlot / 2;
  const int nch = (int)((a.V + CH - 1) / CH);
  return launch_T<uint16_t, false, 1, false, false, true>(a, s, nch, limit_ns);
}

}  // namespace aal
