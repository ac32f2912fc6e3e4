// Forward per-row statistics, GB300 path: one thread-block cluster per logit row, the
// row held on chip.
//
// Same outputs as the generic kernel in rowstats.cu (the normalisers (M, Ls) of z_p/T,
// z_q/T and z_q, x* = argmax z_p, a^greedy = q(x*), and the per-CTA partial sums of
// a^sample = sum_v min(p~_v, q~_v) (Eq. acc_sample) and Qlt = sum_{q~_v < p~_v} q~_v),
// but each row is read from HBM once:
//
//   * The C CTAs of a cluster split the row's V into C contiguous slices; each CTA streams
//     its slice of z_p and z_q into a ring of shared-memory slots with 1-D TMA bulk copies
//     (cp.async.bulk, completion counted on an mbarrier), issued by one producer thread.
//   * Phase-1 warps fold each arriving chunk into online max / log-sum-exp / argmax
//     partials, reduce them across the CTA and push the CTA's partial into every peer's
//     shared memory (DSMEM stores + a remote mbarrier arrive).
//   * Phase-2 warps wait for all C partials of the row, combine them in rank order (every
//     CTA obtains bit-identical row statistics), then sweep the slice again -- from shared
//     memory -- for the overlap sums, and free the ring slots for the next row's copies.
//     Phase 1 of row i+1 runs while phase 2 of row i waits for the cluster exchange.
//
// Every wait is bounded by %globaltimer.  A wait that runs out records AAL_ERR_TIMEOUT
// in the workspace status word and raises a CTA-wide abort flag; from then on every
// thread keeps walking the same loop structure without waiting or computing, so all of
// them meet the same named barriers and the final cluster barrier, in-flight copies are
// drained, and the kernel returns.
#include "aal_internal.cuh"

namespace aal {
namespace {

constexpr int kSlots = 13;                       // ring slots per CTA
constexpr int kSlotBytes = 16384;                // 8 KB of z_p + 8 KB of z_q
constexpr int kHalfSlot = kSlotBytes / 2;
constexpr int kXDepth = 4;                       // depth of the partial-exchange ring
#ifndef AAL_RING_SLACK
#define AAL_RING_SLACK 3
#endif
constexpr int kSlack = AAL_RING_SLACK;           // slots a row leaves free for the next row
constexpr int kBarP1 = 1, kBarP2a = 2, kBarP2b = 3;

// A CTA's phase-1 partial of one row (48 bytes: three 16-byte DSMEM stores).
struct __align__(16) Part {
  float pM, pS, qM, qS;
  float q1M, q1S, av, ac;  // av: max z_p so far, ac: z_q at that index
  int32_t ai;
  int32_t pad[3];
};

struct Smem {
  uint64_t full[kSlots];
  uint64_t empty[kSlots];
  uint64_t xfull[kXDepth];
  uint64_t xempty[kXDepth];
  Part xpart[kXDepth][kMaxCluster];
  Part red1[2][8];
  float2 red2[2][8];
  int abort_flag;
};

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ uint32_t s32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(s32(b)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(s32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(s32(b)) : "memory");
}
// try_wait with a suspend-time hint: a thread whose phase has not completed sleeps in
// hardware (up to kSuspendNs) instead of spinning, leaving the issue slots to the warps
// that have work.
constexpr uint32_t kSuspendNs = 20000;
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(s32(b)), "r"(parity), "r"(kSuspendNs)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_test_cluster(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(s32(b)), "r"(parity), "r"(kSuspendNs)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint32_t map_rank(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(s32(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_remote(uint64_t* b, uint32_t rank) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(map_rank(b, rank)) : "memory");
}
__device__ __forceinline__ void st_remote(void* p, uint32_t rank, const uint4& v) {
  asm volatile("st.shared::cluster.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(map_rank(p, rank)), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ uint64_t evict_first_policy() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                          uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          s32(dst)),
      "l"(src), "r"(bytes), "r"(s32(bar)), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_index() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_barrier() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Named barrier over one warp group; the warp is reconverged first so that it arrives whole.
__device__ __forceinline__ void named_barrier(int id, int n) {
  __syncwarp();
  asm volatile("barrier.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
__device__ __forceinline__ uint64_t now_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait on an mbarrier phase.  Returns false if the abort flag is (or gets) set or
// the time limit passes; a timeout records the status and raises the abort flag.
template <bool CLUSTER>
__device__ __forceinline__ bool wait_phase(uint64_t* b, uint32_t parity, volatile int* abort_flag,
                                           uint64_t limit_ns, WsHeader* hdr) {
  if (CLUSTER ? mbar_test_cluster(b, parity) : mbar_test(b, parity)) return !*abort_flag;
  const uint64_t t0 = now_ns();
  for (uint32_t it = 0; it < kSpinLimit; ++it) {
    if (CLUSTER ? mbar_test_cluster(b, parity) : mbar_test(b, parity)) return true;
    if (*abort_flag) return false;
    if (now_ns() - t0 > limit_ns) break;
  }
  *abort_flag = 1;
  atomicExch(&hdr->status, kStatusTimeout);
  return false;
}

// ---------------------------------------------------------------- row arithmetic

__device__ __forceinline__ void part_init(Part& a) {
  a.pM = a.qM = a.q1M = -INFINITY;
  a.pS = a.qS = a.q1S = 0.f;
  a.av = -INFINITY;
  a.ac = 0.f;
  a.ai = 0x7fffffff;
}

__device__ __forceinline__ void lse_fold(float& M, float& S, float m, float Sb) {
  Lse x{M, S}, y{m, Sb};
  Lse r = lse_merge(x, y);
  M = r.M;
  S = r.S;
}

__device__ __forceinline__ Part part_merge(const Part& a, const Part& b) {
  Part r = a;
  lse_fold(r.pM, r.pS, b.pM, b.pS);
  lse_fold(r.qM, r.qS, b.qM, b.qS);
  lse_fold(r.q1M, r.q1S, b.q1M, b.q1S);
  if (b.av > a.av || (b.av == a.av && b.ai < a.ai)) {
    r.av = b.av;
    r.ai = b.ai;
    r.ac = b.ac;
  }
  return r;
}

__device__ __forceinline__ Part part_shfl(const Part& a, int off) {
  Part b;
  b.pM = __shfl_xor_sync(0xffffffffu, a.pM, off);
  b.pS = __shfl_xor_sync(0xffffffffu, a.pS, off);
  b.qM = __shfl_xor_sync(0xffffffffu, a.qM, off);
  b.qS = __shfl_xor_sync(0xffffffffu, a.qS, off);
  b.q1M = __shfl_xor_sync(0xffffffffu, a.q1M, off);
  b.q1S = __shfl_xor_sync(0xffffffffu, a.q1S, off);
  b.av = __shfl_xor_sync(0xffffffffu, a.av, off);
  b.ac = __shfl_xor_sync(0xffffffffu, a.ac, off);
  b.ai = __shfl_xor_sync(0xffffffffu, a.ai, off);
  return b;
}

// Fold n values of one tensor into an online (M, S): the unit's max first, so the running
// maximum moves at most once per unit and each value costs one fma, one ex2 and one add.
template <int N>
__device__ __forceinline__ void lse_unit(float& M, float& S, const float* v, float vmax, float s) {
  const float xm = __fmul_rn(vmax, s);
  if (xm > M) {
    S *= ex2(M - xm);  // M == -inf: ex2(-inf) = 0 and S is still 0
    M = xm;
  }
  if (M != -INFINITY) {
    float acc = 0.f;
#pragma unroll
    for (int e = 0; e < N; ++e) acc += ex2(fmaf(v[e], s, -M));
    S += acc;
  }
}

template <typename T>
__device__ __forceinline__ void unpack8(const uint4& w, float* o);
template <>
__device__ __forceinline__ void unpack8<uint16_t>(const uint4& w, float* o) {
  o[0] = bf16_lo(w.x);
  o[1] = bf16_hi(w.x);
  o[2] = bf16_lo(w.y);
  o[3] = bf16_hi(w.y);
  o[4] = bf16_lo(w.z);
  o[5] = bf16_hi(w.z);
  o[6] = bf16_lo(w.w);
  o[7] = bf16_hi(w.w);
}
template <>
__device__ __forceinline__ void unpack8<float>(const uint4& w, float* o) {
  o[0] = __uint_as_float(w.x);
  o[1] = __uint_as_float(w.y);
  o[2] = __uint_as_float(w.z);
  o[3] = __uint_as_float(w.w);
}

// ---- packed arithmetic (sm_100+): two fp32 lanes per instruction, exact IEEE rounding
#ifdef AAL_SCALAR_PAIRS
__device__ __forceinline__ float2 f2fma(float2 a, float2 b, float2 c) {
  return make_float2(fmaf(a.x, b.x, c.x), fmaf(a.y, b.y, c.y));
}
__device__ __forceinline__ float2 f2add(float2 a, float2 b) { return make_float2(a.x + b.x, a.y + b.y); }
#else
__device__ __forceinline__ float2 f2fma(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mov.b64 rc, {%6, %7};\n\tfma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 f2add(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
#endif
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ float set_lt(float a, float b) {  // 1.0f if a < b else 0.0f
  float d;
  asm("set.lt.f32.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}
// max of the 16 bf16 values in two 16-byte vectors (exact: max of bf16 values is a bf16 value)
__device__ __forceinline__ float bmax16(const uint4& a, const uint4& b) {
  const uint32_t m = bmax2(bmax2(bmax2(a.x, a.y), bmax2(a.z, a.w)), bmax2(bmax2(b.x, b.y), bmax2(b.z, b.w)));
  return fmaxf(bf16_lo(m), bf16_hi(m));
}
__device__ __forceinline__ float2 bpair(uint32_t w) { return make_float2(bf16_lo(w), bf16_hi(w)); }

// One tensor's 16 bf16 values folded into (M, S): max first, then 2^(z s - M) summed with
// packed fma / add over two independent accumulators.
__device__ __forceinline__ void lse16(float& M, float& S, const uint4& a, const uint4& b, float vmax, float s) {
  const float xm = __fmul_rn(vmax, s);
  if (xm > M) {
    S *= ex2(M - xm);
    M = xm;
  }
  if (M == -INFINITY) return;
  const float2 s2 = make_float2(s, s), m2 = make_float2(-M, -M);
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
  float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < 8; k += 2) {
    const float2 x0 = f2fma(bpair(w[k]), s2, m2);
    const float2 x1 = f2fma(bpair(w[k + 1]), s2, m2);
    acc0 = f2add(acc0, make_float2(ex2(x0.x), ex2(x0.y)));
    acc1 = f2add(acc1, make_float2(ex2(x1.x), ex2(x1.y)));
  }
  const float2 t = f2add(acc0, acc1);
  S += t.x + t.y;
}

// Phase 1 on a full bf16 chunk slice: 16 values of z_p and z_q per thread.
template <bool NEED_Q1>
__device__ __forceinline__ void phase1_bf16x16(Part& A, const uint4& p0, const uint4& p1, const uint4& q0,
                                               const uint4& q1, int64_t idx0, int64_t idx1, float sT) {
  const float pm = bmax16(p0, p1), qm = bmax16(q0, q1);
  if (pm > A.av) {  // new argmax of z_p: its first occurrence (rare after the first chunks)
    const uint32_t pw[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
    const uint32_t qw[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
    int e = 0;
    float carry = 0.f;
#pragma unroll
    for (int k = 15; k >= 0; --k) {
      const float v = (k & 1) ? bf16_hi(pw[k >> 1]) : bf16_lo(pw[k >> 1]);
      if (v == pm) {
        e = k;
        carry = (k & 1) ? bf16_hi(qw[k >> 1]) : bf16_lo(qw[k >> 1]);
      }
    }
    A.av = pm;
    A.ai = (int32_t)(e < 8 ? idx0 + e : idx1 + (e - 8));
    A.ac = carry;
  }
  lse16(A.pM, A.pS, p0, p1, pm, sT);
  lse16(A.qM, A.qS, q0, q1, qm, sT);
  if (NEED_Q1) lse16(A.q1M, A.q1S, q0, q1, qm, kLog2e);
}

// Phase 2 on 8 bf16 values of each tensor: sum_v min(p~, q~) and sum_{q~ < p~} q~.
__device__ __forceinline__ void phase2_bf16x8(float2& smin2, float2& sqlt2, const uint4& pw, const uint4& qw,
                                              float2 s2, float2 negM, float2 negLs) {
  const uint32_t pa[4] = {pw.x, pw.y, pw.z, pw.w};
  const uint32_t qa[4] = {qw.x, qw.y, qw.z, qw.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    // lanes (p, q) of element 2k and of element 2k+1
    const float2 l0 = f2add(f2fma(make_float2(bf16_lo(pa[k]), bf16_lo(qa[k])), s2, negM), negLs);
    const float2 l1 = f2add(f2fma(make_float2(bf16_hi(pa[k]), bf16_hi(qa[k])), s2, negM), negLs);
    const float2 e = make_float2(ex2(fminf(l0.x, l0.y)), ex2(fminf(l1.x, l1.y)));
    smin2 = f2add(smin2, e);
    sqlt2 = f2fma(e, make_float2(set_lt(l0.y, l0.x), set_lt(l1.y, l1.x)), sqlt2);
  }
}

template <typename T, bool NEED_Q1>
__device__ __forceinline__ void phase1_vec(Part& A, const uint4& pw, const uint4& qw, int64_t idx0, float sT) {
  constexpr int E = 16 / sizeof(T);
  float pv[8], qv[8];
  unpack8<T>(pw, pv);
  unpack8<T>(qw, qv);
  float pm = pv[0], qm = qv[0];
#pragma unroll
  for (int e = 1; e < E; ++e) {
    pm = fmaxf(pm, pv[e]);
    qm = fmaxf(qm, qv[e]);
  }
  if (pm > A.av) {  // new argmax of z_p: the first element equal to the unit's max
    int e = 0;
    float carry = qv[0];
#pragma unroll
    for (int k = E - 1; k >= 0; --k) {
      if (pv[k] == pm) {
        e = k;
        carry = qv[k];
      }
    }
    A.av = pm;
    A.ai = (int32_t)(idx0 + e);
    A.ac = carry;
  }
  lse_unit<E>(A.pM, A.pS, pv, pm, sT);
  lse_unit<E>(A.qM, A.qS, qv, qm, sT);
  if (NEED_Q1) lse_unit<E>(A.q1M, A.q1S, qv, qm, kLog2e);
}

template <typename T>
__device__ __forceinline__ void phase2_vec(float& smin, float& sqlt, const uint4& pw, const uint4& qw, float sT,
                                           float Mp, float Lsp, float Mq, float Lsq) {
  constexpr int E = 16 / sizeof(T);
  float pv[8], qv[8];
  unpack8<T>(pw, pv);
  unpack8<T>(qw, qv);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const float lp = fmaf(pv[e], sT, -Mp) - Lsp;
    const float lq = fmaf(qv[e], sT, -Mq) - Lsq;
    const float t = ex2(fminf(lp, lq));
    smin += t;
    sqlt += (lq < lp) ? t : 0.f;
  }
}

// ---------------------------------------------------------------- the kernel

#ifndef AAL_GROUP_WARPS
#define AAL_GROUP_WARPS 8
#endif
constexpr int kGroupWarps = AAL_GROUP_WARPS;  // warps in each of the two consumer groups
constexpr int kVecPerChunk = kHalfSlot / 16;   // 16-byte vectors per tensor per chunk

// Ring position: slot index and phase parity advanced one chunk at a time.
struct RingPos {
  int slot = 0;
  uint32_t phase = 0;
  __device__ __forceinline__ void next() {
    if (++slot == kSlots) {
      slot = 0;
      phase ^= 1u;
    }
  }
};

template <typename T, bool NEED_Q1, int G>
__global__ void __launch_bounds__(32 * (1 + 2 * G), 1)
    rowstats_cluster(RowStatsArgs a, int C, int m, int nch, uint64_t limit_ns) {
  constexpr int GT = 32 * G;                // threads per consumer group
  constexpr int NV = kVecPerChunk / GT;     // vectors per thread per full chunk
  static_assert(NV * GT == kVecPerChunk, "group must tile the chunk");
  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* ring = smem;
  Smem& S = *reinterpret_cast<Smem*>(smem + kSlots * kSlotBytes);
  volatile int* abort_flag = &S.abort_flag;
  WsHeader* hdr = a.ws.hdr;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int64_t cid = cluster_index(), ncl = cluster_count();
  constexpr int ES = sizeof(T);
  constexpr int E = 16 / ES;           // elements per 16-byte vector
  constexpr int CH = kHalfSlot / ES;   // elements per chunk per tensor
  const int V = (int)a.V;
  const int c0 = (int)rank * m;
  const int c1 = min(nch, c0 + m);
  const int nfull = V / CH;            // chunks [0, nfull) are full

  if (threadIdx.x == 0) {
    for (int k = 0; k < kSlots; ++k) {
      mbar_init(&S.full[k], 1);
      mbar_init(&S.empty[k], G);
    }
    for (int k = 0; k < kXDepth; ++k) {
      mbar_init(&S.xfull[k], (uint32_t)C);
      mbar_init(&S.xempty[k], (uint32_t)C);
    }
    S.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  cluster_barrier();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = evict_first_policy();
      RingPos pos;
      uint32_t issued = 0;
      for (int64_t r = cid; r < a.R && !*abort_flag; r += ncl) {
        const char* prow = static_cast<const char*>(a.zp) + r * a.V * ES;
        const char* qrow = static_cast<const char*>(a.zq) + r * a.V * ES;
        for (int c = c0; c < c1; ++c) {
          if (!wait_phase<false>(&S.empty[pos.slot], pos.phase ^ 1u, abort_flag, limit_ns, hdr)) break;
          const int e0 = c * CH;
          const uint32_t bytes = (uint32_t)(min(CH, V - e0) * ES);
          mbar_expect_tx(&S.full[pos.slot], 2u * bytes);
          bulk_load(ring + pos.slot * kSlotBytes, prow + (int64_t)e0 * ES, bytes, &S.full[pos.slot], pol);
          bulk_load(ring + pos.slot * kSlotBytes + kHalfSlot, qrow + (int64_t)e0 * ES, bytes, &S.full[pos.slot], pol);
          pos.next();
          ++issued;
        }
      }
      // drain: every copy issued must have landed before the CTA may exit
      const uint32_t first = issued > (uint32_t)kSlots ? issued - (uint32_t)kSlots : 0u;
      for (uint32_t j = first; j < issued; ++j) {
        const uint64_t t0 = now_ns();
        for (uint32_t it = 0; it < kSpinLimit && !mbar_test(&S.full[j % kSlots], (j / kSlots) & 1u); ++it)
          if (now_ns() - t0 > limit_ns) break;
      }
    }
  } else if (warp <= G) {
    // ------------------------------------------------------------ phase 1
    const int t = threadIdx.x - 32;
    const int w = t >> 5;
    RingPos pos;
    uint32_t j = 0;
    for (int64_t r = cid; r < a.R; r += ncl, ++j) {
      Part A;
      part_init(A);
      for (int c = c0; c < c1; ++c, pos.next()) {
        if (!wait_phase<false>(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr)) continue;
        const int e0 = c * CH;
        const uint4* P = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes);
        const uint4* Q = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes + kHalfSlot);
        if (sizeof(T) == 2 && c < nfull) {
#pragma unroll
          for (int v = 0; v < NV; v += 2) {
            const int i0 = t + v * GT, i1 = i0 + GT;
            phase1_bf16x16<NEED_Q1>(A, P[i0], P[i1], Q[i0], Q[i1], e0 + i0 * E, e0 + i1 * E, a.sT);
          }
        } else {
          const int nvec = min(CH, V - e0) / E;
          for (int i = t; i < nvec; i += GT) phase1_vec<T, NEED_Q1>(A, P[i], Q[i], e0 + i * E, a.sT);
        }
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) A = part_merge(A, part_shfl(A, off));
      if (lane == 0) S.red1[j & 1][w] = A;
      named_barrier(kBarP1, GT);
      if (w == 0) {
        // lanes 0..G-1 hold the warp partials; a fixed butterfly over them (the other lanes
        // carry the identity) leaves the CTA partial in lane 0
        Part tot;
        if (lane < G) tot = S.red1[j & 1][lane];
        else part_init(tot);
#pragma unroll
        for (int off = G / 2; off > 0; off >>= 1) tot = part_merge(tot, part_shfl(tot, off));
        tot = part_shfl(tot, lane);  // lane 0's value to every lane
        const int s = (int)(j % kXDepth);
        bool ok = false;
        if (lane == 0) ok = wait_phase<true>(&S.xempty[s], ((j / kXDepth) & 1u) ^ 1u, abort_flag, limit_ns, hdr);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (ok && lane < C) {  // lane c writes this CTA's partial into peer c, then signals it
          const uint4* src = reinterpret_cast<const uint4*>(&tot);
          uint4* dst = reinterpret_cast<uint4*>(&S.xpart[s][rank]);
          st_remote(dst + 0, (uint32_t)lane, src[0]);
          st_remote(dst + 1, (uint32_t)lane, src[1]);
          st_remote(dst + 2, (uint32_t)lane, src[2]);
          mbar_arrive_remote(&S.xfull[s], (uint32_t)lane);
        }
      }
      __syncwarp();
    }
  } else {
    // ------------------------------------------------------------ phase 2
    const int t = threadIdx.x - 32 * (1 + G);
    const int w = t >> 5;
    RingPos pos;
    uint32_t j = 0;
    for (int64_t r = cid; r < a.R; r += ncl, ++j) {
      const int s = (int)(j % kXDepth);
      Part tot;
      part_init(tot);
      const bool ok = wait_phase<true>(&S.xfull[s], (j / kXDepth) & 1u, abort_flag, limit_ns, hdr);
      if (ok) {
        tot = S.xpart[s][0];
        for (int k = 1; k < C; ++k) tot = part_merge(tot, S.xpart[s][k]);
      }
      named_barrier(kBarP2a, GT);  // every phase-2 thread has read the exchange slot
      if (t == 0 && ok && !*abort_flag)
        for (int cr = 0; cr < C; ++cr) mbar_arrive_remote(&S.xempty[s], (uint32_t)cr);
      __syncwarp();
      const float Mp = tot.pM, Lsp = log2f(tot.pS);
      const float Mq = tot.qM, Lsq = log2f(tot.qS);
      float smin = 0.f, sqlt = 0.f;
      float2 smin2 = make_float2(0.f, 0.f), sqlt2 = make_float2(0.f, 0.f);
      const float2 s2 = make_float2(a.sT, a.sT), negM = make_float2(-Mp, -Mq), negLs = make_float2(-Lsp, -Lsq);
      for (int c = c0; c < c1; ++c, pos.next()) {
        if (wait_phase<false>(&S.full[pos.slot], pos.phase, abort_flag, limit_ns, hdr)) {
          const int e0 = c * CH;
          const uint4* P = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes);
          const uint4* Q = reinterpret_cast<const uint4*>(ring + pos.slot * kSlotBytes + kHalfSlot);
          if (sizeof(T) == 2 && c < nfull) {
#pragma unroll
            for (int v = 0; v < NV; ++v) {
              const int i = t + v * GT;
              phase2_bf16x8(smin2, sqlt2, P[i], Q[i], s2, negM, negLs);
            }
          } else {
            const int nvec = min(CH, V - e0) / E;
            for (int i = t; i < nvec; i += GT) phase2_vec<T>(smin, sqlt, P[i], Q[i], a.sT, Mp, Lsp, Mq, Lsq);
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
      if (lane == 0) S.red2[j & 1][w] = make_float2(smin, sqlt);
      named_barrier(kBarP2b, GT);
      if (t == 0 && !*abort_flag) {
        float2 x = S.red2[j & 1][0];
        for (int k = 1; k < G; ++k) {
          x.x += S.red2[j & 1][k].x;
          x.y += S.red2[j & 1][k].y;
        }
        a.ws.cpart[r * kMaxCluster + rank] = x;
        if (rank == 0) {
          const float Mq1 = NEED_Q1 ? tot.q1M : Mq;
          const float Lsq1 = NEED_Q1 ? log2f(tot.q1S) : Lsq;
          a.ws.Mp[r] = Mp;
          a.ws.Lsp[r] = Lsp;
          a.ws.Mq[r] = Mq;
          a.ws.Lsq[r] = Lsq;
          a.ws.Mq1[r] = Mq1;
          a.ws.Lsq1[r] = Lsq1;
          a.ws.xstar[r] = tot.ai;
          a.ws.ag[r] = exp2f(log2_prob(tot.ac, kLog2e, Mq1, Lsq1));
        }
      }
      __syncwarp();
    }
  }
  __syncwarp();
  cluster_barrier();  // no CTA leaves while a peer may still touch its shared memory
}

constexpr size_t kSmemBytes = (size_t)kSlots * kSlotBytes + sizeof(Smem);

template <typename T, bool NEED_Q1>
cudaError_t launch_T(const RowStatsArgs& a, cudaStream_t s, int C, int m, int nch, uint64_t limit_ns,
                     bool* launched) {
  auto kern = rowstats_cluster<T, NEED_Q1, kGroupWarps>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.blockDim = dim3(32 * (1 + 2 * kGroupWarps));
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cfg.gridDim = dim3((unsigned)C);
  int max_clusters = 0;
  e = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
  if (e != cudaSuccess || max_clusters < 1) {
    cudaGetLastError();  // not launchable this way here: the caller uses the generic kernel
    *launched = false;
    return cudaSuccess;
  }
  int64_t ncl = max_clusters;
  if (ncl > a.R) ncl = a.R;
  cfg.gridDim = dim3((unsigned)(ncl * C));
  *launched = true;
  e = cudaLaunchKernelEx(&cfg, kern, a, C, m, nch, limit_ns);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

// Cluster width for a row of V elements of `elt` bytes: the smallest C whose per-CTA slice
// leaves kSlack ring slots free; 0 when even 8 CTAs cannot hold the row.
int rowstats_cluster_width(int64_t V, int elt, int* m_out, int* nch_out) {
  const int64_t CH = kHalfSlot / elt;
  const int64_t nch = (V + CH - 1) / CH;
  for (int C = 1; C <= kMaxCluster; C *= 2) {
    const int64_t m = (nch + C - 1) / C;
    if (m <= kSlots - kSlack) {
      *m_out = (int)m;
      *nch_out = (int)nch;
      return C;
    }
  }
  return 0;
}

cudaError_t launch_rowstats_cluster(const RowStatsArgs& a, bool bf16, cudaStream_t s, int C, int m, int nch,
                                    uint64_t limit_ns, bool* launched) {
  const bool q1 = a.need_q1;
  if (bf16) return q1 ? launch_T<uint16_t, true>(a, s, C, m, nch, limit_ns, launched)
                      : launch_T<uint16_t, false>(a, s, C, m, nch, limit_ns, launched);
  return q1 ? launch_T<float, true>(a, s, C, m, nch, limit_ns, launched)
            : launch_T<float, false>(a, s, C, m, nch, limit_ns, launched);
}

}  // namespace aal
