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
// first pass also folds D = sum_v e_v (z_p,v - z_q,v) next to the log-sum-exp of z_p.
//
// There is no cross-CTA communication, so all 152 SMs run one CTA each.  Every wait is
// bounded (ptx::wait_phase); after a timeout every thread keeps walking the same loops
// without waiting (a consumer still folds a chunk it finds landed, into results that are
// never written), so all meet the same named barriers, the producer drains its copies,
// and the kernel returns with AAL_ERR_TIMEOUT in the workspace status word.
#include "ptx.cuh"

namespace aal {
namespace {

using namespace ptx;

#ifndef AAL_STREAM_SLOTS
#define AAL_STREAM_SLOTS 4
#endif
#ifndef AAL_STREAM_SLOT_KB
#define AAL_STREAM_SLOT_KB 48
#endif
constexpr int kSlots = AAL_STREAM_SLOTS;               // ring slots
constexpr int kSlotBytes = AAL_STREAM_SLOT_KB * 1024;  // half z_p, half z_q
constexpr int kHalfSlot = kSlotBytes / 2;
constexpr int kVecPerChunk = kHalfSlot / 16;
#ifndef AAL_STREAM_WARPS
#define AAL_STREAM_WARPS 16
#endif
constexpr int kWarps = AAL_STREAM_WARPS;  // consumer warps
constexpr int kConsumers = 32 * kWarps;
constexpr int kThreads = 32 + kConsumers;
#ifndef AAL_STREAM_CTAS
#define AAL_STREAM_CTAS 1
#endif
constexpr int kCtasPerSm = AAL_STREAM_CTAS;  // resident CTAs per SM (each with its own ring)
constexpr int kNV = kVecPerChunk / kConsumers;  // 16-byte vectors per thread per full chunk
static_assert(kNV * kConsumers == kVecPerChunk, "consumers must tile a chunk");
constexpr int kBarRow = 1, kBarSum = 2;

// Phase-1 state of a thread, a warp or a row.  The target argmax is tracked per 16-byte
// vector (8 contiguous elements): av is the largest z_p seen and ab the first element index
// of the first vector that holds it.  Vectors are disjoint contiguous ranges, so the lowest
// ab among equal av contains the first occurrence; the position inside that vector is
// found in the second pass, by the one thread that streams the vector again.
struct RowPart {
  float pM, pS, qM, qS, q1M, q1S;  // online log2-sum-exp states (M = raw max of z)
  float pD;                        // KL anchor: sum 2^((z_p - pM) s) (z_p - z_q), rescaled with pS
  float av;                        // target: largest z_p and the first vector holding it
  int32_t ab;
  float qv;                        // draft: largest z_q and the first vector holding it
  int32_t qb;
};

struct Smem {
  uint64_t full[kSlots];
  uint64_t empty[kSlots];
  RowPart red[2][kWarps];  // by row parity
  float2 red2[2][kWarps];
  int32_t arg_index;  // x*, written by the thread that finds it in the second pass
  float arg_carry;    // z_q at x*
  int32_t yarg_index;  // the draft argmax, found the same way
  float yarg_carry;    // z_p there
  int abort_flag;
};

// Running maxima start at a finite floor far below any logit, so the online updates need
// no -inf special cases: a floor term contributes 2^(-huge) = 0.
constexpr float kMaxFloor = -1e30f;

__device__ __forceinline__ void part_init(RowPart& a) {
  a.pM = a.qM = a.q1M = kMaxFloor;
  a.pS = a.qS = a.q1S = 0.f;
  a.pD = 0.f;
  a.av = -INFINITY;
  a.ab = 0x7fffffff;
  a.qv = -INFINITY;
  a.qb = 0x7fffffff;
}

// Butterfly reductions over a warp: every lane ends with the same, order-fixed result.
__device__ __forceinline__ void warp_lse(float& M, float& S, float scale) {
  float m = M;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  float s = S * ex2((M - m) * scale);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  M = m;
  S = s;
}
__device__ __forceinline__ void warp_amax(float& v, int32_t& i) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, v, off);
    const int32_t i2 = __shfl_xor_sync(0xffffffffu, i, off);
    if (v2 > v || (v2 == v && i2 < i)) {
      v = v2;
      i = i2;
    }
  }
}
// (M, S, D): D rescales with S.
__device__ __forceinline__ void warp_lse_kl(float& M, float& S, float& D, float scale) {
  float m = M;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  const float r = ex2((M - m) * scale);
  float s = S * r, d = D * r;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, off);
    d += __shfl_xor_sync(0xffffffffu, d, off);
  }
  M = m;
  S = s;
  D = d;
}
template <bool NEED_Q1, bool KL = false>
__device__ __forceinline__ void warp_part(RowPart& a, float sT) {
  if (KL) warp_lse_kl(a.pM, a.pS, a.pD, sT);
  else warp_lse(a.pM, a.pS, sT);
  warp_lse(a.qM, a.qS, sT);
  if (NEED_Q1) warp_lse(a.q1M, a.q1S, kLog2e);
  warp_amax(a.av, a.ab);
  warp_amax(a.qv, a.qb);
}
// A vector's maximum beats the running one: remember it and where its vector starts.
__device__ __forceinline__ void amax_vec(float& best, int32_t& at, float vmax, int base) {
  const bool take = vmax > best;
  best = take ? vmax : best;
  at = take ? base : at;
}

// ---------------------------------------------------------------- per-chunk arithmetic

// Fold NW bf16 words (2 NW values) of one tensor into (M, S); vmax is their maximum.
// Each value costs one mixed-precision add (z - M, the bf16 widened inside the add), half
// a packed multiply by s, one ex2 and half a packed add.
template <int NW>
__device__ __forceinline__ void lse_words(float& M, float& S, const uint32_t* w, float vmax, float s) {
  const float m = fmaxf(M, vmax);  // branch-free: rescale by 2^((M - m) s), 1 when unchanged
  S *= ex2((M - m) * s);
  M = m;
  const float nM = -M;
  const float2 s2 = make_float2(s, s), zero2 = make_float2(0.f, 0.f);
  float2 acc0 = zero2, acc1 = zero2;
#pragma unroll
  for (int k = 0; k < NW; ++k) {
    const float2 x = f2fma(make_float2(bf16lo_add(w[k], nM), bf16hi_add(w[k], nM)), s2, zero2);
    const float2 e = make_float2(ex2(x.x), ex2(x.y));
    if (k & 1) acc1 = f2add(acc1, e);
    else acc0 = f2add(acc0, e);
  }
  const float2 t = f2add(acc0, acc1);
  S += t.x + t.y;
}

// lse_words for z_p with the KL sum: D += 2^((z_p - M) s) (z_p - z_q), rescaled with S.
template <int NW>
__device__ __forceinline__ void lse_kl_words(float& M, float& S, float& D, const uint32_t* pw,
                                             const uint32_t* qw, float vmax, float s) {
  const float m = fmaxf(M, vmax);
  const float r = ex2((M - m) * s);
  S *= r;
  D *= r;
  M = m;
  const float nM = -M;
  const float2 s2 = make_float2(s, s), zero2 = make_float2(0.f, 0.f);
  float2 acc = zero2, dacc = zero2;
#pragma unroll
  for (int k = 0; k < NW; ++k) {
    const float2 x = f2fma(make_float2(bf16lo_add(pw[k], nM), bf16hi_add(pw[k], nM)), s2, zero2);
    const float2 e = make_float2(ex2(x.x), ex2(x.y));
    acc = f2add(acc, e);
    // z_p - z_q: the draft value widened, the target's bf16 widened inside the add
    const float2 d = make_float2(bf16lo_add(pw[k], -bf16_lo(qw[k])), bf16hi_add(pw[k], -bf16_hi(qw[k])));
    dacc = f2fma(e, d, dacc);
  }
  S += acc.x + acc.y;
  D += dacc.x + dacc.y;
}

// The first of a thread's NV vectors whose maximum (vm[v], packed bf16 pair) equals m:
// the running argmax moves there.  Called only when m beats the running maximum, which
// after the first chunks of a row is rare.
template <int NV>
__device__ __forceinline__ void first_vec_at(float& best, int32_t& at, const uint32_t* vm, float m, int idx0,
                                             int vstride) {
  int v0 = NV - 1;
#pragma unroll
  for (int v = NV - 2; v >= 0; --v)
    if (fmaxf(bf16_lo(vm[v]), bf16_hi(vm[v])) == m) v0 = v;
  best = m;
  at = idx0 + v0 * vstride;
}

// Phase 1 on NV 16-byte vectors of bf16 per tensor; vector v holds elements
// idx0 + v * vstride + [0, 8).  The maxima are taken on packed bf16 pairs: per vector, then
// over the thread's vectors; only a maximum that beats the running one looks for its vector
// (the first in element order, as a strict per-vector update in that order would).
template <int NV, bool NEED_Q1, bool KL = false>
__device__ __forceinline__ void phase1_bf16(RowPart& A, const uint4* pv, const uint4* qv, int idx0, int vstride,
                                            float sT) {
  constexpr int NW = 4 * NV;
  uint32_t pw[NW], qw[NW];
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    pw[4 * v + 0] = pv[v].x;
    pw[4 * v + 1] = pv[v].y;
    pw[4 * v + 2] = pv[v].z;
    pw[4 * v + 3] = pv[v].w;
    qw[4 * v + 0] = qv[v].x;
    qw[4 * v + 1] = qv[v].y;
    qw[4 * v + 2] = qv[v].z;
    qw[4 * v + 3] = qv[v].w;
  }
  uint32_t vp[NV], vq[NV];
#pragma unroll
  for (int v = 0; v < NV; ++v) {  // per-vector maxima of z_p and z_q, packed
    vp[v] = bmax2(bmax2(pw[4 * v], pw[4 * v + 1]), bmax2(pw[4 * v + 2], pw[4 * v + 3]));
    vq[v] = bmax2(bmax2(qw[4 * v], qw[4 * v + 1]), bmax2(qw[4 * v + 2], qw[4 * v + 3]));
  }
  uint32_t cp = vp[0], cq = vq[0];
#pragma unroll
  for (int v = 1; v < NV; ++v) {
    cp = bmax2(cp, vp[v]);
    cq = bmax2(cq, vq[v]);
  }
  const float pm = fmaxf(bf16_lo(cp), bf16_hi(cp)), qm = fmaxf(bf16_lo(cq), bf16_hi(cq));
  if (pm > A.av) first_vec_at<NV>(A.av, A.ab, vp, pm, idx0, vstride);
  if (qm > A.qv) first_vec_at<NV>(A.qv, A.qb, vq, qm, idx0, vstride);
  if (KL) lse_kl_words<NW>(A.pM, A.pS, A.pD, pw, qw, pm, sT);
  else lse_words<NW>(A.pM, A.pS, pw, pm, sT);
  lse_words<NW>(A.qM, A.qS, qw, qm, sT);
  if (NEED_Q1) lse_words<NW>(A.q1M, A.q1S, qw, qm, kLog2e);
}

// Phase 2 on one 16-byte vector of bf16 per tensor.  With C = M + Ls/s, log2 p~ = (z - C) s;
// since s > 0 the min and the comparison are taken on u = z - C (one mixed-precision add
// each) and only the min is scaled.
__device__ __forceinline__ void phase2_bf16(float2& smin2, float2& sqlt2, const uint4& pw, const uint4& qw,
                                            float s, float nCp, float nCq) {
  const uint32_t pa[4] = {pw.x, pw.y, pw.z, pw.w};
  const uint32_t qa[4] = {qw.x, qw.y, qw.z, qw.w};
  const float2 s2 = make_float2(s, s), zero2 = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float up0 = bf16lo_add(pa[k], nCp), up1 = bf16hi_add(pa[k], nCp);
    const float uq0 = bf16lo_add(qa[k], nCq), uq1 = bf16hi_add(qa[k], nCq);
    const float2 x = f2fma(make_float2(fminf(up0, uq0), fminf(up1, uq1)), s2, zero2);
    const float2 e = make_float2(ex2(x.x), ex2(x.y));
    smin2 = f2add(smin2, e);
    sqlt2 = f2fma(e, make_float2(set_lt(uq0, up0), set_lt(uq1, up1)), sqlt2);
  }
}

// The first element of a 16-byte vector equal to `target` (the row's max of z_p), with
// the z_q value at the same position.
template <typename T>
__device__ __forceinline__ void find_first(const uint4& pw, const uint4& qw, float target, int* at, float* carry);

// Scalar element paths (fp32 rows, and the partial last chunk of a bf16 row).
template <typename T>
__device__ __forceinline__ void unpack_vec(const uint4& w, float* o);
template <>
__device__ __forceinline__ void unpack_vec<uint16_t>(const uint4& w, float* o) {
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
__device__ __forceinline__ void unpack_vec<float>(const uint4& w, float* o) {
  o[0] = __uint_as_float(w.x);
  o[1] = __uint_as_float(w.y);
  o[2] = __uint_as_float(w.z);
  o[3] = __uint_as_float(w.w);
}

template <typename T>
__device__ __forceinline__ void find_first(const uint4& pw, const uint4& qw, float target, int* at, float* carry) {
  constexpr int E = 16 / sizeof(T);
  float pv[8], qv[8];
  unpack_vec<T>(pw, pv);
  unpack_vec<T>(qw, qv);
  int e = 0;
  float c = qv[0];
#pragma unroll
  for (int k = E - 1; k >= 0; --k) {
    if (pv[k] == target) {
      e = k;
      c = qv[k];
    }
  }
  *at = e;
  *carry = c;
}

template <int N>
__device__ __forceinline__ void lse_vals(float& M, float& S, const float* v, float vmax, float s) {
  const float m = fmaxf(M, vmax);
  S *= ex2((M - m) * s);
  M = m;
  float acc = 0.f;
#pragma unroll
  for (int e = 0; e < N; ++e) acc += ex2((v[e] - M) * s);
  S += acc;
}

template <int N>
__device__ __forceinline__ void lse_kl_vals(float& M, float& S, float& D, const float* p, const float* q,
                                            float vmax, float s) {
  const float m = fmaxf(M, vmax);
  const float r = ex2((M - m) * s);
  S *= r;
  D *= r;
  M = m;
  float acc = 0.f, dacc = 0.f;
#pragma unroll
  for (int e = 0; e < N; ++e) {
    const float x = ex2((p[e] - M) * s);
    acc += x;
    dacc = fmaf(x, p[e] - q[e], dacc);
  }
  S += acc;
  D += dacc;
}

template <typename T, bool NEED_Q1, bool KL = false>
__device__ __forceinline__ void phase1_vec(RowPart& A, const uint4& pw, const uint4& qw, int idx0, float sT) {
  constexpr int E = 16 / sizeof(T);
  float pv[8], qv[8];
  unpack_vec<T>(pw, pv);
  unpack_vec<T>(qw, qv);
  float pm = pv[0], qm = qv[0];
#pragma unroll
  for (int e = 1; e < E; ++e) {
    pm = fmaxf(pm, pv[e]);
    qm = fmaxf(qm, qv[e]);
  }
  amax_vec(A.av, A.ab, pm, idx0);
  amax_vec(A.qv, A.qb, qm, idx0);
  if (KL) lse_kl_vals<E>(A.pM, A.pS, A.pD, pv, qv, pm, sT);
  else lse_vals<E>(A.pM, A.pS, pv, pm, sT);
  lse_vals<E>(A.qM, A.qS, qv, qm, sT);
  if (NEED_Q1) lse_vals<E>(A.q1M, A.q1S, qv, qm, kLog2e);
}

template <typename T>
__device__ __forceinline__ void phase2_vec(float& smin, float& sqlt, const uint4& pw, const uint4& qw, float sT,
                                           float nCp, float nCq) {
  constexpr int E = 16 / sizeof(T);
  float pv[8], qv[8];
  unpack_vec<T>(pw, pv);
  unpack_vec<T>(qw, qv);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const float up = pv[e] + nCp, uq = qv[e] + nCq;
    const float t = ex2(fminf(up, uq) * sT);
    smin += t;
    sqlt += (uq < up) ? t : 0.f;
  }
}

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

// ---------------------------------------------------------------- the kernel

// PASSES = 2: the sampling term (normalisers at T, then the overlap sums).  PASSES = 1: no
// sampling term; everything at T = 1 (sT is log2 e), argmaxes resolved by resolve_argmax.
// KL: the anchor's D next to the z_p normaliser (which must then be at T = 1).
template <typename T, bool NEED_Q1, int PASSES, bool KL>
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
    const float sT = PASSES == 2 ? a.sT : kLog2e;
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
            phase1_bf16<kNV, NEED_Q1, KL>(A, pv, qv, e0 + t * E, kConsumers * E, sT);
          } else {
            const int nvec = min(CH, V - e0) / E;
            for (int i = t; i < nvec; i += kConsumers) {
              if (sizeof(T) == 2) phase1_bf16<1, NEED_Q1, KL>(A, P + i, Q + i, e0 + i * E, 0, sT);
              else phase1_vec<T, NEED_Q1, KL>(A, P[i], Q[i], e0 + i * E, sT);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[pos.slot]);
      }
      warp_part<NEED_Q1, KL>(A, sT);
      if (lane == 0) S.red[j & 1][warp] = A;
      named_barrier(kBarRow, kConsumers);
      // every warp combines the warp partials itself (lanes >= kWarps carry the identity)
      RowPart tot;
      if (lane < kWarps) tot = S.red[j & 1][lane];
      else part_init(tot);
      warp_part<NEED_Q1, KL>(tot, sT);
      const float Mp = tot.pM, Lsp = log2f(tot.pS);
      const float Mq = tot.qM, Lsq = log2f(tot.qS);
      if (KL && t == 0 && !*abort_flag) {  // both normalisers are at T = 1 here
        const float Mq1 = NEED_Q1 ? tot.q1M : Mq;
        const float Lsq1 = NEED_Q1 ? log2f(tot.q1S) : Lsq;
        a.ws.Mp1[r] = Mp;
        a.ws.Lsp1[r] = Lsp;
        a.ws.kl[r] = tot.pD / tot.pS - (Mp - Mq1) - kLn2 * (Lsp - Lsq1);
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

template <typename T, bool NEED_Q1, int PASSES, bool KL>
cudaError_t launch_T(const RowStatsArgs& a, cudaStream_t s, int nch, uint64_t limit_ns) {
  auto kern = rowstats_stream<T, NEED_Q1, PASSES, KL>;
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
  constexpr int E = 16 / sizeof(T);
  const T* zp = static_cast<const T*>(a.zp) + r * a.V;
  const T* zq = static_cast<const T*>(a.zq) + r * a.V;
  const int32_t xb = a.ws.xstar[r], yb = a.ws.yhat[r];
  int32_t xs = 0, ys = 0;
  float cx = 0.f, cy = 0.f;
  // a vector is read only at an in-range, vector-aligned start (an all -inf row, or a row
  // of an aborted launch, records none)
  if (xb >= 0 && xb % E == 0 && (int64_t)xb + E <= a.V) {
    const uint4 pw = *reinterpret_cast<const uint4*>(zp + xb), qw = *reinterpret_cast<const uint4*>(zq + xb);
    float pv[8], qv[8];
    unpack_vec<T>(pw, pv);
    unpack_vec<T>(qw, qv);
    float m = pv[0];
    for (int e = 1; e < E; ++e) m = fmaxf(m, pv[e]);
    int at = 0;
    for (int e = E - 1; e >= 0; --e)
      if (pv[e] == m) at = e;
    xs = xb + at;
    cx = qv[at];
  }
  if (yb >= 0 && yb % E == 0 && (int64_t)yb + E <= a.V) {
    const uint4 pw = *reinterpret_cast<const uint4*>(zp + yb), qw = *reinterpret_cast<const uint4*>(zq + yb);
    float pv[8], qv[8];
    unpack_vec<T>(pw, pv);
    unpack_vec<T>(qw, qv);
    float m = qv[0];
    for (int e = 1; e < E; ++e) m = fmaxf(m, qv[e]);
    int at = 0;
    for (int e = E - 1; e >= 0; --e)
      if (qv[e] == m) at = e;
    ys = yb + at;
    cy = pv[at];
  }
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
  if (a.need_kl) return launch_T<T, false, 2, true>(a, s, nch, limit_ns);  // T = 1: no separate q1
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

}  // namespace aal
