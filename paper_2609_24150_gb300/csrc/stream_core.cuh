// Shared pieces of the TMA-streamed row kernels (rowstats_stream.cu: the forward statistics;
// fused.cu: the forward and backward in one pass over each window): the ring geometry, the
// per-thread statistics state, the packed per-chunk arithmetic of both passes, and the CTA
// reductions.  Everything is internal linkage; each kernel file includes it once.
#pragma once

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
  float p1M, p1S;                  // KL anchor beside an overlap at T != 1 (P1): z_p at T = 1,
                                   // and pD then rescales with p1S
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
  a.pM = a.qM = a.q1M = a.p1M = kMaxFloor;
  a.pS = a.qS = a.q1S = a.p1S = 0.f;
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
template <bool NEED_Q1, bool KL = false, bool P1 = false>
__device__ __forceinline__ void warp_part(RowPart& a, float sT) {
  if (KL && P1) {
    warp_lse(a.pM, a.pS, sT);
    warp_lse_kl(a.p1M, a.p1S, a.pD, kLog2e);
  } else if (KL) {
    warp_lse_kl(a.pM, a.pS, a.pD, sT);
  } else {
    warp_lse(a.pM, a.pS, sT);
  }
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
template <int NV, bool NEED_Q1, bool KL = false, bool P1 = false>
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
  if (KL && P1) {
    lse_words<NW>(A.pM, A.pS, pw, pm, sT);
    lse_kl_words<NW>(A.p1M, A.p1S, A.pD, pw, qw, pm, kLog2e);
  } else if (KL) {
    lse_kl_words<NW>(A.pM, A.pS, A.pD, pw, qw, pm, sT);
  } else {
    lse_words<NW>(A.pM, A.pS, pw, pm, sT);
  }
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

template <typename T, bool NEED_Q1, bool KL = false, bool P1 = false>
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
  if (KL && P1) {
    lse_vals<E>(A.pM, A.pS, pv, pm, sT);
    lse_kl_vals<E>(A.p1M, A.p1S, A.pD, pv, qv, pm, kLog2e);
  } else if (KL) {
    lse_kl_vals<E>(A.pM, A.pS, A.pD, pv, qv, pm, sT);
  } else {
    lse_vals<E>(A.pM, A.pS, pv, pm, sT);
  }
  lse_vals<E>(A.qM, A.qS, qv, qm, sT);
  if (NEED_Q1) lse_vals<E>(A.q1M, A.q1S, qv, qm, kLog2e);
}

// The anchor's row statistics from a row's reduced state (Mp, Lsp: z_p's normaliser at the
// pass's temperature; Mq, Lsq: z_q's): z_p's normaliser at T = 1, kept apart when the
// overlap runs at T != 1 (P1), and KL(p || q) = D / S_p - (Mp1 - Mq1) - ln 2 (Lsp1 - Lsq1)
// in nats, with q's normaliser at T = 1.
template <bool NEED_Q1, bool P1>
__device__ __forceinline__ void kl_stats(const RowPart& tot, float Mp, float Lsp, float Mq, float Lsq, float& Mp1,
                                         float& Lsp1, float& kl) {
  const float Mq1 = NEED_Q1 ? tot.q1M : Mq;
  const float Lsq1 = NEED_Q1 ? log2f(tot.q1S) : Lsq;
  Mp1 = P1 ? tot.p1M : Mp;
  Lsp1 = P1 ? log2f(tot.p1S) : Lsp;
  kl = tot.pD / (P1 ? tot.p1S : tot.pS) - (Mp1 - Mq1) - kLn2 * (Lsp1 - Lsq1);
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

// The exact argmaxes inside the 16-byte vectors a one-pass scan recorded: x* = the first
// element of z_p's vector at xb equal to its maximum, with z_q there (cx), and y = the same for
// z_q's vector at yb, with z_p there (cy).  A vector is read only at an in-range,
// vector-aligned start (an all -inf row, or a row of an aborted launch, records none: index 0).
template <typename T>
__device__ __forceinline__ void resolve_vectors(const T* zp, const T* zq, int64_t V, int32_t xb, int32_t yb,
                                                int32_t* xs, float* cx, int32_t* ys, float* cy) {
  constexpr int E = 16 / sizeof(T);
  *xs = 0;
  *ys = 0;
  *cx = 0.f;
  *cy = 0.f;
  if (xb >= 0 && xb % E == 0 && (int64_t)xb + E <= V) {
    const uint4 pw = *reinterpret_cast<const uint4*>(zp + xb), qw = *reinterpret_cast<const uint4*>(zq + xb);
    float pv[8], qv[8];
    unpack_vec<T>(pw, pv);
    unpack_vec<T>(qw, qv);
    float m = pv[0];
    for (int e = 1; e < E; ++e) m = fmaxf(m, pv[e]);
    int at = 0;
    for (int e = E - 1; e >= 0; --e)
      if (pv[e] == m) at = e;
    *xs = xb + at;
    *cx = qv[at];
  }
  if (yb >= 0 && yb % E == 0 && (int64_t)yb + E <= V) {
    const uint4 pw = *reinterpret_cast<const uint4*>(zp + yb), qw = *reinterpret_cast<const uint4*>(zq + yb);
    float pv[8], qv[8];
    unpack_vec<T>(pw, pv);
    unpack_vec<T>(qw, qv);
    float m = qv[0];
    for (int e = 1; e < E; ++e) m = fmaxf(m, qv[e]);
    int at = 0;
    for (int e = E - 1; e >= 0; --e)
      if (qv[e] == m) at = e;
    *ys = yb + at;
    *cy = pv[at];
  }
}

}  // namespace
}  // namespace aal
