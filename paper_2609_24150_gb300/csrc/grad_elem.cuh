// Per-element gradient of the EAL / WTV losses (and the KL anchor and GRPO terms) with
// respect to the draft logits, shared by the backward kernel (backward.cu) and the fused
// forward + backward (rowstats_stream.cu), so that both write bitwise the same gradient.
//
// For row r = (n, j) with g^g = -(dloss/|W|) w_g dE^g_n/da^g_{n,j} and
// g^s = -(dloss/|W|) dE^s_n/da^s_{n,j} (w_s and w_tv already folded into dE^s/da):
//   dz_u = g^g a^g (delta_{u,x*} - q(u))                 greedy term, Eq. acc_greedy
//        + g^s (1/T) q~(u) (c_u - Qlt),  c_u = [q~_u < p~_u]   sampling term, Eq. acc_sample
//        + c^kl (q(u) - p(u))                                  KL anchor (Sec. 4.1), T = 1
//        + c^grpo (delta_{u,y} - q(u))                         GRPO surrogate (Sec. 3.4)
// (the softmax Jacobian applied to d a / d q; at a tie q~_u = p~_u the min follows the
// frozen p~, so c_u = 0).
#pragma once

#include "aal_internal.cuh"
#include "ptx.cuh"

namespace aal {

template <typename T>
struct Io;

template <>
struct Io<float> {
  static constexpr int E = 4;
  __device__ static void unpack(const uint4& w, float* o) {
    o[0] = __uint_as_float(w.x);
    o[1] = __uint_as_float(w.y);
    o[2] = __uint_as_float(w.z);
    o[3] = __uint_as_float(w.w);
  }
  __device__ static uint4 pack(const float* d) {
    return make_uint4(__float_as_uint(d[0]), __float_as_uint(d[1]), __float_as_uint(d[2]),
                      __float_as_uint(d[3]));
  }
  __device__ static void store1(float* p, float d) { *p = d; }
};

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

template <>
struct Io<uint16_t> {
  static constexpr int E = 8;
  __device__ static void unpack(const uint4& w, float* o) {
    o[0] = bf16_lo(w.x);
    o[1] = bf16_hi(w.x);
    o[2] = bf16_lo(w.y);
    o[3] = bf16_hi(w.y);
    o[4] = bf16_lo(w.z);
    o[5] = bf16_hi(w.z);
    o[6] = bf16_lo(w.w);
    o[7] = bf16_hi(w.w);
  }
  __device__ static uint4 pack(const float* d) {
    return make_uint4(pack_bf16x2(d[0], d[1]), pack_bf16x2(d[2], d[3]), pack_bf16x2(d[4], d[5]),
                      pack_bf16x2(d[6], d[7]));
  }
  __device__ static void store1(uint16_t* p, float d) {
    *p = (uint16_t)(pack_bf16x2(d, 0.f) & 0xffffu);
  }
};

// 16-byte streaming store (evict-first): gradient rows are written once and not re-read.
__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

// log2 q~_u = (z_q,u + nCq) s and log2 p~_u = (z_p,u + nCp) s with nC = -(M + Ls / s): the
// same per-row constants, and the same comparison c_u = [z_q,u + nCq < z_p,u + nCp], as the
// forward's overlap pass, so the gradient's c_u is the one the forward's Qlt summed over.
// nCq1, nCp1: the same at T = 1 (s = log2 e) for q and p.
struct RowCoef {
  float sT, nCq, nCp, nCq1, nCp1;
  float Ck;          // c^kl
  float cpos, cneg;  // g^s/T (1 - Qlt) and -g^s/T Qlt
  float Ag;          // g^g a^g
  float Cg;          // c^grpo
  float Aq;          // Ag + Cg, the coefficient of -q(u)
  float q1c;         // Ck - Aq: the coefficient of q(u) in every term but the sampling one
  float cposq, cnegq;  // cpos + q1c, cneg + q1c: with q = q~ (T = 1) the element's whole q~ factor
  int32_t xs, ys;
};

// What a row's coefficient needs from its forward statistics.
struct RowStat {
  float Mq, Lsq, Mp, Lsp, Mq1, Lsq1, Mp1, Lsp1;
  float qlt, ag;
  int32_t xs, ys;
};

// The statistics the instantiation reads, from the workspace (the rest stay 0).
template <bool GREEDY, bool SAMPLING, bool KL>
__device__ __forceinline__ RowStat load_row_stat(const LossWs& ws, int64_t r, bool with_greedy, bool with_grpo) {
  RowStat st{};
  if (SAMPLING) {
    st.Mq = ws.Mq[r];
    st.Lsq = ws.Lsq[r];
    st.Mp = ws.Mp[r];
    st.Lsp = ws.Lsp[r];
    st.qlt = ws.qlt[r];
  }
  if (GREEDY || KL) {
    st.Mq1 = ws.Mq1[r];
    st.Lsq1 = ws.Lsq1[r];
  }
  if (KL) {
    st.Mp1 = ws.Mp1[r];
    st.Lsp1 = ws.Lsp1[r];
  }
  if (GREEDY && with_greedy) {
    st.ag = ws.ag[r];
    st.xs = ws.xstar[r];
  }
  if (GREEDY && with_grpo) st.ys = ws.yhat[r];
  return st;
}

// The row-local part of the coefficients: the offsets nC = -(M + Ls / s) of q~, p~ (at T) and of
// q, p (at T = 1), from the row's own statistics (no window term), each rounding spelled out.
template <bool GREEDY, bool SAMPLING, bool KL>
__device__ __forceinline__ void row_coef_local(const BackwardArgs& a, const RowStat& st, RowCoef& c) {
  c.sT = a.sT;
  c.nCq = SAMPLING ? -__fadd_rn(st.Mq, __fdiv_rn(st.Lsq, a.sT)) : 0.f;
  c.nCp = SAMPLING ? -__fadd_rn(st.Mp, __fdiv_rn(st.Lsp, a.sT)) : 0.f;
  c.nCq1 = (GREEDY || KL) ? -__fadd_rn(st.Mq1, __fdiv_rn(st.Lsq1, kLog2e)) : 0.f;
  c.nCp1 = KL ? -__fadd_rn(st.Mp1, __fdiv_rn(st.Lsp1, kLog2e)) : 0.f;
}

// The row's coefficients from its statistics, dE^g/da (unweighted), dE^s/da (weights folded),
// the GRPO coefficient and whether the row is a valid position (the anchor's rows).  Returns
// false when every term of the row is zero (the row's gradient is all zeros).  LOCAL_DONE: the
// caller already formed the row-local part with row_coef_local (the same values).
template <bool GREEDY, bool SAMPLING, bool KL, bool LOCAL_DONE = false>
__device__ __forceinline__ bool row_coef(const BackwardArgs& a, float scale, float kscale, float dEg, float dEs,
                                         float cgr, bool pos_valid, const RowStat& st, RowCoef& c) {
  // every rounding spelled out (no contraction into fused multiply-adds), so that each kernel
  // that includes this forms the same bits
  const float gg = (GREEDY && a.w_greedy != 0.f) ? __fmul_rn(__fmul_rn(scale, a.w_greedy), dEg) : 0.f;
  const float cg = (GREEDY && a.grpo) ? __fmul_rn(a.dloss, cgr) : 0.f;
  const float gs = SAMPLING ? __fmul_rn(__fmul_rn(scale, a.w_sampling), dEs) : 0.f;
  const float ck = (KL && pos_valid) ? kscale : 0.f;
  if (gg == 0.f && gs == 0.f && ck == 0.f && cg == 0.f) return false;
  if (!LOCAL_DONE) row_coef_local<GREEDY, SAMPLING, KL>(a, st, c);
  c.Ck = ck;
  const float qlt = SAMPLING ? st.qlt : 0.f;
  const float Bs = __fmul_rn(gs, a.invT);
  c.cpos = __fmul_rn(Bs, __fsub_rn(1.f, qlt));
  c.cneg = -__fmul_rn(Bs, qlt);
  c.Ag = gg != 0.f ? __fmul_rn(gg, st.ag) : 0.f;
  c.Cg = cg;
  c.Aq = __fadd_rn(c.Ag, c.Cg);
  c.q1c = __fsub_rn(c.Ck, c.Aq);
  c.cposq = __fadd_rn(c.cpos, c.q1c);
  c.cnegq = __fadd_rn(c.cneg, c.q1c);
  c.xs = gg != 0.f ? st.xs : -1;
  c.ys = cg != 0.f ? st.ys : -1;
  return true;
}

// Every term of element u except the greedy and GRPO spikes (+Ag at x*, +Cg at y), which
// the callers add: once per 16-byte vector in the vector paths, per element in the scalar one.
// (On the element's logits widened to fp32: the vector path below reaches the same values with
// the bf16 widened inside the adds.)
// The terms are grouped by exponential: q~(u) (c_u ? cpos : cneg) + q(u) (Ck - Aq) - Ck p(u),
// and with q = q~ the first two share one factor, q~(u) (c_u ? cposq : cnegq).
template <bool GREEDY, bool SAMPLING, bool Q1_IS_QT, bool KL>
__device__ __forceinline__ float grad_elem(const RowCoef& c, float q, float p) {
  float d = 0.f;
  if (SAMPLING) {
    const float uq = q + c.nCq, up = p + c.nCp;
    const float qt = ex2(uq * c.sT);
    if (Q1_IS_QT) d = qt * (uq < up ? c.cposq : c.cnegq);
    else d = qt * (uq < up ? c.cpos : c.cneg);
  }
  if ((GREEDY || KL) && !(SAMPLING && Q1_IS_QT)) d = fmaf(ex2((q + c.nCq1) * kLog2e), c.q1c, d);
  if (KL) d = fmaf(ex2((p + c.nCp1) * kLog2e), -c.Ck, d);
  return d;
}

// grad_elem on the two bf16 halves of a word of z_q (qw) and of z_p (pw): each widened inside
// a mixed-precision add, the products and sums on fp32 pairs.  The same values as grad_elem on
// the widened logits (the widening is exact and every product or fused add is one rounding
// either way), up to the sign of an exact zero.
template <bool GREEDY, bool SAMPLING, bool Q1_IS_QT, bool KL>
__device__ __forceinline__ float2 grad_pair_bf16(const RowCoef& c, uint32_t qw, uint32_t pw) {
  const float2 zero2 = make_float2(0.f, 0.f), l2e2 = make_float2(kLog2e, kLog2e);
  float2 d = zero2;
  if (SAMPLING) {
    const float uq0 = bf16lo_add(qw, c.nCq), uq1 = bf16hi_add(qw, c.nCq);
    const float up0 = bf16lo_add(pw, c.nCp), up1 = bf16hi_add(pw, c.nCp);
    const float2 x = ptx::f2fma(make_float2(uq0, uq1), make_float2(c.sT, c.sT), zero2);
    const float2 qt = make_float2(ex2(x.x), ex2(x.y));
    const float a = Q1_IS_QT ? c.cposq : c.cpos, b = Q1_IS_QT ? c.cnegq : c.cneg;
    d = ptx::f2fma(qt, make_float2(uq0 < up0 ? a : b, uq1 < up1 ? a : b), zero2);
  }
  if ((GREEDY || KL) && !(SAMPLING && Q1_IS_QT)) {
    const float2 x = ptx::f2fma(make_float2(bf16lo_add(qw, c.nCq1), bf16hi_add(qw, c.nCq1)), l2e2, zero2);
    d = ptx::f2fma(make_float2(ex2(x.x), ex2(x.y)), make_float2(c.q1c, c.q1c), d);
  }
  if (KL) {
    const float2 x = ptx::f2fma(make_float2(bf16lo_add(pw, c.nCp1), bf16hi_add(pw, c.nCp1)), l2e2, zero2);
    d = ptx::f2fma(make_float2(ex2(x.x), ex2(x.y)), make_float2(-c.Ck, -c.Ck), d);
  }
  return d;
}

// One 16-byte vector of gradient (elements i*E ..): the terms, the spikes at x* and y when
// they fall in it, packed in the logits' dtype.
template <typename T, bool GREEDY, bool SAMPLING, bool Q1_IS_QT, bool KL>
__device__ __forceinline__ uint4 grad_vec(const RowCoef& c, const uint4& qw, const uint4& pw, int64_t i,
                                          int64_t xv, int xe, int64_t yv, int ye) {
  constexpr int E = Io<T>::E;
  constexpr bool READ_P = SAMPLING || KL;
  float d[E];
  if constexpr (sizeof(T) == 2) {
    const uint32_t qa[4] = {qw.x, qw.y, qw.z, qw.w};
    const uint32_t pa[4] = {pw.x, pw.y, pw.z, pw.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 dd = grad_pair_bf16<GREEDY, SAMPLING, Q1_IS_QT, KL>(c, qa[k], READ_P ? pa[k] : 0u);
      d[2 * k] = dd.x;
      d[2 * k + 1] = dd.y;
    }
  } else {
    float qv[E], pv[E];
    Io<T>::unpack(qw, qv);
    if (READ_P) Io<T>::unpack(pw, pv);
#pragma unroll
    for (int e = 0; e < E; ++e) d[e] = grad_elem<GREEDY, SAMPLING, Q1_IS_QT, KL>(c, qv[e], READ_P ? pv[e] : 0.f);
  }
  if (GREEDY) {  // the spikes, tested once per vector
    if (i == xv) {
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (e == xe) d[e] += c.Ag;
    }
    if (i == yv) {
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (e == ye) d[e] += c.Cg;
    }
  }
  return Io<T>::pack(d);
}

// The window exchange of the fused forward + backward, run by one whole warp: lane 0 publishes
// this row's (a^greedy, a^sample) as one 64-bit word in the per-row mailbox (preset to
// kMboxEmpty, so the word is its own ready flag), then lane j polls the word of depth j of the
// window (rows r0 .. r0 + K - 1) until none is empty, bounded like the ring waits.  When `need`
// is false (no window term) nothing is polled.  Returns, to every lane, whether the window's
// words arrived; on lane 0, ag[j] and as[j] hold depth j's values (0 beyond K).  The abort flag
// is read once for the warp (another warp may raise it meanwhile).
struct NoPrePoll {
  __device__ void operator()() const {}
};

// This row's mailbox word: (a^greedy, a^sample) as one 64-bit value, never the empty sentinel.
__device__ __forceinline__ uint64_t mbox_word(float ag_r, float as_r) {
  uint64_t word = ((uint64_t)__float_as_uint(as_r) << 32) | __float_as_uint(ag_r);
  return word == kMboxEmpty ? 0 : word;  // (bit patterns no arithmetic yields; never sent)
}

// `publish`: lane 0 writes this row's word first (false when the caller has already written it);
// `pre`: run by lane 0 before the window's words are polled, while the first poll is in flight.
template <typename Pre = NoPrePoll>
__device__ __forceinline__ bool window_exchange(uint64_t* mbox, int64_t r, int64_t r0, int K, int lane, float ag_r,
                                                float as_r, bool need, volatile int* abort_flag, WsHeader* hdr,
                                                uint64_t limit_ns, float* ag, float* as, bool publish = true,
                                                Pre pre = Pre()) {
  if (lane == 0 && publish) ptx::st_relaxed(&mbox[r], mbox_word(ag_r, as_r));
  bool ok = __shfl_sync(0xffffffffu, *abort_flag == 0 ? 1 : 0, 0) != 0;
  uint64_t w = 0;
  if (lane == 0 && !(ok && need)) pre();  // nothing to poll: the caller's work runs now
  if (ok && need) {
    const uint64_t t0 = ptx::now_ns();
    for (uint32_t it = 0;; ++it) {
      if (lane < K) w = ptx::ld_relaxed(&mbox[r0 + lane]);
      if (it == 0 && lane == 0) pre();
      if (__all_sync(0xffffffffu, lane >= K || w != kMboxEmpty)) break;
      int quit = 0;  // lane 0 decides for the warp whether to give up
      if (lane == 0 && (*abort_flag || it >= kSpinLimit || ptx::now_ns() - t0 > limit_ns)) {
        if (!*abort_flag) {
          *abort_flag = 1;
          atomicExch(&hdr->status, kStatusTimeout);
        }
        quit = 1;
      }
      if (__shfl_sync(0xffffffffu, quit, 0)) {
        ok = false;
        break;
      }
      __nanosleep(64);
    }
  }
#pragma unroll
  for (int jj = 0; jj < AAL_MAX_K; ++jj) {
    const float g_ = __shfl_sync(0xffffffffu, __uint_as_float((uint32_t)w), jj);
    const float s_ = __shfl_sync(0xffffffffu, __uint_as_float((uint32_t)(w >> 32)), jj);
    ag[jj] = (jj < K && need) ? g_ : 0.f;
    as[jj] = (jj < K && need) ? s_ : 0.f;
  }
  return ok;
}


// dE/da_j of a window whose depth-i acceptance is held by lane (base + i) of the warp (each lane
// names its own window and depth): the bits of window_term's dE[j], with the same roundings in
// the same order, 0 for j >= kn; every lane of the warp must call it.
__device__ __forceinline__ float window_partial(float a_l, int base, int j, int kn) {
  float P = 1.f, S = 1.f;
#pragma unroll
  for (int i = 0; i < AAL_MAX_K; ++i) {  // P_j = a_0 ... a_{j-1}
    const float v = __shfl_sync(0xffffffffu, a_l, (base + i) & 31);
    if (i < j && i < kn) P = __fmul_rn(P, v);
  }
#pragma unroll
  for (int i = AAL_MAX_K - 1; i >= 0; --i) {  // S_j = 1 + a_{j+1} (1 + a_{j+2} (...)) from the top
    const float v = __shfl_sync(0xffffffffu, a_l, (base + i) & 31);
    if (i > j && i < kn) S = __fmaf_rn(v, S, 1.f);
  }
  return j < kn ? __fmul_rn(P, S) : 0.f;
}

// The exchange of the fused sequence layout, run by one whole warp for row p (position p - lo of
// the sequence whose rows are lo .. hi; every row's word is published with its statistics).
// Lane l < 2K - 1 polls the word of row p - (K - 1) + l when that row is in the sequence,
// bounded like window_exchange.  Lane j < K then forms the window that starts at row p - j (when
// it starts inside the sequence) as the sequence window kernel does: its K_n leading valid
// positions (stopping at the sequence's end or its first invalid position; 0 when full_windows
// and K_n < K), dE/da by window_term, and the depth-j partials (greedy; sampling with w_s and
// the TV term folded in).  Lane 0 adds them in increasing j, as the gather does, into dEg and
// dEs.  Returns, to every lane, whether the words arrived.
template <typename Pre = NoPrePoll>
__device__ __forceinline__ bool seq_exchange(const uint64_t* mbox, const uint8_t* mask, int64_t p, int64_t lo,
                                             int64_t hi, int K, bool full, bool greedy, bool sampling, bool tv,
                                             float w_sampling, float w_tv, bool need, int lane,
                                             volatile int* abort_flag, WsHeader* hdr, uint64_t limit_ns,
                                             float* dEg, float* dEs, Pre pre = Pre()) {
  bool ok = __shfl_sync(0xffffffffu, *abort_flag == 0 ? 1 : 0, 0) != 0;
  // rows p - back .. p + fwd are the sequence's within K - 1 of p; lane l holds row p + l - (K - 1)
  const int back = (int)min(p - lo, (int64_t)(K - 1)), fwd = (int)min(hi - p, (int64_t)(K - 1));
  const int o = lane - (K - 1);
  const bool mine = lane < 2 * K - 1 && o >= -back && o <= fwd;
  const uint64_t* mrow = mbox + p;
  uint64_t w = 0;
  if (lane == 0 && !(ok && need)) pre();
  if (ok && need) {
    const uint64_t t0 = ptx::now_ns();
    for (uint32_t it = 0;; ++it) {
      if (mine) w = ptx::ld_relaxed(mrow + o);
      if (it == 0 && lane == 0) pre();
      if (__all_sync(0xffffffffu, !mine || w != kMboxEmpty)) break;
      int quit = 0;
      if (lane == 0 && (*abort_flag || it >= kSpinLimit || ptx::now_ns() - t0 > limit_ns)) {
        if (!*abort_flag) {
          *abort_flag = 1;
          atomicExch(&hdr->status, kStatusTimeout);
        }
        quit = 1;
      }
      if (__shfl_sync(0xffffffffu, quit, 0)) {
        ok = false;
        break;
      }
      __nanosleep(64);
    }
  }
  const float ag_l = __uint_as_float((uint32_t)w), as_l = __uint_as_float((uint32_t)(w >> 32));
  // lane j: the window starting at row p - j, K_n positions long
  int kn = 0;
  if (need && lane < K && lane <= back) {
    const uint8_t* mrow8 = mask != nullptr ? mask + (p - lane) : nullptr;
    while (kn < K && kn - lane <= fwd && (mrow8 == nullptr || mrow8[kn] != 0)) ++kn;
    if (full && kn < K) kn = 0;
  }
  // row p - j + i was polled by lane (K - 1) - j + i
  const int base = (K - 1) - lane;
  float pg = 0.f, ps = 0.f;
  if (greedy) pg = window_partial(ag_l, base, lane, kn);
  if (sampling || tv) {
    const float d = sampling ? window_partial(as_l, base, lane, kn) : 0.f;
    const float tvc = (tv && kn > 0) ? w_tv / (float)kn : 0.f;
    ps = __fadd_rn(sampling ? __fmul_rn(w_sampling, d) : 0.f, lane < kn ? tvc : 0.f);
  }
  float g = 0.f, s = 0.f;
#pragma unroll
  for (int j = 0; j < AAL_MAX_K; ++j) {
    const float pgj = __shfl_sync(0xffffffffu, pg, j);
    const float psj = __shfl_sync(0xffffffffu, ps, j);
    if (j < K && j <= back) {
      if (greedy) g += pgj;
      if (sampling || tv) s += psj;
    }
  }
  *dEg = g;
  *dEs = s;
  return ok;
}

}  // namespace aal
