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

struct RowCoef {
  float sT, Mq, Lsq, Mp, Lsp, Mq1, Lsq1, Mp1, Lsp1;
  float Ck;          // c^kl
  float cpos, cneg;  // g^s/T (1 - Qlt) and -g^s/T Qlt
  float Ag;          // g^g a^g
  float Cg;          // c^grpo
  float Aq;          // Ag + Cg, the coefficient of -q(u)
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

// The row's coefficients from its statistics, dE^g/da (unweighted), dE^s/da (weights folded),
// the GRPO coefficient and whether the row is a valid position (the anchor's rows).  Returns
// false when every term of the row is zero (the row's gradient is all zeros).
template <bool GREEDY, bool SAMPLING, bool KL>
__device__ __forceinline__ bool row_coef(const BackwardArgs& a, float scale, float kscale, float dEg, float dEs,
                                         float cgr, bool pos_valid, const RowStat& st, RowCoef& c) {
  const float gg = (GREEDY && a.w_greedy != 0.f) ? scale * a.w_greedy * dEg : 0.f;
  const float cg = (GREEDY && a.grpo) ? a.dloss * cgr : 0.f;
  const float gs = SAMPLING ? scale * a.w_sampling * dEs : 0.f;
  const float ck = (KL && pos_valid) ? kscale : 0.f;
  if (gg == 0.f && gs == 0.f && ck == 0.f && cg == 0.f) return false;
  c.sT = a.sT;
  c.Mq = SAMPLING ? st.Mq : 0.f;
  c.Lsq = SAMPLING ? st.Lsq : 0.f;
  c.Mp = SAMPLING ? st.Mp : 0.f;
  c.Lsp = SAMPLING ? st.Lsp : 0.f;
  c.Mq1 = (GREEDY || KL) ? st.Mq1 : 0.f;
  c.Lsq1 = (GREEDY || KL) ? st.Lsq1 : 0.f;
  c.Mp1 = KL ? st.Mp1 : 0.f;
  c.Lsp1 = KL ? st.Lsp1 : 0.f;
  c.Ck = ck;
  const float qlt = SAMPLING ? st.qlt : 0.f;
  const float Bs = gs * a.invT;
  c.cpos = Bs * (1.f - qlt);
  c.cneg = -Bs * qlt;
  c.Ag = gg != 0.f ? gg * st.ag : 0.f;
  c.Cg = cg;
  c.Aq = c.Ag + c.Cg;
  c.xs = gg != 0.f ? st.xs : -1;
  c.ys = cg != 0.f ? st.ys : -1;
  return true;
}

// Every term of element u except the greedy and GRPO spikes (+Ag at x*, +Cg at y), which
// the callers add: once per 16-byte vector in the vector paths, per element in the scalar one.
template <bool GREEDY, bool SAMPLING, bool Q1_IS_QT, bool KL>
__device__ __forceinline__ float grad_elem(const RowCoef& c, float q, float p) {
  float d = 0.f, qt = 0.f;
  if (SAMPLING) {
    const float lq = log2_prob(q, c.sT, c.Mq, c.Lsq);
    const float lp = log2_prob(p, c.sT, c.Mp, c.Lsp);
    qt = ex2(lq);
    d = qt * (lq < lp ? c.cpos : c.cneg);
  }
  if (GREEDY || KL) {
    const float q1 = Q1_IS_QT ? qt : ex2(log2_prob(q, kLog2e, c.Mq1, c.Lsq1));
    if (GREEDY) d = fmaf(-c.Aq, q1, d);
    if (KL) d = fmaf(c.Ck, q1 - ex2(log2_prob(p, kLog2e, c.Mp1, c.Lsp1)), d);
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
  float qv[E], pv[E], d[E];
  Io<T>::unpack(qw, qv);
  if (READ_P) Io<T>::unpack(pw, pv);
#pragma unroll
  for (int e = 0; e < E; ++e) d[e] = grad_elem<GREEDY, SAMPLING, Q1_IS_QT, KL>(c, qv[e], READ_P ? pv[e] : 0.f);
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

}  // namespace aal
