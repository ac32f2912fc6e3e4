// Backward of the EAL / WTV losses with respect to the draft logits.
//
// For row r = (n, j) with g^g = -(dloss/|W|) w_g dE^g_n/da^g_{n,j} and
// g^s = -(dloss/|W|) w_s dE^s_n/da^s_{n,j} (dE/da from the window kernel):
//   dz_u = g^g a^g (delta_{u,x*} - q(u))                 greedy term, Eq. acc_greedy
//        + g^s (1/T) q~(u) (c_u - Qlt),  c_u = [q~_u < p~_u]   sampling term, Eq. acc_sample
//        + c^kl (q(u) - p(u))                                  KL anchor (Sec. 4.1), T = 1
//        + c^grpo (delta_{u,y} - q(u))                         GRPO surrogate (Sec. 3.4), y = argmax z_q
// (the softmax Jacobian applied to d a / d q; at a tie q~_u = p~_u the min follows the
// frozen p~, so c_u = 0).  q(u), q~(u) and c_u are recomputed from the logits and the
// row's saved log-sum-exps; nothing of size V is materialised.  One pass: reads z_q
// (and z_p when the sampling term or the anchor is on), writes dz in the logits' dtype.
// c^kl = dloss w_kl / |positions| on valid positions, 0 elsewhere; c^grpo = dloss times the
// per-row coefficient aal_grpo_from_loss left in the workspace.  The greedy and GRPO terms
// share q(u), so both run in the GREEDY instantiation.
#include "aal_internal.cuh"

namespace aal {
namespace {

constexpr int kBwdThreads = 256;

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

// Every term of element u except the greedy and GRPO spikes (+Ag at x*, +Cg at y), which
// the callers add: once per 16-byte vector in the vector path, per element in the scalar one.
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

template <typename T, bool VEC, bool GREEDY, bool SAMPLING, bool Q1_IS_QT, bool KL>
__device__ __forceinline__ void backward_rows(const BackwardArgs& a) {
  const int nvalid = a.ws.hdr->nvalid;
  const float scale = nvalid > 0 ? -a.dloss / (float)nvalid : 0.f;
  const int npos = KL ? a.ws.hdr->npos : 0;
  const float kscale = npos > 0 ? a.dloss * a.w_kl / (float)npos : 0.f;
  constexpr bool READ_P = SAMPLING || KL;
  constexpr int E = Io<T>::E;
  for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
    const float gg = (GREEDY && a.w_greedy != 0.f) ? scale * a.w_greedy * a.ws.dEg[r] : 0.f;
    const float cg = (GREEDY && a.grpo) ? a.dloss * a.ws.cgr[r] : 0.f;
    const float gs = SAMPLING ? scale * a.w_sampling * a.ws.dEs[r] : 0.f;
    const float ck = (KL && (a.mask == nullptr || a.mask[r] != 0)) ? kscale : 0.f;
    T* out = static_cast<T*>(a.grad) + r * a.V;
    const T* zq = static_cast<const T*>(a.zq) + r * a.V;
    const T* zp = READ_P ? static_cast<const T*>(a.zp) + r * a.V : nullptr;  // (token ids otherwise)
    if (gg == 0.f && gs == 0.f && ck == 0.f && cg == 0.f) {
      if (VEC) {
        uint4* o4 = reinterpret_cast<uint4*>(out);
        for (int64_t i = threadIdx.x; i < a.V / E; i += kBwdThreads) st_stream(o4 + i, make_uint4(0, 0, 0, 0));
      } else {
        for (int64_t v = threadIdx.x; v < a.V; v += kBwdThreads) Io<T>::store1(out + v, 0.f);
      }
      continue;
    }
    RowCoef c;
    c.sT = a.sT;
    c.Mq = SAMPLING ? a.ws.Mq[r] : 0.f;
    c.Lsq = SAMPLING ? a.ws.Lsq[r] : 0.f;
    c.Mp = SAMPLING ? a.ws.Mp[r] : 0.f;
    c.Lsp = SAMPLING ? a.ws.Lsp[r] : 0.f;
    c.Mq1 = (GREEDY || KL) ? a.ws.Mq1[r] : 0.f;
    c.Lsq1 = (GREEDY || KL) ? a.ws.Lsq1[r] : 0.f;
    c.Mp1 = KL ? a.ws.Mp1[r] : 0.f;
    c.Lsp1 = KL ? a.ws.Lsp1[r] : 0.f;
    c.Ck = ck;
    const float qlt = SAMPLING ? a.ws.qlt[r] : 0.f;
    const float Bs = gs * a.invT;
    c.cpos = Bs * (1.f - qlt);
    c.cneg = -Bs * qlt;
    c.Ag = gg != 0.f ? gg * a.ws.ag[r] : 0.f;
    c.Cg = cg;
    c.Aq = c.Ag + c.Cg;
    c.xs = gg != 0.f ? a.ws.xstar[r] : -1;
    c.ys = cg != 0.f ? a.ws.yhat[r] : -1;
    if (VEC) {
      const int64_t nv = a.V / E;
      // the vectors and lanes of the spikes (-1: none)
      const int64_t xv = c.xs >= 0 ? c.xs / E : -1, yv = c.ys >= 0 ? c.ys / E : -1;
      const int xe = c.xs >= 0 ? c.xs % E : 0, ye = c.ys >= 0 ? c.ys % E : 0;
      const uint4* q4 = reinterpret_cast<const uint4*>(zq);
      const uint4* p4 = reinterpret_cast<const uint4*>(zp);
      uint4* o4 = reinterpret_cast<uint4*>(out);
      for (int64_t i = threadIdx.x; i < nv; i += kBwdThreads) {
        float qv[E], pv[E], d[E];
        Io<T>::unpack(ldg_stream(q4 + i), qv);
        if (READ_P) Io<T>::unpack(ldg_stream(p4 + i), pv);
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
        st_stream(o4 + i, Io<T>::pack(d));
      }
    } else {
      for (int64_t v = threadIdx.x; v < a.V; v += kBwdThreads) {
        const float q = load_elem<T>(zq + v);
        const float p = READ_P ? load_elem<T>(zp + v) : 0.f;
        float d = grad_elem<GREEDY, SAMPLING, Q1_IS_QT, KL>(c, q, p);
        if (GREEDY) {
          if (v == c.xs) d += c.Ag;
          if (v == c.ys) d += c.Cg;
        }
        Io<T>::store1(out + v, d);
      }
    }
  }
}

template <typename T, bool VEC, bool G, bool S, bool Q, bool KL>
__global__ void __launch_bounds__(kBwdThreads) backward_kernel(BackwardArgs a) {
  backward_rows<T, VEC, G, S, Q, KL>(a);
}
// The anchor's bf16 vector instances (two exponentials an element) are held to 40
// registers, six blocks an SM, for enough loads in flight (unbounded they took 48, five
// blocks); the others fit six or more unbounded, and fp32 ones would spill at 40.
template <typename T, bool G, bool S, bool Q>
__global__ void __launch_bounds__(kBwdThreads, 6) backward_kernel_kl(BackwardArgs a) {
  backward_rows<T, true, G, S, Q, true>(a);
}

template <typename T, bool VEC, bool G, bool S, bool Q, bool KL>
cudaError_t go(const BackwardArgs& a, cudaStream_t s) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  void (*kern)(BackwardArgs);
  if constexpr (VEC && KL && sizeof(T) == 2) kern = backward_kernel_kl<T, G, S, Q>;
  else kern = backward_kernel<T, VEC, G, S, Q, KL>;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kBwdThreads, 0);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)sms * per_sm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  kern<<<(unsigned)grid, kBwdThreads, 0, s>>>(a);
  return cudaGetLastError();
}

template <typename T, bool VEC, bool KL>
cudaError_t dispatch_mode(const BackwardArgs& a, cudaStream_t s) {
  const bool G = a.w_greedy != 0.f || a.grpo, S = a.w_sampling != 0.f;
  const bool Q = a.q1_is_qT && S && (G || KL);
  if (G && S) return Q ? go<T, VEC, true, true, true, KL>(a, s) : go<T, VEC, true, true, false, KL>(a, s);
  if (G) return go<T, VEC, true, false, false, KL>(a, s);
  if (S) {
    if constexpr (KL) {
      if (Q) return go<T, VEC, false, true, true, KL>(a, s);
    }
    return go<T, VEC, false, true, false, KL>(a, s);
  }
  return go<T, VEC, false, false, false, KL>(a, s);
}

template <typename T>
cudaError_t dispatch(const BackwardArgs& a, cudaStream_t s) {
  // z_p is read only by the sampling term and the anchor (and may be token ids otherwise)
  const bool reads_p = a.w_sampling != 0.f || a.w_kl != 0.f;
  const bool vec = ((a.V * (int64_t)sizeof(T)) % 16 == 0) &&
                   ((reinterpret_cast<uintptr_t>(a.zq) | (reads_p ? reinterpret_cast<uintptr_t>(a.zp) : 0) |
                     reinterpret_cast<uintptr_t>(a.grad)) % 16 == 0);
  if (a.w_kl != 0.f) return vec ? dispatch_mode<T, true, true>(a, s) : dispatch_mode<T, false, true>(a, s);
  return vec ? dispatch_mode<T, true, false>(a, s) : dispatch_mode<T, false, false>(a, s);
}

}  // namespace

cudaError_t launch_backward(const BackwardArgs& a, bool bf16, cudaStream_t s) {
  return bf16 ? dispatch<uint16_t>(a, s) : dispatch<float>(a, s);
}

}  // namespace aal
