// Backward of the EAL / WTV losses with respect to the draft logits (the per-element terms
// are in grad_elem.cuh).  q(u), q~(u) and c_u are recomputed from the logits and the row's
// saved log-sum-exps; nothing of size V is materialised.  One pass: reads z_q (and z_p when
// the sampling term or the anchor is on), writes dz in the logits' dtype.  c^kl = dloss w_kl /
// |positions| on valid positions, 0 elsewhere; c^grpo = dloss times the per-row coefficient
// aal_grpo_from_loss left in the workspace.  The greedy and GRPO terms share q(u), so both
// run in the GREEDY instantiation.
#include "grad_elem.cuh"

namespace aal {
namespace {

constexpr int kBwdThreads = 256;

template <typename T, bool VEC, bool GREEDY, bool SAMPLING, bool Q1_IS_QT, bool KL>
__device__ __forceinline__ void backward_rows(const BackwardArgs& a) {
  const int nvalid = a.ws.hdr->nvalid;
  const float scale = nvalid > 0 ? -a.dloss / (float)nvalid : 0.f;
  const int npos = KL ? a.ws.hdr->npos : 0;
  const float kscale = npos > 0 ? a.dloss * a.w_kl / (float)npos : 0.f;
  constexpr bool READ_P = SAMPLING || KL;
  constexpr int E = Io<T>::E;
  const bool with_greedy = GREEDY && a.w_greedy != 0.f;
  for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
    const float dEg = with_greedy ? a.ws.dEg[r] : 0.f;
    const float cgr = (GREEDY && a.grpo) ? a.ws.cgr[r] : 0.f;
    const float dEs = SAMPLING ? a.ws.dEs[r] : 0.f;
    const bool pos_valid = a.mask == nullptr || a.mask[r] != 0;
    const RowStat st = load_row_stat<GREEDY, SAMPLING, KL>(a.ws, r, with_greedy, GREEDY && a.grpo);
    T* out = static_cast<T*>(a.grad) + r * a.V;
    const T* zq = static_cast<const T*>(a.zq) + r * a.V;
    const T* zp = READ_P ? static_cast<const T*>(a.zp) + r * a.V : nullptr;  // (token ids otherwise)
    RowCoef c;
    if (!row_coef<GREEDY, SAMPLING, KL>(a, scale, kscale, dEg, dEs, cgr, pos_valid, st, c)) {
      if (VEC) {
        uint4* o4 = reinterpret_cast<uint4*>(out);
        for (int64_t i = threadIdx.x; i < a.V / E; i += kBwdThreads) st_stream(o4 + i, make_uint4(0, 0, 0, 0));
      } else {
        for (int64_t v = threadIdx.x; v < a.V; v += kBwdThreads) Io<T>::store1(out + v, 0.f);
      }
      continue;
    }
    if (VEC) {
      const int64_t nv = a.V / E;
      // the vectors and lanes of the spikes (-1: none)
      const int64_t xv = c.xs >= 0 ? c.xs / E : -1, yv = c.ys >= 0 ? c.ys / E : -1;
      const int xe = c.xs >= 0 ? c.xs % E : 0, ye = c.ys >= 0 ? c.ys % E : 0;
      const uint4* q4 = reinterpret_cast<const uint4*>(zq);
      const uint4* p4 = reinterpret_cast<const uint4*>(zp);
      uint4* o4 = reinterpret_cast<uint4*>(out);
      for (int64_t i = threadIdx.x; i < nv; i += kBwdThreads) {
        const uint4 qw = ldg_stream(q4 + i);
        const uint4 pw = READ_P ? ldg_stream(p4 + i) : make_uint4(0, 0, 0, 0);
        st_stream(o4 + i, grad_vec<T, GREEDY, SAMPLING, Q1_IS_QT, KL>(c, qw, pw, i, xv, xe, yv, ye));
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
// The anchor's bf16 vector instances (two exponentials an element) are bounded for enough
// loads in flight: six blocks an SM (40 registers) without the sampling term (unbounded they
// took 48, five blocks), five with it (at 40 registers they spilled; measured 6.47 against
// 6.50 ms); the others fit six or more unbounded, and fp32 ones would spill at 40.
template <typename T, bool G, bool S, bool Q>
__global__ void __launch_bounds__(kBwdThreads, S ? 5 : 6) backward_kernel_kl(BackwardArgs a) {
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
