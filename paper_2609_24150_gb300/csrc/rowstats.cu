// Forward per-row statistics of the EAL / WTV losses.
//
// For every logit row r = (window n, depth j) this computes, from z_p (target)
// and z_q (draft):
//   (M, Ls)  the normalisers of z_p/T and z_q/T (the temperature-scaled distributions
//            of Sec. 2.3) and of z_q (the unscaled draft of Eq. acc_greedy):
//            M = max_v z_v, Ls = log2 sum_v 2^((z_v - M) s),
//   x*       argmax_v z_p (lowest index on ties) and a^greedy = q(x*) (Eq. acc_greedy),
//   a^sample = sum_v min(p~_v, q~_v)   (Eq. acc_sample),
//   Qlt      = sum_{v: q~_v < p~_v} q~_v, which the backward of a^sample needs,
//   KL(p || q) at T = 1 and the normaliser of z_p at T = 1, for the forward-KL anchor of
//            the combined objectives (Sec. 4.1), in the same pass as the normalisers.
// a^sample needs both normalisers before it can be summed, so it is a second phase
// over the row.  This file holds the generic kernel: one CTA per row, both
// phases streamed from global memory (the second mostly from L2), any V and any
// row alignment.
#include "aal_internal.cuh"

namespace aal {
namespace {

constexpr int kGenericThreads = 256;
constexpr int kGenericWarps = kGenericThreads / 32;

template <typename T>
struct Vec {
  static constexpr int E = 16 / sizeof(T);
};

template <typename T>
__device__ __forceinline__ void unpack(const uint4& w, float* out);
template <>
__device__ __forceinline__ void unpack<float>(const uint4& w, float* out) {
  out[0] = __uint_as_float(w.x);
  out[1] = __uint_as_float(w.y);
  out[2] = __uint_as_float(w.z);
  out[3] = __uint_as_float(w.w);
}
template <>
__device__ __forceinline__ void unpack<uint16_t>(const uint4& w, float* out) {
  out[0] = bf16_lo(w.x);
  out[1] = bf16_hi(w.x);
  out[2] = bf16_lo(w.y);
  out[3] = bf16_hi(w.y);
  out[4] = bf16_lo(w.z);
  out[5] = bf16_hi(w.z);
  out[6] = bf16_lo(w.w);
  out[7] = bf16_hi(w.w);
}

struct Phase1 {
  Lse p, q, q1;
  KlAcc kl;
  Amax am;  // target argmax, carrying z_q there
  Amax aq;  // draft argmax, carrying z_p there
};

__device__ __forceinline__ Phase1 merge1(const Phase1& a, const Phase1& b, float sT) {
  Phase1 r;
  r.p = lse_merge(a.p, b.p, sT);
  r.q = lse_merge(a.q, b.q, sT);
  r.q1 = lse_merge(a.q1, b.q1, kLog2e);
  r.kl = kl_merge(a.kl, b.kl);
  r.am = amax_merge(a.am, b.am);
  r.aq = amax_merge(a.aq, b.aq);
  return r;
}

__device__ __forceinline__ Phase1 shfl1(const Phase1& a, int off) {
  Phase1 b;
  b.p = shfl_lse(a.p, off);
  b.q = shfl_lse(a.q, off);
  b.q1 = shfl_lse(a.q1, off);
  b.kl.M = __shfl_xor_sync(0xffffffffu, a.kl.M, off);
  b.kl.S = __shfl_xor_sync(0xffffffffu, a.kl.S, off);
  b.kl.D = __shfl_xor_sync(0xffffffffu, a.kl.D, off);
  b.am = shfl_amax(a.am, off);
  b.aq = shfl_amax(a.aq, off);
  return b;
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kGenericThreads) rowstats_generic(RowStatsArgs a) {
  __shared__ Phase1 red1[kGenericWarps];
  __shared__ float2 red2[kGenericWarps];
  __shared__ Phase1 row1;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
    const T* zq = static_cast<const T*>(a.zq) + r * a.V;
    const T* zp = static_cast<const T*>(a.zp) + r * a.V;

    Phase1 acc;
    lse_init(acc.p);
    lse_init(acc.q);
    lse_init(acc.q1);
    kl_init(acc.kl);
    amax_init(acc.am);
    amax_init(acc.aq);
    auto visit = [&](int64_t v, float p, float q) {
      if (p > acc.am.v) {
        acc.am.v = p;
        acc.am.i = (int32_t)v;
        acc.am.carry = q;
      }
      if (q > acc.aq.v) {
        acc.aq.v = q;
        acc.aq.i = (int32_t)v;
        acc.aq.carry = p;
      }
      if (a.need_p) lse_push(acc.p, p, a.sT);
      if (a.need_q) lse_push(acc.q, q, a.sT);
      if (a.need_q1) lse_push(acc.q1, q, kLog2e);
      if (a.need_kl) kl_push(acc.kl, p, q);
    };
    constexpr int E = Vec<T>::E;
    if (VEC) {
      const int64_t nv = a.V / E;
      const uint4* p4 = reinterpret_cast<const uint4*>(zp);
      const uint4* q4 = reinterpret_cast<const uint4*>(zq);
      for (int64_t i = threadIdx.x; i < nv; i += blockDim.x) {
        float pv[E], qv[E];
        unpack<T>(ldg_stream(p4 + i), pv);
        unpack<T>(ldg_stream(q4 + i), qv);
#pragma unroll
        for (int e = 0; e < E; ++e) visit(i * E + e, pv[e], qv[e]);
      }
    } else {
      for (int64_t v = threadIdx.x; v < a.V; v += blockDim.x)
        visit(v, load_elem<T>(zp + v), load_elem<T>(zq + v));
    }

    // block reduction of phase 1 (fixed butterfly + fixed warp order: deterministic)
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc = merge1(acc, shfl1(acc, off), a.sT);
    if (lane == 0) red1[warp] = acc;
    __syncthreads();
    if (warp == 0) {
      Phase1 x;
      if (lane < kGenericWarps) {
        x = red1[lane];
      } else {
        lse_init(x.p);
        lse_init(x.q);
        lse_init(x.q1);
        kl_init(x.kl);
        amax_init(x.am);
        amax_init(x.aq);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) x = merge1(x, shfl1(x, off), a.sT);
      if (lane == 0) row1 = x;
    }
    __syncthreads();
    const Phase1 tot = row1;
    const float Mp = tot.p.M, Lsp = a.need_p ? lse_ls(tot.p) : 0.f;
    const float Mq = tot.q.M, Lsq = a.need_q ? lse_ls(tot.q) : 0.f;
    const float Mq1 = a.need_q1 ? tot.q1.M : Mq, Lsq1 = a.need_q1 ? lse_ls(tot.q1) : Lsq;

    float s_min = 0.f, s_qlt = 0.f;
    if (a.overlap) {
      auto visit2 = [&](float p, float q) {
        const float lp = log2_prob(p, a.sT, Mp, Lsp);
        const float lq = log2_prob(q, a.sT, Mq, Lsq);
        const float e = ex2(fminf(lp, lq));
        s_min += e;
        if (lq < lp) s_qlt += e;
      };
      if (VEC) {
        const int64_t nv = a.V / E;
        const uint4* p4 = reinterpret_cast<const uint4*>(zp);
        const uint4* q4 = reinterpret_cast<const uint4*>(zq);
        for (int64_t i = threadIdx.x; i < nv; i += blockDim.x) {
          float pv[E], qv[E];
          unpack<T>(ldg_stream(p4 + i), pv);
          unpack<T>(ldg_stream(q4 + i), qv);
#pragma unroll
          for (int e = 0; e < E; ++e) visit2(pv[e], qv[e]);
        }
      } else {
        for (int64_t v = threadIdx.x; v < a.V; v += blockDim.x)
          visit2(load_elem<T>(zp + v), load_elem<T>(zq + v));
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        s_min += __shfl_xor_sync(0xffffffffu, s_min, off);
        s_qlt += __shfl_xor_sync(0xffffffffu, s_qlt, off);
      }
      if (lane == 0) red2[warp] = make_float2(s_min, s_qlt);
      __syncthreads();
      if (threadIdx.x == 0) {
        float2 t = red2[0];
        for (int w = 1; w < kGenericWarps; ++w) {
          t.x += red2[w].x;
          t.y += red2[w].y;
        }
        s_min = t.x;
        s_qlt = t.y;
      }
    }
    if (threadIdx.x == 0) {
      a.ws.Mp[r] = Mp;
      a.ws.Lsp[r] = Lsp;
      a.ws.Mq[r] = Mq;
      a.ws.Lsq[r] = Lsq;
      a.ws.Mq1[r] = Mq1;
      a.ws.Lsq1[r] = Lsq1;
      if (a.need_kl) {
        const float Lsp1 = log2f(tot.kl.S);
        a.ws.Mp1[r] = tot.kl.M;
        a.ws.Lsp1[r] = Lsp1;
        a.ws.kl[r] = tot.kl.D / tot.kl.S - (tot.kl.M - Mq1) - kLn2 * (Lsp1 - Lsq1);
      }
      a.ws.xstar[r] = tot.am.i;
      a.ws.yhat[r] = tot.aq.i;
      a.ws.zpy[r] = tot.aq.carry;
      a.ws.ag[r] = exp2f(log2_prob(tot.am.carry, kLog2e, Mq1, Lsq1));
      a.ws.cpart[r * kMaxCluster] = make_float2(s_min, s_qlt);
    }
    __syncthreads();  // red1/red2/row1 are reused by the next row
  }
}

template <typename T>
cudaError_t launch_generic(const RowStatsArgs& a, cudaStream_t s) {
  const bool vec = ((a.V * (int64_t)sizeof(T)) % 16 == 0) &&
                   ((reinterpret_cast<uintptr_t>(a.zq) | reinterpret_cast<uintptr_t>(a.zp)) % 16 == 0);
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (vec)
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rowstats_generic<T, true>, kGenericThreads, 0);
  else
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rowstats_generic<T, false>, kGenericThreads, 0);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)sms * per_sm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  if (vec)
    rowstats_generic<T, true><<<(unsigned)grid, kGenericThreads, 0, s>>>(a);
  else
    rowstats_generic<T, false><<<(unsigned)grid, kGenericThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

// The TMA-streamed kernel (rowstats_stream.cu) serves rows whose byte length is a multiple
// of 16: in two passes with the sampling term, in one pass without it; bf16 rows under the fused
// call's threshold take its short-row geometry (rowstats_short.cu).  Unaligned rows take the
// generic kernel.
cudaError_t launch_rowstats(const RowStatsArgs& a, bool bf16, cudaStream_t s, int* cluster_used) {
  const int elt = bf16 ? 2 : 4;
  const bool aligned = ((a.V * elt) % 16 == 0) &&
                       ((reinterpret_cast<uintptr_t>(a.zq) | reinterpret_cast<uintptr_t>(a.zp)) % 16 == 0);
  if (aligned) {
    *cluster_used = 1;
    const uint64_t limit = debug_wait_limit_ns();
    if (bf16 && a.V * 2 < fused_min_row_bytes())
      return launch_rowstats_stream_short(a, bf16, s, limit ? limit : kWaitLimitNs);
    return launch_rowstats_stream(a, bf16, s, limit ? limit : kWaitLimitNs);
  }
  *cluster_used = 1;
  return bf16 ? launch_generic<uint16_t>(a, s) : launch_generic<float>(a, s);
}

}  // namespace aal
