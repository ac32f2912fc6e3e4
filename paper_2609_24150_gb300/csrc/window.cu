// Window combination of the per-position acceptances into the losses.
//
// Per window n with K_n leading valid depths (Sec. 3.1, Eq. eal_generic):
//   E_n = sum_{k=1}^{K_n} P_k,   P_k = prod_{j<k} a_{n,j}
//   dE_n/da_{n,j} = P_j * S_j,  S_{K_n-1} = 1,  S_j = 1 + a_{n,j+1} S_{j+1}   (j < K_n)
// for the greedy term (a^greedy, Eq. loss_eal) and the sampling term (a^sample,
// Eq. loss_tv).  The partials go to the workspace for the backward; the loss
// L = -(w_g sum E^g + w_s sum E^s) / |W| (+ w_kl times the mean KL anchor over the
// valid positions, Sec. 4.1) is summed deterministically: each block reduces its
// windows in a fixed tree, and the last block to finish adds the block partials in
// index order.
#include "aal_internal.cuh"

namespace aal {
namespace {

// Sum NV doubles over the block in a fixed order (warp butterflies, then warps in index
// order); the totals land in thread 0.
template <int NT, int NV>
__device__ __forceinline__ void block_sum(double (&x)[NV], double* sm) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
    for (int i = 0; i < NV; ++i) x[i] += __shfl_xor_sync(0xffffffffu, x[i], off);
  }
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < NV; ++i) sm[NV * warp + i] = x[i];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
#pragma unroll
    for (int i = 0; i < NV; ++i) x[i] = sm[i];
    for (int w = 1; w < NT / 32; ++w) {
#pragma unroll
      for (int i = 0; i < NV; ++i) x[i] += sm[NV * w + i];
    }
  }
  __syncthreads();
}

constexpr int kSums = 6;  // sum E^g, sum E^s, |W|, sum KL, |positions|, sum of window TV means

// Block partials -> the last block to finish adds them in block order and writes the loss
//   L = -(w_g sum E^g + w_s sum E^s) / |W| + w_kl sum KL / |positions|
//       + w_tv sum_n (1/K_n) sum_j (1 - a^s_{n,j}) / |W|
// (each term 0 when its count is 0), |W| and |positions|.
template <typename Args>
__device__ __forceinline__ void finish_loss(const Args& a, double (&x)[kSums], double* sm, bool* is_last) {
  block_sum<kWindowThreads, kSums>(x, sm);
  if (threadIdx.x == 0) {
#pragma unroll
    for (int i = 0; i < kSums; ++i) a.ws.wpart[kWpart * blockIdx.x + i] = x[i];
    __threadfence();
    const unsigned ticket = atomicAdd(&a.ws.hdr->done_blocks, 1u);
    *is_last = (ticket == gridDim.x - 1);
  }
  __syncthreads();
  if (!*is_last) return;
  __threadfence();
  double t[kSums];
#pragma unroll
  for (int i = 0; i < kSums; ++i) t[i] = 0.0;
  const volatile double* wp = a.ws.wpart;
  for (int64_t b = threadIdx.x; b < a.nwblk; b += kWindowThreads) {
#pragma unroll
    for (int i = 0; i < kSums; ++i) t[i] += wp[kWpart * b + i];
  }
  block_sum<kWindowThreads, kSums>(t, sm);
  if (threadIdx.x == 0) {
    // the data-parallel normalisers of the whole batch when the caller gives them
    const int nvalid = a.nvalid_g >= 0 ? a.nvalid_g : (int)t[2];
    const int npos = a.npos_g >= 0 ? a.npos_g : (int)t[4];
    const double num = (a.greedy ? (double)a.w_greedy * t[0] : 0.0) +
                       (a.sampling ? (double)a.w_sampling * t[1] : 0.0);
    double L = nvalid > 0 ? -num / (double)nvalid : 0.0;
    if (a.kl && npos > 0) L += (double)a.w_kl * t[3] / (double)npos;
    if (a.tv && nvalid > 0) L += (double)a.w_tv * t[5] / (double)nvalid;
    const float loss = (float)L;
    *a.loss = loss;
    a.ws.hdr->loss = loss;
    a.ws.hdr->nvalid = nvalid;
    a.ws.hdr->npos = npos;
    a.ws.hdr->cluster = a.cluster;
    a.ws.hdr->done_blocks = 0u;
  }
}

__global__ void __launch_bounds__(kWindowThreads) window_kernel(WindowArgs a) {
  __shared__ double sm[kSums * kWindowThreads / 32];
  __shared__ bool is_last;
  const int64_t n = (int64_t)blockIdx.x * kWindowThreads + threadIdx.x;
  double eg = 0.0, es = 0.0, valid = 0.0, ksum = 0.0, kcnt = 0.0, tvs = 0.0;
  const bool ov = a.sampling || a.tv;  // both terms are built from a^sample
  if (n < a.N) {
    const int K = a.K;
    int kn = K;
    if (a.mask != nullptr) {
      kn = 0;
      while (kn < K && a.mask[n * K + kn] != 0) ++kn;
    }
    valid = kn >= 1 ? 1.0 : 0.0;
    const int64_t r0 = n * K;
    float ag[AAL_MAX_K], as[AAL_MAX_K], dE[AAL_MAX_K];
#pragma unroll
    for (int j = 0; j < AAL_MAX_K; ++j) {
      ag[j] = 0.f;
      as[j] = 0.f;
      if (j < K) {
        const int64_t r = r0 + j;
        if (a.greedy) ag[j] = a.ws.ag[r];
        if (ov) {
          float2 t = a.ws.cpart[r * kMaxCluster];
          for (int c = 1; c < a.cluster; ++c) {
            const float2 u = a.ws.cpart[r * kMaxCluster + c];
            t.x += u.x;
            t.y += u.y;
          }
          as[j] = t.x;
          a.ws.as[r] = t.x;
          a.ws.qlt[r] = t.y;
        }
      }
    }
    float Eg = 0.f, Es = 0.f;
    if (a.greedy) {
      Eg = window_term(ag, kn, dE);
#pragma unroll
      for (int j = 0; j < AAL_MAX_K; ++j)
        if (j < K) a.ws.dEg[r0 + j] = dE[j];
    }
    if (ov) {
      // the sampling-side coefficient of each row, weights folded in:
      // w_s dE^s/da + w_tv / K_n (the TV term's derivative, with the sign of -a^s)
      if (a.sampling) Es = window_term(as, kn, dE);
      const float tvc = (a.tv && kn > 0) ? a.w_tv / (float)kn : 0.f;
      float tsum = 0.f;
#pragma unroll
      for (int j = 0; j < AAL_MAX_K; ++j) {
        if (j < K) a.ws.dEs[r0 + j] = __fadd_rn(a.sampling ? __fmul_rn(a.w_sampling, dE[j]) : 0.f, j < kn ? tvc : 0.f);
        if (j < kn) tsum += 1.f - as[j];
      }
      if (a.tv && kn > 0) tvs = tsum / (float)kn;
    }
    if (a.eal != nullptr) {
      a.eal[2 * n + 0] = Eg;
      a.eal[2 * n + 1] = Es;
    }
    eg = Eg;
    es = Es;
    if (a.kl) {
      // the anchor: every valid position (row) of the window, whatever its prefix
      float s = 0.f;
      int c = 0;
      for (int j = 0; j < K; ++j) {
        if (a.mask == nullptr || a.mask[r0 + j] != 0) {
          s += a.ws.kl[r0 + j];
          ++c;
        }
      }
      ksum = s;
      kcnt = c;
    }
  }
  double x[kSums] = {eg, es, valid, ksum, kcnt, tvs};
  finish_loss(a, x, sm, &is_last);
}

// ---------------------------------------------------------------- sequence layout
// Window n = b*T + t starts at position t of sequence b and covers t..t+K-1 (Sec. 3.3, the
// window slides by one), stopping at the first invalid position or the end of the sequence;
// with full_windows a window that stops before K positions is left out of W.  Rows are
// positions, so the window's depth-j row is row n + j.

__device__ __forceinline__ float row_overlap(const LossWs& ws, int64_t r, int cluster, float* qlt) {
  float2 t = ws.cpart[r * kMaxCluster];
  for (int c = 1; c < cluster; ++c) {
    const float2 u = ws.cpart[r * kMaxCluster + c];
    t.x += u.x;
    t.y += u.y;
  }
  if (qlt) *qlt = t.y;
  return t.x;
}

__global__ void __launch_bounds__(kWindowThreads) seq_window_kernel(SeqWindowArgs a) {
  __shared__ double sm[kSums * kWindowThreads / 32];
  __shared__ bool is_last;
  const int64_t N = a.B * a.T;
  const int64_t n = (int64_t)blockIdx.x * kWindowThreads + threadIdx.x;
  double eg = 0.0, es = 0.0, valid = 0.0, ksum = 0.0, kcnt = 0.0, tvs = 0.0;
  const bool ov = a.sampling || a.tv;
  if (n < N) {
    const int K = a.K;
    const int64_t t = n % a.T;
    int kn = 0;
    while (kn < K && t + kn < a.T && (a.mask == nullptr || a.mask[n + kn] != 0)) ++kn;
    if (a.full_windows && kn < K) kn = 0;
    valid = kn >= 1 ? 1.0 : 0.0;
    // this window's first row is position n: finish its per-row overlap sums here
    if (ov) {
      float q;
      a.ws.as[n] = row_overlap(a.ws, n, a.cluster, &q);
      a.ws.qlt[n] = q;
    }
    float ag[AAL_MAX_K], as[AAL_MAX_K], dE[AAL_MAX_K];
#pragma unroll
    for (int j = 0; j < AAL_MAX_K; ++j) {
      ag[j] = 0.f;
      as[j] = 0.f;
      if (j < kn) {
        if (a.greedy) ag[j] = a.ws.ag[n + j];
        if (ov) as[j] = row_overlap(a.ws, n + j, a.cluster, nullptr);
      }
    }
    float Eg = 0.f, Es = 0.f;
    if (a.greedy) {
      Eg = window_term(ag, kn, dE);
#pragma unroll
      for (int j = 0; j < AAL_MAX_K; ++j)
        if (j < K) a.pg[n * K + j] = dE[j];
    }
    if (ov) {  // weighted partials, as in window_kernel
      if (a.sampling) Es = window_term(as, kn, dE);
      const float tvc = (a.tv && kn > 0) ? a.w_tv / (float)kn : 0.f;
      float tsum = 0.f;
#pragma unroll
      for (int j = 0; j < AAL_MAX_K; ++j) {
        if (j < K) a.ps[n * K + j] = __fadd_rn(a.sampling ? __fmul_rn(a.w_sampling, dE[j]) : 0.f, j < kn ? tvc : 0.f);
        if (j < kn) tsum += 1.f - as[j];
      }
      if (a.tv && kn > 0) tvs = tsum / (float)kn;
    }
    if (a.eal != nullptr) {
      a.eal[2 * n + 0] = Eg;
      a.eal[2 * n + 1] = Es;
    }
    eg = Eg;
    es = Es;
    if (a.kl && (a.mask == nullptr || a.mask[n] != 0)) {  // the anchor: position n itself
      ksum = a.ws.kl[n];
      kcnt = 1.0;
    }
  }
  double x[kSums] = {eg, es, valid, ksum, kcnt, tvs};
  finish_loss(a, x, sm, &is_last);
}

// dE/da of position p: the partials of the windows t = p - j (j < K, same sequence) that
// reach it, added in increasing j.
__global__ void __launch_bounds__(256) seq_gather_kernel(SeqWindowArgs a) {
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= a.B * a.T) return;
  const int64_t t = p % a.T;
  const int K = a.K;
  float g = 0.f, s = 0.f;
  for (int j = 0; j < K && j <= t; ++j) {
    const int64_t n = p - j;
    if (a.greedy) g += a.pg[n * K + j];
    if (a.sampling || a.tv) s += a.ps[n * K + j];
  }
  a.ws.dEg[p] = g;
  a.ws.dEs[p] = s;
}

}  // namespace

cudaError_t launch_seq_window(const SeqWindowArgs& a, cudaStream_t s) {
  if (a.nwblk < 1) return cudaSuccess;
  seq_window_kernel<<<(unsigned)a.nwblk, kWindowThreads, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t rows = a.B * a.T;
  seq_gather_kernel<<<(unsigned)((rows + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_window(const WindowArgs& a, cudaStream_t s) {
  if (a.nwblk < 1) return cudaSuccess;
  window_kernel<<<(unsigned)a.nwblk, kWindowThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace aal
