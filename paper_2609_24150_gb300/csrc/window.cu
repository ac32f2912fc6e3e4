// Window combination of the per-position acceptances into the losses.
//
// Per window n with K_n leading valid depths (Sec. 3.1, Eq. eal_generic):
//   E_n = sum_{k=1}^{K_n} P_k,   P_k = prod_{j<k} a_{n,j}
//   dE_n/da_{n,j} = P_j * S_j,  S_{K_n-1} = 1,  S_j = 1 + a_{n,j+1} S_{j+1}   (j < K_n)
// for the greedy term (a^greedy, Eq. loss_eal) and the sampling term (a^sample,
// Eq. loss_tv).  The partials go to the workspace for the backward; the loss
// L = -(w_g sum E^g + w_s sum E^s) / |W| is summed deterministically: each block
// reduces its windows in a fixed tree, and the last block to finish adds the
// block partials in index order.
#include "aal_internal.cuh"

namespace aal {
namespace {

template <int NT>
__device__ __forceinline__ void block_sum3(double& x, double& y, double& z, double* sm) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    x += __shfl_xor_sync(0xffffffffu, x, off);
    y += __shfl_xor_sync(0xffffffffu, y, off);
    z += __shfl_xor_sync(0xffffffffu, z, off);
  }
  if (lane == 0) {
    sm[3 * warp + 0] = x;
    sm[3 * warp + 1] = y;
    sm[3 * warp + 2] = z;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    x = sm[0];
    y = sm[1];
    z = sm[2];
    for (int w = 1; w < NT / 32; ++w) {
      x += sm[3 * w + 0];
      y += sm[3 * w + 1];
      z += sm[3 * w + 2];
    }
  }
  __syncthreads();
}

// Expected length and its partials for one window term; returns E.
__device__ __forceinline__ float window_term(const float* a, int kn, float* dE) {
  float P[AAL_MAX_K + 1];
  P[0] = 1.f;
  float E = 0.f;
#pragma unroll
  for (int j = 0; j < AAL_MAX_K; ++j) {
    if (j < kn) {
      P[j + 1] = P[j] * a[j];
      E += P[j + 1];
    }
  }
  float S = 1.f;
#pragma unroll
  for (int j = AAL_MAX_K - 1; j >= 0; --j) {
    if (j < kn) {
      dE[j] = P[j] * S;
      S = 1.f + a[j] * S;
    } else {
      dE[j] = 0.f;
    }
  }
  return E;
}

__global__ void __launch_bounds__(kWindowThreads) window_kernel(WindowArgs a) {
  __shared__ double sm[3 * kWindowThreads / 32];
  __shared__ bool is_last;
  const int64_t n = (int64_t)blockIdx.x * kWindowThreads + threadIdx.x;
  double eg = 0.0, es = 0.0, valid = 0.0;
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
        if (a.sampling) {
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
    if (a.sampling) {
      Es = window_term(as, kn, dE);
#pragma unroll
      for (int j = 0; j < AAL_MAX_K; ++j)
        if (j < K) a.ws.dEs[r0 + j] = dE[j];
    }
    if (a.eal != nullptr) {
      a.eal[2 * n + 0] = Eg;
      a.eal[2 * n + 1] = Es;
    }
    eg = Eg;
    es = Es;
  }
  block_sum3<kWindowThreads>(eg, es, valid, sm);
  if (threadIdx.x == 0) {
    a.ws.wpart[4 * blockIdx.x + 0] = eg;
    a.ws.wpart[4 * blockIdx.x + 1] = es;
    a.ws.wpart[4 * blockIdx.x + 2] = valid;
    __threadfence();
    const unsigned ticket = atomicAdd(&a.ws.hdr->done_blocks, 1u);
    is_last = (ticket == gridDim.x - 1);
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  // last block: add the block partials in a fixed order
  double sg = 0.0, ss = 0.0, sv = 0.0;
  const volatile double* wp = a.ws.wpart;
  for (int64_t b = threadIdx.x; b < a.nwblk; b += kWindowThreads) {
    sg += wp[4 * b + 0];
    ss += wp[4 * b + 1];
    sv += wp[4 * b + 2];
  }
  block_sum3<kWindowThreads>(sg, ss, sv, sm);
  if (threadIdx.x == 0) {
    const int nvalid = (int)sv;
    const double num = (a.greedy ? (double)a.w_greedy * sg : 0.0) +
                       (a.sampling ? (double)a.w_sampling * ss : 0.0);
    const float loss = nvalid > 0 ? (float)(-num / (double)nvalid) : 0.f;
    *a.loss = loss;
    a.ws.hdr->loss = loss;
    a.ws.hdr->nvalid = nvalid;
    a.ws.hdr->cluster = a.cluster;
    a.ws.hdr->done_blocks = 0u;
  }
}

}  // namespace

cudaError_t launch_window(const WindowArgs& a, cudaStream_t s) {
  if (a.nwblk < 1) return cudaSuccess;
  window_kernel<<<(unsigned)a.nwblk, kWindowThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace aal
