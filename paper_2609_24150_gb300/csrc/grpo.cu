// The GRPO surrogate of Sec. 3.4 on top of a completed loss forward.
//
// The loss forward has already streamed z_p and z_theta and left, per row, x* = argmax z_p,
// the draft's greedy token y = S_k = argmax z_theta and the draft's T = 1 normaliser, so
// log pi_theta(y) = -ln 2 * Ls_q1 (y is where z_theta peaks).  What is left needs the
// reference draft only:
//   one-tensor pass one pass over z_ref (onetensor.cu, mode REF): its normaliser, its own
//                   greedy token (for tau^ref) and z_ref(y), giving log pi_ref(y) and both
//                   acceptance flags;
//   reward_groups   tau, tau^ref, R = tau - tau^ref, rollout means, clipped advantages
//                   (the kernel of aal_accept_reward);
//   grpo_windows    per window: log rho = (1/K) sum_k [log pi_theta(y_k) - log pi_ref(y_k)]
//                   clipped to +-log_rho_clip, rho = exp(log rho) clipped to [rho_min, rho_max],
//                   the surrogate min(rho A, clip(rho, 1 - eps, 1 + eps) A), L_GRPO = -mean,
//                   and per row the coefficient of d log pi_theta(y)/dz = delta_{u,y} - q(u)
//                   that the loss backward adds:  w_grpo (-1/N) A rho / K where the unclipped
//                   term is the minimum and every clip is inside, else 0.
// The group loss is the mean over a group's windows and L_GRPO the mean over equal-sized
// groups, which is -(1/N) sum_t surrogate_t.
#include "aal_internal.cuh"

namespace aal {
namespace {

__global__ void __launch_bounds__(kGrpoThreads) grpo_windows(GrpoWindowArgs a) {
  __shared__ double sm[kGrpoThreads / 32];
  __shared__ bool is_last;
  const int64_t t = (int64_t)blockIdx.x * kGrpoThreads + threadIdx.x;
  double surr = 0.0;
  if (t < a.N) {
    const int K = a.K;
    float sum = 0.f;
    for (int k = 0; k < K; ++k) {
      const int64_t r = t * K + k;
      sum += -kLn2 * a.lws.Lsq1[r] - a.lpr[r];
    }
    const float raw = sum / (float)K;
    const float lr = fminf(fmaxf(raw, -a.log_rho_clip), a.log_rho_clip);
    const float rho_e = expf(lr);
    const float rho = fminf(fmaxf(rho_e, a.rho_min), a.rho_max);
    const float A = a.adv[t / a.wpr];
    const float lo = 1.f - a.eps_clip, hi = 1.f + a.eps_clip;
    const float s = fminf(rho * A, fminf(fmaxf(rho, lo), hi) * A);
    const bool unclipped = (A >= 0.f && rho <= hi) || (A < 0.f && rho >= lo);
    const bool inside = raw >= -a.log_rho_clip && raw <= a.log_rho_clip && rho_e >= a.rho_min &&
                        rho_e <= a.rho_max;
    const float coef = (unclipped && inside) ? a.w_grpo * (-1.f / (float)a.N) * A * rho_e / (float)K : 0.f;
    for (int k = 0; k < K; ++k) a.lws.cgr[t * K + k] = coef;
    if (a.log_rho != nullptr) a.log_rho[t] = lr;
    surr = s;
  }
  // fixed-order block sum, then the last block adds the block partials in order
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) surr += __shfl_xor_sync(0xffffffffu, surr, off);
  if (lane == 0) sm[warp] = surr;
  __syncthreads();
  if (threadIdx.x == 0) {
    double b = sm[0];
    for (int w = 1; w < kGrpoThreads / 32; ++w) b += sm[w];
    a.part[blockIdx.x] = b;
    __threadfence();
    const unsigned ticket = atomicAdd(&a.hdr->done_blocks, 1u);
    is_last = (ticket == gridDim.x - 1);
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    const volatile double* p = a.part;
    double tot = 0.0;
    for (int64_t b = 0; b < a.nblk; ++b) tot += p[b];
    const float loss = a.N > 0 ? (float)(-tot / (double)a.N) : 0.f;
    *a.loss = loss;
    a.hdr->loss = loss;
    a.hdr->done_blocks = 0u;
  }
}

}  // namespace

cudaError_t launch_grpo_windows(const GrpoWindowArgs& a, cudaStream_t s) {
  if (a.nblk < 1) return cudaSuccess;
  grpo_windows<<<(unsigned)a.nblk, kGrpoThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace aal
