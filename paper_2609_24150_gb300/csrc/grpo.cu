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
    // the window's rows: n*K + k, or (sequence layout) positions start + k, whose bounds the
    // gather kernel has checked (a bad start reads position 0 here and is reported there)
    int64_t row0 = t * K;
    if (a.starts != nullptr) {
      const int64_t st = a.starts[t];
      row0 = (st >= 0 && st + K <= a.RP) ? st : 0;
    }
    float sum = 0.f;
    for (int k = 0; k < K; ++k) {
      const int64_t r = row0 + k;
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
    float* out = a.starts != nullptr ? a.cw + t * K : a.lws.cgr + t * K;
    for (int k = 0; k < K; ++k) out[k] = coef;
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

// Sequence layout: each window row (n, k) takes the flags of position starts[n] + k.  A start
// outside [0, RP - K], across a sequence end, or below the previous one records
// AAL_ERR_INVALID_ARG and its rows read nothing (flags 0).
__global__ void __launch_bounds__(256) seq_grpo_gather(SeqGrpoArgs a) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= a.N * a.K) return;
  const int64_t n = i / a.K;
  const int k = (int)(i - n * a.K);
  const int64_t st = a.starts[n];
  const bool ok = st >= 0 && st + a.K <= a.RP && (st % a.T) + a.K <= a.T && (n == 0 || a.starts[n - 1] <= st);
  if (!ok && k == 0) atomicExch(&a.hdr->status, 1u);  // == AAL_ERR_INVALID_ARG
  a.acc[i] = ok ? a.acc_pos[st + k] : 0;
  a.acc_ref[i] = ok ? a.accr_pos[st + k] : 0;
}

// Per position p: the coefficients of the window rows that land on it, windows in start order
// (starts ascending, so they are the windows with start in [p - K + 1, p], found by binary
// search): a fixed order of at most K terms, no atomics.
__global__ void __launch_bounds__(256) seq_grpo_scatter(SeqGrpoArgs a) {
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= a.RP) return;
  const int64_t lo_start = p - a.K + 1;
  int64_t lo = 0, hi = a.N;  // first window with start >= lo_start
  while (lo < hi) {
    const int64_t mid = (lo + hi) >> 1;
    if (a.starts[mid] < lo_start) lo = mid + 1;
    else hi = mid;
  }
  float c = 0.f;
  for (int64_t n = lo; n < a.N && a.starts[n] <= p; ++n) {
    const int64_t k = p - a.starts[n];
    if (k >= 0 && k < a.K) c += a.cw[n * a.K + k];
  }
  a.cgr[p] = c;
}

cudaError_t launch_seq_grpo_gather(const SeqGrpoArgs& a, cudaStream_t s) {
  const int64_t n = a.N * a.K;
  if (n < 1) return cudaSuccess;
  seq_grpo_gather<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_seq_grpo_scatter(const SeqGrpoArgs& a, cudaStream_t s) {
  if (a.RP < 1) return cudaSuccess;
  seq_grpo_scatter<<<(unsigned)((a.RP + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_grpo_windows(const GrpoWindowArgs& a, cudaStream_t s) {
  if (a.nblk < 1) return cudaSuccess;
  grpo_windows<<<(unsigned)a.nblk, kGrpoThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace aal
