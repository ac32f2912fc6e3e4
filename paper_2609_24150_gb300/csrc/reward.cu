// Simulated acceptance reward of the GRPO stage (Sec. 3.4).
//
// Row kernel, per logit row r = (window n, depth k), one pass over V:
//   S_k = argmax z_q (greedy draft trajectory), x*_k = argmax z_p, S^ref_k = argmax z_ref,
//   lowest index on ties.  Greedy verification accepts iff S_k == x*_k.  Sampling
//   verification accepts iff u < min(1, p~(S_k)/q~(S_k)) (Sec. 2.3), with
//   u = Philox4x32-10(counter (n_lo, n_hi, k, 0), key seed) and n the global window
//   index; it needs the log-sum-exps of z_p/T and z_q/T, streamed online.  With a sampled
//   draft (sampled_draft) S_k is instead drawn from q~ by the Gumbel-max method: S_k =
//   argmax_v (z_q(v)/T + G_v), G_v = -ln(-ln U_v), U_v from counter (n_lo, n_hi, k, 1 + v/4)
//   word v mod 4; the reference draft draws with the same G (common random numbers).
// Group kernel, per group of rollouts:
//   tau = sum_{k=1}^{K} prod_{j<=k} accept_j (the leading run), R = tau - tau^ref
//   (Eq. debiased_reward), rollout length = mean R over the rollout's windows,
//   A = clip((x - mean)/(std + 1e-6), -C_A, C_A) with the population std (Eq. advantage).
#include "ptx.cuh"

namespace aal {
namespace {

constexpr int kRowThreads = 256;
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kGroupThreads = 256;

template <typename T>
__device__ __forceinline__ void unpack_any(const uint4& w, float* o);
template <>
__device__ __forceinline__ void unpack_any<float>(const uint4& w, float* o) {
  o[0] = __uint_as_float(w.x);
  o[1] = __uint_as_float(w.y);
  o[2] = __uint_as_float(w.z);
  o[3] = __uint_as_float(w.w);
}
template <>
__device__ __forceinline__ void unpack_any<uint16_t>(const uint4& w, float* o) {
  o[0] = bf16_lo(w.x);
  o[1] = bf16_hi(w.x);
  o[2] = bf16_lo(w.y);
  o[3] = bf16_hi(w.y);
  o[4] = bf16_lo(w.z);
  o[5] = bf16_hi(w.z);
  o[6] = bf16_lo(w.w);
  o[7] = bf16_hi(w.w);
}

struct RowState {
  Amax q, p, r;  // draft (carry: z_p at its argmax), target, reference (carry: z_p)
  Lse lp, lq, lr;
};

// Running best of a perturbed key (Gumbel-max), with z of the drawn tensor and z_p there.
struct Draw {
  float key;
  int32_t i;
  float z, zp;
};
__device__ __forceinline__ void draw_init(Draw& d) {
  d.key = -INFINITY;
  d.i = 0x7fffffff;
  d.z = 0.f;
  d.zp = 0.f;
}
__device__ __forceinline__ Draw draw_merge(const Draw& a, const Draw& b) {
  return (b.key > a.key || (b.key == a.key && b.i < a.i)) ? b : a;
}
__device__ __forceinline__ Draw shfl_draw(const Draw& a, int off) {
  Draw b;
  b.key = __shfl_xor_sync(0xffffffffu, a.key, off);
  b.i = __shfl_xor_sync(0xffffffffu, a.i, off);
  b.z = __shfl_xor_sync(0xffffffffu, a.z, off);
  b.zp = __shfl_xor_sync(0xffffffffu, a.zp, off);
  return b;
}
__device__ __forceinline__ void draw_push(Draw& d, float key, int64_t v, float z, float zp) {
  if (key > d.key) {
    d.key = key;
    d.i = (int32_t)v;
    d.z = z;
    d.zp = zp;
  }
}
// The Gumbel noise in log2 units: G log2(e) = -log2(-ln U) = -log2(-ln2 * log2 U).  Both
// logarithms see normal numbers only: U >= 2^-24, and -ln2 * log2 U >= 5.9e-8 (U <= 1 - 2^-24).
__device__ __forceinline__ float gumbel2(float U) { return -lg2(-kLn2 * lg2(U)); }

__device__ __forceinline__ RowState merge_state(const RowState& a, const RowState& b, float sT) {
  RowState o;
  o.q = amax_merge(a.q, b.q);
  o.p = amax_merge(a.p, b.p);
  o.r = amax_merge(a.r, b.r);
  o.lp = lse_merge(a.lp, b.lp, sT);
  o.lq = lse_merge(a.lq, b.lq, sT);
  o.lr = lse_merge(a.lr, b.lr, sT);
  return o;
}

__device__ __forceinline__ RowState shfl_state(const RowState& a, int off) {
  RowState o;
  o.q = shfl_amax(a.q, off);
  o.p = shfl_amax(a.p, off);
  o.r = shfl_amax(a.r, off);
  o.lp = shfl_lse(a.lp, off);
  o.lq = shfl_lse(a.lq, off);
  o.lr = shfl_lse(a.lr, off);
  return o;
}

__device__ __forceinline__ void init_state(RowState& s) {
  amax_init(s.q);
  amax_init(s.p);
  amax_init(s.r);
  lse_init(s.lp);
  lse_init(s.lq);
  lse_init(s.lr);
}

template <typename T, bool VEC, bool SAMPLING, bool REF, bool SAMPLED = false>
__global__ void __launch_bounds__(kRowThreads) reward_rows(RewardRowArgs a) {
  __shared__ RowState red[kRowWarps];
  __shared__ Draw dred[2][kRowWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
    const T* zq = static_cast<const T*>(a.zq) + r * a.V;
    const T* zp = static_cast<const T*>(a.zp) + r * a.V;
    const T* zr = REF ? static_cast<const T*>(a.zr) + r * a.V : nullptr;
    RowState st;
    init_state(st);
    Draw dq, dr;  // sampled draft tokens (SAMPLED)
    draw_init(dq);
    draw_init(dr);
    const int64_t n_glob = a.row_offset + r / a.K;
    const uint32_t k_depth = (uint32_t)(r % a.K);
    auto draw = [&](int64_t v, float q, float p, float rr, float U) {
      const float g = gumbel2(U);
      draw_push(dq, fmaf(q, a.sT, g), v, q, p);
      if (REF) draw_push(dr, fmaf(rr, a.sT, g), v, rr, p);
    };
    auto visit = [&](int64_t v, float q, float p, float rr) {
      if (q > st.q.v) {
        st.q.v = q;
        st.q.i = (int32_t)v;
        st.q.carry = p;
      }
      if (p > st.p.v) {
        st.p.v = p;
        st.p.i = (int32_t)v;
      }
      if (REF && rr > st.r.v) {
        st.r.v = rr;
        st.r.i = (int32_t)v;
        st.r.carry = p;
      }
      if (SAMPLING) {
        lse_push(st.lp, p, a.sT);
        lse_push(st.lq, q, a.sT);
        if (REF) lse_push(st.lr, rr, a.sT);
      }
    };
    if (VEC) {
      constexpr int E = 16 / sizeof(T);
      const int64_t nv = a.V / E;
      for (int64_t i = threadIdx.x; i < nv; i += kRowThreads) {
        float qv[E], pv[E], rv[E];
        unpack_any<T>(ldg_stream(reinterpret_cast<const uint4*>(zq) + i), qv);
        unpack_any<T>(ldg_stream(reinterpret_cast<const uint4*>(zp) + i), pv);
        if (REF) unpack_any<T>(ldg_stream(reinterpret_cast<const uint4*>(zr) + i), rv);
#pragma unroll
        for (int e = 0; e < E; ++e) visit(i * E + e, qv[e], pv[e], REF ? rv[e] : 0.f);
        if (SAMPLED) {  // E is a multiple of 4: whole counters
#pragma unroll
          for (int h = 0; h < E / 4; ++h) {
            const int64_t v0 = i * E + 4 * h;
            const float4 U = philox_uniform4(a.seed, (uint64_t)n_glob, k_depth, (uint32_t)(1 + v0 / 4));
            draw(v0 + 0, qv[4 * h + 0], pv[4 * h + 0], REF ? rv[4 * h + 0] : 0.f, U.x);
            draw(v0 + 1, qv[4 * h + 1], pv[4 * h + 1], REF ? rv[4 * h + 1] : 0.f, U.y);
            draw(v0 + 2, qv[4 * h + 2], pv[4 * h + 2], REF ? rv[4 * h + 2] : 0.f, U.z);
            draw(v0 + 3, qv[4 * h + 3], pv[4 * h + 3], REF ? rv[4 * h + 3] : 0.f, U.w);
          }
        }
      }
    } else {
      for (int64_t v = threadIdx.x; v < a.V; v += kRowThreads) {
        const float q = load_elem<T>(zq + v), p = load_elem<T>(zp + v), rr = REF ? load_elem<T>(zr + v) : 0.f;
        visit(v, q, p, rr);
        if (SAMPLED) {
          const float4 U4 = philox_uniform4(a.seed, (uint64_t)n_glob, k_depth, (uint32_t)(1 + v / 4));
          const int w = (int)(v & 3);
          draw(v, q, p, rr, w == 0 ? U4.x : w == 1 ? U4.y : w == 2 ? U4.z : U4.w);
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) st = merge_state(st, shfl_state(st, off), a.sT);
    if (SAMPLED) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        dq = draw_merge(dq, shfl_draw(dq, off));
        if (REF) dr = draw_merge(dr, shfl_draw(dr, off));
      }
      if (lane == 0) {
        dred[0][warp] = dq;
        dred[1][warp] = dr;
      }
    }
    if (lane == 0) red[warp] = st;
    __syncthreads();
    if (threadIdx.x == 0) {
      RowState t = red[0];
      for (int w = 1; w < kRowWarps; ++w) t = merge_state(t, red[w], a.sT);
      uint8_t acc, acc_ref = 0;
      if (!SAMPLING) {
        acc = (t.q.i == t.p.i) ? 1 : 0;
        if (REF) acc_ref = (t.r.i == t.p.i) ? 1 : 0;
      } else {
        const int64_t n = r / a.K;
        const uint32_t k = (uint32_t)(r - n * a.K);
        const float u = philox_uniform(a.seed, (uint64_t)(a.row_offset + n), k);
        const float Lsp = lse_ls(t.lp), Lsq = lse_ls(t.lq);
        // the drafted token S: the draft's argmax, or its Gumbel-max draw
        float zqS = t.q.v, zpS = t.q.carry, zrS = t.r.v, zpR = t.r.carry;
        if (SAMPLED) {
          Draw bq = dred[0][0], br = dred[1][0];
          for (int w = 1; w < kRowWarps; ++w) {
            bq = draw_merge(bq, dred[0][w]);
            if (REF) br = draw_merge(br, dred[1][w]);
          }
          zqS = bq.z;
          zpS = bq.zp;
          zrS = br.z;
          zpR = br.zp;
        }
        // log2 p~(S) - log2 q~(S)
        const float d = log2_prob(zpS, a.sT, t.lp.M, Lsp) - log2_prob(zqS, a.sT, t.lq.M, Lsq);
        acc = (u < exp2f(fminf(d, 0.f))) ? 1 : 0;
        if (REF) {
          const float Lsr = lse_ls(t.lr);
          const float dr = log2_prob(zpR, a.sT, t.lp.M, Lsp) - log2_prob(zrS, a.sT, t.lr.M, Lsr);
          acc_ref = (u < exp2f(fminf(dr, 0.f))) ? 1 : 0;
        }
      }
      a.acc[r] = acc;
      if (REF) a.acc_ref[r] = acc_ref;
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- sampled draft, vector path
// The sampled-draft reward is bound by arithmetic, not bytes: one Philox4x32-10 call per four
// vocabulary entries and two logarithms per entry.  This path keeps everything per 16-byte vector
// and branch-free: the log-sum-exps fold a vector's values after one rescale to the vector maximum
// (as in the streamed forward), the Gumbel keys of a vector are maxed first and the element is
// looked up only when the vector beats the running best, and the first Philox round, whose two
// products depend only on the row (window, depth), is computed once per row.
struct PhiloxRow {
  uint32_t x0, x1, x2k, x3;  // round-1 output except the c3 term: x2 = x2k ^ c3
  uint32_t k0[10], k1[10];   // round keys
};

__device__ __forceinline__ PhiloxRow philox_row(uint64_t seed, uint64_t n, uint32_t k) {
  PhiloxRow P;
  uint32_t a = (uint32_t)seed, b = (uint32_t)(seed >> 32);
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    P.k0[r] = a;
    P.k1[r] = b;
    a += 0x9E3779B9u;
    b += 0xBB67AE85u;
  }
  const uint32_t c0 = (uint32_t)n, c1 = (uint32_t)(n >> 32), c2 = k;
  const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
  const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
  P.x0 = hi1 ^ c1 ^ P.k0[0];
  P.x1 = lo1;
  P.x2k = hi0 ^ P.k1[0];
  P.x3 = lo0;
  return P;
}

// The four words of counter (n_lo, n_hi, k, c3): rounds 2..10 after the row's round 1.
__device__ __forceinline__ uint4 philox_rest(const PhiloxRow& P, uint32_t c3) {
  uint4 c = make_uint4(P.x0, P.x1, P.x2k ^ c3, P.x3);
#pragma unroll
  for (int r = 1; r < 10; ++r) {
    // each 32 x 32 -> 64 product in one multiply: high and low halves together
    const uint64_t p0 = (uint64_t)0xD2511F53u * c.x, p1 = (uint64_t)0xCD9E8D57u * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ P.k0[r], (uint32_t)p1, (uint32_t)(p0 >> 32) ^ c.w ^ P.k1[r],
                   (uint32_t)p0);
  }
  return c;
}

// ((w >> 9) * 2 + 1) * 2^-24 without an integer-to-float conversion: the 23 high bits as the
// mantissa of a float in [1, 2), minus (1 - 2^-24) (exact: the result is an odd multiple of
// 2^-24 below 1).
__device__ __forceinline__ float word_uniform(uint32_t w) {
  return __uint_as_float(0x3F800000u | (w >> 9)) - 0.99999994039535522461f;
}

// Fold E values into (M, S) at scale s after one rescale to max(M, vector max).
template <int E>
__device__ __forceinline__ void lse_fold(Lse& L, const float* z, float s) {
  float vm = z[0];
#pragma unroll
  for (int e = 1; e < E; ++e) vm = fmaxf(vm, z[e]);
  const float m = fmaxf(L.M, vm);
  float acc = 0.f;
#pragma unroll
  for (int e = 0; e < E; ++e) acc += ex2((z[e] - m) * s);
  L.S = L.S * ex2((L.M - m) * s) + acc;
  L.M = m;
}

// Offer E Gumbel keys of one vector (elements v0 ..) to a running draw; the target's vector
// (pw, packed) is unpacked only when the vector wins.
template <typename T, int E>
__device__ __forceinline__ void draw_fold(Draw& d, const float* key, const float* z, const uint4& pw, int64_t v0) {
  float km = key[0];
#pragma unroll
  for (int e = 1; e < E; ++e) km = fmaxf(km, key[e]);
  if (km > d.key) {  // rare once the running best has settled
    int at = 0;
#pragma unroll
    for (int e = E - 1; e >= 0; --e)
      if (key[e] == km) at = e;
    float zp[E];
    unpack_any<T>(pw, zp);
    float zz = z[0], pp = zp[0];
#pragma unroll
    for (int e = 1; e < E; ++e)
      if (e == at) {
        zz = z[e];
        pp = zp[e];
      }
    d.key = km;
    d.i = (int32_t)(v0 + at);
    d.z = zz;
    d.zp = pp;
  }
}

// lse_fold for a bf16 vector in its packed form: the maximum by max.bf16x2, z - m with the bf16
// widened inside the add, the scale and the sums on f32 pairs.
__device__ __forceinline__ void lse_fold_bf16(Lse& L, const uint4& w, float s) {
  const uint32_t mw = ptx::bmax2(ptx::bmax2(w.x, w.y), ptx::bmax2(w.z, w.w));
  const float m = fmaxf(L.M, fmaxf(bf16_lo(mw), bf16_hi(mw)));
  const float nm = -m;
  const float2 s2 = make_float2(s, s), zero2 = make_float2(0.f, 0.f);
  const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
  float2 acc = zero2;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float2 x = ptx::f2fma(make_float2(bf16lo_add(ww[k], nm), bf16hi_add(ww[k], nm)), s2, zero2);
    acc = ptx::f2add(acc, make_float2(ex2(x.x), ex2(x.y)));
  }
  L.S = L.S * ex2((L.M - m) * s) + (acc.x + acc.y);
  L.M = m;
}

// Four blocks an SM for both instances: measured against five (without the reference draft,
// 48 registers) and three (with it, 72 registers and no spill), both slower.
// STATS: the normalisers of z_p/T and z_q/T come from a loss forward's workspace (a.lws), so only
// the draft is streamed (for the draws) and the target is read at the drawn token alone.
template <typename T, bool REF, bool STATS = false>
__global__ void __launch_bounds__(kRowThreads, 4) reward_sampled_rows(RewardRowArgs a) {
  __shared__ RowState red[kRowWarps];
  __shared__ Draw dred[2][kRowWarps];
  constexpr int E = 16 / sizeof(T);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
    const uint4* q4 = reinterpret_cast<const uint4*>(static_cast<const T*>(a.zq) + r * a.V);
    const uint4* p4 = reinterpret_cast<const uint4*>(static_cast<const T*>(a.zp) + r * a.V);
    const uint4* r4 = REF ? reinterpret_cast<const uint4*>(static_cast<const T*>(a.zr) + r * a.V) : nullptr;
    const int64_t n_glob = a.row_offset + r / a.K;
    const uint32_t k_depth = (uint32_t)(r % a.K);
    const PhiloxRow P = philox_row(a.seed, (uint64_t)n_glob, k_depth);
    RowState st;
    init_state(st);
    // running maxima start at a finite floor, so lse_fold needs no -inf case (a -inf logit
    // then adds 2^(-inf) = 0)
    st.lp.M = st.lq.M = st.lr.M = -1e30f;
    Draw dq, dr;
    draw_init(dq);
    draw_init(dr);
    const int64_t nv = a.V / E;
    for (int64_t i = threadIdx.x; i < nv; i += kRowThreads) {
      float qv[E], pv[E], rv[E], g[E], kq[E], kr[E];
      const uint4 qw = ldg_stream(q4 + i);
      const uint4 pw = STATS ? make_uint4(0, 0, 0, 0) : ldg_stream(p4 + i);
      uint4 rw = make_uint4(0, 0, 0, 0);
      if (REF) rw = ldg_stream(r4 + i);
      unpack_any<T>(qw, qv);
      if (sizeof(T) != 2 && !STATS) unpack_any<T>(pw, pv);  // (the bf16 path folds z_p packed)
      if (REF) unpack_any<T>(rw, rv);
#pragma unroll
      for (int h = 0; h < E / 4; ++h) {
        const uint4 w = philox_rest(P, (uint32_t)(1 + (i * E) / 4 + h));
        g[4 * h + 0] = gumbel2(word_uniform(w.x));
        g[4 * h + 1] = gumbel2(word_uniform(w.y));
        g[4 * h + 2] = gumbel2(word_uniform(w.z));
        g[4 * h + 3] = gumbel2(word_uniform(w.w));
      }
#pragma unroll
      for (int e = 0; e < E; ++e) {
        kq[e] = fmaf(qv[e], a.sT, g[e]);
        if (REF) kr[e] = fmaf(rv[e], a.sT, g[e]);
      }
      draw_fold<T, E>(dq, kq, qv, pw, i * E);
      if (REF) draw_fold<T, E>(dr, kr, rv, pw, i * E);
      if (STATS) {
        // (the normalisers are the loss forward's)
      } else if (sizeof(T) == 2) {
        lse_fold_bf16(st.lp, pw, a.sT);
        lse_fold_bf16(st.lq, qw, a.sT);
        if (REF) lse_fold_bf16(st.lr, rw, a.sT);
      } else {
        lse_fold<E>(st.lp, pv, a.sT);
        lse_fold<E>(st.lq, qv, a.sT);
        if (REF) lse_fold<E>(st.lr, rv, a.sT);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      if (!STATS) {
        st.lp = lse_merge(st.lp, shfl_lse(st.lp, off), a.sT);
        st.lq = lse_merge(st.lq, shfl_lse(st.lq, off), a.sT);
      }
      if (REF) st.lr = lse_merge(st.lr, shfl_lse(st.lr, off), a.sT);
      dq = draw_merge(dq, shfl_draw(dq, off));
      if (REF) dr = draw_merge(dr, shfl_draw(dr, off));
    }
    if (lane == 0) {
      red[warp] = st;
      dred[0][warp] = dq;
      dred[1][warp] = dr;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      RowState t = red[0];
      Draw bq = dred[0][0], br = dred[1][0];
      for (int w = 1; w < kRowWarps; ++w) {
        if (!STATS) {
          t.lp = lse_merge(t.lp, red[w].lp, a.sT);
          t.lq = lse_merge(t.lq, red[w].lq, a.sT);
        }
        if (REF) t.lr = lse_merge(t.lr, red[w].lr, a.sT);
        bq = draw_merge(bq, dred[0][w]);
        if (REF) br = draw_merge(br, dred[1][w]);
      }
      const float u = philox_uniform(a.seed, (uint64_t)n_glob, k_depth);
      float d;
      if (STATS) {
        // the target's logit at the drawn token (an all -inf draft row draws none: index 0)
        const int64_t y = (bq.i >= 0 && bq.i < a.V) ? bq.i : 0;
        const float zpy = sizeof(T) == 2
                              ? __uint_as_float((uint32_t)static_cast<const uint16_t*>(a.zp)[r * a.V + y] << 16)
                              : static_cast<const float*>(a.zp)[r * a.V + y];
        d = log2_prob(zpy, a.sT, a.lws.Mp[r], a.lws.Lsp[r]) - log2_prob(bq.z, a.sT, a.lws.Mq[r], a.lws.Lsq[r]);
      } else {
        const float Lsp = lse_ls(t.lp), Lsq = lse_ls(t.lq);
        d = log2_prob(bq.zp, a.sT, t.lp.M, Lsp) - log2_prob(bq.z, a.sT, t.lq.M, Lsq);
      }
      a.acc[r] = (u < exp2f(fminf(d, 0.f))) ? 1 : 0;
      if (REF) {
        const float Lsp = lse_ls(t.lp), Lsr = lse_ls(t.lr);
        const float dd = log2_prob(br.zp, a.sT, t.lp.M, Lsp) - log2_prob(br.z, a.sT, t.lr.M, Lsr);
        a.acc_ref[r] = (u < exp2f(fminf(dd, 0.f))) ? 1 : 0;
      }
    }
    __syncthreads();
  }
}

template <typename T, bool REF, bool STATS = false>
cudaError_t go_sampled(const RewardRowArgs& a, cudaStream_t s) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, reward_sampled_rows<T, REF, STATS>, kRowThreads, 0);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)sms * per_sm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  reward_sampled_rows<T, REF, STATS><<<(unsigned)grid, kRowThreads, 0, s>>>(a);
  return cudaGetLastError();
}

template <typename T, bool VEC, bool S, bool R, bool D = false>
cudaError_t go(const RewardRowArgs& a, cudaStream_t s) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, reward_rows<T, VEC, S, R, D>, kRowThreads, 0);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)sms * per_sm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  reward_rows<T, VEC, S, R, D><<<(unsigned)grid, kRowThreads, 0, s>>>(a);
  return cudaGetLastError();
}

template <typename T, bool VEC>
cudaError_t dispatch_flags(const RewardRowArgs& a, cudaStream_t s) {
  const bool ref = a.zr != nullptr;
  if (a.sampling && a.sampled_draft) {
    if (VEC) return ref ? go_sampled<T, true>(a, s) : go_sampled<T, false>(a, s);
    return ref ? go<T, VEC, true, true, true>(a, s) : go<T, VEC, true, false, true>(a, s);
  }
  if (a.sampling) return ref ? go<T, VEC, true, true>(a, s) : go<T, VEC, true, false>(a, s);
  return ref ? go<T, VEC, false, true>(a, s) : go<T, VEC, false, false>(a, s);
}

template <typename T>
cudaError_t dispatch(const RewardRowArgs& a, cudaStream_t s) {
  const bool vec = ((a.V * (int64_t)sizeof(T)) % 16 == 0) &&
                   ((reinterpret_cast<uintptr_t>(a.zq) | reinterpret_cast<uintptr_t>(a.zp) |
                     reinterpret_cast<uintptr_t>(a.zr)) % 16 == 0);
  return vec ? dispatch_flags<T, true>(a, s) : dispatch_flags<T, false>(a, s);
}

__device__ __forceinline__ double block_sum(double x, double* sm) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  __syncthreads();
  if (lane == 0) sm[warp] = x;
  __syncthreads();
  double t = sm[0];
  for (int w = 1; w < kGroupThreads / 32; ++w) t += sm[w];
  return t;
}

// One CTA per advantage group.
__global__ void __launch_bounds__(kGroupThreads) reward_groups(RewardGroupArgs a) {
  __shared__ double sm[kGroupThreads / 32];
  const int64_t g = blockIdx.x;
  const int64_t w0 = g * a.rpg * a.wpr, nw = a.rpg * a.wpr;
  const int K = a.K;
  // per window: tau, tau_ref, R
  for (int64_t i = threadIdx.x; i < nw; i += kGroupThreads) {
    const int64_t n = w0 + i;
    int tau = 0;
    while (tau < K && a.acc[n * K + tau] != 0) ++tau;
    int tr = 0;
    if (a.acc_ref != nullptr)
      while (tr < K && a.acc_ref[n * K + tr] != 0) ++tr;
    a.tau[n] = tau;
    if (a.tau_ref != nullptr) a.tau_ref[n] = tr;
    a.rbuf[n] = (float)(tau - tr);
  }
  __syncthreads();
  // rollout lengths: mean R over each rollout's windows (fixed-order block sums)
  const volatile float* rb = a.rbuf;
  for (int64_t ro = 0; ro < a.rpg; ++ro) {
    double s = 0.0;
    for (int64_t i = threadIdx.x; i < a.wpr; i += kGroupThreads) s += rb[w0 + ro * a.wpr + i];
    s = block_sum(s, sm);
    if (threadIdx.x == 0) a.rollout_len[g * a.rpg + ro] = (float)(s / (double)a.wpr);
  }
  __syncthreads();
  // group mean and population std, then clipped standardised advantages
  const volatile float* rl = a.rollout_len;
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < a.rpg; i += kGroupThreads) s += rl[g * a.rpg + i];
  const double mean = block_sum(s, sm) / (double)a.rpg;
  double v = 0.0;
  for (int64_t i = threadIdx.x; i < a.rpg; i += kGroupThreads) {
    const double d = rl[g * a.rpg + i] - mean;
    v += d * d;
  }
  const double sd = sqrt(block_sum(v, sm) / (double)a.rpg);
  for (int64_t i = threadIdx.x; i < a.rpg; i += kGroupThreads) {
    double A = (rl[g * a.rpg + i] - mean) / (sd + 1e-6);
    A = fmin(fmax(A, -(double)a.adv_clip), (double)a.adv_clip);
    a.advantage[g * a.rpg + i] = (float)A;
  }
}

// One thread per row: the acceptance of the draft's greedy token from the loss forward's
// statistics (x*, the draft argmax y = S_k and z_p(y), and the normalisers), no logit pass.
// Sampling: log2 q~(y) = (z_q(y) - M_q) s - Ls_q = -Ls_q because y is where z_q peaks.
__global__ void __launch_bounds__(256) reward_flags_from_stats(RewardStatsArgs a) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.R) return;
  uint8_t acc;
  if (!a.sampling) {
    acc = (a.ws.yhat[r] == a.ws.xstar[r]) ? 1 : 0;
  } else {
    const int64_t n = r / a.K;
    const uint32_t k = (uint32_t)(r - n * a.K);
    const float u = philox_uniform(a.seed, (uint64_t)(a.row_offset + n), k);
    const float d = log2_prob(a.ws.zpy[r], a.sT, a.ws.Mp[r], a.ws.Lsp[r]) + a.ws.Lsq[r];
    acc = (u < exp2f(fminf(d, 0.f))) ? 1 : 0;
  }
  a.acc[r] = acc;
}

}  // namespace

cudaError_t launch_reward_flags_from_stats(const RewardStatsArgs& a, cudaStream_t s) {
  if (a.R < 1) return cudaSuccess;
  reward_flags_from_stats<<<(unsigned)((a.R + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_reward_rows(const RewardRowArgs& a, bool bf16, cudaStream_t s) {
  return bf16 ? dispatch<uint16_t>(a, s) : dispatch<float>(a, s);
}

cudaError_t launch_reward_sampled_stats(const RewardRowArgs& a, bool bf16, cudaStream_t s) {
  return bf16 ? go_sampled<uint16_t, false, true>(a, s) : go_sampled<float, false, true>(a, s);
}

cudaError_t launch_reward_groups(const RewardGroupArgs& a, cudaStream_t s) {
  const int64_t groups = a.N / (a.wpr * a.rpg);
  if (groups < 1) return cudaSuccess;
  reward_groups<<<(unsigned)groups, kGroupThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace aal
