// One pass over the rows of a single logit tensor, for the calls that need one tensor only:
//
//   REF  aal_grpo_from_loss's reference-draft pass (Sec. 3.4): per row, log pi_ref at the
//        draft's greedy token y, [y == x*] and [argmax z_ref == x*] (x*, y from the loss
//        forward's workspace).
//   IDS  the loss forward when x* is given as target token ids (mode bit AAL_IDS; Sec. 3.2:
//        for greedy target-generated data x* is the ground-truth token): per row, the
//        draft's T = 1 normaliser, a^greedy = q(x*) and the draft's greedy token y.  Only
//        the draft is read: half the forward's bytes of the target-logit form.
//
// Rows whose byte length is a multiple of 16 are streamed through a shared-memory ring by
// TMA (one_tensor_stream); the others take a plain per-row loop (one_tensor_rows).
#include "grad_elem.cuh"
#include "ptx.cuh"

namespace aal {
namespace {

using namespace ptx;

constexpr uint32_t kStatusBadIndex = 1;  // == AAL_ERR_INVALID_ARG

constexpr int kRefThreads = 256;

template <typename T>
struct RefVec;
template <>
struct RefVec<float> {
  static constexpr int E = 4;
  __device__ static void unpack(const uint4& w, float* o) {
    o[0] = __uint_as_float(w.x);
    o[1] = __uint_as_float(w.y);
    o[2] = __uint_as_float(w.z);
    o[3] = __uint_as_float(w.w);
  }
};
template <>
struct RefVec<uint16_t> {
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
};

struct RefAcc {
  Lse l;
  Amax am;
};

__device__ __forceinline__ void ref_push(RefAcc& a, int64_t v, float z) {
  if (z > a.am.v) {
    a.am.v = z;
    a.am.i = (int32_t)v;
  }
  lse_push(a.l, z, kLog2e);
}

__device__ __forceinline__ RefAcc ref_merge(const RefAcc& a, const RefAcc& b) {
  RefAcc r;
  r.l = lse_merge(a.l, b.l, kLog2e);
  r.am = amax_merge(a.am, b.am);
  return r;
}

__device__ __forceinline__ RefAcc ref_shfl(const RefAcc& a, int off) {
  RefAcc b;
  b.l = shfl_lse(a.l, off);
  b.am = shfl_amax(a.am, off);
  return b;
}

// Row outputs of the two modes, by thread 0 once the row's normaliser (M, S), exact argmax
// `am` and the value z(x*) are known.  REF: log pi_ref(y), [y == x*], [argmax == x*].
// IDS: the draft's T = 1 statistics with x* = ids[r]; an id outside [0, V) records
// AAL_ERR_INVALID_ARG in the status word and contributes a^greedy = 0.
template <bool IDS>
__device__ __forceinline__ void row_outputs(const Stream1Args& a, int64_t r, float M, float S, int32_t am_index,
                                            bool am_exact, float zy, float zx, bool first_is_x) {
  const float Ls = log2f(S);
  if (IDS) {
    const int32_t xs = a.ids[r];
    const bool ok = xs >= 0 && (int64_t)xs < a.V;
    if (!ok) atomicExch(&a.hdr->status, kStatusBadIndex);
    a.lws.Mp[r] = 0.f;
    a.lws.Lsp[r] = 0.f;
    a.lws.Mq[r] = M;
    a.lws.Lsq[r] = Ls;
    a.lws.Mq1[r] = M;
    a.lws.Lsq1[r] = Ls;
    a.lws.cpart[r * kMaxCluster] = make_float2(0.f, 0.f);
    a.lws.xstar[r] = ok ? xs : -1;
    a.lws.ag[r] = ok ? exp2f(log2_prob(zx, kLog2e, M, Ls)) : 0.f;
    a.lws.yhat[r] = am_index;  // the exact index, or (am_exact false) its vector's start
    a.lws.zpy[r] = 0.f;
    (void)am_exact;
  } else {
    a.lpr[r] = (zy - M) - kLn2 * Ls;
    const int32_t y = a.lws.yhat[r], xs = a.lws.xstar[r];
    a.acc[r] = (y == xs) ? 1 : 0;
    a.acc_ref[r] = first_is_x ? 1 : 0;
  }
}

// One CTA per row (grid-stride over rows), 16-byte loads, two in flight per thread.
template <typename T, bool VEC, bool IDS>
__global__ void __launch_bounds__(kRefThreads) one_tensor_rows(Stream1Args a) {
  __shared__ RefAcc red[kRefThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x) {
    const T* z = static_cast<const T*>(a.z) + r * a.V;
    RefAcc acc;
    lse_init(acc.l);
    amax_init(acc.am);
    if (VEC) {
      constexpr int E = RefVec<T>::E;
      const int64_t nv = a.V / E;
      const uint4* z4 = reinterpret_cast<const uint4*>(z);
      int64_t i = threadIdx.x;
      for (; i + kRefThreads < nv; i += 2 * kRefThreads) {
        const uint4 w0 = ldg_stream(z4 + i);
        const uint4 w1 = ldg_stream(z4 + i + kRefThreads);
        float f[E];
        RefVec<T>::unpack(w0, f);
#pragma unroll
        for (int e = 0; e < E; ++e) ref_push(acc, i * E + e, f[e]);
        RefVec<T>::unpack(w1, f);
#pragma unroll
        for (int e = 0; e < E; ++e) ref_push(acc, (i + kRefThreads) * E + e, f[e]);
      }
      if (i < nv) {
        float f[E];
        RefVec<T>::unpack(ldg_stream(z4 + i), f);
#pragma unroll
        for (int e = 0; e < E; ++e) ref_push(acc, i * E + e, f[e]);
      }
    } else {
      for (int64_t v = threadIdx.x; v < a.V; v += kRefThreads) ref_push(acc, v, load_elem<T>(z + v));
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc = ref_merge(acc, ref_shfl(acc, off));
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      RefAcc t = red[0];
      for (int w = 1; w < kRefThreads / 32; ++w) t = ref_merge(t, red[w]);
      // indices are read only where they are valid (an all -inf row has no draft argmax; an
      // id may be out of range): nothing is read otherwise
      const int32_t y = IDS ? -1 : a.lws.yhat[r];
      const int32_t xs = IDS ? a.ids[r] : a.lws.xstar[r];
      const float zy = (y >= 0 && (int64_t)y < a.V) ? load_elem<T>(z + y) : -INFINITY;
      const float zx = (xs >= 0 && (int64_t)xs < a.V) ? load_elem<T>(z + xs) : -INFINITY;
      row_outputs<IDS>(a, r, t.l.M, t.l.S, t.am.i, true, zy, zx, t.am.i == xs);
    }
    __syncthreads();  // red is reused by the next row
  }
}

template <typename T, bool VEC, bool IDS>
cudaError_t go_rows(const Stream1Args& a, cudaStream_t s) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, one_tensor_rows<T, VEC, IDS>, kRefThreads, 0);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (int64_t)sms * per_sm;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  one_tensor_rows<T, VEC, IDS><<<(unsigned)grid, kRefThreads, 0, s>>>(a);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- streamed pass
// One CTA per SM, persistent over rows.  A producer thread copies each row in
// 48 KB chunks into a 4-slot ring (1-D TMA bulk copies, completion counted on an mbarrier
// per slot, evict_first: nothing is read twice); 16 consumer warps fold each chunk into
// an online log2-sum-exp and a per-16-byte-vector running maximum.  The indices asked
// about are known before the row starts (REF: y and x* from the loss forward; IDS: x* =
// ids[r]), so the thread that holds y's vector reads z(y), and the one that holds x*'s
// vector reads z(x*) and the first position in that vector with the same value.  At the
// end of the row (REF):
//   log pi_ref(y) = (z_ref(y) - M) - ln 2 * log2 S,
//   argmax z_ref == x*  iff  z_ref(x*) = M, the first vector holding M is x*'s, and no
//                           earlier element of that vector equals z_ref(x*).
// IDS records the first vector holding M as y; resolve_draft_argmax places the element.
// Every wait is bounded as in the loss forward (status word of the given workspace).
constexpr int kRSlots = 4;
constexpr int kRSlotBytes = 48 * 1024;
constexpr int kRWarps = 16;
constexpr int kRConsumers = 32 * kRWarps;
constexpr int kRThreads = 32 + kRConsumers;
constexpr int kRVecPerChunk = kRSlotBytes / 16;
constexpr int kRNV = kRVecPerChunk / kRConsumers;
static_assert(kRNV * kRConsumers == kRVecPerChunk, "consumers must tile a chunk");
constexpr int kRBarRow = 1;

struct RefPart {
  float M, S;    // online log2-sum-exp (M = raw max)
  float av;      // largest value and the first vector (element index) holding it
  int32_t ab;
};

struct RefSmem {
  uint64_t full[kRSlots];
  uint64_t empty[kRSlots];
  RefPart red[2][kRWarps];
  float zy[2], zx[2];   // z_ref(y), z_ref(x*), by row parity
  int32_t fx[2];        // first index of x*'s vector whose value equals z_ref(x*)
  int abort_flag;
};

constexpr float kRefFloor = -1e30f;

__device__ __forceinline__ void refpart_init(RefPart& a) {
  a.M = kRefFloor;
  a.S = 0.f;
  a.av = -INFINITY;
  a.ab = 0x7fffffff;
}

__device__ __forceinline__ void refpart_warp(RefPart& a) {
  float m = a.M;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  float s = a.S * ex2((a.M - m) * kLog2e);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  a.M = m;
  a.S = s;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, a.av, off);
    const int32_t i2 = __shfl_xor_sync(0xffffffffu, a.ab, off);
    if (v2 > a.av || (v2 == a.av && i2 < a.ab)) {
      a.av = v2;
      a.ab = i2;
    }
  }
}

// Fold one 16-byte vector (E values, the first at element idx0) into the part.
template <typename T>
__device__ __forceinline__ void ref_vec(RefPart& A, const uint4& w, int idx0) {
  constexpr int E = RefVec<T>::E;
  float f[E];
  RefVec<T>::unpack(w, f);
  float vm = f[0];
#pragma unroll
  for (int e = 1; e < E; ++e) vm = fmaxf(vm, f[e]);
  if (vm > A.av) {
    A.av = vm;
    A.ab = idx0;
  }
  const float m = fmaxf(A.M, vm);
  A.S *= ex2((A.M - m) * kLog2e);
  A.M = m;
  float acc = 0.f;
#pragma unroll
  for (int e = 0; e < E; ++e) acc += ex2((f[e] - m) * kLog2e);
  A.S += acc;
}

template <typename T>
__device__ __forceinline__ float ref_elem(const uint4& w, int e) {
  constexpr int E = RefVec<T>::E;
  float f[E];
  RefVec<T>::unpack(w, f);
  float v = f[0];
#pragma unroll
  for (int k = 1; k < E; ++k)
    if (k == e) v = f[k];
  return v;
}

// The first lane k <= e of the vector whose value equals lane e's.
template <typename T>
__device__ __forceinline__ int ref_first_equal(const uint4& w, int e) {
  constexpr int E = RefVec<T>::E;
  float f[E];
  RefVec<T>::unpack(w, f);
  const float v = ref_elem<T>(w, e);
  int first = e;
#pragma unroll
  for (int k = E - 1; k >= 0; --k)
    if (k <= e && f[k] == v) first = k;
  return first;
}

template <typename T, bool IDS>
__global__ void __launch_bounds__(kRThreads, 1) one_tensor_stream(Stream1Args a, int nch, uint64_t limit_ns) {
  WsHeader* hdr = a.hdr;
  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* ring = smem;
  RefSmem& S = *reinterpret_cast<RefSmem*>(smem + kRSlots * kRSlotBytes);
  volatile int* abort_flag = &S.abort_flag;
  constexpr int ES = sizeof(T);
  constexpr int E = 16 / ES;
  constexpr int CH = kRSlotBytes / ES;  // elements per chunk
  const int V = (int)a.V;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int k = 0; k < kRSlots; ++k) {
      mbar_init(&S.full[k], 1);
      mbar_init(&S.empty[k], kRWarps);
    }
    S.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == kRWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t drop = policy_evict_first();
      int slot = 0;
      uint32_t phase = 0, armed = 0, last_phase = 0;
      int64_t seq = 0;  // chunks walked, in ring order
      for (int64_t r = blockIdx.x; r < a.R && !*abort_flag; r += gridDim.x) {
        const char* row = static_cast<const char*>(a.z) + r * a.V * ES;
        for (int c = 0; c < nch; ++c, ++seq) {
          if (!wait_phase(&S.empty[slot], phase ^ 1u, abort_flag, limit_ns, hdr)) break;
          const int e0 = c * CH;
          const uint32_t bytes = (uint32_t)(min(CH, V - e0) * ES);
          if (seq != a.skip_chunk) {  // (the test hook leaves one chunk's barrier unarmed)
            mbar_expect_tx(&S.full[slot], bytes);
            bulk_load(ring + slot * kRSlotBytes, row + (int64_t)e0 * ES, bytes, &S.full[slot], drop);
            armed |= 1u << slot;
            last_phase = (last_phase & ~(1u << slot)) | (phase << slot);
          }
          if (++slot == kRSlots) {
            slot = 0;
            phase ^= 1u;
          }
        }
      }
      for (int k = 0; k < kRSlots; ++k) {  // drain the last copy of every slot
        if (!(armed & (1u << k))) continue;
        const uint32_t ph = (last_phase >> k) & 1u;
        const uint64_t t0 = now_ns();
        for (uint32_t it = 0; it < kSpinLimit && !mbar_try(&S.full[k], ph, 100000); ++it)
          if (now_ns() - t0 > limit_ns) break;
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    const int t = threadIdx.x;
    int slot = 0;
    uint32_t phase = 0, j = 0;
    for (int64_t r = blockIdx.x; r < a.R; r += gridDim.x, ++j) {
      const int32_t y = IDS ? -1 : a.lws.yhat[r];
      const int32_t xs = IDS ? a.ids[r] : a.lws.xstar[r];
      // owners of y's and x*'s vectors (none when an index is out of range)
      const bool y_ok = y >= 0 && y < V, x_ok = xs >= 0 && xs < V;
      const int cy = y_ok ? y / CH : -1, iy = y_ok ? (y - cy * CH) / E : 0, ey = y_ok ? y % E : 0;
      const int cx = x_ok ? xs / CH : -1, ix = x_ok ? (xs - cx * CH) / E : 0, ex = x_ok ? xs % E : 0;
      // S.zy/zx/fx[j & 1] are written by the owners before this row's barrier and read by
      // thread 0 after it; the owners of row j + 2 write them only after thread 0 has passed
      // the barrier of row j + 1, so nothing is reset (an absent owner is known from y_ok/x_ok)
      RefPart A;
      refpart_init(A);
      for (int c = 0; c < nch; ++c) {
        if (wait_phase(&S.full[slot], phase, abort_flag, limit_ns, hdr)) {
          const int e0 = c * CH;
          const uint4* Z = reinterpret_cast<const uint4*>(ring + slot * kRSlotBytes);
          if (e0 + CH <= V) {
            uint4 w[kRNV];
#pragma unroll
            for (int v = 0; v < kRNV; ++v) w[v] = Z[t + v * kRConsumers];
#pragma unroll
            for (int v = 0; v < kRNV; ++v) ref_vec<T>(A, w[v], e0 + (t + v * kRConsumers) * E);
          } else {
            const int nvec = (V - e0) / E;
            for (int i = t; i < nvec; i += kRConsumers) ref_vec<T>(A, Z[i], e0 + i * E);
          }
          if (c == cy && t == iy % kRConsumers) S.zy[j & 1] = ref_elem<T>(Z[iy], ey);
          if (c == cx && t == ix % kRConsumers) {
            S.zx[j & 1] = ref_elem<T>(Z[ix], ex);
            S.fx[j & 1] = cx * CH + ix * E + ref_first_equal<T>(Z[ix], ex);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[slot]);
        if (++slot == kRSlots) {
          slot = 0;
          phase ^= 1u;
        }
      }
      refpart_warp(A);
      if (lane == 0) S.red[j & 1][warp] = A;
      named_barrier(kRBarRow, kRConsumers);
      if (t == 0 && !*abort_flag) {
        RefPart tot = S.red[j & 1][0];
        for (int w = 1; w < kRWarps; ++w) {
          const RefPart b = S.red[j & 1][w];
          const float m = fmaxf(tot.M, b.M);
          tot.S = tot.S * ex2((tot.M - m) * kLog2e) + b.S * ex2((b.M - m) * kLog2e);
          tot.M = m;
          if (b.av > tot.av || (b.av == tot.av && b.ab < tot.ab)) {
            tot.av = b.av;
            tot.ab = b.ab;
          }
        }
        const bool first_is_x = x_ok && S.zx[j & 1] == tot.av && tot.ab == xs - ex && S.fx[j & 1] == xs;
        const float zy = y_ok ? S.zy[j & 1] : -INFINITY;
        const float zx = x_ok ? S.zx[j & 1] : -INFINITY;
        row_outputs<IDS>(a, r, tot.M, tot.S, tot.ab, false, zy, zx, first_is_x);
      }
    }
  }
  __syncwarp();
  __syncthreads();
}

constexpr size_t kRSmemBytes = (size_t)kRSlots * kRSlotBytes + sizeof(RefSmem);

template <typename T, bool IDS>
cudaError_t go_stream(const Stream1Args& a, cudaStream_t s, uint64_t limit_ns) {
  auto kern = one_tensor_stream<T, IDS>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kRSmemBytes);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t grid = sms;
  if (grid > a.R) grid = a.R;
  if (grid < 1) return cudaSuccess;
  const int CH = kRSlotBytes / (int)sizeof(T);
  const int nch = (int)((a.V + CH - 1) / CH);
  kern<<<(unsigned)grid, kRThreads, kRSmemBytes, s>>>(a, nch, limit_ns);
  return cudaGetLastError();
}


// The first z maximum inside the vector the IDS stream recorded for each row.
template <typename T>
__global__ void __launch_bounds__(256) resolve_draft_argmax(Stream1Args a) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= a.R) return;
  constexpr int E = 16 / sizeof(T);
  const int32_t b = a.lws.yhat[r];
  int32_t y = 0;
  if (b >= 0 && b % E == 0 && (int64_t)b + E <= a.V) {  // an in-range, vector-aligned start only
    const T* z = static_cast<const T*>(a.z) + r * a.V;
    float f[8];
    RefVec<T>::unpack(*reinterpret_cast<const uint4*>(z + b), f);
    float m = f[0];
    for (int e = 1; e < E; ++e) m = fmaxf(m, f[e]);
    int at = 0;
    for (int e = E - 1; e >= 0; --e)
      if (f[e] == m) at = e;
    y = b + at;
  }
  a.lws.yhat[r] = y;
}

template <typename T>
cudaError_t launch_T(const Stream1Args& a, bool ids, cudaStream_t s) {
  const bool aligned = (a.V * (int64_t)sizeof(T)) % 16 == 0 && reinterpret_cast<uintptr_t>(a.z) % 16 == 0;
  if (!aligned) {
    if (ids) return go_rows<T, false, true>(a, s);
    return go_rows<T, false, false>(a, s);
  }
  const uint64_t limit = debug_wait_limit_ns();
  const uint64_t lim = limit ? limit : kWaitLimitNs;
  if (!ids) return go_stream<T, false>(a, s, lim);
  cudaError_t e = go_stream<T, true>(a, s, lim);
  if (e != cudaSuccess || a.R < 1) return e;
  resolve_draft_argmax<T><<<(unsigned)((a.R + 255) / 256), 256, 0, s>>>(a);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- fused forward + backward, ids
// aal_loss_fwd_bwd with x* as token ids: the K rows of a window held by K CTAs (one cooperative
// launch, one CTA per SM), each row streamed from HBM for the draft's statistics (kept in L2),
// its a^greedy exchanged through the per-row mailbox as in fused.cu, and streamed again from L2
// for the gradient -dloss/|W| w_g dE/da a^g (delta_{u,x*} - q(u)).  Statistics, exchange and
// coefficients reuse the IDS stream's and the backward's code, so the results are bitwise those
// of aal_loss_fwd + aal_loss_bwd; resolve_draft_argmax and the window kernel run after it.
// The SMs that G K leaves over take whole windows as solo CTAs, as in fused.cu.  SEQ: the
// sequence layout (aal_seq_loss_fwd_bwd with token ids), every CTA walking the positions from the
// last one down and exchanging with the 2K - 1 positions around its row, as fused.cu's SEQ
// instances do.
constexpr int kRBarCoef = 3;

struct FusedIdsSmem {
  RefSmem s;
  RowCoef coef;
  int32_t live;
  // a solo CTA's window: its rows' statistics, then their coefficients
  RowStat solo_st[AAL_MAX_K];
  RowCoef solo_coef[AAL_MAX_K];
  int32_t solo_live[AAL_MAX_K];
};

constexpr size_t kFIdsSmemBytes = (size_t)kRSlots * kRSlotBytes + sizeof(FusedIdsSmem);

template <bool SEQ>
__global__ void __launch_bounds__(kRThreads, 1) fused_ids_rows(FusedIdsArgs f, int nch, uint64_t limit_ns) {
  using T = uint16_t;
  constexpr int E = 8;
  constexpr int CH = kRSlotBytes / 2;  // elements per chunk
  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* ring = smem;
  FusedIdsSmem& F = *reinterpret_cast<FusedIdsSmem*>(smem + kRSlots * kRSlotBytes);
  RefSmem& S = F.s;
  const Stream1Args& a = f.st;
  WsHeader* hdr = a.hdr;
  volatile int* abort_flag = &S.abort_flag;
  const int V = (int)a.V;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = f.win.K;
  const int64_t N = f.win.N;
  const int G = f.groups;
  const int64_t NG = f.n_group;  // windows 0 .. NG - 1 go to the groups, the rest to the solo CTAs
  const bool solo = !SEQ && (int)blockIdx.x >= G * K;
  const int g = blockIdx.x / K, k = blockIdx.x % K;  // (a group's CTA)
  const int so = (int)blockIdx.x - G * K;            // (a solo CTA)
  const int C = gridDim.x;                           // (the sequence layout: rows R-1-c, R-1-c-C, ...)

  if (threadIdx.x == 0) {
    for (int q = 0; q < kRSlots; ++q) {
      mbar_init(&S.full[q], 1);
      mbar_init(&S.empty[q], kRWarps);
    }
    S.abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == kRWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t keep = policy_evict_last(), drop = policy_evict_first();
      int slot = 0;
      uint32_t phase = 0, armed = 0, last_phase = 0;
      int64_t seq = 0;
      // pass 0 (statistics, kept in L2) or 1 (gradient, the row's last use) of row r
      auto issue = [&](int64_t r, int pass) {
        const char* row = static_cast<const char*>(a.z) + r * a.V * 2;
        const uint64_t pol = pass == 0 ? keep : drop;
        for (int c = 0; c < nch && !*abort_flag; ++c, ++seq) {
          if (!wait_phase(&S.empty[slot], phase ^ 1u, abort_flag, limit_ns, hdr)) break;
          const int e0 = c * CH;
          const uint32_t bytes = (uint32_t)(min(CH, V - e0) * 2);
          if (seq != a.skip_chunk) {  // (the test hook leaves one chunk's barrier unarmed)
            mbar_expect_tx(&S.full[slot], bytes);
            bulk_load(ring + slot * kRSlotBytes, row + (int64_t)e0 * 2, bytes, &S.full[slot], pol);
            armed |= 1u << slot;
            last_phase = (last_phase & ~(1u << slot)) | (phase << slot);
          }
          if (++slot == kRSlots) {
            slot = 0;
            phase ^= 1u;
          }
        }
      };
      if (SEQ) {
        for (int64_t p = a.R - 1 - blockIdx.x; p >= 0 && !*abort_flag; p -= C) {
          issue(p, 0);
          issue(p, 1);
        }
      } else if (!solo) {
        for (int64_t n = g; n < NG && !*abort_flag; n += G) {
          issue(n * K + k, 0);
          issue(n * K + k, 1);
        }
      } else {
        // a whole window: the statistics of its K rows, then their gradients
        for (int64_t n = NG + so; n < N && !*abort_flag; n += f.solos) {
          for (int kk = 0; kk < K; ++kk) issue(n * K + kk, 0);
          for (int kk = 0; kk < K; ++kk) issue(n * K + kk, 1);
        }
      }
      for (int q = 0; q < kRSlots; ++q) {
        if (!(armed & (1u << q))) continue;
        const uint32_t ph = (last_phase >> q) & 1u;
        const uint64_t t0 = now_ns();
        for (uint32_t it = 0; it < kSpinLimit && !mbar_try(&S.full[q], ph, 100000); ++it)
          if (now_ns() - t0 > limit_ns) break;
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    const int t = threadIdx.x;
    int slot = 0;
    uint32_t phase = 0, j = 0;  // j: rows walked (parity of the reduction buffers)
    float scale = 0.f;          // thread 0: -dloss / |W|
    if (t == 0) {
      const int nvalid = hdr->nvalid;
      scale = nvalid > 0 ? -f.bw.dloss / (float)nvalid : 0.f;
    }

    // ---- pass 1 of row r: the draft's normaliser and greedy token (HBM), written to the
    // workspace; thread 0 gets what the row's coefficients need
    auto stats_row = [&](int64_t r, RowStat& st) {
      const int32_t xs = a.ids[r];
      const bool x_ok = xs >= 0 && xs < V;
      const int cx = x_ok ? xs / CH : -1, ix = x_ok ? (xs - cx * CH) / E : 0, ex = x_ok ? xs % E : 0;
      RefPart A;
      refpart_init(A);
      for (int c = 0; c < nch; ++c) {
        if (wait_full(&S.full[slot], phase, abort_flag, limit_ns, hdr)) {
          const int e0 = c * CH;
          const uint4* Z = reinterpret_cast<const uint4*>(ring + slot * kRSlotBytes);
          if (e0 + CH <= V) {
            uint4 w[kRNV];
#pragma unroll
            for (int v = 0; v < kRNV; ++v) w[v] = Z[t + v * kRConsumers];
#pragma unroll
            for (int v = 0; v < kRNV; ++v) ref_vec<T>(A, w[v], e0 + (t + v * kRConsumers) * E);
          } else {
            const int nvec = (V - e0) / E;
            for (int i = t; i < nvec; i += kRConsumers) ref_vec<T>(A, Z[i], e0 + i * E);
          }
          if (c == cx && t == ix % kRConsumers) S.zx[j & 1] = ref_elem<T>(Z[ix], ex);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[slot]);
        if (++slot == kRSlots) {
          slot = 0;
          phase ^= 1u;
        }
      }
      refpart_warp(A);
      if (lane == 0) S.red[j & 1][warp] = A;
      named_barrier(kRBarRow, kRConsumers);
      if (t == 0) {
        RefPart tot = S.red[j & 1][0];
        for (int w = 1; w < kRWarps; ++w) {
          const RefPart b = S.red[j & 1][w];
          const float m = fmaxf(tot.M, b.M);
          tot.S = tot.S * ex2((tot.M - m) * kLog2e) + b.S * ex2((b.M - m) * kLog2e);
          tot.M = m;
          if (b.av > tot.av || (b.av == tot.av && b.ab < tot.ab)) {
            tot.av = b.av;
            tot.ab = b.ab;
          }
        }
        const float zx = x_ok ? S.zx[j & 1] : -INFINITY;
        if (!*abort_flag) row_outputs<true>(a, r, tot.M, tot.S, tot.ab, false, -INFINITY, zx, false);
        // the same values row_outputs wrote, as the backward reads them
        const float Ls = log2f(tot.S);
        st.Mq1 = tot.M;
        st.Lsq1 = Ls;
        st.ag = x_ok ? exp2f(log2_prob(zx, kLog2e, tot.M, Ls)) : 0.f;
        st.xs = x_ok ? xs : -1;
      }
      ++j;
    };

    // Thread 0: the coefficients of depth kk of window n (row r) from the window's a^greedy
    // (agv), as the window kernel forms its terms and the backward its coefficients.
    auto coef_row = [&](int64_t n, int kk, int64_t r, const float* agv, const RowStat& st, RowCoef& c) -> int32_t {
      int kn = K;
      if (f.win.mask != nullptr) {
        kn = 0;
        while (kn < K && f.win.mask[n * K + kn] != 0) ++kn;
      }
      float dE[AAL_MAX_K];
      window_term(agv, kn, dE);
      const bool pos_valid = f.bw.mask == nullptr || f.bw.mask[r] != 0;
      return row_coef<true, false, false>(f.bw, scale, 0.f, f.bw.w_greedy != 0.f ? dE[kk] : 0.f, 0.f, 0.f,
                                          pos_valid, st, c)
                 ? 1
                 : 0;
    };

    // ---- pass 2 of row r: the gradient row (L2)
    auto grad_row = [&](int64_t r, const RowCoef& c, int32_t live) {
      const int64_t xv = (live && c.xs >= 0) ? c.xs / E : -1;
      const int xe = c.xs >= 0 ? c.xs % E : 0;
      uint4* out4 = reinterpret_cast<uint4*>(static_cast<T*>(f.bw.grad) + r * a.V);
      const uint4 zero4 = make_uint4(0, 0, 0, 0);
      for (int cc = 0; cc < nch; ++cc) {
        if (wait_full(&S.full[slot], phase, abort_flag, limit_ns, hdr)) {
          const int e0 = cc * CH;
          const int64_t vb = e0 / E;
          const uint4* Z = reinterpret_cast<const uint4*>(ring + slot * kRSlotBytes);
          if (e0 + CH <= V) {
#pragma unroll
            for (int v = 0; v < kRNV; ++v) {
              const int i = t + v * kRConsumers;
              st_stream(out4 + vb + i, live ? grad_vec<T, true, false, false, false>(c, Z[i], zero4, vb + i, xv, xe, -1, 0)
                                            : zero4);
            }
          } else {
            const int nvec = (V - e0) / E;
            for (int i = t; i < nvec; i += kRConsumers)
              st_stream(out4 + vb + i, live ? grad_vec<T, true, false, false, false>(c, Z[i], zero4, vb + i, xv, xe, -1, 0)
                                            : zero4);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&S.empty[slot]);
        if (++slot == kRSlots) {
          slot = 0;
          phase ^= 1u;
        }
      }
    };

    if (SEQ) {
      // each row: statistics, its mailbox word, the exchange with the positions around it (warp
      // 0), the coefficients (thread 0), the gradient
      for (int64_t r = a.R - 1 - blockIdx.x; r >= 0; r -= C) {
        RowStat st{};
        stats_row(r, st);
        if (warp == 0) {
          if (lane == 0) ptx::st_relaxed(&a.lws.mbox[r], mbox_word(st.ag, 0.f));
          const int64_t lo = r - r % f.seq_T, hi = lo + f.seq_T - 1;
          float dEg = 0.f, dEs = 0.f;
          const bool ok = seq_exchange(a.lws.mbox, f.seq_mask, r, lo, hi, K, f.seq_full != 0, true, false, false,
                                       0.f, 0.f, true, lane, abort_flag, hdr, limit_ns, &dEg, &dEs);
          if (lane == 0) {
            RowCoef c;
            const bool pos_valid = f.bw.mask == nullptr || f.bw.mask[r] != 0;
            F.live = ok && row_coef<true, false, false>(f.bw, scale, 0.f, f.bw.w_greedy != 0.f ? dEg : 0.f, 0.f, 0.f,
                                                       pos_valid, st, c)
                         ? 1
                         : 0;
            if (F.live) F.coef = c;
          }
        }
        named_barrier(kRBarCoef, kRConsumers);
        const RowCoef c = F.coef;
        grad_row(r, c, F.live);
      }
    } else if (!solo) {
      // one row of each of the group's windows: statistics, the window exchange (warp 0: lane j
      // polls depth j), the coefficients (thread 0), the gradient
      for (int64_t n = g; n < NG; n += G) {
        const int64_t r = n * K + k;
        RowStat st{};
        stats_row(r, st);
        if (warp == 0) {
          float agv[AAL_MAX_K], asv[AAL_MAX_K];
          const bool ok = window_exchange(a.lws.mbox, r, n * K, K, lane, st.ag, 0.f, true, abort_flag, hdr, limit_ns,
                                          agv, asv);
          if (lane == 0) {
            RowCoef c;
            F.live = ok ? coef_row(n, k, r, agv, st, c) : 0;
            if (F.live) F.coef = c;
          }
        }
        named_barrier(kRBarCoef, kRConsumers);
        const RowCoef c = F.coef;
        grad_row(r, c, F.live);
      }
    } else {
      // whole windows: the statistics of the K rows, their coefficients from those rows alone
      // (no exchange), then the K gradient rows
      for (int64_t n = NG + so; n < N; n += f.solos) {
        for (int kk = 0; kk < K; ++kk) {
          RowStat st{};
          stats_row(n * K + kk, st);
          if (t == 0) F.solo_st[kk] = st;
        }
        if (t == 0) {
          float agv[AAL_MAX_K];
#pragma unroll
          for (int jj = 0; jj < AAL_MAX_K; ++jj) agv[jj] = jj < K ? F.solo_st[jj].ag : 0.f;
          for (int kk = 0; kk < K; ++kk) {
            RowCoef c;
            F.solo_live[kk] = !*abort_flag ? coef_row(n, kk, n * K + kk, agv, F.solo_st[kk], c) : 0;
            if (F.solo_live[kk]) F.solo_coef[kk] = c;
          }
        }
        named_barrier(kRBarCoef, kRConsumers);
        for (int kk = 0; kk < K; ++kk) {
          const RowCoef c = F.solo_coef[kk];
          grad_row(n * K + kk, c, F.solo_live[kk]);
        }
      }
    }
  }
  __syncwarp();
  __syncthreads();
}

}  // namespace

namespace {
template <bool SEQ>
cudaError_t go_fused_ids(const FusedIdsArgs& f0, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  *launched = false;
  if (f0.bw.w_greedy == 0.f || f0.bw.grpo) return cudaSuccess;  // only the greedy term is fused here
  auto kern = fused_ids_rows<SEQ>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFIdsSmemBytes);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per_sm = 0, coop = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kRThreads, kFIdsSmemBytes);
  if (e != cudaSuccess) return e;
  const int64_t K = f0.win.K;
  FusedIdsArgs f = f0;
  int64_t grid = 0;
  if (SEQ) {
    // one CTA per SM walking the positions down; deadlock-free when a round spans a window or
    // holds every row (fused.cu, go_fused_seq)
    grid = (int64_t)sms * per_sm;
    if (grid > f.st.R) grid = f.st.R;
    if (!coop || grid < 1 || (grid < K && grid < f.st.R)) return cudaSuccess;
  } else {
    int64_t G = (int64_t)sms * per_sm / K;
    if (G > f0.win.N) G = f0.win.N;
    if (G > kMaxGroups) G = kMaxGroups;
    if (!coop || G < 1) return cudaSuccess;
    // the SMs left over by the groups take whole windows alone
    const int64_t S = (int64_t)sms * per_sm - G * K;
    const int64_t m = solo_windows_each(f0.win.N, K, G, S);
    f.groups = (int32_t)G;
    f.solos = m > 0 ? (int32_t)S : 0;
    f.n_group = f0.win.N - m * f.solos;
    grid = G * K + f.solos;
  }
  const int CH = kRSlotBytes / 2;
  const int nch = (int)((f.st.V + CH - 1) / CH);
  void* args[] = {&f, (void*)&nch, &limit_ns};
  e = cudaLaunchCooperativeKernel((const void*)kern, dim3((unsigned)grid), dim3(kRThreads), args, kFIdsSmemBytes, s);
  if (e == cudaErrorCooperativeLaunchTooLarge) {  // fewer SMs available: the caller runs the two calls
    cudaGetLastError();
    return cudaSuccess;
  }
  if (e != cudaSuccess) return e;
  *launched = true;
  resolve_draft_argmax<uint16_t><<<(unsigned)((f.st.R + 255) / 256), 256, 0, s>>>(f.st);
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_fused_ids(const FusedIdsArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  return go_fused_ids<false>(f, s, limit_ns, launched);
}

cudaError_t launch_fused_ids_seq(const FusedIdsArgs& f, cudaStream_t s, uint64_t limit_ns, bool* launched) {
  return go_fused_ids<true>(f, s, limit_ns, launched);
}

cudaError_t launch_one_tensor(const Stream1Args& a, bool bf16, bool ids, cudaStream_t s) {
  return bf16 ? launch_T<uint16_t>(a, ids, s) : launch_T<float>(a, ids, s);
}

}  // namespace aal
