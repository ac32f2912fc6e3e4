// Inline-PTX building blocks for sm_103a kernels: mbarriers, 1-D TMA bulk copies, cluster
// and named barriers, bounded waits, packed fp32 / bf16 arithmetic.
#pragma once

#include "aal_internal.cuh"

namespace aal {
namespace ptx {

__device__ __forceinline__ uint32_t s32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// ---------------------------------------------------------------- mbarriers
__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(s32(b)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(s32(b)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(s32(b)) : "memory");
}
// Non-blocking test of a phase (no suspension).
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(s32(b)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Potentially blocking test: the thread may sleep in hardware (up to suspend_ns) until the
// phase completes.
__device__ __forceinline__ bool mbar_try(uint64_t* b, uint32_t parity, uint32_t suspend_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(s32(b)), "r"(parity), "r"(suspend_ns)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_try_cluster(uint64_t* b, uint32_t parity, uint32_t suspend_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(s32(b)), "r"(parity), "r"(suspend_ns)
      : "memory");
  return ok != 0;
}

// ---------------------------------------------------------------- TMA bulk copies
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// Global -> this CTA's shared memory, `bytes` (multiple of 16, both addresses 16-byte
// aligned), completion counted on `bar` in bytes.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                          uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          s32(dst)),
      "l"(src), "r"(bytes), "r"(s32(bar)), "l"(policy)
      : "memory");
}

// ---------------------------------------------------------------- barriers, time
// Named barrier over `n` threads; the warp is reconverged first so that it arrives whole.
__device__ __forceinline__ void named_barrier(int id, int n) {
  __syncwarp();
  asm volatile("barrier.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// GPU-scope relaxed 64-bit store and load (single-copy atomic, coherent in L2): the fused
// kernel's mailbox words, whose value is their own ready flag.
__device__ __forceinline__ void st_relaxed(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint64_t ld_relaxed(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ uint64_t now_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait on an mbarrier phase.  Returns false if the CTA's abort flag is (or gets)
// set or the time limit passes; a timeout records AAL_ERR_TIMEOUT in the workspace status
// word and raises the abort flag.
template <bool CLUSTER = false>
__device__ __forceinline__ bool wait_phase(uint64_t* b, uint32_t parity, volatile int* abort_flag,
                                           uint64_t limit_ns, WsHeader* hdr) {
  constexpr uint32_t kSuspendNs = 100000;
  if (*abort_flag) return false;
  if (CLUSTER ? mbar_try_cluster(b, parity, kSuspendNs) : mbar_try(b, parity, kSuspendNs)) return !*abort_flag;
  const uint64_t t0 = now_ns();
  for (uint32_t it = 0; it < kSpinLimit; ++it) {
    if (*abort_flag) return false;
    if (now_ns() - t0 > limit_ns) break;
    if (CLUSTER ? mbar_try_cluster(b, parity, kSuspendNs) : mbar_try(b, parity, kSuspendNs)) return !*abort_flag;
  }
  *abort_flag = 1;
  atomicExch(&hdr->status, kStatusTimeout);
  return false;
}

// Consumer side of a ring slot: a phase that has already completed is taken after one
// non-blocking test, without reading the abort flag; otherwise the bounded wait above.
// After an abort a consumer may so still read a landed (or stale) slot: its results are
// discarded, since every output write is guarded by the abort flag.
__device__ __forceinline__ bool wait_full(uint64_t* b, uint32_t parity, volatile int* abort_flag,
                                          uint64_t limit_ns, WsHeader* hdr) {
  return mbar_test(b, parity) || wait_phase(b, parity, abort_flag, limit_ns, hdr);
}

// ---------------------------------------------------------------- packed arithmetic
// Two fp32 lanes per instruction (sm_100+), IEEE round-to-nearest like the scalar forms.
#ifndef AAL_F2_ASM
#define AAL_F2_ASM 0
#endif
#if !AAL_F2_ASM
// the compiler's own pair operations: it places the pairs in registers itself
__device__ __forceinline__ float2 f2fma(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 f2add(float2 a, float2 b) { return __fadd2_rn(a, b); }
#else
__device__ __forceinline__ float2 f2fma(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mov.b64 rc, {%6, %7};\n\tfma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 f2add(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
#endif
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ float set_lt(float a, float b) {  // 1.0f if a < b else 0.0f
  float d;
  asm("set.lt.f32.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}
__device__ __forceinline__ float2 bpair(uint32_t w) { return make_float2(bf16_lo(w), bf16_hi(w)); }

}  // namespace ptx
}  // namespace aal
