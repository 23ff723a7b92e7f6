// Device-side helpers shared by the sm_103a kernel files: mbarrier ring
// primitives, 1-D TMA bulk copies, bounded waits, shared-memory loads.
// Internal to the library (each translation unit gets its own copies).
#pragma once

#include <cstdint>

namespace wt {
namespace {

constexpr int kStatusTimedOut = -7;  // WT_ETIMEDOUT
constexpr long long kWaitCycles = 1ll << 31;  // ~1 s at 2 GHz

// ------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// 1-D bulk copy global -> this CTA's shared memory, completion counted on `bar`.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes,
                                         uint32_t bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(pol)
      : "memory");
}

__device__ __forceinline__ void named_bar(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// Bounded wait.  Returns false (and raises the CTA's abort flag on a timeout)
// instead of spinning forever.
__device__ __forceinline__ bool bounded_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                             int *status) {
  if (*abort_flag) return false;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort_flag) return false;
    if (clock64() - t0 > kWaitCycles) {
      *abort_flag = 1;
      if (status) atomicCAS(status, 0, kStatusTimedOut);
      return false;
    }
  }
  return true;
}

// Programmatic dependent launch (launch attribute cudaLaunchAttributeProgrammaticStreamSerialization):
// griddep_wait blocks until the grid this one depends on in its stream has completed and its
// memory is visible (a no-op when the launch had no such dependency); griddep_launch lets the
// next grid of the stream be launched, its CTAs taking SMs as this grid's CTAs leave them.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// The global nanosecond timer (comparable across the SMs of one GPU) and the SM this thread
// runs on; read by the stamping instantiation of the one-column kernel only.
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ uint32_t sm_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}


__device__ __forceinline__ uint4 lds_or_zero(uint32_t addr, bool ok) {
  return ok ? lds128(addr) : make_uint4(0, 0, 0, 0);
}

// Two int8 weights as exact f16x2.  With u = b ^ 0x80 (0..255) in the low byte and 0x64 in
// the high byte, a half holds 1024 + u (f16 has unit spacing on [1024, 2048)); subtracting
// 1152 = 1024 + 128 leaves b, an integer in [-128, 127], exactly.
__device__ __forceinline__ uint32_t i8x2_to_f16x2(uint32_t u, uint32_t sel) {
  uint32_t h;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(h) : "r"(__byte_perm(u, 0x64646464u, sel)), "r"(0x64806480u));
  return h;
}

}  // namespace
}  // namespace wt
