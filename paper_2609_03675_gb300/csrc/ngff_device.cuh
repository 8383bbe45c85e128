// Device helpers shared by the frame-streaming kernels: shared-memory
// addresses, the global timer, mbarriers with a bounded wait, and the
// per-pixel grayscale and bin functions of K1 (one definition, used by K1,
// the spatial-signal kernels and the bin check entry point).
#pragma once

#include "ngff_common.cuh"

namespace cofie {
namespace {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
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

// Waits for the phase of parity `parity` to complete; false after timeout_ns.
__device__ __noinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > timeout_ns) return false;
  }
}

// Luma sums v = wR R + wG G + wB B + half of the four pixels packed in three
// little-endian words (bytes R0 G0 B0 R1 | G1 B1 R2 G2 | B2 R3 G3 B3).
__device__ __forceinline__ void luma4(uint32_t w0, uint32_t w1, uint32_t w2, const LumaConsts& L, uint32_t& v0,
                                      uint32_t& v1, uint32_t& v2, uint32_t& v3) {
  v0 = __dp2a_hi(L.w_b0, w0, __dp2a_lo(L.w_rg, w0, L.half));  // R0 G0 | B0
  v1 = __dp2a_lo(L.w_gb, w1, __dp2a_hi(L.w_0r, w0, L.half));  // R1 | G1 B1
  v2 = __dp2a_lo(L.w_b0, w2, __dp2a_hi(L.w_rg, w1, L.half));  // R2 G2 | B2
  v3 = __dp2a_hi(L.w_gb, w2, __dp2a_lo(L.w_0r, w2, L.half));  // R3 | G3 B3
}

template <int kBin>
__device__ __forceinline__ uint32_t bin_of(uint32_t v, const LumaConsts& L) {
  if (kBin == kBinFast) return __umulhi(v, L.magic);  // floor(v / (den * 256 / B)), host-verified
  const uint32_t y = __umulhi(v, L.magic_y);          // floor(v / den), host-verified
  return (y * L.bins) >> 8;
}

}  // namespace
}  // namespace cofie
