// Device helpers shared by the sm_103a kernels: 16-bit element types, the RoPE angle, and PTX
// wrappers for mbarriers, bulk copies, the global timer and programmatic dependent launch.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace kvc {

// ---------------------------------------------------------------------------------------------
// 16-bit element types
// ---------------------------------------------------------------------------------------------
struct F16T {
  static __device__ __forceinline__ float2 f2(uint32_t u) {
    return __half22float2(*reinterpret_cast<const __half2*>(&u));
  }
  static __device__ __forceinline__ float f1(uint16_t u) { return __half2float(__ushort_as_half(u)); }
  static __device__ __forceinline__ uint16_t r(float x) { return __half_as_ushort(__float2half_rn(x)); }
};
struct BF16T {
  static __device__ __forceinline__ float2 f2(uint32_t u) {
    return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u));
  }
  static __device__ __forceinline__ float f1(uint16_t u) { return __bfloat162float(__ushort_as_bfloat16(u)); }
  static __device__ __forceinline__ uint16_t r(float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }
};

// ---------------------------------------------------------------------------------------------
// RoPE angle.  theta = pos * base^(-2i/rot) is reduced in turns: g = base^(-2i/rot) / (2 pi) is
// held as a double-float (hi, lo); pos * hi is split exactly with an FMA (Dekker's two-product),
// the integer part of the turns is removed exactly, leaving f in [-1/2, 1/2] turns with an error
// near 1e-7 at any position below 2^24 (a plain binary32 product would be off by up to half an ulp
// of theta, about 5e-4 rad at position 8192).  The sine and cosine of 2 pi f, an angle in
// [-pi, pi], come from the hardware approximation, whose absolute error there (about 2^-21) is
// far below the 16-bit rounding of the rotated values (2^-11 relative for fp16).
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ void rope_sincos(int32_t pos, float2 g, float* s, float* c) {
  const float p = (float)pos;
  const float a = __fmul_rn(p, g.x);
  const float e = __fmaf_rn(p, g.x, -a);
  const float f = __fadd_rn(__fsub_rn(a, rintf(a)), __fmaf_rn(p, g.y, e));
  __sincosf(6.28318530717958647692f * f, s, c);
}

// ---------------------------------------------------------------------------------------------
// PTX helpers: mbarrier, 1-D bulk copy (TMA), global timer
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Waits for the phase with the given parity; gives up after limit_ns (returns false).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, unsigned long long limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63u) == 0 && global_ns() - t0 > limit_ns) return false;
  }
}
// Programmatic dependent launch: let the next kernel on the stream be scheduled, and wait for
// the preceding one (no-ops when the launch did not opt in).
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_addr(dst)),
               "l"(src), "r"(bytes), "r"(smem_addr(bar))
               : "memory");
}
// Orders this thread's generic-proxy shared-memory writes before later async-proxy accesses
// (bulk copies, tensor-core operand reads).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

}  // namespace kvc
