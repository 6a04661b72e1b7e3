// Device helpers for sm_103a: mbarrier waits with a bound, 1-D TMA bulk
// copies into shared memory, bf16 unpacking and packed fp32x2 FMA.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "reskv.h"

namespace reskv {

// Device status word codes (written with atomicOr, read by reskv_check_status).
enum : uint32_t {
  kStatusWaitTimeout = 1u,    // a bounded mbarrier wait gave up
  kStatusBadIndex = 2u,       // an index left its valid range
};

// Upper bound for one mbarrier wait, in SM clock cycles (~2 s at 2 GHz).
constexpr long long kWaitLimitCycles = 4000000000LL;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Arrive on the barrier and announce `bytes` of transaction count.
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase with the given parity to complete; false after the bound.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitLimitCycles) return false;
  }
  return true;
}

// 1-D bulk copy global -> shared (TMA, non-multicast), completing on `bar`.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Two bf16 packed in a 32-bit word -> two floats (exact).
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// d = a * b + c on float pairs (one packed sm_100+ instruction).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  unsigned long long ra = *reinterpret_cast<unsigned long long*>(&a);
  unsigned long long rb = *reinterpret_cast<unsigned long long*>(&b);
  unsigned long long rc = *reinterpret_cast<unsigned long long*>(&c);
  unsigned long long rd;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(rd) : "l"(ra), "l"(rb), "l"(rc));
  return *reinterpret_cast<float2*>(&rd);
}

__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  unsigned long long ra = *reinterpret_cast<unsigned long long*>(&a);
  unsigned long long rb = *reinterpret_cast<unsigned long long*>(&b);
  unsigned long long rd;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(rd) : "l"(ra), "l"(rb));
  return *reinterpret_cast<float2*>(&rd);
}

// Coefficients (a, c) of o^ = a * acc_M + c * acc_R from the two branch
// states (m: running max in log2 units, l: sum of 2^(logit - m), acc: sum of
// 2^(logit - m) v) and the gate value g.
//   RESKV_SOFTMAX_SHARED (Eq. reskv): x = max(mM, mR), wM = 2^(mM - x),
//     wR = g 2^(mR - x), a = wM / den, c = wR / den, den = wM lM + wR lR;
//   RESKV_SOFTMAX_SEPARATE (ablation): a = (1 - g) / lM, c = g / lR.
// Without residual mass (lR = 0) or with g = 0 both are main-only: a = 1 / lM.
__device__ __forceinline__ float2 branch_coefs(int32_t softmax_mode, float g, float mM, float lM,
                                               float mR, float lR) {
  if (!(lR > 0.f) || !(g > 0.f)) return make_float2(1.0f / lM, 0.f);
  if (softmax_mode == RESKV_SOFTMAX_SEPARATE) return make_float2((1.0f - g) / lM, g / lR);
  const float x = fmaxf(mM, mR);
  const float wM = exp2f(mM - x), wR = g * exp2f(mR - x);
  const float inv = 1.0f / (wM * lM + wR * lR);
  return make_float2(wM * inv, wR * inv);
}

__device__ __forceinline__ void report_status(uint32_t* status, uint32_t code) {
  if (status) atomicOr(status, code);
}

}  // namespace reskv
