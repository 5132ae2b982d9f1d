// Device helpers shared by the probe kernels.
#pragma once
#include <stdint.h>

namespace lc {

// Per-query reduction word of an accepted pair: IEEE bits of the FP32
// squared distance (non-negative, so bit order = value order) above the
// cache index; atomicMin keeps the nearest hit and, on equal distances, the
// lowest index (Eq. 14).
__device__ __forceinline__ unsigned long long pack_hit(float dist2, int64_t index) {
  return ((unsigned long long)__float_as_uint(dist2) << 32) | (unsigned long long)(uint32_t)index;
}

// Canonical FP32 squared distance sum_j (q_j - k_j)^2 over d_pad (multiple
// of 32) zero-padded features: a 32-wide fused-multiply-add chain per chunk,
// chunk sums added in order. Every probe path evaluates exactly this
// sequence of rounded operations, so all paths agree bit for bit. q and k
// are 16-byte aligned.
__device__ __forceinline__ float dist2_canonical(const float* __restrict__ q, const float* __restrict__ k, int dpad) {
  float total = 0.f;
  for (int c = 0; c < dpad; c += 32) {
    float p = 0.f;
#pragma unroll
    for (int j = 0; j < 32; j += 4) {
      const float4 a = *reinterpret_cast<const float4*>(q + c + j);
      const float4 b = *reinterpret_cast<const float4*>(k + c + j);
      float e = __fsub_rn(a.x, b.x);
      p = __fmaf_rn(e, e, p);
      e = __fsub_rn(a.y, b.y);
      p = __fmaf_rn(e, e, p);
      e = __fsub_rn(a.z, b.z);
      p = __fmaf_rn(e, e, p);
      e = __fsub_rn(a.w, b.w);
      p = __fmaf_rn(e, e, p);
    }
    total = __fadd_rn(total, p);
  }
  return total;
}

}  // namespace lc
