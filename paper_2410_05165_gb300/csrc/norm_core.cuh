// RMSNorm sum of squares shared by every norm kernel: a row is reduced by 256 "virtual threads",
// virtual thread vt summing the float4 chunks vt, vt + 256, ... of the row in order; each virtual
// warp of 32 is reduced with a butterfly, then the 8 warp totals with one more butterfly.  A kernel
// with fewer real threads runs several virtual threads per real thread and gets the same sum, bit
// for bit, as the 256-thread kernel.
#pragma once
#include <cuda_bf16.h>

#include "common.cuh"

namespace atspeed {

__device__ __forceinline__ float rms_part(const float* hr, int vt, int d) {
  float ss = 0.f;
  const float4* h4 = reinterpret_cast<const float4*>(hr);
  for (int c = vt; c < d / 4; c += 256) {
    const float4 v = __ldcg(h4 + c);
    ss += v.x * v.x;
    ss += v.y * v.y;
    ss += v.z * v.z;
    ss += v.w * v.w;
  }
  return ss;
}

// Same over an embedding row (bf16), also writing it to the fp32 residual row hr.
__device__ __forceinline__ float rms_part_embed(const __nv_bfloat16* er, float* hr, int vt, int d) {
  float ss = 0.f;
  for (int c = vt; c < d / 4; c += 256) {
    const uint2 raw = *reinterpret_cast<const uint2*>(er + 4 * c);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&raw);
    const float2 f0 = __bfloat1622float2(b[0]), f1 = __bfloat1622float2(b[1]);
    *reinterpret_cast<float4*>(hr + 4 * c) = make_float4(f0.x, f0.y, f1.x, f1.y);
    ss += f0.x * f0.x;
    ss += f0.y * f0.y;
    ss += f1.x * f1.x;
    ss += f1.y * f1.y;
  }
  return ss;
}

// Total of the 8 virtual-warp sums red[0..7]; called by whole warps, every lane gets the total.
__device__ __forceinline__ float rms_total(const float* red) {
  const int lane = threadIdx.x & 31;
  return warp_sum(lane < 8 ? red[lane] : 0.f);
}

}  // namespace atspeed
