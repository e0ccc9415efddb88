// RMSNorm sum of squares shared by every norm kernel: a row is reduced by 256 "virtual threads",
// virtual thread vt summing the float4 chunks vt, vt + 256, ... of the row in order; each virtual
// warp of 32 is reduced with a butterfly, then the 8 warp totals with one more butterfly.  A kernel
// with fewer real threads runs several virtual threads per real thread and gets the same sum, bit
// for bit, as the 256-thread kernel.
#pragma once
#include <cuda_bf16.h>

#include "common.cuh"
#include "gemm_core.cuh"

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

// Embedding row t entering the residual stream, with its norm folded into the next GEMM:
// h[t] = embed row (fp32), xg[t] = bf16(g * h[t]) and the partial sums of squares of h[t] per
// 128-row tile, ssq[mt * ld + t], in the order every partial-sum producer uses (ssq32 quarters,
// then (q0 + q1) + (q2 + q3)).  nthreads (a multiple of 32) threads of one CTA, tid = 0 ..
// nthreads - 1, all of them calling.
__device__ __forceinline__ void embed_row(const __nv_bfloat16* er, const __nv_bfloat16* g, float* hr,
                                          __nv_bfloat16* xr, float* ssq, int ld, int t, int d, int tid,
                                          int nthreads) {
  for (int c = tid; c < d / 4; c += nthreads) {
    const uint2 raw = *reinterpret_cast<const uint2*>(er + 4 * c);
    const uint2 graw = *reinterpret_cast<const uint2*>(g + 4 * c);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&raw);
    const __nv_bfloat162* gb = reinterpret_cast<const __nv_bfloat162*>(&graw);
    const float2 f0 = __bfloat1622float2(b[0]), f1 = __bfloat1622float2(b[1]);
    const float2 g0 = __bfloat1622float2(gb[0]), g1 = __bfloat1622float2(gb[1]);
    *reinterpret_cast<float4*>(hr + 4 * c) = make_float4(f0.x, f0.y, f1.x, f1.y);
    __nv_bfloat162 o[2];
    o[0] = __floats2bfloat162_rn(f0.x * g0.x, f0.y * g0.y);
    o[1] = __floats2bfloat162_rn(f1.x * g1.x, f1.y * g1.y);
    *reinterpret_cast<uint2*>(xr + 4 * c) = *reinterpret_cast<const uint2*>(o);
  }
  const int nq = 4 * ((d + GEMM_BM - 1) / GEMM_BM);   // quarters of all tiles
  const int nq_w = (nq + 31) & ~31;                    // whole warps take part in the shuffles
  for (int qi = tid; qi < nq_w; qi += nthreads) {
    const int mt = qi >> 2, sub = qi & 3;
    const int r0 = mt * GEMM_BM + sub * 32;
    float s = 0.f;
    if (qi < nq) s = ssq32([&](int r) { return r0 + r < d ? __bfloat162float(er[r0 + r]) : 0.f; }, ssq_rot(sub));
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    if (qi < nq && sub == 0) ssq[(size_t)mt * ld + t] = s;
  }
}

// Total of the 8 virtual-warp sums red[0..7]; called by whole warps, every lane gets the total.
__device__ __forceinline__ float rms_total(const float* red) {
  const int lane = threadIdx.x & 31;
  return warp_sum(lane < 8 ? red[lane] : 0.f);
}

}  // namespace atspeed
