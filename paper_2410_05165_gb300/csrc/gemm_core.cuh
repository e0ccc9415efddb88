// Shared pieces of the tcgen05 GEMM: tile constants and the fused epilogue of one 32-token chunk.
#pragma once
#include "common.cuh"
#include "gemm.cuh"

namespace atspeed {

constexpr int GEMM_BK = 64;    // bf16 elements per 128-byte swizzle row (one k-block)
constexpr int GEMM_BM = 128;   // weight rows per tile (MMA M)
constexpr int GEMM_WS_SLOT_FLOATS = 256 * 128;

// st: staging [32 tokens][128 rows] fp32 of one chunk; 128 threads (ep_tid) write the outputs.
template <int BN, int EPI>
__device__ __forceinline__ void epi_chunk(const GemmArgs& a, const float* st, int m_tile, int n_tile, int ch,
                                          int ep_tid) {
  const int tok0 = n_tile * BN + ch * 32;
  if constexpr (EPI == EPI_SWIGLU) {
    // thread owns feature i of the tile and tokens (ep_tid >> 6) + 2k
    const int i = ep_tid & 63, n0 = ep_tid >> 6;
    __nv_bfloat16* out = a.out_bf16 + m_tile * 64 + i;
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      const int n = n0 + 2 * k;
      const int tok = tok0 + n;
      if (tok < a.T) {
        const float g = st[n * GEMM_BM + i];
        const float u = st[n * GEMM_BM + 64 + i];
        out[(size_t)tok * a.ldo] = __float2bfloat16_rn(g / (1.0f + expf(-g)) * u);
      }
    }
  } else {
    // thread owns weight row m of the tile and the 32 tokens of the chunk
    const int m = ep_tid;
    const int row = m_tile * GEMM_BM + m;
    if (row >= a.M) return;
    const int nv = min(32, a.T - tok0);
    if constexpr (EPI == EPI_F32) {
#pragma unroll 8
      for (int n = 0; n < nv; ++n) a.out_f32[(size_t)(tok0 + n) * a.ldo + row] = st[n * GEMM_BM + m];
    } else if constexpr (EPI == EPI_BF16) {
#pragma unroll 8
      for (int n = 0; n < nv; ++n) a.out_bf16[(size_t)(tok0 + n) * a.ldo + row] = __float2bfloat16_rn(st[n * GEMM_BM + m]);
    } else if constexpr (EPI == EPI_RESID) {
      // read-modify-write of the fp32 residual; loads bypass L1 (other CTAs may have written it)
      float old[32];
      float* base = a.out_f32 + (size_t)tok0 * a.ldo + row;
#pragma unroll
      for (int n = 0; n < 32; ++n) old[n] = n < nv ? __ldcg(base + (size_t)n * a.ldo) : 0.f;
#pragma unroll
      for (int n = 0; n < 32; ++n)
        if (n < nv) base[(size_t)n * a.ldo] = old[n] + st[n * GEMM_BM + m];
    } else {  // EPI_QKV: rows of q | k | v; RoPE (rotate-half) on q and k, k / v to their cache rows
      const int d = a.d_model, hd = a.head_dim, half = hd >> 1;
      const int region = row / d;
      const int f = row - region * d;
      const int i = f & (hd - 1);
      const bool lo = i < half;
      const int ii = lo ? i : i - half;
      const int partner = lo ? m + half : m - half;
#pragma unroll 4
      for (int n = 0; n < nv; ++n) {
        const int tok = tok0 + n;
        const float v = st[n * GEMM_BM + m];
        if (region == 2) {
          a.v_cache[(size_t)a.kv_row[tok] * d + f] = __float2half_rn(bf16_round(v));
          continue;
        }
        const size_t cs = (size_t)a.pos[tok] * half + ii;
        const float cth = a.rope_cos[cs], sth = a.rope_sin[cs];
        const float x2 = st[n * GEMM_BM + partner];
        const float out = lo ? v * cth - x2 * sth : v * cth + x2 * sth;
        const __nv_bfloat16 ob = __float2bfloat16_rn(out);
        if (region == 0)
          a.q_out[(size_t)tok * d + f] = ob;
        else
          a.k_cache[(size_t)a.kv_row[tok] * d + f] = ob;
      }
    }
  }
}

}  // namespace atspeed
