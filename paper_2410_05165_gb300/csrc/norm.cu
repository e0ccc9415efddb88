// Embedding gather and RMSNorm (LLaMA pre-norm), one CTA per token row.  (The decoder forward uses
// embed_rows for layer 0 and folds every other norm into its GEMMs; rmsnorm serves the operator API.)
//   h[t] = embed[token[t]]                      (fp32 residual stream; the table is bf16)
//   x[t] = bf16( h[t] / sqrt(mean(h[t]^2) + eps) * g )
#include "common.cuh"
#include "kernels.cuh"
#include "norm_core.cuh"

namespace atspeed {

__global__ void __launch_bounds__(256) rmsnorm_kernel(const float* __restrict__ h, const int* __restrict__ tokens,
                                                      const __nv_bfloat16* __restrict__ embed,
                                                      float* __restrict__ h_out, const __nv_bfloat16* __restrict__ g,
                                                      int d, float eps, __nv_bfloat16* __restrict__ x, int ldx) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.x;
  __shared__ float red[8];
  float* hr = tokens ? h_out + (size_t)t * d : const_cast<float*>(h) + (size_t)t * d;
  float ss = tokens ? rms_part_embed(embed + (size_t)tokens[t] * d, hr, threadIdx.x, d) : rms_part(hr, threadIdx.x, d);
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  const float r = 1.0f / sqrtf(rms_total(red) / (float)d + eps);
  for (int i = threadIdx.x; i < d; i += blockDim.x)
    x[(size_t)t * ldx + i] = __float2bfloat16_rn(hr[i] * r * __bfloat162float(g[i]));
}

// Layer 0's input rows: h[t] = embed[token[t]], xg[t] = bf16(g * h[t]) and the partial sums of
// squares per 128-row tile (the first norm's scale is applied by the QKV epilogue).
__global__ void __launch_bounds__(256) embed_rows_kernel(const int* __restrict__ tokens,
                                                         const __nv_bfloat16* __restrict__ embed,
                                                         const __nv_bfloat16* __restrict__ g, float* __restrict__ h,
                                                         __nv_bfloat16* __restrict__ xg, float* __restrict__ ssq,
                                                         int ld, int d) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.x;
  embed_row(embed + (size_t)tokens[t] * d, g, h + (size_t)t * d, xg + (size_t)t * d, ssq, ld, t, d, threadIdx.x,
            blockDim.x);
}

cudaError_t embed_rows_launch(const int* tokens, const __nv_bfloat16* embed, const __nv_bfloat16* g, float* h,
                              __nv_bfloat16* xg, float* ssq, int ld, int T, int d, cudaStream_t st, bool pdl) {
  if (T <= 0) return cudaSuccess;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(T);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, embed_rows_kernel, tokens, embed, g, h, xg, ssq, ld, d);
}

cudaError_t rmsnorm_launch(const float* h, const int* tokens, const __nv_bfloat16* embed, float* h_out,
                           const __nv_bfloat16* g, int T, int d, float eps, __nv_bfloat16* x, int ldx,
                           cudaStream_t st, bool pdl) {
  if (T <= 0) return cudaSuccess;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(T);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, rmsnorm_kernel, h, tokens, embed, h_out, g, d, eps, x, ldx);
}

}  // namespace atspeed
