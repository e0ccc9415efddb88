// Small kernels around the tree: gather the per-token inputs of a forward over tree nodes, and the
// final RMSNorm over the rows whose logits are needed.
#include "common.cuh"
#include "kernels.cuh"
#include "norm_core.cuh"

namespace atspeed {

__global__ void tree_gather_kernel(TreeDev t, const int* __restrict__ fwd_nodes, int T,
                                   const int* __restrict__ user_P, int code_base, int target, int row_base,
                                   FwdTokens f) {
  pdl_launch_dependents();
  pdl_wait();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= T) return;
  const int node = fwd_nodes[i];
  const int u = node / t.stride;
  const int slot = node - u * t.stride;
  const int lvl = slot < t.slots_in ? 0 : 1 + (slot - t.slots_in) / t.slots_lvl;
  const int depth = t.d[u] + lvl;   // >= 1 for every forwarded node
  const int code = t.code[node];
  const int own = target ? t.row_t[node] : t.row_d[node];
  const int* anc = target ? t.anc_t : t.anc_d;
  f.tok[i] = code_base + TREE_CODES * (depth - 1) + (code >= 0 ? code : 0);
  f.pos[i] = user_P[u] + depth - 1;
  f.kv_row[i] = own;
  f.tok_user[i] = u;
  f.tok_vis[i] = user_P[u];
  if (code >= 0) {
    for (int j = 0; j < 4; ++j) f.anc_row[i * 4 + j] = j < depth ? anc[(size_t)node * 4 + j] : own;
    f.anc_n[i] = depth;
  } else {  // unused slot: attend to the prefix and itself only
    for (int j = 0; j < 4; ++j) f.anc_row[i * 4 + j] = own;
    f.anc_n[i] = 1;
  }
  if (target)
    t.lg_t[node] = row_base + i;
  else
    t.lg_d[node] = row_base + i;
}

cudaError_t tree_gather_launch(const TreeDev& t, const int* fwd_nodes, int T, const int* user_P, int code_base,
                               bool target, int row_base, const FwdTokens& f, cudaStream_t st, bool pdl) {
  if (T <= 0) return cudaSuccess;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t c = {};
  c.gridDim = dim3((T + 127) / 128);
  c.blockDim = dim3(128);
  c.stream = st;
  c.attrs = at;
  c.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&c, tree_gather_kernel, t, fwd_nodes, T, user_P, code_base, target ? 1 : 0, row_base,
                            f);
}

__global__ void __launch_bounds__(256) rmsnorm_rows_kernel(const float* __restrict__ h, const int* __restrict__ rows,
                                                           const __nv_bfloat16* __restrict__ g, int d, float eps,
                                                           __nv_bfloat16* __restrict__ x, int ldx) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float red[8];
  const int i = blockIdx.x;
  const float* hr = h + (size_t)rows[i] * d;
  float ss = warp_sum(rms_part(hr, threadIdx.x, d));
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  const float r = 1.0f / sqrtf(rms_total(red) / (float)d + eps);
  for (int k = threadIdx.x; k < d; k += blockDim.x)
    x[(size_t)i * ldx + k] = __float2bfloat16_rn(hr[k] * r * __bfloat162float(g[k]));
}

cudaError_t rmsnorm_rows_launch(const float* h, const int* rows, int n, const __nv_bfloat16* g, int d, float eps,
                                __nv_bfloat16* x, int ldx, cudaStream_t st, bool pdl) {
  if (n <= 0) return cudaSuccess;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t c = {};
  c.gridDim = dim3(n);
  c.blockDim = dim3(256);
  c.stream = st;
  c.attrs = at;
  c.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&c, rmsnorm_rows_kernel, h, rows, g, d, eps, x, ldx);
}

}  // namespace atspeed
