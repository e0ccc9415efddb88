// Shared-prefix tree attention: TMA-staged K/V pages, tensor cores (mma.sync m16n8k16: bf16 Q K^T;
// P V with P split into two fp16 halves and V in fp16) with an fp32 online softmax, prefix split across CTAs, then a combine kernel that
// merges the splits with each node's path keys (ancestors + self, at most 4).
#include <cudaTypedefs.h>
#include <math.h>
#include <stdio.h>

#include "attention.cuh"
#include "attn_core.cuh"
#include "common.cuh"

namespace atspeed {

namespace {

template <int HD>
__global__ void __launch_bounds__(128)
    attn_prefix_kernel(const __grid_constant__ CUtensorMap mk, const __grid_constant__ CUtensorMap mv,
                       const AttnArgs a) {
  using C = AttCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::SMEM_BODY);
  pdl_launch_dependents();
  pdl_wait();
  if (threadIdx.x == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
    tma_prefetch_desc(&mk);
    tma_prefetch_desc(&mv);
  }
  __syncthreads();
  int use[2] = {0, 0};
  attn_item<HD>(a, &mk, &mv, blockIdx.x, blockIdx.y, blockIdx.z, smem, bars, use, threadIdx.x, 1);
}

// One CTA of 128 threads per (query tile, head, group of 16 queries): merge the prefix splits with
// the path keys.
template <int HD>
__global__ void __launch_bounds__(128) attn_combine_kernel(const AttnArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  attn_combine_group<HD>(a, blockIdx.x, blockIdx.y, blockIdx.z, threadIdx.x);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn_att() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

template <int HD>
cudaError_t launch_hd(const AttnArgs& a, const CUtensorMap& mk, const CUtensorMap& mv, cudaStream_t st, bool pdl) {
  using C = AttCfg<HD>;
  static std::atomic<unsigned long long> attr_done{0};
  {
    const cudaError_t e = smem_attr_once(attr_done, attn_prefix_kernel<HD>, C::SMEM);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_qtiles, a.n_heads, a.max_splits);
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cfg.attrs = at;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, attn_prefix_kernel<HD>, mk, mv, a);
  if (e != cudaSuccess || a.direct) return e;
  cudaLaunchConfig_t c2 = {};
  c2.gridDim = dim3(a.n_qtiles, a.n_heads, ATT_QTILE / ATT_CQ);
  c2.blockDim = dim3(128);
  c2.stream = st;
  c2.attrs = at;
  c2.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&c2, attn_combine_kernel<HD>, a);
}

}  // namespace

bool attn_make_maps(const __nv_bfloat16* k_cache, const __half* v_cache, int rows, int d_model, int head_dim,
                    CUtensorMap* mk, CUtensorMap* mv, char* eb, size_t el) {
  auto fn = encode_fn_att();
  if (!fn) {
    snprintf(eb, el, "cuTensorMapEncodeTiled unavailable");
    return false;
  }
  const int boxw = head_dim >= 64 ? 64 : head_dim;
  cuuint64_t dims[2] = {(cuuint64_t)d_model, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d_model * 2};
  cuuint32_t box[2] = {(cuuint32_t)boxw, (cuuint32_t)ATT_SUB};
  cuuint32_t es[2] = {1, 1};
  const CUtensorMapSwizzle sw = head_dim >= 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE;
  for (int i = 0; i < 2; ++i) {
    CUresult r = fn(i == 0 ? mk : mv, i == 0 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2,
                    i == 0 ? (void*)k_cache : (void*)v_cache, dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
      snprintf(eb, el, "attention tensor map failed (%d)", (int)r);
      return false;
    }
  }
  return true;
}

cudaError_t attn_launch(const AttnArgs& a, const CUtensorMap& mk, const CUtensorMap& mv, cudaStream_t st, bool pdl) {
  switch (a.head_dim) {
    case 32: return launch_hd<32>(a, mk, mv, st, pdl);
    case 64: return launch_hd<64>(a, mk, mv, st, pdl);
    case 128: return launch_hd<128>(a, mk, mv, st, pdl);
  }
  return cudaErrorInvalidValue;
}

}  // namespace atspeed
