// Persistent forward kernel: one cooperative launch runs a whole decoder forward (every layer's
// QKV GEMM + RMSNorm scale + RoPE + KV store, tree attention, O GEMM + residual, gate/up GEMM +
// RMSNorm scale + SwiGLU, down GEMM + residual, then the final norm and the item-code LM head).
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "attention.cuh"

namespace atspeed {

// Tensor-map table layout (device memory, 64-byte aligned CUtensorMap entries):
//   [l*4 + 0..3]    weights of layer l: wqkv, wo, wgate_up, wdown   (box 64 x 64, 128B swizzle)
//   [4L + 2l + 0/1] K / V cache of layer l                          (box hd' x 64, attention)
//   [6L + 0]        item-code rows of the LM head                   (box 64 x 64)
//   [6L + 1..3]     activations x, att, act, token tile 128         (box 64 x 128)
//   [6L + 4..6]     activations x, att, act, token tile 256         (box 64 x 256)
inline int fwd_map_count(int L) { return 6 * L + 7; }

struct FwdParams {
  int T;          // tokens of the forward
  int n_out;      // tokens whose item-code logits are produced (final-norm rows)
  int d, H, hd, ffn, L;
  float eps;
  int G;          // CTAs (one per SM, all co-resident)
  const CUtensorMap* maps;
  // norms, embedding (bf16)
  const __nv_bfloat16* const* attn_norm;  // [L] device pointers
  const __nv_bfloat16* const* mlp_norm;   // [L]
  const __nv_bfloat16* final_norm;
  const __nv_bfloat16* embed;
  // activations
  float* h;                 // [T][d] fp32 residual stream
  float* ssq;               // [ceil(d / 128)][ssq_ld] partial sums of squares of h per 128-row tile
  int ssq_ld;
  __nv_bfloat16* x;         // [Xrows][d] B operand of the QKV / gate-up GEMMs: bf16(g * h) (the norm's
                            // per-token scale is applied in their epilogues); the LM head's: the
                            // final norm's rows
  __nv_bfloat16* q;         // [T][d]
  __nv_bfloat16* att;       // [Xrows][d]
  __nv_bfloat16* act;       // [Xrows][ffn]
  float* logits;            // [n_out][1024]
  // KV caches: layer l at kc + l * layer_elems
  __nv_bfloat16* kc;
  __half* vc;
  size_t layer_elems;
  // per token
  const int* tok;
  const int* pos;
  const int* kv_row;
  const int* out_rows;      // [n_out] rows of h that get logits
  const float* rope_cos;
  const float* rope_sin;
  // attention (k_cache / v_cache of `att_args` are set per layer inside the kernel)
  AttnArgs att_args;
  int att_items;            // n_qtiles * H * max_splits
  int* att_counters;        // [n_qtiles * H], zeroed before the launch (split arrivals, all layers)
  // GEMM split-K scratch
  float* ws;
  int* counters;            // zero, left zero
  int* sk_counters;         // [GEMM phases][G] split-tile arrivals of phases with whole tiles per CTA,
                            // zeroed before the launch
  // grid barrier: monotonic arrival counter, zeroed before the launch
  unsigned int* bar;
  unsigned int* err;
  unsigned long long* trace;  // optional [16][phases][G] globaltimer stamps (phase end, producer and epilogue milestones), or null
};

// Shared memory the persistent kernel needs for (head_dim, token tile) = (hd, bn).
size_t fwd_smem_bytes(int hd, int bn);

// Launches the persistent forward (cooperative, grid = p.G).  p.T decides the token tile
// (128 up to 128 tokens, else 256).
cudaError_t fwd_launch(const FwdParams& p, cudaStream_t st);

}  // namespace atspeed
