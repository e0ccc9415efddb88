// Launch wrappers of the non-GEMM kernels (host-visible).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "tree.cuh"

namespace atspeed {

// h_out/x rows: x[t] = bf16(rmsnorm(h[t]) * g); with `tokens`, h[t] = embed[tokens[t]] first.
cudaError_t rmsnorm_launch(const float* h, const int* tokens, const __nv_bfloat16* embed, float* h_out,
                           const __nv_bfloat16* g, int T, int d, float eps, __nv_bfloat16* x, int ldx,
                           cudaStream_t st, bool pdl);

// Layer 0's rows with the first norm folded into the QKV GEMM: h[t] = embed[tokens[t]],
// xg[t] = bf16(g * h[t]), ssq[mt * ld + t] = partial sums of squares of h[t] per 128-row tile.
cudaError_t embed_rows_launch(const int* tokens, const __nv_bfloat16* embed, const __nv_bfloat16* g, float* h,
                              __nv_bfloat16* xg, float* ssq, int ld, int T, int d, cudaStream_t st, bool pdl);

// x[i] = bf16(rmsnorm(h[rows[i]]) * g) for i < n (final norm of the tokens whose logits are needed)
cudaError_t rmsnorm_rows_launch(const float* h, const int* rows, int n, const __nv_bfloat16* g, int d, float eps,
                                __nv_bfloat16* x, int ldx, cudaStream_t st, bool pdl);

size_t select_smem_bytes(int max_parents);
cudaError_t draft_level_launch(const TreeDev& t, int lvl, int N, bool relaxed, uint64_t seed, cudaStream_t st,
                               bool pdl);
// probe: decide level 1 only (see verify_strict_kernel); users whose level 1 is accepted get
// accepted = -1 and must be verified again by a full launch
cudaError_t verify_launch(const TreeDev& t, int K, bool relaxed, uint64_t seed, const VerifyOut& o, cudaStream_t st,
                          bool pdl, bool probe = false);

// Per-token inputs of a forward over tree nodes, read from the node table.
struct FwdTokens {
  int* tok;        // [T] token id
  int* pos;        // [T] rotary position
  int* kv_row;     // [T] own cache row
  int* tok_user;   // [T]
  int* tok_vis;    // [T] visible prefix length
  int* anc_row;    // [T][4]
  int* anc_n;      // [T]
};
// fwd_nodes[i]: global node index of token i; user_P[u]: prompt length.  Also stores the logits row
// (row_base + i) of every node into lg_t (target == true) or lg_d.
cudaError_t tree_gather_launch(const TreeDev& t, const int* fwd_nodes, int T, const int* user_P, int code_base,
                               bool target, int row_base, const FwdTokens& f, cudaStream_t st, bool pdl);

}  // namespace atspeed
