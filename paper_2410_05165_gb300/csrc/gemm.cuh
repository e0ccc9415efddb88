// Host-visible declarations of the weight-streaming GEMM (tcgen05 + TMA + TMEM).
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace atspeed {

enum EpiKind : int { EPI_F32 = 0, EPI_BF16 = 1, EPI_RESID = 2, EPI_SWIGLU = 3, EPI_QKV = 4, EPI_LSE = 5, EPI_RESNORM = 6 };

// Y[t][m] = sum_k W[m][k] * X[t][k]  (W: weight rows, X: token rows, both bf16 K-major)
// with a fused epilogue.  The MMA runs "swap-AB": weight rows are the MMA M dimension (128 per
// tile), tokens are the MMA N dimension (128 or 256 per tile), so a handful of tokens still
// fills the tensor core while the weights stream from HBM exactly once.
struct GemmArgs {
  EpiKind epi;
  const __nv_bfloat16* W;   // [M_rows][K]
  const __nv_bfloat16* X;   // [X_rows][K], X_rows >= round_up(T, BN) (rows >= T are ignored)
  int M;                    // weight rows (for EPI_SWIGLU: 2 * d_ffn, gate rows then up rows)
  int K;                    // reduction length, multiple of 64
  int T;                    // tokens
  int X_rows;               // allocated token rows of X
  // RMSNorm folded into the GEMMs around it (LLaMA pre-norm: x = h / rms(h) * g; the per-token
  // scale 1 / rms(h) commutes with the projection, so W x = (W (g h)) / rms(h)):
  //  * EPI_RESNORM (O / down projections): h += product, then xg = bf16(g * h) and, per 128-row
  //    tile mt of h, the token's partial sum of squares ssq[mt * ssq_ld + t];
  //  * EPI_QKV / EPI_SWIGLU with ssq_in set: the product is multiplied by the token's
  //    1 / sqrt(sum_mt ssq[mt][t] / nrm_d + eps) before the epilogue's arithmetic.
  const float* ssq_in;      // partial sums of the GEMM input's rows (null: no scaling)
  float* ssq_out;           // EPI_RESNORM: partial sums of the updated residual (null: none)
  int ssq_ld;               // token stride of the partial sums
  int nrm_d;                // norm width (d_model); its ceil(d / 128) tiles are summed
  float eps;
  const __nv_bfloat16* gain;  // EPI_RESNORM: gain of the next norm (null: only h is written)
  __nv_bfloat16* xg_out;      // EPI_RESNORM: [T][ldo] bf16(g * h), the next GEMM's input
  // outputs
  float* out_f32;           // EPI_F32 / EPI_RESID / EPI_RESNORM: [T][ldo]
  __nv_bfloat16* out_bf16;  // EPI_BF16 / EPI_SWIGLU: [T][ldo]
  int ldo;
  // EPI_LSE: per (weight-row tile, token) the tile's (max, sum of exp(y - max)) over its rows,
  // lse_part[m_tile * lse_ld + token] (the logits themselves are not stored)
  float2* lse_part;
  int lse_ld;
  // EPI_QKV
  int d_model, head_dim;
  const int* pos;           // [T] rotary positions
  const int* kv_row;        // [T] destination row of k / v in the caches
  const float* rope_cos;    // [max_pos][head_dim / 2]
  const float* rope_sin;
  __nv_bfloat16* q_out;     // [T][d_model]
  __nv_bfloat16* k_cache;   // [rows][d_model]
  __half* v_cache;          // [rows][d_model]: v rounded to bf16, stored exactly as fp16
};

struct GemmScratch {
  float* ws;                // split partials: [2 * grid][256][128] fp32
  int* counters;            // [max tiles], zero-initialised, restored to zero by every launch
  size_t ws_bytes;
  int max_tiles;
  unsigned int* err;        // device error word
};

// log-sum-exp of each token's whole row from the EPI_LSE partials of m_tiles row tiles, combined in
// tile order: lse[t] = log sum_m s_m exp(max_m - max) + max.
cudaError_t lse_combine_launch(const float2* part, int ld, int m_tiles, int T, float* lse, cudaStream_t st);

// Bytes of split-K workspace / counters needed for a grid of `grid` CTAs.
size_t gemm_ws_bytes(int grid);
int gemm_max_tiles();
// Number of CTAs of the persistent stream-K grid (one per SM).
int gemm_grid_size(int device);

// 2D bf16 tensor map over a row-major [rows][inner] matrix, box {64, box_rows}, 128B swizzle.
bool gemm_make_map(CUtensorMap* m, const void* base, int inner, int rows, int box_rows, char* eb, size_t el);

// gemm_launch's return value when an operand cannot be described by a tensor map (its base
// address or row pitch breaks the TMA alignment rules); cudaErrorInvalidValue means a bad shape.
constexpr cudaError_t kGemmMapError = cudaErrorInvalidDevicePointer;

// Encodes the tensor maps and launches.  `pdl` enables programmatic dependent launch.
cudaError_t gemm_launch(const GemmArgs& a, const GemmScratch& s, int grid, cudaStream_t stream, bool pdl,
                        char* errbuf, size_t errlen);

}  // namespace atspeed
