// Stateless operator entry points of include/atspeed.h (GEMM, SwiGLU GEMM, RMSNorm, tree attention)
// on caller-owned device buffers.  Used by the parity tests and by callers composing their own loop.
#include <cuda.h>
#include <cuda_runtime.h>

#include <stdint.h>

#include <algorithm>
#include <cstring>
#include <mutex>
#include <vector>

#include "atspeed.h"
#include "attention.cuh"
#include "gemm.cuh"
#include "common.cuh"
#include "kernels.cuh"

using namespace atspeed;

namespace {

int current_grid() {
  int dev = 0;
  cudaGetDevice(&dev);
  return gemm_grid_size(dev);
}

GemmScratch scratch_from(void* ws) {
  const int G = current_grid();
  GemmScratch s;
  s.ws = static_cast<float*>(ws);
  s.ws_bytes = gemm_ws_bytes(G);
  s.counters = reinterpret_cast<int*>(static_cast<char*>(ws) + s.ws_bytes);
  s.max_tiles = gemm_max_tiles();
  s.err = reinterpret_cast<unsigned int*>(static_cast<char*>(ws) + s.ws_bytes + (size_t)s.max_tiles * 4);
  return s;
}

// gemm_launch result -> status: a refused shape is E_SHAPE, an operand the tensor-map encoder
// refuses (misaligned base address) is E_ARG, any other launch failure is E_CUDA.
atspeed_status gemm_status(cudaError_t e) {
  if (e == cudaSuccess) return ATSPEED_OK;
  if (e == cudaErrorInvalidValue) return ATSPEED_E_SHAPE;
  if (e == kGemmMapError) return ATSPEED_E_ARG;
  return ATSPEED_E_CUDA;
}

atspeed_status run_gemm(cudaStream_t st, const GemmArgs& a, void* ws) {
  if (!ws) return ATSPEED_E_ARG;
  char eb[256];
  return gemm_status(gemm_launch(a, scratch_from(ws), current_grid(), st, false, eb, sizeof eb));
}

// ---------------------------------------------------------------------------------------------
// Allocation-free GEMM: its split-K scratch lives in a fixed device array of this library.
// ---------------------------------------------------------------------------------------------
constexpr int kNoAllocGrid = 32;        // CTAs of the persistent grid (caps the workspace)
constexpr int kNoAllocTiles = 4096;     // output tiles (128 weight rows x up to 256 tokens)
constexpr size_t kNoAllocWsBytes = (size_t)2 * kNoAllocGrid * 256 * 128 * sizeof(float);  // 8 MiB
constexpr size_t kNoAllocBytes = kNoAllocWsBytes + (size_t)kNoAllocTiles * sizeof(int) + 256;

// One copy per GPU that loads the library, held until the process exits.  Host code must not use
// this name as an address: the device address comes from cudaGetSymbolAddress (per device).
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[64] = {nullptr};

// Device address of the allocation-free scratch on the current device, looked up on first use.
void* noalloc_base() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return nullptr;
    g_noalloc_ptr[dev] = ptr;
  }
  return g_noalloc_ptr[dev];
}

unsigned int* noalloc_err_word(void* base) {
  return reinterpret_cast<unsigned int*>(static_cast<char*>(base) + kNoAllocWsBytes + (size_t)kNoAllocTiles * 4);
}

}  // namespace

extern "C" {

size_t atspeed_op_workspace_bytes(void) {
  return gemm_ws_bytes(current_grid()) + (size_t)gemm_max_tiles() * 4 + 256;
}

atspeed_status atspeed_op_gemm(atspeed_stream stream, const void* d_W, const void* d_X, int M, int K, int T, int x_rows,
                               float* d_Y, int ldy, int accumulate, void* d_ws) {
  if (!d_W || !d_X || !d_Y || M <= 0 || K <= 0 || T <= 0 || ldy < M) return ATSPEED_E_ARG;
  GemmArgs a = {};
  a.epi = accumulate ? EPI_RESID : EPI_F32;
  a.W = static_cast<const __nv_bfloat16*>(d_W);
  a.X = static_cast<const __nv_bfloat16*>(d_X);
  a.M = M;
  a.K = K;
  a.T = T;
  a.X_rows = x_rows;
  a.out_f32 = d_Y;
  a.ldo = ldy;
  return run_gemm((cudaStream_t)stream, a, d_ws);
}

atspeed_status atspeed_op_gemm_swiglu(atspeed_stream stream, const void* d_W, const void* d_X, int F, int K, int T,
                                      int x_rows, void* d_out, int ldo, void* d_ws) {
  // the epilogue stores two adjacent bf16 outputs at once: ldo even, d_out 4-byte aligned
  if (!d_W || !d_X || !d_out || F <= 0 || K <= 0 || T <= 0 || ldo < F || (ldo & 1) ||
      (reinterpret_cast<uintptr_t>(d_out) & 3))
    return ATSPEED_E_ARG;
  GemmArgs a = {};
  a.epi = EPI_SWIGLU;
  a.W = static_cast<const __nv_bfloat16*>(d_W);
  a.X = static_cast<const __nv_bfloat16*>(d_X);
  a.M = 2 * F;
  a.K = K;
  a.T = T;
  a.X_rows = x_rows;
  a.out_bf16 = static_cast<__nv_bfloat16*>(d_out);
  a.ldo = ldo;
  return run_gemm((cudaStream_t)stream, a, d_ws);
}

atspeed_status atspeed_op_rmsnorm(atspeed_stream stream, const float* d_h, const void* d_g, int T, int d, float eps,
                                  void* d_x, int ldx) {
  if (!d_h || !d_g || !d_x || T <= 0 || d <= 0 || ldx < d) return ATSPEED_E_ARG;
  const cudaError_t e = rmsnorm_launch(d_h, nullptr, nullptr, nullptr, static_cast<const __nv_bfloat16*>(d_g), T, d,
                                       eps, static_cast<__nv_bfloat16*>(d_x), ldx, (cudaStream_t)stream, false);
  return e == cudaSuccess ? ATSPEED_OK : ATSPEED_E_CUDA;
}

size_t atspeed_op_attention_scratch(int T, int n_heads, int head_dim, int P) {
  const int pages = (P + ATT_PAGE - 1) / ATT_PAGE;
  const int S = std::max(1, (pages + 1) / 2);
  const int nqt = (T + ATT_QTILE - 1) / ATT_QTILE;
  const size_t floats = (size_t)S * T * n_heads * head_dim + (size_t)S * T * n_heads * 2;
  const size_t ints = (size_t)4 * nqt + (size_t)T * 7 + pages + 1;
  return floats * 4 + ints * 4 + 256;
}

atspeed_status atspeed_op_attention(atspeed_stream stream, const void* d_q, const void* d_kcache, const void* d_vcache,
                                    int cache_rows, int T, int n_heads, int head_dim, int P, const int32_t* h_pages,
                                    const int32_t* h_vis, const int32_t* h_path_rows, const int32_t* h_n_path,
                                    void* d_out, void* d_part) {
  if (!d_q || !d_kcache || !d_vcache || !d_out || !d_part || !h_pages || !h_vis || T <= 0 || P < 0 ||
      cache_rows <= 0)
    return ATSPEED_E_ARG;
  if (head_dim != 32 && head_dim != 64 && head_dim != 128) return ATSPEED_E_SHAPE;
  cudaStream_t st = (cudaStream_t)stream;
  const int pages = (P + ATT_PAGE - 1) / ATT_PAGE;
  const int S = std::max(1, (pages + 1) / 2);
  const int nqt = (T + ATT_QTILE - 1) / ATT_QTILE;
  for (int p = 0; p < pages; ++p)
    if (h_pages[p] < 0 || (h_pages[p] + 1) * ATT_PAGE > cache_rows) return ATSPEED_E_ARG;
  for (int t = 0; t < T; ++t) {
    if (h_vis[t] < 0 || h_vis[t] > P) return ATSPEED_E_ARG;
    const int np = h_n_path ? h_n_path[t] : 0;
    if (np < 0 || np > ATT_MAX_ANC) return ATSPEED_E_ARG;
    for (int j = 0; j < np; ++j)
      if (h_path_rows[t * 4 + j] < 0 || h_path_rows[t * 4 + j] >= cache_rows) return ATSPEED_E_ARG;
  }
  float* part_o = static_cast<float*>(d_part);
  float* part_ml = part_o + (size_t)S * T * n_heads * head_dim;
  int* ip = reinterpret_cast<int*>(part_ml + (size_t)S * T * n_heads * 2);
  std::vector<int> host(4 * nqt + 7 * T + pages + 1, 0);
  int* qt0 = host.data();
  int* qtn = qt0 + nqt;
  int* qtu = qtn + nqt;
  int* tu = qtu + nqt;
  int* tv = tu + T;
  int* an = tv + T;
  int* ann = an + 4 * T;
  int* pg = ann + T;
  int* sp = pg + pages;
  int* qtv = sp + 1;
  for (int i = 0; i < nqt; ++i) {
    qt0[i] = i * ATT_QTILE;
    qtn[i] = std::min(ATT_QTILE, T - i * ATT_QTILE);
    qtu[i] = 0;
  }
  for (int t = 0; t < T; ++t) {
    tv[t] = h_vis[t];
    qtv[t / ATT_QTILE] = std::max(qtv[t / ATT_QTILE], h_vis[t]);
    ann[t] = h_n_path ? h_n_path[t] : 0;
    for (int j = 0; j < 4; ++j) an[t * 4 + j] = (h_path_rows && j < ann[t]) ? h_path_rows[t * 4 + j] : 0;
  }
  for (int p = 0; p < pages; ++p) pg[p] = h_pages[p];
  sp[0] = S;
  if (cudaMemcpyAsync(ip, host.data(), host.size() * 4, cudaMemcpyHostToDevice, st) != cudaSuccess) return ATSPEED_E_CUDA;
  const int d = n_heads * head_dim;
  CUtensorMap mk, mv;
  char eb[256];
  if (!attn_make_maps(static_cast<const __nv_bfloat16*>(d_kcache), static_cast<const __half*>(d_vcache),
                      cache_rows, d, head_dim, &mk, &mv, eb, sizeof eb))
    return ATSPEED_E_CUDA;
  AttnArgs a = {};
  a.T = T;
  a.n_heads = n_heads;
  a.head_dim = head_dim;
  a.q = static_cast<const __nv_bfloat16*>(d_q);
  a.k_cache = static_cast<const __nv_bfloat16*>(d_kcache);
  a.v_cache = static_cast<const __half*>(d_vcache);
  a.kv_rows = cache_rows;
  a.n_qtiles = nqt;
  const int off_qt0 = 0, off_qtn = nqt, off_qtu = 2 * nqt, off_tu = 3 * nqt, off_tv = off_tu + T, off_an = off_tv + T,
            off_ann = off_an + 4 * T, off_pg = off_ann + T, off_sp = off_pg + pages, off_qtv = off_sp + 1;
  a.qt_t0 = ip + off_qt0;
  a.qt_n = ip + off_qtn;
  a.qt_user = ip + off_qtu;
  a.qt_vis = ip + off_qtv;
  a.tok_user = ip + off_tu;
  a.tok_vis = ip + off_tv;
  a.anc_row = ip + off_an;
  a.anc_n = ip + off_ann;
  a.page_table = ip + off_pg;
  a.max_pages = std::max(1, pages);
  a.user_splits = ip + off_sp;
  a.chunks_per_split = 2;
  a.max_splits = S;
  a.out = static_cast<__nv_bfloat16*>(d_out);
  a.part_o = part_o;
  a.part_ml = part_ml;
  a.direct = false;
  a.err = nullptr;
  const cudaError_t e = attn_launch(a, mk, mv, st, false);
  return e == cudaSuccess ? ATSPEED_OK : ATSPEED_E_CUDA;
}

/* See include/atspeed.h.  The device address of the scratch array is looked up once per device, on
 * that device's first call (so the first call on a device should come before any stream capture). */
atspeed_status atspeed_op_gemm_noalloc(atspeed_stream stream, const void* d_W, const void* d_X, int M, int K, int T,
                                       int x_rows, float* d_Y, int ldy, int accumulate) {
  if (!d_W || !d_X || !d_Y || M <= 0 || K <= 0 || T <= 0 || ldy < M) return ATSPEED_E_ARG;
  const int BN = T <= 128 ? 128 : 256;
  const long long tiles = (long long)((M + 127) / 128) * ((T + BN - 1) / BN);
  if (tiles > kNoAllocTiles || K % 64 != 0 || K / 64 > 256) return ATSPEED_E_SHAPE;
  void* base = noalloc_base();
  if (!base) return ATSPEED_E_CUDA;
  GemmScratch s;
  s.ws = static_cast<float*>(base);
  s.ws_bytes = kNoAllocWsBytes;
  s.counters = reinterpret_cast<int*>(static_cast<char*>(base) + kNoAllocWsBytes);
  s.max_tiles = kNoAllocTiles;
  s.err = noalloc_err_word(base);
  // the tile counters must start at zero (a call that failed part-way could have left some set);
  // the error word after them is left alone: it is sticky until atspeed_op_status reads it
  if (cudaMemsetAsync(s.counters, 0, (size_t)kNoAllocTiles * sizeof(int), (cudaStream_t)stream) != cudaSuccess)
    return ATSPEED_E_CUDA;
  GemmArgs a = {};
  a.epi = accumulate ? EPI_RESID : EPI_F32;
  a.W = static_cast<const __nv_bfloat16*>(d_W);
  a.X = static_cast<const __nv_bfloat16*>(d_X);
  a.M = M;
  a.K = K;
  a.T = T;
  a.X_rows = x_rows;
  a.out_f32 = d_Y;
  a.ldo = ldy;
  char eb[256];
  return gemm_status(gemm_launch(a, s, kNoAllocGrid, (cudaStream_t)stream, false, eb, sizeof eb));
}

/* See include/atspeed.h.  Reads (and clears) the error word that the op GEMMs' bounded waits set. */
atspeed_status atspeed_op_status(atspeed_stream stream, void* d_ws) {
  unsigned int* word = nullptr;
  if (d_ws) {
    word = scratch_from(d_ws).err;
  } else {
    void* base = noalloc_base();
    if (!base) return ATSPEED_E_CUDA;
    word = noalloc_err_word(base);
  }
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaStreamSynchronize(st) != cudaSuccess) return ATSPEED_E_CUDA;
  unsigned int v = 0;
  if (cudaMemcpy(&v, word, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return ATSPEED_E_CUDA;
  if (v == 0) return ATSPEED_OK;
  if (cudaMemset(word, 0, sizeof v) != cudaSuccess) return ATSPEED_E_CUDA;
  return (v & ATSPEED_DEV_ERR_TIMEOUT) ? ATSPEED_E_TIMEOUT : ATSPEED_E_CUDA;
}

}  // extern "C"
