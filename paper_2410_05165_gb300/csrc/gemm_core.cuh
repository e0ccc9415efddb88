// Shared pieces of the tcgen05 GEMM: tile constants and the fused epilogue of one 32-token chunk.
#pragma once
#include "common.cuh"
#include "gemm.cuh"

namespace atspeed {

constexpr int GEMM_BK = 64;    // bf16 elements per 128-byte swizzle row (one k-block)
constexpr int GEMM_BM = 128;   // weight rows per tile (MMA M)
constexpr int GEMM_WS_SLOT_FLOATS = 256 * 128;

// ---- work split of a tiled GEMM over G CTAs (tiles of kb k-blocks)
// Each CTA takes q = tiles / G whole tiles; the first r = tiles % G tiles are split by k-blocks into
// G equal contiguous unit ranges (stream-K; unit = one tile's k-block).  A CTA works on its
// stream-K units first and then on its whole tiles r + c, r + c + G, ..., r + c + (q - 1) G, so the
// partial sums of the split tiles are published early and the tail after the last MMA is
// whole-tile epilogues.  Whole tiles go round robin: at each step the grid works on G consecutive
// tiles, i.e. (the token-tile index varying fastest) on every token tile of a few weight row tiles,
// so each weight tile is read from DRAM about once per step and shared through L2 by the CTAs
// that need it, where a contiguous range per CTA would have one CTA read it once per token tile.
// With tiles < G (q = 0) this is plain stream-K over all tiles.
struct WorkSplit {
  int tiles, kb, q, r;
  long long Usk;   // stream-K units: r * kb
  int Gsk;         // CTAs that get stream-K units: min(G, Usk)
  int G;           // CTAs that take work (any others of the grid idle in this GEMM)
};

__host__ __device__ inline WorkSplit work_split(int tiles, int kb, int G) {
  WorkSplit w;
  w.tiles = tiles;
  w.kb = kb;
  w.q = tiles / G;
  w.r = tiles - w.q * G;
  w.Usk = (long long)w.r * kb;
  w.Gsk = (int)(w.Usk < (long long)G ? w.Usk : (long long)G);
  w.G = G;
  return w;
}

// CTAs that take work in a GEMM of `tiles` tiles of kb k-blocks on a grid of `grid` CTAs.  With
// fewer tiles than CTAs, the first `tiles` CTAs take one whole tile each (and the others idle) when
// that costs at most 8 k-blocks more per CTA than spreading the k-blocks over the grid: every split
// tile ends in a sum of its parts whose latency outweighs a short stream (a small model's QKV
// projection).  Both the per-op GEMM and the persistent forward take their split from here, so
// their sums are the same bit for bit.
__host__ __device__ inline int gemm_work_ctas(long long tiles, int kb, int grid) {
  if (tiles < grid && (long long)kb * (grid - tiles) <= 8LL * grid) return (int)tiles;
  const long long U = tiles * kb;
  return (int)(U < (long long)grid ? U : (long long)grid);
}
// stream-K unit range [a, b) of CTA c
__device__ __forceinline__ void sk_range(const WorkSplit& w, int c, long long& a, long long& b) {
  if (c >= w.Gsk) {
    a = b = 0;
    return;
  }
  a = (long long)c * w.Usk / w.Gsk;
  b = (long long)(c + 1) * w.Usk / w.Gsk;
}
__device__ __forceinline__ long long sk_start(const WorkSplit& w, long long c) { return c * w.Usk / w.Gsk; }
__device__ __forceinline__ int sk_owner(const WorkSplit& w, long long u) {
  return (int)(((u + 1) * (long long)w.Gsk - 1) / w.Usk);
}
// number of units of CTA c, and its i-th unit as (tile, k-block)
__device__ __forceinline__ long long cta_units(const WorkSplit& w, int c) {
  if (c >= w.G) return 0;
  long long a, b;
  sk_range(w, c, a, b);
  return (b - a) + (long long)w.q * w.kb;
}
__device__ __forceinline__ void cta_unit(const WorkSplit& w, int c, long long i, int& tile, int& kbi) {
  long long a, b;
  sk_range(w, c, a, b);
  if (i < b - a) {
    const long long u = a + i;
    tile = (int)(u / w.kb);
    kbi = (int)(u - (long long)tile * w.kb);
  } else {
    const long long j = i - (b - a);
    const int t = (int)(j / w.kb);
    tile = w.r + t * w.G + c;
    kbi = (int)(j - (long long)t * w.kb);
  }
}
// the segments (one tile's contiguous k-blocks [k0, k1)) of CTA c in order
struct SegIter {
  long long u, u1;
  int dp, dp1;
  __device__ __forceinline__ void init(const WorkSplit& w, int c) {
    if (c >= w.G) {
      u = u1 = 0;
      dp = dp1 = 0;
      return;
    }
    sk_range(w, c, u, u1);
    dp = w.r + c;                // whole tiles r + c, r + c + G, ... (round robin)
    dp1 = w.r + w.q * w.G + c;
  }
  __device__ __forceinline__ bool next(const WorkSplit& w, int& tile, int& k0, int& k1) {
    if (u < u1) {
      tile = (int)(u / w.kb);
      k0 = (int)(u - (long long)tile * w.kb);
      const long long len = (w.kb - k0) < (u1 - u) ? (w.kb - k0) : (u1 - u);
      k1 = k0 + (int)len;
      u += len;
      return true;
    }
    if (dp < dp1) {
      tile = dp;
      dp += w.G;
      k0 = 0;
      k1 = w.kb;
      return true;
    }
    return false;
  }
  __device__ __forceinline__ bool more() const { return u < u1 || dp < dp1; }
};

// Per-token data of the QKV epilogue for the BN tokens of n-tile n_tile (rotary position and cache
// row), copied to shared memory when a segment starts so that the epilogue's loads do not wait on
// them.  Callers synchronise the 128 threads before the first chunk's epilogue.
template <int BN>
__device__ __forceinline__ void load_tok_tables(const GemmArgs& a, int n_tile, int* tpos, int* tkvr, int ep_tid,
                                                int nthreads = 128) {
  for (int j = ep_tid; j < BN; j += nthreads) {
    const int tok = n_tile * BN + j;
    tpos[j] = tok < a.T ? a.pos[tok] : 0;
    tkvr[j] = tok < a.T ? a.kv_row[tok] : 0;
  }
}

// ---- RMSNorm folded into the GEMMs around it
// Sum of squares of 32 values v(0 .. 31) in the rotated order rot, rot + 1, ... (mod 32), one fused
// multiply-add per value.  A token's partial sum over a 128-row tile of the residual is
// (q0 + q1) + (q2 + q3), q_s = ssq32 over rows 32 s .. 32 s + 31 of the tile with rot = ssq_rot(s);
// rows past d count as zero.  Every producer of partial sums (the O / down epilogue, the embedding
// rows) uses exactly these orders, and none depends on the token's index in the call, so a token's
// sums depend neither on the kernel or schedule that made them nor on the other tokens of the call.
template <class F>
__device__ __forceinline__ float ssq32(F v, int rot) {
  float x[32];   // every value loaded first, then the dependent chain
#pragma unroll
  for (int i = 0; i < 32; ++i) x[i] = v((i + rot) & 31);
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 32; ++i) s = __fmaf_rn(x[i], x[i], s);
  return s;
}
// (the four quarters start on different banks of the staging rows)
__device__ __forceinline__ int ssq_rot(int sub) { return sub * 8; }

// 1 / rms of token t (RMSNorm's per-token scale) from its partial sums, added in tile order.
__device__ __forceinline__ float norm_scale(const float* ssq, int ld, int d, float eps, int t) {
  const int nt = (d + GEMM_BM - 1) / GEMM_BM;
  float s = 0.f;
#pragma unroll 8
  for (int mt = 0; mt < nt; ++mt) s += __ldcg(ssq + (size_t)mt * ld + t);
  return 1.0f / sqrtf(s / (float)d + eps);
}

// The scales of the BN tokens of n-tile n_tile into trs (shared memory); callers synchronise
// before the epilogue reads them.
template <int BN>
__device__ __forceinline__ void load_norm_scales(const GemmArgs& a, int n_tile, float* trs, int tid, int nthreads) {
  for (int j = tid; j < BN; j += nthreads) {
    const int tok = n_tile * BN + j;
    trs[j] = tok < a.T ? norm_scale(a.ssq_in, a.ssq_ld, a.nrm_d, a.eps, tok) : 0.f;
  }
}

// Partial sums of squares of the updated residual of tokens j0 .. j0 + NJ - 1 of a chunk (st holds
// them, [token][128 rows]), nv of them valid: 4 threads per token (warps 0 .. NJ / 8 - 1), token jj
// of the range, quarter sub of the rows.
// sr: the first of those tokens' rows, SR floats apart (the order of the sums does not depend on
// where the rows sit: a row stride of 132 spreads a warp's eight tokens over the banks).
template <int NJ, int SR = GEMM_BM>
__device__ __forceinline__ void resnorm_ssq(const GemmArgs& a, const float* sr, int m_tile, int tok0, int j0, int nv,
                                            int ep_tid) {
  if (ep_tid < 4 * NJ) {
    const int jj = ep_tid >> 2, sub = ep_tid & 3, j = j0 + jj;
    const float* sj = sr + jj * SR + sub * 32;
    float s = ssq32([&](int r) { return sj[r]; }, ssq_rot(sub));
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    if (sub == 0 && jj < nv) a.ssq_out[(size_t)m_tile * a.ssq_ld + tok0 + j] = s;
  }
}

// The updated residual of tokens j0 .. j0 + NJ - 1 of a chunk (st, [token][128 rows]; nv of them
// valid) to h and bf16(g * h) to xg: a thread stores four adjacent rows (one 16-byte h store, one
// 8-byte xg store per token), warp w the tokens j0 + w NJ / 4 .., so a warp's store covers a token's
// 128 rows in one piece.  (M, the residual's width, is a multiple of 4.)
template <int NJ, int SR = GEMM_BM>
__device__ __forceinline__ void resnorm_store(const GemmArgs& a, const float* sr, int m_tile, int tok0, int j0, int nv,
                                              int ep_tid) {
  constexpr int TPW = NJ / 4;   // tokens per warp
  const int rq = ep_tid & 31, w = ep_tid >> 5;
  const int row = m_tile * GEMM_BM + 4 * rq;
  if (row >= a.M) return;
  const bool xg = a.gain != nullptr;
  float2 g01 = make_float2(0.f, 0.f), g23 = g01;
  if (xg) {
    const uint2 graw = *reinterpret_cast<const uint2*>(a.gain + row);
    const __nv_bfloat162* gb = reinterpret_cast<const __nv_bfloat162*>(&graw);
    g01 = __bfloat1622float2(gb[0]);
    g23 = __bfloat1622float2(gb[1]);
  }
#pragma unroll
  for (int k = 0; k < TPW; ++k) {
    const int n = w * TPW + k;
    if (n < nv) {
      const float4 v = *reinterpret_cast<const float4*>(sr + n * SR + 4 * rq);
      const size_t e = (size_t)(tok0 + j0 + n) * a.ldo + row;
      *reinterpret_cast<float4*>(a.out_f32 + e) = v;
      if (xg) {
        __nv_bfloat162 o[2];
        o[0] = __floats2bfloat162_rn(v.x * g01.x, v.y * g01.y);
        o[1] = __floats2bfloat162_rn(v.z * g23.x, v.w * g23.y);
        *reinterpret_cast<uint2*>(a.xg_out + e) = *reinterpret_cast<const uint2*>(o);
      }
    }
  }
}

// EPI_RESNORM over tokens j0 .. j0 + NJ - 1 of one 32-token chunk (O / down projections): h +=
// product (fp32 residual, read-modify-write; every (row, token) belongs to one chunk of one CTA),
// xg = bf16(g * h) for the next GEMM, and the partial sums of squares of the updated rows.  128
// threads (ep_tid = the tile row they own); `bar` is a named barrier of those 128 threads.  st
// (staging, [32 tokens][128 rows]) holds the product in the rows of those tokens and is overwritten
// there with the updated residual.  The arithmetic per token does not depend on NJ or j0.
template <int NJ = 32>
__device__ __forceinline__ void epi_resnorm(const GemmArgs& a, float* st, int m_tile, int tok0, int ep_tid, int bar,
                                            int j0 = 0) {
  const int nv = min(NJ, a.T - tok0 - j0);   // valid tokens of the range
  const int m = ep_tid, row = m_tile * GEMM_BM + m;
  const bool in = row < a.M;
  const float* base = a.out_f32 + (size_t)(tok0 + j0) * a.ldo + row;
  float* sb = st + j0 * GEMM_BM;
  float old[NJ];
#pragma unroll
  for (int n = 0; n < NJ; ++n) old[n] = (in && n < nv) ? __ldcg(base + (size_t)n * a.ldo) : 0.f;
#pragma unroll
  for (int n = 0; n < NJ; ++n) sb[n * GEMM_BM + m] = in ? old[n] + sb[n * GEMM_BM + m] : 0.f;
  // the sums of squares before the stores (their shared-memory reads would queue behind them)
  named_bar_sync(bar, 128);
  if (a.ssq_out != nullptr) resnorm_ssq<NJ>(a, sb, m_tile, tok0, j0, nv, ep_tid);
  resnorm_store<NJ>(a, sb, m_tile, tok0, j0, nv, ep_tid);
}

// Split-K sum (in k order, from zero) of tokens 16 half .. 16 half + 15 of chunk ch of the parts in
// `slot`, then EPI_RESNORM of those tokens: epi_resnorm<16>'s arithmetic, with the residual loads
// issued together with the first parts' loads.  PB parts in flight at once.
template <int PB>
__device__ __forceinline__ void ws_reduce_resnorm_half(const GemmArgs& a, const float* ws, const int* slot, int parts,
                                                       int ch, int half, int m_tile, int tok0, int ep_tid,
                                                       float* st, int bar) {
  const int j0 = 16 * half;
  const int nv = min(16, a.T - tok0 - j0);
  const int m = ep_tid, row = m_tile * GEMM_BM + m;
  const bool in = row < a.M;
  const float* base = a.out_f32 + (size_t)(tok0 + j0) * a.ldo + row;
  float old[16], acc[16];
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    old[n] = (in && n < nv) ? __ldcg(base + (size_t)n * a.ldo) : 0.f;
    acc[n] = 0.f;
  }
  const float4* w4 = reinterpret_cast<const float4*>(ws);
  constexpr long long SLOT4 = GEMM_WS_SLOT_FLOATS / 4;
  for (int p0 = 0; p0 < parts; p0 += PB) {
    float4 v[PB][4];
#pragma unroll
    for (int b = 0; b < PB; ++b) {
      if (p0 + b < parts) {
        const float4* src = w4 + (long long)slot[p0 + b] * SLOT4 + (ch * 8 + 4 * half) * GEMM_BM + m;
#pragma unroll
        for (int j4 = 0; j4 < 4; ++j4) v[b][j4] = __ldcg(src + j4 * GEMM_BM);
      }
    }
#pragma unroll
    for (int b = 0; b < PB; ++b) {
      if (p0 + b < parts) {
#pragma unroll
        for (int j4 = 0; j4 < 4; ++j4) {
          acc[4 * j4] += v[b][j4].x;
          acc[4 * j4 + 1] += v[b][j4].y;
          acc[4 * j4 + 2] += v[b][j4].z;
          acc[4 * j4 + 3] += v[b][j4].w;
        }
      }
    }
  }
  // the updated rows go to the start of st, 132 floats apart (16 x 132 floats fit the 32 x 128 of a
  // staging buffer; float4-aligned rows; conflict-free sums of squares)
  constexpr int SR = GEMM_BM + 4;
#pragma unroll
  for (int n = 0; n < 16; ++n) st[n * SR + m] = in ? old[n] + acc[n] : 0.f;
  named_bar_sync(bar, 128);
  if (a.ssq_out != nullptr) resnorm_ssq<16, SR>(a, st, m_tile, tok0, j0, nv, ep_tid);
  resnorm_store<16, SR>(a, st, m_tile, tok0, j0, nv, ep_tid);
}

// st: staging [32 tokens][128 rows] fp32 of one chunk; 128 threads (ep_tid) write the outputs.
// tpos / tkvr: the n-tile's token tables (EPI_QKV only); trs: the n-tile's norm scales (EPI_QKV /
// EPI_SWIGLU when the input rows are g * h, else null).
template <int BN, int EPI>
__device__ __forceinline__ void epi_chunk(const GemmArgs& a, const float* st, int m_tile, int n_tile, int ch,
                                          int ep_tid, const int* tpos, const int* tkvr, const float* trs = nullptr) {
  const int tok0 = n_tile * BN + ch * 32;
  if constexpr (EPI == EPI_QKV) {
    // rows of q | k | v.  Thread = (two adjacent rotation pairs, token quarter): pairs (i, i + hd/2)
    // and (i + 1, i + 1 + hd/2) of one head (i even) for tokens (ep_tid >> 5) + 4k, so every load of
    // the staged rows and the rotary tables and every store moves two adjacent values (rotate-half
    // RoPE, the same arithmetic per element); k / v rows go to their cache rows, v rounded to bf16
    // and kept as fp16.
    const int d = a.d_model, hd = a.head_dim, half = hd >> 1;
    const int pi = 2 * (ep_tid & 31), n0 = ep_tid >> 5;
    const int hh = pi / half, i = pi - hh * half;
    const int r_lo = hh * hd + i, r_hi = r_lo + half;     // rows within the tile (r_lo even)
    const int row = m_tile * GEMM_BM + r_lo;
    if (row >= a.M) return;                                // padding rows of the last tile
    const int region = row / d;
    const int f_lo = row - region * d, f_hi = f_lo + half;
    const int nv = min(32, a.T - tok0);
    const int tt0 = ch * 32;                               // token-table index of the chunk's first token
    if (region == 2) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int n = n0 + 4 * k;
        if (n < nv) {
          __half* vr = a.v_cache + (size_t)tkvr[tt0 + n] * d;
          float2 lo = *reinterpret_cast<const float2*>(st + n * GEMM_BM + r_lo);
          float2 hi = *reinterpret_cast<const float2*>(st + n * GEMM_BM + r_hi);
          if (trs) {
            const float sc = trs[tt0 + n];
            lo.x *= sc;
            lo.y *= sc;
            hi.x *= sc;
            hi.y *= sc;
          }
          *reinterpret_cast<__half2*>(vr + f_lo) =
              __halves2half2(__float2half_rn(bf16_round(lo.x)), __float2half_rn(bf16_round(lo.y)));
          *reinterpret_cast<__half2*>(vr + f_hi) =
              __halves2half2(__float2half_rn(bf16_round(hi.x)), __float2half_rn(bf16_round(hi.y)));
        }
      }
    } else {
      float2 cth[8], sth[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int n = n0 + 4 * k;
        const size_t cs = (size_t)tpos[tt0 + (n < nv ? n : 0)] * half + i;
        cth[k] = *reinterpret_cast<const float2*>(a.rope_cos + cs);
        sth[k] = *reinterpret_cast<const float2*>(a.rope_sin + cs);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int n = n0 + 4 * k;
        if (n < nv) {
          float2 xl = *reinterpret_cast<const float2*>(st + n * GEMM_BM + r_lo);
          float2 xh = *reinterpret_cast<const float2*>(st + n * GEMM_BM + r_hi);
          if (trs) {
            const float sc = trs[tt0 + n];
            xl.x *= sc;
            xl.y *= sc;
            xh.x *= sc;
            xh.y *= sc;
          }
          const __nv_bfloat16 o_lo0 = __float2bfloat16_rn(xl.x * cth[k].x - xh.x * sth[k].x);
          const __nv_bfloat16 o_hi0 = __float2bfloat16_rn(xh.x * cth[k].x + xl.x * sth[k].x);
          const __nv_bfloat16 o_lo1 = __float2bfloat16_rn(xl.y * cth[k].y - xh.y * sth[k].y);
          const __nv_bfloat16 o_hi1 = __float2bfloat16_rn(xh.y * cth[k].y + xl.y * sth[k].y);
          __nv_bfloat16* orow = region == 0 ? a.q_out + (size_t)(tok0 + n) * d : a.k_cache + (size_t)tkvr[tt0 + n] * d;
          *reinterpret_cast<__nv_bfloat162*>(orow + f_lo) = __halves2bfloat162(o_lo0, o_lo1);
          *reinterpret_cast<__nv_bfloat162*>(orow + f_hi) = __halves2bfloat162(o_hi0, o_hi1);
        }
      }
    }
  } else if constexpr (EPI == EPI_SWIGLU) {
    // thread owns features 2f, 2f + 1 of the tile (one 4-byte store per token) and tokens
    // (ep_tid >> 5) + 4k.  silu(g) = g / (1 + e^-g) with the hardware exponential and an
    // approximate divide (a few ulp, far below the bf16 rounding of the product; for g -> -inf the
    // divisor overflows to inf and the quotient is -0); the IEEE expf and divide made this loop
    // latency-bound (about 2 us per 32-token chunk)
    const int f = ep_tid & 31, n0 = ep_tid >> 5;
    __nv_bfloat16* out = a.out_bf16 + m_tile * 64 + 2 * f;
    const int T = a.T;
    const size_t ldo = (size_t)a.ldo;
    float2 gv[8], uv[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int n = n0 + 4 * k;
      gv[k] = *reinterpret_cast<const float2*>(st + n * GEMM_BM + 2 * f);
      uv[k] = *reinterpret_cast<const float2*>(st + n * GEMM_BM + 64 + 2 * f);
      if (trs) {
        const float sc = trs[ch * 32 + n];
        gv[k].x *= sc;
        gv[k].y *= sc;
        uv[k].x *= sc;
        uv[k].y *= sc;
      }
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int tok = tok0 + n0 + 4 * k;
      if (tok < T) {
        const float y0 = __fdividef(gv[k].x, 1.0f + __expf(-gv[k].x)) * uv[k].x;
        const float y1 = __fdividef(gv[k].y, 1.0f + __expf(-gv[k].y)) * uv[k].y;
        *reinterpret_cast<__nv_bfloat162*>(out + (size_t)tok * ldo) = __floats2bfloat162_rn(y0, y1);
      }
    }
  } else if constexpr (EPI == EPI_LSE) {
    // per token of the chunk, (max, sum of exp(y - max)) over the tile's rows: 4 threads per token
    // take 32 rows each (rotated by token and thread so the shared-memory reads spread over the
    // banks), then combine in a fixed order (pairs, then pairs of pairs)
    const int j = ep_tid >> 2, sub = ep_tid & 3;
    const int valid = min(GEMM_BM, a.M - m_tile * GEMM_BM);
    const float* sj = st + j * GEMM_BM + sub * 32;
    float mx = -INFINITY;
#pragma unroll 8
    for (int i = 0; i < 32; ++i) {
      const int r = (i + sub * 8 + j) & 31;
      if (sub * 32 + r < valid) mx = fmaxf(mx, sj[r]);
    }
    float sm = 0.f;
    if (mx != -INFINITY) {
#pragma unroll 8
      for (int i = 0; i < 32; ++i) {
        const int r = (i + sub * 8 + j) & 31;
        if (sub * 32 + r < valid) sm += expf(sj[r] - mx);
      }
    }
#pragma unroll
    for (int o = 1; o <= 2; o <<= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, mx, o), s2 = __shfl_xor_sync(0xffffffffu, sm, o);
      const float mn = fmaxf(mx, m2);
      sm = (mx == -INFINITY ? 0.f : sm * expf(mx - mn)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - mn));
      mx = mn;
    }
    const int tok = tok0 + j;
    if (sub == 0 && tok < a.T) a.lse_part[(size_t)m_tile * a.lse_ld + tok] = make_float2(mx, sm);
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
    }
  }
}

// ---- split-K partials (stream-K tiles shared by several CTAs)
// A workspace slot holds one CTA's fp32 partial of a 128-row tile for up to 256 tokens, laid out
// [token/4][row][4] so that a thread (one weight row) moves four tokens per 16-byte access.

// TMEM accumulator (this thread's lane = row m) -> workspace slot, chunks ch0, ch0 + step, ... < nch
__device__ __forceinline__ void ws_store_partial(float* wsl, uint32_t tb, int nch, int m, int ch0 = 0, int step = 1) {
  float4* w4 = reinterpret_cast<float4*>(wsl);
  for (int ch = ch0; ch < nch; ch += step) {
    uint32_t r[32];
    tmem_ld_32x32b_x32(tb + ch * 32, r);
    tmem_ld_wait();
#pragma unroll
    for (int j4 = 0; j4 < 8; ++j4)
      __stcg(&w4[(ch * 8 + j4) * GEMM_BM + m],
             make_float4(__uint_as_float(r[4 * j4]), __uint_as_float(r[4 * j4 + 1]), __uint_as_float(r[4 * j4 + 2]),
                         __uint_as_float(r[4 * j4 + 3])));
  }
}

// Sum, in k order (part 0 first, starting from zero), of chunk ch of the parts in `slot` -> this
// thread's row m of the staging buffer [32 tokens][128 rows].  PB parts are in flight at once (the
// result does not depend on PB).
template <int PB = 4>
__device__ __forceinline__ void ws_reduce_chunk(const float* ws, const int* slot, int parts, int ch, int m,
                                             float* staging) {
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  const float4* w4 = reinterpret_cast<const float4*>(ws);
  constexpr long long SLOT4 = GEMM_WS_SLOT_FLOATS / 4;
  for (int p0 = 0; p0 < parts; p0 += PB) {
    float4 v[PB][8];
#pragma unroll
    for (int b = 0; b < PB; ++b) {
      if (p0 + b < parts) {
        const float4* src = w4 + (long long)slot[p0 + b] * SLOT4 + (ch * 8) * GEMM_BM + m;
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) v[b][j4] = __ldcg(src + j4 * GEMM_BM);
      }
    }
#pragma unroll
    for (int b = 0; b < PB; ++b) {
      if (p0 + b < parts) {
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {
          acc[4 * j4] += v[b][j4].x;
          acc[4 * j4 + 1] += v[b][j4].y;
          acc[4 * j4 + 2] += v[b][j4].z;
          acc[4 * j4 + 3] += v[b][j4].w;
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) staging[j * GEMM_BM + m] = acc[j];
}

// As ws_reduce_chunk, with part `own` of the sum taken from registers (this CTA's accumulator, 32
// tokens of row m) instead of the workspace.  One part is in flight at a time.
__device__ __forceinline__ void ws_reduce_chunk_own(const float* ws, const int* slot, int parts, int own,
                                                    const uint32_t (&r)[32], int ch, int m, float* staging) {
  float acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0.f;
  const float4* w4 = reinterpret_cast<const float4*>(ws);
  constexpr long long SLOT4 = GEMM_WS_SLOT_FLOATS / 4;
  for (int pi = 0; pi < parts; ++pi) {
    if (pi == own) {
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] += __uint_as_float(r[j]);
      continue;
    }
    const float4* src = w4 + (long long)slot[pi] * SLOT4 + (ch * 8) * GEMM_BM + m;
    float4 v[8];
#pragma unroll
    for (int j4 = 0; j4 < 8; ++j4) v[j4] = __ldcg(src + j4 * GEMM_BM);
#pragma unroll
    for (int j4 = 0; j4 < 8; ++j4) {
      acc[4 * j4] += v[j4].x;
      acc[4 * j4 + 1] += v[j4].y;
      acc[4 * j4 + 2] += v[j4].z;
      acc[4 * j4 + 3] += v[j4].w;
    }
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) staging[j * GEMM_BM + m] = acc[j];
}

}  // namespace atspeed
