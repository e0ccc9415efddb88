// Weight-streaming GEMM for sm_103a: TMA -> shared memory (128B swizzle) -> tcgen05.mma with the
// fp32 accumulator in TMEM -> tcgen05.ld epilogue with fused QKV+RoPE+KV-store / SwiGLU /
// residual-add (with the next RMSNorm's partial sums) / plain stores.
//
// Decomposition ("stream-K"): the work units are (tile, 64-wide k-block) pairs, tile = (weight-row
// tile of 128, token tile of BN), ordered weight-tile-major.  A persistent grid of one CTA per SM
// takes equal contiguous ranges of units, so every SM streams the same number of weight bytes
// whatever the matrix shape.  A tile whose k-range spans several CTAs is reduced through an fp32
// workspace by the last CTA to finish it (fixed summation order, hence deterministic), which then
// runs the fused epilogue.  The partition depends only on (M, K, the number of token tiles and the
// grid), so a token's output does not depend on the other tokens of the call as long as the calls
// compared have the same number of token tiles (one tile up to 256 tokens); with more token tiles
// the k-split, and so the order of the fp32 sums, can differ.
//
// Roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM allocator + MMA issuer, warps 2-5 =
// epilogue (TMEM lane quadrant = warp % 4).  Two TMEM accumulators alternate between segments so
// the next segment's MMAs overlap the previous segment's epilogue.
#include <cudaTypedefs.h>
#include <stdio.h>

#include "common.cuh"
#include "gemm.cuh"
#include "gemm_core.cuh"

namespace atspeed {

namespace {

constexpr int BK = 64;            // bf16 elements per 128-byte swizzle row
constexpr int BM = 128;           // weight rows per tile (MMA M)
constexpr int WS_SLOT_FLOATS = 256 * 128;
constexpr int MAX_TILES = 1 << 16;

template <int BN>
struct Cfg {
  static constexpr int STAGES = (BN == 128) ? 6 : 4;
  static constexpr int A_BYTES = BM * 128;
  static constexpr int B_BYTES = BN * 128;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGING_FLOATS = 32 * BM;
  static constexpr int BAR_BYTES = 256 + 1024 + 2048 + 1024;  // barriers, flags, split-part slot table, token
                                                              // tables, norm scales
  static constexpr int SMEM = 1024 + STAGES * STAGE_BYTES + STAGING_FLOATS * 4 + BAR_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;
};

struct KParams {
  GemmArgs a;
  int m_tiles, n_tiles, kb;
  WorkSplit w;   // whole tiles per CTA + stream-K over the remaining tiles
  int G;
  int up_row0;
  float* ws;
  int* counters;
  unsigned int* err;
};


template <int BN, int EPI>
__global__ void __launch_bounds__(192, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const KParams p) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* staging = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* full = reinterpret_cast<uint64_t*>(staging + C::STAGING_FLOATS);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  int* flag = reinterpret_cast<int*>(tmem_slot + 1);
  int* failed = flag + 1;
  int* last_fill = failed + 1;  // [STAGES]: parity of the last fill issued per stage, -1 if none
  int* part_slot = last_fill + 8;  // [<= 256] workspace slots of a split tile's parts
  int* tpos = part_slot + 256;     // [BN] QKV epilogue token tables of the current n-tile
  int* tkvr = tpos + 256;
  float* trs = reinterpret_cast<float*>(tkvr + 256);   // [BN] norm scales of the current n-tile

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x;
  const long long nu = cta_units(p.w, c);   // this CTA's units (stream-K units, then whole tiles)
  const int kb = p.kb;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      last_fill[s] = -1;
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 4);
    }
    mbar_init(mma_done, 1);
    *failed = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_launch_dependents();

  if (warp == 0) {
    if (lane == 0 && nu > 0) {
      // ------------------------------------------------------------------ TMA producer
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      const uint64_t pol_w = policy_evict_first();   // weights: streamed once
      const uint64_t pol_x = policy_evict_last();    // activations: re-read by every CTA
      const long long total = nu;
      const int npre = (int)(total < C::STAGES ? total : C::STAGES);
      // units in order, walked segment by segment (no per-unit divisions)
      SegIter it;
      it.init(p.w, c);
      int cur_tile = 0, cur_k = 0, cur_k1 = 0;
      auto a_rows = [&](int& r0, int& r1, int& xk, int& brow) {
        if (cur_k >= cur_k1) it.next(p.w, cur_tile, cur_k, cur_k1);
        const int tile = cur_tile, kbi = cur_k++;
        const int mt = tile / p.n_tiles, nt = tile % p.n_tiles;
        if (EPI == EPI_SWIGLU) {
          r0 = mt * 64;
          r1 = p.up_row0 + mt * 64;
        } else {
          r0 = mt * BM;
          r1 = mt * BM + 64;
        }
        xk = kbi * BK;
        brow = nt * BN;
      };
      // prologue: weights do not depend on the previous kernel, so fetch them before waiting
      int pre_xk[C::STAGES], pre_brow[C::STAGES];
      for (int i = 0; i < npre; ++i) {
        int r0, r1;
        a_rows(r0, r1, pre_xk[i], pre_brow[i]);
        uint8_t* sa = smem + i * C::STAGE_BYTES;
        mbar_arrive_expect_tx(&full[i], C::STAGE_BYTES);
        last_fill[i] = 0;
        tma_load_2d(sa, &tmA, &full[i], pre_xk[i], r0, pol_w);
        tma_load_2d(sa + 8192, &tmA, &full[i], pre_xk[i], r1, pol_w);
      }
      pdl_wait();
      for (int i = 0; i < npre; ++i)
        tma_load_2d(smem + i * C::STAGE_BYTES + C::A_BYTES, &tmB, &full[i], pre_xk[i], pre_brow[i], pol_x);
      int stage = npre % C::STAGES;
      uint32_t phase = (npre == C::STAGES) ? 1u : 0u;
      for (long long i = npre; i < total; ++i) {
        if (!mbar_wait(&empty[stage], phase ^ 1u, p.err)) {
          *failed = 1;
          break;
        }
        int r0, r1, xk, brow;
        a_rows(r0, r1, xk, brow);
        uint8_t* sa = smem + stage * C::STAGE_BYTES;
        mbar_arrive_expect_tx(&full[stage], C::STAGE_BYTES);
        last_fill[stage] = (int)phase;
        tma_load_2d(sa, &tmA, &full[stage], xk, r0, pol_w);
        tma_load_2d(sa + 8192, &tmA, &full[stage], xk, r1, pol_w);
        tma_load_2d(sa + C::A_BYTES, &tmB, &full[stage], xk, brow, pol_x);
        if (++stage == C::STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && nu > 0) {
      // ------------------------------------------------------------------ MMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int si = 0;
      bool ok = true;
      SegIter it;
      it.init(p.w, c);
      int tile, k0, k1;
      for (; ok && it.next(p.w, tile, k0, k1); ++si) {
        const long long len = k1 - k0;
        const int acc = si & 1, use = si >> 1;
        if (!mbar_wait(&tempty[acc], (uint32_t)(use & 1) ^ 1u, p.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dt = tmem_base + (uint32_t)(acc * BN);
        for (long long j = 0; j < len; ++j) {
          if (!mbar_wait(&full[stage], phase, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * C::STAGE_BYTES);
          const uint64_t ad = smem_desc_sw128(sa);
          const uint64_t bd = smem_desc_sw128(sa + C::A_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            // advance the start address by kk * 32 bytes inside the 128-byte swizzle row
            tc_mma_bf16(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), idesc, (j > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(&empty[stage]);
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        tc_commit(&tfull[acc]);
      }
      if (!ok) *failed = 1;
      // drain: no MMA may still be running when TMEM is released
      tc_commit(mma_done);
      mbar_wait(mma_done, 0, p.err);
    }
  } else {
    // -------------------------------------------------------------------- epilogue
    const int q = warp & 3;
    const int ep_tid = threadIdx.x - 64;
    const int m = q * 32 + lane;
    pdl_wait();
    int si = 0;
    SegIter it;
    it.init(p.w, c);
    int tile, k0, k1;
    for (; it.next(p.w, tile, k0, k1); ++si) {
      const int acc = si & 1, use = si >> 1;
      const bool got = named_bar_and(1, 128, mbar_wait(&tfull[acc], (uint32_t)(use & 1), p.err));
      if (!got) {
        *failed = 1;
        break;
      }
      tc_fence_after();
      const int m_tile = tile / p.n_tiles, n_tile = tile % p.n_tiles;
      if constexpr (EPI == EPI_QKV) load_tok_tables<BN>(p.a, n_tile, tpos, tkvr, ep_tid);
      const bool scaled = (EPI == EPI_QKV || EPI == EPI_SWIGLU) && p.a.ssq_in != nullptr;
      if (scaled) load_norm_scales<BN>(p.a, n_tile, trs, ep_tid, 128);
      auto epilogue = [&](int ch) {
        if constexpr (EPI == EPI_RESNORM)
          epi_resnorm(p.a, staging, m_tile, n_tile * BN + ch * 32, ep_tid, 1);
        else
          epi_chunk<BN, EPI>(p.a, staging, m_tile, n_tile, ch, ep_tid, tpos, tkvr, scaled ? trs : nullptr);
      };
      const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
      // 32-token chunks that hold at least one valid token (the rest are padding)
      const int nch = min(BN / 32, (p.a.T - n_tile * BN + 31) / 32);
      if (k0 == 0 && k1 == kb) {
        for (int ch = 0; ch < nch; ++ch) {
          uint32_t r[32];
          tmem_ld_32x32b_x32(tb + ch * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; ++j) staging[j * BM + m] = __uint_as_float(r[j]);
          named_bar_sync(1, 128);
          epilogue(ch);
          named_bar_sync(1, 128);
        }
        tc_fence_before();
        if (lane == 0) mbar_arrive(&tempty[acc]);
      } else {
        const long long slot = (long long)c * 2 + (si == 0 ? 0 : 1);
        ws_store_partial(p.ws + slot * WS_SLOT_FLOATS, tb, nch, m);
        tc_fence_before();
        if (lane == 0) mbar_arrive(&tempty[acc]);
        __threadfence();
        named_bar_sync(1, 128);
        const long long tu0 = (long long)tile * kb;
        const int c_first = sk_owner(p.w, tu0);
        const int c_last = sk_owner(p.w, tu0 + kb - 1);
        const int parts = c_last - c_first + 1;
        if (ep_tid == 0) {
          const int old = atomicAdd(&p.counters[tile], 1);
          const int last = (old == parts - 1);
          if (last) {
            p.counters[tile] = 0;
            __threadfence();
          }
          *flag = last;
        }
        // workspace slot of every part, in k order
        for (int pi = ep_tid; pi < parts; pi += 128) {
          const int cc = c_first + pi;
          part_slot[pi] = cc * 2 + (sk_start(p.w, cc) >= tu0 ? 0 : 1);
        }
        named_bar_sync(1, 128);
        if (*flag) {
          for (int ch = 0; ch < nch; ++ch) {
            ws_reduce_chunk(p.ws, part_slot, parts, ch, m, staging);
            named_bar_sync(1, 128);
            epilogue(ch);
            named_bar_sync(1, 128);
          }
        }
      }
    }
  }

  __syncthreads();
  if (*failed && threadIdx.x == 0) {
    // make sure no TMA write is still headed for this CTA's shared memory
    for (int s = 0; s < C::STAGES; ++s)
      if (last_fill[s] >= 0) mbar_wait(&full[s], (uint32_t)last_fill[s], p.err);
  }
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

bool make_map(CUtensorMap* m, const void* base, int inner, int rows, int box_rows, char* eb, size_t el) {
  auto fn = encode_fn();
  if (!fn) {
    snprintf(eb, el, "cuTensorMapEncodeTiled unavailable");
    return false;
  }
  cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    snprintf(eb, el, "cuTensorMapEncodeTiled failed (%d): inner=%d rows=%d box_rows=%d", (int)r, inner, rows,
             box_rows);
    return false;
  }
  return true;
}

template <int BN, int EPI>
cudaError_t launch_t(const CUtensorMap& ma, const CUtensorMap& mb, const KParams& kp, cudaStream_t st, bool pdl) {
  using C = Cfg<BN>;
  static std::atomic<unsigned long long> attr_done{0};
  const cudaError_t e = smem_attr_once(attr_done, gemm_kernel<BN, EPI>, C::SMEM);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kp.G);
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_kernel<BN, EPI>, ma, mb, kp);
}

template <int BN>
cudaError_t launch_bn(EpiKind e, const CUtensorMap& ma, const CUtensorMap& mb, const KParams& kp, cudaStream_t st,
                      bool pdl) {
  switch (e) {
    case EPI_F32: return launch_t<BN, EPI_F32>(ma, mb, kp, st, pdl);
    case EPI_BF16: return launch_t<BN, EPI_BF16>(ma, mb, kp, st, pdl);
    case EPI_RESID: return launch_t<BN, EPI_RESID>(ma, mb, kp, st, pdl);
    case EPI_SWIGLU: return launch_t<BN, EPI_SWIGLU>(ma, mb, kp, st, pdl);
    case EPI_QKV: return launch_t<BN, EPI_QKV>(ma, mb, kp, st, pdl);
    case EPI_LSE: return launch_t<BN, EPI_LSE>(ma, mb, kp, st, pdl);
    case EPI_RESNORM: return launch_t<BN, EPI_RESNORM>(ma, mb, kp, st, pdl);
  }
  return cudaErrorInvalidValue;
}

__global__ void lse_combine_kernel(const float2* part, int ld, int m_tiles, int T, float* lse) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  float mx = -INFINITY;
  for (int m = 0; m < m_tiles; ++m) mx = fmaxf(mx, part[(size_t)m * ld + t].x);
  float s = 0.f;
  if (mx != -INFINITY)
    for (int m = 0; m < m_tiles; ++m) {
      const float2 v = part[(size_t)m * ld + t];
      if (v.x != -INFINITY) s += v.y * expf(v.x - mx);
    }
  lse[t] = mx + logf(s);
}

}  // namespace

cudaError_t lse_combine_launch(const float2* part, int ld, int m_tiles, int T, float* lse, cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  lse_combine_kernel<<<(T + 127) / 128, 128, 0, st>>>(part, ld, m_tiles, T, lse);
  return cudaGetLastError();
}

bool gemm_make_map(CUtensorMap* m, const void* base, int inner, int rows, int box_rows, char* eb, size_t el) {
  return make_map(m, base, inner, rows, box_rows, eb, el);
}

size_t gemm_ws_bytes(int grid) { return (size_t)2 * grid * WS_SLOT_FLOATS * sizeof(float); }
int gemm_max_tiles() { return MAX_TILES; }

int gemm_grid_size(int device) {
  int sms = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
  return sms > 0 ? sms : 1;
}

cudaError_t gemm_launch(const GemmArgs& a, const GemmScratch& s, int grid, cudaStream_t stream, bool pdl,
                        char* eb, size_t el) {
  if (a.K <= 0 || a.K % BK != 0 || a.K / BK > 256 || a.M <= 0 || a.T <= 0) {
    snprintf(eb, el, "gemm: bad shape M=%d K=%d T=%d", a.M, a.K, a.T);
    return cudaErrorInvalidValue;
  }
  const int BN = a.T <= 128 ? 128 : 256;
  KParams kp;
  kp.a = a;
  kp.n_tiles = (a.T + BN - 1) / BN;
  if (a.X_rows < kp.n_tiles * BN) {
    snprintf(eb, el, "gemm: X has %d rows, needs %d", a.X_rows, kp.n_tiles * BN);
    return cudaErrorInvalidValue;
  }
  if (a.epi == EPI_SWIGLU) {
    if (a.M % 128 != 0) {
      snprintf(eb, el, "gemm: SwiGLU needs 2*d_ffn %% 128 == 0 (M=%d)", a.M);
      return cudaErrorInvalidValue;
    }
    kp.m_tiles = a.M / 128;
    kp.up_row0 = a.M / 2;
  } else {
    kp.m_tiles = (a.M + BM - 1) / BM;
    kp.up_row0 = 0;
  }
  kp.kb = a.K / BK;
  const long long tiles = (long long)kp.m_tiles * kp.n_tiles;
  if (tiles > s.max_tiles) {
    snprintf(eb, el, "gemm: %lld tiles exceed the counter table (%d)", tiles, s.max_tiles);
    return cudaErrorInvalidValue;
  }
  kp.G = gemm_work_ctas(tiles, kp.kb, grid);
  kp.w = work_split((int)tiles, kp.kb, kp.G);
  if (s.ws_bytes < gemm_ws_bytes(kp.G)) {
    snprintf(eb, el, "gemm: workspace too small");
    return cudaErrorInvalidValue;
  }
  kp.ws = s.ws;
  kp.counters = s.counters;
  kp.err = s.err;
  CUtensorMap ma, mb;
  // an operand the tensor-map encoder refuses (typically a base address that is not 16-byte aligned)
  if (!make_map(&ma, a.W, a.K, a.M, 64, eb, el)) return kGemmMapError;
  if (!make_map(&mb, a.X, a.K, a.X_rows, BN, eb, el)) return kGemmMapError;
  return BN == 128 ? launch_bn<128>(a.epi, ma, mb, kp, stream, pdl) : launch_bn<256>(a.epi, ma, mb, kp, stream, pdl);
}

}  // namespace atspeed
