// Persistent forward kernel for sm_103a.
//
// One cooperative launch, one CTA per SM, runs a whole decoder forward as a fixed phase program:
//   EMBED | for each layer: QKV, ATTN, O, GATE_UP, DOWN | final NORM | LM
// with a grid barrier after every phase.  The RMSNorms before the QKV and gate/up projections are
// folded into the GEMMs around them (x = h / rms(h) * g, and W x = (W (g h)) / rms(h)): the O /
// down epilogue adds its product to h and leaves bf16(g h) and per-128-row-tile sums of squares of
// h; the QKV / gate-up epilogue multiplies each token's product by 1 / rms(h) from those sums.  (The
// program keeps the index slots of the two folded norm phases per layer, 7 per layer, for the
// trace.)  The GEMM phases reuse the stream-K decomposition of the standalone GEMM (whole tiles
// and stream-K units per CTA, split tiles summed in k order), but their operands flow through two
// rings that live for the whole launch:
//   * the weight ring (A, 16 KB per stage) is filled by a producer warp that walks every GEMM
//     phase of the forward in order and never waits for a grid barrier -- weights do not depend
//     on activations -- so HBM keeps streaming the next phase's weights during barriers, split-sum
//     tails and attention;
//   * the activation ring (B) is filled by a second producer warp that waits for the barrier that
//     publishes the phase's input.
// Warp roles (384 threads): 0 weight TMA, 1 activation TMA, 2 TMEM + MMA issue, 3 idle; 4..11 two
// compute warpgroups (GEMM epilogues -- a warp reads the TMEM lane quadrant of its id mod 4 --,
// the embedding and final-norm rows, tree attention).
// Every wait is bounded; a timeout (or an error raised by another CTA) makes every role leave its
// loop, in-flight copies are waited for, TMEM is released.
#include <cudaTypedefs.h>
#include <stdio.h>

#include "attn_core.cuh"
#include "common.cuh"
#include "fwd.cuh"
#include "gemm_core.cuh"
#include "norm_core.cuh"

namespace atspeed {

namespace {

constexpr int FWD_THREADS = 384;   // warps 0-3: producers, MMA (3 idle); warps 4-11: two compute warpgroups
constexpr int COMPUTE_WARP0 = 4;
constexpr int CT = 256;            // compute threads (named barrier 1); warpgroup w uses barrier 2 + w
// Registers per thread after the prologue: the launch gives every thread 168 (12 warps, 3 per
// SM sub-partition); warpgroup 0 (producers, MMA issuer, prefetch: little live state) gives back
// down to kRegsRoles and the two compute warpgroups take them up to kRegsCompute, so that the
// epilogues, norms and attention do not spill.  Budget (checked below): 128 * kRegsRoles + 256 *
// kRegsCompute <= 384 * 168, and per sub-partition one role warp and two compute warps.
constexpr int kRegsLaunch = 168, kRegsRoles = 80, kRegsCompute = 208;
static_assert(128 * kRegsRoles + 256 * kRegsCompute <= FWD_THREADS * kRegsLaunch, "register split over the launch's total");
static_assert(32 * (kRegsRoles + 2 * kRegsCompute) <= 16384, "register split over a sub-partition's file");
static_assert(kRegsRoles % 8 == 0 && kRegsCompute % 8 == 0 && kRegsRoles >= 24 && kRegsCompute <= 256, "setmaxnreg range");
// Split parts in flight in a residual-update sum: one.  With two or three the kernel spills
// registers (24 / 136 and 48 / 164 bytes; the attention phase holds the peak), which costs more
// than the round trips they save.
constexpr int RED_PB = 1;
constexpr int ITEM_ROWS_FWD = 1024;   // item-code rows of the LM head (4 levels x 256 codes)

template <int BN>
struct FCfg {
  static constexpr int SA = BN == 128 ? 8 : 5;   // weight stages
  static constexpr int SB = BN == 128 ? 3 : 3;   // activation stages
  static constexpr int A_BYTES = GEMM_BM * 128;
  static constexpr int B_BYTES = BN * 128;
  static constexpr int STAGING = 2 * 32 * GEMM_BM * 4;   // one [32][128] fp32 chunk per warpgroup
  static constexpr int MISC = 8192;
  static constexpr int TMEM_COLS = 2 * BN;
};

template <int HD, int BN>
struct FLayout {
  using C = FCfg<BN>;
  static constexpr int A_OFF = 0;
  static constexpr int B_OFF = C::SA * C::A_BYTES;
  static constexpr int STG_OFF = B_OFF + C::SB * C::B_BYTES;
  // the attention work areas (one per warpgroup) overlap the activation ring and the staging buffers
  // (both idle then)
  static constexpr int ATT_OFF = B_OFF;
  static constexpr int ATT_BODY = ((AttCfg<HD>::SMEM_BODY + 1023) / 1024) * 1024;
  static constexpr int ATT_NEED = 2 * ATT_BODY;
  static constexpr int AFTER_STG = STG_OFF + C::STAGING;
  static constexpr int EXTRA = (ATT_OFF + ATT_NEED > AFTER_STG) ? ((ATT_OFF + ATT_NEED - AFTER_STG + 1023) / 1024) * 1024 : 0;
  static constexpr int MISC_OFF = AFTER_STG + EXTRA;
  static constexpr int TOTAL = 1024 + MISC_OFF + C::MISC;
  static_assert(C::SB * C::B_BYTES >= 8192 * 4, "a final-norm row (d <= 8192 floats) must fit in the activation ring");
};

struct GP {
  int epi;
  int k;         // 0 QKV, 1 O, 2 gate/up, 3 down (of layer `layer`), 4 LM head
  bool dh_out;   // O / down projection: the product is added to h (EPI_RESNORM)
  int M, K, m_tiles, n_tiles, kb, up_row0, rows;  // rows: valid tokens of the phase
  WorkSplit w;   // whole tiles per CTA + stream-K over the remaining tiles
  int mapA, mapB, layer;
};

__device__ __forceinline__ GP gemm_phase(const FwdParams& p, int gi, int BN) {
  GP g;
  const int L = p.L;
  const int act0 = 6 * L + 1 + (BN == 256 ? 3 : 0);   // activation maps: x, att, act
  g.layer = gi / 4;
  g.up_row0 = 0;
  g.rows = p.T;
  g.dh_out = false;
  if (gi == 4 * L) {
    g.k = 4;
    g.epi = EPI_F32;
    g.M = ITEM_ROWS_FWD;
    g.K = p.d;
    g.mapA = 6 * L;
    g.mapB = act0;
    g.rows = p.n_out;
  } else {
    const int k = gi % 4;
    g.k = k;
    g.mapA = g.layer * 4 + k;
    if (k == 0) {
      g.epi = EPI_QKV;
      g.M = 3 * p.d;
      g.K = p.d;
      g.mapB = act0;
    } else if (k == 1) {
      g.epi = EPI_RESNORM;
      g.dh_out = true;
      g.M = p.d;
      g.K = p.d;
      g.mapB = act0 + 1;
    } else if (k == 2) {
      g.epi = EPI_SWIGLU;
      g.M = 2 * p.ffn;
      g.K = p.d;
      g.up_row0 = p.ffn;
      g.mapB = act0;
    } else {
      g.epi = EPI_RESNORM;
      g.dh_out = true;
      g.M = p.d;
      g.K = p.ffn;
      g.mapB = act0 + 2;
    }
  }
  g.m_tiles = (g.epi == EPI_SWIGLU) ? g.M / GEMM_BM : (g.M + GEMM_BM - 1) / GEMM_BM;
  g.n_tiles = (g.rows + BN - 1) / BN;
  g.kb = g.K / GEMM_BK;
  g.w = work_split(g.m_tiles * g.n_tiles, g.kb, gemm_work_ctas((long long)g.m_tiles * g.n_tiles, g.kb, p.G));
  return g;
}

// Weight-tile coordinates of (tile, k-block): k offset and the rows of the two 64-row boxes
// (SwiGLU tiles pair 64 gate rows with the matching 64 up rows).
__device__ __forceinline__ void a_coords(const GP& g, int tile, int kbi, int& x, int& y0, int& y1) {
  const int mt = tile / g.n_tiles;
  x = kbi * GEMM_BK;
  if (g.epi == EPI_SWIGLU) {
    y0 = mt * 64;
    y1 = g.up_row0 + mt * 64;
  } else {
    y0 = mt * GEMM_BM;
    y1 = mt * GEMM_BM + 64;
  }
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* a) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
  return v;
}
// Publishing a CTA's split parts: every thread stores, the CTA synchronises, then one thread's
// release (or acquire-release) add at gpu scope makes all of those stores visible to whoever
// acquires the counter (and synchronises its own CTA after that).
__device__ __forceinline__ void red_release_add(int* a, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(a), "r"(v) : "memory");
}
__device__ __forceinline__ int atom_acq_rel_add(int* a, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.global;" ::: "memory"); }

__device__ __forceinline__ bool err_set(const unsigned* e) { return *(volatile const unsigned*)e != 0u; }

// Waits until barrier `k` (0-based) is complete: count >= (k + 1) * G.  False on timeout or when an
// error was raised anywhere.
__device__ bool grid_wait(const FwdParams& p, int k) {
  const unsigned target = (unsigned)(k + 1) * (unsigned)p.G;
  if (ld_acquire_u32(p.bar) >= target) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned it = 1;; ++it) {
    if (it > 32u) __nanosleep(64);   // back-to-back polls first: the barrier usually completes soon
    if (ld_acquire_u32(p.bar) >= target) return true;
    if ((it & 255u) == 0u) {
      if (err_set(p.err)) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        set_error(p.err, ATSPEED_DEV_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

__device__ __forceinline__ void st_release_cta(int* a, int v) {
  asm volatile("st.release.cta.shared.u32 [%0], %1;" ::"r"(smem_u32(a)), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_cta(const int* a) {
  int v;
  asm volatile("ld.acquire.cta.shared.u32 %0, [%1];" : "=r"(v) : "r"(smem_u32(a)) : "memory");
  return v;
}
// Waits until the shared counter reaches `target` (bounded; false on timeout or a raised error).
__device__ bool cta_count_wait(const int* cnt, int target, unsigned* err) {
  if (ld_acquire_cta(cnt) >= target) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned it = 1;; ++it) {
    __nanosleep(32);
    if (ld_acquire_cta(cnt) >= target) return true;
    if ((it & 1023u) == 0u) {
      if (err_set(err)) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        set_error(err, ATSPEED_DEV_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

// Waits until the global counter reaches `target` (bounded; false on timeout or a raised error).
__device__ bool counter_wait(const int* cnt, int target, unsigned* err) {
  if ((int)ld_acquire_u32(reinterpret_cast<const unsigned*>(cnt)) >= target) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned it = 1;; ++it) {
    if (it > 32u) __nanosleep(64);
    if ((int)ld_acquire_u32(reinterpret_cast<const unsigned*>(cnt)) >= target) return true;
    if ((it & 255u) == 0u) {
      if (err_set(err)) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        set_error(err, ATSPEED_DEV_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

// mbarrier wait that also gives up as soon as an error is raised anywhere
__device__ bool mwait(uint64_t* bar, uint32_t parity, unsigned* err) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 1023u) == 0u) {
      if (err_set(err)) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        set_error(err, ATSPEED_DEV_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

// trs: the n-tile's norm scales (QKV / gate-up); bar: the warpgroup's named barrier (EPI_RESNORM)
template <int BN>
__device__ __noinline__ void epi_dispatch(int epi, const GemmArgs* a, float* st, int mt, int nt, int ch, int t,
                                          const int* tpos, const int* tkvr, const float* trs, int bar) {
  switch (epi) {
    case EPI_F32: epi_chunk<BN, EPI_F32>(*a, st, mt, nt, ch, t, tpos, tkvr); break;
    case EPI_RESNORM: epi_resnorm(*a, st, mt, nt * BN + ch * 32, t, bar); break;
    case EPI_SWIGLU: epi_chunk<BN, EPI_SWIGLU>(*a, st, mt, nt, ch, t, tpos, tkvr, trs); break;
    default: epi_chunk<BN, EPI_QKV>(*a, st, mt, nt, ch, t, tpos, tkvr, trs); break;
  }
}

__device__ GemmArgs epi_args(const FwdParams& p, const GP& g) {
  GemmArgs a = {};
  a.epi = (EpiKind)g.epi;
  a.M = g.M;
  a.K = g.K;
  a.T = g.rows;
  a.d_model = p.d;
  a.head_dim = p.hd;
  a.pos = p.pos;
  a.kv_row = p.kv_row;
  a.rope_cos = p.rope_cos;
  a.rope_sin = p.rope_sin;
  a.q_out = p.q;
  a.k_cache = p.kc + p.layer_elems * g.layer;
  a.v_cache = p.vc + p.layer_elems * g.layer;
  a.ssq_ld = p.ssq_ld;
  a.nrm_d = p.d;
  a.eps = p.eps;
  if (g.k == 0 || g.k == 2) a.ssq_in = p.ssq;   // input rows bf16(g * h): scaled by 1 / rms(h)
  if (g.dh_out) {
    a.out_f32 = p.h;
    a.ldo = p.d;
    // the next norm (of the gate/up or of the next layer's QKV) is folded into this epilogue; after
    // the last layer the final norm normalises the selected rows from h
    const __nv_bfloat16* gn = g.k == 1 ? p.mlp_norm[g.layer] : (g.layer + 1 < p.L ? p.attn_norm[g.layer + 1] : nullptr);
    if (gn) {
      a.gain = gn;
      a.xg_out = p.x;
      a.ssq_out = p.ssq;
    }
  } else if (g.epi == EPI_F32) {
    a.out_f32 = p.logits;
    a.ldo = ITEM_ROWS_FWD;
  } else if (g.epi == EPI_SWIGLU) {
    a.out_bf16 = p.act;
    a.ldo = p.ffn;
  }
  return a;
}

// Norm phases (256 compute threads).  final == false: layer 0's input rows -- the embedding rows
// enter h, and x gets bf16(g * h) with the partial sums of squares (the norm's per-token scale is
// applied by the QKV epilogue, as after every O / down projection).  final == true: RMSNorm of the
// selected rows out_rows[r] of h into x row r, the LM head's input; the per-thread chunks and the
// reduction are those of the 256-thread kernels, so the sums are the same bit for bit.  Between the
// passes the row is kept in shared memory (`rowbuf`, d floats: the activation ring, idle then).
template <int BN>
__device__ __forceinline__ void norm_phase(const FwdParams& p, bool final, const __nv_bfloat16* g, float* red,
                                           float4* rowbuf, int ctid, int ph) {
  const int d = p.d, nc = d / 4;
  if (!final) {
    for (int r = blockIdx.x; r < p.T; r += p.G)
      embed_row(p.embed + (size_t)p.tok[r] * d, g, p.h + (size_t)r * d, p.x + (size_t)r * d, p.ssq, p.ssq_ld, r, d,
                ctid, CT);
    return;
  }
  const int w = ctid >> 5, lane = ctid & 31;
  for (int r = blockIdx.x; r < p.n_out; r += p.G) {
    const float4* h4 = reinterpret_cast<const float4*>(p.h + (size_t)p.out_rows[r] * d);
    float ss = 0.f;
    // the gains do not depend on the row: their loads go out with the row's
    constexpr int NG_MAX = 8192 / 4 / CT;   // chunks per thread, d <= 8192
    uint2 graw[NG_MAX];
#pragma unroll
    for (int k = 0; k < NG_MAX; ++k) {
      const int c = ctid + CT * k;
      graw[k] = c < nc ? *reinterpret_cast<const uint2*>(g + 4 * c) : make_uint2(0, 0);
    }
#pragma unroll
    for (int k = 0; k < NG_MAX; ++k) {
      const int c = ctid + CT * k;
      if (c < nc) {
        const float4 v = __ldcg(h4 + c);
        rowbuf[c] = v;
        ss += v.x * v.x;
        ss += v.y * v.y;
        ss += v.z * v.z;
        ss += v.w * v.w;
      }
    }
    ss = warp_sum(ss);
    if (lane == 0) red[w] = ss;
    named_bar_sync(1, CT);
    if (p.trace && ctid == 0 && r == (int)blockIdx.x) p.trace[((size_t)5 * (7 * p.L + 2) + ph) * p.G + blockIdx.x] = globaltimer_ns();
    const float rs = 1.0f / sqrtf(rms_total(red) / (float)d + p.eps);
    __nv_bfloat16* xr = p.x + (size_t)r * d;
#pragma unroll
    for (int k = 0; k < NG_MAX; ++k) {
      const int c = ctid + CT * k;
      if (c >= nc) break;
      const float4 v = rowbuf[c];
      const __nv_bfloat162* gb = reinterpret_cast<const __nv_bfloat162*>(&graw[k]);
      const float2 g0 = __bfloat1622float2(gb[0]), g1 = __bfloat1622float2(gb[1]);
      __nv_bfloat162 o[2];
      o[0] = __floats2bfloat162_rn(v.x * rs * g0.x, v.y * rs * g0.y);
      o[1] = __floats2bfloat162_rn(v.z * rs * g1.x, v.w * rs * g1.y);
      *reinterpret_cast<uint2*>(xr + 4 * c) = *reinterpret_cast<uint2*>(o);
    }
    named_bar_sync(1, CT);
  }
}

// Tree attention of layer l, one warpgroup (128 threads, `wt`): its work items (query tile, head,
// prefix split) are item c + (2k + wg) G; each is followed by the warpgroup's share of the merge of
// the splits of (tile, head) once all of them are published.
template <int HD>
__device__ __forceinline__ bool attn_phase(const FwdParams& p, int l, uint8_t* att_smem, uint64_t* att_bars,
                                           int (&use_att)[2], int* flag, int wt, int wg, int wbar) {
  const int c = blockIdx.x, G = p.G, L = p.L;
  AttnArgs a = p.att_args;
  a.k_cache = p.kc + p.layer_elems * l;
  a.v_cache = p.vc + p.layer_elems * l;
  const CUtensorMap* mk = p.maps + 4 * L + 2 * l;
  const CUtensorMap* mv = mk + 1;
  const int H = p.H, S = a.max_splits;
  const int NP = 7 * L + 2, ph = 7 * l + 2;
  int nit = 0;
  for (int item = c + wg * G; item < p.att_items; item += 2 * G, ++nit) {
    const int tile = item / (H * S), rem = item % (H * S);
    const int h = rem / S, split = rem % S;
    const bool tr_on = p.trace && wg == 0 && nit == 0;
    unsigned long long* tr = tr_on ? p.trace + ((size_t)8 * NP + ph) * G + c : nullptr;
    if (!attn_item<HD>(a, mk, mv, tile, h, split, att_smem, att_bars, use_att, wt, wbar, tr, (size_t)NP * G))
      return false;
    if (tr_on && wt == 0) p.trace[((size_t)4 * NP + ph) * G + c] = globaltimer_ns();
    if (a.direct) continue;
    const int S_u = a.user_splits[a.qt_user[tile]];
    if (split >= S_u) continue;
    // every split publishes its partials and waits for the others of (tile, h) -- all items run in
    // one round (2 G work slots), or the awaited ones in a later round, never an earlier one -- then
    // split s merges query groups s, s + S_u, ...  The counter only grows during a launch: layer l
    // completes at S_u * (l + 1).
    __threadfence();
    named_bar_sync(wbar, 128);
    if (wt == 0) {
      int* cnt = &p.att_counters[tile * H + h];
      atomicAdd(cnt, 1);
      *flag = counter_wait(cnt, S_u * (l + 1), p.err) ? 1 : 0;
    }
    named_bar_sync(wbar, 128);
    if (!*flag) return false;
    const int nq = a.qt_n[tile];
    for (int qg = split; qg * ATT_CQ < nq; qg += S_u) attn_combine_group<HD>(a, tile, h, qg, wt);
    named_bar_sync(wbar, 128);
    if (tr_on && wt == 0) p.trace[((size_t)5 * NP + ph) * G + c] = globaltimer_ns();
  }
  return true;
}

// GEMM phase gi (program phase ph), compute-warp side (256 threads, ctid).  The 32-token chunks of
// a tile alternate between the two warpgroups (chunk ch by warpgroup ch & 1, each with its own
// staging buffer and named barrier); warp 4 + q and warp 8 + q both read TMEM lane quadrant q.
// For each of this CTA's segments, wait for its accumulator, then:
//  * a whole tile runs the fused epilogue; for a split tile, if every other part is already
//    published (and this is the CTA's last segment) this CTA is the last one and sums the parts
//    with its own part read straight from TMEM; otherwise it publishes its part and the last CTA
//    to arrive does the sum;
//  * shared sums (phases with whole tiles per CTA, whose split tiles come first and finish early;
//    the O / down projections, whose residual update ends the phase; the LM head, whose tiles have
//    many short parts): every part publishes, then each part sums a share of its tile's chunks
//    (chunk ch by part ch mod parts).
// Parts are always summed in k order starting from zero, whichever CTA sums them.  The QKV and
// gate/up epilogues first multiply by each token's norm scale (trs, loaded per token tile).
template <int BN>
__device__ __forceinline__ bool gemm_epi_phase(const FwdParams& p, int gi, int ph, float* staging_base, uint64_t* tfull,
                                               uint64_t* tempty, int* flag, int* part_slot, int* tpos, int* tkvr,
                                               float* trs, GemmArgs* s_ea, uint32_t tmem_base, int ctid, int& si) {
  const int c = blockIdx.x, G = p.G, NP = 7 * p.L + 2;
  const int wg = ctid >> 7, wt = ctid & 127, wbar = 2 + wg;
  // a warp reads the TMEM lane quadrant of its warp id mod 4; each warpgroup (4 consecutive warps)
  // covers all four, so row m of the tile is the quadrant's row of this lane
  const int lane = ctid & 31, q = (threadIdx.x >> 5) & 3, m = q * 32 + lane;
  float* staging = staging_base + wg * (32 * GEMM_BM);
  const GP g = gemm_phase(p, gi, BN);
  // the epilogue's arguments live in shared memory (read by the out-of-line epilogue functions)
  if (ctid == 0) *s_ea = epi_args(p, g);
  named_bar_sync(1, CT);
  const GemmArgs& ea = *s_ea;
  const int kb = g.kb;
  const bool scaled = g.k == 0 || g.k == 2;
  const float* trs_e = scaled ? trs : nullptr;
  // per-token tables of the token tile nt (QKV: rotary positions and cache rows; QKV and gate/up:
  // norm scales), loaded when the tile changes; callers synchronise before their first use
  int tab_nt = -1;
  auto tables = [&](int nt) {
    if ((g.epi != EPI_QKV && !scaled) || nt == tab_nt) return;
    named_bar_sync(1, CT);   // both warpgroups are done with the previous tables
    tab_nt = nt;
    if (g.epi == EPI_QKV) load_tok_tables<BN>(ea, nt, tpos, tkvr, ctid, CT);
    if (scaled) load_norm_scales<BN>(ea, nt, trs, ctid, CT);
  };
  SegIter it;
  it.init(g.w, c);
  int tile, k0, k1;
  auto fill_part_slots = [&](long long tu0, int c_first, int parts) {
    for (int pi = ctid; pi < parts; pi += CT) {
      const int cc = c_first + pi;
      part_slot[pi] = cc * 2 + (sk_start(g.w, cc) >= tu0 ? 0 : 1);
    }
  };
  const bool shared_sums = g.w.q > 0 || g.dh_out || (gi == 4 * p.L && g.w.Gsk > 0 && g.w.Usk / g.w.Gsk + 1 < kb);
  if (shared_sums && it.u < it.u1) {
    int sk_tile[2], nsk = 0;
    while (it.u < it.u1 && nsk < 2) {
      it.next(g.w, tile, k0, k1);
      const int acc = si & 1, use = si >> 1;
      ++si;
      const bool got = named_bar_and(1, CT, mwait(&tfull[acc], (uint32_t)(use & 1), p.err));
      if (!got) return false;
      tc_fence_after();
      const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
      const int nch = min(BN / 32, (g.rows - (tile % g.n_tiles) * BN + 31) / 32);
      ws_store_partial(p.ws + ((long long)c * 2 + nsk) * GEMM_WS_SLOT_FLOATS, tb, nch, m, wg, 2);
      tc_fence_before();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      sk_tile[nsk++] = tile;
    }
    named_bar_sync(1, CT);
    int* skc = p.sk_counters + (size_t)gi * G;
    if (ctid == 0)
      for (int j = 0; j < nsk; ++j) red_release_add(&skc[sk_tile[j]], 1);
    if (p.trace && ctid == 0) p.trace[((size_t)5 * NP + ph) * G + c] = globaltimer_ns();
    for (int j = 0; j < nsk; ++j) {
      const int t = sk_tile[j];
      const long long tu0 = (long long)t * kb;
      const int c_first = sk_owner(g.w, tu0);
      const int parts = sk_owner(g.w, tu0 + kb - 1) - c_first + 1;
      const int m_tile = t / g.n_tiles, n_tile = t % g.n_tiles;
      fill_part_slots(tu0, c_first, parts);
      tables(n_tile);
      if (ctid == 0) *flag = counter_wait(&skc[t], parts, p.err) ? 1 : 0;
      named_bar_sync(1, CT);
      if (!*flag) return false;
      const bool tr_on = p.trace && ctid == 0 && j == 0;
      if (tr_on) p.trace[((size_t)6 * NP + ph) * G + c] = globaltimer_ns();
      const int nch = min(BN / 32, (g.rows - n_tile * BN + 31) / 32);
      if (g.dh_out) {
        // residual updates: both warpgroups on each chunk of this part, 16 tokens each
        for (int ch = c - c_first; ch < nch; ch += parts) {
          if (ch * 32 + 16 * wg >= g.rows - n_tile * BN) continue;   // (warpgroup-uniform)
          ws_reduce_resnorm_half<RED_PB>(ea, p.ws, part_slot, parts, ch, wg, m_tile, n_tile * BN + ch * 32, wt, staging,
                                         wbar);
          named_bar_sync(wbar, 128);
          if (tr_on) p.trace[((size_t)9 * NP + ph) * G + c] = globaltimer_ns();
        }
        named_bar_sync(1, CT);   // flag, part_slot and the token tables are reused
        continue;
      }
      int k = 0;
      for (int ch = c - c_first; ch < nch; ch += parts, ++k) {
        if ((k & 1) != wg) continue;
        ws_reduce_chunk<1>(p.ws, part_slot, parts, ch, m, staging);
        named_bar_sync(wbar, 128);
        if (tr_on && k == 0) p.trace[((size_t)8 * NP + ph) * G + c] = globaltimer_ns();
        epi_dispatch<BN>(g.epi, s_ea, staging, m_tile, n_tile, ch, wt, tpos, tkvr, trs_e, wbar);
        named_bar_sync(wbar, 128);
        if (tr_on && k == 0) p.trace[((size_t)9 * NP + ph) * G + c] = globaltimer_ns();
      }
      named_bar_sync(1, CT);   // flag, part_slot and the token tables are reused
    }
  }
  for (int seg = 0; it.next(g.w, tile, k0, k1); ++si, ++seg) {
    const int acc = si & 1, use = si >> 1;
    const int m_tile = tile / g.n_tiles, n_tile = tile % g.n_tiles;
    const bool whole = (k0 == 0 && k1 == kb);
    tables(n_tile);
    long long tu0 = 0;
    int c_first = 0, parts = 1;
    if (!whole) {
      tu0 = (long long)tile * kb;
      c_first = sk_owner(g.w, tu0);
      parts = sk_owner(g.w, tu0 + kb - 1) - c_first + 1;
      fill_part_slots(tu0, c_first, parts);
    }
    // (the vote is also the barrier after which token tables and part slots are in place)
    const bool got = named_bar_and(1, CT, mwait(&tfull[acc], (uint32_t)(use & 1), p.err));
    if (!got) return false;
    tc_fence_after();
    if (p.trace && ctid == 0) p.trace[((size_t)4 * NP + ph) * G + c] = globaltimer_ns();
    const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
    const int nch = min(BN / 32, (g.rows - n_tile * BN + 31) / 32);
    if (whole) {
      for (int ch = wg; ch < nch; ch += 2) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tb + ch * 32, r);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 32; ++j) staging[j * GEMM_BM + m] = __uint_as_float(r[j]);
        named_bar_sync(wbar, 128);
        epi_dispatch<BN>(g.epi, s_ea, staging, m_tile, n_tile, ch, wt, tpos, tkvr, trs_e, wbar);
        named_bar_sync(wbar, 128);
      }
      tc_fence_before();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      continue;
    }
    // split tile: are the other parts all published already?  (Only for the CTA's last segment of
    // the phase: holding this accumulator through the sum must not stall later MMAs of the phase.)
    if (ctid == 0)
      *flag = !it.more() &&
              (int)ld_acquire_u32(reinterpret_cast<const unsigned*>(&p.counters[tile])) == parts - 1;
    named_bar_sync(1, CT);
    if (*flag) {
      // last part: nobody else touches this tile's counter in this phase
      if (ctid == 0) p.counters[tile] = 0;
      if (p.trace && ctid == 0) p.trace[((size_t)6 * NP + ph) * G + c] = globaltimer_ns();
      const int own = c - c_first;
      for (int ch = wg; ch < nch; ch += 2) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tb + ch * 32, r);
        tmem_ld_wait();
        ws_reduce_chunk_own(p.ws, part_slot, parts, own, r, ch, m, staging);
        named_bar_sync(wbar, 128);
        epi_dispatch<BN>(g.epi, s_ea, staging, m_tile, n_tile, ch, wt, tpos, tkvr, trs_e, wbar);
        named_bar_sync(wbar, 128);
      }
      tc_fence_before();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      named_bar_sync(1, CT);   // flag and part_slot are reused by the next segment
      continue;
    }
    const long long slot = (long long)c * 2 + (seg == 0 ? 0 : 1);
    ws_store_partial(p.ws + slot * GEMM_WS_SLOT_FLOATS, tb, nch, m, wg, 2);
    tc_fence_before();
    if (lane == 0) mbar_arrive(&tempty[acc]);
    named_bar_sync(1, CT);
    if (p.trace && ctid == 0) p.trace[((size_t)5 * NP + ph) * G + c] = globaltimer_ns();
    if (ctid == 0) {
      const int old = atom_acq_rel_add(&p.counters[tile], 1);
      const int last = (old == parts - 1);
      if (last) {
        p.counters[tile] = 0;
        __threadfence();
      }
      *flag = last;
    }
    named_bar_sync(1, CT);
    if (p.trace && ctid == 0) p.trace[((size_t)6 * NP + ph) * G + c] = globaltimer_ns();
    if (*flag) {
      for (int ch = wg; ch < nch; ch += 2) {
        ws_reduce_chunk<1>(p.ws, part_slot, parts, ch, m, staging);
        named_bar_sync(wbar, 128);
        epi_dispatch<BN>(g.epi, s_ea, staging, m_tile, n_tile, ch, wt, tpos, tkvr, trs_e, wbar);
        named_bar_sync(wbar, 128);
      }
    }
    named_bar_sync(1, CT);  // flag and part_slot are reused by the next segment
  }
  return true;
}

template <int HD, int BN>
__global__ void __launch_bounds__(FWD_THREADS, 1) fwd_kernel(const FwdParams p) {
  using C = FCfg<BN>;
  using LY = FLayout<HD, BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* ringA = smem + LY::A_OFF;
  uint8_t* ringB = smem + LY::B_OFF;
  float* staging = reinterpret_cast<float*>(smem + LY::STG_OFF);
  uint8_t* att_smem = smem + LY::ATT_OFF;
  float4* rowbuf = reinterpret_cast<float4*>(ringB);   // final norm: one row, d <= 8192 floats
  uint64_t* fullA = reinterpret_cast<uint64_t*>(smem + LY::MISC_OFF);
  uint64_t* emptyA = fullA + C::SA;
  uint64_t* fullB = emptyA + C::SA;
  uint64_t* emptyB = fullB + C::SB;
  uint64_t* tfull = emptyB + C::SB;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint64_t* att_bars = mma_done + 1;                              // 2 per warpgroup
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(att_bars + 4);
  int* flag = reinterpret_cast<int*>(tmem_slot + 1);
  int* flagw = flag + 1;                                          // 2: one per warpgroup
  int* failed = flagw + 2;
  int* go = failed + 1;   // count of GEMM phases whose input the compute warps have seen published
  int* lastA = go + 1;                                            // [SA] parity of last fill, -1 none
  int* lastB = lastA + C::SA;                                     // [SB]
  float* red = reinterpret_cast<float*>(lastB + C::SB);           // 8
  int* part_slot = reinterpret_cast<int*>(red + 8);               // 256
  int* tpos = part_slot + 256;                                    // [BN] QKV token tables
  int* tkvr = tpos + 256;
  float* trs = reinterpret_cast<float*>(tkvr + 256);              // [BN] norm scales (QKV, gate/up)
  GemmArgs* s_ea = reinterpret_cast<GemmArgs*>((reinterpret_cast<uintptr_t>(trs + 256) + 15) &
                                                ~uintptr_t(15));   // epilogue arguments
  static_assert(8 * (2 * C::SA + 2 * C::SB + 9) + 4 * (6 + C::SA + C::SB + 8 + 256 + 768) + 16 + (int)sizeof(GemmArgs) <=
                    C::MISC,
                "shared-memory misc area too small");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x, G = p.G, L = p.L;
  const int NG = 4 * L + 1;      // GEMM phases
  const int NP = 7 * L + 2;      // all phases

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::SA; ++s) {
      mbar_init(&fullA[s], 1);
      mbar_init(&emptyA[s], 1);
      lastA[s] = -1;
    }
    for (int s = 0; s < C::SB; ++s) {
      mbar_init(&fullB[s], 1);
      mbar_init(&emptyB[s], 1);
      lastB[s] = -1;
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 8);   // one arrival per compute warp
    }
    for (int i = 0; i < 4; ++i) mbar_init(&att_bars[i], 1);
    mbar_init(mma_done, 1);
    *go = 0;
    *failed = 0;
    fence_mbar_init();
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Each warpgroup sets its register count at the top of its own branch (every thread executes
  // it; the compute warpgroups' request waits for the roles' release if it comes first), so that
  // the code of each branch is allocated against its own count.
  if (warp < COMPUTE_WARP0) {
  asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsRoles));
  if (warp == 0) {
    // ------------------------------------------------------------- weight producer (never waits for the grid)
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      long long n = 0;
      bool ok = true;
      for (int gi = 0; gi < NG && ok; ++gi) {
        const GP g = gemm_phase(p, gi, BN);
        const CUtensorMap* mA = p.maps + g.mapA;
        SegIter it;
        it.init(g.w, c);
        int tile, k0, k1;
        while (ok && it.next(g.w, tile, k0, k1)) {
          int kx, r0, r1;
          a_coords(g, tile, k0, kx, r0, r1);
          for (int kbi = k0; kbi < k1; ++kbi, ++n, kx += GEMM_BK) {
            const int s = (int)(n % C::SA);
            const uint32_t ph = (uint32_t)((n / C::SA) & 1);
            if (!mwait(&emptyA[s], ph ^ 1u, p.err)) {
              ok = false;
              break;
            }
            uint8_t* sa = ringA + s * C::A_BYTES;
            mbar_arrive_expect_tx(&fullA[s], C::A_BYTES);
            lastA[s] = (int)ph;
            tma_load_2d(sa, mA, &fullA[s], kx, r0, pol);
            tma_load_2d(sa + 8192, mA, &fullA[s], kx, r1, pol);
          }
        }
      }
      if (!ok) *failed = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- activation producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();
      long long n = 0;
      bool ok = true;
      for (int gi = 0; gi < NG && ok; ++gi) {
        const GP g = gemm_phase(p, gi, BN);
        const long long nu = cta_units(g.w, c);
        // the compute warps pass the grid barrier that publishes this phase's input and count it in
        // `go` (one grid poller per CTA)
        if (!cta_count_wait(go, gi + 1, p.err)) {
          ok = false;
          break;
        }
        if (nu == 0) continue;
        if (p.trace) p.trace[((size_t)1 * (7 * L + 2) + gi) * G + c] = globaltimer_ns();
        fence_proxy_async();
        const CUtensorMap* mB = p.maps + g.mapB;
        SegIter it;
        it.init(g.w, c);
        int tile, k0, k1;
        while (ok && it.next(g.w, tile, k0, k1)) {
          const int nt = tile % g.n_tiles;
          for (int kbi = k0; kbi < k1; ++kbi, ++n) {
            const int s = (int)(n % C::SB);
            const uint32_t ph = (uint32_t)((n / C::SB) & 1);
            if (!mwait(&emptyB[s], ph ^ 1u, p.err)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&fullB[s], C::B_BYTES);
            lastB[s] = (int)ph;
            tma_load_2d(ringB + s * C::B_BYTES, mB, &fullB[s], kbi * GEMM_BK, nt * BN, pol);
          }
        }
        if (p.trace) p.trace[((size_t)2 * (7 * L + 2) + gi) * G + c] = globaltimer_ns();
      }
      if (!ok) *failed = 1;
    }
  } else if (warp == 2) {
    // ------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(GEMM_BM, BN);
      long long n = 0;
      int si = 0;
      int mma_waits = 0;
      bool ok = true;
      for (int gi = 0; gi < NG && ok; ++gi) {
        const GP g = gemm_phase(p, gi, BN);
        SegIter it;
        it.init(g.w, c);
        int tile, k0, k1;
        bool any = false;
        while (ok && it.next(g.w, tile, k0, k1)) {
          any = true;
          const long long len = k1 - k0;
          const int acc = si & 1, use = si >> 1;
          ++si;
          if (!mwait(&tempty[acc], (uint32_t)(use & 1) ^ 1u, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tmem_base + (uint32_t)(acc * BN);
          for (long long j = 0; j < len; ++j, ++n) {
            const int sa = (int)(n % C::SA), sb = (int)(n % C::SB);
            const uint32_t pa = (uint32_t)((n / C::SA) & 1), pb = (uint32_t)((n / C::SB) & 1);
            if (!mwait(&fullA[sa], pa, p.err) || !mwait(&fullB[sb], pb, p.err)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t ad = smem_desc_sw128(smem_u32(ringA + sa * C::A_BYTES));
            const uint64_t bd = smem_desc_sw128(smem_u32(ringB + sb * C::B_BYTES));
#pragma unroll
            for (int kk = 0; kk < GEMM_BK / 16; ++kk)
              tc_mma_bf16(dt, ad + (uint64_t)(kk * 2), bd + (uint64_t)(kk * 2), idesc, (j > 0 || kk > 0) ? 1u : 0u);
            tc_commit(&emptyA[sa]);
            tc_commit(&emptyB[sb]);
          }
          if (!ok) break;
          tc_commit(&tfull[acc]);
        }
        if (p.trace && any) {
          // time the last MMA of this phase completed
          tc_commit(mma_done);
          mbar_wait(mma_done, (uint32_t)(mma_waits & 1), nullptr);
          ++mma_waits;
          p.trace[((size_t)3 * (7 * L + 2) + gi) * G + c] = globaltimer_ns();
        }
      }
      if (!ok) *failed = 1;
      tc_commit(mma_done);
      mbar_wait(mma_done, (uint32_t)(mma_waits & 1), nullptr);
    }
  }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsCompute));
    // ------------------------------------------------------------- compute warps (two warpgroups)
    const int ctid = threadIdx.x - COMPUTE_WARP0 * 32;
    const int wg = ctid >> 7, wt = ctid & 127;
    int si = 0;
    int use_att[2] = {0, 0};
    bool ok = true;
    int nb = 0;   // grid barriers passed
    for (int ph = 0; ph < NP && ok; ++ph) {
      // which phase is this?
      int kind, l = 0;   // 0 EMBED, 1 GEMM, 2 ATTN, 3 NORM (mlp, folded), 4 NORM (next attn: folded; final)
      int gi = -1;
      if (ph == 0) {
        kind = 0;
      } else if (ph == NP - 1) {
        kind = 1;
        gi = 4 * L;
      } else {
        l = (ph - 1) / 7;
        const int r = (ph - 1) % 7;
        if (r == 0 || r == 2 || r == 4 || r == 5) {
          kind = 1;
          gi = 4 * l + (r == 0 ? 0 : r == 2 ? 1 : r == 4 ? 2 : 3);
        } else if (r == 1) {
          kind = 2;
        } else if (r == 3) {
          kind = 3;
        } else {
          kind = 4;
        }
      }
      // the norms before the gate/up projection and before the next layer's QKV are folded into
      // the GEMMs around them: no phase, no barrier
      if (kind == 3 || (kind == 4 && l + 1 < L)) continue;
      if (ph > 0) {
        // Barrier nb-1 must be complete before this CTA can arrive at barrier nb: the arrival counter
        // is shared by all barriers, so an early arrival would count towards the previous one.
        // (Non-GEMM phases also read what the previous phase wrote.)
        if (ctid == 0) {
          *flag = grid_wait(p, nb) ? 1 : 0;
          if (*flag && kind == 1) st_release_cta(go, gi + 1);
        }
        ++nb;
        named_bar_sync(1, CT);
        if (!*flag) {
          ok = false;
          break;
        }
        fence_proxy_async();
        named_bar_sync(1, CT);
      }
      if (kind == 0 || kind == 4) {
        norm_phase<BN>(p, kind == 4, kind == 0 ? p.attn_norm[0] : p.final_norm, red, rowbuf, ctid, ph);
      } else if (kind == 2) {
        // both warpgroups leave together: a failed bounded wait in either ends the program
        const bool aok = attn_phase<HD>(p, l, att_smem + wg * LY::ATT_BODY, att_bars + 2 * wg,
                                        use_att, flagw + wg, wt, wg, 2 + wg);
        if (!named_bar_and(1, CT, aok)) {
          ok = false;
          break;
        }
      } else {
        if (!gemm_epi_phase<BN>(p, gi, ph, staging, tfull, tempty, flag, part_slot, tpos, tkvr, trs, s_ea, tmem_base, ctid, si)) {
          ok = false;
          break;
        }
      }
      if (p.trace && ctid == 0) p.trace[(size_t)ph * G + c] = globaltimer_ns();
      // publish this phase: this CTA's generic-proxy stores must be visible to the other CTAs'
      // TMA (async-proxy) reads of the next phases, hence the proxy fence before the release
      if (ph < NP - 1) {
        fence_proxy_async();
        __threadfence();
        named_bar_sync(1, CT);
        if (ctid == 0) atomicAdd(p.bar, 1u);
      }
    }
    if (!ok) *failed = 1;
  }

  __syncthreads();
  if (*failed && threadIdx.x == 0) {
    set_error(p.err, ATSPEED_DEV_ERR_TIMEOUT);
    for (int s = 0; s < C::SA; ++s)
      if (lastA[s] >= 0) mbar_wait(&fullA[s], (uint32_t)lastA[s], nullptr);
    for (int s = 0; s < C::SB; ++s)
      if (lastB[s] >= 0) mbar_wait(&fullB[s], (uint32_t)lastB[s], nullptr);
  }
  __syncthreads();
  if (warp == 2) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

template <int HD, int BN>
cudaError_t launch_t(const FwdParams& p, cudaStream_t st) {
  using LY = FLayout<HD, BN>;
  static std::atomic<unsigned long long> attr_done{0};
  {
    const cudaError_t e = smem_attr_once(attr_done, fwd_kernel<HD, BN>, LY::TOTAL);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.G);
  cfg.blockDim = dim3(FWD_THREADS);
  cfg.dynamicSmemBytes = LY::TOTAL;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fwd_kernel<HD, BN>, p);
}

template <int HD>
cudaError_t launch_hd(const FwdParams& p, cudaStream_t st) {
  return p.T <= 128 ? launch_t<HD, 128>(p, st) : launch_t<HD, 256>(p, st);
}

}  // namespace

size_t fwd_smem_bytes(int hd, int bn) {
  if (bn == 128) return hd == 32 ? FLayout<32, 128>::TOTAL : hd == 64 ? FLayout<64, 128>::TOTAL : FLayout<128, 128>::TOTAL;
  return hd == 32 ? FLayout<32, 256>::TOTAL : hd == 64 ? FLayout<64, 256>::TOTAL : FLayout<128, 256>::TOTAL;
}

cudaError_t fwd_launch(const FwdParams& p, cudaStream_t st) {
  switch (p.hd) {
    case 32: return launch_hd<32>(p, st);
    case 64: return launch_hd<64>(p, st);
    case 128: return launch_hd<128>(p, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace atspeed
