// Device functions of the shared-prefix tree attention, used by the standalone kernels
// (attention.cu) and by the persistent forward kernel (fwd.cu).
#pragma once
#include <cuda.h>
#include <math.h>

#include "attention.cuh"
#include "common.cuh"

namespace atspeed {

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset of (row, 16-byte chunk) inside a K or V tile of ATT_SUB rows as written by TMA.
// HD >= 64: boxes of 64 columns (128 B rows), 128-byte swizzle: chunk ^= row & 7.
// HD == 32: one box of 64-byte rows, no swizzle.
template <int HD>
__device__ __forceinline__ uint32_t kv_off(int row, int chunk16) {
  if constexpr (HD >= 64) {
    const int box = chunk16 >> 3, c = chunk16 & 7;
    return (uint32_t)(box * (ATT_SUB * 128) + row * 128 + ((c ^ (row & 7)) << 4));
  } else {
    return (uint32_t)(row * (HD * 2) + (chunk16 << 4));
  }
}

// Physical 16-byte chunk of logical chunk c of Q row r (conflict-free ldmatrix without padding).
template <int HD>
__device__ __forceinline__ int q_chunk(int r, int c) {
  return c ^ (r & ((HD / 8 < 8 ? HD / 8 : 8) - 1));
}

template <int HD>
struct AttCfg {
  // SMEM_BODY: bytes from the 1024-aligned base: the K/V double buffer (half pages of ATT_SUB keys);
  // the Q tile (rows of HD bf16, 16-byte chunks XOR-swizzled by row) is staged in the second
  // buffer before its first K/V copy (Q lives in registers from then on)
  static constexpr int Q_BYTES = ATT_QTILE * HD * 2;
  static constexpr int KV_BYTES = ATT_SUB * HD * 2;          // one K (or V) half-page tile
  static constexpr int BUF_BYTES = 2 * KV_BYTES;             // K + V
  static constexpr int SMEM_BODY = 2 * BUF_BYTES;
  static_assert(Q_BYTES <= BUF_BYTES, "the Q tile must fit in one K/V buffer");
  static constexpr int SMEM = 1024 + SMEM_BODY + 64;
};

// One work item (query tile, head, prefix split) with 128 threads (4 warps, 16 queries each).
// smem: 1024-aligned, AttCfg<HD>::SMEM_BODY bytes; bars: two mbarriers initialised by the caller
// (count 1) whose completed uses are tracked in use[0], use[1] identically by every thread.
// Writes the normalised output (a.direct) or the split's unnormalised partials.  Returns false if
// a bounded wait timed out.
template <int HD>
__device__ bool attn_item(const AttnArgs& a, const CUtensorMap* mk, const CUtensorMap* mv, int tile, int h, int split,
                          uint8_t* smem, uint64_t* bars, int (&use)[2], int tid, int bar_id,
                          unsigned long long* tr = nullptr, size_t trs = 0) {
#define ATT_TR(k) do { if (tr && tid == 0) tr[(size_t)(k) * trs] = globaltimer_ns(); } while (0)
  using C = AttCfg<HD>;
  constexpr int NDT = HD / 8;    // dim n-tiles of O
  constexpr int NKS = HD / 16;   // k-steps of Q K^T
  uint8_t* kvbuf = smem;                                             // [2][K | V]
  __nv_bfloat16* qs = reinterpret_cast<__nv_bfloat16*>(smem + C::BUF_BYTES);   // buffer 1, until chunk 2's copy
  const int warp = tid >> 5, lane = tid & 31;
  const int d = a.n_heads * HD;
  const int u = a.qt_user[tile];
  const int t0 = a.qt_t0[tile];
  const int nq = a.qt_n[tile];
  const int S_u = a.user_splits[u];
  if (split >= S_u) return true;

  // this item's prefix pages [c0, c1): the split's share of the pages the tile's queries see
  const int* ptab = a.page_table + (size_t)u * a.max_pages;
  constexpr int NBOX = HD >= 64 ? HD / 64 : 1;
  constexpr int BOXW = HD >= 64 ? 64 : HD;
  const int nch = (a.qt_vis[tile] + ATT_PAGE - 1) / ATT_PAGE;
  int c0 = 0, c1 = nch;
  if (a.chunks_per_split > 0) {
    c0 = min(nch, split * a.chunks_per_split);
    c1 = min(nch, c0 + a.chunks_per_split);
  }
  ATT_TR(0);
  int page0 = 0, page1 = 0;   // cache pages of the first two pages (thread 0)
  // copy of half page sc (keys sc * ATT_SUB ...) into buffer buf
  auto issue = [&](int sc, int buf) {
    const int pg = sc / (ATT_PAGE / ATT_SUB);
    const int row0 = (pg == c0 ? page0 : pg == c0 + 1 ? page1 : ptab[pg]) * ATT_PAGE + (sc % (ATT_PAGE / ATT_SUB)) * ATT_SUB;
    uint8_t* kb = kvbuf + buf * C::BUF_BYTES;
    mbar_arrive_expect_tx(&bars[buf], C::BUF_BYTES);
    const uint64_t pol = policy_evict_last();
    for (int b = 0; b < NBOX; ++b) {
      tma_load_2d(kb + b * (ATT_SUB * BOXW * 2), mk, &bars[buf], h * HD + b * BOXW, row0, pol);
      tma_load_2d(kb + C::KV_BYTES + b * (ATT_SUB * BOXW * 2), mv, &bars[buf], h * HD + b * BOXW, row0, pol);
    }
  };
  constexpr int SUBS = ATT_PAGE / ATT_SUB;
  // the first K / V half page does not depend on Q: start its copy now
  if (tid == 0 && c0 < c1) {
    page0 = ptab[c0];
    if (c0 + 1 < c1) page1 = ptab[c0 + 1];
    issue(c0 * SUBS, 0);
  }
  // Q tile -> shared memory (rows >= nq are zero); all of a thread's loads are issued first
  {
    constexpr int NQL = ATT_QTILE * (HD / 8) / 128;
    uint4 v[NQL];
#pragma unroll
    for (int k = 0; k < NQL; ++k) {
      const int i = tid + 128 * k;
      const int r = i / (HD / 8), c = i % (HD / 8);
      v[k] = r < nq ? __ldcg(reinterpret_cast<const uint4*>(a.q + (size_t)(t0 + r) * d + h * HD + c * 8))
                    : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int k = 0; k < NQL; ++k) {
      const int i = tid + 128 * k;
      const int r = i / (HD / 8), c = i % (HD / 8);
      *reinterpret_cast<uint4*>(qs + r * HD + q_chunk<HD>(r, c) * 8) = v[k];
    }
  }
  named_bar_sync(bar_id, 128);
  ATT_TR(1);

  // Q fragments (A operand) for this warp's 16 rows
  uint32_t qf[NKS][4];
  {
    const uint32_t qbase = smem_u32(qs);
    const int r = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
    const int cofs = lane >> 4;   // 16-byte chunk within the 16-column k-step
#pragma unroll
    for (int kk = 0; kk < NKS; ++kk)
      ldsm_x4(qbase + (uint32_t)((r * HD + q_chunk<HD>(r, kk * 2 + cofs) * 8) * 2), qf[kk][0], qf[kk][1], qf[kk][2],
              qf[kk][3]);
  }
  named_bar_sync(bar_id, 128);   // every warp holds its Q fragments: buffer 1 may receive K/V now
  const int g = lane >> 2, tq = lane & 3;
  const int row_a = warp * 16 + g, row_b = row_a + 8;
  const int vis_a = row_a < nq ? a.tok_vis[t0 + row_a] : 0;
  const int vis_b = row_b < nq ? a.tok_vis[t0 + row_b] : 0;
  const float scale = kLog2e / sqrtf((float)HD);

  float o[NDT][4];
#pragma unroll
  for (int j = 0; j < NDT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;
  bool ok = true;

  for (int sc = c0 * SUBS; sc < c1 * SUBS; ++sc) {
    const int buf = (sc - c0 * SUBS) & 1;
    if (tid == 0 && sc + 1 < c1 * SUBS) issue(sc + 1, buf ^ 1);
    const bool got = named_bar_and(bar_id, 128, mbar_wait(&bars[buf], (uint32_t)(use[buf] & 1), a.err));
    if (sc - c0 * SUBS < 2) ATT_TR(2 + 2 * (sc - c0 * SUBS));
    ++use[buf];
    if (!got) {
      ok = false;
      break;
    }
    const uint32_t kbase = smem_u32(kvbuf + buf * C::BUF_BYTES);
    const uint32_t vbase = kbase + C::KV_BYTES;
    {
      constexpr int hk = 0;   // the buffer holds the half page's ATT_SUB = 32 keys
      float s[4][4];
#pragma unroll
      for (int j = 0; j < 4; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
      for (int jj = 0; jj < 2; ++jj) {
#pragma unroll
        for (int kk = 0; kk < NKS; ++kk) {
          // matrices: (keys 16jj+0..7, dims lo), (keys 0..7, dims hi), (keys 8..15, lo), (keys 8..15, hi)
          const int key = hk * 32 + jj * 16 + (lane & 7) + ((lane >> 4) << 3);
          const int ch = kk * 2 + ((lane >> 3) & 1);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(kbase + kv_off<HD>(key, ch), b0, b1, b2, b3);
          mma_bf16_16816(s[2 * jj], qf[kk], b0, b1);
          mma_bf16_16816(s[2 * jj + 1], qf[kk], b2, b3);
        }
      }
      // scale, mask, online softmax (base 2)
      const int kbase_idx = sc * ATT_SUB;
      float mx_a = m_a, mx_b = m_b;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int k0 = kbase_idx + j * 8 + tq * 2;
        s[j][0] = (k0 < vis_a) ? s[j][0] * scale : -INFINITY;
        s[j][1] = (k0 + 1 < vis_a) ? s[j][1] * scale : -INFINITY;
        s[j][2] = (k0 < vis_b) ? s[j][2] * scale : -INFINITY;
        s[j][3] = (k0 + 1 < vis_b) ? s[j][3] * scale : -INFINITY;
        mx_a = fmaxf(mx_a, fmaxf(s[j][0], s[j][1]));
        mx_b = fmaxf(mx_b, fmaxf(s[j][2], s[j][3]));
      }
      mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
      mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
      mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
      mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
      const float ua = (mx_a == -INFINITY) ? 0.f : mx_a;
      const float ub = (mx_b == -INFINITY) ? 0.f : mx_b;
      const float alpha_a = exp2f(m_a - ua), alpha_b = exp2f(m_b - ub);
      m_a = mx_a;
      m_b = mx_b;
      l_a *= alpha_a;
      l_b *= alpha_b;
#pragma unroll
      for (int j = 0; j < NDT; ++j) {
        o[j][0] *= alpha_a;
        o[j][1] *= alpha_a;
        o[j][2] *= alpha_b;
        o[j][3] *= alpha_b;
      }
      uint32_t ph[2][4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float p0 = exp2f(s[j][0] - ua), p1 = exp2f(s[j][1] - ua);
        const float p2 = exp2f(s[j][2] - ub), p3 = exp2f(s[j][3] - ub);
        l_a += p0 + p1;
        l_b += p2 + p3;
        const int kk = j >> 1, r = (j & 1) * 2;
        const __half2 h01 = __floats2half2_rn(p0, p1), h23 = __floats2half2_rn(p2, p3);
        ph[kk][r] = *reinterpret_cast<const uint32_t*>(&h01);
        ph[kk][r + 1] = *reinterpret_cast<const uint32_t*>(&h23);
      }
      // O += P V with P in fp16 (11 significant bits; the row sum l uses the fp32 values) and V fp16
      // (exactly the bf16-rounded values)
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
#pragma unroll
        for (int dd = 0; dd < NDT / 2; ++dd) {
          // trans matrices: (keys 16kk+0..7, dims 16dd+0..7), (keys +8..15, same), (keys 0..7, dims +8..15), (8..15, +8..15)
          const int key = hk * 32 + kk * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
          const int ch = dd * 2 + (lane >> 4);
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(vbase + kv_off<HD>(key, ch), b0, b1, b2, b3);
          mma_f16_16816(o[2 * dd], ph[kk], b0, b1);
          mma_f16_16816(o[2 * dd + 1], ph[kk], b2, b3);
        }
      }
    }
    named_bar_sync(bar_id, 128);  // buffer `buf` may be refilled next iteration
    if (sc - c0 * SUBS < 2) ATT_TR(3 + 2 * (sc - c0 * SUBS));
  }
  if (!ok) {
    // the copy for the next chunk may still be in flight: wait for it (bounded) before returning
    if (tid == 0) {
      for (int b = 0; b < 2; ++b) mbar_wait(&bars[b], (uint32_t)(use[b] & 1), nullptr);
    }
    named_bar_sync(bar_id, 128);
    return false;
  }
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);

  if (a.direct) {
    const float ia = l_a > 0.f ? 1.f / l_a : 0.f, ib = l_b > 0.f ? 1.f / l_b : 0.f;
#pragma unroll
    for (int j = 0; j < NDT; ++j) {
      const int col = h * HD + j * 8 + tq * 2;
      if (row_a < nq)
        *reinterpret_cast<__nv_bfloat162*>(a.out + (size_t)(t0 + row_a) * d + col) =
            __floats2bfloat162_rn(o[j][0] * ia, o[j][1] * ia);
      if (row_b < nq)
        *reinterpret_cast<__nv_bfloat162*>(a.out + (size_t)(t0 + row_b) * d + col) =
            __floats2bfloat162_rn(o[j][2] * ib, o[j][3] * ib);
    }
  } else {
    const size_t base = (size_t)split * a.T;
#pragma unroll
    for (int j = 0; j < NDT; ++j) {
      const int col = j * 8 + tq * 2;
      if (row_a < nq)
        *reinterpret_cast<float2*>(a.part_o + ((base + t0 + row_a) * a.n_heads + h) * HD + col) =
            make_float2(o[j][0], o[j][1]);
      if (row_b < nq)
        *reinterpret_cast<float2*>(a.part_o + ((base + t0 + row_b) * a.n_heads + h) * HD + col) =
            make_float2(o[j][2], o[j][3]);
    }
    if (tq == 0) {
      if (row_a < nq)
        *reinterpret_cast<float2*>(a.part_ml + ((base + t0 + row_a) * a.n_heads + h) * 2) = make_float2(m_a, l_a);
      if (row_b < nq)
        *reinterpret_cast<float2*>(a.part_ml + ((base + t0 + row_b) * a.n_heads + h) * 2) = make_float2(m_b, l_b);
    }
  }
  ATT_TR(6);
#undef ATT_TR
  return true;
}

// Queries per combine group: the merge of one (query tile, head) is split into ATT_QTILE / 16
// groups of 16 queries, each handled by 128 threads (8 per query).
constexpr int ATT_CQ = 16;

// 128 threads: merge the prefix splits of 16 queries (group qg of the tile) of one head with each
// query's path keys and write the normalised bf16 output.  Eight threads per query, each owning
// HD / 8 consecutive dimensions; a path-key dot product adds the eight partial sums by a butterfly
// over the eight lanes (exact in any lane, as fp32 addition commutes), so the result does not
// depend on the schedule that calls it.
template <int HD>
__device__ void attn_combine_group(const AttnArgs& a, int tile, int h, int qg, int ctid) {
  constexpr int TPQ = 8, DH = HD / TPQ;
  const int ql = qg * ATT_CQ + (ctid >> 3), part = ctid & 7;
  const int t0 = a.qt_t0[tile], nq = a.qt_n[tile];
  const bool active = ql < nq;
  const int t = t0 + (active ? ql : 0);
  const int d = a.n_heads * HD;
  const int S = a.user_splits[a.qt_user[tile]];
  const float scale = kLog2e / sqrtf((float)HD);
  const int dim0 = h * HD + part * DH;
  // loads that do not depend on each other first: q, the path rows, the split statistics
  float qv[DH];
  {
    __nv_bfloat16 qb[DH];
#pragma unroll
    for (int i = 0; i < DH; i += 4) *reinterpret_cast<uint2*>(qb + i) = __ldcg(reinterpret_cast<const uint2*>(a.q + (size_t)t * d + dim0 + i));
#pragma unroll
    for (int i = 0; i < DH; ++i) qv[i] = __bfloat162float(qb[i]);
  }
  const int na = (a.anc_n && active) ? a.anc_n[t] : 0;
  int arow[ATT_MAX_ANC];
#pragma unroll
  for (int j = 0; j < ATT_MAX_ANC; ++j) arow[j] = j < na ? a.anc_row[t * ATT_MAX_ANC + j] : 0;
  float M = -INFINITY;
  for (int s = 0; s < S; ++s) M = fmaxf(M, __ldcg(a.part_ml + (((size_t)s * a.T + t) * a.n_heads + h) * 2));
  // path keys (rows written earlier in this forward; cached loads, queries share ancestors)
  float sa[ATT_MAX_ANC];
#pragma unroll
  for (int j = 0; j < ATT_MAX_ANC; ++j) {
    float pd = 0.f;
    if (j < na) {
      __nv_bfloat16 kb[DH];
#pragma unroll
      for (int i = 0; i < DH; i += 4)
        *reinterpret_cast<uint2*>(kb + i) = *reinterpret_cast<const uint2*>(a.k_cache + (size_t)arow[j] * d + dim0 + i);
#pragma unroll
      for (int i = 0; i < DH; ++i) pd += qv[i] * __bfloat162float(kb[i]);
    }
    pd += __shfl_xor_sync(0xffffffffu, pd, 1);
    pd += __shfl_xor_sync(0xffffffffu, pd, 2);
    pd += __shfl_xor_sync(0xffffffffu, pd, 4);
    sa[j] = pd * scale;
    if (j < na) M = fmaxf(M, sa[j]);
  }
  const float Mu = (M == -INFINITY) ? 0.f : M;
  float L = 0.f, o[DH];
#pragma unroll
  for (int i = 0; i < DH; ++i) o[i] = 0.f;
  for (int s = 0; s < S; ++s) {
    const size_t b = ((size_t)s * a.T + t) * a.n_heads + h;
    const float2 ml = __ldcg(reinterpret_cast<const float2*>(a.part_ml + b * 2));
    const float* po = a.part_o + b * HD + part * DH;
    float4 pv[DH / 4];
#pragma unroll
    for (int i = 0; i < DH; i += 4) pv[i / 4] = __ldcg(reinterpret_cast<const float4*>(po + i));
    const float w = exp2f(ml.x - Mu);
    L += ml.y * w;
#pragma unroll
    for (int i = 0; i < DH; i += 4) {
      o[i] += pv[i / 4].x * w;
      o[i + 1] += pv[i / 4].y * w;
      o[i + 2] += pv[i / 4].z * w;
      o[i + 3] += pv[i / 4].w * w;
    }
  }
#pragma unroll
  for (int j = 0; j < ATT_MAX_ANC; ++j) {
    if (j >= na) continue;
    const float w = exp2f(sa[j] - Mu);
    L += w;
    __half vb[DH];
#pragma unroll
    for (int i = 0; i < DH; i += 4)
      *reinterpret_cast<uint2*>(vb + i) = *reinterpret_cast<const uint2*>(a.v_cache + (size_t)arow[j] * d + dim0 + i);
#pragma unroll
    for (int i = 0; i < DH; ++i) o[i] += w * __half2float(vb[i]);
  }
  if (!active) return;
  const float inv = L > 0.f ? 1.f / L : 0.f;
#pragma unroll
  for (int i = 0; i < DH; i += 2)
    *reinterpret_cast<__nv_bfloat162*>(a.out + (size_t)t * d + dim0 + i) = __floats2bfloat162_rn(o[i] * inv, o[i + 1] * inv);
}

}  // namespace atspeed
