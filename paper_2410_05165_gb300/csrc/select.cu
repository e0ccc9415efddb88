// Discrete logic of speculative beam decoding, one CTA (1024 threads) per user:
//   * trie-masked log-softmax of every beam's item-code logits, cumulative fp32 beam scores;
//   * exact top-W selection by (score desc, candidate index asc) with a 4-pass radix select over
//     order-preserving 32-bit keys held in shared memory, then an in-order compaction;
//   * drafting (Eq. 1): top-N (strict) or Gumbel-top-N sampling without replacement (relaxed);
//   * strict top-K verification (Alg. 1) and relaxed sampling verification (Sec. 3.2, Alg. 2),
//     which also cover plain target beam search / sampling when no level is drafted.
// Randomness: Philox4x32-10 (Salmon et al., SC'11), counter = (draw >> 2, level | stream << 8,
// sd_step, user), key = seed, output word draw & 3.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"
#include "tree.cuh"

namespace atspeed {

namespace {

constexpr int NT = 1024;   // threads per CTA
constexpr int NW = NT / 32;

// ---------------------------------------------------------------------------------------------
// Philox4x32-10
// ---------------------------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

__device__ __forceinline__ uint32_t draw_u32(uint64_t seed, int stream, int level, int sd_step, int user,
                                             uint32_t draw) {
  const uint4 r = philox4x32_10(make_uint4(draw >> 2, (uint32_t)(level | (stream << 8)), (uint32_t)sd_step,
                                           (uint32_t)user),
                                (uint32_t)seed, (uint32_t)(seed >> 32));
  const uint32_t w = draw & 3u;
  return w == 0 ? r.x : (w == 1 ? r.y : (w == 2 ? r.z : r.w));
}

__device__ __forceinline__ float u_accept(uint32_t w) { return ((float)(w >> 8) + 1.0f) * 5.9604644775390625e-8f; }
__device__ __forceinline__ float u_open(uint32_t w) {
  return ((float)(w >> 9) * 2.0f + 1.0f) * 5.9604644775390625e-8f;
}
__device__ __forceinline__ float gumbel(uint32_t w) { return -logf(-logf(u_open(w))); }

enum { STREAM_DRAFT = 0, STREAM_ACCEPT = 1, STREAM_SUBSET = 2, STREAM_RESAMPLE = 3 };

// order-preserving map float -> uint32 (finite values map to >= 0x00800000; 0 marks "invalid")
__device__ __forceinline__ uint32_t ordkey(float x) {
  const uint32_t b = __float_as_uint(x);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// ---------------------------------------------------------------------------------------------
// block primitives (blockDim == NT)
// ---------------------------------------------------------------------------------------------
struct Scratch {
  int hist[256];
  int wsum[NW];
  int misc[8];
  float fred[NW];
};

// exclusive scan of one int per thread; returns the exclusive prefix, total in *total
__device__ int block_excl_scan(int v, Scratch& s, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s.wsum[w] = x;
  __syncthreads();
  if (w == 0) {
    int t = s.wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    s.wsum[lane] = t;  // inclusive
  }
  __syncthreads();
  const int before = (w > 0 ? s.wsum[w - 1] : 0) + x - v;
  *total = s.wsum[NW - 1];
  __syncthreads();
  return before;
}

__device__ float block_max(float v, Scratch& s) {
  v = warp_max(v);
  if ((threadIdx.x & 31) == 0) s.fred[threadIdx.x >> 5] = v;
  __syncthreads();
  float r = s.fred[0];
  for (int i = 1; i < NW; ++i) r = fmaxf(r, s.fred[i]);
  __syncthreads();
  return r;
}

__device__ float block_sum(float v, Scratch& s) {
  v = warp_sum(v);
  if ((threadIdx.x & 31) == 0) s.fred[threadIdx.x >> 5] = v;
  __syncthreads();
  float r = 0.f;
  for (int i = 0; i < NW; ++i) r += s.fred[i];  // same fixed order in every thread
  __syncthreads();
  return r;
}

// Selects the W best candidates among keys[0..n) (key 0 = invalid), ranked by (key desc, index
// asc).  Writes their indices to sel[0..m) and returns m = min(W, #valid).
__device__ int block_select(const uint32_t* keys, int n, int W, int* sel, int* tmp, Scratch& s) {
  const int per = (n + NT - 1) / NT;
  const int i0 = threadIdx.x * per, i1 = min(n, i0 + per);
  int c = 0;
  for (int i = i0; i < i1; ++i) c += keys[i] != 0;
  int valid;
  block_excl_scan(c, s, &valid);
  uint32_t tau = 1;   // select every key >= tau ...
  int need_eq = 0x7fffffff;  // ... taking at most need_eq keys equal to tau (in index order)
  if (valid > W) {
    uint32_t prefix = 0, pmask = 0;
    int rem = W;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int b = threadIdx.x; b < 256; b += NT) s.hist[b] = 0;
      __syncthreads();
      for (int i = i0; i < i1; ++i) {
        const uint32_t k = keys[i];
        if (k != 0 && (k & pmask) == prefix) atomicAdd(&s.hist[(k >> shift) & 255u], 1);
      }
      __syncthreads();
      if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        // lane covers bins 255-8*lane .. 248-8*lane (descending)
        int loc = 0;
        for (int j = 0; j < 8; ++j) loc += s.hist[255 - 8 * lane - j];
        int inc = loc;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += y;
        }
        const int exc = inc - loc;
        if (exc < rem && rem <= inc) {
          int cum = exc;
          for (int j = 0; j < 8; ++j) {
            const int b = 255 - 8 * lane - j;
            if (cum + s.hist[b] >= rem) {
              s.misc[0] = b;
              s.misc[1] = rem - cum;
              break;
            }
            cum += s.hist[b];
          }
        }
      }
      __syncthreads();
      const uint32_t b = (uint32_t)s.misc[0];
      rem = s.misc[1];
      prefix |= b << shift;
      pmask |= 0xFFu << shift;
      __syncthreads();
    }
    tau = prefix;
    need_eq = rem;
  }
  // rank of each tau-equal key among the tau-equal keys (index order)
  int e = 0;
  for (int i = i0; i < i1; ++i) e += keys[i] == tau;
  int etot;
  int ebefore = block_excl_scan(e, s, &etot);
  // final flags and in-order compaction into tmp
  int f = 0;
  {
    int er = ebefore;
    for (int i = i0; i < i1; ++i) {
      const uint32_t k = keys[i];
      if (k == 0) continue;
      if (k > tau) ++f;
      else if (k == tau) {
        if (er < need_eq) ++f;
        ++er;
      }
    }
  }
  int m;
  int pos = block_excl_scan(f, s, &m);
  {
    int er = ebefore;
    for (int i = i0; i < i1; ++i) {
      const uint32_t k = keys[i];
      if (k == 0) continue;
      bool take = false;
      if (k > tau) take = true;
      else if (k == tau) {
        take = er < need_eq;
        ++er;
      }
      if (take) tmp[pos++] = i;
    }
  }
  __syncthreads();
  // rank the m selected by (key desc, index asc)
  if (threadIdx.x < m) {
    const int idx = tmp[threadIdx.x];
    const uint32_t k = keys[idx];
    int r = 0;
    for (int j = 0; j < m; ++j) {
      const int o = tmp[j];
      const uint32_t ko = keys[o];
      r += (ko > k) || (ko == k && o < idx);
    }
    sel[r] = idx;
  }
  __syncthreads();
  return m;
}

__device__ __forceinline__ int trie_child(const TreeDev& t, int x, int c) {
  const uint32_t* mk = t.trie_mask + (size_t)x * 8;
  int r = 0;
  for (int w = 0; w < (c >> 5); ++w) r += __popc(mk[w]);
  r += __popc(mk[c >> 5] & ((1u << (c & 31)) - 1u));
  return t.trie_child[x] + r;
}

// One warp: constrained log-probs of the valid children of trie node `tn`, given the 256 logits of
// the node's level: MASKED (log-sum-exp over the valid children) when lse_full is NaN, else FULL
// (lse_full = log-sum-exp of the node's whole-vocabulary row).  Lane l owns codes 8l .. 8l+7;
// returns the valid bits of those codes.
__device__ __forceinline__ uint32_t warp_logprobs(const float* row, const uint32_t* tmask, int tn, float (&lp)[8],
                                                  float lse_full) {
  const int lane = threadIdx.x & 31;
  const uint32_t bits = (tmask[(size_t)tn * 8 + (lane >> 2)] >> ((lane & 3) * 8)) & 0xFFu;
  const float4 x0 = *reinterpret_cast<const float4*>(row + lane * 8);
  const float4 x1 = *reinterpret_cast<const float4*>(row + lane * 8 + 4);
  const float x[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
  float lse = lse_full;
  if (isnan(lse_full)) {
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (bits >> j & 1u) m = fmaxf(m, x[j]);
    m = warp_max(m);
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (bits >> j & 1u) s += expf(x[j] - m);
    s = warp_sum(s);
    lse = m + logf(s);
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) lp[j] = x[j] - lse;
  return bits;
}

// Writes output beam r of user u as (parent node, code, score).
__device__ void write_out(const TreeDev& t, const VerifyOut& o, int K, int u, int r, int parent, int c, float score) {
  const int dp = t.d[u];
  int depth_parent = 0;
  for (int i = 0; i < TREE_L; ++i) depth_parent += t.path[(size_t)parent * 4 + i] >= 0;
  (void)dp;
  for (int i = 0; i < TREE_L; ++i) {
    int v = t.path[(size_t)parent * 4 + i];
    if (i == depth_parent) v = c;
    o.out_path[((size_t)u * K + r) * 4 + i] = v;
  }
  o.out_score[(size_t)u * K + r] = score;
  o.out_parent[(size_t)u * K + r] = parent;
  o.out_trie[(size_t)u * K + r] = trie_child(t, t.trie[parent], c);
  for (int i = 0; i < TREE_L; ++i) {
    o.out_anc_t[((size_t)u * K + r) * 4 + i] = t.anc_t[(size_t)parent * 4 + i];
    o.out_anc_d[((size_t)u * K + r) * 4 + i] = t.anc_d[(size_t)parent * 4 + i];
  }
}

// ---------------------------------------------------------------------------------------------
// drafting: level `lvl` of every user from level lvl-1 using the draft logits
// ---------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(NT) draft_level_kernel(TreeDev t, int lvl, int N, int relaxed, uint64_t seed) {
  extern __shared__ uint8_t sm[];
  __shared__ Scratch s;
  __shared__ int sel[256], tmp[256];
  const int u = blockIdx.x;
  pdl_launch_dependents();
  pdl_wait();
  if (t.d[u] >= TREE_L || lvl > t.g[u]) return;
  const int d = t.d[u];
  const size_t base = (size_t)u * t.stride;
  const int poff = level_off(t, lvl - 1);
  const int pc = t.cnt[u * (t.max_levels + 1) + lvl - 1];
  const int n = pc * TREE_CODES;
  uint32_t* keys = reinterpret_cast<uint32_t*>(sm);
  float* score = reinterpret_cast<float*>(keys + (size_t)max(t.slots_in, t.slots_lvl) * TREE_CODES);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int p = warp; p < pc; p += NW) {
    const size_t node = base + poff + p;
    const float* row = t.logits_d + (size_t)t.lg_d[node] * ITEM_ROWS + (d + lvl - 1) * TREE_CODES;
    float lp[8];
    const uint32_t bits = warp_logprobs(row, t.trie_mask, t.trie[node], lp, t.lse_d ? t.lse_d[t.lg_d[node]] : NAN);
    const float sq0 = t.sq[node];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int idx = p * TREE_CODES + lane * 8 + j;
      if (bits >> j & 1u) {
        const float sc = sq0 + lp[j];
        score[idx] = sc;
        keys[idx] = relaxed ? ordkey(sc + gumbel(draw_u32(seed, STREAM_DRAFT, d + lvl, t.sd_step[u], u, idx)))
                            : ordkey(sc);
      } else {
        keys[idx] = 0u;
      }
    }
  }
  __syncthreads();
  const int m = block_select(keys, n, N, sel, tmp, s);
  const int off = level_off(t, lvl);
  const int depth = d + lvl;
  for (int r = threadIdx.x; r < t.slots_lvl; r += NT) {
    const size_t node = base + off + r;
    if (r < m) {
      const int idx = sel[r];
      const int p = idx >> 8, c = idx & 255;
      const size_t par = base + poff + p;
      t.code[node] = c;
      t.prank[node] = p;
      t.trie[node] = trie_child(t, t.trie[par], c);
      for (int i = 0; i < TREE_L; ++i) {
        t.path[node * 4 + i] = (i == depth - 1) ? c : t.path[par * 4 + i];
        t.anc_t[node * 4 + i] = (i == depth - 1) ? t.row_t[node] : t.anc_t[par * 4 + i];
        t.anc_d[node * 4 + i] = (i == depth - 1) ? t.row_d[node] : t.anc_d[par * 4 + i];
      }
      t.sq[node] = score[idx];
      t.sp[node] = 0.f;
    } else {
      t.code[node] = -1;
      t.prank[node] = -1;
      t.trie[node] = 0;
      for (int i = 0; i < TREE_L; ++i) t.path[node * 4 + i] = -1;
      t.sq[node] = -INFINITY;
    }
  }
  if (threadIdx.x == 0) t.cnt[u * (t.max_levels + 1) + lvl] = m;
}

// ---------------------------------------------------------------------------------------------
// strict top-K verification (Alg. 1); g = 0 gives one step of plain target beam search.
// probe != 0 (g >= 1): only level 1 is examined -- a user whose level 1 is rejected gets its
// complete output exactly as in the full call (it depends on the level-0 logits alone); a user
// whose level 1 is accepted gets accepted = -1 and nothing else.
// ---------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(NT) verify_strict_kernel(TreeDev t, int K, VerifyOut o, int probe) {
  extern __shared__ uint8_t sm[];
  __shared__ Scratch s;
  __shared__ int sel[256], tmp[256];
  __shared__ int yp_node[256];
  __shared__ float yp_sp[256];
  __shared__ int match[256];
  __shared__ int n_yp, all_ok;
  const int u = blockIdx.x;
  pdl_launch_dependents();
  pdl_wait();
  const int d = t.d[u], g = t.g[u];
  if (d >= TREE_L) return;
  const size_t base = (size_t)u * t.stride;
  uint32_t* keys = reinterpret_cast<uint32_t*>(sm);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) n_yp = t.cnt[u * (t.max_levels + 1)];
  __syncthreads();
  for (int i = threadIdx.x; i < n_yp; i += NT) {
    yp_node[i] = (int)(base + i);
    yp_sp[i] = t.sp[base + i];
  }
  __syncthreads();
  float* score = reinterpret_cast<float*>(keys + (size_t)max(t.slots_in, t.slots_lvl) * TREE_CODES);
  const int last = (d + g < TREE_L) ? g + 1 : g;
  int a = 0, adv = 0, m = 0;
  for (int j = 1; j <= last; ++j) {
    const int n = n_yp * TREE_CODES;
    for (int p = warp; p < n_yp; p += NW) {
      const int node = yp_node[p];
      const float* row = t.logits_t + (size_t)t.lg_t[node] * ITEM_ROWS + (d + j - 1) * TREE_CODES;
      float lp[8];
      const uint32_t bits = warp_logprobs(row, t.trie_mask, t.trie[node], lp, t.lse_t ? t.lse_t[t.lg_t[node]] : NAN);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int idx = p * TREE_CODES + lane * 8 + q;
        const float sc = yp_sp[p] + lp[q];
        score[idx] = sc;
        keys[idx] = (bits >> q & 1u) ? ordkey(sc) : 0u;
      }
    }
    __syncthreads();
    m = block_select(keys, n, K, sel, tmp, s);
    if (j > g) {  // all drafted levels accepted: Y^p_{g+1} is the output
      a = g;
      adv = g + 1;
      break;
    }
    // is every selected (parent, code) a drafted node of level j?
    const int off = level_off(t, j), poff = level_off(t, j - 1);
    const int nq = t.cnt[u * (t.max_levels + 1) + j];
    if (threadIdx.x == 0) all_ok = 1;
    __syncthreads();
    if (threadIdx.x < m) {
      const int idx = sel[threadIdx.x];
      const int pnode = yp_node[idx >> 8], c = idx & 255;
      int f = -1;
      for (int i = 0; i < nq; ++i) {
        const size_t nd = base + off + i;
        if (t.code[nd] == c && (int)(base + poff + t.prank[nd]) == pnode) {
          f = (int)nd;
          break;
        }
      }
      match[threadIdx.x] = f;
      if (f < 0) atomicAnd(&all_ok, 0);
    }
    __syncthreads();
    if (probe && all_ok) {
      if (threadIdx.x == 0) o.accepted[u] = -1;
      return;
    }
    if (!all_ok) {
      a = j - 1;
      adv = j;
      break;
    }
    // accepted: Y^p_j becomes the parents of step j + 1 (all of them are drafted tree nodes)
    float nsp = 0.f;
    if (threadIdx.x < m) nsp = score[sel[threadIdx.x]];
    __syncthreads();
    if (threadIdx.x < m) {
      yp_node[threadIdx.x] = match[threadIdx.x];
      yp_sp[threadIdx.x] = nsp;
      t.sp[match[threadIdx.x]] = nsp;
    }
    if (threadIdx.x == 0) n_yp = m;
    __syncthreads();
    a = j;
    if (j == g && d + g >= TREE_L) {  // item complete: output Y^p_g
      adv = g;
      m = -m;  // marker: output is yp itself
      break;
    }
  }
  if (m < 0) {
    m = -m;
    if (threadIdx.x < m) {
      const int nd = yp_node[threadIdx.x];
      const int par = (int)(base + level_off(t, g - 1) + t.prank[nd]);
      write_out(t, o, K, u, threadIdx.x, par, t.code[nd], yp_sp[threadIdx.x]);
    }
  } else {
    if (threadIdx.x < m) {
      const int idx = sel[threadIdx.x];
      write_out(t, o, K, u, threadIdx.x, yp_node[idx >> 8], idx & 255, score[idx]);
    }
  }
  if (threadIdx.x == 0) {
    o.accepted[u] = a;
    o.advance[u] = adv;
    o.n_out[u] = m;
    o.n_acc_last[u] = 0;
  }
}

// ---------------------------------------------------------------------------------------------
// relaxed sampling verification (Sec. 3.2, Alg. 2); g = 0 gives one step of sampling beam search.
// probe != 0 (g >= 1): as in the strict kernel, a user whose level 1 is rejected (|A| < K) gets
// its complete output, one whose level 1 is accepted gets accepted = -1.
// ---------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(NT) verify_relaxed_kernel(TreeDev t, int K, VerifyOut o, uint64_t seed,
                                                            int probe) {
  extern __shared__ uint8_t sm[];
  __shared__ Scratch s;
  __shared__ int sel[256], tmp[256];
  __shared__ int accd[256];     // accepted drafted slots, draft order
  __shared__ int outc[256];     // output candidate indices
  const int u = blockIdx.x;
  pdl_launch_dependents();
  pdl_wait();
  const int d = t.d[u], g = t.g[u], step = t.sd_step[u];
  if (d >= TREE_L) return;
  const size_t base = (size_t)u * t.stride;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int maxp = max(t.slots_in, t.slots_lvl);
  float* Sp = reinterpret_cast<float*>(sm);
  float* Sq = Sp + maxp * TREE_CODES;      // later reused as keys
  uint32_t* keys = reinterpret_cast<uint32_t*>(Sq);
  int a = 0, adv = 0, nout = 0, nacc_last = 0;
  int plvl = 0;  // level of the current parents (drafted beams Y^q_{j-1})
  for (int j = 1; j <= g + 1; ++j) {
    if (j == g + 1 && d + g >= TREE_L) break;  // cannot happen: handled at j == g
    const int poff = level_off(t, plvl);
    const int pc = t.cnt[u * (t.max_levels + 1) + plvl];
    const int n = pc * TREE_CODES;
    const int lvl_abs = d + j;
    // target and draft sequence scores of every candidate in C_j
    for (int p = warp; p < pc; p += NW) {
      const size_t node = base + poff + p;
      const float* rp = t.logits_t + (size_t)t.lg_t[node] * ITEM_ROWS + (lvl_abs - 1) * TREE_CODES;
      float lp[8];
      const uint32_t bits = warp_logprobs(rp, t.trie_mask, t.trie[node], lp, t.lse_t ? t.lse_t[t.lg_t[node]] : NAN);
      const float spn = t.sp[node];
#pragma unroll
      for (int q = 0; q < 8; ++q) Sp[p * TREE_CODES + lane * 8 + q] = (bits >> q & 1u) ? spn + lp[q] : -INFINITY;
      if (j <= g) {
        const float* rq = t.logits_d + (size_t)t.lg_d[node] * ITEM_ROWS + (lvl_abs - 1) * TREE_CODES;
        float lq[8];
        warp_logprobs(rq, t.trie_mask, t.trie[node], lq, t.lse_d ? t.lse_d[t.lg_d[node]] : NAN);
        const float sqn = (plvl == 0) ? spn : t.sq[node];
#pragma unroll
        for (int q = 0; q < 8; ++q) Sq[p * TREE_CODES + lane * 8 + q] = (bits >> q & 1u) ? sqn + lq[q] : -INFINITY;
      }
    }
    __syncthreads();
    if (j == g + 1) {
      // every drafted level accepted: sample K from p_{g+1} over the extensions of Y^q_g
      for (int i = threadIdx.x; i < n; i += NT) {
        const float v = Sp[i];
        keys[i] = (v == -INFINITY) ? 0u
                                    : ordkey(v + gumbel(draw_u32(seed, STREAM_RESAMPLE, lvl_abs, step, u, i)));
      }
      __syncthreads();
      nout = block_select(keys, n, K, sel, tmp, s);
      if (threadIdx.x < nout) outc[threadIdx.x] = sel[threadIdx.x];
      a = g;
      adv = g + 1;
      __syncthreads();
      break;
    }
    // softmax normalisers over C_j (fp32)
    float mp = -INFINITY, mq = -INFINITY;
    for (int i = threadIdx.x; i < n; i += NT) {
      mp = fmaxf(mp, Sp[i]);
      mq = fmaxf(mq, Sq[i]);
    }
    mp = block_max(mp, s);
    mq = block_max(mq, s);
    float sp_ = 0.f, sq_ = 0.f;
    for (int i = threadIdx.x; i < n; i += NT) {
      if (Sp[i] != -INFINITY) {
        sp_ += expf(Sp[i] - mp);
        sq_ += expf(Sq[i] - mq);
      }
    }
    const float lse_p = mp + logf(block_sum(sp_, s));
    const float lse_q = mq + logf(block_sum(sq_, s));
    // acceptance test of every drafted sequence, in draft order
    const int off = level_off(t, j);
    const int nd = t.cnt[u * (t.max_levels + 1) + j];
    int f = 0, ci = -1;
    if (threadIdx.x < nd) {
      const size_t node = base + off + threadIdx.x;
      ci = t.prank[node] * TREE_CODES + t.code[node];
      const float logp = Sp[ci] - lse_p, logq = Sq[ci] - lse_q;
      const float ratio = fminf(1.0f, expf(logp - logq));
      const float uu = u_accept(draw_u32(seed, STREAM_ACCEPT, lvl_abs, step, u, (uint32_t)threadIdx.x));
      f = uu <= ratio;
    }
    int na;
    const int pos = block_excl_scan(f, s, &na);
    if (f) accd[pos] = threadIdx.x;
    __syncthreads();
    nacc_last = na;
    if (probe && na >= K) {
      if (threadIdx.x == 0) o.accepted[u] = -1;
      return;
    }
    if (na >= K) {
      if (j < g) {
        // step accepted: the drafted beams of level j carry their target scores to step j + 1
        if (threadIdx.x < nd) t.sp[base + off + threadIdx.x] = Sp[ci];
        __syncthreads();
        plvl = j;
        continue;
      }
      if (d + g < TREE_L) {
        if (threadIdx.x < nd) t.sp[base + off + threadIdx.x] = Sp[ci];
        __syncthreads();
        plvl = j;
        continue;  // j == g: sample Y_{g+1} from p_{g+1} at the next iteration
      }
      // item complete: K uniform picks among the accepted drafts: the K smallest Philox words
      // (ties to the lower draft slot), ranked exactly by pairwise comparison
      __shared__ uint32_t wsub[256];
      if (threadIdx.x < na)
        wsub[threadIdx.x] = draw_u32(seed, STREAM_SUBSET, lvl_abs, step, u, (uint32_t)accd[threadIdx.x]);
      __syncthreads();
      int mm = 0;
      if (threadIdx.x < na) {
        const uint32_t w = wsub[threadIdx.x];
        int r = 0;
        for (int q = 0; q < na; ++q) r += (wsub[q] < w) || (wsub[q] == w && q < (int)threadIdx.x);
        if (r < K) {
          const size_t node = base + off + accd[threadIdx.x];
          tmp[r] = t.prank[node] * TREE_CODES + t.code[node];
        }
      }
      __syncthreads();
      mm = min(K, na);
      if (threadIdx.x < mm) outc[threadIdx.x] = tmp[threadIdx.x];
      nout = mm;
      a = g;
      adv = g;
      __syncthreads();
      break;
    }
    // step rejected: A plus K - |A| draws from norm(max(0, p - q)), zero on A
    const int need = K - na;
    // tier 1: candidates outside A with p' > 0, keyed by log p' + Gumbel; tier 2 (only if tier 1
    // runs out, e.g. p = q): the rest of C_j \ A keyed by log p + Gumbel.  Keys overwrite Sq.
    for (int i = threadIdx.x; i < n; i += NT) {
      uint32_t kk = 0u;
      const float spv = Sp[i];
      if (spv != -INFINITY) {
        const float logp = spv - lse_p, logq = Sq[i] - lse_q;
        const float pr = fmaxf(0.f, expf(logp) - expf(logq));
        if (pr > 0.f) kk = ordkey(logf(pr) + gumbel(draw_u32(seed, STREAM_RESAMPLE, lvl_abs, step, u, (uint32_t)i)));
      }
      keys[i] = kk;
    }
    __syncthreads();
    if (threadIdx.x < na) {
      const size_t node = base + off + accd[threadIdx.x];
      keys[t.prank[node] * TREE_CODES + t.code[node]] = 0u;  // A is not resampled
    }
    __syncthreads();
    int mm = block_select(keys, n, need, sel, tmp, s);
    if (threadIdx.x < na) {
      const size_t node = base + off + accd[threadIdx.x];
      outc[threadIdx.x] = t.prank[node] * TREE_CODES + t.code[node];
    }
    if (threadIdx.x < mm) outc[na + threadIdx.x] = sel[threadIdx.x];
    __syncthreads();
    if (mm < need) {
      // tier 2 over the candidates not yet chosen
      for (int i = threadIdx.x; i < n; i += NT) {
        const float spv = Sp[i];
        keys[i] = (spv == -INFINITY)
                      ? 0u
                      : ordkey((spv - lse_p) + gumbel(draw_u32(seed, STREAM_RESAMPLE, lvl_abs, step, u, (uint32_t)i)));
      }
      __syncthreads();
      for (int q = threadIdx.x; q < na + mm; q += NT) keys[outc[q]] = 0u;
      __syncthreads();
      const int m2 = block_select(keys, n, need - mm, sel, tmp, s);
      if (threadIdx.x < m2) outc[na + mm + threadIdx.x] = sel[threadIdx.x];
      mm += m2;
      __syncthreads();
    }
    nout = na + mm;
    a = j - 1;
    adv = j;
    __syncthreads();
    break;
  }
  // rank the output by (target score desc, candidate index asc) and write it
  {
    const int poff = level_off(t, plvl);
    if (threadIdx.x < nout) {
      const int ci = outc[threadIdx.x];
      const float sc = Sp[ci];
      int r = 0;
      for (int q = 0; q < nout; ++q) {
        const int cq = outc[q];
        const float so = Sp[cq];
        r += (so > sc) || (so == sc && cq < ci);
      }
      write_out(t, o, K, u, r, (int)(base + poff + (ci >> 8)), ci & 255, sc);
    }
  }
  if (threadIdx.x == 0) {
    o.accepted[u] = a;
    o.advance[u] = adv;
    o.n_out[u] = nout;
    o.n_acc_last[u] = nacc_last;
  }
}

cudaLaunchConfig_t cfg_for(int B, size_t smem, cudaStream_t st, cudaLaunchAttribute* at, bool pdl) {
  cudaLaunchConfig_t c = {};
  c.gridDim = dim3(B);
  c.blockDim = dim3(NT);
  c.dynamicSmemBytes = smem;
  c.stream = st;
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  c.attrs = at;
  c.numAttrs = pdl ? 1 : 0;
  return c;
}

template <typename Kern>
cudaError_t set_smem(Kern k, size_t smem) {
  return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

}  // namespace

size_t select_smem_bytes(int max_parents) { return (size_t)max_parents * TREE_CODES * 8 + 64; }

cudaError_t draft_level_launch(const TreeDev& t, int lvl, int N, bool relaxed, uint64_t seed, cudaStream_t st,
                               bool pdl) {
  const size_t smem = select_smem_bytes(max(t.slots_in, t.slots_lvl));
  cudaError_t e = set_smem(draft_level_kernel, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute at[1];
  cudaLaunchConfig_t c = cfg_for(t.B, smem, st, at, pdl);
  return cudaLaunchKernelEx(&c, draft_level_kernel, t, lvl, N, relaxed ? 1 : 0, seed);
}

cudaError_t verify_launch(const TreeDev& t, int K, bool relaxed, uint64_t seed, const VerifyOut& o, cudaStream_t st,
                          bool pdl, bool probe) {
  const size_t smem = select_smem_bytes(max(t.slots_in, t.slots_lvl));
  cudaLaunchAttribute at[1];
  cudaLaunchConfig_t c = cfg_for(t.B, smem, st, at, pdl);
  if (relaxed) {
    cudaError_t e = set_smem(verify_relaxed_kernel, smem);
    if (e != cudaSuccess) return e;
    return cudaLaunchKernelEx(&c, verify_relaxed_kernel, t, K, o, seed, probe ? 1 : 0);
  }
  cudaError_t e = set_smem(verify_strict_kernel, smem);
  if (e != cudaSuccess) return e;
  return cudaLaunchKernelEx(&c, verify_strict_kernel, t, K, o, probe ? 1 : 0);
}

}  // namespace atspeed
