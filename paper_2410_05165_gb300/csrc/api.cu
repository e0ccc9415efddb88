// Host runtime behind include/atspeed.h: context (weights, trie, KV arenas, node table, scratch),
// the decoder forward, and the prefill / draft_step / verify / beam_search calls.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <array>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "atspeed.h"
#include "common.cuh"
#include "attention.cuh"
#include "fwd.cuh"
#include "gemm.cuh"
#include "kernels.cuh"
#include "tree.cuh"

using namespace atspeed;
typedef __nv_bfloat16 bf16;

namespace {

thread_local std::string g_create_error;

// Prefix pages per attention split of a model's tree forwards, fixed per context (so a node's
// output does not depend on the call it is in): among 1, 2, 4, ... pages, the one that minimises
// the estimated time of the attention phase -- rounds of work items over the 2 x grid warpgroup
// slots, each item costing a fixed start (Q, first K / V copy, partials; ~9 us) plus ~2.2 us per
// page -- for the limits' typical call: max_users users of min(3 max_N, node slots) tree tokens,
// in query tiles of 64, times the heads.  One user at the bench shape gets 2 pages (256 items in
// one round); 16 users get whole-prefix items (many rounds, so fewer and longer items win).
int attention_pages_per_split(const atspeed_limits& L, int H, int grid) {
  const int pages = std::max(1, (L.max_prompt + ATT_PAGE - 1) / ATT_PAGE);
  const int stride = L.max_K + L.max_gamma * L.max_N;
  const int tokens = std::max(1, std::min(3 * L.max_N, stride));
  const long long pairs = (long long)L.max_users * ((tokens + ATT_QTILE - 1) / ATT_QTILE) * H;
  int best = 1;
  double best_t = 1e30;
  for (int cps = 1; cps < 2 * pages; cps *= 2) {
    const long long items = pairs * ((pages + cps - 1) / cps);
    const long long rounds = (items + 2LL * grid - 1) / (2LL * grid);
    const double t = (double)rounds * (9.0 + 2.2 * std::min(cps, pages));
    if (t < best_t - 1e-9) {
      best_t = t;
      best = cps;
    }
  }
  return best;
}

struct Fail {
  atspeed_status st;
};

struct ModelRt {
  bool present = false;
  bool per_op = false;   // this model's forward runs one kernel per op (else one persistent launch)
  int grid = 0;          // CTAs of its GEMM work splits (both schedules, so both give the same bits)
  int cps = 2;           // prefix pages per attention split of its tree forwards (fixed per context)
  int layers = 0, d = 0, H = 0, hd = 0, ffn = 0, V = 0;
  float eps = 1e-6f, theta = 1e4f;
  const bf16 *embed = nullptr, *final_norm = nullptr, *lm_head = nullptr;
  std::vector<const bf16*> attn_norm, wqkv, wo, mlp_norm, wgate_up, wdown;
  // KV arena: [layers][rows][d]
  bf16* kc = nullptr;
  __half* vc = nullptr;
  int rows = 0;
  std::vector<CUtensorMap> mk, mv;
  float *rope_cos = nullptr, *rope_sin = nullptr;  // [max_pos][hd/2]
  int max_pos = 0;
  // activations
  int Tcap = 0, Xrows = 0;
  float* h = nullptr;
  float* ssq = nullptr;  // [ceil(d / 128)][Tcap] partial sums of squares of the residual rows per
                         // 128-row tile (RMSNorm folded into the GEMMs around it)
  bf16 *x = nullptr, *q = nullptr, *att = nullptr, *act = nullptr;
  float* logits = nullptr;  // [logit_rows][1024]
  int logit_rows = 0;
  // FULL normalisation: whole-vocabulary log-sum-exp per logits row, the LM head's per-tile
  // partials [ceil(V / 128)][lse_ld], and the prefill's final-norm rows of the last history tokens
  float* lse = nullptr;
  float2* lse_part = nullptr;
  int lse_ld = 0;
  bf16* root_x = nullptr;
  int root_rows = 0;
  // per-token forward inputs
  int *tok = nullptr, *pos = nullptr, *kvrow = nullptr, *tuser = nullptr, *tvis = nullptr, *anc = nullptr,
      *ancn = nullptr;
  int *qt_t0 = nullptr, *qt_n = nullptr, *qt_user = nullptr, *qt_vis = nullptr, *rows_sel = nullptr,
      *user_splits = nullptr;
  float *part_o = nullptr, *part_ml = nullptr;
  int max_splits = 1;
  // persistent forward kernel
  CUtensorMap* maps = nullptr;           // device table, layout in fwd.cuh
  const bf16** d_attn_norm = nullptr;    // device arrays of layer pointers
  const bf16** d_mlp_norm = nullptr;
  int* att_counters = nullptr;
  int* plan_blk = nullptr;   // qt_* / user_splits / rows_sel of the current forward, packed
  int max_qt = 0;
};

struct UserState {
  int P = 0;          // prompt length
  int d = 0;          // depth of the incoming beams
  int step = 0;       // speculative steps taken (Philox counter word)
  int region = 0;     // node-row region of the next step (never reused within one decode)
  int g = 0;          // drafted levels of the current step
  bool active = false;
  // incoming beams (level 0 of the next tree)
  std::vector<std::array<int, 4>> path;
  std::vector<float> sp;
  std::vector<int> trie;
  std::vector<std::array<int, 4>> anc_t, anc_d;
  // statistics
  int acc_steps = 0, calls = 0, tree_tokens = 0;
};

}  // namespace

struct atspeed_ctx {
  std::string err;
  int device = 0;
  ModelRt tgt, drf;
  int code_base = 0;
  atspeed_limits lim{};
  // trie
  std::vector<uint32_t> h_mask;
  std::vector<int> h_child;
  uint32_t* trie_mask = nullptr;
  int* trie_child = nullptr;
  // scratch
  GemmScratch gs{};
  int gemm_grid = 1;
  unsigned int* err_word = nullptr;
  // node table
  int cap_nodes = 0, node_rows_per_user = 0, prefix_pages_per_user = 0;
  int *n_code = nullptr, *n_prank = nullptr, *n_trie = nullptr, *n_path = nullptr, *n_row_t = nullptr,
      *n_row_d = nullptr, *n_anc_t = nullptr, *n_anc_d = nullptr, *n_lg_t = nullptr, *n_lg_d = nullptr,
      *n_cnt = nullptr;
  float *n_sq = nullptr, *n_sp = nullptr;
  int *u_d = nullptr, *u_g = nullptr, *u_step = nullptr, *u_P = nullptr, *page_table = nullptr;
  int* fwd_nodes = nullptr;
  // pinned host staging for uploads and downloads: regions are handed out in order and reclaimed
  // at the next synchronisation of the stream (every copy staged before it has then completed)
  uint8_t* h_stage = nullptr;
  size_t stage_cap = 0, stage_used = 0;
  int* n_blk = nullptr;     // node table: the n_* arrays, packed for the current step's size
  int* u_blk = nullptr;     // per-user d, g, step, P (max_users each)
  int* o_blk = nullptr;     // verification outputs (fixed sections, max_users x max_K)
  int* o_anc_t = nullptr;   // [max_users][max_K][4] ancestor rows of the output beams' parents
  int* o_anc_d = nullptr;
  int* fwd_zero = nullptr;  // grid barrier, split arrivals and attention arrivals, zeroed per forward
  size_t fwd_zero_att = 0;  // offset of the attention arrivals in fwd_zero
  // verify outputs
  int *o_acc = nullptr, *o_adv = nullptr, *o_n = nullptr, *o_nacc = nullptr, *o_path = nullptr, *o_parent = nullptr,
      *o_trie = nullptr;
  float* o_score = nullptr;
  // host state
  int B = 0;
  bool prefilled = false;
  bool step_open = false;      // level 0 of the current step is on the device
  bool full_norm = false;      // the current step normalises over the whole vocabulary (FULL)
  int step_K = 0, step_N = 0, step_gamma = 0, levels_done = 0;
  bool roots_drafted = false;
  bool level_fwd_pending = false;  // the draft forward of level `levels_done` has not run yet
  bool early_reject = false;       // decide level 1 of depth-0 steps before any forward over it
  bool tree_injected = false;
  bool have_tree = false;      // a node table exists (debug hooks may read it)
  std::vector<UserState> users;
  std::vector<void*> allocs;
  bool pdl = true;
  // optional per-launch timing (CUDA events on the launching stream)
  bool prof = false;
  struct ProfRec {
    int kind;
    double bytes, flops;
    cudaEvent_t a, b;
  };
  std::vector<ProfRec> prof_recs;
  std::vector<cudaEvent_t> prof_pool;
  long long n_launch = 0;  // kernels launched by this context (all kinds)
  int forward_mode = 0;    // ATSPEED_FORWARD: 0 default (persistent), 1 persistent, 2 one kernel per op
  int fwd_grid = 0;
  unsigned int* fwd_bar = nullptr;
  int* fwd_sk = nullptr;     // split-tile arrival counters of the persistent forward
  size_t fwd_sk_n = 0;
  unsigned long long* fwd_trace = nullptr;  // per-phase timestamps of the last forward (tracing on)
  size_t fwd_trace_n = 0;
};

namespace {

void set_err(atspeed_ctx* c, const char* fmt, ...) {
  char buf[1024];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (c)
    c->err = buf;
  else
    g_create_error = buf;
}

#define CK(call)                                                                              \
  do {                                                                                        \
    cudaError_t e_ = (call);                                                                  \
    if (e_ != cudaSuccess) {                                                                  \
      set_err(c, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, __LINE__); \
      throw Fail{ATSPEED_E_CUDA};                                                             \
    }                                                                                         \
  } while (0)

template <typename T>
T* dalloc(atspeed_ctx* c, size_t n, bool zero = true) {
  void* p = nullptr;
  if (n == 0) n = 1;
  cudaError_t e = cudaMalloc(&p, n * sizeof(T));
  if (e != cudaSuccess) {
    set_err(c, "cudaMalloc of %zu bytes failed: %s", n * sizeof(T), cudaGetErrorString(e));
    throw Fail{ATSPEED_E_OOM};
  }
  c->allocs.push_back(p);
  if (zero) {
    e = cudaMemset(p, 0, n * sizeof(T));
    if (e != cudaSuccess) {
      set_err(c, "cudaMemset failed: %s", cudaGetErrorString(e));
      throw Fail{ATSPEED_E_CUDA};
    }
  }
  return static_cast<T*>(p);
}

void stage_sync(atspeed_ctx* c, cudaStream_t st);
template <typename T>
T* stage_alloc(atspeed_ctx* c, cudaStream_t st, size_t n);

// Synchronises the stream and reads the device error word (one download through the staging
// buffer; regions staged before the call stay readable until the next staging request).
void check_device_error(atspeed_ctx* c, cudaStream_t st) {
  unsigned int* hw = stage_alloc<unsigned int>(c, st, 1);
  CK(cudaMemcpyAsync(hw, c->err_word, sizeof(unsigned int), cudaMemcpyDeviceToHost, st));
  stage_sync(c, st);
  const unsigned int w = *hw;
  if (w) {
    CK(cudaMemset(c->err_word, 0, sizeof w));
    set_err(c, "device error word 0x%x (%s)", w, (w & ATSPEED_DEV_ERR_TIMEOUT) ? "bounded wait timed out" : "bounds");
    throw Fail{(w & ATSPEED_DEV_ERR_TIMEOUT) ? ATSPEED_E_TIMEOUT : ATSPEED_E_CUDA};
  }
}

void stage_sync(atspeed_ctx* c, cudaStream_t st) {
  CK(cudaStreamSynchronize(st));
  c->stage_used = 0;
}

// A region of the pinned staging buffer that stays untouched until the stream's next
// synchronisation by stage_sync (which the next region may force when the buffer is full).
template <typename T>
T* stage_alloc(atspeed_ctx* c, cudaStream_t st, size_t n) {
  const size_t bytes = (n * sizeof(T) + 255) & ~size_t(255);
  if (bytes > c->stage_cap) {
    set_err(c, "staging request of %zu bytes exceeds the %zu-byte staging buffer", bytes, c->stage_cap);
    throw Fail{ATSPEED_E_SHAPE};
  }
  if (c->stage_used + bytes > c->stage_cap) stage_sync(c, st);
  T* p = reinterpret_cast<T*>(c->h_stage + c->stage_used);
  c->stage_used += bytes;
  return p;
}

// Host-to-device copy through the staging buffer (the source may be freed on return).
void upload(atspeed_ctx* c, cudaStream_t st, void* dst, const void* src, size_t bytes) {
  if (bytes == 0) return;
  uint8_t* h = stage_alloc<uint8_t>(c, st, bytes);
  memcpy(h, src, bytes);
  CK(cudaMemcpyAsync(dst, h, bytes, cudaMemcpyHostToDevice, st));
}

// Points the n_* arrays at consecutive sections of the node-table block for n slots and B users
// of g drafted levels (one contiguous upload in open_step).
void carve_nodes(atspeed_ctx* c, size_t n, int B, int g) {
  int* q = c->n_blk;
  c->n_code = q, q += n;
  c->n_prank = q, q += n;
  c->n_trie = q, q += n;
  c->n_path = q, q += 4 * n;
  c->n_row_t = q, q += n;
  c->n_row_d = q, q += n;
  c->n_anc_t = q, q += 4 * n;
  c->n_anc_d = q, q += 4 * n;
  c->n_lg_t = q, q += n;
  c->n_lg_d = q, q += n;
  c->n_sq = reinterpret_cast<float*>(q), q += n;
  c->n_sp = reinterpret_cast<float*>(q), q += n;
  c->n_cnt = q, q += (size_t)B * (g + 1);
}
constexpr size_t NODE_INTS = 21;   // ints per slot in the node table (the n_* arrays above)
size_t o_blk_ints(int mu, int mK) { return 4 * (size_t)mu + 15 * (size_t)mu * mK; }

void init_model(atspeed_ctx* c, ModelRt& m, const atspeed_model_desc* md, const char* name) {
  if (!md) return;
  if (md->n_layers <= 0 || md->d_model <= 0 || md->n_heads <= 0 || md->d_ffn <= 0 || md->vocab <= 0) {
    set_err(c, "%s: non-positive dimension", name);
    throw Fail{ATSPEED_E_ARG};
  }
  if (md->d_model % md->n_heads) {
    set_err(c, "%s: d_model %% n_heads != 0", name);
    throw Fail{ATSPEED_E_SHAPE};
  }
  const int hd = md->d_model / md->n_heads;
  if (hd != 32 && hd != 64 && hd != 128) {
    set_err(c, "%s: head_dim %d not in {32, 64, 128}", name, hd);
    throw Fail{ATSPEED_E_SHAPE};
  }
  if (md->d_model % 64 || md->d_ffn % 64 || md->d_model > 8192) {
    set_err(c, "%s: d_model and d_ffn must be multiples of 64, d_model at most 8192", name);
    throw Fail{ATSPEED_E_SHAPE};
  }
  if (!md->embed || !md->final_norm || !md->lm_head || !md->attn_norm || !md->wqkv || !md->wo || !md->mlp_norm ||
      !md->wgate_up || !md->wdown) {
    set_err(c, "%s: null weight pointer", name);
    throw Fail{ATSPEED_E_ARG};
  }
  m.present = true;
  m.layers = md->n_layers;
  m.d = md->d_model;
  m.H = md->n_heads;
  m.hd = hd;
  m.ffn = md->d_ffn;
  m.V = md->vocab;
  m.eps = md->rms_eps;
  m.theta = md->rope_theta;
  m.embed = (const bf16*)md->embed;
  m.final_norm = (const bf16*)md->final_norm;
  m.lm_head = (const bf16*)md->lm_head;
  for (int l = 0; l < m.layers; ++l) {
    if (!md->attn_norm[l] || !md->wqkv[l] || !md->wo[l] || !md->mlp_norm[l] || !md->wgate_up[l] || !md->wdown[l]) {
      set_err(c, "%s: null weight pointer in layer %d", name, l);
      throw Fail{ATSPEED_E_ARG};
    }
    m.attn_norm.push_back((const bf16*)md->attn_norm[l]);
    m.wqkv.push_back((const bf16*)md->wqkv[l]);
    m.wo.push_back((const bf16*)md->wo[l]);
    m.mlp_norm.push_back((const bf16*)md->mlp_norm[l]);
    m.wgate_up.push_back((const bf16*)md->wgate_up[l]);
    m.wdown.push_back((const bf16*)md->wdown[l]);
  }
}

void alloc_model(atspeed_ctx* c, ModelRt& m) {
  if (!m.present) return;
  const atspeed_limits& L = c->lim;
  const int stride = L.max_K + L.max_gamma * L.max_N;
  m.rows = L.max_users * (c->prefix_pages_per_user * ATT_PAGE + c->node_rows_per_user);
  const size_t per = (size_t)m.rows * m.d;
  m.kc = dalloc<bf16>(c, per * m.layers);
  m.vc = dalloc<__half>(c, per * m.layers);
  m.mk.resize(m.layers);
  m.mv.resize(m.layers);
  {
  char eb[256];
  for (int l = 0; l < m.layers; ++l)
    if (!attn_make_maps(m.kc + per * l, m.vc + per * l, m.rows, m.d, m.hd, &m.mk[l], &m.mv[l], eb, sizeof eb)) {
      set_err(c, "%s", eb);
      throw Fail{ATSPEED_E_CUDA};
    }
  }
  // rotary tables, computed in double precision
  m.max_pos = L.max_prompt + TREE_L + 1;
  const int half = m.hd / 2;
  std::vector<float> hc((size_t)m.max_pos * half), hs((size_t)m.max_pos * half);
  for (int p = 0; p < m.max_pos; ++p)
    for (int i = 0; i < half; ++i) {
      const double ang = (double)p * std::pow((double)m.theta, -2.0 * i / m.hd);
      hc[(size_t)p * half + i] = (float)std::cos(ang);
      hs[(size_t)p * half + i] = (float)std::sin(ang);
    }
  m.rope_cos = dalloc<float>(c, hc.size(), false);
  m.rope_sin = dalloc<float>(c, hs.size(), false);
  CK(cudaMemcpy(m.rope_cos, hc.data(), hc.size() * 4, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(m.rope_sin, hs.data(), hs.size() * 4, cudaMemcpyHostToDevice));
  // activations: the larger of a batched prefill and a full tree
  m.Tcap = std::max(L.max_users * L.max_prompt, L.max_users * stride);
  m.Xrows = ((m.Tcap + 255) / 256) * 256;
  m.h = dalloc<float>(c, (size_t)m.Tcap * m.d);
  m.ssq = dalloc<float>(c, (size_t)((m.d + 127) / 128) * m.Tcap);
  m.x = dalloc<bf16>(c, (size_t)m.Xrows * m.d);
  m.q = dalloc<bf16>(c, (size_t)m.Tcap * m.d);
  m.att = dalloc<bf16>(c, (size_t)m.Xrows * m.d);
  m.act = dalloc<bf16>(c, (size_t)m.Xrows * m.ffn);
  m.logit_rows = L.max_users + L.max_users * stride;
  m.logits = dalloc<float>(c, (size_t)m.logit_rows * ITEM_ROWS);
  m.lse = dalloc<float>(c, m.logit_rows);
  m.lse_ld = m.Tcap;
  m.lse_part = dalloc<float2>(c, (size_t)((m.V + 127) / 128) * m.lse_ld, false);
  m.root_rows = ((L.max_users + 255) / 256) * 256;
  m.root_x = dalloc<bf16>(c, (size_t)m.root_rows * m.d);
  m.tok = dalloc<int>(c, m.Tcap);
  m.pos = dalloc<int>(c, m.Tcap);
  m.kvrow = dalloc<int>(c, m.Tcap);
  m.tuser = dalloc<int>(c, m.Tcap);
  m.tvis = dalloc<int>(c, m.Tcap);
  m.anc = dalloc<int>(c, (size_t)m.Tcap * 4);
  m.ancn = dalloc<int>(c, m.Tcap);
  const int max_qt = m.Tcap / ATT_QTILE + L.max_users + 1;
  char eb[256];
  m.plan_blk = dalloc<int>(c, 4 * (size_t)max_qt + L.max_users + m.Tcap);   // carved per forward
  const int pages = c->prefix_pages_per_user;
  {
    // the grid the model's forward will run on (as set with the schedule) and its split size
    const int grid = std::max(1, std::min(gemm_grid_size(c->device), 2 * m.ffn / 128));
    m.cps = attention_pages_per_split(L, m.H, grid);
  }
  m.max_splits = std::max(1, (pages + m.cps - 1) / m.cps);
  const int Ttree = std::max(L.max_users * stride, m.Tcap);
  m.part_o = dalloc<float>(c, (size_t)m.max_splits * Ttree * m.d, false);
  m.part_ml = dalloc<float>(c, (size_t)m.max_splits * Ttree * m.H * 2, false);
  m.max_qt = max_qt;   // (the attention arrival counters live in the ctx's per-forward zero block)
  // tensor maps of the persistent forward
  const int nmaps = fwd_map_count(m.layers);
  std::vector<CUtensorMap> hm(nmaps);
  for (int l = 0; l < m.layers; ++l) {
    const bool ok = gemm_make_map(&hm[l * 4 + 0], m.wqkv[l], m.d, 3 * m.d, 64, eb, sizeof eb) &&
                    gemm_make_map(&hm[l * 4 + 1], m.wo[l], m.d, m.d, 64, eb, sizeof eb) &&
                    gemm_make_map(&hm[l * 4 + 2], m.wgate_up[l], m.d, 2 * m.ffn, 64, eb, sizeof eb) &&
                    gemm_make_map(&hm[l * 4 + 3], m.wdown[l], m.ffn, m.d, 64, eb, sizeof eb);
    if (!ok) {
      set_err(c, "%s", eb);
      throw Fail{ATSPEED_E_CUDA};
    }
    hm[4 * m.layers + 2 * l] = m.mk[l];
    hm[4 * m.layers + 2 * l + 1] = m.mv[l];
  }
  const int L6 = 6 * m.layers;
  bool ok = gemm_make_map(&hm[L6], m.lm_head + (size_t)c->code_base * m.d, m.d, ITEM_ROWS, 64, eb, sizeof eb);
  for (int v = 0; v < 2 && ok; ++v) {
    const int bn = v == 0 ? 128 : 256;
    ok = gemm_make_map(&hm[L6 + 1 + 3 * v], m.x, m.d, m.Xrows, bn, eb, sizeof eb) &&
         gemm_make_map(&hm[L6 + 2 + 3 * v], m.att, m.d, m.Xrows, bn, eb, sizeof eb) &&
         gemm_make_map(&hm[L6 + 3 + 3 * v], m.act, m.ffn, m.Xrows, bn, eb, sizeof eb);
  }
  if (!ok) {
    set_err(c, "%s", eb);
    throw Fail{ATSPEED_E_CUDA};
  }
  m.maps = dalloc<CUtensorMap>(c, nmaps, false);
  CK(cudaMemcpy(m.maps, hm.data(), nmaps * sizeof(CUtensorMap), cudaMemcpyHostToDevice));
  m.d_attn_norm = dalloc<const bf16*>(c, m.layers, false);
  m.d_mlp_norm = dalloc<const bf16*>(c, m.layers, false);
  CK(cudaMemcpy(m.d_attn_norm, m.attn_norm.data(), m.layers * sizeof(void*), cudaMemcpyHostToDevice));
  CK(cudaMemcpy(m.d_mlp_norm, m.mlp_norm.data(), m.layers * sizeof(void*), cudaMemcpyHostToDevice));
}

void build_trie(atspeed_ctx* c, const atspeed_items_desc* it) {
  std::vector<uint32_t> keys(it->n_items);
  for (int i = 0; i < it->n_items; ++i) {
    uint32_t k = 0;
    for (int l = 0; l < 4; ++l) {
      const int code = it->h_codes[(size_t)i * 4 + l];
      if (code < 0 || code >= 256) {
        set_err(c, "item %d has code %d outside [0, 256)", i, code);
        throw Fail{ATSPEED_E_ARG};
      }
      k = (k << 8) | (uint32_t)code;
    }
    keys[i] = k;
  }
  std::sort(keys.begin(), keys.end());
  keys.erase(std::unique(keys.begin(), keys.end()), keys.end());
  // prefixes per level in lexicographic order; ids assigned level by level
  std::vector<std::vector<uint32_t>> pref(5);
  for (int l = 0; l <= 4; ++l) {
    for (uint32_t k : keys) {
      const uint32_t p = l == 0 ? 0u : (k >> (8 * (4 - l)));
      if (pref[l].empty() || pref[l].back() != p) pref[l].push_back(p);
    }
  }
  std::vector<int> off(5, 0);
  for (int l = 1; l <= 4; ++l) off[l] = off[l - 1] + (int)pref[l - 1].size();
  const int n_nodes = off[4];  // levels 0..3 carry masks
  c->h_mask.assign((size_t)n_nodes * 8, 0u);
  c->h_child.assign(n_nodes, 0);
  for (int l = 0; l < 4; ++l) {
    size_t j = 0;  // index into pref[l+1]
    for (size_t i = 0; i < pref[l].size(); ++i) {
      const int node = off[l] + (int)i;
      const uint32_t p = pref[l][i];
      while (j < pref[l + 1].size() && (pref[l + 1][j] >> 8) < p) ++j;
      c->h_child[node] = (l + 1 < 4 ? off[l + 1] : off[4]) + (int)j;
      size_t jj = j;
      while (jj < pref[l + 1].size() && (pref[l + 1][jj] >> 8) == p) {
        const uint32_t code = pref[l + 1][jj] & 255u;
        c->h_mask[(size_t)node * 8 + code / 32] |= 1u << (code % 32);
        ++jj;
      }
      j = jj;
    }
  }
  c->trie_mask = dalloc<uint32_t>(c, c->h_mask.size(), false);
  c->trie_child = dalloc<int>(c, c->h_child.size(), false);
  CK(cudaMemcpy(c->trie_mask, c->h_mask.data(), c->h_mask.size() * 4, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(c->trie_child, c->h_child.data(), c->h_child.size() * 4, cudaMemcpyHostToDevice));
}

int host_trie_child(const atspeed_ctx* c, int x, int code) {
  const uint32_t* m = &c->h_mask[(size_t)x * 8];
  int r = 0;
  for (int w = 0; w < code / 32; ++w) r += __builtin_popcount(m[w]);
  r += __builtin_popcount(m[code / 32] & ((1u << (code % 32)) - 1u));
  return c->h_child[x] + r;
}
bool host_trie_has(const atspeed_ctx* c, int x, int code) {
  return (c->h_mask[(size_t)x * 8 + code / 32] >> (code % 32)) & 1u;
}

TreeDev tree_dev(atspeed_ctx* c) {
  TreeDev t;
  t.B = c->B;
  t.slots_in = c->step_K;
  t.slots_lvl = c->step_N;
  t.max_levels = c->step_gamma;
  t.stride = c->step_K + c->step_gamma * c->step_N;
  t.d = c->u_d;
  t.g = c->u_g;
  t.sd_step = c->u_step;
  t.cnt = c->n_cnt;
  t.code = c->n_code;
  t.prank = c->n_prank;
  t.trie = c->n_trie;
  t.path = c->n_path;
  t.sq = c->n_sq;
  t.sp = c->n_sp;
  t.row_t = c->n_row_t;
  t.row_d = c->n_row_d;
  t.anc_t = c->n_anc_t;
  t.anc_d = c->n_anc_d;
  t.lg_t = c->n_lg_t;
  t.lg_d = c->n_lg_d;
  t.trie_mask = c->trie_mask;
  t.trie_child = c->trie_child;
  t.logits_t = c->tgt.logits;
  t.logits_d = c->drf.present ? c->drf.logits : c->tgt.logits;
  t.lse_t = c->full_norm ? c->tgt.lse : nullptr;
  t.lse_d = c->full_norm ? (c->drf.present ? c->drf.lse : c->tgt.lse) : nullptr;
  return t;
}

int prefix_row(const atspeed_ctx* c, int u, int p) { return u * c->prefix_pages_per_user * ATT_PAGE + p; }
int node_row(const atspeed_ctx* c, int u, int step, int slot, int stride) {
  return c->lim.max_users * c->prefix_pages_per_user * ATT_PAGE + u * c->node_rows_per_user + step * stride + slot;
}

// ---------------------------------------------------------------------------------------------
// the decoder forward
// ---------------------------------------------------------------------------------------------
struct FwdPlan {
  int T = 0;
  bool prefill = false;
  const int* d_tokens = nullptr;       // prefill: caller's tokens; tree: m.tok (filled by gather)
  std::vector<int> qt_t0, qt_n, qt_user, qt_vis;   // qt_vis: longest visible prefix in the tile
  std::vector<int> splits;             // per user
  std::vector<int> out_rows;           // tokens whose logits are produced, in order
  int logit_row_base = 0;
};

cudaEvent_t prof_event(atspeed_ctx* c) {
  if (!c->prof_pool.empty()) {
    cudaEvent_t e = c->prof_pool.back();
    c->prof_pool.pop_back();
    return e;
  }
  cudaEvent_t e;
  CK(cudaEventCreate(&e));
  return e;
}

// Brackets one kernel launch with events when profiling is on.
struct ProfScope {
  atspeed_ctx* c;
  cudaStream_t st;
  atspeed_ctx::ProfRec r;
  ProfScope(atspeed_ctx* c_, cudaStream_t st_, int kind, double bytes, double flops) : c(c_), st(st_) {
    if (!c->prof) return;
    r.kind = kind;
    r.bytes = bytes;
    r.flops = flops;
    r.a = prof_event(c);
    r.b = prof_event(c);
    CK(cudaEventRecord(r.a, st));
  }
  void done() {
    if (!c->prof) return;
    CK(cudaEventRecord(r.b, st));
    c->prof_recs.push_back(r);
  }
};

void gemm(atspeed_ctx* c, const GemmArgs& a, cudaStream_t st, int kind, int grid) {
  char eb[256] = {0};
  // algorithmic bytes: weights once, activations in, outputs out
  const double out_b = a.epi == EPI_F32 ? 4.0 * a.M : a.epi == EPI_RESID ? 8.0 * a.M
                       : a.epi == EPI_RESNORM ? (a.gain ? 10.0 * a.M : 8.0 * a.M)
                       : a.epi == EPI_SWIGLU ? 1.0 * a.M : 2.0 * a.M;
  ProfScope ps(c, st, kind, 2.0 * a.M * a.K + 2.0 * a.T * a.K + out_b * a.T, 2.0 * a.M * a.K * a.T);
  cudaError_t e = gemm_launch(a, c->gs, grid, st, c->pdl && !c->prof, eb, sizeof eb);
  c->n_launch += 1;
  if (e != cudaSuccess) {
    set_err(c, "gemm launch failed: %s %s", cudaGetErrorString(e), eb);
    throw Fail{ATSPEED_E_CUDA};
  }
  ps.done();
}

void forward(atspeed_ctx* c, ModelRt& m, const FwdPlan& p, cudaStream_t st) {
  const int T = p.T;
  if (T <= 0) return;
  if (T > m.Tcap) {
    set_err(c, "forward of %d tokens exceeds capacity %d", T, m.Tcap);
    throw Fail{ATSPEED_E_SHAPE};
  }
  const int nqt = (int)p.qt_t0.size();
  if (nqt > m.max_qt || (int)p.splits.size() > c->lim.max_users || (int)p.out_rows.size() > m.Tcap) {
    set_err(c, "forward plan exceeds capacity (%d query tiles, %zu users, %zu rows)", nqt, p.splits.size(),
            p.out_rows.size());
    throw Fail{ATSPEED_E_SHAPE};
  }
  {
    // the plan's tables, packed: one upload into the model's plan block
    const size_t ns = p.splits.size(), nr = p.out_rows.size(), tot = 4 * (size_t)nqt + ns + nr;
    int* h = stage_alloc<int>(c, st, tot);
    int* q = h;
    for (const std::vector<int>* v : {&p.qt_t0, &p.qt_n, &p.qt_user, &p.qt_vis, &p.splits, &p.out_rows}) {
      memcpy(q, v->data(), v->size() * sizeof(int));
      q += v->size();
    }
    m.qt_t0 = m.plan_blk;
    m.qt_n = m.qt_t0 + nqt;
    m.qt_user = m.qt_n + nqt;
    m.qt_vis = m.qt_user + nqt;
    m.user_splits = m.qt_vis + nqt;
    m.rows_sel = m.user_splits + ns;
    CK(cudaMemcpyAsync(m.plan_blk, h, tot * sizeof(int), cudaMemcpyHostToDevice, st));
  }
  int max_split = 1;
  for (int s : p.splits) max_split = std::max(max_split, s);
  const size_t per = (size_t)m.rows * m.d;
  const bool pdl = c->pdl;
  if (!m.per_op) {
    // the whole forward in one persistent cooperative launch
    if (nqt > m.max_qt) {
      set_err(c, "forward needs %d query tiles (capacity %d)", nqt, m.max_qt);
      throw Fail{ATSPEED_E_SHAPE};
    }
    FwdParams f = {};
    f.T = T;
    f.n_out = (int)p.out_rows.size();
    f.d = m.d;
    f.H = m.H;
    f.hd = m.hd;
    f.ffn = m.ffn;
    f.L = m.layers;
    f.eps = m.eps;
    f.G = m.grid;
    f.maps = m.maps;
    f.attn_norm = m.d_attn_norm;
    f.mlp_norm = m.d_mlp_norm;
    f.final_norm = m.final_norm;
    f.embed = m.embed;
    f.h = m.h;
    f.ssq = m.ssq;
    f.ssq_ld = m.Tcap;
    f.x = m.x;
    f.q = m.q;
    f.att = m.att;
    f.act = m.act;
    f.logits = m.logits + (size_t)p.logit_row_base * ITEM_ROWS;
    f.kc = m.kc;
    f.vc = m.vc;
    f.layer_elems = per;
    f.tok = p.d_tokens;
    f.pos = m.pos;
    f.kv_row = m.kvrow;
    f.out_rows = m.rows_sel;
    f.rope_cos = m.rope_cos;
    f.rope_sin = m.rope_sin;
    AttnArgs& a = f.att_args;
    a.T = T;
    a.n_heads = m.H;
    a.head_dim = m.hd;
    a.q = m.q;
    a.kv_rows = m.rows;
    a.n_qtiles = nqt;
    a.qt_t0 = m.qt_t0;
    a.qt_n = m.qt_n;
    a.qt_user = m.qt_user;
    a.qt_vis = m.qt_vis;
    a.tok_user = m.tuser;
    a.tok_vis = m.tvis;
    a.anc_row = p.prefill ? nullptr : m.anc;
    a.anc_n = p.prefill ? nullptr : m.ancn;
    a.page_table = c->page_table;
    a.max_pages = c->prefix_pages_per_user;
    a.user_splits = m.user_splits;
    a.chunks_per_split = p.prefill ? 0 : m.cps;
    a.max_splits = max_split;
    a.out = m.att;
    a.part_o = m.part_o;
    a.part_ml = m.part_ml;
    a.direct = p.prefill;
    a.err = c->err_word;
    f.att_items = nqt * m.H * max_split;
    f.att_counters = m.att_counters;
    f.ws = c->gs.ws;
    f.counters = c->gs.counters;
    f.sk_counters = c->fwd_sk;
    f.bar = c->fwd_bar;
    f.err = c->err_word;
    f.trace = c->fwd_trace;
    CK(cudaMemsetAsync(c->fwd_zero, 0, (c->fwd_zero_att + (size_t)nqt * m.H) * sizeof(int), st));
    if (c->fwd_trace) CK(cudaMemsetAsync(c->fwd_trace, 0, c->fwd_trace_n * sizeof(unsigned long long), st));
    const double wbytes = 2.0 * m.layers * (4.0 * m.d * m.d + 3.0 * m.d * m.ffn) + 2.0 * ITEM_ROWS * m.d;
    ProfScope ps(c, st, 6, wbytes, 2.0 * T * (wbytes / 2.0));
    CK(fwd_launch(f, st));
    ps.done();
    c->n_launch += 1;
    return;
  }
  // RMSNorm folded into the GEMMs: the O / down epilogues leave h, bf16(g * h) and per-tile sums of
  // squares; the QKV / gate-up epilogues apply each token's 1 / rms
  CK(embed_rows_launch(p.d_tokens, m.embed, m.attn_norm[0], m.h, m.x, m.ssq, m.Tcap, T, m.d, st, pdl));
  c->n_launch += 1;
  auto folded = [&](GemmArgs& g) {
    g.ssq_ld = m.Tcap;
    g.nrm_d = m.d;
    g.eps = m.eps;
  };
  for (int l = 0; l < m.layers; ++l) {
    GemmArgs g = {};
    folded(g);
    g.ssq_in = m.ssq;
    g.epi = EPI_QKV;
    g.W = m.wqkv[l];
    g.X = m.x;
    g.M = 3 * m.d;
    g.K = m.d;
    g.T = T;
    g.X_rows = m.Xrows;
    g.d_model = m.d;
    g.head_dim = m.hd;
    g.pos = m.pos;
    g.kv_row = m.kvrow;
    g.rope_cos = m.rope_cos;
    g.rope_sin = m.rope_sin;
    g.q_out = m.q;
    g.k_cache = m.kc + per * l;
    g.v_cache = m.vc + per * l;
    gemm(c, g, st, 0, m.grid);
    AttnArgs a = {};
    a.T = T;
    a.n_heads = m.H;
    a.head_dim = m.hd;
    a.q = m.q;
    a.k_cache = m.kc + per * l;
    a.v_cache = m.vc + per * l;
    a.kv_rows = m.rows;
    a.n_qtiles = nqt;
    a.qt_t0 = m.qt_t0;
    a.qt_n = m.qt_n;
    a.qt_user = m.qt_user;
    a.qt_vis = m.qt_vis;
    a.tok_user = m.tuser;
    a.tok_vis = m.tvis;
    a.anc_row = p.prefill ? nullptr : m.anc;
    a.anc_n = p.prefill ? nullptr : m.ancn;
    a.page_table = c->page_table;
    a.max_pages = c->prefix_pages_per_user;
    a.user_splits = m.user_splits;
    a.chunks_per_split = p.prefill ? 0 : m.cps;
    a.max_splits = max_split;
    a.out = m.att;
    a.part_o = m.part_o;
    a.part_ml = m.part_ml;
    a.direct = p.prefill;
    a.err = c->err_word;
    {
      ProfScope ps(c, st, 5, 0.0, 0.0);
      CK(attn_launch(a, m.mk[l], m.mv[l], st, pdl && !c->prof));
      c->n_launch += a.direct ? 1 : 2;
      ps.done();
    }
    g = GemmArgs{};
    folded(g);
    g.epi = EPI_RESNORM;
    g.gain = m.mlp_norm[l];
    g.xg_out = m.x;
    g.ssq_out = m.ssq;
    g.W = m.wo[l];
    g.X = m.att;
    g.M = m.d;
    g.K = m.d;
    g.T = T;
    g.X_rows = m.Xrows;
    g.out_f32 = m.h;
    g.ldo = m.d;
    gemm(c, g, st, 1, m.grid);
    g = GemmArgs{};
    folded(g);
    g.ssq_in = m.ssq;
    g.epi = EPI_SWIGLU;
    g.W = m.wgate_up[l];
    g.X = m.x;
    g.M = 2 * m.ffn;
    g.K = m.d;
    g.T = T;
    g.X_rows = m.Xrows;
    g.out_bf16 = m.act;
    g.ldo = m.ffn;
    gemm(c, g, st, 2, m.grid);
    g = GemmArgs{};
    folded(g);
    g.epi = EPI_RESNORM;
    if (l + 1 < m.layers) {   // (the final norm normalises the selected rows from h itself)
      g.gain = m.attn_norm[l + 1];
      g.xg_out = m.x;
      g.ssq_out = m.ssq;
    }
    g.W = m.wdown[l];
    g.X = m.act;
    g.M = m.d;
    g.K = m.ffn;
    g.T = T;
    g.X_rows = m.Xrows;
    g.out_f32 = m.h;
    g.ldo = m.d;
    gemm(c, g, st, 3, m.grid);
  }
  const int n_out = (int)p.out_rows.size();
  CK(rmsnorm_rows_launch(m.h, m.rows_sel, n_out, m.final_norm, m.d, m.eps, m.x, m.d, st, pdl));
  c->n_launch += 1;
  GemmArgs g = {};
  g.epi = EPI_F32;
  g.W = m.lm_head + (size_t)c->code_base * m.d;
  g.X = m.x;
  g.M = ITEM_ROWS;
  g.K = m.d;
  g.T = n_out;
  g.X_rows = m.Xrows;
  g.out_f32 = m.logits + (size_t)p.logit_row_base * ITEM_ROWS;
  g.ldo = ITEM_ROWS;
  gemm(c, g, st, 4, m.grid);
}

// FULL normalisation (whole-vocabulary log-softmax, then the trie mask): log-sum-exp over the whole
// vocabulary of the n final-norm rows X[0 .. n) (bf16, X_rows allocated) into lse_out[0 .. n): the
// LM head over all V rows with the EPI_LSE epilogue, then the combine of its per-tile partials.
void full_lse(atspeed_ctx* c, ModelRt& m, const bf16* X, int X_rows, int n, float* lse_out, cudaStream_t st) {
  if (n <= 0) return;
  if (n > m.lse_ld) {
    set_err(c, "FULL normalisation of %d rows exceeds the partials buffer (%d)", n, m.lse_ld);
    throw Fail{ATSPEED_E_SHAPE};
  }
  GemmArgs g = {};
  g.epi = EPI_LSE;
  g.W = m.lm_head;
  g.X = X;
  g.M = m.V;
  g.K = m.d;
  g.T = n;
  g.X_rows = X_rows;
  g.lse_part = m.lse_part;
  g.lse_ld = m.lse_ld;
  gemm(c, g, st, 4, m.grid);
  CK(lse_combine_launch(m.lse_part, m.lse_ld, (m.V + 127) / 128, n, lse_out, st));
  c->n_launch += 1;
}

// Query tiles of user u's n consecutive tokens from t0.  vis = the history length every token sees
// (tree nodes), or -1 for the history itself (token i sees i + 1 tokens).
void add_qtiles(FwdPlan& p, int u, int t0, int n, int vis) {
  for (int i = 0; i < n; i += ATT_QTILE) {
    const int cnt = std::min(ATT_QTILE, n - i);
    p.qt_t0.push_back(t0 + i);
    p.qt_n.push_back(cnt);
    p.qt_user.push_back(u);
    p.qt_vis.push_back(vis < 0 ? i + cnt : vis);
  }
}

int splits_for(int P, int cps) {
  const int pages = (P + ATT_PAGE - 1) / ATT_PAGE;
  return std::max(1, (pages + cps - 1) / cps);
}

// Forward of the given node slots of the current step through model m (target or draft).
void forward_nodes(atspeed_ctx* c, ModelRt& m, bool target, const std::vector<int>& nodes, int row_base,
                   cudaStream_t st) {
  if (nodes.empty()) return;
  const int T = (int)nodes.size();
  const TreeDev t = tree_dev(c);
  upload(c, st, c->fwd_nodes, nodes.data(), (size_t)T * 4);
  FwdTokens f{m.tok, m.pos, m.kvrow, m.tuser, m.tvis, m.anc, m.ancn};
  CK(tree_gather_launch(t, c->fwd_nodes, T, c->u_P, c->code_base, target, row_base, f, st, c->pdl));
  c->n_launch += 1;
  FwdPlan p;
  p.T = T;
  p.prefill = false;
  p.d_tokens = m.tok;
  // tokens are grouped by user (nodes sorted by user)
  int i = 0;
  while (i < T) {
    const int u = nodes[i] / t.stride;
    int j = i;
    while (j < T && nodes[j] / t.stride == u) ++j;
    add_qtiles(p, u, i, j - i, c->users[u].P);
    i = j;
  }
  p.splits.resize(c->B);
  for (int u = 0; u < c->B; ++u) p.splits[u] = splits_for(c->users[u].P, m.cps);
  p.out_rows.resize(T);
  for (int k = 0; k < T; ++k) p.out_rows[k] = k;
  p.logit_row_base = row_base;
  forward(c, m, p, st);
  if (c->full_norm) full_lse(c, m, m.x, m.Xrows, T, m.lse + row_base, st);
}

// ---------------------------------------------------------------------------------------------
// speculative-step bookkeeping
// ---------------------------------------------------------------------------------------------
void upload_users(atspeed_ctx* c, cudaStream_t st) {
  const int mu = c->lim.max_users;
  int* h = stage_alloc<int>(c, st, 4 * (size_t)mu);
  for (int u = 0; u < c->B; ++u) {
    const UserState& us = c->users[u];
    h[u] = us.active ? us.d : TREE_L;
    h[mu + u] = us.active ? us.g : 0;
    h[2 * mu + u] = us.step;
    h[3 * mu + u] = us.P;
  }
  CK(cudaMemcpyAsync(c->u_blk, h, 4 * (size_t)mu * sizeof(int), cudaMemcpyHostToDevice, st));
}

// Writes level 0 (incoming beams) and the own-row assignment of every slot of the new step.
void open_step(atspeed_ctx* c, const atspeed_decode_opts* o, cudaStream_t st) {
  const int K = o->K, N = o->N, G = o->gamma;
  c->step_K = K;
  c->step_N = N;
  c->step_gamma = G;
  const int stride = K + G * N;
  const size_t n = (size_t)c->B * stride;
  // the node table of this step: n slots in consecutive sections, filled in the staging buffer and
  // uploaded at once
  const size_t ncnt = (size_t)c->B * (G + 1);
  carve_nodes(c, n, c->B, G);
  int* h = stage_alloc<int>(c, st, NODE_INTS * n + ncnt);
  int* code = h;
  int* prank = code + n;
  int* trie = prank + n;
  int* path = trie + n;
  int* rt = path + 4 * n;
  int* rd = rt + n;
  int* at = rd + n;
  int* ad = at + 4 * n;
  int* lgt = ad + 4 * n;
  int* lgd = lgt + n;
  float* sq = reinterpret_cast<float*>(lgd + n);
  float* sp = sq + n;
  int* cnt = reinterpret_cast<int*>(sp + n);
  std::fill(code, code + 3 * n, -1);           // code, prank: -1
  std::fill(trie, trie + n, 0);
  std::fill(path, path + 4 * n, -1);
  std::fill(at, at + 8 * n, 0);                // at, ad
  std::fill(lgt, lgt + 2 * n, -1);             // lg_t, lg_d
  std::fill(sq, sq + 2 * n, -INFINITY);        // sq, sp
  std::fill(cnt, cnt + ncnt, 0);
  for (int u = 0; u < c->B; ++u) {
    UserState& us = c->users[u];
    us.g = us.active ? std::min(G, TREE_L - us.d) : 0;
    for (int k = 0; k < stride; ++k) {
      const size_t nd = (size_t)u * stride + k;
      rt[nd] = node_row(c, u, us.region, k, stride);
      rd[nd] = rt[nd];
    }
    if (!us.active) continue;
    const int nin = (int)us.path.size();
    cnt[(size_t)u * (G + 1)] = nin;
    for (int k = 0; k < nin && k < K; ++k) {
      const size_t nd = (size_t)u * stride + k;
      code[nd] = us.d > 0 ? us.path[k][us.d - 1] : -1;
      trie[nd] = us.trie[k];
      for (int i = 0; i < 4; ++i) path[nd * 4 + i] = us.path[k][i];
      sp[nd] = us.sp[k];
      sq[nd] = us.sp[k];
      for (int i = 0; i < 4; ++i) {
        at[nd * 4 + i] = us.anc_t[k][i];
        ad[nd * 4 + i] = us.anc_d[k][i];
      }
      if (us.d > 0) {
        at[nd * 4 + us.d - 1] = rt[nd];
        ad[nd * 4 + us.d - 1] = rd[nd];
      } else {
        lgt[nd] = u;  // prefill logits row of the user
        lgd[nd] = u;
      }
    }
  }
  CK(cudaMemcpyAsync(c->n_blk, h, (NODE_INTS * n + ncnt) * sizeof(int), cudaMemcpyHostToDevice, st));
  c->full_norm = o->norm == ATSPEED_NORM_FULL;
  if (c->full_norm) {
    // level 0 of users at depth 0 scores with the prefill's logits rows 0 .. B-1
    bool fresh = false;
    for (int u = 0; u < c->B; ++u) fresh |= c->users[u].active && c->users[u].d == 0;
    if (fresh)
      for (ModelRt* m : {&c->tgt, &c->drf})
        if (m->present) full_lse(c, *m, m->root_x, m->root_rows, c->B, m->lse, st);
  }
  upload_users(c, st);
  c->step_open = true;
  c->have_tree = true;
  c->levels_done = 0;
  c->roots_drafted = false;
  c->level_fwd_pending = false;
  c->tree_injected = false;
}

void check_opts(atspeed_ctx* c, const atspeed_decode_opts* o) {
  if (!o) {
    set_err(c, "null decode options");
    throw Fail{ATSPEED_E_ARG};
  }
  if (o->K < 1 || o->K > c->lim.max_K || o->N < 1 || o->N > c->lim.max_N || o->gamma < 0 ||
      o->gamma > c->lim.max_gamma) {
    set_err(c, "decode options K=%d N=%d gamma=%d outside limits (max_K=%d max_N=%d max_gamma=%d)", o->K, o->N,
            o->gamma, c->lim.max_K, c->lim.max_N, c->lim.max_gamma);
    throw Fail{ATSPEED_E_SHAPE};
  }
  if (o->norm != ATSPEED_NORM_MASKED && o->norm != ATSPEED_NORM_FULL) {
    set_err(c, "unknown normalisation mode %d", (int)o->norm);
    throw Fail{ATSPEED_E_ARG};
  }
}

void ensure_step(atspeed_ctx* c, const atspeed_decode_opts* o, cudaStream_t st) {
  if (!c->prefilled) {
    set_err(c, "prefill must come first");
    throw Fail{ATSPEED_E_STATE};
  }
  if (c->step_open && (o->norm == ATSPEED_NORM_FULL) != c->full_norm) {
    set_err(c, "the normalisation mode cannot change within a speculative step");
    throw Fail{ATSPEED_E_STATE};
  }
  if (!c->step_open) open_step(c, o, st);
  if (o->K != c->step_K || o->N != c->step_N || o->gamma != c->step_gamma) {
    set_err(c, "decode options changed inside a speculative step");
    throw Fail{ATSPEED_E_STATE};
  }
}

std::vector<int> level_nodes(atspeed_ctx* c, int lvl, bool need_forward_rule) {
  std::vector<int> v;
  const int stride = c->step_K + c->step_gamma * c->step_N;
  for (int u = 0; u < c->B; ++u) {
    const UserState& us = c->users[u];
    if (!us.active) continue;
    if (lvl == 0) {
      if (us.d == 0) continue;
      for (int k = 0; k < c->step_K; ++k) v.push_back(u * stride + k);
    } else {
      if (lvl > us.g) continue;
      if (need_forward_rule && lvl > TREE_L - us.d - 1) continue;
      const int off = c->step_K + (lvl - 1) * c->step_N;
      for (int k = 0; k < c->step_N; ++k) v.push_back(u * stride + off + k);
    }
  }
  return v;
}

// Draft forward over the nodes of drafted level `lvl` (their logits draft level lvl + 1).
void draft_level_forward(atspeed_ctx* c, int lvl, cudaStream_t st) {
  std::vector<int> nodes = level_nodes(c, lvl, true);
  // rows of this level's draft logits follow the rows already used in this step
  int base = c->B + (int)level_nodes(c, 0, false).size();
  for (int j = 1; j < lvl; ++j) base += (int)level_nodes(c, j, true).size();
  forward_nodes(c, c->drf, false, nodes, base, st);
  c->level_fwd_pending = false;
}

// forward_level = false leaves the draft forward over the new level pending: the next draft_step
// or verify runs it, an early-rejected step never does.
void draft_step_impl(atspeed_ctx* c, cudaStream_t st, const atspeed_decode_opts* o, atspeed_verify_mode mode,
                     bool forward_level = true) {
  check_opts(c, o);
  if (!c->drf.present) {
    set_err(c, "no draft model in this context");
    throw Fail{ATSPEED_E_STATE};
  }
  ensure_step(c, o, st);
  if (c->tree_injected) {
    set_err(c, "the tree of this step was injected");
    throw Fail{ATSPEED_E_STATE};
  }
  if (c->level_fwd_pending) draft_level_forward(c, c->levels_done, st);
  // draft logits rows: users' prefill rows first, then one row per node slot
  if (!c->roots_drafted) {
    std::vector<int> roots = level_nodes(c, 0, false);
    forward_nodes(c, c->drf, false, roots, c->B, st);  // row = B + index, remapped below
    c->roots_drafted = true;
  }
  const int lvl = c->levels_done + 1;
  int maxg = 0;
  for (auto& us : c->users)
    if (us.active) maxg = std::max(maxg, us.g);
  if (lvl > maxg) return;  // every tree is complete
  const TreeDev t = tree_dev(c);
  CK(draft_level_launch(t, lvl, c->step_N, mode == ATSPEED_RELAXED, o->philox_seed, st, c->pdl));
  c->n_launch += 1;
  c->levels_done = lvl;
  if (forward_level)
    draft_level_forward(c, lvl, st);
  else
    c->level_fwd_pending = true;
}

void commit(atspeed_ctx* c, cudaStream_t st, bool count_stats, const std::vector<int>& T_user) {
  const int B = c->B, K = c->step_K;
  // every output section in one download (fixed section offsets: max_users, max_K)
  const int mu = c->lim.max_users;
  const size_t mk = (size_t)mu * c->lim.max_K, nblk = o_blk_ints(mu, c->lim.max_K);
  int* h = stage_alloc<int>(c, st, nblk);
  CK(cudaMemcpyAsync(h, c->o_blk, nblk * sizeof(int), cudaMemcpyDeviceToHost, st));
  check_device_error(c, st);   // synchronises; the download stays intact until the next staging
  const int* adv = h + mu;
  const int* acc = h;
  const int* nout = h + 2 * mu;
  const int* path = h + 4 * mu;
  const int* parent = path + 4 * mk;
  const int* trie = parent + mk;
  const float* score = reinterpret_cast<const float*>(trie + mk);
  const int* anc_t = reinterpret_cast<const int*>(score + mk);
  const int* anc_d = anc_t + 4 * mk;
  (void)parent;
  for (int u = 0; u < B; ++u) {
    UserState& us = c->users[u];
    if (!us.active) continue;
    const int nd = us.d + adv[u];
    us.path.assign(nout[u], {});
    us.sp.assign(nout[u], 0.f);
    us.trie.assign(nout[u], 0);
    us.anc_t.assign(nout[u], {});
    us.anc_d.assign(nout[u], {});
    for (int k = 0; k < nout[u]; ++k) {
      const size_t o = (size_t)u * K + k;
      for (int i = 0; i < 4; ++i) us.path[k][i] = path[o * 4 + i];
      us.sp[k] = score[o];
      us.trie[k] = trie[o];
      for (int i = 0; i < 4; ++i) {
        us.anc_t[k][i] = i < nd - 1 ? anc_t[o * 4 + i] : 0;
        us.anc_d[k][i] = i < nd - 1 ? anc_d[o * 4 + i] : 0;
      }
    }
    if (count_stats) {
      us.acc_steps += acc[u];
      us.calls += 1;
      us.tree_tokens += T_user[u];
    }
    us.d = nd;
    us.step += 1;
    us.region += 1;
    if (us.d >= TREE_L || nout[u] == 0) us.active = false;
  }
  c->step_open = false;
}

// Early rejection (opt-in, atspeed_set_early_reject).  At depth 0 the target logits of level 0 (the
// empty beam) are the prefill's, so whether drafted level 1 is accepted can be decided before any
// forward over the tree.  A user that rejects level 1 takes its K output beams from level 1's
// candidates (Alg. 1: the top-K of level 1; Alg. 2: A plus draws from the residual), which depend
// on those logits alone: when every active user rejects, the tree forward is skipped and the step
// ends with the same outputs as the full verification.
bool early_reject_eligible(const atspeed_ctx* c) {
  if (!c->early_reject || c->levels_done < 1) return false;
  bool any = false;
  for (const auto& us : c->users) {
    if (!us.active) continue;
    if (us.d != 0 || us.g < 1) return false;
    any = true;
  }
  return any;
}

// One probe launch of the verification kernel; true when every active user was decided at level 1
// (its outputs are then in the o_* buffers, ready for commit).
bool early_reject_probe(atspeed_ctx* c, cudaStream_t st, const atspeed_decode_opts* o, atspeed_verify_mode mode) {
  const TreeDev t = tree_dev(c);
  VerifyOut vo{c->o_acc, c->o_adv, c->o_n, c->o_nacc, c->o_path, c->o_score, c->o_parent, c->o_trie,
               c->o_anc_t, c->o_anc_d};
  CK(verify_launch(t, c->step_K, mode == ATSPEED_RELAXED, o->philox_seed, vo, st, c->pdl, true));
  c->n_launch += 1;
  int* acc = stage_alloc<int>(c, st, c->B);
  CK(cudaMemcpyAsync(acc, c->o_acc, c->B * 4, cudaMemcpyDeviceToHost, st));
  stage_sync(c, st);
  for (int u = 0; u < c->B; ++u)
    if (c->users[u].active && acc[u] < 0) return false;
  return true;
}

void verify_impl(atspeed_ctx* c, cudaStream_t st, const atspeed_decode_opts* o, atspeed_verify_mode mode,
                 bool allow_probe = true) {
  check_opts(c, o);
  ensure_step(c, o, st);
  if (allow_probe && early_reject_eligible(c) && early_reject_probe(c, st, o, mode)) {
    c->level_fwd_pending = false;
    commit(c, st, true, std::vector<int>(c->B, 0));
    return;
  }
  if (c->level_fwd_pending) draft_level_forward(c, c->levels_done, st);
  // target forward over the incoming beams (depth >= 1) and drafted levels 1 .. min(g, L-d-1)
  std::vector<int> nodes;
  std::vector<int> T_user(c->B, 0);
  const int stride = c->step_K + c->step_gamma * c->step_N;
  for (int lvl = 0; lvl <= c->step_gamma; ++lvl) {
    std::vector<int> v = level_nodes(c, lvl, true);
    nodes.insert(nodes.end(), v.begin(), v.end());
  }
  std::stable_sort(nodes.begin(), nodes.end(), [&](int a, int b) { return a / stride < b / stride; });
  for (int n : nodes) T_user[n / stride] += 1;
  // users that drafted fewer levels than gamma' verify only what they have
  for (int u = 0; u < c->B; ++u) {
    UserState& us = c->users[u];
    if (us.active && c->levels_done < us.g && !c->tree_injected) us.g = c->levels_done;
  }
  upload_users(c, st);
  // nodes beyond a user's (possibly reduced) g are not forwarded
  nodes.erase(std::remove_if(nodes.begin(), nodes.end(),
                             [&](int n) {
                               const int u = n / stride, slot = n % stride;
                               const int lvl = slot < c->step_K ? 0 : 1 + (slot - c->step_K) / c->step_N;
                               return lvl > c->users[u].g;
                             }),
              nodes.end());
  std::fill(T_user.begin(), T_user.end(), 0);
  for (int n : nodes) T_user[n / stride] += 1;
  forward_nodes(c, c->tgt, true, nodes, c->B, st);
  const TreeDev t = tree_dev(c);
  VerifyOut vo{c->o_acc, c->o_adv, c->o_n, c->o_nacc, c->o_path, c->o_score, c->o_parent, c->o_trie,
               c->o_anc_t, c->o_anc_d};
  CK(verify_launch(t, c->step_K, mode == ATSPEED_RELAXED, o->philox_seed, vo, st, c->pdl));
  c->n_launch += 1;
  commit(c, st, true, T_user);
}

void prefill_impl(atspeed_ctx* c, cudaStream_t st, int n_users, const int32_t* d_tokens, const int32_t* h_off) {
  if (n_users < 1 || n_users > c->lim.max_users || !d_tokens || !h_off) {
    set_err(c, "prefill: bad arguments (n_users=%d, max_users=%d)", n_users, c->lim.max_users);
    throw Fail{ATSPEED_E_ARG};
  }
  std::vector<int> P(n_users);
  for (int u = 0; u < n_users; ++u) {
    P[u] = h_off[u + 1] - h_off[u];
    if (P[u] < 1 || P[u] > c->lim.max_prompt) {
      set_err(c, "prefill: user %d has history length %d (limit %d)", u, P[u], c->lim.max_prompt);
      throw Fail{ATSPEED_E_SHAPE};
    }
  }
  c->B = n_users;
  c->users.assign(n_users, UserState{});
  const int T = h_off[n_users] - h_off[0];
  std::vector<int> pos(T), kvrow(T), tuser(T), tvis(T);
  FwdPlan p;
  p.T = T;
  p.prefill = true;
  p.d_tokens = d_tokens + h_off[0];
  p.splits.assign(n_users, 1);
  for (int u = 0; u < n_users; ++u) {
    const int t0 = h_off[u] - h_off[0];
    for (int i = 0; i < P[u]; ++i) {
      pos[t0 + i] = i;
      kvrow[t0 + i] = prefix_row(c, u, i);
      tuser[t0 + i] = u;
      tvis[t0 + i] = i + 1;
    }
    add_qtiles(p, u, t0, P[u], -1);
    p.out_rows.push_back(t0 + P[u] - 1);
    UserState& us = c->users[u];
    us.P = P[u];
    us.d = 0;
    us.step = 0;
    us.region = 0;
    us.active = true;
    us.path.assign(1, {-1, -1, -1, -1});
    us.sp.assign(1, 0.f);
    us.trie.assign(1, 0);
    us.anc_t.assign(1, {0, 0, 0, 0});
    us.anc_d.assign(1, {0, 0, 0, 0});
  }
  p.logit_row_base = 0;
  for (ModelRt* m : {&c->tgt, &c->drf}) {
    if (!m->present) continue;
    upload(c, st, m->pos, pos.data(), (size_t)T * 4);
    upload(c, st, m->kvrow, kvrow.data(), (size_t)T * 4);
    upload(c, st, m->tuser, tuser.data(), (size_t)T * 4);
    upload(c, st, m->tvis, tvis.data(), (size_t)T * 4);
    forward(c, *m, p, st);
    // the last history tokens' final-norm rows, for a FULL-normalised first step
    CK(cudaMemcpyAsync(m->root_x, m->x, (size_t)n_users * m->d * sizeof(bf16), cudaMemcpyDeviceToDevice, st));
  }
  upload(c, st, c->u_P, P.data(), (size_t)n_users * 4);
  stage_sync(c, st);
  c->prefilled = true;
  c->step_open = false;
}


// Writes caller-supplied item-code logits of node slots [off, off + width) of every active user into
// rows B + u * stride + slot of the model's logits buffer and points the nodes' logits rows there.
void inject_logits(atspeed_ctx* c, bool target, int off, int width, const float* h, size_t h_user_stride,
                   cudaStream_t st) {
  const int stride = c->step_K + c->step_gamma * c->step_N;
  ModelRt& m = (target || !c->drf.present) ? c->tgt : c->drf;
  int* lg = target ? c->n_lg_t : c->n_lg_d;
  const size_t n = (size_t)c->B * stride;
  std::vector<int> rows(n);
  stage_sync(c, st);
  CK(cudaMemcpy(rows.data(), lg, n * 4, cudaMemcpyDeviceToHost));
  for (int u = 0; u < c->B; ++u) {
    if (!c->users[u].active) continue;
    const int r0 = c->B + u * stride + off;
    CK(cudaMemcpy(m.logits + (size_t)r0 * ITEM_ROWS, h + (size_t)u * h_user_stride, (size_t)width * ITEM_ROWS * 4,
                  cudaMemcpyHostToDevice));
    for (int k = 0; k < width; ++k) rows[(size_t)u * stride + off + k] = r0 + k;
  }
  CK(cudaMemcpy(lg, rows.data(), n * 4, cudaMemcpyHostToDevice));
}

void draft_step_logits_impl(atspeed_ctx* c, cudaStream_t st, const atspeed_decode_opts* o, atspeed_verify_mode mode,
                            const float* h_logits) {
  check_opts(c, o);
  ensure_step(c, o, st);
  if (!h_logits) {
    set_err(c, "null logits");
    throw Fail{ATSPEED_E_ARG};
  }
  const int lvl = c->levels_done + 1;
  if (lvl > c->step_gamma) {
    set_err(c, "all gamma levels are drafted");
    throw Fail{ATSPEED_E_STATE};
  }
  const int off = lvl == 1 ? 0 : c->step_K + (lvl - 2) * c->step_N;
  const int width = lvl == 1 ? c->step_K : c->step_N;
  if (c->full_norm) {
    set_err(c, "injected logits carry no whole-vocabulary rows: FULL normalisation needs forwarded nodes");
    throw Fail{ATSPEED_E_STATE};
  }
  inject_logits(c, false, off, width, h_logits, (size_t)width * ITEM_ROWS, st);
  const TreeDev t = tree_dev(c);
  CK(draft_level_launch(t, lvl, c->step_N, mode == ATSPEED_RELAXED, o->philox_seed, st, c->pdl));
  c->levels_done = lvl;
  c->roots_drafted = true;
  stage_sync(c, st);
}

void verify_logits_impl(atspeed_ctx* c, cudaStream_t st, const atspeed_decode_opts* o, atspeed_verify_mode mode,
                        const float* h_logits) {
  check_opts(c, o);
  ensure_step(c, o, st);
  if (!h_logits) {
    set_err(c, "null logits");
    throw Fail{ATSPEED_E_ARG};
  }
  const int stride = c->step_K + c->step_gamma * c->step_N;
  for (int u = 0; u < c->B; ++u) {
    UserState& us = c->users[u];
    if (us.active && c->levels_done < us.g && !c->tree_injected) us.g = c->levels_done;
  }
  upload_users(c, st);
  if (c->full_norm) {
    set_err(c, "injected logits carry no whole-vocabulary rows: FULL normalisation needs forwarded nodes");
    throw Fail{ATSPEED_E_STATE};
  }
  inject_logits(c, true, 0, stride, h_logits, (size_t)stride * ITEM_ROWS, st);
  const TreeDev t = tree_dev(c);
  VerifyOut vo{c->o_acc, c->o_adv, c->o_n, c->o_nacc, c->o_path, c->o_score, c->o_parent, c->o_trie,
               c->o_anc_t, c->o_anc_d};
  CK(verify_launch(t, c->step_K, mode == ATSPEED_RELAXED, o->philox_seed, vo, st, c->pdl));
  commit(c, st, true, std::vector<int>(c->B, 0));
}

template <typename F>
atspeed_status guarded(atspeed_ctx* c, F&& f) {
  if (!c) return ATSPEED_E_ARG;
  try {
    CK(cudaSetDevice(c->device));
    f();
    return ATSPEED_OK;
  } catch (const Fail& e) {
    return e.st;
  }
}

void write_outputs(atspeed_ctx* c, cudaStream_t st, int32_t* d_acc, int32_t* d_depth, int32_t* d_beams,
                   float* d_scores, const std::vector<int>& acc) {
  const int B = c->B, K = c->step_K;
  std::vector<int> depth(B), beams((size_t)B * K * 4, -1);
  std::vector<float> sc((size_t)B * K, -INFINITY);
  for (int u = 0; u < B; ++u) {
    const UserState& us = c->users[u];
    depth[u] = us.d;
    for (size_t k = 0; k < us.path.size() && (int)k < K; ++k) {
      for (int i = 0; i < 4; ++i) beams[((size_t)u * K + k) * 4 + i] = us.path[k][i];
      sc[(size_t)u * K + k] = us.sp[k];
    }
  }
  if (d_acc) upload(c, st, d_acc, acc.data(), (size_t)B * 4);
  if (d_depth) upload(c, st, d_depth, depth.data(), (size_t)B * 4);
  if (d_beams) upload(c, st, d_beams, beams.data(), beams.size() * 4);
  if (d_scores) upload(c, st, d_scores, sc.data(), sc.size() * 4);
  stage_sync(c, st);
}

}  // namespace

// =============================================================================================
// C ABI
// =============================================================================================
extern "C" {

atspeed_status atspeed_create(const atspeed_model_desc* target, const atspeed_model_desc* draft,
                              const atspeed_items_desc* items, const atspeed_limits* lim, atspeed_ctx** out) {
  g_create_error.clear();
  if (!out || !target || !items || !lim) {
    g_create_error = "atspeed_create: null argument";
    return ATSPEED_E_ARG;
  }
  *out = nullptr;
  atspeed_ctx* c = new atspeed_ctx();
  try {
    CK(cudaGetDevice(&c->device));
    if (items->L != 4 || items->codes_per_level != 256 || items->n_items < 1 || !items->h_codes) {
      set_err(c, "items: need L = 4, 256 codes per level, n_items >= 1");
      throw Fail{ATSPEED_E_SHAPE};
    }
    if (lim->max_users < 1 || lim->max_prompt < 1 || lim->max_K < 1 || lim->max_K > 256 || lim->max_N < 1 ||
        lim->max_N > 256 || lim->max_gamma < 0 || lim->max_gamma > 4) {
      set_err(c, "limits out of range");
      throw Fail{ATSPEED_E_SHAPE};
    }
    c->lim = *lim;
    c->code_base = items->code_base;
    init_model(c, c->tgt, target, "target");
    init_model(c, c->drf, draft, "draft");
    if (c->code_base < 0 || c->code_base + ITEM_ROWS > c->tgt.V || (c->drf.present && c->code_base + ITEM_ROWS > c->drf.V)) {
      set_err(c, "item codes [code_base, code_base + 1024) exceed the vocabulary");
      throw Fail{ATSPEED_E_SHAPE};
    }
    if (c->drf.present && c->drf.V != c->tgt.V) {
      set_err(c, "draft and target vocabularies differ");
      throw Fail{ATSPEED_E_SHAPE};
    }
    c->prefix_pages_per_user = (lim->max_prompt + ATT_PAGE - 1) / ATT_PAGE;
    const int stride = lim->max_K + lim->max_gamma * lim->max_N;
    c->node_rows_per_user = TREE_L * stride;
    build_trie(c, items);
    alloc_model(c, c->tgt);
    alloc_model(c, c->drf);
    c->gemm_grid = gemm_grid_size(c->device);
    c->fwd_grid = c->gemm_grid;  // one persistent CTA per SM
    {
      // Schedule of a model's forward: one persistent launch; ATSPEED_FORWARD=per_op runs one kernel
      // per op instead (same bits).  GEMM work splits run over min(SMs, gate/up weight tiles) CTAs:
      // a small model (the 4-layer draft: 48 tiles) then takes one whole gate/up tile per CTA with
      // no split sums, and every phase's grid barrier spans fewer CTAs; a 7B-shape model (172 tiles)
      // takes the whole GPU.
      const char* fm = getenv("ATSPEED_FORWARD");
      c->forward_mode = (fm && strcmp(fm, "persistent") == 0) ? 1 : (fm && strcmp(fm, "per_op") == 0) ? 2 : 0;
      for (ModelRt* mr : {&c->tgt, &c->drf}) {
        mr->per_op = c->forward_mode == 2;
        mr->grid = std::max(1, std::min(c->fwd_grid, 2 * mr->ffn / 128));
      }
    }
    {
      // grid barrier, split-tile arrivals and attention split arrivals of the persistent forward:
      // one block, zeroed by one memset before every launch
      const int Lmax = std::max(c->tgt.layers, c->drf.present ? c->drf.layers : 0);
      c->fwd_sk_n = (size_t)(4 * Lmax + 1) * c->fwd_grid;
      size_t att = 0;
      for (ModelRt* mr : {&c->tgt, &c->drf})
        if (mr->present) att = std::max(att, (size_t)mr->max_qt * mr->H);
      c->fwd_zero_att = 32 + c->fwd_sk_n;
      c->fwd_zero = dalloc<int>(c, c->fwd_zero_att + att);
      c->fwd_bar = reinterpret_cast<unsigned int*>(c->fwd_zero);
      c->fwd_sk = c->fwd_zero + 32;
      for (ModelRt* mr : {&c->tgt, &c->drf}) mr->att_counters = c->fwd_zero + c->fwd_zero_att;
    }
    {
      const char* tr = getenv("ATSPEED_FWD_TRACE");
      if (tr && tr[0] == '1') {
        const int Lmax = std::max(c->tgt.layers, c->drf.present ? c->drf.layers : 0);
        c->fwd_trace_n = (size_t)16 * (7 * Lmax + 2) * c->fwd_grid;
        c->fwd_trace = dalloc<unsigned long long>(c, c->fwd_trace_n);
      }
    }
    c->gs.ws_bytes = gemm_ws_bytes(c->gemm_grid);
    c->gs.ws = dalloc<float>(c, c->gs.ws_bytes / 4, false);
    c->gs.max_tiles = gemm_max_tiles();
    c->gs.counters = dalloc<int>(c, c->gs.max_tiles);
    c->err_word = dalloc<unsigned int>(c, 1);
    c->gs.err = c->err_word;
    const size_t nn = (size_t)lim->max_users * stride;
    c->cap_nodes = (int)nn;
    const size_t n_cnt_max = (size_t)lim->max_users * (lim->max_gamma + 1);
    c->n_blk = dalloc<int>(c, NODE_INTS * nn + n_cnt_max);
    carve_nodes(c, nn, lim->max_users, lim->max_gamma);
    const int mu = lim->max_users;
    c->u_blk = dalloc<int>(c, 4 * (size_t)mu);
    c->u_d = c->u_blk;
    c->u_g = c->u_blk + mu;
    c->u_step = c->u_blk + 2 * mu;
    c->u_P = c->u_blk + 3 * mu;
    c->fwd_nodes = dalloc<int>(c, nn);
    // staging: the largest per-step upload is the node table; forward plans and outputs are small
    c->stage_cap = 2 * (NODE_INTS * nn + n_cnt_max) * sizeof(int) + ((size_t)1 << 20);
    {
      void* hp = nullptr;
      CK(cudaMallocHost(&hp, c->stage_cap));
      c->h_stage = static_cast<uint8_t*>(hp);
    }
    std::vector<int> pt((size_t)lim->max_users * c->prefix_pages_per_user);
    for (size_t i = 0; i < pt.size(); ++i) pt[i] = (int)i;  // user u's prefix pages are contiguous
    c->page_table = dalloc<int>(c, pt.size(), false);
    CK(cudaMemcpy(c->page_table, pt.data(), pt.size() * 4, cudaMemcpyHostToDevice));
    {
      // verification outputs in one block, read back by one copy per step
      const size_t mk = (size_t)mu * lim->max_K;
      c->o_blk = dalloc<int>(c, o_blk_ints(mu, lim->max_K));
      int* q = c->o_blk;
      c->o_acc = q, q += mu;
      c->o_adv = q, q += mu;
      c->o_n = q, q += mu;
      c->o_nacc = q, q += mu;
      c->o_path = q, q += 4 * mk;
      c->o_parent = q, q += mk;
      c->o_trie = q, q += mk;
      c->o_score = reinterpret_cast<float*>(q), q += mk;
      c->o_anc_t = q, q += 4 * mk;
      c->o_anc_d = q, q += 4 * mk;
    }
    CK(cudaDeviceSynchronize());
  } catch (const Fail& e) {
    g_create_error = c->err;
    atspeed_destroy(c);
    return e.st;
  }
  *out = c;
  return ATSPEED_OK;
}

void atspeed_destroy(atspeed_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->device);
  cudaDeviceSynchronize();
  for (auto& r : c->prof_recs) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : c->prof_pool) cudaEventDestroy(e);
  for (void* p : c->allocs) cudaFree(p);
  if (c->h_stage) cudaFreeHost(c->h_stage);
  delete c;
}

const char* atspeed_last_error(const atspeed_ctx* c) { return c ? c->err.c_str() : g_create_error.c_str(); }

atspeed_status atspeed_prefill(atspeed_ctx* c, atspeed_stream stream, int n_users, const int32_t* d_tokens,
                               const int32_t* h_offsets) {
  return guarded(c, [&] { prefill_impl(c, (cudaStream_t)stream, n_users, d_tokens, h_offsets); });
}

atspeed_status atspeed_draft_step(atspeed_ctx* c, atspeed_stream stream, const atspeed_decode_opts* opts,
                                  atspeed_verify_mode mode) {
  return guarded(c, [&] { draft_step_impl(c, (cudaStream_t)stream, opts, mode); });
}

atspeed_status atspeed_verify(atspeed_ctx* c, atspeed_stream stream, const atspeed_decode_opts* opts,
                              atspeed_verify_mode mode, int32_t* d_accepted, int32_t* d_depth, int32_t* d_beams,
                              float* d_scores) {
  return guarded(c, [&] {
    cudaStream_t st = (cudaStream_t)stream;
    std::vector<int> before(c->B);
    for (int u = 0; u < c->B; ++u) before[u] = c->users[u].acc_steps;
    verify_impl(c, st, opts, mode);
    std::vector<int> acc(c->B);
    for (int u = 0; u < c->B; ++u) acc[u] = c->users[u].acc_steps - before[u];
    write_outputs(c, st, d_accepted, d_depth, d_beams, d_scores, acc);
  });
}

atspeed_status atspeed_draft_step_logits(atspeed_ctx* c, atspeed_stream stream, const atspeed_decode_opts* opts,
                                         atspeed_verify_mode mode, const float* h_logits) {
  return guarded(c, [&] { draft_step_logits_impl(c, (cudaStream_t)stream, opts, mode, h_logits); });
}

atspeed_status atspeed_verify_logits(atspeed_ctx* c, atspeed_stream stream, const atspeed_decode_opts* opts,
                                     atspeed_verify_mode mode, const float* h_logits, int32_t* d_accepted,
                                     int32_t* d_depth, int32_t* d_beams, float* d_scores) {
  return guarded(c, [&] {
    cudaStream_t st = (cudaStream_t)stream;
    std::vector<int> before(c->B);
    for (int u = 0; u < c->B; ++u) before[u] = c->users[u].acc_steps;
    verify_logits_impl(c, st, opts, mode, h_logits);
    std::vector<int> acc(c->B);
    for (int u = 0; u < c->B; ++u) acc[u] = c->users[u].acc_steps - before[u];
    write_outputs(c, st, d_accepted, d_depth, d_beams, d_scores, acc);
  });
}

atspeed_status atspeed_beam_search(atspeed_ctx* c, atspeed_stream stream, int n_users, const int32_t* d_tokens,
                                   const int32_t* h_offsets, const atspeed_decode_opts* opts,
                                   atspeed_decode_mode mode, int32_t* d_items, float* d_scores, int32_t* h_stats) {
  return guarded(c, [&] {
    cudaStream_t st = (cudaStream_t)stream;
    check_opts(c, opts);
    const bool sd = mode == ATSPEED_SD_STRICT || mode == ATSPEED_SD_RELAXED;
    if (sd && !c->drf.present) {
      set_err(c, "speculative decoding needs a draft model");
      throw Fail{ATSPEED_E_STATE};
    }
    const atspeed_verify_mode vm =
        (mode == ATSPEED_SD_RELAXED || mode == ATSPEED_PLAIN_SAMPLE) ? ATSPEED_RELAXED : ATSPEED_STRICT;
    prefill_impl(c, st, n_users, d_tokens, h_offsets);
    atspeed_decode_opts o = *opts;
    if (!sd) o.gamma = 0;
    std::vector<std::vector<std::array<int, 4>>> fin_path(n_users);
    std::vector<std::vector<float>> fin_sp(n_users);
    for (int guard = 0; guard < 4 * TREE_L; ++guard) {
      bool any = false;
      for (auto& us : c->users) any |= us.active;
      if (!any) break;
      open_step(c, &o, st);
      int maxg = 0;
      for (auto& us : c->users)
        if (us.active) maxg = std::max(maxg, us.g);
      // with early rejection the level-1 decision is taken right after drafting level 1, before the
      // draft forward over it: a step that every user rejects at level 1 runs no further forward
      const bool probe = c->early_reject && maxg >= 1;
      bool decided = false;
      std::vector<bool> was(n_users);
      for (int u = 0; u < n_users; ++u) was[u] = c->users[u].active;
      for (int j = 0; j < maxg && !decided; ++j) {
        draft_step_impl(c, st, &o, vm, !(probe && j == 0));
        if (probe && j == 0 && early_reject_eligible(c) && early_reject_probe(c, st, &o, vm)) decided = true;
      }
      if (decided) {
        c->level_fwd_pending = false;
        commit(c, st, true, std::vector<int>(n_users, 0));
      } else {
        verify_impl(c, st, &o, vm, !probe);
      }
      for (int u = 0; u < n_users; ++u)
        if (was[u] && !c->users[u].active) {
          fin_path[u] = c->users[u].path;
          fin_sp[u] = c->users[u].sp;
        }
    }
    const int K = o.K;
    std::vector<int> items((size_t)n_users * K * 4, -1);
    std::vector<float> sc((size_t)n_users * K, -INFINITY);
    for (int u = 0; u < n_users; ++u)
      for (size_t k = 0; k < fin_path[u].size() && (int)k < K; ++k) {
        for (int i = 0; i < 4; ++i) items[((size_t)u * K + k) * 4 + i] = fin_path[u][k][i];
        sc[(size_t)u * K + k] = fin_sp[u][k];
      }
    if (d_items) upload(c, st, d_items, items.data(), items.size() * 4);
    if (d_scores) upload(c, st, d_scores, sc.data(), sc.size() * 4);
    if (h_stats)
      for (int u = 0; u < n_users; ++u) {
        h_stats[u * 3 + 0] = c->users[u].acc_steps;
        h_stats[u * 3 + 1] = c->users[u].calls;
        h_stats[u * 3 + 2] = c->users[u].tree_tokens;
      }
    stage_sync(c, st);
  });
}

atspeed_status atspeed_begin_step(atspeed_ctx* c, atspeed_stream stream, const atspeed_decode_opts* opts) {
  return guarded(c, [&] {
    check_opts(c, opts);
    if (c->step_open) {
      set_err(c, "a speculative step is already open");
      throw Fail{ATSPEED_E_STATE};
    }
    ensure_step(c, opts, (cudaStream_t)stream);
  });
}

atspeed_status atspeed_set_early_reject(atspeed_ctx* c, int enable) {
  return guarded(c, [&] {
    if (c->step_open) {
      set_err(c, "set_early_reject: a speculative step is open");
      throw Fail{ATSPEED_E_STATE};
    }
    c->early_reject = enable != 0;
  });
}

atspeed_status atspeed_profile(atspeed_ctx* c, int enable) {
  return guarded(c, [&] {
    CK(cudaDeviceSynchronize());
    for (auto& r : c->prof_recs) {
      c->prof_pool.push_back(r.a);
      c->prof_pool.push_back(r.b);
    }
    c->prof_recs.clear();
    c->prof = enable != 0;
  });
}

atspeed_status atspeed_profile_read(atspeed_ctx* c, int kind, int32_t* h_launches, double* h_ms, double* h_bytes,
                                    double* h_flops) {
  return guarded(c, [&] {
    CK(cudaDeviceSynchronize());
    if (kind < 0) {  // total kernel launches of this context since creation
      if (h_launches) *h_launches = (int32_t)c->n_launch;
      if (h_ms) *h_ms = 0;
      if (h_bytes) *h_bytes = 0;
      if (h_flops) *h_flops = 0;
      return;
    }
    int n = 0;
    double ms = 0, by = 0, fl = 0;
    for (auto& r : c->prof_recs) {
      if (r.kind != kind) continue;
      float t = 0.f;
      CK(cudaEventElapsedTime(&t, r.a, r.b));
      ++n;
      ms += t;
      by += r.bytes;
      fl += r.flops;
    }
    if (h_launches) *h_launches = n;
    if (h_ms) *h_ms = ms;
    if (h_bytes) *h_bytes = by;
    if (h_flops) *h_flops = fl;
  });
}

atspeed_status atspeed_debug_buffer(atspeed_ctx* c, int which, int id, void* h_out, size_t bytes) {
  return guarded(c, [&] {
    const ModelRt& m = which == 0 ? c->tgt : c->drf;
    const void* src = nullptr;
    size_t cap = 0;
    switch (id) {
      case 0: src = m.h; cap = (size_t)m.Tcap * m.d * 4; break;
      case 1: src = m.x; cap = (size_t)m.Xrows * m.d * 2; break;
      case 2: src = m.q; cap = (size_t)m.Tcap * m.d * 2; break;
      case 3: src = m.att; cap = (size_t)m.Xrows * m.d * 2; break;
      case 4: src = m.act; cap = (size_t)m.Xrows * m.ffn * 2; break;
      case 5: src = m.kc; cap = (size_t)m.rows * m.d * 2 * m.layers; break;
      case 6: src = m.vc; cap = (size_t)m.rows * m.d * 2 * m.layers; break;
      case 7: src = m.logits; cap = (size_t)m.logit_rows * ITEM_ROWS * 4; break;
      case 8: src = c->fwd_bar; cap = 4; break;
      case 9: src = c->fwd_trace; cap = c->fwd_trace_n * 8; break;
      case 10: src = m.lse; cap = (size_t)m.logit_rows * 4; break;
      case 11: src = m.tok; cap = (size_t)m.Tcap * 4; break;
      case 12: src = m.pos; cap = (size_t)m.Tcap * 4; break;
      case 13: src = m.kvrow; cap = (size_t)m.Tcap * 4; break;
      case 14: src = m.anc; cap = (size_t)m.Tcap * 16; break;
      case 15: src = m.ancn; cap = (size_t)m.Tcap * 4; break;
      case 16: {  // geometry, from the host
        const int32_t g[4] = {m.rows, m.Tcap, m.Xrows, c->prefix_pages_per_user};
        if (!m.present || !h_out || bytes > sizeof g) {
          set_err(c, "debug_buffer: bad arguments");
          throw Fail{ATSPEED_E_ARG};
        }
        memcpy(h_out, g, bytes);
        return;
      }
      default: break;
    }
    if (!m.present || !src || !h_out || bytes > cap) {
      set_err(c, "debug_buffer: bad arguments");
      throw Fail{ATSPEED_E_ARG};
    }
    CK(cudaDeviceSynchronize());
    CK(cudaMemcpy(h_out, src, bytes, cudaMemcpyDeviceToHost));
  });
}

atspeed_status atspeed_tree_shape(const atspeed_ctx* cc, int32_t* h_depth, int32_t* h_levels, int32_t* h_slots_in,
                                  int32_t* h_slots_lvl) {
  if (!cc) return ATSPEED_E_ARG;
  for (int u = 0; u < cc->B; ++u) {
    if (h_depth) h_depth[u] = cc->users[u].d;
    if (h_levels) h_levels[u] = cc->step_open ? std::min(cc->levels_done, cc->users[u].g) : 0;
  }
  if (h_slots_in) *h_slots_in = cc->step_K;
  if (h_slots_lvl) *h_slots_lvl = cc->step_N;
  return ATSPEED_OK;
}

atspeed_status atspeed_debug_tree(atspeed_ctx* c, int32_t* h_path, float* h_sq, float* h_sp, int32_t* h_count) {
  return guarded(c, [&] {
    if (!c->have_tree) {
      set_err(c, "no speculative step has been opened");
      throw Fail{ATSPEED_E_STATE};
    }
    const size_t n = (size_t)c->B * (c->step_K + c->step_gamma * c->step_N);
    CK(cudaDeviceSynchronize());
    if (h_path) CK(cudaMemcpy(h_path, c->n_path, n * 16, cudaMemcpyDeviceToHost));
    if (h_sq) CK(cudaMemcpy(h_sq, c->n_sq, n * 4, cudaMemcpyDeviceToHost));
    if (h_sp) CK(cudaMemcpy(h_sp, c->n_sp, n * 4, cudaMemcpyDeviceToHost));
    if (h_count) CK(cudaMemcpy(h_count, c->n_cnt, (size_t)c->B * (c->step_gamma + 1) * 4, cudaMemcpyDeviceToHost));
  });
}

atspeed_status atspeed_debug_node_logits(atspeed_ctx* c, int which, int user, int slot, float* h_logits) {
  return guarded(c, [&] {
    const int stride = c->step_K + c->step_gamma * c->step_N;
    if (!c->have_tree || user < 0 || user >= c->B || slot < 0 || slot >= stride || !h_logits) {
      set_err(c, "debug_node_logits: bad arguments or no open step");
      throw Fail{ATSPEED_E_ARG};
    }
    CK(cudaDeviceSynchronize());
    int row = -1;
    CK(cudaMemcpy(&row, (which == 0 ? c->n_lg_t : c->n_lg_d) + (size_t)user * stride + slot, 4,
                  cudaMemcpyDeviceToHost));
    if (row < 0) {
      set_err(c, "node was not forwarded");
      throw Fail{ATSPEED_E_STATE};
    }
    const ModelRt& m = which == 0 ? c->tgt : c->drf;
    CK(cudaMemcpy(h_logits, m.logits + (size_t)row * ITEM_ROWS, ITEM_ROWS * 4, cudaMemcpyDeviceToHost));
  });
}

atspeed_status atspeed_debug_node_lse(atspeed_ctx* c, int which, int user, int slot, float* h_lse) {
  return guarded(c, [&] {
    const int stride = c->step_K + c->step_gamma * c->step_N;
    if (!c->have_tree || !c->full_norm || user < 0 || user >= c->B || slot < 0 || slot >= stride || !h_lse) {
      set_err(c, "debug_node_lse: bad arguments, no open step or not a FULL-normalised step");
      throw Fail{ATSPEED_E_ARG};
    }
    CK(cudaDeviceSynchronize());
    int row = -1;
    CK(cudaMemcpy(&row, (which == 0 ? c->n_lg_t : c->n_lg_d) + (size_t)user * stride + slot, 4,
                  cudaMemcpyDeviceToHost));
    if (row < 0) {
      set_err(c, "node was not forwarded");
      throw Fail{ATSPEED_E_STATE};
    }
    const ModelRt& m = (which == 0 || !c->drf.present) ? c->tgt : c->drf;
    CK(cudaMemcpy(h_lse, m.lse + row, 4, cudaMemcpyDeviceToHost));
  });
}

atspeed_status atspeed_set_tree(atspeed_ctx* c, atspeed_stream stream, int n_levels, const int32_t* h_count,
                                const int32_t* h_parent, const int32_t* h_code, const float* h_sq,
                                const float* h_draft_logits) {
  return guarded(c, [&] {
    cudaStream_t st = (cudaStream_t)stream;
    if (!c->step_open) {
      set_err(c, "set_tree: call atspeed_begin_step first");
      throw Fail{ATSPEED_E_STATE};
    }
    if (n_levels < 0 || n_levels > c->step_gamma || !h_count || (n_levels > 0 && (!h_parent || !h_code || !h_sq))) {
      set_err(c, "set_tree: bad arguments");
      throw Fail{ATSPEED_E_ARG};
    }
    const int K = c->step_K, N = c->step_N, G = c->step_gamma, stride = K + G * N, W = c->lim.max_N;
    const size_t n = (size_t)c->B * stride;
    std::vector<int> code(n), prank(n), trie(n), path(n * 4), rt(n), rd(n), at(n * 4), ad(n * 4), lgd(n),
        cnt((size_t)c->B * (G + 1));
    std::vector<float> sq(n), sp(n);
    stage_sync(c, st);
    CK(cudaMemcpy(code.data(), c->n_code, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(trie.data(), c->n_trie, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(path.data(), c->n_path, n * 16, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(rt.data(), c->n_row_t, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(rd.data(), c->n_row_d, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(at.data(), c->n_anc_t, n * 16, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(ad.data(), c->n_anc_d, n * 16, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(lgd.data(), c->n_lg_d, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(sq.data(), c->n_sq, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(sp.data(), c->n_sp, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(prank.data(), c->n_prank, n * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(cnt.data(), c->n_cnt, cnt.size() * 4, cudaMemcpyDeviceToHost));
    int drow = c->B;  // draft logits rows for injected parents
    std::vector<float> dl;
    std::vector<int> dl_rows;
    for (int u = 0; u < c->B; ++u) {
      UserState& us = c->users[u];
      if (!us.active) continue;
      const int gl = std::min(n_levels, TREE_L - us.d);
      us.g = gl;
      for (int j = 1; j <= G; ++j) cnt[(size_t)u * (G + 1) + j] = 0;
      for (int j = 1; j <= gl; ++j) {
        const int m = h_count[u * n_levels + j - 1];
        const int pc = cnt[(size_t)u * (G + 1) + j - 1];
        if (m < 0 || m > N) {
          set_err(c, "set_tree: level %d of user %d has %d nodes (N = %d)", j, u, m, N);
          throw Fail{ATSPEED_E_SHAPE};
        }
        const int poff = j == 1 ? 0 : K + (j - 2) * N, off = K + (j - 1) * N;
        for (int k = 0; k < N; ++k) {
          const size_t nd = (size_t)u * stride + off + k;
          if (k >= m) {
            code[nd] = -1;
            prank[nd] = -1;
            for (int i = 0; i < 4; ++i) path[nd * 4 + i] = -1;
            continue;
          }
          const size_t src = ((size_t)u * n_levels + (j - 1)) * W + k;
          const int p = h_parent[src], cd = h_code[src];
          if (p < 0 || p >= pc || cd < 0 || cd > 255) {
            set_err(c, "set_tree: bad parent/code at user %d level %d node %d", u, j, k);
            throw Fail{ATSPEED_E_ARG};
          }
          const size_t par = (size_t)u * stride + poff + p;
          if (!host_trie_has(c, trie[par], cd)) {
            set_err(c, "set_tree: user %d level %d node %d is not a valid item prefix", u, j, k);
            throw Fail{ATSPEED_E_ARG};
          }
          const int depth = us.d + j;
          code[nd] = cd;
          prank[nd] = p;
          trie[nd] = host_trie_child(c, trie[par], cd);
          for (int i = 0; i < 4; ++i) {
            path[nd * 4 + i] = i == depth - 1 ? cd : path[par * 4 + i];
            at[nd * 4 + i] = i == depth - 1 ? rt[nd] : at[par * 4 + i];
            ad[nd * 4 + i] = i == depth - 1 ? rd[nd] : ad[par * 4 + i];
          }
          sq[nd] = h_sq[src];
          sp[nd] = 0.f;
        }
        cnt[(size_t)u * (G + 1) + j] = m;
      }
      if (h_draft_logits) {
        for (int j = 0; j < gl; ++j) {
          const int poff = j == 0 ? 0 : K + (j - 1) * N;
          const int pc = cnt[(size_t)u * (G + 1) + j];
          for (int k = 0; k < pc; ++k) {
            const size_t nd = (size_t)u * stride + poff + k;
            const float* src = h_draft_logits + (((size_t)u * n_levels + j) * W + k) * ITEM_ROWS;
            dl.insert(dl.end(), src, src + ITEM_ROWS);
            lgd[nd] = drow++;
          }
        }
      }
    }
    if (!dl.empty()) {
      ModelRt& m = c->drf.present ? c->drf : c->tgt;
      if (drow > m.logit_rows) {
        set_err(c, "set_tree: too many draft logits rows");
        throw Fail{ATSPEED_E_SHAPE};
      }
      CK(cudaMemcpy(m.logits + (size_t)c->B * ITEM_ROWS, dl.data(), dl.size() * 4, cudaMemcpyHostToDevice));
    }
    CK(cudaMemcpy(c->n_code, code.data(), n * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_prank, prank.data(), n * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_trie, trie.data(), n * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_path, path.data(), n * 16, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_anc_t, at.data(), n * 16, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_anc_d, ad.data(), n * 16, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_lg_d, lgd.data(), n * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_sq, sq.data(), n * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_sp, sp.data(), n * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(c->n_cnt, cnt.data(), cnt.size() * 4, cudaMemcpyHostToDevice));
    c->levels_done = n_levels;
    c->tree_injected = true;
    upload_users(c, st);
  });
}

}  // extern "C"
