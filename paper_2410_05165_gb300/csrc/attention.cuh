// Tree attention over a paged, shared user-history prefix (Sec. 3.3 "Tree-based Attention",
// App. A.3.1).  A drafted node attends to the whole prefix of its user plus the tree nodes on its
// own path (ancestors and itself), which is exactly what the flattened-sequence tree mask of
// App. A.3.1 selects.  The prefix part is shared by every node of a user, so it is computed with
// tensor cores for a whole tile of queries while each K/V page is read once per tile; the path
// part (at most L = 4 keys per node) is merged afterwards in a combine kernel.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace atspeed {

constexpr int ATT_PAGE = 64;       // rows per KV page
constexpr int ATT_SUB = 32;        // rows per K / V copy of the attention (half a page)
constexpr int ATT_QTILE = 64;      // queries per CTA
constexpr int ATT_MAX_ANC = 4;     // path keys per query (L = 4)

struct AttnArgs {
  int T, n_heads, head_dim;        // d_model = n_heads * head_dim
  const __nv_bfloat16* q;          // [T][d] (RoPE applied)
  const __nv_bfloat16* k_cache;    // [rows][d] for this layer
  const __half* v_cache;           // fp16 holding bf16-rounded values (exact)
  int kv_rows;                     // rows of the cache arena
  // query tiles: consecutive tokens of one user
  int n_qtiles;
  const int* qt_t0;                // [n_qtiles] first token of the tile
  const int* qt_n;                 // [n_qtiles] tokens in the tile (<= 64)
  const int* qt_user;              // [n_qtiles]
  const int* qt_vis;               // [n_qtiles] longest visible prefix of the tile's tokens
  // per token
  const int* tok_user;             // [T] user of each token
  const int* tok_vis;              // [T] visible prefix length (P for tree nodes, pos+1 for prefill)
  const int* anc_row;              // [T][4] cache rows of the path keys (ancestors and self) or null
  const int* anc_n;                // [T] number of path keys
  // per user
  const int* page_table;           // [users][max_pages] page ids (page p = rows 64p .. 64p+63)
  int max_pages;
  const int* user_splits;          // [users] number of prefix splits of this user
  int chunks_per_split;            // prefix pages per split (0 = all pages in one split)
  int max_splits;                  // grid z
  // outputs
  __nv_bfloat16* out;              // [T][d] attention output (bf16)
  float* part_o;                   // [max_splits][T][n_heads][head_dim] unnormalised partials
  float* part_ml;                  // [max_splits][T][n_heads][2] (running max in log2 units, sum)
  bool direct;                     // single split and no path keys: write `out` directly
  unsigned int* err;
};

// Encodes the K/V tensor maps for one layer's cache arena (box = 64 rows x min(head_dim, 64)).
bool attn_make_maps(const __nv_bfloat16* k_cache, const __half* v_cache, int rows, int d_model,
                    int head_dim, CUtensorMap* mk, CUtensorMap* mv, char* eb, size_t el);

cudaError_t attn_launch(const AttnArgs& a, const CUtensorMap& mk, const CUtensorMap& mv, cudaStream_t st, bool pdl);

}  // namespace atspeed
