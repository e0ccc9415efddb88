// Device-side state of one speculative step: the drafted beam tree of every user, laid out as a
// fixed-shape node table so that every kernel launch of a step has a host-known shape.
//
// Per user the table holds level 0 (the incoming beams, `slots_in` slots) followed by drafted
// levels 1 .. max_levels (`slots_lvl` slots each, the draft beam width N).  Unused slots carry
// code -1.  A node at level j of a user at depth d sits at depth d + j of the item identifier.
#pragma once
#include <stdint.h>

namespace atspeed {

constexpr int TREE_L = 4;       // item identifier length
constexpr int TREE_CODES = 256; // codes per level
constexpr int ITEM_ROWS = TREE_L * TREE_CODES;  // item-code logits per forwarded node

struct TreeDev {
  int B, slots_in, slots_lvl, max_levels, stride;   // stride = slots_in + max_levels * slots_lvl
  // per user [B]
  const int* d;        // depth of the incoming beams (0..L-1)
  const int* g;        // drafted levels this step (gamma' = min(gamma, L - d))
  const int* sd_step;  // speculative steps already taken by this user (Philox counter word)
  int* cnt;            // [B][max_levels + 1] valid nodes per level
  // per node [B * stride]
  int* code;           // last code of the node's path (-1: unused slot / empty path)
  int* prank;          // slot of the parent within the previous level (-1 on level 0)
  int* trie;           // trie node of the node's prefix
  int* path;           // [.][4] codes of the whole path, -1 padded
  float* sq;           // draft sequence score (fp32)
  float* sp;           // target sequence score (fp32)
  int* row_t;          // own KV-cache row in the target cache (-1 if never forwarded)
  int* row_d;          // own KV-cache row in the draft cache
  int* anc_t;          // [.][4] target cache rows of the path tokens, depth 1 .. depth
  int* anc_d;          // [.][4]
  int* lg_t;           // row of the target item-code logits buffer (-1 if not forwarded)
  int* lg_d;           // row of the draft item-code logits buffer
  // trie: node 0 is the root; children of node x are trie_child[x] + rank of the code in mask
  const uint32_t* trie_mask;  // [nodes][8]
  const int* trie_child;      // [nodes]
  // item-code logits [rows][1024]: block l*256 .. l*256+255 scores the codes of level l
  const float* logits_t;
  const float* logits_d;
  // FULL normalisation: log-sum-exp of each logits row's whole-vocabulary row (same row index as
  // logits_t / logits_d); null under MASKED normalisation
  const float* lse_t;
  const float* lse_d;
};

__host__ __device__ inline int level_off(const TreeDev& t, int lvl) {
  return lvl == 0 ? 0 : t.slots_in + (lvl - 1) * t.slots_lvl;
}
__host__ __device__ inline int level_width(const TreeDev& t, int lvl) { return lvl == 0 ? t.slots_in : t.slots_lvl; }

struct VerifyOut {
  int* accepted;       // [B] accepted steps a
  int* advance;        // [B] depth gained
  int* n_out;          // [B] output beams (K, or fewer when fewer valid items exist)
  int* n_acc_last;     // [B] |A| at the last verified level (relaxed)
  int* out_path;       // [B][K][4]
  float* out_score;    // [B][K]
  int* out_parent;     // [B][K] global node index of the output beam's parent
  int* out_trie;       // [B][K] trie node of the output beam's prefix
  int* out_anc_t;      // [B][K][4] target cache rows of the parent's path tokens (anc_t of the parent)
  int* out_anc_d;      // [B][K][4] the same in the draft cache
};

}  // namespace atspeed
