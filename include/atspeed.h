/*
 * atspeed.h -- C ABI of the GB300 (sm_103a) implementation of the AtSpeed verification call
 * (speculative beam decoding for LLM-based generative recommendation, arXiv 2410.05165).
 *
 * Problem statement (Sec. 2): a target LLM M_p encodes a user's history x and returns the top-K
 * items {y_{L,i}} by beam search over item identifiers of L = 4 codebook tokens, restricted to
 * valid identifiers (Sec. 3.1).  Speculative decoding (Sec. 2, Alg. 1, Alg. 2) lets a small draft
 * model M_q run gamma beam-search steps of width N; one target call over the whole tree of drafted
 * beams (tree attention, Sec. 3.3 / App. A.3.1) then verifies them, strictly (the target's top-K
 * must be among the drafts at every accepted step) or by relaxed sampling (Sec. 3.2).
 *
 * Conventions shared by every entry point:
 *   - Status codes only: no exceptions cross the ABI, nothing aborts, no kernel traps.  Argument
 *     and shape checks run on the host before the first launch.  A device error word (bounded
 *     waits that timed out, bounds checks) is read at the next synchronisation point and reported
 *     as ATSPEED_E_TIMEOUT / ATSPEED_E_CUDA; atspeed_last_error() gives the message.
 *   - "d_" pointers are device pointers, "h_" pointers are host pointers.  The caller owns every
 *     pointer it passes; the library never frees them.  Weights passed to atspeed_create are
 *     borrowed and must stay alive and unchanged until atspeed_destroy.
 *   - Work is enqueued on the given stream (a cudaStream_t; NULL is the legacy default stream).
 *     Calls that must read results back (verify, beam_search) synchronise that stream.
 *   - One context is not thread-safe; use one context per stream, and pass that same stream to
 *     every call on it (host-to-device copies go through a pinned staging buffer of the context
 *     that is reused after the stream's next synchronisation).  Every GPU buffer the context
 *     needs (KV caches, node pool, activations, workspace) and the staging buffer are allocated
 *     once in atspeed_create, sized by atspeed_limits.
 *   - Token id of code c at identifier level l (0-based) is code_base + 256 * l + c.
 */
#ifndef ATSPEED_H_
#define ATSPEED_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct atspeed_ctx atspeed_ctx;
typedef struct CUstream_st *atspeed_stream; /* same type as cudaStream_t */

typedef enum {
  ATSPEED_OK = 0,
  ATSPEED_E_ARG = -1,         /* null pointer, out-of-range value */
  ATSPEED_E_SHAPE = -2,       /* sizes exceed the limits given at create time, or unsupported dims */
  ATSPEED_E_OOM = -3,         /* device allocation failed in atspeed_create */
  ATSPEED_E_CUDA = -4,        /* a CUDA call failed */
  ATSPEED_E_TIMEOUT = -5,     /* a bounded device wait gave up */
  ATSPEED_E_STATE = -6,       /* wrong call order (e.g. verify before prefill) */
  ATSPEED_E_UNSUPPORTED = -7  /* valid request this build does not implement */
} atspeed_status;

typedef enum { ATSPEED_STRICT = 0, ATSPEED_RELAXED = 1 } atspeed_verify_mode;

/* Normalisation of the constrained token log-probability (the paper does not fix it):
 * MASKED: log-softmax over the valid children only; FULL: over the whole vocabulary, then mask. */
typedef enum { ATSPEED_NORM_MASKED = 0, ATSPEED_NORM_FULL = 1 } atspeed_norm_mode;

typedef enum {
  ATSPEED_PLAIN_TOPK = 0,   /* target-only constrained beam search (the losslessness reference) */
  ATSPEED_PLAIN_SAMPLE = 1, /* target-only sampling beam search at temperature 1 */
  ATSPEED_SD_STRICT = 2,    /* speculative beam decoding, strict top-K verification (Alg. 1)  */
  ATSPEED_SD_RELAXED = 3    /* speculative beam decoding, relaxed sampling verification (Alg. 2) */
} atspeed_decode_mode;

/* LLaMA-style pre-norm decoder (the paper's target is LLaMA-7B, its draft LLaMA-68M, Sec. 4.1).
 * All tensors are bf16, row-major, on the device.  head_dim = d_model / n_heads in {32, 64, 128};
 * d_model and d_ffn multiples of 64. */
typedef struct {
  int n_layers, d_model, n_heads, d_ffn, vocab;
  float rms_eps, rope_theta;
  const void *embed;            /* [vocab][d_model]                                         */
  const void *final_norm;       /* [d_model]                                                */
  const void *lm_head;          /* [vocab][d_model]                                         */
  const void *const *attn_norm; /* n_layers pointers, each [d_model]                        */
  const void *const *wqkv;      /* each [3*d_model][d_model]: rows q | k | v, head-major    */
  const void *const *wo;        /* each [d_model][d_model]                                  */
  const void *const *mlp_norm;  /* each [d_model]                                           */
  const void *const *wgate_up;  /* each [2*d_ffn][d_model]: rows gate | up                  */
  const void *const *wdown;     /* each [d_model][d_ffn]                                    */
} atspeed_model_desc;

/* The valid-item set (Sec. 2 footnote: codebook identifiers of one fixed length).  Copied. */
typedef struct {
  int n_items, L, codes_per_level, code_base; /* L must be 4, codes_per_level 256 */
  const int32_t *h_codes;                     /* host [n_items][L], codes in [0, 256) */
} atspeed_items_desc;

typedef struct {
  int max_users, max_prompt, max_K, max_N, max_gamma; /* max_K, max_N <= 256, max_gamma <= 4 */
} atspeed_limits;

typedef struct {
  int K;                  /* recommended items / target beam width          */
  int N;                  /* draft beam width                                */
  int gamma;              /* drafted beam-search steps per speculative step */
  atspeed_norm_mode norm; /* MASKED or FULL; fixed for a speculative step. FULL runs the LM
                           * head over all V rows of every forwarded node (log-sum-exp
                           * epilogue): V x d_model x 2 more weight bytes per forward      */
  uint64_t philox_seed;   /* key of the Philox4x32-10 streams (relaxed mode) */
} atspeed_decode_opts;

/* Builds the valid-item trie, allocates every device buffer, encodes the TMA descriptors.
 * `draft` may be NULL (then only PLAIN_* decoding and verify-with-injected-trees work). */
atspeed_status atspeed_create(const atspeed_model_desc *target, const atspeed_model_desc *draft,
                              const atspeed_items_desc *items, const atspeed_limits *lim, atspeed_ctx **out);
void atspeed_destroy(atspeed_ctx *ctx);
/* Message of the last failure of this context (or of the last failed create when ctx is NULL). */
const char *atspeed_last_error(const atspeed_ctx *ctx);

/* Prefill (Alg. 1 input "prefix"): causal forward of every user's history through the target (and
 * the draft when present); fills the paged prefix KV caches and the logits p_1 of the first item
 * token, and resets every user to depth 0 with the single empty beam.
 *   d_tokens: device [sum of lengths] int32 token ids, users concatenated;
 *   h_offsets: host [n_users + 1], offsets of each user's history in d_tokens (lengths >= 1). */
atspeed_status atspeed_prefill(atspeed_ctx *ctx, atspeed_stream stream, int n_users, const int32_t *d_tokens,
                               const int32_t *h_offsets);

/* Opens the next speculative step explicitly: level 0 of every user's tree becomes its incoming
 * beams (the single empty beam after prefill).  draft_step and verify open it implicitly; an
 * explicit call is only needed before atspeed_set_tree.  ATSPEED_E_STATE if a step is open. */
atspeed_status atspeed_begin_step(atspeed_ctx *ctx, atspeed_stream stream, const atspeed_decode_opts *opts);

/* Drafting (Eq. 1, Alg. 1/2 drafting loop): appends one drafted level to every user's tree -- the
 * top-N (strict) or N samples without replacement from q_j (relaxed) over the valid extensions of
 * the previous level -- and runs the draft forward over the new level so the next level can be
 * drafted.  The first call of a speculative step also forwards the incoming beams' last tokens.
 * Users whose tree already has gamma' = min(gamma, L - depth) levels are left unchanged.
 * opts must stay the same across the draft_step / verify calls of one speculative step. */
atspeed_status atspeed_draft_step(atspeed_ctx *ctx, atspeed_stream stream, const atspeed_decode_opts *opts,
                                  atspeed_verify_mode mode);

/* The verification call (Alg. 1 / Alg. 2, the hot path): one target forward over every drafted
 * beam of every user (tree attention over the shared prefix, Sec. 3.3), trie-constrained
 * log-softmax, beam scores, exact top-K, then strict or relaxed acceptance; the output beams become
 * the next speculative step's incoming beams (their KV rows are kept, no copy).  Synchronises.
 *   d_accepted [n_users]: accepted steps a of this call;  d_depth [n_users]: depth after the call;
 *   d_beams [n_users][K][4]: output beams (codes, -1 beyond the depth / for missing beams);
 *   d_scores [n_users][K]: their fp32 target log-probabilities (-inf for missing beams).
 * With no drafted level (draft_step not called) this is one step of plain target beam search
 * (strict) or sampling beam search (relaxed). */
atspeed_status atspeed_verify(atspeed_ctx *ctx, atspeed_stream stream, const atspeed_decode_opts *opts,
                              atspeed_verify_mode mode, int32_t *d_accepted, int32_t *d_depth, int32_t *d_beams,
                              float *d_scores);

/* Drafting and verification driven by caller-supplied item-code logits instead of the built-in
 * decoder forwards, for callers that run a model elsewhere (and for kernel-level parity checks).
 *   draft_step_logits: h_logits [n_users][w][1024] are the draft's item-code logits of the nodes of
 *     the previous level (w = K slots for level 0, N slots for drafted levels; unused slots ignored);
 *     appends one drafted level exactly as atspeed_draft_step does, without a draft forward.
 *   verify_logits: h_logits [n_users][K + gamma*N][1024] are the target's item-code logits of every
 *     slot of the node table (level 0, then each drafted level); verifies exactly as atspeed_verify
 *     does, without the target forward.  Both synchronise. */
atspeed_status atspeed_draft_step_logits(atspeed_ctx *ctx, atspeed_stream stream, const atspeed_decode_opts *opts,
                                         atspeed_verify_mode mode, const float *h_logits);
atspeed_status atspeed_verify_logits(atspeed_ctx *ctx, atspeed_stream stream, const atspeed_decode_opts *opts,
                                     atspeed_verify_mode mode, const float *h_logits, int32_t *d_accepted,
                                     int32_t *d_depth, int32_t *d_beams, float *d_scores);

/* One recommendation list per user: prefill, then speculative steps (SD_*) or plain beam-search
 * steps (PLAIN_*) until every user holds complete items.  Synchronises.
 *   d_items [n_users][K][4], d_scores [n_users][K] (ranked, best first);
 *   h_stats [n_users][3] (may be NULL): accepted steps, verification calls, tree tokens. */
atspeed_status atspeed_beam_search(atspeed_ctx *ctx, atspeed_stream stream, int n_users, const int32_t *d_tokens,
                                   const int32_t *h_offsets, const atspeed_decode_opts *opts,
                                   atspeed_decode_mode mode, int32_t *d_items, float *d_scores, int32_t *h_stats);

/* Early rejection (off by default; not part of the paper's method, same outputs bit for bit).
 * At depth 0 the target logits of the empty beam come from the prefill, so the acceptance of
 * drafted level 1 (Alg. 1: are the top-K of level 1 all drafted?  Alg. 2: is |A| >= K?) can be
 * decided before any forward over the tree.  When every active user rejects level 1 -- its output
 * beams are then level-1 candidates scored from those logits alone -- the step ends without the
 * target forward (and, in atspeed_beam_search, without drafting levels 2 .. gamma).  Such a step
 * counts as a verification call with 0 tree tokens.  Costs one extra verification launch and one
 * host synchronisation per depth-0 step when some user accepts.  ATSPEED_E_STATE while a step is
 * open. */
atspeed_status atspeed_set_early_reject(atspeed_ctx *ctx, int enable);

/* ----------------------------------------------------------------------------------------------
 * Introspection / test hooks.
 * ---------------------------------------------------------------------------------------------- */

/* Per-launch timing: while enabled, every kernel launch of the decoder forwards is bracketed by
 * CUDA events on its stream (and programmatic dependent launch is off, so launches do not
 * overlap).  atspeed_profile(ctx, 1) clears previous records.  profile_read sums, over the
 * launches of one kind (0 QKV GEMM, 1 O GEMM, 2 gate/up GEMM, 3 down GEMM, 4 LM-head GEMM,
 * 5 attention, 6 whole persistent forward kernel), the launch count, the device time (ms), and the algorithmic bytes and FLOPs (weights
 * read once, activations in, outputs out).  kind < 0 returns in *h_launches the number of kernels
 * the context has launched since creation (every kind, profiling on or off).  Synchronises. */
atspeed_status atspeed_profile(atspeed_ctx *ctx, int enable);
atspeed_status atspeed_profile_read(atspeed_ctx *ctx, int kind, int32_t *h_launches, double *h_ms, double *h_bytes,
                                    double *h_flops);

/* Copies the first `bytes` of one internal buffer of the target (which = 0) or draft (1) decoder
 * to the host: id 0 residual stream h (fp32 [T][d]), 1 GEMM input rows x (bf16 [T][d]: the final
 * norm's rows after a forward; during it, the gain-scaled residual g * h that feeds the QKV and
 * gate/up projections, whose epilogues apply the norm's per-token scale), 2 q (bf16),
 * 3 attention output (bf16), 4 SwiGLU output (bf16 [T][d_ffn]), 5 K cache (bf16, all layers),
 * 6 V cache (fp16), 7 item-code logits (fp32 [rows][1024]), 8 the persistent forward's barrier
 * counter (u32), 9 its per-phase timestamps ([phases][CTAs] u64 ns, recorded only when the
 * environment variable ATSPEED_FWD_TRACE=1 was set at create time), 10 the whole-vocabulary
 * log-sum-exp of each logits row (fp32 [rows], written under FULL normalisation); the last
 * forward's per-token tables (int32 [T]): 11 token ids, 12 rotary positions, 13 K/V cache rows,
 * 14 the cache rows of each token's path keys ([T][4]), 15 their count; 16 the buffer geometry
 * (int32 [4]: K/V cache rows per layer, token capacity, allocated rows of x, prefix pages per
 * user; user u's history token p sits in cache row u * 64 * pages + p).
 * Synchronises the device (except id 16). */
atspeed_status atspeed_debug_buffer(atspeed_ctx *ctx, int which, int id, void *h_out, size_t bytes);

/* Shape of the current speculative step: h_depth[n_users], h_levels[n_users] (drafted levels),
 * and the node-table geometry (*h_slots_in slots on level 0, *h_slots_lvl per drafted level). */
atspeed_status atspeed_tree_shape(const atspeed_ctx *ctx, int32_t *h_depth, int32_t *h_levels, int32_t *h_slots_in,
                                  int32_t *h_slots_lvl);

/* Copies the node table of the current step to the host: for each user u and slot s of the
 * table (stride = slots_in + gamma * slots_lvl), h_path[(u*stride+s)*4 .. +3] are the node's
 * codes (-1 padded, all -1 for an unused slot) and h_sq / h_sp its draft / target scores.
 * h_count[u*(gamma+1)+j] is the number of valid nodes on level j. */
atspeed_status atspeed_debug_tree(atspeed_ctx *ctx, int32_t *h_path, float *h_sq, float *h_sp, int32_t *h_count);

/* Item-code logits [1024] of a node of the current step (which = 0 target, 1 draft), for the
 * node in slot `slot` of user `user`, copied to the host.  ATSPEED_E_STATE if it was not forwarded. */
atspeed_status atspeed_debug_node_logits(atspeed_ctx *ctx, int which, int user, int slot, float *h_logits);

/* Under FULL normalisation: the log-sum-exp over the whole vocabulary of the same node's logits row
 * (which = 0 target, 1 draft), one float copied to the host.  ATSPEED_E_ARG outside a FULL step,
 * ATSPEED_E_STATE if the node was not forwarded. */
atspeed_status atspeed_debug_node_lse(atspeed_ctx *ctx, int which, int user, int slot, float *h_lse);

/* Replaces the drafted tree of the current step (after prefill / a previous verify, before
 * verify): levels j = 1..n_levels, each with h_count[u*n_levels + j-1] nodes given as
 * (parent slot in level j-1, code, draft score) in draft order; row-major arrays
 * [n_users][n_levels][width] with width = the context's max_N.  Runs the target forward needed by
 * verify but no draft forward, so relaxed verification of an injected tree also needs h_draft_logits:
 * [n_users][levels 0 .. n_levels-1][width][1024] draft item-code logits of every parent node
 * (may be NULL for strict).  Used to verify trees produced outside this library. */
atspeed_status atspeed_set_tree(atspeed_ctx *ctx, atspeed_stream stream, int n_levels, const int32_t *h_count,
                                const int32_t *h_parent, const int32_t *h_code, const float *h_sq,
                                const float *h_draft_logits);

/* ----------------------------------------------------------------------------------------------
 * Stateless operators (the building blocks of the calls above), on caller-owned device buffers.
 * ---------------------------------------------------------------------------------------------- */

/* Y[t][m] = sum_k W[m][k] X[t][k] (+ Y when accumulate) with W bf16 [M][K], X bf16 [x_rows][K]
 * (x_rows >= T rounded up to 128, or to 256 when T > 128), Y fp32 [T][ldy].  tcgen05 tensor cores,
 * fp32 accumulation.  K must be a multiple of 64.  Needs atspeed_op_workspace_bytes() of d_ws
 * (zero-filled before its first use; every call leaves its counter part zeroed again).  Returns
 * ATSPEED_E_SHAPE for a shape it cannot run, ATSPEED_E_ARG for a null or misaligned operand (W, X
 * need 16-byte aligned rows), ATSPEED_E_CUDA for a failed launch; device-side timeouts surface
 * through atspeed_op_status. */
size_t atspeed_op_workspace_bytes(void);
atspeed_status atspeed_op_gemm(atspeed_stream stream, const void *d_W, const void *d_X, int M, int K, int T,
                               int x_rows, float *d_Y, int ldy, int accumulate, void *d_ws);

/* Same result as atspeed_op_gemm, for callers that cannot allocate device memory: code that runs
 * while a stream is being captured into a CUDA graph (an allocation there breaks or is not part of
 * the capture), serving loops with a fixed, pre-reserved memory budget, and hosts whose device
 * memory is owned by another allocator or pool that forbids direct cudaMalloc.  This entry point
 * allocates nothing: its split-K scratch is a static device array inside this library, 8 MiB of
 * partial sums (a 32-CTA grid, two 128 KiB slots per CTA) plus 16 KiB of tile counters and an error
 * word, held by every GPU that loads the library until the process exits.  It therefore runs on at
 * most 32 CTAs (slower than atspeed_op_gemm at large sizes) and accepts at most 4096 output tiles,
 * ceil(M/128) * ceil(T/BN) with BN = 128 for T <= 128 and 256 above (ATSPEED_E_SHAPE otherwise),
 * and K a multiple of 64 up to 16384.  Every call shares the one scratch array, which keeps the
 * previous call's contents (the tile counters are cleared at the start of each call): calls that
 * overlap on one GPU (issued on different streams, or from several host threads) race on it.  The
 * first call on a device looks up the array's device address (no allocation); make that first call
 * before any stream capture.  The paper has no counterpart: it is a deployment convenience. */
atspeed_status atspeed_op_gemm_noalloc(atspeed_stream stream, const void *d_W, const void *d_X, int M, int K, int T,
                                       int x_rows, float *d_Y, int ldy, int accumulate);

/* Device-side failures of the op GEMMs above (atspeed_op_gemm, atspeed_op_gemm_swiglu,
 * atspeed_op_gemm_noalloc).  Their launches return ATSPEED_OK once enqueued; a bounded wait inside
 * the kernel that gives up (a copy or a peer CTA that never arrives) does not trap but sets an error
 * word in the call's scratch, which stays set (sticky) across later calls until this function reads
 * it.  Synchronises `stream`, reads and clears the word of the workspace d_ws (or, with d_ws = NULL,
 * of the allocation-free entry point's scratch on the current device) and returns ATSPEED_OK,
 * ATSPEED_E_TIMEOUT (a bounded wait gave up: the outputs of the calls since the last check are not
 * valid) or ATSPEED_E_CUDA (the synchronisation or the read failed).  Not part of the paper: it is
 * how the stateless operators report device errors. */
atspeed_status atspeed_op_status(atspeed_stream stream, void *d_ws);

/* out[t][j] = bf16(silu(G[t][j]) * U[t][j]) with G = X W[0:F]^T, U = X W[F:2F]^T (SwiGLU), W bf16
 * [2F][K]; out bf16 [T][ldo] with ldo even and d_out 4-byte aligned (ATSPEED_E_ARG otherwise). */
atspeed_status atspeed_op_gemm_swiglu(atspeed_stream stream, const void *d_W, const void *d_X, int F, int K, int T,
                                      int x_rows, void *d_out, int ldo, void *d_ws);

/* x[t] = bf16(h[t] / sqrt(mean(h[t]^2) + eps) * g), h fp32 [T][d], g bf16 [d], x bf16 [T][ldx]. */
atspeed_status atspeed_op_rmsnorm(atspeed_stream stream, const float *d_h, const void *d_g, int T, int d, float eps,
                                  void *d_x, int ldx);

/* Tree attention of T query tokens of ONE user over a paged prefix of length P plus per-token path
 * keys (Sec. 3.3, App. A.3.1).  q bf16 [T][H*hd]; K cache bf16 [rows][H*hd]; V cache fp16
 * [rows][H*hd] holding bf16-rounded values (the library's own layout: P V runs in fp16 with P split
 * into two fp16 halves); prefix row p of the
 * user is cache row 64*h_pages[p/64] + p%64; token t also attends to the n_path[t] <= 4 cache rows
 * path_rows[t][0..], and sees prefix positions < vis[t] (vis[t] = P for tree nodes, t+1 for a
 * causal prefill).  out bf16 [T][H*hd].  d_part: fp32 scratch of atspeed_op_attention_scratch(T,H,hd,P). */
size_t atspeed_op_attention_scratch(int T, int n_heads, int head_dim, int P);
atspeed_status atspeed_op_attention(atspeed_stream stream, const void *d_q, const void *d_kcache, const void *d_vcache,
                                    int cache_rows, int T, int n_heads, int head_dim, int P, const int32_t *h_pages,
                                    const int32_t *h_vis, const int32_t *h_path_rows, const int32_t *h_n_path,
                                    void *d_out, void *d_part);

#ifdef __cplusplus
}
#endif
#endif /* ATSPEED_H_ */
