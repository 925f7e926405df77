/*
 * presto.h - C ABI of the PRESTO tree draft-and-verify step on one GB300 (sm_103a).
 *
 * One round of tree-based diffusion speculative decoding (PRESTO: prefix-aligned
 * scoring and priority-based tree search):
 *
 *   presto_topk             per-position log-softmax and top-k of the drafter logits
 *   presto_topk_entropy     the same, plus each row's entropy and adaptive lambda_d
 *   presto_topk_slots       the same over the mask slots of the accepted node
 *                           (self-speculative rounds)
 *   presto_score_build_tree prefix-aligned scores + best-first tree up to N nodes
 *                           (_ex: beam search / printed Alg. 2, per-position lambda;
 *                           _mask: the tree mask and position ids in the same kernel)
 *   presto_tree_mask        ancestor bitmask and position ids of the tree tokens
 *   presto_tree_attention   tree-masked GQA attention against the KV-cache prefix
 *   presto_accept           longest accepted root path under greedy verification
 *
 * Conventions shared by every call
 *   - All array pointers are DEVICE pointers owned by the caller.  The library never
 *     allocates, frees or synchronises; each call only enqueues work on `stream`
 *     (a cudaStream_t; NULL is the legacy default stream) and returns.
 *   - Arrays are dense, row-major (C order) with the shapes given below, unless a
 *     stride argument says otherwise.
 *   - Return value: PRESTO_OK, or a negative PRESTO_ERR_* code found on the host
 *     before anything is enqueued (arguments, limits, workspace size), or
 *     PRESTO_ERR_CUDA when a launch fails (cudaGetLastError).
 *   - `dev_status` (nullable) points to one device int32.  Kernels OR PRESTO_DEV_*
 *     bits into it when they meet bad data (an out-of-range parent or token, a
 *     kv_len above Tmax, ...) or a bounded wait that ran out; they never trap.
 *     The caller clears it and reads it back when it wants to check.
 *   - Workspaces are device scratch of at least the size the matching
 *     presto_*_workspace() query returns (256-byte aligned).  Their contents on
 *     entry do not matter.  Two calls that run at the same time need two
 *     workspaces.
 *   - Limits: V < 2^18, 1 <= L <= 63, 1 <= b <= k <= 16, 1 <= N <= 1024 (these let
 *     the tree-order key pack into 64 bits: S, depth, the token's rank among its
 *     depth's k candidates, and a 22-bit parent field), D in {64, 128},
 *     Hq % Hkv == 0 with Hq / Hkv a power of two <= 128.
 *
 * Sizes: B batch (sequences), L drafter block length (tree depth limit), V vocab,
 * k candidates per position, b branching factor, N node budget including the root,
 * Tmax KV-cache capacity, kv_len[b] <= Tmax committed tokens of sequence b,
 * Hq / Hkv query / key-value heads, D head dim.
 */
#ifndef PRESTO_H
#define PRESTO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* presto_stream_t;  /* same type as cudaStream_t */

/* ---- host status codes ---------------------------------------------------- */
#define PRESTO_OK 0
#define PRESTO_ERR_INVALID_ARG (-1)   /* null pointer, bad size or dtype          */
#define PRESTO_ERR_UNSUPPORTED (-2)   /* a documented limit is exceeded           */
#define PRESTO_ERR_CUDA (-3)          /* a CUDA call or kernel launch failed      */
#define PRESTO_ERR_WORKSPACE (-4)     /* workspace missing or too small           */

/* ---- device status bits (ORed into *dev_status) --------------------------- */
#define PRESTO_DEV_BAD_PARENT 0x1     /* parent index not in [0, node index)      */
#define PRESTO_DEV_BAD_TOKEN 0x2      /* token id outside [0, V) / [0, 2^18)      */
#define PRESTO_DEV_BAD_KVLEN 0x4      /* kv_len < 0 or kv_len > Tmax              */
#define PRESTO_DEV_BAD_NNODES 0x8     /* n_nodes outside [1, N]                   */
#define PRESTO_DEV_POSITIVE_SCORE 0x10 /* a token score s > 0 (log-probs must be <= 0) */
#define PRESTO_DEV_TIMEOUT 0x20       /* a bounded in-kernel wait ran out         */
#define PRESTO_DEV_DUP_SIBLING 0x40   /* two candidates of one position share a token */
#define PRESTO_DEV_TABLE_FULL 0x80    /* n-gram insert found no free slot         */
#define PRESTO_DEV_NONFINITE 0x100    /* a logits row has no finite maximum       */
#define PRESTO_DEV_BAD_PATH 0x200     /* accept_len / accept_path entry out of range */
#define PRESTO_DEV_BOUNDS 0x400       /* an index failed a bounds check of a debug build
                                         (built with PRESTO_CHECKS); the access was skipped */

/* ---- element types -------------------------------------------------------- */
#define PRESTO_F32 0
#define PRESTO_BF16 1

/* Human-readable name of a PRESTO_OK / PRESTO_ERR_* code (static string). */
const char* presto_status_string(int status);

/* ABI version: (major << 16) | minor. */
/* Build flags of the loaded library: PRESTO_BUILD_CHECKS when it was compiled with
 * device-side bounds checks (-DPRESTO_CHECKS; a debug build: every data-dependent index
 * into a buffer the kernels write or a table they read is checked, and a failing one
 * reports PRESTO_DEV_BOUNDS and skips the access instead of faulting). */
#define PRESTO_BUILD_CHECKS 0x1
int presto_build_flags(void);
int presto_version(void);

/*
 * presto_selftest_wait_timeout - a diagnostic with no counterpart in the paper: it
 * exercises the bounded in-kernel waits.  One GPU thread waits up to wait_cycles SM
 * cycles (0 <= wait_cycles <= about 2e9, the library's own limit, roughly a
 * second) for a barrier phase that nothing completes; the wait runs out, ORs
 * PRESTO_DEV_TIMEOUT into *dev_status (device int32, required) and the kernel
 * returns normally, leaving the context usable.  Enqueued on `stream`.
 */
int presto_selftest_wait_timeout(int32_t* dev_status, long long wait_cycles,
                                 presto_stream_t stream);

/*
 * presto_topk - per-row log-softmax and top-k (the drafter's position-wise
 * marginals q_d of §2.3, Eq. marginal-surrogate; "extracts top-k diffusion
 * candidates", §4.3; k = 10 in §5.1).
 *
 *   logits      [B*L rows, row_stride elements]  dtype PRESTO_F32 or PRESTO_BF16;
 *               row r = b*L + (d-1) holds position d of sequence b; only the
 *               first V entries of a row are read.  Values must be finite or -inf.
 *   topk_ids    [B, L, k] int32 out: the k largest logits of each row in
 *               descending order; equal values are ordered by lower token id.
 *   topk_logq   [B, L, k] float32 out: log q_d(t) = x_t - log sum_v exp(x_v).
 *   lse         [B, L] float32 out, nullable: log sum_v exp(x_v).
 *   ws          presto_topk_workspace(B, L, V, k) bytes (currently 256 for every
 *               shape and unused: a row's spans merge inside one thread-block
 *               cluster; the argument is kept so that a plan may use it).
 *   dev_status  nullable; PRESTO_DEV_NONFINITE when a row has no finite maximum.
 * One pass over the logits; accumulation in float32.  The base pointer must be
 * aligned to the element size; rows need not be 16-byte aligned.
 */
size_t presto_topk_workspace(int B, int L, int V, int k);
int presto_topk(const void* logits, int dtype, int B, int L, int V, long long row_stride,
                int k, int32_t* topk_ids, float* topk_logq, float* lse, void* ws,
                size_t ws_bytes, int32_t* dev_status, presto_stream_t stream);

/*
 * presto_topk_entropy - presto_topk that also yields each row's entropy and the
 * entropy-adaptive lambda_d of App. F, in the same single pass over the logits.
 *
 *   H_d = -sum_w q_d(w) log q_d(w)  (nats; q_d the row's softmax, §2.3)
 *   lambda_d(H_d) = beta * H_d / (H_d + C)
 *
 *   beta, C     > 0 and finite when lambda_d is given (the largest correction
 *               strength and the stabilising constant; the paper fixes neither).
 *   entropy     [B, L] float32 out, nullable: H_d of every row.
 *   lambda_d    [B, L] float32 out, nullable: lambda_d(H_d), float32 with correctly
 *               rounded multiply, add and divide; it is the layout that
 *               presto_score_build_tree_ex takes as its lambda_d.
 * At least one of entropy, lambda_d is non-null.  Every other argument and result
 * is as presto_topk.  Where presto_topk reports PRESTO_DEV_NONFINITE for a row,
 * its entropy and lambda_d are unspecified.
 */
int presto_topk_entropy(const void* logits, int dtype, int B, int L, int V,
                        long long row_stride, int k, float beta, float C, int32_t* topk_ids,
                        float* topk_logq, float* lse, float* entropy, float* lambda_d, void* ws,
                        size_t ws_bytes, int32_t* dev_status, presto_stream_t stream);

/*
 * presto_topk_slots - presto_topk over the mask slots of the accepted path, for
 * self-speculative rounds (App. C (II)): one forward of the dLLM verified the
 * previous tree and denoised a block of mask slots attached to every one of its
 * nodes; only the slots of the deepest accepted node a*_b stay valid, and they are
 * the next round's drafter rows.
 *
 *   slot_logits  [B, n_prev, n_slots, row_stride] dtype PRESTO_F32 or PRESTO_BF16:
 *                the logits at slot j of node i of sequence b (first V entries
 *                of a row are read).  Only the rows named below are read; the
 *                slots of every other node are never touched.
 *   accept_len, accept_path  [B], [B, path_len] int32, as written by presto_accept
 *                (path_len = its L + 1): a*_b = accept_path[b][accept_len[b]].
 *                Read on the device after the kernel before this one on `stream`
 *                finishes, so presto_accept may run just before with no host sync.
 *   slot_offset, L  drafter row j (depth j + 1 of the next tree) is slot
 *                slot_offset + j of a*_b; 0 <= slot_offset <= n_slots - L.  Which
 *                slot holds the position after the bonus token depends on the model
 *                (the paper does not fix it): 1 when slot j of a node predicts the
 *                token j + 1 places after it, since the bonus takes the first place.
 *   node_token, bonus, ctx2_next  nullable together: [B, n_prev], [B] int32 in
 *                (presto_score_build_tree's node_token and presto_accept's bonus),
 *                [B, 2] int32 out = (node_token[b][a*_b], bonus[b]), the last two
 *                committed tokens, i.e. the next round's ctx2.  Must not alias the
 *                inputs.
 *   topk_ids, topk_logq, lse, ws, dev_status  as presto_topk with B x L rows.
 *                PRESTO_DEV_BAD_PATH when accept_len[b] is outside [0, path_len) or
 *                the node it selects is outside [0, n_prev); that sequence then
 *                reads the root's slots.
 */
int presto_topk_slots(const void* slot_logits, int dtype, int B, int n_prev, int n_slots, int V,
                      long long row_stride, const int32_t* accept_len,
                      const int32_t* accept_path, int path_len, int slot_offset, int L, int k,
                      const int32_t* node_token, const int32_t* bonus, int32_t* ctx2_next,
                      int32_t* topk_ids, float* topk_logq, float* lse, void* ws, size_t ws_bytes,
                      int32_t* dev_status, presto_stream_t stream);

/*
 * Trigram prefix signal rho_d(t | t_{d-2}, t_{d-1}) (§4.1; the paper instantiates
 * it with an n = 3 n-gram model, §5.1).  An open-addressing hash table in device
 * memory with 2^log2_cap slots:
 *   keys    [2^log2_cap] uint64, key = presto_ngram3_key(a, b, t); empty slots hold
 *           PRESTO_NGRAM3_EMPTY.
 *   logrho  [2^log2_cap] float32 log rho values (must be <= 0).
 * A lookup that finds no key returns miss_logrho (<= 0).  The struct itself is a
 * host value; its pointers are device pointers owned by the caller.
 */
#define PRESTO_NGRAM3_EMPTY 0xFFFFFFFFFFFFFFFFull
typedef struct {
  uint64_t* keys;
  float* logrho;
  uint32_t log2_cap;
  float miss_logrho;
} presto_ngram3;

static inline uint64_t presto_ngram3_key(uint32_t a, uint32_t b, uint32_t t) {
  return ((uint64_t)a << 36) | ((uint64_t)b << 18) | (uint64_t)t;
}

/* Mark every slot empty.  log2_cap in [4, 30]. */
int presto_ngram3_clear(const presto_ngram3* table, presto_stream_t stream);

/* Insert n (key, logrho) pairs (device arrays).  Keys must be unique and below
 * 2^54; a key already present keeps one of its values.  A full table sets
 * PRESTO_DEV_TABLE_FULL.  Keep the load factor below ~0.5 for short probes. */
int presto_ngram3_insert(const presto_ngram3* table, const uint64_t* keys,
                         const float* logrho, int n, int32_t* dev_status,
                         presto_stream_t stream);

/*
 * presto_score_build_tree - prefix-aligned scoring and best-first tree search.
 *
 * Score (§4.1, Eq. path-score): s_{d,t}(c_d) = log q_d(t) + lambda * log rho(t |
 * t_{d-2}, t_{d-1}), the context taken from (ctx2[b,0], ctx2[b,1], t_1, ...,
 * t_{d-1}); computed in float32 as fl(fl(lambda * log rho) + log q).  With
 * ngram == NULL the score is log q (marginal-only scoring, Eq.
 * marginal-surrogate).  Path score S(child) = fl(S(parent) + s); S(root) = 0.
 *
 * Tree (§4.2, Alg. 2 with a node committed when it is popped): node 0 is the root
 * (token ctx2[b,1], depth 0); a node at depth d < L has as children the top-b of
 * the k candidates of depth d+1 ranked by (s desc, token asc); the result is the
 * N nodes of this candidate tree that come first in the order
 *   S desc, depth asc, token asc, parent index asc,
 * stored in that order (so parent index < child index), which is the top-N
 * prefix-closed set of §4.2 whenever every s <= 0.  Fewer than N nodes when the
 * candidate tree is smaller.
 *
 *   topk_ids, topk_logq  [B, L, k] as written by presto_topk (row d-1 = depth d);
 *                        tokens of one row must be distinct.
 *   ctx2        [B, 2] int32: the last two committed tokens; ctx2[b,1] is the root.
 *   ngram       host pointer to the table descriptor, or NULL.
 *   lambda      >= 0 (0.2 in §5.1).
 *   node_token  [B, N] int32 out  (-1 in unused slots)
 *   node_parent [B, N] int32 out  (-1 for the root and unused slots)
 *   node_depth  [B, N] int32 out  (-1 in unused slots)
 *   node_score  [B, N] float32 out S (-inf in unused slots)
 *   n_nodes     [B] int32 out
 *   ws          presto_build_workspace(B, L, k, N) bytes.
 */
size_t presto_build_workspace(int B, int L, int k, int N);
int presto_score_build_tree(const int32_t* topk_ids, const float* topk_logq, int B, int L,
                            int k, int b, const int32_t* ctx2, const presto_ngram3* ngram,
                            float lambda, int N, int32_t* node_token, int32_t* node_parent,
                            int32_t* node_depth, float* node_score, int32_t* n_nodes,
                            void* ws, size_t ws_bytes, int32_t* dev_status,
                            presto_stream_t stream);

/*
 * presto_score_build_tree_ex - presto_score_build_tree with a choice of search
 * policy (§4.2) and of a per-position lambda.
 *
 *   lambda_d    nullable [B, L] float32 (device): lambda of each drafter row (row d-1
 *               scores depth d), e.g. the entropy-adaptive lambda_d(H_d) of App. F
 *               written by presto_topk_entropy; NULL uses `lambda` everywhere.
 *               Values must be >= 0.
 *   policy      PRESTO_SEARCH_BEST_FIRST: as presto_score_build_tree (Alg. 2 with a
 *                 node committed when it is popped: the N best nodes of the
 *                 candidate tree).
 *               PRESTO_SEARCH_BEAM: beam search with global retention (Alg. 1): from
 *                 the beam {root}, while the tree T holds fewer than N nodes, every
 *                 beam node gains its top-b children (all join T) and the
 *                 `beam_width` best of them form the next beam; the result is the
 *                 N best nodes of T.  The paper's default (beam width 10, §5.1).
 *               PRESTO_SEARCH_EAGER: Alg. 2 as printed: pop the best frontier node,
 *                 add all its children to T, until |T| >= N; the N best nodes of T.
 *   beam_width  >= 1 (used by PRESTO_SEARCH_BEAM; <= 1024).
 * "Best" is always the order S desc, depth asc, token asc, parent index asc, and
 * the output is stored in that order (parent index < child index).
 *   ws          presto_build_workspace_ex(B, L, k, N, beam_width) bytes.
 */
#define PRESTO_SEARCH_BEST_FIRST 0
#define PRESTO_SEARCH_BEAM 1
#define PRESTO_SEARCH_EAGER 2
size_t presto_build_workspace_ex(int B, int L, int k, int N, int beam_width);
int presto_score_build_tree_ex(const int32_t* topk_ids, const float* topk_logq, int B, int L,
                               int k, int b, const int32_t* ctx2, const presto_ngram3* ngram,
                               float lambda, const float* lambda_d, int policy, int beam_width,
                               int N, int32_t* node_token, int32_t* node_parent,
                               int32_t* node_depth, float* node_score, int32_t* n_nodes,
                               void* ws, size_t ws_bytes, int32_t* dev_status,
                               presto_stream_t stream);

/*
 * presto_score_build_tree_mask - presto_score_build_tree_ex that also writes the
 * tree-attention mask and position ids of the tree it builds, exactly as
 * presto_tree_mask computes them (§4.3; App. C (I), (IV)), in the same kernel: one
 * launch and one dependency fewer per round.
 *
 *   kv_len, mask, pos_ids  as presto_tree_mask's ([B] int32 in; [B, N, ceil(N/32)]
 *               uint32 and [B, N] int32 out); non-null together.
 * Every other argument is as presto_score_build_tree_ex; PRESTO_DEV_BAD_KVLEN when
 * kv_len[b] < 0.
 */
int presto_score_build_tree_mask(const int32_t* topk_ids, const float* topk_logq, int B, int L,
                                 int k, int b, const int32_t* ctx2, const presto_ngram3* ngram,
                                 float lambda, const float* lambda_d, int policy, int beam_width,
                                 int N, int32_t* node_token, int32_t* node_parent,
                                 int32_t* node_depth, float* node_score, int32_t* n_nodes,
                                 const int32_t* kv_len, uint32_t* mask, int32_t* pos_ids,
                                 void* ws, size_t ws_bytes, int32_t* dev_status,
                                 presto_stream_t stream);

/*
 * presto_score_build_tree_noalloc - presto_score_build_tree_mask for callers that
 * cannot allocate device memory.  The paper has no counterpart: this is a
 * deployment variant of the same kernel.
 *
 * Some callers have no way to hand this library a workspace: a plugin inside a
 * serving framework whose allocator owns all of the GPU's memory, a C program with
 * no allocator at all, or a latency-critical loop that must never block in
 * cudaMalloc (which can synchronise the device and can fail once memory is
 * fragmented).  Large node budgets (N = 512, 1024) make the tree build keep its
 * level-selection scratch and child tables in global memory; this entry point keeps
 * them in a fixed device array inside the library instead, of
 * PRESTO_BUILD_STATIC_SCRATCH_BYTES (1 MiB).  Every GPU that loads the library
 * holds that array until the process exits.  It fits, for example, two sequences at
 * N = 1024 (k = b = 8, with a trigram table) or sixteen at N = 512.
 *
 * Arguments and results are those of presto_score_build_tree_mask without ws and
 * ws_bytes.  Returns PRESTO_ERR_UNSUPPORTED, enqueueing nothing, when the call
 * needs more scratch than the array holds (B times the per-sequence need of the
 * shape; see presto_build_workspace_ex).  Calls no cudaMalloc, cudaFree or other
 * allocating routine.  The first call on a device looks up the array's device
 * address (cudaGetSymbolAddress, with that device current) and caches it; make that
 * first call before any stream capture.  All calls on a device share the one array
 * and it keeps the last call's contents; nothing in it has to start at zero (every
 * call writes each scratch entry before reading it).  Calls whose kernels may
 * overlap on the GPU (different streams with no ordering between them) race on the
 * array: order them on one stream.
 */
#define PRESTO_BUILD_STATIC_SCRATCH_BYTES (1u << 20)
int presto_score_build_tree_noalloc(const int32_t* topk_ids, const float* topk_logq, int B,
                                    int L, int k, int b, const int32_t* ctx2,
                                    const presto_ngram3* ngram, float lambda,
                                    const float* lambda_d, int policy, int beam_width, int N,
                                    int32_t* node_token, int32_t* node_parent,
                                    int32_t* node_depth, float* node_score, int32_t* n_nodes,
                                    const int32_t* kv_len, uint32_t* mask, int32_t* pos_ids,
                                    int32_t* dev_status, presto_stream_t stream);

/*
 * presto_tree_mask - tree attention mask and position ids (§4.3 and App. C (I),
 * (IV): each draft token attends to its ancestors in the draft tree).
 *
 *   node_parent, node_depth [B, N], n_nodes [B], kv_len [B]  int32 inputs.
 *   mask    [B, N, ceil(N/32)] uint32 out: bit j of row i is set iff node j is node
 *           i or one of its ancestors; rows of unused slots are 0.
 *   pos_ids [B, N] int32 out: kv_len[b] + depth(i); -1 in unused slots.
 */
int presto_tree_mask(const int32_t* node_parent, const int32_t* node_depth,
                     const int32_t* n_nodes, const int32_t* kv_len, int B, int N,
                     uint32_t* mask, int32_t* pos_ids, int32_t* dev_status,
                     presto_stream_t stream);

/*
 * presto_tree_attention - one layer's tree-masked GQA attention of the N tree
 * tokens (target verification with a tree-structured mask, §5.1; App. C (I)).
 *
 * out[b,i,h] = sum_j softmax_j(sm_scale * <q[b,i,h], key_j>) value_j over
 *   - the committed prefix: key_j = k_cache[b,g,j], value_j = v_cache[b,g,j],
 *     j < kv_len[b], and
 *   - the tree: key = k_tree[b,j,g], value = v_tree[b,j,g] for every j with bit j
 *     of mask[b,i] set,
 * with g = h / (Hq/Hkv).  bf16 inputs, float32 softmax and accumulation, bf16 out.
 *
 *   q        [B, N, Hq, D] bf16 (positions / RoPE already applied)
 *   k_cache, v_cache [B, Hkv, Tmax, D] bf16; rows >= kv_len[b] get zero weight
 *   kv_len   [B] int32 in [0, Tmax]
 *   k_tree, v_tree   [B, N, Hkv, D] bf16
 *   mask     [B, N, ceil(N/32)] uint32 from presto_tree_mask
 *   n_nodes  [B] int32; rows i >= n_nodes[b] are written as zeros (lse -inf)
 *   out      [B, N, Hq, D] bf16 out
 *   lse      [B, N, Hq] float32 out, nullable: natural-log softmax denominator
 *   ws       presto_attn_workspace(B, N, Hq, Hkv, D, Tmax) bytes (for the current
 *            device).
 * All base pointers must be 16-byte aligned.  Rows of k_cache / v_cache at or past
 * kv_len[b], and rows of k_tree / v_tree at or past n_nodes[b] (up to N), get zero
 * weight but are read with the 128-key tile that holds them: they must hold finite
 * values (a zero weight times a NaN is a NaN).
 * Under programmatic dependent launch, the KV cache and kv_len may be read before the
 * kernel waits for the previous kernels on the stream (no kernel of a round writes
 * them: the caller must not write them from a kernel that lets this one start early);
 * q, k_tree, v_tree, mask and n_nodes are read after that wait.
 */
size_t presto_attn_workspace(int B, int N, int Hq, int Hkv, int D, int Tmax);
/* Kernels one presto_tree_attention call of these shapes launches on the current
 * device: 2 when its KV splits are merged by a second kernel, else 1; 0 for shapes
 * the call refuses (the checks of presto_attn_workspace). */
int presto_attn_launches(int B, int N, int Hq, int Hkv, int D, int Tmax);
int presto_tree_attention(const void* q, const void* k_cache, const void* v_cache,
                          const int32_t* kv_len, int Tmax, const void* k_tree,
                          const void* v_tree, const uint32_t* mask, const int32_t* n_nodes,
                          int B, int N, int Hq, int Hkv, int D, float sm_scale, void* out,
                          float* lse, void* ws, size_t ws_bytes, int32_t* dev_status,
                          presto_stream_t stream);

/*
 * presto_accept - greedy (temperature 0) verification of the tree (§2.1: tokens
 * are accepted left to right until the first mismatch; App. A alpha_T(P); App. C
 * (I): the position after the last accepted token takes the target's own token).
 *
 *   node_token, node_parent, node_depth [B, N], n_nodes [B], mask [B, N, ceil(N/32)]
 *   target_token [B, N] int32: the target model's greedy next token after node i.
 *   accept_len  [B] int32 out: depth of the deepest node whose every ancestor-or-self
 *               j != 0 has node_token[j] == target_token[parent(j)].
 *   accept_path [B, L+1] int32 out: node ids root..deepest, then -1.
 *   bonus       [B] int32 out: target_token of the deepest accepted node.
 * The ancestor sets are walked through node_parent (the sets the mask rows hold), so
 * node_depth and mask are not read; they stay in the signature (non-null) so that a
 * caller can pass the round's arrays unchanged.
 */
int presto_accept(const int32_t* node_token, const int32_t* node_parent,
                  const int32_t* node_depth, const uint32_t* mask, const int32_t* n_nodes,
                  const int32_t* target_token, int B, int N, int L, int32_t* accept_len,
                  int32_t* accept_path, int32_t* bonus, int32_t* dev_status,
                  presto_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* PRESTO_H */
