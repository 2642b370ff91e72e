/*
 * seed.h -- C ABI of the SEED draft/verify attention path for NVIDIA GB300
 * (sm_103a).
 *
 * SEED (Self-Speculative Decoding via Implicit Encoder-Decoder) drafts tokens
 * with the last decoder layers of the model, fed raw token embeddings and
 * attending to the deep KV cache the previous verification left behind
 * (Sec. 4.1), then verifies d drafts with one (d+1)-token pass of the full
 * model and keeps the greedy longest matching prefix plus a bonus token
 * (Alg. 2).  This library implements the memory-bound steps of that loop:
 *
 *   seed_draft_kv_append / seed_draft_attn   -- one draft step, per decoder layer
 *   seed_kv_append       / seed_verify_attn  -- the verify pass, per layer
 *   seed_accept_commit                       -- acceptance and cache commit
 *
 * Conventions shared by every call
 * --------------------------------
 * - All tensor pointers are DEVICE pointers, row-major, densely packed, owned
 *   by the caller; the library never allocates, frees or synchronises, and
 *   keeps no state between calls.  Calls are asynchronous on `stream` (a
 *   cudaStream_t; NULL is the legacy default stream) and are safe to call
 *   from several host threads on different streams.
 * - bf16 tensors hold IEEE bfloat16 bit patterns; f32 outputs are IEEE float.
 * - Host-side checks (null pointers, unsupported shapes, a too-small
 *   workspace) return a status synchronously and launch nothing.
 * - Data-dependent checks run on the device: a violation ORs a SEED_DEVERR_*
 *   bit into *err_flag (an int32 in device memory, which the caller zeroes and
 *   reads) and the offending work is skipped.  No kernel ever traps; outputs
 *   of a call that raised a device error are unspecified, but no memory
 *   outside the arguments is touched.
 * - KV cache of one layer (a "paged" cache): K and V are each
 *   [num_pages, hkv, page_size, head_dim] bf16.  Logical position `pos` of
 *   sequence b lives in page page_table[b * max_pages + pos / page_size] at
 *   offset pos % page_size.  A contiguous cache is the identity page order.
 * - GQA: query head h reads KV head h / (hq / hkv).
 * - Attention outputs are f32; lse is the natural-log sum of exp(scores).
 */
#ifndef SEED_H_
#define SEED_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SEED_ABI_VERSION 4
#define SEED_MAX_KMAX 31        /* largest supported draft length d (32 rows per sequence) */

typedef enum {
  SEED_OK = 0,
  SEED_ERR_NULL = 1,          /* a required pointer is NULL                    */
  SEED_ERR_SHAPE = 2,         /* batch < 0, hq % hkv != 0, kmax out of range   */
  SEED_ERR_RANGE = 3,         /* max_pages / num_pages out of range            */
  SEED_ERR_UNSUPPORTED = 4,   /* head_dim, group size or page_size not built   */
  SEED_ERR_CUDA = 5,          /* a CUDA runtime call failed (launch error)     */
  SEED_ERR_WORKSPACE = 6,     /* workspace too small or misaligned             */
  SEED_ERR_SCRATCH_LIMIT = 7  /* problem too large for the built-in scratch    */
} seed_status_t;

/* Device error bits (OR-ed into *err_flag). */
#define SEED_DEVERR_CTX_LEN   1   /* ctx_len < 0, or rows past max_pages*page_size */
#define SEED_DEVERR_DRAFT_LEN 2   /* draft_len outside [0, kmax]                    */
#define SEED_DEVERR_NQ        4   /* n_q / n_new outside [0, kmax+1]                */
#define SEED_DEVERR_PAGE      8   /* page id outside [0, num_pages)                 */
#define SEED_DEVERR_KB        16  /* k_b outside [0, kmax]                          */
#define SEED_DEVERR_WORKSPACE 32  /* more work units than the workspace holds       */
#define SEED_DEVERR_TIMEOUT   64  /* a bounded on-chip wait gave up (never expected) */
#define SEED_DEVERR_TREE      128 /* a draft tree's parents or accepted path are invalid */
#define SEED_DEVERR_TOKEN     256 /* a token id outside [0, vocab)                      */

/* Shapes of one model's attention.  Supported: head_dim in {64, 128};
 * hq / hkv in {1, 2, 4, 8}; page_size == 16; 1 <= kmax <= SEED_MAX_KMAX.
 * scale == 0 selects 1/sqrt(head_dim) (the paper leaves the softmax scale to
 * the base model; this is the usual one). */
typedef struct {
  int32_t hq;
  int32_t hkv;
  int32_t head_dim;
  int32_t page_size;
  int32_t kmax;
  float scale;
} seed_cfg_t;

/* One layer's paged KV cache.  k, v: bf16 [num_pages, hkv, page_size,
 * head_dim] (written only by the *_append calls); page_table: int32
 * [batch, max_pages]. */
typedef struct {
  void* k;
  void* v;
  const int32_t* page_table;
  int32_t max_pages;
  int32_t num_pages;
} seed_kv_t;

int32_t seed_abi_version(void);
const char* seed_status_string(seed_status_t status);

/* Bytes of device workspace that seed_draft_attn and seed_verify_attn need
 * for `batch` sequences with this cfg (independent of lengths).  The
 * workspace must be 256-byte aligned and ZERO-FILLED before its first use;
 * every call leaves it zero-filled again (it holds split partials and
 * per-(sequence, KV head) arrival counters).  Returns 0 for an invalid cfg. */
size_t seed_workspace_bytes(const seed_cfg_t* cfg, int32_t batch);

/* Draft step, cache side (Alg. 2, drafting phase; Sec. 4.1 "Cheap drafting"):
 * store the K/V row the drafter computed for X_draft[i-1] in one decoder layer
 * as row i-1 of that layer's draft scratch.
 *   k_new, v_new   bf16 [batch, hkv, head_dim]
 *   draft_lens     int32 [batch]: i, the number of draft rows after this
 *                  append (1..kmax); 0 skips the sequence
 *   draft_k/v      bf16 [batch, hkv, kmax, head_dim], written at row i-1
 * Device errors: SEED_DEVERR_DRAFT_LEN. */
seed_status_t seed_draft_kv_append(const seed_cfg_t* cfg, int32_t batch,
                                   const void* k_new, const void* v_new,
                                   const int32_t* draft_lens,
                                   void* draft_k, void* draft_v,
                                   int32_t* err_flag, void* stream);

/* Draft attention (Sec. 4.1 eq. for X_{n+1} from f_dec(H^0_n, KV^dec_{<n});
 * Alg. 2 drafting phase): for each sequence b and query head h, softmax
 * attention of q[b, h] over the ctx_lens[b] committed rows of this decoder
 * layer's cache (the deep KV the last verification wrote) followed by the
 * draft_lens[b] rows of the draft scratch (X_draft[0..i-1], the query's own
 * row included).
 *   q            bf16 [batch, hq, head_dim]
 *   ctx_kv       this layer's cache (read only)
 *   draft_k/v    bf16 [batch, hkv, kmax, head_dim]
 *   ctx_lens     int32 [batch] >= 0
 *   draft_lens   int32 [batch] in [0, kmax]; 0 skips the sequence (its out
 *                and lse rows are left untouched)
 *   out          f32 [batch, hq, head_dim]
 *   lse          f32 [batch, hq], or NULL
 *   ws           workspace of ws_bytes >= seed_workspace_bytes(cfg, batch)
 * Device errors: SEED_DEVERR_CTX_LEN, _DRAFT_LEN, _PAGE, _WORKSPACE. */
seed_status_t seed_draft_attn(const seed_cfg_t* cfg, int32_t batch, const void* q,
                              seed_kv_t ctx_kv, const void* draft_k, const void* draft_v,
                              const int32_t* ctx_lens, const int32_t* draft_lens,
                              float* out, float* lse, void* ws, size_t ws_bytes,
                              int32_t* err_flag, void* stream);

/* Verify pass, cache side (Alg. 2 verification phase; Sec. 4.1 "Verification
 * already does the encoder's work"): write the n_new[b] K/V rows the verifier
 * computed for X_draft[0..n_new-1] at logical positions ctx_lens[b] ..
 * ctx_lens[b] + n_new[b] - 1 of this layer's cache.
 *   k_new, v_new  bf16 [batch, kmax+1, hkv, head_dim]
 *   n_new         int32 [batch] in [0, kmax+1]
 *   ctx_lens      int32 [batch] (not modified)
 * Device errors: SEED_DEVERR_CTX_LEN, _NQ, _PAGE. */
seed_status_t seed_kv_append(const seed_cfg_t* cfg, int32_t batch, seed_kv_t kv,
                             const void* k_new, const void* v_new, const int32_t* n_new,
                             const int32_t* ctx_lens, int32_t* err_flag, void* stream);

/* Verify attention (Alg. 2 verification phase: (f_dec o f_enc) over
 * X_draft[0..d] with the cache KV_{1..t-1}): query j of sequence b (token
 * X_draft[j], j < n_q[b]) attends to rows 0 .. ctx_lens[b] + j of this
 * layer's cache, which already holds the n_q[b] new rows (seed_kv_append):
 * causal among the new rows, all committed rows visible.
 *   q         bf16 [batch, kmax+1, hq, head_dim]
 *   n_q       int32 [batch] in [0, kmax+1] (k_b + 1; 0 skips the sequence)
 *   kv        this layer's cache (read only)
 *   ctx_lens  int32 [batch]: committed rows before the new ones
 *   out       f32 [batch, kmax+1, hq, head_dim] (rows j >= n_q untouched)
 *   lse       f32 [batch, kmax+1, hq], or NULL
 * Device errors: SEED_DEVERR_CTX_LEN, _NQ, _PAGE, _WORKSPACE. */
seed_status_t seed_verify_attn(const seed_cfg_t* cfg, int32_t batch, const void* q,
                               const int32_t* n_q, seed_kv_t kv, const int32_t* ctx_lens,
                               float* out, float* lse, void* ws, size_t ws_bytes,
                               int32_t* err_flag, void* stream);

/* Which kernel seed_draft_attn (draft != 0) or seed_verify_attn (draft == 0)
 * runs for this cfg, batch and page-table width max_pages on the current
 * device (the calls choose the same way; for diagnostics and tests):
 *   SEED_ROUTE_CUDA_CORE   split-KV kernel on CUDA cores
 *   SEED_ROUTE_TC_ROWS     tensor cores, the query rows of a KV head as MMA
 *                          rows (head_dim 128, up to 128 rows)
 *   SEED_ROUTE_TC_KEYS     tensor cores, the keys as MMA rows (head_dim 64,
 *                          up to 48 query rows)
 *   SEED_ROUTE_CLUSTER_8, _12, _16
 *                          few (sequence, KV head) pairs and short page tables
 *                          (head_dim 128, up to 32 query rows): one cluster of
 *                          8, 12 or 16 CTAs per pair, merged on chip; the
 *                          largest cluster whose clusters all fit the device
 *                          at once and whose CTAs hold max_pages + 2 pages
 * seed_tree_verify_attn always takes a tensor-core route.  Returns -1 for an
 * invalid cfg, batch < 1 or max_pages < 1. */
typedef enum {
  SEED_ROUTE_CUDA_CORE = 0,
  SEED_ROUTE_TC_ROWS = 1,
  SEED_ROUTE_TC_KEYS = 2,
  SEED_ROUTE_CLUSTER_8 = 8,
  SEED_ROUTE_CLUSTER_12 = 12,
  SEED_ROUTE_CLUSTER_16 = 16
} seed_route_t;
int32_t seed_attn_route(const seed_cfg_t* cfg, int32_t batch, int32_t draft, int32_t max_pages);

/* Greedy acceptance and cache commit/rollback (Alg. 2, after verification):
 * n_b = number of leading i < k_b[b] with draft_ids[b,i] == target_ids[b,i];
 * tokens[b] = draft_ids[b, 0..n_b-1] then the bonus target_ids[b, n_b];
 * the rows of X_draft[0..n_b] (positions ctx_lens[b] .. ctx_lens[b]+n_b) are
 * committed and their physical slots (page * page_size + offset) reported;
 * rows past them are rolled back (left in place, never read again);
 * ctx_lens[b] += n_b + 1.
 *   draft_ids        int32 [batch, kmax]   (X_draft[1..kmax])
 *   target_ids       int32 [batch, kmax+1] (argmax p_1..p_{kmax+1})
 *   k_b              int32 [batch] in [0, kmax]
 *   page_table       int32 [batch, max_pages]
 *   ctx_lens         int32 [batch], updated in place
 *   accepted         int32 [batch]: n_b
 *   tokens           int32 [batch, kmax+1], -1 past n_b
 *   committed_slots  int32 [batch, kmax+1], -1 past n_b
 * Device errors: SEED_DEVERR_KB, _CTX_LEN (committed rows past capacity);
 * the sequence is then left unchanged. */
seed_status_t seed_accept_commit(int32_t batch, int32_t kmax, const int32_t* draft_ids,
                                 const int32_t* target_ids, const int32_t* k_b,
                                 const int32_t* page_table, int32_t max_pages,
                                 int32_t page_size, int32_t* ctx_lens, int32_t* accepted,
                                 int32_t* tokens, int32_t* committed_slots,
                                 int32_t* err_flag, void* stream);

/* ------------------------------------------------------------------------
 * Tree-based verification (Sec. D.1).  The drafter proposes a tree of
 * candidates instead of one chain; the verifier checks all of them in one
 * pass, each candidate seeing the verified prefix and its own ancestral path
 * only; the tree is then walked greedily from the root and the cache keeps
 * the accepted path.
 *
 * A tree of sequence b has n_nodes[b] <= kmax + 1 nodes, numbered so that
 * every node comes after its parent.  Node 0 is the root: the last verified
 * token (X_draft[0] of the linear case), whose row is not in the cache yet.
 * Node i's K/V row is written with seed_kv_append (n_new = n_nodes) at packed
 * position ctx_lens[b] + i; its model position, for position embeddings, is
 * ctx_lens[b] + depth(i).  One round is:
 *   per layer:  seed_kv_append, seed_tree_verify_attn
 *   then:       seed_tree_accept_commit (once), seed_tree_kv_compact (per layer)
 * ------------------------------------------------------------------------ */

/* Verify attention over a draft tree (Sec. D.1, tree-structured mask): node
 * j (j < n_nodes[b]) of sequence b attends to cache rows 0 .. ctx_lens[b]-1
 * and to the packed rows ctx_lens[b] + a of the nodes a whose bit is set in
 * anc[b, j] (its ancestors; the node's own bit is always added, bits at or
 * past n_nodes[b] are ignored).
 *   q         bf16 [batch, kmax+1, hq, head_dim] (row j = node j)
 *   n_nodes   int32 [batch] in [0, kmax+1] (0 skips the sequence)
 *   anc       uint32 [batch, kmax+1]: bit a of anc[b, j] = node a is an
 *             ancestor of node j
 *   others    as seed_verify_attn (same workspace size)
 * Built for head_dim 128 with (hq/hkv) * (kmax+1) <= 128 and for head_dim
 * 64 with (hq/hkv) * (kmax+1) <= 48; other shapes return
 * SEED_ERR_UNSUPPORTED.
 * Device errors: SEED_DEVERR_CTX_LEN, _NQ, _PAGE. */
seed_status_t seed_tree_verify_attn(const seed_cfg_t* cfg, int32_t batch, const void* q,
                                    const int32_t* n_nodes, const uint32_t* anc,
                                    seed_kv_t kv, const int32_t* ctx_lens,
                                    float* out, float* lse, void* ws, size_t ws_bytes,
                                    int32_t* err_flag, void* stream);

/* Greedy acceptance over a draft tree (Sec. D.1): from the root, take the
 * child of the current node whose token equals target_ids at the current
 * node (the lowest node index if several do), until no child matches.  n_b =
 * accepted drafts; tokens[b] = their tokens then the bonus target_ids[b, last
 * accepted node]; path[b, d] = node at depth d of the accepted path
 * (path[b, 0] = 0); committed_slots = slots of positions ctx_lens[b] ..
 * ctx_lens[b] + n_b (where seed_tree_kv_compact puts the path's rows);
 * ctx_lens[b] += n_b + 1.
 *   tok         int32 [batch, kmax+1]: node tokens (tok[b, 0] = root)
 *   parent      int32 [batch, kmax+1]: parent[b, i] < i for 1 <= i < n_nodes
 *   n_nodes     int32 [batch] in [1, kmax+1]
 *   target_ids  int32 [batch, kmax+1]: the verifier's argmax at each node
 *   accepted    int32 [batch]; tokens, path, committed_slots int32
 *               [batch, kmax+1], -1 past the used entries
 * Device errors: SEED_DEVERR_NQ (n_nodes), _TREE (a parent not before its
 * node), _CTX_LEN (the tree's rows past capacity); that sequence is then left
 * unchanged. */
seed_status_t seed_tree_accept_commit(int32_t batch, int32_t kmax, const int32_t* tok,
                                      const int32_t* parent, const int32_t* n_nodes,
                                      const int32_t* target_ids, const int32_t* page_table,
                                      int32_t max_pages, int32_t page_size, int32_t* ctx_lens,
                                      int32_t* accepted, int32_t* tokens, int32_t* path,
                                      int32_t* committed_slots, int32_t* err_flag,
                                      void* stream);

/* Cache side of the tree commit, per layer: moves the rows of the accepted
 * path from their packed positions L + path[b, d] to L + d (d = 1..n_b), with
 * L = ctx_lens[b] - accepted[b] - 1 (ctx_lens and accepted as
 * seed_tree_accept_commit left them).
 * Device errors: SEED_DEVERR_TREE (path not increasing from depth d on, or
 * past capacity), _CTX_LEN, _PAGE. */
seed_status_t seed_tree_kv_compact(const seed_cfg_t* cfg, int32_t batch, seed_kv_t kv,
                                   const int32_t* path, const int32_t* accepted,
                                   const int32_t* ctx_lens, int32_t* err_flag, void* stream);

/* ------------------------------------------------------------------------
 * Confidence-aware dynamic drafting (Sec. D.1).  After each draft step the
 * drafter's LM head gives a distribution p = softmax(W_out h) over the
 * vocabulary.  Its top-1 probability p0 sets how many sibling candidates the
 * tree gets at this step,
 *     k = 1 if p0 > 0.95, 3 if 0.8 < p0 <= 0.95, 5 if 0.5 < p0 <= 0.8, else 10,
 * and drafting goes on after a step only while p0 > tau (the step that falls
 * to p0 <= tau still adds its k candidates).
 * ------------------------------------------------------------------------ */
#define SEED_DRAFT_TOPK 10             /* candidates returned per sequence */
#define SEED_DRAFT_HEAD_MAX_BATCH 128  /* sequences per call */

/* Bytes of workspace seed_draft_head_topk needs for `batch` sequences (no
 * zeroing needed); 0 for a batch outside [1, SEED_DRAFT_HEAD_MAX_BATCH]. */
size_t seed_draft_head_workspace_bytes(int32_t batch);

/* The drafter's LM head with a fused softmax: for each sequence b, logits
 * z = W_out h[b] (no bias, no temperature) over the whole vocabulary, never
 * written out.
 *   h          bf16 [batch, d_model]: the drafter's final hidden states (after
 *              its output norm); d_model a multiple of 64
 *   w_out      bf16 [vocab, d_model]: the LM head, row v = token v
 *   tau        stop threshold
 *   ids        int32 [batch, 10]: the 10 most probable tokens, decreasing
 *              probability, equal logits in increasing id order
 *   probs      f32 [batch, 10]: their probabilities (probs[b, 0] = p0)
 *   n_sib      int32 [batch]: k by the rule above
 *   stop       int32 [batch]: 1 when p0 <= tau
 *   lse        f32 [batch]: natural log of sum_v exp(z_v), or NULL
 * Runs on the tensor cores (bf16 inputs, f32 accumulation).  batch <= 128,
 * vocab >= 10.  Device errors: SEED_DEVERR_TIMEOUT only. */
seed_status_t seed_draft_head_topk(int32_t batch, int32_t d_model, int32_t vocab,
                                   const void* h, const void* w_out, float tau,
                                   int32_t* ids, float* probs, int32_t* n_sib,
                                   int32_t* stop, float* lse, void* ws, size_t ws_bytes,
                                   int32_t* err_flag, void* stream);

/* ------------------------------------------------------------------------
 * The whole draft step on the device (Sec. 4.1 "cheap drafting"; the work per
 * draft token that the paper's computational-cost appendix counts: per
 * decoder layer W_Q, W_K, W_V, W_O and three MLP matrices, then the head).
 * The decoder layers are the model's last l - l' layers, in the pre-norm form
 * of the paper's Qwen3 models:
 *   a = RMSNorm(x; g_attn); q, k, v = a W_qkv^T (q heads, then k, then v);
 *   q, k = RoPE(RMSNorm_head(q; g_q)), RoPE(RMSNorm_head(k; g_k));
 *   (k, v) -> draft row i-1; o = draft attention; x += o W_o^T;
 *   m = RMSNorm(x; g_mlp); x += (silu(m W_gate^T) * (m W_up^T)) W_down^T.
 * The residual stream x is f32; the operands of every product (a, q, k, v,
 * o, m and the MLP activation) are bf16.  RoPE pairs element i with i + D/2
 * at angle pos * theta^(-2i/D), pos = ctx_len + draft_len - 1.
 * Weights are bf16, row-major in nn.Linear layout [out, in], 16-byte aligned.
 * ------------------------------------------------------------------------ */

/* The three epilogues of seed_linear. */
#define SEED_LINEAR_F32       0  /* y  = x W^T, f32 [batch, n_out]                   */
#define SEED_LINEAR_RESID_F32 1  /* y += x W^T, f32 [batch, n_out] updated in place   */
#define SEED_LINEAR_SWIGLU    2  /* y  = bf16(silu(x W^T) * (x W2^T)), bf16 [batch, n_out] */
#define SEED_LINEAR_MAX_BATCH 128

/* Workspace bytes of seed_linear for these sizes and epilogue: a fixed block
 * of per-tile arrival counters, then an f32 scratch of (1, or 2 for SwiGLU)
 * x batch x n_out sums.  It must be 256-byte aligned and ZERO-FILLED before
 * its first use; every call leaves all of it zero again, so one workspace (of
 * the largest size needed) serves any sequence of calls on one stream.  0 for
 * sizes seed_linear rejects. */
size_t seed_linear_workspace_bytes(int32_t batch, int32_t n_out, int32_t k_in, int32_t epilogue);

/* y (epilogue) x W^T on the tensor cores, one pass over W.  Work is split
 * evenly over the SMs by (128-row tile, 64-wide K slab); a tile whose slabs
 * fall on several CTAs is summed in f32 with atomic adds, so its last bits
 * can differ between runs (tiles computed whole are bit-reproducible).
 *   x      bf16 [batch, k_in], batch in [1, SEED_LINEAR_MAX_BATCH], k_in % 64 == 0,
 *          n_out <= 524288
 *   w      bf16 [n_out, k_in]; w2 bf16 [n_out, k_in] for SEED_LINEAR_SWIGLU
 *          (the up projection, w being the gate), else NULL
 *   y      see the epilogue; never aliases x
 * Errors: SEED_ERR_SHAPE (sizes, epilogue), SEED_ERR_NULL, SEED_ERR_RANGE
 * (a pointer not 16-byte aligned), SEED_ERR_WORKSPACE.  batch 0 is a no-op.
 * Device errors: SEED_DEVERR_TIMEOUT only. */
seed_status_t seed_linear(int32_t batch, int32_t k_in, int32_t n_out, const void* x,
                          const void* w, const void* w2, int32_t epilogue, void* y,
                          void* ws, size_t ws_bytes, int32_t* err_flag, void* stream);

/* x[b] = W_emb[tokens[b]] as f32 [batch, d_model] (the raw embedding H^0 the
 * drafter is fed, Sec. 4.1).  W_emb bf16 [vocab, d_model] (8-byte aligned),
 * x 16-byte aligned, d_model % 4 == 0.
 * Device errors: SEED_DEVERR_TOKEN (that row is left untouched). */
seed_status_t seed_embed(int32_t batch, int32_t d_model, int32_t vocab, const int32_t* tokens,
                         const void* w_emb, float* x, int32_t* err_flag, void* stream);

/* y = bf16(x / sqrt(mean(x^2) + eps) * gamma) row by row; x f32 [rows, n]
 * (16-byte aligned), gamma bf16 [n] and y bf16 [rows, n] (8-byte aligned),
 * n % 4 == 0. */
seed_status_t seed_rmsnorm(int32_t rows, int32_t n, const float* x, const void* gamma,
                           float eps, void* y, void* stream);

/* One decoder layer's weights (all bf16, nn.Linear layout). */
typedef struct {
  int32_t d_model;       /* multiple of 64 */
  int32_t d_ff;          /* multiple of 64 */
  float rms_eps;         /* e.g. 1e-6 */
  float rope_theta;      /* e.g. 1e6 */
  const void* g_attn;    /* [d_model] */
  const void* w_qkv;     /* [(hq + 2 hkv) head_dim, d_model] */
  const void* g_q;       /* [head_dim] */
  const void* g_k;       /* [head_dim] */
  const void* w_o;       /* [d_model, hq head_dim] */
  const void* g_mlp;     /* [d_model] */
  const void* w_gate;    /* [d_ff, d_model] */
  const void* w_up;      /* [d_ff, d_model] */
  const void* w_down;    /* [d_model, d_ff] */
} seed_decoder_layer_t;

/* Workspace bytes of seed_draft_layer (256-byte aligned, ZERO-FILLED before
 * its first use; every call leaves its counters zeroed again). */
size_t seed_draft_layer_workspace_bytes(const seed_cfg_t* cfg, const seed_decoder_layer_t* layer,
                                        int32_t batch);

/* One decoder layer of draft step i for a batch (head_dim 64 or 128):
 *   x          f32 [batch, d_model], the residual stream, updated in place
 *   ctx_kv     this layer's committed cache (the deep KV, read only)
 *   ctx_lens   int32 [batch] committed rows L
 *   draft_k/v  this layer's draft scratch; row i-1 is written
 *   draft_lens int32 [batch]: i after this step (1..kmax); 0 skips the
 *              sequence (its x row is then unspecified)
 * The step's token sits at position L + i - 1.  Launches norm, QKV product,
 * q/k norm + RoPE (which writes the step's K/V row into the draft scratch),
 * draft attention, output product with residual, norm, gate/up product with
 * SwiGLU and down product with residual, in this order on `stream`.
 * Errors: as seed_draft_attn and seed_linear.  Device errors: as
 * seed_draft_attn, plus SEED_DEVERR_TIMEOUT. */
seed_status_t seed_draft_layer(const seed_cfg_t* cfg, int32_t batch,
                               const seed_decoder_layer_t* layer, float* x, seed_kv_t ctx_kv,
                               const int32_t* ctx_lens, void* draft_k, void* draft_v,
                               const int32_t* draft_lens, void* ws, size_t ws_bytes,
                               int32_t* err_flag, void* stream);

/* ------------------------------------------------------------------------
 * The decoder's block-causal training attention (Sec. 4.2, "Training with
 * Block Attention"; Fig. 2, right), forward pass.  Sequences of n tokens are
 * cut into blocks of b; the query at position p sees
 *   - the deep keys/values k_dec/v_dec (the decoder layer's KV^dec from the
 *     full forward pass) at every position < s(p) = (p / b) * b, and
 *   - the layer's own keys/values over the raw embeddings, k_spec/v_spec,
 *     at positions s(p) .. p (causal within the block).
 *   cfg        hq, hkv, head_dim (64 or 128) and scale as for the other
 *              calls; page_size and kmax are not used
 *   n, block   n % block == 0, 2 <= block <= SEED_MAX_KMAX + 1 (a block of one
 *              token is the draft call's shape: use seed_draft_attn)
 *   q          bf16 [batch, n, hq, head_dim]
 *   k_dec, v_dec, k_spec, v_spec   bf16 [batch, n, hkv, head_dim]
 *   out        f32 [batch, n, hq, head_dim]; lse f32 [batch, n, hq] or NULL
 *   ws         seed_block_attn_workspace_bytes(...) bytes, 256-byte aligned,
 *              ZERO-FILLED before its first use.  head_dim 128 with 1, 2 or
 *              4 query heads per KV head runs one tensor-core kernel that
 *              reads q and the four inputs directly (the size is then 256,
 *              the workspace is not touched, and ws may be NULL with
 *              ws_bytes 0); other shapes run the
 *              verify kernel on one virtual sequence per block, and the
 *              workspace holds its counters (every call leaves them zeroed)
 *              and a paged copy of the rows that each call rewrites.
 * Errors: SEED_ERR_SHAPE (sizes, block, head_dim, group), SEED_ERR_NULL,
 * SEED_ERR_RANGE (a tensor not 16-byte aligned), SEED_ERR_WORKSPACE.
 * Device errors: none expected; a wait inside a kernel that runs out raises
 * SEED_DEVERR_TIMEOUT (as seed_verify_attn). */
size_t seed_block_attn_workspace_bytes(const seed_cfg_t* cfg, int32_t batch, int32_t n,
                                       int32_t block);
seed_status_t seed_block_attn(const seed_cfg_t* cfg, int32_t batch, int32_t n, int32_t block,
                              const void* q, const void* k_dec, const void* v_dec,
                              const void* k_spec, const void* v_spec, float* out, float* lse,
                              void* ws, size_t ws_bytes, int32_t* err_flag, void* stream);

/* ------------------------------------------------------------------------
 * Library convenience with no counterpart in the paper: verify attention
 * without a caller-provided workspace.
 *
 * seed_verify_attn_noalloc computes exactly what seed_verify_attn computes,
 * with the same arguments minus ws / ws_bytes. Its workspace is a scratch
 * array of SEED_NOALLOC_SCRATCH_BYTES built into the library (one per
 * device), so neither the caller nor the library allocates device memory.
 * It is meant for callers that cannot provide device memory: a plain C host
 * with no allocator of its own to expose, or a server that has handed all
 * free HBM to its KV page pool.
 *
 *   - Size limit: the call returns SEED_ERR_SCRATCH_LIMIT and launches
 *     nothing when seed_workspace_bytes(cfg, batch) exceeds
 *     SEED_NOALLOC_SCRATCH_BYTES.
 *   - Set-up: the first call on a device, with that device current, resolves
 *     the scratch's device address (this can load the library's module on
 *     the device) and caches it with the id of the device's current context.
 *   - Context changes: the scratch belongs to that context. When the device's
 *     current context is a different one (after cudaDeviceReset, or with
 *     another context made current), the next call resolves the address
 *     again; nothing in the scratch carries over from one call to the next,
 *     so no state is lost.
 *   - Zeroing: each call clears the scratch's counters on `stream` before its
 *     kernels (one small memset), so the caller never zeroes anything, and a
 *     call after a device error starts clean.
 *   - Concurrency: calls on one device that overlap in time (different
 *     streams, or host threads with no ordering between them) share the
 *     scratch and RACE. Serialise them: one stream, or events between them.
 *   - Errors: as seed_verify_attn, plus SEED_ERR_SCRATCH_LIMIT, and
 *     SEED_ERR_CUDA when the device or the scratch address cannot be
 *     obtained.
 * ------------------------------------------------------------------------ */
#define SEED_NOALLOC_SCRATCH_BYTES (32u << 20)

seed_status_t seed_verify_attn_noalloc(const seed_cfg_t* cfg, int32_t batch,
                                       const void* q, const int32_t* n_q,
                                       seed_kv_t kv, const int32_t* ctx_lens,
                                       float* out, float* lse,
                                       int32_t* err_flag, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SEED_H_ */
