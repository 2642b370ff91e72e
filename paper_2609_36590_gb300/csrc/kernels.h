// Internal launch interface between the C ABI (seed_api.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <utility>

namespace seedk {

constexpr int kPageTokens = 16;   // tokens per KV page; the only page size built

// Launch with programmatic stream serialisation: the kernel may begin while
// the previous kernel of the stream finishes (it must call pdl_wait() before
// touching global memory).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Split-KV flash-decoding work description (see decode_attn.cu).
struct DecodeParams {
  const uint16_t* q;          // bf16 [NV, hq, D]
  const uint16_t* k_cache;    // bf16 [num_pages, hkv, 16, D]
  const uint16_t* v_cache;
  const int32_t* page_table;  // [B, max_pages]
  int32_t max_pages;
  int32_t num_pages;
  const uint16_t* draft_k;    // bf16 [B, hkv, kmax, D] (draft mode only)
  const uint16_t* draft_v;
  const int32_t* ctx_lens;    // [B]
  const int32_t* aux;         // draft: draft_lens [B]; verify: n_q [B]
  float* out;                 // f32 [NV, hq, D]
  float* lse;                 // f32 [NV, hq] or null
  float* part;                // split partial records
  int32_t* counters;          // [NV * hkv] arrival counters (zero between calls)
  int32_t* err;
  int32_t B, hq, hkv, kmax;
  int32_t nq_per_seq;         // virtual sequences per real sequence: 1 or kmax+1
  int32_t verify;             // 0: draft rows after the context; 1: causal verify
  int32_t ppu;                // pages per work unit (multiple of 4)
  int32_t cmax;               // work units per (virtual sequence, KV head)
  int32_t n_units;            // NV * hkv * cmax
  float scale_log2;           // softmax scale * log2(e)
};

// Work split shared by the host-side planner and the workspace-size bound.
constexpr int kTargetUnits = 2048;

struct DecodePlan {
  int32_t nv, ppu, cmax, n_units;
  size_t counters_bytes, part_bytes;
};

DecodePlan plan_decode(int32_t nv, int32_t hkv, int32_t group, int32_t head_dim,
                       int32_t max_pages);
size_t decode_workspace_bound(int32_t nv_max, int32_t hkv, int32_t group, int32_t head_dim);

cudaError_t launch_decode(const DecodeParams& p, int head_dim, int group, cudaStream_t st);

cudaError_t launch_draft_append(int32_t B, int32_t hkv, int32_t head_dim, int32_t kmax,
                                const uint16_t* k_new, const uint16_t* v_new,
                                const int32_t* draft_lens, uint16_t* draft_k, uint16_t* draft_v,
                                int32_t* err, cudaStream_t st);

cudaError_t launch_kv_append(int32_t B, int32_t hkv, int32_t head_dim, int32_t kmax,
                             uint16_t* k_cache, uint16_t* v_cache, const int32_t* page_table,
                             int32_t max_pages, int32_t num_pages, const uint16_t* k_new,
                             const uint16_t* v_new, const int32_t* n_new,
                             const int32_t* ctx_lens, int32_t* err, cudaStream_t st);

cudaError_t launch_accept(int32_t B, int32_t kmax, const int32_t* draft_ids,
                          const int32_t* target_ids, const int32_t* k_b,
                          const int32_t* page_table, int32_t max_pages, int32_t page_size,
                          int32_t* ctx_lens, int32_t* accepted, int32_t* tokens,
                          int32_t* slots, int32_t* err, cudaStream_t st);

cudaError_t launch_tree_accept(int32_t B, int32_t kmax, const int32_t* tok, const int32_t* parent,
                               const int32_t* n_nodes, const int32_t* target_ids,
                               const int32_t* page_table, int32_t max_pages, int32_t page_size,
                               int32_t* ctx_lens, int32_t* accepted, int32_t* tokens,
                               int32_t* path, int32_t* slots, int32_t* err, cudaStream_t st);

cudaError_t launch_tree_compact(int32_t B, int32_t hkv, int32_t head_dim, int32_t kmax,
                                uint16_t* k_cache, uint16_t* v_cache, const int32_t* page_table,
                                int32_t max_pages, int32_t num_pages, const int32_t* path,
                                const int32_t* accepted, const int32_t* ctx_lens, int32_t* err,
                                cudaStream_t st);

int device_sm_count();

// Drafter LM head with fused softmax and top-10 (head_tc.cu).
constexpr int kHeadMaxCtas = 256;
struct HeadParams {
  float* part;        // [ctas * 4, B, 24] partial records
  int32_t* ids;       // [B, 10]
  float* probs;       // [B, 10]
  int32_t* n_sib;     // [B]
  int32_t* stop;      // [B]
  float* lse;         // [B] or null
  int32_t* err;
  int32_t B, d, V;
  float tau;
};
int head_ctas(int32_t vocab);
size_t head_workspace_bytes(int32_t batch);
cudaError_t launch_head(const HeadParams& p, const void* h, const void* w, int nctas,
                        cudaStream_t st);

// Skinny GEMM for the drafter's decoder layers (linear_tc.cu).
constexpr int kLinearMaxCtas = 256;
constexpr int kLinearMaxTiles = 4096;                  // n_out <= 4096 * 128
constexpr size_t kLinearCntBytes = kLinearMaxTiles * sizeof(int32_t);
enum LinearEpi : int32_t { kEpiF32 = 0, kEpiResidF32 = 1, kEpiSwigluBf16 = 2 };
struct LinearParams {
  void* y;            // f32 [B, N] (kEpiF32, kEpiResidF32) or bf16 [B, N] (kEpiSwigluBf16)
  float* acc;         // [(1|2), B, N] f32 scratch for tiles split over CTAs, zero between calls
  int32_t* cnt;       // [kLinearMaxTiles] arrival counters, zero between calls
  int32_t* err;
  int32_t B, K, N, epi;
};
int linear_ctas(int32_t n_out, int32_t k_in);
size_t linear_workspace_bytes(int32_t batch, int32_t n_out, int32_t k_in, int32_t epi);
cudaError_t launch_linear(LinearParams p, const void* x, const void* w, const void* w2, void* ws,
                          cudaStream_t st);

// The small steps of a draft step (draft_ops.cu).
cudaError_t launch_embed(int32_t B, int32_t d, int32_t vocab, const int32_t* tokens,
                         const void* w, float* x, int32_t* err, cudaStream_t st);
cudaError_t launch_rmsnorm(int32_t rows, int32_t n, const float* x, const void* gamma, float eps,
                           void* y, cudaStream_t st);
cudaError_t launch_qk_norm_rope(int32_t B, int32_t hq, int32_t hkv, int32_t D, const float* qkv,
                                const void* gq, const void* gk, const int32_t* ctx_lens,
                                const int32_t* draft_lens, float theta, float eps, int32_t kmax,
                                void* q, void* draft_k, void* draft_v, int32_t* err,
                                cudaStream_t st);
cudaError_t launch_f32_to_bf16(size_t n, const float* x, void* y, cudaStream_t st);

// Tensor-core draft and verify attention (attn_tc.cu).
constexpr int kTcMaxCtas = 256;     // most CTAs of one launch (two record slots each)
constexpr int kPlanInts = 8;        // int32 per merge plan entry

struct AttnTcParams {
  const int32_t* page_table;
  int32_t max_pages;
  int32_t num_pages;
  const int32_t* ctx_lens;    // [B]
  const int32_t* aux;         // verify: n_q [B]; draft: draft_lens [B]
  const uint32_t* anc;        // tree verify: [B, W1] ancestor masks; else null
  float* out;                 // f32 [B, W1, hq, 128]
  float* lse;                 // f32 [B, W1, hq] or null
  float* part;                // partial records: two slots per CTA
  int32_t* plan;              // merge plan: 8 int32 per CTA range boundary
  int32_t* err;
  int32_t B, hq, hkv, kmax, G;
  int32_t draft;              // 1: draft attention (cache rows + draft scratch rows)
  int32_t W1;                 // query positions per sequence: kmax+1 (verify) or 1 (draft)
  int32_t nctas;              // CTAs of the attention kernel (static tile partition)
  float scale_log2;
  // raw inputs for the keys-as-rows kernel's exact recomputation of a piece
  // (bf16): q [B, W1, hq, D], the paged caches, the draft scratch (draft only)
  const uint16_t* q;
  const uint16_t* k_cache;
  const uint16_t* v_cache;
  const uint16_t* draft_k;
  const uint16_t* draft_v;
  int32_t D;
};

bool attn_tc_supported(int head_dim, int group, int w1);
int attn_tc_ctas();
// Bytes at the start of a draft / verify workspace that must be zero before
// a call (every kernel leaves them zero again): 256 bytes of work-dispenser
// state, then one int32 arrival counter per (sequence, query slot, KV head)
// with at least 4 slots per sequence, rounded up to 256 bytes.  The rest of
// the workspace holds split records and plans, always written before read.
size_t workspace_zero_prefix_bytes(int32_t kmax, int32_t hkv, int32_t batch);

// Workspace of either tensor-core kernel, after its counters: two split
// records per CTA (rows x (head_dim + 1) floats each), then, at
// attn_tc_plan_offset, one 32-byte merge plan per CTA range boundary.
size_t attn_tc_plan_offset(int32_t ctas, int32_t rows, int32_t head_dim);
size_t attn_tc_records_bytes(int32_t ctas, int32_t rows, int32_t head_dim);
// attn_tc_records_bytes at the most CTAs a launch uses.
size_t attn_tc_part_bound(int32_t group, int32_t w1, int32_t head_dim);
cudaError_t launch_attn_tc(const AttnTcParams& p, const void* q, const void* k_cache,
                           const void* v_cache, const void* draft_k, const void* draft_v,
                           cudaStream_t st);

// Keys-as-rows tensor-core attention for at most 64 query rows per KV head
// (attn_kt.cu); head_dim 64 or 128.
bool attn_kt_supported(int head_dim, int group, int w1);
cudaError_t launch_attn_kt(const AttnTcParams& p, int head_dim, const void* q,
                           const void* k_cache, const void* v_cache, const void* draft_k,
                           const void* draft_v, cudaStream_t st);

// Cluster attention for launches with few (sequence, KV head) pairs
// (attn_cluster.cu): one cluster of 8, 12 or 16 CTAs per pair, each CTA at
// most kClMaxPages pages of the pair, at most kClRows query rows per KV head,
// head_dim 128.  attn_cl_route gives the cluster size for a launch (0: not
// this kernel): the largest whose clusters are all resident at once and whose
// CTAs hold every sequence the page table allows.
constexpr int kClMaxPages = 19;
constexpr int kClRows = 32;
int attn_cl_route(int head_dim, int group, int w1, int batch, int hkv, int max_pages);
cudaError_t launch_attn_cl(const AttnTcParams& p, int cluster, const void* k_cache,
                           const void* v_cache, const void* draft_k, const void* draft_v,
                           cudaStream_t st);

}  // namespace seedk
