// KV appends and greedy accept/commit: the integer and copy steps of SEED's
// decode loop (Alg. 2).
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace seedk {
namespace {

// One thread moves 16 bytes (8 bf16) of one KV head's row.
// grid (batch, rows per sequence), block hkv * D / 8 threads.

// Draft scratch append: row draft_lens[b]-1 of [B, hkv, kmax, D].
__global__ void draft_append_kernel(int32_t hkv, int32_t D, int32_t kmax,
                                    const uint16_t* __restrict__ k_new,
                                    const uint16_t* __restrict__ v_new,
                                    const int32_t* __restrict__ draft_lens,
                                    uint16_t* __restrict__ draft_k,
                                    uint16_t* __restrict__ draft_v, int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int chunks = D / 8;
  const int h = threadIdx.x / chunks, c = threadIdx.x - h * chunks;
  const int dl = draft_lens[b];
  if (dl < 0 || dl > kmax) {
    if (threadIdx.x == 0) raise_err(err, SEED_DEVERR_DRAFT_LEN);
    return;
  }
  if (dl == 0 || h >= hkv) return;
  const size_t src = ((size_t)b * hkv + h) * D + c * 8;
  const size_t dst = (((size_t)b * hkv + h) * kmax + (dl - 1)) * D + c * 8;
  *reinterpret_cast<uint4*>(draft_k + dst) = __ldg(reinterpret_cast<const uint4*>(k_new + src));
  *reinterpret_cast<uint4*>(draft_v + dst) = __ldg(reinterpret_cast<const uint4*>(v_new + src));
}

// Verify rows: row j of [B, kmax+1, hkv, D] goes to logical position
// ctx_lens[b] + j of the paged cache.
__global__ void kv_append_kernel(int32_t hkv, int32_t D, int32_t kmax,
                                 uint16_t* __restrict__ k_cache, uint16_t* __restrict__ v_cache,
                                 const int32_t* __restrict__ page_table, int32_t max_pages,
                                 int32_t num_pages, const uint16_t* __restrict__ k_new,
                                 const uint16_t* __restrict__ v_new,
                                 const int32_t* __restrict__ n_new,
                                 const int32_t* __restrict__ ctx_lens, int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, j = blockIdx.y;
  const int chunks = D / 8;
  const int h = threadIdx.x / chunks, c = threadIdx.x - h * chunks;
  const int n = n_new[b];
  const int L = ctx_lens[b];
  if (n < 0 || n > kmax + 1) {
    if (j == 0 && threadIdx.x == 0) raise_err(err, SEED_DEVERR_NQ);
    return;
  }
  if (L < 0 || (long long)L + n > (long long)max_pages * kPage) {
    if (j == 0 && threadIdx.x == 0) raise_err(err, SEED_DEVERR_CTX_LEN);
    return;
  }
  if (j >= n || h >= hkv) return;
  const int pos = L + j;
  const int pid = page_table[(size_t)b * max_pages + pos / kPage];
  if (pid < 0 || pid >= num_pages) {
    if (threadIdx.x == 0) raise_err(err, SEED_DEVERR_PAGE);
    return;
  }
  const size_t src = (((size_t)b * (kmax + 1) + j) * hkv + h) * D + c * 8;
  const size_t dst = (((size_t)pid * hkv + h) * kPage + pos % kPage) * D + c * 8;
  *reinterpret_cast<uint4*>(k_cache + dst) = __ldg(reinterpret_cast<const uint4*>(k_new + src));
  *reinterpret_cast<uint4*>(v_cache + dst) = __ldg(reinterpret_cast<const uint4*>(v_new + src));
}

// Greedy longest-prefix acceptance (Alg. 2): one warp per sequence.  Lane i
// compares X_draft[i+1] with argmax p_{i+1}; the first mismatch among the
// k_b drafts (ballot + find-first-set) gives n.  Lanes 0..n emit the tokens
// and the committed slots of positions L..L+n; lane 0 advances the length.
__global__ void accept_kernel(int32_t B, int32_t kmax, const int32_t* __restrict__ draft_ids,
                              const int32_t* __restrict__ target_ids,
                              const int32_t* __restrict__ k_b,
                              const int32_t* __restrict__ page_table, int32_t max_pages,
                              int32_t page_size, int32_t* __restrict__ ctx_lens,
                              int32_t* __restrict__ accepted, int32_t* __restrict__ tokens,
                              int32_t* __restrict__ slots, int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;
  const int width = kmax + 1;
  const int kb = k_b[b];
  const int L = ctx_lens[b];
  const bool bad_k = kb < 0 || kb > kmax;
  const bool bad_len = L < 0 || (long long)L + kb + 1 > (long long)max_pages * page_size;
  if (bad_k || bad_len) {
    if (lane == 0) {
      raise_err(err, (bad_k ? SEED_DEVERR_KB : 0) | (bad_len ? SEED_DEVERR_CTX_LEN : 0));
      accepted[b] = 0;
    }
    for (int i = lane; i < width; i += 32) {
      tokens[(size_t)b * width + i] = -1;
      slots[(size_t)b * width + i] = -1;
    }
    return;
  }
  const bool mism = lane < kb && draft_ids[(size_t)b * kmax + lane] !=
                                     target_ids[(size_t)b * width + lane];
  const unsigned mask = __ballot_sync(0xffffffffu, mism);
  const int n = mask ? (__ffs(mask) - 1) : kb;
  for (int i = lane; i < width; i += 32) {
    int tok = -1, slot = -1;
    if (i < n) tok = draft_ids[(size_t)b * kmax + i];
    else if (i == n) tok = target_ids[(size_t)b * width + i];
    if (i <= n) {
      const int pos = L + i;
      slot = page_table[(size_t)b * max_pages + pos / page_size] * page_size + pos % page_size;
    }
    tokens[(size_t)b * width + i] = tok;
    slots[(size_t)b * width + i] = slot;
  }
  if (lane == 0) {
    accepted[b] = n;
    ctx_lens[b] = L + n + 1;
  }
}

}  // namespace

// Tree acceptance (Sec. D.1): one warp per sequence, lane i = node i of the
// linearised tree (at most 32 nodes).  From the root, the walk takes the
// lowest-index child whose token equals the verifier's argmax at the current
// node, until no child matches; the bonus token is the argmax at the last
// accepted node.  Outputs follow seed_accept_commit, plus the accepted path.
__global__ void tree_accept_kernel(int32_t B, int32_t kmax, const int32_t* __restrict__ tok,
                                   const int32_t* __restrict__ parent,
                                   const int32_t* __restrict__ n_nodes,
                                   const int32_t* __restrict__ target_ids,
                                   const int32_t* __restrict__ page_table, int32_t max_pages,
                                   int32_t page_size, int32_t* __restrict__ ctx_lens,
                                   int32_t* __restrict__ accepted, int32_t* __restrict__ tokens,
                                   int32_t* __restrict__ path, int32_t* __restrict__ slots,
                                   int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) return;
  const int W = kmax + 1;
  const size_t row = (size_t)b * W;
  const int n = n_nodes[b];
  const int L = ctx_lens[b];
  const bool bad_n = n < 1 || n > W;
  const bool in = !bad_n && lane < n;
  const int par = (in && lane > 0) ? parent[row + lane] : -1;
  const int t = in ? tok[row + lane] : -1;
  const int tg = in ? target_ids[row + lane] : -1;
  const bool bad_par = __any_sync(0xffffffffu, in && lane > 0 && (par < 0 || par >= lane));
  const long long cap = (long long)max_pages * page_size;
  const bool bad_len = L < 0 || (!bad_n && (long long)L + n > cap);
  if (bad_n || bad_par || bad_len) {
    if (lane == 0)
      raise_err(err, bad_n ? SEED_DEVERR_NQ : bad_par ? SEED_DEVERR_TREE : SEED_DEVERR_CTX_LEN);
    return;
  }
  // the walk; lane d keeps the node at depth d of the accepted path
  int cur = 0, depth = 0, mypath = lane == 0 ? 0 : -1;
  for (int it = 0; it < 32; ++it) {
    const int want = __shfl_sync(0xffffffffu, tg, cur);
    const unsigned m = __ballot_sync(0xffffffffu, in && lane > 0 && par == cur && t == want);
    if (m == 0u) break;
    cur = __ffs((int)m) - 1;
    ++depth;
    if (lane == depth) mypath = cur;
  }
  const int bonus = __shfl_sync(0xffffffffu, tg, cur);
  const int next = __shfl_sync(0xffffffffu, mypath, (lane + 1) & 31);   // path[lane + 1]
  const int tnext = __shfl_sync(0xffffffffu, t, next < 0 ? 0 : next);
  if (lane < W) {
    int out_tok = -1, out_slot = -1;
    if (lane < depth) out_tok = tnext;
    else if (lane == depth) out_tok = bonus;
    if (lane <= depth) {
      const int pos = L + lane;
      out_slot = page_table[(size_t)b * max_pages + pos / page_size] * page_size + pos % page_size;
    }
    tokens[row + lane] = out_tok;
    slots[row + lane] = out_slot;
    path[row + lane] = lane <= depth ? mypath : -1;
  }
  if (lane == 0) {
    accepted[b] = depth;
    ctx_lens[b] = L + depth + 1;
  }
}

// Commit of a tree's accepted path in one layer's cache: the row of the node at
// depth d moves from packed position L + path[d] to L + d (d = 1..n), one
// depth at a time (a later move never reads a row an earlier one wrote).
// grid (batch), block hkv * D / 8 threads; runs after tree_accept_kernel, whose
// updated ctx_lens and accepted give L = ctx_lens - accepted - 1.
__global__ void tree_compact_kernel(int32_t hkv, int32_t D, int32_t kmax,
                                    uint16_t* __restrict__ k_cache,
                                    uint16_t* __restrict__ v_cache,
                                    const int32_t* __restrict__ page_table, int32_t max_pages,
                                    int32_t num_pages, const int32_t* __restrict__ path,
                                    const int32_t* __restrict__ accepted,
                                    const int32_t* __restrict__ ctx_lens, int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int chunks = D / 8;
  const int h = threadIdx.x / chunks, c = threadIdx.x - h * chunks;
  const int W = kmax + 1;
  const int n = accepted[b];
  const int L = ctx_lens[b] - n - 1;
  if (n < 0 || n > kmax || L < 0) {
    if (threadIdx.x == 0) raise_err(err, n < 0 || n > kmax ? SEED_DEVERR_TREE : SEED_DEVERR_CTX_LEN);
    return;
  }
  const long long cap = (long long)max_pages * kPage;
  for (int d = 1; d <= n; ++d) {
    const int pd = path[(size_t)b * W + d];
    if (pd < d || pd > kmax || (long long)L + pd >= cap) {
      if (threadIdx.x == 0) raise_err(err, SEED_DEVERR_TREE);
      return;
    }
  }
  for (int d = 1; d <= n; ++d) {
    const int src = L + path[(size_t)b * W + d], dst = L + d;
    if (src != dst && h < hkv) {
      const int ps = page_table[(size_t)b * max_pages + src / kPage];
      const int pdst = page_table[(size_t)b * max_pages + dst / kPage];
      if (ps < 0 || ps >= num_pages || pdst < 0 || pdst >= num_pages) {
        raise_err(err, SEED_DEVERR_PAGE);
      } else {
        const size_t so = (((size_t)ps * hkv + h) * kPage + src % kPage) * D + c * 8;
        const size_t dof = (((size_t)pdst * hkv + h) * kPage + dst % kPage) * D + c * 8;
        *reinterpret_cast<uint4*>(k_cache + dof) = *reinterpret_cast<const uint4*>(k_cache + so);
        *reinterpret_cast<uint4*>(v_cache + dof) = *reinterpret_cast<const uint4*>(v_cache + so);
      }
    }
    __syncthreads();
  }
}

cudaError_t launch_draft_append(int32_t B, int32_t hkv, int32_t head_dim, int32_t kmax,
                                const uint16_t* k_new, const uint16_t* v_new,
                                const int32_t* draft_lens, uint16_t* draft_k, uint16_t* draft_v,
                                int32_t* err, cudaStream_t st) {
  const int threads = hkv * head_dim / 8;
  return launch_pdl(draft_append_kernel, dim3(B), dim3(threads), 0, st, hkv, head_dim, kmax, k_new,
                    v_new, draft_lens, draft_k, draft_v, err);
}

cudaError_t launch_kv_append(int32_t B, int32_t hkv, int32_t head_dim, int32_t kmax,
                             uint16_t* k_cache, uint16_t* v_cache, const int32_t* page_table,
                             int32_t max_pages, int32_t num_pages, const uint16_t* k_new,
                             const uint16_t* v_new, const int32_t* n_new,
                             const int32_t* ctx_lens, int32_t* err, cudaStream_t st) {
  const int threads = hkv * head_dim / 8;
  dim3 grid(B, kmax + 1);
  return launch_pdl(kv_append_kernel, grid, dim3(threads), 0, st, hkv, head_dim, kmax, k_cache,
                    v_cache, page_table, max_pages, num_pages, k_new, v_new, n_new, ctx_lens, err);
}

cudaError_t launch_accept(int32_t B, int32_t kmax, const int32_t* draft_ids,
                          const int32_t* target_ids, const int32_t* k_b,
                          const int32_t* page_table, int32_t max_pages, int32_t page_size,
                          int32_t* ctx_lens, int32_t* accepted, int32_t* tokens,
                          int32_t* slots, int32_t* err, cudaStream_t st) {
  constexpr int kWarpsPerBlock = 4;
  const int grid = (B + kWarpsPerBlock - 1) / kWarpsPerBlock;
  return launch_pdl(accept_kernel, dim3(grid), dim3(32 * kWarpsPerBlock), 0, st, B, kmax,
                    draft_ids, target_ids, k_b, page_table, max_pages, page_size, ctx_lens,
                    accepted, tokens, slots, err);
}

cudaError_t launch_tree_accept(int32_t B, int32_t kmax, const int32_t* tok, const int32_t* parent,
                               const int32_t* n_nodes, const int32_t* target_ids,
                               const int32_t* page_table, int32_t max_pages, int32_t page_size,
                               int32_t* ctx_lens, int32_t* accepted, int32_t* tokens,
                               int32_t* path, int32_t* slots, int32_t* err, cudaStream_t st) {
  constexpr int kWarpsPerBlock = 4;
  const int grid = (B + kWarpsPerBlock - 1) / kWarpsPerBlock;
  return launch_pdl(tree_accept_kernel, dim3(grid), dim3(32 * kWarpsPerBlock), 0, st, B, kmax,
                    tok, parent, n_nodes, target_ids, page_table, max_pages, page_size, ctx_lens,
                    accepted, tokens, path, slots, err);
}

cudaError_t launch_tree_compact(int32_t B, int32_t hkv, int32_t head_dim, int32_t kmax,
                                uint16_t* k_cache, uint16_t* v_cache, const int32_t* page_table,
                                int32_t max_pages, int32_t num_pages, const int32_t* path,
                                const int32_t* accepted, const int32_t* ctx_lens, int32_t* err,
                                cudaStream_t st) {
  const int threads = hkv * head_dim / 8;
  return launch_pdl(tree_compact_kernel, dim3(B), dim3(threads), 0, st, hkv, head_dim, kmax,
                    k_cache, v_cache, page_table, max_pages, num_pages, path, accepted, ctx_lens,
                    err);
}

}  // namespace seedk
