// Block-causal training attention of the decoder (Sec. 4.2, "Training with
// Block Attention"; Fig. 2): with blocks of b tokens, the query at position p
// sees the decoder's deep keys/values (KV^dec) at positions < s(p) = (p/b)*b
// and, causally, its own keys/values over the raw embeddings at positions
// s(p) .. p.
//
// For the queries of one block starting at s, that is exactly verify
// attention (Alg. 2's k+1 causal queries) over a sequence whose L = s
// committed rows are the deep rows of positions [0, s) and whose b new rows
// are the raw-embedding rows of positions [s, s + b).  So the call builds one
// such virtual sequence per (sequence, block) in a paged layout -- the deep
// rows of each sequence are paged once and shared by all its blocks' page
// tables; each block gets private pages only for the page its boundary falls
// in and the pages of its own rows -- and runs the tensor-core verify kernel
// on all blocks at once: q [batch, n, hq, D] is already the virtual batch's
// [batch * n/b, b, hq, D] layout, and so are out and lse.
//
// head_dim 128 with groups of 1, 2 or 4 query heads per KV head goes to the
// prefill-style tensor-core kernel of block_tc.cu instead, which reads each
// query tile's prefix once for 128 query rows; the virtual-sequence route
// (which re-reads each block's prefix, about n^2 / 2b rows per sequence and
// KV head) serves the other shapes.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "../../include/seed.h"
#include "common.cuh"
#include "kernels.h"

namespace seedk {
bool block_tc_supported(int32_t head_dim, int32_t group);
cudaError_t launch_block_tc(int32_t B, int32_t n, int32_t blk, int32_t hq, int32_t hkv,
                            float scale, const void* q, const void* k_dec, const void* v_dec,
                            const void* k_spec, const void* v_spec, float* out, float* lse,
                            int32_t* err, cudaStream_t st);
}  // namespace seedk

namespace {

constexpr int kPg = 16;                       // rows per page (the cache's page size)
constexpr int kPackThreads = 256;

struct BlockGeom {
  int32_t B, n, b, hkv, D, nblk;              // nblk = n / b blocks per sequence
  int32_t pd;                                 // deep pages per sequence: ceil(n / 16)
  int32_t pp;                                 // private pages per block: ceil((15 + b) / 16)
  int32_t max_pages;                          // page-table width: pd + pp
  int64_t num_pages;                          // B * pd + B * nblk * pp
};

BlockGeom geom(int32_t B, int32_t n, int32_t b, int32_t hkv, int32_t D) {
  BlockGeom g{};
  g.B = B;
  g.n = n;
  g.b = b;
  g.hkv = hkv;
  g.D = D;
  g.nblk = n / b;
  g.pd = (n + kPg - 1) / kPg;
  g.pp = (15 + b + kPg - 1) / kPg;
  g.max_pages = g.pd + g.pp;
  g.num_pages = (int64_t)B * g.pd + (int64_t)B * g.nblk * g.pp;
  return g;
}

size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

struct BlockWs {
  size_t k, v, pt, ctx, nq, attn, total;
};

BlockWs layout(const BlockGeom& g, const seed_cfg_t& vcfg) {
  BlockWs w{};
  const size_t page_bytes = (size_t)g.hkv * kPg * g.D * 2;
  const int32_t Bv = g.B * g.nblk;
  size_t off = 0;
  auto take = [&](size_t n) {
    const size_t o = off;
    off += up256(n);
    return o;
  };
  w.k = take(page_bytes * g.num_pages);
  w.v = take(page_bytes * g.num_pages);
  w.pt = take((size_t)Bv * g.max_pages * 4);
  w.ctx = take((size_t)Bv * 4);
  w.nq = take((size_t)Bv * 4);
  w.attn = take(seed_workspace_bytes(&vcfg, Bv));
  w.total = off;
  return w;
}

// One block per page.  Deep page (sequence, j) holds deep rows 16 j ..; the
// private page t of block (sequence, blk) holds positions 16 (s/16 + t) ..,
// taking deep rows below s, raw-embedding rows in [s, s + b), zeros above.
// 16-byte copies (D is 64 or 128).
__global__ void __launch_bounds__(kPackThreads) pack_pages_kernel(
    const BlockGeom g, const uint4* k_dec, const uint4* v_dec, const uint4* k_spec,
    const uint4* v_spec, uint4* kp, uint4* vp) {
  if (threadIdx.x == 0) seedk::pdl_trigger();
  seedk::pdl_wait();
  const int64_t page = blockIdx.x;
  const int vec = g.D / 8;                    // uint4 per row of one head
  const int per_page = g.hkv * kPg * vec;
  int seq, first_pos, s = 0, e = 0;
  bool priv;
  if (page < (int64_t)g.B * g.pd) {
    seq = (int)(page / g.pd);
    first_pos = (int)(page % g.pd) * kPg;
    priv = false;
  } else {
    const int64_t r = page - (int64_t)g.B * g.pd;
    const int64_t blk = r / g.pp;             // virtual sequence index
    seq = (int)(blk / g.nblk);
    s = (int)(blk % g.nblk) * g.b;
    e = s + g.b;
    first_pos = (s / kPg + (int)(r % g.pp)) * kPg;
    priv = true;
  }
  uint4* kd = kp + page * per_page;
  uint4* vd = vp + page * per_page;
  for (int i = threadIdx.x; i < per_page; i += blockDim.x) {
    const int h = i / (kPg * vec), rr = (i / vec) % kPg, c = i % vec;
    const int pos = first_pos + rr;
    uint4 kv = make_uint4(0, 0, 0, 0), vv = kv;
    if (pos < g.n) {
      const size_t src = (((size_t)seq * g.n + pos) * g.hkv + h) * vec + c;
      if (!priv || pos < s) {
        kv = k_dec[src];
        vv = v_dec[src];
      } else if (pos < e) {
        kv = k_spec[src];
        vv = v_spec[src];
      }
    }
    kd[i] = kv;
    vd[i] = vv;
  }
}

// Page tables, committed lengths and query counts of the virtual sequences.
__global__ void block_tables_kernel(const BlockGeom g, int32_t* pt, int32_t* ctx, int32_t* nq) {
  if (threadIdx.x == 0) seedk::pdl_trigger();
  seedk::pdl_wait();
  const int blk = blockIdx.x;                 // virtual sequence
  const int seq = blk / g.nblk, s = (blk % g.nblk) * g.b;
  const int t0 = s / kPg;
  const int64_t priv0 = (int64_t)g.B * g.pd + (int64_t)blk * g.pp;
  for (int j = threadIdx.x; j < g.max_pages; j += blockDim.x) {
    int32_t id;
    if (j < t0)
      id = seq * g.pd + j;                    // shared deep page
    else if (j < t0 + g.pp)
      id = (int32_t)(priv0 + (j - t0));       // this block's private pages
    else
      id = 0;                                 // never read (past the block's rows)
    pt[(size_t)blk * g.max_pages + j] = id;
  }
  if (threadIdx.x == 0) {
    ctx[blk] = s;
    nq[blk] = g.b;
  }
}

seed_cfg_t virtual_cfg(const seed_cfg_t* cfg, int32_t b) {
  seed_cfg_t v = *cfg;
  v.page_size = kPg;
  v.kmax = b - 1;
  return v;
}

bool block_ok(const seed_cfg_t* cfg, int32_t batch, int32_t n, int32_t b) {
  if (cfg == nullptr || batch < 0 || n < 1 || b < 2 || b > SEED_MAX_KMAX + 1 || n % b != 0)
    return false;
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return false;
  const seed_cfg_t v = virtual_cfg(cfg, b);
  return seed_workspace_bytes(&v, 1) != 0;
}

}  // namespace

extern "C" {

size_t seed_block_attn_workspace_bytes(const seed_cfg_t* cfg, int32_t batch, int32_t n,
                                       int32_t block) {
  if (!block_ok(cfg, batch, n, block) || batch == 0) return 0;
  if (seedk::block_tc_supported(cfg->head_dim, cfg->hq / cfg->hkv)) return 256;   // unused
  const BlockGeom g = geom(batch, n, block, cfg->hkv, cfg->head_dim);
  if (g.num_pages > INT32_MAX) return 0;
  const seed_cfg_t v = virtual_cfg(cfg, block);
  return layout(g, v).total;
}

seed_status_t seed_block_attn(const seed_cfg_t* cfg, int32_t batch, int32_t n, int32_t block,
                              const void* q, const void* k_dec, const void* v_dec,
                              const void* k_spec, const void* v_spec, float* out, float* lse,
                              void* ws, size_t ws_bytes, int32_t* err_flag, void* stream) {
  if (cfg == nullptr) return SEED_ERR_NULL;
  if (!block_ok(cfg, batch, n, block)) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!q || !k_dec || !v_dec || !k_spec || !v_spec || !out || !err_flag) return SEED_ERR_NULL;
  auto mis16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; };
  if (mis16(q) || mis16(k_dec) || mis16(v_dec) || mis16(k_spec) || mis16(v_spec) || mis16(out))
    return SEED_ERR_RANGE;
  if (seedk::block_tc_supported(cfg->head_dim, cfg->hq / cfg->hkv)) {
    // the tensor-core kernel uses no workspace: ws may be NULL, ws_bytes 0
    const float scale = cfg->scale > 0.f ? cfg->scale : 1.0f / std::sqrt((float)cfg->head_dim);
    const cudaError_t e = seedk::launch_block_tc(batch, n, block, cfg->hq, cfg->hkv, scale, q,
                                                 k_dec, v_dec, k_spec, v_spec, out, lse,
                                                 err_flag, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? SEED_OK : SEED_ERR_CUDA;
  }
  if (ws == nullptr) return SEED_ERR_NULL;
  const BlockGeom g = geom(batch, n, block, cfg->hkv, cfg->head_dim);
  if (g.num_pages > INT32_MAX) return SEED_ERR_SHAPE;
  const seed_cfg_t v = virtual_cfg(cfg, block);
  const BlockWs w = layout(g, v);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < w.total) return SEED_ERR_WORKSPACE;
  char* base = static_cast<char*>(ws);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int32_t Bv = batch * g.nblk;
  cudaError_t e = seedk::launch_pdl(
      pack_pages_kernel, dim3((unsigned)g.num_pages), dim3(kPackThreads), 0, st, g,
      static_cast<const uint4*>(k_dec), static_cast<const uint4*>(v_dec),
      static_cast<const uint4*>(k_spec), static_cast<const uint4*>(v_spec),
      reinterpret_cast<uint4*>(base + w.k), reinterpret_cast<uint4*>(base + w.v));
  if (e != cudaSuccess) return SEED_ERR_CUDA;
  e = seedk::launch_pdl(block_tables_kernel, dim3(Bv), dim3(64), 0, st, g,
                        reinterpret_cast<int32_t*>(base + w.pt),
                        reinterpret_cast<int32_t*>(base + w.ctx),
                        reinterpret_cast<int32_t*>(base + w.nq));
  if (e != cudaSuccess) return SEED_ERR_CUDA;
  seed_kv_t kv;
  kv.k = base + w.k;
  kv.v = base + w.v;
  kv.page_table = reinterpret_cast<const int32_t*>(base + w.pt);
  kv.max_pages = g.max_pages;
  kv.num_pages = (int32_t)g.num_pages;
  return seed_verify_attn(&v, Bv, q, reinterpret_cast<const int32_t*>(base + w.nq), kv,
                          reinterpret_cast<const int32_t*>(base + w.ctx), out, lse, base + w.attn,
                          seed_workspace_bytes(&v, Bv), err_flag, stream);
}

}  // extern "C"
