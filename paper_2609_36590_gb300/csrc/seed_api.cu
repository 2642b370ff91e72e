// The C ABI of include/seed.h: host-side argument checks, work planning and
// kernel launches.  No allocation, no synchronisation, no state.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "../../include/seed.h"
#include "kernels.h"

namespace {

constexpr size_t kAlign = 256;

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

namespace seedk {

size_t workspace_zero_prefix_bytes(int32_t kmax, int32_t hkv, int32_t batch) {
  const size_t per = (size_t)std::max(kmax + 1, 4);
  return kAlign + round_up((size_t)batch * per * hkv * sizeof(int32_t), kAlign);
}

}  // namespace seedk

namespace {

bool group_supported(int g) { return g == 1 || g == 2 || g == 4 || g == 8; }

seed_status_t check_cfg(const seed_cfg_t* cfg) {
  if (cfg == nullptr) return SEED_ERR_NULL;
  if (cfg->hq <= 0 || cfg->hkv <= 0 || cfg->hq % cfg->hkv != 0) return SEED_ERR_SHAPE;
  if (cfg->kmax < 1 || cfg->kmax > SEED_MAX_KMAX) return SEED_ERR_SHAPE;
  if (!(cfg->scale >= 0.f) || std::isinf(cfg->scale)) return SEED_ERR_SHAPE;
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return SEED_ERR_UNSUPPORTED;
  if (!group_supported(cfg->hq / cfg->hkv)) return SEED_ERR_UNSUPPORTED;
  if (cfg->page_size != seedk::kPageTokens) return SEED_ERR_UNSUPPORTED;
  return SEED_OK;
}

seed_status_t check_kv(const seed_kv_t& kv) {
  if (kv.k == nullptr || kv.v == nullptr || kv.page_table == nullptr) return SEED_ERR_NULL;
  if (kv.max_pages <= 0 || kv.num_pages <= 0) return SEED_ERR_RANGE;
  if ((long long)kv.max_pages * seedk::kPageTokens > INT32_MAX) return SEED_ERR_RANGE;
  return SEED_OK;
}

float scale_of(const seed_cfg_t* cfg) {
  return cfg->scale > 0.f ? cfg->scale : 1.0f / std::sqrt((float)cfg->head_dim);
}

// Workspace layout: [0, 256) the tensor-core verify's unit dispenser; then
// arrival counters for batch*(kmax+1)*hkv (virtual sequence, KV head) pairs;
// then the split partial records.  Every kernel leaves the counters at zero.
// The first two parts are the zero prefix (seedk::workspace_zero_prefix_bytes).
constexpr size_t kSchedBytes = kAlign;

size_t zero_prefix(const seed_cfg_t* cfg, int32_t batch) {
  return seedk::workspace_zero_prefix_bytes(cfg->kmax, cfg->hkv, batch);
}

seed_status_t finish(cudaError_t e) { return e == cudaSuccess ? SEED_OK : SEED_ERR_CUDA; }

seed_status_t run_decode(const seed_cfg_t* cfg, int32_t batch, bool verify, const void* q,
                         const seed_kv_t& kv, const void* draft_k, const void* draft_v,
                         const int32_t* ctx_lens, const int32_t* aux, float* out, float* lse,
                         void* ws, size_t ws_bytes, int32_t* err, void* stream) {
  const int G = cfg->hq / cfg->hkv;
  const int nq = verify ? cfg->kmax + 1 : 1;
  const int nv = batch * nq;
  const seedk::DecodePlan pl = seedk::plan_decode(nv, cfg->hkv, G, cfg->head_dim, kv.max_pages);
  const size_t cb = zero_prefix(cfg, batch);
  if (ws_bytes < cb + pl.part_bytes) return SEED_ERR_WORKSPACE;
  seedk::DecodeParams p{};
  p.q = static_cast<const uint16_t*>(q);
  p.k_cache = static_cast<const uint16_t*>(kv.k);
  p.v_cache = static_cast<const uint16_t*>(kv.v);
  p.page_table = kv.page_table;
  p.max_pages = kv.max_pages;
  p.num_pages = kv.num_pages;
  p.draft_k = static_cast<const uint16_t*>(draft_k);
  p.draft_v = static_cast<const uint16_t*>(draft_v);
  p.ctx_lens = ctx_lens;
  p.aux = aux;
  p.out = out;
  p.lse = lse;
  p.counters = reinterpret_cast<int32_t*>(static_cast<char*>(ws) + kSchedBytes);
  p.part = reinterpret_cast<float*>(static_cast<char*>(ws) + cb);
  p.err = err;
  p.B = batch;
  p.hq = cfg->hq;
  p.hkv = cfg->hkv;
  p.kmax = cfg->kmax;
  p.nq_per_seq = nq;
  p.verify = verify ? 1 : 0;
  p.ppu = pl.ppu;
  p.cmax = pl.cmax;
  p.n_units = pl.n_units;
  p.scale_log2 = scale_of(cfg) * 1.4426950408889634f;
  return finish(seedk::launch_decode(p, cfg->head_dim, G, static_cast<cudaStream_t>(stream)));
}

// Draft / verify attention on the tensor cores: the cluster kernel when the
// launch has few (sequence, KV head) pairs and short sequences (head_dim 128,
// R = G * W1 <= 32), else the keys-as-rows kernel for head_dim 64 when the R
// query rows of a KV head fit 48 MMA columns, the query-rows kernel for
// head_dim 128 (R <= 128).
seed_status_t run_attn_tc(const seed_cfg_t* cfg, int32_t batch, bool draft, const void* q,
                          const int32_t* aux, const seed_kv_t& kv, const void* draft_k,
                          const void* draft_v, const int32_t* ctx_lens, float* out, float* lse,
                          void* ws, size_t ws_bytes, int32_t* err, void* stream,
                          const uint32_t* anc = nullptr) {
  const int G = cfg->hq / cfg->hkv;
  const int W1 = draft ? 1 : cfg->kmax + 1;
  const size_t cb = zero_prefix(cfg, batch);
  const int ctas = seedk::attn_tc_ctas();
  const size_t need = cb + seedk::attn_tc_records_bytes(ctas, G * W1, cfg->head_dim);
  const bool kt = seedk::attn_kt_supported(cfg->head_dim, G, W1);
  if (ws_bytes < need) return SEED_ERR_WORKSPACE;
  seedk::AttnTcParams p{};
  p.page_table = kv.page_table;
  p.max_pages = kv.max_pages;
  p.num_pages = kv.num_pages;
  p.ctx_lens = ctx_lens;
  p.aux = aux;
  p.anc = anc;
  p.out = out;
  p.lse = lse;
  p.part = reinterpret_cast<float*>(static_cast<char*>(ws) + cb);
  p.plan = reinterpret_cast<int32_t*>(static_cast<char*>(ws) + cb +
                                      seedk::attn_tc_plan_offset(ctas, G * W1, cfg->head_dim));
  p.err = err;
  p.B = batch;
  p.hq = cfg->hq;
  p.hkv = cfg->hkv;
  p.kmax = cfg->kmax;
  p.G = G;
  p.draft = draft ? 1 : 0;
  p.W1 = W1;
  p.nctas = ctas;
  p.scale_log2 = scale_of(cfg) * 1.4426950408889634f;
  p.q = static_cast<const uint16_t*>(q);
  p.k_cache = static_cast<const uint16_t*>(kv.k);
  p.v_cache = static_cast<const uint16_t*>(kv.v);
  p.draft_k = static_cast<const uint16_t*>(draft_k);
  p.draft_v = static_cast<const uint16_t*>(draft_v);
  p.D = cfg->head_dim;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int cluster =
      anc == nullptr ? seedk::attn_cl_route(cfg->head_dim, G, W1, batch, cfg->hkv, kv.max_pages)
                     : 0;
  if (cluster > 0)
    return finish(seedk::launch_attn_cl(p, cluster, kv.k, kv.v, draft_k, draft_v, st));
  return finish(kt ? seedk::launch_attn_kt(p, cfg->head_dim, q, kv.k, kv.v, draft_k, draft_v, st)
                   : seedk::launch_attn_tc(p, q, kv.k, kv.v, draft_k, draft_v, st));
}

bool misaligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; }

// Whether a launch with R = group * w1 query rows per KV head runs on one of
// the tensor-core kernels.
bool tc_path(int head_dim, int group, int w1) {
  return seedk::attn_kt_supported(head_dim, group, w1) ||
         seedk::attn_tc_supported(head_dim, group, w1);
}

}  // namespace

extern "C" {

int32_t seed_abi_version(void) { return SEED_ABI_VERSION; }

const char* seed_status_string(seed_status_t s) {
  switch (s) {
    case SEED_OK: return "ok";
    case SEED_ERR_NULL: return "a required pointer is NULL";
    case SEED_ERR_SHAPE: return "invalid shape (batch, heads or kmax)";
    case SEED_ERR_RANGE: return "max_pages / num_pages out of range";
    case SEED_ERR_UNSUPPORTED: return "head_dim, group size or page_size not supported";
    case SEED_ERR_CUDA: return "CUDA launch failed";
    case SEED_ERR_WORKSPACE: return "workspace too small or misaligned";
    case SEED_ERR_SCRATCH_LIMIT:
      return "problem needs more workspace than the built-in scratch holds";
  }
  return "unknown status";
}

size_t seed_workspace_bytes(const seed_cfg_t* cfg, int32_t batch) {
  if (check_cfg(cfg) != SEED_OK || batch < 0) return 0;
  const int G = cfg->hq / cfg->hkv;
  const int32_t nv_max = batch * (cfg->kmax + 1);
  size_t part = seedk::decode_workspace_bound(nv_max, cfg->hkv, G, cfg->head_dim);
  if (tc_path(cfg->head_dim, G, 1))
    part = std::max(part, seedk::attn_tc_part_bound(G, 1, cfg->head_dim));
  if (tc_path(cfg->head_dim, G, cfg->kmax + 1))
    part = std::max(part, seedk::attn_tc_part_bound(G, cfg->kmax + 1, cfg->head_dim));
  return zero_prefix(cfg, batch) + round_up(part, kAlign);
}

seed_status_t seed_draft_kv_append(const seed_cfg_t* cfg, int32_t batch, const void* k_new,
                                   const void* v_new, const int32_t* draft_lens, void* draft_k,
                                   void* draft_v, int32_t* err_flag, void* stream) {
  seed_status_t st = check_cfg(cfg);
  if (st != SEED_OK) return st;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!k_new || !v_new || !draft_lens || !draft_k || !draft_v || !err_flag) return SEED_ERR_NULL;
  if (misaligned16(k_new) || misaligned16(v_new) || misaligned16(draft_k) || misaligned16(draft_v))
    return SEED_ERR_RANGE;
  return finish(seedk::launch_draft_append(
      batch, cfg->hkv, cfg->head_dim, cfg->kmax, static_cast<const uint16_t*>(k_new),
      static_cast<const uint16_t*>(v_new), draft_lens, static_cast<uint16_t*>(draft_k),
      static_cast<uint16_t*>(draft_v), err_flag, static_cast<cudaStream_t>(stream)));
}

seed_status_t seed_draft_attn(const seed_cfg_t* cfg, int32_t batch, const void* q,
                              seed_kv_t ctx_kv, const void* draft_k, const void* draft_v,
                              const int32_t* ctx_lens, const int32_t* draft_lens, float* out,
                              float* lse, void* ws, size_t ws_bytes, int32_t* err_flag,
                              void* stream) {
  seed_status_t st = check_cfg(cfg);
  if (st != SEED_OK) return st;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!q || !draft_k || !draft_v || !ctx_lens || !draft_lens || !out || !ws || !err_flag)
    return SEED_ERR_NULL;
  if ((st = check_kv(ctx_kv)) != SEED_OK) return st;
  if (misaligned16(q) || misaligned16(ctx_kv.k) || misaligned16(ctx_kv.v) ||
      misaligned16(draft_k) || misaligned16(draft_v))
    return SEED_ERR_RANGE;
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0) return SEED_ERR_WORKSPACE;
  if (tc_path(cfg->head_dim, cfg->hq / cfg->hkv, 1))
    return run_attn_tc(cfg, batch, true, q, draft_lens, ctx_kv, draft_k, draft_v, ctx_lens, out,
                       lse, ws, ws_bytes, err_flag, stream);
  return run_decode(cfg, batch, false, q, ctx_kv, draft_k, draft_v, ctx_lens, draft_lens, out, lse,
                    ws, ws_bytes, err_flag, stream);
}

seed_status_t seed_kv_append(const seed_cfg_t* cfg, int32_t batch, seed_kv_t kv,
                             const void* k_new, const void* v_new, const int32_t* n_new,
                             const int32_t* ctx_lens, int32_t* err_flag, void* stream) {
  seed_status_t st = check_cfg(cfg);
  if (st != SEED_OK) return st;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!k_new || !v_new || !n_new || !ctx_lens || !err_flag) return SEED_ERR_NULL;
  if ((st = check_kv(kv)) != SEED_OK) return st;
  if (misaligned16(k_new) || misaligned16(v_new) || misaligned16(kv.k) || misaligned16(kv.v))
    return SEED_ERR_RANGE;
  return finish(seedk::launch_kv_append(
      batch, cfg->hkv, cfg->head_dim, cfg->kmax, static_cast<uint16_t*>(kv.k),
      static_cast<uint16_t*>(kv.v), kv.page_table, kv.max_pages, kv.num_pages,
      static_cast<const uint16_t*>(k_new), static_cast<const uint16_t*>(v_new), n_new, ctx_lens,
      err_flag, static_cast<cudaStream_t>(stream)));
}

seed_status_t seed_verify_attn(const seed_cfg_t* cfg, int32_t batch, const void* q,
                               const int32_t* n_q, seed_kv_t kv, const int32_t* ctx_lens,
                               float* out, float* lse, void* ws, size_t ws_bytes,
                               int32_t* err_flag, void* stream) {
  seed_status_t st = check_cfg(cfg);
  if (st != SEED_OK) return st;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!q || !n_q || !ctx_lens || !out || !ws || !err_flag) return SEED_ERR_NULL;
  if ((st = check_kv(kv)) != SEED_OK) return st;
  if (misaligned16(q) || misaligned16(kv.k) || misaligned16(kv.v)) return SEED_ERR_RANGE;
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0) return SEED_ERR_WORKSPACE;
  if (tc_path(cfg->head_dim, cfg->hq / cfg->hkv, cfg->kmax + 1))
    return run_attn_tc(cfg, batch, false, q, n_q, kv, nullptr, nullptr, ctx_lens, out, lse, ws,
                       ws_bytes, err_flag, stream);
  return run_decode(cfg, batch, true, q, kv, nullptr, nullptr, ctx_lens, n_q, out, lse, ws,
                    ws_bytes, err_flag, stream);
}

int32_t seed_attn_route(const seed_cfg_t* cfg, int32_t batch, int32_t draft, int32_t max_pages) {
  if (check_cfg(cfg) != SEED_OK || batch < 1 || max_pages < 1) return -1;
  const int G = cfg->hq / cfg->hkv;
  const int W1 = draft ? 1 : cfg->kmax + 1;
  if (!tc_path(cfg->head_dim, G, W1)) return SEED_ROUTE_CUDA_CORE;
  const int cluster = seedk::attn_cl_route(cfg->head_dim, G, W1, batch, cfg->hkv, max_pages);
  if (cluster > 0) return cluster;
  return seedk::attn_kt_supported(cfg->head_dim, G, W1) ? SEED_ROUTE_TC_KEYS : SEED_ROUTE_TC_ROWS;
}

seed_status_t seed_tree_verify_attn(const seed_cfg_t* cfg, int32_t batch, const void* q,
                                    const int32_t* n_nodes, const uint32_t* anc, seed_kv_t kv,
                                    const int32_t* ctx_lens, float* out, float* lse, void* ws,
                                    size_t ws_bytes, int32_t* err_flag, void* stream) {
  seed_status_t st = check_cfg(cfg);
  if (st != SEED_OK) return st;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (!tc_path(cfg->head_dim, cfg->hq / cfg->hkv, cfg->kmax + 1)) return SEED_ERR_UNSUPPORTED;
  if (batch == 0) return SEED_OK;
  if (!q || !n_nodes || !anc || !ctx_lens || !out || !ws || !err_flag) return SEED_ERR_NULL;
  if ((st = check_kv(kv)) != SEED_OK) return st;
  if (misaligned16(q) || misaligned16(kv.k) || misaligned16(kv.v)) return SEED_ERR_RANGE;
  if ((reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0) return SEED_ERR_WORKSPACE;
  return run_attn_tc(cfg, batch, false, q, n_nodes, kv, nullptr, nullptr, ctx_lens, out, lse, ws,
                     ws_bytes, err_flag, stream, anc);
}

seed_status_t seed_accept_commit(int32_t batch, int32_t kmax, const int32_t* draft_ids,
                                 const int32_t* target_ids, const int32_t* k_b,
                                 const int32_t* page_table, int32_t max_pages,
                                 int32_t page_size, int32_t* ctx_lens, int32_t* accepted,
                                 int32_t* tokens, int32_t* committed_slots, int32_t* err_flag,
                                 void* stream) {
  if (batch < 0 || kmax < 1 || kmax > SEED_MAX_KMAX) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!draft_ids || !target_ids || !k_b || !page_table || !ctx_lens || !accepted || !tokens ||
      !committed_slots || !err_flag)
    return SEED_ERR_NULL;
  if (max_pages <= 0 || page_size <= 0 || (long long)max_pages * page_size > INT32_MAX)
    return SEED_ERR_RANGE;
  return finish(seedk::launch_accept(batch, kmax, draft_ids, target_ids, k_b, page_table,
                                     max_pages, page_size, ctx_lens, accepted, tokens,
                                     committed_slots, err_flag,
                                     static_cast<cudaStream_t>(stream)));
}

seed_status_t seed_tree_accept_commit(int32_t batch, int32_t kmax, const int32_t* tok,
                                      const int32_t* parent, const int32_t* n_nodes,
                                      const int32_t* target_ids, const int32_t* page_table,
                                      int32_t max_pages, int32_t page_size, int32_t* ctx_lens,
                                      int32_t* accepted, int32_t* tokens, int32_t* path,
                                      int32_t* committed_slots, int32_t* err_flag,
                                      void* stream) {
  if (batch < 0 || kmax < 1 || kmax > SEED_MAX_KMAX) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!tok || !parent || !n_nodes || !target_ids || !page_table || !ctx_lens || !accepted ||
      !tokens || !path || !committed_slots || !err_flag)
    return SEED_ERR_NULL;
  if (max_pages <= 0 || page_size <= 0 || (long long)max_pages * page_size > INT32_MAX)
    return SEED_ERR_RANGE;
  return finish(seedk::launch_tree_accept(batch, kmax, tok, parent, n_nodes, target_ids,
                                          page_table, max_pages, page_size, ctx_lens, accepted,
                                          tokens, path, committed_slots, err_flag,
                                          static_cast<cudaStream_t>(stream)));
}

seed_status_t seed_tree_kv_compact(const seed_cfg_t* cfg, int32_t batch, seed_kv_t kv,
                                   const int32_t* path, const int32_t* accepted,
                                   const int32_t* ctx_lens, int32_t* err_flag, void* stream) {
  seed_status_t st = check_cfg(cfg);
  if (st != SEED_OK) return st;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!path || !accepted || !ctx_lens || !err_flag) return SEED_ERR_NULL;
  if ((st = check_kv(kv)) != SEED_OK) return st;
  if (misaligned16(kv.k) || misaligned16(kv.v)) return SEED_ERR_RANGE;
  return finish(seedk::launch_tree_compact(
      batch, cfg->hkv, cfg->head_dim, cfg->kmax, static_cast<uint16_t*>(kv.k),
      static_cast<uint16_t*>(kv.v), kv.page_table, kv.max_pages, kv.num_pages, path, accepted,
      ctx_lens, err_flag, static_cast<cudaStream_t>(stream)));
}

size_t seed_draft_head_workspace_bytes(int32_t batch) {
  if (batch < 1 || batch > SEED_DRAFT_HEAD_MAX_BATCH) return 0;
  return seedk::head_workspace_bytes(batch);
}

seed_status_t seed_draft_head_topk(int32_t batch, int32_t d_model, int32_t vocab,
                                   const void* h, const void* w_out, float tau, int32_t* ids,
                                   float* probs, int32_t* n_sib, int32_t* stop, float* lse,
                                   void* ws, size_t ws_bytes, int32_t* err_flag, void* stream) {
  if (batch < 0 || batch > SEED_DRAFT_HEAD_MAX_BATCH) return SEED_ERR_SHAPE;
  if (d_model <= 0 || d_model % 64 != 0 || vocab < SEED_DRAFT_TOPK) return SEED_ERR_SHAPE;
  if (!(tau >= 0.f) || std::isinf(tau)) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!h || !w_out || !ids || !probs || !n_sib || !stop || !ws || !err_flag) return SEED_ERR_NULL;
  if (misaligned16(h) || misaligned16(w_out)) return SEED_ERR_RANGE;
  if ((reinterpret_cast<uintptr_t>(ws) & 15u) != 0 ||
      ws_bytes < seedk::head_workspace_bytes(batch))
    return SEED_ERR_WORKSPACE;
  seedk::HeadParams p{};
  p.part = static_cast<float*>(ws);
  p.ids = ids;
  p.probs = probs;
  p.n_sib = n_sib;
  p.stop = stop;
  p.lse = lse;
  p.err = err_flag;
  p.B = batch;
  p.d = d_model;
  p.V = vocab;
  p.tau = tau;
  return finish(seedk::launch_head(p, h, w_out, seedk::head_ctas(vocab),
                                   static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
