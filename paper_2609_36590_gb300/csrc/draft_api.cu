// C ABI of the draft step on the device (include/seed.h, "The whole draft
// step"): the skinny products, embedding, RMS norm, and one decoder layer of
// a draft step composed from them and the draft attention calls.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "../../include/seed.h"
#include "kernels.h"

namespace {

seed_status_t fin(cudaError_t e) { return e == cudaSuccess ? SEED_OK : SEED_ERR_CUDA; }
bool mis16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; }
bool mis8(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 7u) != 0; }
size_t up256(size_t n) { return (n + 255) & ~(size_t)255; }

bool linear_shape_ok(int32_t batch, int32_t n_out, int32_t k_in, int32_t epi) {
  return batch >= 0 && batch <= SEED_LINEAR_MAX_BATCH && n_out > 0 &&
         n_out <= seedk::kLinearMaxTiles * 128 && k_in > 0 && k_in % 64 == 0 &&
         (epi == SEED_LINEAR_F32 || epi == SEED_LINEAR_RESID_F32 || epi == SEED_LINEAR_SWIGLU);
}

// The layer's temporaries, carved from its workspace.
struct LayerWs {
  size_t attn, lin, a, qkv, q, o, ob, m, act, total;
};

LayerWs layer_ws(const seed_cfg_t* cfg, const seed_decoder_layer_t* L, int32_t B) {
  LayerWs w{};
  const int32_t D = cfg->head_dim, hq = cfg->hq, hkv = cfg->hkv;
  const int32_t nqkv = (hq + 2 * hkv) * D;
  size_t lin = seedk::linear_workspace_bytes(B, nqkv, L->d_model, SEED_LINEAR_F32);
  lin = std::max(lin, seedk::linear_workspace_bytes(B, L->d_model, hq * D, SEED_LINEAR_RESID_F32));
  lin = std::max(lin, seedk::linear_workspace_bytes(B, L->d_ff, L->d_model, SEED_LINEAR_SWIGLU));
  lin = std::max(lin, seedk::linear_workspace_bytes(B, L->d_model, L->d_ff, SEED_LINEAR_RESID_F32));
  size_t off = 0;
  auto take = [&](size_t n) {
    const size_t o = off;
    off += up256(n);
    return o;
  };
  w.attn = take(seed_workspace_bytes(cfg, B));
  w.lin = take(lin);
  w.a = take((size_t)B * L->d_model * 2);
  w.qkv = take((size_t)B * nqkv * 4);
  w.q = take((size_t)B * hq * D * 2);
  w.o = take((size_t)B * hq * D * 4);
  w.ob = take((size_t)B * hq * D * 2);
  w.m = take((size_t)B * L->d_model * 2);
  w.act = take((size_t)B * L->d_ff * 2);
  w.total = off;
  return w;
}

bool layer_ok(const seed_cfg_t* cfg, const seed_decoder_layer_t* L) {
  if (cfg == nullptr || L == nullptr) return false;
  if (cfg->head_dim != 64 && cfg->head_dim != 128) return false;
  if (L->d_model <= 0 || L->d_model % 64 != 0 || L->d_ff <= 0 || L->d_ff % 64 != 0) return false;
  if (!(L->rms_eps > 0.f) || !(L->rope_theta > 1.f) || std::isinf(L->rope_theta)) return false;
  return true;
}

}  // namespace

extern "C" {

size_t seed_linear_workspace_bytes(int32_t batch, int32_t n_out, int32_t k_in, int32_t epilogue) {
  if (!linear_shape_ok(batch, n_out, k_in, epilogue) || batch == 0) return 0;
  return seedk::linear_workspace_bytes(batch, n_out, k_in, epilogue);
}

seed_status_t seed_linear(int32_t batch, int32_t k_in, int32_t n_out, const void* x,
                          const void* w, const void* w2, int32_t epilogue, void* y, void* ws,
                          size_t ws_bytes, int32_t* err_flag, void* stream) {
  if (!linear_shape_ok(batch, n_out, k_in, epilogue)) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  const bool swiglu = epilogue == SEED_LINEAR_SWIGLU;
  if (!x || !w || !y || !ws || !err_flag || (swiglu && !w2)) return SEED_ERR_NULL;
  if (mis16(x) || mis16(w) || (swiglu && mis16(w2)) || mis16(y)) return SEED_ERR_RANGE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 ||
      ws_bytes < seedk::linear_workspace_bytes(batch, n_out, k_in, epilogue))
    return SEED_ERR_WORKSPACE;
  seedk::LinearParams p{};
  p.y = y;
  p.err = err_flag;
  p.B = batch;
  p.K = k_in;
  p.N = n_out;
  p.epi = epilogue;
  return fin(seedk::launch_linear(p, x, w, swiglu ? w2 : nullptr, ws,
                                  static_cast<cudaStream_t>(stream)));
}

seed_status_t seed_embed(int32_t batch, int32_t d_model, int32_t vocab, const int32_t* tokens,
                         const void* w_emb, float* x, int32_t* err_flag, void* stream) {
  if (batch < 0 || d_model <= 0 || d_model % 4 != 0 || vocab <= 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  if (!tokens || !w_emb || !x || !err_flag) return SEED_ERR_NULL;
  if (mis8(w_emb) || mis16(x)) return SEED_ERR_RANGE;
  return fin(seedk::launch_embed(batch, d_model, vocab, tokens, w_emb, x, err_flag,
                                 static_cast<cudaStream_t>(stream)));
}

seed_status_t seed_rmsnorm(int32_t rows, int32_t n, const float* x, const void* gamma, float eps,
                           void* y, void* stream) {
  if (rows < 0 || n <= 0 || n % 4 != 0 || !(eps > 0.f)) return SEED_ERR_SHAPE;
  if (rows == 0) return SEED_OK;
  if (!x || !gamma || !y) return SEED_ERR_NULL;
  if (mis16(x) || mis8(gamma) || mis8(y)) return SEED_ERR_RANGE;
  return fin(seedk::launch_rmsnorm(rows, n, x, gamma, eps, y, static_cast<cudaStream_t>(stream)));
}

size_t seed_draft_layer_workspace_bytes(const seed_cfg_t* cfg, const seed_decoder_layer_t* layer,
                                        int32_t batch) {
  if (!layer_ok(cfg, layer) || batch < 1 || batch > SEED_LINEAR_MAX_BATCH) return 0;
  if (seed_workspace_bytes(cfg, batch) == 0) return 0;
  return layer_ws(cfg, layer, batch).total;
}

seed_status_t seed_draft_layer(const seed_cfg_t* cfg, int32_t batch,
                               const seed_decoder_layer_t* layer, float* x, seed_kv_t ctx_kv,
                               const int32_t* ctx_lens, void* draft_k, void* draft_v,
                               const int32_t* draft_lens, void* ws, size_t ws_bytes,
                               int32_t* err_flag, void* stream) {
  if (cfg == nullptr || layer == nullptr) return SEED_ERR_NULL;
  if (!layer_ok(cfg, layer)) return SEED_ERR_UNSUPPORTED;
  if (batch < 0 || batch > SEED_LINEAR_MAX_BATCH) return SEED_ERR_SHAPE;
  if (seed_workspace_bytes(cfg, batch > 0 ? batch : 1) == 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  const seed_decoder_layer_t& L = *layer;
  if (!x || !ctx_lens || !draft_k || !draft_v || !draft_lens || !ws || !err_flag || !L.g_attn ||
      !L.w_qkv || !L.g_q || !L.g_k || !L.w_o || !L.g_mlp || !L.w_gate || !L.w_up || !L.w_down)
    return SEED_ERR_NULL;
  if (mis16(L.w_qkv) || mis16(L.w_o) || mis16(L.w_gate) || mis16(L.w_up) || mis16(L.w_down) ||
      mis16(x) || mis8(L.g_attn) || mis8(L.g_mlp))
    return SEED_ERR_RANGE;
  const LayerWs w = layer_ws(cfg, layer, batch);
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0 || ws_bytes < w.total) return SEED_ERR_WORKSPACE;
  char* base = static_cast<char*>(ws);
  auto at = [&](size_t off) { return static_cast<void*>(base + off); };
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int32_t D = cfg->head_dim, hq = cfg->hq, hkv = cfg->hkv, dm = L.d_model, F = L.d_ff;
  const int32_t nqkv = (hq + 2 * hkv) * D;
  const size_t lin_bytes = w.a - w.lin;
  seed_status_t s;

  if ((s = fin(seedk::launch_rmsnorm(batch, dm, x, L.g_attn, L.rms_eps, at(w.a), st))) != SEED_OK)
    return s;
  if ((s = seed_linear(batch, dm, nqkv, at(w.a), L.w_qkv, nullptr, SEED_LINEAR_F32, at(w.qkv),
                       at(w.lin), lin_bytes, err_flag, stream)) != SEED_OK)
    return s;
  // q/k norms and RoPE; k and v land in row i-1 of the draft scratch (the
  // draft KV append of this step)
  if ((s = fin(seedk::launch_qk_norm_rope(
           batch, hq, hkv, D, static_cast<const float*>(at(w.qkv)), L.g_q, L.g_k, ctx_lens,
           draft_lens, L.rope_theta, L.rms_eps, cfg->kmax, at(w.q), draft_k, draft_v, err_flag,
           st))) != SEED_OK)
    return s;
  if ((s = seed_draft_attn(cfg, batch, at(w.q), ctx_kv, draft_k, draft_v, ctx_lens, draft_lens,
                           static_cast<float*>(at(w.o)), nullptr, at(w.attn),
                           seed_workspace_bytes(cfg, batch), err_flag, stream)) != SEED_OK)
    return s;
  if ((s = fin(seedk::launch_f32_to_bf16((size_t)batch * hq * D,
                                         static_cast<const float*>(at(w.o)), at(w.ob), st))) !=
      SEED_OK)
    return s;
  if ((s = seed_linear(batch, hq * D, dm, at(w.ob), L.w_o, nullptr, SEED_LINEAR_RESID_F32, x,
                       at(w.lin), lin_bytes, err_flag, stream)) != SEED_OK)
    return s;
  if ((s = fin(seedk::launch_rmsnorm(batch, dm, x, L.g_mlp, L.rms_eps, at(w.m), st))) != SEED_OK)
    return s;
  if ((s = seed_linear(batch, dm, F, at(w.m), L.w_gate, L.w_up, SEED_LINEAR_SWIGLU, at(w.act),
                       at(w.lin), lin_bytes, err_flag, stream)) != SEED_OK)
    return s;
  return seed_linear(batch, F, dm, at(w.act), L.w_down, nullptr, SEED_LINEAR_RESID_F32, x,
                     at(w.lin), lin_bytes, err_flag, stream);
}

}  // extern "C"
