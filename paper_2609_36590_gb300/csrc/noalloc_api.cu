// seed_verify_attn_noalloc: the verify attention of seed_verify_attn with the
// workspace taken from a fixed scratch array that lives in this library's
// device image, so that the caller allocates nothing at all.
//
// Who needs it: a caller that cannot hand the library device memory of its
// own. Examples are a plain C host with no device allocator it wants to
// expose, and a serving engine that has given all free HBM to its KV page
// pool, so that a workspace allocated at call time could fail. A cudaFree
// elsewhere would also stall the whole device. Both kinds of caller get the
// same kernels and the same numbers as seed_verify_attn.
//
// Cost and limits: the scratch is SEED_NOALLOC_SCRATCH_BYTES of device
// memory on every device where the library's module is loaded. A problem is
// accepted only while seed_workspace_bytes(cfg, batch) fits in it. There is
// one scratch per device, so calls on one device that overlap in time (two
// streams, or two host threads without ordering between them) race on it;
// the caller serialises them.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "../../include/seed.h"

namespace {

// The scratch itself. 256-byte alignment is what the workspace of
// seed_verify_attn requires.
static __device__ __align__(256) unsigned char g_scratch[SEED_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

struct DeviceScratch {
  std::mutex mu;
  void* ptr[kMaxDevices] = {};
};

DeviceScratch& scratch_table() {
  static DeviceScratch t;
  return t;
}

// Device address of g_scratch on the current device. The first call on a
// device resolves it with that device current (this may load the library's
// module on the device); later calls read the cached value.
seed_status_t scratch_on_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return SEED_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return SEED_ERR_CUDA;
  DeviceScratch& t = scratch_table();
  std::lock_guard<std::mutex> lock(t.mu);
  if (t.ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr)
      return SEED_ERR_CUDA;
    t.ptr[dev] = p;
  }
  *out = t.ptr[dev];
  return SEED_OK;
}

// Bytes at the start of the workspace that seed_verify_attn requires to be
// zero: 256 bytes of work-dispenser state, then one int32 arrival counter per
// (sequence, query slot, KV head) with at least 4 slots per sequence, rounded
// up to 256 bytes. The rest of the workspace holds split partial records,
// which are always written before they are read.
size_t zero_prefix_bytes(const seed_cfg_t* cfg, int32_t batch) {
  const size_t slots = (size_t)std::max(cfg->kmax + 1, 4);
  const size_t counters = (size_t)batch * slots * cfg->hkv * sizeof(int32_t);
  return 256 + (counters + 255) / 256 * 256;
}

}  // namespace

extern "C" seed_status_t seed_verify_attn_noalloc(const seed_cfg_t* cfg, int32_t batch,
                                                  const void* q, const int32_t* n_q, seed_kv_t kv,
                                                  const int32_t* ctx_lens, float* out,
                                                  float* lse, int32_t* err_flag, void* stream) {
  if (cfg == nullptr) return SEED_ERR_NULL;
  if (batch < 0) return SEED_ERR_SHAPE;
  if (batch == 0) return SEED_OK;
  const size_t need = seed_workspace_bytes(cfg, batch);
  if (need == 0)  // an invalid cfg: seed_verify_attn's host checks name the reason
    return seed_verify_attn(cfg, batch, q, n_q, kv, ctx_lens, out, lse, nullptr, 0, err_flag,
                            stream);
  if (need > (size_t)SEED_NOALLOC_SCRATCH_BYTES) return SEED_ERR_SCRATCH_LIMIT;
  if (!q || !n_q || !ctx_lens || !out || !err_flag || !kv.k || !kv.v || !kv.page_table)
    return SEED_ERR_NULL;
  void* ws = nullptr;
  seed_status_t st = scratch_on_current_device(&ws);
  if (st != SEED_OK) return st;
  // Clear what must start at zero on the caller's stream, so that a call
  // after one that raised a device error starts from a clean state too.
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(ws, 0, zero_prefix_bytes(cfg, batch), s) != cudaSuccess)
    return SEED_ERR_CUDA;
  return seed_verify_attn(cfg, batch, q, n_q, kv, ctx_lens, out, lse, ws,
                          (size_t)SEED_NOALLOC_SCRATCH_BYTES, err_flag, stream);
}
