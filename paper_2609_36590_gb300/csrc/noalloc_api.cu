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
// the caller serialises them. The scratch's address belongs to the device's
// current context: it is cached with that context's id and looked up again
// when the id changes (after cudaDeviceReset, for instance).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "../../include/seed.h"
#include "kernels.h"

namespace {

// The scratch itself. 256-byte alignment is what the workspace of
// seed_verify_attn requires.
static __device__ __align__(256) unsigned char g_scratch[SEED_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

struct DeviceScratch {
  std::mutex mu;
  void* ptr[kMaxDevices] = {};
  unsigned long long ctx[kMaxDevices] = {};   // id of the context ptr belongs to
};

// Driver entry points for the current context and its id (ids are unique for
// the life of the process, so a new context never matches an old entry).
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

struct DriverFns {
  CtxGetCurrentFn get_current = nullptr;
  CtxGetIdFn get_id = nullptr;
};

const DriverFns& driver_fns() {
  static DriverFns f;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      f.get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  return f;
}

// Id of the calling thread's current context; 0 when there is none or it
// cannot be read (the scratch address is then looked up on every call).
unsigned long long current_context_id() {
  const DriverFns& f = driver_fns();
  if (f.get_current == nullptr || f.get_id == nullptr) return 0;
  CUcontext c = nullptr;
  if (f.get_current(&c) != CUDA_SUCCESS || c == nullptr) return 0;
  unsigned long long id = 0;
  if (f.get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}

DeviceScratch& scratch_table() {
  static DeviceScratch t;
  return t;
}

// Device address of g_scratch on the current device. The first call on a
// device, and the first after the device's context changed, resolves it with
// that device current (this may load the library's module on the device);
// other calls read the cached value.
seed_status_t scratch_on_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return SEED_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return SEED_ERR_CUDA;
  DeviceScratch& t = scratch_table();
  std::lock_guard<std::mutex> lock(t.mu);
  const unsigned long long id = current_context_id();
  if (t.ptr[dev] == nullptr || id == 0 || id != t.ctx[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr)
      return SEED_ERR_CUDA;
    t.ptr[dev] = p;
    t.ctx[dev] = current_context_id();   // the lookup made the context current
  }
  *out = t.ptr[dev];
  return SEED_OK;
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
  if (cudaMemsetAsync(ws, 0, seedk::workspace_zero_prefix_bytes(cfg->kmax, cfg->hkv, batch), s) !=
      cudaSuccess)
    return SEED_ERR_CUDA;
  return seed_verify_attn(cfg, batch, q, n_q, kv, ctx_lens, out, lse, ws,
                          (size_t)SEED_NOALLOC_SCRATCH_BYTES, err_flag, stream);
}
