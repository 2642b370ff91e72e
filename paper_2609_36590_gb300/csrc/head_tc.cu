// The drafter's LM head with a fused softmax and top-k, for confidence-aware
// dynamic drafting (Sec. D.1): per sequence, logits z = W_out h over the whole
// vocabulary are never stored; the kernel keeps the log-sum-exp and the ten
// most probable tokens, from which the top-1 probability p0 gives the number
// of sibling candidates k (1, 3, 5 or 10) and the stop decision p0 <= tau.
//
// Design.  The contraction [B, d] x [d, V] is a dense GEMM, memory-bound on
// the 2 V d bytes of W for small B, so it runs on the tensor cores: sequences
// are the M = 128 rows of a tcgen05 MMA (bf16 -> f32), 256 vocabulary rows the
// N columns, and K runs over d in slabs of 64.  A 4-stage TMA ring holds each
// slab's h (B rows) and W (256 rows) tiles; two TMEM accumulators of 256
// columns let the MMAs of one vocabulary tile run while the previous tile's
// logits are consumed.  Each epilogue thread owns one sequence (one TMEM
// lane): per tile it takes the maximum, accumulates sum 2^(z log2 e - max) and
// keeps a register top-10 (scanning ids upwards, so equal logits keep the
// lower id first).  CTAs take contiguous ranges of vocabulary tiles; each
// leaves per-sequence partials that a small kernel merges.
//
// Warp roles (192 threads): warps 0-3 epilogue (TMEM lane quarters), warp 4
// TMA producer, warp 5 MMA issuer and TMEM owner.  Every wait is bounded; a
// wait that gives up raises SEED_DEVERR_TIMEOUT.
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace seedk {
namespace {

constexpr int kHN = 256;                       // vocabulary rows per tile
constexpr int kHK = 64;                        // head dims per K slab
constexpr int kHStages = 4;
constexpr int kHTopK = 10;
constexpr int kHThreads = 192;
constexpr int kHWarpProd = 4, kHWarpMma = 5;
constexpr uint32_t kHSlabA = 128u * 128u;      // h slab: 128 rows x 128 B (B rows loaded)
constexpr uint32_t kHSlabB = kHN * 128u;       // W slab: 256 rows x 128 B
constexpr uint32_t kHStage = kHSlabA + kHSlabB;
constexpr uint32_t kHOffCtrl = kHStages * kHStage;
constexpr uint32_t kHIdesc = idesc_bf16_f32(128, kHN, 0, 0);
constexpr unsigned kFullH = 0xffffffffu;
constexpr float kLog2e = 1.4426950408889634f;

struct HCtrl {
  uint64_t full[kHStages], empty[kHStages];
  uint64_t d_full[2], d_empty[2];
  uint32_t tmem_base;
  volatile int32_t abort_flag;
};

constexpr size_t kSmemHead = kHOffCtrl + sizeof(HCtrl) + 1024;
static_assert(kSmemHead <= 232448, "shared memory budget");

__device__ __noinline__ bool hwait(uint64_t* bar, uint32_t parity, HCtrl* c, int32_t* err) {
  for (uint32_t i = 0; i < kSuspendTries; ++i) {
    if (mbar_try_wait_sleep(bar, parity, kSuspendNs)) return true;
    if (c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ bool hwarp_wait(uint64_t* bar, uint32_t parity, HCtrl* c,
                                           int32_t* err) {
  return __all_sync(kFullH, hwait(bar, parity, c, err));
}

// Insert (z, id) into a descending top-10 (equal values keep the earlier id).
__device__ __forceinline__ void top_insert(float (&tv)[kHTopK], int (&ti)[kHTopK], float z, int id) {
  if (!(z > tv[kHTopK - 1])) return;
  tv[kHTopK - 1] = z;
  ti[kHTopK - 1] = id;
#pragma unroll
  for (int k = kHTopK - 1; k > 0; --k) {
    if (tv[k] > tv[k - 1]) {
      const float a = tv[k];
      tv[k] = tv[k - 1];
      tv[k - 1] = a;
      const int b = ti[k];
      ti[k] = ti[k - 1];
      ti[k - 1] = b;
    }
  }
}

// Partial record of one (CTA, sequence): [0] running max (log2 units), [1]
// sum 2^(zs - max), [2..11] top logits (natural units), [12..21] their ids.
constexpr int kHRec = 24;

__global__ void __launch_bounds__(kHThreads) head_tc_kernel(
    const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_w,
    const HeadParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  HCtrl* ctrl = reinterpret_cast<HCtrl*>(smem + kHOffCtrl);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  if (tid == 0) pdl_trigger();
  const int nqa = (p.B + 31) / 32;   // epilogue warps with sequences
  if (tid == 0) {
    for (int s = 0; s < kHStages; ++s) {
      mbar_init(&ctrl->full[s], 1);
      mbar_init(&ctrl->empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->d_full[i], 1);
      mbar_init(&ctrl->d_empty[i], nqa);
    }
    ctrl->abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kHWarpMma) {
    tmem_alloc(&ctrl->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctrl->tmem_base;
  pdl_wait();

  // this CTA's vocabulary tiles [t0, t1)
  const int ntiles = (p.V + kHN - 1) / kHN;
  const int t0 = (int)((long long)ntiles * blockIdx.x / gridDim.x);
  const int t1 = (int)((long long)ntiles * (blockIdx.x + 1) / gridDim.x);
  const int nslab = p.d / kHK;
  const uint32_t bpad = (uint32_t)((p.B + 7) & ~7);

  if (warp == kHWarpProd) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_h);
      tma_prefetch_desc(&tm_w);
    }
    int it = 0;
    bool ok = true;
    for (int t = t0; t < t1 && ok; ++t) {
      for (int k = 0; k < nslab && ok; ++k, ++it) {
        const int s = it % kHStages;
        if (it >= kHStages) ok = hwarp_wait(&ctrl->empty[s], ((it / kHStages) - 1) & 1, ctrl, p.err);
        if (ok && lane == 0) {
          uint8_t* st = smem + (size_t)s * kHStage;
          mbar_arrive_expect_tx(&ctrl->full[s], bpad * 128u + kHSlabB);
          tma_load_2d(st, &tm_h, k * kHK, 0, &ctrl->full[s]);
          tma_load_2d(st + kHSlabA, &tm_w, k * kHK, t * kHN, &ctrl->full[s]);
        }
        __syncwarp();
      }
    }
  } else if (warp == kHWarpMma) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      int it = 0;
      for (int t = t0, n = 0; t < t1; ++t, ++n) {
        const uint32_t d = tmem + (uint32_t)(n & 1) * kHN;
        if (n >= 2 && !hwait(&ctrl->d_empty[n & 1], ((n >> 1) - 1) & 1, ctrl, p.err)) break;
        bool ok = true;
        for (int k = 0; k < nslab; ++k, ++it) {
          const int s = it % kHStages;
          if (!hwait(&ctrl->full[s], (it / kHStages) & 1, ctrl, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = sbase + (uint32_t)s * kHStage;
          const uint32_t b0 = a0 + kHSlabA;
#pragma unroll 1
          for (int kk = 0; kk < kHK / 16; ++kk) {
            const uint64_t a = smem_desc_sw128(a0 + kk * 32, 16, 1024);
            const uint64_t b = smem_desc_sw128(b0 + kk * 32, 16, 1024);
            mma_ss(d, a, b, kHIdesc, (k > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(&ctrl->empty[s]);
        }
        if (!ok) break;
        mma_commit(&ctrl->d_full[n & 1]);
      }
    }
    __syncwarp();
  } else if (warp < 4 && warp < nqa) {
    // ---------------------------------------------------------- epilogue
    const int b = warp * 32 + lane;           // this thread's sequence
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    float m2 = -INFINITY, l = 0.f;
    float tv[kHTopK];
    int ti[kHTopK];
#pragma unroll
    for (int k = 0; k < kHTopK; ++k) {
      tv[k] = -INFINITY;
      ti[k] = -1;
    }
    for (int t = t0, n = 0; t < t1; ++t, ++n) {
      if (!hwarp_wait(&ctrl->d_full[n & 1], (n >> 1) & 1, ctrl, p.err)) break;
      tc_fence_after();
      const uint32_t col = tmem + lane_off + (uint32_t)(n & 1) * kHN;
      const int v0 = t * kHN;
      // pass 1: the tile's maximum
      float mx = -INFINITY;
#pragma unroll 1
      for (int c = 0; c < kHN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(col + c * 32, r);
        tmem_wait_ld();
        const int nv = min(32, p.V - (v0 + 32 * c));
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (i < nv) mx = fmaxf(mx, __uint_as_float(r[i]));
      }
      const float mt = mx * kLog2e;
      if (mt > m2) {
        l *= (m2 == -INFINITY) ? 0.f : ex2_approx(m2 - mt);
        m2 = mt;
      }
      // pass 2: the sum and the top tokens
      float ls = 0.f;
#pragma unroll 1
      for (int c = 0; c < kHN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(col + c * 32, r);
        tmem_wait_ld();
        const int nv = min(32, p.V - (v0 + 32 * c));
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          if (i < nv) {
            const float z = __uint_as_float(r[i]);
            ls += ex2_approx(fmaf(z, kLog2e, -m2));
            top_insert(tv, ti, z, v0 + 32 * c + i);
          }
        }
      }
      l += ls;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->d_empty[n & 1]);
    }
    if (b < p.B) {
      float* rec = p.part + ((size_t)blockIdx.x * p.B + b) * kHRec;
      rec[0] = m2;
      rec[1] = l;
#pragma unroll
      for (int k = 0; k < kHTopK; ++k) {
        rec[2 + k] = tv[k];
        rec[2 + kHTopK + k] = __int_as_float(ti[k]);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kHWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// One warp per sequence: merge the CTAs' partials into the log-sum-exp and
// the global top-10, then apply the sibling-count rule and the stop rule.
__global__ void head_merge_kernel(const HeadParams p, int nctas) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, lane = threadIdx.x;
  if (b >= p.B) return;
  float M = -INFINITY;
  for (int c = lane; c < nctas; c += 32) M = fmaxf(M, p.part[((size_t)c * p.B + b) * kHRec]);
  for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(kFullH, M, o));
  float L = 0.f;
  float tv[kHTopK];
  int ti[kHTopK];
#pragma unroll
  for (int k = 0; k < kHTopK; ++k) {
    tv[k] = -INFINITY;
    ti[k] = -1;
  }
  for (int c = lane; c < nctas; c += 32) {
    const float* rec = p.part + ((size_t)c * p.B + b) * kHRec;
    if (rec[0] != -INFINITY) L += rec[1] * ex2_approx(rec[0] - M);
#pragma unroll
    for (int k = 0; k < kHTopK; ++k) {
      const int id = __float_as_int(rec[2 + kHTopK + k]);
      if (id < 0) continue;
      // equal logits from a later CTA carry larger ids: keep the earlier one
      const float z = rec[2 + k];
      if (z > tv[kHTopK - 1] || (z == tv[kHTopK - 1] && id < ti[kHTopK - 1])) {
        tv[kHTopK - 1] = z;
        ti[kHTopK - 1] = id;
#pragma unroll
        for (int j = kHTopK - 1; j > 0; --j) {
          if (tv[j] > tv[j - 1] || (tv[j] == tv[j - 1] && ti[j] < ti[j - 1])) {
            const float a = tv[j];
            tv[j] = tv[j - 1];
            tv[j - 1] = a;
            const int q = ti[j];
            ti[j] = ti[j - 1];
            ti[j - 1] = q;
          }
        }
      }
    }
  }
  for (int o = 16; o; o >>= 1) L += __shfl_xor_sync(kFullH, L, o);
  const float lse2 = M + log2f(L);
  // pop the best head of all lanes' lists ten times
  float p0 = 0.f;
  for (int k = 0; k < kHTopK; ++k) {
    float bz = tv[0];
    int bi = ti[0], bl = lane;
    for (int o = 16; o; o >>= 1) {
      const float oz = __shfl_xor_sync(kFullH, bz, o);
      const int oi = __shfl_xor_sync(kFullH, bi, o);
      const int ol = __shfl_xor_sync(kFullH, bl, o);
      const bool take = (oi >= 0) && (bi < 0 || oz > bz || (oz == bz && oi < bi));
      if (take) {
        bz = oz;
        bi = oi;
        bl = ol;
      }
    }
    if (lane == bl) {
#pragma unroll
      for (int j = 0; j < kHTopK - 1; ++j) {
        tv[j] = tv[j + 1];
        ti[j] = ti[j + 1];
      }
      tv[kHTopK - 1] = -INFINITY;
      ti[kHTopK - 1] = -1;
    }
    const float pr = bi >= 0 ? exp2f(fmaf(bz, kLog2e, -lse2)) : 0.f;
    if (k == 0) p0 = pr;
    if (lane == 0) {
      p.ids[(size_t)b * kHTopK + k] = bi;
      p.probs[(size_t)b * kHTopK + k] = pr;
    }
  }
  if (lane == 0) {
    p.n_sib[b] = p0 > 0.95f ? 1 : p0 > 0.8f ? 3 : p0 > 0.5f ? 5 : 10;
    p.stop[b] = p0 <= p.tau ? 1 : 0;
    if (p.lse != nullptr) p.lse[b] = lse2 / kLog2e;
  }
}

// ------------------------------------------------------------- host side
using EncodeTiledFn2 = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                    const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                    const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                    CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn2 encode_fn2() {
  static EncodeTiledFn2 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn2>(ptr);
  });
  return fn;
}

// 2-d bf16 map [rows, d], 64-element x `box_rows` boxes, 128-byte swizzle.
bool encode_2d(CUtensorMap* map, const void* base, uint64_t d, uint64_t rows,
               uint32_t box_rows) {
  EncodeTiledFn2 fn = encode_fn2();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {d, rows};
  const cuuint64_t strides[1] = {d * 2ull};
  const cuuint32_t box[2] = {(cuuint32_t)kHK, box_rows};
  const cuuint32_t elem[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

std::atomic<uint64_t> g_head_attr_set{0};

}  // namespace

int head_ctas(int32_t vocab) {
  const int ntiles = (vocab + kHN - 1) / kHN;
  return std::max(1, std::min(std::min(device_sm_count(), kHeadMaxCtas), ntiles));
}

cudaError_t launch_head(const HeadParams& prm, const void* h, const void* w, int nctas,
                        cudaStream_t st) {
  CUtensorMap th, tw;
  const uint32_t bpad = (uint32_t)((prm.B + 7) & ~7);
  if (!encode_2d(&th, h, (uint64_t)prm.d, (uint64_t)prm.B, bpad)) return cudaErrorInvalidValue;
  if (!encode_2d(&tw, w, (uint64_t)prm.d, (uint64_t)prm.V, kHN)) return cudaErrorInvalidValue;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(g_head_attr_set.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(head_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmemHead);
    if (e != cudaSuccess) return e;
    g_head_attr_set.fetch_or(bit, std::memory_order_acq_rel);
  }
  e = launch_pdl(head_tc_kernel, dim3(nctas), dim3(kHThreads), kSmemHead, st, th, tw, prm);
  if (e != cudaSuccess) return e;
  return launch_pdl(head_merge_kernel, dim3(prm.B), dim3(32), 0, st, prm, nctas);
}

size_t head_workspace_bytes(int32_t batch) {
  return (size_t)kHeadMaxCtas * batch * kHRec * sizeof(float);
}

}  // namespace seedk
