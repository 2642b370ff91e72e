// Skinny GEMM y = x W^T for the drafter's decoder layers (Sec. 4.1 drafting;
// the per-token work the paper's cost appendix counts: W_Q, W_K, W_V, W_O and
// three MLP matrices per decoder layer).  x is [B, K] bf16 with B <= 128, W is
// [N, K] bf16 (nn.Linear layout); the product is bound by reading W once.
//
// Design.  As in the drafter's head, 128 rows of W are the M = 128 operand of
// a tcgen05 MMA and the B sequences (padded to 16) the N operand, so small
// batches issue small MMAs; K runs in 64-element slabs through a TMA ring of
// as many stages as shared memory holds.  Work is split stream-K: the
// (tile, slab) units of the whole product are cut into equal contiguous
// ranges, one per CTA, so every SM streams the same number of bytes whatever
// N and K are.  A tile whose slabs span several CTAs is finished by the last
// of them to arrive: each adds its share to an f32 scratch with atomic adds
// (so the split sum's order, and its last bits, may vary between runs), bumps
// the tile's counter, and the one that completes it applies the epilogue to
// the sums and zeroes the scratch and the counter again.
//
// Epilogues: y = acc (f32); y += acc (f32 residual stream); and SwiGLU, where
// a second weight matrix (the up projection) runs as a second MMA on the same
// x slab and y = bf16(silu(acc_gate) * acc_up).
//
// Before the previous kernel in the stream has finished (programmatic
// dependent launch), a CTA already streams the W slabs of its first stages:
// weights are never written by the path.  x, y and the workspace are touched
// only after griddepcontrol.wait.
//
// Warp roles (192 threads): warps 0-3 epilogue (one TMEM lane quarter each),
// warp 4 TMA producer, warp 5 MMA issuer and TMEM owner.  Every wait is
// bounded; on a timeout the kernel raises SEED_DEVERR_TIMEOUT, still drains
// its copies and MMAs, and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace seedk {
namespace {

constexpr int kLRows = 128;                    // rows of W per tile (MMA M)
constexpr int kLK = 64;                        // K per slab
constexpr int kLMaxStages = 12;
constexpr int kLThreads = 192;
constexpr int kLWarpProd = 4, kLWarpMma = 5;
constexpr uint32_t kLSlabW = kLRows * 128u;    // one W slab: 128 rows x 128 B
constexpr uint32_t kLCtrlBytes = 256;
constexpr uint32_t kLSmemMax = 232448;
constexpr unsigned kFullL = 0xffffffffu;

struct LCtrl {
  uint64_t full[kLMaxStages], empty[kLMaxStages];
  uint64_t d_full[2], d_empty[2];
  uint64_t mma_done;
  uint32_t tmem_base;
  volatile int32_t abort_flag;
  volatile int32_t last;
};
static_assert(sizeof(LCtrl) <= kLCtrlBytes, "control block");

__host__ __device__ constexpr int lin_nb(int B) { return (B + 15) & ~15; }
__host__ __device__ constexpr uint32_t lin_stage_bytes(int nb, int nw) {
  return (uint32_t)nw * kLSlabW + (uint32_t)nb * 128u;
}
__host__ __device__ constexpr int lin_stages(int nb, int nw) {
  const uint32_t n = (kLSmemMax - 1024u - kLCtrlBytes) / lin_stage_bytes(nb, nw);
  return n < (uint32_t)kLMaxStages ? (int)n : kLMaxStages;
}
__host__ __device__ constexpr size_t lin_smem_bytes(int nb, int nw) {
  return (size_t)lin_stages(nb, nw) * lin_stage_bytes(nb, nw) + kLCtrlBytes + 1024u;
}
// TMEM columns of one accumulator buffer: a power of two >= 32 holding every
// column the epilogue reads (x32 loads of nch chunks, after nb gate columns
// for SwiGLU)
__host__ __device__ constexpr uint32_t lin_bufcols(int nb, int nw, int nch) {
  uint32_t p = 32;
  while (p < (uint32_t)((nw - 1) * nb + 32 * nch)) p <<= 1;
  return p;
}
static_assert(lin_stages(128, 2) >= 3 && lin_smem_bytes(128, 2) <= kLSmemMax, "stage budget");
static_assert(lin_smem_bytes(16, 1) <= kLSmemMax, "stage budget");
static_assert(2 * lin_bufcols(128, 2, 4) <= 512, "TMEM budget");

// CTA c's units are [lin_start(c), lin_start(c + 1)); unit u lies in CTA
// lin_cta_of(u) (the largest c whose start is <= u).
__host__ __device__ inline long long lin_start(long long U, int c, int n) {
  return U * c / n;
}
__device__ inline int lin_cta_of(long long U, long long u, int n) {
  return (int)(((u + 1) * n - 1) / U);
}

__device__ __noinline__ bool lwait(uint64_t* bar, uint32_t parity, LCtrl* c, int32_t* err) {
  for (uint32_t i = 0; i < kSuspendTries; ++i) {
    if (mbar_try_wait_sleep(bar, parity, kSuspendNs)) return true;
    if (c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ bool lwarp_wait(uint64_t* bar, uint32_t parity, LCtrl* c,
                                           int32_t* err) {
  return __all_sync(kFullL, lwait(bar, parity, c, err));
}

// Inline polling wait of the producer and MMA threads (bounded: ~2^26 polls).
__device__ __forceinline__ bool lpoll(uint64_t* bar, uint32_t parity, LCtrl* c, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 26); ++i) {
    if (mbar_test(bar, parity)) return true;
    if ((i & 1023u) == 1023u && c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ void ldrain(uint64_t* bar, uint32_t parity, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 26); ++i)
    if (mbar_test(bar, parity)) return;
  raise_err(err, SEED_DEVERR_TIMEOUT);
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// The epilogue of 32 output elements (b0 + i, n), i < 32, b0 + i < B, from
// the finished sums g (and u for SwiGLU).  For the residual epilogue all 32
// old values are loaded before any store, so that their latencies overlap.
template <int NW>
__device__ __forceinline__ void finish32(const LinearParams& p, int b0, int n, const float (&g)[32],
                                         const float (&u)[32]) {
  if (NW == 2) {
    __nv_bfloat16* y = static_cast<__nv_bfloat16*>(p.y);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      if (b0 + i < p.B) {
        const float s = g[i] / (1.f + __expf(-g[i]));
        y[(size_t)(b0 + i) * p.N + n] = __float2bfloat16_rn(s * u[i]);
      }
    }
  } else {
    float* y = static_cast<float*>(p.y);
    float old[32];
#pragma unroll
    for (int i = 0; i < 32; ++i)
      old[i] = (p.epi == kEpiResidF32 && b0 + i < p.B) ? y[(size_t)(b0 + i) * p.N + n] : 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (b0 + i < p.B) y[(size_t)(b0 + i) * p.N + n] = old[i] + g[i];
  }
}

// NW: weight matrices (1, or 2 for SwiGLU); NCH: 32-column chunks per matrix.
template <int NW, int NCH>
__global__ void __launch_bounds__(kLThreads, 1) linear_tc_kernel(
    const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
    const __grid_constant__ CUtensorMap tm_w2, const LinearParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int nb = lin_nb(p.B);
  const int S = lin_stages(nb, NW);
  const uint32_t stage_bytes = lin_stage_bytes(nb, NW);
  const uint32_t bufcols = lin_bufcols(nb, NW, NCH);
  LCtrl* ctrl = reinterpret_cast<LCtrl*>(smem + (size_t)S * stage_bytes);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  if (tid == 0) pdl_trigger();
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&ctrl->full[s], 1);
      mbar_init(&ctrl->empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->d_full[i], 1);
      mbar_init(&ctrl->d_empty[i], 4);
    }
    mbar_init(&ctrl->mma_done, 1);
    ctrl->abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kLWarpMma) {
    tmem_alloc(&ctrl->tmem_base, 2 * bufcols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctrl->tmem_base;

  const int nslab = p.K / kLK;
  const int ntiles = (p.N + kLRows - 1) / kLRows;
  const long long U = (long long)ntiles * nslab;
  const int nct = gridDim.x;
  const long long u0 = lin_start(U, blockIdx.x, nct), u1 = lin_start(U, blockIdx.x + 1, nct);
  const int total = (int)(u1 - u0);
  const int t_first = (int)(u0 / nslab), k_first = (int)(u0 % nslab);
  const int t_last = (int)((u1 - 1) / nslab);

  if (warp == kLWarpProd) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_x);
      tma_prefetch_desc(&tm_w);
      if (NW == 2) tma_prefetch_desc(&tm_w2);
      // the first stages' weights, while the previous kernel may still run
      const int pre = total < S ? total : S;
      {
        int t = t_first, k = k_first;
        for (int i = 0; i < pre; ++i) {
          uint8_t* st = smem + (size_t)i * stage_bytes;
          mbar_arrive_expect_tx(&ctrl->full[i], stage_bytes);
          tma_load_2d(st, &tm_w, k * kLK, t * kLRows, &ctrl->full[i]);
          if (NW == 2) tma_load_2d(st + kLSlabW, &tm_w2, k * kLK, t * kLRows, &ctrl->full[i]);
          if (++k == nslab) {
            k = 0;
            ++t;
          }
        }
      }
      pdl_wait();
      int it = 0, s = 0, t = t_first, k = k_first;
      uint32_t ph = 0;
      for (; it < total; ++it) {
        uint8_t* st = smem + (size_t)s * stage_bytes;
        if (it >= S) {
          if (!lpoll(&ctrl->empty[s], ph ^ 1u, ctrl, p.err)) break;
          mbar_arrive_expect_tx(&ctrl->full[s], stage_bytes);
          tma_load_2d(st, &tm_w, k * kLK, t * kLRows, &ctrl->full[s]);
          if (NW == 2) tma_load_2d(st + kLSlabW, &tm_w2, k * kLK, t * kLRows, &ctrl->full[s]);
        }
        tma_load_2d(st + NW * kLSlabW, &tm_x, k * kLK, 0, &ctrl->full[s]);
        if (++k == nslab) {
          k = 0;
          ++t;
        }
        if (++s == S) {
          s = 0;
          ph ^= 1u;
        }
      }
      // every stage's last fill has landed before the CTA moves on (the loop
      // cannot stop before it = S, so the first round's x is always issued)
      for (int j = 0; j < S && j < it; ++j) {
        const int lastj = j + S * ((it - 1 - j) / S);
        ldrain(&ctrl->full[j], (lastj / S) & 1, p.err);
      }
    }
    __syncwarp();
  } else if (warp == kLWarpMma) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kLRows, nb, 0, 0);
      int s = 0;
      uint32_t ph = 0;
      int t = t_first, k = k_first;
      for (int n = 0; t <= t_last; ++t, k = 0, ++n) {
        const int kend = t == t_last ? (int)((u1 - 1) % nslab) + 1 : nslab;
        const uint32_t d = tmem + (uint32_t)(n & 1) * bufcols;
        if (n >= 2 && !lpoll(&ctrl->d_empty[n & 1], ((n >> 1) - 1) & 1, ctrl, p.err)) break;
        tc_fence_after();
        bool ok = true;
        for (int kk = k; kk < kend; ++kk) {
          if (!lpoll(&ctrl->full[s], ph, ctrl, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = sbase + (uint32_t)s * stage_bytes;   // W slab(s)
          const uint32_t b0 = a0 + NW * kLSlabW;                   // x slab
#pragma unroll
          for (int j = 0; j < kLK / 16; ++j) {
            const uint64_t bx = smem_desc_sw128(b0 + j * 32, 16, 1024);
            const uint32_t acc = (kk > k || j > 0) ? 1u : 0u;
            mma_ss(d, smem_desc_sw128(a0 + j * 32, 16, 1024), bx, idesc, acc);
            if (NW == 2)
              mma_ss(d + (uint32_t)nb, smem_desc_sw128(a0 + kLSlabW + j * 32, 16, 1024), bx,
                     idesc, acc);
          }
          mma_commit(&ctrl->empty[s]);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(&ctrl->d_full[n & 1]);
      }
      mma_commit(&ctrl->mma_done);
      ldrain(&ctrl->mma_done, 0, p.err);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------- epilogue
    pdl_wait();
    const int q = warp;
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const int row = q * 32 + lane;
    const size_t accn = (size_t)p.B * p.N;   // one matrix's accumulator in the scratch
    bool ok = true;
    int t = t_first, k = k_first;
    for (int n = 0; t <= t_last; ++t, k = 0, ++n) {
      const int kend = t == t_last ? (int)((u1 - 1) % nslab) + 1 : nslab;
      const bool whole = k == 0 && kend == nslab;
      if (ok) ok = lwarp_wait(&ctrl->d_full[n & 1], (n >> 1) & 1, ctrl, p.err);
      tc_fence_after();
      const uint32_t col0 = tmem + lane_off + (uint32_t)(n & 1) * bufcols;
      const int nrow = t * kLRows + row;
      const bool vrow = nrow < p.N;
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        uint32_t rg[32], ru[32];
        if (ok) {
          tmem_ld32(col0 + c * 32, rg);
          if (NW == 2) tmem_ld32(col0 + (uint32_t)nb + c * 32, ru);
          tmem_wait_ld();
          if (c == NCH - 1) {                 // the accumulator is free for piece n + 2
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctrl->d_empty[n & 1]);
          }
          if (vrow) {
            if (whole) {
              float g[32], u[32];
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                g[i] = __uint_as_float(rg[i]);
                u[i] = NW == 2 ? __uint_as_float(ru[i]) : 0.f;
              }
              finish32<NW>(p, c * 32, nrow, g, u);
            } else {
              // a share of a tile split over CTAs: add it to the scratch
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const int b = c * 32 + i;
                if (b < p.B) {
                  atomicAdd(p.acc + (size_t)b * p.N + nrow, __uint_as_float(rg[i]));
                  if (NW == 2) atomicAdd(p.acc + accn + (size_t)b * p.N + nrow, __uint_as_float(ru[i]));
                }
              }
            }
          }
        }
      }
      if (whole) continue;
      // the last CTA of the tile to arrive applies the epilogue to the sums
      // and leaves the scratch zeroed
      __threadfence();
      epi_bar();
      if (tid == 0) {
        const int cf = lin_cta_of(U, (long long)t * nslab, nct);
        const int cl = lin_cta_of(U, (long long)(t + 1) * nslab - 1, nct);
        const int old = atomicAdd(p.cnt + t, 1);
        ctrl->last = old == cl - cf;
      }
      epi_bar();
      if (ctrl->last) {
        __threadfence();
        if (vrow) {
          for (int b0 = 0; b0 < p.B; b0 += 32) {
            float g[32], u[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const size_t at = (size_t)(b0 + i) * p.N + nrow;
              g[i] = b0 + i < p.B ? __ldcg(p.acc + at) : 0.f;
              u[i] = NW == 2 && b0 + i < p.B ? __ldcg(p.acc + accn + at) : 0.f;
            }
            finish32<NW>(p, b0, nrow, g, u);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              if (b0 + i < p.B) {
                const size_t at = (size_t)(b0 + i) * p.N + nrow;
                p.acc[at] = 0.f;
                if (NW == 2) p.acc[accn + at] = 0.f;
              }
            }
          }
        }
        if (tid == 0) p.cnt[t] = 0;           // the workspace stays zeroed
      }
      epi_bar();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kLWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * bufcols);
  }
}

// ------------------------------------------------------------- host side
using EncodeTiledFnL = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                    const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                    const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                    CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFnL encode_fn_l() {
  static EncodeTiledFnL fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFnL>(ptr);
  });
  return fn;
}

// 2-d bf16 map [rows, k], 64-element x `box_rows` boxes, 128-byte swizzle.
bool encode_rows(CUtensorMap* map, const void* base, uint64_t k, uint64_t rows,
                 uint32_t box_rows) {
  EncodeTiledFnL fn = encode_fn_l();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {k, rows};
  const cuuint64_t strides[1] = {k * 2ull};
  const cuuint32_t box[2] = {(cuuint32_t)kLK, box_rows};
  const cuuint32_t elem[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

std::atomic<uint64_t> g_lin_attr[6];

template <int NW, int NCH>
cudaError_t launch_nw(const LinearParams& prm, const CUtensorMap& tx, const CUtensorMap& tw,
                      const CUtensorMap& tw2, int nctas, int slot, cudaStream_t st) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(g_lin_attr[slot].load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(linear_tc_kernel<NW, NCH>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kLSmemMax);
    if (e != cudaSuccess) return e;
    g_lin_attr[slot].fetch_or(bit, std::memory_order_acq_rel);
  }
  const size_t smem = lin_smem_bytes(lin_nb(prm.B), NW);
  return launch_pdl(linear_tc_kernel<NW, NCH>, dim3(nctas), dim3(kLThreads), smem, st, tx, tw, tw2,
                    prm);
}

}  // namespace

int linear_ctas(int32_t n_out, int32_t k_in) {
  const long long units = (long long)((n_out + kLRows - 1) / kLRows) * (k_in / kLK);
  return (int)std::max(1LL, std::min((long long)std::min(device_sm_count(), kLinearMaxCtas), units));
}

// Workspace: a fixed prefix of kLinearMaxTiles counters (so that calls of any
// size can share one workspace), then the f32 scratch [nw][batch][n_out].
// Both are zero between calls.
size_t linear_workspace_bytes(int32_t batch, int32_t n_out, int32_t k_in, int32_t epi) {
  const int nw = epi == kEpiSwigluBf16 ? 2 : 1;
  (void)k_in;
  return kLinearCntBytes + (size_t)nw * batch * n_out * sizeof(float);
}

cudaError_t launch_linear(LinearParams prm, const void* x, const void* w, const void* w2, void* ws,
                          cudaStream_t st) {
  const int nw = prm.epi == kEpiSwigluBf16 ? 2 : 1;
  const int nb = lin_nb(prm.B);
  prm.cnt = static_cast<int32_t*>(ws);
  prm.acc = reinterpret_cast<float*>(static_cast<char*>(ws) + kLinearCntBytes);
  CUtensorMap tx, tw, tw2;
  if (!encode_rows(&tx, x, (uint64_t)prm.K, (uint64_t)prm.B, (uint32_t)nb))
    return cudaErrorInvalidValue;
  if (!encode_rows(&tw, w, (uint64_t)prm.K, (uint64_t)prm.N, kLRows)) return cudaErrorInvalidValue;
  if (!encode_rows(&tw2, nw == 2 ? w2 : w, (uint64_t)prm.K, (uint64_t)prm.N, kLRows))
    return cudaErrorInvalidValue;
  const int nctas = linear_ctas(prm.N, prm.K);
  const int nch = (nb + 31) / 32;
  if (nw == 1) {
    if (nch == 1) return launch_nw<1, 1>(prm, tx, tw, tw2, nctas, 0, st);
    if (nch == 2) return launch_nw<1, 2>(prm, tx, tw, tw2, nctas, 1, st);
    return launch_nw<1, 4>(prm, tx, tw, tw2, nctas, 2, st);
  }
  if (nch == 1) return launch_nw<2, 1>(prm, tx, tw, tw2, nctas, 3, st);
  if (nch == 2) return launch_nw<2, 2>(prm, tx, tw, tw2, nctas, 4, st);
  return launch_nw<2, 4>(prm, tx, tw, tw2, nctas, 5, st);
}

}  // namespace seedk
