// The drafter's LM head with a fused softmax and top-k, for confidence-aware
// dynamic drafting (Sec. D.1): per sequence, logits z = W_out h over the whole
// vocabulary are never stored; the kernel keeps the log-sum-exp and the ten
// most probable tokens, from which the top-1 probability p0 gives the number
// of sibling candidates k (1, 3, 5 or 10) and the stop decision p0 <= tau.
//
// Design.  The contraction [B, d] x [d, V] is memory-bound on the 2 V d bytes
// of W for B <= 128, so it runs on the tensor cores with W as the 128-row M
// operand (a vocabulary tile of 128 rows) and the B sequences, padded to a
// multiple of 16, as the N operand; K runs over d in slabs of 64.  A TMA ring
// of as many stages as shared memory holds (W slab 16 KiB + h slab) feeds one
// MMA thread; two TMEM accumulators of 128 columns let one tile's MMAs run
// while the previous tile's logits are consumed.  Small MMAs (N = B) keep
// each stage busy only briefly after its bytes land, which is what lets the
// ring stream W near the copy rate.
//
// Epilogue.  TMEM lane = vocabulary row, column = sequence, so each of the
// four epilogue warps holds 32 rows.  Per chunk of 32 sequences the warps
// transpose their rows into shared memory; thread (q, j) then scans the 32
// logits of sequence j in row quarter q with an online max / sum 2^(.) and a
// register top-10 (ids rise during the scan, so equal logits keep the lower
// id).  At the end the four quarters of each sequence merge in shared memory
// into one partial record per (CTA, sequence); a small kernel merges CTAs.
//
// Warp roles (192 threads): warps 0-3 epilogue, warp 4 TMA producer, warp 5
// MMA issuer and TMEM owner.  Every wait is bounded; a wait that gives up
// raises SEED_DEVERR_TIMEOUT, the producer still waits (bounded) for its
// copies in flight and the MMA thread for its MMAs before TMEM is freed.
// The epilogue warps run the same sequence of named barriers whatever their
// waits return, so an abort cannot leave one of them behind at a barrier.
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

constexpr int kHRows = 128;                    // vocabulary rows per tile (MMA M)
constexpr int kHK = 64;                        // head dims per K slab
constexpr int kHMaxStages = 12;
constexpr int kHTopK = 10;
constexpr int kHThreads = 192;
constexpr int kHWarpProd = 4, kHWarpMma = 5;
constexpr uint32_t kHSlabW = kHRows * 128u;    // W slab: 128 rows x 128 B
constexpr int kHTStride = 129;                 // transpose row stride in floats (bank-conflict free)
constexpr uint32_t kHTBytes = 32u * kHTStride * 4u;
constexpr uint32_t kHCtrlBytes = 256;
constexpr uint32_t kHColsBuf = 128;            // TMEM columns per accumulator
constexpr uint32_t kHSmemMax = 232448;
constexpr unsigned kFullH = 0xffffffffu;
constexpr float kLog2e = 1.4426950408889634f;

struct HCtrl {
  uint64_t full[kHMaxStages], empty[kHMaxStages];
  uint64_t d_full[2], d_empty[2];
  uint64_t mma_done;
  uint32_t tmem_base;
  volatile int32_t abort_flag;
};
static_assert(sizeof(HCtrl) <= kHCtrlBytes, "control block");

// Sequences padded to the MMA's N granularity.
__host__ __device__ constexpr int head_nb(int B) { return (B + 15) & ~15; }
__host__ __device__ constexpr uint32_t head_stage_bytes(int nb) {
  return kHSlabW + (uint32_t)nb * 128u;
}
__host__ __device__ constexpr int head_stages(int nb) {
  const uint32_t n = (kHSmemMax - 1024u - kHTBytes - kHCtrlBytes) / head_stage_bytes(nb);
  return n < (uint32_t)kHMaxStages ? (int)n : kHMaxStages;
}
__host__ __device__ constexpr size_t head_smem_bytes(int nb) {
  return (size_t)head_stages(nb) * head_stage_bytes(nb) + kHTBytes + kHCtrlBytes + 1024u;
}
static_assert(head_stages(128) >= 4 && head_smem_bytes(128) <= kHSmemMax, "stage budget");
static_assert(head_smem_bytes(16) <= kHSmemMax, "stage budget");

// Suspending wait (epilogue warps, off the streaming path).
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

// Polling wait of the producer and MMA threads: these waits sit on the
// streaming path, where the wake-up latency of a suspended wait costs
// bandwidth.  About 2^26 polls (seconds) before giving up.
__device__ __forceinline__ bool hpoll(uint64_t* bar, uint32_t parity, HCtrl* c, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 26); ++i) {
    if (mbar_test(bar, parity)) return true;
    if ((i & 1023u) == 1023u && c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

// Wait for an async operation this CTA started, abort or not (bounded).
__device__ __forceinline__ void hdrain(uint64_t* bar, uint32_t parity, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 26); ++i)
    if (mbar_test(bar, parity)) return;
  raise_err(err, SEED_DEVERR_TIMEOUT);
}

// Named barrier of the four epilogue warps.
__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Insert (z, id) into a descending top-10 while ids arrive in increasing
// order: equal values keep the earlier (lower) id.
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

// Insert with ids in any order: larger logit first, equal logits by lower id.
__device__ __forceinline__ void top_insert_any(float (&tv)[kHTopK], int (&ti)[kHTopK], float z,
                                               int id) {
  if (id < 0) return;
  if (!(z > tv[kHTopK - 1] || (z == tv[kHTopK - 1] && (ti[kHTopK - 1] < 0 || id < ti[kHTopK - 1]))))
    return;
  tv[kHTopK - 1] = z;
  ti[kHTopK - 1] = id;
#pragma unroll
  for (int k = kHTopK - 1; k > 0; --k) {
    if (tv[k] > tv[k - 1] || (tv[k] == tv[k - 1] && (ti[k - 1] < 0 || ti[k] < ti[k - 1]))) {
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

// NCH = chunks of 32 sequences (1, 2 or 4).
template <int NCH>
__global__ void __launch_bounds__(kHThreads, 1) head_tc_kernel(
    const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_w,
    const HeadParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const int nb = head_nb(p.B);
  const int S = head_stages(nb);
  const uint32_t stage_bytes = head_stage_bytes(nb);
  float* T = reinterpret_cast<float*>(smem + (size_t)S * stage_bytes);
  HCtrl* ctrl = reinterpret_cast<HCtrl*>(smem + (size_t)S * stage_bytes + kHTBytes);
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
  if (warp == kHWarpMma) {
    tmem_alloc(&ctrl->tmem_base, 2 * kHColsBuf);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctrl->tmem_base;
  pdl_wait();

  // this CTA's vocabulary tiles [t0, t1)
  const int ntiles = (p.V + kHRows - 1) / kHRows;
  const int t0 = (int)((long long)ntiles * blockIdx.x / gridDim.x);
  const int t1 = (int)((long long)ntiles * (blockIdx.x + 1) / gridDim.x);
  const int nslab = p.d / kHK;

  if (warp == kHWarpProd) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_h);
      tma_prefetch_desc(&tm_w);
      int it = 0, s = 0;
      uint32_t ph = 0;                        // phase of stage s's current fill
      bool ok = true;
      for (int t = t0; t < t1 && ok; ++t) {
        for (int k = 0; k < nslab; ++k, ++it) {
          if (it >= S && !hpoll(&ctrl->empty[s], ph ^ 1u, ctrl, p.err)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + (size_t)s * stage_bytes;
          mbar_arrive_expect_tx(&ctrl->full[s], stage_bytes);
          tma_load_2d(st, &tm_w, k * kHK, t * kHRows, &ctrl->full[s]);
          tma_load_2d(st + kHSlabW, &tm_h, k * kHK, 0, &ctrl->full[s]);
          if (++s == S) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      // the last copy issued into each stage has landed before the CTA moves on
      for (int j = 0; j < S && j < it; ++j) {
        const int last = j + S * ((it - 1 - j) / S);
        hdrain(&ctrl->full[j], (last / S) & 1, p.err);
      }
    }
    __syncwarp();
  } else if (warp == kHWarpMma) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kHRows, nb, 0, 0);
      int s = 0;
      uint32_t ph = 0;
      for (int t = t0, n = 0; t < t1; ++t, ++n) {
        const uint32_t d = tmem + (uint32_t)(n & 1) * kHColsBuf;
        if (n >= 2 && !hpoll(&ctrl->d_empty[n & 1], ((n >> 1) - 1) & 1, ctrl, p.err)) break;
        tc_fence_after();
        bool ok = true;
        for (int k = 0; k < nslab; ++k) {
          if (!hpoll(&ctrl->full[s], ph, ctrl, p.err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = sbase + (uint32_t)s * stage_bytes;   // W slab
          const uint32_t b0 = a0 + kHSlabW;                        // h slab
#pragma unroll
          for (int kk = 0; kk < kHK / 16; ++kk) {
            const uint64_t a = smem_desc_sw128(a0 + kk * 32, 16, 1024);
            const uint64_t b = smem_desc_sw128(b0 + kk * 32, 16, 1024);
            mma_ss(d, a, b, idesc, (k > 0 || kk > 0) ? 1u : 0u);
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
      // every MMA issued has completed before TMEM is released
      mma_commit(&ctrl->mma_done);
      hdrain(&ctrl->mma_done, 0, p.err);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------- epilogue
    const int q = warp;                       // row quarter = TMEM lane quarter
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    // per-thread sequence states (chunk c: sequence 32 c + lane)
    float m2[NCH], l[NCH], tv[NCH][kHTopK];
    int ti[NCH][kHTopK];
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      m2[c] = -INFINITY;
      l[c] = 0.f;
#pragma unroll
      for (int k = 0; k < kHTopK; ++k) {
        tv[c][k] = -INFINITY;
        ti[c][k] = -1;
      }
    }
    bool ok = true;
    for (int t = t0, n = 0; t < t1; ++t, ++n) {
      if (ok) ok = hwarp_wait(&ctrl->d_full[n & 1], (n >> 1) & 1, ctrl, p.err);
      tc_fence_after();
      const uint32_t col0 = tmem + lane_off + (uint32_t)(n & 1) * kHColsBuf;
      const int id0 = t * kHRows + q * 32;    // vocabulary id of this quarter's first row
      const int nv = min(32, p.V - id0);
#pragma unroll
      for (int c = 0; c < NCH; ++c) {
        uint32_t r[32];
        if (ok) {
          tmem_ld32(col0 + c * 32, r);
          tmem_wait_ld();
          if (c == NCH - 1) {                 // the accumulator is free for tile n + 2
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctrl->d_empty[n & 1]);
          }
        }
        epi_bar();                            // readers of the previous chunk are done
        if (ok) {
#pragma unroll
          for (int x = 0; x < 32; ++x) T[x * kHTStride + q * 32 + lane] = __uint_as_float(r[x]);
        }
        epi_bar();
        const int b = c * 32 + lane;
        if (ok && b < p.B && nv > 0) {
          const float* col = T + lane * kHTStride + q * 32;
          float v[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = col[i];
          float mx = -INFINITY;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (i < nv) mx = fmaxf(mx, v[i]);
          const float mt = mx * kLog2e;
          if (mt > m2[c]) {
            l[c] *= (m2[c] == -INFINITY) ? 0.f : ex2_approx(m2[c] - mt);
            m2[c] = mt;
          }
          // sum, and a mask of the logits above the current tenth best
          float ls = 0.f;
          uint32_t cand = 0;
          const float thr = tv[c][kHTopK - 1];
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            if (i < nv) {
              ls += ex2_approx(fmaf(v[i], kLog2e, -m2[c]));
              cand |= (v[i] > thr ? 1u : 0u) << i;
            }
          }
          l[c] += ls;
          // the few candidates, in increasing id order (one copy of the insert)
#pragma unroll 1
          while (cand != 0u) {
            const int i = __ffs(cand) - 1;
            cand &= cand - 1u;
            top_insert(tv[c], ti[c], col[i], id0 + i);
          }
        }
      }
    }
    // one partial record per (CTA, row quarter, sequence)
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int b = c * 32 + lane;
      if (b < p.B) {
        float4* rec = reinterpret_cast<float4*>(p.part + ((size_t)(blockIdx.x * 4 + q) * p.B + b) * kHRec);
        const float* z = tv[c];
        const int* id = ti[c];
        rec[0] = make_float4(m2[c], l[c], z[0], z[1]);
        rec[1] = make_float4(z[2], z[3], z[4], z[5]);
        rec[2] = make_float4(z[6], z[7], z[8], z[9]);
        rec[3] = make_float4(__int_as_float(id[0]), __int_as_float(id[1]), __int_as_float(id[2]),
                             __int_as_float(id[3]));
        rec[4] = make_float4(__int_as_float(id[4]), __int_as_float(id[5]), __int_as_float(id[6]),
                             __int_as_float(id[7]));
        rec[5] = make_float4(__int_as_float(id[8]), __int_as_float(id[9]), 0.f, 0.f);
      }
    }
  }

  tc_fence_before();
  __syncthreads();                            // ring drained, MMAs complete
  if (warp == kHWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * kHColsBuf);
  }
}

// Order-preserving 32-bit key of a (non-NaN) float.
__device__ __forceinline__ uint32_t fkey(float z) {
  const uint32_t u = __float_as_uint(z);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Pop the best head (largest logit, then lowest id) of the warp's sorted
// lists ten times; lane 0 writes the merged list to (zo, io).
__device__ __forceinline__ void warp_top10(float (&tv)[kHTopK], int (&ti)[kHTopK], int lane,
                                           float* zo, int* io) {
#pragma unroll 1
  for (int k = 0; k < kHTopK; ++k) {
    const uint32_t key = ti[0] >= 0 ? fkey(tv[0]) : 0u;
    const uint32_t kmax = __reduce_max_sync(kFullH, key);
    const int cand = (key == kmax && ti[0] >= 0) ? ti[0] : 0x7fffffff;
    const int imin = __reduce_min_sync(kFullH, cand);
    const bool win = cand == imin && imin != 0x7fffffff;
    const unsigned wl = __ballot_sync(kFullH, win);
    const float z = __shfl_sync(kFullH, tv[0], wl ? __ffs(wl) - 1 : 0);
    if (lane == 0) {
      zo[k] = wl ? z : -INFINITY;
      io[k] = wl ? imin : -1;
    }
    if (win) {
#pragma unroll
      for (int j = 0; j < kHTopK - 1; ++j) {
        tv[j] = tv[j + 1];
        ti[j] = ti[j + 1];
      }
      tv[kHTopK - 1] = -INFINITY;
      ti[kHTopK - 1] = -1;
    }
  }
}

// Online combine of (max, sum) pairs in log2 units.
__device__ __forceinline__ void lse_combine(float& M, float& L, float M2, float L2) {
  const float Mn = fmaxf(M, M2);
  L = (M == -INFINITY ? 0.f : L * ex2_approx(M - Mn)) +
      (M2 == -INFINITY ? 0.f : L2 * ex2_approx(M2 - Mn));
  M = Mn;
}

// One block per sequence: merge the (CTA, row quarter) partial records into
// the log-sum-exp and the global top-10, then apply the sibling-count rule
// and the stop rule.
constexpr int kMergeThreads = 512;
constexpr int kMergeRecs = 4 * kHeadMaxCtas / kMergeThreads;   // records per thread, at most
__global__ void __launch_bounds__(kMergeThreads) head_merge_kernel(const HeadParams p, int nrec) {
  __shared__ float s_m[kMergeThreads / 32], s_l[kMergeThreads / 32];
  __shared__ float s_z[kMergeThreads / 32][kHTopK];
  __shared__ int s_i[kMergeThreads / 32][kHTopK];
  __shared__ float s_zf[kHTopK];
  __shared__ int s_if[kHTopK];
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float M = -INFINITY, L = 0.f, tv[kHTopK];
  int ti[kHTopK];
#pragma unroll
  for (int k = 0; k < kHTopK; ++k) {
    tv[k] = -INFINITY;
    ti[k] = -1;
  }
  // this thread's records (at most kMergeRecs), all loads issued before any use
  float4 rv[kMergeRecs][kHRec / 4];
#pragma unroll
  for (int j = 0; j < kMergeRecs; ++j) {
    const int r = tid + j * kMergeThreads;
    if (r < nrec) {
      const float4* rec = reinterpret_cast<const float4*>(p.part + ((size_t)r * p.B + b) * kHRec);
#pragma unroll
      for (int v = 0; v < kHRec / 4; ++v) rv[j][v] = rec[v];
    }
  }
#pragma unroll
  for (int j = 0; j < kMergeRecs; ++j) {
    if (tid + j * kMergeThreads >= nrec) break;
    const float f[kHRec] = {rv[j][0].x, rv[j][0].y, rv[j][0].z, rv[j][0].w, rv[j][1].x, rv[j][1].y,
                            rv[j][1].z, rv[j][1].w, rv[j][2].x, rv[j][2].y, rv[j][2].z, rv[j][2].w,
                            rv[j][3].x, rv[j][3].y, rv[j][3].z, rv[j][3].w, rv[j][4].x, rv[j][4].y,
                            rv[j][4].z, rv[j][4].w, rv[j][5].x, rv[j][5].y, rv[j][5].z, rv[j][5].w};
    lse_combine(M, L, f[0], f[1]);
    if (j == 0) {                             // the first list is taken as it is
#pragma unroll
      for (int k = 0; k < kHTopK; ++k) {
        tv[k] = f[2 + k];
        ti[k] = __float_as_int(f[2 + kHTopK + k]);
      }
      continue;
    }
    // each record's list is sorted: stop at the first entry that stays out
#pragma unroll
    for (int k = 0; k < kHTopK; ++k) {
      const int id = __float_as_int(f[2 + kHTopK + k]);
      const float z = f[2 + k];
      if (id < 0 || !(z > tv[kHTopK - 1] || (z == tv[kHTopK - 1] && (ti[kHTopK - 1] < 0 ||
                                                                      id < ti[kHTopK - 1]))))
        break;
      top_insert_any(tv, ti, z, id);
    }
  }
  for (int o = 16; o; o >>= 1) {
    const float M2 = __shfl_xor_sync(kFullH, M, o), L2 = __shfl_xor_sync(kFullH, L, o);
    lse_combine(M, L, M2, L2);
  }
  warp_top10(tv, ti, lane, s_z[warp], s_i[warp]);
  if (lane == 0) {
    s_m[warp] = M;
    s_l[warp] = L;
  }
  __syncthreads();
  if (warp != 0) return;
  constexpr int kW = kMergeThreads / 32;
  static_assert(kW <= 32, "one list per lane");
  M = lane < kW ? s_m[lane] : -INFINITY;
  L = lane < kW ? s_l[lane] : 0.f;
  for (int o = 16; o; o >>= 1) {
    const float M2 = __shfl_xor_sync(kFullH, M, o), L2 = __shfl_xor_sync(kFullH, L, o);
    lse_combine(M, L, M2, L2);
  }
  const float lse2 = M + log2f(L);
  // lane w holds warp w's sorted list
#pragma unroll
  for (int k = 0; k < kHTopK; ++k) {
    tv[k] = lane < kW ? s_z[lane][k] : -INFINITY;
    ti[k] = lane < kW ? s_i[lane][k] : -1;
  }
  warp_top10(tv, ti, lane, s_zf, s_if);
  __syncwarp();
  if (lane < kHTopK) {
    const int id = s_if[lane];
    p.ids[(size_t)b * kHTopK + lane] = id;
    p.probs[(size_t)b * kHTopK + lane] = id >= 0 ? exp2f(fmaf(s_zf[lane], kLog2e, -lse2)) : 0.f;
  }
  if (lane == 0) {
    const float p0 = s_if[0] >= 0 ? exp2f(fmaf(s_zf[0], kLog2e, -lse2)) : 0.f;
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

std::atomic<uint64_t> g_head_attr_set[3];

template <int NCH>
cudaError_t launch_head_nch(const HeadParams& prm, const CUtensorMap& th, const CUtensorMap& tw,
                            int nctas, int slot, cudaStream_t st) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(g_head_attr_set[slot].load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(head_tc_kernel<NCH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kHSmemMax);
    if (e != cudaSuccess) return e;
    g_head_attr_set[slot].fetch_or(bit, std::memory_order_acq_rel);
  }
  const size_t smem = head_smem_bytes(head_nb(prm.B));
  return launch_pdl(head_tc_kernel<NCH>, dim3(nctas), dim3(kHThreads), smem, st, th, tw, prm);
}

}  // namespace

int head_ctas(int32_t vocab) {
  const int ntiles = (vocab + kHRows - 1) / kHRows;
  return std::max(1, std::min(std::min(device_sm_count(), kHeadMaxCtas), ntiles));
}

cudaError_t launch_head(const HeadParams& prm, const void* h, const void* w, int nctas,
                        cudaStream_t st) {
  CUtensorMap th, tw;
  const int nb = head_nb(prm.B);
  if (!encode_2d(&th, h, (uint64_t)prm.d, (uint64_t)prm.B, (uint32_t)nb)) return cudaErrorInvalidValue;
  if (!encode_2d(&tw, w, (uint64_t)prm.d, (uint64_t)prm.V, kHRows)) return cudaErrorInvalidValue;
  cudaError_t e;
  if (prm.B <= 32)
    e = launch_head_nch<1>(prm, th, tw, nctas, 0, st);
  else if (prm.B <= 64)
    e = launch_head_nch<2>(prm, th, tw, nctas, 1, st);
  else
    e = launch_head_nch<4>(prm, th, tw, nctas, 2, st);
  if (e != cudaSuccess) return e;
  return launch_pdl(head_merge_kernel, dim3(prm.B), dim3(kMergeThreads), 0, st, prm, 4 * nctas);
}

size_t head_workspace_bytes(int32_t batch) {
  return (size_t)kHeadMaxCtas * 4 * batch * kHRec * sizeof(float);
}

}  // namespace seedk
