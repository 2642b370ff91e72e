// Block-causal training attention on the tensor cores (Sec. 4.2, "Training
// with Block Attention"; Fig. 2): the query at position p sees the deep rows
// KV^dec at positions < s(p) = (p / b) * b and its own block's raw-embedding
// rows at positions s(p) .. p.
//
// A prefill-style kernel for head_dim 128.  A work item is 128 query rows --
// 128 / G consecutive positions times the G query heads of one KV head, the
// row of (position i, head j) being i * G + j -- and the key tiles it needs,
// each read once: the deep rows below the item's last block start, then the
// raw-embedding rows from its first block start to its last position.  Per
// key tile, S = Q K^T (tcgen05, bf16 -> f32 in TMEM), an online softmax in
// the log2 domain with the block mask, and O += P V with P split into bf16
// hi + lo terms (within 2^-14 of P, relative).  Two S/P buffers let S(t + 1)
// run while tile t's softmax runs.
//
// Persistent: one CTA per SM walks the items (longest prefixes first,
// strided over the CTAs).  Every counter runs over the CTA's whole sequence
// of key tiles, and O is double-buffered by item, so the next item's Q and
// key tiles load and its first S and PV run while the softmax warps write
// out the previous item: they do that epilogue after handing over the next
// item's first P.
//
// Warp roles (320 threads): warps 0-7 softmax and epilogue -- warp w takes
// TMEM lane quarter w % 4 and key / output columns [64 (w / 4), + 64), the
// two halves of a row trading their maxima through shared memory -- warp 8
// TMA producer, warp 9 MMA issuer and TMEM owner.  Every wait is bounded; a
// wait that gives up raises SEED_DEVERR_TIMEOUT, and the CTA still drains its
// copies and MMAs before it frees TMEM and exits.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace seedk {
namespace {

constexpr int kBD = 128;                       // head_dim
constexpr int kBN = 128;                       // keys per tile
constexpr int kBThreads = 320;
constexpr int kBSoftWarps = 8;
constexpr int kBWarpProd = 8, kBWarpMma = 9;
constexpr uint32_t kBHalf = 128 * 128;         // 128 rows x 128 B
constexpr uint32_t kBTile = 2 * kBHalf;        // one tile of Q, K or V: two head-dim halves
constexpr uint32_t kBOffK = kBTile;            // Q at 0, then the K ring, then the V ring
constexpr uint32_t kBOffV = kBOffK + 2 * kBTile;
constexpr uint32_t kBOffCtrl = kBOffV + 2 * kBTile;
constexpr uint32_t kBOffX = kBOffCtrl + 256;   // f32 [2 tiles][2 halves][128 rows] row maxima
constexpr uint32_t kBOffL = kBOffX + 2048;     // f32 [2 items][2 halves][128 rows] row sums
constexpr uint32_t kBOffE = kBOffL + 2048;     // epilogue staging: 4 KiB per softmax warp
constexpr uint32_t kBColO = 256;               // S/P buffers [0, 256), O buffers [256, 512)
constexpr uint32_t kBIdescS = idesc_bf16_f32(128, kBN, 0, 0);   // K-major A and B
constexpr uint32_t kBIdescPV = idesc_bf16_f32(128, kBD, 0, 1);  // B (V) MN-major
constexpr float kBRescale = 8.0f;
constexpr float kBLn2 = 0.69314718055994531f;
constexpr unsigned kBFull = 0xffffffffu;

struct BCtrl {
  uint64_t q_full, q_empty;
  uint64_t k_full[2], k_empty[2], v_full[2], v_empty[2];
  uint64_t s_full[2], p_full[2];
  uint64_t x_full[2], l_full[2];               // the softmax warps' exchanges
  uint64_t o_full, o_done[2], mma_done;
  uint32_t tmem_base;
  volatile int32_t abort_flag;
};
constexpr size_t kBSmem = kBOffE + kBSoftWarps * 4096 + 1024;
static_assert(sizeof(BCtrl) <= 256, "control block");

struct BlockTcParams {
  float* out;          // f32 [B, n, hq, D]
  float* lse;          // f32 [B, n, hq] or null
  int32_t* err;
  int32_t B, n, blk, hq, hkv, G, P, nqt, nitems;
  float c2;            // softmax scale * log2(e)
};

// The softmax and epilogue warps' waits: try_wait without a sleep hint (the
// thread resumes as soon as the phase completes; a sleeping wait wakes
// later), bounded (2^22 tries; the abort flag is read every 64).
__device__ __forceinline__ bool bwait_hot(uint64_t* bar, uint32_t parity, BCtrl* c, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 22); ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 63u && c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ bool bwarp_hot(uint64_t* bar, uint32_t parity, BCtrl* c,
                                          int32_t* err) {
  return __all_sync(kBFull, bwait_hot(bar, parity, c, err));
}

__device__ __forceinline__ bool bpoll(uint64_t* bar, uint32_t parity, BCtrl* c, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 26); ++i) {
    if (mbar_test(bar, parity)) return true;
    if ((i & 1023u) == 1023u && c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ void bdrain(uint64_t* bar, uint32_t parity, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 26); ++i)
    if (mbar_test(bar, parity)) return;
  raise_err(err, SEED_DEVERR_TIMEOUT);
}

// Pull a 4-d box of a tensor map into L2 (no shared memory, no completion).
__device__ __forceinline__ void tma_prefetch_l2_4d(const CUtensorMap* map, int x, int y, int z,
                                                   int w) {
  asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z), "r"(w)
               : "memory");
}

// Bits of the 32 keys k0 .. k0 + 31 that lie in [lo, hi].
__device__ __forceinline__ uint32_t key_bits(int k0, int lo, int hi) {
  const int a = max(lo - k0, 0), e = min(hi - k0, 31);
  if (e < a) return 0u;
  const uint32_t w = (uint32_t)(e - a + 1);
  return (w == 32u ? 0xffffffffu : ((1u << w) - 1u)) << a;
}

// Two probabilities as bf16 hi + lo pairs by truncation: hi keeps the top 16
// bits of each f32, lo the top 16 bits of the exact f32 remainder, so hi + lo
// is within 2^-14 of the value (relative) and never above it.  First
// argument in the low half of each word.
__device__ __forceinline__ void split_pair(float p0, float p1, uint32_t& hi, uint32_t& lo) {
  const uint32_t b0 = __float_as_uint(p0), b1 = __float_as_uint(p1);
  hi = __byte_perm(b0, b1, 0x7632);
  const float r0 = p0 - __uint_as_float(b0 & 0xffff0000u);
  const float r1 = p1 - __uint_as_float(b1 & 0xffff0000u);
  lo = __byte_perm(__float_as_uint(r0), __float_as_uint(r1), 0x7632);
}

// Warp-uniform class of a 32-key chunk: 2 when every lane sees all its keys,
// 0 when no lane sees any, 1 otherwise.
__device__ __forceinline__ int chunk_kind(uint32_t bits) {
  if (__all_sync(kBFull, bits == 0xffffffffu)) return 2;
  if (__all_sync(kBFull, bits == 0u)) return 0;
  return 1;
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Maximum of a chunk's visible scores (-inf if none).
__device__ __forceinline__ float chunk_max(const uint32_t (&r)[32], uint32_t bits, int kind) {
  if (kind == 2) {
    float a[11];
#pragma unroll
    for (int i = 0; i < 10; ++i)
      a[i] = fmax3(__uint_as_float(r[3 * i]), __uint_as_float(r[3 * i + 1]),
                   __uint_as_float(r[3 * i + 2]));
    a[10] = fmaxf(__uint_as_float(r[30]), __uint_as_float(r[31]));
    const float b0 = fmax3(a[0], a[1], a[2]), b1 = fmax3(a[3], a[4], a[5]);
    const float b2 = fmax3(a[6], a[7], a[8]), b3 = fmaxf(a[9], a[10]);
    return fmaxf(fmax3(b0, b1, b2), b3);
  }
  float m = -INFINITY;
  if (kind == 1) {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      m = fmaxf(m, ((bits >> i) & 1u) ? __uint_as_float(r[i]) : -INFINITY);
  }
  return m;
}

// P = 2^(s c2 - mc) of a chunk (0 where masked) as bf16 hi + lo pairs;
// returns the chunk's sum of P.
__device__ __forceinline__ float chunk_p(const uint32_t (&r)[32], uint32_t bits, int kind,
                                         float c2, float mc, uint32_t (&wh)[16],
                                         uint32_t (&wl)[16]) {
  float ls = 0.f;
  if (kind == 2) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float p0 = ex2_approx(fmaf(__uint_as_float(r[2 * i]), c2, -mc));
      const float p1 = ex2_approx(fmaf(__uint_as_float(r[2 * i + 1]), c2, -mc));
      ls += p0 + p1;
      split_pair(p0, p1, wh[i], wl[i]);
    }
  } else if (kind == 1) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float x0 = ((bits >> (2 * i)) & 1u) ? fmaf(__uint_as_float(r[2 * i]), c2, -mc) : -INFINITY;
      const float x1 =
          ((bits >> (2 * i + 1)) & 1u) ? fmaf(__uint_as_float(r[2 * i + 1]), c2, -mc) : -INFINITY;
      const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);   // 2^-inf = +0
      ls += p0 + p1;
      split_pair(p0, p1, wh[i], wl[i]);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 16; ++i) wh[i] = wl[i] = 0u;
  }
  return ls;
}

// A work item's query tile and its key tiles.
struct BTiles {
  int b, g, p0, plast, s_lo, nd, nt;
};

__device__ __forceinline__ BTiles tiles_of(const BlockTcParams& p, int item) {
  BTiles t;
  const int per = p.B * p.hkv;
  const int qt = p.nqt - 1 - item / per;       // longest prefixes first
  const int rest = item - (item / per) * per;
  t.b = rest / p.hkv;
  t.g = rest - t.b * p.hkv;
  t.p0 = qt * p.P;
  t.plast = min(t.p0 + p.P, p.n) - 1;
  t.s_lo = (t.p0 / p.blk) * p.blk;
  const int s_hi = (t.plast / p.blk) * p.blk;
  t.nd = (s_hi + kBN - 1) / kBN;                          // deep tiles: rows [0, s_hi)
  t.nt = t.nd + (t.plast + 1 - t.s_lo + kBN - 1) / kBN;   // then rows [s_lo, plast]
  return t;
}

// The MMA issuer's position in the CTA's sequence of items and key tiles.
struct BCursor {
  int item, wi, t, nt;
};

__device__ __forceinline__ void cursor_next(BCursor& c, const BlockTcParams& p) {
  if (++c.t < c.nt) return;
  c.t = 0;
  ++c.wi;
  c.item += (int)gridDim.x;
  c.nt = c.item < p.nitems ? tiles_of(p, c.item).nt : 0;
}

__global__ void __launch_bounds__(kBThreads, 1) block_tc_kernel(
    const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kd,
    const __grid_constant__ CUtensorMap tm_vd, const __grid_constant__ CUtensorMap tm_ks,
    const __grid_constant__ CUtensorMap tm_vs, const BlockTcParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  BCtrl* ctrl = reinterpret_cast<BCtrl*>(smem + kBOffCtrl);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  if (tid == 0) pdl_trigger();
  if (tid == 0) {
    mbar_init(&ctrl->q_full, 1);
    mbar_init(&ctrl->q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->k_full[i], 1);
      mbar_init(&ctrl->k_empty[i], 1);
      mbar_init(&ctrl->v_full[i], 1);
      mbar_init(&ctrl->v_empty[i], 1);
      mbar_init(&ctrl->s_full[i], 1);
      mbar_init(&ctrl->p_full[i], kBSoftWarps);
      mbar_init(&ctrl->x_full[i], kBSoftWarps);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->l_full[i], kBSoftWarps);
      mbar_init(&ctrl->o_done[i], 1);
    }
    mbar_init(&ctrl->o_full, 1);
    mbar_init(&ctrl->mma_done, 1);
    ctrl->abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == kBWarpMma) {
    tmem_alloc(&ctrl->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctrl->tmem_base;
  pdl_wait();

  if (warp == kBWarpProd) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_kd);
      tma_prefetch_desc(&tm_vd);
      tma_prefetch_desc(&tm_ks);
      tma_prefetch_desc(&tm_vs);
      int it = 0, qiss = 0, kiss = 0, viss = 0;   // key tiles; Q, K and V tiles issued
      bool run = true;
      for (int item = blockIdx.x, wi = 0; run && item < p.nitems; item += gridDim.x, ++wi) {
        const BTiles T = tiles_of(p, item);
        // the single Q buffer is free once every S of the previous item is done
        if (wi > 0 && !bpoll(&ctrl->q_empty, (uint32_t)((wi - 1) & 1), ctrl, p.err)) break;
        mbar_arrive_expect_tx(&ctrl->q_full, kBTile);
        tma_load_4d(smem, &tm_q, 0, T.g * p.G, T.p0, T.b, &ctrl->q_full);
        tma_load_4d(smem + kBHalf, &tm_q, 64, T.g * p.G, T.p0, T.b, &ctrl->q_full);
        ++qiss;
        // the next item's Q is read once from HBM: start it towards L2 now, so
        // that its load after this item's last S does not wait on HBM latency
        if (item + (int)gridDim.x < p.nitems) {
          const BTiles N = tiles_of(p, item + (int)gridDim.x);
          tma_prefetch_l2_4d(&tm_q, 0, N.g * p.G, N.p0, N.b);
          tma_prefetch_l2_4d(&tm_q, 64, N.g * p.G, N.p0, N.b);
        }
        for (int t = 0; t < T.nt; ++t, ++it) {
          const int s = it & 1;
          const uint32_t ph = (uint32_t)(((it >> 1) - 1) & 1);
          const bool deep = t < T.nd;
          const int k0 = deep ? t * kBN : T.s_lo + (t - T.nd) * kBN;
          const CUtensorMap* mk = deep ? &tm_kd : &tm_ks;
          const CUtensorMap* mv = deep ? &tm_vd : &tm_vs;
          if (it >= 2 && !bpoll(&ctrl->k_empty[s], ph, ctrl, p.err)) { run = false; break; }
          uint8_t* kb = smem + kBOffK + s * kBTile;
          mbar_arrive_expect_tx(&ctrl->k_full[s], kBTile);
          tma_load_4d(kb, mk, 0, T.g, k0, T.b, &ctrl->k_full[s]);
          tma_load_4d(kb + kBHalf, mk, 64, T.g, k0, T.b, &ctrl->k_full[s]);
          ++kiss;
          if (it >= 2 && !bpoll(&ctrl->v_empty[s], ph, ctrl, p.err)) { run = false; break; }
          uint8_t* vb = smem + kBOffV + s * kBTile;
          mbar_arrive_expect_tx(&ctrl->v_full[s], kBTile);
          tma_load_4d(vb, mv, 0, T.g, k0, T.b, &ctrl->v_full[s]);
          tma_load_4d(vb + kBHalf, mv, 64, T.g, k0, T.b, &ctrl->v_full[s]);
          ++viss;
        }
      }
      // every copy this CTA started has landed before it moves on (the last
      // fill of each buffer; earlier fills were consumed before reuse)
      if (qiss > 0) bdrain(&ctrl->q_full, (uint32_t)((qiss - 1) & 1), p.err);
      for (int j = max(0, kiss - 2); j < kiss; ++j)
        bdrain(&ctrl->k_full[j & 1], (uint32_t)((j >> 1) & 1), p.err);
      for (int j = max(0, viss - 2); j < viss; ++j)
        bdrain(&ctrl->v_full[j & 1], (uint32_t)((j >> 1) & 1), p.err);
    }
    __syncwarp();
  } else if (warp == kBWarpMma) {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      BCursor cs{(int)blockIdx.x, 0, 0, 0}, cp{(int)blockIdx.x, 0, 0, 0};
      cs.nt = cp.nt = cs.item < p.nitems ? tiles_of(p, cs.item).nt : 0;
      int ts = 0, tp = 0;                      // S and PV issued, over all items
      uint32_t idle = 0;
      while (cp.item < p.nitems && !ctrl->abort_flag) {
        bool did = false;
        if (cs.item < p.nitems && ts <= tp + 1 &&
            (cs.t > 0 || mbar_test(&ctrl->q_full, (uint32_t)(cs.wi & 1))) &&
            mbar_test(&ctrl->k_full[ts & 1], (uint32_t)((ts >> 1) & 1))) {
          tc_fence_after();
          const uint32_t d = tmem + (uint32_t)(ts & 1) * kBN;
          const uint32_t kb = sbase + kBOffK + (uint32_t)(ts & 1) * kBTile;
#pragma unroll
          for (int kk = 0; kk < kBD / 16; ++kk) {
            const uint32_t h = kk >> 2, off = (kk & 3) * 32;
            const uint64_t a = smem_desc_sw128(sbase + h * kBHalf + off, 16, 1024);
            const uint64_t bd = smem_desc_sw128(kb + h * kBHalf + off, 16, 1024);
            mma_ss(d, a, bd, kBIdescS, kk > 0 ? 1u : 0u);
          }
          mma_commit(&ctrl->s_full[ts & 1]);
          mma_commit(&ctrl->k_empty[ts & 1]);
          if (cs.t == cs.nt - 1) mma_commit(&ctrl->q_empty);   // the item's last S
          ++ts;
          cursor_next(cs, p);
          did = true;
        }
        if (tp < ts && mbar_test(&ctrl->p_full[tp & 1], (uint32_t)((tp >> 1) & 1)) &&
            mbar_test(&ctrl->v_full[tp & 1], (uint32_t)((tp >> 1) & 1))) {
          tc_fence_after();
          const uint32_t pcol = tmem + (uint32_t)(tp & 1) * kBN;
          const uint32_t ocol = tmem + kBColO + (uint32_t)(cp.wi & 1) * kBD;
          const uint32_t vb = sbase + kBOffV + (uint32_t)(tp & 1) * kBTile;
          // keys [16 kk, 16 kk + 16): P_hi at packed column 32 (kk / 2) + 8 (kk % 2),
          // P_lo 16 columns further
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk) {
            const uint64_t bd = smem_desc_sw128(vb + kk * 2048u, kBHalf, 1024);
            const uint32_t a = pcol + 32 * (kk >> 1) + 8 * (kk & 1);
            mma_ts(ocol, a, bd, kBIdescPV, (cp.t > 0 || kk > 0) ? 1u : 0u);
            mma_ts(ocol, a + 16, bd, kBIdescPV, 1u);
          }
          mma_commit(&ctrl->o_full);
          mma_commit(&ctrl->v_empty[tp & 1]);
          if (cp.t == cp.nt - 1) mma_commit(&ctrl->o_done[cp.wi & 1]);   // the item's O is final
          ++tp;
          cursor_next(cp, p);
          did = true;
        }
        if (did) {
          idle = 0;
        } else if (++idle > (1u << 28)) {
          ctrl->abort_flag = 1;
          raise_err(p.err, SEED_DEVERR_TIMEOUT);
        }
      }
      mma_commit(&ctrl->mma_done);
      bdrain(&ctrl->mma_done, 0, p.err);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------- softmax + epilogue
    const int q4 = warp & 3, hf = warp >> 2;  // lane quarter, column half
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int lg = p.G >> 1;                  // log2 G for G in {1, 2, 4}
    float* xs = reinterpret_cast<float*>(smem + kBOffX);
    float* ls_sh = reinterpret_cast<float*>(smem + kBOffL);
    uint8_t* stage = smem + kBOffE + warp * 4096;
    bool ok = true, pend = false;             // pend: the previous item awaits its epilogue
    BTiles PT{};
    int pwi = 0;
    float pm = 0.f;
    int it = 0;                               // key tiles, over all items
    int item = blockIdx.x, wi = 0, t = 0;
    BTiles T = tiles_of(p, item);
    int pos = T.p0 + (row >> lg);
    bool real = pos <= T.plast;
    int sp = (pos / p.blk) * p.blk;           // this row's block start
    float m_used = -INFINITY, l = 0.f;
    // One step per key tile, then one more after the last item: a tile's step
    // ends by handing its P to the MMA warp; the step of an item's first tile
    // (or the final step) then writes out the previous item.
    while (ok) {
      const bool active = item < p.nitems;
      if (active) {
        ok = bwarp_hot(&ctrl->s_full[it & 1], (uint32_t)((it >> 1) & 1), ctrl, p.err);
        if (!ok) break;
        tc_fence_after();
        const bool deep = t < T.nd;
        const int k0 = (deep ? t * kBN : T.s_lo + (t - T.nd) * kBN) + 64 * hf;
        const int lo = real ? (deep ? 0 : sp) : 1;
        const int hi = real ? (deep ? sp - 1 : pos) : 0;   // visible keys [lo, hi]
        const uint32_t scol = tmem + lane_off + (uint32_t)(it & 1) * kBN + 64u * hf;
        uint32_t ra[32], rb[32];
        tmem_ld32(scol, ra);
        tmem_ld32(scol + 32, rb);
        const uint32_t ba = key_bits(k0, lo, hi), bb = key_bits(k0 + 32, lo, hi);
        const int ka = chunk_kind(ba), kb = chunk_kind(bb);
        tmem_wait_ld();
        float mx = fmaxf(chunk_max(ra, ba, ka), chunk_max(rb, bb, kb));
        // the row's maximum over both column halves
        float* xt = xs + (it & 1) * 256;
        xt[hf * 128 + row] = mx;
        __syncwarp();
        if (lane == 0) mbar_arrive(&ctrl->x_full[it & 1]);
        ok = bwarp_hot(&ctrl->x_full[it & 1], (uint32_t)((it >> 1) & 1), ctrl, p.err);
        if (!ok) break;
        mx = fmaxf(mx, xt[(hf ^ 1) * 128 + row]);
        const float mt = mx * p.c2;
        bool resc = false;
        float fo = 1.f;
        if (mt > m_used + kBRescale) {
          const float f = (m_used == -INFINITY) ? 0.f : ex2_approx(m_used - mt);
          if (t > 0 && m_used != -INFINITY) {
            resc = true;
            fo = f;
          }
          l *= f;
          m_used = mt;
        }
        const float mc = (m_used == -INFINITY) ? 0.f : m_used;
        // P = 2^(s c2 - m) as bf16 hi + lo pairs, in place of S; the second
        // chunk goes through the same code after a register copy
        uint32_t bits = ba;
        int kind = ka;
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          uint32_t wh[16], wl[16];
          l += chunk_p(ra, bits, kind, p.c2, mc, wh, wl);
          tmem_st16(scol + 32 * c, wh);
          tmem_st16(scol + 32 * c + 16, wl);
          if (c == 0) {
#pragma unroll
            for (int i = 0; i < 32; ++i) ra[i] = rb[i];
            bits = bb;
            kind = kb;
          }
        }
        tmem_wait_st();
        // O must be rescaled before PV(t) adds to it: wait for PV(t - 1)
        if (__any_sync(kBFull, resc)) {
          ok = bwarp_hot(&ctrl->o_full, (uint32_t)((it - 1) & 1), ctrl, p.err);
          if (!ok) break;
          tc_fence_after();
          const uint32_t ocol = tmem + lane_off + kBColO + (uint32_t)(wi & 1) * kBD + 64u * hf;
#pragma unroll 1
          for (int c = 0; c < 2; ++c) {
            uint32_t r[32];
            tmem_ld32(ocol + c * 32, r);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * fo);
            tmem_st32(ocol + c * 32, r);
          }
          tmem_wait_st();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&ctrl->p_full[it & 1]);
      }
      // The previous item's O (the other buffer) goes out while PV(t) runs:
      // the row sum over both halves, then O / l through a per-warp staging
      // tile, so that the stores go out as whole 128-byte row pieces (lane i
      // writes its row's 32 values, then each group of 8 lanes writes one row
      // piece; 16-byte chunks swizzled by row).
      if (pend && (t == 0 || !active)) {
        pend = false;
        ok = bwarp_hot(&ctrl->l_full[pwi & 1], (uint32_t)((pwi >> 1) & 1), ctrl, p.err);
        if (!ok) break;
        const float el = ls_sh[(pwi & 1) * 256 + row] + ls_sh[(pwi & 1) * 256 + 128 + row];
        ok = bwarp_hot(&ctrl->o_done[pwi & 1], (uint32_t)((pwi >> 1) & 1), ctrl, p.err);
        if (!ok) break;
        tc_fence_after();
        const uint32_t ocol = tmem + lane_off + kBColO + (uint32_t)(pwi & 1) * kBD + 64u * hf;
        const float inv = el > 0.f ? 1.f / el : 0.f;
        // rows q4 * 32 + 4 i + lane / 8: position p0 + (q4 * 32 + 4 i) / G + (lane / 8) / G
        const int ebase = (PT.b * p.n + PT.p0) * p.hq + PT.g * p.G;
        const int sub = lane >> 3, ch = lane & 7;
        const int eoff = (sub >> lg) * (p.hq - p.G) + sub;    // the lane's part of R + (R / G)(hq - G)
#pragma unroll 1
        for (int c = 0; c < 2; ++c) {
          uint32_t r[32];
          tmem_ld32(ocol + c * 32, r);
          tmem_wait_ld();
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(stage + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                make_float4(__uint_as_float(r[4 * j]) * inv, __uint_as_float(r[4 * j + 1]) * inv,
                            __uint_as_float(r[4 * j + 2]) * inv,
                            __uint_as_float(r[4 * j + 3]) * inv);
          __syncwarp();
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int rr = i * 4 + sub;
            const int R0 = q4 * 32 + i * 4;                   // a multiple of G
            const float4 v =
                *reinterpret_cast<const float4*>(stage + rr * 128 + ((ch ^ (rr & 7)) << 4));
            if (PT.p0 + ((R0 + sub) >> lg) <= PT.plast) {
              const size_t orow = (size_t)ebase + R0 + (R0 >> lg) * (p.hq - p.G) + eoff;
              *reinterpret_cast<float4*>(p.out + orow * kBD + 64 * hf + 32 * c + 4 * ch) = v;
            }
          }
          __syncwarp();
        }
        const int epos = PT.p0 + (row >> lg);
        if (epos <= PT.plast && hf == 0 && p.lse != nullptr)
          p.lse[((size_t)PT.b * p.n + epos) * p.hq + PT.g * p.G + (row & (p.G - 1))] =
              (pm + log2f(el)) * kBLn2;
        tc_fence_before();
      }
      if (!active) break;
      ++it;
      if (++t == T.nt) {
        // the item's last tile: publish its row sum and leave its epilogue
        // for the next step that starts an item
        ls_sh[(wi & 1) * 256 + hf * 128 + row] = l;
        __syncwarp();
        if (lane == 0) mbar_arrive(&ctrl->l_full[wi & 1]);
        pend = true;
        PT = T;
        pwi = wi;
        pm = m_used;
        item += gridDim.x;
        ++wi;
        t = 0;
        if (item < p.nitems) {
          T = tiles_of(p, item);
          pos = T.p0 + (row >> lg);
          real = pos <= T.plast;
          sp = (pos / p.blk) * p.blk;
          m_used = -INFINITY;
          l = 0.f;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kBWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------------------- host side
using EncodeFnB = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                               const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                               const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                               CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFnB encode_fn_b() {
  static EncodeFnB fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFnB>(ptr);
  });
  return fn;
}

// 4-d bf16 map [B, n, heads, 128] with (64, hbox, rows, 1) boxes, 128-byte swizzle.
bool encode_bthd(CUtensorMap* map, const void* base, int B, int n, int heads, int hbox,
                 int rows) {
  EncodeFnB fn = encode_fn_b();
  if (fn == nullptr) return false;
  const cuuint64_t dims[4] = {(cuuint64_t)kBD, (cuuint64_t)heads, (cuuint64_t)n, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)kBD * 2, (cuuint64_t)heads * kBD * 2,
                                 (cuuint64_t)n * heads * kBD * 2};
  const cuuint32_t box[4] = {64, (cuuint32_t)hbox, (cuuint32_t)rows, 1};
  const cuuint32_t elem[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

std::atomic<uint64_t> g_block_attr{0};

}  // namespace

bool block_tc_supported(int32_t head_dim, int32_t group) {
  return head_dim == kBD && (group == 1 || group == 2 || group == 4);
}

cudaError_t launch_block_tc(int32_t B, int32_t n, int32_t blk, int32_t hq, int32_t hkv,
                            float scale, const void* q, const void* k_dec, const void* v_dec,
                            const void* k_spec, const void* v_spec, float* out, float* lse,
                            int32_t* err, cudaStream_t st) {
  BlockTcParams p{};
  p.out = out;
  p.lse = lse;
  p.err = err;
  p.B = B;
  p.n = n;
  p.blk = blk;
  p.hq = hq;
  p.hkv = hkv;
  p.G = hq / hkv;
  p.P = 128 / p.G;
  p.nqt = (n + p.P - 1) / p.P;
  const long long items = (long long)B * hkv * p.nqt;
  if (items <= 0 || items > 0x7fffffffLL) return cudaErrorInvalidValue;
  p.nitems = (int32_t)items;
  p.c2 = scale * 1.4426950408889634f;
  CUtensorMap tq, tkd, tvd, tks, tvs;
  if (!encode_bthd(&tq, q, B, n, hq, p.G, p.P) || !encode_bthd(&tkd, k_dec, B, n, hkv, 1, kBN) ||
      !encode_bthd(&tvd, v_dec, B, n, hkv, 1, kBN) ||
      !encode_bthd(&tks, k_spec, B, n, hkv, 1, kBN) ||
      !encode_bthd(&tvs, v_spec, B, n, hkv, 1, kBN))
    return cudaErrorInvalidValue;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(g_block_attr.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(block_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kBSmem);
    if (e != cudaSuccess) return e;
    g_block_attr.fetch_or(bit, std::memory_order_acq_rel);
  }
  const int grid = (int)std::min<long long>(items, std::max(1, device_sm_count()));
  return launch_pdl(block_tc_kernel, dim3((unsigned)grid), dim3(kBThreads), kBSmem, st, tq, tkd,
                    tvd, tks, tvs, p);
}

}  // namespace seedk
