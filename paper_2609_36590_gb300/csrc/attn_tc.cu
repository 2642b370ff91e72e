// Draft and verify attention on the 5th-generation tensor cores (tcgen05,
// TMEM, TMA).
//
// What it computes (Sec. 4.1: the drafter's cross-attention is ordinary
// self-attention over the cache; Alg. 2 fixes the visible rows), for sequence
// b and each of the G query heads of KV head g:
//   verify: query j < n_q[b] (token X_draft[j]) over cache rows 0 .. L + j,
//           L = ctx_lens[b] (the cache already holds the n_q new rows);
//   draft:  one query over cache rows 0 .. L - 1 (the deep KV the last
//           verification left) followed by draft rows 0 .. nd - 1 of the
//           draft scratch (X_draft[0 .. nd-1], the query's own row included).
//
// Design.  All G * n_q query rows of one (sequence, KV head) sit in the rows
// of one M=128 MMA tile, so every K/V byte is read from HBM once per call
// whatever k is.  A sequence is a list of 16-token pages (cache pages, then for
// the draft one page holding the draft rows); 8 pages make a 128-token tile
// that flows through a 3-stage TMA ring (128-byte swizzled boxes of one page x
// 64 head dims).  Per tile one thread issues S = Q K^T (8 MMAs, M=128 N=128
// K=16) into a double-buffered TMEM accumulator; four softmax warps (one per
// TMEM lane quarter, one thread per query row) read S, mask it per column,
// run the online softmax in log2 units (the output accumulator is rescaled
// only when the running maximum grows by more than 2^8) and write the
// probabilities back into the same TMEM columns as two bf16 halves
// P = P_hi + P_lo (P_hi = bf16(P), P_lo = bf16(P - P_hi)); the MMA thread
// then accumulates O += P_hi V + P_lo V with A read from TMEM and V read
// MN-major from shared memory.  The two-term split keeps ~16 bits of each
// probability, enough for 2e-3 absolute accuracy on the peaked rows of the
// x8-key workload (one bf16 term alone is not).  V rows of columns that no
// query may see (past the sequence end, unfilled page slots) are zeroed in
// shared memory before PV so that stale or poisoned rows contribute nothing.
//
// Work: the launch's tiles, ordered by (sequence, KV head, tile), are cut
// into one contiguous range per CTA of (almost) equal length.  A CTA's range
// covers whole (b, g) pairs, whose outputs it writes directly, and at most
// two pieces of pairs shared with its neighbours; for those it leaves a
// normalised partial and its log2-sum-exps in one of its two record slots.
// A second, small kernel merges the pieces of every shared pair in range
// order, so results are deterministic and no CTA ever waits for another.
//
// Warp roles (384 threads): warps 0-7 softmax / epilogue (two groups of four,
// one warp per TMEM lane quarter), warp 10 TMA producer and scheduler, warp 11
// MMA issuer and TMEM owner; warps 8-9 only keep the role warps off the
// sub-partition of lane quarter 0.  Every wait is bounded;
// a wait that gives up raises SEED_DEVERR_TIMEOUT and all roles drain out.
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <mutex>

#include "attn_sched.cuh"
#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace seedk {
namespace {

using namespace sched;

constexpr int kD = 128;
constexpr int kN = 128;                      // tokens (columns) per tile
constexpr int kStagesTC = 3;
constexpr int kThreadsTC = 384;   // warps 0-7 softmax, 8 idle, 9 V loads, 10 K loads, 11 MMA
constexpr int kWarpLoadV = 9, kWarpProducer = 10, kWarpMma = 11;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 256;              // O accumulators: [256, 384) and [384, 512)
constexpr float kRescale = 8.0f;
constexpr float kLn2 = 0.69314718055994531f;

constexpr int kMetaRing = 2 * kStagesTC;      // tile descriptors in flight

constexpr uint32_t kHalf = kN * 128;                   // 16 KiB: 128 rows x 128 B
constexpr uint32_t kQBytes = 2 * kHalf;                // Q: two head-dim halves
constexpr uint32_t kKV = 2 * kHalf;                    // one tile's K (or V): two halves
constexpr uint32_t kOffK = kQBytes;                    // K ring
constexpr uint32_t kOffV = kOffK + kStagesTC * kKV;    // V ring
constexpr uint32_t kOffCtrl = kOffV + kStagesTC * kKV;

constexpr uint32_t kIdescS = idesc_bf16_f32(128, kN, 0, 0);     // K-major A and B
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, kD, 0, 1);    // B (V) MN-major

struct TileMeta {
  int32_t unit;        // < 0: no more tiles (else: index of the piece in the CTA)
  int32_t b, g;
  int32_t tile;        // tile index within the sequence
  int32_t k, ntu;      // tile index within the unit; tiles in the unit
  int32_t nq, nd;      // query positions; draft rows (draft mode)
  int32_t ncp;         // cache pages of the sequence
  int32_t cvalid;      // cache rows that exist (L, or L + n_q for verify)
  int32_t lim0;        // query j sees cache positions <= lim0 + j
  int32_t slot;        // partial record of this piece, or -1: the whole pair
  int32_t dslot;       // page slot of draft page 0 (outside [0, 8) when not in this tile)
  int32_t pad[3];
  int32_t pids[kPagesPerTile];   // cache page of each page slot, -1: none
};

struct Ctrl {
  uint64_t k_full[kStagesTC], k_empty[kStagesTC];   // K ring
  uint64_t v_full[kStagesTC], v_empty[kStagesTC];   // V ring
  uint64_t q_full[2], q_empty[2];             // Q buffers (two when the rows fit 64)
  uint64_t meta_full[kMetaRing], meta_empty[kMetaRing];   // K warp -> V warp
  uint64_t s_full[2], p_full[2], o_full[2];   // per tile parity
  uint64_t stats_bar[4], orel_bar[4];         // per TMEM lane quarter
  uint32_t tmem_base;
  volatile int32_t abort_flag;
  int32_t end_tile;                           // first tile index past the CTA's work
  TileMeta meta[kMetaRing];
  float xm[4][32], xl[4][32];                 // row statistics handed to the epilogue owner
};

constexpr size_t kSmemTC = kOffCtrl + sizeof(Ctrl) + 1024;   // + alignment slack
static_assert(kSmemTC <= 232448, "shared memory budget");

// Bounded wait (about 2 s) on an mbarrier phase; the waiting thread sleeps in
// hardware between tries.  Gives up early if another role has aborted.  Out of
// line, like the other cold helpers below: the kernel's code must stay small
// enough for the instruction cache, or its warps stall on instruction fetch.
__device__ __noinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, Ctrl* c,
                                           int32_t* err) {
  for (uint32_t i = 0; i < kSuspendTries; ++i) {
    if (mbar_try_wait_sleep(bar, parity, kSuspendNs)) return true;
    if (c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

// Bounded wait by a whole warp: the lanes agree on the outcome, so that an
// abort racing with the barrier's completion cannot split the warp.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, Ctrl* c, int32_t* err) {
  return __all_sync(0xffffffffu, wait_or_abort(bar, parity, c, err));
}

// The softmax and epilogue warps' waits: try_wait without a sleep hint, so the
// warp resumes as soon as the phase completes (a sleeping wait's wake-up
// comes later, which each tile of a short launch pays in full); bounded like
// wait_or_abort (the abort flag is read every 64 tries).
__device__ __noinline__ bool wait_hot(uint64_t* bar, uint32_t parity, Ctrl* c, int32_t* err) {
  for (uint32_t i = 0; i < (1u << 22); ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 63u && c->abort_flag) return false;
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ bool warp_wait_hot(uint64_t* bar, uint32_t parity, Ctrl* c,
                                              int32_t* err) {
  return __all_sync(0xffffffffu, wait_hot(bar, parity, c, err));
}

// ------------------------------------------------------------- the kernel
// One softmax row: the visible columns of a tile for query j are the cache
// columns c <= lim (c < dcol) and the draft columns dcol <= c < dend.
// For a tree verify (Sec. D.1) the cache columns of the tree's packed rows
// start at column tb, and bit a of tm makes packed row a visible.
struct ColMask {
  int dcol, dend, lim, tb;
  uint32_t tm;
  // bit i set <=> column c0 + i is visible
  __device__ __forceinline__ uint32_t bits(int c0) const {
    const int nc = min(max(min(lim, dcol - 1) - c0 + 1, 0), 32);
    const int lo = min(max(dcol - c0, 0), 32), hi = min(max(dend - c0, 0), 32);
    const uint32_t mc = nc == 32 ? 0xffffffffu : ((1u << nc) - 1u);
    const uint32_t mh = hi == 32 ? 0xffffffffu : ((1u << hi) - 1u);
    const uint32_t ml = lo == 32 ? 0xffffffffu : ((1u << lo) - 1u);
    const int off = c0 - tb;   // packed row seen at column c0
    const uint32_t mt = (off >= 32 || off <= -32) ? 0u : off >= 0 ? (tm >> off) : (tm << -off);
    return mc | (mh & ~ml) | mt;
  }
};

// Pass 1 of a tile's softmax row: maximum of the raw scores over the visible
// columns.  MASKED = false for the (common) tiles every column of which is
// visible, so that their loop carries no per-column test.
template <bool MASKED>
__device__ __forceinline__ float row_max(uint32_t scol, const ColMask& cm) {
  float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll 1
  for (int c = 0; c < kN / 32; ++c) {
    uint32_t r[32];
    tmem_ld32(scol + c * 32, r);
    tmem_wait_ld();
    const uint32_t bits = MASKED ? cm.bits(32 * c) : 0xffffffffu;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      float v = __uint_as_float(r[i]);
      if (MASKED) v = ((bits >> i) & 1u) ? v : -INFINITY;
      mx[i & 3] = fmaxf(mx[i & 3], v);
    }
  }
  return fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
}

// Pass 2: p = 2^(s*c2 - mc) written back as P_hi / P_lo bf16 pairs -- tokens
// [32c, 32c+32) to packed columns [32c, 32c+16) (P_hi) and [32c+16, 32c+32)
// (P_lo), i.e. inside the S columns this chunk has already consumed; even
// token in the low half-word.  Returns the sum of the p.
template <bool MASKED>
__device__ __forceinline__ float row_p(uint32_t scol, const ColMask& cm, float c2, float mc) {
  float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
  for (int c = 0; c < kN / 32; ++c) {
    uint32_t r[32];
    tmem_ld32(scol + 32 * c, r);
    tmem_wait_ld();
    const uint32_t bits = MASKED ? cm.bits(32 * c) : 0xffffffffu;
    uint32_t wh[16], wl[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float s0 = __uint_as_float(r[2 * i]);
      float s1 = __uint_as_float(r[2 * i + 1]);
      if (MASKED) {
        s0 = ((bits >> (2 * i)) & 1u) ? s0 : -INFINITY;
        s1 = ((bits >> (2 * i + 1)) & 1u) ? s1 : -INFINITY;
      }
      const float p0 = ex2_approx(fmaf(s0, c2, -mc));
      const float p1 = ex2_approx(fmaf(s1, c2, -mc));
      ls[i & 3] += p0 + p1;
      const uint32_t h = pack_bf16x2(p0, p1);
      wh[i] = h;
      wl[i] = pack_bf16x2(p0 - bf16lo(h), p1 - bf16hi(h));
    }
    tmem_st16(scol + 32 * c, wh);
    tmem_st16(scol + 32 * c + 16, wl);
  }
  tmem_wait_st();
  return (ls[0] + ls[1]) + (ls[2] + ls[3]);
}

// Epilogue of one piece for one warp's rows (run by the group that processed
// the piece's last tile): combine the two groups' partial softmax states,
// normalise, and write the output rows -- or, for a piece of a pair shared
// with other CTAs, this piece's partial record (same row-major layout:
// [row][d], then the per-row log2-sum-exp) for the merge kernel.  Kept out of
// line: it runs once per piece and needs more registers than the tile loop.
__device__ __noinline__ void unit_epilogue(const AttnTcParams& p, int b, int g, int nq, int slot,
                                           int row, uint32_t ocol, uint32_t ocol_other,
                                           float m_used, float l, float mo, float lo) {
  const int Rmax = p.G * p.W1;
  const int R = nq * p.G;
  const int j = row / p.G;
  const float M = fmaxf(m_used, lo > 0.f ? mo : -INFINITY);
  const float fa = (l > 0.f) ? ex2_approx(m_used - M) : 0.f;
  const float fb = (lo > 0.f) ? ex2_approx(mo - M) : 0.f;
  const float Ls = l * fa + lo * fb;
  const float inv = (Ls > 0.f) ? 1.f / Ls : 0.f;
  const float lse2 = (Ls > 0.f) ? M + log2f(Ls) : -INFINITY;
  const bool use_other = __any_sync(kFull, lo > 0.f);
  const bool real = row < R;
  const int qh = g * p.G + (row - j * p.G);
  const size_t orow = ((size_t)b * p.W1 + j) * p.hq + qh;   // [b, j, head]
  float* rec = p.part + (size_t)max(slot, 0) * Rmax * (kD + 1);
  float* dst = slot < 0 ? p.out + orow * kD : rec + (size_t)row * kD;
#pragma unroll 1
  for (int c = 0; c < kD / 16; ++c) {
    uint32_t ra[16], rb[16];
    tmem_ld16(ocol + c * 16, ra);
    if (use_other) tmem_ld16(ocol_other + c * 16, rb);
    tmem_wait_ld();
    float v[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float x = __uint_as_float(ra[i]) * fa;
      if (use_other && lo > 0.f) x = fmaf(__uint_as_float(rb[i]), fb, x);
      v[i] = x * inv;
    }
    if (real) {
      float4* dp = reinterpret_cast<float4*>(dst + c * 16);
#pragma unroll
      for (int i = 0; i < 4; ++i)
        dp[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    }
  }
  if (real) {
    if (slot >= 0)
      rec[(size_t)kD * Rmax + row] = lse2;
    else if (p.lse != nullptr)
      p.lse[orow] = lse2 * kLn2;
  }
}

// Merge of the pieces of a pair (b, g) whose tiles span several CTAs of the
// attention kernel: the pieces' records are combined with weights
// 2^(lse_i - M) / sum, in range order.  Block x looks at the boundary where
// CTA x + 1's range starts and merges the pair that boundary splits, if it is
// the pair's first such boundary (the attention kernel's CTA x + 1 leaves
// that in the merge plan); so the grid has one block column per boundary,
// whatever the number of pairs.  One warp per query row (rows
// 8 * blockIdx.y + warp), one lane per 4 head dims; each lane reads every
// piece's log2-sum-exp and values in one online pass, kMergeBatch pieces at a
// time.
constexpr int kMergeThreads = 256;
constexpr int kMergeRows = kMergeThreads / 32;
constexpr int kMergeBatch = 8;

// Per-lane slice of a record row: D / 32 consecutive floats (4 for D = 128,
// 2 for D = 64) moved as one vector.
template <int D> struct MergeVec;
template <> struct MergeVec<128> {
  using T = float4;
  __device__ static void to(const T& v, float* f) { f[0] = v.x; f[1] = v.y; f[2] = v.z; f[3] = v.w; }
  __device__ static T from(const float* f) { return make_float4(f[0], f[1], f[2], f[3]); }
};
template <> struct MergeVec<64> {
  using T = float2;
  __device__ static void to(const T& v, float* f) { f[0] = v.x; f[1] = v.y; }
  __device__ static T from(const float* f) { return make_float2(f[0], f[1]); }
};

template <int D>
__global__ void __launch_bounds__(kMergeThreads) attn_merge_kernel(const AttnTcParams p) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // Block x handles range boundary c = x + 1: its plan entry, written by the
  // attention kernel's CTA c, names the pair to merge (b < 0: none)
  const int c = blockIdx.x + 1;
  const int4* pe = reinterpret_cast<const int4*>(p.plan + (size_t)c * kPlanInts);
  const int4 e0 = __ldcg(pe), e1 = __ldcg(pe + 1);
  const int b = e0.x, g = e0.y, slot_lo = e0.z, c_lo = e0.w;
  const int nseg = e1.x, R = e1.y;
  const int r = blockIdx.y * kMergeRows + warp;   // query row j * G + head
  if (b < 0 || r >= R) return;
  const int Rmax = p.G * p.W1;
  const size_t REC = (size_t)Rmax * (D + 1);
  using V = MergeVec<D>;
  constexpr int kPer = D / 32;
  float M = -INFINITY, S = 0.f;
  float acc[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) acc[e] = 0.f;
  for (int i0 = 0; i0 < nseg; i0 += kMergeBatch) {
    float li[kMergeBatch];
    typename V::T x[kMergeBatch];
    // only the pieces that exist are loaded: the merge's time is its loads
    // once the attention kernel has ended, and a batch padded with repeats of
    // the last piece multiplied them (a pair has 2 or 3 pieces, typically)
#pragma unroll
    for (int u = 0; u < kMergeBatch; ++u) {
      li[u] = -INFINITY;
      x[u] = typename V::T{};
      if (i0 + u < nseg) {
        const int i = i0 + u;
        const float* rc = p.part + (size_t)(i == 0 ? slot_lo : 2 * (c_lo + i)) * REC;
        li[u] = __ldcg(rc + (size_t)D * Rmax + r);
        x[u] = __ldcg(reinterpret_cast<const typename V::T*>(rc + (size_t)r * D) + lane);
      }
    }
#pragma unroll
    for (int u = 0; u < kMergeBatch; ++u) {
      if (li[u] == -INFINITY) continue;
      float w = 1.f;
      if (li[u] > M) {
        const float f = ex2_approx(M - li[u]);   // 0 for the first piece
        S *= f;
#pragma unroll
        for (int e = 0; e < kPer; ++e) acc[e] *= f;
        M = li[u];
      } else {
        w = ex2_approx(li[u] - M);
      }
      S += w;
      float xv[kPer];
      V::to(x[u], xv);
#pragma unroll
      for (int e = 0; e < kPer; ++e) acc[e] = fmaf(w, xv[e], acc[e]);
    }
  }
  const float inv = 1.f / S;
  const int j = r / p.G;
  const size_t orow = ((size_t)b * p.W1 + j) * p.hq + g * p.G + (r - j * p.G);
  float res[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) res[e] = acc[e] * inv;
  reinterpret_cast<typename V::T*>(p.out + orow * D)[lane] = V::from(res);
  if (lane == 0 && p.lse != nullptr) p.lse[orow] = (M + log2f(S)) * kLn2;
}

// No __launch_bounds__: with it ptxas budgets the 320-thread block like a
// 384-thread one and spills in the per-tile loop; without it the kernel fits
// in 168 registers with no spills (a launch that did not fit would fail with
// an error, never run).
__global__ void attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q,
                   const __grid_constant__ PageMaps pm,
                   const __grid_constant__ CUtensorMap tm_dk,
                   const __grid_constant__ CUtensorMap tm_dv, const AttnTcParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // the 128-byte swizzled tiles need a 1 KiB aligned base
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  Ctrl* ctrl = reinterpret_cast<Ctrl*>(smem + kOffCtrl);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  if (tid == 0) pdl_trigger();

  if (tid == 0) {
    // one arrival per lane quarter that can hold query rows in this launch
    const int nqa = min(4, (p.G * p.W1 + 31) / 32);
    for (int s = 0; s < kStagesTC; ++s) {
      mbar_init(&ctrl->k_full[s], 1);
      mbar_init(&ctrl->k_empty[s], 1);
      mbar_init(&ctrl->v_full[s], 1);
      mbar_init(&ctrl->v_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->q_full[i], 1);
      mbar_init(&ctrl->q_empty[i], 1);
    }
    for (int i = 0; i < kMetaRing; ++i) {
      mbar_init(&ctrl->meta_full[i], 1);
      mbar_init(&ctrl->meta_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->s_full[i], 1);
      mbar_init(&ctrl->p_full[i], nqa);
      mbar_init(&ctrl->o_full[i], 1);
    }
    for (int i = 0; i < 4; ++i) {
      mbar_init(&ctrl->stats_bar[i], 1);
      mbar_init(&ctrl->orel_bar[i], 1);
    }
    ctrl->abort_flag = 0;
    ctrl->end_tile = 1 << 30;
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(&ctrl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctrl->tmem_base;
  const int Rmax = p.G * p.W1;
  // Q buffers.  With at most 64 query rows, two compact buffers (rows padded
  // to 8, each head-dim half Rpad x 128 B) share the Q region, so that the Q
  // of the next piece loads while S of the current one runs.  The MMA reads
  // 128 rows from a buffer; rows past its Rpad are unused garbage rows.
  const int Rpad = (Rmax + 7) & ~7;
  const int nqb = Rpad <= 64 ? 2 : 1;
  const uint32_t qhalf = nqb == 2 ? (uint32_t)Rpad * 128u : kHalf;
  if (warp == kWarpProducer) {
    // descriptors are kernel parameters; the lengths are only pulled into L2
    // (a prefetch returns nothing, so a predecessor still writing them is
    // harmless): both before the dependency wait
    if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      for (int i = 0; i < 4; ++i) {
        tma_prefetch_desc(&pm.k[i]);
        tma_prefetch_desc(&pm.v[i]);
      }
      if (p.draft) {
        tma_prefetch_desc(&tm_dk);
        tma_prefetch_desc(&tm_dv);
      }
    }
    prefetch_lens_l2(p, lane);
  }
  // everything above touched only this CTA's shared and tensor memory
  pdl_wait();

  if (warp == kWarpProducer) {
    // ---------------------------------------------------------- producer
    if (blockIdx.x == 0) {
      for (int b = lane; b < p.B; b += 32) {
        const int bad = seq_of(p, b).bad;
        if (bad) raise_err(p.err, bad);
      }
    }
    // this CTA's units [x, x1)
    long long T, x, x1;
    SeqWin win;
    int b = p.B, g = 0, t0 = 0;
    long long pc = 0;   // first unit of pair (b, g)
    lookup_range(p, lane, T, x, x1, win, b, g, t0, pc);
    {
      const SeqT s0 = b < p.B ? win_get(win, b) : SeqT{};
      if (lane == 0) write_merge_plan(p, T, x, x1, b, g, t0, pc, s0);
    }
    // K tiles in range order, each into the K ring as soon as a slot is free
    // (a slot frees when S of its tile is done).  Each tile's descriptor goes
    // to the descriptor ring, from which the V warp issues the tile's V.
    int tk = 0, uo = 0;
    bool ok = true;
    const uint64_t kv_pol = policy_evict_first();   // K is read once per call
    // page ids of tiles t and t + 1 of the piece (lanes 0-7, one page each),
    // loaded ahead so that their latency overlaps the copies
    int pid_a = -1, pid_b = -1;
    SeqT sq{};
    int t1 = 0;
    auto load_pid = [&](int tt) -> int {
      const int vp = tt * kPagesPerTile + (lane & 7);
      return (lane < kPagesPerTile && tt < t1 && vp < sq.ncp)
                 ? __ldg(p.page_table + (size_t)b * p.max_pages + vp)
                 : -1;
    };
    while (ok && b < p.B) {
      // one piece: tiles [t0, t1) of pair (b, g), those whose units lie below x1
      sq = win_get(win, b);
      t1 = (int)min((long long)sq.tiles, x1 - pc - kPairCost);
      if (t1 <= t0) break;
      const int slot = (t0 == 0 && t1 == sq.tiles) ? -1 : 2 * (int)blockIdx.x + (uo > 0 ? 1 : 0);
      pid_a = load_pid(t0);
      pid_b = load_pid(t0 + 1);
      for (int t = t0; t < t1; ++t, ++tk) {
        const int s = tk % kStagesTC, mi = tk % kMetaRing;
        int pid = pid_a;
        pid_a = pid_b;
        pid_b = load_pid(t + 2);
        if (tk >= kStagesTC)
          ok = warp_wait(&ctrl->k_empty[s], ((tk / kStagesTC) - 1) & 1, ctrl, p.err);
        if (ok && tk >= kMetaRing)
          ok = warp_wait(&ctrl->meta_empty[mi], ((tk / kMetaRing) - 1) & 1, ctrl, p.err);
        if (ok && t == t0 && uo >= nqb)
          ok = warp_wait(&ctrl->q_empty[uo % nqb], ((uo / nqb) - 1) & 1, ctrl, p.err);
        if (!ok) break;
        if (lane < kPagesPerTile && t * kPagesPerTile + lane < sq.ncp &&
            (pid < 0 || pid >= p.num_pages)) {
          raise_err(p.err, SEED_DEVERR_PAGE);
          pid = -1;
        }
        // lane pp < 8 owns page slot pp of the tile
        // slot of draft page 0 (may lie outside the tile); lane pp holds
        // draft page dpage when the tile's slot pp is one
        const int dslot = sq.ncp - t * kPagesPerTile;
        const int dpage = lane < kPagesPerTile ? draft_page_of_slot(sq.ncp, sq.nd, t, lane) : -1;
        const bool has = lane < kPagesPerTile && (pid >= 0 || dpage >= 0);
        const uint32_t loads = __ballot_sync(kFull, has);
        const int box = box_size(pid, lane);
        TileMeta& m = ctrl->meta[mi];
        if (lane < kPagesPerTile) m.pids[lane] = pid;
        __syncwarp();
        if (lane == 0) {
          m.unit = uo;
          m.b = b;
          m.g = g;
          m.tile = t;
          m.k = t - t0;
          m.ntu = t1 - t0;
          m.nq = sq.nq;
          m.nd = sq.nd;
          m.ncp = sq.ncp;
          m.cvalid = sq.cvalid;
          m.lim0 = sq.lim0;
          m.slot = slot;
          m.dslot = dslot;
          mbar_arrive(&ctrl->meta_full[mi]);
          if (t == t0) {
            const int qb = uo % nqb;
            uint8_t* qd = smem + (size_t)qb * 2 * qhalf;
            mbar_arrive_expect_tx(&ctrl->q_full[qb], 2u * 128u * (uint32_t)Rmax);
            tma_load_4d(qd, &tm_q, 0, g * p.G, 0, b, &ctrl->q_full[qb]);
            tma_load_4d(qd + qhalf, &tm_q, 64, g * p.G, 0, b, &ctrl->q_full[qb]);
          }
          mbar_arrive_expect_tx(&ctrl->k_full[s], (uint32_t)__popc(loads) * 2u * 2048u);
        }
        __syncwarp();
        if (box > 0 || (has && pid < 0)) {
          // a box of `box` pages from this slot on, or the draft rows' page
          uint8_t* kb = smem + kOffK + (size_t)s * kKV + lane * 2048u;
          const CUtensorMap* mk = box > 0 ? &pm.k[log2_box(box)] : &tm_dk;
          const int w = box > 0 ? pid : b, r0 = box > 0 ? 0 : kPage * dpage;
          tma_load_4d_hint(kb, mk, 0, r0, g, w, &ctrl->k_full[s], kv_pol);
          tma_load_4d_hint(kb + kHalf, mk, 64, r0, g, w, &ctrl->k_full[s], kv_pol);
        }
      }
      if (!ok) break;
      ++uo;
      if (t1 < sq.tiles) break;
      // the range goes on with the next pair
      pc += sq.tiles + kPairCost;
      t0 = 0;
      if (++g == p.hkv) {
        g = 0;
        next_seq(p, lane, win, b);
      }
    }
    // end markers: one for each softmax parity (the MMA thread stops at the
    // first, the V warp too)
    for (int e = 0; e < 2 && ok; ++e, ++tk) {
      const int s = tk % kStagesTC, mi = tk % kMetaRing;
      if (tk >= kStagesTC)
        ok = warp_wait(&ctrl->k_empty[s], ((tk / kStagesTC) - 1) & 1, ctrl, p.err);
      if (ok && tk >= kMetaRing)
        ok = warp_wait(&ctrl->meta_empty[mi], ((tk / kMetaRing) - 1) & 1, ctrl, p.err);
      if (ok && lane == 0) {
        ctrl->meta[mi].unit = -1;
        mbar_arrive(&ctrl->meta_full[mi]);
        mbar_arrive(&ctrl->k_full[s]);
      }
    }
    __syncwarp();
  } else if (warp == kWarpLoadV) {
    // ---------------------------------------------------------- V loads
    // V(t) into the V ring once tile t's descriptor is out and PV(t - 3)
    // has freed the slot
    const uint64_t kv_pol = policy_evict_first();   // V is read once per call
    for (int tv = 0;; ++tv) {
      const int s = tv % kStagesTC, mi = tv % kMetaRing;
      if (!warp_wait(&ctrl->meta_full[mi], (tv / kMetaRing) & 1, ctrl, p.err)) break;
      const TileMeta& m = ctrl->meta[mi];
      if (m.unit < 0) break;
      const int pid = lane < kPagesPerTile ? m.pids[lane] : -1;
      const int mb = m.b, mg = m.g, dslot = m.dslot, nd = m.nd;
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->meta_empty[mi]);
      if (tv >= kStagesTC &&
          !warp_wait(&ctrl->v_empty[s], ((tv / kStagesTC) - 1) & 1, ctrl, p.err))
        break;
      const int dpage =
          (lane < kPagesPerTile && lane >= dslot && lane - dslot < draft_pages(nd)) ? lane - dslot
                                                                                     : -1;
      const bool has = lane < kPagesPerTile && (pid >= 0 || dpage >= 0);
      const uint32_t loads = __ballot_sync(kFull, has);
      if (lane == 0)
        mbar_arrive_expect_tx(&ctrl->v_full[s], (uint32_t)__popc(loads) * 2u * 2048u);
      __syncwarp();
      const int box = box_size(pid, lane);
      if (box > 0 || (has && pid < 0)) {
        uint8_t* vb = smem + kOffV + (size_t)s * kKV + lane * 2048u;
        const CUtensorMap* mv = box > 0 ? &pm.v[log2_box(box)] : &tm_dv;
        const int w = box > 0 ? pid : mb, r0 = box > 0 ? 0 : kPage * dpage;
        tma_load_4d_hint(vb, mv, 0, r0, mg, w, &ctrl->v_full[s], kv_pol);
        tma_load_4d_hint(vb + kHalf, mv, 64, r0, mg, w, &ctrl->v_full[s], kv_pol);
      }
    }
    __syncwarp();
  } else if (warp == kWarpMma) {
    // ---------------------------------------------------------- MMA issuer
    // An event loop over two streams: S(ts) = Q K^T of the next loaded tile
    // and PV(tp) of the next tile whose probabilities are written.  Either is
    // issued as soon as it is ready; the only orderings kept are PV(t) after
    // S(t) and S(t) after PV(t-2) (S(t) overwrites P(t-2) in the same TMEM
    // columns; one thread's MMAs execute in issue order).
    if (lane == 0) {
      int ts = 0, tp = 0, uo = 0, qcur = 0, t_end = 1 << 30;
      int k_of[kStagesTC];               // tile index within its unit, per stage
      uint32_t idle = 0;
      while (tp < t_end && !ctrl->abort_flag) {
        bool did = false;
        if (ts < t_end && ts <= tp + 1) {
          const int s = ts % kStagesTC;
          const TileMeta& mt = ctrl->meta[ts % kMetaRing];
          if (mbar_test(&ctrl->k_full[s], (ts / kStagesTC) & 1)) {
            const int unit = mt.unit;
            if (unit < 0) {
              t_end = ts;   // no more tiles
              did = true;
            } else {
              const int k = mt.k;
              const bool q_ok = (k != 0) || mbar_test(&ctrl->q_full[uo % nqb], (uo / nqb) & 1);
              if (q_ok) {
                if (k == 0) {
                  qcur = uo % nqb;
                  ++uo;
                }
                k_of[s] = k;
                tc_fence_after();
                const uint32_t d = tmem + (uint32_t)(ts & 1) * kN;
                const uint32_t kb = sbase + kOffK + (uint32_t)s * kKV;
#pragma unroll 1
                for (int kk = 0; kk < kD / 16; ++kk) {
                  const uint32_t h = kk >> 2, off = (kk & 3) * 32;
                  const uint64_t a =
                      smem_desc_sw128(sbase + (uint32_t)(qcur * 2 + h) * qhalf + off, 16, 1024);
                  const uint64_t b = smem_desc_sw128(kb + h * kHalf + off, 16, 1024);
                  mma_ss(d, a, b, kIdescS, kk > 0);
                }
                mma_commit(&ctrl->s_full[ts & 1]);
                mma_commit(&ctrl->k_empty[s]);
                if (mt.k == mt.ntu - 1) mma_commit(&ctrl->q_empty[qcur]);
                ++ts;
                did = true;
              }
            }
          }
        }
        if (tp < ts && mbar_test(&ctrl->p_full[tp & 1], (tp >> 1) & 1) &&
            mbar_test(&ctrl->v_full[tp % kStagesTC], (tp / kStagesTC) & 1)) {
          tc_fence_after();
          const int sp = tp % kStagesTC;
          const uint32_t pcol = tmem + (uint32_t)(tp & 1) * kN;
          const uint32_t ocol = tmem + kColO + (uint32_t)(tp & 1) * kD;
          const uint32_t vb = sbase + kOffV + (uint32_t)sp * kKV;
          const bool first = k_of[sp] < 2;
          // tokens [16kk, 16kk+16): P_hi at packed column 32*(kk/2) + 8*(kk%2),
          // P_lo 16 columns further
#pragma unroll 1
          for (int kk = 0; kk < kN / 16; ++kk) {
            const uint64_t b = smem_desc_sw128(vb + kk * 2048u, kHalf, 1024);
            const uint32_t a = pcol + 32 * (kk >> 1) + 8 * (kk & 1);
            mma_ts(ocol, a, b, kIdescPV, !(first && kk == 0));
            mma_ts(ocol, a + 16, b, kIdescPV, 1);
          }
          mma_commit(&ctrl->o_full[tp & 1]);
          mma_commit(&ctrl->v_empty[sp]);
          ++tp;
          did = true;
        }
        // polls without sleeping once the first S is out (a sleep's wake-up
        // granularity would delay the next MMA); before it, nothing can be
        // ready for microseconds, and a spinning warp would take issue slots
        // from the producer's range lookup, so it backs off.  Bounded: a stuck
        // pipeline gives up after ~2^28 polls (~2^22 sleeps before the first S).
        if (did) {
          idle = 0;
        } else if (++idle > (ts == 0 ? (1u << 22) : (1u << 28))) {
          ctrl->abort_flag = 1;
          raise_err(p.err, SEED_DEVERR_TIMEOUT);
        } else if (ts == 0) {
          __nanosleep(128);
        }
      }
      // Wake both softmax groups through their S barriers: their next tiles,
      // t_end and t_end + 1, never get an S.  Only now: every PV has been
      // issued, so each group has consumed all of its S phases and waits (or
      // will wait) for exactly the phase these arrivals complete.
      if (!ctrl->abort_flag) {
        ctrl->end_tile = t_end;
        mbar_arrive(&ctrl->s_full[t_end & 1]);
        mbar_arrive(&ctrl->s_full[(t_end + 1) & 1]);
      }
    }
    __syncwarp();
  } else if (warp < 8 && (warp & 3) < min(4, (p.G * p.W1 + 31) / 32)) {
    // ---------------------------------------------------------- softmax
    // (warps of lane quarters that no query row of this launch reaches skip
    // the role altogether, so that they never gate the pipeline)
    // Warps 0-3 take the even tiles of the CTA, warps 4-7 the odd ones; each
    // group keeps its own running max, sum and O accumulator per row.  (The
    // producer and MMA warps sit on the SM sub-partitions of lane quarters 2
    // and 3, away from quarter 0, which holds the rows of small tiles.)
    const int par = warp >> 2;
    const int q4 = warp & 3;                  // TMEM lane quarter of this warp
    const int row = q4 * 32 + lane;           // query row = j * G + head in group
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const uint32_t ocol = tmem + lane_off + kColO + (uint32_t)par * kD;
    const uint32_t ocol_other = tmem + lane_off + kColO + (uint32_t)(par ^ 1) * kD;
    const int nqa = min(4, (p.G * p.W1 + 31) / 32);   // lane quarters in use
    const float c2 = p.scale_log2;
    float m_used = -INFINITY, l = 0.f;
    uint32_t tmask = 0u;
    int xcnt = 0;
    bool pend_rel = false;
    // (every wait below gives up once another role has aborted; the lanes
    // agree on each outcome, so the loop is left by the whole warp at once)
    for (int t = par, own = 0;; t += 2, ++own) {
      const int s = t % kStagesTC;
      // S(t) done implies K(t) landed and tile t's descriptor is written; the
      // MMA thread also completes this phase, without an S, at the end
      // (the first S comes microseconds after the dependency wait: that wait
      // sleeps between tries, so as not to take issue slots from the
      // producer's lookup on the same sub-partition)
      if (!(own == 0 ? warp_wait(&ctrl->s_full[par], 0, ctrl, p.err)
                     : warp_wait_hot(&ctrl->s_full[par], own & 1, ctrl, p.err)))
        break;
      if (t >= *reinterpret_cast<volatile int32_t*>(&ctrl->end_tile)) break;
      const TileMeta m = ctrl->meta[t % kMetaRing];
      tc_fence_after();
      const bool first_own = m.k < 2;
      const int R = m.nq * p.G;
      const int j = row / p.G;
      if (first_own) {
        m_used = -INFINITY;
        l = 0.f;
        // tree verify: this row's ancestors among the packed rows, clamped to
        // the tree's nodes, the node itself always included
        if (p.anc != nullptr && row < R) {
          const uint32_t below = m.nq >= 32 ? 0xffffffffu : ((1u << m.nq) - 1u);
          tmask = (__ldg(p.anc + (size_t)m.b * p.W1 + j) | (1u << j)) & below;
        }
      }
      const bool warp_active = q4 * 32 < R;
      ColMask cm;
      cm.dcol = (m.ncp - m.tile * kPagesPerTile) * kPage;   // first draft column
      cm.dend = cm.dcol + m.nd;
      if (p.anc == nullptr) {
        cm.lim = m.lim0 + j - m.tile * kN;                   // cache columns <= lim visible
        cm.tb = 0;
        cm.tm = 0u;
      } else {
        cm.lim = m.lim0 - 1 - m.tile * kN;                   // the committed rows
        cm.tb = m.lim0 - m.tile * kN;                        // packed row 0
        cm.tm = tmask;
      }
      bool resc = false;
      float fo = 1.f;
      const uint32_t scol = tmem + lane_off + (uint32_t)par * kN;
      if (warp_active) {
        const bool masked = __any_sync(kFull, !(cm.dcol >= kN && cm.lim >= kN - 1));
        const float mt = (masked ? row_max<true>(scol, cm) : row_max<false>(scol, cm)) * c2;
        if (mt > m_used + kRescale) {
          const float f = (m_used == -INFINITY) ? 0.f : ex2_approx(m_used - mt);
          if (!first_own && m_used != -INFINITY) {
            resc = true;
            fo = f;
          }
          l *= f;
          m_used = mt;
        }
        const float mc = (m_used == -INFINITY) ? 0.f : m_used;
        l += masked ? row_p<true>(scol, cm, c2, mc) : row_p<false>(scol, cm, c2, mc);
      }
      // V rows of columns nobody may see are zeroed, so that a probability of
      // 0 never meets a stale or NaN-poisoned row
      if (m.cvalid - m.tile * kN < kN || cm.dcol < kN) {
        // (after V has landed, or the copy engine would overwrite the zeros)
        if (!warp_wait_hot(&ctrl->v_full[s], (t / kStagesTC) & 1, ctrl, p.err)) break;
        uint8_t* vb = smem + kOffV + (size_t)s * kKV;
        bool wrote = false;
#pragma unroll 1
        for (int col = q4 * 32 + lane; col < kN; col += 32 * nqa) {
          const bool valid = (col < cm.dcol) ? (col < m.cvalid - m.tile * kN) : (col < cm.dend);
          if (valid) continue;
#pragma unroll 1
          for (int ch = 0; ch < 8; ++ch) {
            *reinterpret_cast<uint4*>(vb + col * 128 + ch * 16) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(vb + kHalf + col * 128 + ch * 16) = make_uint4(0, 0, 0, 0);
          }
          wrote = true;
        }
        if (wrote) fence_proxy_async_smem();
      }
      // this group's previous PV must be done before its O is rescaled (the
      // rescale is rare: only when the running maximum jumps by > 2^8)
      const bool do_resc = warp_active && __any_sync(kFull, resc);
      if (own > 0 && do_resc && !warp_wait_hot(&ctrl->o_full[par], (own - 1) & 1, ctrl, p.err))
        break;
      // the first tile of a unit overwrites O: the other group's epilogue of
      // the previous unit must have read it
      if (first_own && pend_rel) {
        if (!warp_wait_hot(&ctrl->orel_bar[q4], (xcnt - 1) & 1, ctrl, p.err)) break;
        pend_rel = false;
      }
      tc_fence_after();
      if (do_resc) {
        const float f = resc ? fo : 1.f;
#pragma unroll 1
        for (int c = 0; c < kD / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(ocol + c * 32, r);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * f);
          tmem_st32(ocol + c * 32, r);
        }
        tmem_wait_st();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->p_full[par]);

      if (m.k + 2 >= m.ntu) {
        // ------------------------------------------------ this group's last tile of the unit
        if (!warp_wait_hot(&ctrl->o_full[par], own & 1, ctrl, p.err)) break;
        tc_fence_after();
        if (m.k != m.ntu - 1) {
          // the other group owns the epilogue: hand over this row's statistics
          ctrl->xm[q4][lane] = m_used;
          ctrl->xl[q4][lane] = l;
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ctrl->stats_bar[q4]);
          pend_rel = true;
          ++xcnt;
        } else {
          // ---------------------------------------------- epilogue (owner)
          float mo = -INFINITY, lo = 0.f;
          if (m.ntu >= 2) {
            if (!warp_wait_hot(&ctrl->stats_bar[q4], xcnt & 1, ctrl, p.err)) break;
            tc_fence_after();
            mo = ctrl->xm[q4][lane];
            lo = ctrl->xl[q4][lane];
          }
          if (warp_active)
            unit_epilogue(p, m.b, m.g, m.nq, m.slot, row, ocol, ocol_other, m_used, l, mo, lo);
          if (m.ntu >= 2) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctrl->orel_bar[q4]);
            ++xcnt;
          }
        }
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------- host side
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

}  // namespace

// 4-d bf16 tensor map, innermost box of 64 elements (128 bytes), 128-byte
// swizzle.
bool encode_4d_bf16(CUtensorMap* map, const void* base, const cuuint64_t dims[4],
                    const cuuint64_t strides[3], const cuuint32_t box[4]) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint32_t elem[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
            elem, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {
std::atomic<uint64_t> g_tc_attr_set{0};
}  // namespace

cudaError_t launch_attn_merge(const AttnTcParams& prm, int head_dim, cudaStream_t st) {
  if (prm.nctas < 2) return cudaSuccess;        // one CTA: no pair is shared
  const dim3 mgrid(prm.nctas - 1, (prm.G * prm.W1 + kMergeRows - 1) / kMergeRows);
  return head_dim == 64
             ? launch_pdl(attn_merge_kernel<64>, mgrid, dim3(kMergeThreads), 0, st, prm)
             : launch_pdl(attn_merge_kernel<128>, mgrid, dim3(kMergeThreads), 0, st, prm);
}

bool attn_tc_supported(int head_dim, int group, int w1) {
  return head_dim == kD && group * w1 <= 128;
}

int attn_tc_ctas() { return std::min(device_sm_count(), kTcMaxCtas); }

cudaError_t launch_attn_tc(const AttnTcParams& prm, const void* q, const void* k_cache,
                           const void* v_cache, const void* draft_k, const void* draft_v,
                           cudaStream_t st) {
  CUtensorMap tq, tdk, tdv;
  PageMaps pm;
  const uint64_t W1 = (uint64_t)prm.W1;
  {
    const cuuint64_t dims[4] = {kD, (cuuint64_t)prm.hq, W1, (cuuint64_t)prm.B};
    const cuuint64_t strides[3] = {kD * 2ull, (cuuint64_t)prm.hq * kD * 2ull,
                                   W1 * prm.hq * kD * 2ull};
    const cuuint32_t box[4] = {64, (cuuint32_t)prm.G, (cuuint32_t)W1, 1};
    if (!encode_4d_bf16(&tq, q, dims, strides, box)) return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[4] = {kD, (cuuint64_t)kPage, (cuuint64_t)prm.hkv,
                                (cuuint64_t)prm.num_pages};
    const cuuint64_t strides[3] = {kD * 2ull, kPage * kD * 2ull,
                                   (cuuint64_t)prm.hkv * kPage * kD * 2ull};
    for (int i = 0; i < 4; ++i) {
      const cuuint32_t box[4] = {64, (cuuint32_t)kPage, 1, 1u << i};
      if (!encode_4d_bf16(&pm.k[i], k_cache, dims, strides, box)) return cudaErrorInvalidValue;
      if (!encode_4d_bf16(&pm.v[i], v_cache, dims, strides, box)) return cudaErrorInvalidValue;
    }
  }
  if (prm.draft) {
    // draft scratch [B, hkv, kmax, D]: one box = the 16-row draft page (rows
    // past kmax are filled with zeros by the copy engine)
    const cuuint64_t dims[4] = {kD, (cuuint64_t)prm.kmax, (cuuint64_t)prm.hkv, (cuuint64_t)prm.B};
    const cuuint64_t strides[3] = {kD * 2ull, (cuuint64_t)prm.kmax * kD * 2ull,
                                   (cuuint64_t)prm.hkv * prm.kmax * kD * 2ull};
    const cuuint32_t box[4] = {64, (cuuint32_t)kPage, 1, 1};
    if (!encode_4d_bf16(&tdk, draft_k, dims, strides, box)) return cudaErrorInvalidValue;
    if (!encode_4d_bf16(&tdv, draft_v, dims, strides, box)) return cudaErrorInvalidValue;
  } else {
    tdk = pm.k[0];
    tdv = pm.v[0];
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(g_tc_attr_set.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmemTC);
    if (e != cudaSuccess) return e;
    g_tc_attr_set.fetch_or(bit, std::memory_order_acq_rel);
  }
  e = launch_pdl(attn_tc_kernel, dim3(prm.nctas), dim3(kThreadsTC), kSmemTC, st, tq, pm, tdk, tdv,
                 prm);
  if (e != cudaSuccess) return e;
  return launch_attn_merge(prm, kD, st);
}

size_t attn_tc_plan_offset(int32_t ctas, int32_t rows, int32_t head_dim) {
  const size_t rec = 2 * (size_t)ctas * rows * (head_dim + 1) * sizeof(float);
  return (rec + 15) & ~(size_t)15;
}

size_t attn_tc_records_bytes(int32_t ctas, int32_t rows, int32_t head_dim) {
  return attn_tc_plan_offset(ctas, rows, head_dim) + (size_t)ctas * kPlanInts * sizeof(int32_t);
}

size_t attn_tc_part_bound(int32_t group, int32_t w1, int32_t head_dim) {
  return attn_tc_records_bytes(kTcMaxCtas, group * w1, head_dim);
}

}  // namespace seedk
