// Draft and verify attention for few query rows per KV head, on the
// tensor cores with the KEYS as the MMA's 128 rows (tcgen05, TMEM, TMA).
//
// What it computes is what attn_tc.cu computes (Sec. 4.1: the drafter's
// cross-attention is ordinary softmax attention over the cache; Alg. 2 fixes
// the visible rows), for sequence b and the G query heads of KV head g:
//   verify: query j < n_q[b] over cache rows 0 .. L + j (L = ctx_lens[b]);
//   draft:  one query over cache rows 0 .. L - 1, then draft rows
//           0 .. nd - 1 of the draft scratch;
//   tree verify (Sec. D.1): node j over the committed rows 0 .. L - 1 and the
//           packed rows L + a of its ancestors a (itself included).
// It serves head_dim 64 launches whose R = G * n_q query rows fit N <= 48
// MMA columns (every draft call; verify and tree verify up to R = 48): each
// K and V row is read from HBM once per call, whatever the number of query
// rows.  (head_dim 128 runs attn_tc.cu, with the query rows as MMA rows.)
//
// Design.  A tile is 128 keys (8 pages).  Per tile:
//   S^T = K Q^T      M = 128 keys, N = R rounded up to 16, K = head_dim;
//                    A = the K tile, B = Q, both K-major in shared memory.
//   softmax          one thread per key (TMEM lane): only N exponentials per
//                    thread, every lane and all four SM sub-partitions busy,
//                    whatever R is.  Each query row's reference maximum m is
//                    the exact maximum over the first tile of the piece (a
//                    block reduction, once per piece); every tile then
//                    writes P = 2^(s - m) in one pass, with no exchange
//                    between warps.  P is kept as two bf16 terms (hi = P
//                    truncated, lo = the remainder truncated: within 2^-14
//                    of P at any magnitude) stacked as rows [0, N) and
//                    [N, 2N) of one shared-memory operand, double-buffered.
//                    An exponent above 2^64 (a score that far above the
//                    first tile's maximum) is clamped and flags the piece;
//                    the epilogue warps then recompute that piece exactly
//                    from global memory, so the fast path never rescales.
//                    That recomputation is slow (CUDA cores, two passes);
//                    it advances a progress counter, and the other roles'
//                    bounded waits restart while it moves.
//   O^T += V^T P^T   M = 128 (head dims), 2N (hi and lo rows), K = 128 keys;
//                    A = the V tile read MN-major, B = the stacked P^T.
//   l^T += 1 P^T     the same B with an all-ones A operand in TMEM: every
//                    lane holds the row sums of the piece's rows.
// The epilogue adds the hi and lo columns, normalises, and writes the
// output rows (or the piece's partial record for the merge).  The S buffer
// is free once the softmax has read it, so S of later tiles never waits for
// PV; S and PV are issued by two threads, each waiting only for its own
// inputs, so copies, products and the softmax overlap across tiles.
//
// Work partition and split merge as in attn_tc.cu (attn_sched.cuh): a static
// cost-line cut of the launch's tiles into one contiguous range per CTA; a
// pair (b, g) shared by neighbouring CTAs leaves one normalised record per
// piece, merged by the merge kernel in range order.
//
// Warp roles (512 threads): warps 0-7 softmax (warp w serves TMEM lane
// quarter w & 3, lane = key, and every other 8-row chunk of the query rows,
// so two softmax warps share each SM sub-partition), warps 8-11 epilogue
// (lane quarter w - 8, lane = head dim), warp 12 K copies and the CTA's work
// walk, warp 13 V copies, warp 14 S issuer, warp 15 PV issuer and TMEM
// owner.  Every wait is bounded; one that gives up raises
// SEED_DEVERR_TIMEOUT and all roles drain out.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>

#include "attn_sched.cuh"
#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace seedk {
namespace {

using namespace sched;

constexpr int kKeys = kTileRows;               // 128 keys per tile
constexpr int kThreadsKT = 512;
constexpr int kWarpEpi = 8, kWarpProdK = 12, kWarpProdV = 13, kWarpS = 14, kWarpPV = 15;
constexpr int kMetaRing = 8;
constexpr int kMaxNQ = 48;
constexpr uint32_t kTmemCols = 512;
constexpr float kClamp = 64.0f;                // largest exponent of P (log2 units)
constexpr float kLn2 = 0.69314718055994531f;

// TMEM columns for N query rows: S^T double buffer (N each), then O^T and
// l^T (2N each: hi and lo columns), double-buffered by piece, then 8 columns
// of ones.  10 N + 8 <= 512.
__host__ __device__ constexpr uint32_t col_s(int NQ) { return 0; }
__host__ __device__ constexpr uint32_t col_o(int NQ) { return 2u * NQ; }
__host__ __device__ constexpr uint32_t col_l(int NQ) { return 6u * NQ; }
__host__ __device__ constexpr uint32_t col_ones(int NQ) { return 10u * NQ; }

template <int D>
struct Geo {
  static constexpr int kSlabs = D / 64;                       // 64-dim slabs
  static constexpr uint32_t kTile = (uint32_t)kKeys * D * 2;  // one K (or V) tile
  static constexpr int kSK = D == 128 ? 2 : 4;                // K ring slots
  static constexpr int kSV = D == 128 ? 2 : 4;                // V ring slots
};

struct KtMeta {
  int32_t unit;        // < 0: no more tiles
  int32_t b, g, tile;  // sequence, KV head, tile index within the sequence
  int32_t k, ntu;      // tile index within the piece; tiles in the piece
  int32_t nq, nd, ncp, cvalid, lim0, slot, dslot;
  int32_t pad[3];
  int32_t pids[kPagesPerTile];
};

struct KtEpi {
  int32_t b, g, nq, slot;
  int32_t tile0, ntiles;        // the piece's tiles within its sequence
  int32_t lim0, ncp, nd;        // the sequence's geometry (as in KtMeta)
  float m[kMaxNQ];     // the piece's reference maxima (log2 units)
};

struct KtCtrl {
  uint64_t k_full[4], k_empty[4], v_full[4], v_empty[4];
  uint64_t q_full[2], q_empty[2];
  uint64_t meta_full[kMetaRing], meta_empty[kMetaRing];
  uint64_t s_full[2], s_empty[2];
  uint64_t p_full[2], pv_done[2];   // P double buffer
  uint64_t o_full[2], o_free[2];
  uint64_t epi_full[2], epi_free[2];
  uint64_t sm_bar;                  // the softmax warps' exchange point
  uint32_t tmem_base;
  volatile int32_t abort_flag;
  volatile int32_t end_tile;
  // advanced by the exact recomputation of a piece: a wait that sees it move
  // restarts its bound, so only a wait without progress anywhere gives up
  volatile uint32_t progress;
  // per piece parity: u + 1 when piece u had an exponent clamped (written
  // after epi_free, read after epi_full: no reset needed)
  int32_t pflag[2];
  KtMeta meta[kMetaRing];
  KtEpi epi[2];
  alignas(16) float red[2][kMaxNQ][4];   // per lane quarter column maxima
  // negated reference maxima (log2 units) of the current piece, one copy per
  // softmax warp (each warp computes the same values)
  alignas(16) float nmrun[8][kMaxNQ];
  uint32_t desc[2][32];                  // tree verify, per piece parity: descendant masks
};

// Shared-memory layout, in bytes from the 1 KiB-aligned base.
struct KtLayout {
  uint32_t q_bytes, nqb, off_k, off_v, off_p, p_bytes, off_ctrl, total;
};

template <int D>
__host__ __device__ constexpr KtLayout kt_layout(int NQ) {
  KtLayout L{};
  L.q_bytes = (uint32_t)Geo<D>::kSlabs * NQ * 128;
  L.p_bytes = 4u * NQ * 128;     // one stacked P^T: two 64-key slabs of 2N rows (hi, then lo)
  const uint32_t rings = (uint32_t)(Geo<D>::kSK + Geo<D>::kSV) * Geo<D>::kTile;
  const uint32_t fixed = rings + 2 * L.p_bytes + (uint32_t)sizeof(KtCtrl) + 1024;
  L.nqb = fixed + 2 * L.q_bytes <= 232448u ? 2u : 1u;
  L.off_k = L.nqb * L.q_bytes;
  L.off_v = L.off_k + Geo<D>::kSK * Geo<D>::kTile;
  L.off_p = L.off_v + Geo<D>::kSV * Geo<D>::kTile;
  L.off_ctrl = L.off_p + 2 * L.p_bytes;
  L.total = L.off_ctrl + (uint32_t)sizeof(KtCtrl) + 1024;   // + alignment slack
  return L;
}

// ------------------------------------------------------------- waits
__device__ __noinline__ bool kt_wait(uint64_t* bar, uint32_t parity, KtCtrl* c, int32_t* err) {
  uint32_t seen = c->progress;
  for (uint32_t i = 0; i < kSuspendTries; ++i) {
    if (mbar_try_wait_sleep(bar, parity, kSuspendNs)) return true;
    if (c->abort_flag) return false;
    if (c->progress != seen) {
      seen = c->progress;
      i = 0;
    }
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

// A whole warp waits; the lanes agree on the outcome.
__device__ __forceinline__ bool kt_warp_wait(uint64_t* bar, uint32_t parity, KtCtrl* c,
                                             int32_t* err) {
  return __all_sync(kFull, kt_wait(bar, parity, c, err));
}

// One thread polls without sleeping (a sleep's wake-up granularity would
// delay the hot path), bounded like the others.
__device__ __noinline__ bool kt_poll1(uint64_t* bar, uint32_t parity, KtCtrl* c, int32_t* err) {
  uint32_t seen = c->progress;
  for (uint32_t i = 0; i < (1u << 26); ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if (c->abort_flag) return false;
    if ((i & 1023u) == 1023u && c->progress != seen) {
      seen = c->progress;
      i = 0;
    }
  }
  c->abort_flag = 1;
  raise_err(err, SEED_DEVERR_TIMEOUT);
  return false;
}

// A whole warp waits on a hot barrier, every lane polling (measured faster
// than lane 0 polling alone and the others taking the phase after a
// shuffle); the lanes agree on the outcome.
__device__ __forceinline__ bool kt_warp_poll(uint64_t* bar, uint32_t parity, KtCtrl* c,
                                             int32_t* err) {
  return __all_sync(kFull, kt_poll1(bar, parity, c, err));
}

// Exchange point of the eight softmax warps (an mbarrier counting one
// arrival per warp, so that the wait is bounded and an abort cannot strand a
// warp).  ns counts the exchanges so far; it is the same in every softmax
// thread.
__device__ __forceinline__ bool softmax_sync(KtCtrl* c, uint32_t& ns, int lane, int32_t* err) {
  __syncwarp();
  if (lane == 0) mbar_arrive(&c->sm_bar);
  const bool ok = kt_warp_poll(&c->sm_bar, ns & 1u, c, err);
  ++ns;
  return ok;
}

// Order-preserving map of a float onto uint32 (for redux.sync max).
__device__ __forceinline__ uint32_t f2ord(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord2f(uint32_t u) {
  return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}

// One column of a block reduction over the 128 keys: this warp's maximum of
// e over the 32 keys of lane quarter q4.  After the softmax warps' next
// exchange, red_max(c, buf, q) is the largest e[q] over all keys (-inf when
// no key is visible to query row q).
__device__ __forceinline__ void warp_col_max(float e, KtCtrl* c, int buf, int q, int q4,
                                             int lane) {
  const uint32_t u = __reduce_max_sync(kFull, f2ord(e));
  if (lane == (q & 31)) c->red[buf][q][q4] = ord2f(u);
}

__device__ __forceinline__ float red_max(const KtCtrl* c, int buf, int q) {
  const float4 w = *reinterpret_cast<const float4*>(&c->red[buf][q][0]);
  return fmaxf(fmaxf(w.x, w.y), fmaxf(w.z, w.w));
}

// Visibility of the softmax rows for this thread's key, as a bit mask over
// rows q < 64: rows [qmin, R) see the key, and, for a tree verify, the rows
// q < R of the nodes in tdesc (node j owns rows [jG, jG + G)).
__device__ __forceinline__ uint64_t row_mask(int R, int qmin, uint32_t tdesc, int G) {
  const uint64_t below = R >= 64 ? ~0ull : ((1ull << R) - 1ull);
  const uint64_t from = qmin >= 64 ? 0ull : (~0ull << qmin);
  uint64_t m = below & from;
  if (tdesc) {
    const uint64_t grp = G >= 64 ? ~0ull : ((1ull << G) - 1ull);
    for (uint32_t t = tdesc; t; t &= t - 1) m |= (grp << ((__ffs(t) - 1) * G)) & below;
  }
  return m;
}

// 8 consecutive floats of a shared-memory row (16-byte aligned).
__device__ __forceinline__ void lds8(const float* src, float (&v)[8]) {
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float4 x = reinterpret_cast<const float4*>(src)[i];
    v[4 * i] = x.x;
    v[4 * i + 1] = x.y;
    v[4 * i + 2] = x.z;
    v[4 * i + 3] = x.w;
  }
}

// After an abort: wait (bounded, whatever the abort flag says) until the
// newest copy issued into each ring slot has landed, so that no copy writes
// this CTA's shared memory after it exits.  n = copies issued in order.
__device__ __noinline__ void drain_copies(uint64_t* full, int slots, int n) {
  for (int s = 0; s < slots && s < n; ++s) {
    const int last = s + (n - 1 - s) / slots * slots;   // newest tile in slot s
    for (uint32_t i = 0; i < (1u << 20); ++i)
      if (mbar_try_wait(&full[s], (last / slots) & 1)) break;
  }
}

// Exact attention of one piece -- tiles [tile0, tile0 + ntiles) of pair
// (b, g) -- for a piece whose exponents the fast path had to clamp: two
// passes over the piece's visible rows, straight from global memory
// (maximum, then sum and weighted values), one warp per query row (rows
// q4, q4 + 4, ...), D / 32 head dims per lane.  Writes what the epilogue
// writes: the output rows of a whole pair, or the piece's record.  Slow, and
// reached only by scores more than 2^64 above the first tile's maximum.
template <int D>
__device__ __noinline__ void exact_piece(const AttnTcParams& p, const KtEpi& ep, int q4, int lane,
                                         KtCtrl* ctrl) {
  constexpr int kPer = D / 32;
  const int G = p.G, Rmax = G * p.W1, R = ep.nq * G;
  const int b = ep.b, g = ep.g;
  const int k0 = ep.tile0 * kKeys, k1 = (ep.tile0 + ep.ntiles) * kKeys;
  const int dcol = ep.ncp * kPage;
  float* rec = p.part + (size_t)max(ep.slot, 0) * Rmax * (D + 1);
  for (int r = q4; r < R; r += 4) {
    const int j = r / G;
    const int head = g * G + (r - j * G);
    const size_t orow = ((size_t)b * p.W1 + j) * p.hq + head;
    float qv[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const uint16_t bits = p.q[orow * D + lane * kPer + e];
      qv[e] = __uint_as_float((uint32_t)bits << 16);
    }
    uint32_t tm = 0;   // tree: packed rows this node sees
    if (p.anc != nullptr) {
      const uint32_t below = ep.nq >= 32 ? 0xffffffffu : ((1u << ep.nq) - 1u);
      tm = (__ldg(p.anc + (size_t)b * p.W1 + j) | (1u << j)) & below;
    }
    float m = -INFINITY, l = 0.f, o[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) o[e] = 0.f;
    for (int pass = 0; pass < 2; ++pass) {
      for (int kpos = k0; kpos < k1; ++kpos) {
        if (lane == 0 && (kpos & 63) == 0) ctrl->progress = ctrl->progress + 1;
        bool vis;
        if (p.anc != nullptr) {
          const int a = kpos - ep.lim0;
          vis = a < 0 || (a < ep.nq && ((tm >> a) & 1u));
        } else if (p.draft) {
          vis = kpos <= ep.lim0 || (kpos >= dcol && kpos < dcol + ep.nd);
        } else {
          vis = kpos <= ep.lim0 + j;
        }
        if (!vis) continue;
        size_t row;
        const uint16_t *kb, *vb;
        if (p.draft && kpos >= dcol) {
          row = ((size_t)b * p.hkv + g) * p.kmax + (kpos - dcol);
          kb = p.draft_k;
          vb = p.draft_v;
        } else {
          const int pid = __ldg(p.page_table + (size_t)b * p.max_pages + kpos / kPage);
          if (pid < 0 || pid >= p.num_pages) continue;   // raised by the fast path
          row = ((size_t)pid * p.hkv + g) * kPage + (kpos % kPage);
          kb = p.k_cache;
          vb = p.v_cache;
        }
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < kPer; ++e)
          s = fmaf(qv[e], __uint_as_float((uint32_t)kb[row * D + lane * kPer + e] << 16), s);
#pragma unroll
        for (int w = 16; w; w >>= 1) s += __shfl_xor_sync(kFull, s, w);
        s *= p.scale_log2;
        if (pass == 0) {
          m = fmaxf(m, s);
        } else {
          const float w = ex2_approx(s - m);
          l += w;
#pragma unroll
          for (int e = 0; e < kPer; ++e)
            o[e] = fmaf(w, __uint_as_float((uint32_t)vb[row * D + lane * kPer + e] << 16), o[e]);
        }
      }
    }
    const float inv = l > 0.f ? 1.f / l : 0.f;
    const float lse2 = l > 0.f ? m + log2f(l) : -INFINITY;
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      if (ep.slot < 0)
        p.out[orow * D + lane * kPer + e] = o[e] * inv;
      else
        rec[(size_t)r * D + lane * kPer + e] = o[e] * inv;
    }
    if (lane == 0) {
      if (ep.slot >= 0)
        rec[(size_t)D * Rmax + r] = lse2;
      else if (p.lse != nullptr)
        p.lse[orow] = lse2 * kLn2;
    }
  }
}

// ------------------------------------------------------------- the kernel
template <int D, int NQ>
__global__ void __launch_bounds__(kThreadsKT, 1)
    attn_kt_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ PageMaps pm,
                   const __grid_constant__ CUtensorMap tm_dk,
                   const __grid_constant__ CUtensorMap tm_dv, const AttnTcParams p) {
  using GE = Geo<D>;
  constexpr KtLayout LY = kt_layout<D>(NQ);
  constexpr uint32_t kColS = col_s(NQ), kColO = col_o(NQ), kColL = col_l(NQ),
                     kColOnes = col_ones(NQ);
  static_assert(col_ones(NQ) + 8 <= kTmemCols, "tensor memory budget");
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  KtCtrl* ctrl = reinterpret_cast<KtCtrl*>(smem + LY.off_ctrl);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  if (tid == 0) pdl_trigger();

  if (tid == 0) {
    for (int s = 0; s < 4; ++s) {
      mbar_init(&ctrl->k_full[s], 1);
      mbar_init(&ctrl->k_empty[s], 1);
      mbar_init(&ctrl->v_full[s], 1);
      mbar_init(&ctrl->v_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ctrl->q_full[i], 1);
      mbar_init(&ctrl->q_empty[i], 1);
      mbar_init(&ctrl->s_full[i], 1);
      mbar_init(&ctrl->s_empty[i], 8);
      mbar_init(&ctrl->p_full[i], 8);
      mbar_init(&ctrl->pv_done[i], 1);
      mbar_init(&ctrl->o_full[i], 1);
      mbar_init(&ctrl->o_free[i], 4);
      mbar_init(&ctrl->epi_full[i], 8);
      mbar_init(&ctrl->epi_free[i], 4);
      ctrl->pflag[i] = 0;
    }
    for (int i = 0; i < kMetaRing; ++i) {
      mbar_init(&ctrl->meta_full[i], 1);
      mbar_init(&ctrl->meta_empty[i], 2);   // V copies and PV issuer
    }
    mbar_init(&ctrl->sm_bar, 8);
    ctrl->abort_flag = 0;
    ctrl->progress = 0;
    ctrl->end_tile = 1 << 30;
    fence_mbar_init();
  }
  if (warp == kWarpPV) {
    tmem_alloc(&ctrl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kWarpProdK && lane == 0) {
    // descriptors are kernel parameters: prefetch before the dependency wait
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
  if (warp == kWarpProdK) prefetch_lens_l2(p, lane);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctrl->tmem_base;
  if (warp < 4) {
    // the all-ones A operand of the row-sum product (8 columns of bf16 pairs)
    uint32_t ones[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) ones[i] = 0x3F803F80u;
    tmem_st8(tmem + ((uint32_t)(warp * 32) << 16) + kColOnes, ones);
    tmem_wait_st();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const int G = p.G;
  const int Rmax = G * p.W1;
  const int nqb = (int)LY.nqb;
  // everything above touched only this CTA's shared and tensor memory
  pdl_wait();

  if (warp == kWarpProdK) {
    // ------------------------------------------------------------ K copies
    if (blockIdx.x == 0) {
      for (int b = lane; b < p.B; b += 32) {
        const int bad = seq_of(p, b).bad;
        if (bad) raise_err(p.err, bad);
      }
    }
    long long T, x, x1;
    SeqWin win;
    int b = p.B, g = 0, t0 = 0;
    long long pc = 0;
    lookup_range(p, lane, T, x, x1, win, b, g, t0, pc);
    {
      const SeqT s0 = b < p.B ? win_get(win, b) : SeqT{};
      if (lane == 0) write_merge_plan(p, T, x, x1, b, g, t0, pc, s0);
    }
    int tk = 0, uo = 0;
    const uint64_t kv_pol = policy_evict_first();   // K is read once per call
    bool ok = true;
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
      sq = win_get(win, b);
      t1 = (int)min((long long)sq.tiles, x1 - pc - kPairCost);
      if (t1 <= t0) break;
      const int slot = (t0 == 0 && t1 == sq.tiles) ? -1 : 2 * (int)blockIdx.x + (uo > 0 ? 1 : 0);
      pid_a = load_pid(t0);
      pid_b = load_pid(t0 + 1);
      for (int t = t0; t < t1; ++t, ++tk) {
        const int s = tk % GE::kSK, mi = tk % kMetaRing;
        int pid = pid_a;
        pid_a = pid_b;
        pid_b = load_pid(t + 2);
        if (tk >= GE::kSK)
          ok = kt_warp_wait(&ctrl->k_empty[s], ((tk / GE::kSK) - 1) & 1, ctrl, p.err);
        if (ok && tk >= kMetaRing)
          ok = kt_warp_wait(&ctrl->meta_empty[mi], ((tk / kMetaRing) - 1) & 1, ctrl, p.err);
        if (ok && t == t0 && uo >= nqb)
          ok = kt_warp_wait(&ctrl->q_empty[uo % nqb], ((uo / nqb) - 1) & 1, ctrl, p.err);
        if (!ok) break;
        if (lane < kPagesPerTile && t * kPagesPerTile + lane < sq.ncp &&
            (pid < 0 || pid >= p.num_pages)) {
          raise_err(p.err, SEED_DEVERR_PAGE);
          pid = -1;
        }
        // slot of draft page 0 (may lie outside the tile); lane pp holds
        // draft page dpage when the tile's slot pp is one
        const int dslot = sq.ncp - t * kPagesPerTile;
        const int dpage = lane < kPagesPerTile ? draft_page_of_slot(sq.ncp, sq.nd, t, lane) : -1;
        const bool has = lane < kPagesPerTile && (pid >= 0 || dpage >= 0);
        const uint32_t loads = __ballot_sync(kFull, has);
        const int box = box_size(pid, lane);
        KtMeta& m = ctrl->meta[mi];
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
            uint8_t* qd = smem + (size_t)qb * LY.q_bytes;
            mbar_arrive_expect_tx(&ctrl->q_full[qb], (uint32_t)GE::kSlabs * 128u * Rmax);
#pragma unroll
            for (int h = 0; h < GE::kSlabs; ++h)
              tma_load_4d(qd + h * (NQ * 128), &tm_q, 64 * h, g * G, 0, b, &ctrl->q_full[qb]);
          }
          mbar_arrive_expect_tx(&ctrl->k_full[s], (uint32_t)__popc(loads) * GE::kSlabs * 2048u);
        }
        __syncwarp();
        if (box > 0 || (has && pid < 0)) {
          uint8_t* kb = smem + LY.off_k + (size_t)s * GE::kTile + lane * 2048u;
          const CUtensorMap* mk = box > 0 ? &pm.k[log2_box(box)] : &tm_dk;
          const int w = box > 0 ? pid : b, r0 = box > 0 ? 0 : kPage * dpage;
#pragma unroll
          for (int h = 0; h < GE::kSlabs; ++h)
            tma_load_4d_hint(kb + h * (kKeys * 128), mk, 64 * h, r0, g, w, &ctrl->k_full[s],
                             kv_pol);
        }
      }
      if (!ok) break;
      ++uo;
      if (t1 < sq.tiles) break;
      pc += sq.tiles + kPairCost;
      t0 = 0;
      if (++g == p.hkv) {
        g = 0;
        next_seq(p, lane, win, b);
      }
    }
    // end marker for the S issuer and the V warp
    if (ok) {
      const int s = tk % GE::kSK, mi = tk % kMetaRing;
      if (tk >= GE::kSK)
        ok = kt_warp_wait(&ctrl->k_empty[s], ((tk / GE::kSK) - 1) & 1, ctrl, p.err);
      if (ok && tk >= kMetaRing)
        ok = kt_warp_wait(&ctrl->meta_empty[mi], ((tk / kMetaRing) - 1) & 1, ctrl, p.err);
      if (ok && lane == 0) {
        ctrl->meta[mi].unit = -1;
        mbar_arrive(&ctrl->meta_full[mi]);
        mbar_arrive(&ctrl->k_full[s]);
      }
    }
    __syncwarp();
    if (ctrl->abort_flag && lane == 0) drain_copies(ctrl->k_full, GE::kSK, tk);
    __syncwarp();
  } else if (warp == kWarpProdV) {
    // ------------------------------------------------------------ V copies
    int tv = 0;
    const uint64_t kv_pol = policy_evict_first();   // V is read once per call
    for (;; ++tv) {
      const int s = tv % GE::kSV, mi = tv % kMetaRing;
      if (!kt_warp_wait(&ctrl->meta_full[mi], (tv / kMetaRing) & 1, ctrl, p.err)) break;
      const KtMeta& m = ctrl->meta[mi];
      if (m.unit < 0) break;
      const int pid = lane < kPagesPerTile ? m.pids[lane] : -1;
      const int mb = m.b, mg = m.g, dslot = m.dslot, nd = m.nd;
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->meta_empty[mi]);
      if (tv >= GE::kSV &&
          !kt_warp_wait(&ctrl->v_empty[s], ((tv / GE::kSV) - 1) & 1, ctrl, p.err))
        break;
      const int dpage =
          (lane < kPagesPerTile && lane >= dslot && lane - dslot < draft_pages(nd)) ? lane - dslot
                                                                                     : -1;
      const bool has = lane < kPagesPerTile && (pid >= 0 || dpage >= 0);
      const uint32_t loads = __ballot_sync(kFull, has);
      if (lane == 0)
        mbar_arrive_expect_tx(&ctrl->v_full[s], (uint32_t)__popc(loads) * GE::kSlabs * 2048u);
      __syncwarp();
      const int box = box_size(pid, lane);
      if (box > 0 || (has && pid < 0)) {
        uint8_t* vb = smem + LY.off_v + (size_t)s * GE::kTile + lane * 2048u;
        const CUtensorMap* mv = box > 0 ? &pm.v[log2_box(box)] : &tm_dv;
        const int w = box > 0 ? pid : mb, r0 = box > 0 ? 0 : kPage * dpage;
#pragma unroll
        for (int h = 0; h < GE::kSlabs; ++h)
          tma_load_4d_hint(vb + h * (kKeys * 128), mv, 64 * h, r0, mg, w, &ctrl->v_full[s],
                           kv_pol);
      }
    }
    __syncwarp();
    if (ctrl->abort_flag && lane == 0) drain_copies(ctrl->v_full, GE::kSV, tv);
    __syncwarp();
  } else if (warp == kWarpS) {
    // ------------------------------------------------------------ S issuer
    // S^T(t) = K(t) Q^T as soon as K(t) has landed and the softmax has read
    // S(t - 2) out of the same TMEM columns
    if (lane == 0) {
      constexpr uint32_t kIdescS = idesc_bf16_f32(128, NQ, 0, 0);   // K, Q both K-major
      int uq = 0, qcur = 0;
      for (int ts = 0;; ++ts) {
        const int s = ts % GE::kSK;
        if (!kt_poll1(&ctrl->k_full[s], (ts / GE::kSK) & 1, ctrl, p.err)) break;
        // S(ts - 2) has been read (also before the end marker: an s_full
        // phase must never complete twice ahead of the softmax's wait)
        if (ts >= 2 && !kt_poll1(&ctrl->s_empty[ts & 1], ((ts >> 1) - 1) & 1, ctrl, p.err)) break;
        const KtMeta& mt = ctrl->meta[ts % kMetaRing];
        if (mt.unit < 0) {
          // no more tiles: wake the softmax warps, whose next tile never gets an S
          ctrl->end_tile = ts;
          mbar_arrive(&ctrl->s_full[ts & 1]);
          break;
        }
        const int k = mt.k, ntu = mt.ntu;
        if (k == 0) {
          if (!kt_poll1(&ctrl->q_full[uq % nqb], (uq / nqb) & 1, ctrl, p.err)) break;
          qcur = uq % nqb;
          ++uq;
        }
        tc_fence_after();
        // descriptors of operand slices differ from their base by the
        // slice's byte offset / 16 (addresses stay below 2^18)
        const uint64_t kdesc = smem_desc_sw128(sbase + LY.off_k + (uint32_t)s * GE::kTile, 16, 1024);
        const uint64_t qdesc = smem_desc_sw128(sbase + (uint32_t)qcur * LY.q_bytes, 16, 1024);
        const uint32_t d = tmem + kColS + (uint32_t)(ts & 1) * NQ;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t h = kk >> 2, off = (kk & 3) * 32;
          mma_ss(d, kdesc + (uint64_t)((h * (kKeys * 128) + off) >> 4),
                 qdesc + (uint64_t)((h * (NQ * 128) + off) >> 4), kIdescS, kk > 0);
        }
        mma_commit(&ctrl->s_full[ts & 1]);
        mma_commit(&ctrl->k_empty[s]);
        if (k == ntu - 1) mma_commit(&ctrl->q_empty[qcur]);
      }
    }
    __syncwarp();
  } else if (warp == kWarpPV) {
    // ------------------------------------------------------------ PV issuer
    // O^T += V^T P^T and l^T += 1 P^T for tile t as soon as P(t) is written
    // and V(t) has landed
    if (lane == 0) {
      constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 2 * NQ, 1, 0);  // V^T MN-major, P^T K-major
      constexpr uint32_t kIdescL = idesc_bf16_f32(128, 2 * NQ, 0, 0);   // ones (TMEM), P^T
      constexpr uint32_t kVLbo = D == 128 ? (uint32_t)kKeys * 128 : 0u;
      int u = -1;
      for (int tp = 0;; ++tp) {
        // P(tp) written, or the end of the CTA's tiles
        bool got = false;
        uint32_t seen = ctrl->progress;
        for (uint32_t i = 0; i < (1u << 26) && !got; ++i) {
          if (mbar_try_wait(&ctrl->p_full[tp & 1], (tp >> 1) & 1)) got = true;
          else if (tp >= ctrl->end_tile || ctrl->abort_flag) break;
          else if ((i & 1023u) == 1023u && ctrl->progress != seen) {
            seen = ctrl->progress;
            i = 0;
          }
        }
        if (!got) {
          if (tp < ctrl->end_tile && !ctrl->abort_flag) {
            ctrl->abort_flag = 1;
            raise_err(p.err, SEED_DEVERR_TIMEOUT);
          }
          break;
        }
        const int mi = tp % kMetaRing;
        const KtMeta& mt = ctrl->meta[mi];
        const bool first = mt.k == 0, last = mt.k == mt.ntu - 1;
        mbar_arrive(&ctrl->meta_empty[mi]);
        if (first) ++u;
        const int sv = tp % GE::kSV;
        if (!kt_poll1(&ctrl->v_full[sv], (tp / GE::kSV) & 1, ctrl, p.err)) break;
        // the first product of a piece overwrites O and l of piece u - 2: its
        // epilogue must have read them
        if (first && u >= 2 && !kt_poll1(&ctrl->o_free[u & 1], ((u >> 1) - 1) & 1, ctrl, p.err))
          break;
        tc_fence_after();
        const uint64_t vdesc =
            smem_desc_sw128(sbase + LY.off_v + (uint32_t)sv * GE::kTile, kVLbo, 1024);
        const uint64_t pdesc =
            smem_desc_sw128(sbase + LY.off_p + (uint32_t)(tp & 1) * LY.p_bytes, 16, 1024);
        const uint32_t ocol = tmem + kColO + (uint32_t)(u & 1) * (2 * NQ);
        const uint32_t lcol = tmem + kColL + (uint32_t)(u & 1) * (2 * NQ);
#pragma unroll
        for (int kk = 0; kk < kKeys / 16; ++kk) {
          const uint64_t bp = pdesc + (uint64_t)(((kk >> 2) * (2 * NQ * 128) + (kk & 3) * 32) >> 4);
          mma_ss(ocol, vdesc + (uint64_t)((kk * 2048u) >> 4), bp, kIdescPV, !(first && kk == 0));
          mma_ts(lcol, tmem + kColOnes, bp, kIdescL, !(first && kk == 0));
        }
        mma_commit(&ctrl->pv_done[tp & 1]);
        mma_commit(&ctrl->v_empty[sv]);
        if (last) mma_commit(&ctrl->o_full[u & 1]);
      }
    }
    __syncwarp();
  } else if (warp < 8) {
    // ------------------------------------------------------------ softmax
    // Warp w serves TMEM lane quarter w & 3 (keys 32 (w & 3) .. + 31, one per
    // lane) and the 8-row chunks c = h, h + 2, ... of the query rows (h = w >> 2),
    // so that each SM sub-partition runs two softmax warps.
    const int q4 = warp & 3, h = warp >> 2;
    const int key = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const float c2 = p.scale_log2;
    // this key's byte address inside row 0 of the stacked P^T operand (two
    // 64-key slabs of 2N rows of 128 bytes, 128-byte swizzle)
    const int kin = key & 63;
    uint8_t* pkey0 = smem + LY.off_p + (key >> 6) * (2 * NQ * 128) + (kin & 7) * 2;
    const int kchunk = kin >> 3;
    float* nmw = ctrl->nmrun[warp];   // this warp's copy of the negated reference maxima
    int u = -1;
    uint32_t ns = 0;   // softmax exchanges so far
    bool pclamp = false;   // this lane clamped an exponent in the current piece
    for (int t = 0;; ++t) {
      if (!kt_warp_poll(&ctrl->s_full[t & 1], (t >> 1) & 1, ctrl, p.err)) break;
      if (t >= ctrl->end_tile) {
        // no more tiles: tell the epilogue (all eight warps arrive)
        const int uu = u + 1;
        if (uu >= 2 && !kt_warp_wait(&ctrl->epi_free[uu & 1], ((uu >> 1) - 1) & 1, ctrl, p.err))
          break;
        if (warp == 0 && lane == 0) ctrl->epi[uu & 1].b = -1;
        __syncwarp();
        if (lane == 0) mbar_arrive(&ctrl->epi_full[uu & 1]);
        break;
      }
      KtMeta mt;
      {
        const KtMeta& ms = ctrl->meta[t % kMetaRing];
        mt.b = ms.b;
        mt.g = ms.g;
        mt.tile = ms.tile;
        mt.k = ms.k;
        mt.ntu = ms.ntu;
        mt.nq = ms.nq;
        mt.nd = ms.nd;
        mt.ncp = ms.ncp;
        mt.cvalid = ms.cvalid;
        mt.lim0 = ms.lim0;
        mt.slot = ms.slot;
      }
      tc_fence_after();
      const bool first = mt.k == 0;
      if (first) ++u;
      const int R = mt.nq * G;
      const int kpos = mt.tile * kKeys + key;
      const int rb = u & 1;   // first-tile maxima: one buffer per piece parity
      const uint32_t scol = tmem + lane_off + kColS + (uint32_t)(t & 1) * NQ;
      // tree verify: at the piece's first tile, the descendant mask of each
      // packed row a < nq (bit j: node j has a as an ancestor, or is a)
      if (p.anc != nullptr && first) {
        if (warp == 0) {
          uint32_t dm = 0;
          if (lane < mt.nq) {
            const uint32_t below = mt.nq >= 32 ? 0xffffffffu : ((1u << mt.nq) - 1u);
            for (int j = 0; j < mt.nq; ++j) {
              const uint32_t an = (__ldg(p.anc + (size_t)mt.b * p.W1 + j) | (1u << j)) & below;
              dm |= ((an >> lane) & 1u) << j;
            }
          }
          ctrl->desc[u & 1][lane] = dm;
        }
        if (!softmax_sync(ctrl, ns, lane, p.err)) break;
      }
      // visibility of (this key, query row q)
      const int dcol = mt.ncp * kPage;                 // first draft row position (draft)
      const bool in_draft = mt.nd > 0 && kpos >= dcol && kpos < dcol + mt.nd;
      uint32_t tdesc = 0;
      int qmin;
      if (p.anc != nullptr) {
        const int a = kpos - mt.lim0;
        if (a >= 0 && a < mt.nq) tdesc = ctrl->desc[u & 1][a];
        qmin = a < 0 ? 0 : 64;
      } else if (p.draft) {
        qmin = (kpos <= mt.lim0 || in_draft) ? 0 : 64;
      } else {
        const int dl = kpos - mt.lim0;
        qmin = dl <= 0 ? 0 : min(dl * G, 64);
      }
      const uint64_t vis = row_mask(R, qmin, tdesc, G);
      const int nch = (R + 7) >> 3;                // 8-row chunks holding rows < R
      if (first) {
        // the piece's reference maxima: the exact maxima over this tile
        // (rows that see no key here keep m = 0)
#pragma unroll 1
        for (int c = h; c < NQ / 8; c += 2) {
          if (c < nch) {
            uint32_t x[8];
            tmem_ld8(scol + 8 * c, x);
            tmem_wait_ld();
            const uint32_t vb = (uint32_t)(vis >> (8 * c));
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float ev = ((vb >> i) & 1u) ? __uint_as_float(x[i]) * c2 : -INFINITY;
              warp_col_max(ev, ctrl, rb, 8 * c + i, q4, lane);
            }
          } else if (lane < 8) {
            ctrl->red[rb][8 * c + lane][q4] = -INFINITY;   // rows past R
          }
        }
        if (!softmax_sync(ctrl, ns, lane, p.err)) break;
        for (int q = lane; q < NQ; q += 32) {
          const float mx = red_max(ctrl, rb, q);
          nmw[q] = mx == -INFINITY ? 0.f : -mx;
        }
        __syncwarp();
      }
      // P buffer t & 1 is free once PV(t - 2) is done
      if (t >= 2 && !kt_warp_poll(&ctrl->pv_done[t & 1], ((t >> 1) - 1) & 1, ctrl, p.err)) break;
      // one pass: P = 2^(s c - m), hi = P truncated to bf16, lo = the
      // remainder truncated, into rows q and N + q of the stacked operand.
      // (Rows from R to the chunk's end are padding: their P is written,
      // never used.)
      uint8_t* pbase = pkey0 + (t & 1) * LY.p_bytes;
#pragma unroll 1
      for (int c = h; c < nch; c += 2) {
        uint32_t x[8];
        tmem_ld8(scol + 8 * c, x);
        float nm[8];
        lds8(nmw + 8 * c, nm);
        tmem_wait_ld();
        const uint32_t vb = (uint32_t)(vis >> (8 * c)) & 0xffu;
        // the common chunk: every row visible to every key of the warp
        const bool full = __all_sync(kFull, vb == 0xffu);
        uint8_t* prow = pbase + (8 * c) * 128;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float a = fmaf(__uint_as_float(x[i]), c2, nm[i]);
          if (!full) a = ((vb >> i) & 1u) ? a : -INFINITY;
          pclamp |= a > kClamp;
          const float pv = ex2_approx(fminf(a, kClamp));
          const uint32_t hb = __float_as_uint(pv) & 0xffff0000u;
          const uint32_t lb = __float_as_uint(pv - __uint_as_float(hb));
          // row 8c + i of the operand: its 16-byte chunks are swizzled by i
          uint8_t* a16 = prow + i * 128 + ((kchunk ^ i) << 4);
          *reinterpret_cast<uint16_t*>(a16) = (uint16_t)(hb >> 16);
          *reinterpret_cast<uint16_t*>(a16 + NQ * 128) = (uint16_t)(lb >> 16);
        }
      }
      // S(t) has been read: its TMEM columns may take S(t + 2)
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->s_empty[t & 1]);
      // V rows of keys nobody may see (past the sequence end, unfilled page
      // slots, draft rows past nd) are zeroed, so that a probability of 0
      // never meets a stale or NaN-poisoned row (one warp per lane quarter)
      const int tbase = mt.tile * kKeys;
      if (h == 0 && (mt.cvalid - tbase < kKeys || dcol - tbase < kKeys)) {
        const bool valid = kpos < dcol ? kpos < mt.cvalid : in_draft;
        // (after V has landed, or the copy engine would overwrite the zeros)
        if (!kt_warp_wait(&ctrl->v_full[t % GE::kSV], (t / GE::kSV) & 1, ctrl, p.err)) break;
        if (!valid) {
          uint8_t* vr = smem + LY.off_v + (size_t)(t % GE::kSV) * GE::kTile + key * 128;
#pragma unroll
          for (int hh = 0; hh < GE::kSlabs; ++hh)
#pragma unroll
            for (int ch = 0; ch < 8; ++ch)
              *reinterpret_cast<uint4*>(vr + hh * (kKeys * 128) + ch * 16) = make_uint4(0, 0, 0, 0);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->p_full[t & 1]);
      if (mt.k == mt.ntu - 1) {
        // the piece ends here: hand its description to the epilogue
        if (u >= 2 && !kt_warp_wait(&ctrl->epi_free[u & 1], ((u >> 1) - 1) & 1, ctrl, p.err))
          break;
        if (__any_sync(kFull, pclamp) && lane == 0) ctrl->pflag[u & 1] = u + 1;
        pclamp = false;
        if (warp == 0) {
          KtEpi& ep = ctrl->epi[u & 1];
          for (int q = lane; q < NQ; q += 32) ep.m[q] = -nmw[q];
          if (lane == 0) {
            ep.b = mt.b;
            ep.g = mt.g;
            ep.nq = mt.nq;
            ep.slot = mt.slot;
            ep.tile0 = mt.tile - mt.k;
            ep.ntiles = mt.ntu;
            ep.lim0 = mt.lim0;
            ep.ncp = mt.ncp;
            ep.nd = mt.nd;
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&ctrl->epi_full[u & 1]);
      }
    }
  } else if (warp < kWarpEpi + 4) {
    // ------------------------------------------------------------ epilogue
    const int q4 = warp - kWarpEpi;
    const int d = q4 * 32 + lane;                  // head dim of this lane
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const bool has_d = d < D;
    const int lg = 31 - __clz(G);
    for (int u = 0;; ++u) {
      if (!kt_warp_wait(&ctrl->epi_full[u & 1], (u >> 1) & 1, ctrl, p.err)) break;
      const KtEpi& ep = ctrl->epi[u & 1];
      const int b = ep.b, g = ep.g, nq = ep.nq, slot = ep.slot;
      if (b < 0) break;
      if (!kt_warp_wait(&ctrl->o_full[u & 1], (u >> 1) & 1, ctrl, p.err)) break;
      tc_fence_after();
      const int R = nq * G;
      float* rec = p.part + (size_t)max(slot, 0) * Rmax * (D + 1);
      if (ctrl->pflag[u & 1] == u + 1) {
        // an exponent was clamped: this piece is recomputed exactly
        exact_piece<D>(p, ep, q4, lane, ctrl);
      } else {
      const uint32_t oc = tmem + lane_off + kColO + (uint32_t)(u & 1) * (2 * NQ);
      const uint32_t lc = tmem + lane_off + kColL + (uint32_t)(u & 1) * (2 * NQ);
#pragma unroll 1
      for (int c = 0; c < NQ / 8; ++c) {
        if (8 * c >= R) break;
        uint32_t oh[8], ol[8], lh[8], ll[8];
        tmem_ld8(oc + 8 * c, oh);
        tmem_ld8(oc + NQ + 8 * c, ol);
        tmem_ld8(lc + 8 * c, lh);
        tmem_ld8(lc + NQ + 8 * c, ll);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int q = 8 * c + i;
          if (q < R) {
            const float lq = __uint_as_float(lh[i]) + __uint_as_float(ll[i]);
            const float o = __uint_as_float(oh[i]) + __uint_as_float(ol[i]);
            const float val = lq > 0.f ? o / lq : 0.f;
            const int j = q >> lg;
            const size_t orow = ((size_t)b * p.W1 + j) * p.hq + g * G + (q - j * G);
            if (has_d) {
              if (slot < 0)
                p.out[orow * D + d] = val;
              else
                rec[(size_t)q * D + d] = val;
            }
            if (d == 0) {
              const float lse2 = lq > 0.f ? ep.m[q] + log2f(lq) : -INFINITY;
              if (slot >= 0)
                rec[(size_t)D * Rmax + q] = lse2;
              else if (p.lse != nullptr)
                p.lse[orow] = lse2 * kLn2;
            }
          }
        }
      }
      }
      // every read of this piece is done: O and l may take piece u + 2
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&ctrl->o_free[u & 1]);
        mbar_arrive(&ctrl->epi_free[u & 1]);
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpPV) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int D, int NQ>
cudaError_t launch_kt(const AttnTcParams& prm, const CUtensorMap& tq, const PageMaps& pm,
                      const CUtensorMap& tdk, const CUtensorMap& tdv, cudaStream_t st) {
  static std::atomic<uint64_t> attr_set{0};
  constexpr KtLayout LY = kt_layout<D>(NQ);
  static_assert(LY.total <= 232448u, "shared memory budget");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_set.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(attn_kt_kernel<D, NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)LY.total);
    if (e != cudaSuccess) return e;
    attr_set.fetch_or(bit, std::memory_order_acq_rel);
  }
  return launch_pdl(attn_kt_kernel<D, NQ>, dim3(prm.nctas), dim3(kThreadsKT), (size_t)LY.total,
                    st, tq, pm, tdk, tdv, prm);
}

}  // namespace

bool attn_kt_supported(int head_dim, int group, int w1) {
  return head_dim == 64 && group * w1 <= kMaxNQ;
}

cudaError_t launch_attn_kt(const AttnTcParams& prm, int head_dim, const void* q,
                           const void* k_cache, const void* v_cache, const void* draft_k,
                           const void* draft_v, cudaStream_t st) {
  const int D = head_dim;
  CUtensorMap tq, tdk, tdv;
  PageMaps pm;
  const uint64_t W1 = (uint64_t)prm.W1;
  {
    const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)prm.hq, W1, (cuuint64_t)prm.B};
    const cuuint64_t strides[3] = {(cuuint64_t)D * 2ull, (cuuint64_t)prm.hq * D * 2ull,
                                   W1 * prm.hq * D * 2ull};
    const cuuint32_t box[4] = {64, (cuuint32_t)prm.G, (cuuint32_t)W1, 1};
    if (!encode_4d_bf16(&tq, q, dims, strides, box)) return cudaErrorInvalidValue;
  }
  {
    const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)kPage, (cuuint64_t)prm.hkv,
                                (cuuint64_t)prm.num_pages};
    const cuuint64_t strides[3] = {(cuuint64_t)D * 2ull, (cuuint64_t)kPage * D * 2ull,
                                   (cuuint64_t)prm.hkv * kPage * D * 2ull};
    for (int i = 0; i < 4; ++i) {
      const cuuint32_t box[4] = {64, (cuuint32_t)kPage, 1, 1u << i};
      if (!encode_4d_bf16(&pm.k[i], k_cache, dims, strides, box)) return cudaErrorInvalidValue;
      if (!encode_4d_bf16(&pm.v[i], v_cache, dims, strides, box)) return cudaErrorInvalidValue;
    }
  }
  if (prm.draft) {
    // draft scratch [B, hkv, kmax, D]: one box = the 16-row draft page (rows
    // past kmax are filled with zeros by the copy engine)
    const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)prm.kmax, (cuuint64_t)prm.hkv,
                                (cuuint64_t)prm.B};
    const cuuint64_t strides[3] = {(cuuint64_t)D * 2ull, (cuuint64_t)prm.kmax * D * 2ull,
                                   (cuuint64_t)prm.hkv * prm.kmax * D * 2ull};
    const cuuint32_t box[4] = {64, (cuuint32_t)kPage, 1, 1};
    if (!encode_4d_bf16(&tdk, draft_k, dims, strides, box)) return cudaErrorInvalidValue;
    if (!encode_4d_bf16(&tdv, draft_v, dims, strides, box)) return cudaErrorInvalidValue;
  } else {
    tdk = pm.k[0];
    tdv = pm.v[0];
  }
  const int R = prm.G * prm.W1;
  const int nq = (R + 15) / 16 * 16;
  cudaError_t e;
  if (D != 64 || nq > kMaxNQ) return cudaErrorInvalidValue;
  e = nq <= 16   ? launch_kt<64, 16>(prm, tq, pm, tdk, tdv, st)
      : nq <= 32 ? launch_kt<64, 32>(prm, tq, pm, tdk, tdv, st)
                 : launch_kt<64, 48>(prm, tq, pm, tdk, tdv, st);
  if (e != cudaSuccess) return e;
  return launch_attn_merge(prm, D, st);
}

}  // namespace seedk
