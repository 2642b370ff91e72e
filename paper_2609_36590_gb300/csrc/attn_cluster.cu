// Draft and verify attention for launches with few (sequence, KV head) pairs:
// one thread-block cluster per pair, the split merge on chip.
//
// What it computes is what attn_tc.cu computes (Sec. 4.1: the drafter attends
// to the cached deep KV with ordinary self-attention; Alg. 2 fixes the visible
// rows), for sequence b and the G query heads of KV head g:
//   verify: query j < n_q[b] over cache rows 0 .. L + j (L = ctx_lens[b]);
//   draft:  one query over cache rows 0 .. L - 1, then draft rows 0 .. nd - 1
//           of the draft scratch (nd = draft_lens[b]).
//
// Why a kernel of its own.  At batch 1 a call streams one layer's KV (8 MB at
// prefix 2048): well under one tile per SM, so its time is a chain of fixed
// latencies, not bandwidth.  Here the chain is the copies, one pass of
// products over resident keys and one on-chip merge:
//  * a fixed grid: cluster (b, g) of S CTAs (S = 8, 12 or 16, the largest
//    whose clusters are all resident at once); CTA r takes pages
//    [r np / S, (r + 1) np / S) of the pair's np pages (cache pages, then one
//    or two pages of draft rows), found from ctx_lens[b] and the aux length
//    alone -- no cost line, no lookup;
//  * before the dependency wait the CTA reads those lengths and page ids
//    (perhaps stale: the previous kernel may still write them) and keeps the
//    page window; after the wait, the lengths and the page ids of that window
//    are loaded together, so when the lengths did not change (all layers of a
//    verify pass) the copies start one load latency after the wait;
//  * all of a CTA's pages (at most 19) land at once: one TMA copy per 64-dim
//    half and run of consecutive page ids (1, 2, 4 or 8 pages; the copy
//    engine takes ~30 ns per copy), K of every tile before any V, one
//    mbarrier per tile and tensor, and nothing waits for the copy warp but
//    the products that need its pages;
//  * products on the tensor cores with the keys as MMA rows:
//      S^T = K Q^T   (tcgen05, M = 128 keys, N = 16 or 32 query rows),
//      O^T = V^T P^T (M = 128 head dims, N = 64: P_hi and P_lo of 32 query
//                    rows side by side, K = 16 keys per instruction);
//    each 128-key tile has its own group of four softmax warps (one thread
//    per key), its own maxima and its own O^T accumulators, so no tile waits
//    for another's softmax; only the NC query rows rounded up to 8 are read
//    and exponentiated (8 for a draft call at G = 4), the column maxima and
//    sums over a warp's 32 keys come from redux.sync (the sums on P in 24-bit
//    fixed point), and the epilogue adds the tiles' accumulators with
//    weights 2^(m_t - M);
//  * each CTA sends its partial state to the CTA that owns each 1/S of the
//    head dims with asynchronous distributed-shared-memory stores that count
//    their bytes on the owner's mbarrier; an owner merges as soon as every
//    byte it expects has landed: no workspace records, no merge kernel and
//    no cluster-wide barrier at the end.
// P = P_hi + P_lo (two bf16 terms: the truncated value and the truncated
// remainder) keeps ~16 bits of each probability.  V rows that no query may
// see (past the sequence end, draft rows past nd, pages with a bad id) are
// zeroed in shared memory before PV, so that stale or NaN rows add nothing.
// Every wait is bounded: one that gives up raises SEED_DEVERR_TIMEOUT, and
// the CTA still frees its tensor memory after its copies and products end.
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

constexpr int kClSoftWarps = 12;          // warps 0-11: softmax (warp 4 m + q: tile m, lane quarter q)
constexpr int kClThreads = (kClSoftWarps + 2) * 32;
constexpr int kWarpMmaCl = 12, kWarpLoadCl = 13;   // MMA, copies and TMEM; Q
constexpr int kClTiles = (kClMaxPages * kPage + 127) / 128;   // 128-key tiles: 3
constexpr int kClKeys = kClMaxPages * kPage;                  // 304
constexpr uint32_t kClTmemCols = 512;
// TMEM columns: S^T of tile m at [32 m, 32 m + 32); O^T of tile m in two
// accumulators (even and odd pages, which halves the dependent chain of
// products) at [128 + 128 m, + 64) and [192 + 128 m, + 64), each P_hi
// columns then P_lo columns
constexpr uint32_t kClColO = 128;
constexpr float kClLn2 = 0.69314718055994531f;
constexpr int kClRecvStride = 36;          // floats per received (source, dim) row of 32 columns

// The head dims CTA r of S merges: [dim0(r), dim0(r + 1)).
__host__ __device__ constexpr int dim0(int r, int S) { return r * 128 / S; }
// ... and the CTA that merges dim d.
__device__ __forceinline__ int dim_owner(int d, int S) { return ((d + 1) * S - 1) / 128; }

template <int D, int S>
struct ClLayout {
  static constexpr int kHalves = D / 64;
  static constexpr int kDsMax = (128 + S - 1) / S;             // dims merged per CTA, at most
  static constexpr uint32_t kPageBytes = kPage * D * 2;       // one page of K (or V)
  static constexpr uint32_t kHalfBytes = kClKeys * 128;       // one 64-dim half of K (or V)
  static constexpr uint32_t kOffK = 0;                         // [half][key][128 B]
  static constexpr uint32_t kOffV = kHalves * kHalfBytes;
  // P^T, MN-major: one 128-byte row per key = P_hi of query rows 0-31, then
  // P_lo of the same rows (bf16), 16-byte chunks XOR-swizzled by key & 7
  static constexpr uint32_t kOffP = 2 * kHalves * kHalfBytes;
  static constexpr uint32_t kOffQ = kOffP + kClKeys * 128;    // [half][32 rows][128 B]
  // the partial states the cluster sends here: O [source][dim][column],
  // then (max, sum) [source][column]
  static constexpr uint32_t kOffRecvO = kOffQ + kHalves * kClRows * 128;
  static constexpr uint32_t kOffRecvS = kOffRecvO + S * kDsMax * kClRecvStride * 4;
  static constexpr uint32_t kOffCtrl = kOffRecvS + S * kClRows * 8;
};

struct ClCtrl {
  uint64_t kfull[kClTiles], vfull[kClTiles];
  uint64_t s_full[kClTiles], p_full[kClTiles], o_full[kClTiles];
  uint64_t q_ready, codes_ready, recv_full;
  uint32_t tmem_base;
  int32_t spec_p0, spec_n;                    // page window read before the dependency wait
  int32_t code[kClMaxPages];                  // page id; -2 - i: draft page i; -1: none
  float wmax[kClTiles][4][kClRows];           // per tile and lane quarter: column maxima
  float wsum[kClTiles][4][kClRows];           // ... and sums
  float tmax[kClTiles][kClRows];              // per tile: column maxima (log2 units)
  float tw[kClTiles][kClRows];                // per tile: weight of its O in the CTA's
};

template <int D, int S>
constexpr size_t cl_smem_bytes() {
  return ClLayout<D, S>::kOffCtrl + sizeof(ClCtrl) + 1024;   // + alignment slack
}
static_assert(cl_smem_bytes<128, 8>() <= 232448, "shared memory budget");
static_assert(cl_smem_bytes<128, 12>() <= 232448, "shared memory budget");
static_assert(cl_smem_bytes<128, 16>() <= 232448, "shared memory budget");

// ------------------------------------------------------------- PTX helpers
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// The two halves of a cluster barrier: every CTA of the cluster has arrived
// (so has started: its shared memory may take remote stores) once the wait
// returns.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_peer(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}

// Asynchronous stores into another CTA's shared memory whose bytes complete a
// transaction count on that CTA's mbarrier (both addresses shared::cluster).
__device__ __forceinline__ void st_async2(uint32_t a, float x, float y, uint32_t bar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(a),
      "f"(x), "f"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void st_async4(uint32_t a, float x, float y, float z, float w,
                                          uint32_t bar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, "
      "[%5];" ::"r"(a),
      "f"(x), "f"(y), "f"(z), "f"(w), "r"(bar)
      : "memory");
}

// Bulk prefetch of `bytes` (a multiple of 16) from global memory into L2.
__device__ __forceinline__ void prefetch_l2_bulk(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Barrier of the softmax warps (named barrier 1), and of the four warps of
// tile m's group (named barrier 2 + m).
__device__ __forceinline__ void softmax_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(kClSoftWarps * 32) : "memory");
}
__device__ __forceinline__ void tile_bar(int m) {
  asm volatile("bar.sync %0, 128;" ::"r"(2 + m) : "memory");
}

// Bounded wait on an mbarrier phase by one thread (polling).
__device__ __forceinline__ bool cl_wait(uint64_t* bar, uint32_t parity) {
  for (uint32_t i = 0; i < (1u << 22); ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

// The same by a whole warp, which agrees on the outcome.
__device__ __forceinline__ bool cl_warp_wait(uint64_t* bar, uint32_t parity) {
  return __all_sync(kFull, cl_wait(bar, parity));
}

// Bounded wait with cluster-scope acquire: the phase was completed by other
// CTAs' asynchronous stores.
__device__ __forceinline__ bool cl_wait_cluster(uint64_t* bar, uint32_t parity) {
  for (uint32_t i = 0; i < (1u << 22); ++i) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (ok) return true;
  }
  return false;
}

// N (8, 16, 24 or 32) consecutive TMEM columns of this thread's lane, added
// to v (the loads are issued together and waited for once).
template <int N>
__device__ __forceinline__ void tmem_add_cols(uint32_t taddr, float (&v)[N]) {
  static_assert(N % 8 == 0 && N <= 32, "column count");
  if constexpr (N == 32) {
    uint32_t r[32];
    tmem_ld32(taddr, r);
    tmem_wait_ld();
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] += __uint_as_float(r[i]);
  } else if constexpr (N == 24) {
    uint32_t r[16], r2[8];
    tmem_ld16(taddr, r);
    tmem_ld8(taddr + 16, r2);
    tmem_wait_ld();
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] += __uint_as_float(r[i]);
#pragma unroll
    for (int i = 0; i < 8; ++i) v[16 + i] += __uint_as_float(r2[i]);
  } else if constexpr (N == 16) {
    uint32_t r[16];
    tmem_ld16(taddr, r);
    tmem_wait_ld();
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] += __uint_as_float(r[i]);
  } else {
    uint32_t r[8];
    tmem_ld8(taddr, r);
    tmem_wait_ld();
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] += __uint_as_float(r[i]);
  }
}

// Warp-wide sum of one value per lane (every lane gets it).
__device__ __forceinline__ uint32_t warp_sum_u32(uint32_t x) {
  uint32_t r;
  asm volatile("redux.sync.add.u32 %0, %1, 0xffffffff;" : "=r"(r) : "r"(x));
  return r;
}

// Warp-wide maximum of one value per lane (every lane gets it).
__device__ __forceinline__ float warp_max(float x) {
  float r;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(x));
  return r;
}

// A tile's O^T columns 0 .. N - 1 of this thread's lane: the sum of its two
// accumulators (even and odd pages; the odd one is unwritten when the tile
// has a single page), each P_hi columns plus P_lo columns.
template <int N>
__device__ __forceinline__ void tile_o(uint32_t taddr, int pages, float (&o)[N]) {
  tmem_add_cols<N>(taddr, o);
  tmem_add_cols<N>(taddr + 32u, o);
  if (pages >= 2) {
    tmem_add_cols<N>(taddr + 64u, o);
    tmem_add_cols<N>(taddr + 96u, o);
  }
}

// Pages [p0, p0 + npg) of the np pages of a pair, for CTA `rank` of S.
__device__ __forceinline__ void cta_pages(int np, int rank, int S, int& p0, int& npg) {
  p0 = rank * np / S;
  npg = (rank + 1) * np / S - p0;
}

// The pair's cache and draft page counts from the lengths L, a (nq or nd);
// false for a sequence with bad arguments or nothing to do.
__device__ __forceinline__ bool pair_pages(const AttnTcParams& p, int L, int a, int& ncp,
                                           int& nd) {
  const long long cap = (long long)p.max_pages * kPage;
  if (p.draft) {
    if (a <= 0 || a > p.kmax || L < 0 || L > cap) return false;
    ncp = (L + kPage - 1) / kPage;
    nd = a;
  } else {
    if (a <= 0 || a > p.kmax + 1 || L < 0 || (long long)L + a > cap) return false;
    ncp = (L + a + kPage - 1) / kPage;
    nd = 0;
  }
  return true;
}

// Before the dependency wait (one warp): read the lengths through L2 only (no
// stale copy stays in L1) and record this CTA's page window; pull the pair's
// query rows into L2.  Stale values cost a useless prefetch or a second page
// id load at most.
template <int D, int S>
__device__ __forceinline__ void prepare(const AttnTcParams& p, int b, int g, int rank, int lane,
                                        ClCtrl* ctrl) {
  int ncp = 0, nd = 0, p0 = 0, npg = 0;
  if (pair_pages(p, __ldcg(p.ctx_lens + b), __ldcg(p.aux + b), ncp, nd)) {
    cta_pages(ncp + draft_pages(nd), rank, S, p0, npg);
    npg = min(npg, kClMaxPages);
  }
  if (lane == 0) {
    ctrl->spec_p0 = p0;
    ctrl->spec_n = npg;
  }
  // the query rows of the pair: G heads x W1 positions, G * D * 2 bytes each
  if (lane < p.W1)
    prefetch_l2_bulk(p.q + (((size_t)b * p.W1 + lane) * p.hq + (size_t)g * p.G) * D,
                     (uint32_t)p.G * D * 2);
}

// ------------------------------------------------------------- the kernel
// Grid (S, hkv, B), clusters of S along x: cluster (b, g), CTA rank r.
// NC = query rows G * W1 rounded up to 8: the columns the softmax reads.
template <int D, int NC, int S>
__global__ void __launch_bounds__(kClThreads, 1)
    attn_cl_kernel(const __grid_constant__ PageMaps pm, const __grid_constant__ CUtensorMap tm_dk,
                   const __grid_constant__ CUtensorMap tm_dv, const AttnTcParams p) {
  using LY = ClLayout<D, S>;
  static_assert(D == 128, "the epilogue warps hold one head dim per thread");
  constexpr int NQ = NC <= 16 ? 16 : 32;        // the S MMA's N
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 128-byte swizzled operands need a 1 KiB aligned base (the same offset in
  // every CTA, so the receive buffers sit at the same address in each)
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  ClCtrl* ctrl = reinterpret_cast<ClCtrl*>(smem + LY::kOffCtrl);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = blockIdx.y, b = blockIdx.z;
  const int rank = (int)cluster_rank();
  const uint32_t sbase = smem_u32(smem);
  const int ds = dim0(rank + 1, S) - dim0(rank, S);   // head dims this CTA merges
  if (tid == 0) pdl_trigger();
  if (tid == 0) {
    for (int m = 0; m < kClTiles; ++m) {
      mbar_init(&ctrl->kfull[m], 1);
      mbar_init(&ctrl->vfull[m], 1);
      mbar_init(&ctrl->s_full[m], 1);
      mbar_init(&ctrl->p_full[m], 4);
      mbar_init(&ctrl->o_full[m], 1);
    }
    mbar_init(&ctrl->q_ready, kClSoftWarps + 1);
    mbar_init(&ctrl->codes_ready, 1);
    mbar_init(&ctrl->recv_full, 1);
    fence_mbar_init();
  }
  if (warp == kWarpMmaCl) {
    tmem_alloc(&ctrl->tmem_base, kClTmemCols);
    tmem_relinquish();
    if (lane < 4) {
      tma_prefetch_desc(&pm.k[lane]);
      tma_prefetch_desc(&pm.v[lane]);
    }
    if (lane == 0 && p.draft) {
      tma_prefetch_desc(&tm_dk);
      tma_prefetch_desc(&tm_dv);
    }
  }
  if (warp == kWarpLoadCl) prepare<D, S>(p, b, g, rank, lane, ctrl);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_arrive_relaxed();
  const uint32_t tmem = ctrl->tmem_base;
  pdl_wait();

  // ---- Q first (its rows do not depend on the lengths): rows n = j * G +
  // head of all W1 positions (rows past them zero), K-major with 128-byte
  // swizzle: row n of half h at n * 128, 16-byte chunks XOR-ed with n & 7
  if (warp != kWarpMmaCl) {
    constexpr int kCpr = D / 8;   // 16-byte chunks per row
    const int rq_all = p.G * p.W1;
    const int t0 = warp == kWarpLoadCl ? lane : 32 + tid;
    for (int i = t0; i < NQ * kCpr; i += (kClSoftWarps + 1) * 32) {
      const int n = i / kCpr, c = i % kCpr;
      uint4 v = make_uint4(0u, 0u, 0u, 0u);
      if (n < rq_all) {
        const int j = n / p.G, hh = n - j * p.G;
        v = reinterpret_cast<const uint4*>(
            p.q + (((size_t)b * p.W1 + j) * p.hq + (size_t)g * p.G + hh) * D)[c];
      }
      *reinterpret_cast<uint4*>(smem + LY::kOffQ + (c >> 3) * (NQ * 128) + n * 128 +
                                (((c & 7) ^ (n & 7)) << 4)) = v;
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctrl->q_ready);
  }

  // ---- the pair's geometry (the same in every CTA of the cluster).  The
  // copy warp loads the page ids of the pre-wait window with the lengths.
  int pid_spec = -1;
  const int sp0 = ctrl->spec_p0, sn = ctrl->spec_n;
  if (warp == kWarpMmaCl && lane < sn && sp0 + lane < p.max_pages)
    pid_spec = __ldcg(p.page_table + (size_t)b * p.max_pages + sp0 + lane);
  const SeqT sq = seq_of(p, b);
  const bool skip = sq.bad != 0 || sq.nq == 0;
  if (sq.bad && rank == 0 && g == 0 && tid == 0) raise_err(p.err, sq.bad);
  int p0 = 0, npg = 0;
  if (!skip) cta_pages(sq.ncp + draft_pages(sq.nd), rank, S, p0, npg);
  if (npg > kClMaxPages) {   // excluded by the host's routing; never silently wrong
    if (tid == 0) raise_err(p.err, SEED_DEVERR_WORKSPACE);
    npg = 0;
  }
  const int ntiles = (npg * kPage + 127) / 128;
  bool ok = true;
  // what the cluster sends here: from each of the S CTAs, (max, sum) of the
  // rq query rows with outputs and this CTA's dims of them (rows in fours).
  // Posted now, when rq is known: bytes that land first only take the
  // transaction count below zero until then.
  const int rq_s = skip ? 0 : sq.nq * p.G, rq4 = (rq_s + 3) & ~3;
  if (tid == 0 && !skip)
    mbar_arrive_expect_tx(&ctrl->recv_full, (uint32_t)(S * rq_s * 8 + S * ds * rq4 * 4));

  // ---- copies: the MMA warp puts page p0 + s into key rows [16 s, 16 s + 16)
  // of K and V
  if (warp == kWarpMmaCl && npg > 0) {
    const int vp = p0 + lane;
    const bool hit = lane < npg && vp < sq.ncp && vp >= sp0 && vp - sp0 < sn;
    const int spec = __shfl_sync(kFull, pid_spec, hit ? vp - sp0 : 0);
    int code = -1;
    if (lane < npg) {
      if (vp < sq.ncp) {
        const int id = hit ? spec : __ldcg(p.page_table + (size_t)b * p.max_pages + vp);
        if (id >= 0 && id < p.num_pages)
          code = id;
        else
          raise_err(p.err, SEED_DEVERR_PAGE);
      } else {
        code = -2 - (vp - sq.ncp);
      }
      ctrl->code[lane] = code;
    }
    const uint32_t loads = __ballot_sync(kFull, lane < npg && code != -1);
    __syncwarp();
    if (lane == 0) {
      mbar_arrive(&ctrl->codes_ready);
      for (int m = 0; m < ntiles; ++m) {
        const uint32_t bytes = (uint32_t)__popc((loads >> (8 * m)) & 0xffu) * LY::kPageBytes;
        mbar_arrive_expect_tx(&ctrl->kfull[m], bytes);
        mbar_arrive_expect_tx(&ctrl->vfull[m], bytes);
      }
    }
    __syncwarp();
    // cache pages: per 128-key tile, one copy per run of consecutive ids
    // (lane i < 8 of tile m holds slot 8 m + i); K of every tile first, so
    // that the scores and the softmax overlap the V copies
    int box[kClTiles], bpid[kClTiles];
#pragma unroll
    for (int m = 0; m < kClTiles; ++m) {
      box[m] = 0;
      bpid[m] = -1;
      if (m < ntiles) {
        const int slot = 8 * m + (lane & 7);
        const int cs = __shfl_sync(kFull, code, slot);
        bpid[m] = (lane < 8 && slot < npg && cs >= 0) ? cs : -1;
        box[m] = box_size(bpid[m], lane);
      }
    }
    const int y = code <= -2 ? kPage * (-2 - code) : 0;
    const uint64_t kv_pol = policy_evict_first();   // cache pages are read once per call
#pragma unroll
    for (int kv = 0; kv < 2; ++kv) {
      const uint32_t off = kv == 0 ? LY::kOffK : LY::kOffV;
#pragma unroll
      for (int m = 0; m < kClTiles; ++m) {
        if (box[m] > 0) {
          const CUtensorMap* mp = kv == 0 ? &pm.k[log2_box(box[m])] : &pm.v[log2_box(box[m])];
          uint64_t* bar = kv == 0 ? &ctrl->kfull[m] : &ctrl->vfull[m];
#pragma unroll
          for (int h = 0; h < LY::kHalves; ++h)
            tma_load_4d_hint(smem + off + h * LY::kHalfBytes + (8 * m + lane) * 2048, mp,
                             64 * h, 0, g, bpid[m], bar, kv_pol);
        }
      }
      // draft pages: one copy each from the draft scratch
      if (lane < npg && code <= -2) {
        uint64_t* bar = kv == 0 ? &ctrl->kfull[lane >> 3] : &ctrl->vfull[lane >> 3];
#pragma unroll
        for (int h = 0; h < LY::kHalves; ++h)
          tma_load_4d(smem + off + h * LY::kHalfBytes + lane * 2048, kv == 0 ? &tm_dk : &tm_dv,
                      64 * h, y, g, b, bar);
      }
    }
  }

  if (skip) {
    // nothing to do for this pair (the same in every CTA of the cluster);
    // the Q loads above have landed (their warps waited for them)
    if (warp == kWarpMmaCl) {
      tc_fence_after();
      tmem_dealloc(tmem, kClTmemCols);
    }
    return;
  }

  const int lg = __ffs(p.G) - 1;   // G is a power of two
  const int rq = sq.nq * p.G;      // query rows with outputs
  if (warp == kWarpMmaCl) {
    // ---------------------------------------------------------- MMA issuer
    // S^T(m) for every tile as its K lands, then PV(m) into tile m's own O^T
    // as its P is written: no tile waits for another's softmax
    if (lane == 0) {
      constexpr uint32_t kIdescS = idesc_bf16_f32(128, NQ, 0, 0);   // K, Q K-major
      constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 64, 1, 1);  // V^T, P^T MN-major
      const uint32_t sK = sbase + LY::kOffK, sV = sbase + LY::kOffV;
      const uint32_t sP = sbase + LY::kOffP, sQ = sbase + LY::kOffQ;
      ok = cl_wait(&ctrl->q_ready, 0);
      for (int m = 0; m < ntiles && ok; ++m) {
        if (!cl_wait(&ctrl->kfull[m], 0)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t h = kk >> 2, off = (kk & 3) * 32;
          const uint64_t a = smem_desc_sw128(sK + h * LY::kHalfBytes + m * 16384u + off, 16, 1024);
          const uint64_t bq = smem_desc_sw128(sQ + h * (NQ * 128) + off, 16, 1024);
          mma_ss(tmem + 32u * m, a, bq, kIdescS, kk > 0);
        }
        mma_commit(&ctrl->s_full[m]);
      }
      for (int m = 0; m < ntiles && ok; ++m) {
        // P(m) written (its softmax warps zeroed V rows first, after V landed)
        ok = cl_wait(&ctrl->p_full[m], 0) && cl_wait(&ctrl->vfull[m], 0);
        if (!ok) break;
        tc_fence_after();
        const int k1 = min(8 * m + 8, npg);
        for (int kk = 8 * m; kk < k1; ++kk) {
          const uint64_t a = smem_desc_sw128(sV + kk * 2048u, LY::kHalfBytes, 1024);
          const uint64_t bp = smem_desc_sw128(sP + kk * 2048u, 0, 1024);
          const uint32_t acc = kClColO + 128u * m + 64u * ((kk - 8 * m) & 1);
          mma_ss(tmem + acc, a, bp, kIdescPV, kk - 8 * m >= 2);
        }
        mma_commit(&ctrl->o_full[m]);
      }
      if (!ok) raise_err(p.err, SEED_DEVERR_TIMEOUT);
    }
    __syncwarp();
    cluster_wait();   // (every CTA of the cluster is running)
  } else if (warp < kClSoftWarps) {
    // ---------------------------------------------------------- softmax
    // Warp 4 m + q reads TMEM lane quarter q of tile m's S^T: key
    // 128 m + 32 q + lane.  The group of tile m works on it alone: the
    // tile's column maxima, P = 2^(s - max) and the column sums.
    const int m = warp >> 2, q4 = warp & 3;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    if (m < ntiles) {
      const float c2 = p.scale_log2;
      const int key = m * 128 + q4 * 32 + lane, s = key >> 4;
      // keys past the CTA's pages (the end of the last tile) are never read
      // by PV and have no row in the P operand
      const bool in_pages = s < npg;
      int nmin = NC;   // first query row that sees the key (NC: none)
      const bool gotc = cl_warp_wait(&ctrl->codes_ready, 0);
      ok = ok && gotc;
      if (in_pages && gotc) {
        const int code = ctrl->code[s];
        if (code <= -2) {
          nmin = (kPage * (-2 - code) + (key & 15) < sq.nd) ? 0 : NC;
        } else if (code >= 0) {
          const int kpos = (p0 + s) * kPage + (key & 15);
          nmin = kpos < sq.cvalid ? min(max(kpos - sq.lim0, 0) << lg, NC) : NC;
        }
      }
      const bool got = cl_warp_wait(&ctrl->s_full[m], 0);
      ok = ok && got;
      tc_fence_after();
      float sv[NC];
#pragma unroll
      for (int c = 0; c < NC; ++c) sv[c] = 0.f;
      if (got) tmem_add_cols<NC>(tmem + lane_off + 32u * m, sv);
#pragma unroll
      for (int c = 0; c < NC; ++c) sv[c] = c >= nmin ? sv[c] * c2 : -INFINITY;
      // the tile's column maxima: over the warp's 32 keys, then the group's
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        const float wm = warp_max(sv[c]);
        if (lane == 0) ctrl->wmax[m][q4][c] = wm;
      }
      tile_bar(m);
      if (q4 == 0 && lane < NC) {
        float t = -INFINITY;
#pragma unroll
        for (int w = 0; w < 4; ++w) t = fmaxf(t, ctrl->wmax[m][w][lane]);
        ctrl->tmax[m][lane] = t;
      }
      tile_bar(m);
      // P^T row of this key: P_hi of query rows 0-31 (16-byte chunks 0-3),
      // then P_lo (chunks 4-7); only the chunks of the NC rows are written
      // (the others feed output columns nobody reads)
      float pv[NC];
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        const float t = ctrl->tmax[m][c];
        pv[c] = ex2_approx(sv[c] - (t == -INFINITY ? 0.f : t));
      }
      if (in_pages) {
        uint8_t* prow = smem + LY::kOffP + key * 128;
#pragma unroll
        for (int j = 0; j < NC / 8; ++j) {
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float p0 = pv[8 * j + 2 * e], p1 = pv[8 * j + 2 * e + 1];
            const uint32_t h0 = __float_as_uint(p0) & 0xffff0000u;
            const uint32_t h1 = __float_as_uint(p1) & 0xffff0000u;
            const uint32_t l0 = __float_as_uint(p0 - __uint_as_float(h0)) & 0xffff0000u;
            const uint32_t l1 = __float_as_uint(p1 - __uint_as_float(h1)) & 0xffff0000u;
            hi[e] = (h0 >> 16) | h1;
            lo[e] = (l0 >> 16) | l1;
          }
          *reinterpret_cast<uint4*>(prow + ((j ^ (key & 7)) << 4)) =
              make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(prow + (((j + 4) ^ (key & 7)) << 4)) =
              make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
      }
      // column sums over the warp's keys: P in [0, 1] as 24-bit fixed point,
      // summed exactly by redux (error <= 2^-20 against a tile sum >= 1)
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        const uint32_t u = warp_sum_u32(__float2uint_rn(pv[c] * 16777216.f));
        if (lane == 0) ctrl->wsum[m][q4][c] = (float)u * (1.f / 16777216.f);
      }
      // V rows of keys nobody may see are zeroed (after V has landed, or the
      // copy engine would overwrite the zeros); only warps holding such keys
      // (the tail of a sequence, a draft page, a bad page id) wait for V
      const bool zero = nmin >= NC && in_pages;
      if (__any_sync(kFull, zero)) ok = ok && cl_warp_wait(&ctrl->vfull[m], 0);
      if (zero) {
#pragma unroll
        for (int h = 0; h < LY::kHalves; ++h)
#pragma unroll
          for (int ch = 0; ch < 8; ++ch)
            *reinterpret_cast<uint4*>(smem + LY::kOffV + h * LY::kHalfBytes + key * 128 + ch * 16) =
                make_uint4(0u, 0u, 0u, 0u);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctrl->p_full[m]);
    }
    // epilogue (group 0: thread = head dim d): tile 0's O^T (P_hi columns +
    // P_lo columns) is read while the other tiles' products run
    float o0[NC];
#pragma unroll
    for (int c = 0; c < NC; ++c) o0[c] = 0.f;
    if (m == 0 && ntiles > 0) {
      const bool got = cl_warp_wait(&ctrl->o_full[0], 0);
      ok = ok && got;
      tc_fence_after();
      if (got) tile_o<NC>(tmem + lane_off + kClColO, min(npg, 8), o0);
    }
    // every tile's statistics are written: the CTA's (max, sum) per column,
    // sent to every CTA of the cluster (all of which are running once the
    // cluster wait returns), and each tile's weight
    cluster_wait();
    softmax_bar();
    if (warp == 0 && lane < rq) {
      float M = -INFINITY;   // (rq <= NC)
      for (int t = 0; t < ntiles; ++t) M = fmaxf(M, ctrl->tmax[t][lane]);
      float L = 0.f;
      for (int t = 0; t < ntiles; ++t) {
        float st = 0.f;
#pragma unroll
        for (int w = 0; w < 4; ++w) st += ctrl->wsum[t][w][lane];
        const float tm = ctrl->tmax[t][lane];
        const float f = (st > 0.f) ? ex2_approx(tm - M) : 0.f;
        ctrl->tw[t][lane] = f;
        L = fmaf(st, f, L);
      }
      const uint32_t a = sbase + LY::kOffRecvS + (uint32_t)(rank * kClRows + lane) * 8u;
      const uint32_t bar = smem_u32(&ctrl->recv_full);
#pragma unroll
      for (int q = 0; q < S; ++q) st_async2(map_peer(a, q), M, L, map_peer(bar, q));
    }
    softmax_bar();
    if (m == 0) {
      // the other tiles' O^T, then O^T = sum over tiles of weight x O_t,
      // sent to the CTA that merges dim d (the rows with outputs only)
      const int d = q4 * 32 + lane;
      float o[NC];
#pragma unroll
      for (int c = 0; c < NC; ++c) o[c] = ntiles > 0 ? ctrl->tw[0][c] * o0[c] : 0.f;
#pragma unroll 1
      for (int t = 1; t < ntiles; ++t) {
        const bool got = cl_warp_wait(&ctrl->o_full[t], 0);
        ok = ok && got;
        tc_fence_after();
        float ot[NC];
#pragma unroll
        for (int c = 0; c < NC; ++c) ot[c] = 0.f;
        if (got) tile_o<NC>(tmem + lane_off + kClColO + 128u * t, min(npg - 8 * t, 8), ot);
#pragma unroll
        for (int c = 0; c < NC; ++c) o[c] = fmaf(ctrl->tw[t][c], ot[c], o[c]);
      }
      const int owner = dim_owner(d, S);
      const uint32_t a = map_peer(
          sbase + LY::kOffRecvO +
              (uint32_t)((rank * LY::kDsMax + (d - dim0(owner, S))) * kClRecvStride) * 4u,
          (uint32_t)owner);
      const uint32_t bar = map_peer(smem_u32(&ctrl->recv_full), (uint32_t)owner);
#pragma unroll
      for (int c = 0; c < NC; c += 4)
        if (c < rq) st_async4(a + c * 4u, o[c], o[c + 1], o[c + 2], o[c + 3], bar);
    }
    if (!ok && lane == 0) raise_err(p.err, SEED_DEVERR_TIMEOUT);
  } else {
    cluster_wait();   // (the load warp: every CTA of the cluster is running)
  }

  // ---- merge this CTA's slice, head dims [dim0(r), dim0(r + 1)) of every
  // row, once every byte the cluster sends here has landed
  if (cl_wait_cluster(&ctrl->recv_full, 0)) {
    const float* recv_o = reinterpret_cast<const float*>(smem + LY::kOffRecvO);
    const float2* recv_s = reinterpret_cast<const float2*>(smem + LY::kOffRecvS);
    const int d0 = dim0(rank, S);
    for (int i = tid; i < rq * ds; i += kClThreads) {
      const int n = i / ds, dd = i - n * ds;
      float2 st[S];
      float vq[S];
#pragma unroll
      for (int q = 0; q < S; ++q) {
        st[q] = recv_s[q * kClRows + n];
        vq[q] = recv_o[(q * LY::kDsMax + dd) * kClRecvStride + n];
      }
      float M = -INFINITY;
#pragma unroll
      for (int q = 0; q < S; ++q)
        if (st[q].y > 0.f) M = fmaxf(M, st[q].x);
      float L = 0.f, acc = 0.f;
#pragma unroll
      for (int q = 0; q < S; ++q) {
        if (st[q].y > 0.f) {
          const float f = ex2_approx(st[q].x - M);
          L = fmaf(st[q].y, f, L);
          acc = fmaf(f, vq[q], acc);
        }
      }
      const int j = n >> lg, hh = n - (j << lg);
      const size_t orow = ((size_t)b * p.W1 + j) * p.hq + (size_t)g * p.G + hh;
      p.out[orow * D + d0 + dd] = L > 0.f ? acc / L : 0.f;
      if (rank == 0 && dd == 0 && p.lse != nullptr)
        p.lse[orow] = L > 0.f ? (M + log2f(L)) * kClLn2 : -INFINITY;
    }
  } else if (tid == 0) {
    raise_err(p.err, SEED_DEVERR_TIMEOUT);
  }
  // no copy may still be landing, and no product running, when the CTA
  // exits and frees its tensor memory (only after a wait gave up can one be)
  if (warp == kWarpMmaCl) {
    if (lane < npg && ctrl->code[lane] != -1) {
      cl_wait(&ctrl->kfull[lane >> 3], 0);
      cl_wait(&ctrl->vfull[lane >> 3], 0);
    }
    if (lane < ntiles) cl_wait(&ctrl->o_full[lane], 0);
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kClTmemCols);
  }
}

// ------------------------------------------------------------- host side
std::atomic<uint64_t> g_cl_attr_set{0};
std::atomic<int> g_cl_clusters[64][3];   // resident clusters of 8, 12, 16 CTAs

constexpr int kClSizes[3] = {8, 12, 16};

template <int NC, int S>
cudaError_t set_cl_attr() {
  cudaError_t e = cudaFuncSetAttribute(attn_cl_kernel<128, NC, S>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)cl_smem_bytes<128, S>());
  if (e != cudaSuccess || S <= 8) return e;
  return cudaFuncSetAttribute(attn_cl_kernel<128, NC, S>,
                              cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

template <int S>
cudaError_t set_cl_attrs_s() {
  cudaError_t e;
  if ((e = set_cl_attr<8, S>()) != cudaSuccess) return e;
  if ((e = set_cl_attr<16, S>()) != cudaSuccess) return e;
  if ((e = set_cl_attr<24, S>()) != cudaSuccess) return e;
  return set_cl_attr<32, S>();
}

cudaError_t set_cl_attrs(int dev) {
  const uint64_t bit = 1ull << (dev & 63);
  if (g_cl_attr_set.load(std::memory_order_acquire) & bit) return cudaSuccess;
  cudaError_t e;
  if ((e = set_cl_attrs_s<8>()) != cudaSuccess) return e;
  if ((e = set_cl_attrs_s<12>()) != cudaSuccess) return e;
  if ((e = set_cl_attrs_s<16>()) != cudaSuccess) return e;
  g_cl_attr_set.fetch_or(bit, std::memory_order_acq_rel);
  return cudaSuccess;
}

void cl_launch_config(cudaLaunchConfig_t& cfg, cudaLaunchAttribute (&at)[2], dim3 grid, int S,
                      size_t smem, cudaStream_t st, bool pdl) {
  cfg = cudaLaunchConfig_t{};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kClThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = (unsigned)S;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = pdl ? 2 : 1;
}

template <int S>
int query_clusters() {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute at[2];
  cl_launch_config(cfg, at, dim3(S, 1, 1), S, cl_smem_bytes<128, S>(), nullptr, false);
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_cl_kernel<128, 32, S>, &cfg) != cudaSuccess) n = 0;
  return n;
}

// Clusters of kClSizes[i] CTAs that are resident at once on the current
// device (queried once per device).
int cl_clusters(int i) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int cached = g_cl_clusters[dev][i].load(std::memory_order_relaxed);
  if (cached != 0) return cached > 0 ? cached : 0;
  int n = 0;
  if (set_cl_attrs(dev) == cudaSuccess)
    n = i == 0 ? query_clusters<8>() : i == 1 ? query_clusters<12>() : query_clusters<16>();
  (void)cudaGetLastError();   // a failed query leaves no sticky error behind
  g_cl_clusters[dev][i].store(n > 0 ? n : -1, std::memory_order_relaxed);
  return n > 0 ? n : 0;
}

template <int S>
cudaError_t launch_cl_t(int nc, const PageMaps& pm, const CUtensorMap& tdk,
                        const CUtensorMap& tdv, const AttnTcParams& prm, cudaStream_t st) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute at[2];
  cl_launch_config(cfg, at, dim3(S, prm.hkv, prm.B), S, cl_smem_bytes<128, S>(), st, true);
  switch (nc) {
    case 8: return cudaLaunchKernelEx(&cfg, attn_cl_kernel<128, 8, S>, pm, tdk, tdv, prm);
    case 16: return cudaLaunchKernelEx(&cfg, attn_cl_kernel<128, 16, S>, pm, tdk, tdv, prm);
    case 24: return cudaLaunchKernelEx(&cfg, attn_cl_kernel<128, 24, S>, pm, tdk, tdv, prm);
    case 32: return cudaLaunchKernelEx(&cfg, attn_cl_kernel<128, 32, S>, pm, tdk, tdv, prm);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int attn_cl_route(int head_dim, int group, int w1, int batch, int hkv, int max_pages) {
  if (head_dim != 128 || group * w1 > kClRows) return 0;
  const long long pairs = (long long)batch * hkv;
  // the largest cluster whose clusters are all resident at once and whose
  // CTAs hold every sequence the page table allows (plus two draft pages)
  for (int i = 2; i >= 0; --i) {
    const int S = kClSizes[i];
    if ((long long)max_pages + 2 > (long long)S * kClMaxPages) continue;
    if (pairs <= cl_clusters(i)) return S;
  }
  return 0;
}

cudaError_t launch_attn_cl(const AttnTcParams& prm, int cluster, const void* k_cache,
                           const void* v_cache, const void* draft_k, const void* draft_v,
                           cudaStream_t st) {
  constexpr int D = 128;
  PageMaps pm;
  CUtensorMap tdk, tdv;
  {
    const cuuint64_t dims[4] = {D, (cuuint64_t)kPage, (cuuint64_t)prm.hkv,
                                (cuuint64_t)prm.num_pages};
    const cuuint64_t strides[3] = {D * 2ull, kPage * D * 2ull,
                                   (cuuint64_t)prm.hkv * kPage * D * 2ull};
    for (int i = 0; i < 4; ++i) {
      const cuuint32_t box[4] = {64, (cuuint32_t)kPage, 1, 1u << i};
      if (!encode_4d_bf16(&pm.k[i], k_cache, dims, strides, box)) return cudaErrorInvalidValue;
      if (!encode_4d_bf16(&pm.v[i], v_cache, dims, strides, box)) return cudaErrorInvalidValue;
    }
  }
  if (prm.draft) {
    // draft scratch [B, hkv, kmax, D]: a box is one 16-row draft page (rows
    // past kmax are filled with zeros by the copy engine)
    const cuuint64_t dims[4] = {D, (cuuint64_t)prm.kmax, (cuuint64_t)prm.hkv, (cuuint64_t)prm.B};
    const cuuint64_t strides[3] = {D * 2ull, (cuuint64_t)prm.kmax * D * 2ull,
                                   (cuuint64_t)prm.hkv * prm.kmax * D * 2ull};
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
  if ((e = set_cl_attrs(dev)) != cudaSuccess) return e;
  const int nc = (prm.G * prm.W1 + 7) & ~7;   // query rows rounded up to 8
  switch (cluster) {
    case 8: return launch_cl_t<8>(nc, pm, tdk, tdv, prm, st);
    case 12: return launch_cl_t<12>(nc, pm, tdk, tdv, prm, st);
    case 16: return launch_cl_t<16>(nc, pm, tdk, tdv, prm, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace seedk
