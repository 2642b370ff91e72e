// Work description shared by the tensor-core draft / verify attention kernels
// (attn_tc.cu, attn_kt.cu) and their split merge: the geometry of one
// sequence's visible rows, the static cost-line partition of a launch's tiles
// over CTAs, and the TMA boxes that copy runs of consecutive cache pages.
//
// What a sequence sees (Sec. 4.1, Alg. 2): in draft mode one query over cache
// rows 0 .. L - 1 followed by draft rows 0 .. nd - 1 of the draft scratch; in
// verify mode query j < n_q over cache rows 0 .. L + j.  Rows are handled in
// 16-token pages (the draft rows in one or two pages after the cache pages);
// 8 pages make a 128-row tile.
#pragma once

#include <cuda.h>

#include <cstdint>

#include "common.cuh"
#include "kernels.h"

namespace seedk {
namespace sched {
namespace {   // internal linkage: each kernel file has its own copy

constexpr int kTileRows = 128;                       // rows (tokens) per tile
constexpr int kPagesPerTile = kTileRows / kPage;     // 8
constexpr unsigned kFull = 0xffffffffu;

struct SeqT {
  int nq, nd, ncp, cvalid, lim0, tiles, bad;
};

// Pages that hold nd draft rows: rows 16 i .. 16 i + 15 of the draft scratch
// make draft page i, placed after the sequence's cache pages.
__device__ __forceinline__ int draft_pages(int nd) { return (nd + kPage - 1) / kPage; }

// Draft page held by page slot `slot` of tile t (-1: none), for a sequence
// with ncp cache pages and nd draft rows.
__device__ __forceinline__ int draft_page_of_slot(int ncp, int nd, int t, int slot) {
  const int dp = t * kPagesPerTile + slot - ncp;
  return (dp >= 0 && dp < draft_pages(nd)) ? dp : -1;
}

// Geometry of sequence b: query positions nq, draft rows nd, cache pages ncp,
// rows that exist cvalid, query j sees cache positions <= lim0 + j, tiles.
// A sequence with bad arguments (bad != 0) or no queries has no tiles.
__device__ __forceinline__ SeqT seq_of(const AttnTcParams& p, int b) {
  SeqT s{};
  const int L = p.ctx_lens[b];
  const int a = p.aux[b];
  const long long cap = (long long)p.max_pages * kPage;
  if (p.draft) {
    if (a < 0 || a > p.kmax) s.bad |= SEED_DEVERR_DRAFT_LEN;
    if (L < 0 || (long long)L > cap) s.bad |= SEED_DEVERR_CTX_LEN;
    if (s.bad || a == 0) return s;
    s.nq = 1;
    s.nd = a;
    s.cvalid = L;
    s.lim0 = L - 1;
    s.ncp = (L + kPage - 1) / kPage;
    s.tiles = (s.ncp + draft_pages(a) + kPagesPerTile - 1) / kPagesPerTile;
  } else {
    if (a < 0 || a > p.kmax + 1) s.bad |= SEED_DEVERR_NQ;
    if (L < 0 || (long long)L + a > cap) s.bad |= SEED_DEVERR_CTX_LEN;
    if (s.bad || a == 0) return s;
    s.nq = a;
    s.cvalid = L + a;
    s.lim0 = L;
    s.ncp = (s.cvalid + kPage - 1) / kPage;
    s.tiles = (s.ncp + kPagesPerTile - 1) / kPagesPerTile;
  }
  return s;
}

// ------------------------------------------------------------- partition
// The launch's work as a line of cost units: pair (b, g) with tiles(b) > 0
// takes kPairCost units for its fixed cost (descriptor and Q load, first-tile
// latency, epilogue), then one unit per tile; pairs in (b, g) order.  CTA c of
// N owns the units [start(c), start(c+1)) with start(c) = floor(c T / N) when
// T >= N, else min(c, T), and so the tiles whose units fall there: a
// contiguous run of pieces, and the CTAs holding one pair are consecutive.
constexpr int kPairCost = 2;
__device__ __forceinline__ long long range_start(long long T, int c, int N) {
  return T >= N ? T * c / N : min((long long)c, T);
}

// The CTA whose range holds unit x (0 <= x < T).
__device__ __forceinline__ int cta_of(long long x, long long T, int N) {
  return T >= N ? (int)(((x + 1) * N - 1) / T) : (int)x;
}

// Cost units of all pairs of sequence b.
__device__ __forceinline__ long long seq_cost(const AttnTcParams& p, int tiles) {
  return tiles > 0 ? (long long)p.hkv * (tiles + kPairCost) : 0;
}

// Warp-cooperative: T.
__device__ __noinline__ long long total_cost(const AttnTcParams& p, int lane) {
  long long tot = 0;
  for (int b = lane; b < p.B; b += 32) tot += seq_cost(p, seq_of(p, b).tiles);
  for (int o = 16; o; o >>= 1) tot += __shfl_xor_sync(kFull, tot, o);
  return tot;
}

// A window of 32 sequences [wb, wb + 32); lane i holds sequence wb + i.
struct SeqWin {
  int wb;
  SeqT mine;
};

__device__ __forceinline__ SeqT seq_or_empty(const AttnTcParams& p, int b) {
  return b < p.B ? seq_of(p, b) : SeqT{};
}

__device__ __forceinline__ SeqT win_get(const SeqWin& w, int b) {
  const int src = b - w.wb;
  SeqT s;
  s.nq = __shfl_sync(kFull, w.mine.nq, src);
  s.nd = __shfl_sync(kFull, w.mine.nd, src);
  s.ncp = __shfl_sync(kFull, w.mine.ncp, src);
  s.cvalid = __shfl_sync(kFull, w.mine.cvalid, src);
  s.lim0 = __shfl_sync(kFull, w.mine.lim0, src);
  s.tiles = __shfl_sync(kFull, w.mine.tiles, src);
  s.bad = 0;
  return s;
}

// Warp-cooperative: the pair (sequence b, KV head g) whose units hold unit
// x < T, the first unit pc of that pair, and the first tile t at or after x
// (0 when x falls in the pair's fixed-cost units); with the window that holds b.
__device__ __noinline__ void locate(const AttnTcParams& p, long long x, int lane, SeqWin& w,
                                    int& b, int& g, int& t, long long& pc) {
  long long base = 0;
  for (w.wb = 0; w.wb < p.B; w.wb += 32) {
    w.mine = seq_or_empty(p, w.wb + lane);
    const long long a = seq_cost(p, w.mine.tiles);
    long long inc = a;
    for (int o = 1; o < 32; o <<= 1) {
      const long long v = __shfl_up_sync(kFull, inc, o);
      if (lane >= o) inc += v;
    }
    const long long tot = __shfl_sync(kFull, inc, 31);
    if (x < base + tot) {
      const unsigned m = __ballot_sync(kFull, base + inc - a <= x && x < base + inc);
      const int src = __ffs(m) - 1;
      const long long sb = base + __shfl_sync(kFull, inc - a, src);
      const int per = __shfl_sync(kFull, w.mine.tiles, src) + kPairCost;
      b = w.wb + src;
      g = (int)((x - sb) / per);
      pc = sb + (long long)g * per;
      t = (int)max(0LL, x - pc - kPairCost);
      return;
    }
    base += tot;
  }
  b = p.B;
  g = t = 0;
  pc = 0;
}

// Warp-cooperative: this CTA's units [x, x1) of the T units of the launch, and
// (when x < x1) what locate() gives for x.  Up to 32 sequences the lengths
// are loaded once: the lanes keep their sequence's geometry from the total
// and find x in it; larger batches take total_cost() and locate().
__device__ __noinline__ void lookup_range(const AttnTcParams& p, int lane, long long& T,
                                          long long& x, long long& x1, SeqWin& w, int& b, int& g,
                                          int& t, long long& pc) {
  const int c = (int)blockIdx.x;
  b = p.B;
  g = t = 0;
  pc = 0;
  if (p.B > 32) {
    T = total_cost(p, lane);
    x = range_start(T, c, p.nctas);
    x1 = range_start(T, c + 1, p.nctas);
    if (x < x1) locate(p, x, lane, w, b, g, t, pc);
    return;
  }
  w.wb = 0;
  w.mine = seq_or_empty(p, lane);
  const long long a = seq_cost(p, w.mine.tiles);
  long long inc = a;
  for (int o = 1; o < 32; o <<= 1) {
    const long long v = __shfl_up_sync(kFull, inc, o);
    if (lane >= o) inc += v;
  }
  T = __shfl_sync(kFull, inc, 31);
  x = range_start(T, c, p.nctas);
  x1 = range_start(T, c + 1, p.nctas);
  if (x >= x1) return;
  const unsigned m = __ballot_sync(kFull, inc - a <= x && x < inc);
  const int src = __ffs(m) - 1;
  const long long sb = __shfl_sync(kFull, inc - a, src);
  const int per = __shfl_sync(kFull, w.mine.tiles, src) + kPairCost;
  b = src;
  g = (int)((x - sb) / per);
  pc = sb + (long long)g * per;
  t = (int)max(0LL, x - pc - kPairCost);
}

// Warp-cooperative: the next sequence after b with at least one tile (p.B if
// none), moving the window forward as needed.
__device__ __noinline__ void next_seq(const AttnTcParams& p, int lane, SeqWin& w, int& b) {
  for (;;) {
    const unsigned m = __ballot_sync(kFull, w.mine.tiles > 0 && w.wb + lane > b);
    if (m) {
      b = w.wb + __ffs(m) - 1;
      return;
    }
    w.wb += 32;
    if (w.wb >= p.B) {
      b = p.B;
      return;
    }
    w.mine = seq_or_empty(p, w.wb + lane);
  }
}

// Warp-cooperative: pull the launch's lengths (ctx_lens, aux) into L2, one
// 128-byte line per lane, so that the lookup after the dependency wait does
// not pay DRAM latency for them.
// A page table of at most 32 KiB is pulled in whole (the CTA's first pages
// are not known before the lookup), a larger one not at all.
__device__ __forceinline__ void prefetch_lens_l2(const AttnTcParams& p, int lane) {
  const int lines = (p.B * 4 + 127) / 128;
  for (int i = lane; i < 2 * lines; i += 32) {
    const int32_t* base = i < lines ? p.ctx_lens : p.aux;
    const int li = i < lines ? i : i - lines;
    asm volatile("prefetch.global.L2 [%0];" ::"l"(base + li * 32) : "memory");
  }
  const long long pt_bytes = (long long)p.B * p.max_pages * 4;
  if (pt_bytes <= 32768) {
    const int pl = (int)((pt_bytes + 127) / 128);
    for (int i = lane; i < pl; i += 32)
      asm volatile("prefetch.global.L2 [%0];" ::"l"(p.page_table + (size_t)i * 32) : "memory");
  }
}

// ------------------------------------------------------------- merge plan
// Entry c of the merge plan describes range boundary c (the first unit of
// CTA c's range, c >= 1): when that boundary splits the tiles of a pair
// (b, g) and is the first boundary to do so (CTA c - 1 holds the pair's first
// tile), the entry is {b, g, slot of the first piece's record, c - 1, number
// of pieces, query rows of the pair}; else b = -1.  CTA c writes it from the
// lookup of its own range start, so that the merge kernel finds its pair with
// one load instead of a scan of the cost line.  Lane 0 stores it; x, x1 are
// the CTA's units, (b, g, t0, pc) what locate() gave for x and sq the
// geometry of sequence b.
__device__ __forceinline__ void write_merge_plan(const AttnTcParams& p, long long T, long long x,
                                                 long long x1, int b, int g, int t0, long long pc,
                                                 const SeqT& sq) {
  const int c = (int)blockIdx.x;
  if (c == 0) return;
  int4 e0 = make_int4(-1, 0, 0, 0), e1 = make_int4(0, 0, 0, 0);
  if (x < x1 && b < p.B && t0 > 0) {
    const long long u0 = pc + kPairCost, u1 = u0 + sq.tiles - 1;
    const int c_lo = cta_of(u0, T, p.nctas);
    if (c_lo == c - 1) {
      const int c_hi = cta_of(u1, T, p.nctas);
      const int slot_lo = 2 * c_lo + (range_start(T, c_lo, p.nctas) >= pc ? 0 : 1);
      e0 = make_int4(b, g, slot_lo, c_lo);
      e1 = make_int4(c_hi - c_lo + 1, sq.nq * p.G, 0, 0);
    }
  }
  int4* dst = reinterpret_cast<int4*>(p.plan + (size_t)c * kPlanInts);
  dst[0] = e0;
  dst[1] = e1;
}

// ------------------------------------------------------------- page boxes
// Tensor maps of the paged cache for boxes of 1, 2, 4 and 8 consecutive pages
// (64 head dims x 16 rows x 1 KV head x n pages): n pages whose ids follow one
// another are one copy, and land as 16 n consecutive 128-byte rows, the
// swizzled K-major layout the MMAs read.
struct PageMaps {
  CUtensorMap k[4];
  CUtensorMap v[4];
};

// Warp-cooperative: the copy box that lane s < 8 issues for page slot s of a
// tile.  Runs of slots holding consecutive page ids are cut greedily into
// boxes of 8, 4, 2 and 1 pages; the result is the box size if slot s starts a
// box, else 0.  A slot at offset o of a run of n slots starts a box of
// 2^floor(log2(n - o)) pages exactly when n with the bits below that box size
// cleared equals o.
__device__ __forceinline__ int box_size(int pid, int lane) {
  const int pid_next = __shfl_down_sync(kFull, pid, 1);
  const uint32_t valid = __ballot_sync(kFull, lane < kPagesPerTile && pid >= 0) & 0xffu;
  const uint32_t cont =
      __ballot_sync(kFull, lane < kPagesPerTile - 1 && pid >= 0 && pid_next == pid + 1) & 0x7fu;
  if (lane >= kPagesPerTile || !((valid >> lane) & 1u)) return 0;
  const uint32_t starts = valid & ~(cont << 1) & 0xffu;
  const int r = 31 - __clz((int)(starts & ((2u << lane) - 1u)));   // first slot of the run
  const int n = lane + __ffs((int)~(cont >> lane)) - r;            // slots in the run
  const int o = lane - r;
  const int sz = 1 << (31 - __clz(n - o));
  return (n & ~(2 * sz - 1)) == o ? sz : 0;
}

__device__ __forceinline__ int log2_box(int sz) {
  return sz >= 8 ? 3 : sz >= 4 ? 2 : sz >= 2 ? 1 : 0;
}

}  // namespace
}  // namespace sched

// Host side (attn_tc.cu): 4-d bf16 tensor map with a 64-element (128-byte)
// innermost box and 128-byte swizzle.
bool encode_4d_bf16(CUtensorMap* map, const void* base, const cuuint64_t dims[4],
                    const cuuint64_t strides[3], const cuuint32_t box[4]);

// The merge kernel of split pairs (attn_tc.cu), for head_dim 64 or 128.
cudaError_t launch_attn_merge(const AttnTcParams& p, int head_dim, cudaStream_t st);

}  // namespace seedk
