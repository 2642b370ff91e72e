// Split-KV flash-decoding attention on CUDA cores: the draft step and (for
// now) the verify step of SEED's decode loop.
//
// What it computes (Sec. 4.1: the drafter attends to the cached deep KV with
// ordinary self-attention; Alg. 2 fixes the visible rows): for a virtual
// sequence v and query head h, softmax(scale * q K^T) V over
//   draft  (v = b):           cache rows 0..ctx_len-1, then draft rows
//                             0..draft_len-1 of the draft scratch;
//   verify (v = b*(kmax+1)+j): cache rows 0..ctx_len+j (causal among the
//                             k+1 new rows, which the cache already holds).
//
// Work decomposition.  The rows of (v, KV head g) are split into units of
// `ppu` 16-token pages; a persistent grid of 2 CTAs per SM walks the units.
// Each CTA (4 warps) streams its unit's pages through a 3-stage TMA bulk-copy
// ring (one page of K and one of V per warp per stage, 4 KiB each at D=128),
// and each warp works on its page with the G query heads of the group packed
// together (GQA head packing: every K/V byte in shared memory feeds G heads).
// Inside a warp, eight lanes ("an octet") share one token: each lane holds 16
// of the 128 head dimensions, so the 8 lanes read the 256-byte row
// conflict-free and the dot product closes with three xor-shuffles.  Scores
// are kept in log2 units (q pre-scaled by scale*log2 e) and the online softmax
// rescales its accumulator only when the running maximum grows by more than
// 2^8 (values stay far inside fp32 range).  Units of the same (v, g) leave a
// normalised partial and its log-sum-exp in the workspace; the last one to
// finish (arrival counter) merges them in fixed unit order, so results are
// deterministic and do not depend on the physical page order.
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace seedk {
namespace {

constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;
constexpr int kTilePages = kWarps;   // one page per warp per stage
constexpr int kStages = 3;
constexpr float kRescale = 8.0f;     // log2 units the reference max may lag
constexpr float kLn2 = 0.69314718055994531f;
constexpr unsigned kFull = 0xffffffffu;
static_assert(kPage == kPageTokens, "page size");

struct Seq {
  int b;
  int nctx;    // rows read from the paged cache
  int ndraft;  // rows read from the draft scratch
  int npages;  // context pages, plus one for the draft rows
  int bad;     // SEED_DEVERR_* bits of this sequence's arguments
};

__device__ __forceinline__ Seq load_seq(const DecodeParams& p, int v) {
  Seq s{};
  if (p.verify) {
    s.b = v / p.nq_per_seq;
    const int j = v - s.b * p.nq_per_seq;
    const int L = p.ctx_lens[s.b];
    const int nq = p.aux[s.b];
    if (nq < 0 || nq > p.kmax + 1) s.bad |= SEED_DEVERR_NQ;
    if (L < 0 || (long long)L + nq > (long long)p.max_pages * kPage) s.bad |= SEED_DEVERR_CTX_LEN;
    if (s.bad || j >= nq) return s;
    s.nctx = L + j + 1;
  } else {
    s.b = v;
    const int L = p.ctx_lens[v];
    const int dl = p.aux[v];
    if (dl < 0 || dl > p.kmax) s.bad |= SEED_DEVERR_DRAFT_LEN;
    if (L < 0 || (long long)L > (long long)p.max_pages * kPage) s.bad |= SEED_DEVERR_CTX_LEN;
    if (s.bad || dl == 0) return s;
    s.nctx = L;
    s.ndraft = dl;
  }
  // the draft rows fill one or two pages after the cache pages
  s.npages = (s.nctx + kPage - 1) / kPage + (s.ndraft + kPage - 1) / kPage;
  return s;
}

struct Cursor {
  int u;               // dense unit index; >= n_units once exhausted
  int v, g, c;
  Seq s;
  int page0, page1;    // pages [page0, page1) of the sequence
  int tile, ntiles;
};

__device__ __forceinline__ bool unit_at(const DecodeParams& p, int u, Cursor& cu, bool report) {
  const int per_v = p.hkv * p.cmax;
  cu.v = u / per_v;
  const int r = u - cu.v * per_v;
  cu.g = r / p.cmax;
  cu.c = r - cu.g * p.cmax;
  cu.s = load_seq(p, cu.v);
  if (report && cu.s.bad && cu.c == 0 && cu.g == 0 && threadIdx.x == 0) raise_err(p.err, cu.s.bad);
  cu.page0 = cu.c * p.ppu;
  if (cu.page0 >= cu.s.npages) return false;
  cu.page1 = min(cu.page0 + p.ppu, cu.s.npages);
  cu.ntiles = (cu.page1 - cu.page0 + kTilePages - 1) / kTilePages;
  cu.tile = 0;
  return true;
}

__device__ __forceinline__ void seek(const DecodeParams& p, Cursor& cu, int u_from, bool report) {
  for (int u = u_from; u < p.n_units; u += gridDim.x) {
    if (unit_at(p, u, cu, report)) {
      cu.u = u;
      return;
    }
  }
  cu.u = p.n_units;
}

__device__ __forceinline__ void advance(const DecodeParams& p, Cursor& cu, bool report) {
  if (++cu.tile < cu.ntiles) return;
  seek(p, cu, cu.u + gridDim.x, report);
}

__device__ __forceinline__ int ctx_pages(const Seq& s) { return (s.nctx + kPage - 1) / kPage; }

// Valid rows of page `pg` of the sequence (0 if its page id is out of range).
__device__ __forceinline__ int page_rows(const DecodeParams& p, const Seq& s, int pg, int* pid_out) {
  if (pg < ctx_pages(s)) {
    const int pid = p.page_table[(size_t)s.b * p.max_pages + pg];
    *pid_out = pid;
    if (pid < 0 || pid >= p.num_pages) return 0;
    return min(kPage, s.nctx - pg * kPage);
  }
  *pid_out = -1;
  return min(kPage, s.ndraft - (pg - ctx_pages(s)) * kPage);   // draft page pg - ctx_pages
}

// Producer: one thread puts the K and V pages of the cursor's current tile
// into stage `stage` of the ring.
template <int D>
__device__ void issue_tile(const DecodeParams& p, const Cursor& cu, int stage, uint16_t* kbuf,
                           uint16_t* vbuf, uint64_t* full, uint64_t pol) {
  const uint16_t* src_k[kTilePages];
  const uint16_t* src_v[kTilePages];
  uint32_t bytes[kTilePages];
  uint32_t total = 0;
#pragma unroll
  for (int w = 0; w < kTilePages; ++w) {
    bytes[w] = 0;
    src_k[w] = src_v[w] = nullptr;
    const int pg = cu.page0 + cu.tile * kTilePages + w;
    if (pg >= cu.page1) continue;
    int pid;
    const int rows = page_rows(p, cu.s, pg, &pid);
    if (pid >= 0) {
      if (rows == 0) {
        raise_err(p.err, SEED_DEVERR_PAGE);
        continue;
      }
      const size_t off = ((size_t)pid * p.hkv + cu.g) * kPage * D;
      src_k[w] = p.k_cache + off;
      src_v[w] = p.v_cache + off;
      bytes[w] = kPage * D * 2;   // whole page; rows past the length are masked
    } else {
      const size_t off =
          (((size_t)cu.s.b * p.hkv + cu.g) * p.kmax + (size_t)(pg - ctx_pages(cu.s)) * kPage) * D;
      src_k[w] = p.draft_k + off;
      src_v[w] = p.draft_v + off;
      bytes[w] = (uint32_t)rows * D * 2;
    }
    total += 2 * bytes[w];
  }
  mbar_arrive_expect_tx(&full[stage], total);
#pragma unroll
  for (int w = 0; w < kTilePages; ++w) {
    if (bytes[w] == 0) continue;
    const size_t slot = ((size_t)stage * kTilePages + w) * kPage * D;
    bulk_g2s(kbuf + slot, src_k[w], bytes[w], &full[stage], pol);
    bulk_g2s(vbuf + slot, src_v[w], bytes[w], &full[stage], pol);
  }
}

template <int D, int G>
__device__ __forceinline__ void consume_page(const uint16_t* __restrict__ kb,
                                             const uint16_t* __restrict__ vb, int rows,
                                             const float (&q)[G][D / 8], float (&o)[G][D / 8],
                                             float (&m)[G], float (&l)[G], int lane) {
  constexpr int CH = D / 64;   // 16-byte chunks per lane
  constexpr int E = D / 8;     // head dims per lane
  const int oct = lane >> 3, sub = lane & 7;
  float s[G][4];
#pragma unroll
  for (int ps = 0; ps < 4; ++ps) {
    const int t = ps * 4 + oct;
    float kf[E];
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const uint4 u = *reinterpret_cast<const uint4*>(kb + t * D + (sub + 8 * c) * 8);
      unpack8(u, kf + 8 * c);
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float a = 0.f;
#pragma unroll
      for (int e = 0; e < E; ++e) a = fmaf(q[h][e], kf[e], a);
      s[h][ps] = a;
    }
  }
#pragma unroll
  for (int h = 0; h < G; ++h)
#pragma unroll
    for (int ps = 0; ps < 4; ++ps) {
      s[h][ps] += __shfl_xor_sync(kFull, s[h][ps], 1);
      s[h][ps] += __shfl_xor_sync(kFull, s[h][ps], 2);
      s[h][ps] += __shfl_xor_sync(kFull, s[h][ps], 4);
    }
  bool valid[4];
#pragma unroll
  for (int ps = 0; ps < 4; ++ps) valid[ps] = (ps * 4 + oct) < rows;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    float mt = -INFINITY;
#pragma unroll
    for (int ps = 0; ps < 4; ++ps)
      if (valid[ps]) mt = fmaxf(mt, s[h][ps]);
    if (mt > m[h] + kRescale) {
      const float f = exp2f(m[h] - mt);
      l[h] *= f;
#pragma unroll
      for (int e = 0; e < E; ++e) o[h][e] *= f;
      m[h] = mt;
    }
#pragma unroll
    for (int ps = 0; ps < 4; ++ps) {
      s[h][ps] = valid[ps] ? exp2f(s[h][ps] - m[h]) : 0.f;
      l[h] += s[h][ps];
    }
  }
#pragma unroll
  for (int ps = 0; ps < 4; ++ps) {
    if (!valid[ps]) continue;   // rows past the length may hold anything (NaN)
    const int t = ps * 4 + oct;
    float vf[E];
#pragma unroll
    for (int c = 0; c < CH; ++c) {
      const uint4 u = *reinterpret_cast<const uint4*>(vb + t * D + (sub + 8 * c) * 8);
      unpack8(u, vf + 8 * c);
    }
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
      for (int e = 0; e < E; ++e) o[h][e] = fmaf(s[h][ps], vf[e], o[h][e]);
  }
}

// Merge the 16 octet states of the CTA into the unit's result; write it out
// directly (single-unit rows) or as a partial, and let the last unit of the
// (v, g) pair merge all partials.
template <int D, int G>
__device__ void finish_unit(const DecodeParams& p, const Cursor& cu, float (&o)[G][D / 8],
                            float (&m)[G], float (&l)[G], float* scratch, int* s_last) {
  constexpr int CH = D / 64;
  constexpr int E = D / 8;
  constexpr int REC = G * D + G;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int oct = lane >> 3, sub = lane & 7;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    float mw = fmaxf(m[h], __shfl_xor_sync(kFull, m[h], 8));
    mw = fmaxf(mw, __shfl_xor_sync(kFull, mw, 16));
    const float f = (m[h] == -INFINITY) ? 0.f : exp2f(m[h] - mw);
    float lw = l[h] * f;
    lw += __shfl_xor_sync(kFull, lw, 8);
    lw += __shfl_xor_sync(kFull, lw, 16);
#pragma unroll
    for (int e = 0; e < E; ++e) {
      float x = o[h][e] * f;
      x += __shfl_xor_sync(kFull, x, 8);
      x += __shfl_xor_sync(kFull, x, 16);
      o[h][e] = x;
    }
    m[h] = mw;
    l[h] = lw;
  }
  float* so = scratch;                     // [warp][G][D]
  float* sm = scratch + kWarps * G * D;    // [warp][G]
  float* sl = sm + kWarps * G;             // [warp][G]
  if (oct == 0) {
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
      for (int c = 0; c < CH; ++c)
#pragma unroll
        for (int e = 0; e < 8; ++e) so[(warp * G + h) * D + (sub + 8 * c) * 8 + e] = o[h][8 * c + e];
  }
  if (lane == 0) {
#pragma unroll
    for (int h = 0; h < G; ++h) {
      sm[warp * G + h] = m[h];
      sl[warp * G + h] = l[h];
    }
  }
  __syncthreads();

  const int nu = (cu.s.npages + p.ppu - 1) / p.ppu;
  const int pair = cu.v * p.hkv + cu.g;
  float* rec = p.part + (size_t)cu.u * REC;
  for (int idx = tid; idx < G * D; idx += kThreads) {
    const int h = idx / D, d = idx - h * D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm[w * G + h]);
    float Ls = 0.f, Os = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float mw = sm[w * G + h];
      const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
      Ls = fmaf(sl[w * G + h], f, Ls);
      Os = fmaf(so[(w * G + h) * D + d], f, Os);
    }
    const float of = Os / Ls;
    const float lse2 = M + log2f(Ls);
    const int hh = cu.g * G + h;
    if (nu == 1) {
      p.out[((size_t)cu.v * p.hq + hh) * D + d] = of;
      if (d == 0 && p.lse != nullptr) p.lse[(size_t)cu.v * p.hq + hh] = lse2 * kLn2;
    } else {
      rec[idx] = of;
      if (d == 0) rec[G * D + h] = lse2;
    }
  }
  if (nu > 1) {
    __threadfence();
    __syncthreads();
    if (tid == 0) *s_last = (atomicAdd(&p.counters[pair], 1) == nu - 1);
    __syncthreads();
    if (*s_last) {
      __threadfence();
      const float* base = p.part + (size_t)pair * p.cmax * REC;
      for (int idx = tid; idx < G * D; idx += kThreads) {
        const int h = idx / D, d = idx - h * D;
        float M = -INFINITY;
        for (int c = 0; c < nu; ++c) M = fmaxf(M, __ldcg(base + (size_t)c * REC + G * D + h));
        float S = 0.f, O = 0.f;
        for (int c = 0; c < nu; ++c) {
          const float w = exp2f(__ldcg(base + (size_t)c * REC + G * D + h) - M);
          S += w;
          O = fmaf(w, __ldcg(base + (size_t)c * REC + idx), O);
        }
        const int hh = cu.g * G + h;
        p.out[((size_t)cu.v * p.hq + hh) * D + d] = O / S;
        if (d == 0 && p.lse != nullptr) p.lse[(size_t)cu.v * p.hq + hh] = (M + log2f(S)) * kLn2;
      }
      if (tid == 0) p.counters[pair] = 0;
    }
  }
  __syncthreads();
}

template <int D, int G>
__global__ void __launch_bounds__(kThreads, 2) decode_attn_kernel(const DecodeParams p) {
  constexpr int E = D / 8;
  constexpr int CH = D / 64;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t full[kStages];
  __shared__ __align__(8) uint64_t empty[kStages];
  __shared__ int s_last;

  uint16_t* kbuf = reinterpret_cast<uint16_t*>(smem);
  uint16_t* vbuf = kbuf + (size_t)kStages * kTilePages * kPage * D;
  float* scratch = reinterpret_cast<float*>(vbuf + (size_t)kStages * kTilePages * kPage * D);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int sub = lane & 7;

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kWarps);
    }
    fence_mbar_init();
  }
  __syncthreads();

  uint64_t pol = 0;
  if (tid == 0) pol = p.verify ? policy_evict_normal() : policy_evict_first();

  Cursor cons, prod;
  seek(p, cons, blockIdx.x, true);
  prod = cons;
  if (tid == 0) {
    for (int s = 0; s < kStages && prod.u < p.n_units; ++s) {
      issue_tile<D>(p, prod, s, kbuf, vbuf, full, pol);
      advance(p, prod, false);
    }
  }

  float q[G][E], o[G][E], m[G], l[G];
  bool timed_out = false;
  for (int it = 0; cons.u < p.n_units; ++it) {
    if (cons.tile == 0) {
      const uint16_t* qp = p.q + ((size_t)cons.v * p.hq + cons.g * G) * D;
#pragma unroll
      for (int h = 0; h < G; ++h) {
#pragma unroll
        for (int c = 0; c < CH; ++c) {
          const uint4 u = __ldg(reinterpret_cast<const uint4*>(qp + h * D + (sub + 8 * c) * 8));
          unpack8(u, &q[h][8 * c]);
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
          q[h][e] *= p.scale_log2;
          o[h][e] = 0.f;
        }
        m[h] = -INFINITY;
        l[h] = 0.f;
      }
    }
    const int s = it % kStages;
    const uint32_t ph = (uint32_t)(it / kStages) & 1u;
    if (!timed_out && !mbar_wait(&full[s], ph)) timed_out = true;

    const int pg = cons.page0 + cons.tile * kTilePages + warp;
    if (!timed_out && pg < cons.page1) {
      int pid;
      const int rows = page_rows(p, cons.s, pg, &pid);
      if (rows > 0) {
        const size_t slot = ((size_t)s * kTilePages + warp) * kPage * D;
        consume_page<D, G>(kbuf + slot, vbuf + slot, rows, q, o, m, l, lane);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
    if (tid == 0 && prod.u < p.n_units) {
      if (!timed_out && !mbar_wait(&empty[s], ph)) timed_out = true;
      if (!timed_out) issue_tile<D>(p, prod, s, kbuf, vbuf, full, pol);
      advance(p, prod, false);
    }
    const bool last_tile = (cons.tile == cons.ntiles - 1);
    if (last_tile) finish_unit<D, G>(p, cons, o, m, l, scratch, &s_last);
    advance(p, cons, true);
  }
  if (timed_out) raise_err(p.err, SEED_DEVERR_TIMEOUT);
}

std::atomic<uint64_t> g_smem_set[8];   // per instantiation: devices configured

template <int D, int G>
constexpr size_t smem_bytes() {
  return (size_t)2 * kStages * kTilePages * kPage * D * 2 + (size_t)kWarps * G * (D + 2) * 4;
}

template <int D, int G>
cudaError_t launch_t(const DecodeParams& p, int slot, cudaStream_t st) {
  constexpr size_t smem = smem_bytes<D, G>();
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(g_smem_set[slot].load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(decode_attn_kernel<D, G>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    g_smem_set[slot].fetch_or(bit, std::memory_order_acq_rel);
  }
  const int grid = std::min(p.n_units, 2 * device_sm_count());
  if (grid <= 0) return cudaSuccess;
  decode_attn_kernel<D, G><<<grid, kThreads, smem, st>>>(p);
  return cudaGetLastError();
}

}  // namespace

DecodePlan plan_decode(int32_t nv, int32_t hkv, int32_t group, int32_t head_dim,
                       int32_t max_pages) {
  DecodePlan pl{};
  pl.nv = nv;
  const long long pages_cap = (long long)max_pages + 2;   // + up to two draft pages
  const long long total = (long long)nv * hkv * pages_cap;
  long long ppu = 4 * ((total + 4LL * kTargetUnits - 1) / (4LL * kTargetUnits));
  if (ppu < 4) ppu = 4;
  pl.ppu = (int32_t)ppu;
  pl.cmax = (int32_t)((pages_cap + ppu - 1) / ppu);
  pl.n_units = nv * hkv * pl.cmax;
  pl.part_bytes = (size_t)pl.n_units * (group * head_dim + group) * 4;
  return pl;
}

size_t decode_workspace_bound(int32_t nv_max, int32_t hkv, int32_t group, int32_t head_dim) {
  return ((size_t)kTargetUnits + (size_t)nv_max * hkv) * (group * head_dim + group) * 4;
}

int device_sm_count() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  int v = cache[dev & 63].load(std::memory_order_relaxed);
  if (v > 0) return v;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
    v = 1;
  cache[dev & 63].store(v, std::memory_order_relaxed);
  return v;
}

cudaError_t launch_decode(const DecodeParams& p, int head_dim, int group, cudaStream_t st) {
  if (head_dim == 128) {
    switch (group) {
      case 1: return launch_t<128, 1>(p, 0, st);
      case 2: return launch_t<128, 2>(p, 1, st);
      case 4: return launch_t<128, 4>(p, 2, st);
      case 8: return launch_t<128, 8>(p, 3, st);
    }
  } else if (head_dim == 64) {
    switch (group) {
      case 1: return launch_t<64, 1>(p, 4, st);
      case 2: return launch_t<64, 2>(p, 5, st);
      case 4: return launch_t<64, 4>(p, 6, st);
      case 8: return launch_t<64, 8>(p, 7, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace seedk
