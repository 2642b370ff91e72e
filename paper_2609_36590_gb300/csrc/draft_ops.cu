// The small steps of a draft step (Sec. 4.1 drafting through the model's last
// layers): the raw token embedding, RMS norms, the per-head q/k norms with the
// rotary position embedding, and an f32 -> bf16 conversion of the attention
// output.  All are a few KB to a few hundred KB per call and bound by launch
// latency; each is launched as a programmatic dependent of the kernel before
// it and waits for it before reading.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "kernels.h"

namespace seedk {
namespace {

constexpr int kOpsThreads = 256;

__device__ __forceinline__ float block_sum(float v, float* sh) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0) sh[w] = v;
  __syncthreads();
  float t = l < (int)(blockDim.x >> 5) ? sh[l] : 0.f;
#pragma unroll
  for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  __syncthreads();
  return t;
}

// x[b] = W_emb[tokens[b]] (bf16 -> f32).  One block per sequence; 8-byte
// loads (d is a multiple of 4).
__global__ void __launch_bounds__(kOpsThreads) embed_kernel(int32_t d, int32_t vocab,
                                                            const int32_t* tokens,
                                                            const __nv_bfloat16* w, float* x,
                                                            int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int tok = tokens[b];
  if (tok < 0 || tok >= vocab) {
    if (threadIdx.x == 0) raise_err(err, SEED_DEVERR_TOKEN);
    return;
  }
  const uint2* row = reinterpret_cast<const uint2*>(w + (size_t)tok * d);
  float4* out = reinterpret_cast<float4*>(x + (size_t)b * d);
  for (int i = threadIdx.x; i < d / 4; i += blockDim.x) {
    const uint2 v = row[i];
    out[i] = make_float4(__uint_as_float(v.x << 16), __uint_as_float(v.x & 0xffff0000u),
                         __uint_as_float(v.y << 16), __uint_as_float(v.y & 0xffff0000u));
  }
}

// y[b] = bf16(x[b] / sqrt(mean(x[b]^2) + eps) * gamma).  One block per row;
// a row of up to 4 * 4 * 256 floats stays in registers between the two
// passes (longer rows read x twice).  n is a multiple of 4.
constexpr int kNormVec = 4;                   // float4 per thread kept in registers
__global__ void __launch_bounds__(kOpsThreads) rmsnorm_kernel(int32_t n, const float* x,
                                                              const __nv_bfloat16* gamma,
                                                              float eps, __nv_bfloat16* y) {
  __shared__ float sh[kOpsThreads / 32];
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)blockIdx.x * n);
  const int n4 = n / 4;
  float4 v[kNormVec];
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < kNormVec; ++j) {
    const int i = threadIdx.x + j * kOpsThreads;
    v[j] = i < n4 ? xr[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
#pragma unroll
  for (int j = 0; j < kNormVec; ++j)
    ss += v[j].x * v[j].x + v[j].y * v[j].y + v[j].z * v[j].z + v[j].w * v[j].w;
  for (int i = threadIdx.x + kNormVec * kOpsThreads; i < n4; i += kOpsThreads) {
    const float4 u = xr[i];
    ss += u.x * u.x + u.y * u.y + u.z * u.z + u.w * u.w;
  }
  const float r = rsqrtf(block_sum(ss, sh) / (float)n + eps);
  const uint2* gr = reinterpret_cast<const uint2*>(gamma);
  uint2* yr = reinterpret_cast<uint2*>(y + (size_t)blockIdx.x * n);
  auto put = [&](int i, float4 u) {
    const uint2 g = gr[i];
    const float2 lo = make_float2(u.x * r * __uint_as_float(g.x << 16),
                                  u.y * r * __uint_as_float(g.x & 0xffff0000u));
    const float2 hi = make_float2(u.z * r * __uint_as_float(g.y << 16),
                                  u.w * r * __uint_as_float(g.y & 0xffff0000u));
    const __nv_bfloat162 a = __float22bfloat162_rn(lo), c = __float22bfloat162_rn(hi);
    yr[i] = make_uint2(*reinterpret_cast<const uint32_t*>(&a), *reinterpret_cast<const uint32_t*>(&c));
  };
#pragma unroll
  for (int j = 0; j < kNormVec; ++j) {
    const int i = threadIdx.x + j * kOpsThreads;
    if (i < n4) put(i, v[j]);
  }
  for (int i = threadIdx.x + kNormVec * kOpsThreads; i < n4; i += kOpsThreads) put(i, xr[i]);
}

// From qkv f32 [B, (hq + 2 hkv) D]: q, k normed per head (gain g_q / g_k) and
// rotated (rotate-half pairs (i, i + D/2), angle pos * theta^(-2i/D)); v
// copied; all three rounded to bf16.  q goes to q [B, hq, D]; k and v go
// straight to row draft_len - 1 of the layer's draft scratch [B, hkv, kmax,
// D] (the draft KV append of this step).  pos = ctx_len + draft_len - 1: the
// position of the token this draft step feeds.  One warp per (sequence,
// head).  The frequencies theta^(-2i/D) come from the host in double; each
// lane forms its angle pos * w in double and reduces it by 2 pi (split in two
// doubles) before a single-precision sincos, so positions of 10^6 and more
// keep their angles to ~1e-10 rad.
constexpr int kRopeWarps = 8;
struct RopeFreq {
  double w[64];
};
__global__ void __launch_bounds__(kRopeWarps * 32) qk_norm_rope_kernel(
    int32_t hq, int32_t hkv, int32_t D, const float* qkv, const __nv_bfloat16* gq,
    const __nv_bfloat16* gk, const int32_t* ctx_lens, const int32_t* draft_lens,
    const RopeFreq fr, float eps, int32_t kmax, __nv_bfloat16* q, __nv_bfloat16* dk,
    __nv_bfloat16* dv, int32_t* err) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nh = hq + 2 * hkv;
  const int h = blockIdx.y * kRopeWarps + warp;
  if (h >= nh) return;
  const int dl = draft_lens[b];
  if (dl <= 0) return;                        // skipped sequence
  if (dl > kmax) {
    if (lane == 0) raise_err(err, SEED_DEVERR_DRAFT_LEN);
    return;
  }
  const float* xh = qkv + ((size_t)b * nh + h) * D;
  const int half = D / 2;                     // 32 or 64: one or two pairs per lane
  if (h >= hq + hkv) {                        // v: copy
    __nv_bfloat16* dst = dv + (((size_t)b * hkv + (h - hq - hkv)) * kmax + dl - 1) * D;
    for (int i = lane; i < D; i += 32) dst[i] = __float2bfloat16_rn(xh[i]);
    return;
  }
  const bool isq = h < hq;
  const __nv_bfloat16* g = isq ? gq : gk;
  __nv_bfloat16* dst = isq ? q + ((size_t)b * hq + h) * D
                            : dk + (((size_t)b * hkv + (h - hq)) * kmax + dl - 1) * D;
  const int np = half / 32;                   // pairs per lane
  float a[2], c[2];
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    if (j < np) {
      a[j] = xh[lane + 32 * j];
      c[j] = xh[lane + 32 * j + half];
      ss = fmaf(a[j], a[j], fmaf(c[j], c[j], ss));
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float r = rsqrtf(ss / (float)D + eps);
  const double pos = (double)((long long)ctx_lens[b] + dl - 1);
  constexpr double kTwoPiHi = 6.283185307179586, kTwoPiLo = 2.4492935982947064e-16;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    if (j < np) {
      const int i = lane + 32 * j;
      const double ang = pos * fr.w[i];
      const double m = rint(ang * (1.0 / kTwoPiHi));
      const float red = (float)fma(-m, kTwoPiLo, fma(-m, kTwoPiHi, ang));
      float sn, cs;
      sincosf(red, &sn, &cs);
      const float x0 = a[j] * r * __bfloat162float(g[i]);
      const float x1 = c[j] * r * __bfloat162float(g[i + half]);
      dst[i] = __float2bfloat16_rn(x0 * cs - x1 * sn);
      dst[i + half] = __float2bfloat16_rn(x1 * cs + x0 * sn);
    }
  }
}

__global__ void __launch_bounds__(kOpsThreads) f32_to_bf16_kernel(size_t n, const float* x,
                                                                  __nv_bfloat16* y) {
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (size_t)gridDim.x * blockDim.x)
    y[i] = __float2bfloat16_rn(x[i]);
}

}  // namespace

cudaError_t launch_embed(int32_t B, int32_t d, int32_t vocab, const int32_t* tokens,
                         const void* w, float* x, int32_t* err, cudaStream_t st) {
  return launch_pdl(embed_kernel, dim3(B), dim3(kOpsThreads), 0, st, d, vocab, tokens,
                    static_cast<const __nv_bfloat16*>(w), x, err);
}

cudaError_t launch_rmsnorm(int32_t rows, int32_t n, const float* x, const void* gamma, float eps,
                           void* y, cudaStream_t st) {
  return launch_pdl(rmsnorm_kernel, dim3(rows), dim3(kOpsThreads), 0, st, n, x,
                    static_cast<const __nv_bfloat16*>(gamma), eps,
                    static_cast<__nv_bfloat16*>(y));
}

cudaError_t launch_qk_norm_rope(int32_t B, int32_t hq, int32_t hkv, int32_t D, const float* qkv,
                                const void* gq, const void* gk, const int32_t* ctx_lens,
                                const int32_t* draft_lens, float theta, float eps, int32_t kmax,
                                void* q, void* draft_k, void* draft_v, int32_t* err,
                                cudaStream_t st) {
  RopeFreq fr{};
  for (int i = 0; i < D / 2 && i < 64; ++i) fr.w[i] = std::pow((double)theta, -2.0 * i / D);
  const dim3 grid(B, (hq + 2 * hkv + kRopeWarps - 1) / kRopeWarps);
  return launch_pdl(qk_norm_rope_kernel, grid, dim3(kRopeWarps * 32), 0, st, hq, hkv, D, qkv,
                    static_cast<const __nv_bfloat16*>(gq), static_cast<const __nv_bfloat16*>(gk),
                    ctx_lens, draft_lens, fr, eps, kmax, static_cast<__nv_bfloat16*>(q),
                    static_cast<__nv_bfloat16*>(draft_k), static_cast<__nv_bfloat16*>(draft_v), err);
}

cudaError_t launch_f32_to_bf16(size_t n, const float* x, void* y, cudaStream_t st) {
  const int grid = (int)std::min<size_t>((n + kOpsThreads - 1) / kOpsThreads, 1024);
  return launch_pdl(f32_to_bf16_kernel, dim3(grid > 0 ? grid : 1), dim3(kOpsThreads), 0, st, n, x,
                    static_cast<__nv_bfloat16*>(y));
}

}  // namespace seedk
