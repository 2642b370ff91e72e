// The small steps of a draft step (Sec. 4.1 drafting through the model's last
// layers): the raw token embedding, RMS norms, the per-head q/k norms with the
// rotary position embedding, and an f32 -> bf16 conversion of the attention
// output.  All are a few KB to a few hundred KB per call and bound by launch
// latency; each is launched as a programmatic dependent of the kernel before
// it and waits for it before reading.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>

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

// x[b] = W_emb[tokens[b]] (bf16 -> f32).  One block per sequence.
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
  const __nv_bfloat16* row = w + (size_t)tok * d;
  for (int i = threadIdx.x; i < d; i += blockDim.x)
    x[(size_t)b * d + i] = __bfloat162float(row[i]);
}

// y[b] = bf16(x[b] / sqrt(mean(x[b]^2) + eps) * gamma).  One block per row.
__global__ void __launch_bounds__(kOpsThreads) rmsnorm_kernel(int32_t n, const float* x,
                                                              const __nv_bfloat16* gamma,
                                                              float eps, __nv_bfloat16* y) {
  __shared__ float sh[kOpsThreads / 32];
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const float* xr = x + (size_t)blockIdx.x * n;
  float ss = 0.f;
  for (int i = threadIdx.x; i < n; i += blockDim.x) ss = fmaf(xr[i], xr[i], ss);
  const float r = rsqrtf(block_sum(ss, sh) / (float)n + eps);
  __nv_bfloat16* yr = y + (size_t)blockIdx.x * n;
  for (int i = threadIdx.x; i < n; i += blockDim.x)
    yr[i] = __float2bfloat16_rn(xr[i] * r * __bfloat162float(gamma[i]));
}

// From qkv f32 [B, (hq + 2 hkv) D]: q, k normed per head (gain g_q / g_k) and
// rotated (rotate-half pairs (i, i + D/2), angle pos * theta^(-2i/D)); v
// copied; all three rounded to bf16.  pos = ctx_len + draft_len - 1: the
// position of the token this draft step feeds.  One block per sequence; the
// angles are reduced in double precision (positions reach 10^5 and more).
__global__ void __launch_bounds__(kOpsThreads) qk_norm_rope_kernel(
    int32_t hq, int32_t hkv, int32_t D, const float* qkv, const __nv_bfloat16* gq,
    const __nv_bfloat16* gk, const int32_t* ctx_lens, const int32_t* draft_lens, float theta,
    float eps, __nv_bfloat16* q, __nv_bfloat16* k, __nv_bfloat16* v) {
  __shared__ float cs[64], sn[64];
  if (threadIdx.x == 0) pdl_trigger();
  pdl_wait();
  const int b = blockIdx.x;
  const int dl = draft_lens[b];
  if (dl <= 0) return;                        // skipped sequence
  const long long pos = (long long)ctx_lens[b] + dl - 1;
  const int half = D / 2;
  for (int i = threadIdx.x; i < half; i += blockDim.x) {
    const double inv = exp(-(2.0 * i / D) * log((double)theta));
    double s, c;
    sincos((double)pos * inv, &s, &c);
    cs[i] = (float)c;
    sn[i] = (float)s;
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nh = hq + 2 * hkv;
  const float* src = qkv + (size_t)b * nh * D;
  for (int h = warp; h < nh; h += blockDim.x >> 5) {
    const float* xh = src + (size_t)h * D;
    if (h >= hq + hkv) {                      // v: copy
      __nv_bfloat16* dst = v + ((size_t)b * hkv + (h - hq - hkv)) * D;
      for (int i = lane; i < D; i += 32) dst[i] = __float2bfloat16_rn(xh[i]);
      continue;
    }
    const bool isq = h < hq;
    const __nv_bfloat16* g = isq ? gq : gk;
    __nv_bfloat16* dst = isq ? q + ((size_t)b * hq + h) * D : k + ((size_t)b * hkv + (h - hq)) * D;
    float ss = 0.f;
    for (int i = lane; i < D; i += 32) ss = fmaf(xh[i], xh[i], ss);
#pragma unroll
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const float r = rsqrtf(ss / (float)D + eps);
    for (int i = lane; i < half; i += 32) {
      const float a = xh[i] * r * __bfloat162float(g[i]);
      const float c = xh[i + half] * r * __bfloat162float(g[i + half]);
      dst[i] = __float2bfloat16_rn(a * cs[i] - c * sn[i]);
      dst[i + half] = __float2bfloat16_rn(c * cs[i] + a * sn[i]);
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
                                const int32_t* draft_lens, float theta, float eps, void* q,
                                void* k, void* v, cudaStream_t st) {
  return launch_pdl(qk_norm_rope_kernel, dim3(B), dim3(kOpsThreads), 0, st, hq, hkv, D, qkv,
                    static_cast<const __nv_bfloat16*>(gq), static_cast<const __nv_bfloat16*>(gk),
                    ctx_lens, draft_lens, theta, eps, static_cast<__nv_bfloat16*>(q),
                    static_cast<__nv_bfloat16*>(k), static_cast<__nv_bfloat16*>(v));
}

cudaError_t launch_f32_to_bf16(size_t n, const float* x, void* y, cudaStream_t st) {
  const int grid = (int)std::min<size_t>((n + kOpsThreads - 1) / kOpsThreads, 1024);
  return launch_pdl(f32_to_bf16_kernel, dim3(grid > 0 ? grid : 1), dim3(kOpsThreads), 0, st, n, x,
                    static_cast<__nv_bfloat16*>(y));
}

}  // namespace seedk
