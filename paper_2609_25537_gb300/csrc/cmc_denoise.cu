// Graph-based context denoising (Section 2.1): token i of a context is kept
// when its cosine similarity to at least one of its g following tokens
// reaches tau, and the keep-minimum constraint of the appendix on the
// threshold forces one kept token into every run of `keep_every` positions.
//
// Two kernels:
//  1. denoise_pass_kernel -- one warp per token: the token's row and the rows
//     of its g followers are read with 16-byte loads through L1 (each row is
//     read from HBM once; the CTA's warps take consecutive tokens, so its
//     re-reads as a follower mostly hit L1 or L2),
//     the norms and dot products reduced in a fixed order, and the pass flag
//     (max cosine >= tau, decided in fp32) written as one byte.
//  2. denoise_compact_kernel -- one CTA per context.  Walking left to right,
//     the keep-minimum forces token i exactly when it fails the test and its
//     distance to the last token that passed (or to position -1) is a
//     multiple of keep_every, so the walk is data-parallel: a block-wide
//     prefix maximum gives every thread's chunk the last passing position
//     before it, and a block-wide prefix sum places the kept positions, which
//     are written in ascending order.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kDenoiseMaxG = 8;
constexpr int kPassThreads = 256;
constexpr int kCompactThreads = 1024;

__global__ void __launch_bounds__(kPassThreads)
denoise_pass_kernel(const float* __restrict__ emb, const int32_t* __restrict__ n_tokens, int B,
                    int n_max, int H, int g, float tau, uint8_t* __restrict__ pass) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const long long warp0 = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long nwarps = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  const long long total = static_cast<long long>(B) * n_max;
  const int H4 = H >> 2;
  for (long long t = warp0; t < total; t += nwarps) {
    const int b = static_cast<int>(t / n_max);
    const int i = static_cast<int>(t - static_cast<long long>(b) * n_max);
    int n = n_tokens ? n_tokens[b] : n_max;
    n = n < 0 ? 0 : (n > n_max ? n_max : n);
    if (i >= n) {
      if (lane == 0) pass[t] = 0;
      continue;
    }
    const int gg = min(g, n - 1 - i);  // followers that exist
    const float4* ei = reinterpret_cast<const float4*>(emb + t * H);
    float ni = 0.f, dot[kDenoiseMaxG], nj[kDenoiseMaxG];
#pragma unroll
    for (int s = 0; s < kDenoiseMaxG; ++s) dot[s] = nj[s] = 0.f;
    // The CTA's warps take consecutive tokens, so a row read here (through
    // L1) is mostly the follower row of the warps just before: each row
    // crosses from L2 about once.
#pragma unroll 2
    for (int c = lane; c < H4; c += 32) {
      const float4 a = __ldg(ei + c);
      ni += (a.x * a.x + a.y * a.y) + (a.z * a.z + a.w * a.w);
#pragma unroll
      for (int s = 0; s < kDenoiseMaxG; ++s) {
        if (s < gg) {
          const float4 v = __ldg(ei + static_cast<long long>(s + 1) * H4 + c);
          dot[s] += (a.x * v.x + a.y * v.y) + (a.z * v.z + a.w * v.w);
          nj[s] += (v.x * v.x + v.y * v.y) + (v.z * v.z + v.w * v.w);
        }
      }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      ni += __shfl_xor_sync(0xffffffffu, ni, off);
#pragma unroll
      for (int s = 0; s < kDenoiseMaxG; ++s) {
        dot[s] += __shfl_xor_sync(0xffffffffu, dot[s], off);
        nj[s] += __shfl_xor_sync(0xffffffffu, nj[s], off);
      }
    }
    if (lane == 0) {
      bool ok = false;
#pragma unroll
      for (int s = 0; s < kDenoiseMaxG; ++s) {
        if (s < gg) {
          const float c = (ni > 0.f && nj[s] > 0.f) ? dot[s] / (sqrtf(ni) * sqrtf(nj[s])) : 0.f;
          ok = ok || c >= tau;
        }
      }
      pass[t] = ok ? 1 : 0;
    }
  }
}

__global__ void __launch_bounds__(kCompactThreads)
denoise_compact_kernel(const uint8_t* __restrict__ pass, const int32_t* __restrict__ n_tokens,
                       int n_max, int keep_every, int32_t* __restrict__ kept_idx,
                       int32_t* __restrict__ kept_count) {
  __shared__ int wred[kCompactThreads / 32];
  __shared__ int wtot;
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int n = n_tokens ? n_tokens[b] : n_max;
  n = n < 0 ? 0 : (n > n_max ? n_max : n);
  const uint8_t* pb = pass + static_cast<long long>(b) * n_max;
  int32_t* out = kept_idx + static_cast<long long>(b) * n_max;
  const int C = (n + kCompactThreads - 1) / kCompactThreads;  // tokens per thread
  const int t0 = tid * C;
  const int t1 = min(t0 + C, n);

  // last passing position in this thread's chunk, then the prefix maximum
  // over the threads before it (-1: none)
  int last = -1;
  for (int i = t0; i < t1; ++i)
    if (pb[i]) last = i;
  int incl = last;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl = max(incl, v);
  }
  if (lane == 31) wred[warp] = incl;
  __syncthreads();
  int carry = -1;  // last passing position before this thread's chunk
  for (int w = 0; w < warp; ++w) carry = max(carry, wred[w]);
  const int prev_lane = __shfl_up_sync(0xffffffffu, incl, 1);
  if (lane > 0) carry = max(carry, prev_lane);
  __syncthreads();  // wred is reused below

  // kept tokens of the chunk: passed, or forced by the keep-minimum
  auto kept = [&](int i, int lastp) {
    return pb[i] != 0 || (keep_every > 0 && (i - lastp) % keep_every == 0);
  };
  int cnt = 0;
  int lp = carry;
  for (int i = t0; i < t1; ++i) {
    if (kept(i, lp)) ++cnt;
    if (pb[i]) lp = i;
  }
  // exclusive prefix sum of the counts
  int inc = cnt;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += v;
  }
  if (lane == 31) wred[warp] = inc;
  __syncthreads();
  int before = 0;
  for (int w = 0; w < warp; ++w) before += wred[w];
  if (tid == kCompactThreads - 1) wtot = before + inc;
  int slot = before + inc - cnt;
  lp = carry;
  for (int i = t0; i < t1; ++i) {
    if (kept(i, lp)) out[slot++] = i;
    if (pb[i]) lp = i;
  }
  __syncthreads();
  const int total = wtot;
  for (int i = total + tid; i < n_max; i += kCompactThreads) out[i] = -1;
  if (tid == 0) kept_count[b] = total;
}

}  // namespace cmc

extern "C" {

size_t cmc_denoise_workspace_size(int B, int n_max) {
  if (B < 1 || n_max < 1) return 0;
  return cmc::align_up(static_cast<size_t>(B) * static_cast<size_t>(n_max), 256);
}

int cmc_denoise(const float* emb, const int32_t* n_tokens, int B, int n_max, int H, int g,
                float tau, int keep_every, int32_t* kept_idx, int32_t* kept_count,
                void* workspace, size_t workspace_bytes, void* stream) {
  using namespace cmc;
  if (B < 1 || B > 65535 || n_max < 1 || n_max > (1 << 24) || H < 4 || H > 65536 || (H & 3))
    return CMC_ERR_SHAPE;
  if (g < 1 || g > kDenoiseMaxG || keep_every < 0 || !isfinite(tau)) return CMC_ERR_RANGE;
  if (!emb || !kept_idx || !kept_count || !workspace) return CMC_ERR_NULL;
  if (!aligned16(emb)) return CMC_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(n_tokens) & 3) || (reinterpret_cast<uintptr_t>(kept_idx) & 3) ||
      (reinterpret_cast<uintptr_t>(kept_count) & 3))
    return CMC_ERR_ALIGN;
  if (workspace_bytes < cmc_denoise_workspace_size(B, n_max)) return CMC_ERR_WORKSPACE;
  if (static_cast<long long>(B) * n_max * H >= (1LL << 40)) return CMC_ERR_SHAPE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* pass = static_cast<uint8_t*>(workspace);
  const long long warps = static_cast<long long>(B) * n_max;
  long long blocks = (warps * 32 + kPassThreads - 1) / kPassThreads;
  const long long cap = static_cast<long long>(sm_count()) * (2048 / kPassThreads) * 4;
  if (blocks > cap) blocks = cap;
  int st = launch_pdl(denoise_pass_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kPassThreads),
                      0, s, emb, n_tokens, B, n_max, H, g, tau, pass);
  if (st != CMC_OK) return st;
  return launch_pdl(denoise_compact_kernel, dim3(B), dim3(kCompactThreads), 0, s,
                    static_cast<const uint8_t*>(pass), n_tokens, n_max, keep_every, kept_idx,
                    kept_count);
}

}  // extern "C"
