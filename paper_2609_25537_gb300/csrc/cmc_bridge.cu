// MemoryBridge output (Section 2.2, the norm-calibrated tanh equation): the
// decoder-ready CMEs from the output x of the MemoryBridge MLP,
//   m_hat = LayerNorm(x)  (mean and biased variance over the H_d features,
//                          eps, per-feature gamma and beta: PyTorch's default
//                          LayerNorm, as the hyperparameter appendix states)
//   m     = nu tanh(m_hat) min(1, 2 nu / ||nu tanh(m_hat)||_2)
// so that every CME's norm is at most 2 nu.  The MLP's two matrix products
// are plain library GEMMs and stay with the caller; this is the row-wise
// epilogue that turns their output into the bank the Tier-1 scoring reads.
//
// One CTA per row (grid-stride): the row is streamed once into shared memory
// with 16-byte loads, the three row reductions (sum, squared deviations,
// squared norm of nu tanh) meet in a fixed tree, and the row is written once.
// HBM-bound: 8 * H_d bytes per row.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kBridgeThreads = 256;
constexpr int kBridgeMaxD = 16384;  // 64 KB of shared memory per row

// Block-wide sum in a fixed order (warp shuffles, then the warps in order);
// every thread receives the total.  `red` holds kBridgeThreads / 32 + 1 floats.
__device__ __forceinline__ float bridge_block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = red[0];
#pragma unroll
    for (int w = 1; w < kBridgeThreads / 32; ++w) t += red[w];
    red[kBridgeThreads / 32] = t;
  }
  __syncthreads();
  const float total = red[kBridgeThreads / 32];
  __syncthreads();  // red is reused by the next call
  return total;
}

__global__ void __launch_bounds__(kBridgeThreads)
bridge_epilogue_kernel(const float* __restrict__ x, const float* __restrict__ gamma,
                       const float* __restrict__ beta, long long rows, int D, float eps, float nu,
                       float* out) {
  extern __shared__ float4 srow[];  // the row being processed, D / 4 vectors
  __shared__ float red[kBridgeThreads / 32 + 1];
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x;
  const int D4 = D >> 2;
  const float4* g4 = reinterpret_cast<const float4*>(gamma);
  const float4* b4 = reinterpret_cast<const float4*>(beta);
  for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
    const float4* xr = reinterpret_cast<const float4*>(x + r * D);
    float s = 0.f;
    // four 16-byte loads per thread in flight before any is used
    for (int base = 0; base < D4; base += 4 * kBridgeThreads) {
      float4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = base + u * kBridgeThreads + tid;
        v[u] = i < D4 ? ld_stream_f4(xr + i) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = base + u * kBridgeThreads + tid;
        if (i < D4) srow[i] = v[u];
        s += (v[u].x + v[u].y) + (v[u].z + v[u].w);
      }
    }
    const float mean = bridge_block_sum(s, red) / static_cast<float>(D);
    float q = 0.f;
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 v = srow[i];
      const float a = v.x - mean, b = v.y - mean, c = v.z - mean, d = v.w - mean;
      q += (a * a + b * b) + (c * c + d * d);
    }
    const float var = bridge_block_sum(q, red) / static_cast<float>(D);
    const float rstd = 1.0f / sqrtf(var + eps);
    float n2 = 0.f;
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 v = srow[i];
      const float4 g = gamma ? __ldg(g4 + i) : make_float4(1.f, 1.f, 1.f, 1.f);
      const float4 b = beta ? __ldg(b4 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
      float4 t;
      t.x = nu * tanhf(fmaf(g.x, (v.x - mean) * rstd, b.x));
      t.y = nu * tanhf(fmaf(g.y, (v.y - mean) * rstd, b.y));
      t.z = nu * tanhf(fmaf(g.z, (v.z - mean) * rstd, b.z));
      t.w = nu * tanhf(fmaf(g.w, (v.w - mean) * rstd, b.w));
      srow[i] = t;
      n2 += (t.x * t.x + t.y * t.y) + (t.z * t.z + t.w * t.w);
    }
    const float norm = sqrtf(bridge_block_sum(n2, red));
    const float f = (norm > 2.f * nu) ? (2.f * nu) / norm : 1.f;
    float4* orow = reinterpret_cast<float4*>(out + r * D);
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 t = srow[i];
      orow[i] = make_float4(t.x * f, t.y * f, t.z * f, t.w * f);
    }
    __syncthreads();  // srow is refilled by the next row
  }
}

}  // namespace cmc

extern "C" {

int cmc_bridge_epilogue(const float* x, const float* gamma, const float* beta, int64_t rows, int D,
                        float eps, float nu, float* out, void* stream) {
  using namespace cmc;
  if (rows < 1 || D < 4 || D > kBridgeMaxD || (D & 3)) return CMC_ERR_SHAPE;
  if (!(eps > 0.f) || !(nu > 0.f) || !isfinite(eps) || !isfinite(nu)) return CMC_ERR_RANGE;
  if (!x || !out) return CMC_ERR_NULL;
  if (!aligned16(x) || !aligned16(out) || (gamma && !aligned16(gamma)) || (beta && !aligned16(beta)))
    return CMC_ERR_ALIGN;
  const size_t smem = static_cast<size_t>(D) * sizeof(float);
  static bool attr_set[64] = {false};
  int dev = 0;
  int st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    st = record_cuda_error(cudaFuncSetAttribute(bridge_epilogue_kernel,
                                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                static_cast<int>(kBridgeMaxD * sizeof(float))));
    if (st != CMC_OK) return st;
    attr_set[dev] = true;
  }
  long long grid = rows;
  const long long cap = static_cast<long long>(sm_count()) * (2048 / kBridgeThreads);
  if (grid > cap) grid = cap;
  return launch_pdl(bridge_epilogue_kernel, dim3(static_cast<unsigned>(grid)), dim3(kBridgeThreads),
                    smem, static_cast<cudaStream_t>(stream), x, gamma, beta,
                    static_cast<long long>(rows), D, eps, nu, out);
}

}  // extern "C"
