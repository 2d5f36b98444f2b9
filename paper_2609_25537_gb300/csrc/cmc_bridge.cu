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
// Rows of up to 4,096 features stay in registers, one 128-thread CTA per
// row (bridge_epilogue_reg_kernel, below).  Longer rows: a CTA walks its rows (grid-stride) through three
// shared-memory row buffers: while it reduces and writes row r, rows r + grid and r + 2 grid are
// already on their way (16-byte cp.async copies), so each SM overlaps the HBM
// reads of later rows with the arithmetic and the writes of the current one.
// The three row reductions (sum, squared deviations, squared norm of
// nu tanh) meet in a fixed tree; each thread touches only its own float4s of
// the row, so the buffers need a barrier only when a buffer is refilled.
// tanh(z) is evaluated as 1 - 2 / (1 + e^{2z}) with the hardware base-2
// exponential (ex2.approx, relative error ~2^-22) and a fast division:
// absolute error below 1e-6, saturating correctly to +-1.
// HBM-bound: 8 * H_d bytes per row.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <atomic>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kBridgeThreads = 256;
constexpr int kBridgeMaxD = 16384;  // 64 KB of shared memory per row buffer
constexpr int kBridgeBufs = 3;      // the row being processed + two in flight
constexpr int kBridgeCtasPerSm = 2;

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

// tanh(z) = 1 - 2 / (1 + 2^(2 z log2 e)).
__device__ __forceinline__ float tanh_ex2(float z) {
  float e;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(e) : "f"(z * 2.8853900817779268f));
  return 1.f - __fdividef(2.f, 1.f + e);
}

__device__ __forceinline__ void br_cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void br_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void br_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

__global__ void __launch_bounds__(kBridgeThreads, kBridgeCtasPerSm)
bridge_epilogue_kernel(const float* x, const float* __restrict__ gamma,
                       const float* __restrict__ beta, long long rows, int D, float eps, float nu,
                       float* out) {
  extern __shared__ float4 sbuf[];  // kBridgeBufs row buffers of D / 4 vectors
  __shared__ float red[kBridgeThreads / 32 + 1];
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x;
  const int D4 = D >> 2;
  const float4* g4 = reinterpret_cast<const float4*>(gamma);
  const float4* b4 = reinterpret_cast<const float4*>(beta);
  const long long step = gridDim.x;
  auto load = [&](long long r, int buf) {
    const float4* src = reinterpret_cast<const float4*>(x + r * D);
    float4* dst = sbuf + static_cast<long long>(buf) * D4;
    for (int i = tid; i < D4; i += kBridgeThreads) br_cp_async16(dst + i, src + i);
  };
  // prologue: the first kBridgeBufs - 1 rows of this CTA (one group each)
#pragma unroll
  for (int k = 0; k < kBridgeBufs - 1; ++k) {
    const long long r = blockIdx.x + k * step;
    if (r < rows) load(r, k);
    br_commit();
  }
  int k = 0;
  for (long long r = blockIdx.x; r < rows; r += step, ++k) {
    const long long ra = r + (kBridgeBufs - 1) * step;  // row whose load starts now
    if (ra < rows) load(ra, (k + kBridgeBufs - 1) % kBridgeBufs);
    br_commit();
    br_wait<kBridgeBufs - 1>();  // this thread's copies of row r have landed
    float4* row = sbuf + static_cast<long long>(k % kBridgeBufs) * D4;
    float s = 0.f;
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 v = row[i];
      s += (v.x + v.y) + (v.z + v.w);
    }
    const float mean = bridge_block_sum(s, red) / static_cast<float>(D);
    float q = 0.f;
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 v = row[i];
      const float a = v.x - mean, b = v.y - mean, c = v.z - mean, d = v.w - mean;
      q += (a * a + b * b) + (c * c + d * d);
    }
    const float var = bridge_block_sum(q, red) / static_cast<float>(D);
    const float rstd = 1.0f / sqrtf(var + eps);
    float n2 = 0.f;
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 v = row[i];
      const float4 g = gamma ? __ldg(g4 + i) : make_float4(1.f, 1.f, 1.f, 1.f);
      const float4 b = beta ? __ldg(b4 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
      float4 t;
      t.x = nu * tanh_ex2(fmaf(g.x, (v.x - mean) * rstd, b.x));
      t.y = nu * tanh_ex2(fmaf(g.y, (v.y - mean) * rstd, b.y));
      t.z = nu * tanh_ex2(fmaf(g.z, (v.z - mean) * rstd, b.z));
      t.w = nu * tanh_ex2(fmaf(g.w, (v.w - mean) * rstd, b.w));
      row[i] = t;
      n2 += (t.x * t.x + t.y * t.y) + (t.z * t.z + t.w * t.w);
    }
    const float norm = sqrtf(bridge_block_sum(n2, red));
    const float f = (norm > 2.f * nu) ? (2.f * nu) / norm : 1.f;
    float4* orow = reinterpret_cast<float4*>(out + r * D);
    for (int i = tid; i < D4; i += kBridgeThreads) {
      const float4 t = row[i];
      orow[i] = make_float4(t.x * f, t.y * f, t.z * f, t.w * f);
    }
    __syncthreads();  // this buffer is refilled at the next iteration
  }
  br_wait<0>();
}

// Rows of at most 4,096 features: one CTA of 128 threads per row, a thread
// keeping its V float4s of the row in registers; eight CTAs per SM, so that
// a bank of up to 8 x SMs rows is one wave whose loads are all issued at
// once (more rows: grid-stride).  No shared-memory staging; each of the
// three reductions takes one barrier (its own partials array, summed by every
// thread in the same order).  Before the grid dependency wait a CTA asks L2
// to prefetch its first row, so that under programmatic dependent launch the
// row streams in while the kernel before drains (a prefetch is a hint: L2
// stays coherent with that kernel's writes to x).
constexpr int kBridgeRegThreads = 128;
constexpr int kBridgeRegMaxV = 8;  // float4s per thread: D <= 4 * 8 * kBridgeRegThreads
constexpr int kBridgeRegCtasPerSm = 8;

template <int V>
__global__ void __launch_bounds__(kBridgeRegThreads, kBridgeRegCtasPerSm)
bridge_epilogue_reg_kernel(const float* x, const float* __restrict__ gamma,
                           const float* __restrict__ beta, long long rows, int D, float eps,
                           float nu, float* out) {
  constexpr int NW = kBridgeRegThreads / 32;
  __shared__ float red[3][NW];
  if (threadIdx.x == 0 && static_cast<long long>(blockIdx.x) < rows)
    // D * 4 bytes of a 16-byte aligned row (D a multiple of 4): the bulk
    // prefetch's alignment and size rules hold
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(
                     x + static_cast<long long>(blockIdx.x) * D),
                 "r"(static_cast<unsigned int>(D) * 4u)
                 : "memory");
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int D4 = D >> 2;
  const float4* g4 = reinterpret_cast<const float4*>(gamma);
  const float4* b4 = reinterpret_cast<const float4*>(beta);
  auto block_sum = [&](float v, float* part) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0) part[warp] = v;
    __syncthreads();
    float t = part[0];
#pragma unroll
    for (int w = 1; w < NW; ++w) t += part[w];
    return t;
  };
  for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
    float4 cur[V];
    const float4* src = reinterpret_cast<const float4*>(x + r * D);
#pragma unroll
    for (int e = 0; e < V; ++e) {
      const int i = tid + e * kBridgeRegThreads;
      cur[e] = i < D4 ? __ldcs(src + i) : make_float4(0.f, 0.f, 0.f, 0.f);  // coherent: x may be out
    }
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < V; ++e) s += (cur[e].x + cur[e].y) + (cur[e].z + cur[e].w);
    const float mean = block_sum(s, red[0]) / static_cast<float>(D);
    float q = 0.f;
#pragma unroll
    for (int e = 0; e < V; ++e) {
      if (tid + e * kBridgeRegThreads < D4) {
        const float a = cur[e].x - mean, b = cur[e].y - mean, c = cur[e].z - mean, d = cur[e].w - mean;
        q += (a * a + b * b) + (c * c + d * d);
      }
    }
    const float var = block_sum(q, red[1]) / static_cast<float>(D);
    const float rstd = 1.0f / sqrtf(var + eps);
    float n2 = 0.f;
#pragma unroll
    for (int e = 0; e < V; ++e) {
      const int i = tid + e * kBridgeRegThreads;
      if (i < D4) {
        const float4 g = gamma ? __ldg(g4 + i) : make_float4(1.f, 1.f, 1.f, 1.f);
        const float4 b = beta ? __ldg(b4 + i) : make_float4(0.f, 0.f, 0.f, 0.f);
        float4& t = cur[e];
        t.x = nu * tanh_ex2(fmaf(g.x, (t.x - mean) * rstd, b.x));
        t.y = nu * tanh_ex2(fmaf(g.y, (t.y - mean) * rstd, b.y));
        t.z = nu * tanh_ex2(fmaf(g.z, (t.z - mean) * rstd, b.z));
        t.w = nu * tanh_ex2(fmaf(g.w, (t.w - mean) * rstd, b.w));
        n2 += (t.x * t.x + t.y * t.y) + (t.z * t.z + t.w * t.w);
      }
    }
    const float norm = sqrtf(block_sum(n2, red[2]));
    const float f = (norm > 2.f * nu) ? (2.f * nu) / norm : 1.f;
    float4* orow = reinterpret_cast<float4*>(out + r * D);
#pragma unroll
    for (int e = 0; e < V; ++e) {
      const int i = tid + e * kBridgeRegThreads;
      if (i < D4) orow[i] = make_float4(cur[e].x * f, cur[e].y * f, cur[e].z * f, cur[e].w * f);
    }
    __syncthreads();  // red is rewritten by the next row of this CTA
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
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int D4 = D / 4;
  if (D4 <= kBridgeRegMaxV * kBridgeRegThreads) {
    long long grid = rows;
    const long long cap = static_cast<long long>(sm_count()) * kBridgeRegCtasPerSm;
    if (grid > cap) grid = cap;
    const dim3 gd(static_cast<unsigned>(grid)), bd(kBridgeRegThreads);
    const long long R = static_cast<long long>(rows);
    switch ((D4 + kBridgeRegThreads - 1) / kBridgeRegThreads) {
      case 1: return launch_pdl(bridge_epilogue_reg_kernel<1>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      case 2: return launch_pdl(bridge_epilogue_reg_kernel<2>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      case 3: return launch_pdl(bridge_epilogue_reg_kernel<3>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      case 4: return launch_pdl(bridge_epilogue_reg_kernel<4>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      case 5: return launch_pdl(bridge_epilogue_reg_kernel<5>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      case 6: return launch_pdl(bridge_epilogue_reg_kernel<6>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      case 7: return launch_pdl(bridge_epilogue_reg_kernel<7>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
      default: return launch_pdl(bridge_epilogue_reg_kernel<8>, gd, bd, 0, s, x, gamma, beta, R, D, eps, nu, out);
    }
  }
  const size_t smem = static_cast<size_t>(kBridgeBufs) * D * sizeof(float);
  static std::atomic<bool> attr_set[64];  // per device: the attribute is set (idempotent)
  int dev = 0;
  int st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  if (dev >= 0 && dev < 64 && !attr_set[dev].load(std::memory_order_acquire)) {
    st = record_cuda_error(cudaFuncSetAttribute(bridge_epilogue_kernel,
                                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                static_cast<int>(kBridgeBufs * kBridgeMaxD * sizeof(float))));
    if (st != CMC_OK) return st;
    attr_set[dev].store(true, std::memory_order_release);
  }
  // Persistent CTAs, kBridgeCtasPerSm per SM (one when the row buffers leave
  // room for only one): each walks about rows / grid rows.
  const int per_sm = D * 4 * kBridgeBufs * kBridgeCtasPerSm <= 200 * 1024 ? kBridgeCtasPerSm : 1;
  long long grid = rows;
  const long long cap = static_cast<long long>(sm_count()) * per_sm;
  if (grid > cap) grid = cap;
  return launch_pdl(bridge_epilogue_kernel, dim3(static_cast<unsigned>(grid)), dim3(kBridgeThreads),
                    smem, s, x, gamma, beta, static_cast<long long>(rows), D, eps, nu, out);
}

}  // extern "C"
