// Staging copies between pinned host memory and device memory inside a
// stream of kernels: the input and output traffic of a serving loop, moved
// by a kernel so that the decode kernels around it keep programmatic
// dependent launch (a copy-engine copy between two kernels, or a wait on
// another stream's copy, ends it for the kernel after it).
//
// One launch performs up to kMaxCopies byte ranges with 16-byte loads and
// stores, each thread keeping kInFlight loads in flight (host memory is reached
// over the chip-to-chip link, with a latency of a microsecond or more).  The
// kernel starts its copies without waiting for the kernel before it on the
// stream and waits for that kernel only at its end (griddepcontrol.wait), so
// the copies overlap that kernel while the launch still completes after it:
// work later on the stream sees both.  With `wait_first` it waits before
// copying instead (for sources that the previous kernel writes).
#include <cuda_runtime.h>
#include <stdint.h>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kMaxCopies = 4;
constexpr int kIoThreads = 256;
constexpr int kInFlight = 4;
constexpr int kIoMaxCtas = 64;

struct IoArgs {
  const uint4* src[kMaxCopies];
  uint4* dst[kMaxCopies];
  long long chunks[kMaxCopies];  // 16-byte chunks of each copy
  int n;
  int wait_first;
};

__global__ void __launch_bounds__(kIoThreads) stage_copy_kernel(const __grid_constant__ IoArgs a) {
  if (a.wait_first) pdl_wait();
  pdl_trigger();
  const long long stride = static_cast<long long>(gridDim.x) * kIoThreads;
  const long long t0 = static_cast<long long>(blockIdx.x) * kIoThreads + threadIdx.x;
  for (int c = 0; c < a.n; ++c) {
    const uint4* __restrict__ src = a.src[c];
    uint4* __restrict__ dst = a.dst[c];
    const long long n = a.chunks[c];
    for (long long base = t0; base < n; base += stride * kInFlight) {
      uint4 v[kInFlight];
#pragma unroll
      for (int e = 0; e < kInFlight; ++e) {
        const long long i = base + e * stride;
        if (i < n) v[e] = src[i];
      }
#pragma unroll
      for (int e = 0; e < kInFlight; ++e) {
        const long long i = base + e * stride;
        if (i < n) dst[i] = v[e];
      }
    }
  }
  // complete only after the kernel before this one on the stream
  if (!a.wait_first) pdl_wait();
}

}  // namespace cmc

extern "C" int cmc_stage_copies(const cmc_copy* copies, int n, int wait_first, void* stream) {
  using namespace cmc;
  if (n < 0 || n > kMaxCopies) return CMC_ERR_RANGE;
  if (n > 0 && !copies) return CMC_ERR_NULL;
  IoArgs a;
  a.n = 0;
  a.wait_first = wait_first ? 1 : 0;
  long long most = 0;
  for (int i = 0; i < n; ++i) {
    const cmc_copy& c = copies[i];
    if (c.bytes == 0) continue;
    if (!c.src || !c.dst) return CMC_ERR_NULL;
    if (!aligned16(c.src) || !aligned16(c.dst) || (c.bytes & 15u)) return CMC_ERR_ALIGN;
    a.src[a.n] = static_cast<const uint4*>(c.src);
    a.dst[a.n] = static_cast<uint4*>(c.dst);
    a.chunks[a.n] = static_cast<long long>(c.bytes / 16);
    if (a.chunks[a.n] > most) most = a.chunks[a.n];
    ++a.n;
  }
  for (int i = a.n; i < kMaxCopies; ++i) {
    a.src[i] = nullptr;
    a.dst[i] = nullptr;
    a.chunks[i] = 0;
  }
  // enough CTAs for every thread to hold kInFlight chunks of the largest copy,
  // at most kIoMaxCtas (the kernel shares the GPU with the decode kernels)
  long long ctas = (most + static_cast<long long>(kIoThreads) * kInFlight - 1) /
                   (static_cast<long long>(kIoThreads) * kInFlight);
  if (ctas < 1) ctas = 1;
  if (ctas > kIoMaxCtas) ctas = kIoMaxCtas;
  return launch_pdl(stage_copy_kernel, dim3(static_cast<unsigned>(ctas)), dim3(kIoThreads), 0,
                    static_cast<cudaStream_t>(stream), a);
}
