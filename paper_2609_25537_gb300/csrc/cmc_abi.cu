// Status strings, CUDA error bookkeeping and shared host-side validation of
// the libcmc C ABI.
#include <cuda_runtime.h>

#include "cmc_internal.cuh"

namespace cmc {

static thread_local int g_last_cuda_error = 0;

int record_cuda_error(cudaError_t e) {
  if (e == cudaSuccess) return CMC_OK;
  g_last_cuda_error = static_cast<int>(e);
  return CMC_ERR_CUDA;
}

int check_launch() { return record_cuda_error(cudaGetLastError()); }

int sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
  if (dev < 64 && cache[dev] > 0) return cache[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    n = 148;
  if (dev < 64) cache[dev] = n;
  return n;
}

int validate_dims(const cmc_dims* dims, bool need_bank) {
  if (!dims) return CMC_ERR_NULL;
  const cmc_dims& m = *dims;
  if (m.B < 1 || m.B > 65535 || m.L < 1 || m.Hkv < 1 || m.W < 1) return CMC_ERR_SHAPE;
  if (m.d != 64 && m.d != 128) return CMC_ERR_SHAPE;
  if ((long long)m.B * m.L * m.Hkv > (1LL << 24)) return CMC_ERR_SHAPE;
  if (m.W > (1 << 24)) return CMC_ERR_SHAPE;
  if (need_bank) {
    if (m.Hq < 1 || m.Hq % m.Hkv != 0) return CMC_ERR_SHAPE;
    const int G = m.Hq / m.Hkv;
    if (G != 1 && G != 2 && G != 4 && G != 8) return CMC_ERR_SHAPE;
    if (m.N < 1 || m.N > (1 << 24)) return CMC_ERR_SHAPE;
    if (m.k < 0 || m.k > m.N) return CMC_ERR_RANGE;
  }
  return CMC_OK;
}

}  // namespace cmc

extern "C" {

const char* cmc_status_string(int status) {
  switch (status) {
    case CMC_OK: return "CMC_OK";
    case CMC_ERR_NULL: return "CMC_ERR_NULL: a required pointer is NULL";
    case CMC_ERR_SHAPE: return "CMC_ERR_SHAPE: a size is outside the supported range";
    case CMC_ERR_RANGE: return "CMC_ERR_RANGE: an index-like argument is out of range";
    case CMC_ERR_ALIGN: return "CMC_ERR_ALIGN: a tensor pointer is not 16-byte aligned";
    case CMC_ERR_WORKSPACE: return "CMC_ERR_WORKSPACE: workspace missing or too small";
    case CMC_ERR_CUDA: return "CMC_ERR_CUDA: a CUDA call failed";
    default: return "unknown cmc_status";
  }
}

int cmc_last_cuda_error(void) {
  int e = cmc::g_last_cuda_error;
  cmc::g_last_cuda_error = 0;
  return e;
}

int cmc_read_status(void* workspace, int clear, uint32_t* flags, void* stream) {
  if (!workspace || !flags) return CMC_ERR_NULL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t v = 0;
  int st = cmc::record_cuda_error(
      cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, s));
  if (st != CMC_OK) return st;
  st = cmc::record_cuda_error(cudaStreamSynchronize(s));
  if (st != CMC_OK) return st;
  *flags = v;
  if (clear) st = cmc::record_cuda_error(cudaMemsetAsync(workspace, 0, sizeof(uint32_t), s));
  return st;
}

}  // extern "C"
