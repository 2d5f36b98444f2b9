// Tier-1 question-guided selection (Section 2.5, the score_j equation and the
// top-K re-ordering by document position that follows it).
//
// Two kernels:
//  1. cosine_scores_kernel -- one CTA of 256 threads per CME row (grid-stride
//     over rows): every thread streams its share of the row with 16-byte loads
//     issued four at a time, accumulating m.q, m.m and q.q in fp32; the
//     partial sums meet in a fixed tree (warp shuffles, then the eight warps
//     in order), so equal rows produce bit-identical scores.  HBM-bound:
//     4*D bytes per row, with a whole row per CTA in flight.
//  2. topk_select_kernel -- one CTA per sequence.  Scores are mapped to
//     order-preserving uint32 keys; a 4-pass MSB radix select (8 bits a pass)
//     finds the key T of the k-th largest score and how many of the keys equal
//     to T are needed; an ordered compaction then writes the selected indices
//     in ascending order (keys > T, plus the lowest-index keys == T), which is
//     the document-order re-ordering and the lower-index tie rule at once.
// Both launch with programmatic stream serialization, so the selection
// kernel's launch overlaps the scoring kernel.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kScoreThreads = 256;
constexpr int kScoreUnroll = 4;
constexpr int kSelectThreads = 1024;

__global__ void __launch_bounds__(kScoreThreads)
cosine_scores_kernel(const float* __restrict__ qv, const float* __restrict__ bank, int N, int D,
                     long long rows, float* __restrict__ scores) {
  constexpr int kWarpsPerCta = kScoreThreads / 32;
  __shared__ float part[3][kWarpsPerCta];
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int D4 = D >> 2;
  pdl_wait();
  pdl_trigger();
  for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
    const long long b = r / N;
    const float4* m = reinterpret_cast<const float4*>(bank + r * D);
    const float4* q = reinterpret_cast<const float4*>(qv + b * D);
    float dot = 0.f, mm = 0.f, qq = 0.f;
    int i = tid;
    for (; i + kScoreThreads * (kScoreUnroll - 1) < D4; i += kScoreThreads * kScoreUnroll) {
      float4 a[kScoreUnroll], c[kScoreUnroll];
#pragma unroll
      for (int u = 0; u < kScoreUnroll; ++u) a[u] = ld_stream_f4(m + i + kScoreThreads * u);
#pragma unroll
      for (int u = 0; u < kScoreUnroll; ++u) c[u] = __ldg(q + i + kScoreThreads * u);
#pragma unroll
      for (int u = 0; u < kScoreUnroll; ++u) {
        dot = fmaf(a[u].x, c[u].x, dot); dot = fmaf(a[u].y, c[u].y, dot);
        dot = fmaf(a[u].z, c[u].z, dot); dot = fmaf(a[u].w, c[u].w, dot);
        mm = fmaf(a[u].x, a[u].x, mm); mm = fmaf(a[u].y, a[u].y, mm);
        mm = fmaf(a[u].z, a[u].z, mm); mm = fmaf(a[u].w, a[u].w, mm);
        qq = fmaf(c[u].x, c[u].x, qq); qq = fmaf(c[u].y, c[u].y, qq);
        qq = fmaf(c[u].z, c[u].z, qq); qq = fmaf(c[u].w, c[u].w, qq);
      }
    }
    for (; i < D4; i += kScoreThreads) {
      const float4 a = ld_stream_f4(m + i);
      const float4 c = __ldg(q + i);
      dot = fmaf(a.x, c.x, dot); dot = fmaf(a.y, c.y, dot);
      dot = fmaf(a.z, c.z, dot); dot = fmaf(a.w, c.w, dot);
      mm = fmaf(a.x, a.x, mm); mm = fmaf(a.y, a.y, mm);
      mm = fmaf(a.z, a.z, mm); mm = fmaf(a.w, a.w, mm);
      qq = fmaf(c.x, c.x, qq); qq = fmaf(c.y, c.y, qq);
      qq = fmaf(c.z, c.z, qq); qq = fmaf(c.w, c.w, qq);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      dot += __shfl_xor_sync(0xffffffffu, dot, off);
      mm += __shfl_xor_sync(0xffffffffu, mm, off);
      qq += __shfl_xor_sync(0xffffffffu, qq, off);
    }
    if (lane == 0) {
      part[0][warp] = dot;
      part[1][warp] = mm;
      part[2][warp] = qq;
    }
    __syncthreads();
    if (tid == 0) {
      float sd = part[0][0], sm = part[1][0], sq = part[2][0];
#pragma unroll
      for (int w = 1; w < kWarpsPerCta; ++w) {
        sd += part[0][w];
        sm += part[1][w];
        sq += part[2][w];
      }
      float sc = 0.f;
      if (sm > 0.f && sq > 0.f) sc = sd / (sqrtf(sm) * sqrtf(sq));
      if (sc == 0.f) sc = 0.f;  // -0 -> +0, so that -0 and +0 tie
      scores[r] = sc;
    }
    __syncthreads();  // part[] is reused by the next row
  }
}

// Exclusive block-wide prefix count of a per-thread flag (1024 threads).
// `warp_sums` is a 32-entry shared scratch array; returns the exclusive count
// for this thread and the block total in *total.
__device__ __forceinline__ uint32_t block_exclusive_count(bool flag, uint32_t* warp_sums,
                                                          uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t ballot = __ballot_sync(0xffffffffu, flag);
  const uint32_t lane_ex = __popc(ballot & ((1u << lane) - 1u));
  if (lane == 0) warp_sums[warp] = __popc(ballot);
  __syncthreads();
  if (warp == 0) {
    const uint32_t v = (lane < (int)(blockDim.x >> 5)) ? warp_sums[lane] : 0u;
    uint32_t inc = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t t = __shfl_up_sync(0xffffffffu, inc, off);
      if (lane >= off) inc += t;
    }
    warp_sums[lane] = inc - v;                       // exclusive
    if (lane == 31) warp_sums[32] = inc;             // block total
  }
  __syncthreads();
  const uint32_t r = warp_sums[warp] + lane_ex;
  *total = warp_sums[32];
  __syncthreads();  // warp_sums is reused by the next call
  return r;
}

__global__ void __launch_bounds__(kSelectThreads)
topk_select_kernel(const float* __restrict__ scores, int N, int k, int32_t* __restrict__ idx_out) {
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  pdl_wait();  // the scores of the kernel before
  pdl_trigger();
  const float* s = scores + static_cast<long long>(b) * N;
  int32_t* out = idx_out + static_cast<long long>(b) * k;
  if (k <= 0) return;
  if (k >= N) {
    for (int j = tid; j < N; j += blockDim.x) out[j] = j;
    return;
  }
  __shared__ uint32_t hist[256];
  __shared__ uint32_t sh_prefix, sh_krem;
  __shared__ uint32_t warp_sums[33];

  uint32_t prefix = 0u, mask = 0u, krem = static_cast<uint32_t>(k);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0u;
    __syncthreads();
    for (int j = tid; j < N; j += blockDim.x) {
      const uint32_t key = orderable(s[j]);
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      // lane l owns digits 255-8l down to 248-8l; scan from the top digit down
      const int lane = tid;
      uint32_t c = 0;
#pragma unroll
      for (int t = 0; t < 8; ++t) c += hist[255 - 8 * lane - t];
      uint32_t inc = c;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += t;
      }
      const uint32_t hit = __ballot_sync(0xffffffffu, inc >= krem);
      const int first = __ffs(hit) - 1;  // krem <= count of matching keys, so hit != 0
      if (lane == first) {
        uint32_t above = inc - c;  // keys in digits above this lane's range
        for (int t = 0; t < 8; ++t) {
          const int digit = 255 - 8 * lane - t;
          const uint32_t h = hist[digit];
          if (above + h >= krem) {
            sh_prefix = prefix | (static_cast<uint32_t>(digit) << shift);
            sh_krem = krem - above;
            break;
          }
          above += h;
        }
      }
    }
    __syncthreads();
    prefix = sh_prefix;
    krem = sh_krem;
    mask |= 0xFFu << shift;
    __syncthreads();
  }

  // prefix == T, the key of the k-th largest score; krem keys equal to T are needed.
  const uint32_t T = prefix;
  uint32_t run_sel = 0u, run_eq = 0u;
  for (int base = 0; base < N; base += blockDim.x) {
    const int j = base + tid;
    const uint32_t key = (j < N) ? orderable(s[j]) : 0u;
    const bool gt = (j < N) && key > T;
    const bool eq = (j < N) && key == T;
    uint32_t eq_total, sel_total;
    const uint32_t eq_rank = run_eq + block_exclusive_count(eq, warp_sums, &eq_total);
    const bool sel = gt || (eq && eq_rank < krem);
    const uint32_t slot = run_sel + block_exclusive_count(sel, warp_sums, &sel_total);
    if (sel && slot < static_cast<uint32_t>(k)) out[slot] = j;  // exactly k are selected
    run_eq += eq_total;
    run_sel += sel_total;
  }
}

// The two selection kernels, scores written to `sc` (device, B * N floats).
static int launch_score_select(const float* question_emb, const float* cme_bank, int B, int N,
                               int D, int k, int32_t* idx_out, float* sc, cudaStream_t s) {
  const long long rows = static_cast<long long>(B) * N;
  long long blocks = rows;
  const long long cap = static_cast<long long>(sm_count()) * (2048 / kScoreThreads);
  if (blocks > cap) blocks = cap;
  int st = launch_pdl(cosine_scores_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kScoreThreads),
                      0, s, question_emb, cme_bank, N, D, rows, sc);
  if (st != CMC_OK || k == 0) return st;
  return launch_pdl(topk_select_kernel, dim3(B), dim3(kSelectThreads), 0, s,
                    static_cast<const float*>(sc), N, k, idx_out);
}

}  // namespace cmc

extern "C" {

size_t cmc_score_select_workspace_size(int B, int N) {
  if (B < 1 || N < 1) return 0;
  return cmc::align_up(static_cast<size_t>(B) * static_cast<size_t>(N) * sizeof(float), 256);
}

int cmc_score_select(const float* question_emb, const float* cme_bank, int B, int N, int D, int k,
                     int32_t* idx_out, float* scores_out, void* workspace, size_t workspace_bytes,
                     void* stream) {
  using namespace cmc;
  if (B < 1 || B > 65535 || N < 1 || N > (1 << 20) || D < 4 || D > 65536 || (D & 3))
    return CMC_ERR_SHAPE;
  if (k < 0 || k > N) return CMC_ERR_RANGE;
  if (!question_emb || !cme_bank) return CMC_ERR_NULL;
  if (k > 0 && !idx_out) return CMC_ERR_NULL;
  if (!aligned16(question_emb) || !aligned16(cme_bank)) return CMC_ERR_ALIGN;
  if ((scores_out && (reinterpret_cast<uintptr_t>(scores_out) & 3)) ||
      (idx_out && (reinterpret_cast<uintptr_t>(idx_out) & 3)))
    return CMC_ERR_ALIGN;
  float* sc = scores_out;
  if (!sc) {
    if (!workspace) return CMC_ERR_WORKSPACE;
    if (workspace_bytes < cmc_score_select_workspace_size(B, N)) return CMC_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(workspace) & 3) return CMC_ERR_ALIGN;
    sc = static_cast<float*>(workspace);
  }
  return launch_score_select(question_emb, cme_bank, B, N, D, k, idx_out, sc,
                             static_cast<cudaStream_t>(stream));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant: the score scratch is a file-scope device array.
// ---------------------------------------------------------------------------

// One copy per device that loads the library; shared by every call.
static __device__ __align__(256) float g_static_scores[CMC_STATIC_SCORES_MAX];

namespace cmc {

constexpr int kStaticMaxDevices = 64;
static std::mutex g_static_mu;
static float* g_static_scores_dev[kStaticMaxDevices] = {};

// Device address of g_static_scores on the current device; looked up once per
// device (host code cannot use the symbol itself as a device pointer).
static int static_scores_address(float** out) {
  int dev = -1;
  int st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  if (dev < 0 || dev >= kStaticMaxDevices) return CMC_ERR_SHAPE;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static_scores_dev[dev]) {
    void* p = nullptr;
    st = record_cuda_error(cudaGetSymbolAddress(&p, g_static_scores));
    if (st != CMC_OK) return st;
    if (!p) return CMC_ERR_CUDA;
    g_static_scores_dev[dev] = static_cast<float*>(p);
  }
  *out = g_static_scores_dev[dev];
  return CMC_OK;
}

}  // namespace cmc

extern "C" int cmc_score_select_static(const float* question_emb, const float* cme_bank, int B,
                                       int N, int D, int k, int32_t* idx_out, void* stream) {
  using namespace cmc;
  if (B < 1 || B > 65535 || N < 1 || N > (1 << 20) || D < 4 || D > 65536 || (D & 3))
    return CMC_ERR_SHAPE;
  if (static_cast<long long>(B) * N > CMC_STATIC_SCORES_MAX) return CMC_ERR_SHAPE;
  if (k < 0 || k > N) return CMC_ERR_RANGE;
  if (!question_emb || !cme_bank) return CMC_ERR_NULL;
  if (k > 0 && !idx_out) return CMC_ERR_NULL;
  if (!aligned16(question_emb) || !aligned16(cme_bank)) return CMC_ERR_ALIGN;
  if (idx_out && (reinterpret_cast<uintptr_t>(idx_out) & 3)) return CMC_ERR_ALIGN;
  float* sc = nullptr;
  int st = static_scores_address(&sc);
  if (st != CMC_OK) return st;
  return launch_score_select(question_emb, cme_bank, B, N, D, k, idx_out, sc,
                             static_cast<cudaStream_t>(stream));
}
