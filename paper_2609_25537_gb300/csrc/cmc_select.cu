// Tier-1 question-guided selection (Section 2.5, the score_j equation and the
// top-K re-ordering by document position that follows it), and the
// question-side prologue before it (the mean-pooled question vector, and the
// CME-guided start of the Tier-2 window).
//
// Small banks (the request sizes of a single decode): one launch,
// score_select_fused_kernel -- CTAs score a few rows each and the CTA that
// completes a sequence's scores selects its top k (see there); the prologue's
// pooling and localisation run in the same launch.
//
// Larger banks, two launches:
//  1. cosine_scores_kernel -- one CTA of 256 threads per CME row (grid-stride
//     over rows): every thread streams its share of the row with 16-byte loads
//     issued four at a time, accumulating m.q, m.m and q.q in fp32; the
//     partial sums meet in a fixed tree (warp shuffles, then the eight warps
//     in order), so equal rows produce bit-identical scores.  HBM-bound:
//     4*D bytes per row, with a whole row per CTA in flight.
//  2. topk_select_kernel -- one CTA per sequence (above 8,192 CMEs,
//     topk_select_cluster_kernel: a cluster of 8, see there).  Scores are mapped to
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
// Threads of the selection CTA: 512 for banks of up to kSelectWideN CMEs, 1024
// above (measured: the wider block halves the top-k time at 16,384 CMEs and
// costs a little at 1,024).
constexpr int kSelectThreadsMax = 1024;
constexpr int kSelectWideN = 8192;

__global__ void __launch_bounds__(kScoreThreads)
cosine_scores_kernel(const float* __restrict__ qv, const float* __restrict__ bank, int N, int D,
                     long long rows, float* __restrict__ scores, float* __restrict__ sqnorm) {
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
      if (sqnorm) sqnorm[r] = sm;  // for the CME-guided localisation
    }
    __syncthreads();  // part[] is reused by the next row
  }
}

// q_vec[b] = mean of the first q_len[b] question-token embeddings (Section
// 2.5, Tier-1); an empty question gives the zero vector.  A CTA covers 32
// four-column groups: lane c of warp s sums the tokens s, s + 8, s + 16, ...
// of its group (so every warp reads whole 512-byte row segments, and all of a
// question's rows are in flight at once), then the eight partial sums of a
// group are added in warp order and divided by the count.
constexpr int kPoolThreads = 256;
constexpr int kPoolSlices = kPoolThreads / 32;  // token slices (warps) per CTA

__global__ void __launch_bounds__(kPoolThreads)
question_pool_kernel(const float* __restrict__ tokens, const int32_t* __restrict__ q_len, int Lq,
                     int D, float* __restrict__ q_vec) {
  __shared__ float4 part[kPoolSlices][32];
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y;
  const int lane = threadIdx.x & 31, sl = threadIdx.x >> 5;
  const int c4 = blockIdx.x * 32 + lane;
  const int D4 = D >> 2;
  int n = q_len ? q_len[b] : Lq;
  n = n < 0 ? 0 : (n > Lq ? Lq : n);
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (c4 < D4) {
    const float4* t = reinterpret_cast<const float4*>(tokens + static_cast<long long>(b) * Lq * D) + c4;
    for (int i = sl; i < n; i += kPoolSlices) {
      const float4 v = __ldg(t + static_cast<long long>(i) * D4);
      acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
    }
  }
  part[sl][lane] = acc;
  __syncthreads();
  if (sl == 0 && c4 < D4) {
    float4 tot = part[0][lane];
#pragma unroll
    for (int w = 1; w < kPoolSlices; ++w) {
      const float4 v = part[w][lane];
      tot.x += v.x; tot.y += v.y; tot.z += v.z; tot.w += v.w;
    }
    if (n > 0) {
      const float fn = static_cast<float>(n);
      tot.x /= fn; tot.y /= fn; tot.z /= fn; tot.w /= fn;
    }
    reinterpret_cast<float4*>(q_vec + static_cast<long long>(b) * D)[c4] = tot;
  }
}

// Exclusive prefix sum of one value per thread over the block (NT threads,
// warps in order); `wsum` is an NT/32-entry shared array
// used by this call only.  Returns this thread's exclusive prefix; *total gets
// the block total.
template <int NT>
__device__ __forceinline__ uint32_t block_exclusive_sum(uint32_t v, uint32_t* wsum, uint32_t* total) {
  constexpr int kW = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t inc = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += t;
  }
  if (lane == 31) wsum[warp] = inc;
  __syncthreads();
  uint32_t before = 0, all = 0;
#pragma unroll
  for (int w = 0; w < kW; ++w) {
    const uint32_t x = wsum[w];
    before += (w < warp) ? x : 0u;
    all += x;
  }
  *total = all;
  return before + inc - v;
}

// Sequences of at most this many CMEs keep their keys in shared memory for
// the radix passes and the compaction; longer ones re-read the scores.  Key
// j sits at word j + j / 32, so that the compaction's threads, each reading
// its own run of consecutive keys, hit different banks.
constexpr int kSelectSmemKeys = 49152;
__host__ __device__ constexpr size_t select_smem_words(int n) {
  return static_cast<size_t>(n) + static_cast<size_t>(n) / 32 + 1;
}

// CME-guided localisation for the Tier-2 window (optional part of the
// selection CTA): alpha = offset of the chunk behind the CME of largest norm
// (the argmax over the squared norms the scoring kernel wrote, ties to the
// lower index), start = max(0, min(|C| - W, alpha - W/2)).
struct LocateArgs {
  float* sqnorm;                // [B, N], or NULL: no localisation
  const int32_t* chunk_offset;  // [B, N]
  const int32_t* ctx_len;       // [B]
  int W;
  int32_t* alpha_out;           // [B] (nullable)
  int32_t* start_out;           // [B] (nullable)
  // [B] or NULL: the one-launch path's argmax slots, (orderable squared norm
  // << 32) | ~index, raised by every scoring CTA (zero before, zero after)
  unsigned long long* best = nullptr;
};

__device__ __forceinline__ void locate_window(const LocateArgs& la, int b, int N) {
  __shared__ float wbest[kSelectThreadsMax / 32];
  __shared__ int wbidx[kSelectThreadsMax / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* sq = la.sqnorm + static_cast<long long>(b) * N;
  float best = -1.f;
  int bi = 0x7fffffff;
  for (int j = tid; j < N; j += blockDim.x) {  // ascending j: strict > keeps the lowest index
    const float v = sq[j];
    if (v > best) { best = v; bi = j; }
  }
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, best, off);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
    if (ov > best || (ov == best && oi < bi)) { best = ov; bi = oi; }
  }
  if (lane == 0) { wbest[warp] = best; wbidx[warp] = bi; }
  __syncthreads();
  if (tid == 0) {
    for (int w = 1; w < static_cast<int>(blockDim.x >> 5); ++w)
      if (wbest[w] > best || (wbest[w] == best && wbidx[w] < bi)) { best = wbest[w]; bi = wbidx[w]; }
    const long long alpha = la.chunk_offset[static_cast<long long>(b) * N + bi];
    long long st = static_cast<long long>(la.ctx_len[b]) - la.W;
    const long long centred = alpha - la.W / 2;
    if (centred < st) st = centred;
    if (st < 0) st = 0;
    if (la.alpha_out) la.alpha_out[b] = static_cast<int32_t>(alpha);
    if (la.start_out) la.start_out[b] = static_cast<int32_t>(st);
  }
}

template <int NT>
__global__ void __launch_bounds__(NT)
topk_select_kernel(const float* __restrict__ scores, int N, int k, int32_t* __restrict__ idx_out,
                   const LocateArgs la) {
  extern __shared__ uint32_t skeys[];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t wsum[3][NT / 32];
  __shared__ uint32_t sh_prefix, sh_krem;
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  pdl_wait();  // the scores of the kernel before
  pdl_trigger();
  if (la.sqnorm) locate_window(la, b, N);
  const float* s = scores + static_cast<long long>(b) * N;
  int32_t* out = idx_out + static_cast<long long>(b) * k;
  if (k <= 0) return;
  if (k >= N) {
    for (int j = tid; j < N; j += blockDim.x) out[j] = j;
    return;
  }
  const bool in_smem = N <= kSelectSmemKeys;
  for (int j = tid; j < 256; j += blockDim.x) hist[j] = 0u;
  if (in_smem)
    for (int j = tid; j < N; j += blockDim.x) skeys[j + (j >> 5)] = orderable(s[j]);
  __syncthreads();
  auto key_at = [&](int j) -> uint32_t { return in_smem ? skeys[j + (j >> 5)] : orderable(s[j]); };

  // Radix select, 8 bits a pass from the top: after the passes `prefix` is the
  // key T of the k-th largest score and krem of the keys equal to T are kept.
  uint32_t prefix = 0u, mask = 0u, krem = static_cast<uint32_t>(k);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    // Scores cluster (cosines near 0 share their top bits), so lanes that hit
    // the same bin add their count with one atomic (warp-aggregated).
    for (int base = 0; base < N; base += blockDim.x) {
      const int j = base + tid;
      const uint32_t key = j < N ? key_at(j) : 0u;
      const bool part = j < N && (key & mask) == prefix;
      const uint32_t bin = part ? ((key >> shift) & 255u) : 0xFFFFFFFFu;
      const uint32_t peers = __match_any_sync(0xffffffffu, bin);
      if (part && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
    }
    __syncthreads();
    // Threads 0..255 own the digits from the top (255 - tid): an inclusive
    // scan over them counts the matching keys at or above each digit; the one
    // thread whose digit holds the krem-th key records it.  Reading a bin also
    // clears it for the next pass.
    uint32_t c = 0u, inc = 0u;
    if (tid < 256) {
      c = hist[255 - tid];
      hist[255 - tid] = 0u;
      inc = c;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += t;
      }
      if (lane == 31) wsum[0][warp] = inc;
    }
    __syncthreads();
    if (tid < 256) {
      for (int w = 0; w < warp; ++w) inc += wsum[0][w];
      const uint32_t excl = inc - c;
      if (excl < krem && inc >= krem) {
        sh_prefix = prefix | (static_cast<uint32_t>(255 - tid) << shift);
        sh_krem = krem - excl;
      }
    }
    __syncthreads();
    prefix = sh_prefix;
    krem = sh_krem;
    mask |= 0xFFu << shift;
  }

  // Ordered compaction: keys > T, and the first krem keys == T in index
  // order, written in ascending index order.  Each thread owns a run of
  // consecutive keys of a chunk; two block scans place its outputs.
  const uint32_t T = prefix;
  const int per = (N + static_cast<int>(blockDim.x) - 1) / static_cast<int>(blockDim.x);
  const int C = per < 32 ? per : 32;  // keys per thread and chunk
  const int chunk = C * static_cast<int>(blockDim.x);
  uint32_t run_eq = 0u, run_sel = 0u;
  for (int base = 0; base < N; base += chunk) {
    const int j0 = base + tid * C;
    uint32_t n_eq = 0u;
    for (int e = 0; e < C; ++e) {
      const int j = j0 + e;
      if (j < N && key_at(j) == T) ++n_eq;
    }
    uint32_t eq_total, sel_total;
    const uint32_t eq0 = run_eq + block_exclusive_sum<NT>(n_eq, wsum[1], &eq_total);
    uint32_t n_sel = 0u, r = eq0;
    for (int e = 0; e < C; ++e) {
      const int j = j0 + e;
      if (j < N) {
        const uint32_t key = key_at(j);
        if (key > T) ++n_sel;
        else if (key == T) n_sel += (r++ < krem) ? 1u : 0u;
      }
    }
    uint32_t slot = run_sel + block_exclusive_sum<NT>(n_sel, wsum[2], &sel_total);
    r = eq0;
    for (int e = 0; e < C; ++e) {
      const int j = j0 + e;
      if (j < N) {
        const uint32_t key = key_at(j);
        const bool sel = key > T || (key == T && r++ < krem);
        if (sel && slot < static_cast<uint32_t>(k)) out[slot++] = j;  // exactly k are selected
      }
    }
    run_eq += eq_total;
    run_sel += sel_total;
    __syncthreads();  // wsum[1], wsum[2] are reused by the next chunk
  }
}

// --- thread-block cluster helpers (barrier over every thread of the
// cluster; loads from a peer CTA's shared memory).
__device__ __forceinline__ void sel_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire;\n" ::: "memory");
}
__device__ __forceinline__ uint32_t sel_cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t sel_ld_peer(const uint32_t* local, uint32_t rank) {
  uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(local)), r, v;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(rank));
  asm volatile("ld.shared::cluster.u32 %0, [%1];\n" : "=r"(v) : "r"(r) : "memory");
  return v;
}

// Banks of more than kSelectWideN CMEs: one cluster of kSelectClusterCtas
// CTAs per sequence, CTA r holding the keys of indices [r N / 8, (r+1) N / 8)
// in its shared memory.  Each radix pass builds the CTA's histogram, and after
// a cluster barrier every CTA adds the eight histograms (distributed shared
// memory, rank order) and takes the same decision; the histograms are
// double-buffered by pass parity.  The compaction counts each CTA's keys above
// and equal to T, combines the counts across the cluster (exclusive sums over
// the ranks) to place the keys equal to T in global index order and each
// CTA's outputs, then writes.  Every thread of the cluster passes the same
// seven cluster barriers.
constexpr int kSelectClusterCtas = 8;

__global__ void __launch_bounds__(kSelectThreadsMax)
topk_select_cluster_kernel(const float* __restrict__ scores, int N, int k,
                           int32_t* __restrict__ idx_out, const LocateArgs la) {
  constexpr int NT = kSelectThreadsMax;
  constexpr int CS = kSelectClusterCtas;
  extern __shared__ uint32_t skeys[];
  __shared__ uint32_t hist[2][256];
  __shared__ uint32_t wsum[3][NT / 32];
  __shared__ uint32_t pub[2];  // this CTA's keys equal to T, and its selected keys
  __shared__ uint32_t sh_prefix, sh_krem;
  const int b = blockIdx.x / CS;
  const uint32_t rank = sel_cluster_rank();
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;
  pdl_wait();  // the scores of the kernel before
  pdl_trigger();
  if (la.sqnorm && rank == 0) locate_window(la, b, N);
  const float* s = scores + static_cast<long long>(b) * N;
  int32_t* out = idx_out + static_cast<long long>(b) * k;
  if (k <= 0) return;  // the same for every CTA of the cluster
  if (k >= N) {
    if (rank == 0)
      for (int j = tid; j < N; j += NT) out[j] = j;
    return;
  }
  const int jb = static_cast<int>((static_cast<long long>(rank) * N) / CS);  // this CTA's first key
  const int n = static_cast<int>((static_cast<long long>(rank + 1) * N) / CS) - jb;
  for (int j = tid; j < 2 * 256; j += NT) hist[j >> 8][j & 255] = 0u;
  for (int j = tid; j < n; j += NT) skeys[j + (j >> 5)] = orderable(s[jb + j]);
  __syncthreads();
  auto key_at = [&](int j) -> uint32_t { return skeys[j + (j >> 5)]; };

  uint32_t prefix = 0u, mask = 0u, krem = static_cast<uint32_t>(k);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    uint32_t* h = hist[pass & 1];
    for (int base = 0; base < n; base += NT) {
      const int j = base + tid;
      const uint32_t key = j < n ? key_at(j) : 0u;
      const bool part = j < n && (key & mask) == prefix;
      const uint32_t bin = part ? ((key >> shift) & 255u) : 0xFFFFFFFFu;
      const uint32_t peers = __match_any_sync(0xffffffffu, bin);
      if (part && lane == __ffs(peers) - 1) atomicAdd(&h[bin], __popc(peers));
    }
    sel_cluster_sync();  // every CTA's histogram of this pass is complete
    uint32_t c = 0u, inc = 0u;
    if (tid < 256) {
      for (int r = 0; r < CS; ++r) c += sel_ld_peer(&h[255 - tid], static_cast<uint32_t>(r));
      inc = c;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += t;
      }
      if (lane == 31) wsum[0][warp] = inc;
      // the other buffer was read by every peer before this pass's barrier
      hist[(pass + 1) & 1][tid] = 0u;
    }
    __syncthreads();
    if (tid < 256) {
      for (int w = 0; w < warp; ++w) inc += wsum[0][w];
      const uint32_t excl = inc - c;
      if (excl < krem && inc >= krem) {
        sh_prefix = prefix | (static_cast<uint32_t>(255 - tid) << shift);
        sh_krem = krem - excl;
      }
    }
    __syncthreads();
    prefix = sh_prefix;
    krem = sh_krem;
    mask |= 0xFFu << shift;
  }

  // This CTA's keys above T and equal to T; then, across the cluster, the
  // keys equal to T before this CTA (they rank first among the equal keys)
  // and the selected keys before this CTA (its first output slot).
  const uint32_t T = prefix;
  uint32_t n_gt = 0u, n_eq = 0u;
  for (int j = tid; j < n; j += NT) {
    const uint32_t key = key_at(j);
    n_gt += key > T ? 1u : 0u;
    n_eq += key == T ? 1u : 0u;
  }
  uint32_t gt_total, eq_total;
  block_exclusive_sum<NT>(n_gt, wsum[1], &gt_total);
  block_exclusive_sum<NT>(n_eq, wsum[2], &eq_total);
  if (tid == 0) pub[0] = eq_total;
  sel_cluster_sync();
  uint32_t eq_before = 0u;
  for (int r = 0; r < static_cast<int>(rank); ++r) eq_before += sel_ld_peer(&pub[0], static_cast<uint32_t>(r));
  const uint32_t eq_take = krem > eq_before ? min(krem - eq_before, eq_total) : 0u;
  if (tid == 0) pub[1] = gt_total + eq_take;
  sel_cluster_sync();
  uint32_t sel_before = 0u;
  for (int r = 0; r < static_cast<int>(rank); ++r) sel_before += sel_ld_peer(&pub[1], static_cast<uint32_t>(r));
  __syncthreads();  // wsum is reused below

  // Ordered compaction of this CTA's keys, as in topk_select_kernel, with
  // the running counts starting from the cluster-wide offsets.
  const int per = (n + NT - 1) / NT;
  const int C = per < 32 ? per : 32;
  const int chunk = C * NT;
  uint32_t run_eq = eq_before, run_sel = sel_before;
  for (int base = 0; base < n; base += chunk) {
    const int j0 = base + tid * C;
    uint32_t m_eq = 0u;
    for (int e = 0; e < C; ++e) {
      const int j = j0 + e;
      if (j < n && key_at(j) == T) ++m_eq;
    }
    uint32_t eqc, selc;
    const uint32_t eq0 = run_eq + block_exclusive_sum<NT>(m_eq, wsum[1], &eqc);
    uint32_t m_sel = 0u, r = eq0;
    for (int e = 0; e < C; ++e) {
      const int j = j0 + e;
      if (j < n) {
        const uint32_t key = key_at(j);
        if (key > T) ++m_sel;
        else if (key == T) m_sel += (r++ < krem) ? 1u : 0u;
      }
    }
    uint32_t slot = run_sel + block_exclusive_sum<NT>(m_sel, wsum[2], &selc);
    r = eq0;
    for (int e = 0; e < C; ++e) {
      const int j = j0 + e;
      if (j < n) {
        const uint32_t key = key_at(j);
        const bool sel = key > T || (key == T && r++ < krem);
        if (sel && slot < static_cast<uint32_t>(k)) out[slot++] = jb + j;
      }
    }
    run_eq += eqc;
    run_sel += selc;
    __syncthreads();
  }
  sel_cluster_sync();  // the published counts stay readable until every CTA is done
}

// ---------------------------------------------------------------------------
// One launch for scoring and selection, for small banks: every CTA scores R
// rows of one sequence (R <= kFusedRows divides N, and B N / R CTAs fit in one
// wave of one CTA per SM).
//
// CTA c (1,024 threads) copies its R rows into shared memory with cp.async,
// thread t taking float4 t of each row, so all of them are requested at
// once; while they are in flight it reduces q_vec . q_vec of its sequence.
// Before the grid dependency wait the CTA asks L2 to prefetch its rows, so
// under programmatic dependent launch the bank streams in while the previous
// kernel drains (a prefetch is a hint and leaves L2 coherent with that
// kernel's writes).  Each thread's partial dot and squared norm of the R rows
// (16 values, zero past R) meet across the lanes in a halving butterfly -- at
// lane offset o the lanes with bit o set keep the upper half of their values
// and add their partner's upper half, then the lane pairs add -- which adds
// the same pairs as a plain xor butterfly for every value, in a quarter of
// the shuffles; then warp r adds row r's 32 warp sums in the same butterfly.
// Equal rows thus get bit-identical scores.
//
// The CTA then adds R to the sequence's counter with an acq_rel atomic (which
// releases the CTA's score writes and acquires those of the CTAs before it);
// the CTA whose addition completes N is the last to score that sequence and
// selects its top k itself.  Keys are the order-
// preserving uint32 images of the scores; each scoring CTA adds its rows to a
// histogram of the top 11 key bits in the workspace, and the selecting CTA
// finds the k-th largest key T from it and two shared-memory histogram levels
// (bits 20..10, 9..0); an ordered compaction then writes the keys > T and
// the lowest-index keys == T in ascending index order.  It puts the counter back to zero for
// the next call.  No CTA waits on another.
// ---------------------------------------------------------------------------

constexpr int kFusedThreads = 1024;
constexpr int kFusedWarps = kFusedThreads / 32;
constexpr int kFusedRows = 8;                    // rows per CTA at most
constexpr int kFusedMaxD = 4 * kFusedThreads;    // one float4 per thread and row
constexpr int kFusedMaxN = 2 * kFusedThreads;    // two keys per thread in the selection
constexpr int kHistTop = 2048;                   // bins of the top 11 bits of a key

struct FusedArgs {
  const float* qv;        // [B, D], or NULL: pooled from q_tokens
  const float* q_tokens;  // [B, Lq, D] question-token embeddings (when qv is NULL)
  const int32_t* q_len;   // [B] or NULL (Lq each)
  int Lq;
  float* q_vec_out;       // [B, D]: the pooled q_vec (when qv is NULL)
  const float* bank;      // [B, N, D]
  int N, D, k;
  int rows_per_cta;       // R: divides N
  float* scores;          // [B, N]
  unsigned int* counters; // [B]: zero before the call, zero after it
  int32_t* idx_out;       // [B, k]
  LocateArgs la;          // la.sqnorm: also write squared norms and localise
  unsigned int* hist;     // [B, kHistTop]: counts of the scores' top 11 key bits (zero before, zero after)
};

// Exclusive prefix sum over the block of one value per thread (warps in
// order); `ws` is a kFusedWarps-entry array used by this call only.  Each
// warp scans its values with shuffles, and after one barrier every warp scans
// the 32 warp totals itself (kFusedWarps == 32) and takes the prefix at its
// own index.
__device__ __forceinline__ uint32_t fused_scan(uint32_t v, uint32_t* ws) {
  static_assert(kFusedWarps == 32, "one warp total per lane");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t inc = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += t;
  }
  if (lane == 31) ws[warp] = inc;
  __syncthreads();
  const uint32_t tot = ws[lane];
  uint32_t tinc = tot;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t t = __shfl_up_sync(0xffffffffu, tinc, off);
    if (lane >= off) tinc += t;
  }
  const uint32_t before = __shfl_sync(0xffffffffu, tinc - tot, warp);
  return before + inc - v;
}

// One level of the histogram search for the k-th largest key: thread t holds
// the counts of bins bin_a > bin_b (the bins in descending order across the
// threads); an exclusive prefix sum over the block gives the keys in the bins
// above, and the thread whose bins hold the rem-th key (counting from the
// top) publishes the bin, the rank of that key within it and the bin's count.
__device__ __forceinline__ void hist_level(uint32_t ha, uint32_t bin_a, uint32_t hb, uint32_t bin_b,
                                           uint32_t& rem, uint32_t& digit, uint32_t& count,
                                           uint32_t* ws, uint32_t* pick) {
  const uint32_t above = fused_scan(ha + hb, ws);
  if (above < rem && rem <= above + ha) {
    pick[0] = bin_a;
    pick[1] = rem - above;
    pick[2] = ha;
  } else if (above + ha < rem && rem <= above + ha + hb) {
    pick[0] = bin_b;
    pick[1] = rem - above - ha;
    pick[2] = hb;
  }
  __syncthreads();
  digit = pick[0];
  rem = pick[1];
  count = pick[2];
}

// Top k of one sequence's N scores (N <= KPT * kFusedThreads), written to
// out[0..k) in ascending index order.  Thread t holds the keys of indices
// t*KPT .. t*KPT + KPT - 1 in registers (index order is thread order, then
// position).  Every thread of the CTA calls it.
//
// The k-th largest key T is found in up to three histogram levels: its top
// 11 bits from the histogram the scoring CTAs built in `ghist` (thread t's
// two bins 2047 - 2t and 2046 - 2t read by the caller with the keys, as ga
// and gb; zeroed here for the next call), bits 20..10 from a shared-memory
// histogram of the keys with those top bits, bits 9..0 likewise; each level
// is one prefix sum over the bins (two a thread) -- at most eight barriers,
// against 32 counting barriers for a bit-by-bit search.  A level whose
// chosen bin holds exactly the keys still to take ends the search: every
// key of that bin is selected, so the compaction compares the keys' prefix
// P = key >> s with the bin (s = 21 or 10) instead of the whole key with T,
// and no tie is left to break.  (At the Llama shape the bins of the top 21
// bits hold one key each almost always, so level 3 is rarely run.)  The
// ordered compaction then writes the keys (prefixes) > P and the
// lowest-index ones == P, its output slots from one prefix sum of both
// counts packed in a word.
template <int KPT>
__device__ __forceinline__ void fused_topk(const uint32_t (&key)[KPT], int N, int k, int32_t* out,
                                           uint32_t* ghist, uint32_t ga, uint32_t gb,
                                           uint32_t* scan_sel) {
  __shared__ uint32_t h2[kHistTop], h3[kHistTop / 2], pick[3];
  const int tid = threadIdx.x;
  static_assert(kHistTop == 2 * kFusedThreads, "two top bins a thread");
  h2[2 * tid] = 0u;
  h2[2 * tid + 1] = 0u;
  h3[tid] = 0u;
  // level 1 (bits 31..21): thread t takes bins 2047 - 2t and 2046 - 2t
  const uint32_t ba = kHistTop - 1 - 2 * tid, bb = ba - 1;
  ghist[ba] = 0u;
  ghist[bb] = 0u;
  uint32_t rem = static_cast<uint32_t>(k), d, cnt;
  hist_level(ga, ba, gb, bb, rem, d, cnt, scan_sel, pick);
  uint32_t P = d;  // the boundary keys' prefix key >> s
  int s = 21;
  if (cnt != rem) {  // rem and cnt came through shared memory: the branch is CTA-uniform
    // level 2 (bits 20..10) among the keys with those top bits
#pragma unroll
    for (int e = 0; e < KPT; ++e)
      if (tid * KPT + e < N && (key[e] >> 21) == P) atomicAdd(h2 + ((key[e] >> 10) & 2047u), 1u);
    __syncthreads();
    hist_level(h2[ba], ba, h2[bb], bb, rem, d, cnt, scan_sel, pick);
    P = (P << 11) | d;
    s = 10;
    if (cnt != rem) {
      // level 3 (bits 9..0): thread t takes bin 1023 - t
#pragma unroll
      for (int e = 0; e < KPT; ++e)
        if (tid * KPT + e < N && (key[e] >> 10) == P) atomicAdd(h3 + (key[e] & 1023u), 1u);
      __syncthreads();
      const uint32_t bc = kHistTop / 2 - 1 - tid;
      hist_level(h3[bc], bc, 0u, 0u, rem, d, cnt, scan_sel, pick);
      P = (P << 10) | d;  // T itself
      s = 0;
    }
  }
  // prefixes == P to keep, lowest index first (k - need keys have a larger
  // prefix); with s > 0, need is the bin's whole count
  const uint32_t need = rem;
  uint32_t n_gt = 0, n_eq = 0;
#pragma unroll
  for (int e = 0; e < KPT; ++e) {
    const uint32_t kp = key[e] >> s;
    n_gt += kp > P ? 1u : 0u;
    n_eq += kp == P ? 1u : 0u;
  }
  // the prefixes > P and == P before this thread's, from one prefix sum: both
  // counts total at most N <= 2048 < 2^16, so the low half never carries
  const uint32_t before = fused_scan(n_gt | (n_eq << 16), scan_sel);
  const uint32_t eq_before = before >> 16;
  // the keys > P before this thread's, and the first `need` keys == P
  uint32_t slot = (before & 0xFFFFu) + min(eq_before, need);
  uint32_t r = eq_before;
#pragma unroll
  for (int e = 0; e < KPT; ++e) {
    const uint32_t kp = key[e] >> s;
    const bool sel = kp > P || (kp == P && r++ < need);
    if (sel && slot < static_cast<uint32_t>(k)) out[slot++] = tid * KPT + e;  // exactly k
  }
}

// The selection (and, with la.sqnorm, the localisation) of sequence b by the
// CTA that completed its scores.  Every thread of the CTA calls it.  Thread
// 0's acq_rel counter addition acquired the other CTAs' writes (scores, and
// their raises of the argmax slot); the caller's barrier passed that order on
// to every thread.  The localisation is one slot read by thread 0, issued
// with the score loads; its chunk-offset load then runs under the search and
// its result is written at the end.
template <int KPT>
__device__ __forceinline__ void fused_select_impl(const FusedArgs& a, int b) {
  __shared__ uint32_t scan_sel[kFusedWarps];
  const int tid = threadIdx.x;
  const int N = a.N, k = a.k;
  const bool topk = k > 0 && k < N;
  const float* sc = a.scores + static_cast<long long>(b) * N;
  uint32_t* ghist = a.hist + static_cast<long long>(b) * kHistTop;
  uint32_t key[KPT];
#pragma unroll
  for (int e = 0; e < KPT; ++e) {
    const int j = tid * KPT + e;
    key[e] = (topk && j < N) ? orderable(__ldcg(sc + j)) : 0u;
  }
  // this thread's two bins of the top-bits histogram, in flight with the keys
  uint32_t ga = 0u, gb = 0u;
  if (topk) {
    ga = __ldcg(ghist + (kHistTop - 1 - 2 * tid));
    gb = __ldcg(ghist + (kHistTop - 2 - 2 * tid));
  }
  const bool locate = a.la.sqnorm && tid == 0;
  int32_t alpha = 0, clen = 0;
  if (locate) {
    const unsigned long long packed = __ldcg(a.la.best + b);
    a.la.best[b] = 0ull;  // ready for the next call
    const int bi = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(packed & 0xFFFFFFFFull));
    alpha = __ldg(a.la.chunk_offset + static_cast<long long>(b) * N + bi);
    clen = __ldg(a.la.ctx_len + b);
  }
  int32_t* out = a.idx_out + static_cast<long long>(b) * k;
  if (k >= N) {
    for (int j = tid; j < N; j += kFusedThreads) out[j] = j;
  } else if (k > 0) {
    fused_topk<KPT>(key, N, k, out, ghist, ga, gb, scan_sel);
  }
  if (locate) {
    long long st = static_cast<long long>(clen) - a.la.W;
    const long long centred = static_cast<long long>(alpha) - a.la.W / 2;
    if (centred < st) st = centred;
    if (st < 0) st = 0;
    if (a.la.alpha_out) a.la.alpha_out[b] = alpha;
    if (a.la.start_out) a.la.start_out[b] = static_cast<int32_t>(st);
  }
  if (tid == 0) a.counters[b] = 0u;  // ready for the next call
  __syncthreads();                    // the shared scratch is reused by the caller
}

__device__ __noinline__ void fused_select(const FusedArgs& a, int b) {
  if (a.N <= kFusedThreads) fused_select_impl<1>(a, b);
  else fused_select_impl<2>(a, b);
}

// 16-byte asynchronous copy global -> shared (cp.async), through L2 only.
__device__ __forceinline__ void sel_cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}

__host__ __device__ constexpr size_t fused_smem_bytes() {
  return static_cast<size_t>(kFusedRows) * kFusedThreads * 16;
}

__global__ void __launch_bounds__(kFusedThreads, 1)
score_select_fused_kernel(const __grid_constant__ FusedArgs a) {
  constexpr int RG = kFusedRows;
  // [row][thread]: thread t copies float4 t of each row into its own slot
  extern __shared__ float4 rows_s[];
  __shared__ float part[kFusedWarps][2 * RG];
  __shared__ float qq_part[kFusedWarps];
  __shared__ float rsq_s[kFusedRows];  // the rows' squared norms (localisation)
  __shared__ int last_flag;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int D4 = a.D >> 2;
  const bool own = tid < D4;
  const int R = a.rows_per_cta;
  const int r0 = static_cast<int>(blockIdx.x) * R;  // B N <= kFusedRows x SMs rows
  const int b = r0 / a.N;                            // all R rows are of sequence b
  const float4* rows_g = reinterpret_cast<const float4*>(a.bank) + static_cast<long long>(r0) * D4;
  if (tid == 0) {
    // L2 prefetch of this CTA's rows (a hint: see above)
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(rows_g),
                 "r"(static_cast<unsigned int>(R) * D4 * 16u)
                 : "memory");
  }
  pdl_wait();
  pdl_trigger();
  if (own)
    for (int r = 0; r < R; ++r) sel_cp_async16(rows_s + r * kFusedThreads + tid, rows_g + r * D4 + tid);
  asm volatile("cp.async.commit_group;\n" ::: "memory");
  // q_vec and q_vec . q_vec while the rows are in flight
  float4 qr = make_float4(0.f, 0.f, 0.f, 0.f);
  if (a.qv) {
    if (own) qr = __ldg(reinterpret_cast<const float4*>(a.qv + static_cast<long long>(b) * a.D) + tid);
  } else if (own) {
    // the mean of the first n question-token rows: eight rows at a time,
    // all eight loads in flight, added in a fixed tree, then divided by n
    int n = a.q_len ? a.q_len[b] : a.Lq;
    n = n < 0 ? 0 : (n > a.Lq ? a.Lq : n);
    const float4* tk = reinterpret_cast<const float4*>(a.q_tokens + static_cast<long long>(b) * a.Lq * a.D) + tid;
    for (int i0 = 0; i0 < n; i0 += 8) {
      float4 v[8];
#pragma unroll
      for (int e = 0; e < 8; ++e)
        v[e] = i0 + e < n ? __ldg(tk + static_cast<long long>(i0 + e) * D4) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int w = 1; w < 8; w <<= 1)
#pragma unroll
        for (int e = 0; e < 8; e += 2 * w) {
          v[e].x += v[e + w].x; v[e].y += v[e + w].y; v[e].z += v[e + w].z; v[e].w += v[e + w].w;
        }
      qr.x += v[0].x; qr.y += v[0].y; qr.z += v[0].z; qr.w += v[0].w;
    }
    if (n > 0) {
      const float fn = static_cast<float>(n);
      qr.x /= fn; qr.y /= fn; qr.z /= fn; qr.w /= fn;
    }
    if (r0 == b * a.N) reinterpret_cast<float4*>(a.q_vec_out + static_cast<long long>(b) * a.D)[tid] = qr;
  }
  {
    float acc = 0.f;
    acc = fmaf(qr.x, qr.x, acc); acc = fmaf(qr.y, qr.y, acc);
    acc = fmaf(qr.z, qr.z, acc); acc = fmaf(qr.w, qr.w, acc);
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) qq_part[warp] = acc;
  }
  asm volatile("cp.async.wait_group 0;\n" ::: "memory");
  // this thread's partials: value 2r is row r's dot, 2r + 1 its squared norm
  float v[2 * RG];
#pragma unroll
  for (int r = 0; r < RG; ++r) {
    const float4 m = (r < R && own) ? rows_s[r * kFusedThreads + tid] : make_float4(0.f, 0.f, 0.f, 0.f);
    float d0 = 0.f, s0 = 0.f;
    d0 = fmaf(m.x, qr.x, d0); d0 = fmaf(m.y, qr.y, d0); d0 = fmaf(m.z, qr.z, d0); d0 = fmaf(m.w, qr.w, d0);
    s0 = fmaf(m.x, m.x, s0); s0 = fmaf(m.y, m.y, s0); s0 = fmaf(m.z, m.z, s0); s0 = fmaf(m.w, m.w, s0);
    v[2 * r] = d0;
    v[2 * r + 1] = s0;
  }
  // halving butterfly over the 16 values: afterwards lanes 2i and 2i + 1 both
  // hold value i (i from lane bits 4..1) summed over the warp
#pragma unroll
  for (int o = 16, n = 2 * RG; o >= 2; o >>= 1, n >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < n / 2; ++i) {
      const float send = up ? v[i] : v[i + n / 2];
      const float keep = up ? v[i + n / 2] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  v[0] += __shfl_xor_sync(0xffffffffu, v[0], 1);
  if ((lane & 1) == 0) part[warp][lane >> 1] = v[0];
  __syncthreads();
  float qq = qq_part[0];
#pragma unroll 4
  for (int w = 1; w < kFusedWarps; ++w) qq += qq_part[w];
  // warp r: row r's 32 warp sums, in the same butterfly; lane 0 writes the score
  if (warp < R) {
    float sd = part[lane][2 * warp], sm = part[lane][2 * warp + 1];
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      sd += __shfl_xor_sync(0xffffffffu, sd, off);
      sm += __shfl_xor_sync(0xffffffffu, sm, off);
    }
    if (lane == 0) {
      float sc = 0.f;
      if (sm > 0.f && qq > 0.f) sc = sd / (sqrtf(sm) * sqrtf(qq));
      if (sc == 0.f) sc = 0.f;  // -0 -> +0, so that -0 and +0 tie
      a.scores[r0 + warp] = sc;
      atomicAdd(a.hist + static_cast<long long>(b) * kHistTop + (orderable(sc) >> 21), 1u);
      if (a.la.sqnorm) a.la.sqnorm[r0 + warp] = sm;
      rsq_s[warp] = sm;
    }
  }
  __syncthreads();
  if (tid == 0) {
    if (a.la.sqnorm) {
      // this CTA's largest squared norm (lowest index on ties, NaN lowest),
      // raised into the sequence's argmax slot
      unsigned long long top = 0ull;
      for (int r = 0; r < R; ++r) {
        const float v = rsq_s[r];
        const unsigned long long key = isnan(v) ? 0ull : orderable(v);
        const unsigned long long p =
            (key << 32) | (0xFFFFFFFFu - static_cast<uint32_t>(r0 + r - b * a.N));
        top = p > top ? p : top;
      }
      atomicMax(a.la.best + b, top);
    }
    // acq_rel at GPU scope: releases the CTA's writes (they precede it through
    // the barrier, and this thread's raise in program order) and, for the
    // last CTA, acquires everyone else's
    unsigned int old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;\n"
                 : "=r"(old)
                 : "l"(a.counters + b), "r"(static_cast<unsigned int>(R))
                 : "memory");
    last_flag = (old + R == static_cast<unsigned int>(a.N)) ? 1 : 0;
  }
  __syncthreads();
  if (last_flag) fused_select(a, b);
}

// Rows per CTA of the one-launch path for B sequences of N CMEs of
// dimension D: the largest R <= kFusedRows dividing N with B N / R CTAs in
// one wave of one CTA per SM; 0 when there is none (or a limit is exceeded).
static int fused_rows_per_cta(int B, int N, int D) {
  if (N > kFusedMaxN || D > kFusedMaxD) return 0;
  const long long rows = static_cast<long long>(B) * N;
  for (int R = kFusedRows; R >= 1; --R)
    if (N % R == 0 && rows / R <= sm_count()) return R;
  return 0;
}

// Launches score_select_fused_kernel with R rows per CTA.
static int launch_score_select_fused(const float* question_emb, const float* cme_bank, int B,
                                     int N, int D, int k, int32_t* idx_out, float* sc,
                                     unsigned int* counters, cudaStream_t s, const LocateArgs& la,
                                     int R, const float* q_tokens = nullptr,
                                     const int32_t* q_len = nullptr, int Lq = 0,
                                     float* q_vec_out = nullptr) {
  static std::once_flag attr_once[64];
  int dev = 0;
  int st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  if (dev < 0 || dev >= 64) return CMC_ERR_CUDA;
  std::call_once(attr_once[dev], [&] {
    st = record_cuda_error(cudaFuncSetAttribute(score_select_fused_kernel,
                                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                static_cast<int>(fused_smem_bytes())));
  });
  if (st != CMC_OK) return st;
  FusedArgs a;
  a.qv = question_emb;
  a.q_tokens = q_tokens;
  a.q_len = q_len;
  a.Lq = Lq;
  a.q_vec_out = q_vec_out;
  a.bank = cme_bank;
  a.N = N;
  a.D = D;
  a.k = k;
  a.rows_per_cta = R;
  a.scores = sc;
  a.counters = counters;
  a.idx_out = idx_out;
  a.la = la;
  // the histograms follow the counters in the workspace
  a.hist = reinterpret_cast<unsigned int*>(reinterpret_cast<char*>(counters) +
                                           align_up(static_cast<size_t>(B) * sizeof(unsigned int), 256));
  const long long ctas = static_cast<long long>(B) * N / R;
  return launch_pdl(score_select_fused_kernel, dim3(static_cast<unsigned>(ctas)),
                    dim3(kFusedThreads), fused_smem_bytes(), s, a);
}

// The two selection kernels, scores written to `sc` (device, B * N floats);
// with la.sqnorm set, the squared norms too and the localisation runs in the
// selection kernel.
// With `counters` (B zeroed words) and a bank within the limits of
// score_select_fused_kernel, one launch; otherwise the two kernels.
static int launch_score_select(const float* question_emb, const float* cme_bank, int B, int N,
                               int D, int k, int32_t* idx_out, float* sc, cudaStream_t s,
                               unsigned int* counters = nullptr,
                               const LocateArgs& la = LocateArgs{nullptr, nullptr, nullptr, 0,
                                                                 nullptr, nullptr}) {
  const int fused_rows = counters ? fused_rows_per_cta(B, N, D) : 0;
  if (fused_rows > 0)
    return launch_score_select_fused(question_emb, cme_bank, B, N, D, k, idx_out, sc, counters, s,
                                     la, fused_rows);
  const long long rows = static_cast<long long>(B) * N;
  long long blocks = rows;
  const long long cap = static_cast<long long>(sm_count()) * (2048 / kScoreThreads);
  if (blocks > cap) blocks = cap;
  int st = launch_pdl(cosine_scores_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kScoreThreads),
                      0, s, question_emb, cme_bank, N, D, rows, sc, la.sqnorm);
  if (st != CMC_OK || (k == 0 && !la.sqnorm)) return st;
  static std::once_flag attr_once[64];
  int dev = 0;
  st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  if (dev >= 0 && dev < 64) {
    std::call_once(attr_once[dev], [&] {
      const int bytes = static_cast<int>(select_smem_words(kSelectSmemKeys) * sizeof(uint32_t));
      st = record_cuda_error(cudaFuncSetAttribute(topk_select_kernel<512>,
                                                  cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
      if (st == CMC_OK)
        st = record_cuda_error(cudaFuncSetAttribute(topk_select_kernel<kSelectThreadsMax>,
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
      if (st == CMC_OK)
        st = record_cuda_error(cudaFuncSetAttribute(topk_select_cluster_kernel,
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize, bytes));
    });
    if (st != CMC_OK) return st;
  }
  const size_t smem =
      (N <= kSelectSmemKeys && k > 0 && k < N) ? select_smem_words(N) * sizeof(uint32_t) : 0;
  const int per_cta = (N + kSelectClusterCtas - 1) / kSelectClusterCtas;
  if (N > kSelectWideN && k > 0 && k < N && per_cta <= kSelectSmemKeys) {
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = kSelectClusterCtas;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(B) * kSelectClusterCtas);
    cfg.blockDim = dim3(kSelectThreadsMax);
    cfg.dynamicSmemBytes = select_smem_words(per_cta) * sizeof(uint32_t);
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return record_cuda_error(cudaLaunchKernelEx(&cfg, topk_select_cluster_kernel,
                                                static_cast<const float*>(sc), N, k, idx_out, la));
  }
  if (N > kSelectWideN)
    return launch_pdl(topk_select_kernel<kSelectThreadsMax>, dim3(B), dim3(kSelectThreadsMax), smem, s,
                      static_cast<const float*>(sc), N, k, idx_out, la);
  return launch_pdl(topk_select_kernel<512>, dim3(B), dim3(512), smem, s,
                    static_cast<const float*>(sc), N, k, idx_out, la);
}

}  // namespace cmc

extern "C" {

// [scores: B N fp32][B completion counters][B x kHistTop histogram counts],
// each part 256-byte aligned; the last two zero between calls.
size_t cmc_score_select_workspace_size(int B, int N) {
  if (B < 1 || N < 1) return 0;
  return cmc::align_up(static_cast<size_t>(B) * static_cast<size_t>(N) * sizeof(float), 256) +
         cmc::align_up(static_cast<size_t>(B) * sizeof(unsigned int), 256) +
         static_cast<size_t>(B) * cmc::kHistTop * sizeof(unsigned int);
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
  // Workspace: [B * N fp32 scores, 256-byte aligned][B completion counters].
  // Without one (scores_out given) the two-launch path runs, which needs no
  // counters.
  float* sc = scores_out;
  unsigned int* counters = nullptr;
  if (workspace) {
    if (workspace_bytes < cmc_score_select_workspace_size(B, N)) return CMC_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(workspace) & 3) return CMC_ERR_ALIGN;
    const size_t scores_bytes = align_up(static_cast<size_t>(B) * N * sizeof(float), 256);
    counters = reinterpret_cast<unsigned int*>(static_cast<char*>(workspace) + scores_bytes);
    if (!sc) sc = static_cast<float*>(workspace);
  } else if (!sc) {
    return CMC_ERR_WORKSPACE;
  }
  return launch_score_select(question_emb, cme_bank, B, N, D, k, idx_out, sc,
                             static_cast<cudaStream_t>(stream), counters);
}

size_t cmc_question_select_workspace_size(int B, int N) {
  if (B < 1 || N < 1) return 0;
  return 2 * cmc::align_up(static_cast<size_t>(B) * static_cast<size_t>(N) * sizeof(float), 256) +
         cmc::align_up(static_cast<size_t>(B) * sizeof(unsigned int), 256) +
         static_cast<size_t>(B) * cmc::kHistTop * sizeof(unsigned int) +
         cmc::align_up(static_cast<size_t>(B) * sizeof(unsigned long long), 256);
}

int cmc_question_select(const float* question_tokens, const int32_t* q_len, int Lq,
                        const float* cme_bank, int B, int N, int D, int k,
                        const int32_t* chunk_offset, const int32_t* ctx_len, int W,
                        float* q_vec_out, int32_t* idx_out, int32_t* alpha_out,
                        int32_t* start_out, void* workspace, size_t workspace_bytes,
                        void* stream) {
  using namespace cmc;
  if (B < 1 || B > 65535 || N < 1 || N > (1 << 20) || D < 4 || D > 65536 || (D & 3) || Lq < 1 ||
      static_cast<long long>(Lq) * D > (1LL << 31))
    return CMC_ERR_SHAPE;
  if (k < 0 || k > N) return CMC_ERR_RANGE;
  const bool locate = alpha_out || start_out;
  if (locate && W < 1) return CMC_ERR_RANGE;
  if (!question_tokens || !cme_bank || !q_vec_out || !workspace) return CMC_ERR_NULL;
  if (k > 0 && !idx_out) return CMC_ERR_NULL;
  if (locate && (!chunk_offset || !ctx_len)) return CMC_ERR_NULL;
  if (!aligned16(question_tokens) || !aligned16(cme_bank) || !aligned16(q_vec_out) ||
      !aligned16(workspace))
    return CMC_ERR_ALIGN;
  for (const void* ptr : {static_cast<const void*>(q_len), static_cast<const void*>(idx_out),
                          static_cast<const void*>(chunk_offset), static_cast<const void*>(ctx_len),
                          static_cast<const void*>(alpha_out), static_cast<const void*>(start_out)})
    if (reinterpret_cast<uintptr_t>(ptr) & 3) return CMC_ERR_ALIGN;
  if (workspace_bytes < cmc_question_select_workspace_size(B, N)) return CMC_ERR_WORKSPACE;
  // Workspace: [scores][squared norms] (B * N fp32 each, 256-byte aligned)
  // [B completion counters][B x kHistTop histogram counts][B argmax slots]
  // (the last three zero between calls).
  const size_t scores_bytes = align_up(static_cast<size_t>(B) * N * sizeof(float), 256);
  float* sc = static_cast<float*>(workspace);
  float* sq = sc + scores_bytes / sizeof(float);
  unsigned int* counters =
      reinterpret_cast<unsigned int*>(static_cast<char*>(workspace) + 2 * scores_bytes);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned long long* best = reinterpret_cast<unsigned long long*>(
      static_cast<char*>(workspace) + 2 * scores_bytes +
      align_up(static_cast<size_t>(B) * sizeof(unsigned int), 256) +
      static_cast<size_t>(B) * kHistTop * sizeof(unsigned int));
  LocateArgs la{locate ? sq : nullptr, chunk_offset, ctx_len, W, alpha_out, start_out, best};
  // small banks: pooling, scoring, selection and localisation in one launch
  const int fused_rows = fused_rows_per_cta(B, N, D);
  if (fused_rows > 0)
    return launch_score_select_fused(nullptr, cme_bank, B, N, D, k, idx_out, sc, counters, s, la,
                                     fused_rows, question_tokens, q_len, Lq, q_vec_out);
  const int D4 = D / 4;
  int st = launch_pdl(question_pool_kernel, dim3((D4 + 31) / 32, B),
                      dim3(kPoolThreads), 0, s, question_tokens, q_len, Lq, D, q_vec_out);
  if (st != CMC_OK) return st;
  return launch_score_select(q_vec_out, cme_bank, B, N, D, k, idx_out, sc, s, counters, la);
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
