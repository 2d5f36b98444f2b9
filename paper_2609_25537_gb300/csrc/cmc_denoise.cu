// Graph-based context denoising (Section 2.1): token i of a context is kept
// when its cosine similarity to at least one of its g following tokens
// reaches tau, and the keep-minimum constraint of the appendix on the
// threshold forces one kept token into every run of `keep_every` positions.
//
// Two kernels:
//  1. denoise_pass_kernel -- a CTA takes a tile of 32 consecutive tokens of
//     one context.  Their rows and the rows of the g tokens that follow the
//     tile (together one contiguous span of the [n, H] matrix) are streamed
//     through shared memory in chunks of 128 features (512 bytes per row),
//     four stages of 16-byte cp.async copies (two CTAs per SM); rows past the
//     context's tokens are zero-filled, never read.  Each warp owns four
//     tokens: per chunk a lane takes one float4 of each of the warp's rows
//     and of the g rows after them, and accumulates their squared norms and
//     the dot products of every token with its g followers; the lanes meet
//     once per tile in a halving butterfly (fixed order), and lane t g + s
//     decides the cosine of token t with follower s (>= tau, in fp32), one
//     vote per warp giving its four pass flags.  Every row crosses from HBM
//     once (the g halo rows are the next tile's first rows, read by the
//     neighbouring CTA at about the same time).  The tile's 32 pass bits also
//     go to a word of the workspace, and the tile's positions of kept_idx are
//     set to -1 (the compaction overwrites the kept ones).  For a context of
//     at most 256 tiles (8,192 tokens) the CTA that finishes its last tile (a
//     counter per context, acq_rel) also runs the keep-minimum and the
//     compaction below for that context (pass_compact_small: one pass word
//     per thread, two barriers), and the second kernel is not launched.
//  2. denoise_compact_kernel -- one cluster of 8 CTAs per longer context.
//     Walking left to right, the keep-minimum forces token i exactly when it
//     fails the test and its distance to the last token that passed (or to
//     position -1) is a multiple of keep_every, so the walk is data-parallel.
//     A thread takes one 32-token pass word per segment of 262,144 tokens
//     (the next segment's word is loaded ahead); a cluster-wide prefix
//     maximum gives it the last passing position before its word, from which
//     the forced positions of each gap follow (keep_mask); a cluster-wide
//     prefix sum places its kept positions; both carry from one segment to
//     the next.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <atomic>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kDenoiseMaxG = 8;
constexpr int kPassThreads = 256;
constexpr int kPassTokPerWarp = 4;
constexpr int kPassTile = kPassTokPerWarp * (kPassThreads / 32);  // 32 tokens per tile
constexpr int kPassChunk = 128;                                   // features per stage
constexpr int kPassStageRows = kPassTile + kDenoiseMaxG;          // 40
constexpr int kPassStageBytes = kPassStageRows * kPassChunk * 4;  // 20 KB
constexpr int kPassStages = 4;                                    // two CTAs per SM
__host__ __device__ constexpr int pass_smem(int stages) { return stages * kPassStageBytes; }
constexpr int kCompactThreads = 1024;
constexpr int kCompactWords = 4;  // pass words per 16-byte group of the word array's rows
constexpr int kCompactCtas = 8;   // CTAs (one thread-block cluster) per context

__device__ __forceinline__ void dn_cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void dn_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void dn_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}
__device__ __forceinline__ float dot4(const float4& a, const float4& b) {
  return (a.x * b.x + a.y * b.y) + (a.z * b.z + a.w * b.w);
}

// Kept tokens among the 32 tokens i0 .. i0+31 whose pass bits are `m`, given
// lp, the last passing position before i0 (-1: none): the passing tokens,
// and in every gap between a passing token (or lp) and the next one, the
// positions at multiples of K after it.  The gap from lp takes one division;
// a later gap holds a forced position only when the K bits after its passing
// token are all zero, which a run mask of the zero bits finds for the whole
// word at once (bit x of r: bits x .. x+K-1 of ~m all set, built by doubling),
// so the loop visits only those gaps.
__device__ __forceinline__ uint32_t keep_mask(uint32_t m, int lp, int i0, int K) {
  uint32_t kept = m;
  if (K <= 0) return kept;
  const int first = m ? __ffs(m) - 1 : 32;  // first passing token (word-relative)
  for (int f = lp + K * ((i0 - lp + K - 1) / K) - i0; f < first; f += K) kept |= 1u << f;
  if (K >= 32) return kept;  // a later gap fits no multiple of K inside the word
  uint32_t r = ~m;
  int len = 1;
  while (2 * len <= K) {
    r &= r >> len;
    len *= 2;
  }
  if (K > len) r &= r >> (K - len);
  uint32_t cand = m & (r >> 1);  // passing tokens followed by K failing ones
  while (cand) {
    const int p = __ffs(cand) - 1;
    cand &= cand - 1;
    const uint32_t after = m & ~((2u << p) - 1u);  // passing tokens after p
    const int q = after ? __ffs(after) - 1 : 32;
    for (int f = p + K; f < q; f += K) kept |= 1u << f;
  }
  return kept;
}

// The keep-minimum and the compaction of context b by the pass CTA that
// finished its last tile, for a context of at most kPassThreads tiles:
// thread t takes pass word t; the last passing position before its word is a
// prefix maximum (a warp scan, then the warp totals before it from shared
// memory), its kept positions follow from keep_mask, and their first slot in
// kept_idx is a prefix sum in the same two steps; it writes its kept
// positions itself.  Two barriers.  The words were written by the other CTAs
// of this launch before their counter additions, which this CTA's thread 0
// acquired.
__device__ void pass_compact_small(const uint32_t* masks, int n, int keep_every,
                                   int32_t* out, int32_t* count, int* wmax, int* wsum) {
  constexpr int NW = kPassThreads / 32;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nw = (n + 31) / 32;  // words that hold tokens (at most kPassThreads)
  const int i0 = 32 * tid;
  const int nv = tid < nw ? min(n - i0, 32) : 0;
  const uint32_t valid = nv >= 32 ? ~0u : ((1u << nv) - 1u);
  const uint32_t m = tid < nw ? (__ldcg(masks + tid) & valid) : 0u;
  int lp = m ? i0 + 31 - __clz(m) : -1;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, lp, off);
    if (lane >= off) lp = max(lp, u);
  }
  if (lane == 31) wmax[warp] = lp;
  lp = __shfl_up_sync(0xffffffffu, lp, 1);
  if (lane == 0) lp = -1;
  __syncthreads();
#pragma unroll
  for (int w = 0; w < NW; ++w)
    if (w < warp) lp = max(lp, wmax[w]);
  uint32_t kept = nv > 0 ? keep_mask(m, lp, i0, keep_every) & valid : 0u;
  const int c = __popc(kept);
  int incl = c;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += u;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  int slot = incl - c, total = 0;
#pragma unroll
  for (int w = 0; w < NW; ++w) {
    const int x = wsum[w];
    slot += w < warp ? x : 0;
    total += x;
  }
  while (kept) {
    out[slot++] = i0 + __ffs(kept) - 1;
    kept &= kept - 1;
  }
  if (tid == 0) *count = total;
}

// FUSE (a context of at most kPassThreads tiles): the CTA that finishes a
// context's last tile also runs its keep-minimum and compaction
// (pass_compact_small), counting finished tiles in `counters` (zero before
// the call, zero after it).
template <int G, int NST, bool FUSE>
__global__ void __launch_bounds__(kPassThreads, 2)
denoise_pass_kernel(const float* __restrict__ emb, const int32_t* __restrict__ n_tokens, int n_max,
                    int H, float tau, uint8_t* __restrict__ pass, uint32_t* __restrict__ masks,
                    int32_t* __restrict__ kept_idx, long long tiles, int tiles_per_ctx,
                    int words_stride, unsigned int* __restrict__ counters, int keep_every,
                    int32_t* __restrict__ kept_count) {
  constexpr int TPW = kPassTokPerWarp;
  constexpr int SROWS = kPassTile + G;                                // rows staged per chunk
  constexpr int NCP = (SROWS * 32 + kPassThreads - 1) / kPassThreads;  // copies per thread
  // per warp: the squared norms of its TPW rows and the G rows after them,
  // then the TPW x G dot products; padded to whole groups of 16
  constexpr int NV = TPW + G + TPW * G;
  constexpr int NV16 = (NV + 15) / 16 * 16;
  constexpr int KV = NV16 / 16;  // values a lane holds after the halving rounds
  extern __shared__ __align__(16) float4 dn_stage[];
  __shared__ float red_s[kPassThreads / 32][NV16];  // each warp's reduced values
  __shared__ uint32_t nib[kPassThreads / 32];        // each warp's four pass bits
  __shared__ int wmax[kPassThreads / 32], wsum[kPassThreads / 32];  // the fused compaction's scans
  __shared__ int last_flag;
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nchunks = (H + kPassChunk - 1) / kPassChunk;
  const uint32_t sbase = static_cast<uint32_t>(__cvta_generic_to_shared(dn_stage));
  const int r0 = warp * TPW;  // this warp's first token row in the tile
  for (long long tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
    const int b = static_cast<int>(tile / tiles_per_ctx);
    const int i0 = static_cast<int>(tile - static_cast<long long>(b) * tiles_per_ctx) * kPassTile;
    int n = n_tokens ? n_tokens[b] : n_max;
    n = n < 0 ? 0 : (n > n_max ? n_max : n);
    uint8_t* pb = pass + static_cast<long long>(b) * n_max;
    // the compaction overwrites the kept positions; everything else stays -1
    if (tid < kPassTile && i0 + tid < n_max) kept_idx[static_cast<long long>(b) * n_max + i0 + tid] = -1;
    // Thread 0 writes the tile's pass word (after the barrier that makes the
    // warps' bits and every thread's writes precede it) and, fused, adds the
    // tile to the context's count with an acq_rel atomic (releasing this CTA's
    // writes, acquiring the other CTAs' for the last one); the CTA that
    // completes the count compacts the context.
    auto tile_done = [&](bool empty) {
      __syncthreads();
      if (tid == 0) {
        uint32_t word = 0;
        if (!empty) {
#pragma unroll
          for (int w = 0; w < kPassThreads / 32; ++w) word |= nib[w] << (w * TPW);
        }
        masks[static_cast<long long>(b) * words_stride + i0 / kPassTile] = word;
        if (FUSE) {
          unsigned int old;
          asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;\n"
                       : "=r"(old)
                       : "l"(counters + b)
                       : "memory");
          last_flag = (old + 1 == static_cast<unsigned int>(tiles_per_ctx)) ? 1 : 0;
        }
      }
      if (FUSE) {
        __syncthreads();
        if (last_flag) {
          pass_compact_small(masks + static_cast<long long>(b) * words_stride, n, keep_every,
                             kept_idx + static_cast<long long>(b) * n_max, kept_count + b, wmax,
                             wsum);
          if (tid == 0) counters[b] = 0u;  // ready for the next call
        }
      }
    };
    if (i0 >= n) {  // a tile past the context's tokens: flags 0
      if (tid < kPassTile && i0 + tid < n_max) pb[i0 + tid] = 0;
      tile_done(true);
      continue;
    }
    const int rows = min(SROWS, n - i0);  // staged rows that hold tokens
    const float* src0 = emb + (static_cast<long long>(b) * n_max + i0) * H;
    // this thread's copies: 16-byte piece x = tid + m * kPassThreads of a
    // chunk, row x / 32, column 4 (x % 32) of the chunk
    const float* src[NCP];
    bool live[NCP];
#pragma unroll
    for (int m = 0; m < NCP; ++m) {
      const int x = tid + m * kPassThreads;
      live[m] = x < SROWS * 32 && (x >> 5) < rows;
      src[m] = src0 + static_cast<long long>(x >> 5) * H + 4 * (x & 31);
    }
    auto issue = [&](int c) {
      const uint32_t dst0 = sbase + (c % NST) * kPassStageBytes;
      const int col0 = c * kPassChunk;
#pragma unroll
      for (int m = 0; m < NCP; ++m) {
        const int x = tid + m * kPassThreads;
        if (x < SROWS * 32) {
          const bool ok = live[m] && col0 + 4 * (x & 31) < H;
          dn_cp_async16(dst0 + x * 16, ok ? src[m] + col0 : src0, ok ? 16u : 0u);
        }
      }
    };
#pragma unroll
    for (int c = 0; c < NST - 1; ++c) {
      if (c < nchunks) issue(c);
      dn_commit();
    }
    // v: the norms of rows r0 .. r0+TPW+G-1, then dot(t, s) at TPW + G + t G + s
    float v[NV16];
#pragma unroll
    for (int j = 0; j < NV16; ++j) v[j] = 0.f;
    for (int c = 0; c < nchunks; ++c) {
      dn_wait<NST - 2>();  // chunk c has landed (this thread's copies)
      __syncthreads();             // ... everyone's; and chunk c-1's stage is free
      if (c + NST - 1 < nchunks) issue(c + NST - 1);
      dn_commit();
      const float4* st = dn_stage + (c % NST) * (kPassStageBytes / 16) + r0 * 32 + lane;
      float4 x[TPW + G];
#pragma unroll
      for (int j = 0; j < TPW + G; ++j) x[j] = st[j * 32];
#pragma unroll
      for (int j = 0; j < TPW + G; ++j) v[j] += dot4(x[j], x[j]);
#pragma unroll
      for (int t = 0; t < TPW; ++t)
#pragma unroll
        for (int s = 0; s < G; ++s) v[TPW + G + t * G + s] += dot4(x[t], x[t + 1 + s]);
    }
    dn_wait<0>();
    // Halving butterfly over the lanes: at offset o the lanes with bit o set
    // keep the upper half of their values and add their partner's upper
    // half; the others the lower half.  It adds the same pairs as a plain xor
    // butterfly for every value (so every warp that reduces a row's norm
    // gets the same bits), in a fraction of the shuffles.  Afterwards lanes
    // 2i and 2i+1 hold values KV i .. KV i + KV-1 summed over the warp.
#pragma unroll
    for (int o = 16, nh = NV16 / 2; o >= 2; o >>= 1, nh >>= 1) {
      const bool up = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < nh; ++i) {
        const float send = up ? v[i] : v[i + nh];
        const float keep = up ? v[i + nh] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
#pragma unroll
    for (int i = 0; i < KV; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], 1);
    if ((lane & 1) == 0) {
#pragma unroll
      for (int i = 0; i < KV; ++i) red_s[warp][KV * (lane >> 1) + i] = v[i];
    }
    __syncwarp();
    {
      // the test of token t against its follower s on lane t G + s, then one
      // vote per warp
      const int my_t = lane / G, my_s = lane - (lane / G) * G;
      const int i = i0 + r0 + my_t;
      bool ok = false;
      if (lane < TPW * G && i < n && my_s < min(G, n - 1 - i)) {
        const float ni = red_s[warp][my_t], nj = red_s[warp][my_t + 1 + my_s];
        const float d = red_s[warp][TPW + G + lane];
        const float c = (ni > 0.f && nj > 0.f) ? d / (sqrtf(ni) * sqrtf(nj)) : 0.f;
        ok = c >= tau;
      }
      const uint32_t vote = __ballot_sync(0xffffffffu, ok);
      uint32_t bits = 0;
#pragma unroll
      for (int t = 0; t < TPW; ++t)
        bits |= ((vote >> (t * G)) & ((1u << G) - 1u)) ? (1u << t) : 0u;
      if (lane < TPW && i0 + r0 + lane < n_max) pb[i0 + r0 + lane] = (bits >> lane) & 1u;
      if (lane == 0) nib[warp] = bits;
    }
    tile_done(false);
  }
}

// Block-wide exclusive scans over kCompactThreads = 32 warps (identity -1
// for the maximum, 0 for the sum): a warp scan, then every warp scans the 32
// warp totals.  `red` holds one int per warp.  Every thread gets the value
// over the threads before it and the block total.
static_assert(kCompactThreads == 1024, "the scans take one warp total per lane");
__device__ __forceinline__ int block_excl_max(int v, int* red, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, v, off);
    if (lane >= off) v = max(v, u);
  }
  int ex = __shfl_up_sync(0xffffffffu, v, 1);
  if (lane == 0) ex = -1;
  if (lane == 31) red[warp] = v;
  __syncthreads();
  int wv = red[lane];
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, wv, off);
    if (lane >= off) wv = max(wv, u);
  }
  const int before = __shfl_sync(0xffffffffu, wv, (warp + 31) & 31);
  *total = __shfl_sync(0xffffffffu, wv, 31);
  __syncthreads();
  return warp > 0 ? max(before, ex) : ex;
}
__device__ __forceinline__ int block_excl_sum(int v, int* red, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int mine = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, v, off);
    if (lane >= off) v += u;
  }
  if (lane == 31) red[warp] = v;
  __syncthreads();
  int wv = red[lane];
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int u = __shfl_up_sync(0xffffffffu, wv, off);
    if (lane >= off) wv += u;
  }
  const int before = __shfl_sync(0xffffffffu, wv, (warp + 31) & 31);
  *total = __shfl_sync(0xffffffffu, wv, 31);
  __syncthreads();
  return (warp > 0 ? before : 0) + v - mine;
}

__device__ __forceinline__ void dn_cluster_sync() {
  asm volatile("barrier.cluster.arrive.release;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire;\n" ::: "memory");
}
__device__ __forceinline__ uint32_t dn_cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}
// Value of an int in the shared memory of CTA `rank` of the cluster, at the
// same offset as `local` in this CTA.
__device__ __forceinline__ int dn_ld_peer(const int* local, uint32_t rank) {
  uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(local)), r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(a), "r"(rank));
  int v;
  asm volatile("ld.shared::cluster.s32 %0, [%1];\n" : "=r"(v) : "r"(r) : "memory");
  return v;
}

// One cluster of kCompactCtas CTAs per context.  A segment is
// kCompactCtas * kCompactThreads pass words (32 tokens each), one per
// thread, CTA r taking the r-th run of kCompactThreads words.  Both scans
// (the last passing position, then the kept counts) go block-wide first;
// each CTA then publishes its block total in shared memory, and after a
// cluster barrier every thread adds the totals of the CTAs before its own
// (distributed shared memory).  The published totals are double-buffered by
// segment parity, so two cluster barriers per segment suffice; a last one
// keeps them readable until every CTA is done.  Every thread of the cluster
// passes the same barriers (all CTAs of a cluster walk the same context).
__global__ void __launch_bounds__(kCompactThreads)
denoise_compact_kernel(const uint32_t* __restrict__ masks, const int32_t* __restrict__ n_tokens,
                       int n_max, int words_stride, int keep_every,
                       int32_t* __restrict__ kept_idx, int32_t* __restrict__ kept_count) {
  constexpr int CS = kCompactCtas;
  constexpr int SEGW = CS * kCompactThreads;  // words per segment
  __shared__ int red[kCompactThreads / 32];
  __shared__ int pub[2][2];  // [segment parity][last passing position, kept count]
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x / CS;
  const int rank = static_cast<int>(dn_cluster_rank());
  const int tid = threadIdx.x;
  int n = n_tokens ? n_tokens[b] : n_max;
  n = n < 0 ? 0 : (n > n_max ? n_max : n);
  const uint32_t* mb = masks + static_cast<long long>(b) * words_stride;
  int32_t* out = kept_idx + static_cast<long long>(b) * n_max;
  const int nw = (n + 31) / 32;  // words that hold tokens
  int carry_last = -1;           // last passing position before the segment
  int carry_cnt = 0;             // tokens kept before the segment
  const int mine = rank * kCompactThreads + tid;  // this thread's word within a segment
  uint32_t next = mine < nw ? mb[mine] : 0u;
  int par = 0;
  for (int w0 = 0; w0 < nw; w0 += SEGW, par ^= 1) {
    const int wi = w0 + mine;
    const uint32_t raw = next;
    if (wi + SEGW < nw) next = mb[wi + SEGW];  // the next segment's word
    const int i0 = 32 * wi;
    const int nv = min(max(n - i0, 0), 32);  // tokens of this word that exist
    const uint32_t valid = nv >= 32 ? ~0u : ((1u << nv) - 1u);
    const uint32_t m = raw & valid;
    const int last = m ? i0 + 31 - __clz(m) : -1;
    int cta_last;
    int lp = block_excl_max(last, red, &cta_last);
    if (tid == 0) pub[par][0] = cta_last;
    dn_cluster_sync();
    int seg_last = carry_last;
    for (int r = 0; r < CS; ++r) {
      const int v = dn_ld_peer(&pub[par][0], static_cast<uint32_t>(r));
      if (r < rank) lp = max(lp, v);
      seg_last = max(seg_last, v);
    }
    lp = max(lp, carry_last);
    uint32_t kept = nv > 0 ? keep_mask(m, lp, i0, keep_every) & valid : 0u;
    int cta_cnt;
    int slot = block_excl_sum(__popc(kept), red, &cta_cnt);
    if (tid == 0) pub[par][1] = cta_cnt;
    dn_cluster_sync();
    int seg_cnt = 0;
    for (int r = 0; r < CS; ++r) {
      const int v = dn_ld_peer(&pub[par][1], static_cast<uint32_t>(r));
      if (r < rank) slot += v;
      seg_cnt += v;
    }
    slot += carry_cnt;
    while (kept) {
      out[slot++] = i0 + __ffs(kept) - 1;
      kept &= kept - 1;
    }
    carry_last = seg_last;
    carry_cnt += seg_cnt;
  }
  dn_cluster_sync();  // the peers' published totals stay readable until here
  if (rank == 0 && tid == 0) kept_count[b] = carry_cnt;
}

}  // namespace cmc

extern "C" {

// [0, B * n_max): one pass byte per token; then, 256-byte aligned, one
// 32-bit pass word per tile of 32 tokens, [B, words_stride] with the row
// stride rounded up to whole 16-byte groups; then, 256-byte aligned, one
// 32-bit tile counter per context (zero-filled once by the caller; every
// call leaves them zero).
static size_t dn_words_offset(int B, int n_max) {
  return cmc::align_up(static_cast<size_t>(B) * static_cast<size_t>(n_max), 256);
}
static int dn_words_stride(int n_max) {
  const int words = (n_max + 31) / 32;
  return (words + cmc::kCompactWords - 1) / cmc::kCompactWords * cmc::kCompactWords;
}

static size_t dn_counters_offset(int B, int n_max) {
  const size_t words = static_cast<size_t>(B) * static_cast<size_t>(dn_words_stride(n_max));
  return cmc::align_up(dn_words_offset(B, n_max) + 4 * words, 256);
}

size_t cmc_denoise_workspace_size(int B, int n_max) {
  if (B < 1 || n_max < 1) return 0;
  return dn_counters_offset(B, n_max) + cmc::align_up(4 * static_cast<size_t>(B), 256);
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
  uint32_t* masks = reinterpret_cast<uint32_t*>(pass + dn_words_offset(B, n_max));
  unsigned int* counters = reinterpret_cast<unsigned int*>(pass + dn_counters_offset(B, n_max));
  static std::atomic<bool> attr_set[64];  // per device: the attribute is set (idempotent)
  int dev = 0;
  int st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  if (dev >= 0 && dev < 64 && !attr_set[dev].load(std::memory_order_acquire)) {
#define CMC_DN_ATTR(GG)                                                                                 \
    st = record_cuda_error(cudaFuncSetAttribute(denoise_pass_kernel<GG, kPassStages, false>,           \
                                                cudaFuncAttributeMaxDynamicSharedMemorySize,           \
                                                pass_smem(kPassStages)));                               \
    if (st != CMC_OK) return st;                                                                        \
    st = record_cuda_error(cudaFuncSetAttribute(denoise_pass_kernel<GG, kPassStages, true>,       \
                                                cudaFuncAttributeMaxDynamicSharedMemorySize,           \
                                                pass_smem(kPassStages)));                          \
    if (st != CMC_OK) return st;
    CMC_DN_ATTR(1) CMC_DN_ATTR(2) CMC_DN_ATTR(3) CMC_DN_ATTR(4)
    CMC_DN_ATTR(5) CMC_DN_ATTR(6) CMC_DN_ATTR(7) CMC_DN_ATTR(8)
#undef CMC_DN_ATTR
    attr_set[dev].store(true, std::memory_order_release);
  }
  const int tiles_per_ctx = (n_max + kPassTile - 1) / kPassTile;
  const long long tiles = static_cast<long long>(B) * tiles_per_ctx;
  long long blocks = tiles;
  const long long cap = static_cast<long long>(sm_count()) * 2 * 64;  // grid-stride beyond
  if (blocks > cap) blocks = cap;
  // Contexts of at most kPassThreads tiles (8,192 tokens): the compaction in
  // the same launch; longer ones: the cluster compaction kernel after the pass.
  const bool fuse = tiles_per_ctx <= kPassThreads;
  switch (g) {
#define CMC_DN_CASE(GG)                                                                             \
  case GG:                                                                                          \
    st = fuse ? launch_pdl(denoise_pass_kernel<GG, kPassStages, true>,                         \
                           dim3(static_cast<unsigned>(blocks)), dim3(kPassThreads),                 \
                           static_cast<size_t>(pass_smem(kPassStages)), s, emb, n_tokens,      \
                           n_max, H, tau, pass, masks, kept_idx, tiles, tiles_per_ctx,              \
                           dn_words_stride(n_max), counters, keep_every, kept_count)                \
              : launch_pdl(denoise_pass_kernel<GG, kPassStages, false>,                             \
                           dim3(static_cast<unsigned>(blocks)), dim3(kPassThreads),                 \
                           static_cast<size_t>(pass_smem(kPassStages)), s, emb, n_tokens, n_max, H, \
                           tau, pass, masks, kept_idx, tiles, tiles_per_ctx,                        \
                           dn_words_stride(n_max), counters, keep_every, kept_count);               \
    break;
    CMC_DN_CASE(1) CMC_DN_CASE(2) CMC_DN_CASE(3) CMC_DN_CASE(4)
    CMC_DN_CASE(5) CMC_DN_CASE(6) CMC_DN_CASE(7) CMC_DN_CASE(8)
#undef CMC_DN_CASE
    default: return CMC_ERR_RANGE;
  }
  if (st != CMC_OK || fuse) return st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = kCompactCtas;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(B) * kCompactCtas);
  cfg.blockDim = dim3(kCompactThreads);
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return record_cuda_error(cudaLaunchKernelEx(&cfg, denoise_compact_kernel,
                                              static_cast<const uint32_t*>(masks), n_tokens, n_max,
                                              dn_words_stride(n_max), keep_every, kept_idx, kept_count));
}

}  // extern "C"
