// Tier-2 ring append, Tier-1 gather and decode attention over the two-tier
// cache (Section 2.5, "Tier-1", "Tier-2: local context window" and "KV cache
// assembly"; cost model in the appendix "Attention MACs Analysis").
//
// Work decomposition.  A unit is one (sequence b, layer l, KV head g).  Its
// keys are cut into tiles of 64: ceil(k / 64) Tier-1 tiles, then ceil(W / 64)
// tiles of ring slots; no tile mixes the two tiers.  With m = resident CTAs
// per unit (at most one per tile, at most 8): m = 1 (the Llama- and
// Mistral-shaped steps) gives one CTA per unit, nothing split; m >= 2 (long
// units, few of them) gives thread-block clusters of m CTAs per unit, each
// CTA taking a contiguous share of the unit's tiles: at the end every CTA
// leaves its fp32 (max, sum, output) record in its own shared memory, and
// after a cluster barrier each CTA merges a slice of the output columns from
// all m records (distributed shared memory, log-sum-exp rescale).  More units
// than resident CTAs: one wave of CTAs, each taking a contiguous run of whole
// units when that is balanced enough, else an equal share of the flattened
// (unit, tile) list (stream-K) with partial records in global memory that a
// small combine kernel following on the stream merges.  No CTA ever
// waits on another outside its cluster's two barriers.
//
// Inside a CTA one producer warp streams the tiles through a ring of shared-
// memory stages.  Ring tiles, and Tier-1 tiles when the Tier-1 rows are the
// first k rows of their tensor (the cache the prefill of M* leaves, or the
// output of cmc_tier1_gather), are two 64-row x 64-column boxes per K and per
// V loaded by the Tensor Memory Accelerator.  Tier-1 tiles gathered by an
// index list are copied with 16-byte cp.async by the producer lanes.  Both
// land in the 128-byte swizzled layout, which places 16-byte chunk c of a row
// at position c ^ (row & 7) within its 128-byte line, so the consumers'
// ldmatrix reads are conflict-free.  Rows that hold no key are masked, and
// their V rows zeroed, so stale or unwritten memory never reaches the output.
// The unit's query rows travel with each tile (1-D bulk copy) and a small
// header written by the producer.  A stage is "full" when its TMA transaction
// bytes (expect_tx / complete_tx) and its cp.async copies
// (cp.async.mbarrier.arrive) have landed; four consumer warps, each owning 16
// keys of a tile, compute
//   S^T = K Q^T   with mma.sync m16n8k16: the warp's 16 keys as the M rows,
//                 the G query heads sharing the KV head as the N = 8 columns
//                 (padded to 8), d in k-steps of 16,
// an online softmax in the log2 domain (running max / sum per head), and
//   O^T += V^T P^T  with mma.sync: 16 rows of the head dimension per m-tile,
//                 the heads as columns, the 16 keys as the k-step; P^T comes
//                 from the S^T accumulators, packed to bf16 and transposed in
//                 registers (movmatrix),
// reading K with ldmatrix and V with ldmatrix.trans, then hand the stage back
// through an "empty" mbarrier.  Every mbarrier wait has a wall-time limit.
// Warps are merged in shared memory at the end of a unit.
//
// K/V rows are read once per launch, so their loads carry an L2 evict-first
// policy.  Before its grid dependency wait (programmatic dependent launch)
// each CTA prefetches its first four box tiles into L2: CTAs that become
// resident in free slots or in the slots of the previous launch's exiting
// CTAs thus pull their first tiles from HBM while that launch drains, and the
// evict-first stream of the running launch does not push them out again.
//
// The fused decode step also appends the new token: the producer copies the
// new token's K/V rows next to the tile that holds its ring slot, a consumer
// warp patches them over the stale ring row in shared memory and stores them
// into the ring.  pos[b] is advanced by the last CTA to read it: each CTA adds
// the number of tiles of sequence b it has read pos[b] for to a per-sequence
// count in the workspace, and the CTA whose addition completes the count
// (L * Hkv * tiles per unit) writes pos[b] + 1 and clears the count.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <atomic>
#include <cstring>
#include <mutex>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kTileKeys = 64;  // keys per pipeline tile
constexpr int kWarps = 4;      // consumer warps; each owns 16 keys of a tile
constexpr int kThreads = 32 * kWarps;
constexpr size_t kWsHeader = 256;
constexpr int kHalfBytes = kTileKeys * 128;  // one 64-row x 128-byte swizzled box
constexpr int kMetaSlots = 4;                // producer metadata prefetch distance (tiles)

// fp32 partial record of one CTA's share of a unit: max[G], sum[G], then, from
// a 16-byte aligned offset, the unnormalised output [G][d].
__host__ __device__ constexpr int rec_out_offset(int G) { return (2 * G + 3) & ~3; }
__host__ __device__ constexpr int rec_floats(int G, int D) { return rec_out_offset(G) + G * D; }

// Tensor maps of one launch (passed by value, in the kernel's parameter space).
struct AttnMaps {
  CUtensorMap rk_box, rv_box;      // ring [units * W, d], box 64 cols x 64 rows
  CUtensorMap t1k_box, t1v_box;    // Tier-1 [units * N, d] (identity selection only)
};

struct AttnParams {
  const uint16_t* q;      // [B, L, Hq, d]
  const uint16_t* t1k;    // [B, L, Hkv, N, d]
  const uint16_t* t1v;    // [B, L, Hkv, N, d]
  const int32_t* idx;     // [B, k], or NULL: Tier-1 is rows 0 .. k-1 of t1k / t1v
  uint16_t* ring_k;       // [B, L, Hkv, W, d]
  uint16_t* ring_v;       // [B, L, Hkv, W, d]
  int64_t* pos;           // [B]
  const uint16_t* k_new;  // [B, L, Hkv, d]   (fused step only)
  const uint16_t* v_new;  // [B, L, Hkv, d]
  uint16_t* out;          // [B, L, Hq, d]
  uint32_t* status;       // workspace status word
  unsigned long long* tickets;  // [B] tiles whose pos read is done (fused step)
  float* partials;        // [units, tpu, G * (d + 2)]
  int B, L, Hq, Hkv, N, k, W;
  int tpu;                // tiles per unit: t1_tiles Tier-1 tiles, then the ring tiles
  int t1_tiles;           // ceil(k / 64)
  int rot;                // in-unit processing order: tile (j + rot) % tpu at position j
  long long base;         // tiles per CTA (CTAs below `rem` take one more)
  long long rem;
  int cm;                 // > 0: clusters of cm CTAs share each unit (CTA j of the cluster
                          // takes positions [j tpu / cm, (j+1) tpu / cm)); 0: flat split
  int gran;               // flat split: tiles per granule (1, or tpu: whole units per CTA)
  float scale_log2;       // softmax scale * log2(e)
  long long rope_offset;  // rotary embedding (GQA-layer step): position of ring token 0
  int l2_prefetch;        // box tiles per CTA prefetched into L2 before the grid dependency wait
  unsigned long long rope_turns[64];  // theta^(-2i/d) / (2 pi) of the d/2 pairs as 0.64 fixed
                                      // point (turns per position), computed on the host
  int rope_slot;          // >= 0: the same table in g_rope_tables[rope_slot] (read from there)
  uint32_t stall_tx;      // 0; the failure-path test hook: bytes every stage expects beyond
                          // what its loads deliver, so that no stage ever completes
};

// Rotary frequency tables in device memory, one per (theta, d) a device has
// seen, written once by the host before the first launch that uses it and
// never changed afterwards.  The producer reads its lanes' two entries with
// plain global loads before the grid dependency wait; reading them from the
// kernel parameters instead (lane-indexed parameter space) measured 0.2-0.3 us
// more per launch.  When no slot is available the parameters are used.
constexpr int kRopeSlots = 16;
__device__ unsigned long long g_rope_tables[kRopeSlots][64];

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// C[16x8] += A[16x16] B[16x8], bf16 inputs, fp32 accumulators (all 16 rows of A).
__device__ __forceinline__ void mma_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                          uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Transpose of an 8x8 matrix of 16-bit elements held one pair per thread
// (thread l: row l/4, columns 2(l%4) and 2(l%4)+1).
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(d) : "r"(a));
  return d;
}

// 2^x with the ex2.approx instruction (ex2(-inf) = +0).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

// Two fp32 -> bf16x2 (round to nearest even); `lo` lands in the low half.
__device__ __forceinline__ uint32_t pack_bf16_rn(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;\n" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// --- mbarrier (shared::cta).  Every wait is bounded in wall time: a waiter
// that has not seen its phase complete kWaitNs after it started polling
// (%globaltimer, nanoseconds) raises the CTA's abort flag, reports
// CMC_DEVFLAG_TIMEOUT and gives up; once the flag is up every other wait of
// the CTA gives up at its next poll.  A poll-count cap backs the deadline up
// in case the timer ever stood still.  Named-barrier and cluster-barrier
// participation never depends on whether a wait succeeded (see the kernel),
// so a CTA whose waits gave up still reaches its end.
constexpr uint32_t kWaitNs = 1000000000u;  // 1 s: the kernel runs for microseconds
constexpr uint32_t kDrainNs = 2000000u;    // after a timeout: wait for issued loads
constexpr uint32_t kMaxWaitPolls = 1u << 28;

// Low 32 bits of %globaltimer (nanoseconds).  Differences of readings less
// than 2^32 ns (4.29 s) apart are exact in unsigned 32-bit arithmetic.
__device__ __forceinline__ uint32_t global_ns32() {
  uint32_t t;
  asm volatile("mov.u32 %0, %%globaltimer_lo;\n" : "=r"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_addr(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}\n" ::"r"(
                   smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile(
      "{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}\n" ::"r"(
          smem_addr(bar)),
      "r"(bytes)
      : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// The CTA's abort flag: raised by the first wait that times out.
__shared__ int attn_abort;

__device__ __forceinline__ bool attn_aborted() { return *static_cast<volatile int*>(&attn_abort) != 0; }

// Waits for the phase of `bar` with the given parity to complete.  False when
// the CTA's abort flag is (or goes) up, or on timeout, which raises it.
__device__ __forceinline__ bool mbar_wait_slow(uint64_t* bar, uint32_t parity) {
  const uint32_t t0 = global_ns32();
  for (uint32_t it = 0; it < kMaxWaitPolls; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if (attn_aborted()) return false;
    if (global_ns32() - t0 > kWaitNs) break;
  }
  *static_cast<volatile int*>(&attn_abort) = 1;
  return false;
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  return mbar_try_wait(bar, parity) || mbar_wait_slow(bar, parity);
}

// --- TMA loads into shared memory, completing on an mbarrier.
// A 2-D TMA box load into shared memory, completing on an mbarrier, with an
// L2 cache policy (createpolicy) attached.
__device__ __forceinline__ void tma_box_hint(uint32_t dst, const CUtensorMap* map, int col, int row,
                                             uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;\n" ::"r"(dst),
      "l"(map), "r"(col), "r"(row), "r"(smem_addr(bar)), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// L2 prefetch of one TMA box and of a contiguous byte range.  These are hints:
// no data reaches the issuing thread and the L2 stays coherent with the
// previous kernel's writes, so they may be issued before the grid dependency
// wait.
__device__ __forceinline__ void tma_prefetch_l2(const CUtensorMap* map, int col, int row) {
  asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];\n" ::"l"(map),
               "r"(col), "r"(row)
               : "memory");
}
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(src), "r"(bytes) : "memory");
}

// Named barrier over the consumer warps only (the producer warp never joins).
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;\n" ::"n"(kWarps * 32) : "memory");
}

// --- thread-block cluster: barrier (every thread of every CTA of the
// cluster arrives, then waits) and loads from a peer CTA's shared memory.
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire;\n" ::: "memory");
}
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t peer_smem(uint32_t local_addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(local_addr), "r"(rank));
  return r;
}
__device__ __forceinline__ float ld_peer_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];\n" : "=f"(v) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ float4 ld_peer_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];\n"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}

// ---------------------------------------------------------------------------
// Shared-memory layout of one pipeline stage (1024-byte aligned)
// ---------------------------------------------------------------------------

template <int D, int G, bool ROPE = false>
struct Stage {
  static constexpr int kHalves = D / 64;               // 128-byte column boxes per row
  static constexpr int kK = 0;                         // K boxes [half][64 rows][128 B]
  static constexpr int kV = kHalves * kHalfBytes;      // V boxes
  static constexpr int kBytes = 2 * kHalves * kHalfBytes;  // a multiple of 1024
  // Small per-stage areas, kept apart so that stages stay 1024-byte aligned:
  static constexpr int kQ = 0;                         // query rows [G][D] bf16
  static constexpr int kNew = G * D * 2;               // new token K row, V row (fused step)
  static constexpr int kHdr = kNew + 2 * D * 2;        // header words (H_*)
  static constexpr int kRope = kHdr + 128;             // rotary table: d/2 (cos, sin) pairs
  static constexpr int kAuxBytes = kRope + (ROPE ? D * 4 : 0);
};

// Per-stage header words: rows of the tile that may hold a key, the new
// token's ring slot and tile row (fused step; -1 if not in this tile),
// whether any of the 64 rows holds no key (its V row must be zeroed), and the
// bit masks of rows 0-31 / 32-63 whose Tier-1 index is out of range.
enum { H_NROWS = 0, H_NEWSLOT = 1, H_NEWROW = 2, H_MASKED = 3, H_BADLO = 4, H_BADHI = 5 };

// Row length (floats) of the end-of-unit merge buffer: d + 4, so that the
// rows of the four head pairs a warp stores to start 8 banks apart and its
// 32 lanes hit distinct banks.
__host__ __device__ constexpr int merge_row_floats(int D) { return D + 4; }

template <int D, int G, int NST, bool ROPE>
constexpr size_t attn_smem_bytes() {
  return 1024 /* alignment slack */ +
         static_cast<size_t>(NST) * (Stage<D, G, ROPE>::kBytes + Stage<D, G, ROPE>::kAuxBytes) +
         kMetaSlots * (kTileKeys * 4 + 16) +
         static_cast<size_t>(kWarps) * (2 * 8 + G * merge_row_floats(D)) * sizeof(float);
}

// Byte offset of 16-byte chunk c (0 .. D/8-1) of tile row r within a K or V
// region: 128-byte column box c / 8, swizzled position (c % 8) ^ (r % 8).
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return static_cast<uint32_t>((c >> 3) * kHalfBytes + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

__device__ __forceinline__ long long cta_first_tile(long long c, long long base, long long rem) {
  return c * base + (c < rem ? c : rem);
}
__device__ __forceinline__ long long cta_of_tile(long long t, long long base, long long rem) {
  const long long big = rem * (base + 1);
  return t < big ? t / (base + 1) : rem + (t - big) / base;
}
// Partial-record slot (tile position within the unit) of CTA c's share of
// the unit whose first tile is ut0: the position of c's first tile in it.
__device__ __forceinline__ long long rec_slot(const AttnParams& p, long long c, long long ut0) {
  const long long t = cta_first_tile(c, p.base, p.rem);
  return t > ut0 ? t - ut0 : 0;
}

// Unit coordinates of the tile at a position of the flattened (unit, j)
// order, advanced one tile at a time so that the main loop does no integer
// division.  Within a unit, position j holds key tile lt = (j + rot) % tpu:
// the ring tiles come first, so a CTA's first loads need no idx entries.
struct TileCursor {
  int u, j, lt, b, l, g;  // unit, position and key tile within it, the unit's (b, l, g)
  __device__ __forceinline__ void init(long long t, const AttnParams& p) {
    const int LH = p.L * p.Hkv;
    u = static_cast<int>(t / p.tpu);
    j = static_cast<int>(t - static_cast<long long>(u) * p.tpu);
    lt = j + p.rot;
    if (lt >= p.tpu) lt -= p.tpu;
    b = u / LH;
    const int lg = u - b * LH;
    l = lg / p.Hkv;
    g = lg - l * p.Hkv;
  }
  __device__ __forceinline__ void next(const AttnParams& p) {
    if (++j == p.tpu) {
      j = 0;
      ++u;
      if (++g == p.Hkv) {
        g = 0;
        if (++l == p.L) {
          l = 0;
          ++b;
        }
      }
    }
    lt = j + p.rot;
    if (lt >= p.tpu) lt -= p.tpu;
  }
};

// What the producer needs to issue one tile -- the idx entries of its 64 rows
// (gathered Tier-1 tiles only) and pos of its sequence -- staged in shared
// memory by asynchronous 4- and 8-byte copies kMetaSlots tiles ahead of their
// use, so the producer never waits on a global load.
struct MetaSlot {
  int32_t idx[kTileKeys];
  long long pos;
  long long pad;
};

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async16_hint(uint32_t dst, const void* src, uint32_t src_bytes,
                                                uint64_t policy) {
  asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2, %3;\n" ::"r"(dst), "l"(src),
               "r"(src_bytes), "l"(policy));
}
// Adds one pending arrival to `bar` now and completes it once every cp.async
// this thread issued so far has landed.
__device__ __forceinline__ void mbar_arrive_cp_async(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.shared::cta.b64 [%0];\n" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ void cp_async_4(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_8(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(dst), "l"(src));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

__device__ __forceinline__ bool gathered_tile(const AttnParams& p, const TileCursor& c) {
  return p.idx != nullptr && c.lt < p.t1_tiles;
}

// Every producer lane commits exactly one copy group per call.
__device__ __forceinline__ void prefetch_meta(const AttnParams& p, const TileCursor& c, bool live,
                                              int lane, MetaSlot* slot) {
  if (live) {
    if (gathered_tile(p, c)) {
      const int key0 = c.lt * kTileKeys;
      const int32_t* irow = p.idx + static_cast<long long>(c.b) * p.k;
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int i = key0 + lane + 32 * e;
        cp_async_4(smem_addr(&slot->idx[lane + 32 * e]), i < p.k ? irow + i : irow, i < p.k ? 4u : 0u);
      }
    }
    if (lane == 0) cp_async_8(smem_addr(&slot->pos), p.pos + c.b);
  }
  cp_async_commit();
}

struct TileMeta {
  long long pos;
  int idx_lo, idx_hi;  // idx entries of rows lane and lane + 32 (gathered tiles)
};

// What a sequence's pos gives every tile of that sequence: the ring slots
// that hold keys and the new token's slot (fused step).  Computed once per
// run of tiles of one sequence.
struct SeqState {
  long long pos;
  int count;     // occupied ring slots (after the append in the fused step)
  int new_slot;  // ring slot of the new token, -1 if none
  bool bad;      // pos < 0: the sequence is skipped
};

template <bool FUSED>
__device__ __forceinline__ SeqState seq_state(const AttnParams& p, long long pos) {
  SeqState q;
  q.pos = pos;
  q.bad = pos < 0;
  q.count = 0;
  q.new_slot = -1;
  if (!q.bad) {
    if (FUSED) {
      q.count = static_cast<int>(pos + 1 < p.W ? pos + 1 : p.W);
      q.new_slot = static_cast<int>(pos % p.W);
    } else {
      q.count = static_cast<int>(pos < p.W ? pos : p.W);
    }
  }
  return q;
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;\n" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

// Rotary embedding of a GQA-layer step: (cos, sin) of the angle
// p * theta^(-2i/d) of pairs i = lane and lane + 32 (i < d/2) at the new
// token's position p = rope_offset + pos.  Angles reach 10^5 rad and more, so
// they are reduced in turns with integer arithmetic: with F_i =
// theta^(-2i/d) / (2 pi) held as a 64-bit binary fraction (rounded on the
// host), p * F_i mod 2^64 is the fractional turn of the angle, off by at most
// p * 2^-65 turns; its top 32 bits, read as a signed fraction of a half turn,
// give the angle in [-pi, pi) for sincospif.  Below p = 2^32 the (cos, sin)
// pairs are within 1e-7 of exact (checked against 200-bit arithmetic); a
// double-precision product p * theta^(-2i/d) would be off by p * 2^-53 rad.
// `turns` holds F_lane and F_(lane+32) (0 past d/2), loaded from the kernel
// parameters before the grid dependency wait.
template <int D>
__device__ __forceinline__ void rope_pairs(const AttnParams& p, long long pos,
                                           const unsigned long long (&turns)[2], int lane,
                                           float2 (&cs)[2]) {
  const unsigned long long pp = static_cast<unsigned long long>(p.rope_offset + pos);
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int i = lane + 32 * e;
    cs[e] = make_float2(1.f, 0.f);
    if (i < D / 2) {
      const unsigned long long frac = pp * turns[e];  // mod 2^64: the fractional turn
      const int hi = static_cast<int>(static_cast<long long>(frac) >> 32);  // [-2^31, 2^31)
      // angle / pi = 2 * turn in [-1, 1)
      const float x = static_cast<float>(hi) * 4.656612873077393e-10f;  // 2^-31
      float sn, cn;
      sincospif(x, &sn, &cn);
      cs[e] = make_float2(cn, sn);
    }
  }
}

// Producer lane 0, box tiles: what does not depend on pos -- the K/V boxes and
// the unit's query rows -- issued as soon as the stage is free.  Two-
// dimensional boxes of 64 consecutive rows of the ring, or of the Tier-1
// tensor under identity selection; rows past the unit's keys are masked later,
// rows past the tensor are zero-filled by the TMA unit.
template <int D, int G>
__device__ __forceinline__ void issue_box_loads(const AttnParams& p, const AttnMaps& maps,
                                                uint8_t* stage, uint8_t* aux, const TileCursor& c,
                                                uint64_t* full) {
  using S = Stage<D, G>;
  constexpr int H = S::kHalves;
  const bool t1 = c.lt < p.t1_tiles;
  const int row = t1 ? c.u * p.N + c.lt * kTileKeys : c.u * p.W + (c.lt - p.t1_tiles) * kTileKeys;
  const CUtensorMap* mk = t1 ? &maps.t1k_box : &maps.rk_box;
  const CUtensorMap* mv = t1 ? &maps.t1v_box : &maps.rv_box;
  const uint32_t sK = smem_addr(stage + S::kK);
  const uint32_t sV = smem_addr(stage + S::kV);
  mbar_expect_tx(full, 2 * H * kHalfBytes + G * D * 2);
  // K/V rows are read once per step: evict-first keeps them from displacing
  // what is worth keeping in L2 (the prefetched first tiles of the next launch)
  const uint64_t pol = policy_evict_first();
#pragma unroll
  for (int h = 0; h < H; ++h) {
    tma_box_hint(sK + h * kHalfBytes, mk, h * 64, row, full, pol);
    tma_box_hint(sV + h * kHalfBytes, mv, h * 64, row, full, pol);
  }
  const uint16_t* qsrc =
      p.q + ((static_cast<long long>(c.b) * p.L + c.l) * p.Hq + static_cast<long long>(c.g) * G) * D;
  bulk_copy(smem_addr(aux + S::kQ), qsrc, G * D * 2, full);
}

// Producer lane 0, before the grid dependency wait: the boxes of a box tile
// (and, for the first tile of a unit, the unit's query rows) prefetched into
// L2.  A CTA that becomes resident while the previous kernel on the stream is
// still running (a free slot, or one that kernel's exiting CTAs freed) thus
// pulls its first tile from HBM during that kernel's tail; its loads after
// the wait then hit L2.
template <int D, int G>
__device__ __forceinline__ void prefetch_box_tile(const AttnParams& p, const AttnMaps& maps,
                                                  const TileCursor& c, bool with_q) {
  constexpr int H = D / 64;
  const bool t1 = c.lt < p.t1_tiles;
  const int row = t1 ? c.u * p.N + c.lt * kTileKeys : c.u * p.W + (c.lt - p.t1_tiles) * kTileKeys;
  const CUtensorMap* mk = t1 ? &maps.t1k_box : &maps.rk_box;
  const CUtensorMap* mv = t1 ? &maps.t1v_box : &maps.rv_box;
#pragma unroll
  for (int h = 0; h < H; ++h) {
    tma_prefetch_l2(mk, h * 64, row);
    tma_prefetch_l2(mv, h * 64, row);
  }
  if (with_q)
    bulk_prefetch_l2(p.q + ((static_cast<long long>(c.b) * p.L + c.l) * p.Hq +
                            static_cast<long long>(c.g) * G) * D,
                     G * D * 2);
}

// Producer warp, once pos (and, for a gathered tile, its idx entries) is
// known: the tile's header (rows that may hold keys, rows with a bad index,
// the new token's row), the new token's K/V rows in the fused step, the loads
// of a gathered tile, and the arrive that, once every byte has landed,
// releases the stage to the consumers.
template <int D, int G, bool FUSED, bool ROPE>
__device__ __forceinline__ void finish_tile(const AttnParams& p, uint8_t* stage, uint8_t* aux,
                                            const TileCursor& c, const TileMeta& meta,
                                            const SeqState& sq, const float2 (&rope)[2], int lane,
                                            uint64_t* full) {
  using S = Stage<D, G, ROPE>;
  if (ROPE) {  // the sequence's rotary table travels with every tile
    float2* tab = reinterpret_cast<float2*>(aux + S::kRope);
    tab[lane] = rope[0];
    if (lane + 32 < D / 2) tab[lane + 32] = rope[1];
    __syncwarp();
  }
  const bool t1 = c.lt < p.t1_tiles;
  int n_rows, new_row = -1;
  if (t1) {
    n_rows = sq.bad ? 0 : min(p.k - c.lt * kTileKeys, kTileKeys);
  } else {
    const int slot0 = (c.lt - p.t1_tiles) * kTileKeys;  // ring slot of row 0
    n_rows = min(max(sq.count - slot0, 0), kTileKeys);
    if (FUSED && sq.new_slot >= slot0 && sq.new_slot - slot0 < n_rows) new_row = sq.new_slot - slot0;
  }
  uint32_t bad_lo = 0, bad_hi = 0;  // rows with an out-of-range index (gathered tiles)
  const bool gath = t1 && p.idx != nullptr;
  if (gath) {
    // Tier-1 rows gathered by idx: 16-byte cp.async copies by the producer
    // lanes (d/8 lanes sweep a row) to the swizzled positions; rows past k and
    // rows with an out-of-range index are zero-filled.  Each lane's copies
    // reach the full barrier through cp.async.mbarrier.arrive.
    constexpr int LPR = D / 8;     // lanes per row
    constexpr int RPP = 32 / LPR;  // rows per pass
    const uint32_t sK = smem_addr(stage + S::kK);
    const uint32_t sV = smem_addr(stage + S::kV);
    const int chunk = lane % LPR;
    const int rsub = lane / LPR;
    const long long ubase = static_cast<long long>(c.u) * p.N * D + chunk * 8;
    const uint64_t pol = policy_evict_first();
#pragma unroll 8
    for (int jj = 0; jj < kTileKeys / RPP; ++jj) {
      const int r = jj * RPP + rsub;
      const int row = __shfl_sync(0xffffffffu, (jj * RPP < 32) ? meta.idx_lo : meta.idx_hi, r & 31);
      const bool ok = r < n_rows && static_cast<unsigned>(row) < static_cast<unsigned>(p.N);
      const long long e = ubase + static_cast<long long>(ok ? row : 0) * D;
      const uint32_t off = swz(r, chunk);
      cp_async16_hint(sK + off, p.t1k + e, ok ? 16u : 0u, pol);
      cp_async16_hint(sV + off, p.t1v + e, ok ? 16u : 0u, pol);
    }
    mbar_arrive_cp_async(full);
    bad_lo = __ballot_sync(0xffffffffu, lane < n_rows && static_cast<unsigned>(meta.idx_lo) >= static_cast<unsigned>(p.N));
    bad_hi = __ballot_sync(0xffffffffu, lane + 32 < n_rows && static_cast<unsigned>(meta.idx_hi) >= static_cast<unsigned>(p.N));
    __syncwarp();
  }
  if (lane == 0) {
    if (bad_lo | bad_hi) atomicOr(p.status, CMC_DEVFLAG_BAD_INDEX);
    if (sq.bad && c.lt == 0) atomicOr(p.status, CMC_DEVFLAG_BAD_POS);
    int* hw = reinterpret_cast<int*>(aux + S::kHdr);
    hw[H_NROWS] = n_rows;
    hw[H_NEWSLOT] = sq.new_slot;
    hw[H_NEWROW] = new_row;
    hw[H_MASKED] = (n_rows < kTileKeys || (bad_lo | bad_hi)) ? 1 : 0;
    hw[H_BADLO] = static_cast<int>(bad_lo);
    hw[H_BADHI] = static_cast<int>(bad_hi);
    uint32_t tx = p.stall_tx;   // 0 outside the failure-path test
    if (gath) tx += G * D * 2;  // query rows (box tiles: issued with the boxes)
    if (new_row >= 0) tx += 2 * D * 2;
    mbar_arrive_expect_tx(full, tx);  // releases the header
    if (gath) {
      const uint16_t* qsrc =
          p.q + ((static_cast<long long>(c.b) * p.L + c.l) * p.Hq + static_cast<long long>(c.g) * G) * D;
      bulk_copy(smem_addr(aux + S::kQ), qsrc, G * D * 2, full);
    }
    if (new_row >= 0) {
      bulk_copy(smem_addr(aux + S::kNew), p.k_new + static_cast<long long>(c.u) * D, D * 2, full);
      bulk_copy(smem_addr(aux + S::kNew + D * 2), p.v_new + static_cast<long long>(c.u) * D, D * 2, full);
    }
  }
}

// Fused step: a CTA has read pos[b] for its run of `tiles` tiles of sequence
// b.  The run that brings the sequence's count to all of its tiles is the last
// reader of pos[b]; it advances pos[b] and clears the count for the next call.
__device__ __forceinline__ void seq_run_done(const AttnParams& p, int b, long long tiles,
                                             const SeqState& sq) {
  const unsigned long long total = static_cast<unsigned long long>(p.L) * p.Hkv * p.tpu;
  const unsigned long long old = atomicAdd(p.tickets + b, static_cast<unsigned long long>(tiles));
  if (old + static_cast<unsigned long long>(tiles) == total) {
    if (!sq.bad) p.pos[b] = sq.pos + 1;
    p.tickets[b] = 0ull;
  }
}

// One CTA = kWarps consumer warps + 1 producer warp.  The producer streams
// the CTA's tiles through NST shared-memory stages; stage s is handed over by
// full[s] (its bytes have landed and its header is written) and handed back
// by empty[s] (every consumer warp is done with it).
template <int D, int G, bool FUSED, int NST, bool ROPE>
__global__ void __launch_bounds__(kThreads + 32)
two_tier_attn_kernel(const __grid_constant__ AttnMaps maps, const AttnParams p) {
  using S = Stage<D, G, ROPE>;
  constexpr int KS = D / 16;  // k-steps of the Q K^T product
  constexpr int DP = merge_row_floats(D);  // padded row of the merge buffer
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* aux0 = smem + NST * S::kBytes;                              // NST aux areas
  uint8_t* meta0 = aux0 + NST * S::kAuxBytes;                          // kMetaSlots slots
  float* merge_m = reinterpret_cast<float*>(meta0 + kMetaSlots * sizeof(MetaSlot));  // [kWarps][8]
  float* merge_l = merge_m + kWarps * 8;                               // [kWarps][8]
  float* merge_o = merge_l + kWarps * 8;                               // [kWarps][G][D]
  __shared__ __align__(8) uint64_t full_bar[NST];
  __shared__ __align__(8) uint64_t empty_bar[NST];

  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;

  const long long cta = blockIdx.x;
  long long t_begin, t_end;
  if (p.cm > 0) {  // clusters of cm CTAs per unit
    const long long u = cta / p.cm;
    const int j = static_cast<int>(cta - u * p.cm);
    t_begin = u * p.tpu + (static_cast<long long>(j) * p.tpu) / p.cm;
    t_end = u * p.tpu + (static_cast<long long>(j + 1) * p.tpu) / p.cm;
  } else {
    t_begin = cta_first_tile(cta, p.base, p.rem) * p.gran;
    t_end = t_begin + (p.base + (cta < p.rem ? 1 : 0)) * p.gran;
  }
  const int n_tiles = static_cast<int>(t_end - t_begin);

  if (tid == 0) {
    for (int s = 0; s < NST; ++s) {
      mbar_init(&full_bar[s], 1);        // the producer's arrive (plus tracked cp.async arrivals)
      mbar_init(&empty_bar[s], kWarps);  // one arrive per consumer warp
    }
    attn_abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
  }
  __syncthreads();
  if (warp == kWarps && lane == 0 && p.l2_prefetch > 0) {
    asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.rk_box) : "memory");
    asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.rv_box) : "memory");
    if (p.idx == nullptr && p.k > 0) {
      asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.t1k_box) : "memory");
      asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.t1v_box) : "memory");
    }
    TileCursor cp;
    cp.init(t_begin, p);
    const int npf = n_tiles < p.l2_prefetch ? n_tiles : p.l2_prefetch;
    for (int i = 0; i < npf; ++i) {
      if (!gathered_tile(p, cp)) prefetch_box_tile<D, G>(p, maps, cp, i == 0 || cp.j == 0);
      cp.next(p);
    }
  }
  // The producer lanes' rotary frequencies from their device table (written
  // long before this launch, never by the kernel before it).
  unsigned long long turns_g[2] = {0ull, 0ull};
  if (ROPE && warp == kWarps && p.rope_slot >= 0) {
    turns_g[0] = g_rope_tables[p.rope_slot][lane];
    if (lane + 32 < D / 2) turns_g[1] = g_rope_tables[p.rope_slot][lane + 32];
  }
  // Programmatic dependent launch: everything above overlapped the previous
  // kernel; inputs may be that kernel's outputs, so wait for it here.  Then let
  // the combine kernel that follows launch early.
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  if (warp == kWarps) {
    // ======================= producer warp =======================
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.rk_box) : "memory");
      asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.rv_box) : "memory");
      if (p.idx == nullptr && p.k > 0) {
        asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.t1k_box) : "memory");
        asm volatile("prefetch.tensormap [%0];\n" ::"l"(&maps.t1v_box) : "memory");
      }
    }
    TileCursor cm, ci;  // tile whose metadata is prefetched, tile issued
    cm.init(t_begin, p);
    ci = cm;
    MetaSlot* slots = reinterpret_cast<MetaSlot*>(meta0);
#pragma unroll
    for (int m = 0; m < kMetaSlots; ++m) {
      prefetch_meta(p, cm, m < n_tiles, lane, &slots[m]);
      cm.next(p);
    }
    {
      // The box tiles of the first NST stages: their loads do not depend on
      // pos, so they go out before any metadata has arrived.
      TileCursor cl = ci;
      for (int i = 0; i < NST && i < n_tiles; ++i) {
        if (lane == 0 && !gathered_tile(p, cl))
          issue_box_loads<D, G>(p, maps, smem + i * S::kBytes, aux0 + i * S::kAuxBytes, cl, &full_bar[i]);
        cl.next(p);
      }
    }
    int issued = 0;
    int run_b = -1;           // sequence of the current run of tiles
    long long run_tiles = 0;  // tiles in that run so far
    SeqState sq;
    sq.pos = 0; sq.count = 0; sq.new_slot = -1; sq.bad = true;
    float2 rope[2] = {make_float2(1.f, 0.f), make_float2(1.f, 0.f)};
    unsigned long long turns[2] = {0ull, 0ull};  // this lane's rotary frequencies (ROPE)
    if (ROPE) {
      if (p.rope_slot >= 0) {
        turns[0] = turns_g[0];
        turns[1] = turns_g[1];
      } else {
        turns[0] = p.rope_turns[lane];
        if (lane + 32 < D / 2) turns[1] = p.rope_turns[lane + 32];
      }
    }
    for (int i = 0; i < n_tiles; ++i) {
      const int s = i % NST;
      if (i >= NST) {
        // Lane 0 waits for the consumers to release the stage; the warp barrier
        // orders the other lanes' copies into it after that, and the broadcast
        // makes the whole warp leave together if the wait gave up.
        int ok = 0;
        if (lane == 0) ok = mbar_wait(&empty_bar[s], static_cast<uint32_t>((i / NST - 1) & 1)) ? 1 : 0;
        __syncwarp();
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        if (lane == 0 && !gathered_tile(p, ci))
          issue_box_loads<D, G>(p, maps, smem + s * S::kBytes, aux0 + s * S::kAuxBytes, ci, &full_bar[s]);
      }
      MetaSlot* ms = &slots[i % kMetaSlots];
      cp_async_wait<kMetaSlots - 1>();  // this tile's metadata has landed
      __syncwarp();
      TileMeta meta;
      meta.pos = ms->pos;
      meta.idx_lo = meta.idx_hi = -1;
      if (gathered_tile(p, ci)) {
        meta.idx_lo = ms->idx[lane];
        meta.idx_hi = ms->idx[lane + 32];
      }
      if (ci.b != run_b) {  // a new sequence: pos-derived state, once per run
        if (FUSED && run_b >= 0 && lane == 0) seq_run_done(p, run_b, run_tiles, sq);
        run_b = ci.b;
        run_tiles = 0;
        sq = seq_state<FUSED>(p, meta.pos);
        if (ROPE && !sq.bad) rope_pairs<D>(p, meta.pos, turns, lane, rope);
      }
      ++run_tiles;
      finish_tile<D, G, FUSED, ROPE>(p, smem + s * S::kBytes, aux0 + s * S::kAuxBytes, ci, meta, sq,
                                     rope, lane, &full_bar[s]);
      ci.next(p);
      issued = i + 1;
      __syncwarp();
      prefetch_meta(p, cm, i + kMetaSlots < n_tiles, lane, ms);  // the slot just read
      cm.next(p);
    }
    if (FUSED && run_b >= 0 && issued == n_tiles && lane == 0) seq_run_done(p, run_b, run_tiles, sq);
    cp_async_wait<0>();  // this lane's cp.async copies (metadata, gathered rows) have landed
    // No CTA exits while bulk loads it issued may still be writing into its
    // shared memory.  Normally the consumers have waited for every stage but
    // the last few, and this wait for the last issued stage covers the rest
    // (a stage's bytes complete its barrier phase).  If waits gave up (abort
    // flag), barrier phases are no evidence, so the warp stays kDrainNs longer
    // -- every bulk load was issued before that, and loads of valid addresses
    // land within microseconds -- with a sleep-count cap behind the timer.
    if (lane == 0 && issued > 0 &&
        !mbar_wait(&full_bar[(issued - 1) % NST], static_cast<uint32_t>(((issued - 1) / NST) & 1))) {
      const uint32_t t0 = global_ns32();
      for (uint32_t it = 0; it < (1u << 16) && global_ns32() - t0 < kDrainNs; ++it) __nanosleep(1000);
    }
    if (lane == 0 && attn_aborted()) atomicOr(p.status, CMC_DEVFLAG_TIMEOUT);
    __syncwarp();
    // A cluster plan: the consumers of every CTA of the cluster pass two
    // cluster barriers at the end of their (one) unit; this warp passes the
    // same two, so every thread of the cluster arrives at each.
    if (p.cm > 0) {
      cluster_sync_all();
      cluster_sync_all();
    }
    return;
  }

  // ======================= consumer warps =======================
  // Both products take the warp's 16 keys (S^T = K Q^T) or 16 rows of the
  // head dimension (O^T = V^T P^T) as the M rows of m16n8k16 and the query
  // heads of the group as the N = 8 columns, so no M row is padding.
  // Fragment coordinates: gq = lane / 4, tq = lane % 4.  S^T: keys gq and
  // gq + 8 of the warp's 16, heads 2 tq and 2 tq + 1.  O^T m-tile mt: head
  // dimension rows 16 mt + gq and 16 mt + 8 + gq, heads 2 tq and 2 tq + 1.
  // A thread keeps the running max and sum of heads 2 tq and 2 tq + 1
  // (heads >= G are padding: zero queries, never written out).
  const int gq = lane >> 2;
  const int tq = lane & 3;
  constexpr int MT = D / 16;  // m-tiles of O^T
  TileCursor cc;
  cc.init(t_begin, p);
  int cur_u = -1;
  uint32_t qa[KS][2];  // Q^T fragments (B operand): head gq, columns of k-step ks
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  float o[MT][4];
#pragma unroll
  for (int j = 0; j < MT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
#pragma unroll
  for (int ks = 0; ks < KS; ++ks) qa[ks][0] = qa[ks][1] = 0u;

  for (int i = 0; i < n_tiles; ++i) {
    const int s = i % NST;
    uint8_t* stage = smem + s * S::kBytes;
    const uint8_t* aux = aux0 + s * S::kAuxBytes;
    // A stage whose wait gave up (this warp's or another's: the CTA's abort
    // flag) is skipped: no key, no patch.  The vote makes that decision the
    // same for every lane of the warp (the shuffles and votes below take the
    // whole warp); barrier participation below does not depend on it.
    const bool dead = __any_sync(0xffffffffu, attn_aborted() ||
                                                  !mbar_wait(&full_bar[s], static_cast<uint32_t>((i / NST) & 1)));
    const int* hw = reinterpret_cast<const int*>(aux + S::kHdr);
    const int u = cc.u;
    const int n_rows = dead ? 0 : hw[H_NROWS];
    const int new_row = dead ? -1 : hw[H_NEWROW];
    // bit r: row r holds a key (the new token's row included)
    const unsigned long long keys =
        (n_rows >= kTileKeys ? ~0ull : ((1ull << n_rows) - 1ull)) &
        ~((static_cast<unsigned long long>(static_cast<uint32_t>(hw[H_BADHI])) << 32) |
          static_cast<uint32_t>(hw[H_BADLO]));
    bool wrote_stage = false;  // generic-proxy writes into the stage by this warp

    if (FUSED && new_row >= 0 && (new_row >> 4) == warp) {
      // Patch the new token over its stale ring row (swizzled) and append it
      // to the ring in global memory.  Each consumer warp reads only its own
      // 16 rows of K and V, so the warp that owns the row does it alone.
      if (lane < 2 * (D / 8)) {
        const int which = lane / (D / 8);  // 0: K, 1: V
        const int c = lane - which * (D / 8);
        uint4 v = *reinterpret_cast<const uint4*>(aux + S::kNew + which * D * 2 + c * 16);
        if (ROPE && which == 0) {
          // rotate the new key: columns 8c .. 8c+7 with their partners in the
          // other half (chunk c ^ d/16), round to bf16
          const uint4 pv = *reinterpret_cast<const uint4*>(aux + S::kNew + (c ^ (D / 16)) * 16);
          const float2* tab = reinterpret_cast<const float2*>(aux + S::kRope);
          const int i0 = (8 * c) & (D / 2 - 1);
          const float sg = (8 * c < D / 2) ? -1.f : 1.f;
          const uint32_t xs[4] = {v.x, v.y, v.z, v.w};
          const uint32_t ps[4] = {pv.x, pv.y, pv.z, pv.w};
          uint32_t r[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 t0 = tab[i0 + 2 * e], t1 = tab[i0 + 2 * e + 1];
            const float lo = fmaf(bf16lo_to_f32(xs[e]), t0.x, sg * bf16lo_to_f32(ps[e]) * t0.y);
            const float hi = fmaf(bf16hi_to_f32(xs[e]), t1.x, sg * bf16hi_to_f32(ps[e]) * t1.y);
            r[e] = pack_bf16_rn(lo, hi);
          }
          v = make_uint4(r[0], r[1], r[2], r[3]);
        }
        *reinterpret_cast<uint4*>(stage + (which ? S::kV : S::kK) + swz(new_row, c)) = v;
        uint16_t* ring = which ? p.ring_v : p.ring_k;
        *reinterpret_cast<uint4*>(ring + (static_cast<long long>(u) * p.W + hw[H_NEWSLOT]) * D + c * 8) = v;
      }
      __syncwarp();
      wrote_stage = true;
    }

    if (u != cur_u) {  // first tile of a unit in this CTA
      cur_u = u;
      const uint8_t* qs = aux + S::kQ;
      if (ROPE && gq < G && !dead) {
        // rotate the query: column c of the first half pairs with c + d/2,
        // and k-step ks + KS/2 holds exactly those partners, so each pair of
        // columns is read once and gives both rotated values
        const float2* tab = reinterpret_cast<const float2*>(aux + S::kRope);
#pragma unroll
        for (int ks = 0; ks < KS / 2; ++ks) {
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            const int c = 16 * ks + 2 * tq + 8 * hf;  // < d/2
            const uint32_t xv = *reinterpret_cast<const uint32_t*>(qs + (gq * D + c) * 2);
            const uint32_t pv = *reinterpret_cast<const uint32_t*>(qs + (gq * D + c + D / 2) * 2);
            const float2 t0 = tab[c], t1 = tab[c + 1];
            const float xl = bf16lo_to_f32(xv), xh = bf16hi_to_f32(xv);
            const float pl = bf16lo_to_f32(pv), ph = bf16hi_to_f32(pv);
            qa[ks][hf] = pack_bf16_rn(fmaf(xl, t0.x, -1.f * pl * t0.y), fmaf(xh, t1.x, -1.f * ph * t1.y));
            qa[ks + KS / 2][hf] = pack_bf16_rn(fmaf(pl, t0.x, 1.f * xl * t0.y), fmaf(ph, t1.x, 1.f * xh * t1.y));
          }
        }
      }
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        if (gq < G && !dead) {
          if (ROPE) {
            // rotated above
          } else {
            qa[ks][0] = *reinterpret_cast<const uint32_t*>(qs + gq * D * 2 + (16 * ks + 2 * tq) * 2);
            qa[ks][1] = *reinterpret_cast<const uint32_t*>(qs + gq * D * 2 + (16 * ks + 2 * tq + 8) * 2);
          }
        }
      }
      m_run[0] = m_run[1] = -INFINITY;
      l_run[0] = l_run[1] = 0.f;
#pragma unroll
      for (int j = 0; j < MT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    }

    if (n_rows > 0) {
      if (hw[H_MASKED]) {
        // Zero the V rows of this warp's 16 keys that hold no key: their
        // probabilities are 0, but the rows may hold stale or unwritten
        // memory, and 0 times a non-finite value is not 0.
        constexpr int CPR = D / 8;  // 16-byte chunks per row
        for (int x = lane; x < 16 * CPR; x += 32) {
          const int r = 16 * warp + x / CPR;
          if (!((keys >> r) & 1ull))
            *reinterpret_cast<uint4*>(stage + S::kV + swz(r, x % CPR)) = make_uint4(0u, 0u, 0u, 0u);
        }
        __syncwarp();
        wrote_stage = true;
      }
      const uint32_t sK = smem_addr(stage + S::kK);
      const uint32_t sV = smem_addr(stage + S::kV);
      // ---- S^T = K Q^T over this warp's 16 keys: 16 x 8 per k-step, in
      // four independent accumulator chains (the last tile's latency is on
      // every launch's critical path) ----
      float sacc[4][4];
#pragma unroll
      for (int cidx = 0; cidx < 4; ++cidx) sacc[cidx][0] = sacc[cidx][1] = sacc[cidx][2] = sacc[cidx][3] = 0.f;
      {
        // ldmatrix x4: lanes 0-7 / 8-15 / 16-23 / 24-31 address keys 0-7 / 8-15 /
        // 0-7 / 8-15 at columns 16 ks .. +7 / same / 16 ks + 8 .. +15 / same
        const int key = 16 * warp + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4(sK + swz(key, 2 * ks + (lane >> 4)), a0, a1, a2, a3);
          mma_16816(sacc[ks & 3], a0, a1, a2, a3, qa[ks][0], qa[ks][1]);
        }
      }
      float sa[4], sb[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        sa[e] = sacc[0][e] + sacc[2][e];
        sb[e] = sacc[1][e] + sacc[3][e];
      }
      // ---- online softmax (log2 domain), heads 2 tq and 2 tq + 1 ----
      const bool ok0 = (keys >> (16 * warp + gq)) & 1ull;
      const bool ok1 = (keys >> (16 * warp + gq + 8)) & 1ull;
      float v[4];
      v[0] = ok0 ? (sa[0] + sb[0]) * p.scale_log2 : -INFINITY;
      v[1] = ok0 ? (sa[1] + sb[1]) * p.scale_log2 : -INFINITY;
      v[2] = ok1 ? (sa[2] + sb[2]) * p.scale_log2 : -INFINITY;
      v[3] = ok1 ? (sa[3] + sb[3]) * p.scale_log2 : -INFINITY;
      float mx0 = fmaxf(v[0], v[2]), mx1 = fmaxf(v[1], v[3]);
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {  // over the 8 key rows (lane bits 2-4)
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
      }
      const float mn0 = fmaxf(m_run[0], mx0), mn1 = fmaxf(m_run[1], mx1);
      float alpha0 = 1.f, alpha1 = 1.f;
      float pr[4] = {0.f, 0.f, 0.f, 0.f};
      if (mn0 != -INFINITY) {
        alpha0 = ex2(m_run[0] - mn0);
        pr[0] = ex2(v[0] - mn0);
        pr[2] = ex2(v[2] - mn0);
      }
      if (mn1 != -INFINITY) {
        alpha1 = ex2(m_run[1] - mn1);
        pr[1] = ex2(v[1] - mn1);
        pr[3] = ex2(v[3] - mn1);
      }
      m_run[0] = mn0;
      m_run[1] = mn1;
      l_run[0] = l_run[0] * alpha0 + (pr[0] + pr[2]);
      l_run[1] = l_run[1] * alpha1 + (pr[1] + pr[3]);
      if (!__all_sync(0xffffffffu, alpha0 == 1.f && alpha1 == 1.f)) {
#pragma unroll
        for (int j = 0; j < MT; ++j) {
          o[j][0] *= alpha0;
          o[j][1] *= alpha1;
          o[j][2] *= alpha0;
          o[j][3] *= alpha1;
        }
      }
      // ---- O^T += V^T P^T ----
      // P^T as the B operand: the S^T fragments (keys gq / gq + 8, heads
      // 2 tq, 2 tq + 1) packed to bf16 and transposed (head gq, keys 2 tq, +1)
      const uint32_t pb0 = movmatrix_trans(pack_bf16_rn(pr[0], pr[1]));
      const uint32_t pb1 = movmatrix_trans(pack_bf16_rn(pr[2], pr[3]));
      {
        // ldmatrix x4 .trans of V: lanes 0-7 / 8-15 / 16-23 / 24-31 address
        // keys 0-7 / 0-7 / 8-15 / 8-15 at columns 16 mt .. +7 / 16 mt + 8 .. +15 / ...
        const int key = 16 * warp + (lane & 7) + ((lane >> 4) & 1) * 8;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4_t(sV + swz(key, 2 * mt + ((lane >> 3) & 1)), a0, a1, a2, a3);
          mma_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
        }
      }
    }
    if (wrote_stage) {
      // generic-proxy writes to this stage must be ordered before the
      // producer's next TMA writes into it
      asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty_bar[s]);  // this warp is done with stage s

    // ---- end of a unit within this CTA: merge warps, write out or a partial ----
    const bool unit_end = (i + 1 == n_tiles) || (cc.j == p.tpu - 1);
    if (unit_end) {
      // Merge the four warps' states of each head: every warp leaves its
      // running max, sum and unnormalised output (rows of DP floats, padded so
      // that the warp's stores hit distinct banks); after one barrier each
      // thread takes four columns of one head, rescales the warps' outputs and
      // sums to the heads' common max and adds them in warp order.
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {  // sums over the 8 key rows
        l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], off);
        l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], off);
      }
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int hh = 2 * tq + e;
        if (hh < G) {
          float* ow = merge_o + (warp * G + hh) * DP;
#pragma unroll
          for (int j = 0; j < MT; ++j) {
            ow[16 * j + gq] = o[j][e];
            ow[16 * j + 8 + gq] = o[j][2 + e];
          }
          if (gq == 0) {
            merge_m[warp * 8 + hh] = m_run[e];
            merge_l[warp * 8 + hh] = l_run[e];
          }
        }
      }
      consumer_sync();

      // The unit is whole in this CTA unless the CTA's tile range cuts it; a
      // cut unit's record goes to the slot of this CTA's first tile in it.
      const long long ut0 = static_cast<long long>(u) * p.tpu;
      const bool whole = ut0 >= t_begin && ut0 + p.tpu <= t_end;
      const long long out_base =
          ((static_cast<long long>(cc.b) * p.L + cc.l) * p.Hq + static_cast<long long>(cc.g) * G) * D;
      constexpr int NGR = G * D / 4;                      // 4-column groups of the unit's output
      constexpr int XPT = (NGR + kThreads - 1) / kThreads;  // groups per thread
      const bool clus = !whole && p.cm > 0;
      float4 cacc[XPT];
      float cls[XPT];
#pragma unroll
      for (int xi = 0; xi < XPT; ++xi) {
        const int x = tid + xi * kThreads;
        if (x >= NGR) break;
        const int hh = (4 * x) / D;
        const int c = (4 * x) % D;
        float M = merge_m[hh];
#pragma unroll
        for (int w = 1; w < kWarps; ++w) M = fmaxf(M, merge_m[w * 8 + hh]);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        float Ls = 0.f;
        if (M != -INFINITY) {
#pragma unroll
          for (int w = 0; w < kWarps; ++w) {
            const float f = ex2(merge_m[w * 8 + hh] - M);
            const float4 v = *reinterpret_cast<const float4*>(merge_o + (w * G + hh) * DP + c);
            acc.x = fmaf(f, v.x, acc.x); acc.y = fmaf(f, v.y, acc.y);
            acc.z = fmaf(f, v.z, acc.z); acc.w = fmaf(f, v.w, acc.w);
            Ls = fmaf(f, merge_l[w * 8 + hh], Ls);
          }
        }
        if (whole) {
          const float inv = Ls > 0.f ? __fdividef(1.f, Ls) : 0.f;
          *reinterpret_cast<uint2*>(p.out + out_base + hh * D + c) =
              make_uint2(pack_bf16_rn(acc.x * inv, acc.y * inv), pack_bf16_rn(acc.z * inv, acc.w * inv));
        } else if (clus) {  // merged across the cluster below
          cacc[xi] = acc;
          cls[xi] = Ls;
        } else {  // merged by two_tier_combine_kernel
          constexpr int PW = rec_floats(G, D);
          float* rec = p.partials + (ut0 + (ut0 > t_begin ? 0 : t_begin - ut0)) * PW;
          if (c == 0) {
            rec[hh] = M;
            rec[G + hh] = Ls;
          }
          *reinterpret_cast<float4*>(rec + rec_out_offset(G) + hh * D + c) = acc;
        }
      }
      if (clus) {
        // Each CTA of the cluster holds one share of the unit.  Its (max, sum,
        // output) record goes to its own shared memory (over the merge
        // buffer, now read); after a cluster barrier every CTA merges a slice
        // of the output columns from all the records (log-sum-exp rescale, in
        // rank order) and writes them; a second barrier keeps each record
        // alive until every peer has read it.
        float* rec = merge_o;
        consumer_sync();
#pragma unroll
        for (int xi = 0; xi < XPT; ++xi) {
          const int x = tid + xi * kThreads;
          if (x >= NGR) break;
          const int hh = (4 * x) / D;
          const int c = (4 * x) % D;
          if (c == 0) {  // merge_m still holds the warps' maxima
            float M = merge_m[hh];
#pragma unroll
            for (int w = 1; w < kWarps; ++w) M = fmaxf(M, merge_m[w * 8 + hh]);
            rec[hh] = M;
            rec[G + hh] = cls[xi];
          }
          *reinterpret_cast<float4*>(rec + rec_out_offset(G) + hh * D + c) = cacc[xi];
        }
        cluster_sync_all();
        const int cm = p.cm;
        const int rank = static_cast<int>(cluster_ctarank());
        const int x0 = (rank * NGR) / cm, x1 = ((rank + 1) * NGR) / cm;
        const uint32_t rec_local = smem_addr(rec);
        for (int x = x0 + tid; x < x1; x += kThreads) {
          const int hh = (4 * x) / D;
          const int c = (4 * x) % D;
          float M = -INFINITY;
          for (int r = 0; r < cm; ++r)
            M = fmaxf(M, ld_peer_f32(peer_smem(rec_local + hh * 4, r)));
          float Ls = 0.f;
          float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
          if (M != -INFINITY) {
            for (int r = 0; r < cm; ++r) {
              const uint32_t base = peer_smem(rec_local, r);
              const float f = ex2(ld_peer_f32(base + hh * 4) - M);
              const float4 o4 = ld_peer_f4(base + (rec_out_offset(G) + hh * D + c) * 4);
              Ls = fmaf(f, ld_peer_f32(base + (G + hh) * 4), Ls);
              O.x = fmaf(f, o4.x, O.x);
              O.y = fmaf(f, o4.y, O.y);
              O.z = fmaf(f, o4.z, O.z);
              O.w = fmaf(f, o4.w, O.w);
            }
          }
          const float inv = Ls > 0.f ? __frcp_rn(Ls) : 0.f;
          *reinterpret_cast<uint2*>(p.out + out_base + hh * D + c) =
              make_uint2(pack_bf16_rn(O.x * inv, O.y * inv), pack_bf16_rn(O.z * inv, O.w * inv));
        }
        cluster_sync_all();
      }
      if (i + 1 < n_tiles) consumer_sync();  // merge buffers are reused by the next unit
    }
    cc.next(p);
  }
  if (tid == 0 && attn_aborted()) atomicOr(p.status, CMC_DEVFLAG_TIMEOUT);
}

// Finishes the units that two_tier_attn_kernel split between CTAs: merges
// their fp32 partial records (max, sum, output per head) with a log-sum-exp
// rescale and writes the bf16 output.  Runs after two_tier_attn_kernel on the
// same stream, only when some unit was split; one CTA per unit.
template <int D, int G>
__global__ void __launch_bounds__(kThreads)
two_tier_combine_kernel(const AttnParams p) {
  asm volatile("griddepcontrol.wait;\n" ::: "memory");  // the attention kernel's records
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  const int u = blockIdx.x;
  const int LH = p.L * p.Hkv;
  const int b = u / LH;
  const int lg = u - b * LH;
  const int l = lg / p.Hkv;
  const int g = lg - l * p.Hkv;
  const long long ut0 = static_cast<long long>(u) * p.tpu;
  const long long c0 = cta_of_tile(ut0, p.base, p.rem);
  const long long c1 = cta_of_tile(ut0 + p.tpu - 1, p.base, p.rem);
  if (c0 == c1) return;  // written by the attention kernel
  // one record per CTA that holds part of the unit, at the slot of that
  // CTA's first tile in the unit (slot 0 for c0)
  const int nrec = static_cast<int>(c1 - c0 + 1);
  constexpr int PW = rec_floats(G, D);
  const float* recs = p.partials + ut0 * PW;
  const long long out_base =
      ((static_cast<long long>(b) * p.L + l) * p.Hq + static_cast<long long>(g) * G) * D;
  for (int x = threadIdx.x; x < G * D / 2; x += blockDim.x) {
    const int hh = (2 * x) / D;
    const int c = (2 * x) % D;
    float M = -INFINITY;
    for (int r = 0; r < nrec; ++r) M = fmaxf(M, recs[rec_slot(p, c0 + r, ut0) * PW + hh]);
    float Ls = 0.f, O0 = 0.f, O1 = 0.f;
    if (M != -INFINITY) {
      for (int r = 0; r < nrec; ++r) {
        const float* pr = recs + rec_slot(p, c0 + r, ut0) * PW;
        const float f = ex2(pr[hh] - M);
        const float2 o2 = *reinterpret_cast<const float2*>(pr + rec_out_offset(G) + hh * D + c);
        Ls = fmaf(f, pr[G + hh], Ls);
        O0 = fmaf(f, o2.x, O0);
        O1 = fmaf(f, o2.y, O1);
      }
    }
    const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
    *reinterpret_cast<uint32_t*>(p.out + out_base + hh * D + c) = pack_bf16x2(O0 * inv, O1 * inv);
  }
}

__global__ void window_append_kernel(uint16_t* __restrict__ ring_k, uint16_t* __restrict__ ring_v,
                                     int64_t* __restrict__ pos, const uint16_t* __restrict__ k_new,
                                     const uint16_t* __restrict__ v_new, int LH, int W, int d) {
  const int b = blockIdx.x;
  const long long pb = pos[b];
  if (pb >= 0) {
    const int slot = static_cast<int>(pb % W);
    const int vpr = d / 8;  // 16-byte vectors per row
    const int total = LH * vpr;
    for (int t = threadIdx.x; t < total; t += blockDim.x) {
      const int row = t / vpr;
      const int v = t - row * vpr;
      const long long unit = static_cast<long long>(b) * LH + row;
      reinterpret_cast<uint4*>(ring_k + (unit * W + slot) * d)[v] =
          reinterpret_cast<const uint4*>(k_new + unit * d)[v];
      reinterpret_cast<uint4*>(ring_v + (unit * W + slot) * d)[v] =
          reinterpret_cast<const uint4*>(v_new + unit * d)[v];
    }
  }
  __syncthreads();  // every thread has read pos[b]
  if (threadIdx.x == 0 && pb >= 0) pos[b] = pb + 1;
}

// Tier-1 compaction (the "M*" of Section 2.5, formed once per question):
//   tier1[b, l, g, i] = bank[b, l, g, idx[b, i]]   for i < k.
// A CTA copies a block of kGatherRows output rows of one unit: each thread
// issues all of its 16-byte streaming loads (K and V) before its stores, so a
// whole block is in flight at once.  Out-of-range indices give a zero row and
// CMC_DEVFLAG_BAD_INDEX.
constexpr int kGatherRows = 64;
constexpr int kGatherThreads = 256;

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

template <int CPR>  // 16-byte chunks per row: d / 8
__global__ void __launch_bounds__(kGatherThreads)
tier1_gather_kernel(const uint4* __restrict__ bank_k, const uint4* __restrict__ bank_v,
                    const int32_t* __restrict__ idx, uint4* __restrict__ out_k,
                    uint4* __restrict__ out_v, uint32_t* status, long long blocks, int row_blocks,
                    int LH, int N, int k) {
  constexpr int kPer = kGatherRows * CPR / kGatherThreads;  // chunks per thread and tensor
  pdl_wait();
  pdl_trigger();
  bool bad = false;
  for (long long blk = blockIdx.x; blk < blocks; blk += gridDim.x) {
    const long long u = blk / row_blocks;
    const int i0 = static_cast<int>(blk - u * row_blocks) * kGatherRows;
    const int32_t* irow = idx + (u / LH) * k;
    uint4 kv[kPer], vv[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int x = threadIdx.x + e * kGatherThreads;
      const int i = i0 + x / CPR;
      kv[e] = vv[e] = make_uint4(0u, 0u, 0u, 0u);
      if (i < k) {
        const int j = __ldg(irow + i);
        if (static_cast<unsigned>(j) < static_cast<unsigned>(N)) {
          const long long src = (u * N + j) * CPR + x % CPR;
          kv[e] = ld_stream(bank_k + src);
          vv[e] = ld_stream(bank_v + src);
        } else {
          bad = true;
        }
      }
    }
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int x = threadIdx.x + e * kGatherThreads;
      const int i = i0 + x / CPR;
      if (i < k) {
        const long long dst = (u * k + i) * CPR + x % CPR;
        out_k[dst] = kv[e];
        out_v[dst] = vv[e];
      }
    }
  }
  if (bad && status) atomicOr(status, CMC_DEVFLAG_BAD_INDEX);
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

struct WsLayout {
  size_t tickets_off, partials_off, total;
};

static int tier1_tiles(const cmc_dims& m) { return (m.k + kTileKeys - 1) / kTileKeys; }
static int tiles_per_unit(const cmc_dims& m) { return tier1_tiles(m) + (m.W + kTileKeys - 1) / kTileKeys; }

// [0, 256): status word; then one 8-byte pos-read count per sequence (padded
// to 256 bytes); then one partial record per (unit, tile) slot (16-byte
// aligned: rec_floats is a multiple of 4).
static WsLayout ws_layout(const cmc_dims& m) {
  WsLayout w;
  const long long units = static_cast<long long>(m.B) * m.L * m.Hkv;
  const int G = m.Hq / m.Hkv;
  w.tickets_off = kWsHeader;
  w.partials_off = w.tickets_off + ((static_cast<size_t>(m.B) * 8 + 255) / 256) * 256;
  w.total = w.partials_off + static_cast<size_t>(units) * tiles_per_unit(m) * rec_floats(G, m.d) * sizeof(float);
  return w;
}

// cuTensorMapEncodeTiled, reached through the runtime's driver entry point.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
  });
  return fn;
}

// A [rows, d] bf16 tensor viewed by boxes of 64 columns x box_rows rows,
// 128-byte swizzle, zero fill outside the tensor.
static bool encode_rows(CUtensorMap* map, const void* base, long long rows, int d, int box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t es[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Pipeline depth: stages of 64 keys per CTA.  Three stages keep a CTA at
// ~110 KB of shared memory at d = 128, G <= 4, so two CTAs share an SM.
constexpr int kStages = 3;
// Box tiles per CTA prefetched into L2 before the grid dependency wait.  With
// the streamed K/V loads marked evict-first, five tiles (160 KB per CTA, some
// in free slots while the previous launch runs, most in its tail) measured
// best at the Llama-3-8B shape (14.20 us against 14.34 for four, 14.30 for six,
// 14.7 for three or eight); without the evict-first policy one tile was best.
// A rolling prefetch a few tiles ahead of the TMA issue, on top, was slower at
// every distance (16.2-16.9 us).  That is for one stream of launches: with
// independent requests' launches on four streams, whose launches already run
// through each other's edges, no prefetch measured best (11.92 us against
// 12.11 for one tile, 12.32 for two, 12.89 for five), so the depth is a
// setting (cmc_set_l2_prefetch_tiles) with this default.
constexpr int kL2PrefetchTiles = 5;
constexpr int kMaxL2PrefetchTiles = 64;
static std::atomic<int> g_l2_prefetch_tiles{kL2PrefetchTiles};

// Launch plan of one attention call on the current device.
struct AttnPlan {
  long long ctas, base, rem;  // grid size; flat split: granules per CTA (the first `rem` take one more)
  int gran;                   // flat split: tiles per granule
  int cm;                     // > 0: clusters of cm CTAs per unit (DSMEM merge, no combine)
  bool split;                 // flat split cuts some unit: the combine kernel runs
};

// Largest cluster of CTAs that share one unit (the portable cluster size).
constexpr int kMaxClusterCtas = 8;

template <int D, int G, bool FUSED, bool ROPE>
static int plan_attn(long long total_tiles, int tpu, AttnPlan* pl) {
  constexpr size_t smem = attn_smem_bytes<D, G, kStages, ROPE>();
  auto kern = two_tier_attn_kernel<D, G, FUSED, kStages, ROPE>;
  static std::atomic<int> configured[64];  // per device: attribute set and occupancy known (idempotent)
  int dev = 0;
  int st = record_cuda_error(cudaGetDevice(&dev));
  if (st != CMC_OK) return st;
  int per_sm = (dev >= 0 && dev < 64) ? configured[dev].load(std::memory_order_acquire) : 0;
  if (per_sm <= 0) {
    st = record_cuda_error(
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)));
    if (st != CMC_OK) return st;
    st = record_cuda_error(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads + 32, smem));
    if (st != CMC_OK) return st;
    if (per_sm < 1) per_sm = 1;
    if (dev >= 0 && dev < 64) configured[dev].store(per_sm, std::memory_order_release);
  }
  // Grid.  With no more units than resident CTAs: m = resident CTAs per unit,
  // at most one per tile and at most 8 (the portable cluster size).  m = 1:
  // one CTA per unit, nothing is split.  m >= 2: clusters of m CTAs per unit,
  // merged in distributed shared memory.  More units than resident CTAs: one
  // wave of CTAs, each taking a run of whole units or, when that would leave
  // too few CTAs for the last round, an equal share of the flattened tiles
  // (stream-K; the combine kernel merges the units cut between CTAs).  (A flat split
  // for few, long units -- m up to 38 at one sequence of one layer -- left
  // about one tile per CTA and a combine over 38 records: 33.4 us against
  // 9.4 us for clusters of 8 at k = 1024, W = 2048.)
  const long long slots = static_cast<long long>(per_sm) * sm_count();
  const long long units = total_tiles / tpu;
  pl->cm = 0;
  long long ctas;
  if (units <= slots) {
    long long m = slots / units;
    if (m > tpu) m = tpu;
    if (m > kMaxClusterCtas) m = kMaxClusterCtas;
    if (m >= 2) pl->cm = static_cast<int>(m);
    ctas = units * m;
  } else {
    ctas = slots;
  }
  if (ctas > total_tiles) ctas = total_tiles;
  if (ctas < 1) ctas = 1;
  pl->ctas = ctas;
  pl->gran = 1;
  pl->base = total_tiles / ctas;
  pl->rem = total_tiles % ctas;
  // More units than resident CTAs: whole units per CTA (contiguous runs, no
  // combine launch) when they divide evenly or when at least half of the CTAs
  // take one unit more -- enough CTAs then stream the last round to keep HBM
  // busy; with fewer, those few CTAs would stream their extra unit alone and
  // the balanced stream-K split with its combine is faster.  Measured at
  // 128 + 512-key units: 312 units 21.1 us stream-K / 23.7 us whole units,
  // 384 units 24.5 / 25.5, 448 units 26.0 / 26.2, 512 units 30.1 / 27.1.
  const long long ru = units % ctas;
  if (units > slots && (ru == 0 || 2 * ru >= ctas)) {
    pl->gran = tpu;
    pl->base = units / ctas;
    pl->rem = ru;
  }
  // Flat split: is any unit cut between CTAs (a CTA boundary inside a unit)?
  pl->split = false;
  for (long long c = 1; pl->cm == 0 && pl->gran == 1 && c < ctas && !pl->split; ++c) {
    const long long t = c * pl->base + (c < pl->rem ? c : pl->rem);
    pl->split = (t % tpu) != 0;
  }
  return CMC_OK;
}

// Launches the attention kernel with programmatic stream serialization and,
// for a cluster plan, the cluster dimension.
template <int D, int G, bool FUSED, bool ROPE>
static int launch_attn_kernel(const AttnMaps& maps, const AttnParams& p, const AttnPlan& pl,
                              cudaStream_t s) {
  constexpr size_t smem = attn_smem_bytes<D, G, kStages, ROPE>();
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  int na = 1;
  if (pl.cm > 0) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = static_cast<unsigned>(pl.cm);
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    na = 2;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(pl.ctas));
  cfg.blockDim = dim3(kThreads + 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return record_cuda_error(cudaLaunchKernelEx(&cfg, two_tier_attn_kernel<D, G, FUSED, kStages, ROPE>, maps, p));
}

template <int D, int G, bool FUSED, bool ROPE>
static int launch_attn(const AttnMaps& maps, const AttnParams& p0, long long total_tiles,
                       cudaStream_t s) {
  AttnPlan pl;
  int st = plan_attn<D, G, FUSED, ROPE>(total_tiles, p0.tpu, &pl);
  if (st != CMC_OK) return st;
  AttnParams p = p0;
  p.base = pl.base;
  p.rem = pl.rem;
  p.cm = pl.cm;
  p.gran = pl.gran;
  st = launch_attn_kernel<D, G, FUSED, ROPE>(maps, p, pl, s);
  if (st != CMC_OK || !pl.split) return st;
  return launch_pdl(two_tier_combine_kernel<D, G>, dim3(static_cast<unsigned>(total_tiles / p.tpu)),
                    dim3(kThreads), 0, s, p);
}

template <bool FUSED, bool ROPE>
static int dispatch_plan(int d, int G, long long tiles, int tpu, AttnPlan* pl) {
  if (d == 128) {
    switch (G) {
      case 1: return plan_attn<128, 1, FUSED, ROPE>(tiles, tpu, pl);
      case 2: return plan_attn<128, 2, FUSED, ROPE>(tiles, tpu, pl);
      case 4: return plan_attn<128, 4, FUSED, ROPE>(tiles, tpu, pl);
      default: return plan_attn<128, 8, FUSED, ROPE>(tiles, tpu, pl);
    }
  }
  switch (G) {
    case 1: return plan_attn<64, 1, FUSED, ROPE>(tiles, tpu, pl);
    case 2: return plan_attn<64, 2, FUSED, ROPE>(tiles, tpu, pl);
    case 4: return plan_attn<64, 4, FUSED, ROPE>(tiles, tpu, pl);
    default: return plan_attn<64, 8, FUSED, ROPE>(tiles, tpu, pl);
  }
}

template <bool FUSED, bool ROPE>
static int dispatch_attn(const AttnMaps& maps, const AttnParams& p, int d, int G, long long tiles,
                         cudaStream_t s) {
  if (d == 128) {
    switch (G) {
      case 1: return launch_attn<128, 1, FUSED, ROPE>(maps, p, tiles, s);
      case 2: return launch_attn<128, 2, FUSED, ROPE>(maps, p, tiles, s);
      case 4: return launch_attn<128, 4, FUSED, ROPE>(maps, p, tiles, s);
      default: return launch_attn<128, 8, FUSED, ROPE>(maps, p, tiles, s);
    }
  }
  switch (G) {
    case 1: return launch_attn<64, 1, FUSED, ROPE>(maps, p, tiles, s);
    case 2: return launch_attn<64, 2, FUSED, ROPE>(maps, p, tiles, s);
    case 4: return launch_attn<64, 4, FUSED, ROPE>(maps, p, tiles, s);
    default: return launch_attn<64, 8, FUSED, ROPE>(maps, p, tiles, s);
  }
}

// The failure-path test hook (cmc_test_stall_attention_waits): bytes every
// stage of the attention launches that follow expects beyond its loads; 0 in
// normal use.
static std::atomic<uint32_t> g_stall_tx{0};

// theta^(-2i/d) / (2 pi) -- the pair's turns per position, below 1/6 -- as a
// 64-bit binary fraction, rounded to nearest, computed in long double.
static unsigned long long rope_turns_fixed(double theta, int i, int d) {
  const long double two_pi = 6.283185307179586476925286766559L;
  const long double t = powl(static_cast<long double>(theta), -2.0L * i / d) / two_pi;
  return static_cast<unsigned long long>(t * 18446744073709551616.0L + 0.5L);  // t * 2^64
}

// The slot of g_rope_tables holding the table of (theta, d) on the current
// device, writing it on first use; -1 (use the kernel parameters) when the
// slots are full, the stream is being captured into a graph, or the copy
// fails.  The copy is synchronous, so every later launch sees the table.
struct RopeSlots {
  std::mutex mu;
  int n = 0;
  double theta[kRopeSlots];
  int d[kRopeSlots];
};
static RopeSlots g_rope_slots[64];

static int rope_slot(double theta, int d, const unsigned long long* table, cudaStream_t s) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return -1;
  }
  RopeSlots& c = g_rope_slots[dev];
  std::lock_guard<std::mutex> lock(c.mu);
  for (int i = 0; i < c.n; ++i)
    if (c.theta[i] == theta && c.d[i] == d) return i;
  if (c.n >= kRopeSlots) return -1;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) {
    cudaGetLastError();
    return -1;
  }
  if (cudaMemcpyToSymbol(g_rope_tables, table, 64 * sizeof(unsigned long long),
                         static_cast<size_t>(c.n) * 64 * sizeof(unsigned long long),
                         cudaMemcpyHostToDevice) != cudaSuccess) {
    cudaGetLastError();
    return -1;
  }
  c.theta[c.n] = theta;
  c.d[c.n] = d;
  return c.n++;
}

static int run_attention(const void* q, const void* tier1_k, const void* tier1_v,
                         const int32_t* idx, void* ring_k, void* ring_v, int64_t* pos,
                         const void* k_new, const void* v_new, const cmc_dims* dims, float scale,
                         void* out, void* workspace, size_t workspace_bytes, void* stream,
                         bool fused, bool rope = false, double rope_theta = 0.0,
                         long long rope_offset = 0) {
  int st = validate_dims(dims, true);
  if (st != CMC_OK) return st;
  const cmc_dims& m = *dims;
  if (!q || !tier1_k || !tier1_v || !ring_k || !ring_v || !pos || !out) return CMC_ERR_NULL;
  if (fused && (!k_new || !v_new)) return CMC_ERR_NULL;
  if (rope && !(rope_theta > 0.0 && rope_theta < 1e300)) return CMC_ERR_RANGE;
  if (rope && (rope_offset < 0 || rope_offset > (1LL << 32))) return CMC_ERR_RANGE;
  if (!aligned16(q) || !aligned16(tier1_k) || !aligned16(tier1_v) || !aligned16(ring_k) ||
      !aligned16(ring_v) || !aligned16(out))
    return CMC_ERR_ALIGN;
  if (fused && (!aligned16(k_new) || !aligned16(v_new))) return CMC_ERR_ALIGN;
  if ((reinterpret_cast<uintptr_t>(pos) & 7) || (idx && (reinterpret_cast<uintptr_t>(idx) & 3)))
    return CMC_ERR_ALIGN;
  const WsLayout w = ws_layout(m);
  if (!workspace || workspace_bytes < w.total) return CMC_ERR_WORKSPACE;
  if (!aligned16(workspace)) return CMC_ERR_ALIGN;

  const long long units = static_cast<long long>(m.B) * m.L * m.Hkv;
  const int tpu = tiles_per_unit(m);
  const long long tiles = units * tpu;
  // tile indices, unit ids and tensor-map row coordinates are 32-bit
  if (tiles >= (1LL << 31) || units * m.N >= (1LL << 31) || units * m.W >= (1LL << 31))
    return CMC_ERR_SHAPE;

  AttnMaps maps;
  memset(&maps, 0, sizeof(maps));
  if (!encode_rows(&maps.rk_box, ring_k, units * m.W, m.d, kTileKeys) ||
      !encode_rows(&maps.rv_box, ring_v, units * m.W, m.d, kTileKeys))
    return CMC_ERR_CUDA;
  if (!idx && m.k > 0 &&
      (!encode_rows(&maps.t1k_box, tier1_k, units * m.N, m.d, kTileKeys) ||
       !encode_rows(&maps.t1v_box, tier1_v, units * m.N, m.d, kTileKeys)))
    return CMC_ERR_CUDA;

  AttnParams p;
  p.q = static_cast<const uint16_t*>(q);
  p.t1k = static_cast<const uint16_t*>(tier1_k);
  p.t1v = static_cast<const uint16_t*>(tier1_v);
  p.idx = m.k > 0 ? idx : nullptr;
  p.ring_k = static_cast<uint16_t*>(ring_k);
  p.ring_v = static_cast<uint16_t*>(ring_v);
  p.pos = pos;
  p.k_new = static_cast<const uint16_t*>(k_new);
  p.v_new = static_cast<const uint16_t*>(v_new);
  p.out = static_cast<uint16_t*>(out);
  char* ws = static_cast<char*>(workspace);
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.tickets = reinterpret_cast<unsigned long long*>(ws + w.tickets_off);
  p.partials = reinterpret_cast<float*>(ws + w.partials_off);
  p.B = m.B; p.L = m.L; p.Hq = m.Hq; p.Hkv = m.Hkv; p.N = m.N; p.k = m.k; p.W = m.W;
  p.tpu = tpu;
  p.t1_tiles = tier1_tiles(m);
  p.rot = p.t1_tiles % tpu;  // the first ring tile
  p.base = 0;
  p.rem = 0;
  p.cm = 0;
  p.gran = 1;
  const float sc = scale > 0.f ? scale : 1.0f / sqrtf(static_cast<float>(m.d));
  p.scale_log2 = sc * 1.4426950408889634f;
  p.rope_offset = rope ? rope_offset : 0;
  p.l2_prefetch = g_l2_prefetch_tiles.load(std::memory_order_relaxed);
  p.stall_tx = g_stall_tx.load(std::memory_order_relaxed);
  for (int i = 0; i < 64; ++i)
    p.rope_turns[i] = (rope && i < m.d / 2) ? rope_turns_fixed(rope_theta, i, m.d) : 0ull;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  p.rope_slot = rope ? rope_slot(rope_theta, m.d, p.rope_turns, s) : -1;
  const int G = m.Hq / m.Hkv;
  if (rope) return dispatch_attn<true, true>(maps, p, m.d, G, tiles, s);
  return fused ? dispatch_attn<true, false>(maps, p, m.d, G, tiles, s)
               : dispatch_attn<false, false>(maps, p, m.d, G, tiles, s);
}

}  // namespace cmc

extern "C" {

size_t cmc_decode_attn_workspace_size(const cmc_dims* dims) {
  if (cmc::validate_dims(dims, true) != CMC_OK) return 0;
  return cmc::ws_layout(*dims).total;
}

int cmc_two_tier_decode_attn(const void* q, const void* tier1_k, const void* tier1_v,
                             const int32_t* idx, const void* ring_k, const void* ring_v,
                             const int64_t* pos, const cmc_dims* dims, float scale, void* out,
                             void* workspace, size_t workspace_bytes, void* stream) {
  return cmc::run_attention(q, tier1_k, tier1_v, idx, const_cast<void*>(ring_k),
                            const_cast<void*>(ring_v), const_cast<int64_t*>(pos), nullptr, nullptr,
                            dims, scale, out, workspace, workspace_bytes, stream, false);
}

int cmc_decode_step(const void* q, const void* tier1_k, const void* tier1_v, const int32_t* idx,
                    void* ring_k, void* ring_v, int64_t* pos, const void* k_new, const void* v_new,
                    const cmc_dims* dims, float scale, void* out, void* workspace,
                    size_t workspace_bytes, void* stream) {
  return cmc::run_attention(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, k_new, v_new, dims,
                            scale, out, workspace, workspace_bytes, stream, true);
}

int cmc_decode_step_rope(const void* q, const void* tier1_k, const void* tier1_v,
                         const int32_t* idx, void* ring_k, void* ring_v, int64_t* pos,
                         const void* k_new, const void* v_new, const cmc_dims* dims, float scale,
                         double rope_theta, int64_t rope_offset, void* out, void* workspace,
                         size_t workspace_bytes, void* stream) {
  return cmc::run_attention(q, tier1_k, tier1_v, idx, ring_k, ring_v, pos, k_new, v_new, dims,
                            scale, out, workspace, workspace_bytes, stream, true, true, rope_theta,
                            rope_offset);
}

int cmc_tier1_gather(const void* bank_k, const void* bank_v, const int32_t* idx,
                     const cmc_dims* dims, void* tier1_k, void* tier1_v, uint32_t* status,
                     void* stream) {
  using namespace cmc;
  if (!dims) return CMC_ERR_NULL;
  cmc_dims m = *dims;
  m.Hq = m.Hkv;  // query heads play no part here
  int st = validate_dims(&m, true);
  if (st != CMC_OK) return st;
  if (m.k == 0) return CMC_OK;
  if (!bank_k || !bank_v || !idx || !tier1_k || !tier1_v) return CMC_ERR_NULL;
  if (!aligned16(bank_k) || !aligned16(bank_v) || !aligned16(tier1_k) || !aligned16(tier1_v) ||
      (reinterpret_cast<uintptr_t>(idx) & 3) || (reinterpret_cast<uintptr_t>(status) & 3))
    return CMC_ERR_ALIGN;
  const long long units = static_cast<long long>(m.B) * m.L * m.Hkv;
  const int row_blocks = (m.k + kGatherRows - 1) / kGatherRows;
  const long long blocks = units * row_blocks;
  const long long grid = blocks < (1LL << 30) ? blocks : (1LL << 30);
  auto kern = m.d == 128 ? tier1_gather_kernel<16> : tier1_gather_kernel<8>;
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(kGatherThreads), 0,
                    static_cast<cudaStream_t>(stream), static_cast<const uint4*>(bank_k),
                    static_cast<const uint4*>(bank_v), idx, static_cast<uint4*>(tier1_k),
                    static_cast<uint4*>(tier1_v), status, blocks, row_blocks, m.L * m.Hkv, m.N,
                    m.k);
}

int cmc_decode_attn_plan(const cmc_dims* dims, int fused, int* ctas, int* launches) {
  using namespace cmc;
  int st = validate_dims(dims, true);
  if (st != CMC_OK) return st;
  if (!ctas || !launches) return CMC_ERR_NULL;
  const cmc_dims& m = *dims;
  const long long units = static_cast<long long>(m.B) * m.L * m.Hkv;
  const int tpu = tiles_per_unit(m);
  const long long tiles = units * tpu;
  if (tiles >= (1LL << 31)) return CMC_ERR_SHAPE;
  AttnPlan pl;
  if (fused < 0 || fused > 2) return CMC_ERR_RANGE;
  st = fused == 2 ? dispatch_plan<true, true>(m.d, m.Hq / m.Hkv, tiles, tpu, &pl)
       : fused    ? dispatch_plan<true, false>(m.d, m.Hq / m.Hkv, tiles, tpu, &pl)
                  : dispatch_plan<false, false>(m.d, m.Hq / m.Hkv, tiles, tpu, &pl);
  if (st != CMC_OK) return st;
  *ctas = static_cast<int>(pl.ctas);
  *launches = pl.split ? 2 : 1;
  return CMC_OK;
}

int cmc_window_append(void* ring_k, void* ring_v, int64_t* pos, const void* k_new,
                      const void* v_new, const cmc_dims* dims, void* stream) {
  using namespace cmc;
  int st = validate_dims(dims, false);
  if (st != CMC_OK) return st;
  if (!ring_k || !ring_v || !pos || !k_new || !v_new) return CMC_ERR_NULL;
  if (!aligned16(ring_k) || !aligned16(ring_v) || !aligned16(k_new) || !aligned16(v_new) ||
      (reinterpret_cast<uintptr_t>(pos) & 7))
    return CMC_ERR_ALIGN;
  const cmc_dims& m = *dims;
  window_append_kernel<<<m.B, 256, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<uint16_t*>(ring_k), static_cast<uint16_t*>(ring_v), pos,
      static_cast<const uint16_t*>(k_new), static_cast<const uint16_t*>(v_new), m.L * m.Hkv, m.W,
      m.d);
  return check_launch();
}

int cmc_set_l2_prefetch_tiles(int tiles) {
  if (tiles < 0 || tiles > cmc::kMaxL2PrefetchTiles) return CMC_ERR_RANGE;
  cmc::g_l2_prefetch_tiles.store(tiles, std::memory_order_relaxed);
  return CMC_OK;
}

int cmc_test_stall_attention_waits(int on) {
  cmc::g_stall_tx.store(on ? 16u : 0u, std::memory_order_relaxed);
  return CMC_OK;
}

}  // extern "C"
