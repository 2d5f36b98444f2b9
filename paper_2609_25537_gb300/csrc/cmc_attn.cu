// Tier-2 ring append and decode attention over the two-tier cache
// (Section 2.5, "Tier-2: local context window" and "KV cache assembly"; cost
// model in the appendix "Attention MACs Analysis").
//
// Work decomposition: a unit is one (sequence b, layer l, KV head g).  Its
// keys are the k Tier-1 rows gathered by idx followed by the occupied ring
// slots; the key range is cut into `splits` chunks and one CTA handles one
// (chunk, unit) pair (split-K / flash-decoding).  Inside a CTA each group of
// d/8 lanes owns one key at a time and each lane one 16-byte slice of it
// (8 bf16): keys of a warp step are adjacent rows, so a ring span is read as
// contiguous 16-byte vectors and a gathered Tier-1 row as whole 256-byte
// (d = 128) rows.  The G = Hq/Hkv query heads of the unit share every K/V
// load.  Logits are reduced across the d/8 lanes with xor shuffles, the
// softmax is an online (running max / sum) softmax in the log2 domain, and the
// per-group (m, l, o) states are merged in shared memory.  With splits > 1 each
// CTA writes its (m, l, o) partial to the workspace and the last CTA of the
// unit to arrive (an atomic ticket, no waiting) merges the partials with a
// log-sum-exp rescale and writes the bf16 output.
//
// The fused decode step additionally appends the new token: every reader of
// the ring slot being overwritten takes the new token's K/V from k_new/v_new
// instead, the CTA whose chunk holds that slot stores it into the ring, and
// the last CTA of the sequence to arrive (a second ticket) advances pos[b].
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "cmc_internal.cuh"

namespace cmc {

constexpr int kAttnWarps = 4;
constexpr int kAttnThreads = 32 * kAttnWarps;
constexpr int kAttnUnroll = 4;
constexpr int kMinChunk = 32;   // smallest chunk the split planner uses
constexpr int kMaxChunk = 512;  // largest chunk (bounds the shared idx buffer)
constexpr size_t kWsHeader = 256;

struct AttnParams {
  const uint16_t* q;      // [B, L, Hq, d]
  const uint16_t* t1k;    // [B, L, Hkv, N, d]
  const uint16_t* t1v;    // [B, L, Hkv, N, d]
  const int32_t* idx;     // [B, k]
  uint16_t* ring_k;       // [B, L, Hkv, W, d]
  uint16_t* ring_v;       // [B, L, Hkv, W, d]
  int64_t* pos;           // [B]
  const uint16_t* k_new;  // [B, L, Hkv, d]   (fused step only)
  const uint16_t* v_new;  // [B, L, Hkv, d]
  uint16_t* out;          // [B, L, Hq, d]
  uint32_t* status;       // workspace status word
  uint32_t* unit_ticket;  // [B * L * Hkv]
  uint32_t* seq_ticket;   // [B]
  float* partials;        // [units, splits, G * (d + 2)]
  int B, L, Hq, Hkv, N, k, W;
  int splits, chunk;
  float scale_log2;       // softmax scale * log2(e)
};

// Split plan: number of chunks per unit and keys per chunk.
struct SplitPlan {
  int splits, chunk;
};

static int max_splits(int n_max) { return (n_max + kMinChunk - 1) / kMinChunk; }

static SplitPlan plan_splits(long long units, int n_max) {
  const long long target = 4LL * sm_count();
  long long s = (target + units - 1) / units;
  if (s < 1) s = 1;
  if (s > max_splits(n_max)) s = max_splits(n_max);
  int chunk = static_cast<int>((n_max + s - 1) / s);
  chunk = (chunk + kMinChunk - 1) / kMinChunk * kMinChunk;
  if (chunk > kMaxChunk) chunk = kMaxChunk;
  if (chunk < kMinChunk) chunk = kMinChunk;
  SplitPlan p;
  p.chunk = chunk;
  p.splits = (n_max + chunk - 1) / chunk;
  if (p.splits < 1) p.splits = 1;
  return p;
}

template <int D, int G, bool FUSED>
__global__ void __launch_bounds__(kAttnThreads)
two_tier_attn_kernel(const AttnParams p) {
  constexpr int LPK = D / 8;                 // lanes per key
  constexpr int KPW = 32 / LPK;              // keys per warp step
  constexpr int GROUPS = kAttnWarps * KPW;   // key groups per CTA
  constexpr int STEP = GROUPS * kAttnUnroll; // keys per CTA iteration

  __shared__ int s_idx[kMaxChunk];
  __shared__ float s_m[GROUPS][G];
  __shared__ float s_l[GROUPS][G];
  __shared__ float s_o[GROUPS][G][D];
  __shared__ int s_last;

  const int split = blockIdx.x;
  const int unit = blockIdx.y;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int sub = lane / LPK;
  const int kl = lane % LPK;
  const int grp = warp * KPW + sub;

  const int LH = p.L * p.Hkv;
  const int b = unit / LH;
  const int lg = unit - b * LH;
  const int l = lg / p.Hkv;
  const int g = lg - l * p.Hkv;

  const long long pos_b = p.pos[b];
  const bool bad_pos = pos_b < 0;
  int count = 0, new_slot = -1;
  if (!bad_pos) {
    if (FUSED) {
      count = static_cast<int>(pos_b + 1 < p.W ? pos_b + 1 : p.W);
      new_slot = static_cast<int>(pos_b % p.W);
    } else {
      count = static_cast<int>(pos_b < p.W ? pos_b : p.W);
    }
  }
  const int k_eff = bad_pos ? 0 : p.k;
  const int n_keys = k_eff + count;
  const int kbeg = split * p.chunk;
  const int kend = min(kbeg + p.chunk, n_keys);
  if (bad_pos && split == 0 && tid == 0) atomicOr(p.status, CMC_DEVFLAG_BAD_POS);

  // Tier-1 rows of this chunk
  const int t1_end = min(kend, k_eff);
  for (int i = kbeg + tid; i < t1_end; i += kAttnThreads) {
    int r = p.idx[static_cast<long long>(b) * p.k + i];
    if (r < 0 || r >= p.N) {
      atomicOr(p.status, CMC_DEVFLAG_BAD_INDEX);
      r = -1;
    }
    s_idx[i - kbeg] = r;
  }

  const long long unit_l = unit;
  // Fused step: store the new token into its slot if this chunk owns the slot.
  if (FUSED && !bad_pos) {
    const int key_new = k_eff + new_slot;
    if (key_new >= kbeg && key_new < kend) {
      const uint4* sk = reinterpret_cast<const uint4*>(p.k_new + unit_l * D);
      const uint4* sv = reinterpret_cast<const uint4*>(p.v_new + unit_l * D);
      uint4* dk = reinterpret_cast<uint4*>(p.ring_k + (unit_l * p.W + new_slot) * D);
      uint4* dv = reinterpret_cast<uint4*>(p.ring_v + (unit_l * p.W + new_slot) * D);
      for (int v = tid; v < D / 8; v += kAttnThreads) {
        dk[v] = sk[v];
        dv[v] = sv[v];
      }
    }
  }

  // This lane's slice of the G query heads, pre-multiplied by scale*log2(e).
  float qf[G][8];
  {
    const long long qbase = (static_cast<long long>(b) * p.L + l) * p.Hq + static_cast<long long>(g) * G;
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const uint4 v = *reinterpret_cast<const uint4*>(p.q + (qbase + h) * D + kl * 8);
      float f[8];
      unpack8(v, f);
#pragma unroll
      for (int e = 0; e < 8; ++e) qf[h][e] = f[e] * p.scale_log2;
    }
  }
  __syncthreads();

  float m[G], lsum[G], o[G][8];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    m[h] = -INFINITY;
    lsum[h] = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) o[h][e] = 0.f;
  }

  const long long bank_row0 = unit_l * p.N;
  const long long ring_row0 = unit_l * p.W;
  for (int base = kbeg; base < kend; base += STEP) {
    uint4 kr[kAttnUnroll], vr[kAttnUnroll];
    bool valid[kAttnUnroll];
#pragma unroll
    for (int u = 0; u < kAttnUnroll; ++u) {
      const int i = base + u * GROUPS + grp;
      const uint16_t* kp = nullptr;
      const uint16_t* vp = nullptr;
      if (i < kend) {
        if (i < k_eff) {
          const int r = s_idx[i - kbeg];
          if (r >= 0) {
            kp = p.t1k + (bank_row0 + r) * D;
            vp = p.t1v + (bank_row0 + r) * D;
          }
        } else {
          const int slot = i - k_eff;
          if (FUSED && slot == new_slot) {
            kp = p.k_new + unit_l * D;
            vp = p.v_new + unit_l * D;
          } else {
            kp = p.ring_k + (ring_row0 + slot) * D;
            vp = p.ring_v + (ring_row0 + slot) * D;
          }
        }
      }
      valid[u] = kp != nullptr;
      if (valid[u]) {
        kr[u] = ld_stream_u4(kp + kl * 8);
        vr[u] = ld_stream_u4(vp + kl * 8);
      } else {
        kr[u] = make_uint4(0u, 0u, 0u, 0u);
        vr[u] = make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int u = 0; u < kAttnUnroll; ++u) {
      float kf[8];
      unpack8(kr[u], kf);
      float z[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        float acc = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc = fmaf(qf[h][e], kf[e], acc);
        z[h] = acc;
      }
#pragma unroll
      for (int off = LPK / 2; off >= 1; off >>= 1) {
#pragma unroll
        for (int h = 0; h < G; ++h) z[h] += __shfl_xor_sync(0xffffffffu, z[h], off);
      }
      if (valid[u]) {
        float vf[8];
        unpack8(vr[u], vf);
#pragma unroll
        for (int h = 0; h < G; ++h) {
          if (z[h] > m[h]) {
            const float a = exp2f(m[h] - z[h]);
            lsum[h] *= a;
#pragma unroll
            for (int e = 0; e < 8; ++e) o[h][e] *= a;
            m[h] = z[h];
          }
          const float pr = exp2f(z[h] - m[h]);
          lsum[h] += pr;
#pragma unroll
          for (int e = 0; e < 8; ++e) o[h][e] = fmaf(pr, vf[e], o[h][e]);
        }
      }
    }
  }

  // Merge the key groups of this CTA.
  if (kl == 0) {
#pragma unroll
    for (int h = 0; h < G; ++h) {
      s_m[grp][h] = m[h];
      s_l[grp][h] = lsum[h];
    }
  }
#pragma unroll
  for (int h = 0; h < G; ++h) {
#pragma unroll
    for (int e = 0; e < 8; ++e) s_o[grp][h][kl * 8 + e] = o[h][e];
  }
  __syncthreads();

  constexpr int PAIRS = G * D / 2;  // output element pairs of the unit
  const long long out_base = ((static_cast<long long>(b) * p.L + l) * p.Hq + static_cast<long long>(g) * G) * D;
  const int PW = G * (D + 2);       // floats per partial
  float* my_part = p.partials + (unit_l * p.splits + split) * PW;

  for (int t = tid; t < PAIRS; t += kAttnThreads) {
    const int h = (2 * t) / D;
    const int c = (2 * t) % D;
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < GROUPS; ++q) M = fmaxf(M, s_m[q][h]);
    float Ls = 0.f, O0 = 0.f, O1 = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int q = 0; q < GROUPS; ++q) {
        const float f = exp2f(s_m[q][h] - M);
        Ls = fmaf(f, s_l[q][h], Ls);
        O0 = fmaf(f, s_o[q][h][c], O0);
        O1 = fmaf(f, s_o[q][h][c + 1], O1);
      }
    }
    if (p.splits == 1) {
      const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
      reinterpret_cast<uint32_t*>(p.out + out_base + h * D + c)[0] = pack_bf16x2(O0 * inv, O1 * inv);
    } else {
      if (c == 0) {
        my_part[h] = M;
        my_part[G + h] = Ls;
      }
      my_part[2 * G + h * D + c] = O0;
      my_part[2 * G + h * D + c + 1] = O1;
    }
  }

  bool unit_done = true;  // this CTA finishes the unit
  if (p.splits > 1) {
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const uint32_t ticket = atomicAdd(&p.unit_ticket[unit], 1u);
      s_last = (ticket == static_cast<uint32_t>(p.splits - 1)) ? 1 : 0;
    }
    __syncthreads();
    unit_done = s_last != 0;
    if (unit_done) {
      __threadfence();
      const float* parts = p.partials + unit_l * p.splits * PW;
      for (int t = tid; t < PAIRS; t += kAttnThreads) {
        const int h = (2 * t) / D;
        const int c = (2 * t) % D;
        float M = -INFINITY;
        for (int s = 0; s < p.splits; ++s) M = fmaxf(M, __ldcg(parts + s * PW + h));
        float Ls = 0.f, O0 = 0.f, O1 = 0.f;
        if (M != -INFINITY) {
          for (int s = 0; s < p.splits; ++s) {
            const float* ps = parts + s * PW;
            const float f = exp2f(__ldcg(ps + h) - M);
            Ls = fmaf(f, __ldcg(ps + G + h), Ls);
            O0 = fmaf(f, __ldcg(ps + 2 * G + h * D + c), O0);
            O1 = fmaf(f, __ldcg(ps + 2 * G + h * D + c + 1), O1);
          }
        }
        const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
        reinterpret_cast<uint32_t*>(p.out + out_base + h * D + c)[0] = pack_bf16x2(O0 * inv, O1 * inv);
      }
      if (tid == 0) p.unit_ticket[unit] = 0u;
    }
  }

  if (FUSED && unit_done && tid == 0) {
    // Every CTA of this unit has read pos[b]; count the unit towards its sequence.
    __threadfence();
    const uint32_t t = atomicAdd(&p.seq_ticket[b], 1u);
    if (t == static_cast<uint32_t>(LH - 1)) {
      p.seq_ticket[b] = 0u;
      if (!bad_pos) p.pos[b] = pos_b + 1;
    }
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

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

struct WsLayout {
  size_t tickets_off, partials_off, total;
  int smax;
};

static WsLayout ws_layout(const cmc_dims& m) {
  WsLayout w;
  const long long units = static_cast<long long>(m.B) * m.L * m.Hkv;
  const int n_max = m.k + m.W;
  w.smax = max_splits(n_max);
  const int G = m.Hq / m.Hkv;
  w.tickets_off = kWsHeader;
  w.partials_off = w.tickets_off + align_up(sizeof(uint32_t) * static_cast<size_t>(units + m.B), 256);
  w.total = w.partials_off + static_cast<size_t>(units) * w.smax * G * (m.d + 2) * sizeof(float);
  return w;
}

template <int D, int G, bool FUSED>
static void launch_attn(const AttnParams& p, dim3 grid, cudaStream_t s) {
  two_tier_attn_kernel<D, G, FUSED><<<grid, kAttnThreads, 0, s>>>(p);
}

template <bool FUSED>
static void dispatch_attn(const AttnParams& p, int d, int G, dim3 grid, cudaStream_t s) {
  if (d == 128) {
    switch (G) {
      case 1: launch_attn<128, 1, FUSED>(p, grid, s); break;
      case 2: launch_attn<128, 2, FUSED>(p, grid, s); break;
      case 4: launch_attn<128, 4, FUSED>(p, grid, s); break;
      default: launch_attn<128, 8, FUSED>(p, grid, s); break;
    }
  } else {
    switch (G) {
      case 1: launch_attn<64, 1, FUSED>(p, grid, s); break;
      case 2: launch_attn<64, 2, FUSED>(p, grid, s); break;
      case 4: launch_attn<64, 4, FUSED>(p, grid, s); break;
      default: launch_attn<64, 8, FUSED>(p, grid, s); break;
    }
  }
}

static int run_attention(const void* q, const void* tier1_k, const void* tier1_v,
                         const int32_t* idx, void* ring_k, void* ring_v, int64_t* pos,
                         const void* k_new, const void* v_new, const cmc_dims* dims, float scale,
                         void* out, void* workspace, size_t workspace_bytes, void* stream,
                         bool fused) {
  int st = validate_dims(dims, true);
  if (st != CMC_OK) return st;
  const cmc_dims& m = *dims;
  if (!q || !tier1_k || !tier1_v || !ring_k || !ring_v || !pos || !out) return CMC_ERR_NULL;
  if (m.k > 0 && !idx) return CMC_ERR_NULL;
  if (fused && (!k_new || !v_new)) return CMC_ERR_NULL;
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
  if (units > 65535) return CMC_ERR_SHAPE;  // grid.y limit
  const SplitPlan plan = plan_splits(units, m.k + m.W);

  AttnParams p;
  p.q = static_cast<const uint16_t*>(q);
  p.t1k = static_cast<const uint16_t*>(tier1_k);
  p.t1v = static_cast<const uint16_t*>(tier1_v);
  p.idx = idx;
  p.ring_k = static_cast<uint16_t*>(ring_k);
  p.ring_v = static_cast<uint16_t*>(ring_v);
  p.pos = pos;
  p.k_new = static_cast<const uint16_t*>(k_new);
  p.v_new = static_cast<const uint16_t*>(v_new);
  p.out = static_cast<uint16_t*>(out);
  char* ws = static_cast<char*>(workspace);
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.unit_ticket = reinterpret_cast<uint32_t*>(ws + w.tickets_off);
  p.seq_ticket = p.unit_ticket + units;
  p.partials = reinterpret_cast<float*>(ws + w.partials_off);
  p.B = m.B; p.L = m.L; p.Hq = m.Hq; p.Hkv = m.Hkv; p.N = m.N; p.k = m.k; p.W = m.W;
  p.splits = plan.splits;
  p.chunk = plan.chunk;
  const float sc = scale > 0.f ? scale : 1.0f / sqrtf(static_cast<float>(m.d));
  p.scale_log2 = sc * 1.4426950408889634f;

  const dim3 grid(static_cast<unsigned>(plan.splits), static_cast<unsigned>(units));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int G = m.Hq / m.Hkv;
  if (fused) dispatch_attn<true>(p, m.d, G, grid, s);
  else dispatch_attn<false>(p, m.d, G, grid, s);
  return check_launch();
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

}  // extern "C"
