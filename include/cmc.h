/*
 * cmc.h -- C ABI of the CMC two-tier KV-cache decode path (GB300, sm_103a).
 *
 * The method (Section 2.5 of "Compressing Long Context into Answer-Aligned
 * Memory Embeddings for LLM Inference", "Inference with Two-Tier KV Cache
 * Policy") keeps, for every sequence, a KV cache of two tiers:
 *
 *   Tier-1  the K Context Memory Embeddings (CMEs) whose cosine similarity to
 *           the mean-pooled question vector is highest, re-ordered by
 *           document position (the score_j equation and the top-K text that
 *           follows it);
 *   Tier-2  a local window of W tokens at full resolution; generated tokens
 *           enter it, so the cache never exceeds K + W + |q| tokens ("KV
 *           cache assembly").
 *
 * Each decode step attends over [Tier-1 | Tier-2]; the appendix ("Attention
 * MACs Analysis") costs it as MACs_t = 2 n_h d_h n_l L_t.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every tensor argument is a DEVICE pointer to memory the caller owns.  The
 *    library allocates no memory and keeps no state between calls apart from
 *    the thread-local last CUDA error, a per-device SM-count cache, the
 *    per-device rotary frequency tables of cmc_decode_step_rope (written once
 *    per (theta, d)), the static score array of cmc_score_select_static and
 *    two process-wide settings of the attention launches
 *    (cmc_set_l2_prefetch_tiles, cmc_test_stall_attention_waits).
 *  - All work is enqueued on `stream` (a cudaStream_t passed as void*; NULL is
 *    the legacy default stream) and is asynchronous: a return of CMC_OK means
 *    the launch was accepted, not that it has finished.
 *  - Tensors are dense, row-major, with the shapes given below (last index
 *    fastest).  bf16 tensors must be 16-byte aligned; so must fp32 tensors.
 *  - Arguments are checked on the host before any launch; a failed check
 *    launches nothing and returns the status below.  Kernels never trap.
 *  - Calls that share a workspace must be ordered on one stream.
 */
#ifndef CMC_H_
#define CMC_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define CMC_API __attribute__((visibility("default")))
#else
#define CMC_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum cmc_status {
  CMC_OK = 0,
  CMC_ERR_NULL = 1,      /* a required pointer is NULL                              */
  CMC_ERR_SHAPE = 2,     /* a size outside the supported range (see each call)      */
  CMC_ERR_RANGE = 3,     /* an index-like argument out of range (k > N, W < 1, ...) */
  CMC_ERR_ALIGN = 4,     /* a tensor pointer is not 16-byte aligned                 */
  CMC_ERR_WORKSPACE = 5, /* workspace NULL or smaller than the size query returns   */
  CMC_ERR_CUDA = 6       /* a CUDA call failed; cmc_last_cuda_error() has the code  */
} cmc_status;

/* Device-side status bits, accumulated in a workspace's status word (see
 * cmc_read_status).  Kernels skip the offending element and carry on. */
#define CMC_DEVFLAG_BAD_INDEX 1u /* an idx entry outside [0, N): that row was skipped   */
#define CMC_DEVFLAG_BAD_POS 2u   /* a negative pos: that sequence was skipped            */
#define CMC_DEVFLAG_TIMEOUT 4u   /* a pipeline wait gave up after its time limit (1 s of
                                    %globaltimer): the call's outputs and ring update are
                                    invalid (never expected in operation)                 */

/* Shapes of one decode problem. */
typedef struct cmc_dims {
  int32_t B;   /* sequences, >= 1                                                  */
  int32_t L;   /* decoder layers handled by one call, >= 1                         */
  int32_t Hq;  /* query heads, >= 1                                                */
  int32_t Hkv; /* KV heads; Hq % Hkv == 0 and Hq / Hkv in {1, 2, 4, 8}             */
  int32_t d;   /* head dimension: 64 or 128                                        */
  int32_t N;   /* rows of the Tier-1 K/V bank per (sequence, layer, KV head), >= 1 */
  int32_t k;   /* selected Tier-1 rows per sequence, 0 <= k <= N                   */
  int32_t W;   /* Tier-2 ring capacity in tokens, >= 1                             */
} cmc_dims;

/* Human-readable name of a cmc_status value (static storage). */
CMC_API const char* cmc_status_string(int status);

/* cudaError_t of the most recent failed CUDA call made by this library on the
 * calling thread; 0 if none.  Reading it clears it. */
CMC_API int cmc_last_cuda_error(void);

/* ------------------------------------------------------------------------ *
 * Graph-based context denoising (Section 2.1)                               *
 * ------------------------------------------------------------------------ */

/* Bytes of workspace cmc_denoise needs for B contexts of n_max tokens. */
CMC_API size_t cmc_denoise_workspace_size(int B, int n_max);

/*
 * Keeps token i of context b when its cosine similarity to at least one of
 * its g following tokens j = i+1 .. min(i+g, n-1) is at least tau (the last
 * token has no follower and fails); the keep-minimum of the paper's
 * threshold appendix then forces one kept token into every run of
 * keep_every consecutive positions (walking left to right, a token is also
 * kept when the previous kept token is keep_every positions back, or, before
 * any, when it is token keep_every - 1; keep_every == 0 disables it).
 * Cosines with a zero vector are 0; the comparison is taken in fp32.
 *
 *   emb         fp32 [B, n_max, H]  token embeddings of each context
 *   n_tokens    int32 [B] tokens per context (clamped to [0, n_max]), or NULL
 *   kept_idx    int32 [B, n_max] output: the kept positions in ascending
 *               order, then -1
 *   kept_count  int32 [B] output: how many were kept
 *   workspace   >= cmc_denoise_workspace_size(B, n_max) bytes, zero-filled
 *               before its first use: its last bytes hold one completion
 *               counter per context, which every call leaves zero (calls
 *               that share a workspace must be ordered, e.g. one stream);
 *               on completion its first B * n_max bytes hold each token's
 *               threshold-test result (1 passed, 0 not or past n_tokens)
 *
 * When the contexts' 32-token tiles fit one CTA per SM (B * ceil(n_max / 32)
 * <= SM count), the whole call is one kernel launch: the CTA that finishes a
 * context's last tile also walks its keep-minimum and writes kept_idx.
 *
 * Limits: 1 <= B <= 65535, 1 <= n_max <= 2^24, 4 <= H <= 65536, H % 4 == 0,
 * 1 <= g <= 8, keep_every >= 0, tau finite.
 */
CMC_API int cmc_denoise(const float* emb, const int32_t* n_tokens, int B, int n_max, int H, int g,
                        float tau, int keep_every, int32_t* kept_idx, int32_t* kept_count,
                        void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------ *
 * MemoryBridge output (Section 2.2, the norm-calibrated tanh equation)       *
 * ------------------------------------------------------------------------ */

/*
 * Turns the output x of the MemoryBridge MLP into decoder-ready CMEs:
 *     m_hat = gamma * (x - mean(x)) / sqrt(var(x) + eps) + beta
 *             (LayerNorm over the D features, biased variance: PyTorch's
 *             default, as the paper's hyperparameter appendix states)
 *     m     = nu tanh(m_hat) * min(1, 2 nu / ||nu tanh(m_hat)||_2)
 * row by row, so every CME's norm is at most 2 nu (nu = s * mean embedding
 * norm of the decoder, a scalar the caller passes).  The MLP's matrix
 * products are plain GEMMs left to the caller.
 *
 *   x      fp32 [rows, D]      out  fp32 [rows, D] (may be x: in place)
 *   gamma, beta  fp32 [D], or NULL for ones / zeros
 *
 * Limits: rows >= 1, 4 <= D <= 16384, D % 4 == 0; eps > 0 and nu > 0 finite.
 */
CMC_API int cmc_bridge_epilogue(const float* x, const float* gamma, const float* beta,
                                int64_t rows, int D, float eps, float nu, float* out,
                                void* stream);

/* ------------------------------------------------------------------------ *
 * Tier-1: question-guided scoring and top-K selection                       *
 * (Section 2.5, the score_j equation and the top-K re-ordering after it)    *
 * ------------------------------------------------------------------------ */

/* Bytes of workspace cmc_score_select needs for B sequences of N CMEs: the
 * B * N fp32 scores (rounded up to 256 bytes), then B completion counters
 * (rounded up to 256 bytes), then B histograms of 2,048 32-bit counts. */
CMC_API size_t cmc_score_select_workspace_size(int B, int N);

/*
 * For each sequence b, scores every CME j by cosine similarity
 *     score[b, j] = (m_j . q_b) / (||m_j|| ||q_b||)
 * and writes the k indices with the highest scores, in ascending index order
 * (document order), to idx_out[b, 0..k).
 *
 *   question_emb  fp32 [B, D]       the question vectors q_vec
 *   cme_bank      fp32 [B, N, D]    the decoder-ready CMEs m_j of each sequence
 *   idx_out       int32 [B, k]      output, ascending within each row
 *   scores_out    fp32 [B, N]       optional output (NULL: not written)
 *   workspace     >= cmc_score_select_workspace_size(B, N) bytes, 16-byte
 *                 aligned, ZERO-FILLED ONCE before its first use: it holds
 *                 one completion counter and one histogram of the scores'
 *                 top 11 key bits per sequence, which every call leaves at
 *                 zero again (the scores part may hold anything).  Calls that
 *                 share a workspace must be ordered (e.g. one stream).  It may
 *                 be NULL when scores_out is given.
 *
 * Small banks with a workspace (D <= 4096, N <= 2048, and B * N rows that
 * CTAs of at most 8 rows of one sequence cover in one wave of one CTA per SM)
 * take one kernel launch: the CTA that writes the last score of a sequence (a
 * counter in the workspace tells it) selects that sequence's top k, starting
 * from the histogram the scoring CTAs built.  Larger
 * banks, or no workspace, take two launches (scoring, then selection).  Both
 * give the same selection.
 *
 * Scores are computed in fp32 with a fixed summation order, so equal rows get
 * bit-identical scores.  Equal scores go to the lower index; -0 equals +0.  A
 * zero-norm CME or question vector scores 0.  Non-finite inputs are outside
 * the contract (no fault, unspecified selection).
 * Limits: 1 <= B <= 65535, 1 <= N <= 1048576, 4 <= D <= 65536, D % 4 == 0,
 * 0 <= k <= N.
 */
CMC_API int cmc_score_select(const float* question_emb, const float* cme_bank, int B, int N, int D,
                             int k, int32_t* idx_out, float* scores_out, void* workspace,
                             size_t workspace_bytes, void* stream);

/* Bytes of workspace cmc_question_select needs for B sequences of N CMEs. */
CMC_API size_t cmc_question_select_workspace_size(int B, int N);

/*
 * The question-side prologue of a request, on the device:
 *   q_vec[b]  = mean of the first q_len[b] rows of question_tokens[b] (the
 *               question tokens' input embeddings, mean-pooled: Section 2.5,
 *               Tier-1); an empty question gives the zero vector;
 *   idx[b]    = the Tier-1 selection of cmc_score_select for q_vec;
 *   alpha[b]  = chunk_offset[b, j*] where j* is the CME of largest norm
 *               (CME-guided localisation, the appendix on deployment without
 *               annotations; norms compared in fp32, ties to the lower index);
 *   start[b]  = max(0, min(ctx_len[b] - W, alpha[b] - W/2)) (W/2 rounded
 *               down), the first context token of the W-token Tier-2 window
 *               (Section 2.5, Tier-2).
 *
 *   question_tokens  fp32 [B, Lq, D]
 *   q_len            int32 [B] tokens per question, or NULL for Lq each;
 *                    values are clamped to [0, Lq]
 *   cme_bank         fp32 [B, N, D]
 *   chunk_offset     int32 [B, N] context position of the chunk behind each
 *                    CME (same unit as ctx_len and W)
 *   ctx_len          int32 [B] context length |C|
 *   q_vec_out        fp32 [B, D] (required)
 *   idx_out          int32 [B, k] ascending (may be NULL when k == 0)
 *   alpha_out, start_out  int32 [B]; either may be NULL; when both are NULL
 *                    chunk_offset, ctx_len and W are not used
 *   workspace        >= cmc_question_select_workspace_size(B, N) bytes,
 *                    16-byte aligned, zero-filled once before its first use
 *                    (as for cmc_score_select: scores, squared norms, then
 *                    B completion counters, B histograms of 2,048 counts and
 *                    B 64-bit argmax slots, all left at zero by every call)
 *
 * Small banks (as for cmc_score_select) take one kernel launch for the whole
 * prologue; larger ones three (pooling, scoring, selection).  q_vec is the
 * fp32 mean in either case, summed in a fixed order (the two paths' orders
 * differ, within fp32 rounding).
 *
 * Limits: those of cmc_score_select, Lq >= 1, Lq * D <= 2^31, W >= 1 when
 * localising.
 */
CMC_API int cmc_question_select(const float* question_tokens, const int32_t* q_len, int Lq,
                                const float* cme_bank, int B, int N, int D, int k,
                                const int32_t* chunk_offset, const int32_t* ctx_len, int W,
                                float* q_vec_out, int32_t* idx_out, int32_t* alpha_out,
                                int32_t* start_out, void* workspace, size_t workspace_bytes,
                                void* stream);

/* ------------------------------------------------------------------------ *
 * Tier-2: local-window ring append (Section 2.5, Tier-2 and the K + W + |q| *
 * bound of "KV cache assembly")                                             *
 * ------------------------------------------------------------------------ */

/*
 * Appends one token per sequence to the ring.  Token number pos[b] (counting
 * from 0) is written to slot pos[b] mod W of every (layer, KV head); once more
 * than W tokens have been appended this overwrites the oldest one.  pos[b] is
 * then incremented on the device.
 *
 *   ring_k, ring_v  bf16 [B, L, Hkv, W, d]   updated in place
 *   pos             int64 [B]                tokens appended so far; updated
 *   k_new, v_new    bf16 [B, L, Hkv, d]      the new token's keys and values
 *
 * dims->Hq, N and k are ignored.  A sequence with pos[b] < 0 is left unchanged.
 */
CMC_API int cmc_window_append(void* ring_k, void* ring_v, int64_t* pos, const void* k_new,
                              const void* v_new, const cmc_dims* dims, void* stream);

/* ------------------------------------------------------------------------ *
 * Decode attention over [Tier-1 | Tier-2]                                   *
 * (Section 2.5 "KV cache assembly"; cost model in "Attention MACs Analysis")*
 * ------------------------------------------------------------------------ */

/* Bytes of workspace the two attention entry points need for `dims`.  The
 * workspace holds the device status word (read by cmc_read_status), one
 * 8-byte counter per sequence that the fused step uses to advance pos, and
 * fp32 partial results.  Zero-fill it once before its first use; every call
 * leaves the counters at zero again.  After a call that raised
 * CMC_DEVFLAG_TIMEOUT, zero-fill it again. */
CMC_API size_t cmc_decode_attn_workspace_size(const cmc_dims* dims);

/*
 * For every sequence b, layer l and query head h (KV head g = h / (Hq/Hkv)):
 *     out[b,l,h] = sum_i softmax_i(scale * q[b,l,h] . key_i) value_i
 * over the keys of
 *     Tier-1: tier1_k[b,l,g, idx[b,i]] for i < k (gathered by index), or,
 *             when idx is NULL, tier1_k[b,l,g, i] for i < k (the selected
 *             rows already stored in order, as cmc_tier1_gather or the
 *             prefill of the selected CMEs leaves them), then
 *     Tier-2: ring_k[b,l,g, s] for the occupied slots s < min(pos[b], W).
 * An empty cache gives a zero output.
 *
 *   q                 bf16 [B, L, Hq, d]
 *   tier1_k, tier1_v  bf16 [B, L, Hkv, N, d]   (N >= k)
 *   idx               int32 [B, k] in any order, or NULL (identity selection;
 *                     the Tier-1 tiles then stream as contiguous boxes, which
 *                     is the fast path)
 *   ring_k, ring_v    bf16 [B, L, Hkv, W, d]
 *   pos               int64 [B]      tokens appended so far (read only)
 *   scale             softmax scale; <= 0 selects 1/sqrt(d)
 *   out               bf16 [B, L, Hq, d]  (round to nearest even)
 *   workspace         see cmc_decode_attn_workspace_size
 *
 * Accumulation is fp32.  idx entries outside [0, N) are skipped and flagged
 * with CMC_DEVFLAG_BAD_INDEX.  A sequence with pos[b] < 0 gets a zero output
 * and sets CMC_DEVFLAG_BAD_POS.
 */
CMC_API int cmc_two_tier_decode_attn(const void* q, const void* tier1_k, const void* tier1_v,
                                     const int32_t* idx, const void* ring_k, const void* ring_v,
                                     const int64_t* pos, const cmc_dims* dims, float scale, void* out,
                                     void* workspace, size_t workspace_bytes, void* stream);

/*
 * One fused decode step: cmc_window_append followed by
 * cmc_two_tier_decode_attn, in one launch.  The new token is appended before
 * attention, so it attends to itself.  On return (in stream order) the ring
 * holds the new token at slot pos[b] mod W and pos[b] has grown by one.
 * Arguments are those of the two calls it fuses.  A sequence with pos[b] < 0
 * is left unchanged, its output is zero and CMC_DEVFLAG_BAD_POS is set.
 */
CMC_API int cmc_decode_step(const void* q, const void* tier1_k, const void* tier1_v,
                            const int32_t* idx, void* ring_k, void* ring_v, int64_t* pos,
                            const void* k_new, const void* v_new, const cmc_dims* dims, float scale,
                            void* out, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Tier-1 compaction, once per question: copies the selected rows of the
 * per-CME K/V bank into a dense Tier-1 cache,
 *     tier1_k[b,l,g,i] = bank_k[b,l,g, idx[b,i]]   for i < k  (same for V),
 * the cache that Section 2.5's prefill of the selected CMEs M* (re-ordered by
 * document position) leaves.  Decode steps then pass tier1_k/v with N = k and
 * idx = NULL.
 *
 *   bank_k, bank_v    bf16 [B, L, Hkv, N, d]
 *   idx               int32 [B, k]   (from cmc_score_select)
 *   tier1_k, tier1_v  bf16 [B, L, Hkv, k, d]   output; must not overlap the bank
 *   status            NULL, or a device uint32 word (for example the start of an
 *                     attention workspace) that receives CMC_DEVFLAG_BAD_INDEX
 *                     when an idx entry is outside [0, N); that row is zeroed
 *
 * dims->Hq and W are ignored.  k == 0 launches nothing.
 */
CMC_API int cmc_tier1_gather(const void* bank_k, const void* bank_v, const int32_t* idx,
                             const cmc_dims* dims, void* tier1_k, void* tier1_v, uint32_t* status,
                             void* stream);

/*
 * Launch plan of cmc_two_tier_decode_attn (fused == 0), cmc_decode_step
 * (fused == 1) or cmc_decode_step_rope (fused == 2) for `dims` on the
 * current device: *ctas receives the grid size
 * of the attention kernel and *launches the number of kernels one call
 * enqueues: 1 when every (sequence, layer, KV head) unit is handled whole by
 * one CTA (several units per CTA when there are more units than resident
 * CTAs and they share out evenly enough) or by a thread-block cluster of 2 to
 * 8 CTAs that merge their partial results in distributed shared memory; 2
 * when, with more units than resident CTAs, the tiles are split evenly
 * instead (units cut between CTAs) and a combine kernel merges the partial
 * results.  No work is enqueued.  Useful for sizing CUDA graphs and for
 * counting launches.
 */
CMC_API int cmc_decode_attn_plan(const cmc_dims* dims, int fused, int* ctas, int* launches);

/*
 * The decode step of a real GQA layer: cmc_decode_step with rotary position
 * embedding applied inside the same launch.  The decoders of Section 2.5
 * (Llama-3, Mistral) rotate queries and keys and cache the rotated keys; the
 * paper does not restate the rotation, so it follows the half-split pairing
 * of those decoders: element i pairs with element i + d/2 and the pair is
 * rotated by the angle p * rope_theta^(-2i/d).
 *
 * q and k_new are taken BEFORE rotation.  For sequence b the new token's
 * position is p = rope_offset + pos[b] (pos[b] before the append; rope_offset
 * counts the positions that precede the ring, e.g. k for the Tier-1 rows of
 * the prefill input [M* | C_local | q]).  The kernel rotates every query head
 * and the new key at p, appends the rotated key (bf16, round to nearest even)
 * and the value to the ring, and attends with the rotated query over
 * [Tier-1 | Tier-2] exactly as cmc_decode_step.  Other arguments are those of
 * cmc_decode_step.
 *
 * Angles.  The host turns each pair's frequency rope_theta^(-2i/d) / (2 pi)
 * into a 64-bit binary fraction F_i (turns per position, rounded to
 * nearest).  The kernel forms p * F_i mod 2^64 in integer arithmetic -- the
 * angle's fractional turn, exact but for the rounding of F_i, so off by at
 * most p * 2^-65 turns -- and passes its top 32 bits, as a signed fraction of
 * a half turn, to sincospif.  The angle error is thus below
 * 2 pi (p * 2^-65 + 2^-32) rad plus sincospif's, and (cos, sin) are within
 * about 1e-7 of exact for p up to 2^33; from there the first term grows as
 * p * 1.7e-19 rad.
 *
 * Errors: as cmc_decode_step; rope_theta must be positive and finite and
 * 0 <= rope_offset <= 2^32 (else CMC_ERR_RANGE).
 */
CMC_API int cmc_decode_step_rope(const void* q, const void* tier1_k, const void* tier1_v,
                                 const int32_t* idx, void* ring_k, void* ring_v, int64_t* pos,
                                 const void* k_new, const void* v_new, const cmc_dims* dims,
                                 float scale, double rope_theta, int64_t rope_offset, void* out,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* Copies the device status word of an attention workspace (CMC_DEVFLAG_*
 * bits) into *flags, waiting for `stream`, and clears it when `clear` != 0. */
CMC_API int cmc_read_status(void* workspace, int clear, uint32_t* flags, void* stream);

/* Tuning of the attention launches (cmc_two_tier_decode_attn,
 * cmc_decode_step, cmc_decode_step_rope) made afterwards, from any thread:
 * before its grid dependency wait every CTA asks L2 to prefetch the K/V boxes
 * of its first `tiles` tiles (64 keys each), so that under programmatic
 * dependent launch they stream in while the kernel before it on the stream
 * drains.  A hint only: results do not depend on it.  Default 5, the best at
 * the Llama-3-8B shape when one stream carries the launches; 0 was best when
 * four independent requests' launches ran on four streams (their launches
 * already overlap).  CMC_ERR_RANGE unless 0 <= tiles <= 64. */
CMC_API int cmc_set_l2_prefetch_tiles(int tiles);

/* Test hook for the failure path of the attention kernels (not part of the
 * method; off unless called).  With on != 0, every pipeline stage of the
 * attention launches made afterwards (cmc_two_tier_decode_attn,
 * cmc_decode_step, cmc_decode_step_rope, from any thread) expects 16 bytes
 * more than its loads deliver, so no stage ever completes: each CTA's first
 * wait gives up after its 1 s limit, the CTA's other waits end at once, the
 * launch returns and the workspace's status word gets CMC_DEVFLAG_TIMEOUT.
 * Outputs, ring and pos of such a call are invalid, and its workspace must be
 * zero-filled again.  on == 0 restores normal operation.  Always CMC_OK. */
CMC_API int cmc_test_stall_attention_waits(int on);

/* ------------------------------------------------------------------------ *
 * Staging copies for a serving loop (not a step of the paper's method: the  *
 * input and output traffic of the decode loop around it)                    *
 * ------------------------------------------------------------------------ */

/* One byte range to copy. */
typedef struct cmc_copy {
  const void* src; /* device memory, or pinned host memory the device can address */
  void* dst;       /* likewise                                                     */
  size_t bytes;    /* a multiple of 16; src and dst 16-byte aligned                */
} cmc_copy;

/*
 * Copies up to 4 byte ranges in one kernel launch, with 16-byte loads and
 * stores, so either side may be pinned host memory (cudaHostAlloc, or
 * cudaHostRegister with cudaHostRegisterMapped: on systems with unified
 * addressing its host address is also its device address).  This moves the
 * per-step inputs in and outputs out of a decode loop without a copy engine:
 * a copy-engine copy between two kernels on the stream, or a wait on another
 * stream's copy, ends programmatic dependent launch for the kernel after it,
 * and with it the overlap of that kernel's start with its predecessor's end.
 *
 * wait_first == 0: the copies start without waiting for the work enqueued
 * before them on `stream`, and the launch completes only after that work
 * (it waits at its end), so the copies overlap the preceding kernel and
 * everything enqueued after the call sees both.  The caller guarantees that
 * the preceding work neither writes any source nor reads or writes any
 * destination (double-buffer the device buffers).
 * wait_first != 0: the copies start after the preceding work, like an
 * ordinary stream operation.
 *
 * Errors: n outside [0, 4] -> CMC_ERR_RANGE; copies NULL with n > 0, or a NULL
 * src / dst with bytes > 0 -> CMC_ERR_NULL; misaligned pointer or size ->
 * CMC_ERR_ALIGN.  Copies of 0 bytes are skipped.  The library does not check
 * that a host pointer is pinned and mapped: an unmapped one faults.
 */
CMC_API int cmc_stage_copies(const cmc_copy* copies, int n, int wait_first, void* stream);

/* ------------------------------------------------------------------------ *
 * Allocation-free Tier-1 selection                                          *
 * ------------------------------------------------------------------------ */

/* Largest B * N that cmc_score_select_static accepts (1 MiB of fp32 scores). */
#define CMC_STATIC_SCORES_MAX 262144

/*
 * cmc_score_select without a caller-provided workspace.  The paper has no
 * counterpart: this is a deployment variant of the same computation.
 *
 * Some callers cannot hand the library a workspace: a serving engine that
 * reserves all free HBM for its KV-cache pool at start-up and forbids any
 * later allocation, or a plain C host program that links only this library
 * and owns no device allocator.  This entry point allocates nothing and calls
 * no allocating routine.  Its score scratch is one file-scope device array of
 * CMC_STATIC_SCORES_MAX floats (1 MiB), which every GPU that loads the library
 * holds until the process exits.
 *
 * Arguments, results and limits are those of cmc_score_select, except that
 * there is no scores_out and no workspace, and B * N must not exceed
 * CMC_STATIC_SCORES_MAX (otherwise CMC_ERR_SHAPE, nothing launched).
 *
 * The first call on a device looks up the array's device address (with that
 * device current); make that first call before any stream capture.  All calls
 * share the one array: each call overwrites the B * N scores it then reads,
 * so nothing in it needs to start at zero, but calls whose kernels overlap on
 * the GPU (different streams, no ordering between them) race on it.
 */
CMC_API int cmc_score_select_static(const float* question_emb, const float* cme_bank, int B,
                                    int N, int D, int k, int32_t* idx_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* CMC_H_ */
