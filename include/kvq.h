/*
 * kvq.h — C ABI of the low-bit KV-cache decode step and the DGAP epilogue.
 *
 * One decode step of the method of arXiv 2607.16248 ("High-accuracy Low-Bit
 * KV-Cache Quantization via Local Distribution Restoration"), built for one
 * GB300 (sm_103a):
 *
 *   kvq_pack         append the step's new K/V to a KbVb cache (Sec. 3.1)
 *   kvq_decode_attn  softmax(q K^T / sqrt(d)) V over that cache (Sec. 1)
 *   dgap_restore     features, detector, gate, top-K corrector, sparse merge
 *                    on the step's logits (Sec. 4.1-4.3, Eqs. 2, 6, 11-13)
 *   kvq_drift_*      offline drift metrics on paired FP16 / low-bit logits and
 *                    the recovery-window rule (Sec. 4.1, Sec. 4.2)
 *
 * Conventions for every call
 * --------------------------
 * - Pointers named "device" point to GPU memory owned by the caller; the
 *   library never allocates, frees or synchronises.  Work is enqueued on the
 *   CUDA stream passed as `stream` (a cudaStream_t; NULL = legacy default).
 * - fp16 data is IEEE binary16 passed as uint16_t bit patterns.
 * - Every call validates its arguments on the host first and returns a
 *   kvq_status; on failure nothing is enqueued and kvq_last_error() (a
 *   thread-local string) says why.  KVQ_ERR_CUDA reports a launch error.
 * - Errors that only the device can see (a sequence pushed past max_len)
 *   never fault the GPU: the kernel skips the write and sets a bit in the
 *   cache's flag word (see kvq_cache).
 * - KVQ_TRACE=1 in the environment prints one line per launch to stderr
 *   (entry point, shapes, grid and split choices).
 */
#ifndef KVQ_H
#define KVQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum kvq_status {
  KVQ_OK = 0,
  KVQ_ERR_ARG = 1,         /* null pointer, bad scalar argument           */
  KVQ_ERR_SHAPE = 2,       /* inconsistent sizes                           */
  KVQ_ERR_UNSUPPORTED = 3, /* bits not in {1,2,4,8}, head_dim != 128 ...   */
  KVQ_ERR_CAPACITY = 4,    /* workspace or cache too small                 */
  KVQ_ERR_ALIGN = 5,       /* pointer not 16-byte aligned                  */
  KVQ_ERR_CUDA = 6         /* kernel launch failed                         */
} kvq_status;

/* Device-side flag bits (cache flag word). */
#define KVQ_FLAG_OVERFLOW 1u /* an append would have passed max_len */
#define KVQ_FLAG_WAIT_TIMEOUT 2u /* an attention kernel's copy wait gave up (~2 s);
                                    its output for that call is not valid */
#define KVQ_FLAG_BAD_PAGE 4u /* a paged cache's block table mapped a block that a
                                call had to read or write outside [0, n_pages):
                                the write was skipped, and an output that needed
                                the block is not valid */

/*
 * Cache configuration.  KbVb with b_k = bits_k and b_v = bits_v (Sec. 3.1
 * names the symmetric settings K1V1..K8V8; Table "ablation_target" of Sec. 5.5
 * also uses K2V1 and K1V2, so the two widths are independent here).
 *   head_dim  must be 128;  group must be 32;
 *   residual  R, fp16 recent-token window, a positive multiple of 32;
 *   max_len   capacity in tokens per sequence, a positive multiple of 32.
 * Grouped-query attention: query head i reads kv-head i / (n_q_heads /
 * n_kv_heads); n_q_heads / n_kv_heads must be an integer in [1, 8].
 */
typedef struct kvq_config {
  int32_t batch;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t bits_k;
  int32_t bits_v;
  int32_t group;
  int32_t residual;
  int32_t max_len;
} kvq_config;

/*
 * Cache storage (all device pointers, caller-owned; kvq_cache_layout gives
 * the sizes and kvq_cache_bind carves them out of one buffer).
 *
 * Token groups are aligned to absolute position 0.  With L tokens cached,
 * Lq = 32 * floor(max(L - R, 0) / 32) tokens live in quantized 32-token
 * blocks and the other L - Lq (R <= L - Lq <= R + 31 once L >= R) stay fp16.
 *
 * pages   [batch][n_kv_heads][max_len / 32][page_bytes], one page per 32-token
 *         block, page_bytes = 512 * (bits_k + bits_v) + 1024:
 *           K codes  [128 channel][bits_k] uint32   (group = 32 tokens of one channel)
 *           K meta   fp16 scale[128 channel], then fp16 zero[128 channel]
 *           V codes  [4 group][32 token][bits_v] uint32 (group = 32 channels of one token)
 *           V meta   fp16 scale[128], then fp16 zero[128]; (group g, token t)
 *                    at 32 g + 8 (t / 8) + 2 (t mod 4) + (t / 4) mod 2, i.e. the
 *                    tokens of each 8-token run in the order 0 4 1 5 2 6 3 7
 *         For b >= 2, element i of a group occupies bits [(i*b) mod 32, +b)
 *         of word floor(i*b / 32).  1-bit codes (512 bytes per tensor) are
 *         stored in the order the attention kernel's MMA fragments read
 *         them: with gid = t / 4, j = t mod 4 (keys: token t, channel
 *         c = 16 ks + 4 tig + 2 h + e) the key code sits in word
 *         16 gid + 4 tig + ks / 2 at bit (10 + 16 e + j - 4 (2 (ks mod 2) + h))
 *         mod 32; with gid = (c mod 32) / 4, j = c mod 4, tig = t / 8,
 *         r = t mod 4, e = (t / 4) mod 2 (values: token t, channel c) the
 *         value code sits in word 16 gid + 4 tig + c / 32 at bit
 *         (10 + 16 e + j - 4 r) mod 32.  Quantizer (b bits, group x_1..x_32):
 *           zero  = min x_i
 *           scale = RU16(RU32(RU32(max x_i - min x_i) / (2^b - 1)))
 *           code  = clamp(rint(RN32(RN32(x - zero) / scale)), 0, 2^b - 1)
 *         (RU = IEEE round toward +inf, RN = to nearest even; scale 0 gives
 *         code 0).  Dequantized value: zero + scale * code.
 * k_resid, v_resid  [batch][n_kv_heads][R + 32][128] fp16 ring; token at
 *         absolute position p sits in slot p mod (R + 32).
 * seq_len [batch + 2] int32: [0, batch) token counts L, [batch] the flag word
 *         (KVQ_FLAG_*), [batch + 1] reserved; followed by `batch` uint32
 *         tickets used by kvq_pack and kvq_decode_step.  kvq_cache_reset
 *         zeroes all of it.
 */
typedef struct kvq_cache {
  void* pages;
  uint16_t* k_resid;
  uint16_t* v_resid;
  int32_t* seq_len;
  const int32_t* block_table; /* NULL: the contiguous page layout above */
  int32_t n_pages;            /* page sets in the pool (paged layout only) */
} kvq_cache;

/*
 * Paged layout (block_table != NULL; Sec. 3.1's 32-token groups as the unit
 * of a shared page pool, for ragged batches that should not reserve max_len
 * per sequence):
 *   pages        device pool [n_pages][n_kv_heads][page_bytes]: one page set
 *                holds one 32-token block of one sequence for every kv-head;
 *                16-byte aligned.
 *   block_table  device int32 [batch][max_len / 32]: entry (b, j) is the page
 *                set of block j (tokens [32 j, 32 j + 32)) of sequence b.
 *   n_pages      1 .. 2^31 - 1.
 * The caller owns both and assigns the entries: every block a call reads
 * (j < Lq / 32) or writes must be mapped to a page set in [0, n_pages) before
 * the call is enqueued, and distinct blocks of live sequences must map to
 * distinct page sets.  kvq_pack of n_new tokens writes blocks
 * [Lq(L) / 32, Lq(L + n_new) / 32); a kvq_decode_step from L to L + 1 tokens
 * writes block Lq(L + 1) / 32 - 1 exactly when Lq(L + 1) > Lq(L), i.e. when
 * L + 1 - R is a positive multiple of 32 (Lq as above; the caller knows the
 * lengths).  An entry of a block that holds data must not change while a
 * call that may read it is in flight.  A block mapped outside [0, n_pages)
 * is never dereferenced: the kernel skips it and sets KVQ_FLAG_BAD_PAGE.
 * The fp16 window and seq_len keep the layout above (kvq_paged_cache_layout).
 */

/* Thread-local description of the last failure ("" after success). */
const char* kvq_last_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t kvq_version(void);

/* Host-only: KVQ_OK when `cfg` is supported. */
kvq_status kvq_validate_config(const kvq_config* cfg);

/* Host-only: bytes of one 32-token page (0 on an invalid config). */
size_t kvq_page_bytes(const kvq_config* cfg);

/*
 * Host-only layout query.  *total_bytes receives the size of one buffer that
 * holds the whole cache; offsets[0..3] the byte offsets of pages, k_resid,
 * v_resid and seq_len inside it (each 256-byte aligned).
 */
kvq_status kvq_cache_layout(const kvq_config* cfg, size_t* total_bytes,
                            size_t offsets[4]);

/* Host-only: fill *cache with pointers into `base` (device, >= total_bytes,
 * 256-byte aligned) following kvq_cache_layout (contiguous pages;
 * block_table = NULL, n_pages = 0). */
kvq_status kvq_cache_bind(const kvq_config* cfg, void* base, kvq_cache* cache);

/* Host-only: bytes of a page pool of n_pages page sets (0 if invalid). */
size_t kvq_page_pool_bytes(const kvq_config* cfg, int32_t n_pages);

/*
 * Host-only layout query of a paged cache: the fp16 rings and seq_len only
 * (the pages live in the caller's pool).  offsets[0] is 0 and the page
 * region is empty; offsets[1..3] as in kvq_cache_layout.
 */
kvq_status kvq_paged_cache_layout(const kvq_config* cfg, size_t* total_bytes,
                                  size_t offsets[4]);

/*
 * Host-only: a paged cache.  `base` (device, >= the paged total, 256-byte
 * aligned) holds the rings and seq_len; `pool` (device, 16-byte aligned,
 * >= kvq_page_pool_bytes(cfg, n_pages)) the page sets; `block_table` (device
 * int32 [batch][max_len / 32]) the caller's mapping (see the paged layout).
 */
kvq_status kvq_paged_cache_bind(const kvq_config* cfg, void* base, void* pool,
                                int32_t n_pages, const int32_t* block_table,
                                kvq_cache* cache);

/* Empty every sequence: zero seq_len, the flag word and the tickets. */
kvq_status kvq_cache_reset(const kvq_config* cfg, const kvq_cache* cache,
                           void* stream);

/*
 * kvq_pack — append n_new tokens to sequences [batch_begin, batch_begin +
 * batch_count) and quantize every 32-token group that leaves the residual
 * window (Sec. 3.1, KbVb).
 *   k_new, v_new  device fp16 [batch_count][n_kv_heads][n_new][128], 16-byte
 *                 aligned; the new tokens of each sequence, oldest first.
 *   n_new         1 for a decode step; larger for prefill.  Sequences of
 *                 different lengths are prefilled by calls with
 *                 batch_count = 1.
 * Each sequence's current length is read on the device, so the call can be
 * captured once in a CUDA graph and replayed every step.  A sequence that
 * would pass max_len is left unchanged and KVQ_FLAG_OVERFLOW is set.
 * Must be ordered before the kvq_decode_attn of the same step (the query
 * attends to its own token).
 */
kvq_status kvq_pack(const kvq_config* cfg, const kvq_cache* cache,
                    const uint16_t* k_new, const uint16_t* v_new,
                    int32_t n_new, int32_t batch_begin, int32_t batch_count,
                    void* stream);

/*
 * Split-K workspace for kvq_decode_attn / kvq_decode_step with the given
 * n_splits (see kvq_decode_attn: > 0 the split plan, 0 the flat plan): a
 * partial max, sum and fp32 output row per query head for every CTA of the
 * launch and two per (sequence, kv-head) pair, one ticket per pair and one
 * counter.  Returns 0 on an invalid config or n_splits outside [0, 255].
 */
size_t kvq_attn_workspace_bytes(const kvq_config* cfg, int32_t n_splits);

/*
 * The split plan's count for one wave: one 512-thread CTA per SM over all
 * (sequence, kv-head) pairs, SMs / (batch * n_kv_heads), between 1 and 255
 * (capped at a quarter of the blocks of max_len).
 */
int32_t kvq_attn_default_splits(const kvq_config* cfg);

/*
 * The n_splits to pass kvq_decode_attn / kvq_decode_step for the sequence
 * lengths, which the caller knows on the host (the library keeps them on the
 * device).  lengths: host int32 [batch], each in [0, max_len].
 *   kvq_attn_default_splits (the split plan) when one wave of its CTAs fills
 *   at least 90% of the GPU, as for batch-1 decoding, where a launch is
 *   bound by latency and dedicated window warps keep the fp16 chunks off the
 *   block warps' path; otherwise 0, the flat plan, which streams every pair
 *   in one wave (no CTA start and merges per wave).
 * Returns -1 on an invalid argument.
 */
int32_t kvq_attn_splits_for_lengths(const kvq_config* cfg, const int32_t* lengths);

/*
 * Zero a workspace (attention or DGAP) once after allocating it.  Both
 * kernels leave their tickets at zero when they finish, so one
 * initialisation serves any number of calls.
 */
kvq_status kvq_workspace_init(void* workspace, size_t ws_bytes, void* stream);

/*
 * kvq_decode_attn — one decode step of grouped-query attention
 *   out[b, i] = softmax(q[b, i] . K_hat[b, g(i)]^T * softmax_scale) V_hat[b, g(i)]
 * over all L = seq_len[b] cached tokens (Sec. 1 gives softmax(QK^T/sqrt(d_k))V;
 * g(i) = i / (n_q_heads / n_kv_heads)).  K_hat, V_hat are the dequantized
 * blocks plus the fp16 residual window.  Accumulation is fp32; the result is
 * rounded once to fp16 (round to nearest even) when it is stored.
 *   q              device fp16 [batch][n_q_heads][128], 16-byte aligned.
 *   out            device fp16 [batch][n_q_heads][128], 16-byte aligned.
 *   softmax_scale  0 selects 1/sqrt(128).
 *   n_splits       the work plan.  1..255: the split plan, n_splits CTAs per
 *                  (sequence, kv-head) pair share its 32-token blocks
 *                  (contiguous ranges, one per warp) and its window chunks
 *                  (dedicated warps).  0: the flat plan, one CTA per SM; all
 *                  pairs' blocks and window chunks lie end to end, weighted
 *                  by their measured cost, and every warp takes an equal
 *                  contiguous share, crossing pair boundaries as it goes.
 *                  Either way a pair's CTAs (and a warp that leaves a pair
 *                  for the next) write partials (max, sum, output row) to the
 *                  workspace and the last to finish merges them; a pair with
 *                  a single partial is written directly.
 *   workspace      device, >= kvq_attn_workspace_bytes(cfg, n_splits), zeroed
 *                  once by kvq_workspace_init.
 * A sequence with L = 0 gets a zero output.  Calls that share a workspace
 * must not overlap on the GPU.
 */
kvq_status kvq_decode_attn(const kvq_config* cfg, const kvq_cache* cache,
                           const uint16_t* q, uint16_t* out,
                           float softmax_scale, int32_t n_splits,
                           void* workspace, size_t ws_bytes, void* stream);

/*
 * kvq_decode_attn_f32 — kvq_decode_attn with the fp32 accumulation result
 * stored unrounded: out is device fp32 [batch][n_q_heads][128].  Rounding it
 * to fp16 to nearest even gives kvq_decode_attn's output bit for bit.
 */
kvq_status kvq_decode_attn_f32(const kvq_config* cfg, const kvq_cache* cache,
                               const uint16_t* q, float* out,
                               float softmax_scale, int32_t n_splits,
                               void* workspace, size_t ws_bytes, void* stream);

/*
 * kvq_decode_step — one decode step of one layer: kvq_pack of one token per
 * sequence followed by kvq_decode_attn, in one kernel (Sec. 3.1 quantizer,
 * Sec. 1 attention).  The token at position L = seq_len[b] is attended from
 * k_new / v_new directly and written to its window slot; when it pushes a
 * 32-token group out of the window, that group is quantized (bit-identical to
 * kvq_pack) into its page and attended in quantized form; seq_len[b] becomes
 * L + 1 when the kernel ends.
 *   k_new, v_new   device fp16 [batch][n_kv_heads][128], 16-byte aligned.
 *   q, out, softmax_scale, n_splits, workspace, ws_bytes: as kvq_decode_attn
 *                  (out fp16).
 * A sequence at max_len is not appended (KVQ_FLAG_OVERFLOW is set) and
 * attends over its L tokens.  Results equal kvq_pack(n_new = 1) then
 * kvq_decode_attn on the same inputs.
 */
kvq_status kvq_decode_step(const kvq_config* cfg, const kvq_cache* cache,
                           const uint16_t* k_new, const uint16_t* v_new,
                           const uint16_t* q, uint16_t* out, float softmax_scale,
                           int32_t n_splits, void* workspace, size_t ws_bytes,
                           void* stream);

/* kvq_decode_step_f32 — kvq_decode_step with an fp32 out, as
 * kvq_decode_attn_f32. */
kvq_status kvq_decode_step_f32(const kvq_config* cfg, const kvq_cache* cache,
                               const uint16_t* k_new, const uint16_t* v_new,
                               const uint16_t* q, float* out, float softmax_scale,
                               int32_t n_splits, void* workspace, size_t ws_bytes,
                               void* stream);

/*
 * kvq_decode_attn_noalloc — kvq_decode_attn_f32 without a caller workspace.
 * The paper has no counterpart; this serves callers that cannot allocate
 * device memory where they run a decode step: code inside a framework whose
 * memory pool owns the whole GPU (a raw allocation would fail or fragment
 * it), or a serving loop that must not allocate per step.  The split
 * partials and tickets live in one built-in device array of
 * KVQ_NOALLOC_SCRATCH_BYTES, which every GPU that loads this library holds
 * until the process exits.
 *   Arguments and results: those of kvq_decode_attn_f32 (fp32 out), without
 *   workspace.
 *   Returns KVQ_ERR_CAPACITY, with nothing enqueued, when
 *   kvq_attn_workspace_bytes(cfg, n_splits) > KVQ_NOALLOC_SCRATCH_BYTES.
 *   The first call on a device looks up the array's device address (once
 *   per device, with that device current): make that first call before any
 *   stream capture.  Every call shares the one array and it keeps the last
 *   call's contents; each call zeroes the tickets it uses before its kernel.
 *   Calls that overlap on the GPU (different streams, or unordered work)
 *   race and give wrong results.  Allocates and frees nothing.
 */
#define KVQ_NOALLOC_SCRATCH_BYTES (4u << 20)
kvq_status kvq_decode_attn_noalloc(const kvq_config* cfg, const kvq_cache* cache,
                                   const uint16_t* q, float* out,
                                   float softmax_scale, int32_t n_splits,
                                   void* stream);

/*
 * DGAP parameters (Sec. 4.2 detector, Sec. 4.3 corrector).  Weights are
 * device fp32, row-major [out][in]; H = hidden.
 *   detector  f = w2 . relu(W1 phi + b1) + b2, r = sigmoid(f)   (Eq. 6)
 *             det_w1 [H][8], det_b1 [H], det_w2 [H], det_b2 [1]
 *   corrector Delta = W2 relu(W1 [xi | phi] + b1) + b2          (Eq. 12)
 *             cor_w1 [H][5K + 8], cor_b1 [H], cor_w2 [K][H], cor_b2 [K]
 *   K    recovery window size K_b, 2 <= K <= 64, K < vocab (Eqs. 2, 11)
 *   H    1 <= hidden <= 1024
 *   tau  risk threshold; the corrector runs when r > tau (Eq. 13); the
 *        paper's calibrated value is 0.60 (Sec. 5.5).
 * phi (8 features, in order): entropy of softmax(z); top-K mass; top-1
 * probability; z_(0) - z_(1); (z_(0) - z_(K-1)) / (K - 1); least adjacent gap
 * in the window; population std of the window logits; entropy of the
 * window's renormalised probabilities.  xi (5 per window rank k):
 * z_(k) - z_(0); log p_(k); k / (K - 1); z_(k-1) - z_(k) (0 at k = 0);
 * z_(k) - z_(k+1) (z_(K) is the (K+1)-th logit).
 */
typedef struct dgap_params {
  int32_t K;
  int32_t hidden;
  float tau;
  const float* det_w1;
  const float* det_b1;
  const float* det_w2;
  const float* det_b2;
  const float* cor_w1;
  const float* cor_b1;
  const float* cor_w2;
  const float* cor_b2;
} dgap_params;

/* Workspace bytes for dgap_restore on [batch][vocab] logits (0 if invalid). */
size_t dgap_workspace_bytes(int32_t batch, int32_t vocab, const dgap_params* p);

/*
 * dgap_restore — the DGAP epilogue on one decode step's logits (Sec. 4.1-4.3).
 * For each row z (finite fp32):
 *   S = TopK(z, K): value descending, lowest index first on ties (Eqs. 2, 11);
 *   phi = Phi(z); r = sigmoid(f_theta(phi)) (Eq. 6);
 *   if r > tau: Delta = g_psi(xi_S, phi) and z[S_k] += Delta_k in place
 *   (Eq. 13); every other logit, and every logit of an ungated row, is left
 *   bit-identical.
 *   logits      device fp32 [batch][vocab], updated in place, 16-byte aligned.
 *   topk_idx    device int32 [batch][K]: S in rank order.
 *   topk_val    device fp32 [batch][K]: merged values z~ at S.
 *   risk        device fp32 [batch]: r.
 *   gate        device uint8 [batch]: 1 when the corrector ran.
 *   next_token  device int32 [batch] or NULL: argmax of the merged row
 *               (lowest index on ties), i.e. greedy token selection.
 *   features    device fp32 [batch][8] or NULL: phi.
 *   workspace   device, >= dgap_workspace_bytes(...), zeroed once by
 *               kvq_workspace_init; calls sharing it must not overlap.
 * The gate is decided as f > log(tau / (1 - tau)) (tau >= 1: never; tau <= 0:
 * always), which equals r > tau.
 */
kvq_status dgap_restore(const dgap_params* params, float* logits,
                        int32_t batch, int32_t vocab, int32_t* topk_idx,
                        float* topk_val, float* risk, uint8_t* gate,
                        int32_t* next_token, float* features, void* workspace,
                        size_t ws_bytes, void* stream);

/*
 * kvq_selftest_wait_timeout — checks on the device that a bounded wait gives
 * up instead of hanging.  One warp waits, with a limit of ~10 ms, on an
 * mbarrier armed for 16 bytes that no copy delivers (the loop the attention
 * kernels use for their copy waits, whose limit is ~2 s); the wait runs out
 * and the kernel sets KVQ_FLAG_WAIT_TIMEOUT in *flag and returns, leaving
 * the context usable.
 *   flag  device uint32, 4-byte aligned; the bit is OR-ed in.
 */
kvq_status kvq_selftest_wait_timeout(uint32_t* flag, void* stream);

/*
 * Offline drift metrics (Sec. 4.1 "Adaptive recovery-window selection",
 * Sec. 4.2 "Offline supervision and calibration").  Tooling for paired
 * traces: each row holds one decode step's FP16-cache logits z_fp and
 * low-bit-cache logits z_q.  With p = softmax(z), both orders taking values
 * descending and the lowest index first among equal values:
 *   C(alpha)  the shortest prefix of the z_fp order whose p_fp mass reaches
 *             alpha (all of the vocabulary if it never does); M_t = |C|;
 *   S         TopK(z_q, window);
 *   c_t       sum of p_fp over C and S (recoverable coverage);
 *   d_loc     || p_fp / p_fp(U) - p_q / p_q(U) ||_2 over U = C union S;
 *   y_t       1 if d_loc > eps and c_t >= rho_c, else 0 (the label);
 *   cov[k-1]  sum of p_fp over C and TopK(z_q, k), k = 1 .. k_max.
 * The paper gives no values for alpha, eps, rho_c or rho_K.
 */
typedef struct kvq_drift_params {
  float alpha;     /* FP16 candidate mass, 0 < alpha <= 1 */
  int32_t window;  /* K of S, 1 <= window <= k_max */
  int32_t k_max;   /* coverage curve length, 1 <= k_max <= 256 and <= vocab */
  float eps;       /* d_loc threshold of the label, finite */
  float rho_c;     /* coverage threshold of the label, finite */
} kvq_drift_params;

/* Largest vocab kvq_drift_metrics accepts (163840). */
int32_t kvq_drift_max_vocab(void);

/*
 * kvq_drift_metrics — the metrics above for `rows` steps.
 *   z_fp, z_q  device fp32 [rows][vocab], finite (no NaN or +inf; -inf is a
 *              zero-probability logit), read only.  16-byte alignment of
 *              each row (vocab a multiple of 4) gives vector loads.
 *   m_t        device int32 [rows]; c_t, d_loc device fp32 [rows];
 *   y_t        device uint8 [rows]; cov device fp32 [rows][k_max].
 * Probabilities are e^(z - max z) in fp32, summed in fp64 (c_t, d_loc are
 * the fp64 results rounded to fp32).  rows <= 65535, vocab <= 163840.
 * No workspace; calls on different outputs may overlap.
 */
kvq_status kvq_drift_metrics(const float* z_fp, const float* z_q, int32_t rows,
                             int32_t vocab, const kvq_drift_params* params,
                             int32_t* m_t, float* c_t, float* d_loc,
                             uint8_t* y_t, float* cov, void* stream);

/*
 * kvq_drift_window — K_b of Sec. 4.1: the smallest k whose coverage
 * cov[.][k-1], averaged over the rows, reaches rho_k; 0 if none does.
 *   cov       device fp32 [rows][k_max] (from kvq_drift_metrics).
 *   mean_cov  device fp32 [k_max]: the column means (fp64 sums, row order).
 *   k_b       device int32 [1].
 */
kvq_status kvq_drift_window(const float* cov, int32_t rows, int32_t k_max,
                            float rho_k, float* mean_cov, int32_t* k_b,
                            void* stream);

#ifdef __cplusplus
}
#endif

#endif /* KVQ_H */
