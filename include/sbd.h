/*
 * sbd.h -- C ABI of the Set Block Decoding (SBD) block step on GB300 (sm_103a).
 *
 * One SBD forward over a block of k positions (arXiv 2509.04185, Sec. 2.3,
 * Eq. 5 and Algorithm 3) is served by three calls, issued in this order on
 * one CUDA stream:
 *
 *   sbd_block_attention      block queries attend to the exact KV cache and,
 *                            bidirectionally, to each other (Eq. 5; Fig. 3);
 *   sbd_head_entropy_sample  LM head over the masked positions, reduced in
 *                            the same kernel to a softmax entropy and a
 *                            Gumbel-max token per position (Eqs. 6-7);
 *   sbd_eb_select            entropy-bounded unmasking (Eq. 3).
 *
 * Conventions shared by every call
 *   - Every tensor argument is a caller-owned DEVICE pointer to contiguous
 *     row-major memory, aligned to 16 bytes.  Shapes are given in the call's
 *     descriptor; the library never keeps a pointer after the call returns.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is
 *     enqueued asynchronously; the calls never synchronise the device.
 *   - The library allocates no device memory.  Calls that need scratch take
 *     a caller-owned `workspace` of at least the size returned by the
 *     matching *_workspace_size() query; the scratch content between calls
 *     is irrelevant (nothing needs zeroing).
 *   - Argument errors are detected on the host before anything is enqueued
 *     and returned as a status; sbd_last_error() then gives a one-line
 *     explanation (per calling thread).  Launch failures return
 *     SBD_ERR_CUDA.  No C++ exception crosses this interface.
 *   - Device-side faults that the host cannot see before launch (a cache
 *     length outside [0, max_cache_len], a wait that timed out) are recorded
 *     in a device error word read by sbd_device_error().
 *   - Calls are thread-safe; concurrent calls may share nothing but
 *     read-only inputs (each needs its own outputs and workspace).
 */
#ifndef SBD_H
#define SBD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SBD_OK = 0,
  SBD_ERR_INVALID_ARG = 1, /* null pointer, bad size, misalignment, bad gamma/tau */
  SBD_ERR_UNSUPPORTED = 2, /* valid but outside what the kernels implement */
  SBD_ERR_WORKSPACE = 3,   /* workspace missing or smaller than required */
  SBD_ERR_CUDA = 4         /* a CUDA runtime/driver call or a launch failed */
} sbd_status;

typedef enum { SBD_DTYPE_F32 = 0, SBD_DTYPE_BF16 = 1 } sbd_dtype;

/* ------------------------------------------------------------------------
 * Block attention (Eq. 5 with the inference mask of Fig. 3 and of the
 * FlexAttention appendix listing): every block query row i of sequence b
 * sees the cached keys 0 .. cache_len[b]-1 and all k block keys.
 *
 *   q        [B, k, Hq, D]          block queries (already position-encoded)
 *   k_cache  [B, Lmax, Hkv, D]      exact KV cache of x_<t; slots at or past
 *   v_cache  [B, Lmax, Hkv, D]      cache_len[b] are never used (may hold NaN)
 *   cache_len[B] int32 (device)     0 <= cache_len[b] <= Lmax
 *   k_blk    [B, k, Hkv, D]         keys/values of the k block positions
 *   v_blk    [B, k, Hkv, D]         (recomputed every forward, not cached)
 *   out      [B, k, Hq, D]          attention output, same dtype as q
 *
 * Query head h reads KV head h / (Hq / Hkv).  s = scale * q.k with
 * scale = desc->scale, or 1/sqrt(D) when desc->scale == 0.  All inputs share
 * desc->dtype; accumulation is fp32.
 * Supported: 1 <= k <= 32, D in {64, 128}, Hq % Hkv == 0,
 * (Hq/Hkv) * k <= 128.  desc->num_splits = 0 picks the KV split count.
 * ---------------------------------------------------------------------- */
typedef struct {
  int32_t batch;          /* B   */
  int32_t block_k;        /* k   */
  int32_t n_q_heads;      /* Hq  */
  int32_t n_kv_heads;     /* Hkv */
  int32_t head_dim;       /* D   */
  int32_t max_cache_len;  /* Lmax (row count of k_cache / v_cache) */
  int32_t dtype;          /* sbd_dtype */
  float scale;            /* 0 -> 1/sqrt(D) */
  int32_t num_splits;     /* 0 -> automatic; else KV splits per (b, kv head) */
} sbd_attn_desc;

size_t sbd_block_attention_workspace_size(const sbd_attn_desc* desc);

sbd_status sbd_block_attention(const sbd_attn_desc* desc, const void* q,
                               const void* k_cache, const void* v_cache,
                               const int32_t* cache_len, const void* k_blk,
                               const void* v_blk, void* out, void* workspace,
                               size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Block attention of the first iteration of a block after the previous one
 * (Algorithm 3, "first iteration and t >= k"; the inference mask of the
 * FlexAttention appendix listing with its causal point at the new block).
 * The forward carries the n_causal tokens of the previous block, which the
 * cache does not hold yet, as the leading block rows:
 *   block row i <  n_causal  sees the cached keys and block keys j <= i;
 *   block row i >= n_causal  sees the cached keys and all block keys;
 * and the keys/values of rows i < n_causal are written into the caches at
 * positions cache_len[b] + i.  cache_len itself is not changed: the caller
 * advances it by n_causal once the call has completed.  Arguments, layouts,
 * workspace and errors are those of sbd_block_attention, except that
 * k_cache / v_cache are written (only at the n_causal new positions), and
 * 0 <= n_causal <= block_k (else SBD_ERR_INVALID_ARG).  A sequence with
 * cache_len[b] + n_causal > max_cache_len gets no append and sets
 * SBD_DEVERR_CACHE_LEN.  n_causal = 0 is sbd_block_attention.
 * ---------------------------------------------------------------------- */
sbd_status sbd_block_attention_causal_prefix(const sbd_attn_desc* desc, int32_t n_causal,
                                             const void* q, void* k_cache, void* v_cache,
                                             const int32_t* cache_len, const void* k_blk,
                                             const void* v_blk, void* out, void* workspace,
                                             size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * LM head + entropy + Gumbel-max sample (Eqs. 6-7; Algorithm 3 "compute
 * probabilities"), over the MASKED block positions only.  For masked
 * position (b, i) with hidden row h = hidden[b, i, :]:
 *   z_v      = sum_c h_c * w[v, c]                (fp32 accumulate)
 *   entropy  = -sum_v p_v log p_v, p = softmax(z)  (nats)
 *   token    = argmax_v (z_v + tau * gumbel[b, i, v]), lowest v on ties
 * Logits are never written to memory.  Unmasked positions get
 * entropy = +inf and token = -1.
 *
 *   hidden [B, k, H], w [V, H] (nn.Linear layout), same dtype
 *   masked [B, k] uint8 (nonzero = masked)
 *   gumbel [B, k, V] fp32, indexed by block position; may be NULL iff
 *          tau == 0 (greedy); rows of unmasked positions are not read
 *   entropy [B, k] fp32 out, token [B, k] int32 out
 * Supported: B * k <= 512, H % 64 == 0 for bf16 (H % 4 == 0 for fp32),
 * tau >= 0 and finite.
 * ---------------------------------------------------------------------- */
typedef struct {
  int32_t batch;    /* B */
  int32_t block_k;  /* k */
  int32_t hidden;   /* H */
  int32_t vocab;    /* V */
  int32_t dtype;    /* sbd_dtype of hidden and w */
} sbd_head_desc;

size_t sbd_head_entropy_sample_workspace_size(const sbd_head_desc* desc);

sbd_status sbd_head_entropy_sample(const sbd_head_desc* desc, const void* hidden,
                                   const void* w, const uint8_t* masked,
                                   const float* gumbel, float tau, float* entropy,
                                   int32_t* token, void* workspace,
                                   size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * sbd_head_entropy_sample plus the confidence of every masked position, for
 * the confidence-ordered selection rules of the Appendix "Sampling
 * algorithm" (Factor decoding; EB-Sampler with the confidence proxy):
 *   confidence = max_v p_v,  p = softmax(z) at temperature 1,
 * computed from the same merged statistics as the entropy (1 / sum_v
 * exp(z_v - max z)).  Unmasked positions get confidence = 0.
 *   confidence [B, k] fp32 out; every other argument, the workspace (size
 *   from sbd_head_entropy_sample_workspace_size) and the errors are those of
 *   sbd_head_entropy_sample.
 * ---------------------------------------------------------------------- */
sbd_status sbd_head_entropy_confidence_sample(const sbd_head_desc* desc, const void* hidden,
                                              const void* w, const uint8_t* masked,
                                              const float* gumbel, float tau, float* entropy,
                                              float* confidence, int32_t* token,
                                              void* workspace, size_t workspace_bytes,
                                              void* stream);

/* ------------------------------------------------------------------------
 * sbd_head_entropy_sample with counter-based Gumbel noise generated inside
 * the kernel instead of read from a [B, k, V] buffer (the buffer read is
 * 4 R V bytes per call).  The noise of block position n = b * k + i and
 * vocabulary id v is
 *   x = word (v mod 4) of Philox4x32-10(counter = (v div 4, n, offset_lo,
 *       offset_hi), key = (seed_lo, seed_hi))
 *       (Salmon, Moraes, Dror, Shaw, SC 2011; 10 rounds),
 *   u = ((x >> 9) + 1/2) * 2^-23   (exact in fp32, strictly inside (0, 1)),
 *   g = -ln(-ln u)                 (fp32, full-precision logarithms),
 * and token = argmax_v (z_v + tau * g).  A new offset (or seed) per step
 * gives fresh noise.  Every other argument, the workspace and the errors are
 * those of sbd_head_entropy_sample; tau = 0 is greedy.
 * ---------------------------------------------------------------------- */
sbd_status sbd_head_entropy_sample_philox(const sbd_head_desc* desc, const void* hidden,
                                          const void* w, const uint8_t* masked, uint64_t seed,
                                          uint64_t offset, float tau, float* entropy,
                                          int32_t* token, void* workspace,
                                          size_t workspace_bytes, void* stream);

/* The same noise written out: out[r, v] = g(row_ids[r], v) for 0 <= v < vocab.
 *   row_ids [n_rows] int32 (device): block positions n = b * k + i
 *   out [n_rows, vocab] fp32 (device)
 * Supported: n_rows <= 65535. */
sbd_status sbd_gumbel_philox(int32_t n_rows, const int32_t* row_ids, int32_t vocab,
                             uint64_t seed, uint64_t offset, float* out, void* stream);

/* ------------------------------------------------------------------------
 * A plain linear layer on the LM-head kernel: y = x W^T, the GEMMs of a
 * transformer layer at decode shapes (few rows, weights streamed once).
 * Used to time full forwards of a model around the block step (the
 * paper's timing section models the linear layers as GEMMs); it is not
 * part of the block step itself.
 *
 *   x [rows, in_features]           bf16, row-major (device)
 *   w [out_features, in_features]   bf16, row-major, nn.Linear layout (device)
 *   y [rows, out_features]          bf16, row-major (device, written)
 *   workspace                       sbd_linear_workspace_size(desc) bytes
 *                                   (device, 16-byte aligned; may be NULL
 *                                   when the size is 0)
 *
 * y is the fp32 sum over in_features of the bf16 products, rounded to
 * bf16 (round to nearest even).  When a layer has too few output tiles to
 * fill the GPU, the in_features are cut into ranges whose fp32 partials go
 * through the workspace and are summed by a second kernel (the split is
 * chosen per call from the shape).  Above 160 rows the product runs on
 * pairs of SMs (2-SM tensor-core MMAs).  All pointers 16-byte aligned,
 * caller-owned.  Asynchronous on `stream`.
 * Supported: dtype bf16, 0 <= rows <= 512, in_features a positive multiple
 * of 64, out_features >= 1; SBD_ERR_UNSUPPORTED otherwise; a workspace
 * smaller than needed gives SBD_ERR_WORKSPACE.
 * ---------------------------------------------------------------------- */
typedef struct {
  int32_t rows, in_features, out_features;
  sbd_dtype dtype;
} sbd_linear_desc;

/* Bytes for the largest split the call may choose: a function of the
 * shape only, the same on every device (0 when no split is possible); 0
 * for an invalid descriptor. */
size_t sbd_linear_workspace_size(const sbd_linear_desc* desc);
sbd_status sbd_linear(const sbd_linear_desc* desc, const void* x, const void* w, void* y,
                      void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * No-allocation variant of sbd_head_entropy_sample.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory -- a host framework that owns the whole device memory pool,
 * a latency-critical loop that cannot afford the device synchronisation of
 * cudaMalloc/cudaFree, or a plug-in with no allocator to borrow a workspace
 * from.  Same arguments, semantics and results as sbd_head_entropy_sample,
 * minus the workspace: the scratch is a fixed array inside the library, of
 * SBD_HEAD_NOALLOC_MAX_SCRATCH bytes, which every GPU that loads the library
 * holds until the process exits.
 *   - Shapes whose scratch (sbd_head_entropy_sample_workspace_size) exceeds
 *     that size are rejected with SBD_ERR_UNSUPPORTED before any launch.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current); make that first
 *     call before any stream capture on that device.
 *   - All calls on a device share the one array, which keeps the last
 *     call's contents (nothing in it needs to start at zero).  Calls whose
 *     kernels overlap on the GPU -- on different streams, or from several
 *     host threads -- race on it: serialise them (one stream, or events).
 *   - Allocates nothing: no cudaMalloc/cudaFree or allocating library call.
 * ---------------------------------------------------------------------- */
#define SBD_HEAD_NOALLOC_MAX_SCRATCH (8u << 20) /* 8 MiB */

sbd_status sbd_head_entropy_sample_noalloc(const sbd_head_desc* desc, const void* hidden,
                                           const void* w, const uint8_t* masked,
                                           const float* gumbel, float tau, float* entropy,
                                           int32_t* token, void* stream);

/* ------------------------------------------------------------------------
 * Entropy-bounded select, entropy proxy (Eq. 3; Algorithm 3 "unmask").  Per
 * sequence b: sort the masked positions by (entropy, position) ascending,
 * i_1, i_2, ...; accept the first s >= 1 positions, s the largest value with
 *   H_{i_1} + ... + H_{i_{s-1}} <= gamma     (fp32 prefix sums)
 * capped at the number of masked positions; for each accepted i write
 * block_tokens[b, i] = token[b, i] and masked[b, i] = 0, and set
 * n_unmasked[b] = s (0 when nothing is masked).  Entropies of masked
 * positions must be >= 0 (as produced by sbd_head_entropy_sample); a NaN
 * sorts last.  Entropies/tokens of unmasked positions are not read.
 *
 *   entropy [B, k] fp32, token [B, k] int32   inputs
 *   masked [B, k] uint8, block_tokens [B, k] int32 (-1 = mask)   in/out
 *   n_unmasked [B] int32 out (may be NULL)
 * Supported: 1 <= k <= 32, gamma >= 0 and finite.
 * ---------------------------------------------------------------------- */
sbd_status sbd_eb_select(int32_t batch, int32_t block_k, const float* entropy,
                         const int32_t* token, float gamma, uint8_t* masked,
                         int32_t* block_tokens, int32_t* n_unmasked, void* stream);

/* ------------------------------------------------------------------------
 * One unmasking step under a selectable rule (Algorithm 3 "unmask"; the
 * rules of Eq. 3 and of the Appendix "Sampling algorithm").  Per sequence b
 * the masked positions are ordered by the rule's key (ties to the lower
 * position), the first s accepted, their tokens committed and their flags
 * cleared, exactly as in sbd_eb_select:
 *   SBD_SELECT_EB_ENTROPY          entropy ascending; s of Eq. 3 with
 *                                  threshold = gamma.  Identical to
 *                                  sbd_eb_select (confidence not read).
 *   SBD_SELECT_EB_CONFIDENCE       confidence descending; s >= 1 the largest
 *                                  count with  sum_{j<=s} H_{i_j} -
 *                                  max_{j'<=s} H_{i_j'} <= gamma  (the
 *                                  general EB bound), capped at |M|.
 *   SBD_SELECT_FACTOR              confidence descending, c^1 >= c^2 >= ...;
 *                                  s the largest n in 1..|M| with
 *                                  (n + 1) c^n < f  (threshold = f), s = 1
 *                                  when no n qualifies.
 *   SBD_SELECT_FACTOR_COMPLEMENT   as FACTOR with (n + 1)(1 - c^n) < f.
 * Sums, maxima and products in fp32.  A NaN key sorts last.
 *
 *   entropy [B, k] fp32, confidence [B, k] fp32 (may be NULL for
 *   SBD_SELECT_EB_ENTROPY), token [B, k] int32   inputs
 *   masked [B, k] uint8, block_tokens [B, k] int32 (-1 = mask)   in/out
 *   n_unmasked [B] int32 out (may be NULL)
 * Supported: 1 <= k <= 32; threshold finite and >= 0.  An unknown rule is
 * SBD_ERR_INVALID_ARG.
 * ---------------------------------------------------------------------- */
typedef enum {
  SBD_SELECT_EB_ENTROPY = 0,
  SBD_SELECT_EB_CONFIDENCE = 1,
  SBD_SELECT_FACTOR = 2,
  SBD_SELECT_FACTOR_COMPLEMENT = 3
} sbd_select_rule;

sbd_status sbd_select(int32_t rule, int32_t batch, int32_t block_k, const float* entropy,
                      const float* confidence, const int32_t* token, float threshold,
                      uint8_t* masked, int32_t* block_tokens, int32_t* n_unmasked,
                      void* stream);

/* Status name ("SBD_OK", ...). Never NULL. */
const char* sbd_status_string(sbd_status status);

/* Detail of the last failing call on this thread ("" if none). */
const char* sbd_last_error(void);

/* Reads and clears the device error word of the current device
 * (synchronises the device).  *code = 0 when no kernel recorded a fault;
 * otherwise a bit set of SBD_DEVERR_* values. */
sbd_status sbd_device_error(int32_t* code);

#define SBD_DEVERR_CACHE_LEN 1   /* a cache_len entry was outside [0, Lmax] */
#define SBD_DEVERR_TIMEOUT 2     /* a bounded wait inside a kernel gave up  */
#define SBD_DEVERR_ROWS 4        /* more masked rows than the head supports */

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t sbd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SBD_H */
