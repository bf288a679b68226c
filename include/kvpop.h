/*
 * kvpop.h -- C ABI of the KVpop decode hot path on one GB300 (sm_103a).
 *
 * KVpop ("KV cache compression with predictive online pruning") keeps, per KV
 * head, the first s tokens (sinks), the last w tokens, which are never
 * evicted, and a long-range top-k set chosen by a learned scorer (Sec. 3,
 * Eq. 1).  Per decode step this library
 *   1. ingests the new token's q/k/v into the window,
 *   2. scores the token u = p - w that has just left the window with the
 *      delayed scorer (Sec. 3.3, App. E.4): a two-layer MLP on
 *      [k_u; v_u; mean of the next w queries of the KV head's query group],
 *   3. keeps or drops u under the fixed budget (Sec. 3.2 running top-k,
 *      App. C.1): a free slot while one exists, else it replaces the slot of
 *      lowest static priority (App. B.3; ties -> lowest slot index) iff its
 *      priority is strictly larger,
 *   4. scatters u's K/V into that slot, and
 *   5. runs GQA decode attention over the compact cache only -- the kept slots
 *      plus the window (App. C, first paragraph).
 *
 * Notation: b = batch, H = KV heads, G = query heads per KV head, d = head
 * dim, D = window (the paper's w), B = slots (sinks + long-range top-k; the
 * paper's s + k), F = scorer hidden width.  Query head index = h * G + g.
 *
 * Conventions for every call:
 *  - Pointers named *_dev are device pointers; *_host are host pointers.
 *    q/k/v/Q/K/V/out device pointers must be 16-byte aligned and the small
 *    per-(sequence, head) arrays (score overrides, evict_info, score_out)
 *    4-byte aligned, else KVPOP_ERR_ALIGN.
 *  - Calls are asynchronous on `stream` unless stated; the caller owns every
 *    input/output buffer, the library owns the cache.
 *  - No call aborts or throws; each returns a status.  After a CUDA error the
 *    cache is poisoned and later calls return KVPOP_ERR_STATE.
 *  - One cache per attention layer.  Calls on one cache must be serialised
 *    (one stream, or stream-ordered) -- they share its workspace.
 */
#ifndef KVPOP_H
#define KVPOP_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  KVPOP_OK = 0,
  KVPOP_ERR_INVALID_ARG = 1,   /* a size or pointer argument is out of range  */
  KVPOP_ERR_ALIGN = 2,         /* a device pointer is not 16-byte aligned     */
  KVPOP_ERR_OOM = 3,           /* device allocation failed                    */
  KVPOP_ERR_CUDA = 4,          /* a CUDA runtime call failed                  */
  KVPOP_ERR_STATE = 5,         /* cache poisoned by an earlier error, or freed */
  KVPOP_ERR_DEVICE_CHECK = 6   /* a kernel reported a failed check / timeout  */
} kvpop_status;

typedef enum { KVPOP_F32 = 0, KVPOP_BF16 = 1 } kvpop_dtype;

typedef struct {
  int32_t batch;          /* b >= 1                                            */
  int32_t n_kv_heads;     /* H >= 1                                            */
  int32_t q_per_kv;       /* G in {1, 2, 4}                                    */
  int32_t head_dim;       /* d in {64, 128}                                    */
  int32_t budget_B;       /* B >= 1: sink + long-range slots (Eq. 1: s + k)    */
  int32_t delay_D;        /* D >= 1: protected window w (Eq. 4); scoring delay */
  int32_t n_sink;         /* s, 0 <= s < B: first s tokens are never evicted   */
  int32_t scorer_hidden;  /* F in [1, 1024]; scorer input width is 3 * d       */
  kvpop_dtype kv_dtype;   /* element type of q, k, v and the K/V store         */
} kvpop_config;

/* Stateless scorer parameters (Sec. 3.3, App. E.2): the per-head two-layer MLP
 *   r = w2 . act(W1^T x + b1) + b2
 * on x = [k (d); v (d); qbar (d)] (input_kind 0; qbar = mean of the next D
 * queries over the G heads) or x = [k; v] (input_kind 1, the plain SiLU-MLP
 * scorer of Sec. 3.3), with act = GELU(erf) (activation 0), SiLU (1) or the
 * identity (2, a linear scorer when F = 1 and w2 = 1).  Host or device fp32
 * arrays; copied into the cache at init (caller keeps ownership).  A zeroed
 * struct with the five pointers set is the GELU [k; v; qbar] scorer. */
typedef struct {
  const float* W1;         /* [H][3d][F], or [H][2d][F] with input_kind 1     */
  const float* b1;         /* [H][F]                                          */
  const float* w2;         /* [H][F]                                          */
  const float* b2;         /* [H]                                             */
  const float* log_gamma;  /* [H] per-head log decay (App. B.3, n = 1) or NULL
                              for none; stored priority = r - u * log_gamma   */
  int32_t input_kind;      /* 0: [k; v; qbar]   1: [k; v]                     */
  int32_t activation;      /* 0: GELU (erf)   1: SiLU   2: identity           */
} kvpop_scorer;

/* Stateful delayed mLSTM scorer (App. A, App. E.3, App. E.4), per KV head.
 * With x = [k; v]: q~ = phi(W_q x), k~ = phi(W_k x), v~ = W_v x, phi the
 * Hedgehog map [softmax(y); softmax(-y)]; gates i = exp(w_i.x + b_i),
 * f = sigmoid(w_f.x + b_f); state C <- f C + i k~ v~^T, z <- f z + i k~ (kept
 * stabilised); after absorbing token p the token u = p - D is scored
 * r = a . SiLU((q~_u^T C) / (q~_u^T z)) + b.  Host or device fp32 arrays,
 * copied at init. */
typedef struct {
  const float* Wq;         /* [H][2d][d/2]                                    */
  const float* Wk;         /* [H][2d][d/2]                                    */
  const float* Wv;         /* [H][2d][d/2]                                    */
  const float* wi;         /* [H][2d] input-gate weights                      */
  const float* wf;         /* [H][2d] forget-gate weights                     */
  const float* bi;         /* [H]                                             */
  const float* bf;         /* [H]                                             */
  const float* a;          /* [H][d/2] output projection                      */
  const float* b;          /* [H]                                             */
  const float* log_gamma;  /* [H] per-head log decay or NULL (as kvpop_scorer) */
} kvpop_mlstm_scorer;

typedef struct kvpop_cache kvpop_cache;   /* opaque, library-owned device state */

/* Human-readable name of a status (static string, never NULL). */
const char* kvpop_status_string(kvpop_status s);

/* Create an empty cache (length 0 for every sequence) on the current device:
 * the per-KV-head state the method keeps under its fixed budget (Sec. 3,
 * Eq. 1: s sink + k long-range slots, here B = s + k, and the window of w = D
 * tokens held apart) plus the stateless scorer of Sec. 3.3.  Allocates the slot store [b][H][B][d] for K and V, the window rings
 * [b][H][D][d], per-slot score/position arrays and the attention workspace.
 * Synchronises `stream` before returning.  *out is NULL on failure. */
kvpop_status kvpop_init_cache(const kvpop_config* cfg, const kvpop_scorer* scorer,
                              cudaStream_t stream, kvpop_cache** out);

/* As kvpop_init_cache with the mLSTM scorer; cfg->scorer_hidden is ignored.
 * The cache additionally holds the recurrent state (C, z, m) of every
 * (sequence, KV head), which prefill builds over the prompt and every decode
 * step advances by one token (in prefill, the chunkwise form of the recurrence:
 * 64-token chunks one after another per pair, the tokens of a chunk together). */
kvpop_status kvpop_init_cache_mlstm(const kvpop_config* cfg, const kvpop_mlstm_scorer* scorer,
                                    cudaStream_t stream, kvpop_cache** out);

/* Release the cache and all its device memory (resource management; the paper
 * has no counterpart).  kvpop_free(NULL) is KVPOP_OK.
 * Synchronises the device work of the cache first. */
kvpop_status kvpop_free(kvpop_cache* cache);

/* Prompt compression (the prefill of the running top-k, Sec. 3.2 / App. C.1).
 * For sequences first_seq .. first_seq + n_seq - 1, whose prompt lengths are
 * prompt_len_host[0 .. n_seq-1] (0 <= P <= Pmax), score every token
 * u <= P - 1 - D with the delayed scorer, keep the s sinks plus the top (B - s)
 * of the rest by (priority desc, position asc), store them in ascending
 * position order, and fill the window with the last min(P, D) tokens.
 * Replaces any state those sequences had.
 *   Q_dev  [n_seq][H*G][Pmax][d]    K_dev, V_dev [n_seq][H][Pmax][d]
 *   score_override_dev  [n_seq][H][Pmax] fp32 raw scores used instead of the
 *                        scorer (entry u), or NULL
 * Uses a stream-ordered temporary of n_seq*H*Pmax*4 bytes and synchronises
 * `stream` before returning (the host length array may be reused at once).
 * The lengths are host values and the batch may come in chunks of sequences
 * because a whole batch's prompts need not fit in device memory at once (128
 * ragged prompts of up to 65536 tokens are about 35 GB of bf16 Q/K/V); the
 * temporary is sized from the chunk, and the call returns only once the host
 * length array is no longer read. */
kvpop_status kvpop_prefill_compress(kvpop_cache* cache, const void* Q_dev, const void* K_dev,
                                    const void* V_dev, const int32_t* prompt_len_host,
                                    int32_t first_seq, int32_t n_seq, int32_t Pmax,
                                    const float* score_override_dev, cudaStream_t stream);

/* Prompt compression with outputs (App. C.1 mask, App. C.3): everything
 * kvpop_prefill_compress does, plus the attention output of every prompt query
 * under the running top-k mask
 *   M[q,t] = t < s  or  q - t < D  or  (s <= t <= q - D and rank(t) <= tau_q)
 * (causal, t <= q), where rank orders the prompt tokens by static priority
 * (higher first, earlier position on ties; the last D tokens, which have no
 * score yet, rank last) and tau_q is the rank of the min(B - s, |E(q)|)-th best
 * token of E(q) = {s <= t <= q - D} (-1 while E(q) is empty).  At q = P - 1 the
 * retained set is exactly the cache prompt compression leaves.
 *   Y_dev    [n_seq][H*G][Pmax][d] fp32 out   (rows q >= P untouched)
 *   lse_dev  [n_seq][H*G][Pmax] fp32 out, natural log of the softmax
 *            normaliser over the retained keys (the sparse LSE of App. D.3),
 *            or NULL
 *   rank_dev, tau_dev [n_seq][H][Pmax] int32 out (-1 past P), or NULL
 *   order_dev [n_seq][H][Pmax] int32 out, position of each rank (entries from P on
 *            untouched), or NULL; with rank_dev and tau_dev it is what
 *            kvpop_prompt_attention takes to recompute the outputs
 * Other arguments as kvpop_prefill_compress.  Needs Pmax <= 262144,
 * n_seq*H <= 65535, d in {64, 128}, G in {1, 2, 4} and per-tile key lists of
 * 4*(B + s + 2*128 + D) bytes that fit in shared memory (else
 * KVPOP_ERR_INVALID_ARG).  bf16 runs on tensor cores, fp32 on CUDA cores.
 * Temporaries: 24 bytes per (sequence, head, token) on top of the compression's. */
kvpop_status kvpop_prefill_attend(kvpop_cache* cache, const void* Q_dev, const void* K_dev,
                                  const void* V_dev, const int32_t* prompt_len_host,
                                  int32_t first_seq, int32_t n_seq, int32_t Pmax,
                                  const float* score_override_dev, float* Y_dev, float* lse_dev,
                                  int32_t* rank_dev, int32_t* tau_dev, int32_t* order_dev,
                                  cudaStream_t stream);

/* Bytes of device workspace kvpop_topk_cutoff needs (0 for an empty problem). */
size_t kvpop_topk_workspace_bytes(int32_t n_rows, int32_t S);

/* Running top-k cutoffs of n_rows independent rows (App. C.1 ranks, App. C.2 /
 * Algorithm 2 cutoffs), no cache involved.  Row r holds lengths_dev[r] tokens
 * (S for every row if lengths_dev is NULL) with fp32 static priorities
 * prio_dev[r][t] (NaN counts as -inf, -0 as +0).  Outputs:
 *   rank_dev [n_rows][S]  rank of token t: 0 = highest priority, equal
 *                         priorities by position; -1 past the row length
 *   tau_dev  [n_rows][S]  rank of the min(k, |E(q)|)-th best token of
 *                         E(q) = {n_sink <= t <= q - window}; -1 while E(q) is
 *                         empty and past the row length
 *   order_dev [n_rows][S] (or NULL) position of each rank: order[r][rank[r][t]] = t
 *                         for t below the row length (entries past it untouched)
 * Where Algorithm 2 leaves tau_q = -1 while fewer than k tokens are eligible,
 * this keeps all of them (the top k of a set smaller than k is the set).
 * workspace_dev: kvpop_topk_workspace_bytes(n_rows, S) bytes, 256-byte aligned,
 * owned by the caller.  S <= 262144, window >= 1, k >= 1.  Asynchronous on
 * `stream`; no allocation. */
kvpop_status kvpop_topk_cutoff(const float* prio_dev, const int32_t* lengths_dev, int32_t n_rows,
                               int32_t S, int32_t n_sink, int32_t window, int32_t k,
                               int32_t* rank_dev, int32_t* tau_dev, int32_t* order_dev,
                               void* workspace_dev, size_t workspace_bytes, cudaStream_t stream);

/* Masked causal attention over prompts under the running top-k mask given by
 * rank / tau from kvpop_topk_cutoff (same n_sink, window and k), no cache
 * involved.  Per KV head h and query head g = 0..G-1:
 *   y[q] = sum_t softmax_t(M[q,t] ? q.k_t / sqrt(d) : -inf) v_t
 *   Q_dev [n_seq][H*G][S][d], K_dev, V_dev [n_seq][H][S][d]  (dtype)
 *   rank_dev, tau_dev [n_seq][H][S] int32;  lengths_dev [n_seq] or NULL (= S)
 *   order_dev [n_seq][H][S] int32, the order output of the same kvpop_topk_cutoff
 *   call, or NULL: with it a tile's key lists are built from the ranks up to its
 *   largest cutoff when that is shorter than its eligible positions (same outputs)
 *   Y_dev [n_seq][H*G][S][d] fp32 out; lse_dev [n_seq][H*G][S] fp32 out or NULL
 * Limits as kvpop_prefill_attend.  Asynchronous on `stream`; no allocation.
 * rank / tau that did not come from kvpop_topk_cutoff give unspecified outputs
 * but never an out-of-bounds access. */
kvpop_status kvpop_prompt_attention(const void* Q_dev, const void* K_dev, const void* V_dev,
                                    const int32_t* rank_dev, const int32_t* tau_dev,
                                    const int32_t* order_dev, const int32_t* lengths_dev,
                                    int32_t n_seq, int32_t n_kv_heads,
                                    int32_t q_per_kv, int32_t head_dim, int32_t S, int32_t n_sink,
                                    int32_t window, int32_t k, kvpop_dtype dtype, float* Y_dev,
                                    float* lse_dev, cudaStream_t stream);

/* First device-side error (a bounded wait that expired) recorded by the
 * cache-free calls kvpop_prompt_attention, kvpop_causal_lse,
 * kvpop_future_target and kvpop_attend_noalloc since the last call of this
 * function: KVPOP_OK, or
 * KVPOP_ERR_DEVICE_CHECK (details in kvpop_last_error).  Synchronises `stream`
 * and clears the record. */
kvpop_status kvpop_standalone_status(cudaStream_t stream);

/* Dense causal log-normalisers (App. D.1), the exact-target variant of the
 * normaliser fed to kvpop_future_target:
 *   lse[q] = log sum_{t <= q} exp(q.k_t / sqrt(d))   per query head, natural log
 *   Q_dev [n_seq][H*G][S][d], K_dev [n_seq][H][S][d] (dtype); lengths_dev [n_seq]
 *   or NULL (= S); lse_dev [n_seq][H*G][S] fp32 out (rows past a length untouched)
 * d in {64, 128}, G in {1, 2, 4}, n_seq*H <= 65535.  Asynchronous; no allocation. */
kvpop_status kvpop_causal_lse(const void* Q_dev, const void* K_dev, const int32_t* lengths_dev,
                              int32_t n_seq, int32_t n_kv_heads, int32_t q_per_kv,
                              int32_t head_dim, int32_t S, kvpop_dtype dtype, float* lse_dev,
                              cudaStream_t stream);

/* Future-attention target for training the scorer (Sec. 3.4, App. D, App. F).
 * Transposed attention pass (App. D.2), for every key t and query head g:
 *   logm[g][t] = log sum_{d = t+w}^{hi} exp(q_d.k_t / sqrt(d) - lse_dev[g][d])
 * with hi = S_b - 1, or min(S_b - 1, t + w + lookahead) when lookahead > 0
 * (-inf when the range is empty).  lse_dev is the dense normaliser of
 * kvpop_causal_lse (exact target) or the sparse one of kvpop_prompt_attention /
 * kvpop_prefill_attend (approximate target, App. D.3).  If target_dev is not
 * NULL it also receives, per KV head (Eq. 2, App. F.1-F.2),
 *   target[t] = log(eps + Agg_g exp(logm[g][t]) / N_t),
 *   Agg = max (agg 0) or mean (agg 1), N_t = max(1, S_b - (t + w)) clipped to
 *   lookahead + 1 when lookahead > 0, N_t = 1 when count_norm is 0.
 *   Q_dev [n_seq][H*G][S][d], K_dev [n_seq][H][S][d]; lse_dev, logm_dev
 *   [n_seq][H*G][S] fp32; target_dev [n_seq][H][S] fp32; lengths_dev [n_seq] or
 *   NULL (S_b = S).  window >= 0, lookahead >= 0, eps >= 0 finite.
 * Asynchronous on `stream`; no allocation. */
kvpop_status kvpop_future_target(const void* Q_dev, const void* K_dev, const float* lse_dev,
                                 const int32_t* lengths_dev, int32_t n_seq, int32_t n_kv_heads,
                                 int32_t q_per_kv, int32_t head_dim, int32_t S, int32_t window,
                                 int32_t lookahead, kvpop_dtype dtype, float* logm_dev,
                                 float* target_dev, int32_t agg, int32_t count_norm, float eps,
                                 cudaStream_t stream);

/* Decode steps 1-4 for every sequence: ingest the token at position p = len,
 * score u = p - D (if p >= D; the token that has just become eligible, Sec. 3.1
 * Eq. 4) with the delayed scorer (Sec. 3.3, App. E.4), keep or drop it under the
 * budget (Sec. 3.2 running top-k, App. C.1 mask, App. B.3 static priority),
 * scatter it, push p.
 *   q_dev [b][H*G][d], k_dev / v_dev [b][H][d]
 *   score_override_dev [b][H] fp32 raw scores used instead of the scorer, or NULL
 *   evict_info_dev [b][H][2] int32 out: (slot u went to or -1, evicted position
 *                  or -1), or NULL
 *   score_out_dev  [b][H] fp32 out: raw score of u (NaN when no token left the
 *                  window), or NULL */
kvpop_status kvpop_decode_ingest(kvpop_cache* cache, const void* q_dev, const void* k_dev,
                                 const void* v_dev, const float* score_override_dev,
                                 int32_t* evict_info_dev, float* score_out_dev,
                                 cudaStream_t stream);

/* Decode step 5 (App. C, first paragraph: decode attends over the compact cache
 * only): out_g = softmax(q_g K_S^T / sqrt(d)) V_S for every query head, where
 * S = kept slots plus window entries of its KV head.  Split-K over a
 * persistent grid with token-balanced ranges.
 *   q_dev [b][H*G][d] (same as ingest)   out_dev [b][H*G][d] fp32 */
kvpop_status kvpop_decode_attend(kvpop_cache* cache, const void* q_dev, float* out_dev,
                                 cudaStream_t stream);

/* One whole decode step (Sec. 3.1-3.3, App. C): the effect of kvpop_decode_ingest
 * followed by kvpop_decode_attend, with the same arguments and outputs.  For bf16
 * caches with d = 128, a scorer hidden width F <= 256, up to about 2000 (sequence,
 * KV head) pairs, and a K/V stream of at least 600 MB per step at full budget
 * (pairs x (B + D) x 2 d x 2 bytes; below that the scorer would outlast the
 * attention) it runs as one kernel: the attention streams every key that cannot change in this
 * step while the scorer, keep-or-drop and scatter run beside it, and the one slot and
 * the one window row that may change are added when each (sequence, KV head) is
 * merged (kvpop_step_is_fused reports 1).  The attention output may then differ from
 * the two-call path by the order of its fp32 sums; evictions follow the same rule.
 * The environment variables KVPOP_SPLIT_STEP / KVPOP_FUSED_STEP, set before
 * kvpop_init_cache, choose the two-kernel / one-kernel path regardless of the stream
 * size (the shape and shared-memory conditions still apply).  Asynchronous on
 * `stream`. */
kvpop_status kvpop_decode_step(kvpop_cache* cache, const void* q_dev, const void* k_dev,
                               const void* v_dev, float* out_dev,
                               const float* score_override_dev, int32_t* evict_info_dev,
                               float* score_out_dev, cudaStream_t stream);

/* 1 when kvpop_decode_step of this cache runs as one kernel, 0 when it runs the
 * ingest and the attention as two, -1 for an invalid handle. */
int32_t kvpop_step_is_fused(const kvpop_cache* cache);

/* kvpop_decode_step on host buffers (pinned memory recommended), all on `stream`
 * (the caller synchronises before reading out_host or reusing the inputs).  When
 * q_host, k_host and v_host are all pinned memory the device can address (on
 * Grace-Blackwell over NVLink-C2C), the step's kernels read them in place;
 * otherwise they are copied into library-owned device staging first (one copy when
 * k_host and v_host follow q_host directly in one buffer).  Likewise the attention
 * writes a device-addressable pinned out_host directly, and anything else is copied
 * back from device staging. */
kvpop_status kvpop_decode_step_host(kvpop_cache* cache, const void* q_host, const void* k_host,
                                    const void* v_host, float* out_host, cudaStream_t stream);

/* Synchronise `stream` and report any device-side check failure
 * (KVPOP_ERR_DEVICE_CHECK) or CUDA error recorded since the last call. */
kvpop_status kvpop_check(kvpop_cache* cache, cudaStream_t stream);

/* Checkpoint / resume.  kvpop_export_state with host_buf == NULL sets *bytes to
 * the size needed; otherwise it copies the full cache state (including lengths)
 * into host_buf (*bytes >= size) and synchronises.  kvpop_import_state restores
 * a blob exported from a cache with an identical config. */
kvpop_status kvpop_export_state(kvpop_cache* cache, void* host_buf, size_t* bytes,
                                cudaStream_t stream);
kvpop_status kvpop_import_state(kvpop_cache* cache, const void* host_buf, size_t bytes,
                                cudaStream_t stream);

/* Per-sequence lengths (tokens seen so far) copied to host; synchronises. */
kvpop_status kvpop_get_lengths(kvpop_cache* cache, int32_t* len_host, cudaStream_t stream);

/* Diagnostic read of one (sequence, KV head): the positions held by its B
 * slots (pos_host[B], -1 = free) and their stored priorities (score_host[B];
 * either may be NULL), and its number of used slots.  Synchronises. */
kvpop_status kvpop_get_pair_state(kvpop_cache* cache, int32_t seq, int32_t head,
                                  int32_t* pos_host, float* score_host, int32_t* nvalid_host,
                                  cudaStream_t stream);

/* Allocation-free decode attention (no counterpart in the paper: it is an
 * interface convenience).  For callers that may not allocate device memory
 * when they decode -- a serving loop whose device memory is fixed up front and
 * must not grow or stall mid-generation, or a plugin that may only use buffers
 * its host framework hands it.  Computes the same output as
 * kvpop_decode_attend (the CUDA-core kernel, for either dtype) over K/V state
 * the caller owns, and takes the kernel's split-K scratch from a fixed 2 MiB
 * array compiled into the library instead of calling cudaMalloc; nothing it
 * calls allocates.
 *   slotK/slotV [b][H][B][d], ringK/ringV [b][H][D][d] (window entry of
 *   position t at index t % D), nvalid/len [b][H] int32 (used slots, tokens
 *   seen), q [b][H*G][d], out [b][H*G][d] fp32 -- all device pointers.
 * Returns KVPOP_ERR_INVALID_ARG (and a kvpop_last_error message) when
 * b * H > 12288 or the scratch would exceed the array.  The first call on each
 * device does a one-time set-up (the array's device address, kernel
 * attributes) with that device current; make that first call before any
 * stream capture.  Every call on a device shares the one array and the array
 * keeps the last call's contents, so calls that overlap on the GPU race:
 * serialise them.  A bounded wait in the kernel that gives up leaves `out`
 * incomplete and is reported by the next kvpop_standalone_status (which
 * synchronises `stream` and allocates nothing); callers that need to know
 * call it after the attention.  The kernel's shared-memory limit is set to the
 * device maximum by every path of the library, so caches created on other
 * threads never lower it under this call. */
kvpop_status kvpop_attend_noalloc(const void* slotK_dev, const void* slotV_dev,
                                  const void* ringK_dev, const void* ringV_dev,
                                  const int32_t* nvalid_dev, const int32_t* len_dev,
                                  const void* q_dev, float* out_dev, int32_t batch,
                                  int32_t n_kv_heads, int32_t q_per_kv, int32_t head_dim,
                                  int32_t budget_B, int32_t delay_D, kvpop_dtype kv_dtype,
                                  cudaStream_t stream);

/* Description of the last failing CUDA call made by this library on the
 * calling thread ("" if none): call site, error name and message. */
const char* kvpop_last_error(void);

/* Testing hook: make the n-th device allocation from now fail (n >= 1), or
 * disable with n <= 0.  Affects only this library's allocations. */
void kvpop_debug_fail_alloc_after(int32_t n);

/* Testing hook for the failure path of the bounded device waits (no counterpart in
 * the paper): while `on` is non-zero, the copy-issuing thread of the bf16
 * tensor-core decode attention (kvpop_decode_attend, kvpop_decode_step) neither
 * arms a barrier nor issues a copy, so every consumer's first wait runs out after
 * the kernels' wait limit (2 s), records a timeout and skips the rest of its work;
 * `out` is then unspecified and the next kvpop_check returns
 * KVPOP_ERR_DEVICE_CHECK.  Nothing faults and no copy is in flight when the kernel
 * ends.  Affects launches made after the call; 0 (the default) turns it off. */
void kvpop_debug_skip_attention_copies(int32_t on);

#ifdef __cplusplus
}
#endif
#endif /* KVPOP_H */
