/*
 * kvr.h -- C ABI of libkvr: the evicted-KV decode step of KV-Rescue
 * (arXiv 2608.15797) on one GB300 (sm_103a).
 *
 * The operation (Sec. 2.1, Eq. 1): at decode step t each layer keeps, per KV
 * head, a budgeted cache C_t^B of key/value rows.  The step
 *   1. appends the new token's (k_t, v_t),
 *   2. computes Attn(q_t, C) for the G query heads that share the KV head
 *      (grouped-query attention; softmax scale 1/sqrt(d) by default),
 *   3. adds to every live row's importance score s_i ("accumulated attention",
 *      Sec. 2.1) the mean over the G query heads of that row's probability,
 *   4. once the live length exceeds B' = B + W (App. D: eviction then runs on
 *      every step), keeps the W most recent rows (the protected window of
 *      Sec. 4.1 / App. C) plus the B best-scored others (TopB of Eq. 1;
 *      equal scores keep the lower position) and compacts K/V in place.
 * Candidates (Sec. 2.2, Eq. 2; App. C, best-of-(N+N)) fork from one cache
 * state, decode a step each, and the chosen one becomes the persistent state
 * (Algorithm 1).
 *
 * Conventions for every call below:
 *  - A "unit" is one (sequence, layer, KV head).  Query head j of a layer
 *    uses KV head j / G.
 *  - Device pointers ("dev") are caller-owned CUDA device memory; host
 *    pointers ("host") are caller-owned host memory.  The library never
 *    allocates device memory: a handle owns only host metadata.
 *  - Tensors are dense row-major with the shapes given; element type is the
 *    descriptor's kv_dtype unless stated (out_dtype for outputs).
 *  - "stream" is a cudaStream_t (NULL = legacy default stream).  Calls are
 *    asynchronous and stream-ordered unless marked "synchronising".
 *  - Errors are returned as kvr_status, never thrown; kvr_last_error() gives
 *    a thread-local message for the last failing call.  Argument and capacity
 *    errors are detected on the host before anything is enqueued (the handle
 *    keeps a host mirror of every live length).  Errors found by a kernel
 *    (non-finite logits, an inconsistent length) set a device error word that
 *    kvr_sync_status() reports as KVR_EDEVICE.
 *  - Slot order inside a unit is not part of the contract: rows are
 *    identified by their position (token index).
 */
#ifndef KVR_H
#define KVR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  KVR_OK = 0,
  KVR_EINVAL = 1,    /* bad argument (null pointer, range, unsupported shape) */
  KVR_ENOMEM = 2,    /* caller-provided buffer smaller than required */
  KVR_ECAPACITY = 3, /* appended rows would exceed the unit capacity */
  KVR_ECUDA = 4,     /* a CUDA runtime call failed */
  KVR_EDEVICE = 5,   /* a kernel set the device error word */
  KVR_ESTATE = 6     /* call not valid in the handle's current state */
} kvr_status;

typedef enum { KVR_BF16 = 0, KVR_F32 = 1 } kvr_dtype;

typedef struct {
  int n_seq;           /* S, sequences in the batch (>= 1) */
  int n_layers;        /* L (>= 1) */
  int n_kv_heads;      /* H, KV heads per layer (>= 1) */
  int group;           /* G = query heads per KV head, 1..8 */
  int head_dim;        /* d: 64 or 128 */
  int capacity;        /* rows per unit slab (>= 1) */
  kvr_dtype kv_dtype;  /* K, V, q, k_new, v_new element type */
  kvr_dtype out_dtype; /* attention output element type */
  float softmax_scale; /* 0 selects 1/sqrt(d) */
} kvr_cache_desc;

typedef struct kvr_cache kvr_cache; /* opaque; host metadata only */
typedef struct kvr_fork kvr_fork;   /* opaque; host metadata only */

/* ---- cache lifetime ---------------------------------------------------- */

/* Bytes of device memory a cache with this descriptor needs (0 if the
 * descriptor is invalid).  The buffer holds, per unit, the K and V slabs
 * [capacity][d], the fp32 scores and int32 positions [capacity], the live
 * length and next position, a logit scratch area [G][capacity] fp32 used when
 * a unit is too long for on-chip memory, and a device error word. */
size_t kvr_cache_required_bytes(const kvr_cache_desc *desc);

/* Create a cache over dev_buf (>= kvr_cache_required_bytes, 256-byte
 * aligned; owned by the caller and must outlive the handle).  Every unit
 * starts empty at position 0.  The initialisation is enqueued on stream. */
kvr_status kvr_cache_create(const kvr_cache_desc *desc, void *dev_buf,
                            size_t bytes, void *stream, kvr_cache **out);

/* Free the handle's host metadata (not the device buffer). NULL is a no-op. */
void kvr_cache_destroy(kvr_cache *cache);

/* Load a prompt into sequence seq of every layer and KV head:
 * k, v dev [L][H][n_rows][d].  Rows get positions first_pos..first_pos+n-1
 * and score 0 (no prefill scoring: the first decode step supplies the first
 * scores).  Replaces whatever the sequence held.  n_rows <= capacity. */
kvr_status kvr_cache_load(kvr_cache *cache, int seq, const void *k,
                          const void *v, int n_rows, int first_pos,
                          void *stream);

/* ---- the decode step --------------------------------------------------- */

/* Steps 1-3 for layers [layer_begin, layer_end) of every sequence: append,
 * attend, accumulate scores; no eviction.  nl = layer_end - layer_begin.
 *   q     dev [S][nl][H*G][d]
 *   k_new dev [S][nl][H][d], v_new dev [S][nl][H][d]
 *   out   dev [S][nl][H*G][d] (out_dtype)
 * Needs one free row per unit (KVR_ECAPACITY otherwise). */
kvr_status kvr_decode_attend_score(kvr_cache *cache, int layer_begin,
                                   int layer_end, const void *q,
                                   const void *k_new, const void *v_new,
                                   void *out, void *stream);

/* Step 4 alone for layers [layer_begin, layer_end): every unit longer than
 * budget + window is cut back to budget + window rows (window = the W most
 * recent positions, always kept; TopB of the rest; ties keep the lower
 * position), compacting K, V, scores and positions in place.
 * budget >= 0, window >= 0, budget + window >= 1. */
kvr_status kvr_evict_compact(kvr_cache *cache, int layer_begin, int layer_end,
                             int budget, int window, void *stream);

/* Step 4 with the redundancy-aware score of R-KV, the eviction policy of
 * the paper's base model (App. C: cached tokens scored by a mix of
 * query-attention importance and key redundancy by cosine similarity, mix
 * weight lambda = 0.1, keeping the top B plus a recent window).  The paper
 * prints no formula; this library reads it, per unit with n live rows,
 * window rows W (the most recent) and candidates C (the rest), as
 *   r_i = mean over live j != i of cos(k_i, k_j)   (0 for a zero key)
 *   R_i = softmax over C of r,   I_i = s_i / sum over C of s   (0 if 0)
 *   z_i = lambda * I_i - (1 - lambda) * R_i
 * keeping the window and the B candidates first by (z descending, position
 * ascending).  s is the accumulated attention score the decode calls keep,
 * so a step with this policy is kvr_decode_attend_score followed by this
 * call.  lambda = 1 gives kvr_evict_compact's result.  Arguments as
 * kvr_evict_compact, plus 0 <= lambda <= 1 (KVR_EINVAL otherwise). */
kvr_status kvr_evict_compact_rkv(kvr_cache *cache, int layer_begin,
                                 int layer_end, int budget, int window,
                                 float lambda, void *stream);

/* Steps 1-4 fused in one pass: equivalent to kvr_decode_attend_score
 * followed by kvr_evict_compact, with the appended row written straight into
 * the slot the eviction frees. */
kvr_status kvr_decode_step(kvr_cache *cache, int layer_begin, int layer_end,
                           const void *q, const void *k_new, const void *v_new,
                           void *out, int budget, int window, void *stream);

/* Steps 1-4 with the R-KV eviction in one pass (App. C, lambda; App. D:
 * the eviction's key-similarity pass): equivalent to
 * kvr_decode_attend_score followed by kvr_evict_compact_rkv with the same
 * reading of R-KV.  Where every unit holds at most 160 rows after the
 * append and at most one is evicted (bf16, head_dim 128, G <= 8) it is one
 * launch: the redundancy of each row comes from the keys already staged
 * for attention, so no key is read twice; otherwise it runs the two calls.
 * Arguments as kvr_decode_step, plus 0 <= lambda <= 1 (KVR_EINVAL
 * otherwise). */
kvr_status kvr_decode_step_rkv(kvr_cache *cache, int layer_begin,
                               int layer_end, const void *q,
                               const void *k_new, const void *v_new, void *out,
                               int budget, int window, float lambda,
                               void *stream);

/* kvr_decode_step with the step's inputs and output in HOST memory, as a
 * serving loop feeds it (Sec. 2.1 Eq. 1, one decode step of every sequence).
 * Enqueued on stream, in order: the copies of q_host, k_new_host and
 * v_new_host (shapes and element types of kvr_decode_step's q, k_new,
 * v_new) into the caller's device staging buffers q_dev, k_new_dev,
 * v_new_dev; the step, which writes out_dev (kvr_decode_step's out); the
 * copy of out_dev into out_host.  The step waits for the handle's previous
 * kvr_decode_step_host step, on whatever stream that ran, so a caller may
 * alternate two streams, each with its own staging buffers, and have one
 * step's copies overlap the other's compute.  A staging set may be reused on
 * the stream that last used it (stream order covers it).  Host buffers are
 * caller-owned, must stay valid until the stream passes the copy out, and
 * should be page-locked (cudaHostAlloc / cudaHostRegister) for the copies
 * to be asynchronous.  Errors: as kvr_decode_step, KVR_EINVAL for a null
 * host or staging pointer, KVR_ECUDA when a copy or event call fails. */
kvr_status kvr_decode_step_host(kvr_cache *cache, int layer_begin,
                                int layer_end, const void *q_host,
                                const void *k_new_host, const void *v_new_host,
                                void *out_host, void *q_dev, void *k_new_dev,
                                void *v_new_dev, void *out_dev, int budget,
                                int window, void *stream);

/* ---- full-context decode (the helper's cache: no scores, no eviction) -- */

/* The full-context helper of KV-Rescue keeps its whole cache (Sec. 3.1;
 * App. D, Eq. 11): its decode step is Attn(q_t, C_t) of Eq. 1 over every
 * cached row, with no importance scores and no eviction.  This call appends
 * the new row (position = next position, score 0) and attends over all
 * rows, splitting each unit's rows over n_splits CTAs whose partial softmax
 * states are merged afterwards (two kernels).  The other units' scores are
 * not touched.  bf16 caches with head_dim 128 and G <= 8 only (KVR_EINVAL
 * otherwise).  Shapes as kvr_decode_attend_score.  n_splits = 0 lets the
 * library choose; workspace (device, caller-owned, 16-byte aligned) must
 * hold kvr_decode_attend_workspace_bytes(cache, layer_begin, layer_end,
 * n_splits) bytes (KVR_ENOMEM otherwise). */
size_t kvr_decode_attend_workspace_bytes(const kvr_cache *cache,
                                         int layer_begin, int layer_end,
                                         int n_splits);
kvr_status kvr_decode_attend(kvr_cache *cache, int layer_begin, int layer_end,
                             const void *q, const void *k_new,
                             const void *v_new, void *out, int n_splits,
                             void *workspace, size_t workspace_bytes,
                             void *stream);

/* ---- candidates: stepwise best-of-N over one shared cache state -------- */

/* Sec. 2.2 (Eq. 2) and App. C (best-of-(N+N)): each reasoning step draws
 * N candidates from the same committed (evicted) cache state; the selected
 * one becomes the persistent state (Algorithm 1).  The paper forks by
 * copying the live rows; here the candidates share the parent's live rows
 * read-only as a common prefix (the batched kernel reads every prefix row
 * once for all N x G query rows) and keep only what differs: a private copy
 * of the prefix scores and a private tail of appended rows.  Eviction is
 * deferred to the end of the step (kvr_fork_commit), which cuts the chosen
 * candidate to B + W exactly as kvr_evict_compact would cut a private copy
 * that had decoded the same rows without eviction. */

/* Device bytes a fork of `parent` into n_cand candidates with tail_cap rows
 * per unit needs (0 for invalid arguments): per candidate, the prefix score
 * copy [S][L][H][capacity], the tail K and V [S][L][H][tail_cap][d], tail
 * scores, positions and lengths. */
size_t kvr_fork_required_bytes(const kvr_cache *parent, int n_cand,
                               int tail_cap);

/* Fork the parent (all sequences) into n_cand >= 1 candidates over dev_buf
 * (caller-owned, >= kvr_fork_required_bytes, 256-byte aligned).  The parent
 * must not be modified by any other call while the fork is alive; its rows
 * are the candidates' shared prefix.  Copies the parent's scores into every
 * candidate (enqueued on stream). */
kvr_status kvr_fork_candidates(kvr_cache *parent, int n_cand, int tail_cap,
                               void *dev_buf, size_t bytes, void *stream,
                               kvr_fork **out);

/* One decode step of every candidate over layers [layer_begin, layer_end):
 * candidate c appends its row to its tail, attends over prefix + its tail,
 * and adds the mean over the G heads of each row's probability to its own
 * scores.  No eviction.
 *   q     dev [N][S][nl][H*G][d],  k_new, v_new dev [N][S][nl][H][d]
 *   out   dev [N][S][nl][H*G][d] (the parent's out_dtype)
 * KVR_ECAPACITY when a tail is full. */
kvr_status kvr_fork_decode_attend_score(kvr_fork *fork, int layer_begin,
                                        int layer_end, const void *q,
                                        const void *k_new, const void *v_new,
                                        void *out, void *stream);

/* Commit: for every sequence s, candidate chosen[s] (host array [S]) is cut
 * to budget + window rows (window = the W newest positions; TopB of the rest
 * on the candidate's scores, ties to the lower position) and becomes the
 * parent's state: kept prefix rows stay, freed parent slots receive the kept
 * tail rows, and the parent's scores become the candidate's.  Every layer's
 * tails must have the same length.  The fork is spent afterwards (further
 * calls return KVR_ESTATE). */
kvr_status kvr_fork_commit(kvr_fork *fork, const int32_t *chosen, int budget,
                           int window, void *stream);

/* Synchronising: candidate cand's view of sequence seq.  host_prefix_score
 * [L][H][capacity] fp32 (slot order of the parent); host_tail_k/v
 * [L][H][tail_cap][d] (kv_dtype); host_tail_score [L][H][tail_cap] fp32;
 * host_tail_pos [L][H][tail_cap] int32; host_tail_len [L][H] int32.  Any
 * pointer may be NULL. */
kvr_status kvr_fork_export(const kvr_fork *fork, int cand, int seq,
                           float *host_prefix_score, void *host_tail_k,
                           void *host_tail_v, float *host_tail_score,
                           int32_t *host_tail_pos, int32_t *host_tail_len,
                           void *stream);

/* Free the fork's host metadata (not its buffer). NULL is a no-op. */
void kvr_fork_destroy(kvr_fork *fork);

/* Which kernel runs the fork's candidate steps (for testing and
 * measurement; every choice computes the same step, Sec. 2.2 Eq. 2).
 * kernel: 0 = the library's choice (the first of 1, 2, 3 that applies,
 * else 4); 1 = candidate-batched (bf16, head_dim 128, G <= 8, N <= 8: a
 * warp per candidate, each prefix row read once per unit for all
 * candidates); 2 = chunked (one job per candidate and unit); 3 = one CTA per
 * unit; 4 = generic; 5 = candidate-batched on 5th-generation tensor cores
 * (bf16, head_dim 128, G <= 8, N <= 8, at most 128 parent rows and 64 tail
 * rows before the append: the N x G query rows of a unit are one
 * contraction against each shared prefix block).  A choice that does not
 * apply to a call runs the generic kernel for that call.  Returns
 * KVR_EINVAL outside [0, 5]. */
kvr_status kvr_fork_set_kernel(kvr_fork *fork, int kernel);

/* The kernel (1..5, numbered as for kvr_fork_set_kernel) that ran the
 * fork's last candidate step; 0 before the first step or for NULL. */
int kvr_fork_last_kernel(const kvr_fork *fork);

/* Bound, in nanoseconds, of each wait of the step kernels (fused,
 * chunked and streaming) on an asynchronous copy into shared memory for this
 * cache.  A wait that runs out sets the timeout bit of the device error
 * word; the launch then waits (up to the default bound) for the copies it
 * has in flight, leaves the units it had not finished untouched and
 * returns, and the next kvr_sync_status reports KVR_EDEVICE.  The cache's
 * state is then undefined for those units: restore it with
 * kvr_cache_import.  Not tied to a passage of the paper (failure handling
 * only).  ns: 1 .. 2e9; 0 restores the default of 2 s.  KVR_EINVAL above
 * the default or for a null cache. */
kvr_status kvr_cache_set_wait_limit(kvr_cache *cache, uint64_t ns);

/* Testing hook for the timeout path: while enable != 0, the fused and
 * chunked step kernels never load the first unit of their first CTA, so
 * the wait for it runs out after the cache's wait limit (no fault, no
 * hang; the launch returns with the timeout bit set, as above).  Never
 * enabled by the library itself.  enable: 0 or 1. */
kvr_status kvr_cache_set_hold_first_unit(kvr_cache *cache, int enable);

/* Choose whether kvr_decode_attend_score / kvr_decode_step may use the
 * fused single-pass kernel (bf16, head_dim 128, G <= 8, at most 160 live rows
 * per unit, at most one eviction per unit; the default) or must use the
 * generic kernels for every shape.  Both compute the same step; this exists
 * for testing and measurement.  enable: 0 or 1. */
kvr_status kvr_cache_set_fused(kvr_cache *cache, int enable);

/* Tuning of the fused kernel.  groups: how many units each SM computes at
 * once (1..4; 0 = the library's choice, the most the shared-memory ring and
 * thread budget allow).  group_warps: warps sharing one unit, either one
 * 16-row tile per warp or two (other values, and 0, select the library's
 * choice).  Results do not depend on either. */
kvr_status kvr_cache_set_fused_tuning(kvr_cache *cache, int groups,
                                      int group_warps);

/* Tuning of the chunked kernel that runs units of 129..1024 live rows and
 * the candidate step (bf16, head_dim 128, G <= 8): units stream in 32-row
 * chunks through per-group shared-memory rings.  groups: consumer groups per
 * SM (1..4; 0 = the library's choice; -1 = never use this kernel, so the
 * older one-CTA-per-unit kernels run instead).  stages: ring stages per
 * group (2..4; 0 = the library's choice).  A choice that does not fit in
 * shared memory for a call falls back to the older kernels for that call.
 * Results do not depend on either. */
kvr_status kvr_cache_set_chunk_tuning(kvr_cache *cache, int groups,
                                      int stages);

/* Absorb a chunk of `chunk` tokens per sequence in one call, and optionally
 * cut every unit back to B + W once afterwards (Algorithm 1: when a helper
 * step is accepted, the base model encodes its tokens in a single forward
 * pass, so its KV absorbs the step; a prompt absorbed into an empty cache
 * seeds the scores with its prefill attention).  The result is that of
 * `chunk` kvr_decode_attend_score calls followed by one kvr_evict_compact:
 * token j is appended as a new row and attends every live row and the
 * chunk's rows 0..j (causal), adding the head-mean of its probabilities to
 * the accumulated score of every row it attends (Sec. 2.1); then, if evict
 * != 0, each unit keeps its W most recent positions and the best B others
 * (score descending, position ascending; Eq. 1).
 *   q:     [S][layer_end - layer_begin][chunk][H * G][d]
 *   k_new: [S][layer_end - layer_begin][chunk][H][d]  (v_new likewise)
 *   out:   [S][layer_end - layer_begin][chunk][H * G][d], out_dtype
 * Every unit must have room for the chunk (live + chunk <= capacity), else
 * KVR_ECAPACITY before anything runs.  Stream-ordered. */
kvr_status kvr_absorb_chunk(kvr_cache *cache, int layer_begin, int layer_end,
                            int chunk, const void *q, const void *k_new,
                            const void *v_new, void *out, int budget,
                            int window, int evict, void *stream);

/* ---- candidates by copy (the paper's own fork) -------------------------- */

/* App. C ("Best-of-(N+N)"): each reasoning step forks N base candidates by
 * physically copying the accepted sequence's live (post-eviction) KV slots,
 * the candidates decode with eviction on every token like any sequence
 * (kvr_decode_step on a cache that holds them), and the chosen candidate
 * becomes the persistent sequence.  This call does both copies: sequence
 * dst_seqs[i] of dst takes the whole state of sequence src_seqs[i] of src
 * (every layer and KV head: live K/V rows, scores, positions, live length,
 * position counter), i < n.  dst_seqs and src_seqs are host arrays.
 *  - The caches must agree in layers, KV heads, head_dim and kv_dtype
 *    (KVR_EINVAL); capacities may differ, but every copied unit's live
 *    length must fit dst's capacity (KVR_ECAPACITY).
 *  - A dst sequence appears at most once; when dst == src, no sequence is
 *    both read and written (KVR_EINVAL).
 *  - Neither cache may have a live kvr_fork (KVR_ESTATE).
 *  - Stream-ordered; nothing is enqueued on an error. */
kvr_status kvr_cache_copy_sequences(kvr_cache *dst, const int32_t *dst_seqs,
                                    const kvr_cache *src,
                                    const int32_t *src_seqs, int n,
                                    void *stream);

/* ---- degeneration detector: the entropy test ---------------------------- */

/* Sec. 3.2 ("Incoherent generation") and App. C ("Online degeneration
 * detection"): each base candidate is screened while it decodes.  At its e-th
 * generated token (e = 1, 2, ... since the row's last reset) the detector
 * takes the predictive entropy
 *   H_e = -sum_v p_e(v) ln p_e(v),  p_e = softmax(logits / temperature)
 * over the whole vocabulary (natural log; nats), and its moving mean H-bar_e
 * over the last min(e, window) tokens.  The row stops at the first e > guard
 * with H-bar_e > tau; a stopped row stays stopped and its later logits are
 * not read.  App. C uses tau = 7.0, window 12, guard 24.  (The paper's
 * second test, the gzip ratio of the candidate's text, is host text work and
 * not part of this library.)
 *
 * The decision is taken in fp32: the window's entropies are summed oldest
 * first and the row stops when e > guard and sum > tau * min(e, window). */
typedef struct {
  int rows;        /* candidate rows tracked, 1..65535 */
  int vocab;       /* logits per row, >= 1 */
  int window;      /* |W_e|, 1..64 */
  int guard;       /* positions never tested (e <= guard), >= 0 */
  float tau;       /* threshold on the moving mean, nats */
  float temperature; /* softmax temperature, > 0; 0 means 1 */
  kvr_dtype logits_dtype;
} kvr_entropy_desc;

typedef struct kvr_entropy kvr_entropy; /* opaque host handle */

/* Device bytes the detector's state needs (0 for an invalid descriptor). */
size_t kvr_entropy_required_bytes(const kvr_entropy_desc *desc);

/* Lay the state out in the caller's device buffer dev_buf (256-byte aligned,
 * >= required bytes; the caller keeps ownership) and clear it on stream:
 * every row starts live with no tokens seen.  The handle owns host
 * metadata only. */
kvr_status kvr_entropy_create(const kvr_entropy_desc *desc, void *dev_buf,
                              size_t bytes, void *stream, kvr_entropy **out);

/* Rows [row_begin, row_end) take new candidates: no tokens seen, live.
 * Stream-ordered. */
kvr_status kvr_entropy_reset(kvr_entropy *det, int row_begin, int row_end,
                             void *stream);

/* One generated token for every row, in one launch.
 *   logits     dev [rows][row_stride] of logits_dtype; the first vocab of
 *              each row are read.  row_stride >= vocab (elements).
 *   entropy    dev [rows] fp32 or NULL: H_e (NaN for a row already stopped
 *              before this call, whose logits are not read).
 *   mean       dev [rows] fp32 or NULL: H-bar_e (NaN for such a row).
 *   stopped    dev [rows] int32 or NULL: after this token, the position e
 *              at which the row stopped, or 0 while it is live.
 * Rows whose logits hold a NaN or +inf, or only -inf, get H_e = NaN, never
 * stop on it, and set the device error word (kvr_entropy_sync_status).
 * Stream-ordered; calls on one handle must be ordered on one stream. */
kvr_status kvr_entropy_step(kvr_entropy *det, const void *logits,
                            int64_t row_stride, float *entropy, float *mean,
                            int32_t *stopped, void *stream);

/* Synchronising: wait for stream, then copy the state to host.
 * host_hist [rows][window] fp32: each row's last min(count, window)
 * entropies, oldest first, then zeros; host_count [rows] int32: tokens seen
 * since the row's reset; host_stopped [rows] int32 as in kvr_entropy_step.
 * Any pointer may be NULL. */
kvr_status kvr_entropy_export(kvr_entropy *det, float *host_hist,
                              int32_t *host_count, int32_t *host_stopped,
                              void *stream);

/* Synchronising: wait for stream, read and clear the detector's device
 * error word (KVR_EDEVICE if a row's logits were not finite). */
kvr_status kvr_entropy_sync_status(kvr_entropy *det, void *stream);

/* Kernel choice (results agree within rounding): 0 = the library's choice
 * (the streaming kernel where the rows allow it),
 * 1 = the persistent streaming kernel wherever the rows are 16-byte aligned
 * and hold at least one 16-byte vector (the piece kernel otherwise),
 * 2 = the piece kernel (one CTA per 16,384 bf16 / 8,192 fp32 logits). */
kvr_status kvr_entropy_set_kernel(kvr_entropy *det, int kernel);

/* Number of kernels this handle has launched since it was created. */
kvr_status kvr_entropy_launch_count(const kvr_entropy *det, uint64_t *count);

void kvr_entropy_destroy(kvr_entropy *det);

/* Kernel of kvr_absorb_chunk's one-launch path (bf16, head_dim 128, G <= 8,
 * chunk <= 64, at most 192 rows after the chunk, 16-byte aligned q, k_new,
 * v_new and out; other calls run token by token).  Results agree within
 * rounding: 0 = 5th-generation tensor cores with the logits, probabilities
 * and outputs in tensor memory, for units of at most 144 rows after the
 * chunk (larger ones run kernel 1; the default), 1 = mma.sync with register
 * accumulators. */
kvr_status kvr_cache_set_absorb_kernel(kvr_cache *cache, int kernel);

/* How the cache's last kvr_absorb_chunk ran: 0 = the tensor-memory kernel,
 * 1 = the mma.sync kernel, 2 = token by token; -1 before the first call
 * (or for NULL).  Host state only: no synchronisation. */
int kvr_cache_last_absorb_kernel(const kvr_cache *cache);

/* ---- the same step for callers that cannot allocate -------------------- */

/* The paper has no counterpart to this call: it is a deployment variant.
 *
 * Some callers cannot allocate device memory for a call at all: a plug-in
 * running inside a host program that owns every device allocation and hands
 * the plug-in only the tensors of a call, or a service that fixes its device
 * footprint at start-up and may not allocate afterwards.  This entry point
 * does exactly what kvr_decode_attend_score does (same arguments, same
 * results), but keeps the per-unit logits in a static device array inside
 * the library instead of the cache buffer's scratch area, and calls no
 * allocator (no cudaMalloc, cudaFree or allocating library routine).
 *  - Limit: the call needs S x (layer_end - layer_begin) x H x G x
 *    (longest live length + 1) x 4 bytes of logits; more than
 *    KVR_NOALLOC_SCRATCH_BYTES is rejected with KVR_EINVAL before anything
 *    is enqueued.
 *  - Every GPU that loads the library holds the array until the process
 *    exits.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress, with that device current); make that first call
 *    before any stream capture.
 *  - All calls share the array and it keeps the previous call's contents:
 *    every logit is written before it is read, so nothing needs clearing,
 *    but calls that overlap on the GPU (other streams or host threads) race
 *    on it; serialise them. */
#define KVR_NOALLOC_SCRATCH_BYTES (4u << 20)
kvr_status kvr_decode_attend_score_noalloc(kvr_cache *cache, int layer_begin,
                                           int layer_end, const void *q,
                                           const void *k_new,
                                           const void *v_new, void *out,
                                           void *stream);

/* ---- inspection -------------------------------------------------------- */

/* Synchronising: wait for stream, then replace sequence seq's state with a
 * host copy in the layout kvr_cache_export writes (resuming a decode, or a
 * state built outside the library): host_k, host_v [L][H][capacity][d]
 * (kv_dtype); host_score [L][H][capacity] fp32; host_pos [L][H][capacity]
 * int32; host_len and host_next_pos [L][H] int32.  Rows [0, len) of a unit
 * are live; the rest are copied but never read.  Checked on the host before
 * anything is copied (KVR_EINVAL): no pointer is NULL; 0 <= len <=
 * capacity; the KV heads of a layer share len and next_pos (every decode
 * call keeps them equal); 0 <= next_pos < INT32_MAX; live positions are
 * distinct and below next_pos.  KVR_ESTATE while the cache has a live fork.
 * Importing what kvr_cache_export returned and decoding on gives the same
 * results bit for bit. */
kvr_status kvr_cache_import(kvr_cache *cache, int seq, const void *host_k,
                            const void *host_v, const float *host_score,
                            const int32_t *host_pos, const int32_t *host_len,
                            const int32_t *host_next_pos, void *stream);

/* Synchronising: wait for stream, then copy sequence seq's state to host.
 * host_k, host_v [L][H][capacity][d] (kv_dtype); host_score [L][H][capacity]
 * fp32; host_pos [L][H][capacity] int32; host_len and host_next_pos [L][H]
 * int32 (live length; position the next appended row will get).  Any pointer
 * may be NULL.  Slots at or beyond a unit's length hold stale data. */
kvr_status kvr_cache_export(const kvr_cache *cache, int seq, void *host_k,
                            void *host_v, float *host_score, int32_t *host_pos,
                            int32_t *host_len, int32_t *host_next_pos,
                            void *stream);

/* The scores half of the step's result, with no copy: device pointers into
 * the caller's cache buffer, valid for the cache's lifetime.
 *   score  [S][L][H][row_stride] fp32: the accumulated importance score of
 *          the row in each slot (Sec. 2.1)
 *   pos    [S][L][H][row_stride] int32: the row's position (token index)
 *   state  [S][L][H][4] int32: live length, next position, 1 while the
 *          library holds a current sum of the unit's normalised keys for
 *          kvr_decode_step_rkv (else 0), 0
 * Slots [0, live length) of a unit hold its rows, in no particular order.
 * The values are those after the last call enqueued on the cache's stream;
 * read them stream-ordered.  Any output pointer may be NULL. */
kvr_status kvr_cache_scores(const kvr_cache *cache, float **score,
                            int32_t **pos, int32_t **state,
                            int64_t *row_stride);

/* Host mirror of the live length of every (sequence, layer): host_len
 * [S][L].  Not synchronising (the mirror is exact after every call). */
kvr_status kvr_cache_lengths(const kvr_cache *cache, int32_t *host_len);

/* Number of kernels this handle has launched since it was created (each
 * call adds the kernels it enqueued; memsets are not counted). */
kvr_status kvr_cache_launch_count(const kvr_cache *cache, uint64_t *count);

/* Synchronising: wait for stream, read and clear the device error word.
 * KVR_OK if no kernel reported an error since the last call. */
kvr_status kvr_sync_status(kvr_cache *cache, void *stream);

/* Message of the last failing call on this thread ("" if none). */
const char *kvr_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* KVR_H */
