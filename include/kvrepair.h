/*
 * kvrepair.h -- C ABI of libkvrepair: repairing a stale KV cache in place,
 * within a budget of positions, after a same-length document edit, on one
 * GB300 GPU (sm_103a).
 *
 * Method: "Contiguity, Not Importance: Budgeted Repair of Stale KV Caches
 * After Document Edits", Sec. 3.  A context C of n tokens is prefilled and
 * its key/value states K(C) are cached.  An edit replaces the tokens of
 * S = [s_start, s_end) (end excluded) by as many new ones, giving C'.  Repair
 * recomputes the positions P = S u A, A a subset of the pool D = [s_end, n),
 * from C' one layer at a time against the otherwise-stale cache and writes the
 * refreshed K/V back in place (operator R, Eq. 1).  A is chosen by one of the
 * five selection policies of Table 1.
 *
 * Conventions for every entry point:
 *   - Return value: KVR_OK (0) or an error code below; kvr_last_error()
 *     returns a message for the calling thread's last failure.
 *   - Token, position and output arrays are HOST pointers (int32 / float),
 *     owned by the caller and only read/written during the call.
 *   - Model and cache handles are owned by the library and freed with
 *     kvr_model_free / kvr_cache_free.  kvr_model_free also frees every
 *     cache of the model still live; their handles are invalid afterwards.
 *   - Device work is enqueued on the model's stream (kvr_model_set_stream;
 *     default: the legacy default stream).  Calls that return data to the host
 *     (kvr_select, kvr_logits, kvr_cache_read*) synchronise that stream;
 *     kvr_prefill and kvr_repair return once the work is enqueued.
 *   - Argument errors are detected on the host before any device work and
 *     leave the cache unchanged.  A CUDA error during device work marks the
 *     cache poisoned; every later call on it returns KVR_E_POISONED.
 *   - Device waits (mbarrier spins in the tensor-core kernels) are bounded;
 *     a wait that runs out sets a device flag that kvr_synchronize (and the
 *     synchronising calls) report as KVR_E_DEVICE_TIMEOUT.
 *   - Not thread-safe per model: calls on one model (and its caches) must not
 *     overlap.
 */
#ifndef KVREPAIR_H
#define KVREPAIR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t kvr_status;
#define KVR_OK 0
#define KVR_E_INVAL 1          /* malformed argument (NULL handle, bad config) */
#define KVR_E_RANGE 2          /* span / positions / tokens out of range */
#define KVR_E_NOMEM 3          /* device or host allocation failed */
#define KVR_E_CUDA 4           /* CUDA runtime or kernel error */
#define KVR_E_DEVICE_TIMEOUT 5 /* a bounded device wait ran out */
#define KVR_E_UNSUPPORTED 6    /* shape or option this build does not handle */
#define KVR_E_POISONED 7       /* cache was left inconsistent by an earlier CUDA error */

typedef enum { KVR_DTYPE_F32 = 0, KVR_DTYPE_BF16 = 1 } kvr_dtype;

/* Selection policies of Table 1.  All pick from the pool D = [s_end, n). */
typedef enum {
  KVR_POLICY_EDITLOCAL = 0,  /* the first K pool positions, those next to the span */
  KVR_POLICY_STRUCTURAL = 1, /* delimiter tokens of the pool, closest first */
  KVR_POLICY_ATTENTION = 2,  /* top-K stale-cache attention from the span queries */
  KVR_POLICY_CACHEBLEND = 3, /* top-K layer-1 (0-indexed) K/V deviation */
  KVR_POLICY_RANDOM = 4,     /* uniform K-subset, seeded */
  /* EditLocal@boundary (Sec. 5.2): the positions from the span end through
   * the next document boundary (the first delimiter token at or after
   * edit_end, inclusive; the end of the context if there is none), with no
   * selector forward; K caps the window. */
  KVR_POLICY_EDITLOCAL_BOUNDARY = 5
} kvr_policy;

/* Llama-style decoder shape (RMSNorm, rotate-half RoPE, GQA, SwiGLU). */
typedef struct {
  int32_t vocab, d_model, n_layers, n_heads, n_kv_heads, head_dim, ffn;
  int32_t qkv_bias;    /* 1: q/k/v projections carry a bias */
  int32_t dtype;       /* kvr_dtype of weights, GEMM operands and the KV cache */
  int32_t delim_id;    /* structural delimiter token id */
  double rope_theta;   /* RoPE base */
  double rms_eps;      /* RMSNorm epsilon */
  int32_t max_context; /* longest context a cache of this model may hold */
  int32_t max_rows;    /* rows per layer pass (prefill is chunked to this); >= 64 */
} kvr_model_config;

/* Host weights in canonical layout and the model dtype (fp32, or bf16 as
 * uint16 bit patterns).  Matrices are row-major [out_features][in_features]:
 * wq [H*dh][d], wk/wv [G*dh][d], wo [d][H*dh], wg/wu [ffn][d], wd [d][ffn],
 * embed/lm_head [vocab][d]; norms [d]; biases [H*dh] / [G*dh] (NULL without
 * qkv_bias).  Per-layer fields are arrays of n_layers pointers.  The library
 * copies everything; the caller keeps ownership. */
typedef struct {
  const void *embed, *final_norm, *lm_head;
  const void *const *attn_norm, *const *wq, *const *wk, *const *wv, *const *wo;
  const void *const *bq, *const *bk, *const *bv;
  const void *const *mlp_norm, *const *wg, *const *wu, *const *wd;
} kvr_weights;

typedef struct kvr_model kvr_model;
typedef struct kvr_cache kvr_cache;

/* Optional device allocator (e.g. PyTorch's caching allocator).  Must be set
 * before the first kvr_model_create; NULL functions restore cudaMalloc/cudaFree. */
typedef void *(*kvr_alloc_fn)(size_t bytes, void *ctx);
typedef void (*kvr_free_fn)(void *ptr, void *ctx);
kvr_status kvr_set_allocator(kvr_alloc_fn alloc, kvr_free_fn free_fn, void *ctx);

/* Create a model on the current CUDA device.  weights == NULL: seeded random
 * init, generated on the device: tensor t draws from SplitMix64 stream
 * s_t = out(seed, t), element i (canonical row-major index) from
 * r = out(s_t, i), where out(s, i) = mix(s + (i+1) * 0x9E3779B97F4A7C15);
 * the four 16-bit lanes of r are summed, centred and scaled in double to
 * std 0.02, rounded to fp32 and then to the model dtype; norms are 1.  Tensor
 * ids: embed 0, lm_head 1, layer l: 8 + 16 l + {wq 0, wk 1, wv 2, wo 3, wg 4,
 * wu 5, wd 6, bq 7, bk 8, bv 9}.  Errors: KVR_E_INVAL (config),
 * KVR_E_UNSUPPORTED (shape), KVR_E_NOMEM. */
kvr_status kvr_model_create(const kvr_model_config *config, const kvr_weights *weights,
                            uint64_t seed, kvr_model **out);
void kvr_model_free(kvr_model *model);

/* Launch all device work of `model` (and its caches) on `cuda_stream`
 * (a cudaStream_t; NULL = legacy default stream). */
kvr_status kvr_model_set_stream(kvr_model *model, void *cuda_stream);

/* Block until the model's stream is idle; reports device-side timeouts. */
kvr_status kvr_synchronize(kvr_model *model);

/* Full prefill K(C) (Sec. 3: the oracle target; Table 4's baseline).
 * tokens: host int32[n], 0 <= id < vocab, 1 <= n <= max_context.  The new
 * cache owns a device copy of the tokens and paged K/V for every layer. */
kvr_status kvr_prefill(kvr_model *model, const int32_t *tokens, int32_t n, kvr_cache **out);
void kvr_cache_free(kvr_cache *cache);

/* A cache restored from host memory instead of computed: the stored state
 * K(C) of Sec. 3 for a context C of n tokens, e.g. one saved earlier with
 * kvr_cache_read_raw over positions 0..n-1 and all layers.  tokens: host
 * int32[n] (same rules as kvr_prefill); k, v: host arrays
 * [n][n_layers][n_kv_heads][head_dim] in the cache's element type (bf16 bit
 * patterns for a bf16 model, fp32 otherwise), only read during the call.
 * The library does not check that the entries are the prefill of the tokens:
 * repair and the selectors compute against whatever they hold, except that
 * the CACHEBLEND policy takes the layer-0 entries of pool positions as the
 * function of their token and position that every prefill leaves there.
 * Synchronous.  Errors: KVR_E_INVAL (NULL argument), KVR_E_RANGE (n, token
 * ids), KVR_E_NOMEM, KVR_E_CUDA. */
kvr_status kvr_cache_load(kvr_model *model, const int32_t *tokens, int32_t n, const void *k,
                          const void *v, kvr_cache **out);

/* Select A (Table 1; Sec. 3 "Cost accounting": selector work is outside K).
 * The edit [edit_start, edit_start+edit_len) with host new_tokens[edit_len]
 * is applied to a private copy of the context, not to the cache; the
 * ATTENTION and CACHEBLEND policies run their model passes against the stale
 * cache and leave it bit-identical.  positions_out: host int32[K], receives
 * *count_out ascending positions in [edit_end, n).  *count_out == K except
 * for STRUCTURAL when the pool holds fewer delimiters, and when the pool is
 * smaller than K.  Ties go to the lowest position.  Device scratch (the
 * edited tokens; for ATTENTION and CACHEBLEND the saved span rows and the
 * ATTENTION logits) belongs to the model and only grows: a call that fits
 * allocates nothing.  Errors: KVR_E_RANGE (K < 0, span outside the
 * context, token id outside the vocabulary, empty span for ATTENTION or
 * CACHEBLEND), KVR_E_INVAL (NULL argument, cache of another model, unknown
 * policy), KVR_E_POISONED, KVR_E_UNSUPPORTED (span above max_rows,
 * CACHEBLEND with fewer than 2 layers), KVR_E_NOMEM (scratch cannot grow). */
kvr_status kvr_select(kvr_model *model, const kvr_cache *cache, kvr_policy policy, int32_t K,
                      int32_t edit_start, int32_t edit_len, const int32_t *new_tokens,
                      uint64_t seed, int32_t *positions_out, int32_t *count_out);

/* Repair in place (operator R, Sec. 3 "The repair interface", Eq. 1):
 * write new_tokens into [edit_start, edit_start+edit_len) of the cached
 * context, then recompute P = S u positions through every layer; all rows of
 * P get fresh K/V at a layer before any of them attends there, every entry
 * outside P is left unchanged.  positions: host int32[n_positions], strictly
 * increasing, in [edit_end, n).  edit_len may be 0 (recompute positions
 * only).  |P| <= max_rows.  Errors: KVR_E_RANGE (span, positions, token ids),
 * KVR_E_UNSUPPORTED (|P| > max_rows). */
kvr_status kvr_repair(kvr_cache *cache, const int32_t *new_tokens, int32_t edit_start,
                      int32_t edit_len, const int32_t *positions, int32_t n_positions);

/* kvr_repair, returning the recomputed entries (Sec. 3, Eq. 1: the rows of P
 * of the repaired cache) in host memory: k_out, v_out receive
 * [|P|][n_layers][n_kv_heads][head_dim] in the cache's element type (bf16 bit
 * patterns for a bf16 model, fp32 otherwise), rows in P's ascending order
 * (the span, then positions) -- what kvr_cache_read_raw returns for P after
 * kvr_repair.  The rows of each group of layers are copied while the pass
 * computes the later layers; with page-locked k_out/v_out the copies overlap
 * the pass, pageable memory is accepted.  Synchronous: returns once the rows
 * are in host memory, reporting device-side timeouts like kvr_synchronize.
 * A row buffer on the device belongs to the model and only grows.  Errors as
 * kvr_repair; KVR_E_INVAL for NULL k_out or v_out with |P| > 0. */
kvr_status kvr_repair_read(kvr_cache *cache, const int32_t *new_tokens, int32_t edit_start,
                           int32_t edit_len, const int32_t *positions, int32_t n_positions,
                           void *k_out, void *v_out);

/* One repair request of a batch: a cache, its edits and the union of the
 * selected positions.  Edits must not overlap; positions must not fall in
 * any edit span. */
typedef struct {
  kvr_cache *cache;
  int32_t n_edits;
  const int32_t *edit_start; /* [n_edits] */
  const int32_t *edit_len;   /* [n_edits] */
  const int32_t *new_tokens; /* concatenated, sum(edit_len) ids */
  const int32_t *positions;  /* [n_positions], strictly increasing */
  int32_t n_positions;
} kvr_repair_req;

/* Several documents, several edits each (beyond the paper's single edit;
 * P_doc = sorted union of all spans and positions), recomputed in one
 * layer-major pass over all rows of all requests.  All caches belong to
 * `model`.  Sum of |P_doc| <= max_rows. */
kvr_status kvr_repair_batch(kvr_model *model, const kvr_repair_req *reqs, int32_t n_reqs);

/* Transplant (Sec. 3, "Transplant is not recomputation"): copy the K/V of
 * every layer, and the token, at the given positions from `src` into `dst`
 * -- e.g. from a fresh prefill of the edited context into the stale cache.
 * A diagnostic operator: it needs the oracle cache, so it is not a repair.
 * Both caches belong to one model and hold the same number of positions;
 * positions: host int32[n_positions], strictly increasing, in [0, n).
 * Asynchronous on the model's stream.  Errors: KVR_E_INVAL, KVR_E_RANGE. */
kvr_status kvr_transplant(kvr_cache *dst, const kvr_cache *src, const int32_t *positions,
                          int32_t n_positions);

/* Teacher-forced answer log-probability for the margin of Eq. 2: the prompt
 * (m_prompt >= 1 tokens) and the answer (m_answer >= 1 tokens) follow the
 * cached context at positions n.., the answer fed one token behind (teacher
 * forcing); *mean_logprob_out = (1/m_answer) sum_i log p(answer_i | context,
 * prompt, answer_<i) under the cache's K/V, length-averaged as Eq. 2
 * prescribes.  The document's K/V are not modified.  m_prompt + m_answer - 1
 * <= 64.  The margin m_x of a cache state is the difference of this value for
 * a_new and a_old; MR (Eq. 2) follows from m of the repaired, stale and
 * oracle caches. */
kvr_status kvr_answer_logprob(kvr_model *model, const kvr_cache *cache, const int32_t *prompt,
                              int32_t m_prompt, const int32_t *answer, int32_t m_answer,
                              double *mean_logprob_out);

/* The margin m_x of Eq. 2 for one cache state: the length-averaged
 * teacher-forced log-probability (kvr_answer_logprob) of the answer a_new
 * minus that of a_old, both after the same prompt.  MR (Eq. 2) is
 * (m_repaired - m_stale) / (m_oracle - m_stale) over three cache states.
 * Errors as kvr_answer_logprob, and KVR_E_INVAL for a NULL margin_out. */
kvr_status kvr_margin(kvr_model *model, const kvr_cache *cache, const int32_t *prompt,
                      int32_t m_prompt, const int32_t *a_new, int32_t m_new,
                      const int32_t *a_old, int32_t m_old, double *margin_out);

/* Fresh-query logits (Sec. 3: the query that scores a cache state is
 * computed anew each time and kept out of the cache).  The m query tokens (1 <= m <= 64) take positions
 * n..n+m-1 and attend to the cache; the document's K/V are not modified.
 * logits_out: host float[vocab], the logits of the last query row. */
kvr_status kvr_logits(kvr_model *model, const kvr_cache *cache, const int32_t *query, int32_t m,
                      float *logits_out);

/* ---- inspection (tests, benchmarks) ---- */

/* Number of cached positions n. */
int32_t kvr_cache_len(const kvr_cache *cache);

/* Copy the cached context's tokens into host int32[n]. */
kvr_status kvr_cache_tokens(const kvr_cache *cache, int32_t *tokens_out);

/* Read K and V of the given positions for layers [layer_begin, layer_end)
 * into host float arrays laid out [n_pos][layer_end-layer_begin][n_kv_heads]
 * [head_dim] (bf16 entries are widened exactly). */
kvr_status kvr_cache_read(const kvr_cache *cache, const int32_t *positions, int32_t n_pos,
                          int32_t layer_begin, int32_t layer_end, float *k_out, float *v_out);

/* The same rows in the cache's own element type: bf16 bit patterns (2 bytes
 * per entry) for a bf16 model, fp32 otherwise -- the repaired K/V exactly as
 * stored, at half the bytes of kvr_cache_read for bf16.  Same layout; k_out and
 * v_out are host buffers of n_pos * (layer_end - layer_begin) * n_kv_heads *
 * head_dim entries each, which the device writes directly when they are
 * page-locked.  No device allocation during the call (model-owned scratch,
 * grown when a larger read first needs it).  Synchronous.  Errors as
 * kvr_cache_read: KVR_E_INVAL for NULL pointers, KVR_E_RANGE for a layer range
 * or position outside the cache, KVR_E_NOMEM if the scratch cannot grow. */
kvr_status kvr_cache_read_raw(const kvr_cache *cache, const int32_t *positions, int32_t n_pos,
                              int32_t layer_begin, int32_t layer_end, void *k_out, void *v_out);

/* Read one weight tensor back in canonical layout and model dtype into host
 * memory of `bytes` bytes.  name: "embed", "lm_head", "final_norm", or per
 * layer "wq","wk","wv","wo","wg","wu","wd","bq","bk","bv","attn_norm",
 * "mlp_norm".  Norms and biases are returned in the model dtype too. */
kvr_status kvr_model_read_tensor(const kvr_model *model, const char *name, int32_t layer,
                                 void *out, size_t bytes);

/* One projection of the model through the library's GEMM kernels (the
 * operator's a5/a7/a8 contractions, exposed for kernel tests):
 * y[M][N] = x[M][K] . W^T, x host [M][K] in the model dtype, y host float.
 * name "wqkv" (N = (H+2G)*dh: q, k, v rows, bias added), "wo", "wd",
 * "lm_head", or "wgu", which returns the fused SwiGLU activation
 * silu(x Wg^T) * (x Wu^T) [M][ffn] (rounded to the model dtype).  1 <= M <=
 * max_rows.  Synchronous. */
kvr_status kvr_linear(kvr_model *model, const char *name, int32_t layer, const void *x, int32_t M,
                      float *y);

/* kvr_linear without any allocation during the call.  The paper has no
 * counterpart; this serves callers that must not allocate device memory at
 * call time (a serving loop under a memory budget reserved up front, code
 * that cannot take the device-wide synchronisation cudaMalloc/cudaFree may
 * imply, hosts whose allocator belongs to another framework).  x: DEVICE
 * bf16 [M][K], y: DEVICE float [M][N], both owned by the caller; name
 * "wqkv", "wo", "wd" or "lm_head" of a bf16 model on the tensor-core GEMM;
 * 1 <= M <= 64, otherwise KVR_E_UNSUPPORTED; x or y not device memory of the
 * model's device: KVR_E_INVAL (checked before any launch).  The GEMM's
 * scratch (partial tiles, arrival counters) is a fixed ~10.5 MB device array
 * that every GPU loading the library holds until exit; the first call on a
 * device looks up its address (make that call before any stream capture) and
 * keeps it for the process: after cudaDeviceReset or a release of the
 * device's primary context, do not call it on that device again.  All calls
 * share the array: calls whose GPU work overlaps race and give wrong results.
 * Asynchronous on the model's stream; kvr_synchronize reports device
 * timeouts.  Allocates nothing: no cudaMalloc, cudaFree or allocating
 * library call. */
kvr_status kvr_linear_noalloc(kvr_model *model, const char *name, int32_t layer, const void *x,
                              int32_t M, float *y);

/* Per-kernel-class device timing with CUDA events around each launch group.
 * enable != 0 turns it on for later calls; kvr_profile_read returns, for
 * up to `cap` classes, the accumulated milliseconds and launch counts since
 * the last reset, and writes the class names (NUL-separated) into `names`.
 * Returns the number of classes via *n_out. */
kvr_status kvr_profile_enable(kvr_model *model, int32_t enable);
kvr_status kvr_profile_reset(kvr_model *model);
kvr_status kvr_profile_read(kvr_model *model, int32_t cap, double *ms_out, int64_t *launches_out,
                            int64_t *bytes_out, char *names, int32_t names_cap, int32_t *n_out);

/* Device timeline trace (tooling; the paper has no counterpart).  Only the
 * KVR_TRACE build of the library (libkvrepair_trace.so) records; elsewhere
 * kvr_trace_enable with capacity > 0 returns KVR_E_UNSUPPORTED.  With
 * capacity > 0, a device buffer of `capacity` records is attached and every
 * CTA of the pass kernels (embedding, RMSNorm, GEMM, RoPE/scatter,
 * attention, combine) and of the Attention selector's two kernels appends
 * one record of 16 uint64 words:
 *   [0] kind (1 embed, 2 rmsnorm, 3 GEMM, 4 RoPE/scatter, 5 attention,
 *       6 combine, 8 selector logits, 9 selector accumulation) | SM id << 8
 *       | linear block index << 16,
 *   [1] start, [2] return of the wait on the predecessor kernel, [3] end,
 *   [4..11] eight marks, 0 where the kernel sets none.  GEMM, for the CTA's
 *       last tile: first operand stage landed, all MMAs complete,
 *       accumulator taken by the epilogue, partial tile stored, split-tile
 *       arrival counted or partials staged across the cluster, tile reduced
 *       and written, epilogue done, all warps done.  Attention: last key
 *       chunk consumed.  Selector logits: keys and queries staged, logits
 *       computed, chunk statistics stored, arrival counted, softmax
 *       statistics folded (the group's last CTA only).
 *   [12..15] zero,
 * times in ns of the device's global timer.  Records past `capacity` are
 * dropped.  capacity == 0 detaches and frees the buffer.  The buffer is
 * process-wide: the model that attached it last owns it, and kernels of
 * every model on the device write to it.  kvr_trace_read synchronises the
 * model's stream, copies up to `cap` records to host `out` (uint64[16*cap]),
 * returns the number appended via *n_out (which may exceed what fitted),
 * and empties the buffer.  Errors: KVR_E_INVAL, KVR_E_NOMEM,
 * KVR_E_UNSUPPORTED. */
kvr_status kvr_trace_enable(kvr_model *model, int32_t capacity);
kvr_status kvr_trace_read(kvr_model *model, uint64_t *out, int32_t cap, int32_t *n_out);

/* Failure-detection probe (tests): enqueue on the model's stream one thread
 * that waits for a device word nothing sets, bounded by limit_us (1 ..
 * 1e6) like every device wait of the library.  When the bound runs out it
 * sets the model's device flag; the next synchronising call (kvr_synchronize,
 * kvr_select, the readbacks) returns KVR_E_DEVICE_TIMEOUT and clears the
 * flag, and the model stays usable.  Errors: KVR_E_INVAL, KVR_E_RANGE. */
kvr_status kvr_wait_probe(kvr_model *model, int32_t limit_us);

/* Number of library kernels launched so far on this model. */
int64_t kvr_launch_count(const kvr_model *model);

/* Message of the calling thread's last failure ("" if none). */
const char *kvr_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* KVREPAIR_H */
