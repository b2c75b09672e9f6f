/*
 * txs.h — C ABI of libtxs, the GB300 (sm_103a) serving path of TransX:
 * amortised behavior K/V caching and multi-candidate next-action decoding.
 *
 * Paper: "TransX: Scaling Transformer-based Recommendation via Behavioral and
 * Serving Stream Crossings" (KDD '26), arXiv 2607.28940.
 *
 * Conventions for every entry point
 * ---------------------------------
 * - Row-vector convention y = x W + b; matrices are row-major.
 * - "device" pointers are CUDA device (or managed) memory owned by the caller;
 *   the library never frees them.  "host" pointers are ordinary host memory,
 *   read before the call returns.
 * - Floating-point storage type of weights, behavior rows and tokens is the
 *   model's dtype (TXS_FP32: float, TXS_BF16: bfloat16).  Outputs of scores are
 *   always float.
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   Every call enqueues its work on that stream and returns without waiting;
 *   argument errors are detected on the host and returned before anything is
 *   enqueued.  Errors found by kernels (bounds, timeouts) are latched in a
 *   per-model device status word read by txs_device_status().
 * - No entry point throws; all return txs_status.
 * - Handles (txs_model, txs_kv_cache) own the device memory they allocate at
 *   create/build time and free it in the matching destroy call.
 * - Calls on the same handle must be ordered by the caller (same stream, or
 *   events); the library does not lock.
 * - CUDA graphs: txs_rebuild_kv_cache, txs_append_behavior,
 *   txs_score_candidates, txs_rank_candidates and txs_encode_append can be
 *   captured (stream capture) when their host offset
 *   arrays hold at most 8000 ints in all per call (they travel as kernel
 *   parameters).  A replay repeats the captured device work, the uploads of
 *   the offsets and lengths computed at capture included, but not the host
 *   bookkeeping: host-side lengths (txs_cache_lengths, capacity checks) stay
 *   those of the last direct call.
 */
#ifndef TXS_H
#define TXS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  TXS_OK = 0,
  TXS_ERR_INVALID_ARG = 1,    /* bad pointer, size, offset array or config      */
  TXS_ERR_COLD_START = 2,     /* a request has no behavior rows (App. D)         */
  TXS_ERR_CAPACITY = 3,       /* append exceeds the cache's spare capacity       */
  TXS_ERR_STALE_CACHE = 4,    /* cache built by a model with other weights/config*/
  TXS_ERR_CUDA = 5,           /* a CUDA runtime/driver call failed               */
  TXS_ERR_DEVICE_TIMEOUT = 6, /* a bounded device-side wait gave up              */
  TXS_ERR_BOUNDS = 7,         /* a kernel saw an index outside its buffers       */
  TXS_ERR_UNSUPPORTED = 8     /* shape outside what the kernels implement        */
} txs_status;

typedef enum { TXS_FP32 = 0, TXS_BF16 = 1 } txs_dtype;

/* Key set of the cross-attention (Sec. 4.1.2 local-global sparse set):
 * LOCAL_GLOBAL = the l_local most recent behavior rows plus the attention-pooled
 * global anchor; FULL = every cached row, no anchor (the -sparseAttn ablation,
 * Sec. 5.2). */
typedef enum { TXS_ATTN_LOCAL_GLOBAL = 0, TXS_ATTN_FULL = 1 } txs_attn_mode;

typedef struct {
  int32_t d_model;   /* d; multiple of 64 for TXS_BF16, of 32 for TXS_FP32; <= 512 */
  int32_t n_heads;   /* H; d_head = d_model / n_heads must be 32 or 64             */
  int32_t d_ff;      /* F; multiple of 64                                         */
  int32_t n_layers;  /* decoder layers, >= 1                                      */
  int32_t n_actions; /* k action tokens (Sec. 4.1.3), 1..16                       */
  int32_t n_ctx;     /* S serving-context tokens per request (App. B), 0..8       */
  int32_t l_local;   /* L_local (Sec. 4.1.2), >= 1                                */
  int32_t attn_mode; /* txs_attn_mode                                             */
  int32_t dtype;     /* txs_dtype                                                 */
  float ln_eps;      /* LayerNorm epsilon (> 0)                                   */
  int32_t n_kv_heads;/* K/V heads of the behavior cache (MQA/GQA variants cited in
                        Sec. 4.1.2): 0 = n_heads; otherwise divides n_heads, and
                        query head h uses K/V head h / (n_heads / n_kv_heads).  The
                        cached rows are n_kv_heads * d_head wide.                   */
  int32_t cand_mlp_hidden; /* hidden width Fc of the candidate-to-query MLP
                        Phi_candidate (Sec. 4.1.2; multiple of 64, <= 16384), or 0
                        when the candidate tokens already are its outputs       */
  int32_t head_dw_hidden; /* Deep & Wide f_dec (App. B): hidden width Fh of its deep
                        FFN (multiple of 64, <= 16384), or 0 for the linear f_dec */
  int32_t head_dw_in;  /* Deep & Wide: the first dw_in features of a candidate token
                        are its wide (linear) part, the rest its deep part;
                        0 <= dw_in <= d_model, multiple of 64                    */
  int32_t head_dw_out; /* Deep & Wide: width of the wide part of k_dec,
                        0 <= dw_out < d_model (the deep part is the rest)       */
} txs_config;

typedef struct txs_model txs_model;       /* opaque */
typedef struct txs_kv_cache txs_kv_cache; /* opaque */

/* Number of per-layer weight tensors and of head tensors in the `weights`
 * array of txs_model_create. */
#define TXS_WEIGHTS_PER_LAYER 22
#define TXS_HEAD_WEIGHTS 4

/*
 * txs_model_create — copy the decoder weights into the library's device layout.
 *
 * `weights` (host array of device pointers) holds n_layers * 22 + 4 (+ 4)
 * pointers,
 * layer by layer, then the head, in this order and with these shapes
 * (d = d_model, F = d_ff, k = n_actions, dkv = n_kv_heads * d_head, which is d
 * when n_kv_heads is 0 or n_heads), all in the config's dtype:
 *   per layer l (Sec. 4.1.2 crossAttend block; App. B serving-stream attention):
 *     0 W_qkv [d,3d]  1 b_qkv [3d]   2 W_os [d,d]  3 b_os [d]  4 ln1_g [d] 5 ln1_b [d]
 *     6 W_Q  [d,d]    7 b_Q  [d]     8 W_K [d,dkv] 9 b_K [dkv] 10 W_V [d,dkv] 11 b_V [dkv]
 *    12 W_oc [d,d]   13 b_oc [d]    14 ln2_g [d]  15 ln2_b [d]
 *    16 W_1  [d,F]   17 b_1  [F]    18 W_2 [F,d]  19 b_2 [d]  20 ln3_g [d] 21 ln3_b [d]
 *   head (Sec. 4.1.3; attention pooling Sec. 5.1):
 *     w_pool [d], W_dec [2d,d], b_dec [d], Q_dec [k,d]
 *   then, when cand_mlp_hidden = Fc > 0, the candidate MLP (4 more pointers):
 *     W_c1 [d,Fc], b_c1 [Fc], W_c2 [Fc,d], b_c2 [d]
 *   (the decoder sees GELU(x W_c1 + b_c1) W_c2 + b_c2 for each candidate
 *   token x; the head's f_dec(z, x) keeps the raw x)
 *   then, when head_dw_hidden = Fh > 0, the Deep & Wide f_dec (6 more;
 *   a = dw_in, o = dw_out):
 *     W_w [a,o], b_w [o], W_d1 [2d-a,Fh], b_d1 [Fh], W_d2 [Fh,d-o], b_d2 [d-o]
 *   with k_dec = [x[:a] W_w + b_w, GELU([z, x[a:]] W_d1 + b_d1) W_d2 + b_d2];
 *   the head's W_dec and b_dec are then unused and may be NULL, as may
 *   W_w when a or o is 0 and b_w when o is 0.
 * The call synchronises the device first (the weights may still be in flight
 * on any stream) and returns after the copies are done; the inputs may be
 * freed afterwards.  The model keeps a 64-bit content hash of config and weights.
 * Errors: TXS_ERR_INVALID_ARG, TXS_ERR_UNSUPPORTED, TXS_ERR_CUDA.
 */
txs_status txs_model_create(const txs_config* cfg, const void* const* weights, txs_model** out);
void txs_model_destroy(txs_model* model);
/* Content hash of config + weights (identical weights give identical hashes). */
uint64_t txs_model_hash(const txs_model* model);

/*
 * txs_build_kv_cache — nearline cache build (Sec. 4.3, amortised encoding and
 * KV caching; Sec. 4.1.2 K = Phi_b W_K, V = Phi_b W_V).
 *
 * For each request r the rows beh_enc[beh_offsets[r] .. beh_offsets[r+1]) are
 * the encoded behavior stream Phi_b (row-major [sum L_r, d_model], device).
 * For every layer l the cache stores K_l = Phi_b W_K^l + b_K^l and
 * V_l = Phi_b W_V^l + b_V^l in the model dtype, plus the attention-pooled
 * anchor g = softmax(Phi_b w_pool / sqrt(d))^T Phi_b and its projections.
 * `beh_offsets` is a host int32 array [n_req + 1], offsets[0] == 0, strictly
 * increasing (every request needs >= 1 row, else TXS_ERR_COLD_START).
 * `capacity_extra` >= 0 spare rows per request are reserved for appends.
 * Allocates the cache (device memory) and returns it in *out.
 */
txs_status txs_build_kv_cache(txs_model* model, int32_t n_req, const int32_t* beh_offsets,
                              const void* beh_enc, int32_t capacity_extra, void* stream,
                              txs_kv_cache** out);
void txs_cache_destroy(txs_kv_cache* cache);

/*
 * txs_rebuild_kv_cache — nearline refresh in place (App. D, time-based batch
 * re-encoding): recompute every request of an existing cache from new rows,
 * exactly as txs_build_kv_cache would, reusing its memory (no allocation).
 * n_req must equal the cache's; each new L_r must be >= 1 (else
 * TXS_ERR_COLD_START) and fit the request's capacity from the original build
 * (else TXS_ERR_CAPACITY; nothing is changed).
 */
txs_status txs_rebuild_kv_cache(txs_model* model, txs_kv_cache* cache, int32_t n_req, const int32_t* beh_offsets,
                                const void* beh_enc, void* stream);

/*
 * txs_append_behavior — incremental update (App. D, incremental-encoding
 * remark): rows new_enc[new_offsets[r] .. new_offsets[r+1]) (device, model
 * dtype, [sum dL_r, d_model]) are projected into the free slots after request
 * r's current rows; existing rows are untouched; the pooled anchor is merged
 * with the new rows (online softmax) and re-projected.  dL_r may be 0.
 * `new_offsets` host int32 [n_req + 1]; n_req must equal the cache's.
 * Errors: TXS_ERR_CAPACITY if any request would exceed its capacity (nothing
 * is changed), TXS_ERR_STALE_CACHE, TXS_ERR_INVALID_ARG.
 */
txs_status txs_append_behavior(txs_model* model, txs_kv_cache* cache, int32_t n_req,
                               const int32_t* new_offsets, const void* new_enc, void* stream);

/*
 * txs_rebuild_append_kv_cache — txs_rebuild_kv_cache from beh_offsets /
 * beh_enc followed by txs_append_behavior of new_offsets / new_enc, in one
 * call (App. D: the batch re-encode and the streamed tail since it).  The
 * result is exactly that of the two calls; the anchor's projections are
 * computed once, after the append.  Capacity is checked for the sum before
 * anything is enqueued.
 */
txs_status txs_rebuild_append_kv_cache(txs_model* model, txs_kv_cache* cache, int32_t n_req,
                                       const int32_t* beh_offsets, const void* beh_enc,
                                       const int32_t* new_offsets, const void* new_enc, void* stream);

/* Copy rows row0 .. row0+n_rows-1 of request `req`'s cached K (which = 0) or
 * V (which = 1) of layer `layer` into dst (device, model dtype, [n_rows, dkv]),
 * asynchronously on `stream`.  Rows must be < the request's current length. */
txs_status txs_cache_read_rows(const txs_kv_cache* cache, int32_t layer, int32_t which, int32_t req, int32_t row0,
                               int32_t n_rows, void* dst, void* stream);
/* Copy the anchor's projected key (which = 0) or value (which = 1) of `layer`
 * for all requests (device, float, [n_req, dkv]), or the pooled anchor g
 * itself (which = 2, layer ignored; [n_req, d]) into dst. */
txs_status txs_cache_read_anchor(const txs_kv_cache* cache, int32_t layer, int32_t which, float* dst, void* stream);

/*
 * Cache export / import (App. D cache management: warm start from a
 * persisted cache; entries versioned by the model identifier and the feature
 * schema, stale entries never reused).  The host blob holds a header (format
 * version, model hash, schema_version, sizes), the request lengths, each
 * layer's cached K and V rows (current lengths only, not spare capacity), the
 * pooling state and the anchor with its per-layer projections.
 *
 * txs_cache_export_size: bytes of the blob of `cache`.
 * txs_cache_export: writes the blob into host_buf (caller-owned, >= that many
 *   bytes); synchronises `stream` before returning.
 * txs_cache_import: builds a new cache from a blob for `model`, with
 *   capacity_extra spare rows per request; scores, appends and reads of it
 *   give exactly what the exported cache gave.  Synchronises `stream` (the
 *   blob may be freed on return).  Errors: TXS_ERR_STALE_CACHE if the blob
 *   was written for another model hash or schema_version, TXS_ERR_INVALID_ARG
 *   for a blob that is not one (bad magic or format, truncated, inconsistent).
 */
txs_status txs_cache_export_size(const txs_kv_cache* cache, size_t* bytes);
txs_status txs_cache_export(const txs_kv_cache* cache, uint32_t schema_version, void* host_buf, size_t bytes,
                            void* stream);
txs_status txs_cache_import(txs_model* model, uint32_t schema_version, const void* host_buf, size_t bytes,
                            int32_t capacity_extra, void* stream, txs_kv_cache** out);

/* Current per-request lengths L_r (host int32 [n_req]) and request count. */
txs_status txs_cache_lengths(const txs_kv_cache* cache, int32_t* out_len);
int32_t txs_cache_n_req(const txs_kv_cache* cache);

/*
 * txs_score_workspace_size — bytes of device scratch txs_score_candidates needs
 * for n_req requests with total_cand candidates in all (256-byte aligned start).
 */
txs_status txs_score_workspace_size(const txs_model* model, int32_t n_req, int64_t total_cand,
                                    size_t* bytes);

/*
 * txs_score_candidates — multi-candidate next-action decoding against the
 * cache (Sec. 4.1.2 multi-query cross-attention sharing K/V across the m
 * candidates; Sec. 4.1.3 parallel grouped decoding and the action softmax).
 *
 * Request r has candidates cand_tok[cand_offsets[r] .. cand_offsets[r+1])
 * (device, model dtype, [sum M_r, d_model]; M_r >= 0) and n_ctx context tokens
 * ctx_tok[r] (device, [n_req, n_ctx, d_model]; may be NULL iff n_ctx == 0).
 * Every decoder layer runs serving-stream attention (context rows attend to
 * the context rows, a candidate to the context rows and itself), cross-
 * attention to the cached key set, and the FFN, each post-LN with a residual.
 * Outputs (device, float, [sum M_r, n_actions]): out_logits = Q_dec k_dec with
 * k_dec = [z, x] W_dec + b_dec, and out_probs = softmax(out_logits) (may be NULL).
 * `workspace` (device, >= txs_score_workspace_size bytes, 256-byte aligned)
 * is scratch owned by the caller; its contents are overwritten.
 * `cand_offsets` host int32 [n_req + 1]; n_req must equal the cache's.
 * Errors: TXS_ERR_STALE_CACHE if the cache came from a model with another hash.
 */
txs_status txs_score_candidates(txs_model* model, const txs_kv_cache* cache, int32_t n_req,
                                const int32_t* cand_offsets, const void* cand_tok,
                                const void* ctx_tok, void* workspace, size_t workspace_bytes,
                                float* out_logits, float* out_probs, void* stream);

/*
 * txs_score_candidates_after — txs_score_candidates for a cache that may still
 * be being written (rebuilt or appended) on another stream.  The work that
 * does not read the cache (packing, and in the first layer the serving-stream
 * attention, its output projection and the query projection) is enqueued on
 * `stream` at once; `stream` then waits on `cache_ready` (a cudaEvent_t
 * recorded on the writing stream after its last cache call, passed as void*)
 * before the first cross-attention, so that prefix overlaps the cache write.
 * cache_ready == NULL gives txs_score_candidates.  The host-side cache state
 * (lengths) must already be that of the writes the event covers, i.e. the
 * cache calls are issued first.  The caller also orders any later write of
 * the cache after this call's reads (an event recorded on `stream`).
 */
txs_status txs_score_candidates_after(txs_model* model, const txs_kv_cache* cache, int32_t n_req,
                                      const int32_t* cand_offsets, const void* cand_tok, const void* ctx_tok,
                                      void* workspace, size_t workspace_bytes, float* out_logits,
                                      float* out_probs, void* cache_ready, void* stream);

/*
 * txs_events_workspace_size — bytes of device scratch txs_score_events needs
 * for n_events events with total_cand candidates in all, the longest event
 * prefix being max_event_end rows.
 */
txs_status txs_events_workspace_size(const txs_model* model, int32_t n_events, int64_t total_cand,
                                     int32_t max_event_end, size_t* bytes);

/*
 * txs_score_events — streaming multi-event scoring of one user (Sec. 4.2,
 * causal attention and prefix reuse: each serving event slices the behavior
 * prefix before it; Sec. 5.1, a global token pooled for each event timestamp).
 *
 * `user` selects a request of `cache` whose rows hold the whole behavior
 * stream; beh_enc (device, model dtype, [L_user, d_model]) are the encoded
 * rows the cache was built (and appended) from, in order.  Event t sees the
 * first event_ends[t] rows only (1 <= event_ends[t] <= L_user, host int32
 * [n_events], any order): its key set is the most recent l_local of those
 * rows plus the anchor pooled over them (LOCAL_GLOBAL), or all of them
 * (FULL).  Event t's candidates are cand_tok[cand_offsets[t] ..
 * cand_offsets[t+1]) (device, [sum m_t, d_model]) and its context tokens
 * ctx_tok[t] (device, [n_events, n_ctx, d_model]; NULL iff n_ctx == 0).
 * Outputs as for txs_score_candidates, packed by cand_offsets (host int32
 * [n_events + 1]).  The cached K/V rows are reused, not recomputed; the
 * per-event anchors are pooled from beh_enc into `workspace` (device, >=
 * txs_events_workspace_size bytes, 256-byte aligned, caller-owned).
 * Errors: TXS_ERR_COLD_START for an event end of 0, TXS_ERR_INVALID_ARG for
 * an end beyond the user's rows or a bad argument, TXS_ERR_STALE_CACHE,
 * TXS_ERR_UNSUPPORTED for more than 4096 events or d_model > 512.
 */
txs_status txs_score_events(txs_model* model, const txs_kv_cache* cache, int32_t user, const void* beh_enc,
                            int32_t n_events, const int32_t* event_ends, const int32_t* cand_offsets,
                            const void* cand_tok, const void* ctx_tok, void* workspace, size_t workspace_bytes,
                            float* out_logits, float* out_probs, void* stream);

/*
 * txs_rank_candidates — per request, candidate indices (local to the request)
 * sorted by descending probs[:, action]; ties go to the lower index and NaN
 * scores rank last.  `probs` device float [sum M_r, n_actions].
 * top_k == 0: out_idx is device int32 [sum M_r], request r's ranking at
 * out_idx[cand_offsets[r] ...].  top_k > 0: out_idx is [n_req, top_k], padded
 * with -1 when M_r < top_k.  Requires M_r <= 32768.
 */
txs_status txs_rank_candidates(int32_t n_req, const int32_t* cand_offsets, const float* probs,
                               int32_t n_actions, int32_t action, int32_t top_k, int32_t* out_idx,
                               void* stream);

/*
 * txs_pool_anchor_static — the attention-pooled anchor g of each request (the
 * value txs_build_kv_cache keeps and txs_cache_read_anchor returns with
 * which = 2), computed without allocating any memory.  The paper has no
 * counterpart: this entry point is for callers that cannot allocate device
 * memory while serving (a process that reserves its GPU memory up front and
 * forbids driver allocations afterwards, a plugin inside another runtime with
 * no allocator of its own, a path that cannot take the implicit device
 * synchronisation of cudaMalloc/cudaFree).
 *
 * Inputs as for txs_build_kv_cache: `beh_offsets` host int32 [n_req + 1],
 * strictly increasing from 0 (an empty request returns TXS_ERR_COLD_START),
 * `beh_enc` device rows [sum L_r, d_model] in the model dtype.  Output:
 * `out_g` device float [n_req, d_model].  The call itself never calls
 * cudaMalloc, cudaFree or any allocating routine.
 *
 * Scratch: a 4 MiB file-scope device array of the library (held on every GPU
 * that loads it until the process exits) — n_req * 16 * (d_model + 2) floats
 * must fit in 1,048,576 (d_model = 512: up to 127 requests), n_req <= 1024 and
 * d_model <= 512; larger calls return TXS_ERR_UNSUPPORTED (txs_last_error says
 * why) before anything is enqueued.  Every call overwrites all scratch it
 * reads, and all calls share that one array: calls that overlap on the GPU
 * (other streams, other threads) race and must be serialised by the caller.
 * Each call looks up the array's device address in the current device's
 * context (cudaGetSymbolAddress, which allocates nothing); make the first call
 * on a device before any stream capture.
 */
txs_status txs_pool_anchor_static(const txs_model* model, int32_t n_req, const int32_t* beh_offsets,
                                  const void* beh_enc, float* out_g, void* stream);

/* ------------------------------------------------------------------ behavior encoder
 *
 * The behavior-stream encoder Phi_behavior (Sec. 4.1.1; two layers in the
 * paper's setup, Sec. 5.1) and its incremental update (App. D,
 * incremental-encoding remark).  Its outputs are the encoded rows Phi_b that
 * txs_build_kv_cache / txs_append_behavior take.
 *
 * Token of behavior i: x_i = [s_i, E_type[type_i]], s_i the subject
 * embedding (width d_model - type_dim, given) and E_type the behavior-type
 * table.  Each layer, post-LN with residuals:
 *   [q|k|v] = X W_qkv + b_qkv
 *   a_i (head h) = sum_j softmax_j(q_i.k_j / sqrt(d_h) + beta_h[min(i-j, R-1)]) v_j
 *     over the visible j: j <= i, and i - j < window when window > 0
 *   H = LN1(X + A W_o + b_o);  Y = LN2(H + GELU(H W_1 + b_1) W_2 + b_2)
 * The mask is causal and the bias depends only on i - j, so appending tokens
 * leaves the earlier outputs unchanged: an append runs the layers for the new
 * tokens only, against each layer's cached keys/values of the earlier tokens
 * (the encoder state), and gives the same rows, bit for bit, as encoding the
 * whole stream at once.
 */
typedef struct {
  int32_t d_model;   /* d; multiple of 64 for TXS_BF16, of 32 for TXS_FP32; <= 512  */
  int32_t n_heads;   /* H; d_head = d_model / n_heads must be 32 or 64             */
  int32_t d_ff;      /* F; multiple of 64, <= 16384                                */
  int32_t n_layers;  /* encoder layers, 1..16                                      */
  int32_t type_dim;  /* d_t, 0 <= d_t < d_model; subject rows are d_model - d_t wide */
  int32_t n_types;   /* rows of E_type (>= 1 when type_dim > 0)                    */
  int32_t n_rel;     /* R relative-bias entries per head, 1..65536                 */
  int32_t window;    /* 0: every earlier token is visible; w > 0: the w most recent
                        (the token itself included)                                */
  int32_t dtype;     /* txs_dtype                                                  */
  float ln_eps;      /* LayerNorm epsilon (> 0)                                    */
} txs_enc_config;

typedef struct txs_encoder txs_encoder;     /* opaque */
typedef struct txs_enc_state txs_enc_state; /* opaque: per-user K/V of every layer */

#define TXS_ENC_WEIGHTS_PER_LAYER 13

/*
 * txs_encoder_create — copy the encoder weights into the library's layout.
 * `weights` (host array of device pointers, config dtype) holds, per layer:
 *    0 W_qkv [d,3d]  1 b_qkv [3d]  2 rel_bias [H,R]  3 W_o [d,d]  4 b_o [d]
 *    5 ln1_g [d]     6 ln1_b [d]   7 W_1 [d,F]       8 b_1 [F]    9 W_2 [F,d]
 *   10 b_2 [d]      11 ln2_g [d]  12 ln2_b [d]
 * then, when type_dim > 0, E_type [n_types, type_dim].  Synchronises the
 * device first and returns after the copies; keeps a content hash.
 * Errors: TXS_ERR_INVALID_ARG, TXS_ERR_UNSUPPORTED, TXS_ERR_CUDA.
 */
txs_status txs_encoder_create(const txs_enc_config* cfg, const void* const* weights, txs_encoder** out);
void txs_encoder_destroy(txs_encoder* enc);
uint64_t txs_encoder_hash(const txs_encoder* enc);

/* Bytes of device scratch one encode call over n_rows tokens needs. */
txs_status txs_encoder_workspace_size(const txs_encoder* enc, int64_t n_rows, size_t* bytes);

/*
 * txs_encode_build — encode each user's behavior stream from its first token
 * and create the encoder state.  User r's tokens are rows offsets[r] ..
 * offsets[r+1] of `subj` (device, config dtype, [n, d_model - type_dim]) and
 * `types` (device int32 [n]; may be NULL iff type_dim == 0); `offsets` is a
 * host int32 array [n_req + 1], non-decreasing from 0 (a user may have no
 * tokens yet).  Writes Phi_b to phi_out (device, config dtype, [n, d_model])
 * and keeps every layer's K/V rows, with capacity_extra >= 0 spare rows per
 * user for appends.  `workspace`: device, >= txs_encoder_workspace_size(n)
 * bytes, 256-byte aligned, caller-owned.  A type id outside [0, n_types)
 * latches TXS_ERR_BOUNDS in the encoder's device status.
 */
txs_status txs_encode_build(txs_encoder* enc, int32_t n_req, const int32_t* offsets, const void* subj,
                            const int32_t* types, int32_t capacity_extra, void* workspace, size_t workspace_bytes,
                            void* phi_out, void* stream, txs_enc_state** out);

/*
 * txs_encode_append — incremental encoding (App. D remark): user r's new
 * tokens, rows new_offsets[r] .. new_offsets[r+1] of subj/types (as above;
 * zero new tokens allowed), are encoded after that user's current tokens;
 * their Phi_b rows go to phi_out (device, [sum new, d_model]).  Earlier rows
 * and their K/V are not touched.  n_req must equal the state's.
 * Errors: TXS_ERR_CAPACITY if a user would exceed its capacity (nothing is
 * changed), TXS_ERR_STALE_CACHE if the state came from another encoder,
 * TXS_ERR_INVALID_ARG.
 */
txs_status txs_encode_append(txs_encoder* enc, txs_enc_state* state, int32_t n_req, const int32_t* new_offsets,
                             const void* subj, const int32_t* types, void* workspace, size_t workspace_bytes,
                             void* phi_out, void* stream);

/* Per-user token counts (host int32 [n_req]) and user count of a state. */
txs_status txs_enc_state_lengths(const txs_enc_state* state, int32_t* out_len);
int32_t txs_enc_state_n_req(const txs_enc_state* state);
/* Copy rows row0 .. row0+n_rows-1 of user `req`'s cached keys (which = 0) or
 * values (which = 1) of encoder layer `layer` into dst (device, config dtype,
 * [n_rows, d_model]), asynchronously on `stream`. */
txs_status txs_enc_state_read_rows(const txs_enc_state* state, int32_t layer, int32_t which, int32_t req,
                                   int32_t row0, int32_t n_rows, void* dst, void* stream);
void txs_enc_state_destroy(txs_enc_state* state);
/* Synchronise the device, read and clear the encoder's latched device status. */
txs_status txs_encoder_device_status(txs_encoder* enc);

/* Synchronise the device, read and clear the model's latched device status. */
txs_status txs_device_status(txs_model* model);

/* Self-test of the device-side failure path (no paper counterpart): enqueue
 * on `stream` one kernel whose bounded wait, the same wait every pipeline
 * of the library uses, runs out (about a second: nothing ever arrives at
 * its barrier).  The kernel then latches TXS_ERR_DEVICE_TIMEOUT into the
 * model's status word and returns; no fault, the context stays usable.  A
 * following txs_device_status(model) returns TXS_ERR_DEVICE_TIMEOUT and
 * clears the word.  Errors: TXS_ERR_INVALID_ARG (null model), TXS_ERR_CUDA. */
txs_status txs_selftest_wait_timeout(txs_model* model, void* stream);

/* The GELU of the FFN epilogues, element-wise on device float arrays x -> y
 * of n elements, for tests of its accuracy (no paper counterpart; the
 * activation is the exact erf form 0.5 x (1 + erf(x / sqrt 2))).  variant 0:
 * the bf16 tensor-core epilogues' evaluation (erf by Abramowitz & Stegun
 * 7.1.26, absolute error <= 1.5e-7); variant 1: the fp32 path's (erff).
 * Asynchronous on `stream`.  Errors: TXS_ERR_INVALID_ARG, TXS_ERR_CUDA. */
txs_status txs_gelu_eval(const float* x, float* y, int64_t n, int32_t variant, void* stream);

/* Process-wide per-kernel-class timing with CUDA events on the launching
 * stream (off by default).  While enabled, every library launch is bracketed
 * by two events; txs_profile_collect synchronises, writes per-class total
 * milliseconds and launch counts (host arrays of length n >=
 * TXS_N_KERNEL_CLASSES) and clears the record.  Not thread-safe; not for use
 * during CUDA-graph capture. */
#define TXS_N_KERNEL_CLASSES 24
txs_status txs_profile_enable(int32_t enable);
txs_status txs_profile_collect(double* total_ms, int64_t* launches, int32_t n);
const char* txs_kernel_class_name(int32_t cls);

const char* txs_status_string(txs_status s);
/* Text of the last host-side failure of this thread (a CUDA error string or
 * the config field that was rejected); empty if none. */
const char* txs_last_error(void);
const char* txs_version(void);

#ifdef __cplusplus
}
#endif
#endif /* TXS_H */
