/*
 * compresskv.h -- C ABI of the CompressKV prefill-end KV-cache compression
 * path on one GB300 (sm_103a).
 *
 * The method (CompressKV, Sec. 3.3 "Token Selection Driven by Semantic
 * Retrieval Heads", with the SnapKV-style local setting of Sec. 4
 * "Implementation Details"): for every sequence s and GQA KV group g of a
 * layer (a *unit*),
 *   1. score each prefix token j < n = L_s - W by the causal softmax
 *      attention of the last W prompt queries of the group's Semantic
 *      Retrieval Heads (SRH; the SRH mask is an input, identified offline per
 *      Sec. 3.2), summed over the window queries and the SRH heads;
 *   2. smooth the scores with 1-D average pooling of width P over tokens;
 *   3. keep the k = min(B, L_s) - W prefix tokens with the largest pooled
 *      score (ties to the lower position) plus the W window tokens, where B is
 *      the layer's budget from the offline layer-wise allocation (Sec. 3.4);
 *   4. gather the retained K and V rows into a contiguous compressed cache.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All tensor arguments are DEVICE pointers unless marked "host".  The
 *   caller allocates and frees every buffer, including the workspace; the
 *   library allocates no device memory, keeps no per-call global state and
 *   never synchronises the stream (except compresskv_read_device_status).
 * - Work is enqueued on `stream` (a cudaStream_t, NULL = legacy default).
 *   Entry points return after enqueueing; results are ready when the stream
 *   reaches them.  Argument errors are detected on the host before anything
 *   is enqueued; launch failures return CKV_ERR_CUDA.  Errors found by a
 *   kernel (a bounded wait that ran out, an index out of range passed to
 *   compresskv_gather) are written to the status word at the start of the
 *   workspace and read with compresskv_read_device_status.
 * - Sequences are packed: sequence s owns rows cu_seqlens[s] ..
 *   cu_seqlens[s+1]-1 of K and V (host array of batch+1 ints, first entry 0).
 *   L_s = cu_seqlens[s+1] - cu_seqlens[s], n_s = max(L_s - W, 0).
 * - K, V: [T][num_kv_heads][head_dim] elements of `dtype`, head_dim contiguous,
 *   element strides kv_token_stride / kv_head_stride (multiples of 8, base
 *   16-byte aligned).  V shares K's strides.  V (read only by the gather)
 *   may also live in page-locked host memory (cudaHostAlloc /
 *   cudaHostRegister), which the device reads through unified addressing:
 *   only the retained rows then cross the host link.  Pageable host memory
 *   is refused with CKV_ERR_INVALID_ARG (checked with
 *   cudaPointerGetAttributes before anything is enqueued).
 * - Window queries q_win: element (s, h, w, :) at
 *   q_win + s*q_batch_stride + h*q_head_stride + w*q_win_stride, head_dim
 *   contiguous; row w is the query of prompt position L_s - W + w.
 *   Strides are multiples of 8 elements, base 16-byte aligned.  Q and K are
 *   taken as given (post-RoPE); no RoPE is applied.
 * - GQA grouping: query head h belongs to KV group h / (num_q_heads /
 *   num_kv_heads).
 * - Prefix-score layout ("score layout"): float [num_kv_heads][P_total],
 *   P_total = sum_s n_s, sequence s at offset cu_prefix[s] = sum_{s'<s} n_s'.
 * - Output layout: kept_s = min(budget_s, L_s) tokens per sequence,
 *   cu_out[s] = sum_{s'<s} kept_s', O_total = cu_out[batch];
 *   indices: int32 [num_kv_heads][O_total], positions within the sequence in
 *   ascending order (the W window positions are the last W entries of a
 *   compressed sequence); k_out / v_out: [O_total][num_kv_heads][head_dim]
 *   contiguous, in the input dtype, bit-exact copies of the retained rows.
 * - Scores are the sum over SRH heads and window queries (the paper averages
 *   the head vectors; within a unit the head count is fixed, so the ranking
 *   is the same).
 */
#ifndef COMPRESSKV_H_
#define COMPRESSKV_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes returned by every entry point (and stored by kernels in the
 * workspace status word). */
enum {
  CKV_OK = 0,
  CKV_ERR_INVALID_ARG = -1,     /* null pointer, bad shape/stride/alignment */
  CKV_ERR_UNSUPPORTED = -2,     /* valid but outside what the kernels take (see limits) */
  CKV_ERR_BUDGET = -3,          /* a budget smaller than the window W */
  CKV_ERR_EMPTY_SRH_GROUP = -4, /* a KV group with no SRH head but a sequence to score */
  CKV_ERR_WORKSPACE = -5,       /* workspace null or smaller than compresskv_workspace_size */
  CKV_ERR_CUDA = -6,            /* a CUDA runtime call or kernel launch failed */
  CKV_ERR_DEVICE_TIMEOUT = -7,  /* a kernel's bounded wait ran out (device status only) */
  CKV_ERR_DEVICE_INDEX = -8,    /* an index outside its sequence: given to compresskv_gather, or
                                   produced by a selection (a device self-check) */
  CKV_ERR_STATIC_SCRATCH = -9   /* problem needs more than CKV_STATIC_SCRATCH_BYTES of scratch */
};

/* Size of the scratch built into the library for
 * compresskv_compress_layer_noalloc (every GPU that loads the library holds
 * it until the process exits). */
#define CKV_STATIC_SCRATCH_BYTES (16u * 1024u * 1024u)

enum { CKV_DTYPE_F16 = 0, CKV_DTYPE_BF16 = 1 };
/* Pooling across the token dimension (Sec. 3.3, width P of Sec. 4).  AVG:
 * average pooling of the heads' summed window scores (divisor P, zero
 * padding; linear, so the order of pooling and head sum does not matter).
 * MAX: each SRH head's window-summed attention is max-pooled over
 * [j - r, j + r] within the prefix, then the heads' pooled vectors are
 * summed (pooling before the head sum, the paper's order).  MAX is taken by
 * compresskv_compress_layer(s) and compresskv_compress_layer_noalloc (both
 * selection scopes; the heads are scored one SRH head per group at a time,
 * then pooled and selected; the workspace holds one more raw-score row per
 * head of a group) and by compresskv_score (raw scores do not depend on it);
 * compresskv_select (its input is already summed over the heads), the
 * given-LSE and the head-budget calls return CKV_ERR_UNSUPPORTED for it. */
enum { CKV_POOL_AVG = 0, CKV_POOL_MAX = 1 };
/* Selection scope.  PER_GROUP: every KV group keeps the tokens its own SRH
 * heads rank highest, and a group without an SRH head is an error.
 * PER_LAYER (Sec. 3.3 read literally: all heads of a layer share one set of
 * retained tokens chosen by the layer's SRH heads, whose pooled scores are
 * averaged): per sequence, the pooled scores of all groups are summed (a
 * group without an SRH head adds nothing), one top-k is taken and every KV
 * group keeps the same positions. */
enum { CKV_SELECT_PER_GROUP = 0, CKV_SELECT_PER_LAYER = 1 };

/* Kernel kinds reported through ckv_trace. */
enum {
  CKV_KERNEL_SCORE = 1,         /* window logits over K: softmax statistics + exponent table */
  CKV_KERNEL_COMBINE = 2,       /* normalised scores summed over queries, then pooled */
  CKV_KERNEL_SELECT = 3,        /* pooling + top-k + window append */
  CKV_KERNEL_GATHER = 4,        /* retained K/V rows -> compressed cache */
  CKV_KERNEL_FUSED = 5          /* all four steps for every unit of a call, one persistent kernel */
};

/* Optional launch trace.  When ckv_problem.trace is non-null every kernel
 * launch is bracketed by two caller-created CUDA events (cudaEvent_t handles
 * in `events`, 2 per launch) recorded on the call's stream, and its kind is
 * stored in `kinds`.  Inside a stream capture the events are recorded as
 * external event nodes.  Once `count` reaches `capacity` further launches
 * are only counted.  The caller zeroes `count` and `launches`. */
typedef struct ckv_trace {
  void** events;       /* [2*capacity] cudaEvent_t */
  int32_t* kinds;      /* [capacity] host */
  int32_t capacity;
  int32_t count;       /* launches recorded so far */
  int64_t launches;    /* kernels launched so far */
} ckv_trace;

/* One layer's problem description (host memory). */
typedef struct ckv_problem {
  int32_t batch;            /* sequences, 1..512 */
  int32_t num_q_heads;      /* H_q, 1..256, a multiple of num_kv_heads */
  int32_t num_kv_heads;     /* H_kv, 1..64 */
  int32_t head_dim;         /* d; 128 */
  int32_t window;           /* W >= 1, the observation window (Sec. 4) */
  int32_t pool_width;       /* P, odd, 1..63, pooling width (Sec. 4) */
  int32_t dtype;            /* CKV_DTYPE_F16 | CKV_DTYPE_BF16 for Q, K and V */
  int32_t pool_kind;        /* CKV_POOL_AVG | CKV_POOL_MAX */
  float scale;              /* softmax scale; 0 selects 1/sqrt(head_dim) */
  int32_t selection;        /* CKV_SELECT_PER_GROUP or CKV_SELECT_PER_LAYER */
  const int32_t* cu_seqlens;/* host [batch+1] */
  int64_t kv_token_stride;  /* elements between consecutive tokens of K/V */
  int64_t kv_head_stride;   /* elements between KV heads of K/V */
  int64_t q_batch_stride;   /* elements, window queries */
  int64_t q_head_stride;
  int64_t q_win_stride;
  ckv_trace* trace;         /* optional launch trace, NULL for none */
} ckv_problem;

/* Bytes of device workspace the calls below need for problem `p` (depends
 * on the shapes and cu_seqlens only; an upper bound over every SRH mask).
 * Returns 0 if `p` is invalid. */
size_t compresskv_workspace_size(const ckv_problem* p);

/* Zero the workspace header -- the status word and the work counters the
 * kernels share between their CTAs (about 390 KB, enqueued on `stream`).
 * Call once after allocating a workspace, and after reading a non-zero
 * device status (an aborted call can leave the counters set); every call
 * that completes leaves them zero. */
int compresskv_workspace_init(void* workspace, size_t workspace_bytes, void* stream);

/* Host-only: per-sequence offsets of the prefix scores (cu_prefix, [batch+1])
 * and of the compressed output (cu_out, [batch+1]) for the given host
 * budgets ([batch]).  Either output may be NULL.  Returns CKV_ERR_BUDGET if a
 * budget is below W. */
int compresskv_output_layout(const ckv_problem* p, const int32_t* budgets,
                             int32_t* cu_prefix, int32_t* cu_out);

/* Step 1 (Sec. 3.3): raw prefix scores.
 * srh_mask: host uint8 [num_q_heads], non-zero = SRH head of this layer.
 * raw_scores: device float, score layout, written for every prefix token.
 * The per-query attention weights pass through an fp16 table scaled so
 * that each weight keeps a relative error below 2^-11 (plus the fp32 sums).
 * Per unit, |S_g| * W must not exceed 256 query rows (CKV_ERR_UNSUPPORTED). */
int compresskv_score(const ckv_problem* p, const void* q_win, const void* k,
                     const uint8_t* srh_mask, float* raw_scores,
                     void* workspace, size_t workspace_bytes, void* stream);

/* Steps 2-3 (Sec. 3.3, Sec. 4): average pooling of width P, top-k of the
 * pooled prefix scores, window append.
 * budgets: host int32 [batch] (per sequence, including the W window tokens).
 * indices: device int32 [num_kv_heads][O_total] (output layout).
 * cu_out: host int32 [batch+1], written.
 * pooled_scores: optional device float in score layout (NULL for none;
 *   must be NULL under CKV_SELECT_PER_LAYER, whose keys are the pooled sum
 *   of all groups' raw scores).
 * Under CKV_SELECT_PER_LAYER every group's row of `indices` receives the
 * sequence's shared selection. */
int compresskv_select(const ckv_problem* p, const float* raw_scores,
                      const int32_t* budgets, int32_t* indices, int32_t* cu_out,
                      float* pooled_scores, void* workspace, size_t workspace_bytes,
                      void* stream);

/* Step 4 (Sec. 3.3): copy the retained K/V rows.
 * indices / cu_out as produced by compresskv_select (cu_out on the host);
 * an index outside [0, L_s) is skipped and reported as CKV_ERR_DEVICE_INDEX
 * in the device status of `workspace` (which may be NULL to skip
 * reporting). */
int compresskv_gather(const ckv_problem* p, const int32_t* indices, const int32_t* cu_out,
                      const void* k, const void* v, void* k_out, void* v_out,
                      void* workspace, void* stream);

/* Steps 1-4 fused for one layer: score, select, gather.
 * raw_scores / pooled_scores are optional outputs in score layout (NULL: raw
 * scores are not materialised, pooled scores stay in the workspace); they are
 * per group in both selection scopes (a group without an SRH head gets
 * zeros under CKV_SELECT_PER_LAYER), and the per-layer selection ranks their
 * sum over the groups.
 * cu_out: host int32 [batch+1], written. */
int compresskv_compress_layer(const ckv_problem* p, const void* q_win, const void* k,
                              const void* v, const uint8_t* srh_mask, const int32_t* budgets,
                              int32_t* indices, int32_t* cu_out, void* k_out, void* v_out,
                              float* raw_scores, float* pooled_scores,
                              void* workspace, size_t workspace_bytes, void* stream);

/* compresskv_compress_layer for several layers in one call (prefill-end
 * compression of a model: every layer's cache exists, Sec. 3; each layer
 * selects with its own SRH heads, Sec. 3.3).  The batch of `p` packs n_masks blocks of
 * batch / n_masks sequences and sequence s uses SRH mask s / (batch /
 * n_masks): with a KV cache laid out [n_layers][T][H_kv][d], viewed as
 * [n_layers*T][H_kv][d] with cu_seqlens repeated per layer (offset by l*T),
 * and window queries [n_layers][B][H_q][W][d] viewed as
 * [n_layers*B][H_q][W][d], block l is layer l.  One launch of each kernel
 * then covers all the layers' units, so the scoring kernel's start-up and
 * tail are paid once.
 * Under CKV_SELECT_PER_GROUP every step of every unit (scoring, normalising
 * and pooling, top-k, window, gather) runs in one persistent kernel
 * (CKV_KERNEL_FUSED): one CTA per SM streams K from the first layer to the
 * last while other warps of the same CTAs merge, select and gather the units
 * whose scores are complete.  It reads K twice per chunk of 16 tiles of 128
 * keys: a first pass sums each query row's exponentials (softmax statistics
 * of the chunk), and once every chunk of the unit is in and the row's
 * denominator merged, a second pass sums the normalised probabilities of
 * each key (Eq. 1-2) in fp32 from K read again (for long calls mostly from
 * DRAM: the step then moves about twice the bytes of K); no exponent table
 * is stored.  The chunk grid is fixed per unit and every chunk's statistics
 * restart, so the scores depend only on the unit itself: compressing a layer
 * alone or among others gives the same bits.  That kernel takes windows W
 * that are multiples of 16, query strides that are multiples of 8 elements,
 * at most 32 query heads per group and SRH lists of at most 192 query rows
 * (|S_g| W: two Q buffers of them beside a ring of two K tiles fill its
 * shared memory); other per-group problems use the separate kernels.
 * n_masks: 1 <= n_masks, dividing batch (else CKV_ERR_INVALID_ARG); at most
 *   256 under CKV_SELECT_PER_GROUP and 4 under CKV_SELECT_PER_LAYER (or when
 *   the separate kernels run) (else CKV_ERR_UNSUPPORTED).
 * srh_masks: host uint8 [n_masks][num_q_heads].
 * budgets, cu_out and every output follow the packed batch (sequence
 * l*B + s is sequence s of block l); the workspace is sized for `p`.
 * With n_masks = 1 this is compresskv_compress_layer. */
int compresskv_compress_layers(const ckv_problem* p, int n_masks, const void* q_win,
                               const void* k, const void* v, const uint8_t* srh_masks,
                               const int32_t* budgets, int32_t* indices, int32_t* cu_out,
                               void* k_out, void* v_out, float* raw_scores, float* pooled_scores,
                               void* workspace, size_t workspace_bytes, void* stream);

/* compresskv_compress_layer when the softmax denominators of the window
 * queries are already known -- a prefill attention kernel has them as its
 * log-sum-exp (CompressKV's latency study, Sec. 4.4, runs on a
 * FlashAttention prefill; no separate normaliser pass is then needed).
 * lse_win: device float, natural-log LSE of each window query's causal
 *   softmax over keys j <= L_s - W + w with the problem's scale: element
 *   (s, h, w) at lse_win + s*lse_batch_stride + h*lse_head_stride + w (4-byte
 *   aligned; only SRH heads are read).  It must be device (or managed) memory
 *   of the current device covering every (s, h, w) of the batch: host memory
 *   is refused with CKV_ERR_INVALID_ARG.  Scores are then exp(z - LSE) summed
 *   in fp32 straight from the logits (no fp16 table), so their accuracy is
 *   the given LSE's.  Other arguments as for compresskv_compress_layer
 *   (pooled_scores must be NULL under CKV_SELECT_PER_LAYER). */
int compresskv_compress_layer_lse(const ckv_problem* p, const void* q_win, const void* k,
                                  const void* v, const float* lse_win, int64_t lse_batch_stride,
                                  int64_t lse_head_stride, const uint8_t* srh_mask,
                                  const int32_t* budgets, int32_t* indices, int32_t* cu_out,
                                  void* k_out, void* v_out, float* raw_scores,
                                  float* pooled_scores, void* workspace, size_t workspace_bytes,
                                  void* stream);

/* compresskv_compress_layer_lse for several layers in one call: the packed
 * batch, the per-block SRH masks and the outputs as for
 * compresskv_compress_layers, and the window queries' LSE packed the same
 * way (element (s, h, w) of the packed batch at
 * lse_win + s*lse_batch_stride + h*lse_head_stride + w). */
int compresskv_compress_layers_lse(const ckv_problem* p, int n_masks, const void* q_win,
                                   const void* k, const void* v, const float* lse_win,
                                   int64_t lse_batch_stride, int64_t lse_head_stride,
                                   const uint8_t* srh_masks, const int32_t* budgets,
                                   int32_t* indices, int32_t* cu_out, void* k_out, void* v_out,
                                   float* raw_scores, float* pooled_scores, void* workspace,
                                   size_t workspace_bytes, void* stream);

/* compresskv_compress_layer with a budget per (sequence, KV group) -- the
 * head-level allocation CompressKV's token selection combines with (Sec.
 * 4.6, HeadKV / AdaKV style budgets, computed elsewhere).  Per-group
 * selection only (CKV_SELECT_PER_LAYER is CKV_ERR_INVALID_ARG).
 * group_budgets: host int32 [batch][num_kv_heads], each >= W (else
 *   CKV_ERR_BUDGET); unit (s, g) keeps min(budget, L_s) tokens.
 * Outputs are packed group-major: group 0's sequences, then group 1's, ...
 * cu_out: host int32 [num_kv_heads][batch+1], written: cu_out[g][s] is the
 *   first output row of (s, g) and cu_out[g][batch] the end of group g.
 * indices: device int32 [rows] (positions within the sequence, ascending
 *   per unit, window last); k_out / v_out: [rows][head_dim] in the input
 *   dtype, rows = cu_out[num_kv_heads-1][batch].
 * At most 2048 (sequence, group) pairs (CKV_ERR_UNSUPPORTED).  Other
 * arguments as for compresskv_compress_layer. */
int compresskv_compress_layer_head_budgets(const ckv_problem* p, const void* q_win,
                                           const void* k, const void* v,
                                           const uint8_t* srh_mask,
                                           const int32_t* group_budgets, int32_t* indices,
                                           int32_t* cu_out, void* k_out, void* v_out,
                                           float* raw_scores, float* pooled_scores,
                                           void* workspace, size_t workspace_bytes,
                                           void* stream);

/* compresskv_compress_layer for callers that cannot allocate device memory
 * (the paper has no counterpart; this is a deployment convenience).  Some
 * hosts own every byte of device memory and give a plugin no allocator (an
 * inference engine that pre-reserves HBM for its KV cache), and some callers
 * run where cudaMalloc is not allowed or would stall the device.  They pass
 * inputs and outputs exactly as for compresskv_compress_layer, but no
 * workspace: the scratch is a static device array of CKV_STATIC_SCRATCH_BYTES
 * inside the library, and this call allocates nothing.
 * - A problem whose compresskv_workspace_size exceeds CKV_STATIC_SCRATCH_BYTES
 *   is rejected with CKV_ERR_STATIC_SCRATCH before anything is enqueued.
 * - The first call on a device looks up the array's device address (with that
 *   device current); make that first call before any stream capture.  The
 *   address is looked up again when the device's context has changed (after
 *   cudaDeviceReset): the first call after a reset, too, belongs before any
 *   capture.
 * - Every call on a device shares the one array, which keeps the last call's
 *   contents: calls whose work may overlap on the GPU (different streams,
 *   different host threads) race and must be serialised by the caller.
 * - device_status: optional device int32; receives this call's device status
 *   word (0, or a CKV_ERR_DEVICE_* code) in stream order.  NULL skips it. */
int compresskv_compress_layer_noalloc(const ckv_problem* p, const void* q_win, const void* k,
                                      const void* v, const uint8_t* srh_mask,
                                      const int32_t* budgets, int32_t* indices, int32_t* cu_out,
                                      void* k_out, void* v_out, float* raw_scores,
                                      float* pooled_scores, int32_t* device_status,
                                      void* stream);

/* Synchronise `stream`, copy the workspace status word to *status and return
 * CKV_OK (or CKV_ERR_CUDA if the copy fails). */
int compresskv_read_device_status(const void* workspace, void* stream, int32_t* status);

/* Test hook for the failure path of the persistent per-group kernel
 * (CKV_KERNEL_FUSED): the next call that launches it runs with every bounded
 * wait limited to wait_ns (instead of 2 s), and its first CTA's claimer
 * first waits for a counter that nothing sets -- before any copy or UMMA is
 * issued -- so the wait runs out: the call stops every CTA, its device status
 * reads CKV_ERR_DEVICE_TIMEOUT, its outputs are undefined and the context
 * stays usable; compresskv_workspace_init makes the workspace usable again.
 * wait_ns: 0 cancels a pending stall, else 100000 .. 2000000000 (else
 * CKV_ERR_INVALID_ARG).  Process-wide, one-shot; not for production use. */
int compresskv_debug_stall_next_fused_call(long long wait_ns);

/* Error-aware layer budgets (Sec. 3.4: the offline per-layer eviction
 * errors, normalised as in Eq. 4, share the total budget after every layer
 * gets a minimum m, no layer above a maximum M; Sec. 4 uses m = 32 and
 * M = 3 * B_total / L).  Host only: no device work, no stream.
 * layer_errors: host double [n_layers], e^(l) >= 0 in any common scale.
 * total_budget: B_total, retained KV pairs summed over the layers.
 * min_budget, max_budget: m and M; max_budget <= 0 selects 3*B_total/L.
 * budgets: host int32 [n_layers], written: m plus the water-filled share
 *   (a layer whose proportional share would pass M - m is capped and the
 *   rest is shared again), rounded by largest remainder with ties to the
 *   lower layer, so the budgets sum to B_total exactly.
 * Returns CKV_ERR_BUDGET when n_layers*m > B_total or B_total > n_layers*M
 * (or m > M), CKV_ERR_INVALID_ARG for a null pointer, n_layers < 1 or an
 * error that is negative, NaN or infinite.  The layer budgets feed
 * compresskv_compress_layer's `budgets` (one value per sequence). */
int compresskv_allocate_layer_budgets(const double* layer_errors, int32_t n_layers,
                                      int64_t total_budget, int32_t min_budget,
                                      int32_t max_budget, int32_t* budgets);

/* Static text for a status code. */
const char* compresskv_status_string(int status);

#ifdef __cplusplus
}  /* extern "C" */
#endif

#endif  /* COMPRESSKV_H_ */
