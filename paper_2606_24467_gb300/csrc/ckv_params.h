// Kernel parameter blocks shared by the host launcher and the kernels.
// Parameters travel by value (__grid_constant__), so a launch needs no
// device-side tables and can be captured into a CUDA graph as is.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <vector_types.h>

namespace ckv {

constexpr int kHeadDim = 128;       // d: one 256-byte K row per token and group (16-bit types)
constexpr int kTileTokens = 128;    // tokens per K tile = UMMA M = TMEM lanes
constexpr int kStages = 6;          // most K tiles in flight per CTA (fewer when Q rows are large)
constexpr int kMaxQRows = 256;      // |S_g| * W rows per unit (UMMA N limit)
constexpr int kMaxBatch = 512;
constexpr int kMaxQHeads = 256;
constexpr int kMaxKvHeads = 64;
constexpr int kMaxItems = 1024;     // score work items per launch
constexpr int kMaxBudgetUnits = 2048;  // (sequence, group) pairs with their own budget
constexpr int kMaxMasks = 4;        // SRH masks per call (the layers of one multi-layer call)
constexpr int kMaxFusedMasks = 256; // ... per call of the persistent per-group kernel
constexpr int kMaxSrhGroups = kMaxMasks * kMaxKvHeads;
constexpr uint64_t kWaitTimeoutNs = 2000000000ull;  // 2 s: far above any legitimate wait

// Device status codes (mirrors of the public CKV_ERR_* values).
constexpr int CKV_DEV_ERR_TIMEOUT = -7;
constexpr int CKV_DEV_ERR_INDEX = -8;

constexpr int kTileBytes = kTileTokens * kHeadDim * 2;   // 32 KiB
constexpr int kHalfTileBytes = kTileBytes / 2;           // 64 columns (128 B) of d
constexpr int kQHalfBytes = kMaxQRows * 128;             // Q rows, one 64-column half
constexpr int kQuarters = kTileTokens / 32;              // 32-token groups per tile (one warp each)

// One work item: a contiguous range [t0, t1) of one unit -- 128-key tiles
// for the scoring kernel, 32-key quarters for the combine kernel.  `first` /
// `count` locate the unit's scoring items (whose softmax pairs the combine
// kernel merges); `eoff` / `roff` are the unit's offsets in the exponent
// table (fp16 elements) and in the reference table (floats).
struct WorkItem {
  uint16_t seq, group, t0, t1, first, count;
  uint32_t eoff, roff;
};

struct ScoreParams {
  CUtensorMap tmap_k;          // 3-D map over K: (d, kv head, token)
  const uint16_t* q;           // window queries (f16/bf16 bits)
  float2* partials;            // [n_items][kMaxQRows]: (M, S) with sum 2^(z*c) = S * 2^M
  float* bias;                 // [item of the unit's first item][kMaxQRows]: log2 D_q per unit
  int stats_only;              // 1: no exponent / reference tables (first of two passes)
  const float* lse_bias;       // given-LSE kernel: log2 D_q rows of a first pass instead of lse
  int* tickets;                // [kMaxItems]: items of the unit done (zero between calls)
  uint16_t* expo;              // fp16 2^(z*c - R) per prefix key and query row (Nr per key)
  float* refs;                 // per (tile, quarter, query row): the R used for expo
  const float* lse;            // given-LSE mode: natural-log LSE per (sequence, head, window row)
  float* raw_out;              // given-LSE mode: raw scores, score layout
  long long lse_bs, lse_hs;    // LSE strides (elements); window rows are contiguous
  int p_total;
  int cu_prefix[kMaxBatch + 1];
  int* status;                 // device status word
  long long q_bs, q_hs, q_ws;  // window-query strides, elements
  float c;                     // scale * log2(e)
  int window, num_kv_heads, n_items, is_bf16, use_evict_hint;
  int q_half_bytes;            // bytes of one 64-column half of the Q rows in shared memory
  int stages;                  // K tiles in the shared-memory ring (2..kStages)
  int epi_warps;               // 8 (two CTAs per SM) or 16 (one CTA per SM)
  int cu_seqlens[kMaxBatch + 1];
  // SRH lists: sequence s uses mask m = s / seqs_per_mask; the SRH heads of
  // its group g are srh_heads[srh_off[v] .. srh_off[v+1]), v = m*H_kv + g
  int seqs_per_mask;
  uint16_t srh_off[kMaxSrhGroups + 1];
  uint8_t srh_heads[kMaxMasks * kMaxQHeads];
  WorkItem items[kMaxItems];
};

// Combine: normalised scores from the stored exponents, then pooling.
struct CombineParams {
  const float* bias;           // per unit (row = its first scoring item): log2 D_q
  const uint16_t* expo;
  const float* refs;
  float* raw_out;              // optional, score layout
  float* pooled;               // score layout (caller's buffer or workspace)
  int window, pool_width, num_kv_heads, p_total, n_items;
  int cu_seqlens[kMaxBatch + 1];
  int cu_prefix[kMaxBatch + 1];
  int seqs_per_mask;           // as in ScoreParams
  uint16_t srh_off[kMaxSrhGroups + 1];
  WorkItem items[kMaxItems];
};

// SRH list index of (sequence s, group g).
__host__ __device__ inline int srh_group(int s, int g, int seqs_per_mask, int num_kv_heads) {
  return (s / seqs_per_mask) * num_kv_heads + g;
}

// Row length (fp16 elements) of the exponent table for `rows` query rows:
// the next power of two >= max(rows, 8), so that a row is a whole number of
// 16-byte chunks and their count divides 32 when rows <= 256.
__host__ __device__ constexpr int expo_stride(int rows) {
  int r = 8;
  while (r < rows) r <<= 1;
  return r;
}

struct SelectParams {
  const float* raw;            // score layout (pooled here when pooled_in is null)
  const float* pooled_in;      // already pooled scores (score layout), or null
  float* pooled_out;           // optional, score layout
  float* pooled_ws;            // workspace copy of pooled scores, score layout
  int32_t* indices;            // [num_kv_heads][o_total]
  int* status;
  const uint4* k;              // gather sources / destinations (when gather != 0)
  const uint4* v;
  uint4* k_out;
  uint4* v_out;
  long long tok_stride_v16, head_stride_v16;  // K/V strides in 16-byte units
  int window, pool_width, num_kv_heads, p_total, o_total, batch;
  int cluster;                 // CTAs per unit (thread-block cluster size, 1..8)
  int slice;                   // prefix tokens per CTA (multiple of 32)
  int smem_slice;              // 1: raw and pooled slices live in shared memory
  int gather;                  // 1: also copy the retained K/V rows
  int head_budgets;            // 1: a budget per (sequence, group), outputs packed group-major
  int layer_scope;             // 1: one selection per sequence, shared by every KV group
  float* shared_ws;            // layer scope: workspace row for the summed scores [p_total]
  int cu_seqlens[kMaxBatch + 1];
  int cu_prefix[kMaxBatch + 1];
  int cu_out[kMaxBatch + 1];
  int2 unit_out[kMaxBudgetUnits];  // head budgets: (first output row, rows) of unit s*H_kv + g
};

struct GatherParams {
  const uint4* k;
  const uint4* v;
  uint4* k_out;
  uint4* v_out;
  const int32_t* indices;
  int* status;                 // may be null
  long long tok_stride_v16, head_stride_v16;  // K/V strides in 16-byte units
  int num_kv_heads, o_total, batch;
  int cu_seqlens[kMaxBatch + 1];
  int cu_out[kMaxBatch + 1];
};

// ---------------------------------------------------------------------------
// Persistent fused layer call (per-group selection of compresskv_compress_layers
// and compresskv_compress_layers_lse): one kernel streams K for every unit of
// a call in two passes (softmax statistics, then normalised scores with K
// re-read from L2), pools, selects and gathers, with work claimed from
// counters in the workspace.
constexpr int kChunkTiles = 16;         // K tiles per scoring chunk (references restart per chunk)
constexpr int kChunkKeys = kChunkTiles * kTileTokens;
constexpr int kFusedMaxSeqs = kMaxBatch;
constexpr int kFusedMaxLists = 1024;    // (mask, group) SRH lists of one call
constexpr int kFusedMaxUnits = kMaxBatch * kMaxKvHeads;
constexpr int kFusedCtrHead = 64;       // claim / exit / abort counters before the per-unit ones
// Workspace counters of the fused call: the header words, then per unit the
// first-pass contributions (one per epilogue warpgroup and chunk), the
// second-pass contributions (one per epilogue warp and chunk) and the state
// of its merged softmax denominators.
constexpr size_t kFusedCtrBytes = static_cast<size_t>(kFusedCtrHead + 3 * kFusedMaxUnits) * 4;
// top-k candidates of one unit kept in shared memory (more go to the unit's
// raw-score row); with it the merge / select region leaves room for two Q
// buffers of 192 query rows (W = 64 with three SRH heads) and two K stages
constexpr int kFusedCandCap = 3072;
constexpr int kFusedCRegion = 32 * 1024;  // shared memory of the merge / select warps

struct FusedParams {
  CUtensorMap tmap_k;          // 3-D map over K: (d, kv head, token)
  CUtensorMap tmap_q;          // 4-D map over the window queries: (d, w, head, sequence)
  const uint16_t* q;           // window queries (f16/bf16 bits)
  long long q_bs, q_hs, q_ws;  // window-query strides, elements
  const float* lse;            // given-LSE mode: natural-log LSE per (sequence, head, window row)
  long long lse_bs, lse_hs;    // its strides (elements); window rows contiguous
  const uint4* k;              // gather sources (K on the device; V may be mapped host memory)
  const uint4* v;
  uint4* k_out;
  uint4* v_out;
  long long tok_stride_v16, head_stride_v16;  // K/V strides in 16-byte units
  int32_t* indices;            // [num_kv_heads][o_total]
  float* raw;                  // raw scores, score layout (caller's buffer or workspace)
  float* pooled;               // pooled scores, score layout (caller's buffer or workspace)
  int* status;                 // device status word
  int* ctr;                    // counters (kFusedCtrBytes, zero between calls)
  float2* partials;            // [chunk * 4 + warpgroup][part_stride]: (M, S), sum 2^(z c) = S 2^M
  float* bias;                 // [unit][part_stride]: log2 D_q
  int part_stride;             // row length of partials and bias
  float c;                     // scale * log2(e)
  int window, pool_width, num_kv_heads, group_size, p_total, o_total, is_bf16;
  int n_units, n_chunks, batch;
  int do_select;
  int raw_scratch;             // raw scores in the workspace: a unit's row may hold its candidates
  unsigned long long wait_ns;  // limit of every bounded wait of the call
  int stall;                   // test hook: CTA 0's claimer first waits for a counter nothing sets               // 0: scores only (no selection, no gather)
  int given_lse;               // 1: no first pass; denominators from `lse`
  int q_half_bytes;            // bytes of one 64-column half of a Q buffer
  int q_bufs;                  // Q buffers (2 or 3)
  int row_stride;              // floats per epilogue warp row (>= max query rows, multiple of 32)
  int stages;                  // K tiles in the shared-memory ring
  int tstride, nbuf;           // TMEM columns per accumulator buffer, buffers
  int nwg;                     // epilogue warpgroups taking tiles (nbuf / nwg buffers each)
  int seqs_per_mask;
  int cu_seqlens[kFusedMaxSeqs + 1];
  int cu_prefix[kFusedMaxSeqs + 1];
  int cu_out[kFusedMaxSeqs + 1];
  int chunk_off[kFusedMaxSeqs + 1];   // first chunk of sequence s (units of s are consecutive)
  uint32_t srh_bits[kFusedMaxLists];  // per (mask, group): bit i = query head group*G + i is SRH
};

cudaError_t launch_fused(const FusedParams& p, int grid, size_t smem, cudaStream_t s);
size_t fused_smem_bytes(int q_half_bytes, int q_bufs, int stages, int row_stride, int nwg);
constexpr int kFusedPartsPerChunk = 4;  // first-pass pairs per chunk (epilogue warpgroups)
cudaError_t fused_set_smem_limit(size_t bytes);

// Kernel parameters travel by value; CUDA takes at most 32764 bytes of them.
static_assert(sizeof(ScoreParams) <= 32764, "scoring kernel parameters");
static_assert(sizeof(CombineParams) <= 32764, "combine kernel parameters");
static_assert(sizeof(SelectParams) <= 32764, "selection kernel parameters");
static_assert(sizeof(FusedParams) <= 32764, "fused kernel parameters");

// Max pooling of each SRH head's window scores, summed over the heads: head
// slot i of list (mask m, group g) holds the raw scores of that list's i-th
// SRH head (slots of a list beyond its head count are ignored).
struct MaxPoolParams {
  const float* slots;          // [n_slots][H_kv][p_total]
  long long slot_stride;       // H_kv * p_total
  float* pooled;               // [H_kv][p_total]
  float* raw;                  // optional: the slots' raw scores summed
  int num_kv_heads, batch, seqs_per_mask, pool_width, p_total;
  int cu_prefix[kMaxBatch + 1];
  uint8_t heads_of[kFusedMaxLists];  // SRH heads of list srh_group(s, g, ...)
};

// Host-side launchers (defined next to each kernel).
cudaError_t launch_score(const ScoreParams& p, int n_items, size_t smem, cudaStream_t s);
cudaError_t launch_score_lse(const ScoreParams& p, int n_items, size_t smem, cudaStream_t s);
cudaError_t launch_combine(const CombineParams& p, int n_items, size_t smem, cudaStream_t s);
cudaError_t launch_select(const SelectParams& p, int n_units, size_t smem, cudaStream_t s);
// Per-group selection from pooled scores by sampling (clusters of up to 16
// CTAs, `p.slice` <= kScMaxSlice positions per CTA).
constexpr int kScMaxSlice = 16384;
constexpr int kScTargetSlice = 2048;  // slice of the cluster-size occupancy query
constexpr int kScTargetCtas = 80;     // CTAs per sampled-select launch to aim for
cudaError_t launch_select_sampled(const SelectParams& p, int n_units, size_t smem, cudaStream_t s);
size_t select_sampled_smem_bytes(int slice);
int select_sampled_max_cluster(int slice);  // 16 when the device takes such clusters, else 8
cudaError_t launch_gather(const GatherParams& p, long long rows, cudaStream_t s);
cudaError_t launch_maxpool(const MaxPoolParams& p, int max_n, cudaStream_t s);
size_t score_smem_bytes(int q_half_bytes, int stages, int epi_warps);
// Sets every scoring kernel's shared-memory limit: `bytes` for one CTA per
// SM, half of it for the two-CTA form.
cudaError_t score_set_smem_limit(size_t bytes);
// Dynamic shared memory of a combine CTA that covers `quarters` 32-key
// quarters with exponent rows of `nr` columns and pooling width P.
size_t combine_smem_bytes(int quarters, int nr, int pool_width);
// Sets the combine kernel's dynamic shared-memory limit to what `optin`
// leaves beside its static shared memory and returns that limit.
cudaError_t combine_set_smem_limit(size_t optin, size_t* dynamic_max);
cudaError_t select_set_smem_limit(size_t bytes);
int select_max_smem_floats();

}  // namespace ckv
