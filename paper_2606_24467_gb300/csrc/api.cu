// Host side of the C ABI declared in include/compresskv.h: argument
// validation, SRH mask -> per-group head lists, unit-set and work-item
// planning, K tensor map, workspace carving and kernel launches.
// No device memory is allocated and no stream is synchronised here (except
// in compresskv_read_device_status).
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "ckv_params.h"
#include "compresskv.h"

namespace {
// A named range around each entry point for profilers (NVTX; nothing happens
// unless a profiling tool is attached to the process).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};
}  // namespace

using namespace ckv;

namespace {

// Test hook: the wait limit of the next fused call that stalls on purpose
// (0: none pending).
std::atomic<long long> g_stall_next_ns{0};

// Workspace header, zeroed by compresskv_workspace_init: the device status
// word (256 B) and one ticket per scoring item (the scoring kernel's
// last-CTA-per-unit merge resets the tickets it uses).
constexpr size_t kTicketOffset = 256;
constexpr size_t kStatusBytes = kTicketOffset + static_cast<size_t>(kMaxItems) * sizeof(int);
// ... followed by the fused call's counters; the whole header is zeroed by
// compresskv_workspace_init and left zero by every call that completes.
constexpr size_t kFusedCtrOffset = kStatusBytes;
constexpr size_t kHeaderBytes = ((kFusedCtrOffset + kFusedCtrBytes) + 255) & ~static_cast<size_t>(255);

// Units are scored in sets whose exponent tables take at most this many
// bytes; one set's table is written by the scoring kernel and read back by
// the combine kernel while (mostly) still in the 126 MB L2.  The workspace
// reserves a set bounded with every head of a group counted as SRH; a call
// packs its sets with the actual SRH rows.  Measured on GB300: 128 MiB sets
// (four bench layers per call, ~100 MB of table) beat 64 MiB sets, and one
// L=128K layer (~100 MB) runs as fast with its table as in two passes.
#ifndef CKV_EXPO_SET_BYTES
#define CKV_EXPO_SET_BYTES (128ll << 20)
#endif
constexpr long long kExpoSetBytes = CKV_EXPO_SET_BYTES;
constexpr size_t kPartialBytes = static_cast<size_t>(kMaxItems) * kMaxQRows * sizeof(float2);
constexpr size_t kBiasBytes = static_cast<size_t>(kMaxItems) * kMaxQRows * sizeof(float);

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// ------------------------------------------------------------------ device facts
struct DeviceFacts {
  int sms = 0;
  int smem_optin = 0;
  long long l2_bytes = 0;
  size_t combine_smem_max = 0;  // dynamic shared memory the combine kernel may use
  int sampled_cluster = 8;      // largest cluster of the sampled select (16 or 8)
  bool smem_attr_set = false;
};

std::mutex g_mutex;
DeviceFacts g_facts[64];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int device_facts(DeviceFacts** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return CKV_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceFacts& f = g_facts[dev];
  if (f.sms == 0) {
    int sms = 0, l2 = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return CKV_ERR_CUDA;
    if (cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess) return CKV_ERR_CUDA;
    f.sms = sms;
    f.l2_bytes = l2;
  }
  if (!f.smem_attr_set) {
    int optin = 0;
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
      return CKV_ERR_CUDA;
    f.smem_optin = optin;
    if (score_set_smem_limit(static_cast<size_t>(optin)) != cudaSuccess) return CKV_ERR_CUDA;
    if (fused_set_smem_limit(static_cast<size_t>(optin)) != cudaSuccess) return CKV_ERR_CUDA;
    if (combine_set_smem_limit(static_cast<size_t>(optin), &f.combine_smem_max) != cudaSuccess)
      return CKV_ERR_CUDA;
    if (select_set_smem_limit(static_cast<size_t>(select_max_smem_floats()) * 4) != cudaSuccess)
      return CKV_ERR_CUDA;
    f.sampled_cluster = select_sampled_max_cluster(kScTargetSlice);
    f.smem_attr_set = true;
  }
  if (!g_encode) {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return CKV_ERR_CUDA;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  *out = &f;
  return CKV_OK;
}

// ------------------------------------------------------------------ validation
struct Info {
  int B = 0, Hq = 0, Hkv = 0, G = 0, W = 0, P = 0;
  bool bf16 = false;
  bool layer = false;  // CKV_SELECT_PER_LAYER
  bool pool_max = false;  // CKV_POOL_MAX
  float scale = 0.f;
  std::vector<int> cu, len, n, cu_prefix;
  long long T = 0, p_total = 0;
  // SRH masks: sequence s uses mask s / spm (n_masks masks, spm = B / n_masks)
  int n_masks = 1, spm = 1;
  int vgroup(int s, int g) const { return srh_group(s, g, spm, Hkv); }
};

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

// The address under which the device reads `ptr`: device or managed memory
// as is, page-locked host memory through its mapped (unified) address.
// Pageable or unknown memory is refused: a kernel must not touch it.
int device_readable(const void* ptr, const void** dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    (void)cudaGetLastError();
    return CKV_ERR_INVALID_ARG;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) {
    *dev = ptr;
    return CKV_OK;
  }
  if (a.type == cudaMemoryTypeHost && a.devicePointer) {
    *dev = a.devicePointer;
    return CKV_OK;
  }
  return CKV_ERR_INVALID_ARG;
}

// Device (or managed) memory of the current device: what a kernel may read
// through a plain pointer.  Host memory of any kind is refused.
int device_memory(const void* ptr) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    (void)cudaGetLastError();
    return CKV_ERR_INVALID_ARG;
  }
  if (a.type == cudaMemoryTypeManaged) return CKV_OK;
  int dev = -1;
  if (a.type != cudaMemoryTypeDevice || cudaGetDevice(&dev) != cudaSuccess || a.device != dev)
    return CKV_ERR_INVALID_ARG;
  return CKV_OK;
}

int validate(const ckv_problem* p, Info& I) {
  if (!p || !p->cu_seqlens) return CKV_ERR_INVALID_ARG;
  if (p->batch < 1 || p->batch > kMaxBatch) return CKV_ERR_UNSUPPORTED;
  if (p->num_kv_heads < 1 || p->num_q_heads < 1) return CKV_ERR_INVALID_ARG;
  if (p->num_q_heads % p->num_kv_heads != 0) return CKV_ERR_INVALID_ARG;
  if (p->num_kv_heads > kMaxKvHeads || p->num_q_heads > kMaxQHeads) return CKV_ERR_UNSUPPORTED;
  if (p->head_dim != kHeadDim) return CKV_ERR_UNSUPPORTED;
  if (p->window < 1) return CKV_ERR_INVALID_ARG;
  if (p->pool_width < 1 || p->pool_width % 2 == 0 || p->pool_width > 63) return CKV_ERR_INVALID_ARG;
  if (p->dtype != CKV_DTYPE_F16 && p->dtype != CKV_DTYPE_BF16) return CKV_ERR_INVALID_ARG;
  if (p->pool_kind != CKV_POOL_AVG && p->pool_kind != CKV_POOL_MAX) return CKV_ERR_INVALID_ARG;
  if (p->selection != CKV_SELECT_PER_GROUP && p->selection != CKV_SELECT_PER_LAYER)
    return CKV_ERR_INVALID_ARG;
  if (!(p->scale >= 0.f) || std::isinf(p->scale)) return CKV_ERR_INVALID_ARG;
  if (p->kv_token_stride <= 0 || p->kv_head_stride <= 0 || p->kv_token_stride % 8 ||
      p->kv_head_stride % 8)
    return CKV_ERR_INVALID_ARG;
  if (p->q_batch_stride < 0 || p->q_head_stride < 0 || p->q_win_stride < 0 ||
      p->q_batch_stride % 8 || p->q_head_stride % 8 || p->q_win_stride % 8)
    return CKV_ERR_INVALID_ARG;
  I.B = p->batch;
  I.Hq = p->num_q_heads;
  I.Hkv = p->num_kv_heads;
  I.G = I.Hq / I.Hkv;
  I.W = p->window;
  I.P = p->pool_width;
  I.bf16 = p->dtype == CKV_DTYPE_BF16;
  I.layer = p->selection == CKV_SELECT_PER_LAYER;
  I.pool_max = p->pool_kind == CKV_POOL_MAX;
  I.scale = p->scale > 0.f ? p->scale : 1.0f / std::sqrt(static_cast<float>(kHeadDim));
  I.cu.assign(p->cu_seqlens, p->cu_seqlens + I.B + 1);
  if (I.cu[0] != 0) return CKV_ERR_INVALID_ARG;
  I.len.resize(I.B);
  I.n.resize(I.B);
  I.cu_prefix.assign(I.B + 1, 0);
  for (int s = 0; s < I.B; ++s) {
    const long long L = static_cast<long long>(I.cu[s + 1]) - I.cu[s];
    if (L < 0) return CKV_ERR_INVALID_ARG;
    if (L > 65535LL * kTileTokens) return CKV_ERR_UNSUPPORTED;
    I.len[s] = static_cast<int>(L);
    I.n[s] = std::max(I.len[s] - I.W, 0);
    I.cu_prefix[s + 1] = I.cu_prefix[s] + I.n[s];
  }
  I.T = I.cu[I.B];
  I.p_total = I.cu_prefix[I.B];
  I.n_masks = 1;
  I.spm = I.B;
  if (static_cast<long long>(I.Hkv) * I.p_total > (1LL << 31) - 1) return CKV_ERR_UNSUPPORTED;
  return CKV_OK;
}

int output_layout(const Info& I, const int32_t* budgets, std::vector<int>& cu_out) {
  if (!budgets) return CKV_ERR_INVALID_ARG;
  cu_out.assign(I.B + 1, 0);
  for (int s = 0; s < I.B; ++s) {
    if (budgets[s] < I.W) return CKV_ERR_BUDGET;
    cu_out[s + 1] = cu_out[s] + std::min(budgets[s], I.len[s]);
  }
  if (static_cast<long long>(I.Hkv) * cu_out[I.B] > (1LL << 31) - 1) return CKV_ERR_UNSUPPORTED;
  return CKV_OK;
}

// Units (s, g) with a prefix to score, in (s, g) order, cut into sets.  The
// cut uses the largest exponent row any SRH mask can give (all G heads of a
// group), so the workspace size depends on the problem alone.
struct UnitSet {
  int u0, u1;             // units [u0, u1) of the unit list
  long long expo_elems;   // fp16 elements of the set's exponent table (bound)
  long long ref_floats;   // floats of its reference table (bound)
};

int expo_row_bound(const Info& I) { return expo_stride(std::min(I.G * I.W, kMaxQRows)); }

void plan_sets(const Info& I, std::vector<UnitSet>& sets) {
  sets.clear();
  const long long nr = expo_row_bound(I);
  int u = 0, u0 = 0;
  long long e = 0, r = 0;
  for (int s = 0; s < I.B; ++s) {
    if (I.n[s] <= 0) continue;
    const long long ue = static_cast<long long>(I.n[s]) * nr;
    const long long ur =
        static_cast<long long>((I.len[s] + kTileTokens - 1) / kTileTokens) * kQuarters * nr;
    for (int g = 0; g < I.Hkv; ++g, ++u) {
      if (u > u0 && (2 * (e + ue) > kExpoSetBytes || u - u0 >= kMaxItems / 2)) {
        sets.push_back({u0, u, e, r});
        u0 = u;
        e = r = 0;
      }
      e += ue;
      r += ur;
    }
  }
  if (u > u0) sets.push_back({u0, u, e, r});
}

struct Workspace {
  int* status = nullptr;
  int* tickets = nullptr;    // [kMaxItems], in the header
  float2* partials = nullptr;
  float* bias = nullptr;     // [kMaxItems][kMaxQRows] log2 softmax denominators per unit
  float* pooled = nullptr;   // score layout
  uint16_t* expo = nullptr;  // one set's exponent table
  float* refs = nullptr;     // one set's reference table
  float* shared = nullptr;   // per-layer selection: summed scores [sum_s n_s]
  float* raw = nullptr;      // raw scores, score layout (given-LSE calls)
};

struct WorkspaceLayout {
  size_t pooled, expo, refs, shared, raw, total;
};

WorkspaceLayout workspace_layout(const Info& I) {
  std::vector<UnitSet> sets;
  plan_sets(I, sets);
  long long e = 0, r = 0;
  for (const UnitSet& S : sets) {
    e = std::max(e, S.expo_elems);
    r = std::max(r, S.ref_floats);
  }
  WorkspaceLayout W;
  W.pooled = kHeaderBytes + kPartialBytes + kBiasBytes;
  W.expo = W.pooled + align256(static_cast<size_t>(I.Hkv) * I.p_total * sizeof(float));
  W.refs = W.expo + align256(static_cast<size_t>(e) * sizeof(uint16_t));
  W.shared = W.refs + align256(static_cast<size_t>(r) * sizeof(float));
  W.raw = W.shared + (I.layer ? align256(static_cast<size_t>(I.p_total) * sizeof(float)) : 0);
  W.total = W.raw + align256(static_cast<size_t>(I.Hkv) * I.p_total * sizeof(float));
  return W;
}

// Layout of the fused call's workspace (after the header; it aliases the
// layout above, which the other entry points use).  A function of the problem
// alone: rows are bounded with every head of a group counted as SRH.
struct FusedLayout {
  size_t raw, pooled, partials, bias, total;
  long long n_chunks;
  int part_stride;
};

int chunks_per_unit(const Info& I, int s) {
  if (I.n[s] <= 0) return 0;
  const int tiles = (I.len[s] + kTileTokens - 1) / kTileTokens;
  return (tiles + kChunkTiles - 1) / kChunkTiles;
}

FusedLayout fused_layout(const Info& I) {
  FusedLayout F;
  F.part_stride = (std::min(I.G * I.W, kMaxQRows) + 3) & ~3;
  F.n_chunks = 0;
  for (int s = 0; s < I.B; ++s) F.n_chunks += static_cast<long long>(I.Hkv) * chunks_per_unit(I, s);
  const long long units = static_cast<long long>(I.B) * I.Hkv;
  const size_t scores = align256(static_cast<size_t>(I.Hkv) * I.p_total * sizeof(float));
  F.raw = kHeaderBytes;
  F.pooled = F.raw + scores;
  F.partials = F.pooled + scores;
  F.bias = F.partials + align256(static_cast<size_t>(F.n_chunks) * kFusedPartsPerChunk *
                                 F.part_stride * sizeof(float2));
  F.total = F.bias + align256(static_cast<size_t>(units) * F.part_stride * sizeof(float));
  return F;
}

// Max pooling: after both layouts, one raw-score row per SRH head slot (at
// most G) of every group.
size_t maxpool_slots_offset(const Info& I) {
  return align256(std::max(workspace_layout(I).total, fused_layout(I).total));
}

size_t workspace_bytes(const Info& I) {
  const size_t base = std::max(workspace_layout(I).total, fused_layout(I).total);
  if (!I.pool_max) return base;
  return maxpool_slots_offset(I) +
         align256(static_cast<size_t>(I.G) * I.Hkv * I.p_total * sizeof(float));
}

int carve(const Info& I, void* ws, size_t bytes, Workspace& out) {
  const WorkspaceLayout W = workspace_layout(I);
  if (!ws || bytes < workspace_bytes(I) || (reinterpret_cast<uintptr_t>(ws) & 255u))
    return CKV_ERR_WORKSPACE;
  char* b = static_cast<char*>(ws);
  out.status = reinterpret_cast<int*>(b);
  out.tickets = reinterpret_cast<int*>(b + kTicketOffset);
  out.partials = reinterpret_cast<float2*>(b + kHeaderBytes);
  out.bias = reinterpret_cast<float*>(b + kHeaderBytes + kPartialBytes);
  out.pooled = reinterpret_cast<float*>(b + W.pooled);
  out.expo = reinterpret_cast<uint16_t*>(b + W.expo);
  out.refs = reinterpret_cast<float*>(b + W.refs);
  out.shared = reinterpret_cast<float*>(b + W.shared);
  out.raw = reinterpret_cast<float*>(b + W.raw);
  return CKV_OK;
}

// ------------------------------------------------------------------ tracing
// Records the caller's trace events around each launch.  A failed record
// (for example a null event handle) is reported as CKV_ERR_INVALID_ARG and
// the runtime's last-error state is cleared.
struct Tracer {
  ckv_trace* t;
  cudaStream_t s;
  int slot = -1;
  int begin(int kind) {
    slot = -1;
    if (!t) return CKV_OK;
    if (t->count < t->capacity && t->events) {
      slot = t->count++;
      if (t->kinds) t->kinds[slot] = kind;
      return record(static_cast<cudaEvent_t>(t->events[2 * slot]));
    }
    return CKV_OK;
  }
  int end() {
    if (!t) return CKV_OK;
    ++t->launches;
    if (slot >= 0) return record(static_cast<cudaEvent_t>(t->events[2 * slot + 1]));
    return CKV_OK;
  }
  int record(cudaEvent_t e) {
    if (!e) return CKV_ERR_INVALID_ARG;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    cudaError_t err = cudaStreamIsCapturing(s, &cs);
    if (err == cudaSuccess) {
      err = cs == cudaStreamCaptureStatusActive
                ? cudaEventRecordWithFlags(e, s, cudaEventRecordExternal)
                : cudaEventRecord(e, s);
    }
    if (err != cudaSuccess) {
      cudaGetLastError();
      return CKV_ERR_INVALID_ARG;
    }
    return CKV_OK;
  }
};

// Launch `fn` bracketed by the trace: trace errors win over a clean launch.
template <class F>
int traced(Tracer& tr, int kind, F&& fn) {
  int rc = tr.begin(kind);
  if (rc != CKV_OK) return rc;
  const cudaError_t e = fn();
  const int rc2 = tr.end();
  if (e != cudaSuccess) return CKV_ERR_CUDA;
  return rc2;
}

// ------------------------------------------------------------------ scoring
// SRH heads per (mask, group), flattened: list v = m * H_kv + g holds
// heads[off[v] .. off[v+1]) and rows[v] = |S| * W query rows.
struct SrhLists {
  std::vector<uint16_t> off;
  std::vector<uint8_t> heads;
  std::vector<int> rows;
};

// masks: I.n_masks masks of I.Hq bytes each.
int srh_lists(const Info& I, const uint8_t* masks, SrhLists& S) {
  if (!masks) return CKV_ERR_INVALID_ARG;
  const int nv = I.n_masks * I.Hkv;
  S.off.assign(nv + 1, 0);
  S.heads.clear();
  S.rows.assign(nv, 0);
  for (int m = 0; m < I.n_masks; ++m) {
    const uint8_t* mask = masks + static_cast<size_t>(m) * I.Hq;
    bool any_scored = false;  // a sequence of this mask's block has a prefix
    for (int s = m * I.spm; s < (m + 1) * I.spm; ++s) any_scored |= I.n[s] > 0;
    const size_t first_head = S.heads.size();
    for (int g = 0; g < I.Hkv; ++g) {
      const int v = m * I.Hkv + g;
      for (int h = g * I.G; h < (g + 1) * I.G; ++h)
        if (mask[h]) S.heads.push_back(static_cast<uint8_t>(h));
      S.off[v + 1] = static_cast<uint16_t>(S.heads.size());
      const int cnt = S.off[v + 1] - S.off[v];
      // per-group selection needs an SRH head in every group; per-layer
      // selection only somewhere in the layer
      if (cnt == 0 && any_scored && !I.layer) return CKV_ERR_EMPTY_SRH_GROUP;
      S.rows[v] = cnt * I.W;
      if (S.rows[v] > kMaxQRows) return CKV_ERR_UNSUPPORTED;
    }
    if (I.layer && S.heads.size() == first_head && any_scored) return CKV_ERR_EMPTY_SRH_GROUP;
  }
  return CKV_OK;
}

int make_k_map(const Info& I, const ckv_problem* p, const void* k, CUtensorMap* map) {
  if (I.T == 0) return CKV_OK;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(I.Hkv),
                        static_cast<cuuint64_t>(I.T)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(p->kv_head_stride) * 2,
                           static_cast<cuuint64_t>(p->kv_token_stride) * 2};
  cuuint32_t box[3] = {64u, 1u, static_cast<cuuint32_t>(kTileTokens)};
  cuuint32_t estr[3] = {1u, 1u, 1u};
  CUresult r = g_encode(map, I.bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16,
                        3, const_cast<void*>(k), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? CKV_OK : CKV_ERR_INVALID_ARG;
}

// 4-D map over the window queries (d, w, head, sequence); the fused kernel
// loads one box of W rows x 64 columns per SRH head and column half.
int make_q_map(const Info& I, const ckv_problem* p, const void* q_win, CUtensorMap* map) {
  const long long bs = I.B > 1 ? p->q_batch_stride : p->q_head_stride * I.Hq;
  cuuint64_t dims[4] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(I.W),
                        static_cast<cuuint64_t>(I.Hq), static_cast<cuuint64_t>(I.B)};
  cuuint64_t strides[3] = {static_cast<cuuint64_t>(p->q_win_stride) * 2,
                           static_cast<cuuint64_t>(p->q_head_stride) * 2,
                           static_cast<cuuint64_t>(bs) * 2};
  cuuint32_t box[4] = {64u, static_cast<cuuint32_t>(I.W), 1u, 1u};
  cuuint32_t estr[4] = {1u, 1u, 1u, 1u};
  CUresult r = g_encode(map, I.bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16,
                        4, const_cast<void*>(q_win), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? CKV_OK : CKV_ERR_INVALID_ARG;
}

// Scores every unit: per set, the scoring kernel (one pass over K) and the
// combine kernel, which leaves pooled scores (and raw scores when `raw` is
// given) in score layout.
// Window-query log-sum-exps supplied by the caller (given-LSE mode).
struct LseInput {
  const float* lse = nullptr;
  long long batch_stride = 0, head_stride = 0;
};

// Without a given LSE, units are scored in one of two ways:
//  * one pass with the exponent table and the combine kernel (raw and pooled
//    scores), when the layer's table -- with the actual SRH rows -- fits one
//    set of kExpoSetBytes, i.e. stays in L2 between the two kernels;
//  * otherwise two passes over K without a table (*two_pass set): the scoring
//    kernel in stats-only mode leaves the per-unit log2 softmax denominators,
//    and the given-LSE kernel reads them and writes raw scores (into `raw`,
//    else the workspace's raw row); the caller then pools and selects from
//    raw scores.  Reading K twice moves fewer bytes than writing and reading
//    a table that does not stay in L2.
int run_score(const ckv_problem* p, const Info& I, const void* q_win, const void* k,
              const uint8_t* mask, float* raw, float* pooled, const Workspace& ws,
              cudaStream_t stream, const LseInput& lse = LseInput{}, bool* two_pass = nullptr) {
  const bool given_lse = lse.lse != nullptr;
  if (!q_win || !k || (given_lse ? !raw : !pooled)) return CKV_ERR_INVALID_ARG;
  if (!aligned16(q_win) || !aligned16(k)) return CKV_ERR_INVALID_ARG;
  SrhLists S;
  int rc = srh_lists(I, mask, S);
  if (rc != CKV_OK) return rc;
  DeviceFacts* F = nullptr;
  if ((rc = device_facts(&F)) != CKV_OK) return rc;
  if (I.p_total == 0) return CKV_OK;

  static thread_local ScoreParams P;    // large (about 17 KB): kept off the stack
  static thread_local CombineParams C;  // likewise
  std::memset(&P, 0, sizeof(P));
  std::memset(&C, 0, sizeof(C));
  if ((rc = make_k_map(I, p, k, &P.tmap_k)) != CKV_OK) return rc;
  P.q = static_cast<const uint16_t*>(q_win);
  P.partials = ws.partials;
  P.bias = ws.bias;
  P.tickets = ws.tickets;
  P.expo = ws.expo;
  P.refs = ws.refs;
  P.status = ws.status;
  P.q_bs = p->q_batch_stride;
  P.q_hs = p->q_head_stride;
  P.q_ws = p->q_win_stride;
  P.c = static_cast<float>(static_cast<double>(I.scale) * 1.4426950408889634);
  P.window = I.W;
  P.num_kv_heads = I.Hkv;
  P.is_bf16 = I.bf16 ? 1 : 0;
  P.use_evict_hint = 1;
  P.lse = lse.lse;
  P.lse_bs = lse.batch_stride;
  P.lse_hs = lse.head_stride;
  P.raw_out = raw;
  P.p_total = static_cast<int>(I.p_total);
  for (int s = 0; s <= I.B; ++s) P.cu_prefix[s] = I.cu_prefix[s];
  C.bias = ws.bias;
  C.expo = ws.expo;
  C.refs = ws.refs;
  C.raw_out = raw;
  C.pooled = pooled;
  C.window = I.W;
  C.pool_width = I.P;
  C.num_kv_heads = I.Hkv;
  C.p_total = static_cast<int>(I.p_total);
  for (int s = 0; s <= I.B; ++s) {
    P.cu_seqlens[s] = I.cu[s];
    C.cu_seqlens[s] = I.cu[s];
    C.cu_prefix[s] = I.cu_prefix[s];
  }
  P.seqs_per_mask = C.seqs_per_mask = I.spm;
  for (size_t v = 0; v < S.off.size(); ++v) P.srh_off[v] = C.srh_off[v] = S.off[v];
  for (size_t h = 0; h < S.heads.size(); ++h) P.srh_heads[h] = S.heads[h];

  // units (s, g) with v = their SRH list
  struct Unit { int s, g, v, tiles, quarters; };
  std::vector<Unit> units;
  for (int s = 0; s < I.B; ++s)
    if (I.n[s] > 0)
      for (int g = 0; g < I.Hkv; ++g)
        units.push_back({s, g, I.vgroup(s, g), (I.len[s] + kTileTokens - 1) / kTileTokens,
                         (I.n[s] + 31) / 32});
  std::vector<UnitSet> sets;
  // the layer's exponent table with the actual SRH rows
  long long table_bytes = 0;
  for (const Unit& U : units) table_bytes += 2LL * I.n[U.s] * expo_stride(S.rows[U.v]);
  const bool passes2 = !given_lse && table_bytes > kExpoSetBytes;
  if (two_pass) *two_pass = passes2;
  if (passes2) {
    // no table: sets are bounded by the work-item tables only
    sets.clear();
    for (int u0 = 0; u0 < static_cast<int>(units.size()); u0 += kMaxItems / 2)
      sets.push_back({u0, std::min<int>(static_cast<int>(units.size()), u0 + kMaxItems / 2), 0, 0});
    if (!raw) raw = ws.raw;
    P.stats_only = 1;
    P.raw_out = raw;
  } else {
    // sets cut with the actual SRH rows, within the workspace's table space
    const WorkspaceLayout WL = workspace_layout(I);
    const long long cap_e = static_cast<long long>((WL.refs - WL.expo) / sizeof(uint16_t));
    const long long cap_r = static_cast<long long>((WL.shared - WL.refs) / sizeof(float));
    long long e = 0, r = 0;
    int u0 = 0;
    for (int u = 0; u < static_cast<int>(units.size()); ++u) {
      const Unit& U = units[u];
      const long long nr = expo_stride(S.rows[U.v]);
      const long long ue = static_cast<long long>(I.n[U.s]) * nr;
      const long long ur = static_cast<long long>(U.tiles) * kQuarters * nr;
      if (u > u0 && (e + ue > cap_e || r + ur > cap_r || 2 * (e + ue) > kExpoSetBytes ||
                     u - u0 >= kMaxItems / 2)) {
        sets.push_back({u0, u, e, r});
        u0 = u;
        e = r = 0;
      }
      if (ue > cap_e || ur > cap_r) return CKV_ERR_WORKSPACE;  // cannot happen: the bound covers a unit
      e += ue;
      r += ur;
    }
    if (static_cast<int>(units.size()) > u0) sets.push_back({u0, static_cast<int>(units.size()), e, r});
  }
  Tracer tr{p->trace, stream};
  // Per-layer selection sums the groups' scores: a group without an SRH head
  // contributes zeros.
  for (int m = 0; m < I.n_masks; ++m) {
    for (int g = 0; g < I.Hkv; ++g) {
      if (S.rows[m * I.Hkv + g] > 0) continue;
      // the scores of this group for the mask's block of sequences
      const size_t off = static_cast<size_t>(g) * I.p_total + I.cu_prefix[m * I.spm];
      const size_t bytes =
          static_cast<size_t>(I.cu_prefix[(m + 1) * I.spm] - I.cu_prefix[m * I.spm]) * sizeof(float);
      if (bytes == 0) continue;
      if (pooled && cudaMemsetAsync(pooled + off, 0, bytes, stream) != cudaSuccess)
        return CKV_ERR_CUDA;
      if (raw && cudaMemsetAsync(raw + off, 0, bytes, stream) != cudaSuccess) return CKV_ERR_CUDA;
    }
  }
  for (const UnitSet& set : sets) {
    const int u0 = set.u0;
    const int nu = set.u1 - set.u0;
    // Score work items: one wave of exactly max(#units, #SMs) CTAs.  A tile
    // of a unit costs about (64 + query rows) (the epilogue scales with the
    // rows); every unit gets one item, the remaining items go one at a time
    // to the unit with the largest work per item, then each unit's tiles are
    // split into balanced ranges.
    // (Units of a group without an SRH head -- per-layer selection only --
    // get no items.)
    auto cost = [&](const Unit& U) { return 64LL + ((S.rows[U.v] + 15) & ~15); };
    std::vector<int> cnt(nu, 1);
    std::vector<long long> uw(nu);
    int active = 0;
    for (int u = 0; u < nu; ++u) {
      uw[u] = static_cast<long long>(units[u0 + u].tiles) * cost(units[u0 + u]);
      cnt[u] = S.rows[units[u0 + u].v] > 0 ? 1 : 0;
      active += cnt[u];
    }
    if (active == 0) continue;
    // Two CTAs per SM (8 epilogue warps each, two K rings in flight) when
    // their shared memory fits; else one CTA per SM with 16 epilogue warps.
    int max_rows = 16;
    for (int u = 0; u < nu; ++u)
      if (cnt[u] > 0) max_rows = std::max(max_rows, (S.rows[units[u0 + u].v] + 15) & ~15);
    const int q_half = ((max_rows * 128) + 1023) & ~1023;
    const int per_sm =
        score_smem_bytes(q_half, 2, 8) <= static_cast<size_t>(F->smem_optin) / 2 - 1024 ? 2 : 1;
    const int target = std::min(kMaxItems, std::max(active, per_sm * F->sms));
    for (int extra = target - active; extra > 0; --extra) {
      int best = -1;
      for (int u = 0; u < nu; ++u) {
        if (cnt[u] == 0 || cnt[u] >= units[u0 + u].tiles) continue;
        if (best < 0 || uw[u] * cnt[best] > uw[best] * cnt[u]) best = u;
      }
      if (best < 0) break;
      ++cnt[best];
    }
    // Combine items: chunks of 32-token quarters, about three CTAs per SM
    // (measured: 3 and 4 per SM best for four-layer calls, 2, 3 and 4 within
    // 0.5% of each other for one-layer calls), balanced by bytes: a quarter
    // of a unit with exponent rows of nr columns weighs nr + 16 (table bytes
    // plus a fixed share per key).
    constexpr int kQuarterFixed = 16;
    long long weight = 0;
    for (int u = 0; u < nu; ++u)
      if (cnt[u] > 0)
        weight += static_cast<long long>(units[u0 + u].quarters) *
                  (expo_stride(S.rows[units[u0 + u].v]) + kQuarterFixed);
    const long long ctarget = std::max(1, std::min(kMaxItems - nu, 3 * F->sms));
    const long long per_chunk = std::max<long long>(8 * (8 + kQuarterFixed),
                                                    (weight + ctarget - 1) / ctarget);
    std::vector<int> chunk_q(nu, 1);
    size_t csmem = 0;
    for (int u = 0; u < nu; ++u) {
      if (cnt[u] == 0) continue;
      const int nr = expo_stride(S.rows[units[u0 + u].v]);
      int cq = static_cast<int>(std::max(1LL, per_chunk / (nr + kQuarterFixed)));
      // a chunk's weight table and raw scores must fit the shared memory
      while (cq > 1 && combine_smem_bytes(cq, nr, I.P) > F->combine_smem_max) cq = (cq + 1) / 2;
      chunk_q[u] = cq;
      csmem = std::max(csmem, combine_smem_bytes(cq, nr, I.P));
    }
    if (csmem > F->combine_smem_max) return CKV_ERR_UNSUPPORTED;

    int n_items = 0, n_comb = 0;
    uint32_t eoff = 0, roff = 0;
    for (int u = 0; u < nu; ++u) {
      const Unit& U = units[u0 + u];
      const int c_u = cnt[u];
      if (c_u == 0) continue;
      const int nr = expo_stride(S.rows[U.v]);
      if (n_items + c_u > kMaxItems) return CKV_ERR_UNSUPPORTED;
      for (int c = 0; c < c_u; ++c) {
        WorkItem& it = P.items[n_items + c];
        it.seq = static_cast<uint16_t>(U.s);
        it.group = static_cast<uint16_t>(U.g);
        it.t0 = static_cast<uint16_t>(static_cast<long long>(U.tiles) * c / c_u);
        it.t1 = static_cast<uint16_t>(static_cast<long long>(U.tiles) * (c + 1) / c_u);
        it.first = static_cast<uint16_t>(n_items);
        it.count = static_cast<uint16_t>(c_u);
        it.eoff = eoff;
        it.roff = roff;
      }
      for (int q0 = 0; q0 < U.quarters; q0 += chunk_q[u]) {
        if (n_comb >= kMaxItems) return CKV_ERR_UNSUPPORTED;
        WorkItem& it = C.items[n_comb++];
        it = P.items[n_items];
        it.t0 = static_cast<uint16_t>(q0);
        it.t1 = static_cast<uint16_t>(std::min(U.quarters, q0 + chunk_q[u]));
      }
      n_items += c_u;
      eoff += static_cast<uint32_t>(I.n[U.s]) * static_cast<uint32_t>(nr);
      roff += static_cast<uint32_t>(U.tiles * kQuarters * nr);
    }
    P.n_items = n_items;
    C.n_items = n_comb;
    P.q_half_bytes = q_half;
    P.stages = kStages;
    P.epi_warps = per_sm == 2 ? 8 : 16;
    const size_t smem_cap = per_sm == 2 ? static_cast<size_t>(F->smem_optin) / 2 - 1024
                                        : static_cast<size_t>(F->smem_optin);
    while (P.stages > 2 && score_smem_bytes(P.q_half_bytes, P.stages, P.epi_warps) > smem_cap)
      --P.stages;
    const size_t smem = score_smem_bytes(P.q_half_bytes, P.stages, P.epi_warps);
    if (given_lse) {  // raw scores come straight out of the scoring kernel
      rc = traced(tr, CKV_KERNEL_SCORE, [&] { return launch_score_lse(P, n_items, smem, stream); });
      if (rc != CKV_OK) return rc;
      continue;
    }
    if (passes2) {
      // pass 1: denominators only; pass 2: raw scores from them
      rc = traced(tr, CKV_KERNEL_SCORE, [&] { return launch_score(P, n_items, smem, stream); });
      if (rc != CKV_OK) return rc;
      P.lse_bias = ws.bias;
      rc = traced(tr, CKV_KERNEL_SCORE, [&] { return launch_score_lse(P, n_items, smem, stream); });
      P.lse_bias = nullptr;
      if (rc != CKV_OK) return rc;
      continue;
    }
    rc = traced(tr, CKV_KERNEL_SCORE, [&] { return launch_score(P, n_items, smem, stream); });
    if (rc != CKV_OK) return rc;
    rc = traced(tr, CKV_KERNEL_COMBINE,
                [&] { return launch_combine(C, n_comb, csmem, stream); });
    if (rc != CKV_OK) return rc;
  }
  return CKV_OK;
}

// ------------------------------------------------------------------ select / gather
// Arguments of the selection's outputs and, when `k` is given, of the fused
// gather; `v` is replaced by the address the device reads it under.  The
// fused layer calls run this before their first launch.
int check_outputs(const Info& I, const std::vector<int>& cu_out, const int32_t* indices,
                  const void* k, const void*& v, const void* k_out, const void* v_out) {
  if (cu_out[I.B] == 0) return CKV_OK;
  if (!indices) return CKV_ERR_INVALID_ARG;
  if (!k) return CKV_OK;
  if (!v || !k_out || !v_out) return CKV_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || !aligned16(k_out) || !aligned16(v_out))
    return CKV_ERR_INVALID_ARG;
  return device_readable(v, &v);
}

// Pooling (unless `pooled_in` holds the pooled scores already), top-k and
// window append, optionally fused with the K/V gather.
// With `unit_out` (head-level budgets) every unit (s, g) has its own output
// rows (first row, count) in a group-major packing, and cu_out[I.B] is the
// total row count.
int run_select(const ckv_problem* p, const Info& I, const float* raw, const float* pooled_in,
               const std::vector<int>& cu_out, int32_t* indices, float* pooled,
               const Workspace& ws, cudaStream_t stream, const void* k = nullptr,
               const void* v = nullptr, void* k_out = nullptr, void* v_out = nullptr,
               const std::vector<int2>* unit_out = nullptr) {
  if (!raw && !pooled_in && I.p_total > 0) return CKV_ERR_INVALID_ARG;
  const bool gather = k != nullptr;
  const int rg = check_outputs(I, cu_out, indices, k, v, k_out, v_out);
  if (rg != CKV_OK) return rg;
  DeviceFacts* F = nullptr;
  int rc = device_facts(&F);
  if (rc != CKV_OK) return rc;
  if (cu_out[I.B] == 0 && (!pooled || pooled_in)) return CKV_OK;
  static thread_local SelectParams P;
  std::memset(&P, 0, sizeof(P));
  P.raw = raw;
  P.pooled_in = pooled_in;
  P.pooled_out = pooled_in ? nullptr : pooled;
  P.layer_scope = I.layer ? 1 : 0;
  P.shared_ws = ws.shared;
  P.pooled_ws = ws.pooled;
  P.indices = indices;
  P.status = ws.status;
  P.k = static_cast<const uint4*>(k);
  P.v = static_cast<const uint4*>(v);
  P.k_out = static_cast<uint4*>(k_out);
  P.v_out = static_cast<uint4*>(v_out);
  P.tok_stride_v16 = p->kv_token_stride / 8;
  P.head_stride_v16 = p->kv_head_stride / 8;
  P.gather = gather ? 1 : 0;
  P.window = I.W;
  P.pool_width = I.P;
  P.num_kv_heads = I.Hkv;
  P.p_total = static_cast<int>(I.p_total);
  P.o_total = cu_out[I.B];
  if (unit_out) {
    if (unit_out->size() > static_cast<size_t>(kMaxBudgetUnits)) return CKV_ERR_UNSUPPORTED;
    P.head_budgets = 1;
    for (size_t u = 0; u < unit_out->size(); ++u) P.unit_out[u] = (*unit_out)[u];
  }
  P.batch = I.B;
  int max_n = 0;
  for (int s = 0; s <= I.B; ++s) {
    P.cu_seqlens[s] = I.cu[s];
    P.cu_prefix[s] = I.cu_prefix[s];
    P.cu_out[s] = cu_out[s];
    if (s < I.B) max_n = std::max(max_n, I.n[s]);
  }
  if (pooled_in && !I.layer && max_n <= 32 * 1024) {
    // fused layer call, per-group selection: sampled select, one cluster of
    // C CTAs per unit (longer prefixes list too many keys above the sampled
    // bound).  C gives about kScTargetCtas CTAs per launch -- few, busy CTAs
    // leave the SMs to the other calls' kernels (measured on the 32-layer
    // bench: 8 units per launch best with C = 8 of 4/8/16, 32 units with
    // C = 2-4 of 2-16) -- but at least slices of kScMaxSlice positions and
    // at most the device's cluster limit.
    const int units = I.B * I.Hkv;
    const int c_min = (max_n + kScMaxSlice - 1) / kScMaxSlice;
    const int C = std::max(std::max(1, c_min),
                           std::min(F->sampled_cluster, (kScTargetCtas + units - 1) / units));
    const int S = std::max(32, ((max_n + C - 1) / C + 31) / 32 * 32);
    if (S <= kScMaxSlice) {
      P.cluster = C;
      P.slice = S;
      Tracer tr{p->trace, stream};
      const size_t smem = select_sampled_smem_bytes(S);
      return traced(tr, CKV_KERNEL_SELECT,
                    [&] { return launch_select_sampled(P, I.B * I.Hkv, smem, stream); });
    }
  }
  // A cluster of up to 8 CTAs per unit (one CTA per unit is several times
  // slower: the four radix passes over a whole unit's keys serialise in one
  // block), at least 4096 prefix tokens and at most 16384 per CTA, and about
  // 80 CTAs per launch where the units allow: few, busy clusters leave the
  // SMs to the other calls' kernels (the ragged and 80-layer workloads ran
  // 12-13% faster with C = 4 and 2 than with 8).
  const int r = (I.P - 1) / 2;
  const int n_units = I.layer ? I.B : I.B * I.Hkv;
  const int C = std::min(8, std::max(std::max(1, (max_n + 16383) / 16384),
                                     std::min((max_n + 4095) / 4096,
                                              (kScTargetCtas + n_units - 1) / n_units)));
  const int S = std::max(32, ((max_n + C - 1) / C + 31) / 32 * 32);
  const int need = pooled_in ? S : 2 * S + 2 * r;  // floats of shared memory
  const bool fits = need <= select_max_smem_floats();
  P.cluster = C;
  P.slice = S;
  P.smem_slice = fits ? 1 : 0;
  const size_t smem = fits ? static_cast<size_t>(need) * 4 : 0;
  Tracer tr{p->trace, stream};
  return traced(tr, CKV_KERNEL_SELECT, [&] { return launch_select(P, n_units, smem, stream); });
}

int run_gather(const ckv_problem* p, const Info& I, const int32_t* indices,
               const std::vector<int>& cu_out, const void* k, const void* v, void* k_out,
               void* v_out, int* status, cudaStream_t stream) {
  const long long rows = static_cast<long long>(cu_out[I.B]) * I.Hkv;
  if (rows == 0) return CKV_OK;
  if (!indices || !k || !v || !k_out || !v_out) return CKV_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || !aligned16(k_out) || !aligned16(v_out))
    return CKV_ERR_INVALID_ARG;
  const int rv = device_readable(v, &v);
  if (rv != CKV_OK) return rv;
  static thread_local GatherParams P;
  std::memset(&P, 0, sizeof(P));
  P.k = static_cast<const uint4*>(k);
  P.v = static_cast<const uint4*>(v);
  P.k_out = static_cast<uint4*>(k_out);
  P.v_out = static_cast<uint4*>(v_out);
  P.indices = indices;
  P.status = status;
  P.tok_stride_v16 = p->kv_token_stride / 8;
  P.head_stride_v16 = p->kv_head_stride / 8;
  P.num_kv_heads = I.Hkv;
  P.o_total = cu_out[I.B];
  P.batch = I.B;
  for (int s = 0; s <= I.B; ++s) {
    P.cu_seqlens[s] = I.cu[s];
    P.cu_out[s] = cu_out[s];
  }
  Tracer tr{p->trace, stream};
  return traced(tr, CKV_KERNEL_GATHER, [&] { return launch_gather(P, rows, stream); });
}

// Per-group selection of a (multi-layer) fused call in one persistent kernel
// (fused_kernel.cu).  Sets *handled = false, enqueueing nothing, when the
// problem is outside what that kernel takes (the caller then uses the
// scoring / combine / selection kernels).  `lse` given: the window queries'
// log-sum-exp replaces the first pass.
int run_fused(const ckv_problem* p, const Info& I, const SrhLists& S, const void* q_win,
              const void* k, const void* v, const std::vector<int>& co, int32_t* indices,
              void* k_out, void* v_out, float* raw_user, float* pooled_user, void* ws,
              size_t ws_bytes, cudaStream_t stream, bool* handled, bool do_select = true,
              const LseInput& lse = LseInput{}) {
  *handled = false;
  if (I.layer || I.G > 32 || I.n_masks * I.Hkv > kFusedMaxLists || I.B > kFusedMaxSeqs)
    return CKV_OK;
  // query rows by TMA: a head block of W rows keeps the 128-byte swizzle
  // atoms aligned and leaves no padding row (W a multiple of 16), and every
  // query stride is a multiple of 16 bytes
  if (I.W % 16 != 0 || I.W > 256 || p->q_win_stride % 8 != 0 || p->q_head_stride % 8 != 0 ||
      p->q_win_stride <= 0 || p->q_head_stride <= 0 ||
      (I.B > 1 && (p->q_batch_stride % 8 != 0 || p->q_batch_stride <= 0)))
    return CKV_OK;
  int max_rows = 16;
  for (int v_ = 0; v_ < I.n_masks * I.Hkv; ++v_) max_rows = std::max(max_rows, S.rows[v_]);
  const int npad_max = (max_rows + 15) & ~15;
  const int q_half = ((npad_max * 128) + 1023) & ~1023;
  const int row_stride = (max_rows + 31) & ~31;
  // TMEM: 512 columns of accumulator buffers, tstride columns each
  const int tstride = npad_max <= 64 ? 64 : (npad_max <= 128 ? 128 : 256);
  const int nwg = 2;  // epilogue warpgroups that take tiles
  const int nbuf = 512 / tstride;
  DeviceFacts* Fd = nullptr;
  int rc = device_facts(&Fd);
  if (rc != CKV_OK) return rc;
  // three Q buffers when they fit beside a ring of at least four K tiles,
  // else two beside at least two; an even number of stages (each UMMA warp
  // has half of them)
  int stages = 0, q_bufs = 0;
  for (int nq = 3; nq >= 2 && stages == 0; --nq) {
    for (int st = 8; st >= (nq == 3 ? 4 : 2); st -= 2) {
      if (fused_smem_bytes(q_half, nq, st, row_stride, nwg) <=
          static_cast<size_t>(Fd->smem_optin)) {
        stages = st;
        q_bufs = nq;
        break;
      }
    }
  }
  if (stages == 0) return CKV_OK;  // query rows too many for two Q buffers and a ring
  *handled = true;
  if (!q_win || !k || !aligned16(q_win) || !aligned16(k)) return CKV_ERR_INVALID_ARG;
  if (do_select && (rc = check_outputs(I, co, indices, k, v, k_out, v_out)) != CKV_OK) return rc;
  const FusedLayout FL = fused_layout(I);
  if (!ws || ws_bytes < workspace_bytes(I) || (reinterpret_cast<uintptr_t>(ws) & 255u))
    return CKV_ERR_WORKSPACE;
  char* wb = static_cast<char*>(ws);

  static thread_local FusedParams P;  // large (about 15 KB): kept off the stack
  std::memset(&P, 0, sizeof(P));
  if ((rc = make_k_map(I, p, k, &P.tmap_k)) != CKV_OK) return rc;
  if ((rc = make_q_map(I, p, q_win, &P.tmap_q)) != CKV_OK) return rc;
  P.q = static_cast<const uint16_t*>(q_win);
  P.q_bs = p->q_batch_stride;
  P.q_hs = p->q_head_stride;
  P.q_ws = p->q_win_stride;
  P.lse = lse.lse;
  P.lse_bs = lse.batch_stride;
  P.lse_hs = lse.head_stride;
  P.given_lse = lse.lse ? 1 : 0;
  P.k = static_cast<const uint4*>(k);
  P.v = static_cast<const uint4*>(v);
  P.k_out = static_cast<uint4*>(k_out);
  P.v_out = static_cast<uint4*>(v_out);
  P.tok_stride_v16 = p->kv_token_stride / 8;
  P.head_stride_v16 = p->kv_head_stride / 8;
  P.indices = indices;
  P.raw = raw_user ? raw_user : reinterpret_cast<float*>(wb + FL.raw);
  P.raw_scratch = raw_user ? 0 : 1;
  {
    const long long stall = g_stall_next_ns.exchange(0);
    P.wait_ns = stall > 0 ? static_cast<unsigned long long>(stall) : kWaitTimeoutNs;
    P.stall = stall > 0 ? 1 : 0;
  }
  P.pooled = pooled_user ? pooled_user : reinterpret_cast<float*>(wb + FL.pooled);
  P.status = reinterpret_cast<int*>(wb);
  P.ctr = reinterpret_cast<int*>(wb + kFusedCtrOffset);
  P.partials = reinterpret_cast<float2*>(wb + FL.partials);
  P.bias = reinterpret_cast<float*>(wb + FL.bias);
  P.part_stride = FL.part_stride;
  P.c = static_cast<float>(static_cast<double>(I.scale) * 1.4426950408889634);
  P.window = I.W;
  P.pool_width = I.P;
  P.num_kv_heads = I.Hkv;
  P.group_size = I.G;
  P.p_total = static_cast<int>(I.p_total);
  P.o_total = co[I.B];
  P.is_bf16 = I.bf16 ? 1 : 0;
  P.n_units = I.B * I.Hkv;
  P.batch = I.B;
  P.do_select = do_select ? 1 : 0;
  P.chunk_off[0] = 0;
  for (int s_ = 0; s_ < I.B; ++s_) {
    P.cu_seqlens[s_] = I.cu[s_];
    P.cu_prefix[s_] = I.cu_prefix[s_];
    P.cu_out[s_] = co[s_];
    P.chunk_off[s_ + 1] = P.chunk_off[s_] + I.Hkv * chunks_per_unit(I, s_);
  }
  P.cu_seqlens[I.B] = I.cu[I.B];
  P.cu_prefix[I.B] = I.cu_prefix[I.B];
  P.cu_out[I.B] = co[I.B];
  P.n_chunks = P.chunk_off[I.B];
  if (P.n_chunks != FL.n_chunks) return CKV_ERR_WORKSPACE;  // cannot happen: same plan
  P.seqs_per_mask = I.spm;
  for (int m = 0; m < I.n_masks; ++m) {
    for (int g = 0; g < I.Hkv; ++g) {
      const int v_ = m * I.Hkv + g;
      uint32_t bits = 0u;
      for (int j = S.off[v_]; j < S.off[v_ + 1]; ++j) bits |= 1u << (S.heads[j] - g * I.G);
      P.srh_bits[v_] = bits;
    }
  }
  P.q_half_bytes = q_half;
  P.q_bufs = q_bufs;
  P.row_stride = row_stride;
  P.stages = stages;
  P.tstride = tstride;
  P.nbuf = nbuf;
  P.nwg = nwg;
  if (P.n_units == 0 || (P.n_chunks == 0 && (!do_select || co[I.B] == 0))) return CKV_OK;
  const size_t smem = fused_smem_bytes(q_half, q_bufs, stages, row_stride, nwg);
  Tracer tr{p->trace, stream};
  return traced(tr, CKV_KERNEL_FUSED, [&] { return launch_fused(P, Fd->sms, smem, stream); });
}

}  // namespace

// ====================================================================== C ABI
// compresskv_compress_layers under CKV_POOL_MAX: the raw scores of every
// list's i-th SRH head (one head per group at a time, scored by the per-group
// scoring path), then each head max-pooled and the heads summed, then the
// selection from those pooled scores (per group or per layer) with the
// gather.  Lists with fewer heads score their first head again in the later
// rounds (a placeholder the pooling ignores), so every round is a valid
// per-group problem.
int run_maxpool_compress(const ckv_problem* p, const Info& I, const uint8_t* srh_masks,
                         const void* q_win, const void* k, const void* v,
                         const std::vector<int>& co, int32_t* indices, void* k_out, void* v_out,
                         float* raw_scores, float* pooled_scores, const Workspace& ws,
                         void* workspace, size_t workspace_bytes, cudaStream_t st) {
  const int nl = I.n_masks * I.Hkv;
  if (nl > kFusedMaxLists || I.G > 255) return CKV_ERR_UNSUPPORTED;
  std::vector<std::vector<int>> heads(nl);
  int rounds = 0;
  for (int m = 0; m < I.n_masks; ++m)
    for (int g = 0; g < I.Hkv; ++g) {
      std::vector<int>& hl = heads[m * I.Hkv + g];
      for (int i = 0; i < I.G; ++i)
        if (srh_masks[static_cast<size_t>(m) * I.Hq + g * I.G + i]) hl.push_back(g * I.G + i);
      rounds = std::max(rounds, static_cast<int>(hl.size()));
    }
  ckv_problem pg = *p;
  pg.selection = CKV_SELECT_PER_GROUP;
  pg.pool_kind = CKV_POOL_AVG;
  Info Ig = I;
  Ig.layer = false;
  Ig.pool_max = false;
  float* slots = reinterpret_cast<float*>(static_cast<char*>(workspace) + maxpool_slots_offset(I));
  const long long slot_stride = static_cast<long long>(I.Hkv) * I.p_total;
  std::vector<uint8_t> mask_i(static_cast<size_t>(I.n_masks) * I.Hq);
  std::vector<int> co0(I.B + 1, 0);
  int rc = CKV_OK;
  for (int r = 0; r < rounds; ++r) {
    std::fill(mask_i.begin(), mask_i.end(), 0);
    for (int m = 0; m < I.n_masks; ++m)
      for (int g = 0; g < I.Hkv; ++g) {
        const std::vector<int>& hl = heads[m * I.Hkv + g];
        const int h = hl.empty() ? g * I.G : hl[std::min(r, static_cast<int>(hl.size()) - 1)];
        mask_i[static_cast<size_t>(m) * I.Hq + h] = 1;
      }
    SrhLists Si;
    if ((rc = srh_lists(Ig, mask_i.data(), Si)) != CKV_OK) return rc;
    float* raw_r = slots + r * slot_stride;
    bool handled = false;
    rc = run_fused(&pg, Ig, Si, q_win, k, nullptr, co0, nullptr, nullptr, nullptr, raw_r, nullptr,
                   workspace, workspace_bytes, st, &handled, false);
    if (!handled) rc = run_score(&pg, Ig, q_win, k, mask_i.data(), raw_r, ws.pooled, ws, st);
    if (rc != CKV_OK) return rc;
  }
  static thread_local MaxPoolParams M;
  std::memset(&M, 0, sizeof(M));
  M.slots = slots;
  M.slot_stride = slot_stride;
  float* pooled = pooled_scores ? pooled_scores : ws.pooled;
  M.pooled = pooled;
  M.raw = raw_scores;
  M.num_kv_heads = I.Hkv;
  M.batch = I.B;
  M.seqs_per_mask = I.spm;
  M.pool_width = I.P;
  M.p_total = static_cast<int>(I.p_total);
  int max_n = 0;
  for (int s = 0; s <= I.B; ++s) {
    M.cu_prefix[s] = static_cast<int>(I.cu_prefix[s]);
    if (s < I.B) max_n = std::max(max_n, I.n[s]);
  }
  for (int l = 0; l < nl; ++l) M.heads_of[l] = static_cast<uint8_t>(heads[l].size());
  Tracer tr{p->trace, st};
  if ((rc = traced(tr, CKV_KERNEL_COMBINE, [&] { return launch_maxpool(M, max_n, st); })) != CKV_OK)
    return rc;
  return run_select(p, I, nullptr, pooled, co, indices, nullptr, ws, st, k, v, k_out, v_out);
}

extern "C" {

int compresskv_debug_stall_next_fused_call(long long wait_ns) {
  if (wait_ns < 0 || (wait_ns > 0 && (wait_ns < 100000 || wait_ns > 2000000000ll)))
    return CKV_ERR_INVALID_ARG;
  g_stall_next_ns.store(wait_ns);
  return CKV_OK;
}

size_t compresskv_workspace_size(const ckv_problem* p) {
  Info I;
  if (validate(p, I) != CKV_OK) return 0;
  return workspace_bytes(I);
}

int compresskv_workspace_init(void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx_range(__func__);
  if (!workspace || workspace_bytes < kHeaderBytes) return CKV_ERR_WORKSPACE;
  return cudaMemsetAsync(workspace, 0, kHeaderBytes, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? CKV_OK
             : CKV_ERR_CUDA;
}

int compresskv_output_layout(const ckv_problem* p, const int32_t* budgets, int32_t* cu_prefix,
                             int32_t* cu_out) {
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (cu_prefix) std::copy(I.cu_prefix.begin(), I.cu_prefix.end(), cu_prefix);
  if (cu_out) {
    std::vector<int> co;
    if ((rc = output_layout(I, budgets, co)) != CKV_OK) return rc;
    std::copy(co.begin(), co.end(), cu_out);
  }
  return CKV_OK;
}

int compresskv_score(const ckv_problem* p, const void* q_win, const void* k,
                     const uint8_t* srh_mask, float* raw_scores, void* workspace,
                     size_t workspace_bytes, void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  Workspace ws;
  if ((rc = carve(I, workspace, workspace_bytes, ws)) != CKV_OK) return rc;
  if (!raw_scores) return CKV_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (!I.layer) {
    // per-group problems are scored by the kernel the fused layer call runs
    // (the same scores, bit for bit), without its selection
    SrhLists S;
    if ((rc = srh_lists(I, srh_mask, S)) != CKV_OK) return rc;
    bool handled = false;
    std::vector<int> co(I.B + 1, 0);
    rc = run_fused(p, I, S, q_win, k, nullptr, co, nullptr, nullptr, nullptr, raw_scores,
                   nullptr, workspace, workspace_bytes, st, &handled, false);
    if (handled) return rc;
  }
  return run_score(p, I, q_win, k, srh_mask, raw_scores, ws.pooled, ws, st);
}

int compresskv_select(const ckv_problem* p, const float* raw_scores, const int32_t* budgets,
                      int32_t* indices, int32_t* cu_out, float* pooled_scores, void* workspace,
                      size_t workspace_bytes, void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (I.pool_max) return CKV_ERR_UNSUPPORTED;  // needs the per-head scores
  std::vector<int> co;
  if ((rc = output_layout(I, budgets, co)) != CKV_OK) return rc;
  if (!cu_out) return CKV_ERR_INVALID_ARG;
  // per-layer selection pools the groups' summed raw scores: there is no
  // per-group pooled output to write
  if (I.layer && pooled_scores) return CKV_ERR_INVALID_ARG;
  Workspace ws;
  if ((rc = carve(I, workspace, workspace_bytes, ws)) != CKV_OK) return rc;
  std::copy(co.begin(), co.end(), cu_out);
  return run_select(p, I, raw_scores, nullptr, co, indices, pooled_scores, ws,
                    static_cast<cudaStream_t>(stream));
}

int compresskv_gather(const ckv_problem* p, const int32_t* indices, const int32_t* cu_out,
                      const void* k, const void* v, void* k_out, void* v_out, void* workspace,
                      void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (!cu_out) return CKV_ERR_INVALID_ARG;
  std::vector<int> co(cu_out, cu_out + I.B + 1);
  if (co[0] != 0) return CKV_ERR_INVALID_ARG;
  for (int s = 0; s < I.B; ++s)
    if (co[s + 1] < co[s] || co[s + 1] - co[s] > I.len[s]) return CKV_ERR_INVALID_ARG;
  if (static_cast<long long>(I.Hkv) * co[I.B] > (1LL << 31) - 1) return CKV_ERR_UNSUPPORTED;
  int* status = nullptr;
  if (workspace) {
    if (reinterpret_cast<uintptr_t>(workspace) & 255u) return CKV_ERR_WORKSPACE;
    status = static_cast<int*>(workspace);
  }
  return run_gather(p, I, indices, co, k, v, k_out, v_out, status,
                    static_cast<cudaStream_t>(stream));
}

int compresskv_compress_layer(const ckv_problem* p, const void* q_win, const void* k,
                              const void* v, const uint8_t* srh_mask, const int32_t* budgets,
                              int32_t* indices, int32_t* cu_out, void* k_out, void* v_out,
                              float* raw_scores, float* pooled_scores, void* workspace,
                              size_t workspace_bytes, void* stream) {
  NvtxRange nvtx_range(__func__);
  return compresskv_compress_layers(p, 1, q_win, k, v, srh_mask, budgets, indices, cu_out, k_out,
                                    v_out, raw_scores, pooled_scores, workspace, workspace_bytes,
                                    stream);
}

int compresskv_compress_layers(const ckv_problem* p, int n_masks, const void* q_win,
                               const void* k, const void* v, const uint8_t* srh_masks,
                               const int32_t* budgets, int32_t* indices, int32_t* cu_out,
                               void* k_out, void* v_out, float* raw_scores, float* pooled_scores,
                               void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (n_masks < 1 || I.B % n_masks != 0) return CKV_ERR_INVALID_ARG;
  if (n_masks > kMaxFusedMasks) return CKV_ERR_UNSUPPORTED;
  I.n_masks = n_masks;
  I.spm = I.B / n_masks;
  const uint8_t* srh_mask = srh_masks;
  std::vector<int> co;
  if ((rc = output_layout(I, budgets, co)) != CKV_OK) return rc;
  if (!cu_out) return CKV_ERR_INVALID_ARG;
  Workspace ws;
  if ((rc = carve(I, workspace, workspace_bytes, ws)) != CKV_OK) return rc;
  SrhLists S;
  if ((rc = srh_lists(I, srh_mask, S)) != CKV_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (I.pool_max) {
    if ((rc = check_outputs(I, co, indices, k, v, k_out, v_out)) != CKV_OK) return rc;
    std::copy(co.begin(), co.end(), cu_out);
    return run_maxpool_compress(p, I, srh_mask, q_win, k, v, co, indices, k_out, v_out,
                                raw_scores, pooled_scores, ws, workspace, workspace_bytes, st);
  }
  if (!I.layer) {
    // per-group selection: one persistent kernel for every unit of the call
    bool handled = false;
    rc = run_fused(p, I, S, q_win, k, v, co, indices, k_out, v_out, raw_scores, pooled_scores,
                   workspace, workspace_bytes, st, &handled);
    if (handled) {
      if (rc == CKV_OK) std::copy(co.begin(), co.end(), cu_out);
      return rc;
    }
  }
  if (n_masks > kMaxMasks) return CKV_ERR_UNSUPPORTED;
  float* pooled = pooled_scores ? pooled_scores : ws.pooled;
  if ((rc = check_outputs(I, co, indices, k, v, k_out, v_out)) != CKV_OK) return rc;
  std::copy(co.begin(), co.end(), cu_out);
  bool two_pass = false;
  if ((rc = run_score(p, I, q_win, k, srh_mask, raw_scores, pooled, ws, st, LseInput{},
                      &two_pass)) != CKV_OK)
    return rc;
  if (two_pass)  // raw scores only: pool and select from them
    return run_select(p, I, raw_scores ? raw_scores : ws.raw, nullptr, co, indices,
                      pooled_scores, ws, st, k, v, k_out, v_out);
  return run_select(p, I, nullptr, pooled, co, indices, nullptr, ws, st, k, v, k_out, v_out);
}

int compresskv_compress_layer_lse(const ckv_problem* p, const void* q_win, const void* k,
                                  const void* v, const float* lse_win, int64_t lse_batch_stride,
                                  int64_t lse_head_stride, const uint8_t* srh_mask,
                                  const int32_t* budgets, int32_t* indices, int32_t* cu_out,
                                  void* k_out, void* v_out, float* raw_scores,
                                  float* pooled_scores, void* workspace, size_t workspace_bytes,
                                  void* stream) {
  NvtxRange nvtx_range(__func__);
  return compresskv_compress_layers_lse(p, 1, q_win, k, v, lse_win, lse_batch_stride,
                                        lse_head_stride, srh_mask, budgets, indices, cu_out,
                                        k_out, v_out, raw_scores, pooled_scores, workspace,
                                        workspace_bytes, stream);
}

int compresskv_compress_layers_lse(const ckv_problem* p, int n_masks, const void* q_win,
                                   const void* k, const void* v, const float* lse_win,
                                   int64_t lse_batch_stride, int64_t lse_head_stride,
                                   const uint8_t* srh_masks, const int32_t* budgets,
                                   int32_t* indices, int32_t* cu_out, void* k_out, void* v_out,
                                   float* raw_scores, float* pooled_scores, void* workspace,
                                   size_t workspace_bytes, void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (I.pool_max) return CKV_ERR_UNSUPPORTED;  // needs the per-head scores
  if (n_masks < 1 || I.B % n_masks != 0) return CKV_ERR_INVALID_ARG;
  if (n_masks > kMaxFusedMasks) return CKV_ERR_UNSUPPORTED;
  I.n_masks = n_masks;
  I.spm = I.B / n_masks;
  const uint8_t* srh_mask = srh_masks;
  if (!lse_win || lse_batch_stride < 0 || lse_head_stride < 0) return CKV_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(lse_win) & 3u) return CKV_ERR_INVALID_ARG;
  std::vector<int> co;
  if ((rc = output_layout(I, budgets, co)) != CKV_OK) return rc;
  if (!cu_out) return CKV_ERR_INVALID_ARG;
  if (I.layer && pooled_scores) return CKV_ERR_INVALID_ARG;
  Workspace ws;
  if ((rc = carve(I, workspace, workspace_bytes, ws)) != CKV_OK) return rc;
  SrhLists S;
  if ((rc = srh_lists(I, srh_mask, S)) != CKV_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* raw = raw_scores ? raw_scores : ws.raw;
  if ((rc = check_outputs(I, co, indices, k, v, k_out, v_out)) != CKV_OK) return rc;
  // the scoring kernel reads lse_win for every (sequence, SRH head, window row)
  if (I.p_total > 0 && (rc = device_memory(lse_win)) != CKV_OK) return rc;
  std::copy(co.begin(), co.end(), cu_out);
  LseInput lse;
  lse.lse = lse_win;
  lse.batch_stride = lse_batch_stride;
  lse.head_stride = lse_head_stride;
  if (!I.layer) {
    // per-group selection: the persistent kernel with the given LSE in place
    // of its first pass
    bool handled = false;
    rc = run_fused(p, I, S, q_win, k, v, co, indices, k_out, v_out, raw_scores, pooled_scores,
                   workspace, workspace_bytes, st, &handled, true, lse);
    if (handled) return rc;
  }
  if (n_masks > kMaxMasks) return CKV_ERR_UNSUPPORTED;
  if ((rc = run_score(p, I, q_win, k, srh_mask, raw, nullptr, ws, st, lse)) != CKV_OK) return rc;
  return run_select(p, I, raw, nullptr, co, indices, pooled_scores, ws, st, k, v, k_out, v_out);
}

int compresskv_compress_layer_head_budgets(const ckv_problem* p, const void* q_win,
                                           const void* k, const void* v,
                                           const uint8_t* srh_mask,
                                           const int32_t* group_budgets, int32_t* indices,
                                           int32_t* cu_out, void* k_out, void* v_out,
                                           float* raw_scores, float* pooled_scores,
                                           void* workspace, size_t workspace_bytes,
                                           void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (I.pool_max) return CKV_ERR_UNSUPPORTED;  // needs the per-head scores
  if (I.layer) return CKV_ERR_INVALID_ARG;  // one shared selection has one budget
  if (!group_budgets || !cu_out) return CKV_ERR_INVALID_ARG;
  if (static_cast<long long>(I.B) * I.Hkv > kMaxBudgetUnits) return CKV_ERR_UNSUPPORTED;
  // group-major packing: group g's sequences follow each other, then group g+1
  std::vector<int2> unit_out(static_cast<size_t>(I.B) * I.Hkv);
  long long row = 0;
  for (int g = 0; g < I.Hkv; ++g) {
    for (int s = 0; s < I.B; ++s) {
      const int b = group_budgets[static_cast<long long>(s) * I.Hkv + g];
      if (b < I.W) return CKV_ERR_BUDGET;
      const int kept = std::min(b, I.len[s]);
      unit_out[static_cast<size_t>(s) * I.Hkv + g] = make_int2(static_cast<int>(row), kept);
      row += kept;
    }
  }
  if (row > (1LL << 31) - 1) return CKV_ERR_UNSUPPORTED;
  Workspace ws;
  if ((rc = carve(I, workspace, workspace_bytes, ws)) != CKV_OK) return rc;
  SrhLists S;
  if ((rc = srh_lists(I, srh_mask, S)) != CKV_OK) return rc;
  for (int g = 0; g < I.Hkv; ++g) {
    for (int s = 0; s <= I.B; ++s) {
      cu_out[g * (I.B + 1) + s] =
          s < I.B ? unit_out[static_cast<size_t>(s) * I.Hkv + g].x
                  : (g + 1 < I.Hkv ? unit_out[static_cast<size_t>(g + 1)].x : static_cast<int>(row));
    }
  }
  std::vector<int> co(I.B + 1, 0);
  co[I.B] = static_cast<int>(row);
  if ((rc = check_outputs(I, co, indices, k, v, k_out, v_out)) != CKV_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* pooled = pooled_scores ? pooled_scores : ws.pooled;
  bool two_pass = false;
  if ((rc = run_score(p, I, q_win, k, srh_mask, raw_scores, pooled, ws, st, LseInput{},
                      &two_pass)) != CKV_OK)
    return rc;
  if (two_pass)  // raw scores only: pool and select from them
    return run_select(p, I, raw_scores ? raw_scores : ws.raw, nullptr, co, indices,
                      pooled_scores, ws, st, k, v, k_out, v_out, &unit_out);
  return run_select(p, I, nullptr, pooled, co, indices, nullptr, ws, st, k, v, k_out, v_out,
                    &unit_out);
}

int compresskv_read_device_status(const void* workspace, void* stream, int32_t* status) {
  if (!workspace || !status) return CKV_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t v = 0;
  if (cudaMemcpyAsync(&v, workspace, sizeof(v), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return CKV_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return CKV_ERR_CUDA;
  *status = v;
  return CKV_OK;
}

const char* compresskv_status_string(int status) {
  switch (status) {
    case CKV_OK: return "ok";
    case CKV_ERR_INVALID_ARG: return "invalid argument";
    case CKV_ERR_UNSUPPORTED: return "unsupported problem shape";
    case CKV_ERR_BUDGET: return "budget smaller than the observation window";
    case CKV_ERR_EMPTY_SRH_GROUP: return "KV group without an SRH head";
    case CKV_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case CKV_ERR_CUDA: return "CUDA runtime error";
    case CKV_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case CKV_ERR_DEVICE_INDEX: return "gather index outside its sequence";
    case CKV_ERR_STATIC_SCRATCH:
      return "problem needs more scratch than the library's static scratch holds";
    default: return "unknown status";
  }
}

}  // extern "C"

// ====================================================================== no-alloc variant
// Scratch for compresskv_compress_layer_noalloc, for callers that cannot
// allocate device memory.  In host code `g_static_scratch` only names a
// host-side stand-in, so its device address is looked up once per device.
static __device__ __align__(256) unsigned char g_static_scratch[CKV_STATIC_SCRATCH_BYTES];

namespace {

std::mutex g_scratch_mutex;
void* g_scratch_addr[64] = {};
unsigned long long g_scratch_ctx[64] = {};  // context the address belongs to
PFN_cuCtxGetCurrent_v4000 g_ctx_current = nullptr;
PFN_cuCtxGetId_v12000 g_ctx_id = nullptr;

// Unique id of the calling thread's current context (0 if it cannot be
// read).  A device reset destroys the context the array's address was looked
// up in; the next context gets a new id.
unsigned long long current_context_id() {
  if (!g_ctx_current || !g_ctx_id) {
    void* f1 = nullptr;
    void* f2 = nullptr;
    cudaDriverEntryPointQueryResult q1, q2;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f1, 4000, cudaEnableDefault, &q1) !=
            cudaSuccess ||
        q1 != cudaDriverEntryPointSuccess ||
        cudaGetDriverEntryPointByVersion("cuCtxGetId", &f2, 12000, cudaEnableDefault, &q2) !=
            cudaSuccess ||
        q2 != cudaDriverEntryPointSuccess || !f1 || !f2) {
      cudaGetLastError();
      return 0;
    }
    g_ctx_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(f1);
    g_ctx_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(f2);
  }
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || !ctx || g_ctx_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of the static scratch on the current device, looked up once
// per device and context (again after a device reset, whose new context has
// the array at a possibly different address).
int static_scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return CKV_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  const unsigned long long ctx = current_context_id();
  if (!g_scratch_addr[dev] || ctx == 0 || ctx != g_scratch_ctx[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_static_scratch) != cudaSuccess || !ptr) {
      cudaGetLastError();
      g_scratch_addr[dev] = nullptr;
      return CKV_ERR_CUDA;
    }
    g_scratch_addr[dev] = ptr;
    // the lookup makes the device's primary context current if none was
    g_scratch_ctx[dev] = ctx != 0 ? ctx : current_context_id();
  }
  *out = g_scratch_addr[dev];
  return CKV_OK;
}

}  // namespace

extern "C" int compresskv_compress_layer_noalloc(
    const ckv_problem* p, const void* q_win, const void* k, const void* v,
    const uint8_t* srh_mask, const int32_t* budgets, int32_t* indices, int32_t* cu_out,
    void* k_out, void* v_out, float* raw_scores, float* pooled_scores, int32_t* device_status,
    void* stream) {
  NvtxRange nvtx_range(__func__);
  Info I;
  int rc = validate(p, I);
  if (rc != CKV_OK) return rc;
  if (workspace_bytes(I) > static_cast<size_t>(CKV_STATIC_SCRATCH_BYTES))
    return CKV_ERR_STATIC_SCRATCH;
  void* scratch = nullptr;
  if ((rc = static_scratch_address(&scratch)) != CKV_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // The array keeps the previous call's contents; the status word and the
  // counters must start at zero.
  if (cudaMemsetAsync(scratch, 0, kHeaderBytes, st) != cudaSuccess) return CKV_ERR_CUDA;
  rc = compresskv_compress_layer(p, q_win, k, v, srh_mask, budgets, indices, cu_out, k_out, v_out,
                                 raw_scores, pooled_scores, scratch,
                                 static_cast<size_t>(CKV_STATIC_SCRATCH_BYTES), stream);
  if (rc != CKV_OK) return rc;
  if (device_status &&
      cudaMemcpyAsync(device_status, scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice, st) !=
          cudaSuccess)
    return CKV_ERR_CUDA;
  return CKV_OK;
}
