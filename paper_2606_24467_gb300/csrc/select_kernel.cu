// Pooling + budgeted top-k + window append (CompressKV Sec. 3.3: pooled
// window scores, the top-N prefix tokens are retained; Sec. 4: pooling kernel
// over the token dimension, the last W tokens are always kept), optionally
// fused with the K/V gather of the retained rows (Sec. 3.3 eviction).
//
// One thread-block cluster of C CTAs (C <= 8) per unit (sequence, KV group).
// CTA r of the cluster owns the contiguous prefix slice [r*S, (r+1)*S):
//   1. it stages raw[slice - halo] in shared memory (all loads in flight) and
//      computes pooled_j = (sum_{t=-h..h} raw_{j+t}) / P, zero outside [0, n),
//      in a fixed summation order (deterministic);
//   2. the k-th largest pooled value is found exactly by a 4-pass radix
//      select on the fp32 bit patterns (pooled >= 0, so bit order == value
//      order), 8 bits per pass: each CTA builds a shared-memory histogram of
//      its slice, one cluster barrier, then every CTA sums the C histograms
//      over distributed shared memory and picks the same bin (a unit with a
//      single CTA is launched without a cluster and uses __syncthreads);
//   3. ordered compaction: every token above the k-th value plus the
//      lowest-position tokens equal to it; slices are placed by an exclusive
//      scan of the per-CTA counts read over distributed shared memory;
//   4. the last CTA appends the W window positions;
//   5. (gather) each warp copies the K and V rows of the tokens it selected.
// Slices larger than the shared-memory budget keep the pooled scores in the
// workspace instead (re-read from L2).
#include <cooperative_groups.h>
#include <cuda_runtime.h>

#include "ckv_device.cuh"
#include "select_common.cuh"

namespace cg = cooperative_groups;

namespace ckv {

namespace {

constexpr int kSelThreads = 512;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kBins = 256;
constexpr int kSelStaticSmem = 2 * kBins * 4 + kBins * 4 + 8 * kSelWarps * 4 + 256;

// Cluster-wide barrier.  The .aligned forms require every thread of a warp
// to execute them together, so the warp is reconverged first.
__device__ __forceinline__ void cluster_barrier() {
  __syncwarp();
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Barrier over the CTAs that share a unit: the whole cluster, or just this
// CTA when a unit has one CTA (launched without a cluster).
template <bool kCluster>
__device__ __forceinline__ void unit_barrier() {
  if (kCluster) {
    cluster_barrier();
  } else {
    __syncthreads();
  }
}

// Shared-memory word `ptr` of CTA `rank` of this unit's cluster.
template <bool kCluster, class T>
__device__ __forceinline__ T* unit_rank_ptr(T* ptr, int rank) {
  if (kCluster) return cg::this_cluster().map_shared_rank(ptr, rank);
  return ptr;
}

template <bool kCluster>
__global__ void __launch_bounds__(kSelThreads, 1) select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ float s_dyn[];
  __shared__ uint32_t hist[2][kBins];
  __shared__ uint32_t ghist[kBins];
  __shared__ int s_gt[kSelWarps], s_eq[kSelWarps], s_eqbase[kSelWarps], s_selbase[kSelWarps];
  __shared__ int s_bin, s_above, s_cta_gt, s_cta_eq, s_cta_first, s_cta_count;

  const int C = kCluster ? static_cast<int>(cg::this_cluster().num_blocks()) : 1;
  const int crank = kCluster ? static_cast<int>(cg::this_cluster().block_rank()) : 0;
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int u = blockIdx.x / C;
  // per-layer selection: one unit per sequence whose keys are the pooled
  // scores summed over the KV groups, and whose indices every group keeps
  const bool layer = p.layer_scope != 0;
  const int s = layer ? u : u / p.num_kv_heads;
  const int g = layer ? 0 : u - s * p.num_kv_heads;
  const int nrows = layer ? p.num_kv_heads : 1;  // score rows summed into the keys
  const long long rstride = p.p_total;
  const int seq0 = p.cu_seqlens[s];
  const int L = p.cu_seqlens[s + 1] - seq0;
  const int W = p.window;
  const int n = max(L - W, 0);
  // output rows of the unit: per sequence (shared by the groups), or per
  // (sequence, group) with head-level budgets (packed group-major)
  const int out0 = p.head_budgets ? p.unit_out[u].x : p.cu_out[s];
  const int kept = p.head_budgets ? p.unit_out[u].y : p.cu_out[s + 1] - out0;
  int32_t* out = p.indices + (p.head_budgets ? 0 : static_cast<long long>(g) * p.o_total) + out0;
  const long long ostride = p.o_total;  // index rows of the groups (layer scope writes all)
  const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const float* raw = p.raw + soff;
  float* pout = p.pooled_out ? p.pooled_out + soff : nullptr;
  const int r = (p.pool_width - 1) >> 1;
  const int S = p.slice;  // prefix tokens per CTA (multiple of 32)
  const int lo = min(n, crank * S);
  const int hi = min(n, lo + S);
  const int len = hi - lo;
  const bool in_smem = p.smem_slice;
  float* raw_s = s_dyn;                                  // [S + 2r] when in_smem
  const float* pin = p.pooled_in ? p.pooled_in + soff + lo : nullptr;
  // pooled scores of the slice: shared memory, else the workspace copy (or,
  // when they arrive already pooled, the caller's buffer, read only)
  // (already pooled scores need no raw staging area in front of them)
  float* const s_pooled = s_dyn + (pin ? 0 : S + 2 * r);
  float* pooled_w =
      in_smem ? s_pooled : (layer ? p.shared_ws + p.cu_prefix[s] + lo : p.pooled_ws + soff + lo);
  const float* pooled = in_smem || layer || !pin ? pooled_w : pin;  // [len]

  pdl_launch_dependents();
  pdl_wait();  // scores come from the previous kernel

  // 1. pooling ---------------------------------------------------------------
  const float fP = static_cast<float>(p.pool_width);
  if (len > 0 && pin) {
    if (in_smem || layer) {  // already pooled: stage (and sum) the slice
      for (int base = 0; base < len; base += 8 * kSelThreads) {
        float v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int li = base + i * kSelThreads + tid;
          v[i] = li < len ? pin[li] : 0.f;
        }
        for (int rr = 1; rr < nrows; ++rr) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int li = base + i * kSelThreads + tid;
            if (li < len) v[i] += pin[rr * rstride + li];
          }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int li = base + i * kSelThreads + tid;
          if (li < len) pooled_w[li] = v[i];
        }
      }
    }
  } else if (len > 0) {
    if (in_smem) {
      const int span = len + 2 * r;
      for (int base = 0; base < span; base += 8 * kSelThreads) {
        float v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int li = base + i * kSelThreads + tid;
          const int j = lo - r + li;
          v[i] = (li < span && j >= 0 && j < n) ? raw[j] : 0.f;
        }
        for (int rr = 1; rr < nrows; ++rr) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int li = base + i * kSelThreads + tid;
            const int j = lo - r + li;
            if (li < span && j >= 0 && j < n) v[i] += raw[rr * rstride + j];
          }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int li = base + i * kSelThreads + tid;
          if (li < span) raw_s[li] = v[i];
        }
      }
      __syncthreads();
      for (int i = tid; i < len; i += kSelThreads) {
        float a = 0.f;
        for (int t = 0; t <= 2 * r; ++t) a += raw_s[i + t];
        const float pv = a / fP;
        pooled_w[i] = pv;
        if (pout) pout[lo + i] = pv;
      }
    } else {
      for (int i = tid; i < len; i += kSelThreads) {
        const int j = lo + i;
        float a = 0.f;
        for (int t = -r; t <= r; ++t) {
          const int jj = j + t;
          if (jj >= 0 && jj < n) {
            float x = raw[jj];
            for (int rr = 1; rr < nrows; ++rr) x += raw[rr * rstride + jj];
            a += x;
          }
        }
        const float pv = a / fP;
        pooled_w[i] = pv;
        if (pout) pout[j] = pv;
      }
    }
  }

  // keep-everything units (budget >= L, or L <= W): indices 0..L-1
  if (kept >= L) {
    const int per = (L + C - 1) / C;
    const int a0 = min(L, crank * per);
    const int a1 = min(L, a0 + per);
    for (int i = a0 + tid; i < a1; i += kSelThreads)
      for (int rr = 0; rr < nrows; ++rr) out[rr * ostride + i] = i;
    if (p.gather && a1 > a0) {
      __syncthreads();  // the indices written above are read back by the copy
      for (int rr = 0; rr < nrows; ++rr) copy_kv_rows<kSelThreads>(p, seq0, g + rr, out, out0, a0, a1 - a0);
    }
    return;  // uniform over the cluster: no cluster barrier is pending
  }
  const int k = kept - W;  // 0 <= k < n
  if (crank == C - 1) {
    for (int w = tid; w < W; w += kSelThreads)
      for (int rr = 0; rr < nrows; ++rr) out[rr * ostride + k + w] = n + w;
  }
  if (k == 0) {  // window only (uniform over the cluster)
    if (p.gather && crank == C - 1) {
      __syncthreads();
      for (int rr = 0; rr < nrows; ++rr) copy_kv_rows<kSelThreads>(p, seq0, g + rr, out, out0, k, W);
    }
    return;
  }
  __syncthreads();
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(pooled);

  // 2. radix select of the k-th largest key --------------------------------
  uint32_t prefix = 0u, pmask = 0u;
  int rem = k;
#pragma unroll 1
  for (int pass = 0; pass < 4; ++pass) {
    const int sh = 24 - 8 * pass;
    uint32_t* h = hist[pass & 1];
    for (int b = tid; b < kBins; b += kSelThreads) h[b] = 0u;
    __syncthreads();
    for (int base = 0; base < len; base += kSelThreads) {
      const int i = base + tid;
      const uint32_t key = i < len ? keys[i] : 0u;
      const bool match = i < len && (key & pmask) == prefix;
      const uint32_t bin = (key >> sh) & 255u;
      const uint32_t active = __ballot_sync(0xffffffffu, match);
      if (active) {
        // one add per warp when its keys share the bin, else one per
        // distinct bin of the warp
        const int leader = __ffs(active) - 1;
        const uint32_t lb = __shfl_sync(0xffffffffu, bin, leader);
        if (__all_sync(0xffffffffu, !match || bin == lb)) {
          if (lane == leader) atomicAdd(&h[lb], static_cast<uint32_t>(__popc(active)));
        } else if (match) {
          const uint32_t same = __match_any_sync(active, bin);
          if (lane == __ffs(same) - 1) atomicAdd(&h[bin], static_cast<uint32_t>(__popc(same)));
        }
      }
    }
    unit_barrier<kCluster>();
    for (int b = tid; b < kBins; b += kSelThreads) {
      uint32_t part[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) part[q] = q < C ? unit_rank_ptr<kCluster>(h, q)[b] : 0u;
      uint32_t tot = 0u;
#pragma unroll
      for (int q = 0; q < 8; ++q) tot += part[q];
      ghist[b] = tot;
    }
    __syncthreads();
    if (warp == 0) {
      uint32_t cnt = 0u;
#pragma unroll
      for (int b = 0; b < kBins / 32; ++b) cnt += ghist[lane * (kBins / 32) + b];
      uint32_t suf = cnt;  // inclusive suffix sum over lanes
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t y = __shfl_down_sync(0xffffffffu, suf, off);
        if (lane + off < 32) suf += y;
      }
      const uint32_t ok = __ballot_sync(0xffffffffu, suf >= static_cast<uint32_t>(rem));
      const int top = ok ? 31 - __clz(ok) : 0;
      const uint32_t nxt = __shfl_sync(0xffffffffu, suf, top < 31 ? top + 1 : 31);
      if (lane == top) {
        uint32_t above = top < 31 ? nxt : 0u;
        int bsel = lane * (kBins / 32);
        for (int b = lane * (kBins / 32) + kBins / 32 - 1; b >= lane * (kBins / 32); --b) {
          if (above + ghist[b] >= static_cast<uint32_t>(rem)) {
            bsel = b;
            break;
          }
          above += ghist[b];
        }
        s_bin = bsel;
        s_above = static_cast<int>(above);
      }
    }
    __syncthreads();
    rem -= s_above;
    prefix |= static_cast<uint32_t>(s_bin) << sh;
    pmask |= 255u << sh;
  }
  const uint32_t tau = prefix;  // bit pattern of the k-th largest pooled value
  const int need_eq = rem;      // how many of the values equal to tau are kept

  // 3. ordered compaction ----------------------------------------------------
  const int seg = ((len + kSelWarps * 32 - 1) / (kSelWarps * 32)) * 32;
  const int wlo = min(len, warp * seg);
  const int whi = min(len, wlo + seg);
  int cgt = 0, ceq = 0;
  for (int b0 = wlo; b0 < whi; b0 += 32) {
    const int i = b0 + lane;
    const bool in = i < whi;
    const uint32_t key = in ? keys[i] : 0u;
    cgt += __popc(__ballot_sync(0xffffffffu, in && key > tau));
    ceq += __popc(__ballot_sync(0xffffffffu, in && key == tau));
  }
  if (lane == 0) {
    s_gt[warp] = cgt;
    s_eq[warp] = ceq;
  }
  __syncthreads();
  if (warp == 0) {
    const int e = lane < kSelWarps ? s_eq[lane] : 0;
    const int gt = lane < kSelWarps ? s_gt[lane] : 0;
    const int eq_incl = warp_exclusive_scan(e, lane) + e;
    const int gt_incl = warp_exclusive_scan(gt, lane) + gt;
    if (lane == 31) {
      s_cta_gt = gt_incl;
      s_cta_eq = eq_incl;
    }
  }
  unit_barrier<kCluster>();  // every CTA's totals are visible
  if (warp == 0) {
    // totals of the lower-ranked CTAs of the cluster
    int gt_before = 0, eq_before = 0;
    for (int q = 0; q < crank; ++q) {
      gt_before += *unit_rank_ptr<kCluster>(&s_cta_gt, q);
      eq_before += *unit_rank_ptr<kCluster>(&s_cta_eq, q);
    }
    const int take_before = min(need_eq, eq_before);  // ties are taken in position order
    const int e = lane < kSelWarps ? s_eq[lane] : 0;
    const int w_eq_before = eq_before + warp_exclusive_scan(e, lane);
    const int take = min(max(need_eq - w_eq_before, 0), e);
    const int sel = (lane < kSelWarps ? s_gt[lane] : 0) + take;
    const int sel_before = warp_exclusive_scan(sel, lane);  // every lane takes part
    const int sel_total = __shfl_sync(0xffffffffu, sel_before + sel, 31);
    if (lane < kSelWarps) {
      s_eqbase[lane] = w_eq_before;
      s_selbase[lane] = gt_before + take_before + sel_before;
    }
    if (lane == 0) {
      s_cta_first = gt_before + take_before;  // this CTA's first output slot
      s_cta_count = sel_total;                // and how many it fills
    }
  }
  unit_barrier<kCluster>();  // no CTA leaves while others may still read its shared memory
  int eq_seen = s_eqbase[warp];
  int pos = s_selbase[warp];
  for (int b0 = wlo; b0 < whi; b0 += 32) {
    const int i = b0 + lane;
    const bool in = i < whi;
    const uint32_t key = in ? keys[i] : 0u;
    const uint32_t mgt = __ballot_sync(0xffffffffu, in && key > tau);
    const uint32_t meq = __ballot_sync(0xffffffffu, in && key == tau);
    const bool take_eq =
        in && key == tau && (eq_seen + __popc(meq & lanemask_lt(lane))) < need_eq;
    const uint32_t msel = mgt | __ballot_sync(0xffffffffu, take_eq);
    const int o = pos + __popc(msel & lanemask_lt(lane));
    if ((msel & (1u << lane)) && o < k)
      for (int rr = 0; rr < nrows; ++rr) out[rr * ostride + o] = lo + i;
    pos += __popc(msel);
    eq_seen += __popc(meq);
  }
  if (p.gather) {
    // 5. copy this CTA's retained rows (and the window, last CTA)
    __syncthreads();  // the indices written above are read back by the copy
    const int cta_first = s_cta_first;
    const int cta_count = min(k - cta_first, s_cta_count);
    for (int rr = 0; rr < nrows; ++rr) {
      if (cta_count > 0) copy_kv_rows<kSelThreads>(p, seq0, g + rr, out, out0, cta_first, cta_count);
      if (crank == C - 1) copy_kv_rows<kSelThreads>(p, seq0, g + rr, out, out0, k, W);
    }
  }
}


// ---------------------------------------------------------------------------
// Sampled cluster select (per-group selection of a fused layer call): the same
// result as select_kernel -- the top-k prefix positions of every unit by
// pooled score, ties to the lower position, ascending, the window appended,
// the K/V rows copied -- with three cluster barriers (five on a retry)
// instead of one per radix pass.  One cluster of C <= 16 CTAs per unit; CTA r owns the contiguous
// slice [r*S, (r+1)*S) of the unit's prefix positions.
//   1. The slice's pooled scores go to shared memory; each CTA sends 256 / C
//      evenly spaced scores of its slice to every CTA of the cluster.
//   2. Every CTA takes the same lower bound lo for the k-th largest score:
//      the r-th largest sample (found by counting, for every sample, the
//      samples above it), r a few standard deviations above the expected
//      number k * (samples / n) of samples above the k-th score.
//   3. Each CTA lists its keys >= lo in position order and sends the count.
//      If fewer than k keys reach lo (a unit whose few top keys hold several
//      samples), steps 2-3 run once more with the r whose expected count of
//      keys above it is halfway between k and kScCandCap.
//      When between k and kScCandCap keys reach lo (the usual case), every
//      CTA reads all lists (position order across the cluster), finds the
//      k-th largest key tau and how many keys equal to it are kept (radix
//      passes over min(key - lo, 2^16 - 1), which resolve tau whenever it is
//      below lo + 2^16 - 1, else over the keys themselves), and writes its
//      own selected positions at offsets counted in that list.
//      Otherwise every CTA runs the same search over all of the unit's
//      scores (read from global memory) and counts from there.
//   4. The last CTA appends the window; every CTA copies its own K/V rows.
// Pooled scores are >= 0, so their fp32 bit patterns order like the values.
constexpr int kScThreads = 256;
constexpr int kScWarps = kScThreads / 32;
constexpr int kScSampleTotal = 256;  // samples per unit (kScSampleTotal / C per CTA)
constexpr int kScMaxC = 16;       // CTAs per cluster
constexpr int kScCandCap = 4096;  // candidates per unit
static_assert(kScThreads == 256 && kScSampleTotal == kScThreads, "one thread per radix bin and per sample");

struct ScShared {
  int samp[kScSampleTotal];  // keys as int (>= 0); -1 = no sample; written by every CTA
  int samp_cnt[kScMaxC];
  int cand_cnt[kScMaxC];
  int cand_off[kScMaxC + 1];
  int ovf[kScMaxC];
  uint32_t ckey[kScCandCap];  // own candidates, position order
  int cpos[kScCandCap];
  uint32_t all[kScCandCap];   // every CTA's candidates, position order
  RadixShared rs;
  int wcnt[kScWarps];
  int wbase[kScWarps];
  int red[2][2];              // one pair of sums per use
  int red0;
  uint32_t lo;
};

// Zero state the searches below expect (before the kernel's first barrier).
__device__ __forceinline__ void sc_init_shared(ScShared& sh, int sampled_slots) {
  const int tid = threadIdx.x;
  if (tid >= sampled_slots && tid < kScSampleTotal) sh.samp[tid] = -1;  // slots no CTA fills
  radix_init(sh.rs);
  if (tid < 2) {
    sh.red[tid][0] = 0;
    sh.red[tid][1] = 0;
  }
}

__device__ __forceinline__ void cluster_arrive_relaxed() {
  __syncwarp();
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
  __syncwarp();
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  __syncwarp();
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// CTA-wide sums of two ints into sh.red[slot] (zero on entry; every thread
// receives both).
__device__ __forceinline__ void cta_sum2(int a, int b, ScShared& sh, int slot, int* sa, int* sb) {
  a = __reduce_add_sync(0xffffffffu, a);
  b = __reduce_add_sync(0xffffffffu, b);
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(&sh.red[slot][0], a);
    atomicAdd(&sh.red[slot][1], b);
  }
  __syncthreads();
  *sa = sh.red[slot][0];
  *sb = sh.red[slot][1];
}

__global__ void __launch_bounds__(kScThreads)
    select_sampled_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ __align__(16) uint8_t sc_raw[];
  ScShared& sh = *reinterpret_cast<ScShared*>(sc_raw);
  float* s_keys = reinterpret_cast<float*>(sc_raw + ((sizeof(ScShared) + 15) & ~size_t(15)));
  cg::cluster_group cluster = cg::this_cluster();
  const int C = static_cast<int>(cluster.num_blocks());
  const int cr = static_cast<int>(cluster.block_rank());
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int u = blockIdx.x / C;
  const int s = u / p.num_kv_heads;
  const int g = u - s * p.num_kv_heads;
  const int seq0 = p.cu_seqlens[s];
  const int L = p.cu_seqlens[s + 1] - seq0;
  const int W = p.window;
  const int n = max(L - W, 0);
  const int out0 = p.head_budgets ? p.unit_out[u].x : p.cu_out[s];
  const int kept = p.head_budgets ? p.unit_out[u].y : p.cu_out[s + 1] - out0;
  int32_t* out = p.indices + (p.head_budgets ? 0 : static_cast<long long>(g) * p.o_total) + out0;
  const float* pooled = p.pooled_in + static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const uint32_t* gkeys = reinterpret_cast<const uint32_t*>(pooled);
  const int S = p.slice;
  const int lo_c = min(n, cr * S);
  const int len = min(n, lo_c + S) - lo_c;

  pdl_launch_dependents();
  cluster_arrive_relaxed();  // this CTA has started (remote shared memory may be written)
  pdl_wait();                // pooled scores come from the previous kernel

  if (kept >= L) {  // keep everything (uniform over the cluster)
    const int per = (L + C - 1) / C;
    const int a0 = min(L, cr * per);
    const int a1 = min(L, a0 + per);
    for (int i = a0 + tid; i < a1; i += kScThreads) out[i] = i;
    if (p.gather && a1 > a0) {
      __syncthreads();
      copy_kv_rows<kScThreads>(p, seq0, g, out, out0, a0, a1 - a0);
    }
    cluster_wait();
    return;
  }
  const int k = kept - W;  // 0 <= k < n
  if (cr == C - 1)
    for (int w = tid; w < W; w += kScThreads) out[k + w] = n + w;
  if (k == 0) {
    if (p.gather && cr == C - 1) {
      __syncthreads();
      copy_kv_rows<kScThreads>(p, seq0, g, out, out0, 0, W);
    }
    cluster_wait();
    return;
  }

  // 1. slice -> shared memory; samples to every CTA
  const int per_cta = kScSampleTotal / C;
  sc_init_shared(sh, C * per_cta);
  int pc = 0;  // radix passes run so far (histogram rotation)
  for (int i = tid; i < len; i += kScThreads) cp_async4(smem_u32(s_keys + i), pooled + lo_c + i);
  cp_async_wait_all();
  __syncthreads();
  auto key_at = [&](int i) { return __float_as_uint(s_keys[i]); };
  const int ns_c = min(per_cta, len);
  cluster_wait();  // every CTA has started
  if (tid < per_cta) {
    const int v = tid < ns_c
                      ? static_cast<int>(key_at(static_cast<int>((static_cast<long long>(tid) * len) / ns_c)))
                      : -1;
    for (int t = 0; t < C; ++t) *cluster.map_shared_rank(&sh.samp[cr * per_cta + tid], t) = v;
  }
  if (tid < C) *cluster.map_shared_rank(&sh.samp_cnt[cr], tid) = ns_c;
  cluster_arrive_release();
  cluster_wait();

  // 2.-3. A lower bound lo from the samples, then every CTA's candidates
  //    (keys >= lo); a second, looser bound when the first leaves fewer than
  //    k candidates (a unit whose top keys are few and happen to hold
  //    several samples), before the full search.
  int nsamp = 0;
  for (int c = 0; c < C; ++c) nsamp += sh.samp_cnt[c];
  const float mu = static_cast<float>(k) * static_cast<float>(nsamp) / static_cast<float>(n);
  int rs = min(nsamp, static_cast<int>(ceilf(mu + 3.f * sqrtf(mu))) + 2);
  uint32_t lo = 0;
  int own = 0, total = 0, before = 0, any_ovf = 0;
  for (int attempt = 0; attempt < 2; ++attempt) {
    // the rs-th largest sample, by counting for each sample the samples
    // above it and equal to it
    {
      const int v = sh.samp[tid];  // kScThreads == kScSampleTotal: one sample per thread
      const int4* s4 = reinterpret_cast<const int4*>(sh.samp);
      int gt = 0, eq = 0;
#pragma unroll 8
      for (int j = 0; j < kScSampleTotal / 4; ++j) {  // empty slots (-1) never count
        const int4 x = s4[j];
        gt += (x.x > v) + (x.y > v) + (x.z > v) + (x.w > v);
        eq += (x.x == v) + (x.y == v) + (x.z == v) + (x.w == v);
      }
      if (v >= 0 && gt < rs && rs <= gt + eq) sh.lo = static_cast<uint32_t>(v);  // equal samples agree
    }
    __syncthreads();
    lo = sh.lo;

    // own candidates (keys >= lo) in position order; counts to every CTA
    const int seg = ((len + kScThreads - 1) / kScThreads) * 32;  // positions per warp
    const int wlo = min(len, warp * seg);
    const int whi = min(len, wlo + seg);
    int wc = 0;
#pragma unroll 4
    for (int b0 = wlo; b0 < whi; b0 += 32) {
      const int i = b0 + lane;
      wc += __popc(__ballot_sync(0xffffffffu, i < whi && key_at(i) >= lo));
    }
    if (lane == 0) sh.wcnt[warp] = wc;
    __syncthreads();
    if (warp == 0) {
      const int v = lane < kScWarps ? sh.wcnt[lane] : 0;
      const int ex = warp_exclusive_scan(v, lane);
      if (lane < kScWarps) sh.wbase[lane] = ex;
      if (lane == kScWarps - 1) sh.red0 = ex + v;  // own candidate count
    }
    __syncthreads();
    own = sh.red0;
    {
      int o = sh.wbase[warp];
#pragma unroll 2
      for (int b0 = wlo; b0 < whi; b0 += 32) {
        const int i = b0 + lane;
        const uint32_t key = i < whi ? key_at(i) : 0u;
        const bool c = i < whi && key >= lo;
        const uint32_t mm = __ballot_sync(0xffffffffu, c);
        const int slot = o + __popc(mm & lanemask_lt(lane));
        if (c && slot < kScCandCap) {
          sh.ckey[slot] = key;
          sh.cpos[slot] = lo_c + i;
        }
        o += __popc(mm);
      }
    }
    if (tid < C) {
      *cluster.map_shared_rank(&sh.cand_cnt[cr], tid) = own;
      *cluster.map_shared_rank(&sh.ovf[cr], tid) = own > kScCandCap ? 1 : 0;
    }
    __syncthreads();  // own list complete before the others may read it
    cluster_arrive_release();
    cluster_wait();
    total = before = any_ovf = 0;
    for (int c = 0; c < C; ++c) {
      if (c < cr) before += sh.cand_cnt[c];
      total += sh.cand_cnt[c];
      any_ovf |= sh.ovf[c];
    }
    // the same decision in every CTA of the cluster
    if (attempt == 1 || any_ovf || total >= k || rs >= nsamp) break;
    // the rank whose expected count of keys above it lies halfway between k
    // and the candidate capacity
    rs = min(nsamp, max(rs + 1, static_cast<int>(ceilf(0.5f * static_cast<float>(k + kScCandCap) *
                                                       static_cast<float>(nsamp) /
                                                       static_cast<float>(n)))));
    // every CTA has read this round's counts before they are overwritten
    cluster_arrive_release();
    cluster_wait();
  }
  const bool fast = !any_ovf && total >= k && total <= kScCandCap;

  // k-th largest key tau, keys equal to it that are kept, and this CTA's
  // counts of keys > tau / == tau at lower positions of the unit
  uint32_t tau;
  int need_eq, gt_before, eq_before;
  if (fast) {
    // every CTA's list, concatenated in cluster (= position) order
    if (warp == 0) {
      const int cc = lane < C ? sh.cand_cnt[lane] : 0;
      const int ex = warp_exclusive_scan(cc, lane);
      if (lane <= C) sh.cand_off[lane] = ex;
    }
    __syncthreads();
#pragma unroll 4
    for (int j = tid; j < total; j += kScThreads) {
      int c = 0;
      for (int q = 1; q < C; ++q) c += j >= sh.cand_off[q] ? 1 : 0;
      sh.all[j] = *cluster.map_shared_rank(&sh.ckey[j - sh.cand_off[c]], c);
    }
    __syncthreads();
    cluster_arrive_release();  // done reading the other CTAs' shared memory
    // offsets above lo, clamped to 16 bits: at most two passes
    constexpr uint32_t kClamp = 0xFFFFu;
    const uint32_t td = cta_kth_largest(sh.all, total, lo, kClamp, k, sh.rs, 0, pc, &need_eq);
    tau = lo + td;
    if (td == kClamp)  // tau at or above the clamp: the keys themselves
      tau = cta_kth_largest(sh.all, total, 0u, 0xFFFFFFFFu, k, sh.rs, 1, pc, &need_eq);
    int a = 0, b = 0;
#pragma unroll 4
    for (int j = tid; j < before; j += kScThreads) {
      a += sh.all[j] > tau ? 1 : 0;
      b += sh.all[j] == tau ? 1 : 0;
    }
    cta_sum2(a, b, sh, 0, &gt_before, &eq_before);
  } else {
    cluster_arrive_release();
    tau = cta_kth_largest(gkeys, n, 0u, 0xFFFFFFFFu, k, sh.rs, 1, pc, &need_eq);
    int a = 0, b = 0;
    for (int j = tid; j < lo_c; j += kScThreads) {
      const uint32_t key = __ldg(gkeys + j);
      a += key > tau ? 1 : 0;
      b += key == tau ? 1 : 0;
    }
    cta_sum2(a, b, sh, 1, &gt_before, &eq_before);
  }

  // 4. this CTA's selected positions (keys > tau, and keys == tau while fewer
  //    than need_eq equal keys precede them), in position order
  const int take_before = min(eq_before, need_eq);
  const int first = gt_before + take_before;  // first output slot of this CTA
  int count = 0;
  {
    int o = first;
    int eq_seen = eq_before;
    // scan the own keys >= tau in position order: the candidate list when it
    // is complete, else the slice
    const bool use_list = fast;
    const int m = use_list ? own : len;
    for (int j0 = 0; j0 < m; j0 += 32 * kScWarps) {
      // one warp-wide step per 32 entries, warps in order
      const int j = j0 + warp * 32 + lane;
      const bool in = j < m;
      const uint32_t key = in ? (use_list ? sh.ckey[j] : key_at(j)) : 0u;
      const int pos = in ? (use_list ? sh.cpos[j] : lo_c + j) : 0;
      const bool gt = in && key > tau;
      const bool eq = in && key == tau;
      const uint32_t mgt = __ballot_sync(0xffffffffu, gt);
      const uint32_t meq = __ballot_sync(0xffffffffu, eq);
      if (lane == 0) {
        sh.wcnt[warp] = __popc(mgt);
        sh.wbase[warp] = __popc(meq);
      }
      __syncthreads();
      int gtb = 0, eqb = 0;
      for (int w = 0; w < warp; ++w) {
        gtb += sh.wcnt[w];
        eqb += sh.wbase[w];
      }
      int gtt = gtb, eqt = eqb;
      for (int w = warp; w < kScWarps; ++w) {
        gtt += sh.wcnt[w];
        eqt += sh.wbase[w];
      }
      const int eq_rank = eq_seen + eqb + __popc(meq & lanemask_lt(lane));
      const bool take_eq = eq && eq_rank < need_eq;
      const uint32_t msel = mgt | __ballot_sync(0xffffffffu, take_eq);
      // selected entries before this lane: earlier warps' (gt + taken eq) + this warp's
      const int eq_taken_before = max(0, min(need_eq - eq_seen, eqb));
      const int slot = o + gtb + eq_taken_before + __popc(msel & lanemask_lt(lane));
      if ((msel >> lane) & 1u) {
        if (slot < k) out[slot] = pos;
      }
      const int eq_taken = max(0, min(need_eq - eq_seen, eqt));
      o += gtt + eq_taken;
      eq_seen += eqt;
      __syncthreads();  // wcnt / wbase are rewritten by the next step
    }
    count = o - first;
  }
  if (p.gather) {
    __syncthreads();  // the indices written above are read back by the copy
    const int cnt = min(count, k - first);
    if (cnt > 0) copy_kv_rows<kScThreads>(p, seq0, g, out, out0, first, cnt);
    if (cr == C - 1) copy_kv_rows<kScThreads>(p, seq0, g, out, out0, k, W);
  }
  cluster_wait();  // no CTA leaves while another may still read its candidates
}

}  // namespace

size_t select_sampled_smem_bytes(int slice) {
  return ((sizeof(ScShared) + 15) & ~size_t(15)) + static_cast<size_t>(slice) * sizeof(float);
}

int select_sampled_max_cluster(int slice) {
  // clusters of 16 CTAs are a non-portable size: use them when the device
  // can hold one (else 8)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kScMaxC);
  cfg.blockDim = dim3(kScThreads);
  cfg.dynamicSmemBytes = select_sampled_smem_bytes(slice);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kScMaxC;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, select_sampled_kernel, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 8;
  }
  return clusters > 0 ? kScMaxC : 8;
}

cudaError_t launch_select_sampled(const SelectParams& p, int n_units, size_t smem,
                                  cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n_units * p.cluster));
  cfg.blockDim = dim3(kScThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(p.cluster);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, select_sampled_kernel, p);
}

int select_max_smem_floats() { return (227 * 1024 - kSelStaticSmem - 1024) / 4; }

cudaError_t select_set_smem_limit(size_t bytes) {
  cudaError_t e = cudaFuncSetAttribute(select_sampled_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(select_sampled_smem_bytes(kScMaxSlice)));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(select_sampled_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(select_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(bytes));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(select_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(bytes));
}

cudaError_t launch_select(const SelectParams& p, int n_units, size_t smem, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n_units * p.cluster));
  cfg.blockDim = dim3(kSelThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (p.cluster <= 1) return cudaLaunchKernelEx(&cfg, select_kernel<false>, p);
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(p.cluster);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, select_kernel<true>, p);
}

}  // namespace ckv
