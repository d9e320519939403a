// Building blocks shared by the selection kernels (top-k of the pooled
// scores, CompressKV Sec. 3.3) and the combine kernel's per-unit selection:
// warp scans, the K/V row copy of the retained tokens, and a CTA-wide radix
// select on fp32 bit patterns of non-negative scores (bit order == value
// order).  The radix select runs on CTAs of exactly 256 threads.
#pragma once

#include <cstdint>

#include "ckv_device.cuh"

namespace ckv {

__device__ __forceinline__ uint32_t lanemask_lt(int lane) { return (1u << lane) - 1u; }

__device__ __forceinline__ int warp_exclusive_scan(int v, int lane) {
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  return x - v;
}

// The whole CTA copies the K and V rows of `count` tokens to consecutive
// output rows: token i is out[first + i] (a position in the sequence) and goes
// to output row out0 + first + i.  Each thread moves 16-byte chunks, issuing
// a batch of loads before the matching stores.
// Kept out of line (one copy per instantiation): the selection kernels run
// once per SM and are bound by instruction fetch.
template <int kThreads, class Params>
__device__ __noinline__ void copy_kv_rows(const Params& p, int seq0, int g, const int32_t* out,
                                          int out0, int first, int count) {
  constexpr int kChunks = 2 * kHeadDim * 2 / 16;  // 16 K + 16 V chunks per token
  constexpr int kBatch = 4;
  const int total = count * kChunks;
  for (int base = 0; base < total; base += kBatch * kThreads) {
    uint4 v[kBatch];
    long long dst[kBatch];
    bool is_v[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int e = base + u * kThreads + static_cast<int>(threadIdx.x);
      dst[u] = -1;
      if (e < total) {
        const int i = e / kChunks;
        const int ch = e - i * kChunks;
        const int tok = out[first + i];
        is_v[u] = ch >= kChunks / 2;
        const int part = ch & (kChunks / 2 - 1);
        const long long src = static_cast<long long>(seq0 + tok) * p.tok_stride_v16 +
                              static_cast<long long>(g) * p.head_stride_v16 + part;
        v[u] = __ldg((is_v[u] ? p.v : p.k) + src);
        // one row per (token, group), or per token of this group when the
        // output is packed group-major (head-level budgets)
        dst[u] = (p.head_budgets ? static_cast<long long>(out0 + first + i)
                                 : static_cast<long long>(out0 + first + i) * p.num_kv_heads + g) *
                     (kHeadDim * 2 / 16) + part;
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      if (dst[u] >= 0) (is_v[u] ? p.v_out : p.k_out)[dst[u]] = v[u];
    }
  }
}

// Shared state of cta_kth_largest: four radix histograms used in rotation
// and one (OR, AND) pair of the keys per search slot.
struct RadixShared {
  uint32_t hist[4][256];
  uint32_t key_or[2], key_and[2];
};

// Zero the state cta_kth_largest expects (before the CTA's next barrier).
__device__ __forceinline__ void radix_init(RadixShared& sh) {
  const int tid = threadIdx.x;
  for (int i = tid; i < 2 * 256; i += blockDim.x) sh.hist[i >> 8][i & 255] = 0u;
  if (tid < 2) {
    sh.key_or[tid] = 0u;
    sh.key_and[tid] = 0xFFFFFFFFu;
  }
}

// Whole warp: the bin of `h[0..255]` (counts; higher bin = larger keys)
// holding the rem-th largest key, and the count of keys in the bins above it
// (every lane receives both).
__device__ __forceinline__ void warp_pick_bin256(const uint32_t* h, int rem, int lane, int* bin,
                                                 int* above_out) {
  uint32_t c[8];
  uint32_t cnt = 0u;
#pragma unroll
  for (int b = 0; b < 8; ++b) {
    c[b] = h[lane * 8 + b];
    cnt += c[b];
  }
  uint32_t suf = cnt;  // inclusive suffix sum over lanes
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_down_sync(0xffffffffu, suf, off);
    if (lane + off < 32) suf += y;
  }
  const uint32_t ok = __ballot_sync(0xffffffffu, suf >= static_cast<uint32_t>(rem));
  const int top = ok ? 31 - __clz(ok) : 0;
  uint32_t above = __shfl_sync(0xffffffffu, suf - cnt, top);  // keys above lane top's bins
  int bsel = top * 8;
  if (lane == top) {
    for (int b = 7; b >= 0; --b) {
      if (above + c[b] >= static_cast<uint32_t>(rem)) {
        bsel = top * 8 + b;
        break;
      }
      above += c[b];
    }
  }
  *bin = __shfl_sync(0xffffffffu, bsel, top);
  *above_out = static_cast<int>(__shfl_sync(0xffffffffu, above, top));
}

// CTA-wide (256 threads): the r-th largest (1 <= r <= count) of the keys
// min(keys[j] - sub, clamp), j < count, where `keys` may point to shared or
// global memory (keys[j] >= sub).  Returns that value tau; *rem = how many of
// the count keys equal tau among the r largest (the caller takes those in
// position order).  Radix passes of 8 bits start at the highest bit in which
// the keys differ; each pass has one barrier: pass number pc counts into
// hist[pc % 4] (zero on entry, as is hist[(pc + 1) % 4]) while
// hist[(pc + 2) % 4], last read two passes earlier, is cleared, and every warp
// then picks the bin itself.  `slot` selects this search's key_or / key_and
// (zero / all ones on entry).  Kept out of line: the kernels that call it run
// once per SM, so code size (instruction fetch) matters more than inlining.
static __device__ __noinline__ uint32_t cta_kth_largest(const uint32_t* keys, int count, uint32_t sub,
                                                 uint32_t clamp, int r, RadixShared& sh, int slot,
                                                 int& pc, int* rem) {
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int iters = (count + 255) >> 8;  // warp-uniform trip count
  uint32_t ko = 0u, ka = 0xFFFFFFFFu;
#pragma unroll 4
  for (int i = 0; i < iters; ++i) {
    const int j = (i << 8) + tid;
    if (j < count) {
      const uint32_t key = min(keys[j] - sub, clamp);
      ko |= key;
      ka &= key;
    }
  }
  ko = __reduce_or_sync(0xffffffffu, ko);
  ka = __reduce_and_sync(0xffffffffu, ka);
  if (lane == 0) {
    atomicOr(&sh.key_or[slot], ko);
    atomicAnd(&sh.key_and[slot], ka);
  }
  __syncthreads();
  const uint32_t diff = sh.key_or[slot] ^ sh.key_and[slot];
  const uint32_t kand = sh.key_and[slot];
  int remaining = r;
  if (diff == 0u) {  // all keys equal
    *rem = remaining;
    return kand;
  }
  int hb = 31 - __clz(diff);
  uint32_t pmask = hb == 31 ? 0u : ~((2u << hb) - 1u);
  uint32_t prefix = kand & pmask;
#pragma unroll 1
  while (hb >= 0) {
    const int width = min(8, hb + 1);
    const int shf = hb + 1 - width;
    const uint32_t fm = (1u << width) - 1u;
    uint32_t* h = sh.hist[pc & 3];
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
      const int j = (i << 8) + tid;
      const uint32_t key = j < count ? min(keys[j] - sub, clamp) : 0u;
      const bool m = j < count && (key & pmask) == prefix;
      const uint32_t act = __ballot_sync(0xffffffffu, m);
      if (!act) continue;
      const uint32_t bin = (key >> shf) & fm;
      const int leader = __ffs(act) - 1;
      const uint32_t lb = __shfl_sync(0xffffffffu, bin, leader);
      // one add per warp when its keys share the bin (dense scores), else
      // one per distinct bin of the warp
      if (__all_sync(0xffffffffu, !m || bin == lb)) {
        if (lane == leader) atomicAdd(&h[lb], static_cast<uint32_t>(__popc(act)));
      } else if (m) {
        const uint32_t same = __match_any_sync(act, bin);
        if (lane == __ffs(same) - 1) atomicAdd(&h[bin], static_cast<uint32_t>(__popc(same)));
      }
    }
    sh.hist[(pc + 2) & 3][tid] = 0u;  // one thread per bin (256 threads)
    __syncthreads();
    int bin, above;
    warp_pick_bin256(h, remaining, lane, &bin, &above);
    remaining -= above;
    prefix |= static_cast<uint32_t>(bin) << shf;
    pmask |= fm << shf;
    hb = shf - 1;
    ++pc;
  }
  *rem = remaining;
  return prefix;
}

}  // namespace ckv
