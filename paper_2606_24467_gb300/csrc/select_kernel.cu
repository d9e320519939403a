// Pooling + budgeted top-k + window append (CompressKV Sec. 3.3: pooled
// window scores, the top-N prefix tokens are retained; Sec. 4: pooling kernel
// over the token dimension, the last W tokens are always kept).
//
// One CTA of 1024 threads per unit (sequence, KV group):
//   1. pooled_j = (sum_{t=-r..r} raw_{j+t}) / P over the prefix, zero outside
//      [0, n) (fixed summation order, so results are deterministic); the
//      pooled vector lives in shared memory when it fits, otherwise in the
//      workspace (it is re-read from L2);
//   2. the k-th largest pooled value is found exactly by a 3-pass radix select
//      on the fp32 bit patterns (pooled >= 0, so bit order == value order),
//      11/11/10 bits, shared-memory histograms with warp-aggregated atomics;
//   3. ordered compaction: every token above the k-th value plus the
//      lowest-position tokens equal to it, written in ascending position;
//      each warp owns a contiguous segment, segments are placed by one
//      block-wide scan;
//   4. the W window positions n..L-1 follow.
#include <cuda_runtime.h>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kBins = 2048;
constexpr int kSelStaticSmem = kBins * 4 + 4 * kSelWarps * 4 + 64;

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

__global__ void __launch_bounds__(kSelThreads, 1) select_kernel(const __grid_constant__ SelectParams p) {
  extern __shared__ float s_pooled[];
  __shared__ uint32_t hist[kBins];
  __shared__ int s_gt[kSelWarps], s_eq[kSelWarps], s_eqbase[kSelWarps], s_selbase[kSelWarps];
  __shared__ int s_bin, s_above;

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int u = blockIdx.x;
  const int s = u / p.num_kv_heads;
  const int g = u - s * p.num_kv_heads;
  const int L = p.cu_seqlens[s + 1] - p.cu_seqlens[s];
  const int W = p.window;
  const int n = max(L - W, 0);
  const int out0 = p.cu_out[s];
  const int kept = p.cu_out[s + 1] - out0;
  int32_t* out = p.indices + static_cast<long long>(g) * p.o_total + out0;
  const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const float* raw = p.raw + soff;
  float* buf = (n <= p.smem_floats) ? s_pooled : p.pooled_ws + soff;
  float* pout = p.pooled_out ? p.pooled_out + soff : nullptr;

  // 1. average pooling
  const int r = (p.pool_width - 1) >> 1;
  const float fP = static_cast<float>(p.pool_width);
  for (int j = tid; j < n; j += kSelThreads) {
    float a = 0.f;
    for (int t = -r; t <= r; ++t) {
      const int jj = j + t;
      if (jj >= 0 && jj < n) a += raw[jj];
    }
    const float v = a / fP;
    buf[j] = v;
    if (pout) pout[j] = v;
  }
  if (kept >= L) {  // budget covers the sequence (or L <= W): everything kept
    for (int i = tid; i < L; i += kSelThreads) out[i] = i;
    return;
  }
  const int k = kept - W;  // 0 <= k < n
  for (int w = tid; w < W; w += kSelThreads) out[k + w] = n + w;
  if (k == 0) return;
  __syncthreads();
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(buf);

  // 2. radix select of the k-th largest key
  uint32_t prefix = 0u, pmask = 0u;
  int rem = k;
#pragma unroll 1
  for (int pass = 0; pass < 3; ++pass) {
    const int sh = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
    const uint32_t nb = pass == 2 ? 1024u : 2048u;
    for (int b = tid; b < kBins; b += kSelThreads) hist[b] = 0u;
    __syncthreads();
    for (int base = 0; base < n; base += kSelThreads) {
      const int j = base + tid;
      const uint32_t key = j < n ? keys[j] : 0u;
      const bool match = j < n && (key & pmask) == prefix;
      const uint32_t bin = (key >> sh) & (nb - 1u);
      const uint32_t active = __ballot_sync(0xffffffffu, match);
      if (match) {
        const uint32_t peers = __match_any_sync(active, bin);
        if (lane == __ffs(peers) - 1) atomicAdd(&hist[bin], static_cast<uint32_t>(__popc(peers)));
      }
    }
    __syncthreads();
    if (warp == 0) {
      uint32_t cnt = 0u;
      for (int b = 0; b < kBins / 32; ++b) cnt += hist[lane * (kBins / 32) + b];
      uint32_t suf = cnt;  // inclusive suffix sum over lanes
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t y = __shfl_down_sync(0xffffffffu, suf, off);
        if (lane + off < 32) suf += y;
      }
      const uint32_t ok = __ballot_sync(0xffffffffu, suf >= static_cast<uint32_t>(rem));
      const int top = 31 - __clz(ok);  // highest lane whose suffix still holds rem keys
      const uint32_t nxt = __shfl_sync(0xffffffffu, suf, top < 31 ? top + 1 : 31);
      const uint32_t above0 = top < 31 ? nxt : 0u;
      if (lane == top) {
        uint32_t above = above0;
        int bsel = lane * (kBins / 32);
        for (int b = lane * (kBins / 32) + kBins / 32 - 1; b >= lane * (kBins / 32); --b) {
          if (above + hist[b] >= static_cast<uint32_t>(rem)) {
            bsel = b;
            break;
          }
          above += hist[b];
        }
        s_bin = bsel;
        s_above = static_cast<int>(above);
      }
    }
    __syncthreads();
    rem -= s_above;
    prefix |= static_cast<uint32_t>(s_bin) << sh;
    pmask |= (nb - 1u) << sh;
    __syncthreads();
  }
  const uint32_t tau = prefix;  // bit pattern of the k-th largest pooled value
  const int need_eq = rem;      // how many of the values equal to tau are kept

  // 3. ordered compaction
  const int seg = ((n + kSelWarps * 32 - 1) / (kSelWarps * 32)) * 32;
  const int lo = min(n, warp * seg);
  const int hi = min(n, lo + seg);
  int cgt = 0, ceq = 0;
  for (int b0 = lo; b0 < hi; b0 += 32) {
    const int j = b0 + lane;
    const bool in = j < hi;
    const uint32_t key = in ? keys[j] : 0u;
    cgt += __popc(__ballot_sync(0xffffffffu, in && key > tau));
    ceq += __popc(__ballot_sync(0xffffffffu, in && key == tau));
  }
  if (lane == 0) {
    s_gt[warp] = cgt;
    s_eq[warp] = ceq;
  }
  __syncthreads();
  if (warp == 0) {
    const int e = s_eq[lane];
    const int eq_before = warp_exclusive_scan(e, lane);
    const int take = min(max(need_eq - eq_before, 0), e);
    const int sel = s_gt[lane] + take;
    s_eqbase[lane] = eq_before;
    s_selbase[lane] = warp_exclusive_scan(sel, lane);
  }
  __syncthreads();
  int eq_seen = s_eqbase[warp];
  int pos = s_selbase[warp];
  for (int b0 = lo; b0 < hi; b0 += 32) {
    const int j = b0 + lane;
    const bool in = j < hi;
    const uint32_t key = in ? keys[j] : 0u;
    const uint32_t mgt = __ballot_sync(0xffffffffu, in && key > tau);
    const uint32_t meq = __ballot_sync(0xffffffffu, in && key == tau);
    const bool take_eq =
        in && key == tau && (eq_seen + __popc(meq & lanemask_lt(lane))) < need_eq;
    const uint32_t msel = mgt | __ballot_sync(0xffffffffu, take_eq);
    const int o = pos + __popc(msel & lanemask_lt(lane));
    if ((msel & (1u << lane)) && o < k) out[o] = j;
    pos += __popc(msel);
    eq_seen += __popc(meq);
  }
}

}  // namespace

int select_max_smem_floats() { return (227 * 1024 - kSelStaticSmem - 1024) / 4; }

cudaError_t select_set_smem_limit(size_t bytes) {
  return cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(bytes));
}

cudaError_t launch_select(const SelectParams& p, int n_units, size_t smem, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n_units));
  cfg.blockDim = dim3(kSelThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  return cudaLaunchKernelEx(&cfg, select_kernel, p);
}

}  // namespace ckv
