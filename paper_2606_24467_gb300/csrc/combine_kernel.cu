// Normalised window scores and pooling (CompressKV Sec. 3.3 scores summed over
// the SRH window queries; Sec. 4 average pooling over tokens) from the
// exponent table the scoring kernel leaves behind.
//
// For unit (s, g) the scoring kernel stored, per prefix token j and query row
// q, e_qj = 2^(z_qj*c - R) in fp16, where R = refs[tile, quarter, q] is the
// reference its warp used for that 32-token quarter, and per work item the
// pair (M_i, S_i) with  sum over the item's keys of 2^(z*c) = S_i * 2^M_i.
// This kernel
//   1. merges the pairs of the unit's items: M = max M_i,
//      S = sum S_i 2^(M_i - M), bias_q = M + log2 S  (= log2 of the softmax
//      denominator of query q);
//   2. raw_j = sum_q e_qj * 2^(R - bias_q)   (every weight is <= 1);
//   3. pooled_j = (sum_{t=-h..h} raw_{j+t}) / P with zeros outside [0, n),
//      summed in a fixed order.
// One CTA per chunk of 32-token quarters of one unit; the chunk's raw values
// and an h-token halo on each side live in shared memory.  Warps take whole
// quarters: the quarter's exponent block (32 x Nr fp16, contiguous) is read
// with coalesced 16-byte loads, and each lane's 8 columns are weighted with
// the quarter's weights (one shared-memory row per warp).
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr int kCombThreads = 256;
constexpr int kCombWarps = kCombThreads / 32;
constexpr int kLoadBatch = 4;  // 16-byte loads in flight per lane

__device__ __forceinline__ float dot8(const uint4 v, const float* w) {
  const __half2* h = reinterpret_cast<const __half2*>(&v);
  const float4 w0 = *reinterpret_cast<const float4*>(w);
  const float4 w1 = *reinterpret_cast<const float4*>(w + 4);
  const float2 a = __half22float2(h[0]);
  const float2 b = __half22float2(h[1]);
  const float2 c = __half22float2(h[2]);
  const float2 d = __half22float2(h[3]);
  float s = a.x * w0.x;
  s = fmaf(a.y, w0.y, s);
  s = fmaf(b.x, w0.z, s);
  s = fmaf(b.y, w0.w, s);
  s = fmaf(c.x, w1.x, s);
  s = fmaf(c.y, w1.y, s);
  s = fmaf(d.x, w1.z, s);
  s = fmaf(d.y, w1.w, s);
  return s;
}

__global__ void __launch_bounds__(kCombThreads)
    combine_kernel(const __grid_constant__ CombineParams p) {
  extern __shared__ float s_raw[];  // [chunk + 2h]: raw over [a - h, b + h)
  __shared__ float s_bias[kMaxQRows];
  __shared__ __align__(16) float s_w[kCombWarps][kMaxQRows];
  __shared__ float s_row[kCombWarps][32];

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const WorkItem it = p.items[blockIdx.x];
  const int s = it.seq;
  const int g = it.group;
  const int L = p.cu_seqlens[s + 1] - p.cu_seqlens[s];
  const int W = p.window;
  const int n = L - W;
  const int N = (p.srh_off[g + 1] - p.srh_off[g]) * W;
  const int Nr = expo_stride(N);
  const int cpr = Nr >> 3;  // 16-byte chunks per token row
  const int h = (p.pool_width - 1) >> 1;
  const int a = it.t0 * 32;
  const int b = min(it.t1 * 32, n);
  const int base = a - h;  // s_raw[i] holds raw_{base + i}
  const int span = b - a + 2 * h;
  const int ea = max(base, 0);
  const int eb = min(b + h, n);

  pdl_launch_dependents();
  for (int i = tid; i < span; i += kCombThreads) s_raw[i] = 0.f;
  pdl_wait();  // partials, exponents and references come from the scoring kernel

  // 1. per-query log2 softmax denominators
  for (int q = tid; q < N; q += kCombThreads) {
    float m = -INFINITY;
    for (int i = 0; i < it.count; ++i)
      m = fmaxf(m, p.partials[static_cast<long long>(it.first + i) * kMaxQRows + q].x);
    float z = 0.f;
    for (int i = 0; i < it.count; ++i) {
      const float2 pr = p.partials[static_cast<long long>(it.first + i) * kMaxQRows + q];
      if (pr.x != -INFINITY) z = fmaf(pr.y, ex2_approx(pr.x - m), z);
    }
    s_bias[q] = m + __log2f(z);
  }
  __syncthreads();

  // 2. raw scores, one 32-token quarter per warp at a time
  const bool pow2 = (32 % cpr) == 0;
  float* w = s_w[warp];
  for (int qi = (ea >> 5) + warp; qi < ((eb + 31) >> 5); qi += kCombWarps) {
    const float* rq = p.refs + it.roff + static_cast<long long>(qi) * Nr;
    for (int q = lane; q < Nr; q += 32) w[q] = q < N ? ex2_approx(rq[q] - s_bias[q]) : 0.f;
    if (!pow2) s_row[warp][lane] = 0.f;
    __syncwarp();
    const int r0 = max(ea, qi * 32) - qi * 32;
    const int r1 = min(eb, qi * 32 + 32) - qi * 32;
    const uint4* E = reinterpret_cast<const uint4*>(p.expo + it.eoff +
                                                    static_cast<long long>(qi) * 32 * Nr);
    const int fend = r1 * cpr;
    for (int f0 = r0 * cpr; f0 < fend; f0 += 32 * kLoadBatch) {
      uint4 ev[kLoadBatch];
#pragma unroll
      for (int u = 0; u < kLoadBatch; ++u) {
        const int f = f0 + 32 * u + lane;
        ev[u] = f < fend ? __ldg(E + f) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kLoadBatch; ++u) {
        const int f0u = f0 + 32 * u;
        if (f0u >= fend) break;  // uniform over the warp
        const int f = f0u + lane;
        const int row = f / cpr;
        const int col = f - row * cpr;
        float v = f < fend ? dot8(ev[u], w + 8 * col) : 0.f;
        if (pow2) {
          // the cpr lanes of one row are adjacent and aligned
          for (int off = cpr >> 1; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
          if (f < fend && col == 0) s_raw[qi * 32 + row - base] = v;
        } else if (f < fend) {
          atomicAdd(&s_row[warp][row], v);
        }
      }
    }
    __syncwarp();
    if (!pow2) {
      const int t = qi * 32 + lane;
      if (lane >= r0 && lane < r1) s_raw[t - base] = s_row[warp][lane];
      __syncwarp();  // s_row is cleared for the next quarter only after this read
    }
  }
  __syncthreads();

  // 3. pooling (and the raw scores, when asked for)
  const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const float fP = static_cast<float>(p.pool_width);
  for (int j = a + tid; j < b; j += kCombThreads) {
    const int i = j - a;
    float acc = 0.f;
    for (int t = 0; t <= 2 * h; ++t) acc += s_raw[i + t];
    p.pooled[soff + j] = acc / fP;
    if (p.raw_out) p.raw_out[soff + j] = s_raw[i + h];
  }
}

}  // namespace

size_t combine_smem_bytes(int chunk_tokens, int pool_width) {
  return static_cast<size_t>(chunk_tokens + pool_width) * sizeof(float);
}

cudaError_t combine_set_smem_limit(size_t optin, size_t* dynamic_max) {
  cudaFuncAttributes fa;
  cudaError_t e = cudaFuncGetAttributes(&fa, combine_kernel);
  if (e != cudaSuccess) return e;
  const size_t lim = optin > fa.sharedSizeBytes ? optin - fa.sharedSizeBytes : 0;
  *dynamic_max = lim;
  return cudaFuncSetAttribute(combine_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(lim));
}

cudaError_t launch_combine(const CombineParams& p, int n_items, size_t smem, cudaStream_t stream) {
  if (n_items <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n_items));
  cfg.blockDim = dim3(kCombThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, combine_kernel, p);
}

}  // namespace ckv
