// Max-pooling option of the token selection (CompressKV Sec. 3.3: the SRH
// heads' window scores are pooled across the token dimension -- width P of
// Sec. 4 -- and the heads' vectors are then combined by a sum; with max
// pooling each head is pooled before the sum).  One thread per prefix
// position: for every SRH head slot of its (sequence, group) it takes the
// largest raw score within [j - r, j + r] of the prefix and adds it, in head
// order; the raw scores are summed alongside.
#include <cuda_runtime.h>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr int kPoolThreads = 256;

__global__ void __launch_bounds__(kPoolThreads) maxpool_kernel(const __grid_constant__ MaxPoolParams p) {
  const int s = blockIdx.z;
  const int g = blockIdx.y;
  const int j = blockIdx.x * kPoolThreads + threadIdx.x;
  const int n = p.cu_prefix[s + 1] - p.cu_prefix[s];
  if (j >= n) return;
  const int heads = p.heads_of[srh_group(s, g, p.seqs_per_mask, p.num_kv_heads)];
  const long long base = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const int r = (p.pool_width - 1) >> 1;
  const int lo = max(0, j - r);
  const int hi = min(n - 1, j + r);
  float pooled = 0.f, raw = 0.f;
  for (int i = 0; i < heads; ++i) {
    const float* row = p.slots + i * p.slot_stride + base;
    float m = row[lo];
    for (int t = lo + 1; t <= hi; ++t) m = fmaxf(m, row[t]);
    pooled += m;
    raw += row[j];
  }
  p.pooled[base + j] = pooled;
  if (p.raw) p.raw[base + j] = raw;
}

}  // namespace

cudaError_t launch_maxpool(const MaxPoolParams& p, int max_n, cudaStream_t s) {
  if (max_n <= 0) return cudaSuccess;
  const dim3 grid((max_n + kPoolThreads - 1) / kPoolThreads, p.num_kv_heads, p.batch);
  maxpool_kernel<<<grid, kPoolThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace ckv
