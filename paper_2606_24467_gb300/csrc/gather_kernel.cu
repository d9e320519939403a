// Eviction = keep the selected KV pairs (CompressKV Sec. 3.3): copy the
// retained K and V rows of every unit into the contiguous compressed cache.
// One warp per (output token, KV group): lanes 0-15 move the 256-byte K row,
// lanes 16-31 the V row, 16 bytes per lane.  Bit-exact copies.
#include <cuda_runtime.h>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr int kGatherThreads = 256;
constexpr int kRowsPerBlock = kGatherThreads / 32;

__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const __grid_constant__ GatherParams p) {
  pdl_launch_dependents();
  pdl_wait();  // the indices come from the select kernel
  const long long row = static_cast<long long>(blockIdx.x) * kRowsPerBlock + (threadIdx.x >> 5);
  const long long rows = static_cast<long long>(p.o_total) * p.num_kv_heads;
  if (row >= rows) return;
  const int lane = threadIdx.x & 31;
  const int i = static_cast<int>(row / p.num_kv_heads);
  const int g = static_cast<int>(row - static_cast<long long>(i) * p.num_kv_heads);
  int lo = 0, hi = p.batch;  // sequence s with cu_out[s] <= i < cu_out[s+1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.cu_out[mid] <= i) lo = mid; else hi = mid;
  }
  const int s = lo;
  const int L = p.cu_seqlens[s + 1] - p.cu_seqlens[s];
  const int idx = p.indices[static_cast<long long>(g) * p.o_total + i];
  if (idx < 0 || idx >= L) {
    if (lane == 0 && p.status) atomicCAS(p.status, 0, CKV_DEV_ERR_INDEX);
    return;
  }
  const long long src = static_cast<long long>(p.cu_seqlens[s] + idx) * p.tok_stride_v16 +
                        static_cast<long long>(g) * p.head_stride_v16;
  const long long dst = row * (kHeadDim * 2 / 16);
  const int part = lane & 15;
  if (lane < 16) {
    p.k_out[dst + part] = __ldg(p.k + src + part);
  } else {
    p.v_out[dst + part] = __ldg(p.v + src + part);
  }
}

}  // namespace

cudaError_t launch_gather(const GatherParams& p, long long rows, cudaStream_t stream) {
  if (rows <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>((rows + kRowsPerBlock - 1) / kRowsPerBlock));
  cfg.blockDim = dim3(kGatherThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gather_kernel, p);
}

}  // namespace ckv
