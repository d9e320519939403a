// Normalised window scores and pooling (CompressKV Sec. 3.3 scores summed over
// the SRH window queries; Sec. 4 average pooling over tokens) from the tables
// the scoring kernel leaves behind.
//
// For unit (s, g) the scoring kernel stored, per prefix key j and query row
// q, e_qj = 2^(z_qj*c - R) in fp16, where R = refs[quarter(j), q] is the
// reference its warp used for that 32-key quarter, and per query row
// bias_q = log2 D_q, the log2 of its softmax denominator.  This kernel
//   1. raw_j = sum_q e_qj * 2^(R - bias_q)   (every weight is <= 1);
//   2. pooled_j = (sum_{t=-h..h} raw_{j+t}) / P with zeros outside [0, n),
//      summed in a fixed order.
// One CTA per chunk of 32-key quarters of one unit.  The unit's bias row, the
// references of every quarter the chunk touches (the chunk plus an h-key
// halo on each side) and the first exponent rows are requested together;
// the weights 2^(R - bias_q) are then tabulated in shared memory and the
// exponent rows of those keys -- one contiguous region -- are streamed by the
// whole block, two batches of kLoadBatch 16-byte loads in flight per thread.
// Thread tid always meets the same
// 8-column chunk of a row (tid % cpr, where cpr = Nr / 8 divides 32); the
// cpr threads of a row are adjacent lanes and add their dot products by
// shuffles.  Raw scores of the chunk and halo stay in shared memory for the
// pooling.  The table lines only this chunk reads are then discarded from
// L2 (`discard.global.L2`): the table is dead, so its dirty lines need not be
// written back to DRAM.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr int kCombThreads = 256;
constexpr int kLoadBatch = 4;  // 16-byte loads per batch (two batches in flight per thread)
static_assert(kMaxQRows <= kCombThreads, "one thread per query row");

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
  extern __shared__ __align__(16) float s_dyn[];  // weights [nqt][Nr] | raw [span]
  __shared__ float s_bias[kMaxQRows];

  const int tid = threadIdx.x;
  const WorkItem it = p.items[blockIdx.x];
  const int s = it.seq;
  const int g = it.group;
  const int L = p.cu_seqlens[s + 1] - p.cu_seqlens[s];
  const int W = p.window;
  const int n = L - W;
  const int vg = srh_group(s, g, p.seqs_per_mask, p.num_kv_heads);
  const int N = (p.srh_off[vg + 1] - p.srh_off[vg]) * W;
  const int Nr = expo_stride(N);
  const int cpr = Nr >> 3;  // 16-byte chunks per key row (a power of two <= 32)
  const int lg_cpr = __ffs(cpr) - 1;
  const int col = tid & (cpr - 1);
  const int h = (p.pool_width - 1) >> 1;
  const int a = it.t0 * 32;
  const int b = min(it.t1 * 32, n);
  const int base = a - h;  // s_raw[i] holds raw_{base + i}
  const int span = b - a + 2 * h;
  const int ea = max(base, 0);
  const int eb = min(b + h, n);
  const int q0 = ea >> 5;
  const int nqt = ((eb + 31) >> 5) - q0;  // quarters touched
  float* s_w = s_dyn;
  float* s_raw = s_dyn + nqt * Nr;

  for (int i = tid; i < span; i += kCombThreads) s_raw[i] = 0.f;
  pdl_wait();  // denominators and tables come from the scoring kernel

  // Everything below depends on three independent reads -- the unit's
  // denominators, the references of the quarters touched and the exponent
  // rows -- so all three are issued before any of them is waited on.
  const uint4* E4 = reinterpret_cast<const uint4*>(p.expo + it.eoff);
  const int f_lo = ea * cpr;
  const int f_hi = eb * cpr;
  uint4 ev[kLoadBatch];
  auto load_batch = [&](int f0, uint4 (&dst)[kLoadBatch]) {
#pragma unroll
    for (int u = 0; u < kLoadBatch; ++u) {
      const int f = f0 + u * kCombThreads + tid;
      dst[u] = f < f_hi ? __ldg(E4 + f) : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  load_batch(f_lo, ev);
  // references (16-byte chunks: nqt * Nr is a multiple of 8 and the rows are
  // 32-byte aligned) and denominators arrive by asynchronous copies
  const float* R = p.refs + it.roff + static_cast<long long>(q0) * Nr;
  for (int i = 4 * tid; i < nqt * Nr; i += 4 * kCombThreads) cp_async16(smem_u32(s_w + i), R + i);
  if (tid < N) cp_async4(smem_u32(s_bias + tid), p.bias + static_cast<long long>(it.first) * kMaxQRows + tid);
  cp_async_wait_all();
  __syncthreads();

  // weights 2^(R - bias_q) of the quarters touched, in place
  for (int i = tid; i < nqt * Nr; i += kCombThreads) {
    const int cc = i & (Nr - 1);
    s_w[i] = cc < N ? ex2_approx(s_w[i] - s_bias[cc]) : 0.f;
  }
  __syncthreads();

  // 1. raw scores of the keys [ea, eb): one contiguous run of exponent rows,
  //    the next batch in flight while the current one is reduced
  for (int f0 = f_lo; f0 < f_hi; f0 += kLoadBatch * kCombThreads) {
    uint4 nx[kLoadBatch];
    const int f1 = f0 + kLoadBatch * kCombThreads;
    if (f1 < f_hi) load_batch(f1, nx);
#pragma unroll
    for (int u = 0; u < kLoadBatch; ++u) {
      const int f = f0 + u * kCombThreads + tid;
      const int row = f >> lg_cpr;  // key position
      const int qq = min((row >> 5) - q0, nqt - 1);
      float v = dot8(ev[u], s_w + qq * Nr + 8 * col);
      for (int off = cpr >> 1; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (f < f_hi && col == 0) s_raw[row - base] = v;
    }
    if (f1 < f_hi) {
#pragma unroll
      for (int u = 0; u < kLoadBatch; ++u) ev[u] = nx[u];
    }
  }
  __syncthreads();

  // discard the table lines no other chunk reads (rows inside [a + h, b - h)):
  // every load of them has completed, and they need no write-back to DRAM
  {
    const long long row_bytes = static_cast<long long>(Nr) * 2;
    const long long base_b = static_cast<long long>(it.eoff) * 2;
    const long long lo_b = ((base_b + static_cast<long long>(a + h + 1) * row_bytes + 127) / 128) * 128;
    const long long hi_b = ((base_b + static_cast<long long>(b - h - 1) * row_bytes) / 128) * 128;
    for (long long x = lo_b + static_cast<long long>(tid) * 128; x + 128 <= hi_b;
         x += static_cast<long long>(kCombThreads) * 128) {
      const char* line = reinterpret_cast<const char*>(p.expo) + x;
      asm volatile("discard.global.L2 [%0], 128;" ::"l"(line) : "memory");
    }
  }

  // 2. pooling (and the raw scores, when asked for)
  const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const float fP = static_cast<float>(p.pool_width);
  for (int j = a + tid; j < b; j += kCombThreads) {
    const int i = j - a;
    float acc = 0.f;
    for (int t = 0; t <= 2 * h; ++t) acc += s_raw[i + t];
    p.pooled[soff + j] = acc / fP;
    if (p.raw_out) p.raw_out[soff + j] = s_raw[i + h];
  }
  pdl_launch_dependents();  // late: the select kernel needs every chunk anyway
}

}  // namespace

size_t combine_smem_bytes(int quarters, int nr, int pool_width) {
  // the chunk's quarters plus one halo quarter on each side, and its raw
  // scores with the halo
  return (static_cast<size_t>(quarters + 2) * nr + static_cast<size_t>(quarters) * 32 +
          pool_width) *
         sizeof(float);
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
