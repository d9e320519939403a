// Observation-window scoring (CompressKV Sec. 3.3; SnapKV-style window of
// Sec. 4) on sm_103a tensor cores.
//
// For one unit (sequence s, KV group g) let Q_S be the |S_g|*W window-query
// rows of the group's SRH heads and K the unit's L keys.  With
// z = <q, k> * scale and c = log2(e):
//   pass 1 (stats):  m_q = max_j z_qj*c,  Z_q = sum_{j <= p_q} 2^(z_qj*c - m_q)
//                    over the causal keys j <= p_q = L - W + w(q);
//   pass 2 (accum):  raw_j = sum_q 2^(z_qj*c - m_q - log2 Z_q)  for j < n = L - W,
// i.e. the softmax attention of every SRH window query summed over queries,
// for every prefix token.  The normaliser Z_q needs all keys before any
// attention weight is final, hence two passes; pass 2 re-reads K while it is
// still in L2 (the host sizes the units launched together to the L2).
//
// Each CTA owns one work item: a contiguous range of 128-token K tiles of one
// unit.  Warp roles:
//   warp 0     TMA producer: K tiles (two 64-column halves, 128-byte swizzle)
//              into a kStages-deep shared-memory ring;
//   warp 1     UMMA issuer: D[128 tokens x N] = K_tile . Q_S^T  (tcgen05.mma
//              kind::f16, M=128, N = |S_g|*W rounded to 16, K = d = 128),
//              fp32 accumulators in TMEM, 2 or 4 buffers;
//   warp 2     TMEM allocation;
//   warps 4-11 two epilogue warpgroups (alternate tiles); thread = token
//              (TMEM lane), it reads its row of N logits with tcgen05.ld.
// Tokens sit on the MMA's M side so every epilogue lane holds real work for
// any N; in pass 2 the per-token sum over queries stays inside a thread.  In
// pass 1 the per-query sums over tokens are formed with a 32x32 transpose-
// reduction across the warp (31 shuffles per 1024 values) against a per-warp,
// per-query reference that is only raised when a logit exceeds it by more
// than 2^kTau, so the common path costs one exp per logit.
#include <cuda_runtime.h>

#include <cfloat>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr float kTau = 8.0f;  // log2 headroom before a running reference is raised
constexpr int kNumEpiWarps = 8;
constexpr int kEpiThreads = kNumEpiWarps * 32;
constexpr int kMiscBytes = 256 + 2 * kNumEpiWarps * kMaxQRows * 4;
constexpr float kNegInf = -INFINITY;

__device__ __forceinline__ void wait_plain(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  volatile int never = 0;
  mbar_wait_bounded(bar, parity, &never, nullptr, timeout_ns);
}

template <bool kAccum>
__global__ void __launch_bounds__(kScoreThreads, 1)
    score_kernel(const __grid_constant__ ScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = base;
  uint8_t* sQ = base + kStages * kTileBytes;
  const int qh = p.q_half_bytes;
  uint8_t* sMisc = sQ + 2 * qh;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sMisc);  // full[S] empty[S] tfull[4] tempty[4]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(sMisc + 192);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(sMisc + 196);
  float* sRef = reinterpret_cast<float*>(sMisc + 256);   // [8][kMaxQRows] refs / pass-2 bias
  float* sAcc = sRef + kNumEpiWarps * kMaxQRows;         // [8][kMaxQRows]

  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * kStages;
  const uint32_t tfull0 = empty0 + 8 * kStages;
  const uint32_t tempty0 = tfull0 + 8 * 4;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const WorkItem it = p.items[blockIdx.x];
  const int s = it.seq;
  const int g = it.group;
  const int seq0 = p.cu_seqlens[s];
  const int L = p.cu_seqlens[s + 1] - seq0;
  const int W = p.window;
  const int n = L - W;
  const int h0 = p.srh_off[g];
  const int N = (p.srh_off[g + 1] - h0) * W;
  const int Npad = (N + 15) & ~15;
  const int tstride = Npad <= 64 ? 64 : (Npad <= 128 ? 128 : 256);
  const int nbuf = (4 * tstride <= 512) ? 4 : 2;
  const uint32_t tcols = static_cast<uint32_t>(nbuf * tstride);
  const int t0 = it.t0;
  int t1 = it.t1;
  if (kAccum) t1 = min(t1, (n + kTileTokens - 1) / kTileTokens);
  const int ntiles = max(t1 - t0, 0);

  if (ntiles == 0) return;  // uniform over the CTA: nothing allocated yet

  // ------------------------------------------------------------ set-up
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, 1);
    }
    for (int b = 0; b < 4; ++b) {
      mbar_init(tfull0 + 8 * b, 1);
      mbar_init(tempty0 + 8 * b, 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) tma_prefetch_map(&p.tmap_k);
  if (warp == 2) {
    tmem_alloc(smem_u32(tmem_holder), tcols);
    tmem_relinquish();
  }
  // Window-query rows of the SRH heads -> shared memory in the UMMA K-major
  // 128-byte-swizzle layout (row r, 16-byte chunk ch of each 64-column half
  // lands at chunk ch ^ (r & 7)); rows N..Npad-1 are zero.
  for (int idx = threadIdx.x; idx < Npad * 16; idx += blockDim.x) {
    const int r = idx >> 4;
    const int ch = idx & 15;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    if (r < N) {
      const int head = p.srh_heads[h0 + r / W];
      const int w = r - (r / W) * W;
      const uint16_t* src = p.q + static_cast<long long>(s) * p.q_bs +
                            static_cast<long long>(head) * p.q_hs +
                            static_cast<long long>(w) * p.q_ws + ch * 8;
      val = *reinterpret_cast<const uint4*>(src);
    }
    const int half = ch >> 3;
    const int c8 = ch & 7;
    *reinterpret_cast<uint4*>(sQ + half * qh + r * 128 + ((c8 ^ (r & 7)) << 4)) = val;
  }
  fence_proxy_async_smem();
  if (kAccum) {
    // Merge the unit's pass-1 partials (fixed order => deterministic) into
    // the per-query bias m_q + log2 Z_q.
    for (int q = threadIdx.x; q < N; q += blockDim.x) {
      float m = kNegInf;
      for (int i = 0; i < it.count; ++i)
        m = fmaxf(m, p.partials[static_cast<long long>(it.first + i) * kMaxQRows + q].x);
      float z = 0.f;
      for (int i = 0; i < it.count; ++i) {
        const float2 pr = p.partials[static_cast<long long>(it.first + i) * kMaxQRows + q];
        if (pr.x != kNegInf) z += pr.y * ex2_approx(pr.x - m);
      }
      sRef[q] = m + log2f(z);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tmem_holder;

  // ------------------------------------------------------------ roles
  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol =
          (kAccum || !p.use_evict_hint) ? l2_policy_evict_first() : l2_policy_evict_last();
      int issued = 0;
      for (int i = 0; i < ntiles; ++i) {
        const int st = i % kStages;
        const uint32_t ph = static_cast<uint32_t>(i / kStages) & 1u;
        if (!mbar_wait_bounded(empty0 + 8 * st, ph ^ 1u, abort_flag, p.status)) break;
        mbar_arrive_expect_tx(full0 + 8 * st, kTileBytes);
        const int row = seq0 + (t0 + i) * kTileTokens;
        const uint32_t dst = smem_u32(sK + st * kTileBytes);
        tma_load_3d(dst, &p.tmap_k, full0 + 8 * st, 0, g, row, pol);
        tma_load_3d(dst + kHalfTileBytes, &p.tmap_k, full0 + 8 * st, 64, g, row, pol);
        ++issued;
      }
      if (*abort_flag) {
        // let the copies already issued land before the CTA can exit
        for (int i = max(0, issued - kStages); i < issued; ++i)
          wait_plain(full0 + 8 * (i % kStages), static_cast<uint32_t>(i / kStages) & 1u,
                     100000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_f16(kTileTokens, Npad, p.is_bf16 != 0);
      const uint32_t sq = smem_u32(sQ);
      const uint32_t sk = smem_u32(sK);
      int issued = 0;
      for (int i = 0; i < ntiles; ++i) {
        const int st = i % kStages;
        const uint32_t ph = static_cast<uint32_t>(i / kStages) & 1u;
        const int b = i % nbuf;
        const uint32_t use = static_cast<uint32_t>(i / nbuf) & 1u;
        if (!mbar_wait_bounded(tempty0 + 8 * b, use ^ 1u, abort_flag, p.status)) break;
        tc_fence_after();
        if (!mbar_wait_bounded(full0 + 8 * st, ph, abort_flag, p.status)) break;
        tc_fence_after();
        const uint32_t d = tbase + static_cast<uint32_t>(b * tstride);
#pragma unroll
        for (int kk = 0; kk < kHeadDim / 16; ++kk) {
          const uint32_t koff = (kk >> 2) * kHalfTileBytes + (kk & 3) * 32;
          const uint32_t qoff = (kk >> 2) * qh + (kk & 3) * 32;
          umma_f16(d, smem_desc_sw128(sk + st * kTileBytes + koff), smem_desc_sw128(sq + qoff),
                   idesc, kk > 0 ? 1u : 0u);
        }
        umma_commit(empty0 + 8 * st);
        umma_commit(tfull0 + 8 * b);
        ++issued;
      }
      if (*abort_flag && issued > 0) {
        // the last commit covers every MMA issued: wait for it before TMEM is freed
        const int i = issued - 1;
        wait_plain(tfull0 + 8 * (i % nbuf), static_cast<uint32_t>(i / nbuf) & 1u, 100000000ull);
      }
    }
  } else if (warp >= 4) {
    const int ew = warp - 4;  // 0..7
    const int wg = ew >> 2;   // epilogue warpgroup: tiles i with i % 2 == wg
    const int qd = warp & 3;  // TMEM lane quarter this warp may access
    const int nch = (N + 31) >> 5;
    const float c = p.c;
    float* ref = sRef + ew * kMaxQRows;
    float* acc = sAcc + ew * kMaxQRows;
    if (!kAccum) {
      for (int q = lane; q < kMaxQRows; q += 32) {
        ref[q] = kNegInf;
        acc[q] = 0.f;
      }
      __syncwarp();
    }
    for (int i = wg; i < ntiles; i += 2) {
      const int b = i % nbuf;
      const uint32_t use = static_cast<uint32_t>(i / nbuf) & 1u;
      const bool got = mbar_wait_bounded(tfull0 + 8 * b, use, abort_flag, p.status);
      if (!__all_sync(0xffffffffu, got)) break;  // warp-uniform exit on abort
      tc_fence_after();
      const int tok = (t0 + i) * kTileTokens + qd * 32 + lane;  // position in the sequence
      const uint32_t taddr =
          tbase + (static_cast<uint32_t>(qd * 32) << 16) + static_cast<uint32_t>(b * tstride);
      if (kAccum) {
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
        for (int ch = 0; ch < nch; ++ch) {
          float z[32];
          tmem_load32(taddr + ch * 32, z);
          const float* bias = sRef + ch * 32;
          const int lim = N - ch * 32;
#pragma unroll
          for (int j = 0; j < 32; j += 4) {
            const float4 bq = *reinterpret_cast<const float4*>(bias + j);
            if (j + 0 < lim) s0 += ex2_approx(fmaf(z[j + 0], c, -bq.x));
            if (j + 1 < lim) s1 += ex2_approx(fmaf(z[j + 1], c, -bq.y));
            if (j + 2 < lim) s2 += ex2_approx(fmaf(z[j + 2], c, -bq.z));
            if (j + 3 < lim) s3 += ex2_approx(fmaf(z[j + 3], c, -bq.w));
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * b);
        if (tok < n) {
          p.raw[static_cast<long long>(g) * p.p_total + p.cu_prefix[s] + tok] =
              (s0 + s1) + (s2 + s3);
        }
      } else {
        // tiles reaching the window (causal mask) or past the sequence end
        const bool edge = (t0 + i + 1) * kTileTokens > n;
        for (int ch = 0; ch < nch; ++ch) {
          float z[32];
          tmem_load32(taddr + ch * 32, z);
          const float* rf = ref + ch * 32;
          float t[32];
          float tmax = kNegInf;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int q = ch * 32 + j;
            bool valid = q < N;
            if (edge) valid = valid && tok < L && tok <= n + (q % W);
            z[j] = valid ? z[j] * c : kNegInf;
            t[j] = valid ? z[j] - rf[j] : kNegInf;
            tmax = fmaxf(tmax, t[j]);
          }
          if (__any_sync(0xffffffffu, tmax > kTau)) {
            // raise the references of this chunk's queries to their column max
            float zz[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) zz[j] = z[j];
            const float cmax = warp_transpose_max32(zz, lane);
            const int q = ch * 32 + lane;
            const float old = ref[q];
            const float nw = fmaxf(old, cmax);
            if (nw != old) {
              acc[q] *= (old == kNegInf) ? 0.f : ex2_approx(old - nw);
              ref[q] = nw;
            }
            __syncwarp();
#pragma unroll
            for (int j = 0; j < 32; ++j) t[j] = (z[j] == kNegInf) ? kNegInf : z[j] - rf[j];
          }
#pragma unroll
          for (int j = 0; j < 32; ++j) t[j] = ex2_approx(t[j]);
          const float colsum = warp_transpose_sum32(t, lane);
          acc[ch * 32 + lane] += colsum;
          __syncwarp();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * b);
      }
    }
    if (!kAccum) {
      // combine the 8 epilogue warps' (reference, sum) pairs per query
      named_bar_sync(1, kEpiThreads);
      const int te = threadIdx.x - 4 * 32;
      if (te < N && !*abort_flag) {
        float m = kNegInf;
        for (int w = 0; w < kNumEpiWarps; ++w) m = fmaxf(m, sRef[w * kMaxQRows + te]);
        float z = 0.f;
        for (int w = 0; w < kNumEpiWarps; ++w) {
          const float r = sRef[w * kMaxQRows + te];
          if (r != kNegInf) z += sAcc[w * kMaxQRows + te] * ex2_approx(r - m);
        }
        p.partials[static_cast<long long>(blockIdx.x) * kMaxQRows + te] = make_float2(m, z);
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tbase, tcols);
  }
}

template <bool kAccum>
cudaError_t launch(const ScoreParams& p, int n_items, size_t smem, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n_items));
  cfg.blockDim = dim3(kScoreThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  return cudaLaunchKernelEx(&cfg, score_kernel<kAccum>, p);
}

}  // namespace

size_t score_smem_bytes(int q_half_bytes) {
  return 1024 + static_cast<size_t>(kStages) * kTileBytes + 2 * static_cast<size_t>(q_half_bytes) +
         kMiscBytes;
}

cudaError_t score_set_smem_limit(size_t bytes) {
  cudaError_t e = cudaFuncSetAttribute(score_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(bytes));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(score_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(bytes));
}

cudaError_t launch_score_stats(const ScoreParams& p, int n_items, size_t smem, cudaStream_t s) {
  return launch<false>(p, n_items, smem, s);
}
cudaError_t launch_score_accum(const ScoreParams& p, int n_items, size_t smem, cudaStream_t s) {
  return launch<true>(p, n_items, smem, s);
}

}  // namespace ckv
