// Observation-window scoring (CompressKV Sec. 3.3; SnapKV-style window of
// Sec. 4) on sm_103a tensor cores, in one pass over K.
//
// For one unit (sequence s, KV group g) let Q_S be the N = |S_g|*W
// window-query rows of the group's SRH heads and K the unit's L keys.  With
// z = <q, k> * scale and c = log2(e), the attention of query q (window
// position p_q) on key j <= p_q is 2^(z_qj*c) / D_q with
// D_q = sum_{j <= p_q} 2^(z_qj*c).  This kernel computes every logit once
// and leaves
//   * for every prefix key j < n = L - W and query row q, the exponent
//     e_qj = 2^(z_qj*c - R) in an fp16 table (Nr = N rounded up to a power of
//     two >= 8 columns per key; columns N..Nr-1 are 0), where R is a
//     per-query reference kept by the warp that owns the key's 32-token
//     quarter of its tile; the R used for every (tile, quarter, q) goes to a
//     float table;
//   * per work item and query row the pair (M, S) with
//     sum over the item's keys of 2^(z*c) = S * 2^M.
// R stays kShift below the largest scaled logit the warp has seen and is
// raised whenever an exponent would pass 2^kRaise, so every stored exponent
// is at most 2^kRaise (below the fp16 maximum 65504) and keeps a relative
// rounding error <= 2^-11.  The combine kernel forms D_q from the pairs and
// the normalised, pooled scores from the tables.
//
// Each CTA owns one work item: a contiguous range of 128-token K tiles of one
// unit.  Warp roles:
//   warp 0      TMA producer: K tiles (two 64-column halves, 128-byte swizzle)
//               into a shared-memory ring of up to kStages tiles; it starts
//               streaming while the other warps stage the query rows;
//   warp 1      TMEM allocation, then UMMA issue: D[128 tokens x N] =
//               K_tile . Q_S^T  (tcgen05.mma kind::f16, M=128, N rounded to 16,
//               K = d = 128), fp32 accumulators in TMEM, 2 or 4 buffers, each
//               owned by one epilogue warpgroup;
//   warps 2..   two or four epilogue warpgroups (tiles i % #groups; with 2
//               TMEM buffers only the first two work) -- two warpgroups per CTA
//               and two CTAs per SM when their shared memory fits, else four
//               in one CTA per SM; thread = token (TMEM lane): it reads its
//               row of logits from TMEM 32 columns at a time, keeps the
//               warp's running references, writes its exponent row with
//               32-byte stores that ask L2 to keep the table, and adds the
//               exponents into the warp's per-query sums by a 32x32
//               transpose-reduction.
// Tokens sit on the MMA's M side so every epilogue lane holds real work for
// any N.
//
// With the window queries' log-sum-exp given (kLse: the softmax denominators
// a prefill attention kernel already has), no table is needed: every lane
// sums 2^(z*c - LSE_q*log2(e)) over its row -- the normalised attention of all
// query rows on its key -- and writes the prefix key's raw score directly.
#include <cuda_runtime.h>

#include <cfloat>

#include "ckv_device.cuh"

namespace ckv {

namespace {

constexpr float kShift = 7.0f;   // R sits this far below the warp's largest logit (log2 units)
constexpr float kRaise = 15.0f;  // exponents stay <= 2^kRaise
// Epilogue width: 8 warps (two CTAs per SM, when their shared memory fits)
// or 16 warps (one CTA per SM).
template <int kEpi>
struct Shape {
  static constexpr int kWG = kEpi / 4;                    // epilogue warpgroups
  static constexpr int kThreads = 64 + 32 * kEpi;
  static constexpr int kStagedThreads = kThreads - 32;    // warps 1.. stage the Q rows
  static constexpr int kCtasPerSm = kEpi == 8 ? 2 : 1;
  // misc region: barriers (256 B) | running references [kEpi][256] f32 |
  // sums [kEpi][256] f32 | window position of each query row [256] i32
  static constexpr int kMiscBytes = 256 + 2 * kEpi * kMaxQRows * 4 + kMaxQRows * 4;
};
constexpr float kNegInf = -INFINITY;
constexpr int kBarStaged = 2;  // named barrier: warps 1.. after staging Q
constexpr int kBarEpi = 1;     // named barrier: the epilogue warps
constexpr int kFirstEpiWarp = 2;

__device__ __forceinline__ void wait_plain(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  volatile int never = 0;
  mbar_wait_bounded(bar, parity, &never, nullptr, timeout_ns);
}

template <bool kLse, int kEpi>
__global__ void __launch_bounds__(Shape<kEpi>::kThreads, Shape<kEpi>::kCtasPerSm)
    score_kernel(const __grid_constant__ ScoreParams p) {
  constexpr int kNumEpiWarps = kEpi;
  constexpr int kWG = Shape<kEpi>::kWG;
  constexpr int kStagedThreads = Shape<kEpi>::kStagedThreads;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = base;
  const int nst = p.stages;  // K stages in the ring (2..kStages)
  uint8_t* sQ = base + nst * kTileBytes;
  const int qh = p.q_half_bytes;
  uint8_t* sMisc = sQ + 2 * qh;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sMisc);  // full[6] empty[6] tfull[4] tempty[4]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(sMisc + 192);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(sMisc + 196);
  float* sRef = reinterpret_cast<float*>(sMisc + 256);                  // [16][kMaxQRows]
  float* sAcc = sRef + kNumEpiWarps * kMaxQRows;                         // [kEpi][kMaxQRows]
  int* sWpos = reinterpret_cast<int*>(sAcc + kNumEpiWarps * kMaxQRows);  // [kMaxQRows]

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
  const int vg = srh_group(s, g, p.seqs_per_mask, p.num_kv_heads);
  const int h0 = p.srh_off[vg];
  const int N = (p.srh_off[vg + 1] - h0) * W;
  const int Npad = (N + 15) & ~15;
  const int Nr = expo_stride(N);  // row length of the exponent table
  const int tstride = Npad <= 64 ? 64 : (Npad <= 128 ? 128 : 256);
  const int nbuf = (4 * tstride <= 512) ? 4 : 2;
  const uint32_t tcols = static_cast<uint32_t>(nbuf * tstride);
  const int t0 = it.t0;
  const int ntiles = it.t1 - t0;  // >= 1 by construction

  // ------------------------------------------------------------ set-up
  // Window-query rows of the SRH heads -> shared memory in the UMMA K-major
  // 128-byte-swizzle layout (row r, 16-byte chunk ch of each 64-column half
  // lands at chunk ch ^ (r & 7)); rows N..Npad-1 are zero.  The copies are
  // asynchronous and issued first, so their latency overlaps the set-up.
  if (warp != 0) {
    const int st_tid = threadIdx.x - 32;
    for (int idx = st_tid; idx < Npad * 16; idx += kStagedThreads) {
      const int r = idx >> 4;
      const int ch = idx & 15;
      uint8_t* dst = sQ + (ch >> 3) * qh + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
      if (r < N) {
        const int head = p.srh_heads[h0 + r / W];
        const int w = r - (r / W) * W;
        cp_async16(smem_u32(dst), p.q + static_cast<long long>(s) * p.q_bs +
                                      static_cast<long long>(head) * p.q_hs +
                                      static_cast<long long>(w) * p.q_ws + ch * 8);
      } else {
        *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
      }
    }
  }
  const uint64_t kpol = p.use_evict_hint ? l2_policy_evict_first() : l2_policy_evict_last();
  const int prefill = min(nst, ntiles);  // ring stages filled before the CTA-wide barrier
  if (threadIdx.x == 0) {
    for (int i = 0; i < nst; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, 1);
    }
    for (int b = 0; b < 4; ++b) {
      mbar_init(tfull0 + 8 * b, 1);
      // released by every warp of the warpgroups sharing the buffer
      mbar_init(tempty0 + 8 * b, (!kLse && kWG > nbuf) ? 8 : 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
    // the ring starts empty: its first tiles need no wait
    for (int i = 0; i < prefill; ++i) {
      mbar_arrive_expect_tx(full0 + 8 * i, kTileBytes);
      const int row = seq0 + (t0 + i) * kTileTokens;
      const uint32_t dst = smem_u32(sK + i * kTileBytes);
      tma_load_3d(dst, &p.tmap_k, full0 + 8 * i, 0, g, row, kpol);
      tma_load_3d(dst + kHalfTileBytes, &p.tmap_k, full0 + 8 * i, 64, g, row, kpol);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), tcols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tmem_holder;

  if (warp == 0) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0) {
      int issued = prefill;
      for (int i = prefill; i < ntiles; ++i) {
        const int st = i % nst;
        const uint32_t ph = static_cast<uint32_t>(i / nst) & 1u;
        if (!mbar_wait_bounded(empty0 + 8 * st, ph ^ 1u, abort_flag, p.status)) break;
        mbar_arrive_expect_tx(full0 + 8 * st, kTileBytes);
        const int row = seq0 + (t0 + i) * kTileTokens;
        const uint32_t dst = smem_u32(sK + st * kTileBytes);
        tma_load_3d(dst, &p.tmap_k, full0 + 8 * st, 0, g, row, kpol);
        tma_load_3d(dst + kHalfTileBytes, &p.tmap_k, full0 + 8 * st, 64, g, row, kpol);
        ++issued;
      }
      if (*abort_flag) {
        // let the copies already issued land before the CTA can exit
        for (int i = max(0, issued - nst); i < issued; ++i)
          wait_plain(full0 + 8 * (i % nst), static_cast<uint32_t>(i / nst) & 1u, 100000000ull);
      }
    }
    __syncwarp();  // reconverge before the CTA-wide (aligned) barrier below
  } else {
    // ---------------------------------------------------------- staging
    // the Q-row copies issued at entry have landed: make them visible to the
    // tensor cores (async proxy)
    const int st_tid = threadIdx.x - 32;
    cp_async_wait_all();
    fence_proxy_async_smem();
    for (int q = st_tid; q < kMaxQRows; q += kStagedThreads) sWpos[q] = q < N ? q % W : 0;
    if constexpr (kLse) {
      // log2 of every query row's softmax denominator (first rows of sRef);
      // a first pass's rows are read only once that kernel has completed
      if (p.lse_bias) pdl_wait();
      for (int q = st_tid; q < kMaxQRows; q += kStagedThreads) {
        float l2 = 0.f;
        if (q < N) {
          if (p.lse_bias) {  // second pass: the first pass's log2 denominators
            l2 = p.lse_bias[static_cast<long long>(it.first) * kMaxQRows + q];
          } else {
            const int head = p.srh_heads[h0 + q / W];
            const int w = q - (q / W) * W;
            l2 = p.lse[static_cast<long long>(s) * p.lse_bs +
                       static_cast<long long>(head) * p.lse_hs + w] *
                 1.4426950408889634f;
          }
        }
        sRef[q] = l2;
      }
    } else {
      const int ew = warp - kFirstEpiWarp;
      if (ew >= 0) {
        for (int q = lane; q < kMaxQRows; q += 32) {
          sRef[ew * kMaxQRows + q] = kNegInf;
          sAcc[ew * kMaxQRows + q] = 0.f;
        }
      }
    }
    named_bar_sync(kBarStaged, kStagedThreads);

    if (warp == 1) {
      // -------------------------------------------------------- UMMA issuer
      if (lane == 0) {
        const uint32_t idesc = umma_idesc_f16(kTileTokens, Npad, p.is_bf16 != 0);
        // descriptor start addresses advance in 16-byte units (no carry out of
        // the 14-bit field: shared memory is below 256 KB)
        const uint64_t dq0 = smem_desc_sw128(smem_u32(sQ));
        const uint64_t dk0 = smem_desc_sw128(smem_u32(sK));
        int issued = 0;
        for (int i = 0; i < ntiles; ++i) {
          const int st = i % nst;
          const uint32_t ph = static_cast<uint32_t>(i / nst) & 1u;
          const int b = i % nbuf;
          const uint32_t use = static_cast<uint32_t>(i / nbuf) & 1u;
          if (!mbar_wait_bounded(tempty0 + 8 * b, use ^ 1u, abort_flag, p.status)) break;
          tc_fence_after();
          if (!mbar_wait_bounded(full0 + 8 * st, ph, abort_flag, p.status)) break;
          tc_fence_after();
          const uint32_t d = tbase + static_cast<uint32_t>(b * tstride);
#pragma unroll
          for (int kk = 0; kk < kHeadDim / 16; ++kk) {
            const uint32_t koff = st * kTileBytes + (kk >> 2) * kHalfTileBytes + (kk & 3) * 32;
            const uint32_t qoff = (kk >> 2) * qh + (kk & 3) * 32;
            umma_f16(d, dk0 + (koff >> 4), dq0 + (qoff >> 4), idesc, kk > 0 ? 1u : 0u);
          }
          umma_commit(empty0 + 8 * st);
          umma_commit(tfull0 + 8 * b);
          ++issued;
        }
        if (*abort_flag && issued > 0) {
          // the last commit covers every MMA issued: wait for it before TMEM is freed
          const int i = issued - 1;
          wait_plain(tfull0 + 8 * (i % nbuf), static_cast<uint32_t>(i / nbuf) & 1u,
                     100000000ull);
        }
      }
      __syncwarp();  // reconverge before the CTA-wide (aligned) barrier below
    } else if constexpr (kLse) {
      // -------------------------------------------------------- epilogue (given LSE)
      const int ew = warp - kFirstEpiWarp;  // 0..15
      const int wg = ew >> 2;
      const int qd = warp & 3;
      const float c = p.c;
      const float* lse2 = sRef;
      const int nwg = kWG < nbuf ? kWG : nbuf;
      float* raw_row = p.raw_out + static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
      // the raw-score buffer may still be read by an earlier kernel of the stream
      pdl_wait();
      for (int i = wg; wg < nwg && i < ntiles; i += nwg) {
        const int b = i % nbuf;
        const uint32_t use = static_cast<uint32_t>(i / nbuf) & 1u;
        const bool got = mbar_wait_bounded(tfull0 + 8 * b, use, abort_flag, p.status);
        if (!__all_sync(0xffffffffu, got)) break;
        tc_fence_after();
        const int tile = t0 + i;
        const int tok = tile * kTileTokens + qd * 32 + lane;
        const uint32_t taddr =
            tbase + (static_cast<uint32_t>(qd * 32) << 16) + static_cast<uint32_t>(b * tstride);
        const bool edge = (tile + 1) * kTileTokens > n;
        const int vis = n - tok;
        const bool key = tok < L;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        for (int c0 = 0; c0 < N; c0 += 32) {
          uint32_t r[32];
          tmem_load32_async(taddr + c0, r);
          tmem_wait_ld(r);
          const int lim = min(32, N - c0);
          if (edge || lim < 32) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const int4 wq = *reinterpret_cast<const int4*>(sWpos + c0 + j);
              const float4 lq = *reinterpret_cast<const float4*>(lse2 + c0 + j);
              const int wv[4] = {wq.x, wq.y, wq.z, wq.w};
              const float lv[4] = {lq.x, lq.y, lq.z, lq.w};
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const bool ok = (j + u) < lim && (!edge || (key && wv[u] >= -vis));
                acc[u] += ok ? ex2_approx(fmaf(__uint_as_float(r[j + u]), c, -lv[u])) : 0.f;
              }
            }
          } else {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const float4 lq = *reinterpret_cast<const float4*>(lse2 + c0 + j);
              acc[0] += ex2_approx(fmaf(__uint_as_float(r[j + 0]), c, -lq.x));
              acc[1] += ex2_approx(fmaf(__uint_as_float(r[j + 1]), c, -lq.y));
              acc[2] += ex2_approx(fmaf(__uint_as_float(r[j + 2]), c, -lq.z));
              acc[3] += ex2_approx(fmaf(__uint_as_float(r[j + 3]), c, -lq.w));
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * b);
        if (tok < n) raw_row[tok] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
      }
    } else {
      // -------------------------------------------------------- epilogue
      const int ew = warp - kFirstEpiWarp;  // 0..15
      const int wg = ew >> 2;               // epilogue warpgroup: tiles i % nwg == wg
      const int qd = warp & 3;              // TMEM lane quarter this warp may access
      const float c = p.c;
      float* ref = sRef + ew * kMaxQRows;
      float* acc_s = sAcc + ew * kMaxQRows;
      const int ngrp = (Nr + 31) >> 5;  // 32-column groups of an exponent row
      const uint64_t keep = l2_policy_evict_last();
      // Every TMEM buffer must belong to one warpgroup: an mbarrier parity
      // wait cannot tell phase k from phase k+2, so warpgroups sharing a
      // buffer could read it early.
      const int nwg = kWG < nbuf ? kWG : nbuf;
      // With fewer TMEM buffers than warpgroups (query rows > 128: two
      // buffers), two warpgroups share each buffer and split its 32-column
      // groups (even / odd), so every epilogue warp has work.
      const bool csplit = kWG > nbuf;
      const int tg = wg % nwg;                  // tiles i % nwg == tg
      const int gbeg = csplit ? wg / nwg : 0;   // first column group, step gstep
      const int gstep = csplit ? 2 : 1;
      // The exponent and reference tables and the softmax pairs are reused
      // across calls on one workspace.  Their only reader, the combine kernel,
      // triggers its dependents after its last read of them, so this grid
      // (launched no earlier than that trigger) may overwrite them without
      // waiting for the kernels before it.

      for (int i = tg; i < ntiles; i += nwg) {
        const int b = i % nbuf;
        const uint32_t use = static_cast<uint32_t>(i / nbuf) & 1u;
        const bool got = mbar_wait_bounded(tfull0 + 8 * b, use, abort_flag, p.status);
        if (!__all_sync(0xffffffffu, got)) break;  // warp-uniform exit on abort
        tc_fence_after();
        const int tile = t0 + i;                              // tile index in the unit
        const int tok = tile * kTileTokens + qd * 32 + lane;  // position in the sequence
        const uint32_t taddr =
            tbase + (static_cast<uint32_t>(qd * 32) << 16) + static_cast<uint32_t>(b * tstride);
        // tiles that reach the window (causal mask) or pass the sequence end
        const bool edge = (tile + 1) * kTileTokens > n;
        const int vis = n - tok;  // query row q sees this key iff tok < L and wpos(q) >= -vis
        const bool key = tok < L;    // a key of the sequence (the last tile may run past L)
        const bool store = tok < n && !p.stats_only;  // the table holds prefix keys only
        uint16_t* erow = p.expo + it.eoff + static_cast<long long>(tok) * Nr;

        for (int grp = gbeg; grp < ngrp; grp += gstep) {
          const int c0 = 32 * grp;
          const int ncols = min(32, Nr - c0);  // 8, 16 or 32 (Nr is a power of two)
          if (c0 >= N) {
            // padding columns of the table
            if (store) {
              if (ncols == 32) {
                const uint32_t zz[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
                st_global_v8_hint(erow + c0, zz, keep);
                st_global_v8_hint(erow + c0 + 16, zz, keep);
              } else {
                for (int v = 0; v < ncols; v += 8) st_global_v4_hint(erow + c0 + v, 0u, 0u, 0u, 0u, keep);
              }
            }
            continue;
          }
          uint32_t r[32];
          tmem_load32_async(taddr + c0, r);
          tmem_wait_ld(r);
          const int lim = min(32, N - c0);  // valid columns in this group
          const bool masked = edge || lim < 32;
          float* rf = ref + c0;
          // t = z*c - R, -inf where the key is masked for that query
          float t[32];
          float tmax = kNegInf;
          if (masked) {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const int4 wq = *reinterpret_cast<const int4*>(sWpos + c0 + j);
              const float4 rq = *reinterpret_cast<const float4*>(rf + j);
              const int wv[4] = {wq.x, wq.y, wq.z, wq.w};
              const float rv[4] = {rq.x, rq.y, rq.z, rq.w};
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const bool ok = (j + u) < lim && (!edge || (key && wv[u] >= -vis));
                t[j + u] = ok ? fmaf(__uint_as_float(r[j + u]), c, -rv[u]) : kNegInf;
                tmax = fmaxf(tmax, t[j + u]);
              }
            }
          } else {
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const float4 rq = *reinterpret_cast<const float4*>(rf + j);
              t[j + 0] = fmaf(__uint_as_float(r[j + 0]), c, -rq.x);
              t[j + 1] = fmaf(__uint_as_float(r[j + 1]), c, -rq.y);
              t[j + 2] = fmaf(__uint_as_float(r[j + 2]), c, -rq.z);
              t[j + 3] = fmaf(__uint_as_float(r[j + 3]), c, -rq.w);
              tmax = fmaxf(fmaxf(tmax, fmaxf(t[j], t[j + 1])), fmaxf(t[j + 2], t[j + 3]));
            }
          }
          if (__any_sync(0xffffffffu, tmax > kRaise)) {
            // Rare (always on a warp's first tile, where R = -inf): raise
            // each query's R to kShift below its largest scaled logit in this
            // warp's 32 tokens.  Logits are re-read from TMEM (the buffer is
            // still held) and reduced across lanes in registers.
            uint32_t valid = 0u;
#pragma unroll
            for (int j = 0; j < 32; ++j) valid |= (t[j] != kNegInf ? 1u : 0u) << j;
            float v[32];
            tmem_load32_async(taddr + c0, r);
            tmem_wait_ld(r);
#pragma unroll
            for (int j = 0; j < 32; ++j)
              v[j] = ((valid >> j) & 1u) ? __uint_as_float(r[j]) * c : kNegInf;
            const float m = warp_transpose_max32(v, lane);  // column c0 + lane
            const float old = rf[lane];
            const float nw = fmaxf(old, m - kShift);
            // the sums kept against the old R shrink by 2^(old - new)
            acc_s[c0 + lane] *= (nw == old) ? 1.f : ((old == kNegInf) ? 0.f : ex2_approx(old - nw));
            __syncwarp();
            rf[lane] = nw;
            __syncwarp();
            tmem_load32_async(taddr + c0, r);
            tmem_wait_ld(r);
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              const float4 rq = *reinterpret_cast<const float4*>(rf + j);
              const float rv[4] = {rq.x, rq.y, rq.z, rq.w};
#pragma unroll
              for (int u = 0; u < 4; ++u)
                t[j + u] = ((valid >> (j + u)) & 1u) ? fmaf(__uint_as_float(r[j + u]), c, -rv[u])
                                                      : kNegInf;
            }
          }
          // exponents: stored as fp16 (prefix keys), 16 per 32-byte store, and
          // summed per query over the warp's 32 keys
          float e[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) e[j] = ex2_approx(t[j]);
          if (store) {
#pragma unroll
            for (int v = 0; v < 2; ++v) {
              if (16 * v < ncols) {
                uint32_t pk[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) pk[u] = pack_half2(e[16 * v + 2 * u], e[16 * v + 2 * u + 1]);
                if (ncols >= 16) {
                  st_global_v8_hint(erow + c0 + 16 * v, pk, keep);
                } else {  // ncols == 8
                  st_global_v4_hint(erow + c0, pk[0], pk[1], pk[2], pk[3], keep);
                }
              }
            }
          }
          const float colsum = warp_transpose_sum32(e, lane);
          acc_s[c0 + lane] += colsum;
          __syncwarp();
        }
        // the references this tile quarter's exponents are relative to
        if (!p.stats_only) {
          float* rt = p.refs + it.roff + (static_cast<long long>(tile) * kQuarters + qd) * Nr;
          for (int q = 32 * gbeg + lane; q < N; q += 32 * gstep) rt[q] = ref[q];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * b);
      }
      // merge the epilogue warps' (R, sum) pairs per query into the item's pair
      named_bar_sync(kBarEpi, 32 * kNumEpiWarps);
      const int te = static_cast<int>(threadIdx.x) - kFirstEpiWarp * 32;
      // the first epilogue warp writes the item's pairs, makes them visible
      // device-wide and takes the unit's ticket: the last CTA of the unit to
      // get here (no waiting) merges the pairs of all the unit's items,
      // split over 32*E / N threads per query, into bias_q = log2 D_q for
      // the combine kernel, and resets the ticket
      volatile int* last = abort_flag + 1;
      if (te < 32) {
        for (int q = te; q < N && !*abort_flag; q += 32) {
          float m = kNegInf;
          for (int w = 0; w < kNumEpiWarps; ++w) m = fmaxf(m, sRef[w * kMaxQRows + q]);
          float z = 0.f;
          for (int w = 0; w < kNumEpiWarps; ++w) {
            const float rw = sRef[w * kMaxQRows + q];
            if (rw != kNegInf) z += sAcc[w * kMaxQRows + q] * ex2_approx(rw - m);
          }
          p.partials[static_cast<long long>(blockIdx.x) * kMaxQRows + q] = make_float2(m, z);
        }
        __threadfence();
        __syncwarp();
        if (te == 0)
          *last = (!*abort_flag && atomicAdd(p.tickets + it.first, 1) == it.count - 1) ? 1 : 0;
      }
      named_bar_sync(kBarEpi, 32 * kNumEpiWarps);
      if (*last) {
        __threadfence();
        const int nm = (32 * kNumEpiWarps) / N;
        const int q = te % N;
        const int sub = te / N;
        float m = kNegInf, z = 0.f;
        if (sub < nm) {
          // sixteen pairs in flight per batch (L2 reads of the other CTAs' rows)
          for (int i0 = sub; i0 < it.count; i0 += 16 * nm) {
            float2 pr[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) {
              const int i = i0 + u * nm;
              pr[u] = i < it.count
                          ? __ldcg(p.partials + static_cast<long long>(it.first + i) * kMaxQRows + q)
                          : make_float2(kNegInf, 0.f);
            }
#pragma unroll
            for (int u = 0; u < 16; ++u) {
              if (pr[u].x == kNegInf) continue;
              if (pr[u].x > m) {
                z = fmaf(z, ex2_approx(m - pr[u].x), pr[u].y);
                m = pr[u].x;
              } else {
                z = fmaf(pr[u].y, ex2_approx(pr[u].x - m), z);
              }
            }
          }
          sRef[sub * N + q] = m;
          sAcc[sub * N + q] = z;
        }
        named_bar_sync(kBarEpi, 32 * kNumEpiWarps);
        if (te < N) {
          m = kNegInf;
          z = 0.f;
          for (int j = 0; j < nm; ++j) {
            const float pm = sRef[j * N + te];
            const float pz = sAcc[j * N + te];
            if (pm == kNegInf) continue;
            if (pm > m) {
              z = fmaf(z, ex2_approx(m - pm), pz);
              m = pm;
            } else {
              z = fmaf(pz, ex2_approx(pm - m), z);
            }
          }
          p.bias[static_cast<long long>(it.first) * kMaxQRows + te] = m + __log2f(z);
        }
        if (te == 0) p.tickets[it.first] = 0;
      }
    }
  }

  // ------------------------------------------------------------ teardown
  // The next kernel is launched once every CTA has reached this point, so its
  // CTAs spread over all SMs instead of packing the ones that freed first.
  // The tensor memory is released before the wait for the kernels before
  // this one (completion of this grid then implies theirs).
  pdl_launch_dependents();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tbase, tcols);
  }
  pdl_wait();
}

}  // namespace

size_t score_smem_bytes(int q_half_bytes, int stages, int epi_warps) {
  const size_t misc = epi_warps == 8 ? Shape<8>::kMiscBytes : Shape<16>::kMiscBytes;
  return 1024 + static_cast<size_t>(stages) * kTileBytes + 2 * static_cast<size_t>(q_half_bytes) +
         misc;
}

cudaError_t score_set_smem_limit(size_t bytes) {
  const int b = static_cast<int>(bytes);
  const int half = static_cast<int>(bytes / 2 - 1024);  // two CTAs per SM
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(score_kernel<false, 16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, b)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(score_kernel<true, 16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, b)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(score_kernel<false, 8>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, half)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(score_kernel<true, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              half);
}

namespace {

template <bool kLse, int kEpi>
cudaError_t launch(const ScoreParams& p, int n_items, size_t smem, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n_items));
  cfg.blockDim = dim3(Shape<kEpi>::kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, score_kernel<kLse, kEpi>, p);
}

}  // namespace

cudaError_t launch_score(const ScoreParams& p, int n_items, size_t smem, cudaStream_t stream) {
  return p.epi_warps == 8 ? launch<false, 8>(p, n_items, smem, stream)
                          : launch<false, 16>(p, n_items, smem, stream);
}

cudaError_t launch_score_lse(const ScoreParams& p, int n_items, size_t smem, cudaStream_t stream) {
  return p.epi_warps == 8 ? launch<true, 8>(p, n_items, smem, stream)
                          : launch<true, 16>(p, n_items, smem, stream);
}

}  // namespace ckv
