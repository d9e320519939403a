// Persistent fused layer call (CompressKV Sec. 3.3 token selection with the
// SnapKV-style window of Sec. 4) for per-group selection: one launch scores
// every unit (sequence, KV group) of a call -- typically every layer of a
// model at the end of prefill -- pools the scores, takes the budgeted top-k,
// appends the window and gathers the retained K/V rows.
//
// What is computed is what the three-kernel path computes (scoring kernel,
// combine kernel, selection kernel), with the same arithmetic:
//   * per K tile of 128 keys and query row q of the unit's SRH heads, the
//     logits z = <q, k> * scale on tcgen05 tensor cores (fp32 in TMEM), the
//     exponents e = 2^(z c - R) stored as fp16 for prefix keys (R: the
//     owning warp's running reference, 7 below its largest scaled logit),
//     and per query the pair (M, S) with sum 2^(z c) = S 2^M;
//   * per unit, log2 D_q from the pairs, raw_j = sum_q e_qj 2^(R - log2 D_q),
//     pooled_j = (sum_{t=-h..h} raw_{j+t}) / P with zeros outside [0, n);
//   * the k = kept - W largest pooled scores (ties to the lower position) in
//     ascending position, the window positions, and the K/V rows.
//
// One CTA per SM runs for the whole call.  Its warps have fixed roles and
// never wait on another CTA, except where noted:
//   warp 0      claims scoring chunks (kChunkTiles tiles of one unit) from a
//               counter, publishes each in a small descriptor ring and
//               streams the chunk's K tiles into a shared-memory ring by TMA;
//               before the first chunk of unit u it waits until the unit that
//               last used u's exponent-table slot has been combined (other
//               CTAs: bounded);
//   warp 1      TMEM allocation and UMMA issue (M = 128 keys, N = query rows);
//   warp 2      copies each chunk's SRH query rows into one of two Q buffers;
//   warps 4-11  two epilogue warpgroups; tile t of a chunk belongs to
//               warpgroup t % 2, each with its own TMEM buffers;  at the end
//               of a chunk each warpgroup writes its (M, S) pairs and counts
//               itself in the unit's ticket;
//   warps 12-19 combine / select workers: they claim combine pieces (a run of
//               32-key quarters of one unit: wait for the unit's ticket, merge
//               the pairs once per unit, weight, sum and pool the exponent
//               rows) and, once every piece of a unit is done, the unit's
//               selection and gather (one CTA per unit).
// Every wait that depends on another CTA depends only on work that was
// claimed earlier by a running CTA and that never waits on later work, so
// the call completes whatever the number of CTAs resident at once; every
// wait is bounded (kWaitTimeoutNs) and on expiry records
// CKV_ERR_DEVICE_TIMEOUT and stops the call.
// The references restart at every chunk and tile t of a chunk always goes to
// warpgroup t % 2, so the scores depend only on the chunk grid (fixed per
// unit), not on which CTA ran a chunk: results are deterministic and the
// same whatever the other units of the call.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cfloat>

#include "ckv_device.cuh"
#include "select_common.cuh"

namespace ckv {

namespace {

constexpr int kFWarps = 20;
constexpr int kFThreads = 32 * kFWarps;
constexpr int kProdWarp = 0;
constexpr int kMmaWarp = 1;
constexpr int kStageWarp = 2;
constexpr int kEpiWarp0 = 4;  // warps 4..11: two warpgroups (TMEM lane quarter = warp % 4)
constexpr int kEpiWarps = 8;
constexpr int kCWarp0 = 12;   // warps 12..19
constexpr int kCThreads = 256;
constexpr int kDescs = 4;     // chunk descriptors in flight
constexpr int kBarC = 3;      // named barrier of the combine / select warps (1, 2: warpgroups)
constexpr float kShift = 7.0f;
constexpr float kRaise = 15.0f;
constexpr float kNegInf = -INFINITY;
constexpr int kLoadBatch = 4;

// counters (ints at p.ctr)
constexpr int kCtrChunk = 0;  // next scoring chunk
constexpr int kCtrPiece = 1;  // next combine piece
constexpr int kCtrSel = 2;    // next unit to select
constexpr int kCtrExit = 3;   // CTAs finished
constexpr int kCtrAbort = 4;  // set when any wait ran out

constexpr int kTaskEnd = 0;
constexpr int kTaskCombine = 1;
constexpr int kTaskSelect = 2;

struct ChunkDesc {
  int end, s, g, t0, t1, chunk, n_rows, list;
};

// Shared memory of the combine / select workers (one of the two at a time).
struct SelShared {
  int samp[256];
  uint32_t key[kFusedCandCap];
  int pos[kFusedCandCap];
  RadixShared rs;
  int wcnt[8], wbase[8];
  int red[2];
  uint32_t lo;
};
static_assert(sizeof(SelShared) <= kFusedCRegion, "select scratch");

// Fixed part of the dynamic shared memory (after the K ring and Q buffers).
constexpr int kRefBytes = kEpiWarps * kMaxQRows * 4;  // running references per epilogue warp
constexpr int kAccBytes = kEpiWarps * kMaxQRows * 4;  // per-query sums per epilogue warp
constexpr int kWposBytes = kMaxQRows * 4;
constexpr int kBarBytes = 512;
constexpr int kMiscBytes = 256;  // TMEM address, abort flag, task, descriptors
constexpr int kFixedBytes = kRefBytes + kAccBytes + kWposBytes + kBarBytes + kMiscBytes +
                            kDescs * static_cast<int>(sizeof(ChunkDesc));

__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ int ld_volatile(const int* p) {
  return *reinterpret_cast<const volatile int*>(p);
}

__device__ __forceinline__ void cbar() { named_bar_sync(kBarC, kCThreads); }

// Index of the i-th set bit of `bits` (i < popc(bits)).
__device__ __forceinline__ int nth_bit(uint32_t bits, int i) {
  for (int j = 0; j < i; ++j) bits &= bits - 1u;
  return __ffs(bits) - 1;
}

// Largest s in [0, n) with off[s] <= x (off ascending, off[n] > x).
__device__ __forceinline__ int find_seq(const int* off, int n, int x) {
  int lo = 0, hi = n;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (off[mid] <= x) lo = mid; else hi = mid;
  }
  return lo;
}

struct Fused {
  const FusedParams& p;
  int* abort_cta;  // shared-memory abort flag of this CTA

  __device__ int len(int s) const { return p.cu_seqlens[s + 1] - p.cu_seqlens[s]; }
  __device__ int prefix(int s) const { return max(len(s) - p.window, 0); }
  __device__ int tiles(int s) const { return (len(s) + kTileTokens - 1) / kTileTokens; }
  __device__ int chunks_per_unit(int s) const {
    return (p.chunk_off[s + 1] - p.chunk_off[s]) / p.num_kv_heads;
  }
  __device__ int pieces_per_unit(int s) const {
    return (p.piece_off[s + 1] - p.piece_off[s]) / p.num_kv_heads;
  }
  __device__ int list(int s, int g) const { return srh_group(s, g, p.seqs_per_mask, p.num_kv_heads); }
  __device__ int rows(int s, int g) const { return __popc(p.srh_bits[list(s, g)]) * p.window; }
  __device__ int* ticket(int u) const { return p.ctr + kFusedCtrHead + u; }
  __device__ int* combdone(int u) const { return p.ctr + kFusedCtrHead + p.n_units + u; }
  __device__ int* bias_state(int u) const { return p.ctr + kFusedCtrHead + 2 * p.n_units + u; }
  __device__ uint16_t* expo_slot(int u) const {
    return p.expo + static_cast<long long>(u % p.n_slots) * p.slot_expo;
  }
  __device__ float* refs_slot(int u) const {
    return p.refs + static_cast<long long>(u % p.n_slots) * p.slot_refs;
  }
  __device__ bool aborted() const { return ld_volatile(p.ctr + kCtrAbort) != 0; }
  __device__ void raise_abort() const {
    atomicCAS(p.status, 0, CKV_DEV_ERR_TIMEOUT);
    atomicExch(p.ctr + kCtrAbort, 1);
    *reinterpret_cast<volatile int*>(abort_cta) = 1;
  }
  // Bounded wait (another CTA's progress) until *ptr >= target; false when
  // the call was aborted or the wait ran out.
  __device__ bool wait_counter(const int* ptr, int target) const {
    if (ld_acquire(ptr) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
      __nanosleep(128);
      if (ld_acquire(ptr) >= target) return true;
      if (aborted() || *reinterpret_cast<volatile int*>(abort_cta)) return false;
      if (globaltimer_ns() - t0 > kWaitTimeoutNs) {
        raise_abort();
        return false;
      }
    }
  }
  // Bounded wait on one of this CTA's mbarriers; a timeout stops the call.
  __device__ bool wait_bar(uint32_t bar, uint32_t parity) const {
    const bool ok = mbar_wait_bounded(bar, parity, abort_cta, p.status);
    if (!ok && !aborted()) atomicExch(p.ctr + kCtrAbort, 1);
    return ok;
  }
};

// ---------------------------------------------------------------- combine
__device__ __forceinline__ float dot8w(const uint4 v, const float* w) {
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

// One combine piece: quarters [q_first, q_last) of unit (s, g).  All 256
// worker threads (ct = 0..255).  Returns false if the call was aborted.
__device__ __noinline__ bool combine_piece(const Fused& F, int x, uint8_t* creg, int ct) {
  const FusedParams& p = F.p;
  const int s = find_seq(p.piece_off, p.batch, x);
  const int npc = F.pieces_per_unit(s);
  const int local = x - p.piece_off[s];
  const int g = local / npc;
  const int pc = local - g * npc;
  const int u = s * p.num_kv_heads + g;
  const int n = F.prefix(s);
  const int N = F.rows(s, g);
  const int Nr = expo_stride(N);
  const int cpr = Nr >> 3;
  const int lg_cpr = __ffs(cpr) - 1;
  const int col = ct & (cpr - 1);
  const int h = (p.pool_width - 1) >> 1;
  const int quarters = (n + 31) >> 5;
  const int qa = pc * p.piece_quarters;
  const int qb = min(quarters, qa + p.piece_quarters);
  const int a = qa * 32;
  const int b = min(qb * 32, n);
  const int base = a - h;
  const int span = b - a + 2 * h;
  const int ea = max(base, 0);
  const int eb = min(b + h, n);
  const int q0 = ea >> 5;
  const int nqt = ((eb + 31) >> 5) - q0;
  float* s_bias = reinterpret_cast<float*>(creg);             // [256]
  float* s_mm = s_bias + kMaxQRows;                           // [256] merge scratch (M)
  float* s_mz = s_mm + kMaxQRows;                             // [256] merge scratch (S)
  int* s_flag = reinterpret_cast<int*>(s_mz + kMaxQRows);     // [4]
  float* s_w = s_mz + kMaxQRows + 4;                          // [nqt][Nr] (16-byte aligned)
  float* s_raw = s_w + nqt * Nr;                              // [span]

  for (int i = ct; i < span; i += kCThreads) s_raw[i] = 0.f;
  // every scoring contribution of the unit (two per chunk) has landed
  if (ct == 0) {
    const bool ok = F.wait_counter(F.ticket(u), 2 * F.chunks_per_unit(s));
    s_flag[0] = ok ? 1 : 0;
    s_flag[1] = ok ? atomicCAS(F.bias_state(u), 0, 1) : 2;
  }
  cbar();
  if (!s_flag[0]) return false;
  float* bias_g = p.bias + static_cast<long long>(u) * p.part_stride;
  if (s_flag[1] == 0) {
    // this piece merges the unit's pairs once: nm threads per query row,
    // sixteen pairs in flight per thread
    const int nparts = 2 * F.chunks_per_unit(s);
    const float2* parts =
        p.partials + static_cast<long long>(p.chunk_off[s] + g * F.chunks_per_unit(s)) * 2 *
                         p.part_stride;
    const int nm = kCThreads / N;
    const int q = ct % N;
    const int sub = ct / N;
    if (sub < nm) {
      float m = kNegInf, z = 0.f;
      for (int i0 = sub; i0 < nparts; i0 += 16 * nm) {
        float2 pr[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const int i = i0 + k * nm;
          pr[k] = i < nparts ? __ldcg(parts + static_cast<long long>(i) * p.part_stride + q)
                             : make_float2(kNegInf, 0.f);
        }
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          if (pr[k].x == kNegInf) continue;
          if (pr[k].x > m) {
            z = fmaf(z, ex2_approx(m - pr[k].x), pr[k].y);
            m = pr[k].x;
          } else {
            z = fmaf(pr[k].y, ex2_approx(pr[k].x - m), z);
          }
        }
      }
      s_mm[sub * N + q] = m;  // nm * N <= 256
      s_mz[sub * N + q] = z;
    }
    cbar();
    if (ct < N) {
      float m = kNegInf, z = 0.f;
      for (int j = 0; j < nm; ++j) {
        const float pm = s_mm[j * N + ct];
        const float pz = s_mz[j * N + ct];
        if (pm == kNegInf) continue;
        if (pm > m) {
          z = fmaf(z, ex2_approx(m - pm), pz);
          m = pm;
        } else {
          z = fmaf(pz, ex2_approx(pm - m), z);
        }
      }
      const float bq = m + __log2f(z);
      s_bias[ct] = bq;
      bias_g[ct] = bq;
    }
    __threadfence();
    cbar();
    if (ct == 0) atomicExch(F.bias_state(u), 2);
  } else {
    if (ct == 0) s_flag[2] = F.wait_counter(F.bias_state(u), 2) ? 1 : 0;
    cbar();
    if (!s_flag[2]) return false;  // (a slot no thread still reads)
    if (ct < N) s_bias[ct] = __ldcg(bias_g + ct);
  }
  // references of the quarters touched (the piece plus an h-key halo each
  // side), turned into weights 2^(R - log2 D_q) in place
  const float* R = F.refs_slot(u) + static_cast<long long>(q0) * Nr;
  for (int i = 4 * ct; i < nqt * Nr; i += 4 * kCThreads)
    *reinterpret_cast<float4*>(s_w + i) = __ldcg(reinterpret_cast<const float4*>(R + i));
  cbar();
  for (int i = ct; i < nqt * Nr; i += kCThreads) {
    const int cc = i & (Nr - 1);
    s_w[i] = cc < N ? ex2_approx(s_w[i] - s_bias[cc]) : 0.f;
  }
  cbar();
  // raw scores of keys [ea, eb): one contiguous run of exponent rows
  const uint4* E4 = reinterpret_cast<const uint4*>(F.expo_slot(u));
  const int f_lo = ea * cpr;
  const int f_hi = eb * cpr;
  uint4 ev[kLoadBatch];
#pragma unroll
  for (int k = 0; k < kLoadBatch; ++k) {
    const int f = f_lo + k * kCThreads + ct;
    ev[k] = f < f_hi ? __ldcg(E4 + f) : make_uint4(0u, 0u, 0u, 0u);
  }
  for (int f0 = f_lo; f0 < f_hi; f0 += kLoadBatch * kCThreads) {
    uint4 nx[kLoadBatch];
    const int f1 = f0 + kLoadBatch * kCThreads;
    if (f1 < f_hi) {
#pragma unroll
      for (int k = 0; k < kLoadBatch; ++k) {
        const int f = f1 + k * kCThreads + ct;
        nx[k] = f < f_hi ? __ldcg(E4 + f) : make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int k = 0; k < kLoadBatch; ++k) {
      const int f = f0 + k * kCThreads + ct;
      const int row = f >> lg_cpr;
      const int qq = min((row >> 5) - q0, nqt - 1);
      float v = dot8w(ev[k], s_w + qq * Nr + 8 * col);
      for (int off = cpr >> 1; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      if (f < f_hi && col == 0) s_raw[row - base] = v;
    }
    if (f1 < f_hi) {
#pragma unroll
      for (int k = 0; k < kLoadBatch; ++k) ev[k] = nx[k];
    }
  }
  cbar();
  // table lines no other piece reads (inside [a + h, b - h)) need no
  // write-back to DRAM
  {
    const long long row_bytes = static_cast<long long>(Nr) * 2;
    const uintptr_t tb = reinterpret_cast<uintptr_t>(F.expo_slot(u));
    const long long lo_b = ((static_cast<long long>(a + h + 1) * row_bytes + 127) / 128) * 128;
    const long long hi_b = ((static_cast<long long>(b - h - 1) * row_bytes) / 128) * 128;
    for (long long xb = lo_b + static_cast<long long>(ct) * 128; xb + 128 <= hi_b;
         xb += static_cast<long long>(kCThreads) * 128) {
      const char* line = reinterpret_cast<const char*>(tb) + xb;
      asm volatile("discard.global.L2 [%0], 128;" ::"l"(line) : "memory");
    }
  }
  const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  const float fP = static_cast<float>(p.pool_width);
  for (int j = a + ct; j < b; j += kCThreads) {
    const int i = j - a;
    float acc = 0.f;
    for (int t = 0; t <= 2 * h; ++t) acc += s_raw[i + t];
    p.pooled[soff + j] = acc / fP;
    if (p.raw_out) p.raw_out[soff + j] = s_raw[i + h];
  }
  __threadfence();
  cbar();
  if (ct == 0) atomicAdd(F.combdone(u), 1);
  return true;
}

// ---------------------------------------------------------------- select
// Zero the radix state (the workers' form of radix_init).
__device__ __forceinline__ void radix_init_grp(RadixShared& sh, int ct) {
  for (int i = ct; i < 2 * 256; i += kCThreads) sh.hist[i >> 8][i & 255] = 0u;
  if (ct < 2) {
    sh.key_or[ct] = 0u;
    sh.key_and[ct] = 0xFFFFFFFFu;
  }
}

// The workers' form of cta_kth_largest (256 threads, named barrier): the
// r-th largest of min(keys[j] - sub, clamp), j < count; *rem = how many of
// the keys equal to it are among the r largest.
__device__ __noinline__ uint32_t grp_kth_largest(const uint32_t* keys, int count, uint32_t sub,
                                                 uint32_t clamp, int r, RadixShared& sh, int slot,
                                                 int& pc, int* rem, int ct, bool global_keys) {
  const int lane = ct & 31;
  const int iters = (count + 255) >> 8;
  auto key_at = [&](int j) -> uint32_t {
    const uint32_t k = global_keys ? __ldcg(keys + j) : keys[j];
    return min(k - sub, clamp);
  };
  uint32_t ko = 0u, ka = 0xFFFFFFFFu;
#pragma unroll 4
  for (int i = 0; i < iters; ++i) {
    const int j = (i << 8) + ct;
    if (j < count) {
      const uint32_t key = key_at(j);
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
  cbar();
  const uint32_t diff = sh.key_or[slot] ^ sh.key_and[slot];
  const uint32_t kand = sh.key_and[slot];
  int remaining = r;
  if (diff == 0u) {
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
    uint32_t* hh = sh.hist[pc & 3];
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
      const int j = (i << 8) + ct;
      const uint32_t key = j < count ? key_at(j) : 0u;
      const bool m = j < count && (key & pmask) == prefix;
      const uint32_t act = __ballot_sync(0xffffffffu, m);
      if (!act) continue;
      const uint32_t bin = (key >> shf) & fm;
      const int leader = __ffs(act) - 1;
      const uint32_t lb = __shfl_sync(0xffffffffu, bin, leader);
      if (__all_sync(0xffffffffu, !m || bin == lb)) {
        if (lane == leader) atomicAdd(&hh[lb], static_cast<uint32_t>(__popc(act)));
      } else if (m) {
        atomicAdd(&hh[bin], 1u);
      }
    }
    sh.hist[(pc + 2) & 3][ct] = 0u;
    cbar();
    int bin, above;
    warp_pick_bin256(hh, remaining, lane, &bin, &above);
    remaining -= above;
    prefix |= static_cast<uint32_t>(bin) << shf;
    pmask |= fm << shf;
    hb = shf - 1;
    ++pc;
  }
  *rem = remaining;
  return prefix;
}

// Ordered emission of the selected entries of a key list in position order:
// entry j (key key_at(j), position pos_at(j)) is selected when its key is
// above tau, or equal to tau and fewer than need_eq equal keys precede it.
// Selected entries go to out[0..k) in list order.
template <class KeyAt, class PosAt>
__device__ void emit_selected(int count, uint32_t tau, int need_eq, int32_t* out, int k,
                              SelShared& sh, int ct, KeyAt key_at, PosAt pos_at) {
  const int cw = ct >> 5;
  const int lane = ct & 31;
  int o = 0, eq_seen = 0;
  for (int j0 = 0; j0 < count; j0 += kCThreads) {
    const int j = j0 + ct;
    const bool in = j < count;
    const uint32_t key = in ? key_at(j) : 0u;
    const bool gt = in && key > tau;
    const bool eq = in && key == tau;
    const uint32_t mgt = __ballot_sync(0xffffffffu, gt);
    const uint32_t meq = __ballot_sync(0xffffffffu, eq);
    if (lane == 0) {
      sh.wcnt[cw] = __popc(mgt);
      sh.wbase[cw] = __popc(meq);
    }
    cbar();
    int gtb = 0, eqb = 0, gtt = 0, eqt = 0;
    for (int w = 0; w < 8; ++w) {
      if (w < cw) {
        gtb += sh.wcnt[w];
        eqb += sh.wbase[w];
      }
      gtt += sh.wcnt[w];
      eqt += sh.wbase[w];
    }
    const int eq_rank = eq_seen + eqb + __popc(meq & lanemask_lt(lane));
    const bool take_eq = eq && eq_rank < need_eq;
    const uint32_t msel = mgt | __ballot_sync(0xffffffffu, take_eq);
    const int eq_taken_before = max(0, min(need_eq - eq_seen, eqb));
    const int slot = o + gtb + eq_taken_before + __popc(msel & lanemask_lt(lane));
    if (((msel >> lane) & 1u) && slot < k) out[slot] = pos_at(j);
    o += gtt + max(0, min(need_eq - eq_seen, eqt));
    eq_seen += eqt;
    cbar();
  }
}

// Copy the K and V rows of out[0..count) (positions in the sequence) to the
// compressed cache rows out0 .. out0 + count - 1 of group g.  Eight 16-byte
// loads in flight per thread.
__device__ __noinline__ void gather_rows(const FusedParams& p, int seq0, int g,
                                         const int32_t* out, int out0, int count, int ct) {
  constexpr int kChunks = 2 * kHeadDim * 2 / 16;  // 16 K + 16 V chunks per token
  constexpr int kBatch = 8;
  const int total = count * kChunks;
  for (int base = 0; base < total; base += kBatch * kCThreads) {
    uint4 v[kBatch];
    long long dst[kBatch];
    bool is_v[kBatch];
#pragma unroll
    for (int k = 0; k < kBatch; ++k) {
      const int e = base + k * kCThreads + ct;
      dst[k] = -1;
      is_v[k] = false;
      if (e < total) {
        const int i = e / kChunks;
        const int ch = e - i * kChunks;
        const int tok = out[i];
        is_v[k] = ch >= kChunks / 2;
        const int part = ch & (kChunks / 2 - 1);
        const long long src = static_cast<long long>(seq0 + tok) * p.tok_stride_v16 +
                              static_cast<long long>(g) * p.head_stride_v16 + part;
        v[k] = __ldg((is_v[k] ? p.v : p.k) + src);
        dst[k] = (static_cast<long long>(out0 + i) * p.num_kv_heads + g) * (kHeadDim * 2 / 16) + part;
      }
    }
#pragma unroll
    for (int k = 0; k < kBatch; ++k)
      if (dst[k] >= 0) (is_v[k] ? p.v_out : p.k_out)[dst[k]] = v[k];
  }
}

// Selection of unit u: top-k of its pooled scores by a sampled lower bound,
// candidates in position order, an exact radix search among them (all the
// unit's scores when the bound keeps too few or too many), the window, and
// the K/V rows.  Pooled scores are >= 0: their bit patterns order like
// their values.
__device__ __noinline__ void select_unit(const Fused& F, int u, uint8_t* creg, int ct) {
  const FusedParams& p = F.p;
  SelShared& sh = *reinterpret_cast<SelShared*>(creg);
  const int cw = ct >> 5;
  const int lane = ct & 31;
  const int s = u / p.num_kv_heads;
  const int g = u - s * p.num_kv_heads;
  const int seq0 = p.cu_seqlens[s];
  const int L = F.len(s);
  const int W = p.window;
  const int n = F.prefix(s);
  const int out0 = p.cu_out[s];
  const int kept = p.cu_out[s + 1] - out0;
  int32_t* out = p.indices + static_cast<long long>(g) * p.o_total + out0;
  if (kept >= L) {  // keep everything
    for (int i = ct; i < L; i += kCThreads) out[i] = i;
    __threadfence_block();
    cbar();
    gather_rows(p, seq0, g, out, out0, L, ct);
    return;
  }
  const int k = kept - W;  // 0 <= k < n
  for (int w = ct; w < W; w += kCThreads) out[k + w] = n + w;
  if (k == 0) {
    cbar();
    gather_rows(p, seq0, g, out, out0, W, ct);
    return;
  }
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(
      p.pooled + static_cast<long long>(g) * p.p_total + p.cu_prefix[s]);
  // samples: ns evenly spaced keys
  const int ns = min(256, n);
  sh.samp[ct] = ct < ns ? static_cast<int>(__ldcg(keys + static_cast<int>(
                                                  (static_cast<long long>(ct) * n) / ns)))
                        : -1;
  radix_init_grp(sh.rs, ct);
  cbar();
  const float mu = static_cast<float>(k) * static_cast<float>(ns) / static_cast<float>(n);
  int rs = min(ns, static_cast<int>(ceilf(mu + 3.f * sqrtf(mu))) + 2);
  uint32_t lo = 0;
  int total = 0;
  // positions per warp (multiple of 32)
  const int seg = ((n + 8 * 32 - 1) / (8 * 32)) * 32;
  const int wlo = min(n, cw * seg);
  const int whi = min(n, wlo + seg);
  bool fast = false;
  for (int attempt = 0; attempt < 2; ++attempt) {
    {  // the rs-th largest sample
      const int v = sh.samp[ct];
      const int4* s4 = reinterpret_cast<const int4*>(sh.samp);
      int gt = 0, eq = 0;
#pragma unroll 8
      for (int j = 0; j < 64; ++j) {
        const int4 xx = s4[j];
        gt += (xx.x > v) + (xx.y > v) + (xx.z > v) + (xx.w > v);
        eq += (xx.x == v) + (xx.y == v) + (xx.z == v) + (xx.w == v);
      }
      if (v >= 0 && gt < rs && rs <= gt + eq) sh.lo = static_cast<uint32_t>(v);
    }
    cbar();
    lo = sh.lo;
    int wc = 0;
    for (int b0 = wlo; b0 < whi; b0 += 32) {
      const int i = b0 + lane;
      wc += __popc(__ballot_sync(0xffffffffu, i < whi && __ldcg(keys + i) >= lo));
    }
    if (lane == 0) sh.wcnt[cw] = wc;
    cbar();
    total = 0;
    for (int w = 0; w < 8; ++w) total += sh.wcnt[w];
    if (total >= k && total <= kFusedCandCap) {
      fast = true;
      break;
    }
    if (total > kFusedCandCap || rs >= ns) break;
    rs = min(ns, max(rs + 1, static_cast<int>(ceilf(0.5f * static_cast<float>(k + kFusedCandCap) *
                                                    static_cast<float>(ns) /
                                                    static_cast<float>(n)))));
    cbar();  // every thread has read sh.lo and the counts
  }
  int pc = 0, need_eq = 0;
  uint32_t tau;
  if (fast) {
    // candidates (keys >= lo) in position order
    int o = 0;
    for (int w = 0; w < cw; ++w) o += sh.wcnt[w];
    for (int b0 = wlo; b0 < whi; b0 += 32) {
      const int i = b0 + lane;
      const uint32_t key = i < whi ? __ldcg(keys + i) : 0u;
      const bool c = i < whi && key >= lo;
      const uint32_t mm = __ballot_sync(0xffffffffu, c);
      const int slot = o + __popc(mm & lanemask_lt(lane));
      if (c) {
        sh.key[slot] = key;
        sh.pos[slot] = i;
      }
      o += __popc(mm);
    }
    cbar();
    constexpr uint32_t kClamp = 0xFFFFu;
    const uint32_t td = grp_kth_largest(sh.key, total, lo, kClamp, k, sh.rs, 0, pc, &need_eq, ct,
                                        false);
    tau = lo + td;
    if (td == kClamp)
      tau = grp_kth_largest(sh.key, total, 0u, 0xFFFFFFFFu, k, sh.rs, 1, pc, &need_eq, ct, false);
    emit_selected(total, tau, need_eq, out, k, sh, ct, [&](int j) { return sh.key[j]; },
                  [&](int j) { return sh.pos[j]; });
  } else {
    tau = grp_kth_largest(keys, n, 0u, 0xFFFFFFFFu, k, sh.rs, 1, pc, &need_eq, ct, true);
    emit_selected(n, tau, need_eq, out, k, sh, ct, [&](int j) { return __ldcg(keys + j); },
                  [&](int j) { return j; });
  }
  __threadfence_block();
  cbar();  // the indices written above are read back by the copy
  gather_rows(p, seq0, g, out, out0, kept, ct);
}


// Claim the workers' next task (one thread): the next unit to select once all
// its combine pieces are done, else the next combine piece, else wait for
// the next selection to become ready.  Without selection (scores only) the
// workers stop when every piece is claimed.
__device__ void claim_task(const Fused& F, int* task) {
  const FusedParams& p = F.p;
  uint64_t t0 = 0;
  for (;;) {
    if (F.aborted() || *reinterpret_cast<volatile int*>(F.abort_cta)) break;
    const int u = p.do_select ? ld_volatile(p.ctr + kCtrSel) : p.n_units;
    if (u >= p.n_units && ld_volatile(p.ctr + kCtrPiece) >= p.n_pieces)
      break;  // every unit selected (every piece combined), or scores only and no piece left
    if (u < p.n_units && ld_acquire(F.combdone(u)) >= F.pieces_per_unit(u / p.num_kv_heads)) {
      if (atomicCAS(p.ctr + kCtrSel, u, u + 1) == u) {
        task[0] = kTaskSelect;
        task[1] = u;
        return;
      }
      continue;
    }
    if (ld_volatile(p.ctr + kCtrPiece) < p.n_pieces) {
      const int x = atomicAdd(p.ctr + kCtrPiece, 1);
      if (x < p.n_pieces) {
        task[0] = kTaskCombine;
        task[1] = x;
        return;
      }
    }
    // every piece is claimed; the next unit's last pieces are still running
    const uint64_t now = globaltimer_ns();
    if (t0 == 0) {
      t0 = now;
    } else if (now - t0 > kWaitTimeoutNs) {
      F.raise_abort();
      break;
    }
    __nanosleep(256);
  }
  task[0] = kTaskEnd;
  task[1] = 0;
}

__device__ __forceinline__ void wait_plain(uint32_t bar, uint32_t parity, uint64_t timeout_ns) {
  volatile int never = 0;
  mbar_wait_bounded(bar, parity, &never, nullptr, timeout_ns);
}

__global__ void __launch_bounds__(kFThreads, 1) fused_kernel(const __grid_constant__ FusedParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int nst = p.stages;
  const int qh = p.q_half_bytes;
  uint8_t* sK = base;
  uint8_t* sQ = base + nst * kTileBytes;  // two buffers of two 64-column halves
  float* sRef = reinterpret_cast<float*>(sQ + 4 * qh);
  float* sAcc = sRef + kEpiWarps * kMaxQRows;
  int* sWpos = reinterpret_cast<int*>(sAcc + kEpiWarps * kMaxQRows);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sWpos + kMaxQRows);
  uint8_t* misc = reinterpret_cast<uint8_t*>(bars) + kBarBytes;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(misc);
  int* abort_cta = reinterpret_cast<int*>(misc + 4);
  int* s_task = reinterpret_cast<int*>(misc + 16);
  int* s_last = reinterpret_cast<int*>(misc + 32);
  ChunkDesc* descs = reinterpret_cast<ChunkDesc*>(misc + kMiscBytes);
  uint8_t* creg = reinterpret_cast<uint8_t*>(descs + kDescs);

  const uint32_t bar0 = smem_u32(bars);
  auto full = [&](int i) { return bar0 + 8u * i; };             // K stage landed
  auto empty = [&](int i) { return bar0 + 8u * (8 + i); };      // K stage consumed
  auto tfull = [&](int b) { return bar0 + 8u * (16 + b); };     // TMEM buffer written
  auto tempty = [&](int b) { return bar0 + 8u * (24 + b); };    // TMEM buffer read
  auto dfull = [&](int i) { return bar0 + 8u * (32 + i); };     // descriptor written
  auto dempty = [&](int i) { return bar0 + 8u * (36 + i); };    // descriptor read by all
  auto qfull = [&](int i) { return bar0 + 8u * (40 + i); };     // Q buffer staged
  auto qempty = [&](int i) { return bar0 + 8u * (42 + i); };    // Q buffer's MMAs done
  auto wgbar = [&](int w) { return bar0 + 8u * (44 + w); };     // epilogue warpgroup sync

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int W = p.window;
  const int Hkv = p.num_kv_heads;
  const Fused F{p, abort_cta};

  if (threadIdx.x == 0) {
    for (int i = 0; i < nst; ++i) {
      mbar_init(full(i), 1);
      mbar_init(empty(i), 1);
    }
    for (int b = 0; b < p.nbuf; ++b) {
      mbar_init(tfull(b), 1);
      mbar_init(tempty(b), 4);  // the four warps of the owning warpgroup
    }
    for (int i = 0; i < kDescs; ++i) {
      mbar_init(dfull(i), 1);
      mbar_init(dempty(i), 2 + kEpiWarps);  // MMA, stager, epilogue warps
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(qfull(i), 1);
      mbar_init(qempty(i), 1);
      mbar_init(wgbar(i), 4);
    }
    *abort_cta = 0;
    fence_mbar_init();
  }
  for (int q = threadIdx.x; q < kMaxQRows; q += kFThreads) sWpos[q] = q % W;
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_holder), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tmem_holder;

  if (warp == kProdWarp) {
    // ------------------------------------------------------------ chunks + TMA
    if (lane == 0) {
      const uint64_t kpol = l2_policy_evict_first();
      int gt = 0;  // K tiles issued
      for (int c = 0;; ++c) {
        const int ds = c % kDescs;
        if (!F.wait_bar(dempty(ds), ((c / kDescs) & 1) ^ 1)) break;
        ChunkDesc d;
        d.end = 1;
        const int x = F.aborted() ? p.n_chunks : atomicAdd(p.ctr + kCtrChunk, 1);
        if (x < p.n_chunks) {
          const int s = find_seq(p.chunk_off, p.batch, x);
          const int ncu = F.chunks_per_unit(s);
          const int local = x - p.chunk_off[s];
          const int g = local / ncu;
          const int cc = local - g * ncu;
          const int u = s * Hkv + g;
          // the exponent-table slot's previous unit has been combined
          bool ok = true;
          if (u >= p.n_slots) {
            const int up = u - p.n_slots;
            ok = F.wait_counter(F.combdone(up), F.pieces_per_unit(up / Hkv));
          }
          if (ok) {
            d.end = 0;
            d.s = s;
            d.g = g;
            d.t0 = cc * kChunkTiles;
            d.t1 = min(F.tiles(s), d.t0 + kChunkTiles);
            d.chunk = x;
            d.list = F.list(s, g);
            d.n_rows = __popc(p.srh_bits[d.list]) * W;
          }
        }
        descs[ds] = d;
        mbar_arrive(dfull(ds));
        if (d.end) break;
        const int row0 = p.cu_seqlens[d.s];
        bool stop = false;
        for (int t = d.t0; t < d.t1; ++t) {
          const int st = gt % nst;
          if (!F.wait_bar(empty(st), (static_cast<uint32_t>(gt / nst) & 1u) ^ 1u)) {
            stop = true;
            break;
          }
          mbar_arrive_expect_tx(full(st), kTileBytes);
          const uint32_t dst = smem_u32(sK + st * kTileBytes);
          const int row = row0 + t * kTileTokens;
          tma_load_3d(dst, &p.tmap_k, full(st), 0, d.g, row, kpol);
          tma_load_3d(dst + kHalfTileBytes, &p.tmap_k, full(st), 64, d.g, row, kpol);
          ++gt;
        }
        if (stop) break;
      }
      if (*reinterpret_cast<volatile int*>(abort_cta)) {
        // let the copies already issued land before the CTA can exit
        for (int i = max(0, gt - nst); i < gt; ++i)
          wait_plain(full(i % nst), static_cast<uint32_t>(i / nst) & 1u, 100000000ull);
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ UMMA issue
    if (lane == 0) {
      const uint64_t dk0 = smem_desc_sw128(smem_u32(sK));
      const int half = p.nbuf >> 1;
      int gt = 0;
      int kw[2] = {0, 0};
      int last_b = -1;
      uint32_t last_use = 0;
      for (int c = 0;; ++c) {
        const int ds = c % kDescs;
        if (!F.wait_bar(dfull(ds), static_cast<uint32_t>(c / kDescs) & 1u)) break;
        const ChunkDesc d = descs[ds];
        mbar_arrive(dempty(ds));
        if (d.end) break;
        const int qb = c & 1;
        if (!F.wait_bar(qfull(qb), static_cast<uint32_t>(c >> 1) & 1u)) break;
        tc_fence_after();
        const int Npad = (d.n_rows + 15) & ~15;
        const uint32_t idesc = umma_idesc_f16(kTileTokens, Npad, p.is_bf16 != 0);
        const uint64_t dq0 = smem_desc_sw128(smem_u32(sQ + qb * 2 * qh));
        bool stop = false;
        for (int t = d.t0; t < d.t1; ++t) {
          const int wg = (t - d.t0) & 1;
          const int kk = kw[wg]++;
          const int b = wg + 2 * (kk % half);
          const uint32_t use = static_cast<uint32_t>(kk / half) & 1u;
          if (!F.wait_bar(tempty(b), use ^ 1u)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const int st = gt % nst;
          if (!F.wait_bar(full(st), static_cast<uint32_t>(gt / nst) & 1u)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tbase + static_cast<uint32_t>(b * p.tstride);
#pragma unroll
          for (int k8 = 0; k8 < kHeadDim / 16; ++k8) {
            const uint32_t koff = st * kTileBytes + (k8 >> 2) * kHalfTileBytes + (k8 & 3) * 32;
            const uint32_t qoff = (k8 >> 2) * qh + (k8 & 3) * 32;
            umma_f16(dt, dk0 + (koff >> 4), dq0 + (qoff >> 4), idesc, k8 > 0 ? 1u : 0u);
          }
          umma_commit(empty(st));
          umma_commit(tfull(b));
          last_b = b;
          last_use = use;
          ++gt;
        }
        if (stop) break;
        umma_commit(qempty(qb));
      }
      if (*reinterpret_cast<volatile int*>(abort_cta) && last_b >= 0)
        wait_plain(tfull(last_b), last_use, 100000000ull);  // MMAs done before TMEM is freed
    }
    __syncwarp();
  } else if (warp == kStageWarp) {
    // ------------------------------------------------------------ Q rows
    const int G = p.group_size;
    for (int c = 0;; ++c) {
      const int ds = c % kDescs;
      const bool got = F.wait_bar(dfull(ds), static_cast<uint32_t>(c / kDescs) & 1u);
      if (!__all_sync(0xffffffffu, got)) break;
      const ChunkDesc d = descs[ds];
      __syncwarp();
      if (lane == 0) mbar_arrive(dempty(ds));
      if (d.end) break;
      const int qb = c & 1;
      const bool ok = F.wait_bar(qempty(qb), (static_cast<uint32_t>(c >> 1) & 1u) ^ 1u);
      if (!__all_sync(0xffffffffu, ok)) break;
      const int N = d.n_rows;
      const int Npad = (N + 15) & ~15;
      const uint32_t bits = p.srh_bits[d.list];
      uint8_t* qbuf = sQ + qb * 2 * qh;
      const long long sbase = static_cast<long long>(d.s) * p.q_bs;
      for (int idx = lane; idx < Npad * 16; idx += 32) {
        const int r = idx >> 4;
        const int ch = idx & 15;
        uint8_t* dst = qbuf + (ch >> 3) * qh + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
        if (r < N) {
          const int hi = r / W;
          const int w = r - hi * W;
          const int head = d.g * G + nth_bit(bits, hi);
          cp_async16(smem_u32(dst), p.q + sbase + static_cast<long long>(head) * p.q_hs +
                                        static_cast<long long>(w) * p.q_ws + ch * 8);
        } else {
          *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
        }
      }
      cp_async_wait_all();
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(qfull(qb));
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kEpiWarp0;
    const int wg = ew >> 2;
    const int qd = warp & 3;  // TMEM lane quarter of this warp
    const int tw = (ew & 3) * 32 + lane;
    float* ref = sRef + ew * kMaxQRows;
    float* acc_s = sAcc + ew * kMaxQRows;
    const float c = p.c;
    const uint64_t keep = l2_policy_evict_last();
    const int half = p.nbuf >> 1;
    int kc = 0;       // tiles this warpgroup has taken
    int nsync = 0;    // warpgroup syncs so far (mbarrier phase)
    bool stop = false;
    // bounded warpgroup barrier: a warp that stopped cannot hang the others
    auto wg_sync = [&]() -> bool {
      __syncwarp();
      if (lane == 0) mbar_arrive(wgbar(wg));
      const bool ok = F.wait_bar(wgbar(wg), static_cast<uint32_t>(nsync) & 1u);
      ++nsync;
      return __all_sync(0xffffffffu, ok);
    };
    for (int ci = 0; !stop; ++ci) {
      const int ds = ci % kDescs;
      const bool got = F.wait_bar(dfull(ds), static_cast<uint32_t>(ci / kDescs) & 1u);
      if (!__all_sync(0xffffffffu, got)) break;
      const ChunkDesc d = descs[ds];
      __syncwarp();
      if (lane == 0) mbar_arrive(dempty(ds));
      if (d.end) break;
      const int s = d.s;
      const int g = d.g;
      const int N = d.n_rows;
      const int Nr = expo_stride(N);
      const int L = F.len(s);
      const int n = L - W;
      const int u = s * Hkv + g;
      uint16_t* expo_u = F.expo_slot(u);
      float* refs_u = F.refs_slot(u);
      for (int q = lane; q < N; q += 32) {
        ref[q] = kNegInf;
        acc_s[q] = 0.f;
      }
      __syncwarp();
      const int ngrp = (Nr + 31) >> 5;
      for (int tile = d.t0 + wg; tile < d.t1; tile += 2) {
        const int kk = kc++;
        const int b = wg + 2 * (kk % half);
        const uint32_t use = static_cast<uint32_t>(kk / half) & 1u;
        const bool ok = F.wait_bar(tfull(b), use);
        if (!__all_sync(0xffffffffu, ok)) {
          stop = true;
          break;
        }
        tc_fence_after();
        const int tok = tile * kTileTokens + qd * 32 + lane;  // position in the sequence
        const uint32_t taddr = tbase + (static_cast<uint32_t>(qd * 32) << 16) +
                               static_cast<uint32_t>(b * p.tstride);
        const bool edge = (tile + 1) * kTileTokens > n;  // causal mask or sequence end
        const int vis = n - tok;  // query row q sees this key iff tok < L and wpos(q) >= -vis
        const bool key = tok < L;
        const bool store = tok < n;  // the table holds prefix keys only
        uint16_t* erow = expo_u + static_cast<long long>(tok) * Nr;
        for (int grp = 0; grp < ngrp; ++grp) {
          const int c0 = 32 * grp;
          const int ncols = min(32, Nr - c0);  // 8, 16 or 32
          if (c0 >= N) {
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
          const int lim = min(32, N - c0);
          const bool masked = edge || lim < 32;
          float* rf = ref + c0;
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
              for (int k = 0; k < 4; ++k) {
                const bool okk = (j + k) < lim && (!edge || (key && wv[k] >= -vis));
                t[j + k] = okk ? fmaf(__uint_as_float(r[j + k]), c, -rv[k]) : kNegInf;
                tmax = fmaxf(tmax, t[j + k]);
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
            // raise each query's R to kShift below its largest scaled logit in
            // this warp's 32 keys (always on the warp's first tile of a chunk)
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
              for (int k = 0; k < 4; ++k)
                t[j + k] = ((valid >> (j + k)) & 1u) ? fmaf(__uint_as_float(r[j + k]), c, -rv[k])
                                                      : kNegInf;
            }
          }
          float e[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) e[j] = ex2_approx(t[j]);
          if (store) {
#pragma unroll
            for (int v = 0; v < 2; ++v) {
              if (16 * v < ncols) {
                uint32_t pk[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) pk[k] = pack_half2(e[16 * v + 2 * k], e[16 * v + 2 * k + 1]);
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
        float* rt = refs_u + (static_cast<long long>(tile) * kQuarters + qd) * Nr;
        for (int q = lane; q < N; q += 32) rt[q] = ref[q];
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty(b));
      }
      if (stop) break;
      // the warpgroup's (M, S) pairs for this chunk, then its ticket
      if (!wg_sync()) break;
      float2* part = p.partials + (static_cast<long long>(d.chunk) * 2 + wg) * p.part_stride;
      for (int q = tw; q < N; q += 128) {
        float m = kNegInf;
        for (int w = 0; w < 4; ++w) m = fmaxf(m, sRef[(wg * 4 + w) * kMaxQRows + q]);
        float z = 0.f;
        for (int w = 0; w < 4; ++w) {
          const float rw = sRef[(wg * 4 + w) * kMaxQRows + q];
          if (rw != kNegInf) z += sAcc[(wg * 4 + w) * kMaxQRows + q] * ex2_approx(rw - m);
        }
        part[q] = make_float2(m, z);
      }
      __threadfence();
      if (!wg_sync()) break;
      if (tw == 0) atomicAdd(F.ticket(u), 1);
    }
  } else if (warp >= kCWarp0) {
    // ------------------------------------------------------------ combine / select
    const int ct = threadIdx.x - kCWarp0 * 32;
    for (;;) {
      if (ct == 0) claim_task(F, s_task);
      cbar();
      const int type = s_task[0];
      const int idx = s_task[1];
      cbar();
      if (type == kTaskEnd) break;
      if (type == kTaskCombine) {
        if (!combine_piece(F, idx, creg, ct)) break;
      } else {
        select_unit(F, idx, creg, ct);
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tbase, 512);
  }
  if (threadIdx.x == 0) {
    __threadfence();
    *s_last = atomicAdd(p.ctr + kCtrExit, 1) == static_cast<int>(gridDim.x) - 1 ? 1 : 0;
  }
  __syncthreads();
  if (*s_last) {
    // every other CTA has finished: zero the counters for the next call
    __threadfence();
    const int nz = kFusedCtrHead + 3 * p.n_units;
    for (int i = threadIdx.x; i < nz; i += kFThreads) p.ctr[i] = 0;
  }
}

}  // namespace

size_t fused_smem_bytes(int q_half_bytes, int stages) {
  return 1024 + static_cast<size_t>(stages) * kTileBytes + 4 * static_cast<size_t>(q_half_bytes) +
         kFixedBytes + kFusedCRegion;
}

cudaError_t fused_set_smem_limit(size_t bytes) {
  return cudaFuncSetAttribute(fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(bytes));
}

cudaError_t launch_fused(const FusedParams& p, int grid, size_t smem, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kFThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = nullptr;
  cfg.numAttrs = 0;
  return cudaLaunchKernelEx(&cfg, fused_kernel, p);
}

}  // namespace ckv
