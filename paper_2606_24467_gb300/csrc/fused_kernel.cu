// Persistent fused layer call (CompressKV Sec. 3.3 token selection with the
// SnapKV-style window of Sec. 4) for per-group selection: one launch scores
// every unit (sequence, KV group) of a call -- typically every layer of a
// model at the end of prefill -- pools the scores, takes the budgeted top-k,
// appends the window and gathers the retained K/V rows.
//
// For unit (s, g), with Q_S the N = |S_g| * W window-query rows of the
// group's SRH heads, z = <q, k> * scale and c = log2(e), query q (window
// position p_q) attends key j <= p_q with 2^(z_qj c) / D_q,
// D_q = sum_{j <= p_q} 2^(z_qj c).  The kernel makes two passes over the
// unit's K, both on tcgen05 tensor cores (logits in TMEM):
//   pass 1  per query row and epilogue warpgroup the pair (M, S) with
//           sum 2^(z c) = S 2^M over its tiles of a chunk of kChunkTiles K tiles (the epilogue keeps a reference R
//           per warp and query, 7 below the largest scaled logit it has seen,
//           and sums 2^(z c - R) exactly as the scoring kernel of the
//           separate path does); the workers merge a unit's pairs into
//           log2 D_q once every chunk of the unit is in;
//   pass 2  raw_j = sum_q 2^(z_qj c - log2 D_q) over the unit's prefix keys
//           j < n = L - W, straight from the logits in fp32; pass 2 of a
//           chunk is published only once its unit's denominators are merged
//           (it reads K again: in long calls pass 1 runs too far ahead for
//           L2 to keep it, so mostly from DRAM);
// then pooled_j = (sum_{t=-h..h} raw_{j+t}) / P with zeros outside [0, n)
// (inside a chunk by the epilogue from shared memory, within h of a chunk
// edge by the select), the k = kept - W largest pooled scores (ties to the
// lower position) in ascending position, the window, and the K/V rows.
// With the window queries' log-sum-exp given (given_lse) pass 1 is skipped
// and log2 D_q = LSE_q * log2(e).
//
// One CTA per SM runs for the whole call.  Its warps have fixed roles:
//   warp 3      claims chunks (a pass-2 chunk once its unit's denominators
//               are merged, else the next pass-1 chunk) and publishes them,
//               up to kDescs ahead, in a descriptor ring;
//   warp 0      loads each chunk's SRH query rows (one TMA box of W rows per
//               head and 64-column half) into one of two or three Q buffers
//               and streams its K tiles, by TMA, into a shared-memory ring
//               split in two sub-rings, one per UMMA warp (each consumes
//               its own in order);
//   warps 1, 2  UMMA issue (M = 128 keys, N = query rows), warp 1 for the
//               tiles of warpgroup 0 and warp 2 for those of warpgroup 1
//               (a UMMA of this shape holds the tensor core for a fixed 76
//               cycles whatever N up to 128, so two issuing threads, each
//               with its own waits, keep it fed); warp 1 also allocates TMEM;
//   warps 4-11  two epilogue warpgroups; tile t of a chunk belongs to
//               warpgroup t % nwg (nwg = 2), each with its own TMEM buffers;
//   warps 12-19 workers: they merge a unit's pass-1 pairs into its
//               denominators once all its chunks are in, and select and
//               gather a unit once all its pass-2 chunks are in (one CTA per
//               unit).
// A pass-2 chunk is published once its claimer has seen (acquire) its unit's
// denominators merged; workers claim a merge or a selection only
// when it is ready.  Every wait therefore depends only on
// work claimed earlier by a running CTA that never waits on later work, so a
// call completes whatever the number of CTAs resident at once; every wait
// is bounded (FusedParams::wait_ns, kWaitTimeoutNs unless a test shortens it)
// and on expiry records CKV_ERR_DEVICE_TIMEOUT
// and stops the call.
// References restart at every chunk and tile t of a chunk always goes to
// warpgroup t % nwg, so the scores depend only on the chunk grid (fixed per
// unit), not on which CTA ran a chunk or what else the call holds.
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
constexpr int kMmaWarp2 = 2;  // second UMMA issuer (tiles of warpgroup 1)
constexpr int kClaimWarp = 3;
constexpr int kEpiWarp0 = 4;  // warps 4..11: two warpgroups (TMEM lane quarter = warp % 4)
constexpr int kEpiWarps = 8;
constexpr int kCWarp0 = 12;   // warps 12..19
constexpr int kCThreads = 256;
constexpr int kDescs = 2;     // chunk descriptors in flight (claimed ahead; 2 measured faster than 4)
constexpr int kNwg = 2;       // epilogue warpgroups that take tiles (tile t of a chunk: t % 2)
constexpr int kSelSamples = 1024;  // samples of a unit's pooled scores for the select threshold
constexpr int kPub = 6;       // chunks written, not yet published (publish ring)
constexpr int kBarC = 3;      // named barrier of the worker warps
constexpr float kShift = 7.0f;
constexpr float kRaiseSum = 18446744073709551616.0f;  // 2^64: fp32 column sums stay below it before R is raised
constexpr float kNegInf = -INFINITY;

// counters (ints at p.ctr)
constexpr int kCtrPass1 = 0;  // next pass-1 chunk
constexpr int kCtrPass2 = 1;  // next pass-2 chunk
constexpr int kCtrMerge = 2;  // next unit whose denominators to merge
constexpr int kCtrSel = 3;    // next unit to select
constexpr int kCtrExit = 4;   // CTAs finished
constexpr int kCtrAbort = 5;  // set when any wait ran out
constexpr int kCtrNever = 6;  // never set: the test hook's stall waits for it

constexpr int kTaskEnd = 0;
constexpr int kTaskMerge = 1;
constexpr int kTaskSelect = 2;

struct ChunkDesc {
  int end, pass, s, g, t0, t1, chunk, n_rows;
};

// Shared memory of the worker warps (a merge or a selection at a time).
struct SelShared {
  uint32_t key[kFusedCandCap];
  int pos[kFusedCandCap];
  RadixShared rs;
  int wcnt[8], wbase[8];
  int wcnt_ge[8];  // per-warp counts at the best threshold with at least k keys above
  int flag[4];
  uint32_t lo;
};
static_assert(sizeof(SelShared) <= kFusedCRegion, "select scratch");
static_assert(kSelSamples <= kFusedCandCap, "samples live in the position array");
static_assert(3 * kMaxQRows * 4 + 16 <= kFusedCRegion, "merge scratch");

constexpr int kWposBytes = kMaxQRows * 4;
constexpr int kChunkBufBytes = 2 * kChunkKeys * 4;  // raw scores of two pass-2 chunks
constexpr int kBarBytes = 512;
static_assert((51 + 2 * kPub) * 8 <= kBarBytes, "mbarriers (the publish ring's last) fit their block");
constexpr int kMiscBytes = 256;  // TMEM address, abort flag, task
constexpr int kFixedBytes = kWposBytes + kChunkBufBytes + kBarBytes + kMiscBytes +
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
  __device__ int list(int s, int g) const { return srh_group(s, g, p.seqs_per_mask, p.num_kv_heads); }
  __device__ int rows(int s, int g) const { return __popc(p.srh_bits[list(s, g)]) * p.window; }
  __device__ int* ticket(int u) const { return p.ctr + kFusedCtrHead + u; }
  __device__ int* p2done(int u) const { return p.ctr + kFusedCtrHead + p.n_units + u; }
  __device__ int* bias_state(int u) const { return p.ctr + kFusedCtrHead + 2 * p.n_units + u; }
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
      __nanosleep(64);
      if (ld_acquire(ptr) >= target) return true;
      if (aborted() || *reinterpret_cast<volatile int*>(abort_cta)) return false;
      if (globaltimer_ns() - t0 > p.wait_ns) {
        raise_abort();
        return false;
      }
    }
  }
  // Bounded wait on one of this CTA's mbarriers; a timeout stops the call.
  __device__ bool wait_bar(uint32_t bar, uint32_t parity) const {
    if (mbar_test_wait(bar, parity)) return true;
    const bool ok = mbar_wait_bounded(bar, parity, abort_cta, p.status, p.wait_ns);
    if (!ok && !aborted()) atomicExch(p.ctr + kCtrAbort, 1);
    return ok;
  }
};

// ---------------------------------------------------------------- publishing
// The claimer thread publishes the chunks the epilogue has finished, in
// order: after the epilogue warps' arrivals (CTA-scope release/acquire) one
// GPU-scope fence covers a batch of finished chunks, then each chunk adds to
// its unit's counter (pass 1: the ticket the merge waits for; pass 2: the
// count the selection waits for).  The fence's wait for the writes thus
// stalls neither the epilogue nor the tile pipeline.
struct Publisher {
  const Fused& F;
  uint32_t full0, empty0;  // the publish ring's barriers
  int info[kPub];          // chunk i (slot i % kPub): unit * 2 + pass - 1
  int next, issued;        // first chunk not yet published; chunks issued

  __device__ uint32_t full(int i) const { return full0 + 8u * static_cast<uint32_t>(i % kPub); }
  __device__ uint32_t empty(int i) const { return empty0 + 8u * static_cast<uint32_t>(i % kPub); }
  __device__ void pump() {
    int k = next;
    while (k < issued && mbar_test_wait(full(k), static_cast<uint32_t>(k / kPub) & 1u)) ++k;
    if (k == next) return;
    fence_acq_rel_gpu();
    for (; next < k; ++next) {
      const int v = info[next % kPub];
      if (v & 1) {
        atomicAdd(F.p2done(v >> 1), kEpiWarps);
      } else {
        atomicAdd(F.ticket(v >> 1), kNwg);
      }
      mbar_arrive(empty(next));
    }
  }
  // Bounded wait on one of the CTA's mbarriers, publishing meanwhile.
  __device__ bool wait_bar(uint32_t bar, uint32_t parity) {
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
      if (mbar_try_wait(bar, parity)) return true;
      pump();
      if ((it & 63u) == 0 && !still_waiting(t0)) return false;
    }
  }
  // Bounded wait until at most `left` issued chunks are unpublished.
  __device__ bool wait_published(int left) {
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1; issued - next > left; ++it) {
      pump();
      __nanosleep(32);
      if ((it & 63u) == 0 && !still_waiting(t0)) return false;
    }
    return true;
  }
  __device__ bool still_waiting(uint64_t t0) const {
    if (F.aborted() || *reinterpret_cast<volatile int*>(F.abort_cta)) return false;
    if (globaltimer_ns() - t0 > F.p.wait_ns) {
      F.raise_abort();
      return false;
    }
    return true;
  }
};

// ---------------------------------------------------------------- claims
// The next chunk of this CTA.  Each claimer holds at most one pass-2 chunk it
// has claimed (*pending, taken with atomicAdd as soon as the previous one was
// published) and publishes it once its unit's denominators are merged (with
// the LSE given: at once); until then it claims pass-1 chunks.  Pass 1 keeps
// advancing while pass-2 chunks wait, and a pass-2 chunk never reaches the
// epilogue before its denominators.  When pass 1 is exhausted the claimer
// waits (bounded) for its pending chunk's unit, whose pass-1 chunks are then
// all claimed.  Returns false when both passes are exhausted (or aborted).
__device__ bool claim_chunk(const Fused& F, Publisher& pb, int* pending, int* pass, int* x) {
  const FusedParams& p = F.p;
  for (;;) {
    if (F.aborted() || *reinterpret_cast<volatile int*>(F.abort_cta)) return false;
    if (*pending < 0 && ld_volatile(p.ctr + kCtrPass2) < p.n_chunks) {
      const int y = atomicAdd(p.ctr + kCtrPass2, 1);
      if (y < p.n_chunks) *pending = y;
    }
    int u = -1;
    if (*pending >= 0) {
      const int s = find_seq(p.chunk_off, p.batch, *pending);
      u = s * p.num_kv_heads + (*pending - p.chunk_off[s]) / F.chunks_per_unit(s);
      if (p.given_lse || ld_acquire(F.bias_state(u)) >= 2) {
        *pass = 2;
        *x = *pending;
        *pending = -1;
        return true;
      }
    }
    if (!p.given_lse && ld_volatile(p.ctr + kCtrPass1) < p.n_chunks) {
      const int y = atomicAdd(p.ctr + kCtrPass1, 1);
      if (y < p.n_chunks) {
        *pass = 1;
        *x = y;
        return true;
      }
      continue;
    }
    if (*pending < 0) return false;  // both passes exhausted
    // pass 1 is exhausted: every pass-1 chunk of the pending chunk's unit is
    // claimed; wait (bounded) for its merge, publishing meanwhile (the merge
    // may wait for tickets this CTA holds)
    const uint64_t t0 = globaltimer_ns();
    while (ld_acquire(F.bias_state(u)) < 2) {
      pb.pump();
      __nanosleep(64);
      if (!pb.still_waiting(t0)) return false;
    }
  }
}

// ---------------------------------------------------------------- merge
// log2 D_q of unit u from its pass-1 pairs (one per chunk and warpgroup that
// takes tiles; one that got no tile of a chunk leaves (-inf, 0)), 256 worker
// threads: nm threads per query row, sixteen pairs in flight per thread.
__device__ __noinline__ void merge_unit(const Fused& F, int u, uint8_t* creg, int ct) {
  const FusedParams& p = F.p;
  const int s = u / p.num_kv_heads;
  const int g = u - s * p.num_kv_heads;
  const int N = F.rows(s, g);
  const int ncu = F.chunks_per_unit(s);
  float* s_mm = reinterpret_cast<float*>(creg);  // [256]
  float* s_mz = s_mm + kMaxQRows;                 // [256]
  if (ncu > 0 && N > 0) {
    constexpr int nwg = kNwg;
    const int nparts = nwg * ncu;  // the unit's chunks are consecutive
    const float2* parts = p.partials + static_cast<long long>(p.chunk_off[s] + g * ncu) *
                                           kFusedPartsPerChunk * p.part_stride;
    const int nm = kCThreads / N;
    const int q = ct % N;
    const int sub = ct / N;
    if (sub < nm) {
      float m = kNegInf, z = 0.f;
      for (int i0 = sub; i0 < nparts; i0 += 16 * nm) {
        float2 pr[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const int i = i0 + k * nm;  // pair i: chunk i / nwg, warpgroup i % nwg
          pr[k] = i < nparts
                      ? __ldcg(parts + (static_cast<long long>(i / nwg) * kFusedPartsPerChunk +
                                        i % nwg) * p.part_stride + q)
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
      p.bias[static_cast<long long>(u) * p.part_stride + ct] = m + __log2f(z);
    }
  }
  fence_acq_rel_gpu();
  cbar();
  if (ct == 0) atomicExch(F.bias_state(u), 2);
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
    constexpr int kB = 8;  // keys per thread loaded before they are counted
#pragma unroll 1
    for (int i0 = 0; i0 < iters; i0 += kB) {
      uint32_t kv[kB];
#pragma unroll
      for (int q = 0; q < kB; ++q) {
        const int j = ((i0 + q) << 8) + ct;
        kv[q] = j < count ? key_at(j) : 0u;
      }
#pragma unroll
      for (int q = 0; q < kB; ++q) {
        const int j = ((i0 + q) << 8) + ct;
        const uint32_t key = kv[q];
        const bool m = j < count && (key & pmask) == prefix;
        const uint32_t act = __ballot_sync(0xffffffffu, m);
        if (!act) continue;
        const uint32_t bin = (key >> shf) & fm;
        const int leader = __ffs(act) - 1;
        const uint32_t lb = __shfl_sync(0xffffffffu, bin, leader);
        if (__all_sync(0xffffffffu, !m || bin == lb)) {
          if (lane == leader) atomicAdd(&hh[lb], static_cast<uint32_t>(__popc(act)));
        } else if (m) {
          // one add per distinct bin of the warp (no same-address serialisation)
          const uint32_t same = __match_any_sync(act, bin);
          if (lane == __ffs(same) - 1) atomicAdd(&hh[bin], static_cast<uint32_t>(__popc(same)));
        }
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
  uint32_t next = ct < count ? key_at(ct) : 0u;  // one block of keys loaded ahead
  for (int j0 = 0; j0 < count; j0 += kCThreads) {
    const int j = j0 + ct;
    const bool in = j < count;
    const uint32_t key = next;
    if (j + kCThreads < count) next = key_at(j + kCThreads);
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
// loads in flight per thread: a batch's positions are loaded first, then its
// rows, and a position outside the sequence (never, for a correct selection)
// is skipped and recorded after the batch, so no load waits behind another.
__device__ __noinline__ void gather_rows(const FusedParams& p, int seq0, int L, int g,
                                         const int32_t* out, int out0, int count, int ct) {
  constexpr int kChunks = 2 * kHeadDim * 2 / 16;  // 16 K + 16 V chunks per token
  constexpr int kBatch = 8;
  const int total = count * kChunks;
  bool bad = false;
  for (int base = 0; base < total; base += kBatch * kCThreads) {
    int tok[kBatch];
#pragma unroll
    for (int k = 0; k < kBatch; ++k) {
      const int e = base + k * kCThreads + ct;
      tok[k] = e < total ? out[e / kChunks] : 0;
    }
    uint4 v[kBatch];
    long long dst[kBatch];
    bool is_v[kBatch];
#pragma unroll
    for (int k = 0; k < kBatch; ++k) {
      const int e = base + k * kCThreads + ct;
      const int i = e / kChunks;
      const int ch = e - i * kChunks;
      const bool ok = e < total && tok[k] >= 0 && tok[k] < L;
      bad |= e < total && !ok;
      is_v[k] = ch >= kChunks / 2;
      const int part = ch & (kChunks / 2 - 1);
      const long long src = static_cast<long long>(seq0 + (ok ? tok[k] : 0)) * p.tok_stride_v16 +
                            static_cast<long long>(g) * p.head_stride_v16 + part;
      dst[k] = ok ? (static_cast<long long>(out0 + i) * p.num_kv_heads + g) * (kHeadDim * 2 / 16) +
                        part
                  : -1;
      if (ok) v[k] = __ldg((is_v[k] ? p.v : p.k) + src);
    }
#pragma unroll
    for (int k = 0; k < kBatch; ++k)
      if (dst[k] >= 0) (is_v[k] ? p.v_out : p.k_out)[dst[k]] = v[k];
  }
  if (bad) atomicCAS(p.status, 0, CKV_DEV_ERR_INDEX);
}

// Pooled score of prefix key j from the raw scores (zeros outside [0, n)),
// summed in the order the epilogue's chunk pooling uses.
__device__ __forceinline__ float pool_from_global(const float* raw, int n, int j, int h,
                                                  float fP) {
  float acc = 0.f;
  for (int t = 0; t <= 2 * h; ++t) {
    const int jj = j - h + t;
    acc += (jj >= 0 && jj < n) ? __ldcg(raw + jj) : 0.f;
  }
  return acc / fP;
}

// Selection of unit u.  First the pooled scores within h of a chunk edge
// (the epilogue pooled each chunk's interior), then the top-k by a sampled
// lower bound: candidates in position order, an exact radix search among
// them (among all the unit's scores when the bound keeps too few or too
// many), the window, and the K/V rows.  Pooled scores are >= 0: their bit
// patterns order like their values.
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
  const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
  float* pooled = p.pooled + soff;
  const int h = (p.pool_width - 1) >> 1;
  const float fP = static_cast<float>(p.pool_width);
  // chunk-edge pooled scores: [a, a + h) and [b - h, b) of every chunk
  if (h > 0 && n > 0) {
    const float* raw = p.raw + soff;
    const int nct = (n + kChunkKeys - 1) / kChunkKeys;
    for (int e = ct; e < nct * 2 * h; e += kCThreads) {
      const int c = e / (2 * h);
      const int o = e - c * 2 * h;
      const int a = c * kChunkKeys;
      const int b = min(a + kChunkKeys, n);
      const int lo_end = min(a + h, b);
      const int hi_start = max(b - h, lo_end);
      const int j = o < h ? a + o : hi_start + (o - h);
      if (o < h ? j < lo_end : j < b) pooled[j] = pool_from_global(raw, n, j, h, fP);
    }
    __threadfence();
  }
  cbar();
  if (!p.do_select) return;
  int32_t* out = p.indices + static_cast<long long>(g) * p.o_total + out0;
  if (kept >= L) {  // keep everything
    for (int i = ct; i < L; i += kCThreads) out[i] = i;
    __threadfence_block();
    cbar();
    gather_rows(p, seq0, L, g, out, out0, L, ct);
    return;
  }
  const int k = kept - W;  // 0 <= k < n
  for (int w = ct; w < W; w += kCThreads) out[k + w] = n + w;
  if (k == 0) {
    __threadfence_block();
    cbar();
    gather_rows(p, seq0, L, g, out, out0, W, ct);
    return;
  }
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(pooled);
  // threshold lo: the rs-th largest of ns samples spread over the unit,
  // chosen so that the keys >= lo are at least k and at most the shared
  // candidate capacity; the samples sit in the (not yet used) position array
  uint32_t* samp = reinterpret_cast<uint32_t*>(sh.pos);
  const int ns = min(kSelSamples, n);
  for (int i = ct; i < ns; i += kCThreads)
    samp[i] = __ldcg(keys + static_cast<int>((static_cast<long long>(i) * n) / ns));
  radix_init_grp(sh.rs, ct);
  cbar();
  int pc = 0, need_eq = 0;
  const float mu = static_cast<float>(k) * static_cast<float>(ns) / static_cast<float>(n);
  int rs = min(ns, static_cast<int>(ceilf(mu + 3.f * sqrtf(mu))) + 2);
  uint32_t lo = 0, lo_ge = 0;
  int total = 0, tot_ge = -1;
  constexpr int kU = 8;  // loads in flight per lane
  const int seg = ((n + 8 * 32 * kU - 1) / (8 * 32 * kU)) * 32 * kU;  // positions per warp
  const int wlo = min(n, cw * seg);
  const int whi = min(n, wlo + seg);
  bool fast = false;
  for (int attempt = 0; attempt < 2; ++attempt) {
    // (same sample set every attempt: the radix's OR/AND of slot 0 stay valid)
    lo = grp_kth_largest(samp, ns, 0u, 0xFFFFFFFFu, rs, sh.rs, 0, pc, &need_eq, ct, false);
    int wc = 0;
    for (int b0 = wlo; b0 < whi; b0 += 32 * kU) {
      uint32_t kv[kU];
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        const int i = b0 + q * 32 + lane;
        kv[q] = i < whi ? __ldcg(keys + i) : 0u;
      }
#pragma unroll
      for (int q = 0; q < kU; ++q)
        wc += __popc(__ballot_sync(0xffffffffu, b0 + q * 32 + lane < whi && kv[q] >= lo));
    }
    if (lane == 0) sh.wcnt[cw] = wc;
    cbar();
    total = 0;
    for (int w = 0; w < 8; ++w) total += sh.wcnt[w];
    if (total >= k && (tot_ge < 0 || total < tot_ge)) {
      lo_ge = lo;
      tot_ge = total;
      if (ct < 8) sh.wcnt_ge[ct] = sh.wcnt[ct];
    }
    if (total >= k && total <= kFusedCandCap) {
      fast = true;
      break;
    }
    // aim at the middle of [k, capacity] from the density this attempt saw
    const float per = static_cast<float>(max(total, 1)) / static_cast<float>(rs);
    int want = static_cast<int>(ceilf(0.5f * static_cast<float>(k + kFusedCandCap) / per));
    want = total < k ? max(want, rs + 1) : min(want, rs - 1);
    if (want < 1 || want > ns || want == rs) break;
    rs = want;
    cbar();  // every thread has read the counts
  }
  // the candidates' radix starts afresh
  radix_init_grp(sh.rs, ct);
  pc = 0;
  need_eq = 0;
  cbar();
  // The candidates (keys >= lo) in position order: in shared memory when at
  // most kFusedCandCap, else -- when the raw scores are workspace the select
  // no longer reads (the chunk edges above were its last use) -- in the
  // unit's raw-score row, keys in its first half and positions in its second.
  uint32_t* ckey = sh.key;
  int* cpos = sh.pos;
  bool cglob = false;
  if (!fast && p.raw_scratch && tot_ge >= k && tot_ge <= n / 2) {
    lo = lo_ge;
    total = tot_ge;
    ckey = reinterpret_cast<uint32_t*>(p.raw + soff);
    cpos = reinterpret_cast<int*>(ckey + n / 2);
    cglob = true;
    if (ct < 8) sh.wcnt[ct] = sh.wcnt_ge[ct];
    cbar();
    fast = true;
  }
  uint32_t tau;
  if (fast) {
    int o = 0;
    for (int w = 0; w < cw; ++w) o += sh.wcnt[w];
    for (int b0 = wlo; b0 < whi; b0 += 32 * kU) {
      uint32_t kv[kU];
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        const int i = b0 + q * 32 + lane;
        kv[q] = i < whi ? __ldcg(keys + i) : 0u;
      }
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        const int i = b0 + q * 32 + lane;
        const bool c = i < whi && kv[q] >= lo;
        const uint32_t mm = __ballot_sync(0xffffffffu, c);
        const int slot = o + __popc(mm & lanemask_lt(lane));
        if (c && slot < total) {
          ckey[slot] = kv[q];
          cpos[slot] = i;
        } else if (c) {  // more keys above lo than counted: cannot happen; record
          atomicCAS(p.status, 0, CKV_DEV_ERR_INDEX);
        }
        o += __popc(mm);
      }
    }
    if (cglob) __threadfence_block();
    cbar();
    constexpr uint32_t kClamp = 0xFFFFu;
    const uint32_t td = grp_kth_largest(ckey, total, lo, kClamp, k, sh.rs, 0, pc, &need_eq, ct,
                                        cglob);
    tau = lo + td;
    if (td == kClamp)
      tau = grp_kth_largest(ckey, total, 0u, 0xFFFFFFFFu, k, sh.rs, 1, pc, &need_eq, ct, cglob);
    if (cglob) {
      emit_selected(total, tau, need_eq, out, k, sh, ct, [&](int j) { return __ldcg(ckey + j); },
                    [&](int j) { return __ldcg(cpos + j); });
    } else {
      emit_selected(total, tau, need_eq, out, k, sh, ct, [&](int j) { return ckey[j]; },
                    [&](int j) { return cpos[j]; });
    }
  } else {
    tau = grp_kth_largest(keys, n, 0u, 0xFFFFFFFFu, k, sh.rs, 1, pc, &need_eq, ct, true);
    emit_selected(n, tau, need_eq, out, k, sh, ct, [&](int j) { return __ldcg(keys + j); },
                  [&](int j) { return j; });
  }
  __threadfence_block();
  cbar();  // the indices written above are read back by the copy
  gather_rows(p, seq0, L, g, out, out0, kept, ct);
}

// The workers' next task (one thread): the next unit to select once all its
// pass-2 chunks are in, else the next unit to merge once all its pass-1
// chunks are in; waits (bounded) while neither is ready.
__device__ void claim_task(const Fused& F, int* task) {
  const FusedParams& p = F.p;
  uint64_t t0 = 0;
  for (;;) {
    if (F.aborted() || *reinterpret_cast<volatile int*>(F.abort_cta)) break;
    const int u = ld_volatile(p.ctr + kCtrSel);
    if (u >= p.n_units) break;  // every unit selected (and therefore merged)
    const int s = u / p.num_kv_heads;
    if (ld_acquire(F.p2done(u)) >= kEpiWarps * F.chunks_per_unit(s)) {  // kEpiWarps per pass-2 chunk
      if (atomicCAS(p.ctr + kCtrSel, u, u + 1) == u) {
        task[0] = kTaskSelect;
        task[1] = u;
        return;
      }
      continue;
    }
    if (!p.given_lse) {
      const int m = ld_volatile(p.ctr + kCtrMerge);
      if (m < p.n_units &&
          ld_acquire(F.ticket(m)) >= p.nwg * F.chunks_per_unit(m / p.num_kv_heads)) {
        if (atomicCAS(p.ctr + kCtrMerge, m, m + 1) == m) {
          task[0] = kTaskMerge;
          task[1] = m;
          return;
        }
        continue;
      }
    }
    const uint64_t now = globaltimer_ns();
    if (t0 == 0) {
      t0 = now;
    } else if (now - t0 > p.wait_ns) {
      F.raise_abort();
      break;
    }
    __nanosleep(128);
  }
  task[0] = kTaskEnd;
  task[1] = 0;
}

// Pass 1, rare: an exponent of this 32-column group passed 2^64 (or the
// references are still -inf): raise every query's R to kShift below its
// largest scaled logit among the warp's 32 keys, shrink the sums kept against
// the old R, and return this group's column sums against the new R (column
// lane).  The whole warp calls it; taddr is the group's first TMEM column.
__device__ __noinline__ float p1_raise_group(uint32_t taddr, float* rf, float* acc_c,
                                             const int* wpos, int lim, bool edge, bool key,
                                             int vis, float c, int lane) {
  uint32_t r[32];
  tmem_load32_async(taddr, r);
  tmem_wait_ld(r);
  uint32_t valid = 0u;
  float v[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const bool ok = j < lim && (!edge || (key && wpos[j] >= -vis));
    valid |= (ok ? 1u : 0u) << j;
    v[j] = ok ? __uint_as_float(r[j]) * c : kNegInf;
  }
  const float m = warp_transpose_max32(v, lane);  // column lane
  const float old = rf[lane];
  const float nw = fmaxf(old, m - kShift);
  acc_c[lane] *= (nw == old) ? 1.f : ((old == kNegInf) ? 0.f : ex2_approx(old - nw));
  __syncwarp();
  rf[lane] = nw;
  __syncwarp();
#pragma unroll
  for (int j = 0; j < 32; ++j)
    v[j] = ((valid >> j) & 1u) ? ex2_approx(fmaf(__uint_as_float(r[j]), c, -rf[j])) : 0.f;
  return warp_transpose_sum32(v, lane);
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
  const int rstride = p.row_stride;
  uint8_t* sK = base;
  const int nqb = p.q_bufs;
  uint8_t* sQ = base + nst * kTileBytes;  // nqb buffers of two 64-column halves
  const int nrow = 4 * kNwg;  // epilogue warps that take tiles
  float* sRef = reinterpret_cast<float*>(sQ + 2 * nqb * qh);  // [nrow][rstride]
  float* sAcc = sRef + nrow * rstride;                        // [nrow][rstride]
  int* sWpos = reinterpret_cast<int*>(sAcc + nrow * rstride);
  float* sChunk = reinterpret_cast<float*>(sWpos + kMaxQRows);  // [2][kChunkKeys]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sChunk + 2 * kChunkKeys);
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
  auto qempty = [&](int i) { return bar0 + 8u * (43 + i); };    // Q buffer's MMAs done
  auto wgbar = [&](int w) { return bar0 + 8u * (46 + w); };     // epilogue warpgroup sync
  const uint32_t epibar = bar0 + 8u * 50;                       // all epilogue warps
  auto pubfull = [&](int i) { return bar0 + 8u * (51 + i); };   // chunk's results written
  auto pubempty = [&](int i) { return bar0 + 8u * (51 + kPub + i); };  // chunk published

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
      mbar_init(dempty(i), 3 + kEpiWarps);  // TMA producer, both MMA warps, epilogue warps
    }
    for (int i = 0; i < 3; ++i) {
      mbar_init(qfull(i), 1);
      mbar_init(qempty(i), 2);  // one commit from each MMA warp
    }
    for (int i = 0; i < 4; ++i) mbar_init(wgbar(i), 4);
    mbar_init(epibar, kEpiWarps);
    for (int i = 0; i < kPub; ++i) {
      mbar_init(pubfull(i), kEpiWarps);
      mbar_init(pubempty(i), 1);
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

  if (warp == kClaimWarp) {
    // ------------------------------------------------------------ chunk claims
    if (lane == 0) {
      Publisher pb{F, pubfull(0), pubempty(0), {}, 0, 0};
      int pending = -1;  // pass-2 chunk claimed, not yet published
      // test hook: a wait that cannot complete, before anything is issued;
      // it runs out after p.wait_ns and stops the call
      if (p.stall && blockIdx.x == 0) F.wait_counter(p.ctr + kCtrNever, 1);
      for (int c = 0;; ++c) {
        const int ds = c % kDescs;
        if (!pb.wait_bar(dempty(ds), ((c / kDescs) & 1) ^ 1)) break;
        ChunkDesc d;
        d.end = 1;
        int pass = 0, x = 0;
        if (claim_chunk(F, pb, &pending, &pass, &x)) {
          const int s = find_seq(p.chunk_off, p.batch, x);
          const int ncu = F.chunks_per_unit(s);
          const int local = x - p.chunk_off[s];
          const int g = local / ncu;
          const int cc = local - g * ncu;
          d.end = 0;
          d.pass = pass;
          d.s = s;
          d.g = g;
          d.t0 = cc * kChunkTiles;
          d.t1 = min(F.tiles(s), d.t0 + kChunkTiles);
          d.chunk = x;
          d.n_rows = F.rows(s, g);
          if (!pb.wait_published(kPub - 1)) break;  // a free slot in the publish ring
          pb.info[pb.issued % kPub] = (s * Hkv + g) * 2 + (pass - 1);
          ++pb.issued;
        }
        descs[ds] = d;
        mbar_arrive(dfull(ds));
        if (d.end) break;
      }
      pb.wait_published(0);  // every chunk this CTA processed
    }
    __syncwarp();
  } else if (warp == kProdWarp) {
    // ------------------------------------------------------------ TMA
    if (lane == 0) {
      // Pass 1 runs further ahead of pass 2 than L2 holds, so K marked
      // evict-last everywhere would evict itself in order and pass 2 would
      // miss all of it; marking a fixed 15% of its lines evict-last (the rest
      // evict-first) keeps that share in L2 until pass 2 reads it (measured:
      // 0.10-0.25 best, 2-3% faster than all evict-last, 4% slower with
      // none).  Pass 2 reads K for the last time; the query rows are reused
      // by every chunk of their unit.
      uint64_t pol1;
      asm volatile("createpolicy.fractional.L2::evict_last.L2::evict_first.b64 %0, 0.15;"
                   : "=l"(pol1));
      const uint64_t pol2 = l2_policy_evict_first();
      const uint64_t polq = l2_policy_evict_last();
      const int G = p.group_size;
      // Each UMMA warp has its own sub-ring of the K stages (warp w: stages
      // w, w + 2, ...), consumed strictly in order: a warp that skipped the
      // other warp's tiles could otherwise wait on a stage whose previous
      // fill has not landed and mistake an older phase for its own.
      const int nsw = nst >> 1;
      int sw0 = 0, sw1 = 0;       // next slot of each sub-ring
      uint32_t sp0 = 0, sp1 = 0;  // and its phase
      uint32_t k_used = 0, k_phase = 0;  // per stage: filled, parity of its last fill
      int qb = 0;  // Q buffer of the next chunk and its phase
      uint32_t qph = 0;
      uint32_t q_issued = 0, q_phase = 0;  // per Q buffer: loads issued, phase of the last
      for (int c = 0;; ++c) {
        const int ds = c % kDescs;
        if (!F.wait_bar(dfull(ds), static_cast<uint32_t>(c / kDescs) & 1u)) break;
        const ChunkDesc d = descs[ds];
        mbar_arrive(dempty(ds));
        if (d.end) break;
        const uint64_t pol = d.pass == 1 ? pol1 : pol2;
        const int row0 = p.cu_seqlens[d.s];
        // the chunk's query rows: head block hi of the buffer holds the W
        // window rows of the group's hi-th SRH head
        if (!F.wait_bar(qempty(qb), qph ^ 1u)) break;
        {
          uint32_t bits = p.srh_bits[F.list(d.s, d.g)];
          mbar_arrive_expect_tx(qfull(qb), static_cast<uint32_t>(d.n_rows) * (kHeadDim * 2));
          const uint32_t qdst = smem_u32(sQ + qb * 2 * qh);
          for (int hi = 0; bits != 0u; ++hi, bits &= bits - 1u) {
            const int head = d.g * G + (__ffs(bits) - 1);
            const uint32_t dst = qdst + static_cast<uint32_t>(hi * W * 128);
            tma_load_4d(dst, &p.tmap_q, qfull(qb), 0, 0, head, d.s, polq);
            tma_load_4d(dst + qh, &p.tmap_q, qfull(qb), 64, 0, head, d.s, polq);
          }
          q_issued |= 1u << qb;
          q_phase = (q_phase & ~(1u << qb)) | (qph << qb);
          if (++qb == nqb) {
            qb = 0;
            qph ^= 1u;
          }
        }
        bool stop = false;
        for (int t = d.t0; t < d.t1; ++t) {
          const int w = (t - d.t0) & 1;  // the UMMA warp (and warpgroup) of the tile
          const int st = w + 2 * (w ? sw1 : sw0);
          const uint32_t ph = w ? sp1 : sp0;
          if (!F.wait_bar(empty(st), ph ^ 1u)) {
            stop = true;
            break;
          }
          mbar_arrive_expect_tx(full(st), kTileBytes);
          const uint32_t dst = smem_u32(sK + st * kTileBytes);
          const int row = row0 + t * kTileTokens;
          tma_load_3d(dst, &p.tmap_k, full(st), 0, d.g, row, pol);
          tma_load_3d(dst + kHalfTileBytes, &p.tmap_k, full(st), 64, d.g, row, pol);
          k_used |= 1u << st;
          k_phase = (k_phase & ~(1u << st)) | (ph << st);
          if (w) {
            if (++sw1 == nsw) {
              sw1 = 0;
              sp1 ^= 1u;
            }
          } else if (++sw0 == nsw) {
            sw0 = 0;
            sp0 ^= 1u;
          }
        }
        if (stop) break;
      }
      if (*reinterpret_cast<volatile int*>(abort_cta)) {
        // let the copies already issued land before the CTA can exit
        for (int i = 0; i < nst; ++i)
          if ((k_used >> i) & 1u) wait_plain(full(i), (k_phase >> i) & 1u, 100000000ull);
        for (int b = 0; b < nqb; ++b)
          if ((q_issued >> b) & 1u) wait_plain(qfull(b), (q_phase >> b) & 1u, 100000000ull);
      }
      // Tail: the UMMA warps release a stage (empty) and a Q buffer (qempty)
      // with tcgen05.commit arrivals that nobody else waits for at the end;
      // wait for the last ones, so that no asynchronous arrival can land in
      // this CTA's shared memory after it exits (bounded: after an abort some
      // never come).
      const uint64_t tail_ns = *reinterpret_cast<volatile int*>(abort_cta) ? 100000000ull
                                                                           : p.wait_ns;
      for (int i = 0; i < nst; ++i)
        if ((k_used >> i) & 1u) wait_plain(empty(i), (k_phase >> i) & 1u, tail_ns);
      for (int b = 0; b < nqb; ++b)
        if ((q_issued >> b) & 1u) wait_plain(qempty(b), (q_phase >> b) & 1u, tail_ns);
    }
    __syncwarp();
  } else if (warp == kMmaWarp || warp == kMmaWarp2) {
    // ------------------------------------------------------------ UMMA issue
    const int mw = warp == kMmaWarp ? 0 : 1;  // the warpgroup whose tiles this warp issues
    if (lane == 0) {
      const uint64_t dk0 = smem_desc_sw128(smem_u32(sK));
      const int bpw = p.nbuf / kNwg;  // TMEM buffers per warpgroup (a power of two)
      const int lbpw = __ffs(bpw) - 1;
      const int nsw = nst >> 1;
      int st = 0;  // next slot of this warp's K sub-ring (stages mw, mw + 2, ...) and its phase
      uint32_t sph = 0;
      int qb = 0;  // Q buffer of the next chunk and its phase
      uint32_t qph = 0;
      int kw = 0;  // tiles issued for warpgroup mw
      int last_b = -1;
      uint32_t last_use = 0;
      for (int c = 0;; ++c) {
        const int ds = c % kDescs;
        if (!F.wait_bar(dfull(ds), static_cast<uint32_t>(c / kDescs) & 1u)) break;
        const ChunkDesc d = descs[ds];
        mbar_arrive(dempty(ds));
        if (d.end) break;
        if (!F.wait_bar(qfull(qb), qph)) break;
        tc_fence_after();
        const int Npad = (d.n_rows + 15) & ~15;
        const uint32_t idesc = umma_idesc_f16(kTileTokens, Npad, p.is_bf16 != 0);
        const uint64_t dq0 = smem_desc_sw128(smem_u32(sQ + qb * 2 * qh));
        bool stop = false;
        for (int t = d.t0; t < d.t1; ++t) {
          if (((t - d.t0) & 1) != mw) continue;  // the other warp's tile
          const int kk = kw++;
          const int b = mw + kNwg * (kk & (bpw - 1));
          const uint32_t use = static_cast<uint32_t>(kk >> lbpw) & 1u;
          if (!F.wait_bar(tempty(b), use ^ 1u)) {
            stop = true;
            break;
          }
          const int stp = mw + 2 * st;  // the stage
          if (!F.wait_bar(full(stp), sph)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tbase + static_cast<uint32_t>(b * p.tstride);
          const uint64_t dk = dk0 + static_cast<uint64_t>((stp * kTileBytes) >> 4);
#pragma unroll
          for (int k8 = 0; k8 < kHeadDim / 16; ++k8) {
            const uint32_t koff = (k8 >> 2) * kHalfTileBytes + (k8 & 3) * 32;
            const uint32_t qoff = (k8 >> 2) * qh + (k8 & 3) * 32;
            umma_f16(dt, dk + (koff >> 4), dq0 + (qoff >> 4), idesc, k8 > 0 ? 1u : 0u);
          }
          umma_commit(empty(stp));
          umma_commit(tfull(b));
          last_b = b;
          last_use = use;
          if (++st == nsw) {
            st = 0;
            sph ^= 1u;
          }
        }
        if (stop) break;
        umma_commit(qempty(qb));
        if (++qb == nqb) {
          qb = 0;
          qph ^= 1u;
        }
      }
      if (*reinterpret_cast<volatile int*>(abort_cta) && last_b >= 0)
        wait_plain(tfull(last_b), last_use, 100000000ull);  // MMAs done before TMEM is freed
    }
    __syncwarp();
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - kEpiWarp0;
    const int wg = ew >> 2;
    const int qd = warp & 3;  // TMEM lane quarter of this warp
    const int tw = (ew & 3) * 32 + lane;
    const int te = ew * 32 + lane;  // thread among all epilogue threads
    constexpr int nwg = kNwg;
    const bool takes = wg < nwg;  // this warpgroup takes tiles
    float* ref = sRef + (takes ? ew : 0) * rstride;
    float* acc_s = sAcc + (takes ? ew : 0) * rstride;
    const float c = p.c;
    const int bpw = p.nbuf / nwg;  // a power of two
    const int lbpw = __ffs(bpw) - 1;
    const int h = (p.pool_width - 1) >> 1;
    const float fP = static_cast<float>(p.pool_width);
    const int G = p.group_size;
    int kc = 0;       // tiles this warpgroup has taken
    int nsync = 0;    // warpgroup syncs so far (mbarrier phase)
    int nsync8 = 0;   // all-epilogue syncs so far
    int n2 = 0;       // pass-2 chunks so far (raw buffer parity)
    bool stop = false;
    // bounded barriers (a warp that stopped cannot hang the others)
    auto epi_sync = [&]() -> bool {
      __syncwarp();
      if (lane == 0) mbar_arrive(epibar);
      const bool ok = F.wait_bar(epibar, static_cast<uint32_t>(nsync8) & 1u);
      ++nsync8;
      return __all_sync(0xffffffffu, ok);
    };
    // the chunk's results are written: its claimer publishes it (fence, then
    // the unit's counter) off the epilogue's path
    auto publish = [&](int ci) -> bool {
      const int k = ci % kPub;
      bool ok = true;
      if (ci >= kPub && lane == 0) ok = F.wait_bar(pubempty(k), static_cast<uint32_t>(ci / kPub - 1) & 1u);
      __syncwarp();
      if (lane == 0 && ok) mbar_arrive(pubfull(k));
      return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    };
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
      const int L = F.len(s);
      const int n = L - W;
      const int u = s * Hkv + g;
      const long long soff = static_cast<long long>(g) * p.p_total + p.cu_prefix[s];
      if (d.pass == 1) {
        // ---------------------------------------- pass 1: softmax statistics
        // Per query row q the warp keeps a reference R_q and sums
        // 2^(z c - R_q) over its keys, reduced across the lanes every tile.
        if (!takes) continue;  // warpgroups beyond nwg take no first-pass work
        for (int q = lane; q < N; q += 32) {
          ref[q] = kNegInf;
          acc_s[q] = 0.f;
        }
        __syncwarp();
        bool first = true;  // no tile of this chunk accumulated yet
        for (int tile = d.t0 + wg; tile < d.t1; tile += nwg) {
          const int kk = kc++;
          const int b = wg + nwg * (kk & (bpw - 1));
          const uint32_t use = static_cast<uint32_t>(kk >> lbpw) & 1u;
          const bool ok = F.wait_bar(tfull(b), use);
          if (!__all_sync(0xffffffffu, ok)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const int tok = tile * kTileTokens + qd * 32 + lane;
          const uint32_t taddr = tbase + (static_cast<uint32_t>(qd * 32) << 16) +
                                 static_cast<uint32_t>(b * p.tstride);
          const bool edge = (tile + 1) * kTileTokens > n;
          const int vis = n - tok;
          const bool key = tok < L;
          for (int c0 = 0; c0 < N; c0 += 32) {
            uint32_t r[32];  // the logits
            tmem_load32_async(taddr + c0, r);
            tmem_wait_ld(r);
            const int lim = min(32, N - c0);
            const bool masked = edge || lim < 32;
            float* rf = ref + c0;
            float e[32];  // 2^(z c - R)
            if (first && !masked) {
              // the warp's first tile of the chunk: lane 0's scaled logit is
              // the reference of each query row (any reference within 2^64
              // of the largest keeps the fp32 sums exact enough)
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const float v = __uint_as_float(r[j]) * c;
                const float rj = __shfl_sync(0xffffffffu, v, 0);
                e[j] = ex2_approx(v - rj);
                if (lane == 0) rf[j] = rj;
              }
              __syncwarp();
            } else if (masked) {
#pragma unroll
              for (int j = 0; j < 32; j += 4) {
                const int4 wq = *reinterpret_cast<const int4*>(sWpos + c0 + j);
                const float4 rq = *reinterpret_cast<const float4*>(rf + j);
                const int wv[4] = {wq.x, wq.y, wq.z, wq.w};
                const float rv[4] = {rq.x, rq.y, rq.z, rq.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const bool okk = (j + k) < lim && (!edge || (key && wv[k] >= -vis));
                  e[j + k] = okk ? ex2_approx(fmaf(__uint_as_float(r[j + k]), c, -rv[k])) : 0.f;
                }
              }
            } else {
#pragma unroll
              for (int j = 0; j < 32; j += 4) {
                const float4 rq = *reinterpret_cast<const float4*>(rf + j);
                e[j + 0] = ex2_approx(fmaf(__uint_as_float(r[j + 0]), c, -rq.x));
                e[j + 1] = ex2_approx(fmaf(__uint_as_float(r[j + 1]), c, -rq.y));
                e[j + 2] = ex2_approx(fmaf(__uint_as_float(r[j + 2]), c, -rq.z));
                e[j + 3] = ex2_approx(fmaf(__uint_as_float(r[j + 3]), c, -rq.w));
              }
            }
            float colsum = warp_transpose_sum32(e, lane);  // column c0 + lane
            // an exponent above 2^64 shows in its column's sum (inf/NaN
            // when above 2^128 or with the references still -inf)
            if (__any_sync(0xffffffffu, !(colsum <= kRaiseSum)))
              colsum = p1_raise_group(taddr + c0, rf, acc_s + c0, sWpos + c0, lim, edge, key, vis,
                                      c, lane);
            acc_s[c0 + lane] += colsum;
            __syncwarp();
          }
          first = false;
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(tempty(b));
        }
        if (stop) break;
        // the warpgroup's (M, S) pairs for this chunk, then its ticket
        if (!wg_sync()) break;
        float2* part = p.partials +
                       (static_cast<long long>(d.chunk) * kFusedPartsPerChunk + wg) * p.part_stride;
        for (int q = tw; q < N; q += 128) {
          float m = kNegInf;
          for (int w = 0; w < 4; ++w) m = fmaxf(m, sRef[(wg * 4 + w) * rstride + q]);
          float z = 0.f;
          for (int w = 0; w < 4; ++w) {
            const float rw = sRef[(wg * 4 + w) * rstride + q];
            if (rw != kNegInf) z += sAcc[(wg * 4 + w) * rstride + q] * ex2_approx(rw - m);
          }
          part[q] = make_float2(m, z);
        }
        if (!wg_sync()) break;  // every row read (the next chunk reuses them)
        if (!publish(ci)) break;
      } else {
        // ---------------------------------------- pass 2: raw scores
        // log2 D_q of every query row into this warp's row of sRef
        if (p.given_lse) {
          const uint32_t bits = p.srh_bits[F.list(s, g)];
          for (int q = lane; q < N; q += 32) {
            const int hi = q / W;
            const int w = q - hi * W;
            const int head = g * G + nth_bit(bits, hi);
            ref[q] = p.lse[static_cast<long long>(s) * p.lse_bs +
                           static_cast<long long>(head) * p.lse_hs + w] *
                     1.4426950408889634f;
          }
        } else {
          // published only after its claimer saw the unit's denominators
          // merged (acquire), before the descriptor barrier
          const float* bias = p.bias + static_cast<long long>(u) * p.part_stride;
          for (int q = lane; q < N; q += 32) ref[q] = __ldcg(bias + q);
        }
        __syncwarp();
        float* cbuf = sChunk + (n2 & 1) * kChunkKeys;
        ++n2;
        const int a = d.t0 * kTileTokens;  // first key of the chunk
        for (int tile = d.t0 + wg; takes && tile < d.t1; tile += nwg) {
          const int kk = kc++;
          const int b = wg + nwg * (kk & (bpw - 1));
          const uint32_t use = static_cast<uint32_t>(kk >> lbpw) & 1u;
          const bool ok = F.wait_bar(tfull(b), use);
          if (!__all_sync(0xffffffffu, ok)) {
            stop = true;
            break;
          }
          tc_fence_after();
          const int tok = tile * kTileTokens + qd * 32 + lane;
          const uint32_t taddr = tbase + (static_cast<uint32_t>(qd * 32) << 16) +
                                 static_cast<uint32_t>(b * p.tstride);
          const bool edge = (tile + 1) * kTileTokens > n;
          const int vis = n - tok;
          const bool key = tok < L;
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
          // add 2^(z c - log2 D_q) of 32 columns starting at c0 (lim valid)
          auto add_group = [&](const uint32_t (&r)[32], int c0, int lim) {
            if (edge || lim < 32) {
#pragma unroll
              for (int j = 0; j < 32; j += 4) {
                const int4 wq = *reinterpret_cast<const int4*>(sWpos + c0 + j);
                const float4 lq = *reinterpret_cast<const float4*>(ref + c0 + j);
                const int wv[4] = {wq.x, wq.y, wq.z, wq.w};
                const float lv[4] = {lq.x, lq.y, lq.z, lq.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const bool okk = (j + k) < lim && (!edge || (key && wv[k] >= -vis));
                  acc[k] += okk ? ex2_approx(fmaf(__uint_as_float(r[j + k]), c, -lv[k])) : 0.f;
                }
              }
            } else {
#pragma unroll
              for (int j = 0; j < 32; j += 4) {
                const float4 lq = *reinterpret_cast<const float4*>(ref + c0 + j);
                acc[0] += ex2_approx(fmaf(__uint_as_float(r[j + 0]), c, -lq.x));
                acc[1] += ex2_approx(fmaf(__uint_as_float(r[j + 1]), c, -lq.y));
                acc[2] += ex2_approx(fmaf(__uint_as_float(r[j + 2]), c, -lq.z));
                acc[3] += ex2_approx(fmaf(__uint_as_float(r[j + 3]), c, -lq.w));
              }
            }
          };
          for (int c0 = 0; c0 < N; c0 += 32) {
            uint32_t r0[32];
            tmem_load32_async(taddr + c0, r0);
            tmem_wait_ld(r0);
            add_group(r0, c0, min(32, N - c0));
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(tempty(b));
          if (tok < n) {
            const float rv = (acc[0] + acc[1]) + (acc[2] + acc[3]);
            p.raw[soff + tok] = rv;
            cbuf[tok - a] = rv;
          }
        }
        if (stop) break;
        // pooled scores of the chunk's interior [a + h, b - h) from the raw
        // scores of both warpgroups; the select pools the h keys at each edge
        if (!epi_sync()) break;
        const int bnd = min(d.t1 * kTileTokens, n);
        for (int j = a + h + te; j < bnd - h; j += 32 * kEpiWarps) {
          float accp = 0.f;
          for (int t = 0; t <= 2 * h; ++t) accp += cbuf[j - h + t - a];
          p.pooled[soff + j] = accp / fP;
        }
        if (!publish(ci)) break;
      }
    }
  } else if (warp >= kCWarp0 && warp < kCWarp0 + kCThreads / 32) {
    // ------------------------------------------------------------ merge / select
    const int ct = threadIdx.x - kCWarp0 * 32;
    for (;;) {
      if (ct == 0) claim_task(F, s_task);
      cbar();
      const int type = s_task[0];
      const int idx = s_task[1];
      cbar();
      if (type == kTaskEnd) break;
      if (type == kTaskMerge) {
        merge_unit(F, idx, creg, ct);
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

size_t fused_smem_bytes(int q_half_bytes, int q_bufs, int stages, int row_stride, int nwg) {
  return 1024 + static_cast<size_t>(stages) * kTileBytes +
         2 * static_cast<size_t>(q_bufs) * q_half_bytes +
         2 * static_cast<size_t>(4 * nwg) * row_stride * 4 + kFixedBytes + kFusedCRegion;
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
