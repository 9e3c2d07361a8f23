// Exact cosine top-k over the gradient store (Bergson Sec. 3.1: exact top-k
// nearest-neighbour lookup; queries score against unit-normalised rows).
//
// Score kernels (persistent, one CTA per SM): a CTA owns one query group of
// QT x 128 normalised fp16 queries and streams every (grid / n_qg)-th tile of
// 256 store rows.  TMA brings 64-column slices of the store tile and of the
// query tiles into a shared-memory ring; one thread issues tcgen05.mma with
// the queries on M and N = 256 store rows, K = 16, into TMEM (fp32), so that
// TMEM lane = query and column = store row.  Up to 128 queries one CTA runs
// M = 128 on its own (score_kernel); above that CTAs run in pairs whose MMAs
// take M = 256 over both CTAs' query tiles, each CTA loading half of every
// store tile (score_pair_kernel).  Epilogue warps read their query's 256
// scores, drop everything not above the query's running k-th best, and keep a
// per-(CTA, query) 4-ary min-heap of the k best (score, row) keys in global
// memory.  The N x Q score matrix never exists.
// Merge kernel: one CTA per query takes the heaps of the CTAs that covered the
// query, finds the k-th best key by an exact radix select and sorts the top-k
// by score descending, then row ascending.
// Large stores are scored twice: first a prefix of about 128 x topk rows
// (whole rounds of store tiles), whose exact per-query k-th best is a lower
// bound of the final k-th best; the full pass then starts from that threshold,
// so few scores ever reach the heaps.

#include "internal.h"
#include "ptx.cuh"

namespace bergson {

namespace {

constexpr int kSmemBudget = 232448;
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;
constexpr int kStoreBoxBytes = kScoreBN * 128;      // 256 rows x 64 fp16
constexpr int kQBoxBytes = kScoreQT * 128;          // 128 rows x 64 fp16
constexpr unsigned long long kSentinelKey = 0x007FFFFF00000000ull;   // (-inf, row 0xFFFFFFFF)
// L2 policy of store-chunk loads: 0 = evict_normal, 1 = evict_first.  The
// pair kernel with more than one pair of query groups (n_qg counts the
// CTAs' groups, two per pair) keeps the normal policy: every store half is
// read once per pair group, by CTAs that stream the same tiles in the same
// order (paced, below), and the later reads hit L2 more often when the first
// one does not mark the lines for early eviction (1.6x the store in DRAM
// reads with evict_first at 1024 queries).
constexpr int kStoreEvictFirst = 1;

// Candidates a lane may park in shared memory per tile before inserting them
// into its heap after the tile's TMEM buffer is released.
constexpr int kQueueCap = 8;

// Candidate keys the merge keeps in shared memory for its radix select
// (26,624 x 8 bytes = 208 KB); larger candidate sets are merged in sorted rounds.
constexpr int kMergeSmemKeys = 26624;

template <int QT>
struct ScoreCfg {
  static constexpr int kStageBytes = kStoreBoxBytes + QT * kQBoxBytes;
  static constexpr int kBarBytes = 256;
  static constexpr int kQueueBytes = kQueueCap * QT * 128 * 8;
  static constexpr int kStagesFit = (kSmemBudget - 1024 - kBarBytes - kQueueBytes) / kStageBytes;
  static constexpr int kStages = kStagesFit > 6 ? 6 : kStagesFit;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kQueueBytes + kBarBytes;
  static constexpr int kNBuf = 512 / (QT * kScoreBN);   // TMEM accumulator buffers
  static constexpr int kEpiThreads = QT * 128;
  static constexpr int kThreads = 64 + kEpiThreads;
  static_assert(kNBuf >= 1, "TMEM budget");
};

// Order-preserving map of a float onto uint32 (-0 is folded onto +0 first).
__device__ __forceinline__ uint32_t float_order(float s) {
  const uint32_t u = __float_as_uint(s + 0.0f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float order_to_float(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

// Larger key = better: higher score first, then lower row index.
__device__ __forceinline__ unsigned long long make_key(float s, uint32_t row) {
  return (static_cast<unsigned long long>(float_order(s)) << 32) | static_cast<uint32_t>(~row);
}

// Children per node of the per-query min-heaps (a wider heap is shallower:
// fewer dependent global-memory round trips per insertion).
constexpr int kHeapArity = 4;

// Replace the root (worst kept entry) of a kHeapArity-ary min-heap of `k` keys
// stored at base[e * stride] and restore the heap property.  The children of
// one node are loaded together, so each level costs one memory round trip.
__device__ __forceinline__ void heap_replace_root(unsigned long long* base, int stride, int k,
                                                  unsigned long long key) {
  int i = 0;
  for (;;) {
    const int c0 = kHeapArity * i + 1;
    if (c0 >= k) break;
    unsigned long long kc = base[static_cast<int64_t>(c0) * stride];
    int c = c0;
#pragma unroll
    for (int t = 1; t < kHeapArity; ++t) {
      if (c0 + t < k) {
        const unsigned long long kt = base[static_cast<int64_t>(c0 + t) * stride];
        if (kt < kc) { kc = kt; c = c0 + t; }
      }
    }
    if (kc >= key) break;
    base[static_cast<int64_t>(i) * stride] = kc;
    i = c;
  }
  base[static_cast<int64_t>(i) * stride] = key;
}

// v[pos] for a run-time pos in [0, 32) without dynamic register indexing
// (a 5-level select tree keeps v in registers).
__device__ __forceinline__ float select32(const float* v, uint32_t pos) {
  float t16[16], t8[8], t4[4], t2[2];
#pragma unroll
  for (int i = 0; i < 16; ++i) t16[i] = (pos & 16u) ? v[i + 16] : v[i];
#pragma unroll
  for (int i = 0; i < 8; ++i) t8[i] = (pos & 8u) ? t16[i + 8] : t16[i];
#pragma unroll
  for (int i = 0; i < 4; ++i) t4[i] = (pos & 4u) ? t8[i + 4] : t8[i];
#pragma unroll
  for (int i = 0; i < 2; ++i) t2[i] = (pos & 2u) ? t4[i + 2] : t4[i];
  return (pos & 1u) ? t2[1] : t2[0];
}

// Epilogue role (QT x 128 threads, one query per thread): per store tile, wait
// for the accumulators, read the query's 256 scores from TMEM, keep those above
// its running k-th best, release TMEM (on the even CTA of a pair when kPair),
// then insert the parked candidates into the query's heap in global memory.
template <int QT, int kNBuf, bool kPair>
__device__ __forceinline__ void score_epilogue(const ScoreParams& p, uint32_t tmem, uint64_t* tfull,
                                               uint64_t* tempty,
                                               unsigned long long* cand_queue,
                                               volatile int* s_abort, volatile int* s_epi_stop,
                                               int g, int nt0, int cpg, int warp, int lane,
                                               uint64_t tmo) {
  constexpr int kEpiThreads = QT * 128;
  const int et = threadIdx.x - 64;                 // 0 .. QT*128-1
  const int qt = et >> 7;
  const int quarter = warp & 3;
  const int slot = qt * kScoreQT + 32 * quarter + lane;
  const int stride = kEpiThreads;
  unsigned long long* heap =
      p.heaps + static_cast<int64_t>(blockIdx.x) * p.topk * stride + slot;
  for (int e = 0; e < p.topk; ++e) heap[static_cast<int64_t>(e) * stride] = kSentinelKey;
  unsigned long long tau_key = kSentinelKey;
  // Scores below the k-th best of any subset of the rows can never reach the
  // final top-k, so a threshold from a prefix pass (if any) filters from the start.
  const int q_global = (g * QT + qt) * kScoreQT + 32 * quarter + lane;
  float tau0 = -INFINITY;
  if (p.tau0 != nullptr && q_global < p.Q) {
    const float t = p.tau0[static_cast<int64_t>(q_global) * p.topk + p.topk - 1];
    tau0 = p.tau0_negate ? -t : t;
  }
  float tau = tau0;
  // Slots past the last query (ragged query groups) hold zero rows: they take
  // no candidates, so their lanes do not walk every score of every tile.
  const bool live = q_global < p.Q;
  int nq = 0;                                       // parked candidates of this lane
  int ab = 0;
  uint32_t aph = 0;
  for (int nt = nt0; nt < p.n_ntiles; nt += cpg) {
    if (et == 0) {
      if (!mbar_wait(smem_u32(&tfull[ab]), aph, tmo, s_abort))
        raise_device_error(p.status, s_abort, kStatusTimeout);
      *s_epi_stop = *s_abort;
    }
    named_bar_sync(1, kEpiThreads);
    if (*s_epi_stop) break;
    tc_fence_after();
    const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * quarter) << 16) +
                           ab * QT * kScoreBN + qt * kScoreBN;
    const int row_base = nt * kScoreBN;
#pragma unroll 1
    for (int c = 0; c < kScoreBN / 32; ++c) {
      float v[32];
      tmem_ld32(tbase + c * 32, v);
      const int r0 = row_base + c * 32;
      const int nvalid = min(32, p.N - r0);
      // Candidate positions of this lane (the comparison also drops NaN).
      uint32_t cand = 0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (live && j < nvalid && v[j] >= tau) cand |= 1u << j;
      // Warp-uniform rounds: in round r every lane inserts its r-th candidate,
      // so a warp pays for its busiest lane, not for every distinct column.
      while (__any_sync(0xffffffffu, cand != 0)) {
        if (cand != 0) {
          const uint32_t pos = __ffs(cand) - 1;
          cand &= cand - 1;
          const unsigned long long key = make_key(select32(v, pos), static_cast<uint32_t>(r0) + pos);
          if (key > tau_key) {
            if (nq < kQueueCap) {                 // park it; inserted after TMEM is released
              cand_queue[nq * stride + slot] = key;
              ++nq;
            } else {                              // queue full: insert now
              heap_replace_root(heap, stride, p.topk, key);
              tau_key = heap[0];
              tau = fmaxf(tau0, order_to_float(static_cast<uint32_t>(tau_key >> 32)));
            }
          }
        }
      }
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) {
      if (kPair)
        mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[ab]), 0));
      else
        mbar_arrive(smem_u32(&tempty[ab]));
    }
    if (++ab == kNBuf) { ab = 0; aph ^= 1; }
    // The MMA warp is already filling TMEM for the next tile; drain the parked
    // candidates meanwhile (warp-uniform rounds, as above).
    while (__any_sync(0xffffffffu, nq > 0)) {
      if (nq > 0) {
        --nq;
        const unsigned long long key = cand_queue[nq * stride + slot];
        if (key > tau_key) {
          heap_replace_root(heap, stride, p.topk, key);
          tau_key = heap[0];
          tau = fmaxf(tau0, order_to_float(static_cast<uint32_t>(tau_key >> 32)));
        }
      }
    }
    named_bar_sync(1, kEpiThreads);   // keeps the stop broadcast single-writer
  }
}

template <int QT>
__global__ void __launch_bounds__(ScoreCfg<QT>::kThreads, 1)
    score_kernel(const __grid_constant__ CUtensorMap tm_store, const __grid_constant__ CUtensorMap tm_q,
                 const ScoreParams p) {
  using C = ScoreCfg<QT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  unsigned long long* cand_queue =
      reinterpret_cast<unsigned long long*>(smem + C::kStages * C::kStageBytes);  // [cap][lanes]
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes + C::kQueueBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* tfull = empty + C::kStages;       // [kNBuf]
  uint64_t* tempty = tfull + 2;               // [kNBuf]
  uint64_t* drain = tempty + 2;
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  volatile int* s_epi_stop = s_abort + 1;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g_local = blockIdx.x % p.n_qg;
  const int g = p.qg_base + g_local;
  const int cpg = gridDim.x / p.n_qg;
  const int nt0 = blockIdx.x / p.n_qg;
  const int nK = (p.K + kChunk - 1) / kChunk;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int i = 0; i < C::kNBuf; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), QT * 4);
    }
    mbar_init(smem_u32(drain), 1);
    *s_abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(s_tmem), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const uint64_t tmo = p.timeout_ns;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tm_store);
      prefetch_tmap(&tm_q);
      const uint64_t pol_store = kStoreEvictFirst ? policy_evict_first() : policy_evict_normal();
      const uint64_t pol_q = policy_evict_last();
      int stage = 0;
      uint32_t ph = 0;
      uint32_t issued = 0, issued_par = 0;
      bool ok = true;
      for (int nt = nt0; nt < p.n_ntiles && ok; nt += cpg) {
        for (int kc = 0; kc < nK; ++kc) {
          if (!mbar_wait(smem_u32(&empty[stage]), ph ^ 1, tmo, s_abort)) { ok = false; break; }
          const uint32_t fb = smem_u32(&full[stage]);
          mbar_arrive_expect_tx(fb, C::kStageBytes);
          const uint32_t dst = sbase + stage * C::kStageBytes;
          tma_load_2d_hint(dst, &tm_store, fb, kc * kChunk, nt * kScoreBN, pol_store);
#pragma unroll
          for (int qt = 0; qt < QT; ++qt)
            tma_load_2d_hint(dst + kStoreBoxBytes + qt * kQBoxBytes, &tm_q, fb, kc * kChunk,
                             (g * QT + qt) * kScoreQT, pol_q);
          issued |= 1u << stage;
          issued_par = (issued_par & ~(1u << stage)) | (ph << stage);
          if (++stage == C::kStages) { stage = 0; ph ^= 1; }
        }
      }
      if (!ok) {
        raise_device_error(p.status, s_abort, kStatusTimeout);
        for (int s = 0; s < C::kStages; ++s)
          if (issued >> s & 1)
            mbar_wait(smem_u32(&full[s]), (issued_par >> s) & 1, kDrainTimeoutNs, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = make_idesc_f16(kScoreQT, kScoreBN, false);
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (int nt = nt0; nt < p.n_ntiles && ok; nt += cpg) {
        if (!mbar_wait(smem_u32(&tempty[ab]), aph ^ 1, tmo, s_abort)) { ok = false; break; }
        tc_fence_after();
        const uint32_t dbuf = tmem + ab * QT * kScoreBN;
        for (int kc = 0; kc < nK; ++kc) {
          if (!mbar_wait(smem_u32(&full[stage]), ph, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sd = sbase + stage * C::kStageBytes;
          const uint32_t qd = sd + kStoreBoxBytes;
#pragma unroll
          for (int qt = 0; qt < QT; ++qt) {
#pragma unroll
            for (int kk = 0; kk < kChunk / 16; ++kk)
              umma_f16(dbuf + qt * kScoreBN, sw128_desc(qd + qt * kQBoxBytes + kk * 32),
                       sw128_desc(sd + kk * 32), idesc, (kc | kk) != 0);
          }
          umma_commit(smem_u32(&empty[stage]));
          if (++stage == C::kStages) { stage = 0; ph ^= 1; }
        }
        if (!ok) break;
        umma_commit(smem_u32(&tfull[ab]));
        if (++ab == C::kNBuf) { ab = 0; aph ^= 1; }
      }
      if (!ok) raise_device_error(p.status, s_abort, kStatusTimeout);
      umma_commit(smem_u32(drain));
      mbar_wait(smem_u32(drain), 0, kDrainTimeoutNs, nullptr);
    }
    __syncwarp();
  } else {
    score_epilogue<QT, C::kNBuf, false>(p, tmem, tfull, tempty, cand_queue, s_abort, s_epi_stop,
                                        g, nt0, cpg, warp, lane, tmo);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Pair variant for more than 128 queries (QT query tiles per CTA, clusters of
// two CTAs on two SMs).  One tcgen05.mma of M = 256 (the two CTAs' query tiles
// of the same index) x N = 256 store rows serves both SMs: each CTA loads only
// its half of the store tile (128 rows), and the tensor cores of the pair read
// both halves.  With QT = 2 (more than 256 queries, tensor-bound) a 16-column
// step moves 12 KB into shared memory and reads 16 KB out of it per SM for two
// 128 x 256 products, against 16 KB and 24 KB for the single-CTA kernel.  With
// QT = 1 (129..256 queries, bound by the store stream) the smaller stages give
// six of them, i.e. more store bytes in flight per SM, and two TMEM buffers.
//
// Synchronisation: the odd CTA's TMA loads complete on the even CTA's `full`
// barrier, which expects the bytes of both; the even CTA's MMA thread frees a
// stage in both CTAs (commit multicast to `empty`), and signals both CTAs'
// epilogues (commit multicast to `tfull`); both epilogues release the TMEM
// buffer on the even CTA's `tempty`.
constexpr int kPairStoreRows = kScoreBN / 2;               // store rows each CTA loads
constexpr int kPairStoreBoxBytes = kPairStoreRows * 128;   // 128 rows x 64 fp16

// Pacing of the pair groups that read the same store tiles (two or more pair
// groups: more than 512 queries).  Each store half is read once per pair
// group; the second read finds it in L2 only while the groups stay close
// (left alone they drift apart over a pass, and their re-reads then miss).
// Each producer publishes its count of issued store chunks every kPaceEvery
// chunks, tagged with the launch, and before running more than kPaceLead
// chunks ahead of the next pair group's CTA (same tile sequence, same rank;
// the groups form a ring) waits for it, at most kPaceWaitNs per wait; a peer
// that does not catch up in that time ends the pacing for this CTA.  The
// peer's word is read one check ahead, so a producer that is not ahead does
// not wait out the load.  A waiting CTA has published its own count, so no
// ring of CTAs can all wait on one another.  Only timing depends on the
// words: a stale or foreign word just means a wait that runs out.
// Measured at 1024 queries (3.2 GB store): DRAM reads 1.08x the store at a
// lead of 16 (1.07x at 8, but 30% slower; 1.13-1.33x at 32 or unpaced).
constexpr uint32_t kPaceEvery = 8;
constexpr uint32_t kPaceLead = 16;                    // an eighth of a 8192-column tile
constexpr uint64_t kPaceWaitNs = 100000ull;

template <int QT_>
struct PairCfg {
  static constexpr int QT = QT_;
  static constexpr int kStageBytes = kPairStoreBoxBytes + QT * kQBoxBytes;
  static constexpr int kBarBytes = 256;
  static constexpr int kQueueBytes = kQueueCap * QT * 128 * 8;
  static constexpr int kStagesFit = (kSmemBudget - 1024 - kBarBytes - kQueueBytes) / kStageBytes;
  static constexpr int kStages = kStagesFit > 6 ? 6 : kStagesFit;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kQueueBytes + kBarBytes;
  static constexpr int kNBuf = 512 / (QT * kScoreBN);   // TMEM accumulator buffers
  static constexpr int kEpiThreads = QT * 128;
  static constexpr int kThreads = 64 + kEpiThreads;
  static_assert(kStages >= 3, "pipeline depth");
  static_assert(2 * kStages + 4 * kNBuf + 1 <= kBarBytes / 8 - 2, "barrier area");
};

// Bounded wait for this CTA's own TMA loads after an abort: the odd CTA's
// loads complete on the other CTA's barrier, so it waits out a fixed time.
__device__ __forceinline__ void pair_settle_loads() {
  const uint64_t t0 = global_timer_ns();
  while (global_timer_ns() - t0 < 1000000ull) {
  }
}

template <int QT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PairCfg<QT>::kThreads, 1)
    score_pair_kernel(const __grid_constant__ CUtensorMap tm_store,
                      const __grid_constant__ CUtensorMap tm_q, const ScoreParams p) {
  using C = PairCfg<QT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  unsigned long long* cand_queue =
      reinterpret_cast<unsigned long long*>(smem + C::kStages * C::kStageBytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::kStages * C::kStageBytes + C::kQueueBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* tfull = empty + C::kStages;       // [kNBuf]
  uint64_t* tempty = tfull + 2;               // [kNBuf]
  uint64_t* drain = tempty + 2;
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  volatile int* s_epi_stop = s_abort + 1;

  const uint32_t rank = cluster_ctarank();   // 0: issues the MMAs
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g_local = blockIdx.x % p.n_qg;   // even on rank 0, +1 on rank 1
  const int g = p.qg_base + g_local;
  const int cpg = gridDim.x / p.n_qg;
  const int nt0 = blockIdx.x / p.n_qg;       // the same for both CTAs of the pair
  const int nK = (p.K + kChunk - 1) / kChunk;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int i = 0; i < C::kNBuf; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), 2 * QT * 4);   // every epilogue warp of both CTAs
    }
    mbar_init(smem_u32(drain), 1);
    *s_abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(s_tmem), 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();              // both CTAs' barriers initialised and TMEM allocated
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const uint64_t tmo = p.timeout_ns;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&tm_store);
      prefetch_tmap(&tm_q);
      const uint64_t pol_store =
          kStoreEvictFirst && p.n_qg == 2 ? policy_evict_first() : policy_evict_normal();
      const uint64_t pol_q = policy_evict_last();
      int stage = 0;
      uint32_t ph = 0;
      uint32_t issued = 0, issued_par = 0;
      bool ok = true;
      // pacing against the next pair group's CTA on the same tiles (see kPaceLead)
      bool pacing = p.pace != nullptr && p.n_qg >= 4;
      unsigned long long* pace_mine = nullptr;
      const unsigned long long* pace_peer = nullptr;
      if (pacing) {
        const int n_pg = p.n_qg >> 1;
        const int pg = g_local >> 1;
        pace_mine = p.pace + blockIdx.x;
        pace_peer = p.pace + nt0 * p.n_qg + ((pg + 1) % n_pg) * 2 + (g_local & 1);
      }
      const unsigned long long tag = static_cast<unsigned long long>(p.pace_tag) << 32;
      uint32_t n_chunks = 0;
      unsigned long long peer_next = 0;   // peer word read at the previous check
      for (int nt = nt0; nt < p.n_ntiles && ok; nt += cpg) {
        for (int kc = 0; kc < nK; ++kc, ++n_chunks) {
          if (pacing && n_chunks % kPaceEvery == 0) {
            st_relaxed_u64(pace_mine, tag | n_chunks);
            if (n_chunks >= kPaceLead) {
              unsigned long long v = peer_next;
              const uint64_t t0 = global_timer_ns();
              while (!((v >> 32) == p.pace_tag && static_cast<uint32_t>(v) + kPaceLead >= n_chunks)) {
                if (*s_abort || global_timer_ns() - t0 > kPaceWaitNs) {
                  pacing = false;
                  break;
                }
                v = ld_relaxed_u64(pace_peer);
              }
            }
            peer_next = ld_relaxed_u64(pace_peer);
          }
          if (!mbar_wait(smem_u32(&empty[stage]), ph ^ 1, tmo, s_abort)) { ok = false; break; }
          const uint32_t fb_local = smem_u32(&full[stage]);
          const uint32_t fb = mapa_shared(fb_local, 0);
          if (rank == 0) mbar_arrive_expect_tx(fb_local, 2 * C::kStageBytes);
          const uint32_t dst = sbase + stage * C::kStageBytes;
          tma_load_2d_pair(dst, &tm_store, fb, kc * kChunk,
                           nt * kScoreBN + static_cast<int>(rank) * kPairStoreRows, pol_store);
#pragma unroll
          for (int qt = 0; qt < QT; ++qt)
            tma_load_2d_pair(dst + kPairStoreBoxBytes + qt * kQBoxBytes, &tm_q, fb, kc * kChunk,
                             (g * QT + qt) * kScoreQT, pol_q);
          issued |= 1u << stage;
          issued_par = (issued_par & ~(1u << stage)) | (ph << stage);
          if (++stage == C::kStages) { stage = 0; ph ^= 1; }
        }
      }
      if (pacing) st_relaxed_u64(pace_mine, tag | n_chunks);   // releases a peer near the end
      if (!ok) {
        raise_device_error(p.status, s_abort, kStatusTimeout);
        if (rank == 0) {
          for (int s = 0; s < C::kStages; ++s)
            if (issued >> s & 1)
              mbar_wait(smem_u32(&full[s]), (issued_par >> s) & 1, kDrainTimeoutNs, nullptr);
        } else {
          pair_settle_loads();
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (rank == 0 && lane == 0) {
      const uint32_t idesc = make_idesc_f16(2 * kScoreQT, kScoreBN, false);
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (int nt = nt0; nt < p.n_ntiles && ok; nt += cpg) {
        if (!mbar_wait_cluster(smem_u32(&tempty[ab]), aph ^ 1, tmo, s_abort)) { ok = false; break; }
        tc_fence_after();
        const uint32_t dbuf = tmem + ab * QT * kScoreBN;
        for (int kc = 0; kc < nK; ++kc) {
          if (!mbar_wait(smem_u32(&full[stage]), ph, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sd = sbase + stage * C::kStageBytes;
          const uint32_t qd = sd + kPairStoreBoxBytes;
#pragma unroll
          for (int qt = 0; qt < QT; ++qt) {
#pragma unroll
            for (int kk = 0; kk < kChunk / 16; ++kk)
              umma_f16_pair(dbuf + qt * kScoreBN, sw128_desc(qd + qt * kQBoxBytes + kk * 32),
                            sw128_desc(sd + kk * 32), idesc, (kc | kk) != 0);
          }
          umma_commit_pair(smem_u32(&empty[stage]), 0x3);
          if (++stage == C::kStages) { stage = 0; ph ^= 1; }
        }
        if (!ok) break;
        umma_commit_pair(smem_u32(&tfull[ab]), 0x3);
        if (++ab == C::kNBuf) { ab = 0; aph ^= 1; }
      }
      if (!ok) raise_device_error(p.status, s_abort, kStatusTimeout);
      umma_commit_pair(smem_u32(drain), 0x1);
      mbar_wait(smem_u32(drain), 0, kDrainTimeoutNs, nullptr);
    }
    __syncwarp();
  } else {
    score_epilogue<QT, C::kNBuf, true>(p, tmem, tfull, tempty, cand_queue, s_abort, s_epi_stop, g,
                                       nt0, cpg, warp, lane, tmo);
  }

  tc_fence_before();
  cluster_sync();              // no MMA, commit or remote arrival is still in flight
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
}

// Bitonic sort of keys[0, n) (n a power of two) into descending order.
__device__ __forceinline__ void bitonic_desc(unsigned long long* keys, int n) {
  for (int kk = 2; kk <= n; kk <<= 1) {
    for (int j = kk >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const unsigned long long a = keys[i];
          const unsigned long long b = keys[ixj];
          const bool desc = (i & kk) == 0;
          if (desc ? (a < b) : (a > b)) {
            keys[i] = b;
            keys[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
}

// negate: the scores were taken against -q (a bottom-k search); report them
// against q, so the list runs from the lowest score up.  Key rows are global
// (row_base already added).
__device__ __forceinline__ void write_topk(const unsigned long long* keys, int q, int topk,
                                           int negate, float* out_scores, int64_t* out_idx) {
  for (int e = threadIdx.x; e < topk; e += blockDim.x) {
    const unsigned long long k = keys[e];
    const uint32_t lo = static_cast<uint32_t>(k);
    const bool real = lo >= 0x80000000u;          // rows < 2^31 map to ~row >= 2^31
    const float v = real ? order_to_float(static_cast<uint32_t>(k >> 32)) : -INFINITY;
    out_scores[static_cast<int64_t>(q) * topk + e] = negate ? -v : v;
    out_idx[static_cast<int64_t>(q) * topk + e] = real ? static_cast<int64_t>(~lo) : -1;
  }
}

// Candidate i of query q for the merge: i < n_heap comes from the heaps (its
// local row moved to row_base + row), the next topk from the prior result
// (scores against q, negated back into the search's order for a bottom-k
// state).  Empty entries become the sentinel-free key 0.
struct MergeSource {
  const unsigned long long* heaps;
  int n_qg, gsize, topk, gl, slot;
  int64_t n_heap;
  uint32_t row_base;
  const float* prior_scores;
  const int64_t* prior_idx;
  int q;
  int negate;
  __device__ __forceinline__ unsigned long long key(int64_t i) const {
    if (i < n_heap) {
      const int cta = gl + static_cast<int>(i / topk) * n_qg;
      const unsigned long long k =
          heaps[(static_cast<int64_t>(cta) * topk + i % topk) * gsize + slot];
      const uint32_t lo = static_cast<uint32_t>(k);
      if (lo < 0x80000000u || row_base == 0u) return k;      // sentinel, or no offset
      return (k & 0xFFFFFFFF00000000ull) | static_cast<uint32_t>(~(~lo + row_base));
    }
    const int64_t e = static_cast<int64_t>(q) * topk + (i - n_heap);
    const int64_t idx = prior_idx[e];
    if (idx < 0) return 0ull;
    const float v = prior_scores[e];
    return make_key(negate ? -v : v, static_cast<uint32_t>(idx));
  }
};

// Final top-k of one query from the heaps of the CTAs that covered it.
//
// select_n > 0: all cpg * topk candidate keys fit in shared memory.  An exact
// radix select (eight passes over 8-bit digits, most significant first) finds
// the topk-th largest key T; keys are unique (the low word is the row), so
// exactly topk keys are >= T.  They are compacted and bitonic-sorted
// (select_n = a power of two >= topk).  Otherwise (select_n == 0) the keys
// are sorted in rounds of sort_n, keeping the best topk of each round.
__global__ void __launch_bounds__(512) merge_kernel(const unsigned long long* __restrict__ heaps,
                                                    int n_qg, int cpg, int gsize, int topk,
                                                    int q_begin, int q_end, int sort_n,
                                                    int select_n, int negate, uint32_t row_base,
                                                    const float* prior_scores,
                                                    const int64_t* prior_idx, float* out_scores,
                                                    int64_t* out_idx) {
  extern __shared__ unsigned long long keys[];
  __shared__ unsigned int hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_need, s_count;
  const int q = q_begin + blockIdx.x;
  if (q >= q_end) return;
  const int local = q - q_begin;
  MergeSource src;
  src.heaps = heaps;
  src.n_qg = n_qg;
  src.gsize = gsize;
  src.topk = topk;
  src.gl = local / gsize;
  src.slot = local % gsize;
  src.n_heap = static_cast<int64_t>(cpg) * topk;
  src.row_base = row_base;
  src.prior_scores = prior_scores;
  src.prior_idx = prior_idx;
  src.q = q;
  src.negate = negate;
  // Every prior entry is read (into shared memory) before any output is
  // written, so the prior may alias the output.
  const int64_t total = src.n_heap + (prior_idx != nullptr ? topk : 0);
  if (select_n > 0) {
    const int n = static_cast<int>(total);
    for (int i = threadIdx.x; i < n; i += blockDim.x) keys[i] = src.key(i);
    if (threadIdx.x == 0) {
      s_prefix = 0ull;
      s_need = topk;
      s_count = 0;
    }
    __syncthreads();
    for (int shift = 56; shift >= 0; shift -= 8) {
      for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0u;
      __syncthreads();
      const unsigned long long prefix = s_prefix;
      const unsigned long long above = shift == 56 ? 0ull : (~0ull << (shift + 8));
      // Candidates cluster in score, so most share a digit: lanes of a warp
      // with the same digit add their count once (one atomic per group).
      for (int i0 = 0; i0 < n; i0 += blockDim.x) {
        const int i = i0 + threadIdx.x;
        const unsigned long long k = i < n ? keys[i] : 0ull;
        const bool hit = i < n && (k & above) == prefix;
        const unsigned dig = hit ? static_cast<unsigned>((k >> shift) & 255u) : 256u;
        const unsigned peers = __match_any_sync(0xffffffffu, dig);
        if (hit && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[dig], __popc(peers));
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        const int need = s_need;
        int acc = 0, d = 255;
        for (; d > 0; --d) {
          if (acc + static_cast<int>(hist[d]) >= need) break;
          acc += static_cast<int>(hist[d]);
        }
        s_prefix = prefix | (static_cast<unsigned long long>(d) << shift);
        s_need = need - acc;
      }
      __syncthreads();
    }
    const unsigned long long T = s_prefix;       // the topk-th largest key
    unsigned long long* sel = keys + n;
    // Only real keys (a row in the low word) are kept: when fewer than topk
    // exist (NaN scores, or a running result over fewer rows than topk), T is
    // an empty-slot key and more than select_n keys would reach it, so an
    // arbitrary subset -- real keys included -- would otherwise be dropped.
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const unsigned long long k = keys[i];
      if (k >= T && static_cast<uint32_t>(k) >= 0x80000000u) {
        const int pos = atomicAdd(&s_count, 1);
        if (pos < select_n) sel[pos] = k;
      }
    }
    __syncthreads();
    for (int i = min(s_count, select_n) + threadIdx.x; i < select_n; i += blockDim.x) sel[i] = 0ull;
    __syncthreads();
    bitonic_desc(sel, select_n);
    write_topk(sel, q, topk, negate, out_scores, out_idx);
    return;
  }
  int64_t consumed = 0;
  bool first = true;
  while (first || consumed < total) {
    const int start = first ? 0 : topk;
    for (int i = start + threadIdx.x; i < sort_n; i += blockDim.x) {
      const int64_t ci = consumed + (i - start);
      keys[i] = ci < total ? src.key(ci) : 0ull;
    }
    consumed += sort_n - start;
    first = false;
    __syncthreads();
    bitonic_desc(keys, sort_n);
  }
  __syncthreads();
  write_topk(keys, q, topk, negate, out_scores, out_idx);
}

template <int QT>
cudaError_t launch_score_t(const CUtensorMap& tms, const CUtensorMap& tmq, const ScoreParams& p,
                           int grid, cudaStream_t s) {
  using C = ScoreCfg<QT>;
  static PerDeviceOnce attr;
  const cudaError_t e = smem_attr_once(attr, score_kernel<QT>, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  score_kernel<QT><<<grid, C::kThreads, C::kSmemBytes, s>>>(tms, tmq, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score(int qt, const CUtensorMap& tm_store, const CUtensorMap& tm_q,
                         const ScoreParams& p, int grid, cudaStream_t s) {
  if (qt == 1) return launch_score_t<1>(tm_store, tm_q, p, grid, s);
  if (qt == 2) return launch_score_t<2>(tm_store, tm_q, p, grid, s);
  return cudaErrorInvalidValue;
}

template <int QT>
PerDeviceOnce& pair_attr() {
  static PerDeviceOnce attr;
  return attr;
}

template <int QT>
cudaError_t launch_score_pair_t(const CUtensorMap& tm_store, const CUtensorMap& tm_q,
                                const ScoreParams& p, int grid, cudaStream_t s) {
  using C = PairCfg<QT>;
  const cudaError_t e = smem_attr_once(pair_attr<QT>(), score_pair_kernel<QT>, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  score_pair_kernel<QT><<<grid, C::kThreads, C::kSmemBytes, s>>>(tm_store, tm_q, p);
  return cudaGetLastError();
}

template <int QT>
cudaError_t score_pair_max_ctas_t(int sms, int* ctas) {
  using C = PairCfg<QT>;
  cudaError_t e = smem_attr_once(pair_attr<QT>(), score_pair_kernel<QT>, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (sms / 2));
  cfg.blockDim = dim3(C::kThreads);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  int clusters = 0;
  e = cudaOccupancyMaxActiveClusters(&clusters, score_pair_kernel<QT>, &cfg);
  if (e != cudaSuccess) return e;
  *ctas = 2 * clusters;
  return cudaSuccess;
}

cudaError_t launch_score_pair(int qt, const CUtensorMap& tm_store, const CUtensorMap& tm_q,
                              const ScoreParams& p, int grid, cudaStream_t s) {
  if (qt == 1) return launch_score_pair_t<1>(tm_store, tm_q, p, grid, s);
  if (qt == 2) return launch_score_pair_t<2>(tm_store, tm_q, p, grid, s);
  return cudaErrorInvalidValue;
}

// CTAs of the pair kernel that can be resident at once (2 x co-resident clusters).
cudaError_t score_pair_max_ctas(int qt, int sms, int* ctas) {
  if (qt == 1) return score_pair_max_ctas_t<1>(sms, ctas);
  if (qt == 2) return score_pair_max_ctas_t<2>(sms, ctas);
  return cudaErrorInvalidValue;
}

cudaError_t launch_merge(const unsigned long long* heaps, int grid, int n_qg, int qt, int topk,
                         int q_begin, int q_end, int /*qg_base*/, bool negate, int64_t row_base,
                         const float* prior_scores, const int64_t* prior_idx, float* out_scores,
                         int64_t* out_idx, cudaStream_t s) {
  const int nq = q_end - q_begin;
  if (nq <= 0) return cudaSuccess;
  const int cpg = grid / n_qg;
  const int64_t total = static_cast<int64_t>(cpg) * topk + (prior_idx != nullptr ? topk : 0);
  int sort_n = 2;
  while (sort_n < total && sort_n < 8192) sort_n <<= 1;
  int select_n = 2;
  while (select_n < topk) select_n <<= 1;
  const bool radix = total + select_n <= kMergeSmemKeys;
  if (!radix) select_n = 0;
  const size_t smem =
      static_cast<size_t>(radix ? total + select_n : sort_n) * sizeof(unsigned long long);
  static PerDeviceOnce attr;
  const cudaError_t e = smem_attr_once(
      attr, merge_kernel, static_cast<int>(kMergeSmemKeys * sizeof(unsigned long long)));
  if (e != cudaSuccess) return e;
  merge_kernel<<<nq, 512, smem, s>>>(heaps, n_qg, cpg, qt * kScoreQT, topk, q_begin, q_end, sort_n,
                                     select_n, negate ? 1 : 0, static_cast<uint32_t>(row_base),
                                     prior_scores, prior_idx, out_scores, out_idx);
  return cudaGetLastError();
}

}  // namespace bergson
