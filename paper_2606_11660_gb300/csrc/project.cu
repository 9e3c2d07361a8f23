// Fused token projection + masked per-example contraction (Bergson Fig. 1:
// Adafactor normalisation and the double-sided per-module random projection,
// applied to per-example nn.Linear gradients as in App. B, "Gradients").
//
// For one module and example b the projected gradient is
//   G^_b = P_out'^T (sum_t m_t g_t a_t^T) P_in' = sum_t m_t (P_out'^T g_t)(P_in'^T a_t)^T,
// so the kernel never forms the d_out x d_in gradient.  Per 128-token tile:
//   1. TMA streams A and G in 32-token x 64-column bf16 boxes (128-byte
//      swizzle; slices whose 32 tokens are all masked are not read) and the
//      matching 64-column slices of P'^T (hi and lo bf16 rows) into a ring of
//      shared-memory stages;
//   2. one thread issues tcgen05.mma (M = 128 tokens, N = 2k, K = 16) into TMEM:
//      a~ = A P_in' and g~ = G P_out', each as A*[hi|lo] in one MMA whose B
//      operand is the slice's hi rows followed by its lo rows (fp32
//      accumulators, the two halves added by the epilogue);
//   3. four epilogue warps read a~ and g~ out of TMEM (one token per thread),
//      zero masked tokens, stage them in shared memory and accumulate the
//      k_out x k_in outer-product sum in fp32 registers.
// Slots are (module, example, range of tiles); a global counter hands work
// items to persistent CTAs, and each slot writes one k_out x k_in partial that
// a second kernel sums in a fixed order (deterministic result).  Normally one
// item is one slot.  When a launch has too few slots for the SMs to finish
// together, the host cuts large slots into pieces (one side, a range of
// 64-column chunks) listed in a work table: a piece stores its fp32 token
// projections, and the slot's last piece to finish sums them in piece order and
// contracts, so the result does not depend on which CTA finished last.
//
// Warp roles: warp 0 = TMA producer, warp 1 = TMEM owner + MMA issuer,
// warps 2..5 = epilogue.  Every wait is bounded (see ptx.cuh).

#include "internal.h"
#include "ptx.cuh"

namespace bergson {

namespace {

constexpr int kActBoxBytes = kTileTokens * 128;       // 128 rows x 64 bf16 (one tile)
constexpr int kSliceBytes = 32 * 128;                 // one 32-token TMA box
constexpr int kSmemBudget = 232448;                   // 227 KB opt-in per CTA
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;   // waits for own copies after an abort

constexpr int pow2ceil(int x) {
  int p = 32;
  while (p < x) p <<= 1;
  return p;
}

template <int KI, int KO, bool TOKEN = false>
struct ProjCfg {
  // Token mode on the tensor cores (kTC): per tile and block of kTcNQ queries,
  // U = a~ Q^T (M = 128 tokens, K = k_in, N = kTcNQ k_out rows (q, i)) on
  // tcgen05 kind::tf32 (3xTF32), then s_q = sum_i g~_i U[q, i] on the CUDA
  // cores (k_out FMAs per token and query instead of k_out (k_in + 1)).
  // TMEM with one tile per group: the two projection buffers (4 (k_in + k_out)
  // columns), a~ hi / lo (2 k_in) and U (kTcN <= 256) must fit in 512 columns.
  static constexpr int kTcAvail = 512 - 4 * (KI + KO) - 2 * KI;
  static constexpr int kTcNQa = kTcAvail > 0 ? kTcAvail / KO : 0;
  static constexpr int kTcNQb = kTcNQa < 256 / KO ? kTcNQa : 256 / KO;
  static constexpr int kTcNQ = kTcNQb < 16 ? kTcNQb : 16;
  static constexpr bool kTC = TOKEN && kTcNQ >= 1;
  static constexpr int kTcN = kTcNQ * KO;
  static constexpr int kTcAtoms = (KI + 31) / 32;              // 128-byte K atoms of a B row
  static constexpr int kTcBBytes = kTcN * 128 * kTcAtoms;      // one of B_hi / B_lo
  // Tiles sharing one P' slice: each slice is re-read from L2 once per NT
  // tiles, so a larger NT cuts L2 -> SM traffic (NT = 1 -> 2 -> 4 measured
  // 3.05 -> 2.72 -> 2.59 ms on the 48-module bench call).
  static constexpr int NT = kTC ? 1 : ((KI + KO <= 32) ? 4 : ((KI + KO <= 64) ? 2 : 1));
  static constexpr int kPRows = 2 * (KI > KO ? KI : KO);         // hi + lo rows
  static constexpr int kPBytes = kPRows * 128;
  static constexpr int kStageBytes = NT * kActBoxBytes + kPBytes;
  // Epilogue staging: the contraction stages a~ and g~ 64 tokens at a time
  // (half a tile; the room goes to pipeline stages: 4 -> 5 of them at k = 32);
  // token mode keeps the whole tile's worth, where it holds the query blocks.
  static constexpr int kEpiRows = TOKEN ? kTileTokens : kTileTokens / 2;
  static constexpr int kEpiBytes =
      kTC ? 2 * kTcBBytes : kEpiRows * (KI + 4) * 4 + kEpiRows * (KO + 4) * 4;
  static constexpr int kBarBytes = 512;
  static constexpr int kStagesFit = (kSmemBudget - 1024 - kEpiBytes - kBarBytes) / kStageBytes;
  static constexpr int kStages = kStagesFit > 8 ? 8 : kStagesFit;
  static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + kEpiBytes + kBarBytes;
  // Per tile: A*[hi|lo] in 2 KI columns, then G*[hi|lo] in 2 KO columns.
  static constexpr int kTmemPerBuf = NT * 2 * (KI + KO);
  static constexpr int kTmemCols = kTC ? 512 : pow2ceil(2 * kTmemPerBuf);
  static constexpr int kTmA = 2 * kTmemPerBuf;                  // a~ hi, then lo (kTC)
  static constexpr int kTmU = kTmA + 2 * KI;                    // U (kTC)
  static constexpr int kOPT = KO * KI / kTileTokens;            // outputs per epilogue thread
  // Token mode: queries handled per block (held in shared memory at once).
  static constexpr int kQBFit = kEpiBytes / (4 * KI * KO);
  static constexpr int kQB = kTC ? kTcNQ : (kQBFit > 16 ? 16 : kQBFit);
  static_assert(!kTC || (kTcN % 16 == 0 && kTcN <= 256 && kTmU + kTcN <= 512), "token TMEM plan");
  static_assert(kStages >= 2, "shared memory budget too small");
  static_assert(kTmemCols <= 512, "TMEM budget exceeded");
  static_assert(kOPT >= 2 && kOPT % 2 == 0, "unsupported projection sizes");
};

struct ItemCoord {
  int m, b, t_begin, t_end;
  int slot;                 // partial index of the (module, example, tile range)
  int side;                 // 0: fused; 1 / 2: A / G side piece
  int ch_begin, ch_end;     // chunk range of a piece
  int split, n_a, n_g, piece;
  int64_t base;
};

__device__ __forceinline__ ItemCoord decode_item(const ProjParams& p, int item) {
  ItemCoord c;
  c.slot = item;
  c.side = 0;
  c.ch_begin = c.ch_end = 0;
  c.split = c.n_a = c.n_g = c.piece = 0;
  c.base = 0;
  if (p.items != nullptr) {
    const WorkItem& w = p.items[item];
    c.slot = w.slot;
    c.side = w.side;
    c.ch_begin = w.ch_begin;
    c.ch_end = w.ch_end;
    c.split = w.split;
    c.n_a = w.n_a;
    c.n_g = w.n_g;
    c.piece = w.piece;
    c.base = w.base;
  }
  const int chunk = c.slot % p.n_chunks;
  const int mb = c.slot / p.n_chunks;
  c.b = mb % p.B;
  c.m = mb / p.B;
  c.t_begin = chunk * p.tpc;
  c.t_end = min(p.n_tiles, c.t_begin + p.tpc);
  return c;
}

// Valid 32-token slices of the NT tiles starting at tile g: bit 4*nt + q is set
// when slice q of tile g + nt (inside the item) holds a valid token.  Without a
// mask a slice is valid when it starts before T.
template <int NT>
__device__ __forceinline__ uint32_t group_slices(const ProjParams& p, int b, int g, int t_end) {
  uint32_t vm = 0;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int t = g + nt;
    if (t >= t_end) continue;
    uint32_t q4;
    if (p.tile_valid != nullptr) {
      q4 = p.tile_valid[b * p.n_tiles + t] & 0xFu;
    } else {
      const int left = p.T - t * kTileTokens;          // > 0 inside the item
      q4 = left >= kTileTokens ? 0xFu : (1u << ((left + 31) / 32)) - 1u;
    }
    vm |= q4 << (4 * nt);
  }
  return vm;
}

// v[j] = column j + column N + j of this thread's TMEM lane (one token): a
// projection accumulated as its P'hi part (columns [0, N)) and P'lo part.
template <int N>
__device__ __forceinline__ void tmem_ld_hilo(uint32_t taddr, float* v) {
#pragma unroll
  for (int c = 0; c < N / 16; ++c) tmem_ld16(taddr + c * 16, &v[c * 16]);
#pragma unroll
  for (int c = 0; c < N / 8; ++c) {
    float lo[8];
    tmem_ld8(taddr + N + c * 8, lo);
#pragma unroll
    for (int j = 0; j < 8; ++j) v[c * 8 + j] += lo[j];
  }
}

// Copies this thread's token projection (N values, hi + lo parts) to dst
// (fp32, 16-byte aligned).
template <int N>
__device__ __forceinline__ void store_token_row(uint32_t taddr, float* dst) {
  float v[N];
  tmem_ld_hilo<N>(taddr, v);
#pragma unroll
  for (int x = 0; x < N / 4; ++x)
    reinterpret_cast<float4*>(dst)[x] = make_float4(v[4 * x], v[4 * x + 1], v[4 * x + 2], v[4 * x + 3]);
}

// v = sum over pieces q = 0..n-1 (in order) of the token row src + q * stride.
// Other CTAs wrote the rows during this launch: the loads bypass L1.
template <int N>
__device__ __forceinline__ void sum_token_rows(const float* src, int64_t stride, int n, float (&v)[N]) {
#pragma unroll
  for (int x = 0; x < N; ++x) v[x] = 0.0f;
  for (int q = 0; q < n; ++q) {
    const float4* s4 = reinterpret_cast<const float4*>(src + q * stride);
#pragma unroll
    for (int x = 0; x < N / 4; ++x) {
      const float4 w = __ldcg(s4 + x);
      v[4 * x] += w.x;
      v[4 * x + 1] += w.y;
      v[4 * x + 2] += w.z;
      v[4 * x + 3] += w.w;
    }
  }
}

// Tiles (bit nt) that have at least one valid slice.
template <int NT>
__device__ __forceinline__ uint32_t tiles_of(uint32_t slices) {
  uint32_t tm = 0;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
    if ((slices >> (4 * nt)) & 0xFu) tm |= 1u << nt;
  return tm;
}

// Token mode: module m's blocks of queries [q0, q0 + n) into sA (128 threads).
template <int KI, int KO>
__device__ __forceinline__ void load_query_block(const ProjParams& p, int m, int q0, int n,
                                                 float* sA, int et) {
  constexpr int blk = KO * KI;
  const int64_t off = p.mods[m].col_offset;
  for (int e = et; e < n * blk; e += 128)
    sA[e] = p.queries[static_cast<int64_t>(q0 + e / blk) * p.ld_q + off + e % blk];
}

// Token mode on the tensor cores: a block of module m's query rows [q0, q0 +
// n) held in registers between its global loads and its split into the B
// operand of U = a~ Q^T, so that the next block's loads are in flight while
// the current one is used.  B row r = q * k_out + i holds Q~_q[i, 0:k_in],
// K-major in 128-byte rows (32 fp32 per K atom, atoms kN rows apart) with the
// 128-byte swizzle, split into tf32 hi and lo parts; chunk e of a thread is
// 16 bytes, columns 4c .. 4c + 3 of row (q, i).
template <int KI, int KO, int kN, int kNQ>
struct QueryBlockRegs {
  static_assert(KI % 4 == 0, "query rows in 16-byte chunks");
  static constexpr int kPerQ = KO * KI / 4;                  // chunks per query
  static constexpr int kVec = (kNQ * kPerQ + 127) / 128;     // chunks per thread
  float4 v[kVec];
  // vec: the rows are 16-byte aligned (else four 4-byte loads per chunk)
  __device__ __forceinline__ void load(const ProjParams& p, int m, int q0, int n, int et, bool vec) {
    const int64_t off = p.mods[m].col_offset;
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const int e = et + 128 * u;
      if (e < n * kPerQ) {
        const int q = e / kPerQ, i = (e % kPerQ) / (KI / 4), c = e % (KI / 4);
        const float* src = p.queries + static_cast<int64_t>(q0 + q) * p.ld_q + off + i * KI + 4 * c;
        v[u] = vec ? *reinterpret_cast<const float4*>(src)
                   : make_float4(src[0], src[1], src[2], src[3]);
      }
    }
  }
  __device__ __forceinline__ void store(uint8_t* bhi, uint8_t* blo, int n, int et) const {
#pragma unroll
    for (int u = 0; u < kVec; ++u) {
      const int e = et + 128 * u;
      if (e < n * kPerQ) {
        const int q = e / kPerQ, i = (e % kPerQ) / (KI / 4), c = e % (KI / 4);
        const int r = q * KO + i;
        const int j = 4 * c, jj = j & 31;
        const int byte = (j >> 5) * kN * 128 + r * 128 + (((jj >> 2) ^ (r & 7)) << 4);
        const float4 x = v[u];
        const float4 h = make_float4(tf32_rn(x.x), tf32_rn(x.y), tf32_rn(x.z), tf32_rn(x.w));
        *reinterpret_cast<float4*>(bhi + byte) = h;
        *reinterpret_cast<float4*>(blo + byte) = make_float4(
            tf32_rn(x.x - h.x), tf32_rn(x.y - h.y), tf32_rn(x.z - h.z), tf32_rn(x.w - h.w));
      }
    }
  }
};

// 32 lanes x N columns of this thread's TMEM row from v (N = 16, 32 or 64).
template <int N>
__device__ __forceinline__ void tmem_store_row(uint32_t taddr, const float* v) {
  if constexpr (N == 16) {
    tmem_st16(taddr, v);
  } else {
#pragma unroll
    for (int c = 0; c < N; c += 32) tmem_st32(taddr + c, v + c);
  }
}

template <int KI, int KO, bool TOKEN>
__global__ void __launch_bounds__(192, 1) project_kernel(const ProjParams p) {
  using C = ProjCfg<KI, KO, TOKEN>;
  constexpr int NT = C::NT;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  uint8_t* epi = smem + C::kStages * C::kStageBytes;     // 1024-byte aligned
  float* sA = reinterpret_cast<float*>(epi);
  float* sG = sA + C::kEpiRows * (KI + 4);
  uint8_t* sBhi = epi;                                  // token mode on the tensor cores:
  uint8_t* sBlo = epi + C::kTcBBytes;                   //   the query block, tf32 hi / lo
  uint64_t* full = reinterpret_cast<uint64_t*>(epi + C::kEpiBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* tfull = empty + C::kStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* sfull = tempty + 2;
  uint64_t* sempty = sfull + 2;
  uint64_t* drain = sempty + 2;
  uint64_t* ubar = drain + 1;                           // token U products done (kTC)
  int* s_item = reinterpret_cast<int*>(ubar + 1);
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(s_item + 2);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);
  volatile int* s_last = s_abort + 1;        // epilogue leader's broadcast of "last piece"

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), 4);
      mbar_init(smem_u32(&sfull[i]), 1);
      mbar_init(smem_u32(&sempty[i]), 2);
    }
    mbar_init(smem_u32(drain), 1);
    mbar_init(smem_u32(ubar), 1);
    *s_abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(s_tmem), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const uint64_t tmo = p.timeout_ns;
  uint32_t uph = 0;        // token mode on the tensor cores: phase of ubar
  bool u_pending = false;  // an issued U product not yet waited for (epilogue thread 0)
  // Everything above overlaps the preceding grid (P' generation); the work
  // table, item counter, tile flags and P' are its or earlier writes.
  griddep_wait();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_act = policy_evict_first();
      const uint64_t pol_p = policy_evict_last();
      int stage = 0;
      uint32_t ph = 0;
      int ss = 0;
      uint32_t sph = 0;
      uint32_t issued = 0, issued_par = 0;      // per-stage: TMA in flight, its phase parity
      bool ok = true;
      for (;;) {
        const int item = atomicAdd(p.counter, 1);
        if (!mbar_wait(smem_u32(&sempty[ss]), sph ^ 1, tmo, s_abort)) { ok = false; break; }
        s_item[ss] = item;
        mbar_arrive(smem_u32(&sfull[ss]));
        if (++ss == 2) { ss = 0; sph ^= 1; }
        if (item >= p.n_items) break;
        const ItemCoord ic = decode_item(p, item);
        const ModDesc* md = p.mods + ic.m;
        tmap_acquire(&md->tmA);
        tmap_acquire(&md->tmG);
        tmap_acquire(&md->tmPin);
        tmap_acquire(&md->tmPout);
        for (int g = ic.t_begin; g < ic.t_end && ok; g += NT) {
          const uint32_t sl = group_slices<NT>(p, ic.b, g, ic.t_end);
          if (sl == 0) continue;
          const uint32_t act_bytes = __popc(sl) * kSliceBytes;
          for (int side = 0; side < 2 && ok; ++side) {
            if (ic.side != 0 && side != ic.side - 1) continue;
            const void* tact = side ? static_cast<const void*>(&md->tmG) : &md->tmA;
            const void* tp = side ? static_cast<const void*>(&md->tmPout) : &md->tmPin;
            const int d = side ? md->d_out : md->d_in;
            const uint32_t pbytes = (side ? 2 * KO : 2 * KI) * 128;
            const int c0 = ic.side != 0 ? ic.ch_begin : 0;
            const int c1 = ic.side != 0 ? ic.ch_end : (d + kChunk - 1) / kChunk;
            for (int ch = c0; ch < c1; ++ch) {
              if (!mbar_wait(smem_u32(&empty[stage]), ph ^ 1, tmo, s_abort)) { ok = false; break; }
              const uint32_t fb = smem_u32(&full[stage]);
              mbar_arrive_expect_tx(fb, act_bytes + pbytes);
              const uint32_t dst = sbase + stage * C::kStageBytes;
#pragma unroll
              for (int x = 0; x < 4 * NT; ++x)
                if (sl >> x & 1)
                  tma_load_3d_hint(dst + x * kSliceBytes, tact, fb, ch * kChunk,
                                   g * kTileTokens + 32 * x, ic.b, pol_act);
              tma_load_2d_hint(dst + NT * kActBoxBytes, tp, fb, ch * kChunk, 0, pol_p);
              issued |= 1u << stage;
              issued_par = (issued_par & ~(1u << stage)) | (ph << stage);
              if (++stage == C::kStages) { stage = 0; ph ^= 1; }
            }
          }
        }
        if (!ok) break;
      }
      griddep_launch_dependents();   // all loads issued: the reduction grid may launch
      if (!ok) {
        raise_device_error(p.status, s_abort, kStatusTimeout);
        // Let every copy this thread started land before the CTA can exit.
        for (int s = 0; s < C::kStages; ++s)
          if (issued >> s & 1)
            mbar_wait(smem_u32(&full[s]), (issued_par >> s) & 1, kDrainTimeoutNs, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      int ss = 0;
      uint32_t sph = 0;
      bool ok = true;
      for (;;) {
        if (!mbar_wait(smem_u32(&sfull[ss]), sph, tmo, s_abort)) { ok = false; break; }
        const int item = s_item[ss];
        mbar_arrive(smem_u32(&sempty[ss]));
        if (++ss == 2) { ss = 0; sph ^= 1; }
        if (item >= p.n_items) break;
        const ItemCoord ic = decode_item(p, item);
        const ModDesc* md = p.mods + ic.m;
        for (int g = ic.t_begin; g < ic.t_end && ok; g += NT) {
          const uint32_t vm = tiles_of<NT>(group_slices<NT>(p, ic.b, g, ic.t_end));
          if (vm == 0) continue;
          if (!mbar_wait(smem_u32(&tempty[ab]), aph ^ 1, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t dbuf = tmem + ab * C::kTmemPerBuf;
          for (int side = 0; side < 2 && ok; ++side) {
            if (ic.side != 0 && side != ic.side - 1) continue;
            const int N = side ? KO : KI;
            // B = the P' slice's hi rows then lo rows (2N rows, contiguous): one
            // MMA gives A*hi in N columns and A*lo in the next N, reading the
            // activation tile once.
            const uint32_t idesc = make_idesc_f16(kTileTokens, 2 * N, true);
            const int d = side ? md->d_out : md->d_in;
            const int c0 = ic.side != 0 ? ic.ch_begin : 0;
            const int c1 = ic.side != 0 ? ic.ch_end : (d + kChunk - 1) / kChunk;
            for (int ch = c0; ch < c1; ++ch) {
              if (!mbar_wait(smem_u32(&full[stage]), ph, tmo, s_abort)) { ok = false; break; }
              tc_fence_after();
              const uint32_t act = sbase + stage * C::kStageBytes;
              const uint32_t pp = act + NT * kActBoxBytes;
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                if (!(vm >> nt & 1)) continue;
                const uint32_t dcol = dbuf + nt * 2 * (KI + KO) + (side ? 2 * KI : 0);
#pragma unroll
                for (int kk = 0; kk < kChunk / 16; ++kk)
                  umma_f16(dcol, sw128_desc(act + nt * kActBoxBytes + kk * 32),
                           sw128_desc(pp + kk * 32), idesc, ch != c0 || kk != 0);
              }
              umma_commit(smem_u32(&empty[stage]));
              if (++stage == C::kStages) { stage = 0; ph ^= 1; }
            }
          }
          if (!ok) break;
          umma_commit(smem_u32(&tfull[ab]));
          if (++ab == 2) { ab = 0; aph ^= 1; }
        }
        if (!ok) break;
      }
      if (!ok) raise_device_error(p.status, s_abort, kStatusTimeout);
      // Every MMA this thread issued must finish before TMEM is released.
      umma_commit(smem_u32(drain));
      mbar_wait(smem_u32(drain), 0, kDrainTimeoutNs, nullptr);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    constexpr int OPT = C::kOPT;
    const int et = threadIdx.x - 64;                 // 0..127
    const int quarter = warp & 3;                    // TMEM lanes 32*quarter ..
    const int row = 32 * quarter + lane;             // token row within a tile
    const int oi = et * KO / kTileTokens;            // output row (k_out index)
    const int oj = (et % (kTileTokens / KO)) * OPT;  // first output column (k_in index)
    int ab = 0;
    uint32_t aph = 0;
    int ss = 0;
    uint32_t sph = 0;
    float acc[OPT];
    float bias_acc = 0.0f;   // column (et % KO) of g~ summed over rows (et / KO)*KO .. +KO
    // token mode on the tensor cores: the next query block, in registers
    QueryBlockRegs<KI, KO, (C::kTC ? C::kTcN : 16), (C::kTC ? C::kTcNQ : 1)> qregs;
    bool qvec = false;
    for (;;) {
      // The leader's wait and the abort flag decide "stop" for all 128
      // threads at once (the barrier's OR), so no thread can see a later value.
      bool stop = false;
      if (et == 0) {
        if (!mbar_wait(smem_u32(&sfull[ss]), sph, tmo, s_abort))
          raise_device_error(p.status, s_abort, kStatusTimeout);
        stop = *s_abort != 0;
      }
      if (named_bar_any(1, 128, stop)) break;
      const int item = s_item[ss];
      named_bar_sync(1, 128);
      if (et == 0) mbar_arrive(smem_u32(&sempty[ss]));
      if (++ss == 2) { ss = 0; sph ^= 1; }
      if (item >= p.n_items) break;
      const ItemCoord ic = decode_item(p, item);
      bool aborted = false;
      bool finisher = false;       // last piece of its slot: contracts the summed pieces
      const int64_t stride_a = static_cast<int64_t>(p.tpc) * kTileTokens * KI;
      const int64_t stride_g = static_cast<int64_t>(p.tpc) * kTileTokens * KO;
      if constexpr (!TOKEN) {
        if (ic.side != 0) {
          // A piece: store this side's token projections of the slot's tiles.
          float* dst = p.piece_buf + ic.base +
                       (ic.side == 1 ? ic.piece * stride_a : ic.n_a * stride_a + ic.piece * stride_g);
          for (int g = ic.t_begin; g < ic.t_end; g += NT) {
            const uint32_t vm = tiles_of<NT>(group_slices<NT>(p, ic.b, g, ic.t_end));
            if (vm == 0) continue;
            bool stop = false;
            if (et == 0) {
              if (!mbar_wait(smem_u32(&tfull[ab]), aph, tmo, s_abort))
                raise_device_error(p.status, s_abort, kStatusTimeout);
              stop = *s_abort != 0;
            }
            if (named_bar_any(1, 128, stop)) { aborted = true; break; }
            tc_fence_after();
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              if (!(vm >> nt & 1)) continue;
              const uint32_t taddr = tmem + (static_cast<uint32_t>(32 * quarter) << 16) +
                                     ab * C::kTmemPerBuf + nt * 2 * (KI + KO);
              const int64_t tok = static_cast<int64_t>(g - ic.t_begin + nt) * kTileTokens + row;
              if (ic.side == 1)
                store_token_row<KI>(taddr, dst + tok * KI);
              else
                store_token_row<KO>(taddr + 2 * KI, dst + tok * KO);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&tempty[ab]));
            if (++ab == 2) { ab = 0; aph ^= 1; }
          }
          if (aborted) break;
          // Count the piece; the slot's last piece to finish contracts them all.
          __threadfence();
          named_bar_sync(1, 128);
          if (et == 0) *s_last = atomicAdd(p.split_cnt + ic.split, 1) == ic.n_a + ic.n_g - 1;
          named_bar_sync(1, 128);
          if (!*s_last) continue;
          __threadfence();
          finisher = true;
        }
      }
#pragma unroll
      for (int x = 0; x < OPT; ++x) acc[x] = 0.0f;
      bias_acc = 0.0f;
      constexpr int QB = ProjCfg<KI, KO, true>::kQB;   // queries held in shared memory at once
      const int n_qblocks = TOKEN ? (p.n_queries + QB - 1) / QB : 0;
      if constexpr (TOKEN) {
        // This module's k_out x k_in block of the query rows, into the
        // (otherwise unused) staging area: all of them when they fit in one
        // block of QB queries, else block by block for every tile group
        // below.  All threads left the previous item behind the two barriers
        // above.
        if constexpr (C::kTC) {
          // block 0 of this module into registers (stored below per tile, or
          // once here when it is the only block)
          qvec = (reinterpret_cast<uintptr_t>(p.queries) & 15) == 0 && (p.ld_q & 3) == 0 &&
                 (p.mods[ic.m].col_offset & 3) == 0;
          qregs.load(p, ic.m, 0, min(QB, p.n_queries), et, qvec);
        }
        if (n_qblocks == 1) {
          if constexpr (C::kTC) {
            qregs.store(sBhi, sBlo, p.n_queries, et);
            fence_proxy_async_smem();        // the tensor cores read it through the async proxy
          } else {
            load_query_block<KI, KO>(p, ic.m, 0, p.n_queries, sA, et);
          }
          named_bar_sync(1, 128);
        }
      }
      for (int g = ic.t_begin; g < ic.t_end; g += NT) {
        const uint32_t vm = tiles_of<NT>(group_slices<NT>(p, ic.b, g, ic.t_end));
        if (vm == 0) continue;
        if (!finisher) {
          bool stop = false;
          if (et == 0) {
            if (!mbar_wait(smem_u32(&tfull[ab]), aph, tmo, s_abort))
              raise_device_error(p.status, s_abort, kStatusTimeout);
            stop = *s_abort != 0;
          }
          if (named_bar_any(1, 128, stop)) { aborted = true; break; }
          tc_fence_after();
        }
        if constexpr (C::kTC) {
          // Token scores of tile g (one tile per group) on the tensor cores.
          // a~ (hi + lo halves summed) and g~ of this thread's token, then a~
          // split into tf32 hi / lo parts into this lane's A row; the
          // projection buffer is released at once.
          const uint32_t lane_base = static_cast<uint32_t>(32 * quarter) << 16;
          float va[KI];
          float vg[KO];
          {
            const uint32_t taddr = tmem + lane_base + ab * C::kTmemPerBuf;
            tmem_ld_hilo<KI>(taddr, va);
            tmem_ld_hilo<KO>(taddr + 2 * KI, vg);
          }
          {
            float ah[KI], al[KI];
#pragma unroll
            for (int j = 0; j < KI; ++j) {
              ah[j] = tf32_rn(va[j]);
              al[j] = tf32_rn(va[j] - ah[j]);
            }
            tmem_store_row<KI>(tmem + lane_base + C::kTmA, ah);
            tmem_store_row<KI>(tmem + lane_base + C::kTmA + KI, al);
          }
          tmem_st_wait();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&tempty[ab]));
          if (++ab == 2) { ab = 0; aph ^= 1; }
          const int t = g * kTileTokens + row;
          const bool in_range = t < p.T;
          const bool valid =
              in_range && (p.mask == nullptr || p.mask[static_cast<int64_t>(ic.b) * p.T + t] != 0);
          for (int qb = 0; qb < n_qblocks; ++qb) {
            const int q0 = qb * QB;
            const int nqb = min(QB, p.n_queries - q0);
            if (n_qblocks > 1) {
              // No barrier first: the previous block's product, the last
              // reader of sBhi / sBlo, completed before the barrier that
              // preceded its U reads.
              qregs.store(sBhi, sBlo, nqb, et);
              fence_proxy_async_smem();
              // the next block (block 0 of the next tile after the last one)
              // loads while this one is multiplied and reduced
              const int qn = qb + 1 < n_qblocks ? q0 + QB : 0;
              qregs.load(p, ic.m, qn, min(QB, p.n_queries - qn), et, qvec);
            }
            // Every lane's A row, the query block and the previous block's U
            // reads are complete before one thread issues the products:
            // U = A_hi B_hi + A_hi B_lo + A_lo B_hi (3xTF32, fp32 accumulation).
            named_bar_sync(1, 128);
            bool stop = false;
            if (et == 0) {
              tc_fence_after();
              const uint32_t idesc = make_idesc_tf32(kTileTokens, C::kTcN);
              const uint32_t ua = tmem + C::kTmU;
              const uint32_t aa = tmem + C::kTmA;
#pragma unroll
              for (int kk = 0; kk < KI / 8; ++kk) {
                const uint32_t boff = (kk >> 2) * C::kTcN * 128;
                const uint64_t bh = sw128_desc(smem_u32(sBhi) + boff) + 2 * (kk & 3);
                const uint64_t bl = sw128_desc(smem_u32(sBlo) + boff) + 2 * (kk & 3);
                umma_tf32_ta(ua, aa + 8 * kk, bh, idesc, kk != 0);
                umma_tf32_ta(ua, aa + 8 * kk, bl, idesc, 1u);
                umma_tf32_ta(ua, aa + KI + 8 * kk, bh, idesc, 1u);
              }
              umma_commit(smem_u32(ubar));
              u_pending = true;
              if (mbar_wait(smem_u32(ubar), uph, tmo, s_abort)) {
                u_pending = false;
              } else {
                raise_device_error(p.status, s_abort, kStatusTimeout);
              }
              stop = *s_abort != 0;
            }
            uph ^= 1;
            if (named_bar_any(1, 128, stop)) { aborted = true; break; }
            tc_fence_after();
            // s_q = sum_i g~_i U[token, q k_out + i], kLd columns of U (kLd /
            // k_out queries) per TMEM load; columns past the block's queries
            // are allocated and read, not used
            constexpr int kLd = C::kTcN % 64 == 0 ? 64 : (C::kTcN % 32 == 0 ? 32 : 16);
            constexpr int kQPerLd = kLd / KO;
            for (int qg = 0; qg < nqb; qg += kQPerLd) {
              float u[kLd];
              const uint32_t ua = tmem + lane_base + C::kTmU + qg * KO;
              if constexpr (kLd == 64) tmem_ld64(ua, u);
              else if constexpr (kLd == 32) tmem_ld32(ua, u);
              else tmem_ld16(ua, u);
#pragma unroll
              for (int qq = 0; qq < kQPerLd; ++qq) {
                const int q = qg + qq;
                float sq = 0.0f;
#pragma unroll
                for (int i = 0; i < KO; ++i) sq = fmaf(vg[i], u[qq * KO + i], sq);
                if (q < nqb && in_range)
                  p.token_partials[((static_cast<int64_t>(ic.m) * p.n_queries + q0 + q) * p.B +
                                    ic.b) * p.T + t] = valid ? sq : 0.0f;
              }
            }
            tc_fence_before();
          }
          if (aborted) break;
        } else {
        // One tile at a time: its a~ and g~ (hi + lo halves summed) are loaded,
        // used and dropped before the next tile's; the TMEM buffer is released
        // after the group (the MMA warp fills the other buffer meanwhile).
        // Token mode with more queries than one block: every block is streamed
        // through shared memory once per tile group, and the group's tiles are
        // read from TMEM again for each block.
        for (int qb = 0; qb < (TOKEN ? n_qblocks : 1); ++qb) {
        const int q0 = qb * QB;
        const int nqb = TOKEN ? min(QB, p.n_queries - q0) : 0;
        if (TOKEN && n_qblocks > 1) {
          named_bar_sync(1, 128);                    // the previous block's readers are done
          load_query_block<KI, KO>(p, ic.m, q0, nqb, sA, et);
          named_bar_sync(1, 128);
        }
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          if (!(vm >> nt & 1)) continue;
          float va[KI];
          float vg[KO];
          if (finisher) {
            const int64_t tok = static_cast<int64_t>(g - ic.t_begin + nt) * kTileTokens + row;
            sum_token_rows<KI>(p.piece_buf + ic.base + tok * KI, stride_a, ic.n_a, va);
            sum_token_rows<KO>(p.piece_buf + ic.base + ic.n_a * stride_a + tok * KO, stride_g,
                               ic.n_g, vg);
          } else {
            const uint32_t taddr = tmem + (static_cast<uint32_t>(32 * quarter) << 16) +
                                   ab * C::kTmemPerBuf + nt * 2 * (KI + KO);
            tmem_ld_hilo<KI>(taddr, va);
            tmem_ld_hilo<KO>(taddr + 2 * KI, vg);
          }
          const int t = (g + nt) * kTileTokens + row;
          if constexpr (TOKEN) {
            // s[q] = g~^T Q~_q a~ for this thread's token: its share of the
            // query's score (masked tokens score 0).
            if (t < p.T) {
              const bool valid =
                  p.mask == nullptr || p.mask[static_cast<int64_t>(ic.b) * p.T + t] != 0;
              // u_i = (Q~_q a~)_i for 16 rows i at a time, the k_in loop outermost,
              // so that the FMAs form 16 independent chains (one warp per SM
              // sub-partition runs this; a single chain would wait on every
              // FMA's latency), then s = sum_i g~_i u_i.
              constexpr int kIG = KO < 16 ? KO : 16;
              for (int q = 0; q < nqb; ++q) {
                const float* qm = sA + q * (KO * KI);
                float sq = 0.0f;
#pragma unroll
                for (int i0 = 0; i0 < KO; i0 += kIG) {
                  float u[kIG];
#pragma unroll
                  for (int ii = 0; ii < kIG; ++ii) u[ii] = 0.0f;
#pragma unroll
                  for (int j = 0; j < KI; j += 4) {
#pragma unroll
                    for (int ii = 0; ii < kIG; ++ii) {
                      const float4 w = *reinterpret_cast<const float4*>(qm + (i0 + ii) * KI + j);
                      u[ii] = fmaf(w.x, va[j], u[ii]);
                      u[ii] = fmaf(w.y, va[j + 1], u[ii]);
                      u[ii] = fmaf(w.z, va[j + 2], u[ii]);
                      u[ii] = fmaf(w.w, va[j + 3], u[ii]);
                    }
                  }
#pragma unroll
                  for (int ii = 0; ii < kIG; ++ii) sq = fmaf(vg[i0 + ii], u[ii], sq);
                }
                p.token_partials[((static_cast<int64_t>(ic.m) * p.n_queries + q0 + q) * p.B +
                                  ic.b) * p.T + t] = valid ? sq : 0.0f;
              }
            }
          } else {
            constexpr int kHalf = kTileTokens / 2;
            const bool valid = t < p.T &&
                (p.mask == nullptr || p.mask[static_cast<int64_t>(ic.b) * p.T + t] != 0);
            // Two halves of 64 tokens: the half's owners (whole warps) stage their
            // a~, g~ rows, then all 128 threads accumulate over the half's tokens.
#pragma unroll 1
            for (int h = 0; h < 2; ++h) {
              named_bar_sync(1, 128);                // previous half's readers are done
              if ((row >> 6) == h) {
                float4* ra = reinterpret_cast<float4*>(sA + (row - h * kHalf) * (KI + 4));
                float4* rg = reinterpret_cast<float4*>(sG + (row - h * kHalf) * (KO + 4));
                const float4 z4 = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int x = 0; x < KI / 4; ++x)
                  ra[x] = valid ? make_float4(va[4 * x], va[4 * x + 1], va[4 * x + 2], va[4 * x + 3])
                                : z4;
#pragma unroll
                for (int x = 0; x < KO / 4; ++x)
                  rg[x] = valid ? make_float4(vg[4 * x], vg[4 * x + 1], vg[4 * x + 2], vg[4 * x + 3])
                                : z4;
              }
              named_bar_sync(1, 128);
              if (p.bias_partials != nullptr) {  // projected bias gradient: sum_t g~_t
                const int col = et % KO, r0 = (et / KO) * (KO / 2);
#pragma unroll 4
                for (int i = 0; i < KO / 2; ++i) bias_acc += sG[(r0 + i) * (KO + 4) + col];
              }
#pragma unroll 4
              for (int t2 = 0; t2 < kHalf; ++t2) {
                const float gv = sG[t2 * (KO + 4) + oi];
                const float* ar = sA + t2 * (KI + 4) + oj;
                if constexpr (OPT % 4 == 0) {
#pragma unroll
                  for (int x = 0; x < OPT / 4; ++x) {
                    const float4 a4 = reinterpret_cast<const float4*>(ar)[x];
                    acc[4 * x] = fmaf(gv, a4.x, acc[4 * x]);
                    acc[4 * x + 1] = fmaf(gv, a4.y, acc[4 * x + 1]);
                    acc[4 * x + 2] = fmaf(gv, a4.z, acc[4 * x + 2]);
                    acc[4 * x + 3] = fmaf(gv, a4.w, acc[4 * x + 3]);
                  }
                } else {
#pragma unroll
                  for (int x = 0; x < OPT / 2; ++x) {
                    const float2 a2 = reinterpret_cast<const float2*>(ar)[x];
                    acc[2 * x] = fmaf(gv, a2.x, acc[2 * x]);
                    acc[2 * x + 1] = fmaf(gv, a2.y, acc[2 * x + 1]);
                  }
                }
              }
            }
          }
        }
        }                                            // query blocks
        if (!finisher) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&tempty[ab]));
          if (++ab == 2) { ab = 0; aph ^= 1; }
        }
        }                                            // not the tensor-core token path
      }
      if (aborted) break;
      if constexpr (TOKEN) continue;
      float* dst = p.partials + static_cast<int64_t>(ic.slot) * (KO * KI) + et * OPT;
#pragma unroll
      for (int x = 0; x < OPT / 2; ++x)
        reinterpret_cast<float2*>(dst)[x] = make_float2(acc[2 * x], acc[2 * x + 1]);
      if (p.bias_partials != nullptr)
        p.bias_partials[static_cast<int64_t>(ic.slot) * kTileTokens + et] = bias_acc;
    }
  }

  if constexpr (C::kTC) {
    // a U product abandoned after a timeout must finish before TMEM is released
    if (threadIdx.x == 64 && u_pending) mbar_wait(smem_u32(ubar), uph, kDrainTimeoutNs, nullptr);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// out[b, off_m + e] = sum over chunks c (in order) of partials[(m*B + b)*n_chunks + c][e]
// and, for layers with a bias block, out[b, bias_off + i] = sum over chunks and
// row groups (in order) of the items' column sums of g~.
__global__ void reduce_kernel(const ModDesc* __restrict__ mods, int B, int blk, int k_out,
                              int n_chunks, const float* __restrict__ partials,
                              const float* __restrict__ bias_partials, float* __restrict__ out,
                              int64_t ld_out) {
  griddep_wait();
  griddep_launch_dependents();
  const int mb = blockIdx.x;
  const int m = mb / B;
  const int b = mb % B;
  float* dst = out + static_cast<int64_t>(b) * ld_out + mods[m].col_offset;
  const float* src = partials + static_cast<int64_t>(mb) * n_chunks * blk;
  for (int e = threadIdx.x; e < blk; e += blockDim.x) {
    float s = 0.0f;
    for (int c = 0; c < n_chunks; ++c) s += src[static_cast<int64_t>(c) * blk + e];
    dst[e] = s;
  }
  const int64_t boff = mods[m].bias_col_offset;
  if (bias_partials != nullptr && boff >= 0) {
    const float* bsrc = bias_partials + static_cast<int64_t>(mb) * n_chunks * kTileTokens;
    for (int i = threadIdx.x; i < k_out; i += blockDim.x) {
      float s = 0.0f;
      for (int c = 0; c < n_chunks; ++c)
        for (int rg = 0; rg < kTileTokens / k_out; ++rg)
          s += bsrc[static_cast<int64_t>(c) * kTileTokens + rg * k_out + i];
      out[static_cast<int64_t>(b) * ld_out + boff + i] = s;
    }
  }
}

// out[q, b, t] = sum over modules m (in order) of token_partials[m, q, b, t];
// 0 for masked tokens (whose partials may never have been written).
__global__ void token_reduce_kernel(const float* __restrict__ tp, int n_mods, int Q, int B, int T,
                                    const uint8_t* __restrict__ mask, float* __restrict__ out) {
  const int64_t bt = static_cast<int64_t>(B) * T;
  const int64_t n = static_cast<int64_t>(Q) * bt;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i % bt;
    float s = 0.0f;
    for (int m = 0; m < n_mods; ++m) s += tp[static_cast<int64_t>(m) * n + i];
    out[i] = (mask == nullptr || mask[r] != 0) ? s : 0.0f;
  }
}

template <int KI, int KO, bool TOKEN>
cudaError_t launch_project_t(const ProjParams& p, int grid, cudaStream_t s) {
  using C = ProjCfg<KI, KO, TOKEN>;
  static PerDeviceOnce attr;
  const cudaError_t e = smem_attr_once(attr, project_kernel<KI, KO, TOKEN>, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  return launch_dependent(project_kernel<KI, KO, TOKEN>, dim3(grid), dim3(192), C::kSmemBytes, s,
                          p);
}

template <int KI, int KO>
cudaError_t launch_project_mode(bool token, const ProjParams& p, int grid, cudaStream_t s) {
  return token ? launch_project_t<KI, KO, true>(p, grid, s)
               : launch_project_t<KI, KO, false>(p, grid, s);
}

template <int KI, int KO>
constexpr int token_capacity_of() {
  return ProjCfg<KI, KO, true>::kQB;
}

}  // namespace

#define BERGSON_PROJ_DISPATCH(KI_, KO_, EXPR)        \
  if (k_in == KI_ && k_out == KO_) {                 \
    return EXPR;                                     \
  }

cudaError_t launch_project(int k_in, int k_out, bool token, const ProjParams& p, int grid,
                           cudaStream_t s) {
  BERGSON_PROJ_DISPATCH(16, 16, (launch_project_mode<16, 16>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(16, 32, (launch_project_mode<16, 32>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(16, 64, (launch_project_mode<16, 64>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(32, 16, (launch_project_mode<32, 16>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(32, 32, (launch_project_mode<32, 32>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(32, 64, (launch_project_mode<32, 64>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(64, 16, (launch_project_mode<64, 16>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(64, 32, (launch_project_mode<64, 32>(token, p, grid, s)))
  BERGSON_PROJ_DISPATCH(64, 64, (launch_project_mode<64, 64>(token, p, grid, s)))
  return cudaErrorInvalidValue;
}

int token_query_capacity(int k_in, int k_out) {
  BERGSON_PROJ_DISPATCH(16, 16, (token_capacity_of<16, 16>()))
  BERGSON_PROJ_DISPATCH(16, 32, (token_capacity_of<16, 32>()))
  BERGSON_PROJ_DISPATCH(16, 64, (token_capacity_of<16, 64>()))
  BERGSON_PROJ_DISPATCH(32, 16, (token_capacity_of<32, 16>()))
  BERGSON_PROJ_DISPATCH(32, 32, (token_capacity_of<32, 32>()))
  BERGSON_PROJ_DISPATCH(32, 64, (token_capacity_of<32, 64>()))
  BERGSON_PROJ_DISPATCH(64, 16, (token_capacity_of<64, 16>()))
  BERGSON_PROJ_DISPATCH(64, 32, (token_capacity_of<64, 32>()))
  BERGSON_PROJ_DISPATCH(64, 64, (token_capacity_of<64, 64>()))
  return 0;
}

cudaError_t launch_token_reduce(const float* token_partials, int n_mods, int Q, int B, int T,
                                const uint8_t* mask, float* out, cudaStream_t s) {
  const int64_t n = static_cast<int64_t>(Q) * B * T;
  if (n == 0) return cudaSuccess;
  const int64_t blocks = (n + 255) / 256;
  token_reduce_kernel<<<static_cast<unsigned>(blocks < 8192 ? blocks : 8192), 256, 0, s>>>(
      token_partials, n_mods, Q, B, T, mask, out);
  return cudaGetLastError();
}

cudaError_t launch_reduce(const ModDesc* mods, int n_mods, int k_in, int k_out, int B,
                          int n_chunks, const float* partials, const float* bias_partials,
                          float* out, int64_t ld_out, cudaStream_t s) {
  const int blocks = n_mods * B;
  if (blocks == 0) return cudaSuccess;
  const int blk = k_in * k_out;
  return launch_dependent(reduce_kernel, dim3(blocks), dim3(blk < 1024 ? blk : 1024), 0, s, mods,
                          B, blk, k_out, n_chunks, partials, bias_partials, out, ld_out);
}

}  // namespace bergson
