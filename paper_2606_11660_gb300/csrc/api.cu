// Host side of the C ABI declared in include/bergson.h: argument validation,
// workspace layout, TMA descriptor encoding, kernel launches, error mapping.

#include <cudaTypedefs.h>

#include <algorithm>
#include <chrono>
#include <cmath>
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include "bergson.h"
#include "internal.h"

namespace bergson {
namespace {

constexpr int kVersion = 100;                        // 0.1.0
constexpr int kSchedTargetItems = 8192;              // work items per projection launch (target)
// Piece splitting of projection slots.  The planner assumes kPlanCTAs
// persistent CTAs (one per SM of this part; the launch uses the real count).
// A launch is split when its largest slot exceeds kSplitShare of one CTA's
// share of the work, into pieces of about 1/kPiecesPerShare of a share.
constexpr double kSplitShare = 0.4;
constexpr int kPiecesPerShare = 2;
constexpr int kMaxScoreCTAs = 160;                   // upper bound on persistent score CTAs
constexpr int kMaxDevices = 64;
constexpr int kMaxTokenQueries = 256;                // per-token scores: queries per call
constexpr int64_t kPrefixRowsPerTopk = 128;          // prefix pass: 128 * topk store rows
constexpr int64_t kPrefixMinFactor = 8;              // ... only when N >= 8 * prefix
constexpr int64_t kPrefixMinQueries = 129;           // ... and Q > 128 (fewer queries insert
                                                     // too little into their heaps to repay it)

__device__ int g_status_word;                        // device status word (one per device)

thread_local std::string g_last_error;
std::atomic<int> g_inject_status{0};
std::atomic<int> g_inject_count{0};

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

int fail_cuda(cudaError_t e, const char* what) {
  return fail(BERGSON_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

int injected() {
  int n = g_inject_count.load();
  while (n > 0) {
    if (g_inject_count.compare_exchange_weak(n, n - 1)) {
      const int st = g_inject_status.load();
      return fail(st, "injected status %d (test hook)", st);
    }
  }
  return BERGSON_OK;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
bool known_proj_kind(int kind) {
  return kind == BERGSON_PROJ_GAUSSIAN || kind == BERGSON_PROJ_IDENTITY ||
         kind == BERGSON_PROJ_RADEMACHER || kind == BERGSON_PROJ_UNIFORM;
}
size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Makes the device owning `ptr` current for the lifetime of the guard.
struct DeviceGuard {
  int prev = -1;
  int dev = -1;
  cudaError_t err = cudaSuccess;
  explicit DeviceGuard(const void* ptr) {
    cudaPointerAttributes at;
    err = cudaPointerGetAttributes(&at, ptr);
    if (err != cudaSuccess) return;
    if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) {
      err = cudaErrorInvalidDevicePointer;
      return;
    }
    err = cudaGetDevice(&prev);
    if (err != cudaSuccess) return;
    dev = at.device;
    if (dev != prev) err = cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    if (prev >= 0 && dev >= 0 && prev != dev) cudaSetDevice(prev);
  }
};

int* status_word(int dev) {
  static std::mutex mu;
  static int* ptrs[kMaxDevices] = {};
  std::lock_guard<std::mutex> lk(mu);
  if (dev < 0 || dev >= kMaxDevices) return nullptr;
  if (ptrs[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    ptrs[dev] = static_cast<int*>(p);
  }
  return ptrs[dev];
}

int sm_count(int dev) {
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

bool valid_k(int64_t k) { return k == 16 || k == 32 || k == 64; }

// ----------------------------------------------------------- project_grads

struct Group {
  int k_in = 0, k_out = 0;
  std::vector<int> layers;     // indices into the caller's array, largest unit first
  std::vector<std::pair<int, int>> units;   // (first position in layers, count): layers that
                                            // read one A tensor, scheduled side by side
  int first_mod = 0;           // index of its first ModDesc in workspace
  int n_chunks = 0, tpc = 0;
  int n_slots = 0;             // layers * B * n_chunks partials
  int n_items = 0;             // work items of the launch (= n_slots without a table)
  bool has_bias = false;
  size_t partial_off = 0;
  size_t bias_off = 0;
  std::vector<WorkItem> table; // work table (empty: item i is fused slot i)
  int n_split = 0;             // slots cut into pieces
  int64_t piece_floats = 0;    // token projections stored by pieces
  size_t table_off = 0, split_cnt_off = 0, piece_off = 0;
};

struct ProjLayout {
  int n_tiles = 0;
  std::vector<Group> groups;
  std::vector<int> mod_slot;   // layer index -> ModDesc slot
  std::vector<uint8_t> shared; // layer index -> 1 if another layer of its group reads its A
  size_t mods_off = 0, segs_off = 0, ctr_off = 0, tv_off = 0;
  size_t token_off = 0;        // per-token score partials (token mode)
  std::vector<size_t> pin_off, pout_off;
  size_t total = 0;
};

int validate_layers(const bergson_layer* layers, int n_layers, int64_t B, int64_t T) {
  if (layers == nullptr) return fail(BERGSON_EINVAL, "layers is NULL");
  if (n_layers < 1 || n_layers > 16384)
    return fail(BERGSON_EINVAL, "n_layers must be in [1, 16384] (got %d)", n_layers);
  if (B < 0 || T < 0) return fail(BERGSON_EINVAL, "B and T must be >= 0 (B=%lld T=%lld)",
                                  (long long)B, (long long)T);
  if (B > (1ll << 30) || T > (1ll << 30) || B * T > (1ll << 37))
    return fail(BERGSON_EUNSUPPORTED, "B*T too large");
  for (int i = 0; i < n_layers; ++i) {
    const bergson_layer& L = layers[i];
    if ((L.flags & ~BERGSON_LAYER_BIAS) != 0)
      return fail(BERGSON_EINVAL, "layer %d: unknown flags 0x%x", i, L.flags);
    if ((L.flags & BERGSON_LAYER_BIAS) && L.bias_col_offset < 0)
      return fail(BERGSON_EINVAL, "layer %d: negative bias_col_offset", i);
    if (L.d_in < 8 || L.d_out < 8 || L.d_in > (1 << 24) || L.d_out > (1 << 24))
      return fail(BERGSON_EINVAL, "layer %d: d_in/d_out must be in [8, 2^24]", i);
    if (L.d_in % 8 != 0 || L.d_out % 8 != 0)
      return fail(BERGSON_EALIGN, "layer %d: d_in and d_out must be multiples of 8", i);
    if (!known_proj_kind(L.proj_kind))
      return fail(BERGSON_EINVAL, "layer %d: unknown proj_kind %d", i, L.proj_kind);
    if (!valid_k(L.k_in) || !valid_k(L.k_out))
      return fail(BERGSON_EUNSUPPORTED, "layer %d: k_in and k_out must be 16, 32 or 64", i);
    if (L.proj_kind == BERGSON_PROJ_IDENTITY && (L.k_in != L.d_in || L.k_out != L.d_out))
      return fail(BERGSON_EINVAL, "layer %d: identity projection needs k == d", i);
    if ((L.r == nullptr) != (L.c == nullptr))
      return fail(BERGSON_EINVAL, "layer %d: r and c must both be given or both be NULL", i);
    if ((L.r && !aligned(L.r, 4)) || (L.c && !aligned(L.c, 4)))
      return fail(BERGSON_EALIGN, "layer %d: r/c must be 4-byte aligned", i);
    if (B * T > 0) {
      if (L.A == nullptr || L.G == nullptr) return fail(BERGSON_EINVAL, "layer %d: A or G is NULL", i);
      if (!aligned(L.A, 16) || !aligned(L.G, 16))
        return fail(BERGSON_EALIGN, "layer %d: A and G must be 16-byte aligned", i);
    }
    if (L.out_col_offset < 0) return fail(BERGSON_EINVAL, "layer %d: negative out_col_offset", i);
  }
  return BERGSON_OK;
}

int validate_blocks(const bergson_layer* layers, int n_layers, int64_t ld_out,
                    bool with_bias = true) {
  std::vector<std::pair<int64_t, int64_t>> blk;
  for (int i = 0; i < n_layers; ++i) {
    const int64_t a = layers[i].out_col_offset;
    const int64_t e = a + layers[i].k_in * layers[i].k_out;
    if (e > ld_out)
      return fail(BERGSON_EINVAL, "layer %d: block [%lld, %lld) exceeds ld_out=%lld", i,
                  (long long)a, (long long)e, (long long)ld_out);
    blk.emplace_back(a, e);
    if (with_bias && (layers[i].flags & BERGSON_LAYER_BIAS)) {
      const int64_t ba = layers[i].bias_col_offset, be = ba + layers[i].k_out;
      if (be > ld_out)
        return fail(BERGSON_EINVAL, "layer %d: bias block [%lld, %lld) exceeds ld_out=%lld", i,
                    (long long)ba, (long long)be, (long long)ld_out);
      blk.emplace_back(ba, be);
    }
  }
  std::sort(blk.begin(), blk.end());
  for (size_t i = 1; i < blk.size(); ++i)
    if (blk[i].first < blk[i - 1].second)
      return fail(BERGSON_EINVAL, "output column blocks overlap at column %lld",
                  (long long)blk[i].first);
  return BERGSON_OK;
}

int chunks_of(int64_t d) { return static_cast<int>((d + kChunk - 1) / kChunk); }

// Builds a group's work table when its slots need more than "item i is slot i":
// (1) cutting: when the launch is too coarse for the SMs to finish together
// (largest slot above kSplitShare of one CTA's share), large slots are cut
// into pieces (split = allowed only in projection mode); (2) shared inputs:
// the items of a unit's layers for the same example and tiles are listed next
// to each other (A-side pieces too), so the scheduler starts them together.
// Cost unit: one 64-column chunk of one tile; the table runs largest first.
void plan_work(const bergson_layer* layers, int64_t B, int n_tiles, Group& g, bool allow_split) {
  if (g.n_slots == 0) return;
  int64_t total = 0, max_slot = 0;
  for (int li : g.layers) {
    const int64_t c = chunks_of(layers[li].d_in) + chunks_of(layers[li].d_out);
    total += c * n_tiles * B;
    max_slot = std::max<int64_t>(max_slot, c * std::min(g.tpc, n_tiles));
  }
  const double share = static_cast<double>(total) / kPlanCTAs;
  const bool split = allow_split && static_cast<double>(max_slot) > kSplitShare * share;
  bool shared = false;
  for (const auto& u : g.units) shared = shared || u.second > 1;
  if (!split && !shared) return;
  const double target = share / kPiecesPerShare;
  // A piece stores and its slot's finisher reloads 4k fp32 bytes per token,
  // against 128 bytes per token and chunk streamed: pieces of at least 2k
  // chunks keep that under 1/32 of the piece's traffic.  (Fewer, larger
  // pieces measured faster: Llama-8B-shaped block 0.790 ms at a quarter of a
  // share per piece, 0.770 ms at half.)
  auto pieces = [&](int ch, int k) {
    const int n = static_cast<int>(std::ceil(static_cast<double>(ch) * g.tpc / target));
    return std::max(1, std::min(n, ch / (2 * k)));
  };
  struct Entry {
    WorkItem w;
    int64_t key;
  };
  std::vector<Entry> es;
  int64_t base = 0;
  int n_split = 0;
  for (const auto& u : g.units) {
    const int m0 = u.first, cnt = u.second;
    const int ca = chunks_of(layers[g.layers[m0]].d_in);
    bool cut = false;
    int64_t worst = 0;
    std::vector<int> cg(cnt), n_g(cnt, 0);
    for (int j = 0; j < cnt; ++j) {
      cg[j] = chunks_of(layers[g.layers[m0 + j]].d_out);
      worst = std::max<int64_t>(worst, ca + cg[j]);
      cut = cut || (split && static_cast<double>(ca + cg[j]) * g.tpc > target);
    }
    const int n_a = cut ? pieces(ca, g.k_in) : 0;
    if (cut)
      for (int j = 0; j < cnt; ++j) n_g[j] = pieces(cg[j], g.k_out);
    std::vector<int> sid(cnt);
    std::vector<int64_t> sbase(cnt);
    for (int64_t b = 0; b < B; ++b) {
      for (int c = 0; c < g.n_chunks; ++c) {
        const int tiles = std::min(n_tiles, (c + 1) * g.tpc) - c * g.tpc;
        auto slot_of = [&](int j) {
          return static_cast<int>((static_cast<int64_t>(m0 + j) * B + b) * g.n_chunks + c);
        };
        if (!cut) {
          for (int j = 0; j < cnt; ++j)
            es.push_back({WorkItem{slot_of(j), 0, 0, 0, 0, 0, 0, 0, 0}, worst * tiles});
          continue;
        }
        for (int j = 0; j < cnt; ++j) {
          sid[j] = n_split++;
          sbase[j] = base;
          base += (int64_t{n_a} * g.k_in + int64_t{n_g[j]} * g.k_out) * g.tpc * kTileTokens;
        }
        for (int q = 0; q < n_a; ++q) {             // A side: the unit's layers together
          const int c0 = static_cast<int>(static_cast<int64_t>(q) * ca / n_a);
          const int c1 = static_cast<int>(static_cast<int64_t>(q + 1) * ca / n_a);
          for (int j = 0; j < cnt; ++j)
            es.push_back({WorkItem{slot_of(j), 1, c0, c1, sid[j], n_a, n_g[j], q, sbase[j]},
                          int64_t{c1 - c0} * tiles});
        }
        for (int j = 0; j < cnt; ++j) {
          for (int q = 0; q < n_g[j]; ++q) {
            const int c0 = static_cast<int>(static_cast<int64_t>(q) * cg[j] / n_g[j]);
            const int c1 = static_cast<int>(static_cast<int64_t>(q + 1) * cg[j] / n_g[j]);
            es.push_back({WorkItem{slot_of(j), 2, c0, c1, sid[j], n_a, n_g[j], q, sbase[j]},
                          int64_t{c1 - c0} * tiles});
          }
        }
      }
    }
  }
  std::stable_sort(es.begin(), es.end(),
                   [](const Entry& x, const Entry& y) { return x.key > y.key; });
  g.table.resize(es.size());
  for (size_t i = 0; i < es.size(); ++i) g.table[i] = es[i].w;
  g.n_items = static_cast<int>(es.size());
  g.n_split = n_split;
  g.piece_floats = base;
}

// n_queries > 0 lays out per-token score partials [n_layers, n_queries, B, T]
// instead of per-item projection partials.
ProjLayout plan_project(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                        int64_t n_queries = 0) {
  ProjLayout L;
  L.n_tiles = static_cast<int>((T + kTileTokens - 1) / kTileTokens);
  L.mod_slot.assign(n_layers, 0);
  L.shared.assign(n_layers, 0);
  for (int i = 0; i < n_layers; ++i) {
    const int ki = static_cast<int>(layers[i].k_in), ko = static_cast<int>(layers[i].k_out);
    auto it = std::find_if(L.groups.begin(), L.groups.end(),
                           [&](const Group& g) { return g.k_in == ki && g.k_out == ko; });
    if (it == L.groups.end()) {
      L.groups.push_back(Group());
      it = L.groups.end() - 1;
      it->k_in = ki;
      it->k_out = ko;
    }
    it->layers.push_back(i);
    if (layers[i].flags & BERGSON_LAYER_BIAS) it->has_bias = true;
  }
  int slot = 0;
  for (Group& g : L.groups) {
    // Units: layers that read the same A tensor (same pointer and d_in, e.g. a
    // gate and an up projection) are scheduled side by side, so that the second
    // reader of an A tile can find it in L2 (the saving is small: the lines
    // are streamed with evict_first, and L2 turns over in tens of
    // microseconds; keeping them measured slower).  Largest unit first: the scheduler
    // hands items out in order, so the last items a launch waits on are the
    // cheapest ones (longest processing time first); a tile costs d_in + d_out.
    std::vector<std::vector<int>> units;
    for (int li : g.layers) {
      auto u = std::find_if(units.begin(), units.end(), [&](const std::vector<int>& v) {
        return layers[li].A != nullptr && layers[v[0]].A == layers[li].A &&
               layers[v[0]].d_in == layers[li].d_in;
      });
      if (u == units.end()) units.push_back({li});
      else u->push_back(li);
    }
    auto unit_cost = [&](const std::vector<int>& v) {
      int64_t c = 0;
      for (int li : v) c = std::max<int64_t>(c, layers[li].d_in + layers[li].d_out);
      return c;
    };
    std::stable_sort(units.begin(), units.end(),
                     [&](const std::vector<int>& x, const std::vector<int>& y) {
                       return unit_cost(x) > unit_cost(y);
                     });
    g.layers.clear();
    g.units.clear();
    for (const auto& v : units) {
      g.units.emplace_back(static_cast<int>(g.layers.size()), static_cast<int>(v.size()));
      g.layers.insert(g.layers.end(), v.begin(), v.end());
      if (v.size() > 1)
        for (int li : v) L.shared[li] = 1;
    }
    g.first_mod = slot;
    for (int li : g.layers) L.mod_slot[li] = slot++;
    const int nt_per_group = (g.k_in + g.k_out <= 32) ? 4 : ((g.k_in + g.k_out <= 64) ? 2 : 1);
    const int64_t mb = static_cast<int64_t>(g.layers.size()) * B;
    if (L.n_tiles == 0 || mb == 0) {
      g.n_chunks = 0;
      g.tpc = 0;
      g.n_items = 0;
      continue;
    }
    const int max_chunks = (L.n_tiles + nt_per_group - 1) / nt_per_group;
    int64_t want = (kSchedTargetItems + mb - 1) / mb;
    if (want > max_chunks) want = max_chunks;
    if (want < 1) want = 1;
    int tpc = static_cast<int>((L.n_tiles + want - 1) / want);
    tpc = (tpc + nt_per_group - 1) / nt_per_group * nt_per_group;
    g.tpc = tpc;
    g.n_chunks = (L.n_tiles + tpc - 1) / tpc;
    g.n_slots = static_cast<int>(mb * g.n_chunks);
    g.n_items = g.n_slots;
    plan_work(layers, B, L.n_tiles, g, n_queries == 0);
  }
  size_t off = 0;
  L.mods_off = off;
  off += round_up(sizeof(ModDesc) * n_layers, 256);
  L.segs_off = off;
  off += round_up(sizeof(PrepSeg) * 2 * n_layers, 256);
  L.ctr_off = off;
  off += round_up(sizeof(int) * 32 * L.groups.size(), 256);
  for (Group& g : L.groups) {
    if (g.table.empty()) continue;
    g.table_off = off;
    off += round_up(sizeof(WorkItem) * g.table.size(), 256);
    g.split_cnt_off = off;
    off += round_up(sizeof(int) * g.n_split, 256);
  }
  L.tv_off = off;        // everything before this offset is host-staged each call
  off += round_up(static_cast<size_t>(B) * L.n_tiles, 256);
  L.pin_off.resize(n_layers);
  L.pout_off.resize(n_layers);
  for (int i = 0; i < n_layers; ++i) {
    L.pin_off[i] = off;
    off += round_up(2 * layers[i].k_in * layers[i].d_in * sizeof(__nv_bfloat16), 256);
    L.pout_off[i] = off;
    off += round_up(2 * layers[i].k_out * layers[i].d_out * sizeof(__nv_bfloat16), 256);
  }
  if (n_queries > 0) {
    const size_t per_mod = static_cast<size_t>(n_queries) * B * T * sizeof(float);
    L.token_off = off;
    for (Group& g : L.groups) g.partial_off = off + per_mod * g.first_mod;
    off += round_up(per_mod * n_layers, 256);
  } else {
    for (Group& g : L.groups) {
      g.partial_off = off;
      off += round_up(static_cast<size_t>(g.n_slots) * g.k_in * g.k_out * sizeof(float), 256);
      if (g.has_bias) {
        g.bias_off = off;
        off += round_up(static_cast<size_t>(g.n_slots) * kTileTokens * sizeof(float), 256);
      }
      if (g.piece_floats > 0) {
        g.piece_off = off;
        off += round_up(static_cast<size_t>(g.piece_floats) * sizeof(float), 256);
      }
    }
  }
  L.total = off;
  return L;
}

CUresult encode_act(CUtensorMap* tm, const void* ptr, int64_t d, int64_t T, int64_t B) {
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T),
                        static_cast<cuuint64_t>(B)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d * 2), static_cast<cuuint64_t>(T * d * 2)};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(kChunk), 32, 1};   // 32-token slices
  cuuint32_t es[3] = {1, 1, 1};
  return encode_fn()(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

CUresult encode_2d(CUtensorMap* tm, CUtensorMapDataType dt, const void* ptr, int64_t inner,
                   int64_t outer, int64_t row_bytes, int box_inner, int box_outer) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(row_bytes)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_outer)};
  cuuint32_t es[2] = {1, 1};
  return encode_fn()(tm, dt, 2, const_cast<void*>(ptr), dims, strides, box, es,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// ------------------------------------------------------------- score_topk

struct ScoreLayout {
  int qt = 1;
  size_t qh_off = 0, heap_off = 0, pace_off = 0, total = 0;
};

ScoreLayout plan_score(int64_t K, int64_t Q, int64_t topk) {
  ScoreLayout L;
  // Up to 128 queries: one tile per CTA, single-CTA kernel.  129..256: one
  // tile per CTA of a pair.  More: two tiles per CTA of a pair.
  L.qt = Q > 2 * kScoreQT ? 2 : 1;
  L.qh_off = 0;
  L.heap_off = round_up(static_cast<size_t>(Q) * K * sizeof(__half), 256);
  L.pace_off = L.heap_off + round_up(static_cast<size_t>(kMaxScoreCTAs) * topk * L.qt * kScoreQT *
                                         sizeof(unsigned long long),
                                     256);
  // the pair kernel's pacing words, one per CTA (timing only: never initialised)
  L.total = L.pace_off + round_up(static_cast<size_t>(kMaxScoreCTAs) * sizeof(unsigned long long),
                                  256);
  return L;
}

// A tag per pair-kernel launch for its pacing words (never 0), so that words
// left by an earlier launch on the same workspace are told apart.
unsigned int next_pace_tag() {
  static std::atomic<unsigned int> counter{0};
  unsigned int t = counter.fetch_add(1, std::memory_order_relaxed) + 1;
  if (t == 0) t = counter.fetch_add(1, std::memory_order_relaxed) + 1;
  return t;
}

// One score-kernel launch and the merge that follows it.
struct ScoreLaunch {
  int pass = 0;            // index of the pass over query groups
  int stage = 1;           // 0 = prefix threshold pass, 1 = full pass
  int64_t rows = 0;        // store rows this launch scores (a prefix, or N)
  int n_qg = 0;            // query groups of this pass
  int qg_base = 0;         // first query group of this pass
  int cpg = 0;             // CTAs per query group
  int grid = 0;            // n_qg * cpg
  int n_tiles = 0;         // 256-row store tiles of `rows`
  int q_begin = 0, q_end = 0;   // queries this launch's merge writes
};

struct ScoreLaunchPlan {
  bool pair = false;       // clusters of two CTAs (more than 128 queries)
  int qt = 1;              // 128-query tiles per CTA
  int gsize = 0;           // queries per query group
  int ctas = 0;            // resident CTAs the launches are sized for
  bool use_prefix = false;
  std::vector<ScoreLaunch> launches;
};

// Launch sequence of bergson_score_topk for `ctas` resident CTAs (for the pair
// kernel: 2 x its co-resident clusters).  Pure host logic.
ScoreLaunchPlan plan_score_launches(int64_t N, int64_t Q, int64_t topk, int ctas,
                                    bool allow_prefix = true) {
  ScoreLaunchPlan P;
  const ScoreLayout L = plan_score(0, Q, topk);
  P.pair = Q >= kPairMinQueries;
  P.qt = L.qt;
  P.gsize = L.qt * kScoreQT;
  int sms = std::max(1, std::min(ctas, kMaxScoreCTAs));
  if (P.pair) sms &= ~1;
  P.ctas = sms;
  if (Q <= 0 || (P.pair && sms < 2)) return P;
  int n_qg_total = static_cast<int>((Q + P.gsize - 1) / P.gsize);
  if (P.pair) n_qg_total = (n_qg_total + 1) & ~1;   // whole pairs of query groups
  // Prefix pass (large stores only): the exact top-k of the first `prefix` rows
  // lands in the outputs, and its k-th score seeds the full pass's threshold.
  const int64_t prefix_rows = round_up(static_cast<size_t>(kPrefixRowsPerTopk * topk), kScoreBN);
  P.use_prefix = allow_prefix && N >= kPrefixMinFactor * prefix_rows && Q >= kPrefixMinQueries;
  for (int pass = 0; pass < n_qg_total; pass += sms) {
    const int n_qg = std::min(sms, n_qg_total - pass);
    // The prefix is cut to whole rounds of store tiles over the CTAs of a
    // query group (a partial second round would cost as much as a full one).
    const int64_t round_rows = static_cast<int64_t>(sms / n_qg) * kScoreBN;
    const int64_t prefix = prefix_rows > round_rows ? prefix_rows / round_rows * round_rows
                                                    : prefix_rows;
    for (int stage = P.use_prefix ? 0 : 1; stage < 2; ++stage) {
      ScoreLaunch l;
      l.pass = pass;
      l.stage = stage;
      l.rows = stage == 0 ? prefix : N;
      l.n_qg = n_qg;
      l.qg_base = pass;
      l.n_tiles = static_cast<int>((l.rows + kScoreBN - 1) / kScoreBN);
      l.cpg = std::max(1, std::min(sms / n_qg, l.n_tiles));
      l.grid = n_qg * l.cpg;
      l.q_begin = pass * P.gsize;
      l.q_end = static_cast<int>(std::min<int64_t>(Q, static_cast<int64_t>(pass + n_qg) * P.gsize));
      P.launches.push_back(l);
    }
  }
  return P;
}

// Size rules shared by the scoring calls and their workspace query.
int validate_score_sizes(int64_t N, int64_t K, int64_t Q, int64_t topk) {
  if (N < 1 || N >= (1ll << 31)) return fail(BERGSON_EINVAL, "N must be in [1, 2^31)");
  if (K < 8 || K > (1ll << 24)) return fail(BERGSON_EINVAL, "K must be in [8, 2^24]");
  if (K % 8 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 8");
  if (Q < 0 || Q > (1ll << 24)) return fail(BERGSON_EINVAL, "Q must be in [0, 2^24]");
  if (topk < 1 || topk > kMaxTopk)
    return fail(BERGSON_EUNSUPPORTED, "topk must be in [1, %d]", kMaxTopk);
  if (topk > N) return fail(BERGSON_EINVAL, "topk (%lld) > N (%lld)", (long long)topk, (long long)N);
  return BERGSON_OK;
}

int validate_score(const void* store, int64_t N, int64_t K, int64_t ld_store, const float* queries,
                   int64_t Q, int64_t ld_q, int64_t topk) {
  const int st = validate_score_sizes(N, K, Q, topk);
  if (st != BERGSON_OK) return st;
  if (ld_store < K || ld_store % 8 != 0)
    return fail(ld_store < K ? BERGSON_EINVAL : BERGSON_EALIGN,
                "ld_store must be >= K and a multiple of 8");
  if (store == nullptr) return fail(BERGSON_EINVAL, "store is NULL");
  if (!aligned(store, 16)) return fail(BERGSON_EALIGN, "store must be 16-byte aligned");
  if (Q > 0) {
    if (queries == nullptr) return fail(BERGSON_EINVAL, "queries is NULL");
    if (!aligned(queries, 4)) return fail(BERGSON_EALIGN, "queries must be 4-byte aligned");
    if (ld_q < K) return fail(BERGSON_EINVAL, "ld_q must be >= K");
  }
  return BERGSON_OK;
}

}  // namespace

int record_error(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

CUresult encode_tmap_2d(CUtensorMap* tm, CUtensorMapDataType dt, const void* ptr, int64_t inner,
                        int64_t outer, int64_t row_bytes, int box_inner, int box_outer) {
  if (encode_fn() == nullptr) return CUDA_ERROR_NOT_SUPPORTED;
  return encode_2d(tm, dt, ptr, inner, outer, row_bytes, box_inner, box_outer);
}

}  // namespace bergson

using namespace bergson;

extern "C" {

int bergson_version(void) { return kVersion; }

void bergson_module_seeds(uint64_t base_seed, int64_t module_index, uint64_t* seed_in,
                          uint64_t* seed_out) {
  auto mix = [](uint64_t x) {
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
  };
  const uint64_t m = static_cast<uint64_t>(module_index);
  if (seed_in != nullptr) *seed_in = mix(base_seed ^ (2 * m));
  if (seed_out != nullptr) *seed_out = mix(base_seed ^ (2 * m + 1));
}

const char* bergson_last_error(void) { return g_last_error.c_str(); }

int bergson_debug_project_plan(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                               int64_t* n_slots, int64_t* n_items, int64_t* n_pieces,
                               int64_t* n_shared) {
  const int st = validate_layers(layers, n_layers, B, T);
  if (st != BERGSON_OK) return st;
  const ProjLayout L = plan_project(layers, n_layers, B, T);
  int64_t slots = 0, items = 0, pieces = 0;
  for (const Group& g : L.groups) {
    slots += g.n_slots;
    items += g.n_items;
    for (const WorkItem& w : g.table) pieces += w.side != 0;
  }
  if (n_slots != nullptr) *n_slots = slots;
  if (n_items != nullptr) *n_items = items;
  if (n_pieces != nullptr) *n_pieces = pieces;
  if (n_shared != nullptr) {
    int64_t sh = 0;
    for (uint8_t f : L.shared) sh += f;
    *n_shared = sh;
  }
  return BERGSON_OK;
}

int bergson_debug_score_plan(int64_t N, int64_t K, int64_t Q, int64_t topk, int ctas,
                             int64_t* out, int max_launches, int* n_launches) {
  if (n_launches == nullptr) return fail(BERGSON_EINVAL, "n_launches is NULL");
  const int st = validate_score_sizes(N, K, Q, topk);
  if (st != BERGSON_OK) return st;
  if (ctas < 1) return fail(BERGSON_EINVAL, "ctas must be >= 1");
  const ScoreLaunchPlan P = plan_score_launches(N, Q, topk, ctas);
  *n_launches = static_cast<int>(P.launches.size());
  const int n = out == nullptr ? 0 : std::min(max_launches, *n_launches);
  for (int i = 0; i < n; ++i) {
    const ScoreLaunch& l = P.launches[i];
    const int64_t row[12] = {l.pass, l.stage, l.rows, l.n_qg, l.qg_base, l.cpg,
                             l.grid, l.n_tiles, l.q_begin, l.q_end, P.pair ? 1 : 0, P.qt};
    for (int c = 0; c < 12; ++c) out[static_cast<int64_t>(i) * 12 + c] = row[c];
  }
  return BERGSON_OK;
}

int bergson_debug_xgemm_plan(int64_t B, int64_t Q, int64_t K, int64_t* out, int n_out) {
  if (out == nullptr || n_out < 19) return fail(BERGSON_EINVAL, "out needs room for 19 values");
  if (B < 1 || B > (1 << 20) || Q < 1 || Q > (1 << 24) || K < 4 || K > (1 << 26) || K % 4 != 0)
    return fail(BERGSON_EINVAL, "invalid sizes for the skinny-product plan");
  const XGemmPlan pl = xgemm_plan(B, Q, K);
  const int64_t v[19] = {pl.n_pad, pl.n_ntiles, pl.n_mtiles, pl.steps, pl.S, pl.stages,
                         pl.n_chunks, pl.pair ? 1 : 0, pl.n_buf, pl.y_rows, pl.tmem_cols,
                         static_cast<int64_t>(pl.xnorm_off), static_cast<int64_t>(pl.ynorm_off),
                         static_cast<int64_t>(pl.partial_off), static_cast<int64_t>(pl.xh_off),
                         static_cast<int64_t>(pl.xl_off), static_cast<int64_t>(pl.total),
                         pl.a_base, pl.a_slots};
  for (int i = 0; i < 19; ++i) out[i] = v[i];
  return BERGSON_OK;
}

int bergson_debug_attr_once(int n_threads, int n_devices, int fail_device, int64_t* set_calls,
                            int* failures) {
  if (n_threads < 1 || n_threads > 64 || n_devices < 1 || n_devices > 64)
    return fail(BERGSON_EINVAL, "n_threads and n_devices must be in [1, 64]");
  if (set_calls == nullptr || failures == nullptr)
    return fail(BERGSON_EINVAL, "set_calls or failures is NULL");
  PerDeviceOnce once;
  std::vector<std::atomic<int64_t>> calls(n_devices);
  for (auto& c : calls) c.store(0);
  std::atomic<int> fails{0}, ready{0};
  std::atomic<bool> go{false};
  auto body = [&](int t) {
    ready.fetch_add(1);
    while (!go.load()) std::this_thread::yield();
    for (int rep = 0; rep < 3; ++rep) {
      for (int j = 0; j < n_devices; ++j) {
        const int dev = (j + t) % n_devices;
        const cudaError_t e = once.ensure(dev, [&] {
          // A slow setting widens the window in which other threads arrive.
          std::this_thread::sleep_for(std::chrono::milliseconds(2));
          const int64_t n = calls[dev].fetch_add(1);
          return dev == fail_device && n == 0 ? cudaErrorInvalidValue : cudaSuccess;
        });
        if (e != cudaSuccess) fails.fetch_add(1);
      }
    }
  };
  std::vector<std::thread> th;
  for (int t = 0; t < n_threads; ++t) th.emplace_back(body, t);
  while (ready.load() < n_threads) std::this_thread::yield();
  go.store(true);
  for (auto& x : th) x.join();
  for (int d = 0; d < n_devices; ++d) set_calls[d] = calls[d].load();
  *failures = fails.load();
  return BERGSON_OK;
}

void bergson_debug_inject_status(int status, int count) {
  g_inject_status.store(status);
  g_inject_count.store(count > 0 ? count : 0);
}

int bergson_project_grads_workspace(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                                    size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  int st = validate_layers(layers, n_layers, B, T);
  if (st != BERGSON_OK) return st;
  *ws_bytes = plan_project(layers, n_layers, B, T).total;
  return BERGSON_OK;
}

// Projection mode (n_queries == 0): out = fp32 [B, ld_out] projected gradients.
// Token mode (n_queries > 0): out = fp32 [n_queries, B, T] per-token scores
// against queries [n_queries, ld_q] laid out like projection rows.
static int run_projection(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                          const uint8_t* mask, float* out, int64_t ld_out, const float* queries,
                          int64_t n_queries, int64_t ld_q, void* workspace, size_t ws_bytes,
                          void* stream) {
  const bool token = n_queries > 0;
  int st = validate_layers(layers, n_layers, B, T);
  if (st != BERGSON_OK) return st;
  if (token) {
    if (n_queries > kMaxTokenQueries)
      return fail(BERGSON_EUNSUPPORTED, "at most %d queries per call", kMaxTokenQueries);
    if (ld_q < 0) return fail(BERGSON_EINVAL, "ld_q must be >= 0");
    st = validate_blocks(layers, n_layers, ld_q, false);
    if (st != BERGSON_OK) return st;
    if (queries == nullptr) return fail(BERGSON_EINVAL, "queries is NULL");
    if (!aligned(queries, 4)) return fail(BERGSON_EALIGN, "queries must be 4-byte aligned");
    if (B * T > 0 && out == nullptr) return fail(BERGSON_EINVAL, "out is NULL");
  } else {
    if (ld_out < 0) return fail(BERGSON_EINVAL, "ld_out must be >= 0");
    st = validate_blocks(layers, n_layers, ld_out);
    if (st != BERGSON_OK) return st;
    if (B > 0 && out == nullptr) return fail(BERGSON_EINVAL, "out is NULL");
  }
  if (out != nullptr && !aligned(out, 4)) return fail(BERGSON_EALIGN, "out must be 4-byte aligned");
  const ProjLayout L = plan_project(layers, n_layers, B, T, token ? n_queries : 0);
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < L.total)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, L.total);
  if ((st = injected()) != BERGSON_OK) return st;
  if (B == 0 || (token && T == 0)) return BERGSON_OK;

  DeviceGuard dg(workspace);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "workspace device lookup");
  if (T > 0 && encode_fn() == nullptr)
    return fail(BERGSON_ECUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
  int* status = status_word(dg.dev);
  if (status == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);

  // Host-built records: module descriptors, projection segments, zeroed counters.
  std::vector<uint8_t> staging(L.tv_off, 0);
  ModDesc* mods = reinterpret_cast<ModDesc*>(staging.data() + L.mods_off);
  PrepSeg* segs = reinterpret_cast<PrepSeg*>(staging.data() + L.segs_off);
  int64_t max_pairs = 0;
  for (int i = 0; i < n_layers; ++i) {
    const bergson_layer& ly = layers[i];
    ModDesc& md = mods[L.mod_slot[i]];
    md.d_in = static_cast<int32_t>(ly.d_in);
    md.d_out = static_cast<int32_t>(ly.d_out);
    md.col_offset = ly.out_col_offset;
    md.bias_col_offset = (ly.flags & BERGSON_LAYER_BIAS) ? ly.bias_col_offset : -1;
    __nv_bfloat16* pin = reinterpret_cast<__nv_bfloat16*>(ws + L.pin_off[i]);
    __nv_bfloat16* pout = reinterpret_cast<__nv_bfloat16*>(ws + L.pout_off[i]);
    if (T > 0) {
      CUresult r1 = encode_act(&md.tmA, ly.A, ly.d_in, T, B);
      CUresult r2 = encode_act(&md.tmG, ly.G, ly.d_out, T, B);
      CUresult r3 = encode_2d(&md.tmPin, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, pin, ly.d_in,
                              2 * ly.k_in, ly.d_in * 2, kChunk, static_cast<int>(2 * ly.k_in));
      CUresult r4 = encode_2d(&md.tmPout, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, pout, ly.d_out,
                              2 * ly.k_out, ly.d_out * 2, kChunk, static_cast<int>(2 * ly.k_out));
      if (r1 != CUDA_SUCCESS || r2 != CUDA_SUCCESS || r3 != CUDA_SUCCESS || r4 != CUDA_SUCCESS)
        return fail(BERGSON_ECUDA, "layer %d: tensor map encoding failed (%d %d %d %d)", i,
                    (int)r1, (int)r2, (int)r3, (int)r4);
    }
    PrepSeg& si = segs[2 * i];
    si.seed = ly.seed_in;
    si.moment = ly.c;
    si.dst = pin;
    si.begin = 0;
    si.d = static_cast<int32_t>(ly.d_in);
    si.k = static_cast<int32_t>(ly.k_in);
    si.kind = ly.proj_kind;
    max_pairs = std::max<int64_t>(max_pairs, ly.d_in * ly.k_in / 2);
    PrepSeg& so = segs[2 * i + 1];
    so.seed = ly.seed_out;
    so.moment = ly.r;
    so.dst = pout;
    so.begin = 0;
    so.d = static_cast<int32_t>(ly.d_out);
    so.k = static_cast<int32_t>(ly.k_out);
    so.kind = ly.proj_kind;
    max_pairs = std::max<int64_t>(max_pairs, ly.d_out * ly.k_out / 2);
  }
  for (const Group& g : L.groups)
    if (!g.table.empty())
      std::memcpy(staging.data() + g.table_off, g.table.data(), sizeof(WorkItem) * g.table.size());
  cudaError_t e = cudaMemcpyAsync(ws, staging.data(), staging.size(), cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return fail_cuda(e, "staging copy");
  const ModDesc* mods_dev = reinterpret_cast<const ModDesc*>(ws + L.mods_off);
  const bool need_tiles = T > 0;
  // Tile flags first, then P' right before the projection kernel, which is
  // launched as its dependent and sets itself up while P' is generated.
  uint8_t* tile_valid = nullptr;
  if (mask != nullptr && need_tiles) {
    tile_valid = ws + L.tv_off;
    e = launch_tile_valid(mask, static_cast<int>(B), static_cast<int>(T), L.n_tiles, tile_valid, s);
    if (e != cudaSuccess) return fail_cuda(e, "tile flag launch");
  }
  if (need_tiles) {
    e = launch_prep(reinterpret_cast<const PrepSeg*>(ws + L.segs_off), 2 * n_layers, max_pairs,
                    status, s);
    if (e != cudaSuccess) return fail_cuda(e, "prep launch");
  }
  const int sms = sm_count(dg.dev);
  for (size_t gi = 0; gi < L.groups.size(); ++gi) {
    const Group& g = L.groups[gi];
    float* partials = reinterpret_cast<float*>(ws + g.partial_off);
    if (g.n_items > 0) {
      ProjParams p;
      p.mods = mods_dev + g.first_mod;
      p.n_mods = static_cast<int>(g.layers.size());
      p.B = static_cast<int>(B);
      p.T = static_cast<int>(T);
      p.n_tiles = L.n_tiles;
      p.tpc = g.tpc;
      p.n_chunks = g.n_chunks;
      p.n_items = g.n_items;
      p.items = g.table.empty() ? nullptr : reinterpret_cast<const WorkItem*>(ws + g.table_off);
      p.piece_buf = g.piece_floats > 0 ? reinterpret_cast<float*>(ws + g.piece_off) : nullptr;
      p.split_cnt = g.table.empty() ? nullptr : reinterpret_cast<int*>(ws + g.split_cnt_off);
      p.mask = mask;
      p.tile_valid = tile_valid;
      p.partials = partials;
      p.bias_partials = (g.has_bias && !token) ? reinterpret_cast<float*>(ws + g.bias_off) : nullptr;
      p.queries = queries;
      p.ld_q = ld_q;
      p.n_queries = static_cast<int>(n_queries);
      p.token_partials = partials;
      p.counter = reinterpret_cast<int*>(ws + L.ctr_off) + 32 * gi;
      p.status = status;
      p.timeout_ns = kWaitTimeoutNs;
      const int grid = std::max(1, std::min(sms > 0 ? sms : 1, g.n_items));
      e = launch_project(g.k_in, g.k_out, token, p, grid, s);
      if (e != cudaSuccess) return fail_cuda(e, "projection kernel launch");
    }
    if (!token) {
      e = launch_reduce(mods_dev + g.first_mod, static_cast<int>(g.layers.size()), g.k_in,
                        g.k_out, static_cast<int>(B), g.n_chunks, partials,
                        g.has_bias ? reinterpret_cast<const float*>(ws + g.bias_off) : nullptr,
                        out, ld_out, s);
      if (e != cudaSuccess) return fail_cuda(e, "reduce launch");
    }
  }
  if (token) {
    e = launch_token_reduce(reinterpret_cast<const float*>(ws + L.token_off), n_layers, static_cast<int>(n_queries), static_cast<int>(B),
                            static_cast<int>(T), mask, out, s);
    if (e != cudaSuccess) return fail_cuda(e, "token reduce launch");
  }
  return BERGSON_OK;
}

int bergson_project_grads(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                          const uint8_t* mask, float* out, int64_t ld_out, void* workspace,
                          size_t ws_bytes, void* stream) {
  return run_projection(layers, n_layers, B, T, mask, out, ld_out, nullptr, 0, 0, workspace,
                        ws_bytes, stream);
}

int bergson_token_scores_workspace(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                                   int64_t n_queries, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  if (n_queries < 1 || n_queries > kMaxTokenQueries)
    return fail(BERGSON_EUNSUPPORTED, "n_queries must be in [1, %d]", kMaxTokenQueries);
  int st = validate_layers(layers, n_layers, B, T);
  if (st != BERGSON_OK) return st;
  *ws_bytes = plan_project(layers, n_layers, B, T, n_queries).total;
  return BERGSON_OK;
}

int bergson_token_scores(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                         const uint8_t* mask, const float* queries, int64_t n_queries,
                         int64_t ld_q, float* out, void* workspace, size_t ws_bytes,
                         void* stream) {
  if (n_queries < 1) return fail(BERGSON_EINVAL, "n_queries must be >= 1");
  return run_projection(layers, n_layers, B, T, mask, out, 0, queries, n_queries, ld_q, workspace,
                        ws_bytes, stream);
}

int bergson_build_store(const float* proj, int64_t B, int64_t K, int64_t ld_proj,
                        int unit_normalize, void* store, int64_t ld_store, int64_t row_offset,
                        int64_t N_cap, float* norms_out, void* stream) {
  if (B < 0 || B > (1ll << 31) - 1) return fail(BERGSON_EINVAL, "B must be in [0, 2^31)");
  if (K < 8 || K > (1ll << 28)) return fail(BERGSON_EINVAL, "K must be in [8, 2^28]");
  if (K % 8 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 8");
  if (ld_proj < K) return fail(BERGSON_EINVAL, "ld_proj must be >= K");
  if (ld_proj % 4 != 0) return fail(BERGSON_EALIGN, "ld_proj must be a multiple of 4");
  if (ld_store < K) return fail(BERGSON_EINVAL, "ld_store must be >= K");
  if (ld_store % 8 != 0) return fail(BERGSON_EALIGN, "ld_store must be a multiple of 8");
  if (row_offset < 0 || N_cap < 0 || row_offset + B > N_cap)
    return fail(BERGSON_EINVAL, "rows [%lld, %lld) do not fit N_cap=%lld", (long long)row_offset,
                (long long)(row_offset + B), (long long)N_cap);
  if (B > 0) {
    if (proj == nullptr || store == nullptr) return fail(BERGSON_EINVAL, "proj or store is NULL");
    if (!aligned(proj, 16) || !aligned(store, 16))
      return fail(BERGSON_EALIGN, "proj and store must be 16-byte aligned");
    if (norms_out != nullptr && !aligned(norms_out, 4))
      return fail(BERGSON_EALIGN, "norms_out must be 4-byte aligned");
  }
  int st;
  if ((st = injected()) != BERGSON_OK) return st;
  if (B == 0) return BERGSON_OK;
  DeviceGuard dg(store);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "store device lookup");
  __half* dst = static_cast<__half*>(store) + row_offset * ld_store;
  cudaError_t e = launch_build_store(proj, static_cast<int>(B), static_cast<int>(K), ld_proj,
                                     unit_normalize ? 1 : 0, dst, ld_store, norms_out,
                                     static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, "store kernel launch");
  return BERGSON_OK;
}

int bergson_build_store_blocks(const float* proj, int64_t B, int64_t K, int64_t ld_proj,
                               const int64_t* block_offsets, int n_blocks, void* store,
                               int64_t ld_store, int64_t row_offset, int64_t N_cap,
                               float* norms_out, void* stream) {
  if (B < 0 || B > (1ll << 31) - 1) return fail(BERGSON_EINVAL, "B must be in [0, 2^31)");
  if (K < 8 || K > (1ll << 28)) return fail(BERGSON_EINVAL, "K must be in [8, 2^28]");
  if (K % 8 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 8");
  if (block_offsets == nullptr) return fail(BERGSON_EINVAL, "block_offsets is NULL");
  if (n_blocks < 1 || n_blocks > kMaxStoreBlocks)
    return fail(BERGSON_EINVAL, "n_blocks must be in [1, %d]", kMaxStoreBlocks);
  StoreBlocks sb;
  sb.n = n_blocks;
  if (block_offsets[0] != 0 || block_offsets[n_blocks] != K)
    return fail(BERGSON_EINVAL, "block_offsets must start at 0 and end at K");
  for (int j = 0; j <= n_blocks; ++j) {
    if (j > 0 && block_offsets[j] <= block_offsets[j - 1])
      return fail(BERGSON_EINVAL, "block_offsets must increase (block %d is empty)", j - 1);
    if (block_offsets[j] % 8 != 0)
      return fail(BERGSON_EALIGN, "block_offsets must be multiples of 8 (offset %d)", j);
    sb.offset[j] = static_cast<int32_t>(block_offsets[j]);
  }
  if (ld_proj < K) return fail(BERGSON_EINVAL, "ld_proj must be >= K");
  if (ld_proj % 4 != 0) return fail(BERGSON_EALIGN, "ld_proj must be a multiple of 4");
  if (ld_store < K) return fail(BERGSON_EINVAL, "ld_store must be >= K");
  if (ld_store % 8 != 0) return fail(BERGSON_EALIGN, "ld_store must be a multiple of 8");
  if (row_offset < 0 || N_cap < 0 || row_offset + B > N_cap)
    return fail(BERGSON_EINVAL, "rows [%lld, %lld) do not fit N_cap=%lld", (long long)row_offset,
                (long long)(row_offset + B), (long long)N_cap);
  if (B > 0) {
    if (proj == nullptr || store == nullptr) return fail(BERGSON_EINVAL, "proj or store is NULL");
    if (!aligned(proj, 16) || !aligned(store, 16))
      return fail(BERGSON_EALIGN, "proj and store must be 16-byte aligned");
    if (norms_out != nullptr && !aligned(norms_out, 4))
      return fail(BERGSON_EALIGN, "norms_out must be 4-byte aligned");
  }
  int st;
  if ((st = injected()) != BERGSON_OK) return st;
  if (B == 0) return BERGSON_OK;
  DeviceGuard dg(store);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "store device lookup");
  __half* dst = static_cast<__half*>(store) + row_offset * ld_store;
  cudaError_t e = launch_build_store_blocks(proj, static_cast<int>(B), ld_proj, sb, dst, ld_store,
                                            norms_out, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, "store kernel launch");
  return BERGSON_OK;
}

int bergson_score_topk_workspace(int64_t N, int64_t K, int64_t Q, int64_t topk, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  const int st = validate_score_sizes(N, K, Q, topk);
  if (st != BERGSON_OK) return st;
  *ws_bytes = plan_score(K, Q, topk).total;
  return BERGSON_OK;
}

// Top-k (least = false) or bottom-k (least = true: the queries are negated
// when they are normalised, and the final merge reports the scores against
// the original queries).
//
// Update mode (update = true): out_scores / out_idx hold on entry the result of
// earlier calls over other rows (global indices, this call's order); the call
// scores rows [row_base, row_base + N) of the whole store and leaves in them
// the top-k of both.  Its threshold starts at the prior k-th score, so it
// skips the prefix pass.  Rows report row_base + local row in either mode.
static int run_score(const void* store, int64_t N, int64_t K, int64_t ld_store,
                     const float* queries, int64_t Q, int64_t ld_q, int64_t topk,
                     float* out_scores, int64_t* out_idx, void* workspace, size_t ws_bytes,
                     void* stream, bool least, int64_t row_base = 0, bool update = false,
                     bool chunk_rules = false) {
  int st = chunk_rules ? validate_score_sizes(topk, K, Q, topk)
                       : validate_score(store, N, K, ld_store, queries, Q, ld_q, topk);
  if (st != BERGSON_OK) return st;
  if (chunk_rules) {
    if (N < 1) return fail(BERGSON_EINVAL, "the chunk must hold at least one row");
    if (row_base < 0 || row_base + N > (1ll << 31) - 1)
      return fail(BERGSON_EINVAL, "rows [row_base, row_base + N) must lie in [0, 2^31 - 1)");
    if ((st = validate_score(store, std::max(N, topk), K, ld_store, queries, Q, ld_q, topk)) !=
        BERGSON_OK)
      return st;
  }
  if (Q > 0 && (out_scores == nullptr || out_idx == nullptr))
    return fail(BERGSON_EINVAL, "out_scores or out_idx is NULL");
  if ((out_scores && !aligned(out_scores, 4)) || (out_idx && !aligned(out_idx, 8)))
    return fail(BERGSON_EALIGN, "outputs misaligned");
  const ScoreLayout L = plan_score(K, Q, topk);
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < L.total)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, L.total);
  if ((st = injected()) != BERGSON_OK) return st;
  if (Q == 0) return BERGSON_OK;

  DeviceGuard dg(workspace);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "workspace device lookup");
  if (encode_fn() == nullptr)
    return fail(BERGSON_ECUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
  int* status = status_word(dg.dev);
  if (status == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  __half* qh = reinterpret_cast<__half*>(ws + L.qh_off);
  unsigned long long* heaps = reinterpret_cast<unsigned long long*>(ws + L.heap_off);

  cudaError_t e = launch_normalize_queries(queries, static_cast<int>(Q), static_cast<int>(K), ld_q,
                                           least, qh, s);
  if (e != cudaSuccess) return fail_cuda(e, "query normalisation launch");

  // Many queries: clusters of two CTAs share each store tile (128 rows each).
  const bool pair = Q >= kPairMinQueries;
  CUtensorMap tm_store, tm_q;
  CUresult r1 = encode_2d(&tm_store, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, store, K, N, ld_store * 2,
                          kChunk, pair ? kScoreBN / 2 : kScoreBN);
  CUresult r2 = encode_2d(&tm_q, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, qh, K, Q, K * 2, kChunk, kScoreQT);
  if (r1 != CUDA_SUCCESS || r2 != CUDA_SUCCESS)
    return fail(BERGSON_ECUDA, "tensor map encoding failed (%d %d)", (int)r1, (int)r2);

  int ctas = sm_count(dg.dev);
  if (pair) {
    int resident = 0;
    e = score_pair_max_ctas(L.qt, std::max(1, std::min(ctas, kMaxScoreCTAs)), &resident);
    if (e != cudaSuccess) return fail_cuda(e, "score kernel occupancy query");
    ctas = std::min(ctas, resident);
  }
  const ScoreLaunchPlan P = plan_score_launches(N, Q, topk, ctas, !update);
  if (P.launches.empty()) return fail(BERGSON_ECUDA, "no two-SM cluster fits the score kernel");
  for (const ScoreLaunch& l : P.launches) {
    ScoreParams p;
    p.N = static_cast<int>(l.rows);
    p.K = static_cast<int>(K);
    p.Q = static_cast<int>(Q);
    p.topk = static_cast<int>(topk);
    p.n_qg = l.n_qg;
    p.qg_base = l.qg_base;
    p.n_ntiles = l.n_tiles;
    p.heaps = heaps;
    p.tau0 = l.stage == 1 && (P.use_prefix || update) ? out_scores : nullptr;
    // a prefix pass leaves its scores in the search's own order; a prior
    // bottom-k state holds scores against q
    p.tau0_negate = update && least ? 1 : 0;
    p.status = status;
    p.timeout_ns = kWaitTimeoutNs;
    p.pace = pair ? reinterpret_cast<unsigned long long*>(ws + L.pace_off) : nullptr;
    p.pace_tag = pair ? next_pace_tag() : 0;
    e = pair ? launch_score_pair(L.qt, tm_store, tm_q, p, l.grid, s)
             : launch_score(L.qt, tm_store, tm_q, p, l.grid, s);
    if (e != cudaSuccess) return fail_cuda(e, "score kernel launch");
    // The prefix pass's scores seed the full pass's thresholds, so only
    // the final merge converts them back for a bottom-k search.
    const bool final_merge = l.stage == 1;
    e = launch_merge(heaps, l.grid, l.n_qg, L.qt, static_cast<int>(topk), l.q_begin, l.q_end,
                     l.pass, least && final_merge, final_merge ? row_base : 0,
                     update && final_merge ? out_scores : nullptr,
                     update && final_merge ? out_idx : nullptr, out_scores, out_idx, s);
    if (e != cudaSuccess) return fail_cuda(e, "merge kernel launch");
  }
  return BERGSON_OK;
}

int bergson_score_topk(const void* store, int64_t N, int64_t K, int64_t ld_store,
                       const float* queries, int64_t Q, int64_t ld_q, int64_t topk,
                       float* out_scores, int64_t* out_idx, void* workspace, size_t ws_bytes,
                       void* stream) {
  return run_score(store, N, K, ld_store, queries, Q, ld_q, topk, out_scores, out_idx, workspace,
                   ws_bytes, stream, false);
}

int bergson_score_bottomk(const void* store, int64_t N, int64_t K, int64_t ld_store,
                          const float* queries, int64_t Q, int64_t ld_q, int64_t bottomk,
                          float* out_scores, int64_t* out_idx, void* workspace, size_t ws_bytes,
                          void* stream) {
  return run_score(store, N, K, ld_store, queries, Q, ld_q, bottomk, out_scores, out_idx,
                   workspace, ws_bytes, stream, true);
}

int bergson_score_topk_update_workspace(int64_t K, int64_t Q, int64_t topk, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  const int st = validate_score_sizes(topk, K, Q, topk);
  if (st != BERGSON_OK) return st;
  *ws_bytes = plan_score(K, Q, topk).total;
  return BERGSON_OK;
}

int bergson_score_topk_update(const void* store, int64_t N, int64_t K, int64_t ld_store,
                              int64_t row_base, const float* queries, int64_t Q, int64_t ld_q,
                              int64_t topk, int init, float* scores, int64_t* idx,
                              void* workspace, size_t ws_bytes, void* stream) {
  return run_score(store, N, K, ld_store, queries, Q, ld_q, topk, scores, idx, workspace, ws_bytes,
                   stream, false, row_base, init == 0, true);
}

int bergson_score_bottomk_update(const void* store, int64_t N, int64_t K, int64_t ld_store,
                                 int64_t row_base, const float* queries, int64_t Q, int64_t ld_q,
                                 int64_t bottomk, int init, float* scores, int64_t* idx,
                                 void* workspace, size_t ws_bytes, void* stream) {
  return run_score(store, N, K, ld_store, queries, Q, ld_q, bottomk, scores, idx, workspace,
                   ws_bytes, stream, true, row_base, init == 0, true);
}

// Device bytes of one chunk buffer of the host-streaming scorer.
static size_t host_chunk_bytes(int64_t chunk_rows, int64_t K) {
  return round_up(static_cast<size_t>(chunk_rows) * K * sizeof(__half), 256);
}

int bergson_score_topk_host_workspace(int64_t chunk_rows, int64_t K, int64_t Q, int64_t topk,
                                      size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  if (chunk_rows < 1 || chunk_rows > (1ll << 31) - 1)
    return fail(BERGSON_EINVAL, "chunk_rows must be in [1, 2^31)");
  const int st = validate_score_sizes(topk, K, Q, topk);
  if (st != BERGSON_OK) return st;
  *ws_bytes = 2 * host_chunk_bytes(chunk_rows, K) + plan_score(K, Q, topk).total;
  return BERGSON_OK;
}

int bergson_score_topk_host(const void* host_store, int64_t N, int64_t K, int64_t ld_store,
                            const float* queries, int64_t Q, int64_t ld_q, int64_t topk,
                            int least, int64_t chunk_rows, float* out_scores, int64_t* out_idx,
                            void* workspace, size_t ws_bytes, void* stream, void* copy_stream) {
  int st = validate_score_sizes(N, K, Q, topk);
  if (st != BERGSON_OK) return st;
  if (chunk_rows < 1 || chunk_rows > (1ll << 31) - 1)
    return fail(BERGSON_EINVAL, "chunk_rows must be in [1, 2^31)");
  if (host_store == nullptr) return fail(BERGSON_EINVAL, "host_store is NULL");
  if (ld_store < K) return fail(BERGSON_EINVAL, "ld_store must be >= K");
  if (ld_store % 8 != 0 || !aligned(host_store, 16))
    return fail(BERGSON_EALIGN, "host_store needs 16-byte aligned rows");
  if (Q > 0 && (queries == nullptr || out_scores == nullptr || out_idx == nullptr))
    return fail(BERGSON_EINVAL, "queries, out_scores or out_idx is NULL");
  const size_t chunk_bytes = host_chunk_bytes(chunk_rows, K);
  const size_t need = 2 * chunk_bytes + plan_score(K, Q, topk).total;
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  if ((st = injected()) != BERGSON_OK) return st;
  if (Q == 0) return BERGSON_OK;
  DeviceGuard dg(workspace);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "workspace device lookup");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaStream_t cs = copy_stream != nullptr ? static_cast<cudaStream_t>(copy_stream) : s;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  uint8_t* buf[2] = {ws, ws + chunk_bytes};
  uint8_t* score_ws = ws + 2 * chunk_bytes;
  const size_t score_ws_bytes = ws_bytes - 2 * chunk_bytes;
  // Events order the two streams: a chunk is scored once its copy landed, and
  // a buffer is refilled once the chunk scored from it is done.
  cudaEvent_t ev[5] = {};
  cudaError_t e = cudaSuccess;
  for (int i = 0; i < 5 && e == cudaSuccess; ++i)
    e = cudaEventCreateWithFlags(&ev[i], cudaEventDisableTiming);
  cudaEvent_t* copied = ev;          // [2]
  cudaEvent_t* used = ev + 2;        // [2]
  cudaEvent_t start = ev[4];
  int rc = BERGSON_OK;
  if (e != cudaSuccess) rc = fail_cuda(e, "event creation");
  if (rc == BERGSON_OK && cs != s) {
    // the buffers may still be read by work enqueued on `stream` before this call
    if ((e = cudaEventRecord(start, s)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(cs, start, 0)) != cudaSuccess)
      rc = fail_cuda(e, "stream ordering");
  }
  const int64_t n_chunks = (N + chunk_rows - 1) / chunk_rows;
  for (int64_t c = 0; c < n_chunks && rc == BERGSON_OK; ++c) {
    const int b = static_cast<int>(c & 1);
    const int64_t r0 = c * chunk_rows;
    const int64_t rows = std::min(chunk_rows, N - r0);
    if (c >= 2 && (e = cudaStreamWaitEvent(cs, used[b], 0)) != cudaSuccess) {
      rc = fail_cuda(e, "stream ordering");
      break;
    }
    e = cudaMemcpy2DAsync(buf[b], static_cast<size_t>(K) * sizeof(__half),
                          static_cast<const __half*>(host_store) + r0 * ld_store,
                          static_cast<size_t>(ld_store) * sizeof(__half),
                          static_cast<size_t>(K) * sizeof(__half), static_cast<size_t>(rows),
                          cudaMemcpyHostToDevice, cs);
    if (e != cudaSuccess) {
      rc = fail_cuda(e, "chunk copy");
      break;
    }
    if ((e = cudaEventRecord(copied[b], cs)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(s, copied[b], 0)) != cudaSuccess) {
      rc = fail_cuda(e, "stream ordering");
      break;
    }
    rc = run_score(buf[b], rows, K, K, queries, Q, ld_q, topk, out_scores, out_idx, score_ws,
                   score_ws_bytes, stream, least != 0, r0, c > 0, true);
    if (rc != BERGSON_OK) break;
    if ((e = cudaEventRecord(used[b], s)) != cudaSuccess) rc = fail_cuda(e, "stream ordering");
  }
  // Destroying an event whose work is still pending is allowed: its
  // resources are released once that work completes.
  for (int i = 0; i < 5; ++i)
    if (ev[i] != nullptr) cudaEventDestroy(ev[i]);
  return rc;
}

static size_t onthefly_workspace(int64_t B, int64_t K, int64_t Q) {
  return xgemm_plan(B, Q, K).total;
}

// C[b, q] = <x_b, y_q> (scaled to cosines when unit) into out; x [B, ldx] and
// y [Q, ldy] validated by validate_onthefly.
static int run_xgemm(const float* x, int64_t B, int64_t ldx, const float* y, int64_t Q,
                     int64_t ldy, int64_t K, int unit, float* out, int64_t ld_out,
                     void* workspace, void* stream, const char* what) {
  DeviceGuard dg(workspace);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "workspace device lookup");
  if (encode_fn() == nullptr)
    return fail(BERGSON_ECUDA, "cuTensorMapEncodeTiled is unavailable from the driver");
  int* status = status_word(dg.dev);
  if (status == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  XGemmArgs a;
  a.x = x;
  a.ldx = ldx;
  a.y = y;
  a.ldy = ldy;
  a.B = static_cast<int>(B);
  a.Q = static_cast<int>(Q);
  a.K = static_cast<int>(K);
  a.unit = unit;
  a.scores = out;
  a.ld_scores = ld_out;
  a.ws = static_cast<uint8_t*>(workspace);
  a.status = status;
  a.timeout_ns = kWaitTimeoutNs;
  cudaError_t e = xgemm_run(a, sm_count(dg.dev), static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, what);
  return BERGSON_OK;
}

static int validate_onthefly(const float* proj, int64_t B, int64_t K, int64_t ld_proj,
                             const float* queries, int64_t Q, int64_t ld_q, float* scores,
                             int64_t ld_scores) {
  if (B < 0 || B > (1 << 20) || Q < 0 || Q > (1 << 24))
    return fail(BERGSON_EINVAL, "B must be in [0, 2^20] and Q in [0, 2^24]");
  if (K < 4 || K > (1 << 26)) return fail(BERGSON_EINVAL, "K must be in [4, 2^26]");
  if (K % 4 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 4");
  if (B * Q > (1ll << 34)) return fail(BERGSON_EUNSUPPORTED, "B*Q too large");
  if (B > 0 && Q > 0) {
    if (proj == nullptr || queries == nullptr || scores == nullptr)
      return fail(BERGSON_EINVAL, "proj, queries or scores is NULL");
    if (ld_proj < K || ld_q < K) return fail(BERGSON_EINVAL, "ld_proj and ld_q must be >= K");
    if (ld_scores < Q) return fail(BERGSON_EINVAL, "ld_scores must be >= Q");
    if (!aligned(proj, 16) || !aligned(queries, 16) || ld_proj % 4 != 0 || ld_q % 4 != 0)
      return fail(BERGSON_EALIGN, "proj and queries need 16-byte aligned rows");
    if (!aligned(scores, 4)) return fail(BERGSON_EALIGN, "scores must be 4-byte aligned");
  }
  return BERGSON_OK;
}

int bergson_score_grads_workspace(int64_t B, int64_t K, int64_t Q, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  // the calls' size rules (no pointers to check here)
  const int st = validate_onthefly(nullptr, 0, K, K, nullptr, 0, K, nullptr, 0);
  if (st != BERGSON_OK) return st;
  if (B < 0 || B > (1 << 20) || Q < 0 || Q > (1 << 24))
    return fail(BERGSON_EINVAL, "B must be in [0, 2^20] and Q in [0, 2^24]");
  if (B * Q > (1ll << 34)) return fail(BERGSON_EUNSUPPORTED, "B*Q too large");
  *ws_bytes = onthefly_workspace(B, K, Q);
  return BERGSON_OK;
}

int bergson_score_grads(const float* proj, int64_t B, int64_t K, int64_t ld_proj,
                        const float* queries, int64_t Q, int64_t ld_q, int unit_normalize,
                        float* scores, int64_t ld_scores, void* workspace, size_t ws_bytes,
                        void* stream) {
  int st = validate_onthefly(proj, B, K, ld_proj, queries, Q, ld_q, scores, ld_scores);
  if (st != BERGSON_OK) return st;
  const size_t need = onthefly_workspace(B, K, Q);
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  if ((st = injected()) != BERGSON_OK) return st;
  if (B == 0 || Q == 0) return BERGSON_OK;
  return run_xgemm(proj, B, ld_proj, queries, Q, ld_q, K, unit_normalize ? 1 : 0, scores,
                   ld_scores, workspace, stream, "on-the-fly score launch");
}

int bergson_aggregate_rows_workspace(int64_t n, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  if (n < 0 || n > (1ll << 31) - 1) return fail(BERGSON_EINVAL, "n must be in [0, 2^31)");
  *ws_bytes = round_up(sizeof(float) * static_cast<size_t>(n > 0 ? n : 1), 256);
  return BERGSON_OK;
}

int bergson_aggregate_rows(const float* rows, int64_t n, int64_t K, int64_t ld,
                           const int64_t* offsets, int64_t G, int mode, int normalize_each,
                           float* out, int64_t ld_out, void* workspace, size_t ws_bytes,
                           void* stream) {
  if (n < 0 || n > (1ll << 31) - 1 || G < 0 || G > (1ll << 31) - 1)
    return fail(BERGSON_EINVAL, "n and G must be in [0, 2^31)");
  if (K < 4 || K > (1 << 28)) return fail(BERGSON_EINVAL, "K must be in [4, 2^28]");
  if (K % 4 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 4");
  if (mode != BERGSON_AGG_SUM && mode != BERGSON_AGG_MEAN)
    return fail(BERGSON_EINVAL, "unknown aggregation mode %d", mode);
  if (ld < K || ld_out < K) return fail(BERGSON_EINVAL, "ld and ld_out must be >= K");
  if (G > 0) {
    if (offsets == nullptr || out == nullptr)
      return fail(BERGSON_EINVAL, "offsets or out is NULL");
    if (n > 0 && rows == nullptr) return fail(BERGSON_EINVAL, "rows is NULL");
    if ((rows && !aligned(rows, 16)) || !aligned(out, 16) || ld % 4 != 0 || ld_out % 4 != 0)
      return fail(BERGSON_EALIGN, "rows and out need 16-byte aligned rows");
    if (!aligned(offsets, 8)) return fail(BERGSON_EALIGN, "offsets must be 8-byte aligned");
  }
  const size_t need = round_up(sizeof(float) * static_cast<size_t>(n > 0 ? n : 1), 256);
  if (normalize_each && n > 0) {
    if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
    if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
    if (ws_bytes < need)
      return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  }
  int st;
  if ((st = injected()) != BERGSON_OK) return st;
  if (G == 0) return BERGSON_OK;
  DeviceGuard dg(out);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "output device lookup");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* scale = nullptr;
  cudaError_t e = cudaSuccess;
  if (normalize_each && n > 0) {
    scale = static_cast<float*>(workspace);
    e = launch_row_scales(rows, static_cast<int>(n), static_cast<int>(K), ld, 1, scale, s);
    if (e != cudaSuccess) return fail_cuda(e, "row norm launch");
  }
  e = launch_aggregate(rows, n, static_cast<int>(K), ld, offsets, static_cast<int>(G), mode, scale,
                       out, ld_out, s);
  if (e != cudaSuccess) return fail_cuda(e, "aggregation launch");
  return BERGSON_OK;
}

static int check_square(const float* r, int64_t K, int64_t ld, const char* name) {
  if (r == nullptr) return fail(BERGSON_EINVAL, "%s is NULL", name);
  if (ld < K) return fail(BERGSON_EINVAL, "%s: leading dimension < K", name);
  if (!aligned(r, 16) || ld % 4 != 0)
    return fail(BERGSON_EALIGN, "%s needs 16-byte aligned rows", name);
  return BERGSON_OK;
}

int bergson_fisher_fit_workspace(int64_t n, int64_t K, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  if (n < 1 || n > (1 << 24) || K < 4 || K > (1 << 16))
    return fail(BERGSON_EINVAL, "n must be in [1, 2^24] and K in [4, 65536]");
  if (K % 4 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 4");
  *ws_bytes = round_up(fisher_fit_workspace(n, K), 256);
  return BERGSON_OK;
}

int bergson_fisher_fit(const float* rows, int64_t n, int64_t K, int64_t ld, float* R, int64_t ldr,
                       void* workspace, size_t ws_bytes, void* stream) {
  if (n < 1 || n > (1 << 24) || K < 4 || K > (1 << 16))
    return fail(BERGSON_EINVAL, "n must be in [1, 2^24] and K in [4, 65536]");
  if (K % 4 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 4");
  if (rows == nullptr) return fail(BERGSON_EINVAL, "rows is NULL");
  if (ld < K) return fail(BERGSON_EINVAL, "ld must be >= K");
  int st = check_square(R, K, ldr, "R");
  if (st != BERGSON_OK) return st;
  const size_t need = round_up(fisher_fit_workspace(n, K), 256);
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  if ((st = injected()) != BERGSON_OK) return st;
  DeviceGuard dg(R);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "output device lookup");
  int* status = status_word(dg.dev);
  if (status == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  cudaError_t e = launch_fisher_fit(rows, static_cast<int>(n), static_cast<int>(K), ld, R, ldr,
                                    static_cast<float*>(workspace), status, sm_count(dg.dev),
                                    static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, "Fisher fit launch");
  return BERGSON_OK;
}

int bergson_fisher_preconditioner_workspace(int64_t K, size_t* ws_bytes) {
  if (ws_bytes == nullptr) return fail(BERGSON_EINVAL, "ws_bytes is NULL");
  if (K < 4 || K > (1 << 16)) return fail(BERGSON_EINVAL, "K must be in [4, 65536]");
  if (K % 4 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 4");
  *ws_bytes = round_up(fisher_power_workspace(K), 256);
  return BERGSON_OK;
}

static int run_fisher_preconditioner(const float* R1, const float* R2, int64_t K, int64_t ldr,
                                     float lam, float damping, int power, int iterations,
                                     float tol, float* residuals, int* iterations_done, float* M,
                                     int64_t ldm, void* workspace, size_t ws_bytes,
                                     void* stream) {
  if (K < 4 || K > (1 << 16)) return fail(BERGSON_EINVAL, "K must be in [4, 65536]");
  if (K % 4 != 0) return fail(BERGSON_EALIGN, "K must be a multiple of 4");
  int st = check_square(R1, K, ldr, "R1");
  if (st != BERGSON_OK) return st;
  if (R2 != nullptr && (st = check_square(R2, K, ldr, "R2")) != BERGSON_OK) return st;
  if ((st = check_square(M, K, ldm, "M")) != BERGSON_OK) return st;
  if (!(lam >= 0.0f && lam <= 1.0f)) return fail(BERGSON_EINVAL, "lam must be in [0, 1]");
  if (!(damping >= 0.0f)) return fail(BERGSON_EINVAL, "damping must be >= 0");
  if (power != BERGSON_FISHER_INV_SQRT && power != BERGSON_FISHER_INV)
    return fail(BERGSON_EINVAL, "unknown power %d", power);
  if (iterations < 1 || iterations > 100) return fail(BERGSON_EINVAL, "iterations in [1, 100]");
  if (!(tol >= 0.0f)) return fail(BERGSON_EINVAL, "tol must be >= 0");
  const size_t need = round_up(fisher_power_workspace(K), 256);
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  if ((st = injected()) != BERGSON_OK) return st;
  DeviceGuard dg(M);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "output device lookup");
  int* status = status_word(dg.dev);
  if (status == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  cudaError_t e = launch_fisher_power(R1, R2, static_cast<int>(K), ldr, lam, damping,
                                      power == BERGSON_FISHER_INV ? 1 : 0, iterations, tol,
                                      residuals, iterations_done, M, ldm,
                                      static_cast<float*>(workspace), status, sm_count(dg.dev),
                                      static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, "Fisher preconditioner launch");
  return BERGSON_OK;
}

int bergson_fisher_preconditioner(const float* R1, const float* R2, int64_t K, int64_t ldr,
                                  float lam, float damping, int power, int iterations, float* M,
                                  int64_t ldm, void* workspace, size_t ws_bytes, void* stream) {
  return run_fisher_preconditioner(R1, R2, K, ldr, lam, damping, power, iterations, 0.0f, nullptr,
                                   nullptr, M, ldm, workspace, ws_bytes, stream);
}

int bergson_fisher_preconditioner_tol(const float* R1, const float* R2, int64_t K, int64_t ldr,
                                      float lam, float damping, int power, int max_iterations,
                                      float tol, float* M, int64_t ldm, void* workspace,
                                      size_t ws_bytes, float* residuals, int* iterations,
                                      void* stream) {
  return run_fisher_preconditioner(R1, R2, K, ldr, lam, damping, power, max_iterations, tol,
                                   residuals, iterations, M, ldm, workspace, ws_bytes, stream);
}

int bergson_precondition_rows(const float* rows, int64_t B, int64_t K, int64_t ld, const float* M,
                              int64_t ldm, float* out, int64_t ld_out, void* workspace,
                              size_t ws_bytes, void* stream) {
  int st = validate_onthefly(rows, B, K, ld, M, K, ldm, out, ld_out);
  if (st != BERGSON_OK) return st;
  if (B > 0 && !aligned(out, 4)) return fail(BERGSON_EALIGN, "out must be 4-byte aligned");
  const size_t need = onthefly_workspace(B, K, K);
  if (workspace == nullptr) return fail(BERGSON_EINVAL, "workspace is NULL");
  if (!aligned(workspace, 256)) return fail(BERGSON_EALIGN, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(BERGSON_EWORKSPACE, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  if ((st = injected()) != BERGSON_OK) return st;
  if (B == 0) return BERGSON_OK;
  return run_xgemm(rows, B, ld, M, K, ldm, K, 0, out, ld_out, workspace, stream,
                   "preconditioning launch");
}

int bergson_projection_matrix(uint64_t seed, int64_t d, int64_t k, int proj_kind,
                              const float* moment, float* out, void* stream) {
  if (d < 1 || d > (1 << 24)) return fail(BERGSON_EINVAL, "d must be in [1, 2^24]");
  if (!valid_k(k)) return fail(BERGSON_EUNSUPPORTED, "k must be 16, 32 or 64");
  if (!known_proj_kind(proj_kind)) return fail(BERGSON_EINVAL, "unknown proj_kind %d", proj_kind);
  if (proj_kind == BERGSON_PROJ_IDENTITY && k != d)
    return fail(BERGSON_EINVAL, "identity projection needs k == d");
  if (out == nullptr) return fail(BERGSON_EINVAL, "out is NULL");
  if (!aligned(out, 4) || (moment && !aligned(moment, 4)))
    return fail(BERGSON_EALIGN, "out/moment must be 4-byte aligned");
  int st;
  if ((st = injected()) != BERGSON_OK) return st;
  DeviceGuard dg(out);
  if (dg.err != cudaSuccess) return fail_cuda(dg.err, "output device lookup");
  int* status = status_word(dg.dev);
  if (status == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  cudaError_t e = launch_projection_matrix(seed, static_cast<int>(d), static_cast<int>(k),
                                           proj_kind, moment, status, out,
                                           static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, "projection matrix launch");
  return BERGSON_OK;
}

int bergson_sync_status(void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return fail_cuda(e, "stream synchronisation");
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  int* w = status_word(dev);
  if (w == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  int v = 0;
  e = cudaMemcpy(&v, w, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return fail_cuda(e, "status word read");
  if (v != 0) {
    const int zero = 0;
    cudaMemcpy(w, &zero, sizeof(int), cudaMemcpyHostToDevice);
    if (v == BERGSON_EMOMENT)
      return fail(v, "a factored second-moment entry (r or c) was not > 0; the projected "
                     "values computed from it are inf or NaN (device status %d)", v);
    return fail(v, "a bounded device wait gave up (device status %d)", v);
  }
  return BERGSON_OK;
}

int bergson_debug_wait_probe(uint64_t timeout_ns, void* stream) {
  if (timeout_ns < 1 || timeout_ns > 10000000000ull)
    return fail(BERGSON_EINVAL, "timeout_ns must be in [1, 1e10]");
  int st;
  if ((st = injected()) != BERGSON_OK) return st;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail_cuda(e, "cudaGetDevice");
  int* w = status_word(dev);
  if (w == nullptr) return fail(BERGSON_ECUDA, "device status word unavailable");
  e = launch_wait_probe(w, timeout_ns, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return fail_cuda(e, "probe launch");
  return BERGSON_OK;
}

}  // extern "C"
