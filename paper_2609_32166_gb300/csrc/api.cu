// C ABI of the verify step: argument validation on the host, TMA tensor-map
// encoding, launch-shape selection and the kernel launches.  See
// include/pf_verify.h for the contract of every entry point.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <algorithm>
#include <string>
#include <vector>

#include "pf_internal.h"

namespace {

thread_local std::string g_last_error;

pf_status fail(pf_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

pf_status cuda_fail(cudaError_t e, const char* what) {
  return fail(PF_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int num_sms() {
  static pf::DeviceMemo cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (const int n = cache.get(dev)) return n;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  cache.set(dev, n);
  return n;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
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

// bf16 tensor map with the 128-byte swizzle; dims/strides innermost first,
// strides in bytes for dims 1..rank-1.
pf_status make_map(CUtensorMap* m, int rank, const void* base, const cuuint64_t* dims,
                   const cuuint64_t* strides, const cuuint32_t* box, const char* what) {
  auto fn = encode_fn();
  if (!fn) return fail(PF_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable (no CUDA driver?)");
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base),
                  dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PF_ERR_CUDA, "tensor map for %s: CUresult %d", what, (int)r);
  return PF_OK;
}

int elem_size(int dtype) { return dtype == PF_BF16 ? 2 : 4; }

pf_status check_cache_view(const pf_kv_view& c, int need_rows, const char* who) {
  if (!c.k || !c.v) return fail(PF_ERR_NULL, "%s: cache.k/cache.v is NULL", who);
  if (!aligned16(c.k) || !aligned16(c.v))
    return fail(PF_ERR_ALIGN, "%s: cache pointers must be 16-byte aligned", who);
  if (c.layout == PF_KV_CONTIGUOUS) {
    if (c.max_seq < 1) return fail(PF_ERR_SHAPE, "%s: cache.max_seq must be >= 1", who);
    if (need_rows > c.max_seq)
      return fail(PF_ERR_CAPACITY, "%s: %d rows needed but cache.max_seq = %d", who, need_rows,
                  c.max_seq);
  } else if (c.layout == PF_KV_PAGED) {
    if (!c.page_table) return fail(PF_ERR_NULL, "%s: cache.page_table is NULL", who);
    if (c.num_pages < 1 || c.pages_per_seq < 1)
      return fail(PF_ERR_SHAPE, "%s: num_pages and pages_per_seq must be >= 1", who);
    const int pages = (need_rows + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE;
    if (pages > c.pages_per_seq)
      return fail(PF_ERR_CAPACITY, "%s: %d pages needed but pages_per_seq = %d", who, pages,
                  c.pages_per_seq);
  } else {
    return fail(PF_ERR_SHAPE, "%s: unknown cache layout %d", who, c.layout);
  }
  return PF_OK;
}

// ---------------------------------------------------------------------------
// Attention launch shape.  Which kernel runs and how a layer's work is split
// (query rows per CTA, K/V splits per row block, the balanced batch mode)
// follows from the shape, unless the descriptor's launch fields ask for
// something specific; nothing is read from the environment.
// ---------------------------------------------------------------------------
enum class AttnKernel { F32, MMA, TC64, TC128, PAIR, STREAM, BATCH, TWOBLK };

// A distinct epoch for every call of a kernel that merges its own pieces
// (the group tickets in the workspace compare it): 1 .. 2^40 - 1, wrapping.
unsigned long long next_epoch() {
  static std::atomic<unsigned long long> counter{0};
  unsigned long long e;
  do {
    e = (counter.fetch_add(1, std::memory_order_relaxed) + 1) & ((1ull << 40) - 1);
  } while (e == 0);
  return e;
}

// kernel index 0..2: mma.sync BM 32/64/128
int max_cluster_for(int kernel, int D, int want) {
  static std::atomic<int> cache[64][3][2][17];
  int dev = 0;
  cudaGetDevice(&dev);
  const int di = D == 64 ? 0 : 1;
  int w = want;
  while (w > 8) {
    std::atomic<int>& slot = cache[dev & 63][kernel][di][w];
    int c = slot.load(std::memory_order_acquire);
    if (c == 0) {
      const bool fits = pf::attention_cluster_fits(D, 32 << kernel, w);
      c = fits ? 1 : -1;
      slot.store(c, std::memory_order_release);
    }
    if (c > 0) break;
    w -= 1;
  }
  return w;
}

// How many clusters of `cluster` CTAs fit on the device at once, per kernel
// variant (memoised per device): 0 tc64 128 rows, 1 tc64 256 rows, 2 tc128
// 3 stages, 3 tc128 2 stages.
int max_active_clusters(int variant, int cluster) {
  static std::atomic<int> cache[64][5][17];
  int dev = 0;
  cudaGetDevice(&dev);
  std::atomic<int>& slot = cache[dev & 63][variant][cluster];
  int c = slot.load(std::memory_order_acquire);
  if (c == 0) {
    int n = 0;
    switch (variant) {
      case 0: n = pf::attention_tc_max_active_clusters(cluster, 128); break;
      case 1: n = pf::attention_tc_max_active_clusters(cluster, 256); break;
      case 2: n = pf::attention_tc2_max_active_clusters(cluster, 3); break;
      case 3: n = pf::attention_tc2_max_active_clusters(cluster, 2); break;
      default: n = pf::attention_2blk_max_active_clusters(cluster); break;
    }
    c = std::max(1, n) + 1;
    slot.store(c, std::memory_order_release);
  }
  return c - 1;
}

// The widest even cluster of at most `cap` CTAs (and at most `tiles`)
// whose clusters all fit on the GPU at once, so the grid runs in one wave
// (odd cluster sizes strand SMs of an SM pair); `step` CTAs per split.
int widest_split(int variant, int groups, int tiles, int cap, int step) {
  int splits = std::min(cap, tiles);
  if (step == 1 && splits > 1) splits &= ~1;
  for (; splits > 1; splits -= step == 1 ? 2 : 1)
    if (max_active_clusters(variant, splits * step) >= groups) break;
  return std::max(1, splits);
}

struct AttnChoice {
  AttnKernel kernel;
  int stages;       // TC128 ring depth
  size_t ws_need;   // workspace bytes the balanced batch mode needs (0: not used)
  pf::TeamPlan tp;  // TWOBLK with a.team = 1
};

// Team plan of the two-block kernel from host copies of cu_nodes and
// prefix_len: clusters of s CTAs, each (sequence, KV head, pair of row
// blocks) group a team of k CTAs inside one cluster.  For a target of at
// most X tiles per CTA every group needs k = ceil(tiles / X) CTAs; the teams
// are packed largest first into the first cluster with room (first-fit
// decreasing), and the smallest X whose teams fit wins, over every even
// cluster size whose clusters all fit on the GPU at once (ties: the smaller
// cluster).  A cluster's spare CTAs then join its team with the most tiles
// per CTA.  Used only where X is below the one-group clusters' tiles per CTA
// (`uniform_splits` CTAs per group).
bool plan_teams(pf::AttnArgs& a, const int32_t* hcu, const int32_t* hP, int sms,
                int uniform_splits, pf::TeamPlan* tp, int* tiles_per_cta,
                const int32_t* fits = nullptr) {
  struct Grp {
    int id, t;
  };
  if ((long long)a.B * a.Hkv * a.rb_count > 4096) return false;  // 12-bit group ids
  std::vector<Grp> gs;
  for (int b = 0; b < a.B; ++b) {
    const int nn = hcu[b + 1] - hcu[b], P = hP[b];
    if (nn < 1 || nn > a.max_nodes || P < 0 || P > a.max_prefix) return false;
    const int t = (P + 127) / 128 + (nn + 127) / 128;
    const int pairs = (nn + a.nb - 1) / a.nb;
    for (int g = 0; g < a.Hkv; ++g)
      for (int rb = 0; rb < pairs; ++rb) gs.push_back({(b * a.Hkv + g) * a.rb_count + rb, t});
  }
  const int G = (int)gs.size();
  if (G < 2) return false;
  std::stable_sort(gs.begin(), gs.end(), [](const Grp& x, const Grp& y) { return x.t > y.t; });
  long long total = 0;
  for (const Grp& x : gs) total += x.t;
  int best_x = (gs[0].t + uniform_splits - 1) / uniform_splits;  // to beat
  int best_s = 0;
  std::vector<int> best_k, best_c;
  std::vector<int> k(G), cl(G);
  for (int s = 2; s <= 16; s += 2) {
    const int C = std::min(std::min(fits ? (int)fits[s] : max_active_clusters(4, s), sms / s),
                           pf::kTeamMaxCtas / s);
    if (C < 1) continue;
    const long long lo_total = (total + (long long)C * s - 1) / ((long long)C * s);
    const int lo = std::max((int)lo_total, (gs[0].t + s - 1) / s);
    for (int X = std::max(lo, 1); X < best_x; ++X) {
      long long need = 0;
      for (int j = 0; j < G; ++j) need += (k[j] = (gs[j].t + X - 1) / X);
      if (need > (long long)C * s) continue;
      // first-fit decreasing (gs is sorted by tiles, so k is non-increasing)
      std::vector<int> room(C, s);
      bool ok = true;
      for (int j = 0; j < G && ok; ++j) {
        int c = 0;
        while (c < C && room[c] < k[j]) ++c;
        if (c == C) {
          ok = false;
        } else {
          cl[j] = c;
          room[c] -= k[j];
        }
      }
      if (!ok) continue;
      for (int c = 0; c < C; ++c)
        while (room[c] > 0) {
          int jb = -1;
          for (int j = 0; j < G; ++j)
            if (cl[j] == c && (jb < 0 || (long long)gs[j].t * k[jb] > (long long)gs[jb].t * k[j]))
              jb = j;
          if (jb < 0) break;  // a cluster without teams stays empty
          ++k[jb];
          --room[c];
        }
      best_x = X;
      best_s = s;
      best_k = k;
      best_c = cl;
      break;
    }
  }
  if (best_s == 0) return false;
  // Number the used clusters by their longest piece, longest first: CTAs
  // start as the preceding kernel's CTAs leave, the lowest-numbered first,
  // so the last to start get the shortest pieces.  Each cluster's teams are
  // laid out from rank 0.
  const int s = best_s;
  std::vector<int> longest(pf::kTeamMaxCtas, 0), order;
  for (int j = 0; j < G; ++j) {
    const int c = best_c[j];
    if (longest[c] == 0) order.push_back(c);
    longest[c] = std::max(longest[c], (gs[j].t + best_k[j] - 1) / best_k[j]);
  }
  std::stable_sort(order.begin(), order.end(),
                   [&](int x, int y) { return longest[x] > longest[y]; });
  std::vector<int> cidx(pf::kTeamMaxCtas, -1), next_rank(order.size(), 0);
  const int used = (int)order.size();
  for (int i = 0; i < used; ++i) cidx[order[i]] = i;
  for (int i = 0; i < pf::kTeamMaxCtas; ++i) tp->e[i] = pf::team_entry(0, 0, 0, 0);
  for (int j = 0; j < G; ++j) {
    const int c = cidx[best_c[j]], base = next_rank[c];
    for (int part = 0; part < best_k[j]; ++part)
      tp->e[c * s + base + part] = pf::team_entry(gs[j].id, part, best_k[j], base);
    next_rank[c] += best_k[j];
  }
  a.team = 1;
  a.splits = s;
  a.team_ctas = used * s;
  if (tiles_per_cta) *tiles_per_cta = best_x;
  return true;
}

// plan_teams behind a one-entry cache: the calls of one verify step (every
// layer) and the size queries share the same lengths and shape, so the plan
// is made once per step.
bool make_team_plan(pf::AttnArgs& a, const int32_t* hcu, const int32_t* hP, int sms,
                    int uniform_splits, pf::TeamPlan* tp, int* tiles_per_cta = nullptr) {
  struct Entry {
    bool valid = false, ok = false;
    int dev = -1, B = 0, Hkv = 0, rb_count = 0, nb = 0, max_nodes = 0, max_prefix = 0, sms = 0,
        uniform = 0;
    std::vector<int32_t> cu, P;
    pf::TeamPlan tp;
    int splits = 0, team_ctas = 0, per_cta = 0;
  };
  static std::mutex mu;
  static Entry e;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  const bool hit = e.valid && e.dev == dev && e.B == a.B && e.Hkv == a.Hkv &&
                   e.rb_count == a.rb_count && e.nb == a.nb && e.max_nodes == a.max_nodes &&
                   e.max_prefix == a.max_prefix && e.sms == sms && e.uniform == uniform_splits &&
                   std::memcmp(e.cu.data(), hcu, sizeof(int32_t) * (a.B + 1)) == 0 &&
                   std::memcmp(e.P.data(), hP, sizeof(int32_t) * a.B) == 0;
  if (!hit) {
    pf::AttnArgs t = a;
    e.ok = plan_teams(t, hcu, hP, sms, uniform_splits, &e.tp, &e.per_cta);
    e.splits = t.splits;
    e.team_ctas = t.team_ctas;
    e.valid = true;
    e.dev = dev;
    e.B = a.B;
    e.Hkv = a.Hkv;
    e.rb_count = a.rb_count;
    e.nb = a.nb;
    e.max_nodes = a.max_nodes;
    e.max_prefix = a.max_prefix;
    e.sms = sms;
    e.uniform = uniform_splits;
    e.cu.assign(hcu, hcu + a.B + 1);
    e.P.assign(hP, hP + a.B);
  }
  if (!e.ok) return false;
  *tp = e.tp;
  a.team = 1;
  a.splits = e.splits;
  a.team_ctas = e.team_ctas;
  if (tiles_per_cta) *tiles_per_cta = e.per_cta;
  return true;
}

// Validates the launch fields and fills a.bm, a.nb, a.rb_count, a.splits
// and, when `ws_ok` and the shape allows, the balanced batch mode (a.items).
pf_status choose_attention(const pf_attn_desc* d, pf::AttnArgs& a, int sms, bool ws_ok,
                           AttnChoice* out, const char* who) {
  const int D = a.D, G = a.G;
  out->stages = d->stages == 2 ? 2 : 3;
  out->ws_need = 0;
  if (d->dtype == PF_F32) {
    out->kernel = AttnKernel::F32;
    a.nb = 0;
    a.rb_count = (a.max_nodes * G + 31) / 32;
    a.splits = 1;
    return PF_OK;
  }
  const bool batch_ws = ws_ok && a.B > 1;
  // The pair kernel's groups: 256-row blocks of floor(128 / G) nodes per CTA;
  // the continuous-split kernel's: 128-row blocks of floor(128 / G) nodes.
  const int pair_nb = 2 * (128 / G);
  const int tiles64 = (a.max_prefix + 63) / 64 + (a.max_nodes + 63) / 64;
  const int tiles128 = (a.max_prefix + 127) / 128 + (a.max_nodes + 127) / 128;
  const int pair_groups = a.B * a.Hkv * ((a.max_nodes + pair_nb - 1) / pair_nb);
  const int sk_nb = 128 / G;
  const int sk_groups = a.B * a.Hkv * ((a.max_nodes + sk_nb - 1) / sk_nb);
  // The per-sequence balanced split: (sequence, KV head, 128-row block)
  // groups, at most one CTA each per SM and within the plan's capacity.
  const int batch_groups = a.B * a.Hkv * ((a.max_nodes + 128 / G - 1) / (128 / G));
  const bool batch_fits = batch_groups <= std::min(sms, pf::kPlanMaxGroups);
  AttnKernel k;
  int a_bm_auto = 0;  // the automatic choice's rows per CTA for the 64-token kernel
  if (d->kernel == PF_ATTN_KERNEL_AUTO && d->rows_per_cta != 0) {
    k = AttnKernel::TC64;
  } else if (d->kernel == PF_ATTN_KERNEL_AUTO) {
    // Tensor cores for D = 128: 128-row CTAs in clusters that split each
    // row block's tiles, on 128-token tiles once a CTA holds several of them
    // (wider S MMAs), else on 64-token tiles (a CTA with one or two tiles
    // starts sooner on a smaller first tile).  Measured per layer on GB300
    // (us; 128-token clusters / 64-token clusters / 64-token two-block
    // balanced batch / continuous split / SM pairs): 64-node tree 14.9 /
    // 17.2 / - / 23.0 / 24.7, 32K tree 70.0 / 109.8 / - / 79.2 / 84.5,
    // 8-sequence paged batch 41.9 / 46.0 / 43.4 / 50.1 / 49.7.  The
    // continuous split balances the batch's loop, but its per-launch plan
    // (global round trips at kernel start, 5-9 us under the other CTAs'
    // prefetch) and the merge launch cost more than the imbalance it saves.
    // The batch kernel (pieces in proportion to each sequence's tiles,
    // merged by the last piece in the same launch) balances the 8-sequence
    // batch's loop (at most 19 instead of 24 tiles per CTA) but measured
    // 46.4 us (paged) and 34.5 us (contiguous cache) against 37.7 and 32.3
    // for the clusters: its tile loads take longer under 152 one-CTA
    // launches (2.1 against 1.6 us per paged 64 KB tile, the same DRAM
    // bytes), and its last-piece merge adds ~5 us to the layer's tail.
    k = D != 128 ? AttnKernel::MMA : AttnKernel::TC64;  // may become TC128 below
    if (k == AttnKernel::TC64) a_bm_auto = 128;
    // A batch whose KV heads have more than 128 rows, with the host's copies
    // of the lengths: two 128-row blocks per CTA and teams of a cluster's
    // CTAs per group, sized by the groups' tiles, where the plan leaves each
    // CTA at least 4 tiles (its fixed per-launch cost is higher than the
    // one-block kernel's).  8-sequence batch (prefixes 2048..6144, 32-node
    // trees), us per layer: 33.7 against 35.7 (paged), 32.5 against 32.6
    // (contiguous cache).  Single sequences keep the one-block clusters
    // (64-node tree 16.4 against 13.6, 32K tree 87.9 against 68.1).
    if (D == 128 && a.B > 1 && G * a.max_nodes > 128 && d->host_cu_nodes &&
        d->host_prefix_len) {
      pf::AttnArgs t = a;
      t.bm = 256;
      t.nb = pair_nb;
      t.rb_count = (t.max_nodes + t.nb - 1) / t.nb;
      const int uniform = widest_split(4, t.B * t.Hkv * t.rb_count, tiles128, 16, 1);
      int per_cta = 0;
      if (make_team_plan(t, d->host_cu_nodes, d->host_prefix_len, sms, uniform, &out->tp,
                         &per_cta) &&
          per_cta >= 4) {
        a = t;
        out->kernel = AttnKernel::TWOBLK;
        return PF_OK;
      }
    }
  } else {
    k = d->kernel == PF_ATTN_KERNEL_MMA    ? AttnKernel::MMA
        : d->kernel == PF_ATTN_KERNEL_TC64 ? AttnKernel::TC64
        : d->kernel == PF_ATTN_KERNEL_TC128 ? AttnKernel::TC128
        : d->kernel == PF_ATTN_KERNEL_PAIR  ? AttnKernel::PAIR
        : d->kernel == PF_ATTN_KERNEL_BATCH ? AttnKernel::BATCH
        : d->kernel == PF_ATTN_KERNEL_TWO_BLOCK ? AttnKernel::TWOBLK
                                            : AttnKernel::STREAM;
  }

  if (k == AttnKernel::MMA) {
    const int bms[3] = {128, 64, 32};
    int pick = 32;
    for (int bm : bms) {
      if (G > bm) break;
      const int rb = (a.max_nodes + bm / G - 1) / (bm / G);
      const int base = a.B * a.Hkv * rb;
      const int per_sm = bm == 128 ? 1 : 2;
      if (base * std::min(16, tiles64) >= sms * per_sm || bm == 32) {
        pick = bm;
        break;
      }
    }
    if (G > pick) pick = 128;
    a.bm = pick;
    a.nb = pick / G;
    a.rb_count = (a.max_nodes + a.nb - 1) / a.nb;
    const int base = a.B * a.Hkv * a.rb_count;
    const int per_sm = pick == 128 ? 1 : 2;
    int splits = d->splits > 0 ? d->splits : (sms * per_sm) / base;
    splits = std::max(1, std::min(std::min(16, tiles64), splits));
    if (splits > 8) splits = max_cluster_for(pick == 32 ? 0 : pick == 64 ? 1 : 2, D, splits);
    a.splits = splits;
    out->kernel = k;
    return PF_OK;
  }

  if (k == AttnKernel::BATCH) {
    if (!batch_fits)
      return fail(PF_ERR_SHAPE, "%s: the batch kernel handles at most %d (sequence, KV head, "
                  "128-row block) groups on this device", who, std::min(sms, pf::kPlanMaxGroups));
    a.bm = 128;
    a.nb = 128 / G;
    a.rb_count = (a.max_nodes + a.nb - 1) / a.nb;
    a.splits = 1;
    a.items = sms;  // one CTA per SM
    a.slots = 1;
    out->ws_need = pf::attention_balanced_ws_bytes(a.items, a.bm, D, 1);
    out->kernel = k;
    return PF_OK;
  }
  if (k == AttnKernel::TWOBLK) {
    // two 128-row blocks of floor(128 / G) nodes per CTA, clusters over the
    // 128-token tiles: one group per cluster, or (host lengths given) teams
    a.bm = 256;
    a.nb = pair_nb;
    a.rb_count = (a.max_nodes + a.nb - 1) / a.nb;
    const int groups = a.B * a.Hkv * a.rb_count;
    a.splits = d->splits > 0 ? std::min(d->splits, tiles128)
                             : widest_split(4, groups, tiles128, 16, 1);
    if (d->splits == 0 && d->host_cu_nodes && d->host_prefix_len)
      make_team_plan(a, d->host_cu_nodes, d->host_prefix_len, sms, a.splits, &out->tp);
    out->kernel = k;
    return PF_OK;
  }
  if (k == AttnKernel::STREAM) {
    if (sk_groups > pf::kSkMaxGroups)
      return fail(PF_ERR_SHAPE, "%s: the continuous-split kernel handles at most %d (sequence, "
                  "KV head, 128-row block) groups", who, pf::kSkMaxGroups);
    a.bm = 128;
    a.nb = sk_nb;
    a.rb_count = (a.max_nodes + a.nb - 1) / a.nb;
    a.splits = 1;
    a.items = sms;  // one per SM
    a.slots = 2;
    out->ws_need = pf::attention_balanced_ws_bytes(a.items, a.bm, D, 2);
    out->kernel = k;
    return PF_OK;
  }
  if (k == AttnKernel::PAIR) {
    if (pair_groups > pf::kPlanMaxGroups)
      return fail(PF_ERR_SHAPE, "%s: the pair kernel handles at most %d (sequence, KV head, "
                  "256-row block) groups", who, pf::kPlanMaxGroups);
    a.bm = 256;
    a.nb = pair_nb;
    a.rb_count = (a.max_nodes + a.nb - 1) / a.nb;
    a.splits = 1;
    a.items = std::max(1, sms / 2);  // one per SM pair
    a.slots = 2;
    out->ws_need = pf::attention_balanced_ws_bytes(a.items, a.bm, D, 2);
    out->kernel = k;
    return PF_OK;
  }

  // TC64 / TC128: one 128-row block per CTA, or two (256 rows, TC64 only)
  // where that covers all of a KV head's rows
  const int head_rows = G * a.max_nodes;
  a.bm = (k == AttnKernel::TC64 && head_rows > 128 && head_rows <= 256) ? 256 : 128;
  if (a_bm_auto) a.bm = a_bm_auto;
  if (d->rows_per_cta != 0) a.bm = d->rows_per_cta;
  a.nb = a.bm / G;  // >= 1: G <= 128
  a.rb_count = (a.max_nodes + a.nb - 1) / a.nb;
  const int groups = a.B * a.Hkv * a.rb_count;
  if (k == AttnKernel::TC64 && d->kernel == PF_ATTN_KERNEL_TC64 && batch_ws && d->splits == 0 &&
      groups <= sms && groups <= pf::kPlanMaxGroups) {
    a.splits = 1;
    a.items = sms;
    a.slots = 1;
    out->ws_need = pf::attention_balanced_ws_bytes(sms, a.bm, D, 1);
    out->kernel = k;
    return PF_OK;
  }
  a.splits = d->splits > 0 ? std::min(d->splits, tiles64)
                           : widest_split(a.bm > 128 ? 1 : 0, groups, tiles64, 16, 1);
  if (d->kernel == PF_ATTN_KERNEL_AUTO && a.bm == 128 &&
      (tiles64 + a.splits - 1) / a.splits >= 4)
    k = AttnKernel::TC128;
  if (k == AttnKernel::TC128) {
    a.splits = d->splits > 0 ? std::min(d->splits, tiles128)
                             : widest_split(out->stages == 2 ? 3 : 2, groups, tiles128, 16, 1);
  }
  out->kernel = k;
  return PF_OK;
}

// The fields of pf_attn_desc that the launch shape depends on, validated.
pf_status attention_args(const pf_attn_desc* d, pf::AttnArgs& a, const char* who) {
  if (d->dtype != PF_BF16 && d->dtype != PF_F32)
    return fail(PF_ERR_DTYPE, "%s: dtype %d unsupported", who, d->dtype);
  if (d->batch < 1 || d->n_kv_heads < 1 || d->n_q_heads < 1 ||
      d->n_q_heads % d->n_kv_heads != 0)
    return fail(PF_ERR_SHAPE, "%s: need batch >= 1 and n_q_heads a multiple of n_kv_heads", who);
  const int D = d->head_dim;
  const int G = d->n_q_heads / d->n_kv_heads;
  if (d->dtype == PF_BF16 && D != 64 && D != 128)
    return fail(PF_ERR_SHAPE, "%s: bf16 head_dim must be 64 or 128 (got %d)", who, D);
  if (d->dtype == PF_F32 && (D < 1 || D > 128))
    return fail(PF_ERR_SHAPE, "%s: fp32 head_dim must be in 1..128 (got %d)", who, D);
  if (d->dtype == PF_BF16 && G > 128)
    return fail(PF_ERR_SHAPE, "%s: query heads per KV head must be <= 128", who);
  if (d->max_nodes < 1 || d->max_nodes > PF_MAX_NODES || d->total_nodes < 1)
    return fail(PF_ERR_SHAPE, "%s: max_nodes must be in 1..%d and total_nodes >= 1", who,
                PF_MAX_NODES);
  if (d->max_prefix_len < 0) return fail(PF_ERR_SHAPE, "%s: max_prefix_len < 0", who);
  if (d->flags & ~(PF_ATTN_EARLY_PREFETCH | PF_ATTN_NO_PDL))
    return fail(PF_ERR_SHAPE, "%s: unknown flags 0x%x", who, d->flags);
  // launch fields
  if (d->kernel < PF_ATTN_KERNEL_AUTO || d->kernel > PF_ATTN_KERNEL_TWO_BLOCK)
    return fail(PF_ERR_SHAPE, "%s: unknown kernel %d", who, d->kernel);
  if (d->dtype == PF_F32 && (d->kernel != PF_ATTN_KERNEL_AUTO || d->splits != 0 ||
                             d->rows_per_cta != 0 || d->stages != 0))
    return fail(PF_ERR_DTYPE, "%s: the fp32 path has one kernel and takes no launch fields",
                who);
  const bool tc_kernel = d->kernel == PF_ATTN_KERNEL_TC64 || d->kernel == PF_ATTN_KERNEL_TC128 ||
                         d->kernel == PF_ATTN_KERNEL_PAIR || d->kernel == PF_ATTN_KERNEL_STREAM ||
                         d->kernel == PF_ATTN_KERNEL_BATCH || d->kernel == PF_ATTN_KERNEL_TWO_BLOCK;
  if (tc_kernel && D != 128)
    return fail(PF_ERR_SHAPE, "%s: the tcgen05 kernels need head_dim 128", who);
  if (d->splits < 0 || d->splits > 16 ||
      ((d->kernel == PF_ATTN_KERNEL_PAIR || d->kernel == PF_ATTN_KERNEL_STREAM ||
        d->kernel == PF_ATTN_KERNEL_BATCH) &&
       d->splits != 0))
    return fail(PF_ERR_SHAPE,
                "%s: splits must be 0 (automatic) or 1..16, and 0 for the kernels that split "
                "by the plan",
                who);
  if (d->rows_per_cta != 0 &&
      ((d->rows_per_cta != 128 && d->rows_per_cta != 256) || D != 128 ||
       (d->kernel != PF_ATTN_KERNEL_AUTO && d->kernel != PF_ATTN_KERNEL_TC64) ||
       G > d->rows_per_cta))
    return fail(PF_ERR_SHAPE,
                "%s: rows_per_cta (128 or 256, at least G) applies to the 64-token kernel", who);
  if (d->stages != 0 && ((d->stages != 2 && d->stages != 3) || d->kernel != PF_ATTN_KERNEL_TC128))
    return fail(PF_ERR_SHAPE, "%s: stages (2 or 3) applies to the 128-token kernel", who);
  a.B = d->batch;
  a.Hq = d->n_q_heads;
  a.Hkv = d->n_kv_heads;
  a.D = D;
  a.G = G;
  a.T = d->total_nodes;
  a.max_nodes = d->max_nodes;
  a.max_prefix = d->max_prefix_len;
  a.flags = d->flags & PF_ATTN_EARLY_PREFETCH;
  return PF_OK;
}

}  // namespace

namespace pf {
pf_status set_error(pf_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}
}  // namespace pf

namespace pf {
// Every argument check of pf_lmhead_accept that does not involve the
// workspace (pf_lmhead_accept_noalloc runs them before it touches its
// scratch, so that a rejected call queues nothing).
pf_status lmhead_check_desc(const pf_lm_desc* d, const char* who) {
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (!d->cu_nodes || !d->hidden_states || !d->weight || !d->tokens || !d->parent ||
      !d->argmax || !d->accept_len || !d->path || !d->out_tokens)
    return fail(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  if (d->dtype != PF_BF16 && d->dtype != PF_F32)
    return fail(PF_ERR_DTYPE, "%s: dtype %d unsupported", who, d->dtype);
  if (d->batch < 1 || d->hidden < 1 || d->vocab < 1)
    return fail(PF_ERR_SHAPE, "%s: batch, hidden and vocab must be >= 1", who);
  if (d->total_nodes < 1 || d->total_nodes > PF_MAX_LM_ROWS)
    return fail(PF_ERR_SHAPE, "%s: total_nodes = %d outside 1..%d", who, d->total_nodes,
                PF_MAX_LM_ROWS);
  if (d->max_nodes < 1 || d->max_nodes > PF_MAX_NODES)
    return fail(PF_ERR_SHAPE, "%s: max_nodes outside 1..%d", who, PF_MAX_NODES);
  if (d->dtype == PF_BF16 && d->hidden % 8 != 0)
    return fail(PF_ERR_ALIGN, "%s: bf16 hidden size must be a multiple of 8", who);
  if (!aligned16(d->hidden_states) || !aligned16(d->weight))
    return fail(PF_ERR_ALIGN, "%s: hidden and weight must be 16-byte aligned", who);
  if (d->flags & ~(PF_LM_EARLY_WEIGHT | PF_LM_NO_PDL))
    return fail(PF_ERR_SHAPE, "%s: unknown flags", who);
  if (d->stages < 0 || d->stages == 1 || d->stages > 16)
    return fail(PF_ERR_SHAPE, "%s: stages must be 0 (automatic) or 2..16", who);
  return PF_OK;
}
}  // namespace pf

extern "C" {

const char* pf_last_error(void) { return g_last_error.c_str(); }

int32_t pf_version(void) { return 201; }

pf_status pf_tree_prepare(const int32_t* parent, int32_t n_nodes, int32_t* depth_out,
                          uint64_t* mask_out) {
  if (!parent || !mask_out) return fail(PF_ERR_NULL, "pf_tree_prepare: parent/mask_out is NULL");
  if (n_nodes < 1 || n_nodes > PF_MAX_NODES)
    return fail(PF_ERR_SHAPE, "pf_tree_prepare: n_nodes = %d outside 1..%d", n_nodes,
                PF_MAX_NODES);
  if (parent[0] != -1) return fail(PF_ERR_TREE, "pf_tree_prepare: parent[0] must be -1");
  for (int j = 1; j < n_nodes; ++j)
    if (parent[j] < 0 || parent[j] >= j)
      return fail(PF_ERR_TREE, "pf_tree_prepare: parent[%d] = %d is not in [0, %d)", j,
                  parent[j], j);
  // Nodes are topologically ordered, so each node's mask is its parent's
  // mask plus its own bit.
  for (int j = 0; j < n_nodes; ++j) {
    uint64_t* mj = mask_out + (size_t)j * PF_MASK_WORDS;
    if (j == 0) {
      for (int w = 0; w < PF_MASK_WORDS; ++w) mj[w] = 0;
      if (depth_out) depth_out[0] = 0;
    } else {
      const uint64_t* mp = mask_out + (size_t)parent[j] * PF_MASK_WORDS;
      for (int w = 0; w < PF_MASK_WORDS; ++w) mj[w] = mp[w];
      if (depth_out) depth_out[j] = depth_out[parent[j]] + 1;
    }
    mj[j >> 6] |= 1ull << (j & 63);
  }
  return PF_OK;
}

pf_status pf_tree_prepare_device(const int32_t* parent, const int32_t* cu_nodes, int32_t batch,
                                 int32_t total_nodes, int32_t max_nodes, int32_t* depth_out,
                                 uint64_t* mask_out, int32_t* error_flag, void* stream) {
  static const char* who = "pf_tree_prepare_device";
  if (!parent || !cu_nodes || !mask_out)
    return fail(PF_ERR_NULL, "%s: parent, cu_nodes and mask_out are required", who);
  if (batch < 1 || batch > 65535 || total_nodes < 1)
    return fail(PF_ERR_SHAPE, "%s: need 1 <= batch <= 65535 and total_nodes >= 1", who);
  if (max_nodes < 1 || max_nodes > PF_MAX_NODES)
    return fail(PF_ERR_SHAPE, "%s: max_nodes outside 1..%d", who, PF_MAX_NODES);
  if (!aligned16(mask_out)) return fail(PF_ERR_ALIGN, "%s: mask_out must be 16-byte aligned", who);
  if (num_sms() <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  pf::TreeArgs a = {};
  a.B = batch;
  a.T = total_nodes;
  a.max_nodes = max_nodes;
  a.parent = parent;
  a.cu_nodes = cu_nodes;
  a.depth = depth_out;
  a.mask = mask_out;
  a.err = error_flag;
  cudaError_t e = pf::launch_tree_prepare(a, static_cast<cudaStream_t>(stream), true);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

size_t pf_verify_attention_workspace_size(const pf_attn_desc* d) {
  if (!d) return 0;
  const std::string saved = g_last_error;  // a size query leaves the last error alone
  pf::AttnArgs a = {};
  AttnChoice ch;
  const int sms = num_sms();
  const bool ok = sms > 0 && attention_args(d, a, "") == PF_OK &&
                  choose_attention(d, a, sms, true, &ch, "") == PF_OK;
  g_last_error = saved;
  return ok ? ch.ws_need : 0;
}

int32_t pf_verify_attention_team_plan(const int32_t* cu_nodes, const int32_t* prefix_len,
                                      int32_t batch, int32_t n_kv_heads, int32_t group,
                                      int32_t max_nodes, int32_t max_prefix_len, int32_t sms_count,
                                      const int32_t* max_clusters, int32_t uniform_splits,
                                      uint32_t* entries, int32_t* cluster_size, int32_t* ctas,
                                      int32_t* tiles_per_cta) {
  static_assert(PF_TEAM_MAX_CTAS == pf::kTeamMaxCtas, "team plan size");
  if (!cu_nodes || !prefix_len || !entries || !cluster_size || !ctas || !tiles_per_cta) return -1;
  if (batch < 1 || n_kv_heads < 1 || group < 1 || group > 128 || max_nodes < 1 ||
      max_nodes > PF_MAX_NODES || max_prefix_len < 0 || sms_count < 1 || uniform_splits < 1)
    return -1;
  if (!max_clusters && num_sms() <= 0) return -1;  // the device's figures need a GPU
  pf::AttnArgs a = {};
  a.B = batch;
  a.Hkv = n_kv_heads;
  a.G = group;
  a.max_nodes = max_nodes;
  a.max_prefix = max_prefix_len;
  a.nb = 2 * (128 / group);
  a.rb_count = (max_nodes + a.nb - 1) / a.nb;
  pf::TeamPlan tp;
  int per_cta = 0;
  const std::string saved = g_last_error;
  const bool ok = plan_teams(a, cu_nodes, prefix_len, sms_count, uniform_splits, &tp, &per_cta,
                             max_clusters);
  g_last_error = saved;
  if (!ok) return 0;
  std::memcpy(entries, tp.e, sizeof(tp.e));
  *cluster_size = a.splits;
  *ctas = a.team_ctas;
  *tiles_per_cta = per_cta;
  return 1;
}

int32_t pf_verify_attention_launches(const pf_attn_desc* d) {
  if (!d) return 0;
  const std::string saved = g_last_error;  // a query leaves the last error alone
  pf::AttnArgs a = {};
  AttnChoice ch;
  const int sms = num_sms();
  const bool ok = sms > 0 && attention_args(d, a, "") == PF_OK &&
                  choose_attention(d, a, sms, d->workspace != nullptr, &ch, "") == PF_OK;
  g_last_error = saved;
  if (!ok) return 0;
  if ((ch.kernel == AttnKernel::PAIR || ch.kernel == AttnKernel::STREAM ||
       ch.kernel == AttnKernel::BATCH) &&
      !d->workspace)
    return 0;
  return a.items > 0 && ch.kernel != AttnKernel::BATCH ? 2 : 1;
}

pf_status pf_verify_attention(const pf_attn_desc* d, void* stream) {
  static const char* who = "pf_verify_attention";
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (!d->cu_nodes || !d->prefix_len || !d->q || !d->tree_k || !d->tree_v || !d->mask || !d->out)
    return fail(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  pf::AttnArgs a = {};
  pf_status st = attention_args(d, a, who);
  if (st != PF_OK) return st;
  st = check_cache_view(d->cache, d->max_prefix_len, who);
  if (st != PF_OK) return st;
  if (!aligned16(d->q) || !aligned16(d->tree_k) || !aligned16(d->tree_v) || !aligned16(d->out) ||
      !aligned16(d->mask))
    return fail(PF_ERR_ALIGN, "%s: tensor pointers must be 16-byte aligned", who);
  const int D = a.D, G = a.G;
  a.scale = d->scale > 0.f ? d->scale : 1.0f / sqrtf((float)D);
  a.scale_log2 = a.scale * 1.4426950408889634f;
  a.cu_nodes = d->cu_nodes;
  a.prefix_len = d->prefix_len;
  a.mask = d->mask;
  a.out = d->out;
  a.layout = d->cache.layout;
  a.max_seq = d->cache.max_seq;
  a.page_table = d->cache.page_table;
  a.pages_per_seq = d->cache.pages_per_seq;
  a.num_pages = d->cache.num_pages;
  a.err = d->error_flag;
  a.q = d->q;
  a.tk = d->tree_k;
  a.tv = d->tree_v;
  a.ck = d->cache.k;
  a.cv = d->cache.v;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const bool pdl = (d->flags & PF_ATTN_NO_PDL) == 0;
  const int sms = num_sms();
  if (sms <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);

  AttnChoice ch;
  st = choose_attention(d, a, sms, d->workspace != nullptr, &ch, who);
  if (st != PF_OK) return st;
  if (ch.kernel == AttnKernel::F32) {
    cudaError_t e = pf::launch_attention_f32(a, s, pdl);
    return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
  }
  if ((ch.kernel == AttnKernel::PAIR || ch.kernel == AttnKernel::STREAM ||
       ch.kernel == AttnKernel::BATCH) &&
      !d->workspace)
    return fail(PF_ERR_WORKSPACE, "%s: this kernel needs the workspace (%zu bytes)", who,
                ch.ws_need);
  if (a.items > 0) {
    if (d->workspace_bytes < ch.ws_need)
      return fail(PF_ERR_WORKSPACE, "%s: workspace needs %zu bytes", who, ch.ws_need);
    if (!aligned16(d->workspace))
      return fail(PF_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
    a.ws = d->workspace;
  }
  // Tensor maps: K/V boxes of the chosen kernel's tile (the pair kernel
  // loads half a tile per CTA: 64 K rows, 128 V rows of 64 columns).
  const bool pair = ch.kernel == AttnKernel::PAIR;
  const bool wide = ch.kernel == AttnKernel::TC128 || ch.kernel == AttnKernel::STREAM ||
                    ch.kernel == AttnKernel::BATCH || ch.kernel == AttnKernel::TWOBLK;
  const cuuint32_t k_rows = pair ? 64 : wide ? 128 : 64;
  const cuuint32_t v_rows = pair ? 128 : k_rows;
  const cuuint32_t q_nodes =
      pair || ch.kernel == AttnKernel::TWOBLK ? (cuuint32_t)(a.nb / 2) : (cuuint32_t)a.nb;
  pf::AttnMaps m;
  const cuuint64_t es = 2;
  {
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)a.Hq, (cuuint64_t)a.T};
    cuuint64_t str[2] = {D * es, (cuuint64_t)a.Hq * D * es};
    cuuint32_t box[3] = {64, (cuuint32_t)G, q_nodes};  // q_nodes * G <= 128 rows
    if ((st = make_map(&m.q, 3, d->q, dims, str, box, "q")) != PF_OK) return st;
  }
  {
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)a.Hkv, (cuuint64_t)a.T};
    cuuint64_t str[2] = {D * es, (cuuint64_t)a.Hkv * D * es};
    cuuint32_t kbox[3] = {64, 1, k_rows};
    cuuint32_t vbox[3] = {64, 1, v_rows};
    if ((st = make_map(&m.tk, 3, d->tree_k, dims, str, kbox, "tree_k")) != PF_OK) return st;
    if ((st = make_map(&m.tv, 3, d->tree_v, dims, str, vbox, "tree_v")) != PF_OK) return st;
  }
  if (a.layout == PF_KV_CONTIGUOUS) {
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)a.max_seq, (cuuint64_t)a.B * a.Hkv};
    cuuint64_t str[2] = {D * es, (cuuint64_t)a.max_seq * D * es};
    cuuint32_t kbox[3] = {64, k_rows, 1};
    cuuint32_t vbox[3] = {64, v_rows, 1};
    if ((st = make_map(&m.ck, 3, d->cache.k, dims, str, kbox, "cache.k")) != PF_OK) return st;
    if ((st = make_map(&m.cv, 3, d->cache.v, dims, str, vbox, "cache.v")) != PF_OK) return st;
  } else {
    cuuint64_t dims[4] = {(cuuint64_t)D, PF_PAGE_SIZE, (cuuint64_t)a.Hkv,
                          (cuuint64_t)a.num_pages};
    cuuint64_t str[3] = {D * es, PF_PAGE_SIZE * D * es, (cuuint64_t)a.Hkv * PF_PAGE_SIZE * D * es};
    cuuint32_t box[4] = {64, PF_PAGE_SIZE, 1, 1};
    if ((st = make_map(&m.ck, 4, d->cache.k, dims, str, box, "cache.k")) != PF_OK) return st;
    if ((st = make_map(&m.cv, 4, d->cache.v, dims, str, box, "cache.v")) != PF_OK) return st;
    if (wide) {
      // the 128-token kernels' V: both 64-column halves of a page in one box
      cuuint64_t dims5[5] = {64, PF_PAGE_SIZE, 2, (cuuint64_t)a.Hkv, (cuuint64_t)a.num_pages};
      cuuint64_t str5[4] = {D * es, 64 * es, PF_PAGE_SIZE * D * es,
                            (cuuint64_t)a.Hkv * PF_PAGE_SIZE * D * es};
      cuuint32_t box5[5] = {64, PF_PAGE_SIZE, 2, 1, 1};
      if ((st = make_map(&m.cv_page, 5, d->cache.v, dims5, str5, box5, "cache.v pages")) != PF_OK)
        return st;
    }
  }
  cudaError_t e;
  switch (ch.kernel) {
    case AttnKernel::PAIR: e = pf::launch_attention_pair(a, m, s, pdl); break;
    case AttnKernel::STREAM: e = pf::launch_attention_sk(a, m, s, pdl); break;
    case AttnKernel::TC128: e = pf::launch_attention_tc2(a, m, s, pdl, ch.stages, false); break;
    case AttnKernel::BATCH:
      a.epoch = next_epoch();
      e = pf::launch_attention_tc2(a, m, s, pdl, 3, true);
      break;
    case AttnKernel::TWOBLK: e = pf::launch_attention_2blk(a, m, ch.tp, s, pdl); break;
    case AttnKernel::TC64: e = pf::launch_attention_tc(a, m, s, pdl); break;
    default: e = pf::launch_attention_bf16(a, m, s, sms, pdl); break;
  }
  if (e == cudaSuccess && a.items > 0 && ch.kernel != AttnKernel::BATCH)
    e = pf::launch_attention_combine(a, s, pdl);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

size_t pf_lmhead_accept_workspace_size(const pf_lm_desc*) { return pf::kLmWorkspaceBytes; }


pf_status pf_lmhead_accept(const pf_lm_desc* d, void* workspace, size_t workspace_bytes,
                           void* stream) {
  static const char* who = "pf_lmhead_accept";
  const pf_status chk = pf::lmhead_check_desc(d, who);
  if (chk != PF_OK) return chk;
  if (!workspace || workspace_bytes < pf::kLmWorkspaceBytes)
    return fail(PF_ERR_WORKSPACE, "%s: workspace needs %zu bytes", who, pf::kLmWorkspaceBytes);
  if (!aligned16(workspace))
    return fail(PF_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);

  pf::LmArgs a = {};
  a.T = d->total_nodes;
  a.H = d->hidden;
  a.V = d->vocab;
  a.B = d->batch;
  a.max_nodes = d->max_nodes;
  a.npad = (a.T + 15) / 16 * 16;
  a.num_tiles = (a.V + 127) / 128;
  a.nk = (a.H + 63) / 64;
  a.cu_nodes = d->cu_nodes;
  a.tokens = d->tokens;
  a.parent = d->parent;
  a.argmax = d->argmax;
  a.max_logit = d->max_logit;
  a.accept_len = d->accept_len;
  a.path = d->path;
  a.out_tokens = d->out_tokens;
  a.last_node = d->last_node;
  a.best = static_cast<unsigned long long*>(workspace);
  a.ticket = reinterpret_cast<unsigned int*>(static_cast<char*>(workspace) + 8 * PF_MAX_LM_ROWS);
  a.err = d->error_flag;
  a.flags = d->flags & PF_LM_EARLY_WEIGHT;
  const bool pdl = (d->flags & PF_LM_NO_PDL) == 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int sms = num_sms();
  if (sms <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);

  if (d->dtype == PF_F32) {
    a.hidden_f32 = static_cast<const float*>(d->hidden_states);
    a.weight_f32 = static_cast<const float*>(d->weight);
    cudaError_t e = pf::launch_lmhead_f32(a, s, sms, pdl);
    return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
  }
  a.stages = pf::lmhead_bf16_stages(a.npad, d->stages);
  CUtensorMap wm, hm;
  pf_status st;
  {
    cuuint64_t dims[2] = {(cuuint64_t)a.H, (cuuint64_t)a.V};
    cuuint64_t str[1] = {(cuuint64_t)a.H * 2};
    cuuint32_t box[2] = {64, 128};
    if ((st = make_map(&wm, 2, d->weight, dims, str, box, "weight")) != PF_OK) return st;
  }
  {
    cuuint64_t dims[2] = {(cuuint64_t)a.H, (cuuint64_t)a.T};
    cuuint64_t str[1] = {(cuuint64_t)a.H * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)a.npad};
    if ((st = make_map(&hm, 2, d->hidden_states, dims, str, box, "hidden")) != PF_OK) return st;
  }
  cudaError_t e = pf::launch_lmhead_bf16(a, wm, hm, s, sms, pdl);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

pf_status pf_kv_commit(const pf_commit_desc* d, void* stream) {
  static const char* who = "pf_kv_commit";
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (!d->cu_nodes || !d->prefix_len || !d->accept_len || !d->path || !d->tree_k || !d->tree_v ||
      !d->new_len)
    return fail(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  if (d->dtype != PF_BF16 && d->dtype != PF_F32)
    return fail(PF_ERR_DTYPE, "%s: dtype %d unsupported", who, d->dtype);
  if (d->batch < 1 || d->n_layers < 1 || d->n_kv_heads < 1 || d->head_dim < 1 ||
      d->total_nodes < 1)
    return fail(PF_ERR_SHAPE, "%s: batch, n_layers, n_kv_heads, head_dim, total_nodes >= 1", who);
  if (d->max_nodes < 1 || d->max_nodes > PF_MAX_NODES)
    return fail(PF_ERR_SHAPE, "%s: max_nodes outside 1..%d", who, PF_MAX_NODES);
  if (d->max_prefix_len < 0) return fail(PF_ERR_SHAPE, "%s: max_prefix_len < 0", who);
  if ((long long)d->n_layers * d->batch * 2 > 65535)
    return fail(PF_ERR_SHAPE, "%s: n_layers * batch must be <= 32767", who);
  const int es = elem_size(d->dtype);
  const int row_bytes = d->head_dim * es;
  if (row_bytes % 16 != 0)
    return fail(PF_ERR_ALIGN, "%s: head_dim * element size must be a multiple of 16", who);
  if (d->n_layers > 1 && ((d->tree_layer_stride * es) % 16 != 0 ||
                          (d->cache_layer_stride * es) % 16 != 0))
    return fail(PF_ERR_ALIGN, "%s: layer strides must be multiples of 16 bytes", who);
  if (!aligned16(d->tree_k) || !aligned16(d->tree_v))
    return fail(PF_ERR_ALIGN, "%s: tree pointers must be 16-byte aligned", who);
  if (d->new_len == d->prefix_len)
    return fail(PF_ERR_SHAPE, "%s: new_len must not alias prefix_len", who);
  pf_status st = check_cache_view(d->cache, d->max_prefix_len + d->max_nodes, who);
  if (st != PF_OK) return st;

  pf::CommitArgs a = {};
  a.B = d->batch;
  a.L = d->n_layers;
  a.Hkv = d->n_kv_heads;
  a.row_bytes = row_bytes;
  a.max_nodes = d->max_nodes;
  a.T = d->total_nodes;
  a.cu_nodes = d->cu_nodes;
  a.prefix_len = d->prefix_len;
  a.accept_len = d->accept_len;
  a.path = d->path;
  a.tree_k = static_cast<const char*>(d->tree_k);
  a.tree_v = static_cast<const char*>(d->tree_v);
  a.tree_layer_bytes = d->tree_layer_stride * es;
  a.cache_k = static_cast<char*>(d->cache.k);
  a.cache_v = static_cast<char*>(d->cache.v);
  a.cache_layer_bytes = d->cache_layer_stride * es;
  a.layout = d->cache.layout;
  a.max_seq = d->cache.max_seq;
  a.page_table = d->cache.page_table;
  a.pages_per_seq = d->cache.pages_per_seq;
  a.num_pages = d->cache.num_pages;
  a.new_len = d->new_len;
  a.err = d->error_flag;
  const int sms = num_sms();
  if (sms <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  cudaError_t e = pf::launch_kv_commit(a, static_cast<cudaStream_t>(stream), sms, true);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

pf_status pf_kv_shift(const pf_shift_desc* d, void* stream) {
  static const char* who = "pf_kv_shift";
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (d->dtype != PF_BF16 && d->dtype != PF_F32)
    return fail(PF_ERR_DTYPE, "%s: dtype %d unsupported", who, d->dtype);
  if (d->n_layers < 1 || d->n_kv_heads < 1)
    return fail(PF_ERR_SHAPE, "%s: n_layers and n_kv_heads must be >= 1", who);
  const int es = elem_size(d->dtype);
  const int D = d->head_dim;
  if (D < 2 || D % 2 || D > 256 || ((D / 2) * es) % 16)
    return fail(PF_ERR_SHAPE, "%s: head_dim must be even, <= 256, half a row a multiple of 16 B",
                who);
  if (d->count < 0 || d->src < 0 || d->dst < 0)
    return fail(PF_ERR_SHAPE, "%s: src, dst and count must be >= 0", who);
  if (!(d->rope_base > 0.f)) return fail(PF_ERR_SHAPE, "%s: rope_base must be > 0", who);
  if ((long long)d->n_layers * d->n_kv_heads > 65535)
    return fail(PF_ERR_SHAPE, "%s: n_layers * n_kv_heads must be <= 65535", who);
  if (d->seq < 0 || d->seq >= d->batch)
    return fail(PF_ERR_SHAPE, "%s: seq outside 0..batch-1", who);
  pf_status st = check_cache_view(d->cache, std::max(d->src, d->dst) + d->count, who);
  if (st != PF_OK) return st;
  if (d->n_layers > 1 && (d->cache_layer_stride * es) % 16 != 0)
    return fail(PF_ERR_ALIGN, "%s: layer stride must be a multiple of 16 bytes", who);
  if (d->count == 0 || d->src == d->dst) return PF_OK;  // nothing moves, nothing turns

  pf::ShiftArgs a = {};
  a.L = d->n_layers;
  a.Hkv = d->n_kv_heads;
  a.row_bytes = D * es;
  a.elem_bytes = es;
  a.seq = d->seq;
  a.src = d->src;
  a.dst = d->dst;
  a.count = d->count;
  a.layout = d->cache.layout;
  a.max_seq = d->cache.max_seq;
  a.pages_per_seq = d->cache.pages_per_seq;
  a.num_pages = d->cache.num_pages;
  a.page_table = d->cache.page_table;
  a.cache_k = static_cast<char*>(d->cache.k);
  a.cache_v = static_cast<char*>(d->cache.v);
  a.layer_bytes = d->cache_layer_stride * es;
  a.err = d->error_flag;
  const double shift = (double)d->dst - (double)d->src;
  for (int i = 0; i < D / 2; ++i) {
    const double ang = shift * std::pow((double)d->rope_base, -2.0 * i / D);
    a.cs[i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
  }
  const int sms = num_sms();
  if (sms <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  cudaError_t e = pf::launch_kv_shift(a, static_cast<cudaStream_t>(stream), sms, true);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

size_t pf_retrieval_workspace_size(void) { return pf::kRetrievalWsBytes; }

pf_status pf_retrieval_key(const pf_key_desc* d, void* workspace, size_t workspace_bytes,
                           void* stream) {
  static const char* who = "pf_retrieval_key";
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (!d->hidden_state || !d->projection || !d->key_out)
    return fail(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  if (!workspace || workspace_bytes < pf::kRetrievalWsBytes)
    return fail(PF_ERR_WORKSPACE, "%s: workspace needs %zu bytes", who, pf::kRetrievalWsBytes);
  if (!aligned16(workspace)) return fail(PF_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
  if (d->dtype != PF_BF16 && d->dtype != PF_F32)
    return fail(PF_ERR_DTYPE, "%s: dtype %d unsupported", who, d->dtype);
  if (d->hidden < 1) return fail(PF_ERR_SHAPE, "%s: hidden must be >= 1", who);
  pf::KeyArgs a = {};
  a.H = d->hidden;
  a.bf16 = d->dtype == PF_BF16;
  a.vec = (d->hidden * elem_size(d->dtype)) % 16 == 0 && aligned16(d->hidden_state) &&
          aligned16(d->projection);
  a.hidden = d->hidden_state;
  a.proj = d->projection;
  a.key_out = d->key_out;
  a.z = reinterpret_cast<float*>(static_cast<char*>(workspace) + pf::kRetrievalZOff);
  a.ticket = reinterpret_cast<unsigned*>(static_cast<char*>(workspace) + pf::kRetrievalKeyTicketOff);
  a.err = d->error_flag;
  if (num_sms() <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  cudaError_t e = pf::launch_retrieval_key(a, static_cast<cudaStream_t>(stream), true);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

pf_status pf_retrieve(const pf_retrieval_desc* d, void* workspace, size_t workspace_bytes,
                      void* stream) {
  static const char* who = "pf_retrieve";
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (!d->query_key || !d->keys || !d->entry_token || !d->entry_pos || !d->entry_bound ||
      !d->best || !d->similarity)
    return fail(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  if (!workspace || workspace_bytes < pf::kRetrievalWsBytes)
    return fail(PF_ERR_WORKSPACE, "%s: workspace needs %zu bytes", who, pf::kRetrievalWsBytes);
  if (d->n_entries < 0 || d->lo < 0 || d->lo > d->hi || d->hi > d->n_entries)
    return fail(PF_ERR_SHAPE, "%s: need 0 <= lo <= hi <= n_entries", who);
  if (!aligned16(d->keys) || !aligned16(d->query_key) || !aligned16(d->entry_token) ||
      !aligned16(d->entry_pos) || !aligned16(d->entry_bound) || !aligned16(workspace))
    return fail(PF_ERR_ALIGN, "%s: keys, query_key, entry arrays and workspace must be 16-byte aligned",
                who);
  pf::RetrievalArgs a = {};
  a.lo = d->lo;
  a.hi = d->hi;
  a.token = d->token;
  a.query_key = d->query_key;
  a.keys = d->keys;
  a.entry_token = d->entry_token;
  a.entry_pos = d->entry_pos;
  a.entry_bound = d->entry_bound;
  a.best = d->best;
  a.similarity = d->similarity;
  a.block_best = reinterpret_cast<int4*>(static_cast<char*>(workspace) + pf::kRetrievalBestOff);
  a.ticket =
      reinterpret_cast<unsigned*>(static_cast<char*>(workspace) + pf::kRetrievalScanTicketOff);
  a.err = d->error_flag;
  const int sms = num_sms();
  if (sms <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  cudaError_t e = pf::launch_retrieve(a, static_cast<cudaStream_t>(stream), sms, true);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

pf_status pf_selftest_wait(int32_t* error_flag, int64_t limit_ns, int32_t signal,
                           int32_t* waited_ok, void* stream) {
  static const char* who = "pf_selftest_wait";
  if (!error_flag || !waited_ok) return fail(PF_ERR_NULL, "%s: a required pointer is NULL", who);
  if (limit_ns < 1000 || limit_ns > 5000000000LL)
    return fail(PF_ERR_SHAPE, "%s: limit_ns must be in [1e3, 5e9]", who);
  if (num_sms() <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  cudaError_t e = pf::launch_selftest_wait(error_flag, (unsigned long long)limit_ns, signal ? 1 : 0,
                                           waited_ok, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

pf_status pf_prefix_match(const pf_prefix_desc* d, void* stream) {
  static const char* who = "pf_prefix_match";
  if (!d) return fail(PF_ERR_NULL, "%s: desc is NULL", who);
  if (!d->lcp) return fail(PF_ERR_NULL, "%s: lcp is NULL", who);
  if (d->n_prev < 0 || d->n_next < 0 || d->n_prev > (1 << 30) || d->n_next > (1 << 30))
    return fail(PF_ERR_SHAPE, "%s: prompt lengths must be in [0, 2^30]", who);
  if ((d->n_prev > 0 && !d->prev) || (d->n_next > 0 && !d->next))
    return fail(PF_ERR_NULL, "%s: a prompt with keys has a NULL array", who);
  pf::PrefixArgs a = {};
  a.prev = d->prev;
  a.next = d->next;
  a.n_prev = d->n_prev;
  a.n_next = d->n_next;
  a.vec = aligned16(d->prev) && aligned16(d->next);
  a.lcp = d->lcp;
  a.cache_len = d->cache_len;
  if (num_sms() <= 0) return fail(PF_ERR_CUDA, "%s: no CUDA device", who);
  cudaError_t e = pf::launch_prefix_match(a, static_cast<cudaStream_t>(stream), true);
  return e == cudaSuccess ? PF_OK : cuda_fail(e, who);
}

}  // extern "C"
