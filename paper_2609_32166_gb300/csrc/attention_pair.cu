// Tree-masked GQA attention on pairs of SMs (tcgen05 .cta_group::2): one
// 2-SM MMA of M = 256 query rows per 128-token K/V tile.  Each CTA of the
// pair holds 128 query rows (its proposal nodes' G heads) and HALF of every
// K/V tile -- K rows (tokens) c*64 .. c*64+63 and V columns c*64 .. c*64+63
// for CTA c -- and the pair's MMA reads the other half from the peer's
// shared memory.  Every K/V byte that enters an SM therefore serves 256
// query rows, where a one-SM CTA serves 128: for the 7B shapes, whose KV
// heads have 224..896 query rows, the tile bytes each SM must take in per
// query row halve.
//
//   warp 0     TMA producer of this CTA's halves (Q once, then K/V halves
//              into a ring of kPStages stages), completing on this CTA's
//              own barriers
//   warp 1     TMEM (both CTAs, allocated as a pair); in the odd CTA one
//              thread forwards "Q / tile landed" to the leader's barriers
//              (so that each CTA itself sees every load it issued land);
//              in the leader, one thread issues the pair's MMAs:
//                S_i  = Q K_i^T   M=256, N=128, K=D   -> S[i % 2]
//                O   += P_i V_i   M=256, N=D,  K=128  (A = P in TMEM) -> O
//              and commits each to the barriers of both CTAs
//   softmax    one warpgroup per CTA, one query row per thread (its TMEM
//              lane), as in attn_tc2_kernel; each warp reports "S read" and
//              "P written" to the leader with one cluster-scope arrive
//
// Work split: the (sequence, KV head, 256-row block) groups' tiles are
// split over `splits` pairs of a cluster whose partials are merged through
// distributed shared memory (single sequences), or dealt out to one pair
// per SM pair in proportion to length with partials merged by
// attn_combine_kernel (batches; balanced batch mode).
//
// TMEM columns (each CTA, its 128 lanes): S[0] 0..127, S[1] 128..255,
// O 256..383, P[0] 384..447, P[1] 448..511.
#include <cuda_fp16.h>

#include "attn_common.cuh"

namespace cg = cooperative_groups;

namespace pf {

namespace {

constexpr int kPW = 128;             // tokens per K/V tile
constexpr int kPThreads = 192;       // producer, TMEM/MMA, one softmax warpgroup
constexpr uint32_t kPTmemCols = 512;
constexpr uint32_t kPColO = 256, kPColP = 384;
constexpr float kPRescaleLog2 = 8.f;
constexpr int kPStages = 4;

struct PairSmem {
  static constexpr int D = 128;
  static constexpr int kKHalfBytes = 64 * 128;           // 64 tokens x 64 columns
  static constexpr int kKBytes = 2 * kKHalfBytes;        // this CTA's 64 tokens, all columns
  static constexpr int kVBytes = kPW * 128;              // 128 tokens x this CTA's 64 columns
  static constexpr int kStageBytes = kKBytes + kVBytes;  // 32 KB
  static constexpr int kQOff = kPStages * kStageBytes;
  static constexpr int kQHalf = 128 * 128;               // 128 rows x 64 columns
  static constexpr int kQEnd = kQOff + 2 * kQHalf;
  static constexpr int kInboxSlots = 128 + 16;
  static constexpr int kPitch = D + 8;                   // halves
  static constexpr int kRowBytes = kPitch * 2;
  static constexpr int kInboxOff = kQEnd;
  static constexpr int kBarOff = kInboxOff + kInboxSlots * kRowBytes;
  // kv_full[S] kv_empty[S] q_full s_full[2] s_empty[2] p_full[2] pv_done[2] inbox
  static constexpr int kNumBars = 2 * kPStages + 1 + 8 + 1;
  // then the TMEM address (padded to 16 bytes) and the plan entry (16 bytes)
  static constexpr int kTotal = kBarOff + kNumBars * 8 + 32;
  static_assert(128 * kRowBytes <= kQOff, "staged rows fit in the idle ring");
  static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// TMA loads of this CTA's half of one 128-token K/V tile: K rows c*64 ..
// c*64+63 of the tile (both 64-column halves, two 64-row boxes) and V's
// 64-column half c of all 128 rows (one 128-row box); paged caches take one
// box per 16-token page.  Arms this CTA's barrier `bar` with the bytes.
__device__ __forceinline__ void pair_issue_tile(const AttnArgs& a, const CUtensorMap* tm_ck,
                                                const CUtensorMap* tm_cv,
                                                const CUtensorMap* tm_tk,
                                                const CUtensorMap* tm_tv, uint8_t* stage,
                                                uint32_t bar, int t, int n_ptiles, int b,
                                                int g, int node0, int P, Pages8 pg, int c) {
  using S = PairSmem;
  uint8_t* sk = stage;
  uint8_t* sv = stage + S::kKBytes;
  if (t < n_ptiles) {
    const int tok0 = t * kPW;
    if (a.layout == PF_KV_CONTIGUOUS) {
      mbar_arrive_expect_tx(bar, S::kStageBytes);
#pragma unroll
      for (int h = 0; h < 2; ++h)
        tma_load_3d(smem_u32(sk + h * S::kKHalfBytes), tm_ck, h * 64, tok0 + c * 64,
                    b * a.Hkv + g, bar);
      tma_load_3d(smem_u32(sv), tm_cv, c * 64, tok0, b * a.Hkv + g, bar);
    } else {
      // pages 4c .. 4c+3 hold this CTA's K rows; every page holds V rows
      const int npages = min(kPW / PF_PAGE_SIZE, (P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
      const int kpages = max(0, min(4, npages - 4 * c));
      mbar_arrive_expect_tx(bar, (uint32_t)(kpages * 2 + npages) * PF_PAGE_SIZE * 128);
      const int pages[8] = {pg.lo.x, pg.lo.y, pg.lo.z, pg.lo.w, pg.hi.x, pg.hi.y, pg.hi.z, pg.hi.w};
#pragma unroll
      for (int p = 0; p < 8; ++p) {
        if (p >= npages) break;
        if ((p >> 2) == c) {
#pragma unroll
          for (int h = 0; h < 2; ++h)
            tma_load_4d(smem_u32(sk + h * S::kKHalfBytes + (p & 3) * PF_PAGE_SIZE * 128), tm_ck,
                        h * 64, 0, g, pages[p], bar);
        }
        tma_load_4d(smem_u32(sv + p * PF_PAGE_SIZE * 128), tm_cv, c * 64, 0, g, pages[p], bar);
      }
    }
  } else {
    const int j = t - n_ptiles;
    mbar_arrive_expect_tx(bar, S::kStageBytes);
#pragma unroll
    for (int h = 0; h < 2; ++h)
      tma_load_3d(smem_u32(sk + h * S::kKHalfBytes), tm_tk, h * 64, g, node0 + j * kPW + c * 64,
                  bar);
    tma_load_3d(smem_u32(sv), tm_tv, c * 64, g, node0 + j * kPW, bar);
  }
}

template <bool BAL>
__global__ void __launch_bounds__(kPThreads, 1)
    attn_pair_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_tk,
                     const __grid_constant__ CUtensorMap tm_tv,
                     const __grid_constant__ CUtensorMap tm_ck,
                     const __grid_constant__ CUtensorMap tm_cv, const AttnArgs a) {
  using S = PairSmem;
  constexpr int D = 128;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sKV = smem;
  uint8_t* sQ = smem + S::kQOff;
  __half* sInbox = reinterpret_cast<__half*>(smem + S::kInboxOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* kv_full = bars;           // [S] own loads (+ the odd CTA's forward, leader)
  uint64_t* kv_empty = bars + kPStages;
  uint64_t* q_full = bars + 2 * kPStages;
  uint64_t* s_full = q_full + 1;      // [2]
  uint64_t* s_empty = s_full + 2;     // [2] (leader's used)
  uint64_t* p_full = s_full + 4;      // [2] (leader's used)
  uint64_t* pv_done = s_full + 6;     // [2]
  uint64_t* inbox_full = s_full + 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + S::kNumBars);
  int4* plan_slot = reinterpret_cast<int4*>(smem + S::kBarOff + S::kNumBars * 8 + 16);

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int c = rank & 1;              // position in the pair
  const int leader = rank & ~1;        // the pair's even CTA
  const int nsplit = BAL ? 1 : a.splits;
  const int split = BAL ? 0 : rank >> 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // PF_ATTN_EARLY_PREFETCH: as in attn_tc_kernel
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

  // This pair's group (sequence, KV head, 256-row block) and its part of
  // the group's tiles.  Both CTAs of a pair derive the same values, so every
  // return before the pair's first barrier is taken by both.
  int group, part, nparts;
  if constexpr (BAL) {
    const int item = (int)blockIdx.x >> 1;
    if (warp == 0) {
      const int n_groups = a.B * a.Hkv * a.rb_count;
      const int gq = (c == 0 && item < n_groups) ? item : -1;
      PlanItem ge;
      const PlanItem it = balanced_plan(a, item, gq, &ge, kPW);
      if (lane == 0) {
        *plan_slot = make_int4(it.group, it.j, it.k, 0);
        if (gq >= 0) {
          const int bq = gq / (a.rb_count * a.Hkv), nfq = (gq % a.rb_count) * a.nb;
          const int n0 = a.cu_nodes[bq], nnq = a.cu_nodes[bq + 1] - n0;
          plan_table(a)[gq] = make_int4(ge.first, ge.k, n0 + nfq, max(0, min(a.nb, nnq - nfq)) * a.G);
        }
      }
    }
    __syncthreads();
    const int4 pi = *plan_slot;
    if (pi.x < 0) return;  // no work for this pair
    group = pi.x;
    part = pi.y;
    nparts = pi.z;
  } else {
    group = (int)blockIdx.x / (2 * nsplit);
    part = split;
    nparts = nsplit;
  }
  const int rb = group % a.rb_count;
  const int g = (group / a.rb_count) % a.Hkv;
  const int b = group / (a.rb_count * a.Hkv);
  const int node0 = a.cu_nodes[b];
  const int nn = a.cu_nodes[b + 1] - node0;
  const int P = a.prefix_len[b];
  if (node0 < 0 || nn < 1 || nn > a.max_nodes || node0 + nn > a.T || P < 0 ||
      P > a.max_prefix) {
    if (tid == 0 && rank == 0 && rb == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
    return;  // uniform over the cluster (same b)
  }
  const int nbh = a.nb >> 1;                   // proposal nodes per CTA
  const int nfirst_pair = rb * a.nb;
  if (nfirst_pair >= nn) return;               // uniform over the cluster
  const int nfirst = nfirst_pair + c * nbh;    // this CTA's first node
  const int rows = max(0, min(nbh, nn - nfirst)) * a.G;  // may be 0 in the odd CTA
  const int n_ptiles = (P + kPW - 1) / kPW;
  const int n_qtiles = (nn + kPW - 1) / kPW;
  const int ntiles = n_ptiles + n_qtiles;
  // Part s takes tiles [t_begin, t_end) of the order (proposal tiles,
  // prefix tiles) and processes its prefix tiles first (as in attn_tc_kernel).
  const int t_begin = (int)((long long)ntiles * part / nparts);
  const int t_end = (int)((long long)ntiles * (part + 1) / nparts);
  const int my_tiles = t_end - t_begin;
  const int pre_lo = max(t_begin, n_qtiles);
  const int my_ptiles = max(0, t_end - pre_lo);
  auto tile_at = [&](int i) {
    return i < my_ptiles ? pre_lo - n_qtiles + i : n_ptiles + t_begin + (i - my_ptiles);
  };
  const int first = min(kPStages, my_tiles);

  if (tid == 0) {
    // the leader's load barriers also count the odd CTA's "landed" forward
    const uint32_t loads = c == 0 ? 2 : 1;
    for (int i = 0; i < kPStages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), loads);
      mbar_init(smem_u32(&kv_empty[i]), 1);  // the tile's PV (multicast commit)
    }
    mbar_init(smem_u32(q_full), loads);
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_empty[i]), 8);   // the softmax warps of both CTAs
      mbar_init(smem_u32(&p_full[i]), 8);
      mbar_init(smem_u32(&pv_done[i]), 1);
    }
    mbar_init(smem_u32(inbox_full), 1);
    fence_mbar_init();
  }
  // Every CTA's barriers are initialised before any peer signals them (the
  // odd CTA forwards to the leader's barriers, the leader's commits arrive
  // on both, split peers fill each other's inboxes).
  cluster_arrive_release();
  cluster_wait_acquire();

  const uint32_t s_empty_l0 = mapa_cluster(smem_u32(&s_empty[0]), (uint32_t)leader);
  const uint32_t p_full_l0 = mapa_cluster(smem_u32(&p_full[0]), (uint32_t)leader);

  if (tid == 0) {
    Pages8 pg[kPStages];  // every first tile's page entries in one round trip
#pragma unroll
    for (int i = 0; i < kPStages; ++i)
      pg[i] = i < first ? kv_tile_pages8(a, tile_at(i), n_ptiles, b, P) : no_pages8();
#pragma unroll
    for (int i = 0; i < kPStages; ++i)
      if (i < first && i < my_ptiles)
        pair_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                        smem_u32(&kv_full[i]), tile_at(i), n_ptiles, b, g, node0, P, pg[i], c);
  }
  if (early) pdl_wait();
  if (tid == 0) {
    mbar_arrive_expect_tx(smem_u32(q_full), 2u * a.G * nbh * 128);
#pragma unroll
    for (int h = 0; h < 2; ++h)
      tma_load_3d(smem_u32(sQ + h * S::kQHalf), &tm_q, h * 64, g * a.G, node0 + nfirst,
                  smem_u32(q_full));
    for (int i = 0; i < first; ++i)
      if (i >= my_ptiles)  // proposal tiles: no page entries
        pair_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                        smem_u32(&kv_full[i]), tile_at(i), n_ptiles, b, g, node0, P, no_pages8(),
                        c);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), kPTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();

  float m_ref = -INFINITY, l = 0.f;   // softmax threads: running max (log2) and sum of their row
  if (warp == 0) {
    // ---------------- producer: refill this CTA's ring as the PVs release stages
    if (lane == 0) {
      for (int i = kPStages; i < my_tiles; ++i) {
        const int st = i % kPStages;
        const int t = tile_at(i);
        const Pages8 pg = kv_tile_pages8(a, t, n_ptiles, b, P);  // in flight during the wait
        if (!mbar_wait_cl(smem_u32(&kv_empty[st]), ((i / kPStages) & 1) ^ 1, a.err)) break;
        pair_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + st * S::kStageBytes,
                        smem_u32(&kv_full[st]), t, n_ptiles, b, g, node0, P, pg, c);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && c == 1) {
      // ---------------- forwarder (odd CTA): once this CTA's Q, then each
      // of its tile halves, has landed, arrive on the leader's barrier
      const uint32_t q_full_l = mapa_cluster(smem_u32(q_full), (uint32_t)leader);
      const uint32_t kv_full_l0 = mapa_cluster(smem_u32(&kv_full[0]), (uint32_t)leader);
      bool ok = mbar_wait_cl(smem_u32(q_full), 0, a.err);
      if (ok) mbar_arrive_cluster(q_full_l);
      for (int i = 0; ok && i < my_tiles; ++i) {
        const int st = i % kPStages;
        ok = mbar_wait_cl(smem_u32(&kv_full[st]), (i / kPStages) & 1, a.err);
        if (ok) mbar_arrive_cluster(kv_full_l0 + 8 * st);
      }
    }
    // ---------------- MMA issuer (leader only), pair MMAs committed to both CTAs
    if (lane == 0 && c == 0) {
      const uint32_t id_s = umma_idesc_bf16(256, kPW);
      const uint32_t id_o = umma_idesc_bf16_bmn(256, D);
      const uint16_t both = (uint16_t)(3u << leader);
      bool ok = mbar_wait_cl(smem_u32(q_full), 0, a.err);
      const uint32_t q0 = smem_u32(sQ);
      int ns = 0, np = 0;
      unsigned idle = 0;
      unsigned long long t0 = 0;
      while (ok && np < my_tiles) {
        bool progressed = false;
        if (ns < my_tiles) {
          const int n = ns, st = n % kPStages, sb = n & 1;
          if (mbar_test_wait_cl(smem_u32(&kv_full[st]), (n / kPStages) & 1) &&
              mbar_test_wait_cl(smem_u32(&s_empty[sb]), ((n >> 1) & 1) ^ 1)) {
            tc_fence_after();
            const uint32_t k0 = smem_u32(sKV + st * S::kStageBytes);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              umma_pair_ss(tmem + sb * kPW,
                           umma_desc_sw128(q0 + (kk >> 2) * S::kQHalf + (kk & 3) * 32),
                           umma_desc_sw128(k0 + (kk >> 2) * S::kKHalfBytes + (kk & 3) * 32), id_s,
                           kk > 0);
            umma_commit_pair(smem_u32(&s_full[sb]), both);
            ++ns;
            progressed = true;
          }
        }
        if (np < ns) {
          const int j = np, pb = j & 1, stj = j % kPStages;
          if (mbar_test_wait_cl(smem_u32(&p_full[pb]), (j >> 1) & 1)) {
            tc_fence_after();
            const uint32_t v0 = smem_u32(sKV + stj * S::kStageBytes + S::kKBytes);
#pragma unroll
            for (int kt = 0; kt < kPW / 16; ++kt)
              umma_pair_ts(tmem + kPColO, tmem + kPColP + pb * 64 + kt * 8,
                           umma_desc_sw128_lbo(v0 + kt * 16 * 128, S::kVBytes, 1024), id_o,
                           (j > 0 || kt > 0) ? 1u : 0u);
            umma_commit_pair(smem_u32(&pv_done[pb]), both);
            // only stages that will be refilled are released: after the last
            // PV nothing more arrives on the odd CTA's barriers
            if (j + kPStages < my_tiles) umma_commit_pair(smem_u32(&kv_empty[stj]), both);
            ++np;
            progressed = true;
          }
        }
        if (progressed) {
          idle = 0;
        } else if ((++idle & 63u) == 0u) {
          const unsigned long long now = globaltimer();
          if (idle == 64u) t0 = now;
          if (now - t0 > kWaitLimitNs) {
            flag_error(a.err, PF_DEVERR_TIMEOUT);
            ok = false;
          }
        }
      }
    }
  } else {
    // ---------------- softmax / correction: one row per thread, both CTAs
    const int quad = warp & 3;
    const int rl = quad * 32 + lane;       // row within this CTA (its TMEM lane)
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    uint64_t mk0 = 0, mk1 = 0;
    if (rl < rows) {
      const int node = node0 + nfirst + rl / a.G;
      mk0 = a.mask[2 * node];
      mk1 = a.mask[2 * node + 1];
    }
    bool ok = true;
    for (int i = 0; i < my_tiles && ok; ++i) {
      const int sb = i & 1;
      const int st = i % kPStages;
      ok = __all_sync(0xffffffffu, mbar_wait_cl(smem_u32(&s_full[sb]), (i >> 1) & 1, a.err));
      if (!ok) break;  // warp-uniform
      tc_fence_after();
      uint32_t sraw[kPW];
#pragma unroll
      for (int c0 = 0; c0 < kPW; c0 += 32)
        tmem_ld_32(tmem + lane_base + sb * kPW + c0, *reinterpret_cast<uint32_t(*)[32]>(&sraw[c0]));
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(s_empty_l0 + 8 * sb);
      float sv[kPW];
#pragma unroll
      for (int cc = 0; cc < kPW; ++cc) sv[cc] = __uint_as_float(sraw[cc]);

      const int t = tile_at(i);
      const bool is_prefix = t < n_ptiles;
      const int valid = is_prefix ? min(kPW, P - t * kPW) : kPW;
      if (!is_prefix || valid < kPW) {
        uint64_t v0, v1;
        if (is_prefix) {
          v0 = valid >= 64 ? ~0ull : ((1ull << valid) - 1ull);
          v1 = valid >= 128 ? ~0ull : (valid <= 64 ? 0ull : ((1ull << (valid - 64)) - 1ull));
        } else {
          v0 = mk0;
          v1 = mk1;
        }
#pragma unroll
        for (int cc = 0; cc < 64; ++cc) {
          if (!((v0 >> cc) & 1ull)) sv[cc] = -INFINITY;
          if (!((v1 >> cc) & 1ull)) sv[64 + cc] = -INFINITY;
        }
      }
      float m43[43];
#pragma unroll
      for (int k = 0; k < 42; ++k) m43[k] = fmax3(sv[3 * k], sv[3 * k + 1], sv[3 * k + 2]);
      m43[42] = fmaxf(sv[126], sv[127]);
      float m15[15];
#pragma unroll
      for (int k = 0; k < 14; ++k) m15[k] = fmax3(m43[3 * k], m43[3 * k + 1], m43[3 * k + 2]);
      m15[14] = m43[42];
      float m5[5];
#pragma unroll
      for (int k = 0; k < 5; ++k) m5[k] = fmax3(m15[3 * k], m15[3 * k + 1], m15[3 * k + 2]);
      const float mx = fmaxf(fmax3(m5[0], m5[1], m5[2]), fmaxf(m5[3], m5[4])) * a.scale_log2;
      const float m_new = fmaxf(m_ref, mx);
      const bool resc = m_ref != -INFINITY && m_new > m_ref + kPRescaleLog2;
      if (m_ref == -INFINITY) m_ref = m_new;
      if (__any_sync(0xffffffffu, resc)) {
        // O must hold exactly the tiles before i: wait for PV_{i-1}.
        if (i >= 1) mbar_wait_cl(smem_u32(&pv_done[(i - 1) & 1]), ((i - 1) >> 1) & 1, a.err);
        tc_fence_after();
        const float alpha = resc ? ex2_approx(m_ref - m_new) : 1.f;
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t ov[32];
          tmem_ld_32(tmem + lane_base + kPColO + c0, ov);
          tmem_ld_wait();
#pragma unroll
          for (int cc = 0; cc < 32; ++cc) ov[cc] = __float_as_uint(__uint_as_float(ov[cc]) * alpha);
          tmem_st_32(tmem + lane_base + kPColO + c0, ov);
        }
        tmem_st_wait();
        if (resc) {
          l *= alpha;
          m_ref = m_new;
        }
      }
      const float neg_mu = m_ref == -INFINITY ? 0.f : -m_ref;
      const unsigned long long sc2 = f32x2_pack(a.scale_log2, a.scale_log2);
      const unsigned long long mu2 = f32x2_pack(neg_mu, neg_mu);
      unsigned long long rs2[4] = {0ull, 0ull, 0ull, 0ull};
      uint32_t pk[kPW / 2];
#pragma unroll
      for (int cc = 0; cc < kPW / 2; ++cc) {
        float x0, x1;
        f32x2_unpack(ffma2(f32x2_pack(sv[2 * cc], sv[2 * cc + 1]), sc2, mu2), x0, x1);
        const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
        rs2[cc & 3] = fadd2(rs2[cc & 3], f32x2_pack(p0, p1));
        pk[cc] = pack_bf16(p0, p1);
      }
      float r0, r1;
      f32x2_unpack(fadd2(fadd2(rs2[0], rs2[1]), fadd2(rs2[2], rs2[3])), r0, r1);
      l += r0 + r1;
      // P buffer sb was last read by PV_{i-2}.
      if (i >= 2) mbar_wait_cl(smem_u32(&pv_done[sb]), ((i - 2) >> 1) & 1, a.err);
      tc_fence_after();
      tmem_st_32(tmem + lane_base + kPColP + sb * 64, *reinterpret_cast<uint32_t(*)[32]>(&pk[0]));
      tmem_st_32(tmem + lane_base + kPColP + sb * 64 + 32,
                 *reinterpret_cast<uint32_t(*)[32]>(&pk[32]));
      tmem_st_wait();
      if (valid < kPW) {
        // Cache rows past the prefix end may hold anything (even NaN bit
        // patterns): zero this CTA's V half of them so masked columns
        // contribute exactly 0.  They are one contiguous run of 128-byte rows.
        uint4* vt = reinterpret_cast<uint4*>(sKV + st * S::kStageBytes + S::kKBytes);
        const int chunks = (kPW - valid) * 8;
        for (int cc = rl; cc < chunks; cc += 128) vt[valid * 8 + cc] = make_uint4(0, 0, 0, 0);
        fence_proxy_async_smem();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(p_full_l0 + 8 * sb);
    }
    // O of this row is complete once the last PV has landed
    if (my_tiles > 0)
      mbar_wait_cl(smem_u32(&pv_done[(my_tiles - 1) & 1]), ((my_tiles - 1) >> 1) & 1, a.err);
  }
  __syncwarp();  // the producer and MMA lanes rejoin their warps before the barriers

  // ---- epilogue: each softmax thread reads its row of O / l from TMEM
  const bool has_row = warp >= 2;
  const int r = (warp & 3) * 32 + lane;
  const uint32_t o_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16) + kPColO;
  const float inv_l = (my_tiles > 0 && l > 0.f) ? 1.f / l : 0.f;

  if (nsplit == 1) {
    // ---- one pair per group: O / l is the output -- or, for a group that
    // the balanced batch mode spread over several pairs, this part's
    // partial (O / l in fp16, log2-sum-exp in the pad) for the combine kernel
    if (has_row) {
      uint32_t ov[D];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32)
        tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
      tmem_ld_wait();
      if (BAL && r < rows && nparts > 1) {
        if (!(inv_l > 0.f)) {
#pragma unroll
          for (int cc = 0; cc < D; ++cc) ov[cc] = 0u;
        }
        const int pr = c * nbh * a.G + r;  // row within the pair's block
        __half* dst = reinterpret_cast<__half*>(a.ws) +
                      ((size_t)((int)blockIdx.x >> 1) * a.bm + pr) * S::kPitch;
#pragma unroll
        for (int cc = 0; cc < D; cc += 8) {
          uint4 pk;
          pk.x = pack_half(__uint_as_float(ov[cc]) * inv_l, __uint_as_float(ov[cc + 1]) * inv_l);
          pk.y = pack_half(__uint_as_float(ov[cc + 2]) * inv_l, __uint_as_float(ov[cc + 3]) * inv_l);
          pk.z = pack_half(__uint_as_float(ov[cc + 4]) * inv_l, __uint_as_float(ov[cc + 5]) * inv_l);
          pk.w = pack_half(__uint_as_float(ov[cc + 6]) * inv_l, __uint_as_float(ov[cc + 7]) * inv_l);
          *reinterpret_cast<uint4*>(dst + cc) = pk;
        }
        *reinterpret_cast<float*>(dst + D) = inv_l > 0.f ? m_ref + __log2f(l) : -INFINITY;
      } else if (r < rows) {
        const int node = node0 + nfirst + r / a.G;
        const int h = g * a.G + r % a.G;
        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(a.out) + ((size_t)node * a.Hq + h) * D;
#pragma unroll
        for (int cc = 0; cc < D; cc += 8) {
          uint4 pk;
          pk.x = pack_bf16(__uint_as_float(ov[cc]) * inv_l, __uint_as_float(ov[cc + 1]) * inv_l);
          pk.y = pack_bf16(__uint_as_float(ov[cc + 2]) * inv_l, __uint_as_float(ov[cc + 3]) * inv_l);
          pk.z = pack_bf16(__uint_as_float(ov[cc + 4]) * inv_l, __uint_as_float(ov[cc + 5]) * inv_l);
          pk.w = pack_bf16(__uint_as_float(ov[cc + 6]) * inv_l, __uint_as_float(ov[cc + 7]) * inv_l);
          *reinterpret_cast<uint4*>(dst + cc) = pk;
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc_pair(tmem, kPTmemCols);
    }
    return;
  }
  // ---- split-KV merge between the pairs of the cluster: CTA c of every
  // pair holds the same rows, so rank 2q + c is peer q of this CTA.  Each
  // row's normalised partial and its log2-sum-exp are staged in the idle
  // ring (every PV of the pair has completed: the softmax threads waited for
  // the last one, so neither CTA's MMA reads the ring any more), one bulk
  // copy per peer moves the rows it merges into its inbox, and every CTA
  // merges its own rows from its inbox.
  const int per = (rows + nsplit - 1) / nsplit;
  const int cnt_mine = max(0, min(per, rows - split * per));
  __half* stage_rows = reinterpret_cast<__half*>(smem);
  if (tid == 0)
    mbar_arrive_expect_tx(smem_u32(inbox_full), (uint32_t)(nsplit * cnt_mine * S::kRowBytes));
  if (has_row) {
    uint32_t ov[D];
#pragma unroll
    for (int c0 = 0; c0 < D; c0 += 32)
      tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
    tmem_ld_wait();
    if (!(inv_l > 0.f)) {
      // no column reached this row in this part (a part without tiles never
      // writes O): its partial is 0 with lse = -inf
#pragma unroll
      for (int cc = 0; cc < D; ++cc) ov[cc] = 0u;
    }
    if (r < rows) {
      __half* dst = stage_rows + r * S::kPitch;
#pragma unroll
      for (int cc = 0; cc < D; cc += 8) {
        uint4 pk;
        pk.x = pack_half(__uint_as_float(ov[cc]) * inv_l, __uint_as_float(ov[cc + 1]) * inv_l);
        pk.y = pack_half(__uint_as_float(ov[cc + 2]) * inv_l, __uint_as_float(ov[cc + 3]) * inv_l);
        pk.z = pack_half(__uint_as_float(ov[cc + 4]) * inv_l, __uint_as_float(ov[cc + 5]) * inv_l);
        pk.w = pack_half(__uint_as_float(ov[cc + 6]) * inv_l, __uint_as_float(ov[cc + 7]) * inv_l);
        *reinterpret_cast<uint4*>(dst + cc) = pk;
      }
      *reinterpret_cast<float*>(dst + D) = inv_l > 0.f ? m_ref + __log2f(l) : -INFINITY;
    }
  }
  fence_proxy_async_smem();  // staged rows are read by the bulk-copy engine
  tc_fence_before();
  __syncthreads();
  if (tid < nsplit) {
    const int q = tid;
    const int cnt = min(per, rows - q * per);
    if (cnt > 0) {
      const uint32_t peer = (uint32_t)(2 * q + c);
      const uint32_t src = smem_u32(stage_rows + q * per * S::kPitch);
      const uint32_t dst = mapa_cluster(smem_u32(sInbox + split * per * S::kPitch), peer);
      bulk_copy_s2cluster(dst, src, (uint32_t)(cnt * S::kRowBytes),
                          mapa_cluster(smem_u32(inbox_full), peer));
      bulk_commit_group();
    }
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kPTmemCols);
  }
  if (cnt_mine > 0) mbar_wait(smem_u32(inbox_full), 0, a.err);
  inbox_merge<D, kPThreads, S::kPitch>(a, sInbox, rows, split, per, nsplit, node0 + nfirst, g,
                                       tid);
  // this CTA's staged rows must stay readable until its copies have left
  if (tid < nsplit) bulk_wait_read_all();
}

}  // namespace

static int pair_smem_bytes() { return PairSmem::kTotal + 1024; }

template <bool BAL>
static int pair_max_active_clusters_impl(int cluster) {
  const int smem = pair_smem_bytes();
  static DeviceMemo limit;
  if (ensure_smem_limit((const void*)attn_pair_kernel<BAL>, smem, limit) != cudaSuccess) return 0;
  if (cluster > 8 && cudaFuncSetAttribute(attn_pair_kernel<BAL>,
                                          cudaFuncAttributeNonPortableClusterSizeAllowed,
                                          1) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cluster);
  cfg.blockDim = dim3(kPThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = cluster;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_pair_kernel<BAL>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

int attention_pair_max_active_clusters(int cluster, bool balanced) {
  return balanced ? pair_max_active_clusters_impl<true>(cluster)
                  : pair_max_active_clusters_impl<false>(cluster);
}

template <bool BAL>
static cudaError_t launch_pair(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  const int smem = pair_smem_bytes();
  static DeviceMemo limit;
  static DeviceMemo nonportable;
  cudaError_t e = ensure_smem_limit((const void*)attn_pair_kernel<BAL>, smem, limit);
  if (e != cudaSuccess) return e;
  const int cluster = BAL ? 2 : 2 * a.splits;
  if (cluster > 8) {
    e = ensure_nonportable_cluster((const void*)attn_pair_kernel<BAL>, nonportable);
    if (e != cudaSuccess) return e;
  }
  const dim3 grid(BAL ? 2 * a.items : a.B * a.Hkv * a.rb_count * cluster);
  return launch_ex(attn_pair_kernel<BAL>, grid, dim3(kPThreads), smem, s, cluster, pdl, m.q, m.tk,
                   m.tv, m.ck, m.cv, a);
}

cudaError_t launch_attention_pair(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  return a.items > 0 ? launch_pair<true>(a, m, s, pdl) : launch_pair<false>(a, m, s, pdl);
}

}  // namespace pf
