// Tree-masked GQA attention on the tcgen05 tensor cores with 128-token K/V
// tiles, for CTAs of one 128-row block (the shapes whose KV heads have at
// most 128 rows per CTA; same contract, work split and split-KV merge as
// attn_tc_kernel).  An M = 128 UMMA costs about the same for N = 64 and
// N = 128, so S = Q K^T over 128-token tiles takes half the instructions per
// key of 64-token tiles.  The shared memory that the wider tiles need comes
// from keeping P in tensor memory:
//
//   warp 0     TMA producer: Q once, then K/V tiles (64 KB) into a ring of
//              STAGES (3 by default) stages
//   warp 1     TMEM owner and MMA issuer (one thread):
//                S_i  = Q K_i^T   M=128, N=128, K=D, A and B in smem -> S[i % 2]
//                O   += P_i V_i   M=128, N=D,  K=128, A = P in TMEM    -> O
//              each issued as soon as its inputs are ready
//   softmax    one warpgroup, one query row per thread (its TMEM lane): read
//              S, mask, online softmax in the exp2 domain, write P (bf16
//              pairs, one 32-bit column per two keys) into P[i % 2] with
//              tcgen05.st; O is rescaled only when the row maximum grows by
//              more than 2^8; at the end O / l and the log2-sum-exp go to the
//              merge, as in attn_tc_kernel.
//
// Work split: a cluster of a.splits CTAs per (sequence, KV head, row block)
// group, each taking a contiguous slice of the group's tiles, merged through
// distributed shared memory; or (BAL, a batch with the workspace) one CTA per
// SM and no cluster, each group spread over as many CTAs as its share of all
// tiles calls for (balanced_plan: the groups of one sequence get equal
// pieces, so the CTAs of its KV heads and row blocks read the same pages at
// the same time), each piece leaving a normalised partial in the workspace
// and the last piece of a group to finish merging them (group tickets).
//
// TMEM columns: S[0] 0..127, S[1] 128..255, O 256..383, P[0] 384..447,
// P[1] 448..511.
#include <cuda_fp16.h>

#include "attn_common.cuh"

namespace cg = cooperative_groups;

namespace pf {

namespace {

constexpr int kW = 128;              // tokens per K/V tile
constexpr int kW2Threads = 192;      // producer, MMA, one softmax warpgroup
constexpr uint32_t kW2TmemCols = 512;
constexpr uint32_t kColO = 256, kColP = 384;
constexpr float kW2RescaleLog2 = 8.f;

// STAGES = 2: the merge inbox has its own space, so peers may send while
// this CTA still works.  STAGES = 3: no room; the inbox takes the idle ring
// from its second stage on, and peers send only after every CTA of the
// cluster has left its loop.  Partial rows are staged at the ring's start.
template <int STAGES>
struct W2Smem {
  static constexpr int D = 128;
  static constexpr int kHalfBytes = kW * 128;             // 128 tokens x 64 columns
  static constexpr int kTileBytes = 2 * kHalfBytes;       // one K or V tile
  static constexpr int kStageBytes = 2 * kTileBytes;      // K + V
  static constexpr int kQOff = STAGES * kStageBytes;
  static constexpr int kQHalf = 128 * 128;                // 128 rows x 64 columns
  static constexpr int kQEnd = kQOff + 2 * kQHalf;
  static constexpr int kInboxSlots = 128 + 16;
  static constexpr int kPitch = D + 8;                    // halves
  static constexpr int kRowBytes = kPitch * 2;
  static constexpr bool kLateInbox = STAGES > 2;
  static constexpr int kInboxOff = kLateInbox ? kStageBytes : kQEnd;
  static constexpr int kBarOff = kLateInbox ? kQEnd : kInboxOff + kInboxSlots * kRowBytes;
  // kv_full[S] kv_empty[S] q_full s_full[2] s_empty[2] p_full[2] pv_done[2] inbox
  static constexpr int kNumBars = 2 * STAGES + 1 + 8 + 1;
  // then the TMEM address (16 bytes), the balanced mode's plan entry (an
  // int4) and its last-piece flag
  static constexpr int kPlanOff = kBarOff + kNumBars * 8 + 16;
  static constexpr int kTotal = kPlanOff + 32;
  static_assert(128 * kRowBytes <= kStageBytes, "staged rows fit in the ring's first stage");
  static_assert(!kLateInbox || kInboxOff + kInboxSlots * kRowBytes <= kQOff, "inbox fits in the ring");
  static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// TMA loads of one 128-token K/V tile into a ring stage: K then V, each two
// 64-column halves of 128 rows.  Prefix cache: one 3-D box of 128 rows per
// half (contiguous) or, paged, one 4-D box of K per 16-token page and half
// and one 5-D box of V per page holding both halves; past the prefix, the
// proposal's own rows (one box of 128 nodes).  A paged prefix tile's V
// lands page by page, [page][half][16 rows][64 columns] (w2_v_desc); every
// other tile's K and V, and a paged tile's K, half by half, [half][128
// rows][64 columns].
__device__ __forceinline__ void w2_issue_tile(const AttnArgs& a, const CUtensorMap* tm_ck,
                                              const CUtensorMap* tm_cv, const CUtensorMap* tm_cvp,
                                              const CUtensorMap* tm_tk, const CUtensorMap* tm_tv,
                                              uint8_t* stage, uint32_t bar, int t, int n_ptiles,
                                              int b, int g, int node0, int P, Pages8 pg) {
  using S = W2Smem<2>;  // the tile layout does not depend on the ring depth
  uint8_t* sk = stage;
  uint8_t* sv = stage + S::kTileBytes;
  if (t < n_ptiles) {
    const int tok0 = t * kW;
    if (a.layout == PF_KV_CONTIGUOUS) {
      mbar_arrive_expect_tx(bar, 2 * S::kTileBytes);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        tma_load_3d(smem_u32(sk + h * S::kHalfBytes), tm_ck, h * 64, tok0, b * a.Hkv + g, bar);
        tma_load_3d(smem_u32(sv + h * S::kHalfBytes), tm_cv, h * 64, tok0, b * a.Hkv + g, bar);
      }
    } else {
      const int npages = min(kW / PF_PAGE_SIZE, (P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
      mbar_arrive_expect_tx(bar, 2 * 2 * npages * PF_PAGE_SIZE * 128);
      const int pages[8] = {pg.lo.x, pg.lo.y, pg.lo.z, pg.lo.w, pg.hi.x, pg.hi.y, pg.hi.z, pg.hi.w};
#pragma unroll
      for (int p = 0; p < 8; ++p) {
        if (p >= npages) break;
#pragma unroll
        for (int h = 0; h < 2; ++h)
          tma_load_4d(smem_u32(sk + h * S::kHalfBytes + p * PF_PAGE_SIZE * 128), tm_ck, h * 64, 0,
                      g, pages[p], bar);
        tma_load_5d(smem_u32(sv + p * 2 * PF_PAGE_SIZE * 128), tm_cvp, 0, 0, 0, g, pages[p], bar);
      }
    }
  } else {
    const int j = t - n_ptiles;
    mbar_arrive_expect_tx(bar, 2 * S::kTileBytes);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      tma_load_3d(smem_u32(sk + h * S::kHalfBytes), tm_tk, h * 64, g, node0 + j * kW, bar);
      tma_load_3d(smem_u32(sv + h * S::kHalfBytes), tm_tv, h * 64, g, node0 + j * kW, bar);
    }
  }
}

// PV's B operand for keys 16 kt .. 16 kt + 15 of the tile's V at v0: in
// the page layout the 16 keys are one page (its halves 2 KB apart), else
// 16 rows of both 16 KB halves.
__device__ __forceinline__ uint64_t w2_v_desc(uint32_t v0, int kt, bool page_layout) {
  using S = W2Smem<2>;
  return page_layout
             ? umma_desc_sw128_lbo(v0 + kt * 2 * PF_PAGE_SIZE * 128, PF_PAGE_SIZE * 128, 1024)
             : umma_desc_sw128_lbo(v0 + kt * 16 * 128, S::kHalfBytes, 1024);
}

template <int STAGES, bool BAL>
__global__ void __launch_bounds__(kW2Threads, 1)
    attn_tc2_kernel(const __grid_constant__ CUtensorMap tm_q,
                    const __grid_constant__ CUtensorMap tm_tk,
                    const __grid_constant__ CUtensorMap tm_tv,
                    const __grid_constant__ CUtensorMap tm_ck,
                    const __grid_constant__ CUtensorMap tm_cv,
                    const __grid_constant__ CUtensorMap tm_cvp, const AttnArgs a) {
  using S = W2Smem<STAGES>;
  constexpr int kW2Stages = STAGES;
  constexpr int D = 128;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sKV = smem;
  uint8_t* sQ = smem + S::kQOff;
  __half* sInbox = reinterpret_cast<__half*>(smem + S::kInboxOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* kv_full = bars;
  uint64_t* kv_empty = bars + kW2Stages;
  uint64_t* q_full = bars + 2 * kW2Stages;
  uint64_t* s_full = q_full + 1;      // [2]
  uint64_t* s_empty = s_full + 2;     // [2]
  uint64_t* p_full = s_full + 4;      // [2]
  uint64_t* pv_done = s_full + 6;     // [2]
  uint64_t* inbox_full = s_full + 8;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + S::kNumBars);

  cg::cluster_group cluster = cg::this_cluster();
  const int nsplit = a.splits;
  const int split = (int)cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // PF_ATTN_EARLY_PREFETCH: as in attn_tc_kernel
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

  // This CTA's group and its piece of the group's tiles: split `split` of
  // the cluster, or (BAL) the item the plan gives it.
  int group = blockIdx.x / nsplit, part = split, nparts = nsplit, first_item = 0;
  int4* plan_slot = reinterpret_cast<int4*>(smem + S::kPlanOff);
  if constexpr (BAL) {
    if (warp == 0) {
      const PlanItem it = balanced_plan(a, (int)blockIdx.x, -1, nullptr, kW);
      if (lane == 0) *plan_slot = make_int4(it.group, it.j, it.k, it.first);
    }
    __syncthreads();
    const int4 pi = *plan_slot;
    if (pi.x < 0) {
      if (early) pdl_wait();  // the grid completes only after the preceding kernel
      return;                 // uniform over the CTA: no work for this item
    }
    group = pi.x;
    part = pi.y;
    nparts = pi.z;
    first_item = pi.w;
  }
  const int rb = group % a.rb_count;
  const int g = (group / a.rb_count) % a.Hkv;
  const int b = group / (a.rb_count * a.Hkv);
  const int node0 = a.cu_nodes[b];
  const int nn = a.cu_nodes[b + 1] - node0;
  const int P = a.prefix_len[b];
  if (node0 < 0 || nn < 1 || nn > a.max_nodes || node0 + nn > a.T || P < 0 ||
      P > a.max_prefix) {
    if (tid == 0 && split == 0 && rb == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
    return;  // uniform over the cluster (same b)
  }
  const int nfirst = rb * a.nb;
  if (nfirst >= nn) return;  // uniform over the cluster (same b, g, rb)
  const int rows = min(a.nb, nn - nfirst) * a.G;
  const int n_ptiles = (P + kW - 1) / kW;
  const int n_qtiles = (nn + kW - 1) / kW;
  const int ntiles = n_ptiles + n_qtiles;
  // Split s takes tiles [t_begin, t_end) of the order (proposal tiles,
  // prefix tiles), and processes its prefix tiles first (as in attn_tc_kernel).
  // (BAL: piece `part` of the group's `nparts`)
  const int t_begin = (int)((long long)ntiles * part / nparts);
  const int t_end = (int)((long long)ntiles * (part + 1) / nparts);
  const int my_tiles = t_end - t_begin;
  const int pre_lo = max(t_begin, n_qtiles);
  const int my_ptiles = max(0, t_end - pre_lo);
  auto tile_at = [&](int i) {
    return i < my_ptiles ? pre_lo - n_qtiles + i : n_ptiles + t_begin + (i - my_ptiles);
  };
  const int first = min(kW2Stages, my_tiles);

  if (tid == 0) {
    for (int i = 0; i < kW2Stages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), 1);
      mbar_init(smem_u32(&kv_empty[i]), 1);  // released by the tile's PV
    }
    mbar_init(smem_u32(q_full), 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_empty[i]), 128);
      mbar_init(smem_u32(&p_full[i]), 128);
      mbar_init(smem_u32(&pv_done[i]), 1);
    }
    mbar_init(smem_u32(inbox_full), 1);
    fence_mbar_init();
    Pages8 pg[kW2Stages];  // every first tile's page entries in one round trip
#pragma unroll
    for (int i = 0; i < kW2Stages; ++i)
      pg[i] = i < first ? kv_tile_pages8(a, tile_at(i), n_ptiles, b, P)
                        : no_pages8();
#pragma unroll
    for (int i = 0; i < kW2Stages; ++i)
      if (i < first && i < my_ptiles)
        w2_issue_tile(a, &tm_ck, &tm_cv, &tm_cvp, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                      smem_u32(&kv_full[i]), tile_at(i), n_ptiles, b, g, node0, P, pg[i]);
  }
  if (early) pdl_wait();
  if (tid == 0) {
    mbar_arrive_expect_tx(smem_u32(q_full), 2 * a.G * a.nb * 128);
#pragma unroll
    for (int h = 0; h < 2; ++h)
      tma_load_3d(smem_u32(sQ + h * S::kQHalf), &tm_q, h * 64, g * a.G, node0 + nfirst,
                  smem_u32(q_full));
    for (int i = 0; i < first; ++i)
      if (i >= my_ptiles)  // proposal tiles: no page entries
        w2_issue_tile(a, &tm_ck, &tm_cv, &tm_cvp, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                      smem_u32(&kv_full[i]), tile_at(i), n_ptiles, b, g, node0, P,
                      no_pages8());
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kW2TmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // peers may signal this CTA's inbox barrier once it is initialised (and,
  // with the inbox in the ring, once the ring is idle: after the loop)
  if (!S::kLateInbox && nsplit > 1) cluster_arrive_release();
  pdl_launch_dependents();

  float m_ref = -INFINITY, l = 0.f;   // softmax threads: running max (log2) and sum of their row
  if (warp == 0) {
    // ---------------- producer: refill the ring as the PVs release stages
    if (lane == 0) {
      for (int i = kW2Stages; i < my_tiles; ++i) {
        const int st = i % kW2Stages;
        const int t = tile_at(i);
        const Pages8 pg = kv_tile_pages8(a, t, n_ptiles, b, P);  // in flight during the wait
        if (!mbar_wait(smem_u32(&kv_empty[st]), ((i / kW2Stages) & 1) ^ 1, a.err)) break;
        w2_issue_tile(a, &tm_ck, &tm_cv, &tm_cvp, &tm_tk, &tm_tv, sKV + st * S::kStageBytes,
                      smem_u32(&kv_full[st]), t, n_ptiles, b, g, node0, P, pg);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = umma_idesc_bf16(128, kW);
      const uint32_t id_o = umma_idesc_bf16_bmn(128, D);
      bool ok = mbar_wait(smem_u32(q_full), 0, a.err);
      const uint32_t q0 = smem_u32(sQ);
      // S_n as soon as its tile has landed and the softmax has read S_{n-2}
      // out of the same TMEM buffer; PV_j as soon as P_j is in TMEM.
      int ns = 0, np = 0;
      unsigned idle = 0;
      unsigned long long t0 = 0;
      while (ok && np < my_tiles) {
        bool progressed = false;
        if (ns < my_tiles) {
          const int n = ns, st = n % kW2Stages, sb = n & 1;
          if (mbar_test_wait(smem_u32(&kv_full[st]), (n / kW2Stages) & 1) &&
              mbar_test_wait(smem_u32(&s_empty[sb]), ((n >> 1) & 1) ^ 1)) {
            tc_fence_after();
            const uint32_t k0 = smem_u32(sKV + st * S::kStageBytes);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              umma_bf16(tmem + sb * kW,
                        umma_desc_sw128(q0 + (kk >> 2) * S::kQHalf + (kk & 3) * 32),
                        umma_desc_sw128(k0 + (kk >> 2) * S::kHalfBytes + (kk & 3) * 32), id_s,
                        kk > 0);
            umma_commit(smem_u32(&s_full[sb]));
            ++ns;
            progressed = true;
          }
        }
        if (np < ns) {
          const int j = np, pb = j & 1, stj = j % kW2Stages;
          if (mbar_test_wait(smem_u32(&p_full[pb]), (j >> 1) & 1)) {
            tc_fence_after();
            const uint32_t v0 = smem_u32(sKV + stj * S::kStageBytes + S::kTileBytes);
            const bool vpage = a.layout != PF_KV_CONTIGUOUS && tile_at(j) < n_ptiles;
#pragma unroll
            for (int kt = 0; kt < kW / 16; ++kt)
              umma_bf16_tmem_a(tmem + kColO, tmem + kColP + pb * 64 + kt * 8, w2_v_desc(v0, kt, vpage),
                               id_o, (j > 0 || kt > 0) ? 1u : 0u);
            umma_commit(smem_u32(&pv_done[pb]));
            umma_commit(smem_u32(&kv_empty[stj]));
            ++np;
            progressed = true;
          }
        }
        // bounded like mbar_wait: give up (and flag) after kWaitLimitNs
        // without progress
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
    // ---------------- softmax / correction: one row per thread
    const int quad = warp & 3;
    const int rl = quad * 32 + lane;       // row within the block (its TMEM lane)
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
      const int st = i % kW2Stages;
      ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[sb]), (i >> 1) & 1, a.err));
      if (!ok) break;  // warp-uniform
      tc_fence_after();
      uint32_t sraw[kW];
#pragma unroll
      for (int c0 = 0; c0 < kW; c0 += 32)
        tmem_ld_32(tmem + lane_base + sb * kW + c0, *reinterpret_cast<uint32_t(*)[32]>(&sraw[c0]));
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(smem_u32(&s_empty[sb]));
      float sv[kW];
#pragma unroll
      for (int c = 0; c < kW; ++c) sv[c] = __uint_as_float(sraw[c]);

      const int t = tile_at(i);
      const bool is_prefix = t < n_ptiles;
      const int valid = is_prefix ? min(kW, P - t * kW) : kW;
      if (!is_prefix || valid < kW) {
        // masked tile: prefix columns past the end, or proposal columns
        // that are not ancestors of this row's node (columns 0..63 are
        // nodes 0..63, columns 64..127 nodes 64..127)
        uint64_t v0, v1;
        if (is_prefix) {
          v0 = valid >= 64 ? ~0ull : ((1ull << valid) - 1ull);
          v1 = valid >= 128 ? ~0ull : (valid <= 64 ? 0ull : ((1ull << (valid - 64)) - 1ull));
        } else {
          v0 = mk0;
          v1 = mk1;
        }
#pragma unroll
        for (int c = 0; c < 64; ++c) {
          if (!((v0 >> c) & 1ull)) sv[c] = -INFINITY;
          if (!((v1 >> c) & 1ull)) sv[64 + c] = -INFINITY;
        }
      }
      // row maximum of the raw scores (scale > 0 commutes with max): three-
      // input maxima, 128 -> 43 -> 15 -> 5 -> 2 -> 1
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
      const bool resc = m_ref != -INFINITY && m_new > m_ref + kW2RescaleLog2;
      if (m_ref == -INFINITY) m_ref = m_new;
      if (__any_sync(0xffffffffu, resc)) {
        // O must hold exactly the tiles before i: wait for PV_{i-1}.
        if (i >= 1) mbar_wait(smem_u32(&pv_done[(i - 1) & 1]), ((i - 1) >> 1) & 1, a.err);
        tc_fence_after();
        const float alpha = resc ? ex2_approx(m_ref - m_new) : 1.f;
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t ov[32];
          tmem_ld_32(tmem + lane_base + kColO + c0, ov);
          tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 32; ++c) ov[c] = __float_as_uint(__uint_as_float(ov[c]) * alpha);
          tmem_st_32(tmem + lane_base + kColO + c0, ov);
        }
        tmem_st_wait();
        if (resc) {
          l *= alpha;
          m_ref = m_new;
        }
      }
      // p = 2^(s * scale_log2 - m): one paired FMA per two scores, one MUFU
      // per score; the row sum in four paired accumulators
      const float neg_mu = m_ref == -INFINITY ? 0.f : -m_ref;
      const unsigned long long sc2 = f32x2_pack(a.scale_log2, a.scale_log2);
      const unsigned long long mu2 = f32x2_pack(neg_mu, neg_mu);
      unsigned long long rs2[4] = {0ull, 0ull, 0ull, 0ull};
      uint32_t pk[kW / 2];
#pragma unroll
      for (int c = 0; c < kW / 2; ++c) {
        float x0, x1;
        f32x2_unpack(ffma2(f32x2_pack(sv[2 * c], sv[2 * c + 1]), sc2, mu2), x0, x1);
        const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
        rs2[c & 3] = fadd2(rs2[c & 3], f32x2_pack(p0, p1));
        pk[c] = pack_bf16(p0, p1);
      }
      float r0, r1;
      f32x2_unpack(fadd2(fadd2(rs2[0], rs2[1]), fadd2(rs2[2], rs2[3])), r0, r1);
      l += r0 + r1;
      // P buffer sb was last read by PV_{i-2}.
      if (i >= 2) mbar_wait(smem_u32(&pv_done[sb]), ((i - 2) >> 1) & 1, a.err);
      tc_fence_after();
      tmem_st_32(tmem + lane_base + kColP + sb * 64,
                 *reinterpret_cast<uint32_t(*)[32]>(&pk[0]));
      tmem_st_32(tmem + lane_base + kColP + sb * 64 + 32,
                 *reinterpret_cast<uint32_t(*)[32]>(&pk[32]));
      tmem_st_wait();
      if (valid < kW) {
        // Cache rows past the prefix end may hold anything (even NaN bit
        // patterns): zero their V so masked columns contribute exactly 0.
        // The rows from `valid` on are one contiguous run per 64-column half.
        uint4* vt = reinterpret_cast<uint4*>(sKV + st * S::kStageBytes + S::kTileBytes);
        const int per_half = (kW - valid) * 8;   // 16-byte chunks past the end
        if (a.layout == PF_KV_CONTIGUOUS) {
#pragma unroll
          for (int h = 0; h < 2; ++h)
            for (int c = rl; c < per_half; c += 128)
              vt[h * kW * 8 + valid * 8 + c] = make_uint4(0, 0, 0, 0);
        } else {
          // page layout: row r of half h at chunk (r / 16) * 256 + h * 128 + (r % 16) * 8
#pragma unroll
          for (int h = 0; h < 2; ++h)
            for (int c = rl; c < per_half; c += 128) {
              const int r = valid + (c >> 3);
              vt[(r >> 4) * 256 + h * 128 + (r & 15) * 8 + (c & 7)] = make_uint4(0, 0, 0, 0);
            }
        }
        fence_proxy_async_smem();
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&p_full[sb]));
    }
    // O of this row is complete once the last PV has landed
    if (my_tiles > 0)
      mbar_wait(smem_u32(&pv_done[(my_tiles - 1) & 1]), ((my_tiles - 1) >> 1) & 1, a.err);
  }
  __syncwarp();  // the producer and MMA lanes rejoin their warps before the barriers

  // ---- epilogue: each softmax thread reads its row of O / l from TMEM
  const bool has_row = warp >= 2;
  const int r = (warp & 3) * 32 + lane;
  const uint32_t o_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16) + kColO;
  const float inv_l = (my_tiles > 0 && l > 0.f) ? 1.f / l : 0.f;

  if (nsplit == 1) {
    // ---- single split: O / l is the output -- or (BAL, a group spread over
    // several CTAs) this piece's normalised partial and log2-sum-exp
    const bool piece = BAL && nparts > 1;
    if (has_row) {
      uint32_t ov[D];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32)
        tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
      tmem_ld_wait();
      if (piece && r < rows) {
        if (!(inv_l > 0.f)) {
          // no column reached this row in this piece: 0 with lse = -inf
#pragma unroll
          for (int c = 0; c < D; ++c) ov[c] = 0u;
        }
        __half* dst = reinterpret_cast<__half*>(a.ws) + ((size_t)blockIdx.x * a.bm + r) * S::kPitch;
#pragma unroll
        for (int c = 0; c < D; c += 8) {
          uint4 pk;
          pk.x = pack_half(__uint_as_float(ov[c]) * inv_l, __uint_as_float(ov[c + 1]) * inv_l);
          pk.y = pack_half(__uint_as_float(ov[c + 2]) * inv_l, __uint_as_float(ov[c + 3]) * inv_l);
          pk.z = pack_half(__uint_as_float(ov[c + 4]) * inv_l, __uint_as_float(ov[c + 5]) * inv_l);
          pk.w = pack_half(__uint_as_float(ov[c + 6]) * inv_l, __uint_as_float(ov[c + 7]) * inv_l);
          *reinterpret_cast<uint4*>(dst + c) = pk;
        }
        *reinterpret_cast<float*>(dst + D) = inv_l > 0.f ? m_ref + __log2f(l) : -INFINITY;
        __threadfence();  // before this piece's ticket (after the barrier below)
      } else if (r < rows) {
        const int node = node0 + nfirst + r / a.G;
        const int h = g * a.G + r % a.G;
        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(a.out) + ((size_t)node * a.Hq + h) * D;
#pragma unroll
        for (int c = 0; c < D; c += 8) {
          uint4 pk;
          pk.x = pack_bf16(__uint_as_float(ov[c]) * inv_l, __uint_as_float(ov[c + 1]) * inv_l);
          pk.y = pack_bf16(__uint_as_float(ov[c + 2]) * inv_l, __uint_as_float(ov[c + 3]) * inv_l);
          pk.z = pack_bf16(__uint_as_float(ov[c + 4]) * inv_l, __uint_as_float(ov[c + 5]) * inv_l);
          pk.w = pack_bf16(__uint_as_float(ov[c + 6]) * inv_l, __uint_as_float(ov[c + 7]) * inv_l);
          *reinterpret_cast<uint4*>(dst + c) = pk;
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tmem, kW2TmemCols);
    }
    if (piece) {
      // the group's last piece to arrive merges every piece's partial
      int* last_slot = reinterpret_cast<int*>(plan_slot + 1);
      if (tid == 0)
        *last_slot = ticket_arrive_last(&group_tickets(a)[group], a.epoch, nparts, a.err) ? 1 : 0;
      __syncthreads();
      if (*last_slot) {
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out);
        // The pieces' partials sit in consecutive slots: as many as the idle
        // ring holds come in with one bulk copy (one L2 round trip instead of
        // one per merged row); more are merged straight from L2.
        constexpr int kSlotBytes = 128 * S::kRowBytes;  // a.bm = 128 rows
        constexpr int kStaged = STAGES * S::kStageBytes / kSlotBytes;
        if (nparts <= kStaged) {
          if (tid == 0) {
            fence_proxy_async_global();  // the pieces' stores, acquired above, before the copy
            const uint32_t bytes = (uint32_t)(nparts * kSlotBytes);
            mbar_arrive_expect_tx(smem_u32(inbox_full), bytes);
            bulk_load_g2s(smem_u32(smem),
                          static_cast<const uint8_t*>(a.ws) + (size_t)first_item * kSlotBytes,
                          bytes, smem_u32(inbox_full));
          }
          if (mbar_wait(smem_u32(inbox_full), 0, a.err))
            merge_rows_smem<D, kStaged>(a, smem, S::kRowBytes, kSlotBytes, nparts, rows, 0,
                                        node0 + nfirst, g, tid, kW2Threads);
        } else {
          for (int it = tid; it < rows * (D / 8); it += kW2Threads) {
            const int rr = it / (D / 8), c8 = it % (D / 8);
            const int node = node0 + nfirst + rr / a.G;
            const int h = g * a.G + rr % a.G;
            merge_pieces_row<D>(a, first_item, nparts, rr, c8, out + ((size_t)node * a.Hq + h) * D);
          }
        }
      }
    }
    return;
  }
  // ---- split-KV merge, as in attn_tc_kernel (kWG = 1): each row's
  // normalised partial and its log2-sum-exp are staged in the idle ring,
  // one bulk copy per peer moves the rows it merges into its inbox, and
  // every CTA merges its own rows from its inbox.
  const int per = (rows + nsplit - 1) / nsplit;
  const int cnt_mine = max(0, min(per, rows - split * per));
  __half* stage_rows = reinterpret_cast<__half*>(smem);
  if (S::kLateInbox) {
    // every PV of this CTA has completed (the softmax threads waited for the
    // last one): the ring is idle, so peers may now fill the inbox it holds
    __syncthreads();
    cluster_arrive_release();
  }
  if (tid == 0)
    mbar_arrive_expect_tx(smem_u32(inbox_full), (uint32_t)(nsplit * cnt_mine * S::kRowBytes));
  if (has_row) {
    uint32_t ov[D];  // the whole O row: all TMEM loads in flight behind one wait
#pragma unroll
    for (int c0 = 0; c0 < D; c0 += 32)
      tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
    tmem_ld_wait();
    if (!(inv_l > 0.f)) {
      // no column reached this row in this split (a split without tiles
      // never writes O): its partial is 0 with lse = -inf, whatever the
      // unwritten accumulator holds (0 * NaN would poison the merge)
#pragma unroll
      for (int c = 0; c < D; ++c) ov[c] = 0u;
    }
    if (r < rows) {
      __half* dst = stage_rows + r * S::kPitch;
#pragma unroll
      for (int c = 0; c < D; c += 8) {
        uint4 pk;
        pk.x = pack_half(__uint_as_float(ov[c]) * inv_l, __uint_as_float(ov[c + 1]) * inv_l);
        pk.y = pack_half(__uint_as_float(ov[c + 2]) * inv_l, __uint_as_float(ov[c + 3]) * inv_l);
        pk.z = pack_half(__uint_as_float(ov[c + 4]) * inv_l, __uint_as_float(ov[c + 5]) * inv_l);
        pk.w = pack_half(__uint_as_float(ov[c + 6]) * inv_l, __uint_as_float(ov[c + 7]) * inv_l);
        *reinterpret_cast<uint4*>(dst + c) = pk;
      }
      *reinterpret_cast<float*>(dst + D) = inv_l > 0.f ? m_ref + __log2f(l) : -INFINITY;
    }
  }
  fence_proxy_async_smem();  // staged rows are read by the bulk-copy engine
  tc_fence_before();
  __syncthreads();
  cluster_wait_acquire();    // every peer's inbox is ready to be filled
  if (tid < nsplit) {
    const int q = tid;
    const int cnt = min(per, rows - q * per);
    if (cnt > 0) {
      const uint32_t src = smem_u32(stage_rows + q * per * S::kPitch);
      const uint32_t dst = mapa_cluster(smem_u32(sInbox + split * per * S::kPitch), q);
      bulk_copy_s2cluster(dst, src, (uint32_t)(cnt * S::kRowBytes),
                          mapa_cluster(smem_u32(inbox_full), q));
      bulk_commit_group();
    }
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kW2TmemCols);
  }
  if (cnt_mine > 0) mbar_wait(smem_u32(inbox_full), 0, a.err);
  inbox_merge<D, kW2Threads, S::kPitch>(a, sInbox, rows, split, per, nsplit, node0 + nfirst, g,
                                        tid);
  // this CTA's staged rows must stay readable until its copies have left
  if (tid < nsplit) bulk_wait_read_all();
}

}  // namespace

template <int STAGES>
static int tc2_smem_bytes() {
  return W2Smem<STAGES>::kTotal + 1024;
}

template <int STAGES>
static int tc2_max_active_clusters_impl(int cluster) {
  const int smem = tc2_smem_bytes<STAGES>();
  static DeviceMemo limit;
  if (ensure_smem_limit((const void*)attn_tc2_kernel<STAGES, false>, smem, limit) != cudaSuccess)
    return 0;
  if (cluster > 8 && cudaFuncSetAttribute(attn_tc2_kernel<STAGES, false>,
                                          cudaFuncAttributeNonPortableClusterSizeAllowed,
                                          1) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cluster);
  cfg.blockDim = dim3(kW2Threads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = cluster;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_tc2_kernel<STAGES, false>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

template <int STAGES, bool BAL>
static cudaError_t launch_tc2(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  const int smem = tc2_smem_bytes<STAGES>();
  static DeviceMemo limit;
  static DeviceMemo nonportable;
  cudaError_t e = ensure_smem_limit((const void*)attn_tc2_kernel<STAGES, BAL>, smem, limit);
  if (e != cudaSuccess) return e;
  if (BAL) {
    // one CTA per item, no cluster
    return launch_ex(attn_tc2_kernel<STAGES, BAL>, dim3(a.items), dim3(kW2Threads), smem, s, 1,
                     pdl, m.q, m.tk, m.tv, m.ck, m.cv, m.cv_page, a);
  }
  if (a.splits > 8) {
    e = ensure_nonportable_cluster((const void*)attn_tc2_kernel<STAGES, BAL>, nonportable);
    if (e != cudaSuccess) return e;
  }
  const dim3 grid(a.B * a.Hkv * a.rb_count * a.splits);
  return launch_ex(attn_tc2_kernel<STAGES, BAL>, grid, dim3(kW2Threads), smem, s, a.splits, pdl,
                   m.q, m.tk, m.tv, m.ck, m.cv, m.cv_page, a);
}

// Ring depth: 3 stages (inbox in the ring, peers send after every CTA of
// the cluster has left its loop) unless the caller asks for 2.
int attention_tc2_max_active_clusters(int cluster, int stages) {
  return stages == 2 ? tc2_max_active_clusters_impl<2>(cluster)
                     : tc2_max_active_clusters_impl<3>(cluster);
}

cudaError_t launch_attention_tc2(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl,
                                 int stages, bool balanced) {
  if (balanced) return launch_tc2<3, true>(a, m, s, pdl);
  return stages == 2 ? launch_tc2<2, false>(a, m, s, pdl) : launch_tc2<3, false>(a, m, s, pdl);
}

}  // namespace pf
