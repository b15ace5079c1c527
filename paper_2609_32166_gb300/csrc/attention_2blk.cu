// Tree-masked GQA attention (Section 3.2) on the tcgen05 tensor cores for
// KV heads with more than 128 query rows: one CTA holds two 128-row blocks
// of the same (sequence, KV head) and brings each 128-token K/V tile into
// shared memory once for both, so every K/V byte that enters an SM serves up
// to 256 query rows (the 7B trees and the 8-sequence batch have 7 query heads
// per KV head and 32 to 128 nodes: 224 to 896 rows per KV head).  Same
// contract, tile order and cluster split-KV merge as attn_tc2_kernel.
//
//   warp 0     TMA producer: Q of both blocks, then each tile's K and V as
//              separate 32 KB units through a ring of five units (K_i, V_i,
//              K_{i+1}, ...), so loads run two and a half tiles ahead
//   warp 1     TMEM owner and MMA issuer (one thread), in a fixed order that
//              keeps the tensor pipe busy while each block's softmax runs:
//                S_A(0) S_B(0), then per tile i: PV_A(i) S_A(i+1) PV_B(i) S_B(i+1)
//              S_X = Q_X K^T (M = 128, N = 128) into block X's S columns,
//              O_X += P_X V (A = P_X from TMEM, N = D)
//   warps 2-5  softmax of block A, one row per thread (its TMEM lane)
//   warps 6-9  softmax of block B
//
// P_X (bf16 pairs) is written over the first 64 of S_X's columns.  The next
// S_X MMA, which overwrites them, is issued after PV_X by the same thread,
// and one thread's MMAs run through the tensor pipe in issue order; its
// commit also tells the softmax that PV_X has finished reading P_X.
//
// TMEM columns: S_A 0..127, O_A 128..255, S_B 256..383, O_B 384..511.
#include <cuda_fp16.h>

#include "attn_common.cuh"

namespace cg = cooperative_groups;

namespace pf {

namespace {

constexpr int kW = 128;               // tokens per K/V tile
constexpr int kBThreads = 320;        // producer, MMA, two softmax warpgroups
constexpr int kUnits = 5;             // ring units of one K or one V tile
constexpr uint32_t kBTmemCols = 512;
constexpr uint32_t kBlockCols = 256;  // S then O of one block
constexpr float kBRescaleLog2 = 8.f;

// The ring (five 32 KB units) then Q (two blocks of 128 rows x 128
// columns); after the loop the idle ring holds the staged partial rows
// (256 at most) and, behind them, the merge inbox.
struct BSmem {
  static constexpr int D = 128;
  static constexpr int kHalfBytes = kW * 128;        // 128 rows x 64 columns of bf16
  static constexpr int kUnitBytes = 2 * kHalfBytes;  // one tile's K or V
  static constexpr int kQOff = kUnits * kUnitBytes;
  static constexpr int kQHalf = 128 * 128;
  static constexpr int kQBlock = 2 * kQHalf;
  static constexpr int kQEnd = kQOff + 2 * kQBlock;
  static constexpr int kPitch = D + 8;               // halves
  static constexpr int kRowBytes = kPitch * 2;
  static constexpr int kInboxOff = 256 * kRowBytes;
  static constexpr int kInboxSlots = 256 + 16;
  static constexpr int kBarOff = kQEnd;
  // u_full[5] u_empty[5] q_full s_full[2] p_full[2] pv_done[2] inbox
  static constexpr int kNumBars = 2 * kUnits + 1 + 6 + 1;
  static constexpr int kTotal = kBarOff + kNumBars * 8 + 16;  // + the TMEM address
  static_assert(kInboxOff % 16 == 0, "bulk copies need 16-byte aligned rows");
  static_assert(kInboxOff + kInboxSlots * kRowBytes <= kQOff, "staged rows and inbox fit in the ring");
  static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// TMA loads of tile t's K (v = false) or V (v = true) into one ring unit,
// arming `bar` with the bytes they bring.  Prefix cache, contiguous: two
// 3-D boxes of 128 rows, one per 64-column half ([half][row][column]);
// paged: K two 4-D boxes per 16-token page (the same layout), V one 5-D box
// per page holding both halves (the unit lands [page][half][row][column]);
// past the prefix, the proposal's own rows (two 3-D boxes of 128 nodes).
__device__ __forceinline__ void issue_unit(const AttnArgs& a, bool v, const CUtensorMap* tm_c,
                                           const CUtensorMap* tm_cvp, const CUtensorMap* tm_t,
                                           uint8_t* dst, uint32_t bar, int t, int n_ptiles, int b,
                                           int g, int node0, int P, const Pages8& pg) {
  using S = BSmem;
  if (t < n_ptiles) {
    const int tok0 = t * kW;
    if (a.layout == PF_KV_CONTIGUOUS) {
      mbar_arrive_expect_tx(bar, S::kUnitBytes);
#pragma unroll
      for (int h = 0; h < 2; ++h)
        tma_load_3d(smem_u32(dst + h * S::kHalfBytes), tm_c, h * 64, tok0, b * a.Hkv + g, bar);
    } else {
      const int npages = min(kW / PF_PAGE_SIZE, (P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
      mbar_arrive_expect_tx(bar, npages * 2 * PF_PAGE_SIZE * 128);
      const int pages[8] = {pg.lo.x, pg.lo.y, pg.lo.z, pg.lo.w, pg.hi.x, pg.hi.y, pg.hi.z, pg.hi.w};
#pragma unroll
      for (int p = 0; p < 8; ++p) {
        if (p >= npages) break;
        if (v) {
          tma_load_5d(smem_u32(dst + p * 2 * PF_PAGE_SIZE * 128), tm_cvp, 0, 0, 0, g, pages[p],
                      bar);
        } else {
#pragma unroll
          for (int h = 0; h < 2; ++h)
            tma_load_4d(smem_u32(dst + h * S::kHalfBytes + p * PF_PAGE_SIZE * 128), tm_c, h * 64,
                        0, g, pages[p], bar);
        }
      }
    }
  } else {
    const int j = t - n_ptiles;
    mbar_arrive_expect_tx(bar, S::kUnitBytes);
#pragma unroll
    for (int h = 0; h < 2; ++h)
      tma_load_3d(smem_u32(dst + h * S::kHalfBytes), tm_t, h * 64, g, node0 + j * kW, bar);
  }
}

// PV's B operand for keys 16 kt .. 16 kt + 15 of the V unit at v0: in the
// page layout the 16 keys are one page (its halves 2 KB apart), else 16 rows
// of both 16 KB halves.
__device__ __forceinline__ uint64_t blk_v_desc(uint32_t v0, int kt, bool page_layout) {
  return page_layout
             ? umma_desc_sw128_lbo(v0 + kt * 2 * PF_PAGE_SIZE * 128, PF_PAGE_SIZE * 128, 1024)
             : umma_desc_sw128_lbo(v0 + kt * 16 * 128, BSmem::kHalfBytes, 1024);
}

__global__ void __launch_bounds__(kBThreads, 1)
    attn_2blk_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_tk,
                     const __grid_constant__ CUtensorMap tm_tv,
                     const __grid_constant__ CUtensorMap tm_ck,
                     const __grid_constant__ CUtensorMap tm_cv,
                     const __grid_constant__ CUtensorMap tm_cvp, const AttnArgs a,
                     const __grid_constant__ TeamPlan tp) {
  using S = BSmem;
  constexpr int D = 128;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem + S::kQOff;
  __half* sInbox = reinterpret_cast<__half*>(smem + S::kInboxOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* u_full = bars;
  uint64_t* u_empty = bars + kUnits;
  uint64_t* q_full = bars + 2 * kUnits;
  uint64_t* s_full = q_full + 1;   // [block]
  uint64_t* p_full = q_full + 3;   // [block]
  uint64_t* pv_done = q_full + 5;  // [block]
  uint64_t* inbox_full = q_full + 7;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + S::kNumBars);

  cg::cluster_group cluster = cg::this_cluster();
  const int nsplit = a.splits;
  const int split = (int)cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // PF_ATTN_EARLY_PREFETCH: the first prefix units are requested before the
  // dependency wait (as in attn_tc_kernel)
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

  // group = (sequence, KV head, pair of row blocks); a.nb nodes per CTA,
  // a.nb / 2 per block.  One group per cluster, its pieces the cluster's
  // CTAs; or (team plan) a team of the cluster's CTAs per group.
  int group = blockIdx.x / nsplit, part = split, nparts = nsplit, base = 0;
  if (a.team) {
    const uint32_t e = tp.e[blockIdx.x];
    group = (int)(e & 0xfffu);
    part = (int)(e >> 12) & 31;
    nparts = (int)(e >> 17) & 31;
    base = (int)(e >> 22) & 31;
  }
  // A CTA without work leaves at once -- with the whole cluster in the
  // one-group layout, alone in a team plan, after its share of the one
  // cluster barrier that its cluster's teams pass through.
  auto leave = [&]() {
    if (early) pdl_wait();  // the grid completes only after the preceding kernel
    if (a.team && nsplit > 1) {
      __syncthreads();
      cluster_arrive_release();
      cluster_wait_acquire();
    }
  };
  if (nparts < 1) {
    leave();
    return;
  }
  const int rb = group % a.rb_count;
  const int g = (group / a.rb_count) % a.Hkv;
  const int b = min(group / (a.rb_count * a.Hkv), a.B - 1);
  const int node0 = a.cu_nodes[b];
  const int nn = a.cu_nodes[b + 1] - node0;
  const int P = a.prefix_len[b];
  if (node0 < 0 || nn < 1 || nn > a.max_nodes || node0 + nn > a.T || P < 0 ||
      P > a.max_prefix) {
    if (tid == 0 && part == 0 && rb == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
    leave();
    return;  // uniform over the group
  }
  const int nbh = a.nb / 2;
  const int nfirst = rb * a.nb;
  if (nfirst >= nn) {
    leave();
    return;  // uniform over the group (same b, g, rb)
  }
  const int rows_a = min(nbh, nn - nfirst) * a.G;
  const int rows_b = max(0, min(nbh, nn - nfirst - nbh)) * a.G;
  const bool has_b = rows_b > 0;
  const int rows = rows_a + rows_b;  // CTA row r is node nfirst + r / G, head r % G
  const int n_ptiles = (P + kW - 1) / kW;
  const int n_qtiles = (nn + kW - 1) / kW;
  const int ntiles = n_ptiles + n_qtiles;
  // Split s takes tiles [t_begin, t_end) of the order (proposal tiles,
  // prefix tiles) and processes its prefix tiles first.
  const int t_begin = (int)((long long)ntiles * part / nparts);
  const int t_end = (int)((long long)ntiles * (part + 1) / nparts);
  const int my_tiles = t_end - t_begin;
  const int pre_lo = max(t_begin, n_qtiles);
  const int my_ptiles = max(0, t_end - pre_lo);
  auto tile_at = [&](int i) {
    return i < my_ptiles ? pre_lo - n_qtiles + i : n_ptiles + t_begin + (i - my_ptiles);
  };
  // unit u: K (u even) or V (u odd) of the CTA's tile u / 2, in ring unit u % 5
  const int n_units = 2 * my_tiles;
  const int first_units = min(kUnits, n_units);

  if (tid == 0) {
    for (int i = 0; i < kUnits; ++i) {
      mbar_init(smem_u32(&u_full[i]), 1);
      mbar_init(smem_u32(&u_empty[i]), 1);  // released by the unit's last MMA
    }
    mbar_init(smem_u32(q_full), 1);
    for (int x = 0; x < 2; ++x) {
      mbar_init(smem_u32(&s_full[x]), 1);
      mbar_init(smem_u32(&p_full[x]), 128);
      mbar_init(smem_u32(&pv_done[x]), 1);
    }
    mbar_init(smem_u32(inbox_full), 1);
    fence_mbar_init();
    Pages8 pg[3];  // the first units' page entries (tiles 0..2) in one round trip
#pragma unroll
    for (int i = 0; i < 3; ++i)
      pg[i] = 2 * i < first_units && i < my_ptiles ? kv_tile_pages8(a, tile_at(i), n_ptiles, b, P)
                                                    : no_pages8();
#pragma unroll
    for (int u = 0; u < kUnits; ++u) {
      const int i = u >> 1;
      if (u < first_units && i < my_ptiles)
        issue_unit(a, u & 1, (u & 1) ? &tm_cv : &tm_ck, &tm_cvp, (u & 1) ? &tm_tv : &tm_tk,
                   smem + u * S::kUnitBytes, smem_u32(&u_full[u]), tile_at(i), n_ptiles, b, g,
                   node0, P, pg[i]);
    }
  }
  if (early) pdl_wait();
  if (tid == 0) {
    const int nq = has_b ? 2 : 1;
    mbar_arrive_expect_tx(smem_u32(q_full), nq * 2 * a.G * nbh * 128);
    for (int x = 0; x < nq; ++x)
#pragma unroll
      for (int h = 0; h < 2; ++h)
        tma_load_3d(smem_u32(sQ + x * S::kQBlock + h * S::kQHalf), &tm_q, h * 64, g * a.G,
                    node0 + nfirst + x * nbh, smem_u32(q_full));
    for (int u = 0; u < first_units; ++u)
      if ((u >> 1) >= my_ptiles)  // proposal tiles: no page entries
        issue_unit(a, u & 1, (u & 1) ? &tm_cv : &tm_ck, &tm_cvp, (u & 1) ? &tm_tv : &tm_tk,
                   smem + u * S::kUnitBytes, smem_u32(&u_full[u]), tile_at(u >> 1), n_ptiles, b,
                   g, node0, P, no_pages8());
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kBTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();

  float m_ref = -INFINITY, l = 0.f;  // softmax threads: running max (log2) and sum of their row
  if (warp == 0) {
    // ---------------- producer: refill the ring as the MMAs release units
    if (lane == 0) {
      Pages8 pg = no_pages8();
      for (int u = first_units; u < n_units; ++u) {
        const int i = u >> 1, slot = u % kUnits;
        const int t = tile_at(i);
        if (!(u & 1) || u == first_units)
          pg = kv_tile_pages8(a, t, n_ptiles, b, P);  // in flight during the wait
        if (!mbar_wait(smem_u32(&u_empty[slot]), ((u / kUnits) & 1) ^ 1, a.err)) break;
        issue_unit(a, u & 1, (u & 1) ? &tm_cv : &tm_ck, &tm_cvp, (u & 1) ? &tm_tv : &tm_tk,
                   smem + slot * S::kUnitBytes, smem_u32(&u_full[slot]), t, n_ptiles, b, g, node0,
                   P, pg);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0 && my_tiles > 0) {
      const uint32_t id_s = umma_idesc_bf16(128, kW);
      const uint32_t id_o = umma_idesc_bf16_bmn(128, D);
      const int last_blk = has_b ? 1 : 0;  // the block whose MMA releases a unit
      auto unit_landed = [&](int u) {
        return mbar_wait(smem_u32(&u_full[u % kUnits]), (u / kUnits) & 1, a.err);
      };
      auto issue_s = [&](int x, int i) {
        const int slot = (2 * i) % kUnits;
        const uint32_t k0 = smem_u32(smem + slot * S::kUnitBytes);
        const uint32_t q0 = smem_u32(sQ + x * S::kQBlock);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk)
          umma_bf16(tmem + x * kBlockCols,
                    umma_desc_sw128(q0 + (kk >> 2) * S::kQHalf + (kk & 3) * 32),
                    umma_desc_sw128(k0 + (kk >> 2) * S::kHalfBytes + (kk & 3) * 32), id_s,
                    kk > 0);
        umma_commit(smem_u32(&s_full[x]));
        if (x == last_blk) umma_commit(smem_u32(&u_empty[slot]));
      };
      auto issue_pv = [&](int x, int i) {
        const int slot = (2 * i + 1) % kUnits;
        const uint32_t v0 = smem_u32(smem + slot * S::kUnitBytes);
        const bool vpage = a.layout != PF_KV_CONTIGUOUS && tile_at(i) < n_ptiles;
#pragma unroll
        for (int kt = 0; kt < kW / 16; ++kt)
          umma_bf16_tmem_a(tmem + x * kBlockCols + 128, tmem + x * kBlockCols + kt * 8,
                           blk_v_desc(v0, kt, vpage), id_o, (i > 0 || kt > 0) ? 1u : 0u);
        umma_commit(smem_u32(&pv_done[x]));
        if (x == last_blk) umma_commit(smem_u32(&u_empty[slot]));
      };
      bool ok = mbar_wait(smem_u32(q_full), 0, a.err) && unit_landed(0);
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        if (has_b) issue_s(1, 0);
      }
      for (int i = 0; ok && i < my_tiles; ++i) {
        const bool more = i + 1 < my_tiles;
        ok = mbar_wait(smem_u32(&p_full[0]), i & 1, a.err) && unit_landed(2 * i + 1);
        if (!ok) break;
        tc_fence_after();
        issue_pv(0, i);
        if (more) {
          ok = unit_landed(2 * i + 2);
          if (!ok) break;
          tc_fence_after();
          issue_s(0, i + 1);
        }
        if (has_b) {
          ok = mbar_wait(smem_u32(&p_full[1]), i & 1, a.err);
          if (!ok) break;
          tc_fence_after();
          issue_pv(1, i);
          if (more) issue_s(1, i + 1);  // K_{i+1} has landed (checked for block A)
        }
      }
    }
  } else {
    // ---------------- softmax / correction of block x: one row per thread
    const int x = (warp - 2) >> 2;
    const int quad = warp & 3;
    const int rl = quad * 32 + lane;  // row within the block (its TMEM lane)
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const uint32_t col_s = x * kBlockCols, col_o = col_s + 128;
    const int rows_x = x ? rows_b : rows_a;
    if (rows_x > 0) {  // uniform over the warpgroup
      uint64_t mk0 = 0, mk1 = 0;
      if (rl < rows_x) {
        const int node = node0 + nfirst + x * nbh + rl / a.G;
        mk0 = a.mask[2 * node];
        mk1 = a.mask[2 * node + 1];
      }
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[x]), i & 1, a.err));
        if (!ok) break;  // warp-uniform
        tc_fence_after();
        const int t = tile_at(i);
        const bool is_prefix = t < n_ptiles;
        const int valid = is_prefix ? min(kW, P - t * kW) : kW;
        // masked tile: prefix columns past the end, or proposal columns that
        // are not ancestors of this row's node (columns 0..63 are nodes
        // 0..63, columns 64..127 nodes 64..127)
        const bool masked = !is_prefix || valid < kW;
        uint64_t vm[2] = {mk0, mk1};
        if (is_prefix) {
          vm[0] = valid >= 64 ? ~0ull : ((1ull << valid) - 1ull);
          vm[1] = valid >= 128 ? ~0ull : (valid <= 64 ? 0ull : ((1ull << (valid - 64)) - 1ull));
        }
        // The scores are read from TMEM twice, 64 columns at a time (the row
        // maximum, then P), so that no more than 64 of them are in registers:
        // a thread of this 10-warp CTA has 168.  A masked tile's first pass
        // writes the masked scores back, so the second needs no mask.
        auto load_half = [&](int h, float (&sv)[64]) {
          uint32_t sr[64];
          tmem_ld_32(tmem + lane_base + col_s + 64 * h, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
          tmem_ld_32(tmem + lane_base + col_s + 64 * h + 32,
                     *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
          tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 64; ++c) sv[c] = __uint_as_float(sr[c]);
        };
        // row maximum of the raw scores (scale > 0 commutes with max): eight
        // running three-input maxima
        float m8[8];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          float sv[64];
          load_half(h, sv);
          if (masked) {
            uint64_t v = vm[h];
            uint32_t sm[64];
#pragma unroll
            for (int c = 0; c < 64; ++c) {
              if (!(v & 1ull)) sv[c] = -INFINITY;
              v >>= 1;
              sm[c] = __float_as_uint(sv[c]);
            }
            tmem_st_32(tmem + lane_base + col_s + 64 * h, *reinterpret_cast<uint32_t(*)[32]>(&sm[0]));
            tmem_st_32(tmem + lane_base + col_s + 64 * h + 32,
                       *reinterpret_cast<uint32_t(*)[32]>(&sm[32]));
            tmem_st_wait();
          }
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            float m = h ? fmax3(m8[k], sv[k], sv[8 + k]) : fmaxf(sv[k], sv[8 + k]);
#pragma unroll
            for (int j = 2; j < 8; j += 2) m = fmax3(m, sv[8 * j + k], sv[8 * j + 8 + k]);
            m8[k] = m;
          }
        }
        const float mx =
            fmax3(fmax3(m8[0], m8[1], m8[2]), fmax3(m8[3], m8[4], m8[5]), fmaxf(m8[6], m8[7])) *
            a.scale_log2;
        const float m_new = fmaxf(m_ref, mx);
        const bool resc = m_ref != -INFINITY && m_new > m_ref + kBRescaleLog2;
        if (m_ref == -INFINITY) m_ref = m_new;
        const bool any_resc = __any_sync(0xffffffffu, resc);
        float alpha = 1.f;
        if (resc) {
          alpha = ex2_approx(m_ref - m_new);
          l *= alpha;
          m_ref = m_new;
        }
        // p = 2^(s * scale_log2 - m): one paired FMA per two scores, one MUFU
        // per score; the row sum in four paired accumulators.  P_X goes over
        // the S_X columns this thread has read: half h into columns
        // 32 h .. 32 h + 31, once that half's scores are in registers.
        const float neg_mu = m_ref == -INFINITY ? 0.f : -m_ref;
        const unsigned long long sc2 = f32x2_pack(a.scale_log2, a.scale_log2);
        const unsigned long long mu2 = f32x2_pack(neg_mu, neg_mu);
        unsigned long long rs2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          float sv[64];
          load_half(h, sv);
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            float x0, x1;
            f32x2_unpack(ffma2(f32x2_pack(sv[2 * c], sv[2 * c + 1]), sc2, mu2), x0, x1);
            const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
            rs2[c & 3] = fadd2(rs2[c & 3], f32x2_pack(p0, p1));
            pk[c] = pack_bf16(p0, p1);
          }
          tmem_st_32(tmem + lane_base + col_s + 32 * h, pk);
        }
        float r0, r1;
        f32x2_unpack(fadd2(fadd2(rs2[0], rs2[1]), fadd2(rs2[2], rs2[3])), r0, r1);
        l += r0 + r1;
        tmem_st_wait();
        if (any_resc) {
          // O_X *= alpha before PV_X(i) adds this tile (after the scores and
          // P are out of registers).  O holds exactly the tiles before i:
          // PV_X(i-1) has completed (S_X(i) was issued after it); the wait
          // only confirms it.
          if (i >= 1) mbar_wait(smem_u32(&pv_done[x]), (i - 1) & 1, a.err);
          tc_fence_after();
#pragma unroll
          for (int c0 = 0; c0 < D; c0 += 32) {
            uint32_t ov[32];
            tmem_ld_32(tmem + lane_base + col_o + c0, ov);
            tmem_ld_wait();
#pragma unroll
            for (int c = 0; c < 32; ++c) ov[c] = __float_as_uint(__uint_as_float(ov[c]) * alpha);
            tmem_st_32(tmem + lane_base + col_o + c0, ov);
          }
          tmem_st_wait();
        }
        if (x == 0 && valid < kW) {
          // Cache rows past the prefix end may hold anything (even NaN bit
          // patterns): zero their V, once it has landed, so that masked
          // columns contribute exactly 0 to both blocks (PV_B follows PV_A).
          const int vu = 2 * i + 1;
          mbar_wait(smem_u32(&u_full[vu % kUnits]), (vu / kUnits) & 1, a.err);
          uint4* vt = reinterpret_cast<uint4*>(smem + (vu % kUnits) * S::kUnitBytes);
          const int per_half = (kW - valid) * 8;  // 16-byte chunks past the end
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
        mbar_arrive(smem_u32(&p_full[x]));
      }
      // O of this row is complete once the last PV has landed
      if (my_tiles > 0) mbar_wait(smem_u32(&pv_done[x]), (my_tiles - 1) & 1, a.err);
    }
  }
  __syncwarp();  // the producer and MMA lanes rejoin their warps before the barriers

  // ---- epilogue: each softmax thread reads its row of O / l from TMEM
  const bool has_row = warp >= 2;
  const int x = has_row ? (warp - 2) >> 2 : 0;
  const int rl = (warp & 3) * 32 + lane;
  const int rows_x = x ? rows_b : rows_a;
  const int r = x * nbh * a.G + rl;  // CTA row
  const uint32_t o_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16) + x * kBlockCols + 128;
  const float inv_l = (my_tiles > 0 && l > 0.f) ? 1.f / l : 0.f;

  if (nparts == 1) {
    if (has_row) {
      // O in two 64-column halves (a whole row beside the rest would spill)
      const int node = node0 + nfirst + min(r, rows - 1) / a.G;
      const int h = g * a.G + r % a.G;
      __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(a.out) + ((size_t)node * a.Hq + h) * D;
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 64) {
        uint32_t ov[64];
        tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[0]));
        tmem_ld_32(o_addr + c0 + 32, *reinterpret_cast<uint32_t(*)[32]>(&ov[32]));
        tmem_ld_wait();
        if (rl < rows_x) {
#pragma unroll
          for (int c = 0; c < 64; c += 8) {
            uint4 pk;
            pk.x = pack_bf16(__uint_as_float(ov[c]) * inv_l, __uint_as_float(ov[c + 1]) * inv_l);
            pk.y = pack_bf16(__uint_as_float(ov[c + 2]) * inv_l, __uint_as_float(ov[c + 3]) * inv_l);
            pk.z = pack_bf16(__uint_as_float(ov[c + 4]) * inv_l, __uint_as_float(ov[c + 5]) * inv_l);
            pk.w = pack_bf16(__uint_as_float(ov[c + 6]) * inv_l, __uint_as_float(ov[c + 7]) * inv_l);
            *reinterpret_cast<uint4*>(dst + c0 + c) = pk;
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tmem, kBTmemCols);
    }
    leave();
    return;
  }
  // ---- split-KV merge: each row's normalised partial and its
  // log2-sum-exp are staged in the idle ring, one bulk copy per peer moves
  // the rows it merges into its inbox (behind the staged rows), and every
  // CTA merges its own rows from its inbox.  A CTA's partials of the rows it
  // merges itself are staged straight into its own inbox slots.
  // (the group's pieces: CTAs base .. base + nparts - 1 of the cluster)
  const int per = (rows + nparts - 1) / nparts;
  const int cnt_mine = max(0, min(per, rows - part * per));
  __half* stage_rows = reinterpret_cast<__half*>(smem);
  // every PV of this CTA has completed (the softmax threads waited for the
  // last one): the ring is idle, so peers may now fill the inbox it holds
  __syncthreads();
  cluster_arrive_release();
  if (tid == 0)
    mbar_arrive_expect_tx(smem_u32(inbox_full),
                          (uint32_t)((nparts - 1) * cnt_mine * S::kRowBytes));
  if (has_row) {
    // O in two 64-column halves (a whole row beside the rest would spill)
    // (own rows: inbox slot part * per + i is CTA row r itself)
    const bool own = r >= part * per && r < part * per + cnt_mine;
    __half* dst = (own ? sInbox : stage_rows) + min(r, 255) * S::kPitch;
    // no column reached this row in this split (a split without tiles never
    // writes O): its partial is 0 with lse = -inf, whatever the unwritten
    // accumulator holds (0 * NaN would poison the merge)
    const bool empty = !(inv_l > 0.f);
#pragma unroll
    for (int c0 = 0; c0 < D; c0 += 64) {
      uint32_t ov[64];
      tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[0]));
      tmem_ld_32(o_addr + c0 + 32, *reinterpret_cast<uint32_t(*)[32]>(&ov[32]));
      tmem_ld_wait();
      if (rl < rows_x) {
#pragma unroll
        for (int c = 0; c < 64; c += 8) {
          uint4 pk;
          pk.x = pack_half(__uint_as_float(ov[c]) * inv_l, __uint_as_float(ov[c + 1]) * inv_l);
          pk.y = pack_half(__uint_as_float(ov[c + 2]) * inv_l, __uint_as_float(ov[c + 3]) * inv_l);
          pk.z = pack_half(__uint_as_float(ov[c + 4]) * inv_l, __uint_as_float(ov[c + 5]) * inv_l);
          pk.w = pack_half(__uint_as_float(ov[c + 6]) * inv_l, __uint_as_float(ov[c + 7]) * inv_l);
          if (empty) pk = make_uint4(0, 0, 0, 0);
          *reinterpret_cast<uint4*>(dst + c0 + c) = pk;
        }
      }
    }
    if (rl < rows_x)
      *reinterpret_cast<float*>(dst + D) = empty ? -INFINITY : m_ref + __log2f(l);
  }
  fence_proxy_async_smem();  // staged rows are read by the bulk-copy engine
  tc_fence_before();
  __syncthreads();
  cluster_wait_acquire();    // every peer's inbox is ready to be filled
  if (tid < nparts) {
    const int q = tid;
    const int cnt = min(per, rows - q * per);
    if (cnt > 0 && q != part) {
      const uint32_t src = smem_u32(stage_rows + q * per * S::kPitch);
      const uint32_t dst = mapa_cluster(smem_u32(sInbox + part * per * S::kPitch), base + q);
      bulk_copy_s2cluster(dst, src, (uint32_t)(cnt * S::kRowBytes),
                          mapa_cluster(smem_u32(inbox_full), base + q));
      bulk_commit_group();
    }
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kBTmemCols);
  }
  if (cnt_mine > 0) mbar_wait(smem_u32(inbox_full), 0, a.err);
  inbox_merge<D, kBThreads, S::kPitch>(a, sInbox, rows, part, per, nparts, node0 + nfirst, g,
                                       tid);
  // this CTA's staged rows must stay readable until its copies have left
  if (tid < nparts) bulk_wait_read_all();
}

}  // namespace

static int blk2_smem_bytes() { return BSmem::kTotal + 1024; }

int attention_2blk_max_active_clusters(int cluster) {
  const int smem = blk2_smem_bytes();
  static DeviceMemo limit;
  if (ensure_smem_limit((const void*)attn_2blk_kernel, smem, limit) != cudaSuccess) return 0;
  if (cluster > 8 && cudaFuncSetAttribute(attn_2blk_kernel,
                                          cudaFuncAttributeNonPortableClusterSizeAllowed,
                                          1) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cluster);
  cfg.blockDim = dim3(kBThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = cluster;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_2blk_kernel, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_attention_2blk(const AttnArgs& a, const AttnMaps& m, const TeamPlan& tp,
                                  cudaStream_t s, bool pdl) {
  const int smem = blk2_smem_bytes();
  static DeviceMemo limit;
  static DeviceMemo nonportable;
  cudaError_t e = ensure_smem_limit((const void*)attn_2blk_kernel, smem, limit);
  if (e != cudaSuccess) return e;
  if (a.splits > 8) {
    e = ensure_nonportable_cluster((const void*)attn_2blk_kernel, nonportable);
    if (e != cudaSuccess) return e;
  }
  // one-group clusters, or (team plan) a.team_ctas CTAs in clusters of a.splits
  const dim3 grid(a.team ? a.team_ctas : a.B * a.Hkv * a.rb_count * a.splits);
  return launch_ex(attn_2blk_kernel, grid, dim3(kBThreads), smem, s, a.splits, pdl, m.q, m.tk,
                   m.tv, m.ck, m.cv, m.cv_page, a, tp);
}

}  // namespace pf
