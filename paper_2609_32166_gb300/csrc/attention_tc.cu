// Tree-masked GQA attention on the 5th-generation tensor cores (tcgen05).
// Same contract and work split as the mma.sync kernel in attention.cu (one
// CTA = a block of query rows of one KV head x a slice of the 64-token KV
// tiles, clusters merge the slices); the arithmetic moves to UMMA with TMEM
// accumulators:
//
//   warp 0     TMA producer: Q once, then K/V tiles into a 3-stage ring
//   warp 1     TMEM owner and MMA issuer (one thread), per row block w:
//                S_w,i = Q_w K_i^T    M=128, N=64, K=D   -> TMEM S_w[i % 2]
//                O_w  += P_w,i V_i    M=128, N=D,  K=64  -> TMEM O_w
//              issued as their inputs become ready, so the tensor core
//              computes S_{i+1} while the softmax warps work on S_i
//   softmax    one warpgroup per 128-row block, one query row per thread
//              (its TMEM lane): read S, mask (prefix length / ancestor
//              bits), online softmax in the exp2 domain, write P as bf16
//              into shared memory (K-major, 128-byte swizzle); the running
//              maximum is only moved (and O rescaled in TMEM) when it grows
//              by more than 2^8, so the common case never touches O; at the
//              end they read O back and publish (m, l, O) for the merge.
//
// kWG = 1 (128 rows, 192 threads) serves problems of at most 128 rows per
// KV head; kWG = 2 (256 rows, 320 threads: two softmax warpgroups, 512
// TMEM columns) larger ones: each K/V tile then serves twice the rows and
// two warps share every scheduler during the softmax.
//
// V is the B operand of PV in its natural token-major layout (an MN-major
// UMMA operand), so no transpose is needed anywhere.
#include <cuda_fp16.h>

#include "attn_common.cuh"

namespace cg = cooperative_groups;

namespace pf {

namespace {

constexpr int kTcStages = 3;
constexpr float kRescaleLog2 = 8.f;   // move the reference max when it grows by > 2^8

template <int WG>
struct TcShape {
  static constexpr int kThreads = 64 + 128 * WG;      // producer, MMA, softmax warpgroups
  static constexpr uint32_t kTmemCols = 256 * WG;     // per block: S[0] 0..63, S[1] 64..127, O
};

template <int D, int WG>
struct TcSmem {
  static constexpr int kHalves = D / 64;
  static constexpr int kRows = 128 * WG;
  static constexpr int kTileBytes = kBN * D * 2;         // one K or V tile
  static constexpr int kStageBytes = 2 * kTileBytes;     // K + V
  static constexpr int kQBytes = kRows * D * 2;
  static constexpr int kPBytes = 128 * kBN * 2;          // one P tile (bf16) of one block
  static constexpr int kQOff = kTcStages * kStageBytes;
  static constexpr int kPOff = kQOff + kQBytes;
  static constexpr int kPEnd = kPOff + 2 * WG * kPBytes;
  // Merge inbox: one slot per (split, row) a CTA may receive, at most
  // splits * ceil(rows / splits) <= rows + 15 slots.  A slot holds the
  // normalised partial O / l in fp16 (D halves) followed by its log2-sum-exp
  // (one float) in the 16-byte pad; the same format is staged locally.
  // kWG = 1: the inbox has its own space (peers may send while this CTA is
  // still working) and rows are staged in the idle K/V ring.  kWG = 2: no
  // room; the inbox takes the K/V ring and rows are staged over Q and P,
  // and peers send only after every CTA of the cluster has left its loop.
  static constexpr int kInboxSlots = kRows + 16;
  static constexpr int kInboxPitch = D + 8;              // halves
  static constexpr int kRowBytes = kInboxPitch * 2;
  static constexpr int kStageOff = WG == 1 ? 0 : kQOff;
  static constexpr int kInboxOff = WG == 1 ? kPEnd : 0;
  static constexpr int kBarOff = WG == 1 ? kInboxOff + kInboxSlots * kRowBytes : kPEnd;
  static_assert(kRows * kRowBytes <= (WG == 1 ? kQOff : kPEnd - kQOff), "staged rows fit");
  static_assert(WG == 1 || kInboxSlots * kRowBytes <= kQOff, "inbox fits in the ring");
  // kv_full[3] kv_empty[3] q_full, per block s_full[2] s_empty[2] p_full[2] pv_done[2], inbox
  static constexpr int kNumBars = 2 * kTcStages + 1 + 8 * WG + 1;
  // then the TMEM address (4 bytes, padded to 16) and the balanced batch
  // mode's plan entry (16 bytes)
  static constexpr int kTotal = kBarOff + kNumBars * 8 + 32;
  static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// BAL: the balanced batch mode's instance (plan, partials to the workspace);
// the cluster instance carries none of that code.
template <int D, int WG, bool BAL>
__global__ void __launch_bounds__(TcShape<WG>::kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q,
                   const __grid_constant__ CUtensorMap tm_tk,
                   const __grid_constant__ CUtensorMap tm_tv,
                   const __grid_constant__ CUtensorMap tm_ck,
                   const __grid_constant__ CUtensorMap tm_cv, const AttnArgs a) {
  using S = TcSmem<D, WG>;
  constexpr int kThreads = TcShape<WG>::kThreads;
  constexpr uint32_t kTmemCols = TcShape<WG>::kTmemCols;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sKV = smem;
  uint8_t* sQ = smem + S::kQOff;
  uint8_t* sP = smem + S::kPOff;
  __half* sInbox = reinterpret_cast<__half*>(smem + S::kInboxOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* kv_full = bars;
  uint64_t* kv_empty = bars + kTcStages;
  uint64_t* q_full = bars + 2 * kTcStages;
  // per row block w: s_full[2] s_empty[2] p_full[2] pv_done[2] at blk + 8 w
  uint64_t* blk = q_full + 1;
  uint64_t* inbox_full = blk + 8 * WG;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + S::kNumBars);

  cg::cluster_group cluster = cg::this_cluster();
  const int nsplit = a.splits;
  const int split = (int)cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // With PF_ATTN_EARLY_PREFETCH the tree structure, prefix lengths and the
  // prefix cache were complete before the preceding kernel started: read
  // them and request cache tiles before waiting for it (programmatic
  // dependent launch); q and the proposal K/V only after.
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

  // This CTA's group (sequence, KV head, row block) and its part of the
  // group's tiles: split `split` of the cluster, or (balanced batch mode,
  // one CTA per cluster) the item the plan gives it.
  int group = blockIdx.x / nsplit, part = split, nparts = nsplit;
  if constexpr (BAL) {
    // warp 0 derives the plan; the first n_groups CTAs also record group
    // blockIdx.x's (first item, items) for the combine kernel
    int4* plan_slot = reinterpret_cast<int4*>(smem + S::kBarOff + S::kNumBars * 8 + 16);
    if (warp == 0) {
      const int n_groups = a.B * a.Hkv * a.rb_count;
      const int gq = (int)blockIdx.x < n_groups ? (int)blockIdx.x : -1;
      PlanItem ge;
      const PlanItem it = balanced_plan(a, (int)blockIdx.x, gq, &ge);
      if (lane == 0) {
        *plan_slot = make_int4(it.group, it.j, it.k, 0);
        if (gq >= 0) {
          // the group's first node and rows, for the combine kernel
          const int bq = gq / (a.rb_count * a.Hkv), nfq = (gq % a.rb_count) * a.nb;
          const int n0 = a.cu_nodes[bq], nnq = a.cu_nodes[bq + 1] - n0;
          plan_table(a)[gq] = make_int4(ge.first, ge.k, n0 + nfq, max(0, min(a.nb, nnq - nfq)) * a.G);
        }
      }
    }
    __syncthreads();
    const int4 pi = *plan_slot;
    if (pi.x < 0) return;  // uniform over the CTA: no work for this item
    group = pi.x;
    part = pi.y;
    nparts = pi.z;
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
  const int nblk = WG == 1 ? 1 : (rows > 128 ? 2 : 1);  // row blocks with work
  const int n_ptiles = (P + kBN - 1) / kBN;
  const int n_qtiles = (nn + kBN - 1) / kBN;
  const int ntiles = n_ptiles + n_qtiles;
  // Split s takes tiles [t_begin, t_end) of the order (proposal tiles,
  // prefix tiles): the proposal's K/V can only be loaded once the preceding
  // kernel has finished, so those tiles go to the first split, which holds
  // the fewest tiles (ntiles * s / nsplit rounds down).  Within a split the
  // prefix tiles come first (their loads start before that wait).
  const int t_begin = (int)((long long)ntiles * part / nparts);
  const int t_end = (int)((long long)ntiles * (part + 1) / nparts);
  const int my_tiles = t_end - t_begin;
  const int pre_lo = max(t_begin, n_qtiles);        // first prefix tile of the split
  const int my_ptiles = max(0, t_end - pre_lo);
  // cache tile index (prefix tiles 0..n_ptiles-1, then proposal tiles) of
  // the split's i-th tile
  auto tile_at = [&](int i) {
    return i < my_ptiles ? pre_lo - n_qtiles + i : n_ptiles + t_begin + (i - my_ptiles);
  };
  const int first = min(kTcStages, my_tiles);

  if (tid == 0) {
    for (int i = 0; i < kTcStages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), 1);
      mbar_init(smem_u32(&kv_empty[i]), (uint32_t)nblk);  // one PV per active block
    }
    mbar_init(smem_u32(q_full), 1);
    for (int w = 0; w < WG; ++w)
      for (int i = 0; i < 2; ++i) {
        mbar_init(smem_u32(&blk[8 * w + i]), 1);          // s_full
        mbar_init(smem_u32(&blk[8 * w + 2 + i]), 128);    // s_empty
        mbar_init(smem_u32(&blk[8 * w + 4 + i]), 128);    // p_full
        mbar_init(smem_u32(&blk[8 * w + 6 + i]), 1);      // pv_done
      }
    mbar_init(smem_u32(inbox_full), 1);
    fence_mbar_init();
    int4 pg[kTcStages];  // every first tile's page entries in one round trip
#pragma unroll
    for (int i = 0; i < kTcStages; ++i)
      pg[i] = i < first ? kv_tile_pages(a, tile_at(i), n_ptiles, b, P) : make_int4(-1, -1, -1, -1);
#pragma unroll
    for (int i = 0; i < kTcStages; ++i)
      if (i < first && i < my_ptiles)
        issue_kv_tile<D>(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                         smem_u32(&kv_full[i]), tile_at(i), n_ptiles, b, g, node0, P, pg[i]);
  }
  if (early) pdl_wait();
  if (tid == 0) {
    mbar_arrive_expect_tx(smem_u32(q_full), S::kHalves * a.G * a.nb * 128);
#pragma unroll
    for (int h = 0; h < S::kHalves; ++h)
      tma_load_3d(smem_u32(sQ + h * S::kRows * 128), &tm_q, h * 64, g * a.G, node0 + nfirst,
                  smem_u32(q_full));
    for (int i = 0; i < first; ++i)
      if (i >= my_ptiles)  // proposal tiles: no page entries
        issue_kv_tile<D>(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                         smem_u32(&kv_full[i]), tile_at(i), n_ptiles, b, g, node0, P,
                         make_int4(-1, -1, -1, -1));
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // kWG = 1: peers may signal this CTA's inbox barrier once it is
  // initialised: arrive now, wait just before sending partials.  (A single
  // split is launched without a cluster and uses no cluster feature.)
  if (WG == 1 && nsplit > 1) cluster_arrive_release();
  pdl_launch_dependents();

  float m_ref = -INFINITY, l = 0.f;   // softmax threads: running max (log2) and sum of their row
  const int wg = warp >= 2 ? (warp - 2) >> 2 : 0;   // softmax: this thread's row block
  if (warp == 0) {
    // ---------------- producer: refill the ring as the PVs release stages
    if (lane == 0) {
      for (int i = kTcStages; i < my_tiles; ++i) {
        const int st = i % kTcStages;
        const int t = tile_at(i);
        const int4 pg = kv_tile_pages(a, t, n_ptiles, b, P);  // in flight during the wait
        if (!mbar_wait(smem_u32(&kv_empty[st]), ((i / kTcStages) & 1) ^ 1, a.err)) break;
        issue_kv_tile<D>(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + st * S::kStageBytes,
                         smem_u32(&kv_full[st]), t, n_ptiles, b, g, node0, P, pg);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = umma_idesc_bf16(128, kBN);
      const uint32_t id_o = umma_idesc_bf16_bmn(128, D);
      bool ok = mbar_wait(smem_u32(q_full), 0, a.err);
      const uint32_t q0 = smem_u32(sQ);
      // Event-driven issue, per row block w: S_n as soon as its K/V tile
      // has landed and the softmax has read S_{n-2} out of the same TMEM
      // buffer; PV_j as soon as P_j is in shared memory.  S_{n+1} thus
      // never waits behind P_{n-1}.
      int ns[WG], np[WG];
#pragma unroll
      for (int w = 0; w < WG; ++w) ns[w] = np[w] = 0;
      unsigned idle = 0;
      unsigned long long t0 = 0;
      while (ok) {
        bool progressed = false, done = true;
#pragma unroll
        for (int w = 0; w < WG; ++w) {
          if (w >= nblk) continue;
          uint64_t* bw = blk + 8 * w;
          const uint32_t tw = tmem + (uint32_t)(w * 256);
          if (ns[w] < my_tiles) {
            const int n = ns[w], st = n % kTcStages, sb = n & 1;
            if (mbar_test_wait(smem_u32(&kv_full[st]), (n / kTcStages) & 1) &&
                mbar_test_wait(smem_u32(&bw[2 + sb]), ((n >> 1) & 1) ^ 1)) {
              tc_fence_after();
              const uint32_t k0 = smem_u32(sKV + st * S::kStageBytes);
#pragma unroll
              for (int kk = 0; kk < D / 16; ++kk) {
                const uint32_t qa =
                    q0 + (kk >> 2) * (S::kRows * 128) + w * (128 * 128) + (kk & 3) * 32;
                const uint32_t kb = k0 + (kk >> 2) * (kBN * 128) + (kk & 3) * 32;
                umma_bf16(tw + sb * kBN, umma_desc_sw128(qa), umma_desc_sw128(kb), id_s, kk > 0);
              }
              umma_commit(smem_u32(&bw[sb]));
              ++ns[w];
              progressed = true;
            }
          }
          if (np[w] < ns[w]) {
            const int j = np[w], pb = j & 1, stj = j % kTcStages;
            if (mbar_test_wait(smem_u32(&bw[4 + pb]), (j >> 1) & 1)) {
              tc_fence_after();
              const uint32_t p0 = smem_u32(sP + (2 * w + pb) * S::kPBytes);
              const uint32_t v0 = smem_u32(sKV + stj * S::kStageBytes + S::kTileBytes);
#pragma unroll
              for (int kt = 0; kt < kBN / 16; ++kt)
                umma_bf16(tw + 2 * kBN, umma_desc_sw128(p0 + kt * 32),
                          umma_desc_sw128_lbo(v0 + kt * 16 * 128, kBN * 128, 1024), id_o,
                          (j > 0 || kt > 0) ? 1u : 0u);
              umma_commit(smem_u32(&bw[6 + pb]));
              umma_commit(smem_u32(&kv_empty[stj]));
              ++np[w];
              progressed = true;
            }
          }
          if (np[w] < my_tiles) done = false;
        }
        if (done) break;
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
  } else if (wg < nblk) {
    // ---------------- softmax / correction: one row per thread
    uint64_t* bw = blk + 8 * wg;
    const uint32_t tw = tmem + (uint32_t)(wg * 256);
    const int quad = warp & 3;
    const int rl = quad * 32 + lane;       // row within the block (its TMEM lane)
    const int r = wg * 128 + rl;           // row within the CTA
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    uint64_t mk0 = 0, mk1 = 0;
    if (r < rows) {
      const int node = node0 + nfirst + r / a.G;
      mk0 = a.mask[2 * node];
      mk1 = a.mask[2 * node + 1];
    }
    bool ok = true;
    for (int i = 0; i < my_tiles && ok; ++i) {
      const int sb = i & 1;
      const int st = i % kTcStages;
      ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bw[sb]), (i >> 1) & 1, a.err));
      if (!ok) break;  // warp-uniform
      tc_fence_after();
      uint32_t lo[32], hi[32];
      tmem_ld_32(tw + lane_base + sb * kBN, lo);
      tmem_ld_32(tw + lane_base + sb * kBN + 32, hi);
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(smem_u32(&bw[2 + sb]));

      const int t = tile_at(i);
      const bool is_prefix = t < n_ptiles;
      const int valid = is_prefix ? min(kBN, P - t * kBN) : kBN;
      float sv[64];
#pragma unroll
      for (int c = 0; c < 64; ++c) sv[c] = __uint_as_float(c < 32 ? lo[c] : hi[c - 32]);
      if (!is_prefix || valid < kBN) {
        // masked tile: prefix columns past the end, or proposal columns
        // that are not ancestors of this row's node
        const uint64_t vis = is_prefix ? (valid >= 64 ? ~0ull : ((1ull << valid) - 1ull))
                                       : ((t - n_ptiles) ? mk1 : mk0);
#pragma unroll
        for (int c = 0; c < 64; ++c)
          if (!((vis >> c) & 1ull)) sv[c] = -INFINITY;
      }
      // row maximum of the raw scores (scale > 0 commutes with max): a tree
      // of three-input maxima, 64 -> 22 -> 8 -> 3 -> 1 (32 instructions)
      float m22[22];
#pragma unroll
      for (int k = 0; k < 21; ++k) m22[k] = fmax3(sv[3 * k], sv[3 * k + 1], sv[3 * k + 2]);
      m22[21] = sv[63];
      float m8[8];
#pragma unroll
      for (int k = 0; k < 7; ++k) m8[k] = fmax3(m22[3 * k], m22[3 * k + 1], m22[3 * k + 2]);
      m8[7] = m22[21];
      const float mx = fmax3(fmax3(m8[0], m8[1], m8[2]), fmax3(m8[3], m8[4], m8[5]),
                             fmaxf(m8[6], m8[7])) *
                       a.scale_log2;
      const float m_new = fmaxf(m_ref, mx);
      const bool resc = m_ref != -INFINITY && m_new > m_ref + kRescaleLog2;
      if (m_ref == -INFINITY) m_ref = m_new;
      if (__any_sync(0xffffffffu, resc)) {
        // O must hold exactly the tiles before i: wait for PV_{i-1}.
        if (i >= 1) mbar_wait(smem_u32(&bw[6 + ((i - 1) & 1)]), ((i - 1) >> 1) & 1, a.err);
        tc_fence_after();
        const float alpha = resc ? ex2_approx(m_ref - m_new) : 1.f;
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t ov[32];
          tmem_ld_32(tw + lane_base + 2 * kBN + c0, ov);
          tmem_ld_wait();
#pragma unroll
          for (int c = 0; c < 32; ++c) ov[c] = __float_as_uint(__uint_as_float(ov[c]) * alpha);
          tmem_st_32(tw + lane_base + 2 * kBN + c0, ov);
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
      uint32_t pk[32];
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        float x0, x1;
        f32x2_unpack(ffma2(f32x2_pack(sv[2 * c], sv[2 * c + 1]), sc2, mu2), x0, x1);
        const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
        const unsigned long long p2 = f32x2_pack(p0, p1);
        rs2[c & 3] = fadd2(rs2[c & 3], p2);
        pk[c] = pack_bf16(p0, p1);
      }
      float r0, r1;
      f32x2_unpack(fadd2(fadd2(rs2[0], rs2[1]), fadd2(rs2[2], rs2[3])), r0, r1);
      l += r0 + r1;
      // P buffer sb was last read by PV_{i-2}.
      if (i >= 2) mbar_wait(smem_u32(&bw[6 + sb]), ((i - 2) >> 1) & 1, a.err);
      uint8_t* prow = sP + (2 * wg + sb) * S::kPBytes + rl * 128;
#pragma unroll
      for (int c = 0; c < 8; ++c)
        *reinterpret_cast<uint4*>(prow + ((c ^ (rl & 7)) << 4)) =
            make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
      if (valid < kBN) {
        // Cache rows past the prefix end may hold anything (even NaN bit
        // patterns): zero their V so masked columns contribute exactly 0.
        // (With two blocks both write the same zeros before their PV.)
        // Each 64-column half of the V tile holds its rows at 128-byte
        // pitch, so the rows from `valid` on are one contiguous run per half.
        uint4* sv = reinterpret_cast<uint4*>(sKV + st * S::kStageBytes + S::kTileBytes);
        const int per_half = (kBN - valid) * 8;   // 16-byte chunks past the end
#pragma unroll
        for (int h = 0; h < S::kHalves; ++h)
          for (int c = rl; c < per_half; c += 128)
            sv[h * kBN * 8 + valid * 8 + c] = make_uint4(0, 0, 0, 0);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(smem_u32(&bw[4 + sb]));
    }
    // O of this row is complete once the block's last PV has landed
    if (my_tiles > 0)
      mbar_wait(smem_u32(&bw[6 + ((my_tiles - 1) & 1)]), ((my_tiles - 1) >> 1) & 1, a.err);
  }
  __syncwarp();  // the producer and MMA lanes rejoin their warps before the barriers

  // ---- epilogue: each softmax thread reads its row of O / l from TMEM
  const bool has_row = warp >= 2 && wg < nblk;
  const int quad = warp & 3;
  const int r = wg * 128 + quad * 32 + lane;
  const uint32_t o_addr = tmem + (uint32_t)(wg * 256) + ((uint32_t)(quad * 32) << 16) + 2 * kBN;
  const float inv_l = (my_tiles > 0 && l > 0.f) ? 1.f / l : 0.f;

  // ---- split-KV merge.  Each row's partial result, normalised (O / l,
  // fp16) with its log2-sum-exp lse = m + log2(l) in the row's pad, is
  // staged in this CTA's shared memory, row r at slot r, so the rows each
  // peer merges are contiguous.  One bulk copy per peer moves them into the
  // peer's inbox and completes on the peer's inbox barrier, which expects
  // one block from every CTA of the cluster; the peer then merges from its
  // own shared memory:
  //   out = sum_s 2^(lse_s - M) (O/l)_s / sum_s 2^(lse_s - M),  M = max_s lse_s
  if (nsplit == 1) {
    // ---- single split: O / l is the output -- or, for a group that the
    // balanced batch mode spread over several CTAs, this item's partial
    // (same format as a staged row) for the combine kernel
    if (has_row) {
      uint32_t ov[D];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32)
        tmem_ld_32(o_addr + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
      tmem_ld_wait();
      if (BAL && r < rows && nparts > 1) {
        __half* dst = reinterpret_cast<__half*>(a.ws) + ((size_t)blockIdx.x * a.bm + r) * S::kInboxPitch;
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
      tmem_dealloc(tmem, kTmemCols);
    }
    return;
  }
  const int per = (rows + nsplit - 1) / nsplit;
  const int cnt_mine = max(0, min(per, rows - split * per));
  __half* stage_rows = reinterpret_cast<__half*>(smem + S::kStageOff);
  if (WG == 2) {
    // The rows are staged over Q and P: every block's last PV must have
    // completed (each softmax warpgroup waited for its own) -- and the ring
    // is idle, so peers may now fill the inbox it holds.
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
      __half* dst = stage_rows + r * S::kInboxPitch;
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
      const uint32_t src = smem_u32(stage_rows + q * per * S::kInboxPitch);
      const uint32_t dst = mapa_cluster(smem_u32(sInbox + split * per * S::kInboxPitch), q);
      bulk_copy_s2cluster(dst, src, (uint32_t)(cnt * S::kRowBytes),
                          mapa_cluster(smem_u32(inbox_full), q));
      bulk_commit_group();
    }
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (cnt_mine > 0) mbar_wait(smem_u32(inbox_full), 0, a.err);
  inbox_merge<D, kThreads, S::kInboxPitch>(a, sInbox, rows, split, per, nsplit, node0 + nfirst,
                                           g, tid);
  // this CTA's staged rows must stay readable until its copies have left
  if (tid < nsplit) bulk_wait_read_all();
}

// Balanced batch mode, second kernel: for every group that the plan spread
// over k > 1 CTAs, merge the k partials of each row (same rule as the
// cluster merge: out = sum_j 2^(lse_j - M) (O/l)_j / sum_j 2^(lse_j - M)).
// One CTA per (group, 16 rows), one thread per (row, 8 columns).  Every CTA
// waits for the attention kernel before it exits, so kernels that follow in
// the stream see the attention outputs complete.
constexpr int kCombineRows = 16;

__global__ void __launch_bounds__(256) attn_combine_kernel(const AttnArgs a) {
  constexpr int D = 128, C8 = D / 8, kPitch = D + 8, kBatch = 8;
  const int chunks = (a.bm + kCombineRows - 1) / kCombineRows;
  const int group = blockIdx.x / chunks, chunk = blockIdx.x % chunks;
  pdl_wait();
  pdl_launch_dependents();
  const int4 e = plan_table(a)[group];  // from the attention kernel
  const int first = e.x, k = e.y, node_base = e.z, rows = e.w;
  const int r = chunk * kCombineRows + (int)threadIdx.x / C8;
  const int c8 = (int)threadIdx.x % C8;
  if (k <= 1 || r >= rows) return;
  const __half* base = reinterpret_cast<const __half*>(a.ws) + (size_t)r * kPitch;
  const size_t slot_stride = (size_t)a.bm * kPitch;
  // partial slot of piece j (see plan_table)
  auto slot_of = [&](int j) {
    return a.slots == 2 && j > 0 ? 2 * ((first >> 1) + j) : first + j;
  };
  // partials in batches of 8 (all loads of a batch in flight together),
  // folded into a running maximum M, weight sum W and weighted sum acc
  float M = -INFINITY, W = 0.f;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int j0 = 0; j0 < k; j0 += kBatch) {
    float ls[kBatch];
    uint4 v[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      ls[u] = -INFINITY;
      if (j0 + u < k) {
        const __half* row = base + (size_t)slot_of(j0 + u) * slot_stride;
        ls[u] = *reinterpret_cast<const float*>(row + D);
        v[u] = *reinterpret_cast<const uint4*>(row + c8 * 8);
      }
    }
    float Mb = M;
#pragma unroll
    for (int u = 0; u < kBatch; ++u) Mb = fmaxf(Mb, ls[u]);
    if (Mb == -INFINITY) continue;  // nothing but empty partials so far
    const float sc = ex2_approx(M - Mb);  // M = -inf -> 0
    W *= sc;
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[c] *= sc;
    M = Mb;
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      if (ls[u] == -INFINITY) continue;  // absent or empty partial
      const float w = ex2_approx(ls[u] - M);
      W += w;
      const __half2* h2 = reinterpret_cast<const __half2*>(&v[u]);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float2 f = __half22float2(h2[c]);
        acc[2 * c] = fmaf(w, f.x, acc[2 * c]);
        acc[2 * c + 1] = fmaf(w, f.y, acc[2 * c + 1]);
      }
    }
  }
  const float inv = W > 0.f ? __fdividef(1.f, W) : 0.f;
  const int g = (group / a.rb_count) % a.Hkv;
  const int node = node_base + r / a.G;
  const int h = g * a.G + r % a.G;
  uint4 pk;
  pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
  pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
  pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
  pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
  *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(a.out) +
                            ((size_t)node * a.Hq + h) * D + c8 * 8) = pk;
}

}  // namespace

size_t attention_balanced_ws_bytes(int items, int bm, int D, int slots) {
  return (size_t)items * slots * bm * (D + 8) * 2 + kPlanMaxGroups * sizeof(int4) +
         kPlanMaxGroups * sizeof(unsigned long long);
}

cudaError_t launch_attention_combine(const AttnArgs& a, cudaStream_t s, bool pdl) {
  const int chunks = (a.bm + kCombineRows - 1) / kCombineRows;
  const dim3 grid(a.B * a.Hkv * a.rb_count * chunks);
  return launch_ex(attn_combine_kernel, grid, dim3(256), 0, s, 1, pdl, a);
}

template <int WG>
static int tc_smem_bytes() {
  return TcSmem<128, WG>::kTotal + 1024;
}

int attention_tc_smem_bytes() { return tc_smem_bytes<1>(); }

template <int WG>
static int tc_max_active_clusters_impl(int cluster) {
  const int smem = tc_smem_bytes<WG>();
  static DeviceMemo limit;
  if (ensure_smem_limit((const void*)attn_tc_kernel<128, WG, false>, smem, limit) != cudaSuccess)
    return 0;
  if (cluster > 8 && cudaFuncSetAttribute(attn_tc_kernel<128, WG, false>,
                                          cudaFuncAttributeNonPortableClusterSizeAllowed,
                                          1) != cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cluster);
  cfg.blockDim = dim3(TcShape<WG>::kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = cluster;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_tc_kernel<128, WG, false>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

int attention_tc_max_active_clusters(int cluster, int rows_per_cta) {
  return rows_per_cta > 128 ? tc_max_active_clusters_impl<2>(cluster)
                            : tc_max_active_clusters_impl<1>(cluster);
}

template <int WG, bool BAL>
static cudaError_t launch_tc(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  const int smem = tc_smem_bytes<WG>();
  static DeviceMemo limit;
  static DeviceMemo nonportable;
  cudaError_t e = ensure_smem_limit((const void*)attn_tc_kernel<128, WG, BAL>, smem, limit);
  if (e != cudaSuccess) return e;
  if (a.splits > 8) {
    e = ensure_nonportable_cluster((const void*)attn_tc_kernel<128, WG, BAL>, nonportable);
    if (e != cudaSuccess) return e;
  }
  const dim3 grid(BAL ? a.items : a.B * a.Hkv * a.rb_count * a.splits);
  return launch_ex(attn_tc_kernel<128, WG, BAL>, grid, dim3(TcShape<WG>::kThreads), smem, s,
                   a.splits, pdl, m.q, m.tk, m.tv, m.ck, m.cv, a);
}

cudaError_t launch_attention_tc(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  if (a.items > 0) return a.bm > 128 ? launch_tc<2, true>(a, m, s, pdl) : launch_tc<1, true>(a, m, s, pdl);
  return a.bm > 128 ? launch_tc<2, false>(a, m, s, pdl) : launch_tc<1, false>(a, m, s, pdl);
}

}  // namespace pf
