// Tree-masked GQA attention on pairs of SMs (tcgen05 .cta_group::2): one
// 2-SM MMA of M = 256 query rows per 128-token K/V tile.  Each CTA of the
// pair holds 128 query rows (its proposal nodes' G heads) and HALF of every
// K/V tile -- K rows (tokens) c*64 .. c*64+63 and V columns c*64 .. c*64+63
// for CTA c -- and the pair's MMA reads the other half from the peer's
// shared memory, so every K/V byte that enters an SM serves 256 query rows.
//
// Work split (continuous): the (sequence, KV head, 256-row block) groups'
// 128-token tiles are laid end to end and cut into a.items equal ranges,
// one per SM pair, whatever the sequences' lengths.  A range covers pieces
// of one or more groups (parts); a part that is a whole group writes the
// output, any other part a normalised partial (O / l in fp16 and its
// log2-sum-exp) that attn_combine_kernel merges.  Only an item's first and
// last part can be pieces of a longer group, so each item has two partial
// slots.
//
//   warp 0     TMA producer of this CTA's halves: per part its Q rows (two
//              Q buffers, so the next part's Q loads while this one runs),
//              then K/V halves into a ring of kPStages stages, completing on
//              this CTA's own barriers
//   warp 1     TMEM (both CTAs, allocated as a pair); in the odd CTA one
//              thread forwards "Q / tile landed" to the leader's barriers;
//              in the leader one thread issues the pair's MMAs
//                S_i  = Q K_i^T   M=256, N=128, K=D   -> S[i % 2]
//                O   += P_i V_i   M=256, N=D,  K=128  (A = P in TMEM) -> O
//              and commits each to the barriers of both CTAs
//   softmax    one warpgroup per CTA, one query row per thread (its TMEM
//              lane), as in attn_tc2_kernel; per part it resets its row's
//              running maximum and sum, and after the part's last tile
//              reads O / l out of TMEM, reports "O read" to the leader (the
//              next part's first PV overwrites O) and writes the row
//
// Barrier phases run on across parts: tile i of the item (counting all its
// parts) uses ring stage i % kPStages and S / P buffer i % 2.
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
constexpr int kMaxParts = kPlanMaxGroups;
// Exponentials per 8 column pairs computed by polynomial (exp2_poly_x2)
// instead of on the special-function unit.  Measured on the 32K tree: the
// pair's 2-SM MMAs (S ~0.43 us, PV ~0.58 us per 128-token tile) pace the
// tile, not the softmax, so moving exponentials off the special-function
// unit only lengthens the softmax (per-tile compute 0.61 / 0.58 / 0.64 /
// 0.70 us for 0 / 2 / 3 / 4 of 8): none.
constexpr int kPolyOf8 = 0;

struct PairSmem {
  static constexpr int D = 128;
  static constexpr int kKHalfBytes = 64 * 128;           // 64 tokens x 64 columns
  static constexpr int kKBytes = 2 * kKHalfBytes;        // this CTA's 64 tokens, all columns
  static constexpr int kVBytes = kPW * 128;              // 128 tokens x this CTA's 64 columns
  static constexpr int kStageBytes = kKBytes + kVBytes;  // 32 KB
  static constexpr int kQOff = kPStages * kStageBytes;
  static constexpr int kQHalf = 128 * 128;               // 128 rows x 64 columns
  static constexpr int kQBytes = 2 * kQHalf;
  static constexpr int kPartsOff = kQOff + 2 * kQBytes;  // two Q buffers
  static constexpr int kPitch = D + 8;                   // halves per partial row
  static constexpr int kBarOff = kPartsOff + kMaxParts * 8;
  // kv_full[S] kv_empty[S] q_full[2] q_empty[2] s_full[2] s_empty[2]
  // p_full[2] pv_done[2] o_free
  static constexpr int kNumBars = 2 * kPStages + 13;
  // then the TMEM address, the part count and the item's tile count
  static constexpr int kTotal = kBarOff + kNumBars * 8 + 16;
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
                                                uint32_t bar, int t, const PartGeom& geo,
                                                Pages8 pg, int c) {
  using S = PairSmem;
  uint8_t* sk = stage;
  uint8_t* sv = stage + S::kKBytes;
  const int g = geo.g, b = geo.b;
  if (t < geo.n_ptiles) {
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
      const int npages =
          min(kPW / PF_PAGE_SIZE, (geo.P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
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
    const int j = t - geo.n_ptiles;
    mbar_arrive_expect_tx(bar, S::kStageBytes);
#pragma unroll
    for (int h = 0; h < 2; ++h)
      tma_load_3d(smem_u32(sk + h * S::kKHalfBytes), tm_tk, h * 64, g,
                  geo.node0 + j * kPW + c * 64, bar);
    tma_load_3d(smem_u32(sv), tm_tv, c * 64, g, geo.node0 + j * kPW, bar);
  }
}

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
  uint8_t* sQ = smem + S::kQOff;  // [2][kQBytes]
  unsigned long long* parts = reinterpret_cast<unsigned long long*>(smem + S::kPartsOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* kv_full = bars;                // [S] own loads (+ the odd CTA's forward, leader)
  uint64_t* kv_empty = bars + kPStages;    // [S]
  uint64_t* q_full = bars + 2 * kPStages;  // [2] (+ forward, leader)
  uint64_t* q_empty = q_full + 2;          // [2] the part's last S MMA has completed
  uint64_t* s_full = q_full + 4;           // [2]
  uint64_t* s_empty = q_full + 6;          // [2] (leader's used)
  uint64_t* p_full = q_full + 8;           // [2] (leader's used)
  uint64_t* pv_done = q_full + 10;         // [2]
  uint64_t* o_free = q_full + 12;          // (leader's used)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + S::kNumBars);
  int* n_parts_slot = reinterpret_cast<int*>(bars + S::kNumBars) + 1;
  int* my_tiles_slot = reinterpret_cast<int*>(bars + S::kNumBars) + 2;

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int c = rank & 1;              // position in the pair
  const int leader = rank & ~1;        // the pair's even CTA
  const int item = (int)blockIdx.x >> 1;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // PF_ATTN_EARLY_PREFETCH: as in attn_tc_kernel
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

  // Both CTAs of a pair derive the same plan, so every return before the
  // pair's first barrier is taken by both.
  if (warp == 0) {
    const int n = continuous_plan<kPW>(a, item, c == 0, parts);
    __syncwarp();
    if (lane == 0) {
      int tiles = 0;
      for (int p = 0; p < n; ++p) {
        const Part pt = unpack_part(parts[p]);
        tiles += pt.t1 - pt.t0;
      }
      *n_parts_slot = n;
      *my_tiles_slot = tiles;
    }
  }
  __syncthreads();
  const int n_parts = *n_parts_slot;
  const int my_tiles = *my_tiles_slot;
  if (n_parts == 0) {
    if (early) pdl_wait();  // completes only after the preceding kernel, like every CTA
    return;
  }

  if (tid == 0) {
    // the leader's load barriers also count the odd CTA's "landed" forward
    const uint32_t loads = c == 0 ? 2 : 1;
    for (int i = 0; i < kPStages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), loads);
      mbar_init(smem_u32(&kv_empty[i]), 1);  // the tile's PV (multicast commit)
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&q_full[i]), loads);
      mbar_init(smem_u32(&q_empty[i]), 1);
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_empty[i]), 8);   // the softmax warps of both CTAs
      mbar_init(smem_u32(&p_full[i]), 8);
      mbar_init(smem_u32(&pv_done[i]), 1);
    }
    mbar_init(smem_u32(o_free), 8);
    fence_mbar_init();
  }
  // Every CTA's barriers are initialised before any peer signals them (the
  // odd CTA forwards to the leader's barriers, the leader's commits arrive
  // on both).
  cluster_arrive_release();
  cluster_wait_acquire();

  const uint32_t s_empty_l0 = mapa_cluster(smem_u32(&s_empty[0]), (uint32_t)leader);
  const uint32_t p_full_l0 = mapa_cluster(smem_u32(&p_full[0]), (uint32_t)leader);
  const uint32_t o_free_l = mapa_cluster(smem_u32(o_free), (uint32_t)leader);

  // The first part's leading prefix tiles may load before the preceding
  // kernel finishes (early prefetch); everything else after it.
  int n_pre = 0;
  {
    const Part p0 = unpack_part(parts[0]);
    const PartGeom g0 = part_geom(a, p0.q, a.nb >> 1, c, kPW);
    while (n_pre < kPStages && p0.t0 + n_pre < p0.t1 && p0.t0 + n_pre < g0.n_ptiles) ++n_pre;
    if (tid == 0) {
      Pages8 pg[kPStages];
#pragma unroll
      for (int i = 0; i < kPStages; ++i)
        pg[i] = i < n_pre ? kv_tile_pages8(a, p0.t0 + i, g0.n_ptiles, g0.b, g0.P) : no_pages8();
#pragma unroll
      for (int i = 0; i < kPStages; ++i)
        if (i < n_pre)
          pair_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                          smem_u32(&kv_full[i]), p0.t0 + i, g0, pg[i], c);
    }
  }
  if (early) pdl_wait();
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_slot), kPTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();

  if (warp == 0) {
    // ---------------- producer: per part its Q, then its tiles
    if (lane == 0) {
      bool ok = true;
      int gi = 0;  // tile index over the item's parts
      for (int p = 0; p < n_parts && ok; ++p) {
        const Part pt = unpack_part(parts[p]);
        const PartGeom geo = part_geom(a, pt.q, a.nb >> 1, c, kPW);
        const int qb = p & 1;
        // Q buffer qb was last read by part p-2's S MMAs
        if (p >= 2) ok = mbar_wait(smem_u32(&q_empty[qb]), ((p >> 1) & 1) ^ 1, a.err);
        if (!ok) break;
        mbar_arrive_expect_tx(smem_u32(&q_full[qb]), 2u * a.G * (a.nb >> 1) * 128);
#pragma unroll
        for (int h = 0; h < 2; ++h)
          tma_load_3d(smem_u32(sQ + qb * S::kQBytes + h * S::kQHalf), &tm_q, h * 64, geo.g * a.G,
                      geo.node0 + geo.nfirst, smem_u32(&q_full[qb]));
        for (int t = pt.t0; t < pt.t1 && ok; ++t, ++gi) {
          if (gi < n_pre) continue;  // loaded before the dependency wait
          const int st = gi % kPStages;
          const Pages8 pg = kv_tile_pages8(a, t, geo.n_ptiles, geo.b, geo.P);
          if (gi >= kPStages)
            ok = mbar_wait(smem_u32(&kv_empty[st]), ((gi / kPStages) & 1) ^ 1, a.err);
          if (ok)
            pair_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + st * S::kStageBytes,
                            smem_u32(&kv_full[st]), t, geo, pg, c);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && c == 1) {
      // ---------------- forwarder (odd CTA): once this CTA's Q of a part,
      // then each of its tile halves, has landed, arrive on the leader's
      // barrier (in the producer's issue order)
      const uint32_t q_full_l0 = mapa_cluster(smem_u32(&q_full[0]), (uint32_t)leader);
      const uint32_t kv_full_l0 = mapa_cluster(smem_u32(&kv_full[0]), (uint32_t)leader);
      bool ok = true;
      int gi = 0;
      for (int p = 0; p < n_parts && ok; ++p) {
        const Part pt = unpack_part(parts[p]);
        ok = mbar_wait(smem_u32(&q_full[p & 1]), (p >> 1) & 1, a.err);
        if (ok) mbar_arrive_cluster(q_full_l0 + 8 * (p & 1));
        for (int t = pt.t0; t < pt.t1 && ok; ++t, ++gi) {
          const int st = gi % kPStages;
          ok = mbar_wait(smem_u32(&kv_full[st]), (gi / kPStages) & 1, a.err);
          if (ok) mbar_arrive_cluster(kv_full_l0 + 8 * st);
        }
      }
    }
    // ---------------- MMA issuer (leader only), pair MMAs committed to both CTAs
    if (lane == 0 && c == 0) {
      const uint32_t id_s = umma_idesc_bf16(256, kPW);
      const uint32_t id_o = umma_idesc_bf16_bmn(256, D);
      const uint16_t both = (uint16_t)(3u << leader);
      // S side: part ps whose tiles end at s_end (tile counts over the
      // item); PV side: part pp from pv_start to pv_end
      int ps = 0, pp = 0;
      Part pts = unpack_part(parts[0]);
      int s_end = pts.t1 - pts.t0, pv_start = 0, pv_end = s_end;
      bool q_ready = false, o_ready = true;
      int ns = 0, np = 0;
      bool ok = true;
      unsigned idle = 0;
      unsigned long long t0 = 0;
      while (ok && np < my_tiles) {
        bool progressed = false;
        if (ns < my_tiles) {
          const int n = ns, st = n % kPStages, sb = n & 1;
          if (!q_ready) q_ready = mbar_test_wait(smem_u32(&q_full[ps & 1]), (ps >> 1) & 1);
          if (q_ready && mbar_test_wait(smem_u32(&kv_full[st]), (n / kPStages) & 1) &&
              mbar_test_wait(smem_u32(&s_empty[sb]), ((n >> 1) & 1) ^ 1)) {
            tc_fence_after();
            const uint32_t q0 = smem_u32(sQ + (ps & 1) * S::kQBytes);
            const uint32_t k0 = smem_u32(sKV + st * S::kStageBytes);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              umma_pair_ss(tmem + sb * kPW,
                           umma_desc_sw128(q0 + (kk >> 2) * S::kQHalf + (kk & 3) * 32),
                           umma_desc_sw128(k0 + (kk >> 2) * S::kKHalfBytes + (kk & 3) * 32), id_s,
                           kk > 0);
            umma_commit_pair(smem_u32(&s_full[sb]), both);
            ++ns;
            if (ns == s_end) {
              // the part's Q is read: its buffer may take part ps+2's Q (only
              // a part that exists waits for it)
              if (ps + 2 < n_parts) umma_commit_pair(smem_u32(&q_empty[ps & 1]), both);
              ++ps;
              q_ready = false;
              if (ps < n_parts) {
                pts = unpack_part(parts[ps]);
                s_end += pts.t1 - pts.t0;
              }
            }
            progressed = true;
          }
        }
        if (np < ns) {
          const int j = np, pb = j & 1, stj = j % kPStages;
          // the first PV of a part overwrites O: the softmax threads must
          // have read the previous part's O
          if (!o_ready) o_ready = mbar_test_wait(smem_u32(o_free), (pp - 1) & 1);
          if (o_ready && mbar_test_wait(smem_u32(&p_full[pb]), (j >> 1) & 1)) {
            tc_fence_after();
            const uint32_t v0 = smem_u32(sKV + stj * S::kStageBytes + S::kKBytes);
#pragma unroll
            for (int kt = 0; kt < kPW / 16; ++kt)
              umma_pair_ts(tmem + kPColO, tmem + kPColP + pb * 64 + kt * 8,
                           umma_desc_sw128_lbo(v0 + kt * 16 * 128, S::kVBytes, 1024), id_o,
                           (j > pv_start || kt > 0) ? 1u : 0u);
            umma_commit_pair(smem_u32(&pv_done[pb]), both);
            // only stages that will be refilled are released: after the last
            // PV nothing more arrives on the odd CTA's barriers
            if (j + kPStages < my_tiles) umma_commit_pair(smem_u32(&kv_empty[stj]), both);
            ++np;
            if (np == pv_end && np < my_tiles) {
              ++pp;
              const Part pn = unpack_part(parts[pp]);
              pv_start = np;
              pv_end = np + (pn.t1 - pn.t0);
              o_ready = false;
            }
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
    // ---------------- softmax / correction / epilogue: one row per thread
    const int quad = warp & 3;
    const int rl = quad * 32 + lane;       // row within this CTA (its TMEM lane)
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    bool ok = true;
    int gi = 0;
    for (int p = 0; p < n_parts && ok; ++p) {
      const Part pt = unpack_part(parts[p]);
      const PartGeom geo = part_geom(a, pt.q, a.nb >> 1, c, kPW);
      uint64_t mk0 = 0, mk1 = 0;
      if (rl < geo.rows) {
        const int node = geo.node0 + geo.nfirst + rl / a.G;
        mk0 = a.mask[2 * node];
        mk1 = a.mask[2 * node + 1];
      }
      float m_ref = -INFINITY, l = 0.f;  // running max (log2) and sum of this row
      const int gi0 = gi;
      for (int t = pt.t0; t < pt.t1 && ok; ++t, ++gi) {
        const int sb = gi & 1;
        const int st = gi % kPStages;
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[sb]), (gi >> 1) & 1, a.err));
        if (!ok) break;  // warp-uniform
        tc_fence_after();
        uint32_t sraw[kPW];
#pragma unroll
        for (int c0 = 0; c0 < kPW; c0 += 32)
          tmem_ld_32(tmem + lane_base + sb * kPW + c0,
                     *reinterpret_cast<uint32_t(*)[32]>(&sraw[c0]));
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(s_empty_l0 + 8 * sb);
        float sv[kPW];
#pragma unroll
        for (int cc = 0; cc < kPW; ++cc) sv[cc] = __uint_as_float(sraw[cc]);

        const bool is_prefix = t < geo.n_ptiles;
        const int valid = is_prefix ? min(kPW, geo.P - t * kPW) : kPW;
        if (!is_prefix || valid < kPW) {
          // prefix columns past the end, or proposal columns that are not
          // ancestors of this row's node (columns 0..127 are nodes 0..127)
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
          // O must hold exactly the part's tiles before this one: wait for
          // the previous PV (a part's first tile never rescales: m_ref was
          // -inf)
          if (gi > gi0) mbar_wait(smem_u32(&pv_done[(gi - 1) & 1]), ((gi - 1) >> 1) & 1, a.err);
          tc_fence_after();
          const float alpha = resc ? ex2_approx(m_ref - m_new) : 1.f;
#pragma unroll
          for (int c0 = 0; c0 < D; c0 += 32) {
            uint32_t ov[32];
            tmem_ld_32(tmem + lane_base + kPColO + c0, ov);
            tmem_ld_wait();
#pragma unroll
            for (int cc = 0; cc < 32; ++cc)
              ov[cc] = __float_as_uint(__uint_as_float(ov[cc]) * alpha);
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
          // kPolyOf8 of every 8 column pairs on the FMA pipe, the rest on the
          // special-function unit
          float p0, p1;
          if ((cc & 7) < kPolyOf8) {
            exp2_poly_x2(x0, x1, p0, p1);
          } else {
            p0 = ex2_approx(x0);
            p1 = ex2_approx(x1);
          }
          rs2[cc & 3] = fadd2(rs2[cc & 3], f32x2_pack(p0, p1));
          pk[cc] = pack_bf16(p0, p1);
        }
        float r0, r1;
        f32x2_unpack(fadd2(fadd2(rs2[0], rs2[1]), fadd2(rs2[2], rs2[3])), r0, r1);
        l += r0 + r1;
        // P buffer sb was last read by PV_{gi-2}.
        if (gi >= 2) mbar_wait(smem_u32(&pv_done[sb]), ((gi - 2) >> 1) & 1, a.err);
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
      if (!ok) break;
      // ---- the part's epilogue: O / l of this row, once its last PV landed
      const int last = gi - 1;
      mbar_wait(smem_u32(&pv_done[last & 1]), (last >> 1) & 1, a.err);
      tc_fence_after();
      uint32_t ov[D];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32)
        tmem_ld_32(tmem + lane_base + kPColO + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      // the next part's first PV may now overwrite O (after the last part
      // nothing waits for it)
      if (lane == 0 && p + 1 < n_parts) mbar_arrive_cluster(o_free_l);
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
      if (rl < geo.rows) {
        if (pt.whole) {
          const int node = geo.node0 + geo.nfirst + rl / a.G;
          const int h = geo.g * a.G + rl % a.G;
          __nv_bfloat16* dst =
              reinterpret_cast<__nv_bfloat16*>(a.out) + ((size_t)node * a.Hq + h) * D;
#pragma unroll
          for (int cc = 0; cc < D; cc += 8) {
            uint4 v;
            v.x = pack_bf16(__uint_as_float(ov[cc]) * inv_l, __uint_as_float(ov[cc + 1]) * inv_l);
            v.y = pack_bf16(__uint_as_float(ov[cc + 2]) * inv_l, __uint_as_float(ov[cc + 3]) * inv_l);
            v.z = pack_bf16(__uint_as_float(ov[cc + 4]) * inv_l, __uint_as_float(ov[cc + 5]) * inv_l);
            v.w = pack_bf16(__uint_as_float(ov[cc + 6]) * inv_l, __uint_as_float(ov[cc + 7]) * inv_l);
            *reinterpret_cast<uint4*>(dst + cc) = v;
          }
        } else {
          // this piece's partial: row c * (nodes per CTA) * G + rl of its slot
          const int pr = c * (a.nb >> 1) * a.G + rl;
          __half* dst = reinterpret_cast<__half*>(a.ws) + ((size_t)pt.slot * a.bm + pr) * S::kPitch;
#pragma unroll
          for (int cc = 0; cc < D; cc += 8) {
            uint4 v;
            v.x = pack_half(__uint_as_float(ov[cc]) * inv_l, __uint_as_float(ov[cc + 1]) * inv_l);
            v.y = pack_half(__uint_as_float(ov[cc + 2]) * inv_l, __uint_as_float(ov[cc + 3]) * inv_l);
            v.z = pack_half(__uint_as_float(ov[cc + 4]) * inv_l, __uint_as_float(ov[cc + 5]) * inv_l);
            v.w = pack_half(__uint_as_float(ov[cc + 6]) * inv_l, __uint_as_float(ov[cc + 7]) * inv_l);
            *reinterpret_cast<uint4*>(dst + cc) = v;
          }
          *reinterpret_cast<float*>(dst + D) = inv_l > 0.f ? m_ref + __log2f(l) : -INFINITY;
        }
      }
    }
  }
  __syncwarp();  // the producer and MMA lanes rejoin their warps before the barriers
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kPTmemCols);
  }
}

}  // namespace

static int pair_smem_bytes() { return PairSmem::kTotal + 1024; }

cudaError_t launch_attention_pair(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  const int smem = pair_smem_bytes();
  static DeviceMemo limit;
  cudaError_t e = ensure_smem_limit((const void*)attn_pair_kernel, smem, limit);
  if (e != cudaSuccess) return e;
  return launch_ex(attn_pair_kernel, dim3(2 * a.items), dim3(kPThreads), smem, s, 2, pdl, m.q,
                   m.tk, m.tv, m.ck, m.cv, a);
}

}  // namespace pf
