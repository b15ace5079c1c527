// Tree-masked GQA attention for batches: the 128-token, P-in-TMEM pipeline
// of attn_tc2_kernel (one CTA per SM, 128 query rows per CTA) with the
// continuous work split.  The (sequence, KV head, 128-row block) groups'
// tiles are laid end to end and cut into one equal range per SM, so a batch
// whose prefixes differ threefold in length still keeps every SM busy to
// the end (with a fixed number of CTAs per group, the longest sequences'
// CTAs run alone at the end).  A range covers pieces of one or more groups
// (parts); a part that is a whole group writes the output, any other part a
// normalised partial that attn_combine_kernel merges (see continuous_plan).
//
//   warp 0     TMA producer: per part its Q rows (one buffer, reloaded once
//              the part's last S MMA has read it), then K/V tiles (64 KB)
//              into a ring of kSkStages stages
//   warp 1     TMEM owner and MMA issuer (one thread):
//                S_i  = Q K_i^T   M=128, N=128, K=D   -> S[i % 2]
//                O   += P_i V_i   M=128, N=D,  K=128  (A = P in TMEM) -> O
//   softmax    one warpgroup, one query row per thread (its TMEM lane), as
//              in attn_tc2_kernel; per part it resets its row's running
//              maximum and sum, and after the part's last tile reads O / l
//              out of TMEM, reports "O read" (the next part's first PV
//              overwrites O) and writes its row
//
// Barrier phases run on across parts: tile i of the item (counting all its
// parts) uses ring stage i % kSkStages and S / P buffer i % 2.
//
// TMEM columns: S[0] 0..127, S[1] 128..255, O 256..383, P[0] 384..447,
// P[1] 448..511.
#include <cuda_fp16.h>

#include "attn_common.cuh"

namespace pf {

namespace {

constexpr int kSW = 128;             // tokens per K/V tile
constexpr int kSkThreads = 192;      // producer, MMA, one softmax warpgroup
constexpr uint32_t kSkTmemCols = 512;
constexpr uint32_t kSkColO = 256, kSkColP = 384;
constexpr float kSkRescaleLog2 = 8.f;
constexpr int kSkStages = 3;
constexpr int kSkMaxParts = kSkMaxGroups;

struct SkSmem {
  static constexpr int D = 128;
  static constexpr int kHalfBytes = kSW * 128;            // 128 tokens x 64 columns
  static constexpr int kTileBytes = 2 * kHalfBytes;       // one K or V tile
  static constexpr int kStageBytes = 2 * kTileBytes;      // K + V: 64 KB
  static constexpr int kQOff = kSkStages * kStageBytes;
  static constexpr int kQHalf = 128 * 128;                // 128 rows x 64 columns
  static constexpr int kPartsOff = kQOff + 2 * kQHalf;
  static constexpr int kPitch = D + 8;                    // halves per partial row
  static constexpr int kBarOff = kPartsOff + kSkMaxParts * 8;
  // kv_full[S] kv_empty[S] q_full q_empty s_full[2] s_empty[2] p_full[2]
  // pv_done[2] o_free
  static constexpr int kNumBars = 2 * kSkStages + 11;
  // then the TMEM address, the part count and the item's tile count
  static constexpr int kTotal = kBarOff + kNumBars * 8 + 16;
  static_assert(kTotal + 1024 <= 232448, "shared memory budget");
};

// TMA loads of one 128-token K/V tile into a ring stage: K then V, each two
// 64-column halves of 128 rows; prefix cache (contiguous: one 3-D box per
// half; paged: one 4-D box per 16-token page holding prefix rows) or, past
// the prefix, the proposal's own rows.  Arms `bar` with the bytes.
__device__ __forceinline__ void sk_issue_tile(const AttnArgs& a, const CUtensorMap* tm_ck,
                                              const CUtensorMap* tm_cv, const CUtensorMap* tm_tk,
                                              const CUtensorMap* tm_tv, uint8_t* stage,
                                              uint32_t bar, int t, const PartGeom& geo,
                                              Pages8 pg) {
  using S = SkSmem;
  uint8_t* sk = stage;
  uint8_t* sv = stage + S::kTileBytes;
  const int g = geo.g, b = geo.b;
  if (t < geo.n_ptiles) {
    const int tok0 = t * kSW;
    if (a.layout == PF_KV_CONTIGUOUS) {
      mbar_arrive_expect_tx(bar, 2 * S::kTileBytes);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        tma_load_3d(smem_u32(sk + h * S::kHalfBytes), tm_ck, h * 64, tok0, b * a.Hkv + g, bar);
        tma_load_3d(smem_u32(sv + h * S::kHalfBytes), tm_cv, h * 64, tok0, b * a.Hkv + g, bar);
      }
    } else {
      const int npages =
          min(kSW / PF_PAGE_SIZE, (geo.P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
      mbar_arrive_expect_tx(bar, 2 * 2 * npages * PF_PAGE_SIZE * 128);
      const int pages[8] = {pg.lo.x, pg.lo.y, pg.lo.z, pg.lo.w, pg.hi.x, pg.hi.y, pg.hi.z, pg.hi.w};
#pragma unroll
      for (int p = 0; p < 8; ++p) {
        if (p >= npages) break;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int off = h * S::kHalfBytes + p * PF_PAGE_SIZE * 128;
          tma_load_4d(smem_u32(sk + off), tm_ck, h * 64, 0, g, pages[p], bar);
          tma_load_4d(smem_u32(sv + off), tm_cv, h * 64, 0, g, pages[p], bar);
        }
      }
    }
  } else {
    const int j = t - geo.n_ptiles;
    mbar_arrive_expect_tx(bar, 2 * S::kTileBytes);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      tma_load_3d(smem_u32(sk + h * S::kHalfBytes), tm_tk, h * 64, g, geo.node0 + j * kSW, bar);
      tma_load_3d(smem_u32(sv + h * S::kHalfBytes), tm_tv, h * 64, g, geo.node0 + j * kSW, bar);
    }
  }
}

// D[tmem] (+)= A[tmem] * B[smem]^T, kind::f16: A is 128 rows (TMEM lanes) x
// 16 bf16 (8 columns of packed pairs) starting at column a_tmem.
__device__ __forceinline__ void sk_umma_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                               uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p; }" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__global__ void __launch_bounds__(kSkThreads, 1)
    attn_sk_kernel(const __grid_constant__ CUtensorMap tm_q,
                   const __grid_constant__ CUtensorMap tm_tk,
                   const __grid_constant__ CUtensorMap tm_tv,
                   const __grid_constant__ CUtensorMap tm_ck,
                   const __grid_constant__ CUtensorMap tm_cv, const AttnArgs a) {
  using S = SkSmem;
  constexpr int D = 128;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sKV = smem;
  uint8_t* sQ = smem + S::kQOff;
  unsigned long long* parts = reinterpret_cast<unsigned long long*>(smem + S::kPartsOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  uint64_t* kv_full = bars;                  // [S]
  uint64_t* kv_empty = bars + kSkStages;     // [S] the tile's PV has completed
  uint64_t* q_full = bars + 2 * kSkStages;
  uint64_t* q_empty = q_full + 1;            // the part's last S MMA has completed
  uint64_t* s_full = q_full + 2;             // [2]
  uint64_t* s_empty = q_full + 4;            // [2] one arrive per softmax warp
  uint64_t* p_full = q_full + 6;             // [2]
  uint64_t* pv_done = q_full + 8;            // [2]
  uint64_t* o_free = q_full + 10;            // the part's O has been read
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + S::kNumBars);
  int* n_parts_slot = reinterpret_cast<int*>(bars + S::kNumBars) + 1;
  int* my_tiles_slot = reinterpret_cast<int*>(bars + S::kNumBars) + 2;

  const int item = (int)blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // PF_ATTN_EARLY_PREFETCH: as in attn_tc_kernel
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

  if (warp == 0) {
    const int n = continuous_plan<kSW>(a, item, true, parts);
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
    for (int i = 0; i < kSkStages; ++i) {
      mbar_init(smem_u32(&kv_full[i]), 1);
      mbar_init(smem_u32(&kv_empty[i]), 1);
    }
    mbar_init(smem_u32(q_full), 1);
    mbar_init(smem_u32(q_empty), 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s_full[i]), 1);
      mbar_init(smem_u32(&s_empty[i]), 4);
      mbar_init(smem_u32(&p_full[i]), 4);
      mbar_init(smem_u32(&pv_done[i]), 1);
    }
    mbar_init(smem_u32(o_free), 4);
    fence_mbar_init();
  }
  __syncthreads();

  // The first part's leading prefix tiles may load before the preceding
  // kernel finishes (early prefetch); everything else after it.
  int n_pre = 0;
  {
    const Part p0 = unpack_part(parts[0]);
    const PartGeom g0 = part_geom(a, p0.q, a.nb, 0, kSW);
    while (n_pre < kSkStages && p0.t0 + n_pre < p0.t1 && p0.t0 + n_pre < g0.n_ptiles) ++n_pre;
    if (tid == 0) {
      Pages8 pg[kSkStages];
#pragma unroll
      for (int i = 0; i < kSkStages; ++i)
        pg[i] = i < n_pre ? kv_tile_pages8(a, p0.t0 + i, g0.n_ptiles, g0.b, g0.P) : no_pages8();
#pragma unroll
      for (int i = 0; i < kSkStages; ++i)
        if (i < n_pre)
          sk_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                        smem_u32(&kv_full[i]), p0.t0 + i, g0, pg[i]);
    }
  }
  if (early) pdl_wait();
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kSkTmemCols);
    tmem_relinquish();
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
        const PartGeom geo = part_geom(a, pt.q, a.nb, 0, kSW);
        // the Q buffer was last read by part p-1's S MMAs
        if (p >= 1) ok = mbar_wait(smem_u32(q_empty), (p - 1) & 1, a.err);
        if (!ok) break;
        mbar_arrive_expect_tx(smem_u32(q_full), 2u * a.G * a.nb * 128);
#pragma unroll
        for (int h = 0; h < 2; ++h)
          tma_load_3d(smem_u32(sQ + h * S::kQHalf), &tm_q, h * 64, geo.g * a.G,
                      geo.node0 + geo.nfirst, smem_u32(q_full));
        for (int t = pt.t0; t < pt.t1 && ok; ++t, ++gi) {
          if (gi < n_pre) continue;  // loaded before the dependency wait
          const int st = gi % kSkStages;
          const Pages8 pg = kv_tile_pages8(a, t, geo.n_ptiles, geo.b, geo.P);
          if (gi >= kSkStages)
            ok = mbar_wait(smem_u32(&kv_empty[st]), ((gi / kSkStages) & 1) ^ 1, a.err);
          if (ok)
            sk_issue_tile(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + st * S::kStageBytes,
                          smem_u32(&kv_full[st]), t, geo, pg);
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = umma_idesc_bf16(128, kSW);
      const uint32_t id_o = umma_idesc_bf16_bmn(128, D);
      const uint32_t q0 = smem_u32(sQ);
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
          const int n = ns, st = n % kSkStages, sb = n & 1;
          if (!q_ready) q_ready = mbar_test_wait(smem_u32(q_full), ps & 1);
          if (q_ready && mbar_test_wait(smem_u32(&kv_full[st]), (n / kSkStages) & 1) &&
              mbar_test_wait(smem_u32(&s_empty[sb]), ((n >> 1) & 1) ^ 1)) {
            tc_fence_after();
            const uint32_t k0 = smem_u32(sKV + st * S::kStageBytes);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              umma_bf16(tmem + sb * kSW,
                        umma_desc_sw128(q0 + (kk >> 2) * S::kQHalf + (kk & 3) * 32),
                        umma_desc_sw128(k0 + (kk >> 2) * S::kHalfBytes + (kk & 3) * 32), id_s,
                        kk > 0);
            umma_commit(smem_u32(&s_full[sb]));
            ++ns;
            if (ns == s_end) {
              // the part's Q is read: the buffer may take the next part's Q
              if (ps + 1 < n_parts) umma_commit(smem_u32(q_empty));
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
          const int j = np, pb = j & 1, stj = j % kSkStages;
          // the first PV of a part overwrites O: the softmax threads must
          // have read the previous part's O
          if (!o_ready) o_ready = mbar_test_wait(smem_u32(o_free), (pp - 1) & 1);
          if (o_ready && mbar_test_wait(smem_u32(&p_full[pb]), (j >> 1) & 1)) {
            tc_fence_after();
            const uint32_t v0 = smem_u32(sKV + stj * S::kStageBytes + S::kTileBytes);
#pragma unroll
            for (int kt = 0; kt < kSW / 16; ++kt)
              sk_umma_tmem_a(tmem + kSkColO, tmem + kSkColP + pb * 64 + kt * 8,
                             umma_desc_sw128_lbo(v0 + kt * 16 * 128, S::kHalfBytes, 1024), id_o,
                             (j > pv_start || kt > 0) ? 1u : 0u);
            umma_commit(smem_u32(&pv_done[pb]));
            umma_commit(smem_u32(&kv_empty[stj]));
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
    const int rl = quad * 32 + lane;       // row within the block (its TMEM lane)
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    bool ok = true;
    int gi = 0;
    for (int p = 0; p < n_parts && ok; ++p) {
      const Part pt = unpack_part(parts[p]);
      const PartGeom geo = part_geom(a, pt.q, a.nb, 0, kSW);
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
        const int st = gi % kSkStages;
        ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[sb]), (gi >> 1) & 1, a.err));
        if (!ok) break;  // warp-uniform
        tc_fence_after();
        uint32_t sraw[kSW];
#pragma unroll
        for (int c0 = 0; c0 < kSW; c0 += 32)
          tmem_ld_32(tmem + lane_base + sb * kSW + c0,
                     *reinterpret_cast<uint32_t(*)[32]>(&sraw[c0]));
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&s_empty[sb]));
        float sv[kSW];
#pragma unroll
        for (int cc = 0; cc < kSW; ++cc) sv[cc] = __uint_as_float(sraw[cc]);

        const bool is_prefix = t < geo.n_ptiles;
        const int valid = is_prefix ? min(kSW, geo.P - t * kSW) : kSW;
        if (!is_prefix || valid < kSW) {
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
        const bool resc = m_ref != -INFINITY && m_new > m_ref + kSkRescaleLog2;
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
            tmem_ld_32(tmem + lane_base + kSkColO + c0, ov);
            tmem_ld_wait();
#pragma unroll
            for (int cc = 0; cc < 32; ++cc)
              ov[cc] = __float_as_uint(__uint_as_float(ov[cc]) * alpha);
            tmem_st_32(tmem + lane_base + kSkColO + c0, ov);
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
        uint32_t pk[kSW / 2];
#pragma unroll
        for (int cc = 0; cc < kSW / 2; ++cc) {
          float x0, x1;
          f32x2_unpack(ffma2(f32x2_pack(sv[2 * cc], sv[2 * cc + 1]), sc2, mu2), x0, x1);
          const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          rs2[cc & 3] = fadd2(rs2[cc & 3], f32x2_pack(p0, p1));
          pk[cc] = pack_bf16(p0, p1);
        }
        float r0, r1;
        f32x2_unpack(fadd2(fadd2(rs2[0], rs2[1]), fadd2(rs2[2], rs2[3])), r0, r1);
        l += r0 + r1;
        // P buffer sb was last read by PV_{gi-2}.
        if (gi >= 2) mbar_wait(smem_u32(&pv_done[sb]), ((gi - 2) >> 1) & 1, a.err);
        tc_fence_after();
        tmem_st_32(tmem + lane_base + kSkColP + sb * 64,
                   *reinterpret_cast<uint32_t(*)[32]>(&pk[0]));
        tmem_st_32(tmem + lane_base + kSkColP + sb * 64 + 32,
                   *reinterpret_cast<uint32_t(*)[32]>(&pk[32]));
        tmem_st_wait();
        if (valid < kSW) {
          // Cache rows past the prefix end may hold anything (even NaN bit
          // patterns): zero their V so masked columns contribute exactly 0.
          // The rows from `valid` on are one contiguous run per 64-column half.
          uint4* vt = reinterpret_cast<uint4*>(sKV + st * S::kStageBytes + S::kTileBytes);
          const int per_half = (kSW - valid) * 8;   // 16-byte chunks past the end
#pragma unroll
          for (int h = 0; h < 2; ++h)
            for (int cc = rl; cc < per_half; cc += 128)
              vt[h * kSW * 8 + valid * 8 + cc] = make_uint4(0, 0, 0, 0);
          fence_proxy_async_smem();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&p_full[sb]));
      }
      if (!ok) break;
      // ---- the part's epilogue: O / l of this row, once its last PV landed
      const int last = gi - 1;
      mbar_wait(smem_u32(&pv_done[last & 1]), (last >> 1) & 1, a.err);
      tc_fence_after();
      uint32_t ov[D];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32)
        tmem_ld_32(tmem + lane_base + kSkColO + c0, *reinterpret_cast<uint32_t(*)[32]>(&ov[c0]));
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      // the next part's first PV may now overwrite O (after the last part
      // nothing waits for it)
      if (lane == 0 && p + 1 < n_parts) mbar_arrive(smem_u32(o_free));
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
          __half* dst = reinterpret_cast<__half*>(a.ws) + ((size_t)pt.slot * a.bm + rl) * S::kPitch;
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
    tmem_dealloc(tmem, kSkTmemCols);
  }
}

}  // namespace

cudaError_t launch_attention_sk(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  const int smem = SkSmem::kTotal + 1024;
  static DeviceMemo limit;
  cudaError_t e = ensure_smem_limit((const void*)attn_sk_kernel, smem, limit);
  if (e != cudaSuccess) return e;
  return launch_ex(attn_sk_kernel, dim3(a.items), dim3(kSkThreads), smem, s, 1, pdl, m.q, m.tk,
                   m.tv, m.ck, m.cv, a);
}

}  // namespace pf
