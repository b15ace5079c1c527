// Tree-masked GQA attention of the proposal nodes over the reused prefix KV
// (single-pass verification, Section 3.2, over the KV carried forward per
// Section 3.4).  One launch = one layer.
//
// bf16 path.  A CTA owns one (sequence b, KV head g, row block) and one
// slice of the KV tiles.  Its 128 query rows are the G query heads of g for
// up to floor(128 / G) proposal nodes, so every K/V byte brought into shared
// memory serves all G heads.  K/V tiles of 64 tokens stream in by TMA
// (128-byte swizzle) through a multi-stage mbarrier ring; prefix tiles come
// from the cache (contiguous, or one 16-token page per TMA box), the last
// tiles come from the proposal's own K/V under the ancestor bitmap.  S = QK^T
// and O += PV use the m16n8k16 bf16 tensor-core MMA with an fp32 online
// softmax.  The CTAs of a cluster split the KV tiles of one row block and
// merge their (max, sum, O) partials through distributed shared memory, so
// no workspace and no second launch are needed.
#include <cooperative_groups.h>

#include "attn_common.cuh"

namespace cg = cooperative_groups;

namespace pf {

namespace {

constexpr int kStages = 3;

// Shared-memory plan of one CTA with BM query rows (BM / 16 warps).
template <int D, int BM>
struct AttnSmem {
  static constexpr int kThreads = BM * 2;
  static constexpr int kHalves = D / 64;
  static constexpr int kTileBytes = kBN * D * 2;       // one K or V tile
  static constexpr int kStageBytes = 2 * kTileBytes;   // K + V
  static constexpr int kQBytes = BM * D * 2;
  static constexpr int kRedOff = kStages * kStageBytes + kQBytes;
  static constexpr int kBarOff = kRedOff + 2 * BM * 4;
  static constexpr int kTotal = kBarOff + (kStages + 1) * 8 + 16;
  static constexpr int kOStride = D + 4;               // fp32 partial-O row pitch
  static_assert(BM * kOStride * 4 <= kStages * kStageBytes, "partial O must fit the KV ring");
};

template <int D, int BM>
__global__ void __launch_bounds__(BM * 2, 1)
    attn_bf16_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_tk,
                     const __grid_constant__ CUtensorMap tm_tv,
                     const __grid_constant__ CUtensorMap tm_ck,
                     const __grid_constant__ CUtensorMap tm_cv, const AttnArgs a) {
  using S = AttnSmem<D, BM>;
  constexpr int kThreads = S::kThreads;
  constexpr int KS = D / 16;   // k-steps of QK^T
  constexpr int NT = D / 8;    // n8 tiles of O
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sKV = smem;
  uint8_t* sQ = smem + kStages * S::kStageBytes;
  float* sM = reinterpret_cast<float*>(smem + S::kRedOff);
  float* sL = sM + BM;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S::kBarOff);
  float* sO = reinterpret_cast<float*>(smem);  // reuses the KV ring after the loop

  cg::cluster_group cluster = cg::this_cluster();
  const int nsplit = a.splits;
  const int split = (int)cluster.block_rank();
  int cid = blockIdx.x / nsplit;
  const int rb = cid % a.rb_count;
  cid /= a.rb_count;
  const int g = cid % a.Hkv;
  const int b = cid / a.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // With PF_ATTN_EARLY_PREFETCH the tree structure, prefix lengths and the
  // prefix cache were complete before the preceding kernel started, so they
  // are read, and the cache tiles requested, before waiting for that kernel
  // (programmatic dependent launch); q and the proposal K/V are read after.
  const bool early = (a.flags & PF_ATTN_EARLY_PREFETCH) != 0;
  if (!early) pdl_wait();

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
  const int n_ptiles = (P + kBN - 1) / kBN;
  const int ntiles = n_ptiles + (nn + kBN - 1) / kBN;
  const int t_begin = (int)((long long)ntiles * split / nsplit);
  const int my_tiles = (int)((long long)ntiles * (split + 1) / nsplit) - t_begin;
  const int first = min(kStages, my_tiles);

  const uint32_t qbar = smem_u32(&bars[kStages]);
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(smem_u32(&bars[i]), 1);
    mbar_init(qbar, 1);
    fence_mbar_init();
    int4 pg[kStages];  // every first tile's page entries in one round trip
#pragma unroll
    for (int i = 0; i < kStages; ++i)
      pg[i] = i < first ? kv_tile_pages(a, t_begin + i, n_ptiles, b, P) : make_int4(-1, -1, -1, -1);
#pragma unroll
    for (int i = 0; i < kStages; ++i)
      if (i < first && t_begin + i < n_ptiles)
        issue_kv_tile<D>(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                         smem_u32(&bars[i]), t_begin + i, n_ptiles, b, g, node0, P, pg[i]);
  }
  if (early) pdl_wait();
  if (tid == 0) {
    mbar_arrive_expect_tx(qbar, S::kHalves * a.G * a.nb * 128);
#pragma unroll
    for (int h = 0; h < S::kHalves; ++h)
      tma_load_3d(smem_u32(sQ + h * BM * 128), &tm_q, h * 64, g * a.G, node0 + nfirst, qbar);
    for (int i = 0; i < first; ++i)
      if (t_begin + i >= n_ptiles)  // proposal tiles: no page entries
        issue_kv_tile<D>(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, sKV + i * S::kStageBytes,
                         smem_u32(&bars[i]), t_begin + i, n_ptiles, b, g, node0, P,
                         make_int4(-1, -1, -1, -1));
  }
  __syncthreads();
  pdl_launch_dependents();

  // Rows owned by this thread in the m16n8 fragment layout.
  const int r0 = warp * 16 + (lane >> 2), r1 = r0 + 8;
  const bool warp_active = warp * 16 < rows;
  uint64_t mk0[2] = {0, 0}, mk1[2] = {0, 0};
  if (r0 < rows) {
    const int t0 = node0 + nfirst + r0 / a.G;
    mk0[0] = a.mask[2 * t0];
    mk0[1] = a.mask[2 * t0 + 1];
  }
  if (r1 < rows) {
    const int t1 = node0 + nfirst + r1 / a.G;
    mk1[0] = a.mask[2 * t1];
    mk1[1] = a.mask[2 * t1 + 1];
  }

  bool ok = mbar_wait(qbar, 0, a.err);
  uint32_t qa[KS][4];
  {
    const int qrow = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
      const int col = kk * 16 + (lane >> 4) * 8;
      const uint32_t addr = smem_u32(sQ + (col >> 6) * BM * 128) + sw128_off(qrow, col & 63);
      ldsm_x4(addr, qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
    }
  }

  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  float o[NT][4];
#pragma unroll
  for (int j = 0; j < NT; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;

  for (int i = 0; i < my_tiles; ++i) {
    const int st = i % kStages;
    uint8_t* stage = sKV + st * S::kStageBytes;
    if (ok) ok = mbar_wait(smem_u32(&bars[st]), (i / kStages) & 1, a.err);
    const int t = t_begin + i;
    const bool is_prefix = t < n_ptiles;
    const int valid = is_prefix ? min(kBN, P - t * kBN) : kBN;
    if (valid < kBN) {
      // Rows past the prefix end may hold anything (even NaN bit patterns):
      // zero their V so masked-out columns contribute exactly 0.
      // (each 64-column half holds its rows at 128-byte pitch: the rows
      // from `valid` on are one contiguous run per half)
      uint4* sv = reinterpret_cast<uint4*>(stage + S::kTileBytes);
      const int per_half = (kBN - valid) * 8;   // 16-byte chunks past the end
#pragma unroll
      for (int h = 0; h < S::kHalves; ++h)
        for (int c = tid; c < per_half; c += kThreads)
          sv[h * kBN * 8 + valid * 8 + c] = make_uint4(0, 0, 0, 0);
      fence_proxy_async_smem();
      __syncthreads();
    }
    if (warp_active) {
      const uint32_t sk = smem_u32(stage);
      const uint32_t sv = smem_u32(stage + S::kTileBytes);
      float s[8][4];
#pragma unroll
      for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < KS; ++kk) {
#pragma unroll
        for (int j = 0; j < 8; j += 2) {
          const int tok = j * 8 + (lane & 7) + (lane >> 4) * 8;
          const int col = kk * 16 + ((lane >> 3) & 1) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4(sk + (col >> 6) * kBN * 128 + sw128_off(tok, col & 63), b0, b1, b2, b3);
          mma_bf16_16816(s[j], qa[kk], b0, b1);
          mma_bf16_16816(s[j + 1], qa[kk], b2, b3);
        }
      }
      // scale + mask (prefix: column < valid; proposal: ancestor bit)
      const int jt = t - n_ptiles;  // proposal tile index (0 or 1) when !is_prefix
      const uint64_t w0 = is_prefix ? 0 : ((jt & 1) ? mk0[1] : mk0[0]);
      const uint64_t w1 = is_prefix ? 0 : ((jt & 1) ? mk1[1] : mk1[0]);
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int col = j * 8 + (lane & 3) * 2 + (e & 1);
          const bool vis = is_prefix ? (col < valid)
                                     : (((e < 2 ? w0 : w1) >> col) & 1ull) != 0;
          const float v = vis ? s[j][e] * a.scale_log2 : -INFINITY;
          s[j][e] = v;
          if (e < 2) mx0 = fmaxf(mx0, v);
          else mx1 = fmaxf(mx1, v);
        }
      }
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
      const float mn0 = fmaxf(m_run[0], mx0), mn1 = fmaxf(m_run[1], mx1);
      const float mu0 = mn0 == -INFINITY ? 0.f : mn0;
      const float mu1 = mn1 == -INFINITY ? 0.f : mn1;
      const float al0 = exp2f(m_run[0] - mu0), al1 = exp2f(m_run[1] - mu1);
      m_run[0] = mn0;
      m_run[1] = mn1;
      float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        s[j][0] = exp2f(s[j][0] - mu0);
        s[j][1] = exp2f(s[j][1] - mu0);
        s[j][2] = exp2f(s[j][2] - mu1);
        s[j][3] = exp2f(s[j][3] - mu1);
        rs0 += s[j][0] + s[j][1];
        rs1 += s[j][2] + s[j][3];
      }
      l_run[0] = l_run[0] * al0 + rs0;
      l_run[1] = l_run[1] * al1 + rs1;
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        o[j][0] *= al0;
        o[j][1] *= al0;
        o[j][2] *= al1;
        o[j][3] *= al1;
      }
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t pa[4];
        pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
        pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
        pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
        pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
        const int tok = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
        for (int j = 0; j < NT; j += 2) {
          const int col = j * 8 + (lane >> 4) * 8;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(sv + (col >> 6) * kBN * 128 + sw128_off(tok, col & 63), b0, b1, b2, b3);
          mma_bf16_16816(o[j], pa, b0, b1);
          mma_bf16_16816(o[j + 1], pa, b2, b3);
        }
      }
    }
    if (i + kStages < my_tiles) {
      // the refill's page entries are in flight while the warps finish
      const int4 pg = tid == 0 ? kv_tile_pages(a, t + kStages, n_ptiles, b, P)
                               : make_int4(-1, -1, -1, -1);
      __syncthreads();  // every warp is done with this stage before it is refilled
      if (tid == 0)
        issue_kv_tile<D>(a, &tm_ck, &tm_cv, &tm_tk, &tm_tv, stage, smem_u32(&bars[st]),
                         t + kStages, n_ptiles, b, g, node0, P, pg);
    }
  }

  __syncthreads();  // the KV ring is free: every warp has finished its last tile
  if ((lane & 3) == 0) {
    sM[r0] = m_run[0];
    sM[r1] = m_run[1];
  }
  l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 1);
  l_run[0] += __shfl_xor_sync(0xffffffffu, l_run[0], 2);
  l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 1);
  l_run[1] += __shfl_xor_sync(0xffffffffu, l_run[1], 2);
  if ((lane & 3) == 0) {
    sL[r0] = l_run[0];
    sL[r1] = l_run[1];
  }
  if (warp_active) {
#pragma unroll
    for (int j = 0; j < NT; ++j) {
      const int col = j * 8 + (lane & 3) * 2;
      *reinterpret_cast<float2*>(&sO[r0 * (D + 4) + col]) = make_float2(o[j][0], o[j][1]);
      *reinterpret_cast<float2*>(&sO[r1 * (D + 4) + col]) = make_float2(o[j][2], o[j][3]);
    }
  }
  cluster_merge<D, kThreads>(a, cluster, sM, sL, sO, rows, split, nsplit, node0 + nfirst, g, tid);
}

// ---------------------------------------------------------------- fp32 path
// CUDA-core kernel for fp32 inputs: one CTA per (sequence, KV head, 32 query
// rows); each warp keeps four rows' online softmax; K/V tiles of 32 tokens
// are staged in shared memory.
constexpr int kF32Rows = 32;
constexpr int kF32Tile = 32;

// Row of the prefix cache, or nullptr (and a flagged error) for a page-table
// entry outside the pool.
__device__ __forceinline__ const float* prefix_row(const AttnArgs& a, const float* cache, int b,
                                                   int g, int pos) {
  if (a.layout == PF_KV_CONTIGUOUS)
    return cache + (((size_t)b * a.Hkv + g) * a.max_seq + pos) * a.D;
  const int page = a.page_table[(size_t)b * a.pages_per_seq + pos / PF_PAGE_SIZE];
  if (page < 0 || page >= a.num_pages) {
    flag_error(a.err, PF_DEVERR_BOUNDS);
    return nullptr;
  }
  return cache + (((size_t)page * a.Hkv + g) * PF_PAGE_SIZE + pos % PF_PAGE_SIZE) * a.D;
}

__global__ void __launch_bounds__(256) attn_f32_kernel(const AttnArgs a) {
  extern __shared__ float fsm[];
  const int D = a.D, DP = D + 1;
  float* sK = fsm;                       // [32][D+1]
  float* sV = sK + kF32Tile * DP;        // [32][D]
  float* sQ = sV + kF32Tile * D;         // [32][D]
  int cid = blockIdx.x;
  const int rb = cid % a.rb_count;
  cid /= a.rb_count;
  const int g = cid % a.Hkv;
  const int b = cid / a.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  pdl_wait();
  const int node0 = a.cu_nodes[b];
  const int nn = a.cu_nodes[b + 1] - node0;
  const int P = a.prefix_len[b];
  if (node0 < 0 || nn < 1 || nn > a.max_nodes || node0 + nn > a.T || P < 0 ||
      P > a.max_prefix) {
    if (tid == 0 && rb == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
    return;
  }
  const int rows = nn * a.G;
  const int row0 = rb * kF32Rows;
  if (row0 >= rows) return;
  const float* q = static_cast<const float*>(a.q);
  for (int i = tid; i < kF32Rows * D; i += blockDim.x) {
    const int r = row0 + i / D;
    float v = 0.f;
    if (r < rows) v = q[((size_t)(node0 + r / a.G) * a.Hq + g * a.G + r % a.G) * D + i % D];
    sQ[i] = v;
  }
  constexpr int RPW = kF32Rows / 8;  // rows per warp
  constexpr int MAXC = 4;            // D / 32 <= 4
  float m[RPW], l[RPW], o[RPW][MAXC];
  uint64_t mk[RPW][2];
#pragma unroll
  for (int i = 0; i < RPW; ++i) {
    m[i] = -INFINITY;
    l[i] = 0.f;
#pragma unroll
    for (int c = 0; c < MAXC; ++c) o[i][c] = 0.f;
    const int r = row0 + warp * RPW + i;
    mk[i][0] = mk[i][1] = 0;
    if (r < rows) {
      mk[i][0] = a.mask[2 * (node0 + r / a.G)];
      mk[i][1] = a.mask[2 * (node0 + r / a.G) + 1];
    }
  }
  const float* ck = static_cast<const float*>(a.ck);
  const float* cv = static_cast<const float*>(a.cv);
  const float* tk = static_cast<const float*>(a.tk);
  const float* tv = static_cast<const float*>(a.tv);
  const int n_ptiles = (P + kF32Tile - 1) / kF32Tile;
  const int ntiles = n_ptiles + (nn + kF32Tile - 1) / kF32Tile;
  for (int t = 0; t < ntiles; ++t) {
    const bool is_prefix = t < n_ptiles;
    const int base = is_prefix ? t * kF32Tile : (t - n_ptiles) * kF32Tile;
    __syncthreads();
    for (int i = tid; i < kF32Tile * D; i += blockDim.x) {
      const int j = i / D, d = i % D;
      float kv = 0.f, vv = 0.f;
      if (is_prefix) {
        if (base + j < P) {
          const float* rk = prefix_row(a, ck, b, g, base + j);
          const float* rv = prefix_row(a, cv, b, g, base + j);
          kv = rk ? rk[d] : 0.f;
          vv = rv ? rv[d] : 0.f;
        }
      } else if (base + j < nn) {
        kv = tk[((size_t)(node0 + base + j) * a.Hkv + g) * D + d];
        vv = tv[((size_t)(node0 + base + j) * a.Hkv + g) * D + d];
      }
      sK[j * DP + d] = kv;
      sV[j * D + d] = vv;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < RPW; ++i) {
      const int lr = warp * RPW + i;
      if (row0 + lr >= rows) continue;
      float dot = 0.f;
      for (int d = 0; d < D; ++d) dot = fmaf(sQ[lr * D + d], sK[lane * DP + d], dot);
      const int j = base + lane;
      const uint64_t word = (j >> 6) ? mk[i][1] : mk[i][0];
      const bool vis = is_prefix ? (j < P) : (j < nn && ((word >> (j & 63)) & 1ull) != 0);
      const float s = vis ? dot * a.scale : -INFINITY;
      float mx = s;
#pragma unroll
      for (int off = 16; off; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      const float mn = fmaxf(m[i], mx);
      const float mu = mn == -INFINITY ? 0.f : mn;
      const float alpha = expf(m[i] - mu);
      const float p = expf(s - mu);
      float ps = p;
#pragma unroll
      for (int off = 16; off; off >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, off);
      m[i] = mn;
      l[i] = l[i] * alpha + ps;
#pragma unroll
      for (int c = 0; c < MAXC; ++c) o[i][c] *= alpha;
      for (int jj = 0; jj < kF32Tile; ++jj) {
        const float pj = __shfl_sync(0xffffffffu, p, jj);
#pragma unroll
        for (int c = 0; c < MAXC; ++c)
          if (lane + 32 * c < D) o[i][c] = fmaf(pj, sV[jj * D + lane + 32 * c], o[i][c]);
      }
    }
  }
  pdl_launch_dependents();
  float* out = static_cast<float*>(a.out);
#pragma unroll
  for (int i = 0; i < RPW; ++i) {
    const int r = row0 + warp * RPW + i;
    if (r >= rows) continue;
    const float inv = l[i] > 0.f ? 1.f / l[i] : 0.f;
    float* dst = out + ((size_t)(node0 + r / a.G) * a.Hq + g * a.G + r % a.G) * D;
#pragma unroll
    for (int c = 0; c < MAXC; ++c)
      if (lane + 32 * c < D) dst[lane + 32 * c] = o[i][c] * inv;
  }
}

template <int D, int BM>
cudaError_t launch_bf16_t(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  const int smem = AttnSmem<D, BM>::kTotal + 1024;
  static DeviceMemo limit;
  static DeviceMemo nonportable;
  cudaError_t e = ensure_smem_limit((const void*)attn_bf16_kernel<D, BM>, smem, limit);
  if (e != cudaSuccess) return e;
  if (a.splits > 8) {
    e = ensure_nonportable_cluster((const void*)attn_bf16_kernel<D, BM>, nonportable);
    if (e != cudaSuccess) return e;
  }
  const dim3 grid(a.B * a.Hkv * a.rb_count * a.splits);
  return launch_ex(attn_bf16_kernel<D, BM>, grid, dim3(AttnSmem<D, BM>::kThreads), smem, s,
                   a.splits, pdl, m.q, m.tk, m.tv, m.ck, m.cv, a);
}

template <int D>
cudaError_t launch_bf16_d(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl) {
  switch (a.bm) {
    case 32: return launch_bf16_t<D, 32>(a, m, s, pdl);
    case 64: return launch_bf16_t<D, 64>(a, m, s, pdl);
    default: return launch_bf16_t<D, 128>(a, m, s, pdl);
  }
}

}  // namespace

int attention_bf16_smem_bytes(int D, int bm) {
  if (D == 64)
    return (bm == 32 ? AttnSmem<64, 32>::kTotal
                     : bm == 64 ? AttnSmem<64, 64>::kTotal : AttnSmem<64, 128>::kTotal) + 1024;
  return (bm == 32 ? AttnSmem<128, 32>::kTotal
                   : bm == 64 ? AttnSmem<128, 64>::kTotal : AttnSmem<128, 128>::kTotal) + 1024;
}

template <int D, int BM>
bool cluster_fits_t(int cluster) {
  const int smem = AttnSmem<D, BM>::kTotal + 1024;
  static DeviceMemo limit;
  if (ensure_smem_limit((const void*)attn_bf16_kernel<D, BM>, smem, limit) != cudaSuccess)
    return false;
  if (cluster > 8 && cudaFuncSetAttribute(attn_bf16_kernel<D, BM>,
                                          cudaFuncAttributeNonPortableClusterSizeAllowed,
                                          1) != cudaSuccess)
    return false;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(cluster);
  cfg.blockDim = dim3(AttnSmem<D, BM>::kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = cluster;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, attn_bf16_kernel<D, BM>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return n > 0;
}

bool attention_cluster_fits(int D, int bm, int cluster) {
  if (D == 64)
    return bm == 32 ? cluster_fits_t<64, 32>(cluster)
                    : bm == 64 ? cluster_fits_t<64, 64>(cluster) : cluster_fits_t<64, 128>(cluster);
  return bm == 32 ? cluster_fits_t<128, 32>(cluster)
                  : bm == 64 ? cluster_fits_t<128, 64>(cluster) : cluster_fits_t<128, 128>(cluster);
}

cudaError_t launch_attention_bf16(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, int,
                                  bool pdl) {
  if (a.D == 64) return launch_bf16_d<64>(a, m, s, pdl);
  return launch_bf16_d<128>(a, m, s, pdl);
}

cudaError_t launch_attention_f32(const AttnArgs& a, cudaStream_t s, bool pdl) {
  static DeviceMemo limit;
  const int smem = (kF32Tile * (a.D + 1) + kF32Tile * a.D + kF32Rows * a.D) * 4;
  cudaError_t e = ensure_smem_limit((const void*)attn_f32_kernel, smem, limit);
  if (e != cudaSuccess) return e;
  const dim3 grid(a.B * a.Hkv * a.rb_count);
  return launch_ex(attn_f32_kernel, grid, dim3(256), smem, s, 1, pdl, a);
}

}  // namespace pf
