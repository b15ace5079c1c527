// Pieces shared by the two bf16 tree-attention kernels: the TMA loader of
// one 64-token K/V tile (prefix cache, contiguous or paged, or the proposal's
// own K/V) and the merge of split-KV partials across a thread-block cluster.
#pragma once

#include <cooperative_groups.h>
#include <cuda_fp16.h>

#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

constexpr int kBN = 64;  // tokens per KV tile

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Page-table entries of prefix tile t of a paged cache (a 64-token tile is
// four 16-token pages), loaded together so that their latencies overlap:
// callers fetch them before they wait for the ring stage the tile goes to.
// -1 where the tile has no such page (past the prefix end), and for a
// contiguous cache or a proposal tile.
static_assert(kBN == 4 * PF_PAGE_SIZE, "a K/V tile spans four pages");

__device__ __forceinline__ int4 kv_tile_pages(const AttnArgs& a, int t, int n_ptiles, int b,
                                              int P) {
  int4 pg = make_int4(-1, -1, -1, -1);
  if (a.layout != PF_KV_CONTIGUOUS && t < n_ptiles) {
    const int tok0 = t * kBN;
    const int npages = min(4, (P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);  // >= 1
    const int32_t* pt = a.page_table + (size_t)b * a.pages_per_seq + tok0 / PF_PAGE_SIZE;
    pg.x = pt[0];
    if (npages > 1) pg.y = pt[1];
    if (npages > 2) pg.z = pt[2];
    if (npages > 3) pg.w = pt[3];
  }
  return pg;
}

// Page-table entries of the eight 16-token pages of 128-token prefix tile
// t (-1 past the prefix end, and for a contiguous cache or a proposal
// tile), loaded together.
struct Pages8 {
  int4 lo, hi;
};

__device__ __forceinline__ Pages8 no_pages8() {
  return Pages8{make_int4(-1, -1, -1, -1), make_int4(-1, -1, -1, -1)};
}

__device__ __forceinline__ Pages8 kv_tile_pages8(const AttnArgs& a, int t, int n_ptiles, int b,
                                                 int P) {
  Pages8 pg = no_pages8();
  if (a.layout != PF_KV_CONTIGUOUS && t < n_ptiles) {
    const int tok0 = t * 128;
    const int npages = min(128 / PF_PAGE_SIZE, (P - tok0 + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
    const int32_t* pt = a.page_table + (size_t)b * a.pages_per_seq + tok0 / PF_PAGE_SIZE;
    int v[8];
#pragma unroll
    for (int p = 0; p < 8; ++p) v[p] = p < npages ? pt[p] : -1;
    pg.lo = make_int4(v[0], v[1], v[2], v[3]);
    pg.hi = make_int4(v[4], v[5], v[6], v[7]);
  }
  return pg;
}

// TMA loads of one 64-token K/V tile into a ring stage (K then V, each two
// 64-column halves): from the prefix cache (contiguous: one 3-D box per
// half; paged: one 4-D box per 16-token page that holds prefix rows, pages
// from kv_tile_pages) or, past the prefix, from the proposal's own rows.
// Arms `bar` with the bytes it will bring.
template <int D>
__device__ __forceinline__ void issue_kv_tile(const AttnArgs& a, const CUtensorMap* tm_ck,
                                              const CUtensorMap* tm_cv, const CUtensorMap* tm_tk,
                                              const CUtensorMap* tm_tv, uint8_t* stage,
                                              uint32_t bar, int t, int n_ptiles, int b, int g,
                                              int node0, int P, int4 pg) {
  constexpr int kHalves = D / 64;
  constexpr int kTileBytes = kBN * D * 2;
  uint8_t* sk = stage;
  uint8_t* sv = stage + kTileBytes;
  if (t < n_ptiles) {
    const int tok0 = t * kBN;
    if (a.layout == PF_KV_CONTIGUOUS) {
      mbar_arrive_expect_tx(bar, 2 * kTileBytes);
#pragma unroll
      for (int h = 0; h < kHalves; ++h) {
        tma_load_3d(smem_u32(sk + h * kBN * 128), tm_ck, h * 64, tok0, b * a.Hkv + g, bar);
        tma_load_3d(smem_u32(sv + h * kBN * 128), tm_cv, h * 64, tok0, b * a.Hkv + g, bar);
      }
    } else {
      const int left = P - tok0;
      const int npages = min(kBN / PF_PAGE_SIZE, (left + PF_PAGE_SIZE - 1) / PF_PAGE_SIZE);
      mbar_arrive_expect_tx(bar, 2 * kHalves * npages * PF_PAGE_SIZE * 128);
      const int pages[4] = {pg.x, pg.y, pg.z, pg.w};
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        if (p >= npages) break;
#pragma unroll
        for (int h = 0; h < kHalves; ++h) {
          const int off = h * kBN * 128 + p * PF_PAGE_SIZE * 128;
          tma_load_4d(smem_u32(sk + off), tm_ck, h * 64, 0, g, pages[p], bar);
          tma_load_4d(smem_u32(sv + off), tm_cv, h * 64, 0, g, pages[p], bar);
        }
      }
    }
  } else {
    const int j = t - n_ptiles;
    mbar_arrive_expect_tx(bar, 2 * kTileBytes);
#pragma unroll
    for (int h = 0; h < kHalves; ++h) {
      tma_load_3d(smem_u32(sk + h * kBN * 128), tm_tk, h * 64, g, node0 + j * kBN, bar);
      tma_load_3d(smem_u32(sv + h * kBN * 128), tm_tv, h * 64, g, node0 + j * kBN, bar);
    }
  }
}

// Merge of split-KV partials.  Every CTA of the cluster has published, for
// its rows, the running maximum m (log2 domain), the sum l of exp2(s - m)
// and the unnormalised O (fp32, row pitch D + 4) in its shared memory.  After
// one cluster barrier, CTA `split` combines rows [split*per, (split+1)*per):
//   M = max_q m_q,  w_q = exp2(m_q - M),  out = sum_q w_q O_q / sum_q w_q l_q
// reading its peers' shared memory, one warp per row: lane q fetches peer
// q's (m, l), shuffles reduce them, and each lane owns D/32 output columns,
// issuing all of its peers' loads before accumulating.  A second barrier
// keeps every CTA's shared memory alive until its peers are done.
template <int D, int kThreads>
__device__ __forceinline__ void cluster_merge(const AttnArgs& a,
                                              cooperative_groups::cluster_group& cluster,
                                              float* sM, float* sL, float* sO, int rows, int split,
                                              int nsplit, int node_base, int g, int tid) {
  constexpr int kOStride = D + 4;
  constexpr int kMaxSplit = 16;
  constexpr int CPL = D / 32;  // output columns per lane
  static_assert(CPL == 2 || CPL == 4, "head_dim 64 or 128");
  cluster.sync();
  const int warp = tid >> 5, lane = tid & 31;
  const int per = (rows + nsplit - 1) / nsplit;
  const int lo = split * per, hi = min(rows, lo + per);
  __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out);
  for (int r = lo + warp; r < hi; r += kThreads / 32) {
    float mq = -INFINITY, lq = 0.f;
    if (lane < nsplit) {
      mq = cluster.map_shared_rank(sM, lane)[r];
      lq = cluster.map_shared_rank(sL, lane)[r];
    }
    float M = mq;
#pragma unroll
    for (int off = 16; off; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float Mu = M == -INFINITY ? 0.f : M;
    const float wq = lane < nsplit ? exp2f(mq - Mu) : 0.f;
    float L = wq * lq;
#pragma unroll
    for (int off = 16; off; off >>= 1) L += __shfl_xor_sync(0xffffffffu, L, off);
    float v[kMaxSplit][CPL];
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) {
      if (q < nsplit) {
        const float* src = cluster.map_shared_rank(sO, q) + r * kOStride + lane * CPL;
        if constexpr (CPL == 4) {
          const float4 t = *reinterpret_cast<const float4*>(src);
          v[q][0] = t.x;
          v[q][1] = t.y;
          v[q][2] = t.z;
          v[q][3] = t.w;
        } else {
          const float2 t = *reinterpret_cast<const float2*>(src);
          v[q][0] = t.x;
          v[q][1] = t.y;
        }
      }
    }
    float acc[CPL];
#pragma unroll
    for (int c = 0; c < CPL; ++c) acc[c] = 0.f;
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) {
      const float w = __shfl_sync(0xffffffffu, wq, q);
      if (q < nsplit) {
#pragma unroll
        for (int c = 0; c < CPL; ++c) acc[c] = fmaf(w, v[q][c], acc[c]);
      }
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    const int node = node_base + r / a.G;
    const int h = g * a.G + r % a.G;
    __nv_bfloat16* dst = out + ((size_t)node * a.Hq + h) * D + lane * CPL;
    if constexpr (CPL == 4) {
      uint2 pk;
      pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      *reinterpret_cast<uint2*>(dst) = pk;
    } else {
      *reinterpret_cast<uint32_t*>(dst) = pack_bf16(acc[0] * inv, acc[1] * inv);
    }
  }
  cluster.sync();
}

// ---- balanced batch mode: the work plan.  Group q = (b * Hkv + g) *
// rb_count + rb (sequence b, KV head g, row block rb) holds
//   tiles_q = ceil(P_b / W) + ceil(nn_b / W)
// K/V tiles of W tokens (the kernel's tile width) if its row block has nodes (rb * nb < nn_b), else none.  With
// the smallest T for which sum_q ceil(tiles_q / T) <= items, group q gets
// k_q = ceil(tiles_q / T) consecutive items (CTAs), which split its tiles
// evenly, so no CTA holds more than T tiles while every group is served in
// one wave.  Warp 0 of every attention CTA derives the plan from cu_nodes
// and prefix_len (all derive the same one); the combine kernel reads the
// per-group table the attention kernel leaves in the workspace.

struct PlanItem {
  int group;  // -1: nothing for this item
  int j, k;   // the item is the j-th of the group's k (k = 0: the group has no work)
  int first;  // the group's first item
};

// Tiles of group q of sequence (first node node0, nn nodes, prefix P);
// flags PF_DEVERR_BOUNDS and returns 0 for sizes outside the host bounds.
__device__ __forceinline__ int group_tiles(const AttnArgs& a, int q, int node0, int nn, int P,
                                           int tile_tokens) {
  const int rb = q % a.rb_count;
  if (node0 < 0 || nn < 1 || nn > a.max_nodes || node0 + nn > a.T || P < 0 || P > a.max_prefix) {
    flag_error(a.err, PF_DEVERR_BOUNDS);
    return 0;
  }
  if (rb * a.nb >= nn) return 0;
  return (P + tile_tokens - 1) / tile_tokens + (nn + tile_tokens - 1) / tile_tokens;
}

__device__ __forceinline__ int plan_tiles(const AttnArgs& a, int q, int tile_tokens) {
  const int b = q / (a.Hkv * a.rb_count);
  const int node0 = a.cu_nodes[b];
  return group_tiles(a, q, node0, a.cu_nodes[b + 1] - node0, a.prefix_len[b], tile_tokens);
}

// The plan's per-group table in the workspace, after the partials: (first
// partial slot, pieces, first node, rows) of every group, written by the
// attention kernel for the combine kernel.  With one slot per item, piece j
// of a group is slot first + j; with two (the continuous split), piece 0 is
// slot first and piece j > 0 is slot 2 * (first / 2 + j) (the first piece
// of each following item).
__device__ __forceinline__ int4* plan_table(const AttnArgs& a) {
  return reinterpret_cast<int4*>(reinterpret_cast<uint8_t*>(a.ws) +
                                 (size_t)a.items * a.slots * a.bm * (a.D + 8) * 2);
}

// One 64-bit arrival ticket per group after the plan table, for the kernels
// that merge a spread group's pieces themselves (the last piece to finish
// merges).  A ticket holds (call epoch << 24 | pieces arrived); a ticket
// whose epoch is not this call's counts as 0, so the workspace needs no
// initialisation, and the last piece resets the count to 0, so a captured
// launch replayed with the same epoch starts from 0 again.
__device__ __forceinline__ unsigned long long* group_tickets(const AttnArgs& a) {
  return reinterpret_cast<unsigned long long*>(plan_table(a) + kPlanMaxGroups);
}

// One thread per piece, after every write of the piece's partial is ordered
// before it (writers' __threadfence + a CTA barrier): true for the piece
// that completes the group.  Each failed compare-and-swap means another
// piece's arrival succeeded, so the loop ends after at most k rounds; it is
// bounded all the same.
__device__ __forceinline__ bool ticket_arrive_last(unsigned long long* ticket,
                                                   unsigned long long epoch, int k, int32_t* err) {
  constexpr unsigned long long kCount = (1ull << 24) - 1;
  unsigned long long old = atomicAdd(ticket, 0ull);
  for (int round = 0; round < 4096; ++round) {
    const unsigned long long cnt = (old >> 24) == epoch ? (old & kCount) : 0ull;
    const bool last = (int)cnt + 1 == k;
    const unsigned long long want = (epoch << 24) | (last ? 0ull : cnt + 1);
    const unsigned long long seen = atomicCAS(ticket, old, want);
    if (seen == old) {
      __threadfence();  // the other pieces' partials are visible to this CTA
      return last;
    }
    old = seen;
  }
  flag_error(err, PF_DEVERR_TIMEOUT);
  return false;
}

// Merge of group pieces' partials from global memory (the format of
// attn_tc_kernel's staged rows: fp16 O / l, then the log2-sum-exp as a float
// in the row's pad, pitch D + 8 halves): row r, output columns c8*8 ..
// c8*8+7, pieces in slots first .. first + k - 1 of bm rows each, read past
// L1 (other CTAs wrote them during this launch).  Batches of 8 pieces, all
// loads of a batch in flight together, folded into a running maximum.
//   out = sum_j 2^(lse_j - M) (O/l)_j / sum_j 2^(lse_j - M),  M = max_j lse_j
template <int D>
__device__ __forceinline__ void merge_pieces_row(const AttnArgs& a, int first, int k, int r,
                                                 int c8, __nv_bfloat16* dst) {
  constexpr int kPitch = D + 8, kBatch = 8;
  const __half* base = reinterpret_cast<const __half*>(a.ws) + (size_t)r * kPitch;
  const size_t slot_stride = (size_t)a.bm * kPitch;
  float M = -INFINITY, W = 0.f;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int j0 = 0; j0 < k; j0 += kBatch) {
    float ls[kBatch];
    uint4 v[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      ls[u] = -INFINITY;
      if (j0 + u < k) {
        const __half* row = base + (size_t)(first + j0 + u) * slot_stride;
        ls[u] = __ldcg(reinterpret_cast<const float*>(row + D));
        v[u] = __ldcg(reinterpret_cast<const uint4*>(row + c8 * 8));
      }
    }
    float Mb = M;
#pragma unroll
    for (int u = 0; u < kBatch; ++u) Mb = fmaxf(Mb, ls[u]);
    if (Mb == -INFINITY) continue;  // nothing reached this row yet
    const float sc = M == -INFINITY ? 0.f : ex2_approx(M - Mb);
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
  uint4 pk;
  pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
  pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
  pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
  pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
  *reinterpret_cast<uint4*>(dst + c8 * 8) = pk;
}

// Warp-collective (all 32 lanes, warp-uniform arguments): the plan entry
// of item `item`, and in *grp that of group `group` (j = 0) if group >= 0.
static __device__ __noinline__ PlanItem balanced_plan(const AttnArgs& a, int item, int group,
                                                      PlanItem* grp, int tile_tokens = kBN) {
  const int lane = threadIdx.x & 31;
  const int n_groups = a.B * a.Hkv * a.rb_count;  // <= kPlanMaxGroups and <= items (host)
  constexpr int kPer = kPlanMaxGroups / 32;
  const int n_chunks = (n_groups + 31) / 32;
  int t[kPer];
  int U = 0, n_active = 0, t_max = 0;
  // all groups' sizes loaded together (see continuous_plan)
  int n0[kPer], n1[kPer], pl[kPer];
#pragma unroll
  for (int s = 0; s < kPer; ++s) {
    const int q = lane + 32 * s;
    const int b = q / (a.rb_count * a.Hkv);
    n0[s] = n1[s] = pl[s] = 0;
    if (q < n_groups) {
      n0[s] = __ldg(&a.cu_nodes[b]);
      n1[s] = __ldg(&a.cu_nodes[b + 1]);
      pl[s] = __ldg(&a.prefix_len[b]);
    }
  }
#pragma unroll
  for (int s = 0; s < kPer; ++s) {
    const int q = lane + 32 * s;
    t[s] = q < n_groups ? group_tiles(a, q, n0[s], n1[s] - n0[s], pl[s], tile_tokens) : 0;
    U += t[s];
    n_active += t[s] > 0 ? 1 : 0;
    t_max = max(t_max, t[s]);
  }
  U = __reduce_add_sync(0xffffffffu, U);
  n_active = __reduce_add_sync(0xffffffffu, n_active);
  t_max = __reduce_max_sync(0xffffffffu, t_max);
  PlanItem r = {-1, 0, 0, 0};
  if (group >= 0) *grp = PlanItem{group, 0, 0, 0};
  if (U == 0) return r;
  // T in [lo, hi]: count(T) >= U / T exceeds items below lo, and
  // count(T) <= U / T + n_active fits at hi (as does count(t_max) = n_active).
  int hi = t_max;
  if (a.items > n_active) hi = min(hi, (U + (a.items - n_active) - 1) / (a.items - n_active));
  int lo = min(hi, max(1, (U + a.items - 1) / a.items));
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    int c = 0;
#pragma unroll
    for (int s = 0; s < kPer; ++s)
      if (s < n_chunks) c += (t[s] + mid - 1) / mid;
    c = __reduce_add_sync(0xffffffffu, c);
    if (c <= a.items) hi = mid;
    else lo = mid + 1;
  }
  const int T = lo;
  int base = 0;
#pragma unroll
  for (int s = 0; s < kPer; ++s) {
    if (s >= n_chunks) break;
    const int q = lane + 32 * s;
    const int k = (t[s] + T - 1) / T;
    int incl = k;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    const int first = base + incl - k;
    const unsigned mi = __ballot_sync(0xffffffffu, q < n_groups && k > 0 && item >= first &&
                                                       item < first + k);
    if (mi) {
      const int src = __ffs(mi) - 1;
      r.group = __shfl_sync(0xffffffffu, q, src);
      r.k = __shfl_sync(0xffffffffu, k, src);
      r.first = __shfl_sync(0xffffffffu, first, src);
      r.j = item - r.first;
    }
    if (group >= 0 && group / 32 == s) {
      const int src = group % 32;
      grp->k = __shfl_sync(0xffffffffu, k, src);
      grp->first = __shfl_sync(0xffffffffu, first, src);
    }
    base += __shfl_sync(0xffffffffu, incl, 31);
  }
  return r;
}

// ---- continuous split (the pair kernel and attn_sk_kernel): the groups'
// tiles of `tile_tokens` tokens are laid end to end and cut into a.items
// equal ranges.  A range covers pieces of one or more groups (parts); only
// its first and last part can be pieces of a longer group, so each item
// has two partial slots (2 * item for its first part, 2 * item + 1 for its
// last).  A part is packed in 64 bits: group (9 bits), first and end tile
// within the group (16 bits each), whole-group flag, slot (up to 2^22).
struct Part {
  int q, t0, t1, whole, slot;
};

__device__ __forceinline__ unsigned long long pack_part(const Part& p) {
  return (unsigned long long)p.q | ((unsigned long long)p.t0 << 9) |
         ((unsigned long long)p.t1 << 25) | ((unsigned long long)p.whole << 41) |
         ((unsigned long long)p.slot << 42);
}
__device__ __forceinline__ Part unpack_part(unsigned long long v) {
  return Part{(int)(v & 0x1FF), (int)((v >> 9) & 0xFFFF), (int)((v >> 25) & 0xFFFF),
              (int)((v >> 41) & 1), (int)(v >> 42)};
}

// Warp 0 of every CTA (all 32 lanes, the same result in every CTA): group
// q (8 per lane, q = 32 s + lane) holds t_q tiles starting at position
// start_q of the concatenation; item i takes positions [floor(U i / items),
// floor(U (i+1) / items)).  Writes this item's parts in group order to
// `parts` (at most max_parts) and returns their count; with write_table,
// items with index = q (mod items) also write group q's plan-table entry
// (first partial slot, pieces, first node, rows) for the combine kernel.
// Groups: <= kPlanMaxGroups (host); tiles per group < 2^16, so the total U
// < 2^24 and U * items < 2^32: the arithmetic is 32-bit (64-bit divisions
// here took several microseconds per launch).
template <int kTile>
static __device__ __noinline__ int continuous_plan(const AttnArgs& a, int item, bool write_table,
                                                   unsigned long long* parts) {
  constexpr int tile_tokens = kTile;
  const int lane = threadIdx.x & 31;
  const int n_groups = a.B * a.Hkv * a.rb_count;
  constexpr int kPer = kPlanMaxGroups / 32;
  int t[kPer], start[kPer];
  unsigned U = 0;
  {
    // every group's sizes first, all loads in flight together (issued
    // between the scans, or behind plan_tiles' error atomic, they took one
    // round trip per chunk: ~8 us); cu_nodes and prefix_len are read-only
    // for the kernel's lifetime
    int n0[kPer], n1[kPer], pl[kPer];
#pragma unroll
    for (int s = 0; s < kPer; ++s) {
      const int q = lane + 32 * s;
      const int b = q / (a.rb_count * a.Hkv);
      n0[s] = n1[s] = pl[s] = 0;
      if (q < n_groups) {
        n0[s] = __ldg(&a.cu_nodes[b]);
        n1[s] = __ldg(&a.cu_nodes[b + 1]);
        pl[s] = __ldg(&a.prefix_len[b]);
      }
    }
#pragma unroll
    for (int s = 0; s < kPer; ++s) {
      const int q = lane + 32 * s;
      t[s] = q < n_groups ? group_tiles(a, q, n0[s], n1[s] - n0[s], pl[s], tile_tokens) : 0;
    }
    int base = 0;
#pragma unroll
    for (int s = 0; s < kPer; ++s) {
      int incl = t[s];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      start[s] = base + incl - t[s];
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    U = base;
  }
  if (U == 0) return 0;
  const unsigned items = (unsigned)a.items;
  const unsigned R0 = U * (unsigned)item / items, R1 = U * (unsigned)(item + 1) / items;
  auto item_of = [&](unsigned x) { return (int)(((x + 1) * items - 1) / U); };
  auto range_start = [&](unsigned i) { return U * i / items; };
  int n = 0;
#pragma unroll
  for (int s = 0; s < kPer; ++s) {
    const int q = lane + 32 * s;
    const unsigned s0 = (unsigned)start[s], s1 = (unsigned)(start[s] + t[s]);
    const bool mine = t[s] > 0 && s0 < R1 && s1 > R0;
    const unsigned m = __ballot_sync(0xffffffffu, mine);
    if (mine) {
      const int i0 = item_of(s0), i1 = item_of(s1 - 1);
      Part p;
      p.q = q;
      p.t0 = (int)(max(R0, s0) - s0);
      p.t1 = (int)(min(R1, s1) - s0);  // unsigned max / min: every value >= 0
      p.whole = i0 == i1;
      p.slot = 2 * item + (R0 >= s0 ? 0 : 1);  // this item's first part, or its last
      parts[n + __popc(m & ((1u << lane) - 1u))] = pack_part(p);
    }
    n += __popc(m);
    if (write_table && q < n_groups && q % a.items == item) {
      int4 e = make_int4(0, 0, 0, 0);
      if (t[s] > 0) {
        const int i0 = item_of(s0), i1 = item_of(s1 - 1);
        const int bq = q / (a.rb_count * a.Hkv), nfq = (q % a.rb_count) * a.nb;
        const int n0 = a.cu_nodes[bq], nnq = a.cu_nodes[bq + 1] - n0;
        e = make_int4(2 * i0 + (range_start(i0) < s0 ? 1 : 0), i1 - i0 + 1, n0 + nfq,
                      max(0, min(a.nb, nnq - nfq)) * a.G);
      }
      plan_table(a)[q] = e;
    }
  }
  return n;
}

// A part's group decoded for one CTA holding `cta_nodes` of the group's
// nodes from the group's (c * cta_nodes)-th on: sequence, KV head, first
// node and rows (0 when the CTA holds none).
struct PartGeom {
  int b, g, node0, nn, P, nfirst, rows, n_ptiles;
};

__device__ __forceinline__ PartGeom part_geom(const AttnArgs& a, int q, int cta_nodes, int c,
                                              int tile_tokens) {
  PartGeom r;
  const int rb = q % a.rb_count;
  r.g = (q / a.rb_count) % a.Hkv;
  r.b = q / (a.rb_count * a.Hkv);
  r.node0 = a.cu_nodes[r.b];
  r.nn = a.cu_nodes[r.b + 1] - r.node0;
  r.P = a.prefix_len[r.b];  // the plan checked these (plan_tiles)
  r.nfirst = rb * a.nb + c * cta_nodes;
  r.rows = max(0, min(cta_nodes, r.nn - r.nfirst)) * a.G;
  r.n_ptiles = (r.P + tile_tokens - 1) / tile_tokens;
  return r;
}

// Local half of the split-KV merge: this CTA (rank `split`) owns rows
// [split*per, split*per + cnt); peer s delivered, for local row i, its
// normalised partial (O / l, fp16) followed by its log2-sum-exp (a float in
// the row's pad) at inbox slot s*per + i (pitch kPitch halves).
//   M = max_s lse_s,  w_s = 2^(lse_s - M),  out = sum_s w_s (O/l)_s / sum_s w_s
// One thread per (row, 8 output columns); all loads are issued before use.
// kMaxSplit bounds the unrolled loops: the predicated slots of a wider
// instance than the cluster needs still issue (a 16-way instance took ~4 us
// for 2-CTA clusters), so inbox_merge picks the narrowest that holds nsplit.
template <int D, int kThreads, int kPitch, int kMaxSplit>
__device__ __forceinline__ void inbox_merge_n(const AttnArgs& a, const __half* inbox, int rows,
                                              int split, int per, int nsplit, int node_base, int g,
                                              int tid) {
  constexpr int C8 = D / 8;
  const int cnt = min(per, rows - split * per);
  __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out);
  for (int it = tid; it < cnt * C8; it += kThreads) {
    const int i = it / C8, c8 = it - (it / C8) * C8;
    float ls[kMaxSplit];
    uint4 v[kMaxSplit];
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) {
      if (q < nsplit) {
        const __half* slot = inbox + (q * per + i) * kPitch;
        ls[q] = *reinterpret_cast<const float*>(slot + D);
        v[q] = *reinterpret_cast<const uint4*>(slot + c8 * 8);
      } else {
        ls[q] = -INFINITY;
      }
    }
    float M = -INFINITY;
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) M = fmaxf(M, ls[q]);
    const float Mu = M == -INFINITY ? 0.f : M;
    float W = 0.f, acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int q = 0; q < kMaxSplit; ++q) {
      if (q < nsplit) {
        const float w = ex2_approx(ls[q] - Mu);  // -inf -> 0
        W += w;
        const __half2* h2 = reinterpret_cast<const __half2*>(&v[q]);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const float2 f = __half22float2(h2[c]);
          acc[2 * c] = fmaf(w, f.x, acc[2 * c]);
          acc[2 * c + 1] = fmaf(w, f.y, acc[2 * c + 1]);
        }
      }
    }
    const float inv = W > 0.f ? __fdividef(1.f, W) : 0.f;
    const int r = split * per + i;
    const int node = node_base + r / a.G;
    const int h = g * a.G + r % a.G;
    uint4 pk;
    pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
    pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
    pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
    pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
    *reinterpret_cast<uint4*>(out + ((size_t)node * a.Hq + h) * D + c8 * 8) = pk;
  }
}

// The same merge for k <= kMaxK pieces held in shared memory, latency-lean:
// a unit is (row, a quarter of its 8-column chunks); the unit's k
// log-sum-exps are read once and turned into normalised weights, then its
// four chunks' loads of every piece are all issued before any is used (the
// one-CTA-per-SM kernels run 6 warps, too few to hide one load-use chain
// per output chunk).  Piece j of local row i is at base + j * slot_stride +
// i * row_pitch (bytes): fp16 O / l, then the float log2-sum-exp at byte
// 2 * D.  Local row i is output row row0 + i of the group.
template <int D, int kMaxK>
__device__ __forceinline__ void merge_rows_smem(const AttnArgs& a, const uint8_t* base,
                                                int row_pitch, int slot_stride, int k, int nrows,
                                                int row0, int node_base, int g, int tid,
                                                int nthreads) {
  constexpr int C8 = D / 8, kQ = 4, kPer = C8 / kQ;  // 4 chunks per unit
  __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out);
  for (int u = tid; u < nrows * kQ; u += nthreads) {
    const int i = u / kQ, q = u % kQ;
    const uint8_t* row = base + i * row_pitch;
    float w[kMaxK];
    float M = -INFINITY;
#pragma unroll
    for (int j = 0; j < kMaxK; ++j) {
      w[j] = j < k ? *reinterpret_cast<const float*>(row + j * slot_stride + 2 * D) : -INFINITY;
      M = fmaxf(M, w[j]);
    }
    const float Mu = M == -INFINITY ? 0.f : M;
    float W = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxK; ++j) {
      w[j] = w[j] == -INFINITY ? 0.f : ex2_approx(w[j] - Mu);  // absent or empty: 0
      W += w[j];
    }
    const float inv = W > 0.f ? __fdividef(1.f, W) : 0.f;
    uint4 v[kPer][kMaxK];
#pragma unroll
    for (int c = 0; c < kPer; ++c)
#pragma unroll
      for (int j = 0; j < kMaxK; ++j)
        if (w[j] != 0.f)
          v[c][j] = *reinterpret_cast<const uint4*>(row + j * slot_stride + (q * kPer + c) * 16);
    const int r = row0 + i;
    const int node = node_base + r / a.G;
    const int h = g * a.G + r % a.G;
    uint4* dst = reinterpret_cast<uint4*>(out + ((size_t)node * a.Hq + h) * D) + q * kPer;
#pragma unroll
    for (int c = 0; c < kPer; ++c) {
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int j = 0; j < kMaxK; ++j) {
        if (w[j] == 0.f) continue;  // its O may hold anything (0 * NaN)
        const __half2* h2 = reinterpret_cast<const __half2*>(&v[c][j]);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __half22float2(h2[e]);
          acc[2 * e] = fmaf(w[j], f.x, acc[2 * e]);
          acc[2 * e + 1] = fmaf(w[j], f.y, acc[2 * e + 1]);
        }
      }
      uint4 pk;
      pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      pk.z = pack_bf16(acc[4] * inv, acc[5] * inv);
      pk.w = pack_bf16(acc[6] * inv, acc[7] * inv);
      dst[c] = pk;
    }
  }
}

template <int D, int kThreads, int kPitch>
__device__ __forceinline__ void inbox_merge(const AttnArgs& a, const __half* inbox, int rows,
                                            int split, int per, int nsplit, int node_base, int g,
                                            int tid) {
  // up to 4 peers: the latency-lean unit merge; wider clusters have few rows
  // per CTA and keep one thread per (row, chunk)
  const int cnt = max(0, min(per, rows - split * per));
  const uint8_t* base = reinterpret_cast<const uint8_t*>(inbox);
  if (nsplit <= 2)
    merge_rows_smem<D, 2>(a, base, kPitch * 2, per * kPitch * 2, nsplit, cnt, split * per,
                          node_base, g, tid, kThreads);
  else if (nsplit <= 4)
    merge_rows_smem<D, 4>(a, base, kPitch * 2, per * kPitch * 2, nsplit, cnt, split * per,
                          node_base, g, tid, kThreads);
  else if (nsplit <= 8)
    inbox_merge_n<D, kThreads, kPitch, 8>(a, inbox, rows, split, per, nsplit, node_base, g, tid);
  else
    inbox_merge_n<D, kThreads, kPitch, 16>(a, inbox, rows, split, per, nsplit, node_base, g, tid);
}

}  // namespace pf
