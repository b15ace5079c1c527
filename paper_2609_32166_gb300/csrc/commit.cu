// Carry-forward of the accepted rows (Section 1; Section 3.4; Section 4's
// contiguous cache): for every layer, K and V, sequence b and path slot
// k <= accept_len[b], the row of proposal node path[b][k] moves to cache
// position prefix_len[b] + k.  One launch covers all layers.  accept_len and
// path are read on the device, straight from the LM-head kernel's outputs,
// so the host never waits for them.
//
// The step's moves are a few MB spread over 2 * L row sets per sequence, so
// the kernel is bound by its chain of dependent loads, not by bandwidth.  A
// CTA first resolves every path slot of its sequence once -- source row,
// destination row (through the page table for a paged cache) -- into shared
// memory (two round trips, all slots in parallel), then streams 16-byte
// chunks of its share of the row sets with several loads in flight per
// thread before their stores.
#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

constexpr int kCommitThreads = 256;
constexpr int kCommitUnroll = 4;

// grid = (CTAs per sequence, B).  CTA (x, b) moves the row sets
// s = x, x + gridDim.x, ... of the 2 * L (layer, K/V) sets of sequence b.
__global__ void __launch_bounds__(kCommitThreads) kv_commit_kernel(const CommitArgs a) {
  __shared__ long long s_src[PF_MAX_NODES];  // source row of head 0, or -1
  __shared__ long long s_dst[PF_MAX_NODES];  // destination row of head 0, or -1
  __shared__ int s_rows;
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.y;
  const int t = threadIdx.x;
  // ---- prologue: every path slot of sequence b, all loads in flight together
  if (t < a.max_nodes) {
    const int acc = a.accept_len[b];
    const int P = a.prefix_len[b];
    const int node0 = a.cu_nodes[b];
    const int nn = a.cu_nodes[b + 1] - node0;
    const int node = a.path[(size_t)b * a.max_nodes + t];
    if (t == 0) {
      if (blockIdx.x == 0) a.new_len[b] = P + acc + 1;
      s_rows = max(0, min(acc + 1, a.max_nodes));
    }
    long long src = -1, dst = -1;
    if (t <= acc) {
      if (node0 < 0 || node0 + nn > a.T || node < 0 || node >= nn) {
        if (blockIdx.x == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
      } else {
        const int pos = P + t;
        if (a.layout == PF_KV_CONTIGUOUS) {
          if (pos < a.max_seq)
            dst = (long long)b * a.Hkv * a.max_seq + pos;
        } else {
          const int pi = pos / PF_PAGE_SIZE;
          const int page =
              pi < a.pages_per_seq ? a.page_table[(size_t)b * a.pages_per_seq + pi] : -1;
          if (page >= 0 && page < a.num_pages)
            dst = (long long)page * a.Hkv * PF_PAGE_SIZE + pos % PF_PAGE_SIZE;
        }
        if (dst < 0) {
          if (blockIdx.x == 0) flag_error(a.err, PF_DEVERR_CAPACITY);
        } else {
          src = (long long)(node0 + node) * a.Hkv;
        }
      }
    }
    s_src[t] = src;
    s_dst[t] = dst;
  }
  __syncthreads();
  // ---- stream the chunks: item = (row set, path slot, KV head, chunk)
  const int chunks = a.row_bytes >> 4;
  const int per_slot = a.Hkv * chunks;
  const int per_set = s_rows * per_slot;
  const int sets = (2 * a.L - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
  const int total = sets * per_set;
  // consecutive KV heads of a row: one row apart in the proposal scratch,
  // a sequence's (contiguous) or a page's (paged) rows apart in the cache
  const long long dst_head = a.layout == PF_KV_CONTIGUOUS ? a.max_seq : PF_PAGE_SIZE;
  for (int base = t; base < total; base += kCommitThreads * kCommitUnroll) {
    uint4 v[kCommitUnroll];
    char* dst[kCommitUnroll];
#pragma unroll
    for (int u = 0; u < kCommitUnroll; ++u) {
      const int i = base + u * kCommitThreads;
      dst[u] = nullptr;
      if (i < total) {
        const int si = i / per_set;
        const int r = i - si * per_set;
        const int k = r / per_slot;
        const int g = (r - k * per_slot) / chunks;
        const int c = r - k * per_slot - g * chunks;
        const long long sr = s_src[k], dr = s_dst[k];
        if (sr >= 0) {
          const int set = (int)blockIdx.x + si * (int)gridDim.x;
          const int l = set >> 1, kv = set & 1;
          const char* src = (kv ? a.tree_v : a.tree_k) + l * a.tree_layer_bytes +
                            (sr + g) * a.row_bytes + c * 16;
          dst[u] = (kv ? a.cache_v : a.cache_k) + l * a.cache_layer_bytes +
                   (dr + g * dst_head) * a.row_bytes + c * 16;
          v[u] = __ldg(reinterpret_cast<const uint4*>(src));
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kCommitUnroll; ++u)
      if (dst[u]) *reinterpret_cast<uint4*>(dst[u]) = v[u];
  }
}

}  // namespace

cudaError_t launch_kv_commit(const CommitArgs& a, cudaStream_t s, int num_sms, bool pdl) {
  // about two CTAs per SM over the batch, at most one per row set
  const int per_seq = std::max(1, std::min(2 * a.L, (2 * std::max(num_sms, 1) + a.B - 1) / a.B));
  const dim3 grid(per_seq, a.B);
  return launch_ex(kv_commit_kernel, grid, dim3(kCommitThreads), 0, s, 1, pdl, a);
}

}  // namespace pf
