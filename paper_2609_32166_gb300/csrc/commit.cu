// Carry-forward of the accepted rows (Section 1; Section 3.4; Section 4's
// contiguous cache): for every layer, K and V, sequence b and path slot
// k <= accept_len[b], the row of proposal node path[b][k] moves to cache
// position prefix_len[b] + k.  One launch covers all layers; each thread
// moves one 16-byte chunk, so a 256-byte row is one fully coalesced group of
// 16 threads.  accept_len and path are read on the device, straight from the
// LM-head kernel's outputs, so the host never waits for them.
#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

// grid.y = (layer, K/V, sequence); grid.x * 256 threads cover the
// (path slot, KV head, 16-byte chunk) triples of one row set.
__global__ void __launch_bounds__(256) kv_commit_kernel(const CommitArgs a) {
  pdl_wait();
  const int chunks = a.row_bytes >> 4;
  const int y = blockIdx.y;
  const int b = y % a.B;
  const int kv = (y / a.B) & 1;
  const int l = y / (2 * a.B);
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  const int per_slot = a.Hkv * chunks;
  const int k = u / per_slot;
  if (y == 0 && blockIdx.x == 0)
    for (int i = threadIdx.x; i < a.B; i += blockDim.x)
      a.new_len[i] = a.prefix_len[i] + a.accept_len[i] + 1;
  if (k >= a.max_nodes || k > a.accept_len[b]) return;
  const int g = (u - k * per_slot) / chunks;
  const int c = u - k * per_slot - g * chunks;
  const int node0 = a.cu_nodes[b];
  const int nn = a.cu_nodes[b + 1] - node0;
  const int node = a.path[(size_t)b * a.max_nodes + k];
  if (node0 < 0 || node0 + nn > a.T || node < 0 || node >= nn) {
    flag_error(a.err, PF_DEVERR_BOUNDS);
    return;
  }
  const int pos = a.prefix_len[b] + k;
  long long dst_row;
  if (a.layout == PF_KV_CONTIGUOUS) {
    if (pos >= a.max_seq) {
      flag_error(a.err, PF_DEVERR_CAPACITY);
      return;
    }
    dst_row = ((long long)b * a.Hkv + g) * a.max_seq + pos;
  } else {
    const int pi = pos / PF_PAGE_SIZE;
    const int page = pi < a.pages_per_seq ? a.page_table[(size_t)b * a.pages_per_seq + pi] : -1;
    if (page < 0 || page >= a.num_pages) {
      flag_error(a.err, PF_DEVERR_CAPACITY);
      return;
    }
    dst_row = ((long long)page * a.Hkv + g) * PF_PAGE_SIZE + pos % PF_PAGE_SIZE;
  }
  const char* src = (kv ? a.tree_v : a.tree_k) + l * a.tree_layer_bytes +
                    ((long long)(node0 + node) * a.Hkv + g) * a.row_bytes + c * 16;
  char* dst = (kv ? a.cache_v : a.cache_k) + l * a.cache_layer_bytes + dst_row * a.row_bytes +
              c * 16;
  *reinterpret_cast<uint4*>(dst) = __ldg(reinterpret_cast<const uint4*>(src));
}

}  // namespace

cudaError_t launch_kv_commit(const CommitArgs& a, cudaStream_t s, int num_sms, bool pdl) {
  (void)num_sms;
  const int per_seq = a.max_nodes * a.Hkv * (a.row_bytes / 16);
  const dim3 grid((per_seq + 255) / 256, 2 * a.L * a.B);
  return launch_ex(kv_commit_kernel, grid, dim3(256), 0, s, 1, pdl, a);
}

}  // namespace pf
