// pf_tree_prepare_device: ancestor-or-self bitmaps and depths of a batch of
// proposal trees in device memory (the proposal structure verified in one
// pass, Section 3.2).  One CTA of 128 threads per sequence: the tree's
// parent array is staged in shared memory, and thread j walks from node j to
// the root, setting one bit per node on the way (at most 127 steps).
#include <cuda_runtime.h>

#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

__global__ void __launch_bounds__(PF_MAX_NODES) tree_prepare_kernel(const TreeArgs a) {
  __shared__ int32_t par[PF_MAX_NODES];
  const int b = blockIdx.x, j = threadIdx.x;
  pdl_wait();  // the parent array may come from the preceding kernel or copy
  pdl_launch_dependents();
  const int node0 = a.cu_nodes[b];
  const int nn = a.cu_nodes[b + 1] - node0;
  if (node0 < 0 || nn < 1 || nn > a.max_nodes || node0 + nn > a.T) {
    if (j == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
    return;  // uniform over the CTA
  }
  const int p = j < nn ? a.parent[node0 + j] : 0;
  const bool bad = j < nn && (j == 0 ? p != -1 : (p < 0 || p >= j));
  if (j < nn) par[j] = p;
  const bool malformed = __syncthreads_or(bad) != 0;
  if (j >= nn) return;
  uint64_t m0 = 0, m1 = 0;
  int depth = -1;
  if (malformed) {
    if (j == 0) flag_error(a.err, PF_DEVERR_TREE);
    (j < 64 ? m0 : m1) = 1ull << (j & 63);
  } else {
    // every parent index is below its node, so the walk ends at the root
    int u = j;
    depth = 0;
    while (true) {
      (u < 64 ? m0 : m1) |= 1ull << (u & 63);
      if (u == 0) break;
      u = par[u];
      ++depth;
    }
  }
  reinterpret_cast<ulonglong2*>(a.mask)[node0 + j] = make_ulonglong2(m0, m1);
  if (a.depth) a.depth[node0 + j] = depth;
}

}  // namespace

cudaError_t launch_tree_prepare(const TreeArgs& a, cudaStream_t s, bool pdl) {
  return launch_ex(tree_prepare_kernel, dim3(a.B), dim3(PF_MAX_NODES), 0, s, 1, pdl, a);
}

}  // namespace pf
