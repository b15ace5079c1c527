// Prompt-prefix KV carryover (Section 3.4): the length p of the longest
// identical prefix of the cached prompt's token keys and the new prompt's,
// written on the device together with the cache's new length, so that the
// kernels resuming at position p read it without a host round trip.
//
// One CTA of 1024 threads walks both arrays in blocks of 4096 keys (one
// 16-byte load of each array per thread when both are 16-byte aligned);
// a block's first mismatch is a CTA-wide minimum (warp reductions, then one
// warp over the 32 warp minima) and the walk stops at the first block that
// has one.  A prompt of a few thousand tokens is one or two blocks, so the
// call is bound by launch latency; more CTAs would only add a cross-CTA
// reduction to it.
#include <climits>

#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

constexpr int kPrefixThreads = 1024;

__global__ void __launch_bounds__(kPrefixThreads) prefix_match_kernel(const PrefixArgs a) {
  pdl_wait();
  __shared__ int s_min[kPrefixThreads / 32];
  __shared__ int s_block_min;
  const int n = min(a.n_prev, a.n_next);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int p = n;
  for (int base = 0; base < n; base += 4 * kPrefixThreads) {
    const int j = base + 4 * (int)threadIdx.x;
    int first = INT_MAX;
    if (a.vec && j + 3 < n) {
      const int4 x = __ldg(reinterpret_cast<const int4*>(a.prev + j));
      const int4 y = __ldg(reinterpret_cast<const int4*>(a.next + j));
      if (x.w != y.w) first = j + 3;
      if (x.z != y.z) first = j + 2;
      if (x.y != y.y) first = j + 1;
      if (x.x != y.x) first = j;
    } else {
#pragma unroll
      for (int k = 3; k >= 0; --k)
        if (j + k < n && __ldg(a.prev + j + k) != __ldg(a.next + j + k)) first = j + k;
    }
    first = __reduce_min_sync(0xffffffffu, first);
    if (lane == 0) s_min[warp] = first;
    __syncthreads();
    if (warp == 0) {
      const int m = __reduce_min_sync(0xffffffffu, s_min[lane]);
      if (lane == 0) s_block_min = m;
    }
    __syncthreads();
    const int m = s_block_min;
    __syncthreads();  // s_min and s_block_min are rewritten by the next block
    if (m != INT_MAX) {
      p = m;
      break;  // uniform: every thread read the same m
    }
  }
  if (threadIdx.x == 0) {
    a.lcp[0] = p;
    if (a.cache_len) a.cache_len[0] = p;
  }
  pdl_launch_dependents();
}

static_assert(kPrefixThreads / 32 == 32, "one warp reduces the warp minima");

}  // namespace

cudaError_t launch_prefix_match(const PrefixArgs& a, cudaStream_t s, bool pdl) {
  return launch_ex(prefix_match_kernel, dim3(1), dim3(kPrefixThreads), 0, s, 1, pdl, a);
}

}  // namespace pf
