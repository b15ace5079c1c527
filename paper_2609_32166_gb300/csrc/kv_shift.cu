// Rolling-image KV carryover (Section 3.4): move a block of cached rows of
// one sequence to a new span, re-rotating keys from position p to
// p + (dst - src) and copying values, for all layers and KV heads in one
// launch.  HBM-bound: every row is read once and written once.
//
// Disjoint spans run as one flat grid-stride range of independent items.
// Overlapping spans are cut into disjoint segments (below); only a shift so
// small that this would take many launches uses the ordered mode, where one
// CTA per (layer, KV head) stages a block of rows, synchronises, writes it,
// and walks the blocks in the order that keeps the in-place move safe
// (ascending for a move to lower positions, descending for higher).  An
// item is one 16-byte chunk of a row's first half and the matching chunk of
// the second half, i.e. whole rotary pairs (x_i, x_{i+D/2}), of K and V.
#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

constexpr int kShiftThreads = 256;
constexpr int kItemsPerThread = 4;

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;  // elements per 16-byte chunk
  static __device__ __forceinline__ float get(const uint4& v, int e) {
    const uint32_t w = (&v.x)[e >> 1];
    return __uint_as_float((e & 1) ? (w & 0xFFFF0000u) : (w << 16));
  }
  static __device__ __forceinline__ void set_pair(uint4& v, int e2, float lo, float hi) {
    (&v.x)[e2] = pack_bf16(lo, hi);
  }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ float get(const uint4& v, int e) {
    return __uint_as_float((&v.x)[e]);
  }
  static __device__ __forceinline__ void set_pair(uint4& v, int e2, float lo, float hi) {
    (&v.x)[2 * e2] = __float_as_uint(lo);
    (&v.x)[2 * e2 + 1] = __float_as_uint(hi);
  }
};

// Byte offset of (position, head) inside one layer; -1 if the page table
// points outside the pool.
__device__ __forceinline__ long long row_offset(const ShiftArgs& a, int g, int pos) {
  if (a.layout == PF_KV_CONTIGUOUS)
    return (((long long)a.seq * a.Hkv + g) * a.max_seq + pos) * a.row_bytes;
  const int pi = pos / PF_PAGE_SIZE;
  const int page = pi < a.pages_per_seq ? a.page_table[(size_t)a.seq * a.pages_per_seq + pi] : -1;
  if (page < 0 || page >= a.num_pages) return -1;
  return (((long long)page * a.Hkv + g) * PF_PAGE_SIZE + pos % PF_PAGE_SIZE) * a.row_bytes;
}

// K halves (k1, k2) of one 16-byte chunk pair rotated by the table, then K
// and V stored at the destination row.
template <typename T>
__device__ __forceinline__ void rotate_store(const float2* s_cs, int chunk, const uint4& k1,
                                             const uint4& k2, const uint4& v1, const uint4& v2,
                                             char* kdst, char* vdst, int half_bytes) {
  using V = Vec<T>;
  uint4 o1 = k1, o2 = k2;
#pragma unroll
  for (int e = 0; e < V::N; e += 2) {
    const int i0 = chunk * V::N + e;  // frequency index of this pair
    const float2 cs0 = s_cs[i0], cs1 = s_cs[i0 + 1];
    const float x0 = V::get(k1, e), y0 = V::get(k2, e);
    const float x1 = V::get(k1, e + 1), y1 = V::get(k2, e + 1);
    V::set_pair(o1, e >> 1, x0 * cs0.x - y0 * cs0.y, x1 * cs1.x - y1 * cs1.y);
    V::set_pair(o2, e >> 1, x0 * cs0.y + y0 * cs0.x, x1 * cs1.y + y1 * cs1.x);
  }
  *reinterpret_cast<uint4*>(kdst + chunk * 16) = o1;
  *reinterpret_cast<uint4*>(kdst + half_bytes + chunk * 16) = o2;
  *reinterpret_cast<uint4*>(vdst + chunk * 16) = v1;
  *reinterpret_cast<uint4*>(vdst + half_bytes + chunk * 16) = v2;
}

// Disjoint spans: every (layer, head, row, chunk) item is independent, so
// the items form one flat range walked grid-stride by a grid sized to the
// resident CTAs; each thread keeps kItemsPerThread items (16 loads) in
// flight and needs no barrier.
template <typename T>
__global__ void __launch_bounds__(kShiftThreads) kv_shift_flat_kernel(const ShiftArgs a) {
  __shared__ float2 s_cs[128];
  const int D = a.row_bytes / a.elem_bytes;
  for (int i = threadIdx.x; i < D / 2; i += kShiftThreads) s_cs[i] = a.cs[i];
  __syncthreads();
  pdl_wait();
  // a dependent launch (the next segment of an overlapping move) may take
  // the slots of finished CTAs; it reads nothing before its own wait
  pdl_launch_dependents();
  const int hc = a.row_bytes / 32;  // 16-byte chunks per half row
  const int half_bytes = a.row_bytes / 2;
  const long long per_head = (long long)a.count * hc;
  const long long total = per_head * a.L * a.Hkv;
  const long long stride = (long long)gridDim.x * kShiftThreads;
  for (long long i0 = (long long)blockIdx.x * kShiftThreads + threadIdx.x; i0 < total;
       i0 += stride * kItemsPerThread) {
    uint4 k1[kItemsPerThread], k2[kItemsPerThread], v1[kItemsPerThread], v2[kItemsPerThread];
    char* kd[kItemsPerThread];
    char* vd[kItemsPerThread];
    int chunk[kItemsPerThread];
#pragma unroll
    for (int u = 0; u < kItemsPerThread; ++u) {
      const long long item = i0 + u * stride;
      kd[u] = nullptr;
      if (item < total) {
        const int lh = (int)(item / per_head);
        const long long rem = item - (long long)lh * per_head;
        const int j = (int)(rem / hc);
        const int c = (int)(rem - (long long)j * hc);
        const int l = lh / a.Hkv, g = lh - l * a.Hkv;
        const long long so = row_offset(a, g, a.src + j);
        const long long d = row_offset(a, g, a.dst + j);
        if (so < 0 || d < 0) {
          flag_error(a.err, PF_DEVERR_CAPACITY);
          continue;
        }
        const char* kb = a.cache_k + (long long)l * a.layer_bytes + so + c * 16;
        const char* vb = a.cache_v + (long long)l * a.layer_bytes + so + c * 16;
        k1[u] = *reinterpret_cast<const uint4*>(kb);
        k2[u] = *reinterpret_cast<const uint4*>(kb + half_bytes);
        v1[u] = *reinterpret_cast<const uint4*>(vb);
        v2[u] = *reinterpret_cast<const uint4*>(vb + half_bytes);
        kd[u] = a.cache_k + (long long)l * a.layer_bytes + d;
        vd[u] = a.cache_v + (long long)l * a.layer_bytes + d;
        chunk[u] = c;
      }
    }
#pragma unroll
    for (int u = 0; u < kItemsPerThread; ++u)
      if (kd[u]) rotate_store<T>(s_cs, chunk[u], k1[u], k2[u], v1[u], v2[u], kd[u], vd[u], half_bytes);
  }
}

// Overlapping spans with a small shift: one CTA per (layer, KV head) walks
// the passes in the safe order.
template <typename T>
__global__ void __launch_bounds__(kShiftThreads) kv_shift_kernel(const ShiftArgs a) {
  // cos / sin of the frequencies in shared memory: threads index the table
  // by their own chunk, which from the parameter bank would serialise
  __shared__ float2 s_cs[128];
  const int D = a.row_bytes / a.elem_bytes;
  for (int i = threadIdx.x; i < D / 2; i += kShiftThreads) s_cs[i] = a.cs[i];
  __syncthreads();
  pdl_wait();
  const int l = blockIdx.y / a.Hkv, g = blockIdx.y % a.Hkv;
  const int half_chunks = a.row_bytes / 32;  // 16-byte chunks per half row
  const int rows_per_pass = kItemsPerThread * kShiftThreads / half_chunks;
  const int passes = (a.count + rows_per_pass - 1) / rows_per_pass;

  char* kbase = a.cache_k + (long long)l * a.layer_bytes;
  char* vbase = a.cache_v + (long long)l * a.layer_bytes;
  const int half_bytes = a.row_bytes / 2;
  for (int pi = 0; pi < passes; ++pi) {
    const int p = a.descending ? passes - 1 - pi : pi;
    uint4 k1[kItemsPerThread], k2[kItemsPerThread], v1[kItemsPerThread], v2[kItemsPerThread];
    long long dst_off[kItemsPerThread];
    int chunk[kItemsPerThread];
#pragma unroll
    for (int u = 0; u < kItemsPerThread; ++u) {
      const int item = u * kShiftThreads + threadIdx.x;
      const int r = item / half_chunks;  // row within the pass
      const int j = p * rows_per_pass + r;
      const int c = item % half_chunks;
      chunk[u] = c;
      dst_off[u] = -1;
      if (r < rows_per_pass && j < a.count) {
        const long long so = row_offset(a, g, a.src + j);
        const long long d = row_offset(a, g, a.dst + j);
        if (so < 0 || d < 0) {
          flag_error(a.err, PF_DEVERR_CAPACITY);
          continue;
        }
        dst_off[u] = d;
        k1[u] = *reinterpret_cast<const uint4*>(kbase + so + c * 16);
        k2[u] = *reinterpret_cast<const uint4*>(kbase + so + half_bytes + c * 16);
        v1[u] = *reinterpret_cast<const uint4*>(vbase + so + c * 16);
        v2[u] = *reinterpret_cast<const uint4*>(vbase + so + half_bytes + c * 16);
      }
    }
    __syncthreads();  // every source row of this pass is read before any write
#pragma unroll
    for (int u = 0; u < kItemsPerThread; ++u)
      if (dst_off[u] >= 0)
        rotate_store<T>(s_cs, chunk[u], k1[u], k2[u], v1[u], v2[u], kbase + dst_off[u],
                        vbase + dst_off[u], half_bytes);
    __syncthreads();  // writes of this pass land before the next pass reads
  }
  pdl_launch_dependents();
}

}  // namespace

// A move whose spans overlap (shift d = |dst - src| < count) is cut into
// segments of d rows, launched in the order that consumes every source row
// before it is overwritten (from the front for a move to lower positions,
// from the back for a move to higher ones); each segment's spans are then
// disjoint and its passes run in parallel.  A shift so small that this
// would take more than kMaxSegments launches instead walks the passes in
// order inside one CTA per (layer, head).
constexpr int kMaxSegments = 8;

cudaError_t launch_kv_shift(const ShiftArgs& a0, cudaStream_t s, int num_sms, bool pdl) {
  static DeviceMemo resident[2];  // resident CTAs per SM, fp32 / bf16 kernel
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const int bf = a0.elem_bytes == 2;
  int per_sm = resident[bf].get(dev);
  if (per_sm == 0) {
    e = bf ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                 &per_sm, kv_shift_flat_kernel<__nv_bfloat16>, kShiftThreads, 0)
           : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kv_shift_flat_kernel<float>,
                                                            kShiftThreads, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    resident[bf].set(dev, per_sm);
  }
  auto launch = [&](const ShiftArgs& a) {
    if (a.overlap) {
      const dim3 grid(1, (unsigned)(a.L * a.Hkv));
      return bf ? launch_ex(kv_shift_kernel<__nv_bfloat16>, grid, dim3(kShiftThreads), 0, s, 1,
                            pdl, a)
                : launch_ex(kv_shift_kernel<float>, grid, dim3(kShiftThreads), 0, s, 1, pdl, a);
    }
    const long long items = (long long)a.count * (a.row_bytes / 32) * a.L * a.Hkv;
    const long long want = (items + (long long)kShiftThreads * kItemsPerThread - 1) /
                           ((long long)kShiftThreads * kItemsPerThread);
    const unsigned grid = (unsigned)std::max<long long>(
        1, std::min<long long>(want, (long long)num_sms * per_sm));
    return bf ? launch_ex(kv_shift_flat_kernel<__nv_bfloat16>, dim3(grid), dim3(kShiftThreads), 0,
                          s, 1, pdl, a)
              : launch_ex(kv_shift_flat_kernel<float>, dim3(grid), dim3(kShiftThreads), 0, s, 1,
                          pdl, a);
  };
  ShiftArgs a = a0;
  const int d = a0.dst > a0.src ? a0.dst - a0.src : a0.src - a0.dst;
  a.descending = a0.dst > a0.src;
  if (d >= a0.count) {
    a.overlap = 0;
    return launch(a);
  }
  const int segs = (a0.count + d - 1) / d;
  if (segs > kMaxSegments) {
    a.overlap = 1;
    return launch(a);
  }
  a.overlap = 0;
  for (int k = 0; k < segs; ++k) {
    const int idx = a.descending ? segs - 1 - k : k;
    const int off = idx * d;
    a.src = a0.src + off;
    a.dst = a0.dst + off;
    a.count = std::min(d, a0.count - off);
    e = launch(a);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace pf
