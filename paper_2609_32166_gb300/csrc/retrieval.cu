// Decoding-experience retrieval (Section 3.2 "Context-compatible retrieval";
// Section 4 "Memory and retrieval").
//
// pf_retrieval_key: z = P h (128 threads per output row, 16-byte loads
// when the rows allow), then the last CTA to finish (ticket) scales by
// 127 / max|z| and rounds half to even into the int8 key.  Normalising h
// first does not change the key (the scale cancels), so it is skipped.
//
// pf_retrieve: one CTA per SM at most; each warp filters groups of 128
// entries (16-byte token loads, 4 entries per lane) and lists the eligible
// ones (token match, position before boundary).  The first group is
// filtered before the grid-dependency wait, overlapping the kernel that
// produces the query key.  Listed keys are copied 32 at a time into shared
// memory with asynchronous 16-byte copies (all in flight together) and
// scored one per lane with dp4a.  The
// winner is chosen exactly: cos_a > cos_b  <=>  dot_a^2 kk_b > dot_b^2 kk_a
// (with signs), in 128-bit integer arithmetic, ties to the lower index.
// Per-CTA winners meet in the workspace; the last CTA picks the overall one.
#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

constexpr int kKeyThreads = 256;
constexpr int kKeyRowThreads = 128;
constexpr int kKeyRowsPerCta = kKeyThreads / kKeyRowThreads;
static_assert(kKeyThreads >= PF_KEY_DIM, "the last CTA writes one code per thread");
constexpr int kScanThreads = 512;
constexpr int kScanWarps = kScanThreads / 32;
constexpr int kScanGroup = 128;  // entries a warp filters at once (4 per lane)
constexpr int kScanRound = 32;   // keys a warp stages and scores at once (one per lane)
constexpr int kScanWarpSmem = kScanGroup * 4 + kScanRound * PF_KEY_DIM;
constexpr int kScanSmem = kScanWarps * kScanWarpSmem;

struct Cand {
  int j;    // entry index, -1 = none
  int dot;  // query . key
  int kk;   // key . key
  float s;  // dot / sqrt(kk) in fp32 (the cosine times |query|, to a few ulp)
};

__device__ __forceinline__ Cand make_cand(int j, int dot, int kk) {
  return Cand{j, dot, kk, (float)dot * rsqrtf((float)kk)};
}

// Is candidate a strictly better than b (higher cosine, or equal cosine and
// lower index)?  b.j < 0 means "no candidate".  dot and kk are below 2^24,
// so s carries a relative error of a few 1e-7: a difference in s above
// 1e-5 of its size decides; closer calls are settled exactly in integers.
__device__ __forceinline__ bool cand_better(const Cand& a, const Cand& b) {
  if (a.j < 0) return false;
  if (b.j < 0) return true;
  const float d = a.s - b.s;
  const float tol = 1e-5f * fmaxf(fabsf(a.s), fabsf(b.s));
  if (d > tol) return true;
  if (d < -tol) return false;
  if ((a.dot >= 0) != (b.dot >= 0)) return a.dot >= 0;
  const unsigned long long da = (unsigned long long)((long long)a.dot * a.dot);
  const unsigned long long db = (unsigned long long)((long long)b.dot * b.dot);
  const unsigned long long lo1 = da * (unsigned long long)b.kk;
  const unsigned long long hi1 = __umul64hi(da, (unsigned long long)b.kk);
  const unsigned long long lo2 = db * (unsigned long long)a.kk;
  const unsigned long long hi2 = __umul64hi(db, (unsigned long long)a.kk);
  const bool eq = hi1 == hi2 && lo1 == lo2;
  if (eq) return a.j < b.j;
  const bool gt = hi1 > hi2 || (hi1 == hi2 && lo1 > lo2);
  return a.dot >= 0 ? gt : !gt;  // negative cosines: the smaller ratio is the larger cosine
}

// atomicAdd with release (publishes this thread's earlier writes) and
// acquire (sees what earlier arrivals published) at GPU scope.
__device__ __forceinline__ unsigned atomic_add_acq_rel(unsigned* p, unsigned v) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ float dot8_bf16(const uint4& x, const uint4& y, float acc) {
  const uint32_t* xa = &x.x;
  const uint32_t* ya = &y.x;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    acc = fmaf(__uint_as_float(xa[i] << 16), __uint_as_float(ya[i] << 16), acc);
    acc = fmaf(__uint_as_float(xa[i] & 0xFFFF0000u), __uint_as_float(ya[i] & 0xFFFF0000u), acc);
  }
  return acc;
}

// 128 CTAs x 2 rows; 128 threads (4 warps) per row.
__global__ void __launch_bounds__(kKeyThreads) retrieval_key_kernel(const KeyArgs a) {
  pdl_wait();
  // the scan may start filtering entries now; it waits for this grid to
  // finish before it reads the key
  pdl_launch_dependents();
  __shared__ int s_last;
  __shared__ float s_part[kKeyThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = threadIdx.x / kKeyRowThreads, t = threadIdx.x % kKeyRowThreads;
  const int row = blockIdx.x * kKeyRowsPerCta + r;
  float acc = 0.f;
  if (a.vec && a.bf16) {
    const uint4* h = static_cast<const uint4*>(a.hidden);
    const uint4* p = static_cast<const uint4*>(a.proj) + (size_t)row * (a.H / 8);
    const int n = a.H / 8;
#pragma unroll 4
    for (int c = t; c < n; c += kKeyRowThreads) acc = dot8_bf16(__ldg(p + c), __ldg(h + c), acc);
  } else if (a.vec) {
    const float4* h = static_cast<const float4*>(a.hidden);
    const float4* p = static_cast<const float4*>(a.proj) + (size_t)row * (a.H / 4);
    const int n = a.H / 4;
#pragma unroll 4
    for (int c = t; c < n; c += kKeyRowThreads) {
      const float4 x = __ldg(p + c), y = __ldg(h + c);
      acc = fmaf(x.x, y.x, fmaf(x.y, y.y, fmaf(x.z, y.z, fmaf(x.w, y.w, acc))));
    }
  } else if (a.bf16) {
    const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(a.hidden);
    const __nv_bfloat16* p = static_cast<const __nv_bfloat16*>(a.proj) + (size_t)row * a.H;
    for (int c = t; c < a.H; c += kKeyRowThreads)
      acc = fmaf(__bfloat162float(p[c]), __bfloat162float(h[c]), acc);
  } else {
    const float* h = static_cast<const float*>(a.hidden);
    const float* p = static_cast<const float*>(a.proj) + (size_t)row * a.H;
    for (int c = t; c < a.H; c += kKeyRowThreads) acc = fmaf(p[c], h[c], acc);
  }
#pragma unroll
  for (int off = 16; off; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (lane == 0) s_part[warp] = acc;
  __syncthreads();
  if (t == 0) {
    float z = 0.f;
#pragma unroll
    for (int w = 0; w < kKeyRowThreads / 32; ++w) z += s_part[r * (kKeyRowThreads / 32) + w];
    a.z[row] = z;
  }
  // one release/acquire atomic per CTA publishes this CTA's rows (ordered
  // before it by the barrier) and, in the last CTA, makes every row visible
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomic_add_acq_rel(a.ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __shared__ float s_max[kKeyThreads / 32];
  const float z = threadIdx.x < PF_KEY_DIM ? __ldcg(&a.z[threadIdx.x]) : 0.f;
  float m = fabsf(z);
#pragma unroll
  for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  if (lane == 0) s_max[warp] = m;
  __syncthreads();
  if (warp == 0) {
    m = lane < kKeyThreads / 32 ? s_max[lane] : 0.f;
#pragma unroll
    for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    if (lane == 0) s_max[0] = m;
  }
  __syncthreads();
  m = s_max[0];
  if (threadIdx.x < PF_KEY_DIM) {
    const float x = m > 0.f ? 127.f * z / m : 0.f;
    a.key_out[threadIdx.x] = (int8_t)(int)rintf(fminf(fmaxf(x, -127.f), 127.f));
    a.z[threadIdx.x] = 0.f;  // leave the workspace zeroed
  }
  if (threadIdx.x == 0) *a.ticket = 0u;
}

// The best of a warp's candidates, in every lane (cand_better is a strict
// total order, so the butterfly agrees across lanes).
__device__ __forceinline__ Cand warp_best(Cand b) {
#pragma unroll
  for (int off = 16; off; off >>= 1) {
    const Cand o = {__shfl_xor_sync(0xffffffffu, b.j, off), __shfl_xor_sync(0xffffffffu, b.dot, off),
                    __shfl_xor_sync(0xffffffffu, b.kk, off), __shfl_xor_sync(0xffffffffu, b.s, off)};
    if (cand_better(o, b)) b = o;
  }
  return b;
}

// Filter one group of kScanGroup entries starting at j0 (a multiple of 4):
// lane l tests entries j0 + 4l .. j0 + 4l + 3 (token match, p < b, inside
// [lo, hi)) and the eligible ones are listed in entry order in `list`.
// Returns how many there are.  Needs no query key.
__device__ __forceinline__ int filter_group(const RetrievalArgs& a, long long j0, int lane,
                                            int* list) {
  const long long j = j0 + 4 * lane;
  unsigned bits = 0;
  if (j >= a.lo && j + 3 < a.hi) {
    // the three 16-byte loads go out together (no dependent round trip)
    const int4 t = __ldg(reinterpret_cast<const int4*>(a.entry_token + j));
    const int4 p = __ldg(reinterpret_cast<const int4*>(a.entry_pos + j));
    const int4 b = __ldg(reinterpret_cast<const int4*>(a.entry_bound + j));
    bits = (t.x == a.token && p.x < b.x) | (t.y == a.token && p.y < b.y) << 1 |
           (t.z == a.token && p.z < b.z) << 2 | (t.w == a.token && p.w < b.w) << 3;
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (j + k >= a.lo && j + k < a.hi && __ldg(a.entry_token + j + k) == a.token &&
          __ldg(a.entry_pos + j + k) < __ldg(a.entry_bound + j + k))
        bits |= 1u << k;
  }
  const int cnt = __popc(bits);
  int incl = cnt;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += v;
  }
  int at = incl - cnt;
#pragma unroll
  for (int k = 0; k < 4; ++k)
    if (bits >> k & 1) list[at++] = (int)(j + k);
  __syncwarp();
  return __shfl_sync(0xffffffffu, incl, 31);
}

// Score up to kScanRound listed keys: all their bytes are copied to the
// warp's stage with asynchronous 16-byte copies (coalesced, all in flight
// at once), then lane i scores key i from shared memory (chunks visited in
// a lane-rotated order, so a warp's reads spread over all banks).
__device__ __forceinline__ Cand score_round(const int8_t* keys, const int* list, int m,
                                            int8_t* stage, const int8_t* s_q, int lane, Cand best) {
  const uint32_t sbase = static_cast<uint32_t>(__cvta_generic_to_shared(stage));
#pragma unroll
  for (int i = 0; i < kScanRound * PF_KEY_DIM / 16 / 32; ++i) {
    const int u = lane + 32 * i;
    const int key = u >> 4, c = u & 15;
    if (key < m)
      cp_async16(sbase + key * PF_KEY_DIM + c * 16, keys + (size_t)list[key] * PF_KEY_DIM + c * 16);
  }
  cp_async_wait_all();
  __syncwarp();
  if (lane < m) {
    const uint4* kp = reinterpret_cast<const uint4*>(stage + lane * PF_KEY_DIM);
    const uint4* qp = reinterpret_cast<const uint4*>(s_q);
    int dot = 0, kk = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int c = (i + lane) & 15;
      const uint4 k = kp[c], q = qp[c];
      dot = __dp4a((int)k.x, (int)q.x, dot);
      dot = __dp4a((int)k.y, (int)q.y, dot);
      dot = __dp4a((int)k.z, (int)q.z, dot);
      dot = __dp4a((int)k.w, (int)q.w, dot);
      kk = __dp4a((int)k.x, (int)k.x, kk);
      kk = __dp4a((int)k.y, (int)k.y, kk);
      kk = __dp4a((int)k.z, (int)k.z, kk);
      kk = __dp4a((int)k.w, (int)k.w, kk);
    }
    if (kk > 0) {
      const Cand cand = make_cand(list[lane], dot, kk);
      if (cand_better(cand, best)) best = cand;
    }
  }
  __syncwarp();  // the stage is refilled in the next pass
  return best;
}

__global__ void __launch_bounds__(kScanThreads) retrieve_kernel(const RetrievalArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ __align__(16) int8_t s_q[PF_KEY_DIM];
  __shared__ Cand s_cand[kScanWarps];
  __shared__ int s_last, s_qq;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int* list = reinterpret_cast<int*>(smem + warp * kScanWarpSmem);
  int8_t* stage = reinterpret_cast<int8_t*>(smem + warp * kScanWarpSmem + kScanGroup * 4);
  const long long base = a.lo & ~3LL;
  const long long stride = (long long)gridDim.x * kScanWarps * kScanGroup;
  long long j0 = base + ((long long)blockIdx.x * kScanWarps + warp) * kScanGroup;
  // the first group is filtered before waiting for the kernel that writes
  // the query key (entry metadata does not depend on it)
  int n = j0 < a.hi ? filter_group(a, j0, lane, list) : 0;
  pdl_wait();
  if (threadIdx.x < PF_KEY_DIM / 16)
    reinterpret_cast<uint4*>(s_q)[threadIdx.x] =
        __ldg(reinterpret_cast<const uint4*>(a.query_key) + threadIdx.x);
  __syncthreads();
  if (warp == 0) {
    const int q0 = reinterpret_cast<const int*>(s_q)[lane];
    const int q1 = reinterpret_cast<const int*>(s_q)[lane + 32];
    int qq = __dp4a(q0, q0, __dp4a(q1, q1, 0));
#pragma unroll
    for (int off = 16; off; off >>= 1) qq += __shfl_xor_sync(0xffffffffu, qq, off);
    if (lane == 0) s_qq = qq;
  }
  Cand best = {-1, 0, 1, 0.f};
  while (j0 < a.hi) {
    for (int r0 = 0; r0 < n; r0 += kScanRound)
      best = score_round(a.keys, list + r0, min(kScanRound, n - r0), stage, s_q, lane, best);
    j0 += stride;
    n = j0 < a.hi ? filter_group(a, j0, lane, list) : 0;
  }
  best = warp_best(best);
  if (lane == 0) s_cand[warp] = best;
  __syncthreads();
  static_assert(kScanWarps <= 32, "one warp reduces the per-warp winners");
  const Cand none = {-1, 0, 1, 0.f};
  if (gridDim.x > 1) {
    if (warp == 0) {
      const Cand b = warp_best(lane < kScanWarps ? s_cand[lane] : none);
      if (lane == 0) {
        a.block_best[blockIdx.x] = make_int4(b.j, b.dot, b.kk, __float_as_int(b.s));
        s_last = atomic_add_acq_rel(a.ticket, 1u) == gridDim.x - 1;
      }
    }
    __syncthreads();
    if (!s_last) return;
    Cand b = none;
    for (int i = threadIdx.x; i < (int)gridDim.x; i += kScanThreads) {
      const int4 v = __ldcg(&a.block_best[i]);
      const Cand c = {v.x, v.y, v.z, __int_as_float(v.w)};
      if (cand_better(c, b)) b = c;
      a.block_best[i] = make_int4(0, 0, 0, 0);
    }
    b = warp_best(b);
    __syncthreads();  // s_cand of the scan phase has been read
    if (lane == 0) s_cand[warp] = b;
    __syncthreads();
  }
  if (warp == 0) {
    const Cand b = warp_best(lane < kScanWarps ? s_cand[lane] : none);
    if (lane == 0) {
      a.best[0] = b.j;
      // fp32: dot, qq and kk are exact, the product, root and quotient
      // each round once (relative error below 3e-7)
      a.similarity[0] =
          b.j < 0 ? __int_as_float(0x7fc00000) : (float)b.dot / sqrtf((float)s_qq * (float)b.kk);
      if (gridDim.x > 1) *a.ticket = 0u;
    }
  }
  pdl_launch_dependents();
}

}  // namespace

cudaError_t launch_retrieval_key(const KeyArgs& a, cudaStream_t s, bool pdl) {
  return launch_ex(retrieval_key_kernel, dim3(PF_KEY_DIM / kKeyRowsPerCta), dim3(kKeyThreads), 0,
                   s, 1, pdl, a);
}

cudaError_t launch_retrieve(const RetrievalArgs& a, cudaStream_t s, int num_sms, bool pdl) {
  static DeviceMemo smem_set;
  cudaError_t e = ensure_smem_limit(reinterpret_cast<const void*>(retrieve_kernel), kScanSmem,
                                    smem_set);
  if (e != cudaSuccess) return e;
  const long long range = (long long)a.hi - (a.lo & ~3LL);
  long long blocks = (range + kScanWarps * kScanGroup - 1) / (kScanWarps * kScanGroup);
  const long long cap = std::min<long long>(kRetrievalMaxBlocks, num_sms);
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return launch_ex(retrieve_kernel, dim3((unsigned)blocks), dim3(kScanThreads), kScanSmem, s, 1,
                   pdl, a);
}

}  // namespace pf
