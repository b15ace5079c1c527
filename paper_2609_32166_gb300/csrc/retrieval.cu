// Decoding-experience retrieval (Section 3.2 "Context-compatible retrieval";
// Section 4 "Memory and retrieval").
//
// pf_retrieval_key: z = P h (one warp per output row, lanes across the
// hidden dimension), then the last CTA to finish (ticket) scales by
// 127 / max|z| and rounds half to even into the int8 key.  Normalising h
// first does not change the key (the scale cancels), so it is skipped.
//
// pf_retrieve: warps sweep groups of 32 entries; a ballot of the cheap
// filter (token match, position before boundary) decides which 256-byte
// keys are read at all.  Each eligible key is read by one warp (8 bytes per
// lane, two dp4a for the dot product and two for the squared norm) and the
// winner is chosen exactly: cos_a > cos_b  <=>  dot_a^2 kk_b > dot_b^2 kk_a
// (with signs), in 128-bit integer arithmetic, ties to the lower index.
// Per-CTA winners meet in the workspace; the last CTA picks the overall one.
#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

constexpr int kKeyThreads = 256;
constexpr int kScanThreads = 256;

struct Cand {
  int j;    // entry index, -1 = none
  int dot;  // query . key
  int kk;   // key . key
};

// Is candidate a strictly better than b (higher cosine, or equal cosine and
// lower index)?  b.j < 0 means "no candidate".
__device__ __forceinline__ bool cand_better(const Cand& a, const Cand& b) {
  if (a.j < 0) return false;
  if (b.j < 0) return true;
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

__global__ void __launch_bounds__(kKeyThreads) retrieval_key_kernel(const KeyArgs a) {
  pdl_wait();
  __shared__ int s_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * (kKeyThreads / 32) + warp;
  if (row < PF_KEY_DIM) {
    float acc = 0.f;
    if (a.bf16) {
      const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(a.hidden);
      const __nv_bfloat16* p = static_cast<const __nv_bfloat16*>(a.proj) + (size_t)row * a.H;
      for (int c = lane; c < a.H; c += 32)
        acc = fmaf(__bfloat162float(p[c]), __bfloat162float(h[c]), acc);
    } else {
      const float* h = static_cast<const float*>(a.hidden);
      const float* p = static_cast<const float*>(a.proj) + (size_t)row * a.H;
      for (int c = lane; c < a.H; c += 32) acc = fmaf(p[c], h[c], acc);
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) a.z[row] = acc;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(a.ticket, 1u) == gridDim.x - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
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

__device__ __forceinline__ void warp_sum2(int& x, int& y) {
#pragma unroll
  for (int off = 16; off; off >>= 1) {
    x += __shfl_xor_sync(0xffffffffu, x, off);
    y += __shfl_xor_sync(0xffffffffu, y, off);
  }
}

__global__ void __launch_bounds__(kScanThreads) retrieve_kernel(const RetrievalArgs a) {
  pdl_wait();
  __shared__ Cand s_cand[kScanThreads / 32];
  __shared__ int s_last;
  __shared__ int s_qq;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // this lane's 8 bytes of the query key, and the query's squared norm
  const uint2 q = *reinterpret_cast<const uint2*>(a.query_key + lane * 8);
  int qq = __dp4a((int)q.x, (int)q.x, __dp4a((int)q.y, (int)q.y, 0));
  {
    int dummy = 0;
    warp_sum2(qq, dummy);
  }
  Cand best = {-1, 0, 1};
  const int nwarps = gridDim.x * (kScanThreads / 32);
  for (long long j0 = a.lo + (long long)(blockIdx.x * (kScanThreads / 32) + warp) * 32; j0 < a.hi;
       j0 += (long long)nwarps * 32) {
    const long long jl = j0 + lane;
    bool elig = false;
    if (jl < a.hi)
      elig = __ldg(&a.entry_token[jl]) == a.token && __ldg(&a.entry_pos[jl]) < __ldg(&a.entry_bound[jl]);
    unsigned mask = __ballot_sync(0xffffffffu, elig);
    while (mask) {
      // up to two eligible keys in flight per iteration
      const int e0 = __ffs(mask) - 1;
      mask &= mask - 1;
      const int e1 = mask ? __ffs(mask) - 1 : -1;
      if (e1 >= 0) mask &= mask - 1;
      const uint2 k0 = __ldg(reinterpret_cast<const uint2*>(a.keys + (j0 + e0) * PF_KEY_DIM) + lane);
      uint2 k1 = make_uint2(0, 0);
      if (e1 >= 0)
        k1 = __ldg(reinterpret_cast<const uint2*>(a.keys + (j0 + e1) * PF_KEY_DIM) + lane);
      int d0 = __dp4a((int)k0.x, (int)q.x, __dp4a((int)k0.y, (int)q.y, 0));
      int n0 = __dp4a((int)k0.x, (int)k0.x, __dp4a((int)k0.y, (int)k0.y, 0));
      int d1 = __dp4a((int)k1.x, (int)q.x, __dp4a((int)k1.y, (int)q.y, 0));
      int n1 = __dp4a((int)k1.x, (int)k1.x, __dp4a((int)k1.y, (int)k1.y, 0));
      warp_sum2(d0, n0);
      warp_sum2(d1, n1);
      if (n0 > 0) {
        const Cand c = {(int)(j0 + e0), d0, n0};
        if (cand_better(c, best)) best = c;
      }
      if (e1 >= 0 && n1 > 0) {
        const Cand c = {(int)(j0 + e1), d1, n1};
        if (cand_better(c, best)) best = c;
      }
    }
  }
  if (lane == 0) s_cand[warp] = best;
  if (threadIdx.x == 0) s_qq = qq;
  __syncthreads();
  if (threadIdx.x == 0) {
    Cand b = s_cand[0];
    for (int w = 1; w < kScanThreads / 32; ++w)
      if (cand_better(s_cand[w], b)) b = s_cand[w];
    a.block_best[blockIdx.x] = make_int4(b.j, b.dot, b.kk, 0);
    __threadfence();
    s_last = (atomicAdd(a.ticket, 1u) == gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    Cand b = {-1, 0, 1};
    for (int i = 0; i < (int)gridDim.x; ++i) {
      const int4 v = __ldcg(&a.block_best[i]);
      const Cand c = {v.x, v.y, v.z};
      if (cand_better(c, b)) b = c;
      a.block_best[i] = make_int4(0, 0, 0, 0);
    }
    a.best[0] = b.j;
    a.similarity[0] =
        b.j < 0 ? __int_as_float(0x7fc00000) : (float)((double)b.dot / sqrt((double)s_qq * b.kk));
    *a.ticket = 0u;
  }
  pdl_launch_dependents();
}

}  // namespace

cudaError_t launch_retrieval_key(const KeyArgs& a, cudaStream_t s, bool pdl) {
  return launch_ex(retrieval_key_kernel, dim3(PF_KEY_DIM / (kKeyThreads / 32)), dim3(kKeyThreads),
                   0, s, 1, pdl, a);
}

cudaError_t launch_retrieve(const RetrievalArgs& a, cudaStream_t s, int num_sms, bool pdl) {
  const long long range = (long long)a.hi - a.lo;
  long long blocks = (range + kScanThreads - 1) / kScanThreads;  // 8 warps x 32 entries
  const long long cap = std::min<long long>(kRetrievalMaxBlocks, 4LL * num_sms);
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return launch_ex(retrieve_kernel, dim3((unsigned)blocks), dim3(kScanThreads), 0, s, 1, pdl, a);
}

}  // namespace pf
