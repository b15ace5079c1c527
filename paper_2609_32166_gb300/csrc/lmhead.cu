// LM head, greedy prediction and acceptance (Section 3.2).
//
// logits = hidden . W^T is a skinny GEMM: M = vocabulary (~152K rows of W,
// the dominant bytes of the whole verify step), N = proposal nodes (<= 256),
// K = hidden size.  The bf16 kernel is persistent (one CTA per SM) and
// streams 128-row tiles of W by TMA through a shared-memory ring; one thread
// issues tcgen05 UMMAs (M = 128, N = nodes rounded up to 16, K = 16) whose
// fp32 accumulators live in TMEM, double-buffered so the epilogue of one
// vocabulary tile overlaps the MMAs of the next.  Four epilogue warps read
// the accumulators back (tcgen05.ld), reduce each node's column to a packed
// (logit, index) maximum with a transposing warp-shuffle tree, and keep the
// CTA's best per node in shared memory.  Logits never reach global memory.
// Every CTA then folds its per-node best into the workspace with a 64-bit
// atomicMax; the last CTA to finish (a ticket counter, no spinning) decodes
// the argmax of every node and walks each proposal tree.
#include <cstdlib>

#include "pf_internal.h"
#include "pf_ptx.cuh"

namespace pf {

namespace {

constexpr int kBM = 128;           // vocabulary rows per tile (UMMA M)
constexpr int kBK = 64;            // hidden elements per stage (128 bytes of bf16)
constexpr int kABytes = kBM * kBK * 2;
constexpr int kTcThreads = 192;    // warp 0 TMA, warp 1 MMA, warps 2..5 epilogue
constexpr int kMaxStages = 12;

// Greedy descent of every proposal tree of the batch.  Runs in the last CTA
// after all per-node maxima are final.  One warp per sequence.
__device__ void finalize_accept(const LmArgs& a, int32_t* s_argmax) {
  for (int t = threadIdx.x; t < a.T; t += blockDim.x) {
    const unsigned long long k = __ldcg(&a.best[t]);
    const int am = (int)argmax_key_index(k);
    s_argmax[t] = am;
    a.argmax[t] = am;
    if (a.max_logit) a.max_logit[t] = argmax_key_logit(k);
    a.best[t] = 0ull;  // leave the workspace zeroed for the next call
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = blockDim.x >> 5;
  for (int b = warp; b < a.B; b += nwarps) {
    const int off = a.cu_nodes[b];
    int n = a.cu_nodes[b + 1] - off;
    if (off < 0 || n < 1 || n > a.max_nodes || off + n > a.T) {
      if (lane == 0) flag_error(a.err, PF_DEVERR_BOUNDS);
      n = 0;  // walk nothing; report the root alone
      if (off < 0 || off >= a.T) {
        if (lane == 0) a.accept_len[b] = -1;
        continue;
      }
    }
    int32_t* path = a.path + (size_t)b * a.max_nodes;
    int32_t* out = a.out_tokens + (size_t)b * a.max_nodes;
    int u = 0, depth = 0;
    if (lane == 0) path[0] = 0;
    for (int step = 0; step < n; ++step) {
      const int want = s_argmax[off + u];
      int found = -1;
      for (int c0 = u + 1; c0 < n && found < 0; c0 += 32) {
        const int c = c0 + lane;
        const bool match = c < n && a.parent[off + c] == u && a.tokens[off + c] == want;
        const unsigned bal = __ballot_sync(0xffffffffu, match);
        if (bal) found = c0 + __ffs(bal) - 1;
      }
      if (found < 0) break;
      ++depth;
      if (lane == 0) {
        path[depth] = found;
        out[depth - 1] = a.tokens[off + found];
      }
      u = found;
    }
    if (lane == 0) {
      out[depth] = s_argmax[off + u];
      a.accept_len[b] = depth;
      if (a.last_node) a.last_node[b] = u;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *a.ticket = 0u;
}

// Fold this CTA's per-node maxima into the workspace; the last CTA finalizes.
__device__ void merge_and_finish(const LmArgs& a, const unsigned long long* s_best,
                                 int32_t* s_argmax, int* s_last) {
  for (int t = threadIdx.x; t < a.T; t += blockDim.x)
    if (s_best[t]) atomicMax(&a.best[t], s_best[t]);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) *s_last = (atomicAdd(a.ticket, 1u) == gridDim.x - 1);
  __syncthreads();
  if (*s_last) {
    __threadfence();
    finalize_accept(a, s_argmax);
  }
}

// Max over the 32 lanes of a warp for each of 16 columns: after the five
// exchange rounds lane l (and l ^ 1) holds column ((l >> 1) & 15).
__device__ __forceinline__ unsigned long long warp_colmax16(unsigned long long (&k)[16],
                                                            int lane) {
#pragma unroll
  for (int s = 0; s < 4; ++s) {
    const int off = 16 >> s;
    const int n = 8 >> s;
    const bool hi = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < n; ++i) {
      const unsigned long long send = hi ? k[i] : k[i + n];
      const unsigned long long keep = hi ? k[i + n] : k[i];
      k[i] = umax64(keep, __shfl_xor_sync(0xffffffffu, send, off));
    }
  }
  return umax64(k[0], __shfl_xor_sync(0xffffffffu, k[0], 1));
}

__global__ void __launch_bounds__(kTcThreads, 1)
    lmhead_tc_kernel(const __grid_constant__ CUtensorMap tm_w,
                     const __grid_constant__ CUtensorMap tm_h, const LmArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int ns = a.stages;
  const int npad = a.npad;
  const uint32_t b_bytes = (uint32_t)npad * 128;
  uint8_t* sA = smem;
  uint8_t* sB = smem + ns * kABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sB + ns * b_bytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kMaxStages;
  uint64_t* tfull = bars + 2 * kMaxStages;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  unsigned long long* s_best = reinterpret_cast<unsigned long long*>(tmem_slot + 2);
  int32_t* s_argmax = reinterpret_cast<int32_t*>(s_best + PF_MAX_LM_ROWS);
  int* s_misc = s_argmax + PF_MAX_LM_ROWS;  // [0] last-CTA flag, [1] TMA loads issued, [2] consumed

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t ncols = 32;
  while (ncols < (uint32_t)(2 * npad)) ncols <<= 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < ns; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), 128);
    }
    fence_mbar_init();
    tma_prefetch_desc(&tm_w);
    tma_prefetch_desc(&tm_h);
    s_misc[1] = 0;
    s_misc[2] = 0;
  }
  // With PF_LM_EARLY_WEIGHT the first `pre` stages of weight tiles are
  // requested before waiting for the preceding kernel (programmatic
  // dependent launch); their hidden-state halves follow after the wait.
  const int my_tiles = blockIdx.x < a.num_tiles
                           ? (a.num_tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                           : 0;
  const int pre = (a.flags & PF_LM_EARLY_WEIGHT) ? min(ns, my_tiles * a.nk) : 0;
  if (threadIdx.x == 0) {
    const uint64_t pol = l2_policy_evict_first();
    for (int it = 0; it < pre; ++it) {
      const int tile = blockIdx.x + (it / a.nk) * gridDim.x, kc = it % a.nk;
      const uint32_t fb = smem_u32(&full[it]);
      mbar_arrive_expect_tx(fb, kABytes + b_bytes);
      tma_load_2d_hint(smem_u32(sA + it * kABytes), &tm_w, kc * kBK, tile * kBM, fb, pol);
    }
  }
  for (int i = threadIdx.x; i < PF_MAX_LM_ROWS; i += blockDim.x) s_best[i] = 0ull;

  // Wait for whatever produced the hidden states (programmatic dependent
  // launch) before touching global memory or TMEM.
  pdl_wait();
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      const uint64_t pol = l2_policy_evict_first();
      int it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < a.num_tiles && ok; tile += gridDim.x) {
        for (int kc = 0; kc < a.nk; ++kc, ++it) {
          const int st = it % ns;
          const uint32_t fb = smem_u32(&full[st]);
          if (it >= pre) {
            if (!mbar_wait(smem_u32(&empty[st]), ((it / ns) & 1) ^ 1, a.err)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(fb, kABytes + b_bytes);
            tma_load_2d_hint(smem_u32(sA + st * kABytes), &tm_w, kc * kBK, tile * kBM, fb, pol);
          }
          tma_load_2d(smem_u32(sB + st * b_bytes), &tm_h, kc * kBK, 0, fb);
          s_misc[1] = it + 1;
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      const uint32_t idesc = umma_idesc_bf16(kBM, npad);
      int it = 0, lt = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < a.num_tiles && ok; tile += gridDim.x, ++lt) {
        const int acc = lt & 1;
        if (!mbar_wait(smem_u32(&tempty[acc]), ((lt >> 1) & 1) ^ 1, a.err)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * npad);
        for (int kc = 0; kc < a.nk; ++kc, ++it) {
          const int st = it % ns;
          if (!mbar_wait(smem_u32(&full[st]), (it / ns) & 1, a.err)) {
            ok = false;
            break;
          }
          s_misc[2] = it + 1;
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + st * kABytes);
          const uint32_t b0 = smem_u32(sB + st * b_bytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16(d_tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), idesc,
                      (kc | k) != 0);
          umma_commit(smem_u32(&empty[st]));
        }
        if (ok) umma_commit(smem_u32(&tfull[acc]));
      }
    }
  } else {
    // ---------------- epilogue: TMEM -> per-node (logit, index) maxima
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    int lt = 0;
    for (int tile = blockIdx.x; tile < a.num_tiles; tile += gridDim.x, ++lt) {
      const int acc = lt & 1;
      if (!mbar_wait(smem_u32(&tfull[acc]), (lt >> 1) & 1, a.err)) break;
      tc_fence_after();
      const int row = tile * kBM + q * 32 + lane;
      const bool row_ok = row < a.V;
      for (int c0 = 0; c0 < npad; c0 += 16) {
        uint32_t r[16];
        tmem_ld_16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * npad + c0), r);
        tmem_ld_wait();
        unsigned long long k[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          k[j] = (row_ok && c0 + j < a.T) ? argmax_key(__uint_as_float(r[j]), (uint32_t)row)
                                          : 0ull;
        const unsigned long long best = warp_colmax16(k, lane);
        const int col = c0 + ((lane >> 1) & 15);
        if ((lane & 1) == 0 && col < a.T && best) atomicMax(&s_best[col], best);
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&tempty[acc]));
    }
  }
  __syncwarp();  // the producer and MMA lanes rejoin their warps before the barrier

  __syncthreads();
  if (threadIdx.x == 0 && s_misc[1] > s_misc[2]) {
    // A wait ran out: let every TMA load still in flight land before exit.
    for (int it = s_misc[2]; it < s_misc[1]; ++it)
      mbar_wait(smem_u32(&full[it % ns]), (it / ns) & 1, a.err);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, ncols);
  }
  pdl_launch_dependents();
  merge_and_finish(a, s_best, s_argmax, &s_misc[0]);
}

// ---------------------------------------------------------------- fp32 path
// CUDA-core kernel: each warp takes vocabulary rows in turn and forms their
// dot products with every node's hidden state (lanes split the hidden dim).
__global__ void __launch_bounds__(256) lmhead_f32_kernel(const LmArgs a) {
  __shared__ unsigned long long s_best[PF_MAX_LM_ROWS];
  __shared__ int32_t s_argmax[PF_MAX_LM_ROWS];
  __shared__ int s_last;
  for (int i = threadIdx.x; i < PF_MAX_LM_ROWS; i += blockDim.x) s_best[i] = 0ull;
  pdl_wait();
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gw = blockIdx.x * (blockDim.x >> 5) + warp;
  const int nw = gridDim.x * (blockDim.x >> 5);
  for (int v = gw; v < a.V; v += nw) {
    const float* wrow = a.weight_f32 + (size_t)v * a.H;
    for (int t = 0; t < a.T; ++t) {
      const float* h = a.hidden_f32 + (size_t)t * a.H;
      float acc = 0.f;
      for (int c = lane; c < a.H; c += 32) acc = fmaf(h[c], wrow[c], acc);
#pragma unroll
      for (int off = 16; off; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
      if (lane == 0) atomicMax(&s_best[t], argmax_key(acc, (uint32_t)v));
    }
  }
  __syncthreads();
  pdl_launch_dependents();
  merge_and_finish(a, s_best, s_argmax, &s_last);
}

}  // namespace

int lmhead_bf16_smem_bytes(int npad, int stages) {
  return 1024 + stages * (kABytes + npad * 128) + (2 * kMaxStages + 4) * 8 + 8 +
         PF_MAX_LM_ROWS * 8 + PF_MAX_LM_ROWS * 4 + 16;
}

// Ring depth: as many stages as about 200 KB of shared memory holds (at
// most kMaxStages, at least 2); a caller's request (`want` > 0) overrides it
// within what the 227 KB per-CTA limit allows.
int lmhead_bf16_stages(int npad, int want) {
  const int stage = kABytes + npad * 128;
  int ns = (200 * 1024) / stage;
  if (want > 0) ns = want;
  if (ns > kMaxStages) ns = kMaxStages;
  while (ns > 2 && lmhead_bf16_smem_bytes(npad, ns) > 232448) --ns;
  if (ns < 2) ns = 2;
  return ns;
}

cudaError_t launch_lmhead_bf16(const LmArgs& a, const CUtensorMap& w_map,
                               const CUtensorMap& h_map, cudaStream_t s, int num_sms, bool pdl) {
  static DeviceMemo limit;
  const int smem = lmhead_bf16_smem_bytes(a.npad, a.stages);
  cudaError_t e = ensure_smem_limit((const void*)lmhead_tc_kernel, smem, limit);
  if (e != cudaSuccess) return e;
  const int grid = a.num_tiles < num_sms ? a.num_tiles : num_sms;
  return launch_ex(lmhead_tc_kernel, dim3(grid), dim3(kTcThreads), smem, s, 1, pdl, w_map, h_map,
                   a);
}

cudaError_t launch_lmhead_f32(const LmArgs& a, cudaStream_t s, int num_sms, bool pdl) {
  int grid = (a.V + 7) / 8;
  if (grid > 2 * num_sms) grid = 2 * num_sms;
  if (grid < 1) grid = 1;
  return launch_ex(lmhead_f32_kernel, dim3(grid), dim3(256), 0, s, 1, pdl, a);
}

}  // namespace pf
