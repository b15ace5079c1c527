// Internal interface between the C-ABI layer (api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <atomic>
#include <utility>

#include "pf_verify.h"

namespace pf {

// ------------------------------------------------------------ attention
struct AttnArgs {
  int B, Hq, Hkv, D, G;
  int T, max_nodes, max_prefix;
  int bm;          // query rows per CTA (bf16: 32, 64 or 128)
  int nb;          // proposal nodes per row block (bf16: floor(bm / G))
  int rb_count;    // row blocks per (sequence, KV head)
  int splits;      // CTAs of one cluster, each taking a slice of the KV tiles
  int flags;       // PF_ATTN_* flags
  // Balanced batch mode (tcgen05 kernel, splits == 1, no cluster): `items`
  // CTAs share the groups' tiles in proportion to their lengths (see
  // balanced_plan); a group spread over several CTAs leaves normalised
  // partials in `ws` ([items][bm][D + 8] halves) for the combine kernel.
  int items;       // 0 = off
  // partial slots per item: 1 (tc64: one group part per CTA) or 2 (the pair
  // kernel's continuous split: an item's first and last group piece)
  int slots;
  // two-block kernel: 1 = the CTAs follow a TeamPlan (teams of a cluster's
  // CTAs per group) instead of one group per cluster; team_ctas = its CTAs
  // (a multiple of the cluster size a.splits)
  int team;
  int team_ctas;
  void* ws;
  // this call's epoch for the group tickets of the kernels that merge their
  // own pieces (see group_tickets): distinct for every call, < 2^40
  unsigned long long epoch;
  float scale_log2;  // softmax scale * log2(e)
  float scale;
  const int32_t* cu_nodes;
  const int32_t* prefix_len;
  const uint64_t* mask;
  void* out;
  int layout;
  int max_seq;
  const int32_t* page_table;
  int pages_per_seq;
  int num_pages;
  int32_t* err;
  // raw pointers (fp32 path; the bf16 path reads through tensor maps)
  const void* q;
  const void* tk;
  const void* tv;
  const void* ck;
  const void* cv;
};

struct AttnMaps {
  CUtensorMap q, tk, tv, ck, cv;
  // paged cache only: V of one (page, KV head) as a 5-D map (64 columns, 16
  // rows, the two 64-column halves, head, page), so that one box brings both
  // halves of a page in [half][row][column] order
  CUtensorMap cv_page;
};

cudaError_t launch_attention_bf16(const AttnArgs& a, const AttnMaps& m, cudaStream_t s,
                                  int num_sms, bool pdl);
cudaError_t launch_attention_f32(const AttnArgs& a, cudaStream_t s, bool pdl);
int attention_bf16_smem_bytes(int D, int bm);
// Whether a cluster of `cluster` CTAs of the bf16 attention kernel can be
// resident at once on this device.
bool attention_cluster_fits(int D, int bm, int cluster);
// tcgen05 variant (bf16, D = 128, a.bm = 128 or 256 query rows per CTA).
cudaError_t launch_attention_tc(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl);
// tcgen05 variant with 128-token K/V tiles and P in tensor memory (bf16,
// D = 128, a.bm = 128); its tensor maps hold 128-row cache boxes and
// 128-node proposal boxes.  Cluster split-KV (a.items = 0), or with
// `balanced` one CTA per item (a.items = SMs, a.slots = 1, no cluster):
// groups spread over CTAs in proportion to their tiles (balanced_plan), the
// last piece of a group to finish merging the pieces' partials from the
// workspace (group tickets, a.epoch); no combine kernel.
cudaError_t launch_attention_tc2(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl,
                                 int stages, bool balanced);
int attention_tc2_max_active_clusters(int cluster, int stages);
// tcgen05 variant with 128-token K/V tiles and two 128-row blocks per CTA
// (bf16, D = 128, a.bm = 256, a.nb = 2 * floor(128 / G) nodes per CTA),
// cluster split-KV over a.splits CTAs; needs the 128-token tensor maps and,
// for a paged cache, m.cv_page.
// The two-block kernel's team plan: CTA x works on piece part of the
// nparts pieces of group `group`, whose pieces are the CTAs base ..
// base + nparts - 1 of x's cluster (cluster ranks); nparts = 0: no work.
// Packed as group | part << 12 | nparts << 17 | base << 22.
constexpr int kTeamMaxCtas = 160;
struct TeamPlan {
  uint32_t e[kTeamMaxCtas];
};
__host__ __device__ constexpr uint32_t team_entry(int group, int part, int nparts, int base) {
  return (uint32_t)group | (uint32_t)part << 12 | (uint32_t)nparts << 17 | (uint32_t)base << 22;
}
cudaError_t launch_attention_2blk(const AttnArgs& a, const AttnMaps& m, const TeamPlan& tp,
                                  cudaStream_t s, bool pdl);
int attention_2blk_max_active_clusters(int cluster);
// tcgen05 variant on SM pairs (2-SM MMA, M = 256 rows per pair, 128-token
// tiles; bf16, D = 128): a.bm = 256, a.nb = 2 * floor(128 / G) nodes per
// pair, a.items pairs sharing all groups' tiles in equal contiguous ranges
// (a.slots = 2; needs the workspace and the combine kernel).  Tensor maps:
// K boxes of 64 rows, V boxes of 128 rows (cache), tree K boxes of 64
// nodes, tree V boxes of 128, Q boxes of a.nb / 2 nodes.
cudaError_t launch_attention_pair(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl);
// 128-token, P-in-TMEM kernel (one CTA per SM, 128 query rows, bf16,
// D = 128) with the continuous split: a.items = SMs, a.bm = 128, a.slots =
// 2, at most kSkMaxGroups groups; needs the workspace and the combine
// kernel.  Tensor maps as attn_tc2_kernel's.
constexpr int kSkMaxGroups = 128;
cudaError_t launch_attention_sk(const AttnArgs& a, const AttnMaps& m, cudaStream_t s, bool pdl);
// Merge of the balanced batch mode's partials (launched after the tcgen05
// kernel when a.items > 0).
cudaError_t launch_attention_combine(const AttnArgs& a, cudaStream_t s, bool pdl);
// Groups (sequence, KV head, row block) the balanced batch mode's plan can
// hold (8 per lane of a warp).
constexpr int kPlanMaxGroups = 256;
// Bytes of a.ws for the balanced batch mode with `items` work items of a.bm
// rows and `slots` partial slots per item: the partials, the plan table
// (kPlanMaxGroups int4) and the group tickets (kPlanMaxGroups u64).
size_t attention_balanced_ws_bytes(int items, int bm, int D, int slots = 1);
// How many clusters of `cluster` CTAs of the tcgen05 kernel fit at once.
// rows_per_cta: 128 (one softmax warpgroup) or 256 (two).
int attention_tc_max_active_clusters(int cluster, int rows_per_cta);
int attention_tc_smem_bytes();

// ------------------------------------------------------------ LM head
struct LmArgs {
  int T, H, V, B, max_nodes;
  int npad;        // T rounded up to a multiple of 16 (UMMA N)
  int num_tiles;   // ceil(V / 128)
  int nk;          // ceil(H / 64)
  int stages;      // TMA pipeline depth
  int flags;       // PF_LM_* flags
  const int32_t* cu_nodes;
  const int32_t* tokens;
  const int32_t* parent;
  int32_t* argmax;
  float* max_logit;
  int32_t* accept_len;
  int32_t* path;
  int32_t* out_tokens;
  int32_t* last_node;
  unsigned long long* best;  // workspace [PF_MAX_LM_ROWS]
  unsigned int* ticket;      // workspace
  int32_t* err;
  const float* hidden_f32;
  const float* weight_f32;
};

cudaError_t launch_lmhead_bf16(const LmArgs& a, const CUtensorMap& w_map,
                               const CUtensorMap& h_map, cudaStream_t s, int num_sms, bool pdl);
cudaError_t launch_lmhead_f32(const LmArgs& a, cudaStream_t s, int num_sms, bool pdl);
int lmhead_bf16_stages(int npad, int want);
int lmhead_bf16_smem_bytes(int npad, int stages);

constexpr size_t kLmWorkspaceBytes = 8 * PF_MAX_LM_ROWS + 64;

// ------------------------------------------------------------ device tree prepare
struct TreeArgs {
  int B, T, max_nodes;
  const int32_t* parent;
  const int32_t* cu_nodes;
  int32_t* depth;
  uint64_t* mask;
  int32_t* err;
};

cudaError_t launch_tree_prepare(const TreeArgs& a, cudaStream_t s, bool pdl);

// ------------------------------------------------------------ commit
struct CommitArgs {
  int B, L, Hkv, row_bytes, max_nodes, T;
  const int32_t* cu_nodes;
  const int32_t* prefix_len;
  const int32_t* accept_len;
  const int32_t* path;
  const char* tree_k;
  const char* tree_v;
  long long tree_layer_bytes;
  char* cache_k;
  char* cache_v;
  long long cache_layer_bytes;
  int layout;
  int max_seq;
  const int32_t* page_table;
  int pages_per_seq;
  int num_pages;
  int32_t* new_len;
  int32_t* err;
};

cudaError_t launch_kv_commit(const CommitArgs& a, cudaStream_t s, int num_sms, bool pdl);

// ------------------------------------------------------------ KV shift
struct ShiftArgs {
  int L, Hkv, row_bytes, elem_bytes;
  int seq, src, dst, count;
  int overlap;     // spans overlap: one CTA per (layer, head) walks every pass
  int descending;  // move to higher positions: passes run from the end
  int layout, max_seq, pages_per_seq, num_pages;
  const int32_t* page_table;
  char* cache_k;
  char* cache_v;
  long long layer_bytes;
  int32_t* err;
  float2 cs[128];  // cos / sin of shift * theta_i, i < D/2 (host, double precision)
};

cudaError_t launch_kv_shift(const ShiftArgs& a, cudaStream_t s, int num_sms, bool pdl);

// ------------------------------------------------------------ retrieval
constexpr int kRetrievalMaxBlocks = 1024;
// workspace: [0, 1024) z floats | [1024, 1040) key ticket |
// [1088, 1088 + 16 * kRetrievalMaxBlocks) per-CTA winners | then scan ticket
constexpr size_t kRetrievalZOff = 0;
constexpr size_t kRetrievalKeyTicketOff = 1024;
constexpr size_t kRetrievalBestOff = 1088;
constexpr size_t kRetrievalScanTicketOff = kRetrievalBestOff + 16 * kRetrievalMaxBlocks;
constexpr size_t kRetrievalWsBytes = kRetrievalScanTicketOff + 64;

struct KeyArgs {
  int H, bf16;
  int vec;  // rows and pointers allow 16-byte loads
  const void* hidden;
  const void* proj;
  int8_t* key_out;
  float* z;
  unsigned int* ticket;
  int32_t* err;
};

struct RetrievalArgs {
  int lo, hi, token;
  const int8_t* query_key;
  const int8_t* keys;
  const int32_t* entry_token;
  const int32_t* entry_pos;
  const int32_t* entry_bound;
  int32_t* best;
  float* similarity;
  int4* block_best;
  unsigned int* ticket;
  int32_t* err;
};

cudaError_t launch_retrieval_key(const KeyArgs& a, cudaStream_t s, bool pdl);
cudaError_t launch_retrieve(const RetrievalArgs& a, cudaStream_t s, int num_sms, bool pdl);

// ------------------------------------------------------------ prefix carryover
struct PrefixArgs {
  const int32_t* prev;
  const int32_t* next;
  int n_prev, n_next;
  int vec;  // both arrays 16-byte aligned
  int32_t* lcp;
  int32_t* cache_len;
};

cudaError_t launch_prefix_match(const PrefixArgs& a, cudaStream_t s, bool pdl);

cudaError_t launch_selftest_wait(int32_t* err, unsigned long long limit_ns, int signal,
                                 int32_t* waited_ok, cudaStream_t s);

// pf_lmhead_accept's argument checks that do not involve the workspace.
pf_status lmhead_check_desc(const pf_lm_desc* d, const char* who);

// Record the message pf_last_error() returns on this thread; returns s.
pf_status set_error(pf_status s, const char* fmt, ...);

// Raise a kernel's dynamic shared-memory limit once per device (never while
// a stream is being captured after the first call on that device).
// Per-device memo of one int (0: not yet known), safe to read and fill
// from several host threads at once (a racing fill stores the same value).
struct DeviceMemo {
  std::atomic<int> v[64];
  int get(int dev) const {
    return dev >= 0 && dev < 64 ? v[dev].load(std::memory_order_acquire) : 0;
  }
  void set(int dev, int x) {
    if (dev >= 0 && dev < 64) v[dev].store(x, std::memory_order_release);
  }
};

inline cudaError_t ensure_smem_limit(const void* func, int bytes, DeviceMemo& per_device) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (per_device.get(dev) >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) per_device.set(dev, bytes);
  return e;
}

// Allow cluster sizes above 8 for a kernel, once per device.
inline cudaError_t ensure_nonportable_cluster(const void* func, DeviceMemo& per_device) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (per_device.get(dev)) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess) per_device.set(dev, 1);
  return e;
}

// Shared launch helper: optional cluster dimension and programmatic
// dependent launch.
template <typename... KArgs, typename... Args>
cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                      cudaStream_t s, int cluster_x, bool pdl, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attrs[2];
  int na = 0;
  if (cluster_x > 1) {
    attrs[na].id = cudaLaunchAttributeClusterDimension;
    attrs[na].val.clusterDim.x = cluster_x;
    attrs[na].val.clusterDim.y = 1;
    attrs[na].val.clusterDim.z = 1;
    ++na;
  }
  if (pdl) {
    attrs[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attrs[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attrs;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace pf
