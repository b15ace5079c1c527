// pf_lmhead_accept_noalloc: pf_lmhead_accept with its scratch memory held in
// a fixed, file-scope device array instead of a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they verify
// a proposal: plug-ins whose host framework owns every device allocation
// (they get tensors handed to them and have no allocator of their own), and
// latency-critical decode loops that must never reach an allocator, which
// can synchronise the device or fail under memory pressure.  This entry
// point needs no workspace argument: the LM head's scratch (one packed
// maximum per proposal row and a completion ticket, kLmWorkspaceBytes =
// 2112 bytes, enough for PF_MAX_LM_ROWS = 256 rows) lives in g_lm_scratch
// below, which every GPU that loads this library holds until the process
// exits.
#include <cuda_runtime.h>

#include <mutex>

#include "pf_internal.h"

namespace {

__device__ __align__(256) unsigned char g_lm_scratch[pf::kLmWorkspaceBytes];

std::mutex g_mu;
void* g_scratch_ptr[64] = {};

}  // namespace

extern "C" PF_API pf_status pf_lmhead_accept_noalloc(const pf_lm_desc* d, void* stream) {
  static const char* who = "pf_lmhead_accept_noalloc";
  // Every argument check comes first, so that a rejected call queues
  // nothing; the scratch's capacity first of all, with its own message.
  if (d && d->total_nodes > PF_MAX_LM_ROWS)
    return pf::set_error(PF_ERR_SHAPE,
                         "%s: total_nodes = %d exceeds the %d rows its fixed %zu-byte scratch "
                         "holds",
                         who, d->total_nodes, PF_MAX_LM_ROWS, pf::kLmWorkspaceBytes);
  const pf_status chk = pf::lmhead_check_desc(d, who);
  if (chk != PF_OK) return chk;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return pf::set_error(PF_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return pf::set_error(PF_ERR_CUDA, "%s: device %d >= 64", who, dev);
  void* ptr = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
      // In host code g_lm_scratch names a host-side stand-in, not the
      // device array: its device address is looked up once per device,
      // with that device current, and kept for the life of the process.
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_lm_scratch);
      if (e != cudaSuccess || !p)
        return pf::set_error(PF_ERR_CUDA, "%s: cudaGetSymbolAddress: %s", who,
                             cudaGetErrorString(e));
      g_scratch_ptr[dev] = p;
    }
    ptr = g_scratch_ptr[dev];
  }
  // Every call shares the array and it keeps the last call's contents:
  // clear it so this call starts from zero.
  e = cudaMemsetAsync(ptr, 0, pf::kLmWorkspaceBytes, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess)
    return pf::set_error(PF_ERR_CUDA, "%s: clearing the scratch: %s", who, cudaGetErrorString(e));
  return pf_lmhead_accept(d, ptr, pf::kLmWorkspaceBytes, stream);
}
