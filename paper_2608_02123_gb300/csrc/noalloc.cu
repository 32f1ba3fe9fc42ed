// pctree_draft_noalloc: a drafting round whose scratch memory lives in a
// fixed array inside this library instead of a workspace the caller
// allocates.
//
// Some callers cannot allocate device memory when they draft: code that runs
// inside a host framework that owns a fixed memory budget and forbids side
// allocations, plug-ins that only receive the buffers their host hands them,
// and latency-critical serving loops where cudaMalloc / cudaFree would
// synchronise the device.  Those callers still pass the round's inputs and
// output tensors; the scratch comes from kStaticScratchBytes of memory that
// every GPU which loads this library reserves until the process exits.
//
// Set-up: the first call on a device (with that device current) looks up the
// array's device address with cudaGetSymbolAddress and caches it; make that
// first call before any stream capture begins.  Later calls only read the
// cache.
//
// Sharing: every call on a device uses the same array, which keeps whatever
// the previous call left in it.  pctree_draft clears the parts that must
// start at zero (status word, stage counters and flags) at the start of each
// round.  Calls whose work overlaps on the GPU -- on different streams, or
// from different host threads -- race on the array and must not be issued.
#include <mutex>

#include "pctree_common.cuh"

namespace pct {
namespace {

// 16 MiB: enough for batch-1 Qwen3-shaped rounds (pctree_workspace_bytes is
// 4.74 MB for V=151936, H=2560, B=16, k=8, N=64 and 5.54 MB for V=151936,
// H=5120, B=16, k=16, N=128); larger rounds are rejected.
constexpr size_t kStaticScratchBytes = size_t(16) << 20;

static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of the array on the current device (looked up once).
pctree_status static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return PCTREE_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr)
      return PCTREE_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return PCTREE_OK;
}

}  // namespace
}  // namespace pct

extern "C" {

pctree_status pctree_draft_noalloc(const pctree_config* cfg,
                                   const float* base_logits,
                                   const void* head_emb, const void* head_out,
                                   const int32_t* root_token,
                                   const pctree_tree* out, void* stream) {
  pctree_status st = pctree_check_config(cfg);
  if (st != PCTREE_OK) return st;
  if (pctree_workspace_bytes(cfg) > pct::kStaticScratchBytes)
    return PCTREE_ERR_WORKSPACE;   // round too large for the fixed array
  void* scratch = nullptr;
  st = pct::static_scratch(&scratch);
  if (st != PCTREE_OK) return st;
  return pctree_draft(cfg, base_logits, head_emb, head_out, root_token, out,
                      scratch, pct::kStaticScratchBytes, stream);
}

}  // extern "C"
