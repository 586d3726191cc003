// cmsd_confidence_verify_static: the fused pass with its scratch in a fixed
// array of the library's device image instead of a caller workspace.
//
// For callers that cannot allocate device memory when they make the call: a
// serving loop that divides all of HBM once at start-up (weights, KV cache,
// activations) and treats any later allocation as a failure, or a plain C
// caller without an allocator of its own.  The call allocates nothing; the
// scratch below is part of the loaded module, one copy per device.
#include <cuda_runtime.h>
#include <stdint.h>

#include <map>
#include <mutex>

#include "cmsd.h"
#include "cmsd_internal.h"

namespace {

// The scratch of every call on one device.  Zero-filled at the start of each
// call (only the bytes the call's layout uses), so no state carries over.
static __device__ __align__(256) unsigned char g_scratch[CMSD_STATIC_SCRATCH_BYTES];

std::mutex g_mu;
std::map<int, void*> g_addr;   // device -> device address of g_scratch

// One-time set-up per device, with that device current: look up the address
// of the scratch array in this device's copy of the module.
int scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return CMSD_ECUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_addr.find(dev);
  if (it == g_addr.end()) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess || p == nullptr) return CMSD_ECUDA;
    it = g_addr.emplace(dev, p).first;
  }
  *out = it->second;
  return CMSD_OK;
}

}  // namespace

extern "C" int cmsd_confidence_verify_static(
    const void* draft_logits, const void* target_logits, const int32_t* draft_tokens,
    const int32_t* k_row, int B, int K, int V, int dtype, const cmsd_params* p, uint64_t seed,
    uint32_t iteration, float* H, float* margin, int32_t* argmax, float* conf, float* lse,
    int32_t* k_next, int32_t* n_accept, int32_t* out_tokens, uint8_t* accept, void* stream) {
  // every argument check first: an invalid call enqueues nothing
  int rc = cmsd::validate_fused(draft_logits, target_logits, draft_tokens, k_row, B, K, V, dtype, p,
                                n_accept, out_tokens);
  if (rc) return rc;
  if (B == 0 || K == 0) return CMSD_OK;
  const size_t need = cmsd_workspace_bytes(B, K, V);
  if (need == 0) return CMSD_ECUDA;
  if (need > (size_t)CMSD_STATIC_SCRATCH_BYTES) return CMSD_ESCRATCH;
  void* ws = nullptr;
  rc = scratch_address(&ws);
  if (rc) return rc;
  if (cudaMemsetAsync(ws, 0, need, (cudaStream_t)stream) != cudaSuccess) return CMSD_ECUDA;
  return cmsd_confidence_verify(draft_logits, target_logits, draft_tokens, k_row, B, K, V, dtype,
                                p, seed, iteration, H, margin, argmax, conf, lse, k_next, n_accept,
                                out_tokens, accept, ws, need, stream);
}
