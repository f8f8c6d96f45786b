// hf_transfer_noalloc: a transfer whose per-transfer metadata lives in a
// fixed device array owned by the library instead of a caller workspace.
//
// For callers that cannot allocate device memory per call: code that runs
// inside a host framework owning every device allocation (an inference
// server or plugin that hands in only the caches), code with a fixed memory
// budget that must not grow, or a caller that has no allocator handle at
// the point where the transfer is issued.
//
// The scratch is a file-scope __device__ array, so every GPU that loads the
// library holds kNoAllocScratchBytes of it until the process exits.  Host
// code may not use the array's name as a device address (it names a host
// shadow); the device address comes from cudaGetSymbolAddress, fetched once
// per device with that device current.
#include <mutex>
#include <string>

#include "hf_internal.h"

namespace hf {
namespace {

constexpr size_t kNoAllocScratchBytes = 8u << 20;  // 8 MiB: ~340K receiver tokens
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_scratch_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch on the current device (looked up once).
hf_status scratch_for_current_device(void** out) {
  int dev = 0;
  HF_CUDA_TRY(cudaGetDevice(&dev), "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) {
    set_error("hf_transfer_noalloc: device ordinal out of range");
    return HF_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "hf_transfer_noalloc: cudaGetSymbolAddress");
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return HF_OK;
}

}  // namespace
}  // namespace hf

extern "C" hf_status hf_transfer_noalloc(const hf_plan_desc* desc, const void* sender_kv,
                                         void* receiver_kv, hf_stream_t stream) {
  using namespace hf;
  size_t need = 0;
  hf_status s = hf_plan_workspace_size(desc, &need);
  if (s != HF_OK) return s;
  if (need > kNoAllocScratchBytes) {
    set_error("hf_transfer_noalloc: this transfer needs " + std::to_string(need) +
              " bytes of metadata but the built-in scratch holds " +
              std::to_string(kNoAllocScratchBytes) +
              " bytes (about 340K receiver tokens); use hf_plan_create with a workspace");
    return HF_ERR_UNSUPPORTED;
  }
  // the cache checks come before any work is queued: a rejected call leaves
  // the shared scratch untouched (desc and its r_tok_ptr were checked above)
  if (desc->r_tok_ptr[desc->n_req] > 0 && (!sender_kv || !receiver_kv)) {
    set_error("hf_transfer_noalloc: null cache pointer");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if ((reinterpret_cast<uintptr_t>(sender_kv) | reinterpret_cast<uintptr_t>(receiver_kv) |
       reinterpret_cast<uintptr_t>(desc->d_W)) & 15u) {
    set_error("hf_transfer_noalloc: caches and maps must be 16-byte aligned");
    return HF_ERR_INVALID_ARGUMENT;
  }
  void* ws = nullptr;
  s = scratch_for_current_device(&ws);
  if (s != HF_OK) return s;
  // plan state on the host stack: the call allocates no memory of any kind
  hf_plan_s plan{};
  PlanTables tables;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  s = plan_build(desc, ws, kNoAllocScratchBytes, st, &plan, &tables);
  if (s != HF_OK) return s;
  return launch_transfer(&plan, sender_kv, receiver_kv, st);
}
