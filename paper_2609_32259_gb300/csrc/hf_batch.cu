// hf_transfer_batch: several transfer directions (each its own plan: model
// pair, maps, alignment, caches) in one call.  Directions that share the
// dtype and the operand path run in ONE launch of the persistent kernel:
// its tiles are the concatenation of the directions' tiles and every role
// reads its tile's direction parameters, so short transfers (a few waves
// each) fill one another's tails.  Otherwise each direction's kernel goes to
// its own stream of a per-device pool, forked from and joined back into the
// caller's stream.
#include <mutex>
#include <string>

#include "hf_internal.h"

namespace hf {
namespace {

constexpr int kMaxDevices = 64;

struct StreamPool {
  bool ready = false;
  cudaStream_t streams[kMaxBatch] = {};
  cudaEvent_t fork = nullptr;
  cudaEvent_t join[kMaxBatch] = {};
};

std::mutex g_pool_mutex;
StreamPool g_pools[kMaxDevices];

hf_status get_pool(StreamPool** out) {
  int dev = 0;
  HF_CUDA_TRY(cudaGetDevice(&dev), "hf_transfer_batch: current device");
  if (dev < 0 || dev >= kMaxDevices) {
    set_error("hf_transfer_batch: device index out of range");
    return HF_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_pool_mutex);
  StreamPool& p = g_pools[dev];
  if (!p.ready) {
    for (int i = 0; i < kMaxBatch; ++i) {
      HF_CUDA_TRY(cudaStreamCreateWithFlags(&p.streams[i], cudaStreamNonBlocking), "batch stream");
      HF_CUDA_TRY(cudaEventCreateWithFlags(&p.join[i], cudaEventDisableTiming), "batch event");
    }
    HF_CUDA_TRY(cudaEventCreateWithFlags(&p.fork, cudaEventDisableTiming), "batch event");
    p.ready = true;
  }
  *out = &p;
  return HF_OK;
}

}  // namespace
}  // namespace hf

using namespace hf;

extern "C" hf_status hf_transfer_batch(const hf_plan* plans, const void* const* sender_kv,
                                       void* const* receiver_kv, int32_t n,
                                       hf_stream_t stream_) {
  if (n < 0 || n > kMaxBatch || (n > 0 && (!plans || !sender_kv || !receiver_kv))) {
    set_error("hf_transfer_batch: n must be in [0, 16] with non-null arrays");
    return HF_ERR_INVALID_ARGUMENT;
  }
  for (int i = 0; i < n; ++i) {
    const hf_plan p = plans[i];
    if (!p) {
      set_error("hf_transfer_batch: null plan");
      return HF_ERR_INVALID_ARGUMENT;
    }
    if (p->T_r > 0 && (!sender_kv[i] || !receiver_kv[i])) {
      set_error("hf_transfer_batch: null cache pointer");
      return HF_ERR_INVALID_ARGUMENT;
    }
    if ((reinterpret_cast<uintptr_t>(sender_kv[i]) | reinterpret_cast<uintptr_t>(receiver_kv[i]) |
         reinterpret_cast<uintptr_t>(p->desc.d_W)) & 15u) {
      set_error("hf_transfer_batch: caches and maps must be 16-byte aligned");
      return HF_ERR_INVALID_ARGUMENT;
    }
    for (int k = 0; k < i; ++k)
      if (plans[k] == p) {
        set_error("hf_transfer_batch: a plan appears twice in one batch");
        return HF_ERR_INVALID_ARGUMENT;
      }
  }
  if (n == 0) return HF_OK;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  if (n == 1) return launch_transfer(plans[0], sender_kv[0], receiver_kv[0], stream);
  if (batch_compatible(plans, n))
    return launch_transfer_batch(plans, sender_kv, receiver_kv, n, stream);
  StreamPool* pool = nullptr;
  hf_status s = get_pool(&pool);
  if (s != HF_OK) return s;
  // One batch at a time per device uses the pool: the fork/join events are
  // recorded and waited on within this call, under the lock.
  std::lock_guard<std::mutex> lock(g_pool_mutex);
  HF_CUDA_TRY(cudaEventRecord(pool->fork, stream), "hf_transfer_batch: record");
  // Directions already launched are joined back into `stream` even when a
  // later one fails, so the caller's stream never runs ahead of kernels that
  // still use its caches.
  int launched = 0;
  for (int i = 0; i < n && s == HF_OK; ++i) {
    cudaError_t e = cudaStreamWaitEvent(pool->streams[i], pool->fork, 0);
    if (e != cudaSuccess) {
      s = cuda_fail(e, "hf_transfer_batch: wait");
      break;
    }
    s = launch_transfer(plans[i], sender_kv[i], receiver_kv[i], pool->streams[i]);
    launched = i + 1;  // a failed launch may still have queued nothing; joining it is harmless
  }
  for (int i = 0; i < launched; ++i) {
    cudaError_t e = cudaEventRecord(pool->join[i], pool->streams[i]);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, pool->join[i], 0);
    if (e != cudaSuccess && s == HF_OK) s = cuda_fail(e, "hf_transfer_batch: join");
  }
  return s;
}
