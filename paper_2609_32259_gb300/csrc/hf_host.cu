// hf_transfer_host: one transfer whose sender and receiver caches live in
// page-locked host memory.  The receiver layers are split into groups; the
// sender layers a group reads are brought in, the group's layers are
// computed on the caller's stream, and the finished receiver layers are
// copied out (a copy engine) while later groups are still being brought in
// and computed.  When every alignment row is one sender token (Token
// Alignment, same-index) only the referenced sender rows are read: a small
// gather kernel reads them from the mapped host memory (about a quarter of
// the sender cache for Token Alignment); otherwise whole layers are copied.
#include <algorithm>
#include <cstring>
#include <string>

#include "hf_internal.h"

namespace hf {
namespace {

hf_status require_pinned(const void* ptr, const char* what, const void** dev_alias = nullptr) {
  cudaPointerAttributes a;
  std::memset(&a, 0, sizeof(a));
  const cudaError_t e = cudaPointerGetAttributes(&a, ptr);
  if (e != cudaSuccess) return cuda_fail(e, "hf_transfer_host: pointer attributes");
  if (a.type != cudaMemoryTypeHost) {
    set_error(std::string("hf_transfer_host: ") + what + " is not page-locked host memory");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (dev_alias) *dev_alias = a.devicePointer;
  return HF_OK;
}

// Copies the referenced sender rows (ucol[0 .. U), U read on the device) of
// sender layers [t0, t1), both roles, from mapped host memory into the same
// rows of the device sender cache: 16 bytes per thread, one row's chunks on
// consecutive threads.
__global__ void __launch_bounds__(128) gather_sender_rows(const uint4* __restrict__ src,
                                                          uint4* __restrict__ dst,
                                                          const int32_t* __restrict__ ucol,
                                                          const int32_t* __restrict__ n_distinct,
                                                          int t0, int t1, int64_t s_rows,
                                                          int chunks) {
  const int64_t U = *n_distinct;
  const int64_t total = static_cast<int64_t>(t1 - t0) * 2 * U * chunks;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t rest = i / chunks;
    const int64_t ch = i - rest * chunks;
    const int64_t lcs = rest / U;             // (t - t0) * 2 + c
    const int64_t u = rest - lcs * U;
    const int64_t row = (2 * static_cast<int64_t>(t0) + lcs) * s_rows + ucol[u];
    dst[row * chunks + ch] = src[row * chunks + ch];
  }
}

// The plan's two copy streams (created on first use, on the current device)
// and at least n events.
hf_status ensure_aux(hf_plan_s* p, int n) {
  int dev = 0;
  HF_CUDA_TRY(cudaGetDevice(&dev), "hf_transfer_host: current device");
  if (p->s_h2d && p->aux_device != dev) {
    set_error("hf_transfer_host: the plan's copy streams belong to another device");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (!p->s_h2d) {
    HF_CUDA_TRY(cudaStreamCreateWithFlags(&p->s_h2d, cudaStreamNonBlocking), "copy stream");
    HF_CUDA_TRY(cudaStreamCreateWithFlags(&p->s_d2h, cudaStreamNonBlocking), "copy stream");
    p->aux_device = dev;
  }
  if (p->n_events < n) {
    cudaEvent_t* ev = new cudaEvent_t[n];
    for (int i = 0; i < p->n_events; ++i) ev[i] = p->events[i];
    for (int i = p->n_events; i < n; ++i) {
      const cudaError_t e = cudaEventCreateWithFlags(&ev[i], cudaEventDisableTiming);
      if (e != cudaSuccess) {
        for (int k = p->n_events; k < i; ++k) cudaEventDestroy(ev[k]);
        delete[] ev;
        return cuda_fail(e, "hf_transfer_host: event");
      }
    }
    delete[] p->events;
    p->events = ev;
    p->n_events = n;
  }
  return HF_OK;
}

}  // namespace
}  // namespace hf

using namespace hf;

extern "C" hf_status hf_transfer_host(hf_plan plan, const void* h_sender_kv, void* d_sender_kv,
                                      void* d_receiver_kv, void* h_receiver_kv,
                                      int32_t n_groups, hf_stream_t stream_) {
  if (!plan) {
    set_error("hf_transfer_host: null plan");
    return HF_ERR_INVALID_ARGUMENT;
  }
  const hf_plan_desc& d = plan->desc;
  if (n_groups < 0 || n_groups > d.L_r) {
    set_error("hf_transfer_host: n_groups must be in [0, L_r]");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (plan->T_r == 0) return HF_OK;
  if (!h_sender_kv || !d_sender_kv || !d_receiver_kv) {
    set_error("hf_transfer_host: null cache pointer");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if ((reinterpret_cast<uintptr_t>(d_sender_kv) | reinterpret_cast<uintptr_t>(d_receiver_kv) |
       reinterpret_cast<uintptr_t>(d.d_W)) & 15u) {
    set_error("hf_transfer_host: device caches and maps must be 16-byte aligned");
    return HF_ERR_INVALID_ARGUMENT;
  }
  const void* h_sender_dev = nullptr;  // the sender cache as the device addresses it
  hf_status s = require_pinned(h_sender_kv, "h_sender_kv", &h_sender_dev);
  if (s != HF_OK) return s;
  const size_t row_bytes = static_cast<size_t>(plan->d_s) * (d.dtype == HF_BF16 ? 2 : 4);
  const bool gather = plan->gather && h_sender_dev != nullptr && row_bytes % 16 == 0 &&
                      (reinterpret_cast<uintptr_t>(h_sender_dev) & 15u) == 0;
  const int32_t* ucol = reinterpret_cast<const int32_t*>(plan->ws + plan->lay.ucol);
  const int32_t* n_distinct = reinterpret_cast<const int32_t*>(plan->ws + plan->lay.n_distinct);
  const bool copy_out = h_receiver_kv != nullptr;  // NULL: the cache stays on the device
  if (copy_out && (s = require_pinned(h_receiver_kv, "h_receiver_kv")) != HF_OK) return s;
  // default: one group per receiver layer (the copy out of a layer starts as
  // soon as it is computed; measured best on a 40-layer, 32K-token transfer)
  const int G = n_groups == 0 ? d.L_r : n_groups;
  s = ensure_aux(plan, 2 * G + 2);
  if (s != HF_OK) return s;

  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  const size_t esize = d.dtype == HF_BF16 ? 2 : 4;
  const size_t sender_layer = 2 * static_cast<size_t>(plan->s_rows) * plan->d_s * esize;
  const int64_t recv_rows = d.paged ? static_cast<int64_t>(d.n_blocks) * d.block_size : plan->T_r;
  const size_t recv_layer = 2 * static_cast<size_t>(recv_rows) * plan->d_r * esize;
  const char* hs = static_cast<const char*>(h_sender_kv);
  char* ds = static_cast<char*>(d_sender_kv);
  char* dr = static_cast<char*>(d_receiver_kv);
  char* hr = static_cast<char*>(h_receiver_kv);
  cudaEvent_t* ev = plan->events;
  cudaEvent_t ev_start = ev[0], ev_done = ev[1];

  // nothing is overwritten before the caller's earlier work on `stream`
  HF_CUDA_TRY(cudaEventRecord(ev_start, stream), "hf_transfer_host: record");
  HF_CUDA_TRY(cudaStreamWaitEvent(plan->s_h2d, ev_start, 0), "hf_transfer_host: wait");
  HF_CUDA_TRY(cudaStreamWaitEvent(plan->s_d2h, ev_start, 0), "hf_transfer_host: wait");
  int copied = 0;  // sender layers [0, copied) are on their way to the device
  for (int g = 0; g < G; ++g) {
    const int l0 = static_cast<int>(static_cast<int64_t>(g) * d.L_r / G);
    const int l1 = static_cast<int>(static_cast<int64_t>(g + 1) * d.L_r / G);
    int need = 0;
    for (int l = l0; l < l1; ++l) need = std::max(need, plan->max_sender_layer[l] + 1);
    if (need > copied) {
      if (gather) {
        // small blocks at few registers: the gather of group g + 1 runs
        // wherever an SM frees up (the transfer kernel's CTAs hold the whole
        // register file while they run), ahead of the group's own kernel
        gather_sender_rows<<<4 * device_sm_count(), 128, 0, plan->s_h2d>>>(
            static_cast<const uint4*>(h_sender_dev), reinterpret_cast<uint4*>(ds), ucol,
            n_distinct, copied, need, plan->s_rows, static_cast<int>(row_bytes / 16));
        HF_CUDA_TRY(cudaGetLastError(), "hf_transfer_host: sender gather");
      } else {
        HF_CUDA_TRY(cudaMemcpyAsync(ds + copied * sender_layer, hs + copied * sender_layer,
                                    (need - copied) * sender_layer, cudaMemcpyHostToDevice,
                                    plan->s_h2d),
                    "hf_transfer_host: sender copy");
      }
      copied = need;
    }
    cudaEvent_t ev_in = ev[2 + 2 * g], ev_out = ev[3 + 2 * g];
    HF_CUDA_TRY(cudaEventRecord(ev_in, plan->s_h2d), "hf_transfer_host: record");
    HF_CUDA_TRY(cudaStreamWaitEvent(stream, ev_in, 0), "hf_transfer_host: wait");
    s = launch_transfer(plan, d_sender_kv, d_receiver_kv, stream, l0, l1);
    if (s != HF_OK) return s;
    if (copy_out) {
      HF_CUDA_TRY(cudaEventRecord(ev_out, stream), "hf_transfer_host: record");
      HF_CUDA_TRY(cudaStreamWaitEvent(plan->s_d2h, ev_out, 0), "hf_transfer_host: wait");
      HF_CUDA_TRY(cudaMemcpyAsync(hr + l0 * recv_layer, dr + l0 * recv_layer,
                                  (l1 - l0) * recv_layer, cudaMemcpyDeviceToHost, plan->s_d2h),
                  "hf_transfer_host: receiver copy");
    }
  }
  // `stream` is ordered after the last copy out
  HF_CUDA_TRY(cudaEventRecord(ev_done, plan->s_d2h), "hf_transfer_host: record");
  HF_CUDA_TRY(cudaStreamWaitEvent(stream, ev_done, 0), "hf_transfer_host: wait");
  return HF_OK;
}
