// hf_align_build: the alignment CSR from character-end offsets.
//
// Token Alignment (Section 3.1 "Token and Layer Alignment", Appendix B.1):
// receiver token j takes the sender token ending at the latest shared
// character-end boundary at or before its own end, and the request's first
// sender token before the first shared boundary.  On the device this is
//   1. a match pass: a binary search of each receiver end among the request's
//      sender ends gives the global index of the sender token ending there,
//      or -1; each request's first receiver token gets at least the
//      request's first sender index;
//   2. an inclusive max-scan over all receiver tokens.  Global sender
//      indices grow with the request and with the boundary, so the running
//      maximum is the latest match of the current request (or its first
//      sender token).
// Overlap mean pooling counts the overlapping sender tokens of every
// receiver span with two binary searches, sums the counts into row
// pointers, and fills columns and fp32 weights 1/n.
#include <algorithm>

#include "hf_device.cuh"
#include "hf_internal.h"
#include "hf_scan.cuh"

namespace hf {
namespace {

struct ReqPtrs {
  int32_t n_req;
  int32_t s_ptr[kMaxReq + 1];
  int32_t r_ptr[kMaxReq + 1];
};

constexpr int kThreads = 256;

__device__ __forceinline__ void flag(int32_t* info, int bits) { atomicOr(info + 1, bits); }

// Sender ends must be positive and strictly increasing within a request.
__global__ void check_sender_kernel(ReqPtrs rq, const int32_t* __restrict__ s_end, int64_t T_s,
                                    int32_t* info) {
  __shared__ int32_t sp[kMaxReq + 1];
  for (int i = threadIdx.x; i <= rq.n_req; i += blockDim.x) sp[i] = rq.s_ptr[i];
  __syncthreads();
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < T_s;
       k += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(sp, rq.n_req, k);
    const int32_t prev = (k > sp[q]) ? s_end[k - 1] : 0;
    if (s_end[k] <= prev) flag(info, HF_CHECK_BAD_OFFSETS);
  }
}

// Checks of receiver token j shared by the TA and overlap passes.
__device__ __forceinline__ void check_receiver(const int32_t* __restrict__ s_end,
                                               const int32_t* __restrict__ r_end, int64_t j,
                                               int32_t r0, int32_t r1, int32_t s0, int32_t s1,
                                               int32_t e, int32_t* info) {
  const int32_t prev = (j > r0) ? r_end[j - 1] : 0;
  if (e <= prev) flag(info, HF_CHECK_BAD_OFFSETS);
  if (j == r1 - 1 && s_end[s1 - 1] != e) flag(info, HF_CHECK_BAD_OFFSETS);
  (void)s0;
}

__global__ void ta_match_kernel(ReqPtrs rq, const int32_t* __restrict__ s_end,
                                const int32_t* __restrict__ r_end, int64_t T_r,
                                int32_t* __restrict__ row_ptr, int32_t* __restrict__ col,
                                float* __restrict__ w, int32_t* info) {
  __shared__ int32_t sp[kMaxReq + 1], rp[kMaxReq + 1];
  for (int i = threadIdx.x; i <= rq.n_req; i += blockDim.x) {
    sp[i] = rq.s_ptr[i];
    rp[i] = rq.r_ptr[i];
  }
  __syncthreads();
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < T_r;
       j += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(rp, rq.n_req, j);
    const int32_t r0 = rp[q], r1 = rp[q + 1], s0 = sp[q], s1 = sp[q + 1];
    const int32_t e = r_end[j];
    check_receiver(s_end, r_end, j, r0, r1, s0, s1, e, info);
    const int ns = s1 - s0;
    const int k = lower_bound_i32(s_end + s0, ns, e);
    int32_t m = (k < ns && s_end[s0 + k] == e) ? s0 + k : -1;  // shared boundary?
    if (j == r0 && m < s0) m = s0;  // before the first match: first sender token
    col[j] = m;
    row_ptr[j] = static_cast<int32_t>(j);
    w[j] = 1.0f;
    if (j == T_r - 1) {
      row_ptr[T_r] = static_cast<int32_t>(T_r);
      info[0] = static_cast<int32_t>(T_r);
    }
  }
}

__global__ void same_index_kernel(ReqPtrs rq, int64_t T_r, int32_t* __restrict__ row_ptr,
                                  int32_t* __restrict__ col, float* __restrict__ w,
                                  int32_t* info) {
  __shared__ int32_t sp[kMaxReq + 1], rp[kMaxReq + 1];
  for (int i = threadIdx.x; i <= rq.n_req; i += blockDim.x) {
    sp[i] = rq.s_ptr[i];
    rp[i] = rq.r_ptr[i];
  }
  __syncthreads();
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < T_r;
       j += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(rp, rq.n_req, j);
    const int32_t ns = sp[q + 1] - sp[q];
    const int32_t t = static_cast<int32_t>(j - rp[q]);
    col[j] = sp[q] + (t < ns - 1 ? t : ns - 1);  // a(j) = min(j, n_S), one-based
    row_ptr[j] = static_cast<int32_t>(j);
    w[j] = 1.0f;
    if (j == T_r - 1) {
      row_ptr[T_r] = static_cast<int32_t>(T_r);
      info[0] = static_cast<int32_t>(T_r);
    }
  }
}

// Sender tokens overlapping receiver token j: [k0, k1] (request-local).
__device__ __forceinline__ void overlap_range(const int32_t* __restrict__ s_end,
                                              const int32_t* __restrict__ r_end, int64_t j,
                                              int32_t r0, int32_t s0, int32_t ns, int* k0,
                                              int* k1, int32_t* info) {
  const int32_t start = (j > r0) ? r_end[j - 1] : 0;
  const int32_t e = r_end[j];
  int a = upper_bound_i32(s_end + s0, ns, start);  // first sender end > start
  int b = lower_bound_i32(s_end + s0, ns, e);      // first sender end >= end
  if (b >= ns) {
    b = ns - 1;
    flag(info, HF_CHECK_BAD_OFFSETS);
  }
  if (a > b) {
    a = b;
    flag(info, HF_CHECK_BAD_OFFSETS);
  }
  *k0 = a;
  *k1 = b;
}

__global__ void overlap_count_kernel(ReqPtrs rq, const int32_t* __restrict__ s_end,
                                     const int32_t* __restrict__ r_end, int64_t T_r,
                                     int32_t* __restrict__ row_ptr, int32_t* info) {
  __shared__ int32_t sp[kMaxReq + 1], rp[kMaxReq + 1];
  for (int i = threadIdx.x; i <= rq.n_req; i += blockDim.x) {
    sp[i] = rq.s_ptr[i];
    rp[i] = rq.r_ptr[i];
  }
  __syncthreads();
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < T_r;
       j += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(rp, rq.n_req, j);
    const int32_t r0 = rp[q], r1 = rp[q + 1], s0 = sp[q], s1 = sp[q + 1];
    check_receiver(s_end, r_end, j, r0, r1, s0, s1, r_end[j], info);
    int k0, k1;
    overlap_range(s_end, r_end, j, r0, s0, s1 - s0, &k0, &k1, info);
    row_ptr[j + 1] = k1 - k0 + 1;
    if (j == 0) row_ptr[0] = 0;
  }
}

__global__ void overlap_fill_kernel(ReqPtrs rq, const int32_t* __restrict__ s_end,
                                    const int32_t* __restrict__ r_end, int64_t T_r,
                                    const int32_t* __restrict__ row_ptr, int32_t* __restrict__ col,
                                    float* __restrict__ w, int64_t capacity, int32_t* info) {
  __shared__ int32_t sp[kMaxReq + 1], rp[kMaxReq + 1];
  for (int i = threadIdx.x; i <= rq.n_req; i += blockDim.x) {
    sp[i] = rq.s_ptr[i];
    rp[i] = rq.r_ptr[i];
  }
  __syncthreads();
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < T_r;
       j += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(rp, rq.n_req, j);
    const int32_t r0 = rp[q], s0 = sp[q], s1 = sp[q + 1];
    int k0, k1;
    overlap_range(s_end, r_end, j, r0, s0, s1 - s0, &k0, &k1, info);
    const int64_t e0 = row_ptr[j], e1 = row_ptr[j + 1];
    if (e1 > capacity) {
      flag(info, HF_CHECK_CAPACITY);
      continue;
    }
    const int n = static_cast<int>(e1 - e0);
    const float wt = 1.0f / static_cast<float>(n);  // IEEE division: fp32 RN(1/n)
    for (int i = 0; i < n; ++i) {
      col[e0 + i] = s0 + k0 + i;
      w[e0 + i] = wt;
    }
  }
}

int grid_for(int64_t n) {
  const int64_t want = (n + kThreads - 1) / kThreads;
  const int64_t cap = 8LL * device_sm_count();
  return static_cast<int>(std::max<int64_t>(1, std::min(want, cap)));
}

}  // namespace
}  // namespace hf

extern "C" hf_status hf_align_build(hf_align_mode mode, int32_t n_req, const int32_t* s_tok_ptr,
                                    const int32_t* r_tok_ptr, const int32_t* d_s_end,
                                    const int32_t* d_r_end, int32_t* d_row_ptr, int32_t* d_col,
                                    float* d_w, int64_t nnz_capacity, int32_t* d_info,
                                    hf_stream_t stream_) {
  using namespace hf;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  if (n_req < 1 || n_req > kMaxReq) {
    set_error("hf_align_build: n_req must be in [1, 1024]");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (!s_tok_ptr || !r_tok_ptr || !d_row_ptr || !d_info) {
    set_error("hf_align_build: null pointer argument");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (mode != HF_ALIGN_TA && mode != HF_ALIGN_OVERLAP_MEAN && mode != HF_ALIGN_SAME_INDEX) {
    set_error("hf_align_build: unknown alignment mode");
    return HF_ERR_INVALID_ARGUMENT;
  }
  ReqPtrs rq;
  rq.n_req = n_req;
  if (s_tok_ptr[0] != 0 || r_tok_ptr[0] != 0) {
    set_error("hf_align_build: token pointers must start at 0");
    return HF_ERR_INVALID_ARGUMENT;
  }
  for (int q = 0; q <= n_req; ++q) {
    rq.s_ptr[q] = s_tok_ptr[q];
    rq.r_ptr[q] = r_tok_ptr[q];
    if (q > 0 && (s_tok_ptr[q] < s_tok_ptr[q - 1] || r_tok_ptr[q] < r_tok_ptr[q - 1])) {
      set_error("hf_align_build: token pointers must be non-decreasing");
      return HF_ERR_INVALID_ARGUMENT;
    }
    if (q < n_req && r_tok_ptr[q + 1] > r_tok_ptr[q] && s_tok_ptr[q + 1] == s_tok_ptr[q]) {
      set_error("hf_align_build: a request has receiver tokens but no sender token");
      return HF_ERR_INVALID_ARGUMENT;
    }
  }
  const int64_t T_s = s_tok_ptr[n_req], T_r = r_tok_ptr[n_req];
  const int64_t need = (mode == HF_ALIGN_OVERLAP_MEAN) ? T_r + T_s : T_r;
  if (nnz_capacity < need) {
    set_error("hf_align_build: nnz_capacity too small for this mode");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (T_r > 0 && (!d_col || !d_w)) {
    set_error("hf_align_build: null CSR output");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (mode != HF_ALIGN_SAME_INDEX && T_r > 0 && (!d_s_end || !d_r_end)) {
    set_error("hf_align_build: null offsets");
    return HF_ERR_INVALID_ARGUMENT;
  }
  HF_CUDA_TRY(cudaMemsetAsync(d_info, 0, 2 * sizeof(int32_t), stream), "memset info");
  if (T_r == 0) {
    HF_CUDA_TRY(cudaMemsetAsync(d_row_ptr, 0, sizeof(int32_t), stream), "memset row_ptr");
    return HF_OK;
  }
  const int g = grid_for(T_r);
  if (mode != HF_ALIGN_SAME_INDEX && T_s > 0)
    check_sender_kernel<<<grid_for(T_s), kThreads, 0, stream>>>(rq, d_s_end, T_s, d_info);
  if (mode == HF_ALIGN_TA) {
    ta_match_kernel<<<g, kThreads, 0, stream>>>(rq, d_s_end, d_r_end, T_r, d_row_ptr, d_col, d_w,
                                                d_info);
    scan_inplace_kernel<ScanMax><<<1, kScanThreads, 0, stream>>>(d_col, T_r, nullptr);
  } else if (mode == HF_ALIGN_SAME_INDEX) {
    same_index_kernel<<<g, kThreads, 0, stream>>>(rq, T_r, d_row_ptr, d_col, d_w, d_info);
  } else {
    overlap_count_kernel<<<g, kThreads, 0, stream>>>(rq, d_s_end, d_r_end, T_r, d_row_ptr,
                                                     d_info);
    scan_inplace_kernel<ScanSum><<<1, kScanThreads, 0, stream>>>(d_row_ptr + 1, T_r, d_info);
    overlap_fill_kernel<<<g, kThreads, 0, stream>>>(rq, d_s_end, d_r_end, T_r, d_row_ptr, d_col,
                                                    d_w, nnz_capacity, d_info);
  }
  HF_CUDA_TRY(cudaGetLastError(), "align kernels launch");
  return HF_OK;
}
