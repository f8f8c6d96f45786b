// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "heterofold.h"

namespace hf {

constexpr int kMaxReq = 1024;        // requests per call
constexpr int kMaxLayersR = 128;     // receiver layers
constexpr int kMaxSeg = 8;           // map input segments per receiver layer (Eq. 1: 3;
                                     // KV Ridge's layer routing: 8)
constexpr int kMaxTerms = 2;         // sender layers blended into one segment
constexpr int kMaxHeadDim = 256;
constexpr int kMaxBatch = 16;        // directions per hf_transfer_batch call

// One receiver layer's map input: n_seg segments of d_S features each;
// segment s is sum_t w[s][t] * (pooled sender layer layer[s][t]).
struct LayerSegs {
  int32_t n_seg;
  int32_t n_terms[kMaxSeg];
  int32_t layer[kMaxSeg][kMaxTerms];
  float w[kMaxSeg][kMaxTerms];
};

// Per-plan metadata that lives in the caller's device workspace.
struct WorkspaceLayout {
  size_t status;     // int32: device status bits
  size_t n_distinct; // int32: number of distinct alignment rows U
  size_t segs;       // LayerSegs[L_r]
  size_t inv_r;      // float[L_r * 2]  (1 / r)
  size_t inv_freq;   // float[D_r / 2]
  size_t inv_freq_s; // float[D_s / 2]: sender RoPE (sender_k_rotated)
  size_t r_tok_ptr;  // int32[n_req + 1]
  size_t r_pos0;     // int32[n_req]
  size_t s_tok_ptr;  // int32[n_req + 1]
  size_t s_pos0;     // int32[n_req]
  size_t spos;       // int32[T_s] sender RoPE positions (sender_k_rotated), else one word
  size_t s_row0;     // int32[n_req] sender-cache row of each request's span
  size_t srow;       // int32[T_s] sender-cache row of each aligned token (spans), else one word
  size_t run_ptr;    // int32[T_r + 1]: first receiver row of each distinct row
  size_t ucol;       // int32[T_r]: sender column of each distinct row (one-entry rows)
  size_t upos;       // int32[T_r]: RoPE position of each distinct row's first receiver row
  size_t pos;        // int32[T_r]: RoPE position of each receiver row
  size_t dst_row;    // int32[T_r]: destination row of each receiver row
  size_t new_flag;   // int32[T_r]: 1 where a receiver row starts a new distinct row
  // pooling after the map (overlap mean pooling): windows of 128 aligned
  // sender tokens with stride S = 128 - h, h the widest row's column span
  size_t win_info;   // int32[4]: h, S, number of windows, unused
  size_t row_key;    // int32[T_r]: first column of each row, then its running maximum
  size_t win_ptr;    // int32[T_s + 2]: first receiver row of each window
  size_t total;
};

WorkspaceLayout workspace_layout(const hf_plan_desc& d);

// Constant tables copied into the workspace by the plan kernels.  They are
// passed by value as kernel parameters, so plan creation issues no host
// copies; the layer table goes to a kernel of its own because one launch's
// parameters are limited to 32 KB.
struct PlanConsts {
  int32_t L_r, D_r, D_s, n_req;
  float inv_r[2 * kMaxLayersR];
  float inv_freq[kMaxHeadDim / 2];
  float inv_freq_s[kMaxHeadDim / 2];
  int32_t r_tok_ptr[kMaxReq + 1];
  int32_t r_pos0[kMaxReq];
  int32_t s_tok_ptr[kMaxReq + 1];
  int32_t s_pos0[kMaxReq];
  int32_t s_row0[kMaxReq];
};
struct SegTables {
  int32_t L_r;
  LayerSegs segs[kMaxLayersR];
};
struct PlanTables {
  PlanConsts c;
  SegTables s;
};
static_assert(sizeof(PlanConsts) < 32000, "PlanConsts must fit the kernel parameter space");
static_assert(sizeof(SegTables) < 32000, "SegTables must fit the kernel parameter space");

}  // namespace hf

struct hf_plan_s {
  hf_plan_desc desc;  // host-array fields are cleared after copying
  int d_s, d_r, K, n_seg;
  int64_t T_s, T_r, nnz_hint;
  int BN, groups, stages;
  bool gather;  // every map input row is a single unweighted sender row
  bool split;   // computed bf16 operand rows go to the tensor core as value + residual
  bool staged;  // split rows of one entry each: raw sender atoms staged by cp.async
  bool rope;    // receiver keys get RoPE
  bool unrot;   // sender keys carry RoPE and are rotated back in the builder
  bool span;    // aligned sender tokens are spans inside a longer sender cache
  bool pam;     // pooling after the map: map input rows are sender rows in windows
  bool wide;    // tiles of two 256-column blocks (operand rows built by the loader warps)
  int64_t s_rows;  // sender-cache rows per (layer, role)
  char* ws;
  size_t ws_bytes;
  hf::WorkspaceLayout lay;
  int32_t s_tok_ptr_last;
  int32_t max_sender_layer[hf::kMaxLayersR];  // highest sender layer each receiver layer reads
  // hf_transfer_host: copy streams and events, created on first use
  int aux_device = -1;
  cudaStream_t s_h2d = nullptr, s_d2h = nullptr;
  cudaEvent_t* events = nullptr;
  int n_events = 0;
};

namespace hf {

void set_error(const std::string& msg);
hf_status cuda_fail(cudaError_t e, const char* what);
int device_sm_count();

hf_status launch_plan_kernels(hf_plan_s* p, const PlanTables& tables, cudaStream_t stream);
hf_status plan_build(const hf_plan_desc* desc, void* d_workspace, size_t workspace_bytes,
                     cudaStream_t stream, hf_plan_s* p, PlanTables* t);
// One transfer-kernel launch over receiver layers [l_begin, l_end) (l_end < 0: all).
// stall (test hook): the map producer withholds its first atom, so the
// launch ends through the bounded waits with HF_CHECK_TIMEOUT.
hf_status launch_transfer(hf_plan_s* p, const void* sender, void* receiver, cudaStream_t stream,
                          int l_begin = 0, int l_end = -1, bool stall = false);
// Several plans in one launch: they must share the dtype, the operand path
// and where the pooling happens (batch_compatible); n <= kMaxBatch.
bool batch_compatible(const hf_plan_s* const* plans, int n);
hf_status launch_transfer_batch(hf_plan_s* const* plans, const void* const* senders,
                                void* const* receivers, int n, cudaStream_t stream);

// Device buffers of gemm_f32 (part of hf_recolor_fit's workspace): the bf16
// planes of both operands, split-K partials, and an error word (set when a
// pipeline wait of the product kernel ran out).
struct GemmWork {
  void* planes_a;
  size_t planes_a_bytes;
  void* planes_b;
  size_t planes_b_bytes;
  float* partial;
  size_t partial_bytes;
  int32_t* err;
};
// Bytes of the three bf16 planes of an operand with `rows` rows and K columns.
size_t gemm_planes_bytes(int64_t rows, int64_t K);
// C[M x N] = alpha op(A) op(B) + beta C_in + diag I (row-major C and C_in,
// leading dimension ldc; C_in NULL = C), op(A)(i, k) = A[i * a_i + k * a_k],
// op(B)(k, j) = B[k * b_k + j * b_j], in fp32 accuracy on the tensor cores
// (hf_gemm.cu).  Asynchronous on s.
hf_status gemm_f32(cudaStream_t s, const GemmWork& wk, int M, int N, int K, float alpha,
                   const float* A, int64_t a_i, int64_t a_k, const float* B, int64_t b_k,
                   int64_t b_j, float beta, float* C, int64_t ldc, const float* Cin = nullptr,
                   float diag = 0.f);

}  // namespace hf

#define HF_CUDA_TRY(expr, what)                      \
  do {                                               \
    cudaError_t e__ = (expr);                        \
    if (e__ != cudaSuccess) return hf::cuda_fail(e__, what); \
  } while (0)
