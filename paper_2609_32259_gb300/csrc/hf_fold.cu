// hf_fold: folds the output-aware low-rank correction (Eq. 7) into the
// affine maps (Eq. 9): A_final = A (I + B G), b_final = b (I + B G).
// In the ABI's layout W = A^T ([d_R][K] per map), so
//   T = B^T W                      (rho x K)
//   W_final = W + G^T T            (element [n][k] += sum_r G[r][n] T[r][k])
//   b_final = b + (b B) G.
// A block reads its columns of W twice (the second time from L2) and
// writes them once.  Plain fp32 CUDA-core arithmetic (4 rank FLOP per
// element, which at rank 16 outweighs the memory time): a rank of 16 is
// too thin a contraction for the tensor cores, and fp32 maps need fp32
// accuracy.
#include <cuda_bf16.h>

#include <string>

#include "hf_internal.h"

namespace hf {
namespace {

constexpr int kMaxRank = 32;
constexpr int kFoldThreads = 256;

// CPT consecutive columns of one row: values from shared memory, stores of
// 4 * CPT (fp32) or 2 * CPT (bf16) bytes.
template <int CPT>
__device__ __forceinline__ void smem_cols(const __nv_bfloat16* p, float* x) {
#pragma unroll
  for (int j = 0; j < CPT; j += 2) {
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p + j));
    x[j] = a.x;
    x[j + 1] = a.y;
  }
}
template <int CPT>
__device__ __forceinline__ void smem_cols(const float* p, float* x) {
#pragma unroll
  for (int j = 0; j < CPT; j += 2) {
    const float2 a = *reinterpret_cast<const float2*>(p + j);
    x[j] = a.x;
    x[j + 1] = a.y;
  }
}
template <int CPT>
__device__ __forceinline__ void store_cols(__nv_bfloat16* p, const float* x) {
  if constexpr (CPT == 4) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(x[0], x[1]), b = __floats2bfloat162_rn(x[2], x[3]);
    *reinterpret_cast<uint2*>(p) = make_uint2(*reinterpret_cast<const uint32_t*>(&a),
                                              *reinterpret_cast<const uint32_t*>(&b));
  } else {
    *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(x[0], x[1]);
  }
}
template <int CPT>
__device__ __forceinline__ void store_cols(float* p, const float* x) {
  if constexpr (CPT == 4)
    *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
  else
    *reinterpret_cast<float2*>(p) = make_float2(x[0], x[1]);
}

// Asynchronous copy of N (4, 8 or 16) bytes from global to shared memory.
template <int N>
__device__ __forceinline__ void fold_cp_async(void* dst, const void* src) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst));
  if constexpr (N == 16)
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(src) : "memory");
  else
    asm volatile("cp.async.ca.shared.global [%0], [%1], %2;" ::"r"(d), "l"(src), "n"(N) : "memory");
}
__device__ __forceinline__ void fold_cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void fold_cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

constexpr int kFoldSlices = kFoldThreads / 32;  // row slices (8): one warp each
constexpr int kFoldRing = 16;                    // rows of W in flight per thread

// Shared memory of one block, in floats: a region holding B [d_r][R] in
// pass 1, then the slices' partial sums [slices][R][32 CPT], then G^T
// [d_r][R + 4]; after it, each thread's ring of kFoldRing rows x CPT columns.
template <typename T>
__host__ __device__ constexpr size_t fold_region_floats(int d_r, int R, int CPT) {
  const size_t b = static_cast<size_t>(d_r) * R, g = static_cast<size_t>(d_r) * (R + 4);
  const size_t p = static_cast<size_t>(kFoldSlices) * R * 32 * CPT;
  const size_t m = g > p ? g : p;
  return m > b ? m : b;
}
template <typename T>
__host__ __device__ constexpr size_t fold_smem_bytes(int d_r, int R, int CPT) {
  return fold_region_floats<T>(d_r, R, CPT) * sizeof(float) +
         static_cast<size_t>(kFoldThreads) * kFoldRing * CPT * sizeof(T);
}

// This thread's ring of W rows: rows n = sl, sl + 8, ... < d_r of its CPT
// columns, kFoldRing in flight, each thread copying and reading only its own
// bytes (so a wait on its own copies is all the synchronisation needed).
// Slot i of thread tid is at (i * 256 + tid) * CPT elements: a warp's reads
// of one slot are consecutive.
template <typename T, int CPT>
struct FoldRing {
  static constexpr int kBytes = CPT * static_cast<int>(sizeof(T));
  static constexpr int kStride = kFoldThreads * CPT;  // slots are thread-interleaved
  const T* col0;
  int64_t K;
  int d_r, sl;
  T* ring;
  // issues the first kFoldRing rows (one commit group per row)
  __device__ __forceinline__ void start() const {
#pragma unroll 1
    for (int i = 0; i < kFoldRing; ++i) {
      const int n = sl + kFoldSlices * i;
      if (n < d_r) fold_cp_async<kBytes>(ring + i * kStride, col0 + static_cast<int64_t>(n) * K);
      fold_cp_commit();
    }
  }
  // waits for the row held in `slot` and reads it
  __device__ __forceinline__ void take(int slot, float* x) const {
    fold_cp_wait<kFoldRing - 1>();
    smem_cols<CPT>(ring + slot * kStride, x);
  }
  // refills `slot` (row n, already used) with row n + 8 kFoldRing
  __device__ __forceinline__ void refill(int n, int slot) const {
    const int nn = n + kFoldSlices * kFoldRing;
    if (nn < d_r) fold_cp_async<kBytes>(ring + slot * kStride, col0 + static_cast<int64_t>(nn) * K);
    fold_cp_commit();
  }
};

// One block folds columns [k0, k0 + 32 CPT) of one map; thread (column
// group cg = lane, row slice sl = warp) owns columns k0 + CPT cg .. + CPT - 1
// and streams them, rows n = sl (mod 8), through its shared-memory ring:
//  pass 1: T = B^T W for those columns, B from shared memory (float4
//          broadcasts); the slices' partial sums go through shared memory
//          (where B was) and every thread sums its columns' R values;
//  pass 2: W_final = W + G^T T row by row (the rows come from L2 again), G^T
//          staged in shared memory with rows padded to R + 4 floats.
// Every element of the block's columns is read in pass 1 before any is
// written in pass 2, so W_final may alias W.
template <typename T, int R, int CPT>
__global__ void __launch_bounds__(kFoldThreads) fold_kernel(const T* W, const float* __restrict__ Bm,
                                                            const float* __restrict__ Gm, T* Wf,
                                                            int d_r, int64_t K) {
  extern __shared__ __align__(16) float fsm[];
  constexpr int kGs = R + 4;            // padded G^T row
  constexpr int kCols = 32 * CPT;       // columns per block
  float* const Bs = fsm;                // [d_r][R]
  float* const Ps = fsm;                // [slices][R][kCols]
  float* const Gs = fsm;                // [d_r][kGs]
  const int map = blockIdx.y;
  const int tid = threadIdx.x;
  const int cg = tid & 31, sl = tid >> 5;
  T* const ring = reinterpret_cast<T*>(fsm + fold_region_floats<T>(d_r, R, CPT)) + tid * CPT;
  const int64_t k = static_cast<int64_t>(blockIdx.x) * kCols + CPT * cg;
  const bool live = k < K;  // K is a multiple of CPT: a group's columns all exist or none
  const T* col0 = W + static_cast<int64_t>(map) * d_r * K + k;
  T* const out0 = Wf + static_cast<int64_t>(map) * d_r * K + k;
  const float* B = Bm + static_cast<int64_t>(map) * d_r * R;
  const float* G = Gm + static_cast<int64_t>(map) * R * d_r;
  for (int i = tid; i < R * d_r / 4; i += kFoldThreads)
    reinterpret_cast<float4*>(Bs)[i] = __ldg(reinterpret_cast<const float4*>(B) + i);
  __syncthreads();
  // pass 1
  float acc[R][CPT];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int j = 0; j < CPT; ++j) acc[r][j] = 0.f;
  const FoldRing<T, CPT> rg{col0, K, d_r, sl, ring};
  if (live) {
    rg.start();
    int slot = 0;
#pragma unroll 1
    for (int n = sl; n < d_r; n += kFoldSlices) {
      float x[CPT];
      rg.take(slot, x);
      const float4* bn = reinterpret_cast<const float4*>(Bs + n * R);
#pragma unroll
      for (int q = 0; q < R / 4; ++q) {
        const float4 b = bn[q];
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
          acc[4 * q][j] = fmaf(b.x, x[j], acc[4 * q][j]);
          acc[4 * q + 1][j] = fmaf(b.y, x[j], acc[4 * q + 1][j]);
          acc[4 * q + 2][j] = fmaf(b.z, x[j], acc[4 * q + 2][j]);
          acc[4 * q + 3][j] = fmaf(b.w, x[j], acc[4 * q + 3][j]);
        }
      }
      rg.refill(n, slot);  // after x is consumed
      if (++slot == kFoldRing) slot = 0;
    }
    fold_cp_wait<0>();
  }
  __syncthreads();  // B is no longer read: the partial sums take its place
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int j = 0; j < CPT; ++j) Ps[(sl * R + r) * kCols + CPT * cg + j] = acc[r][j];
  __syncthreads();
  float t[R][CPT];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int j = 0; j < CPT; ++j) t[r][j] = 0.f;
#pragma unroll 1
  for (int s2 = 0; s2 < kFoldSlices; ++s2)
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int j = 0; j < CPT; ++j) t[r][j] += Ps[(s2 * R + r) * kCols + CPT * cg + j];
  __syncthreads();  // the partial sums are read: G^T takes their place
  for (int i = tid; i < R * d_r; i += kFoldThreads) {
    const int r = i / d_r, n = i - r * d_r;
    Gs[n * kGs + r] = __ldg(G + i);
  }
  __syncthreads();
  if (!live) return;
  // pass 2
  rg.start();
  int slot = 0;
#pragma unroll 1
  for (int n = sl; n < d_r; n += kFoldSlices) {
    float v[CPT];
    rg.take(slot, v);
    const float4* g = reinterpret_cast<const float4*>(Gs + n * kGs);
#pragma unroll
    for (int q = 0; q < R / 4; ++q) {
      const float4 gq = g[q];
#pragma unroll
      for (int j = 0; j < CPT; ++j) {
        v[j] = fmaf(gq.x, t[4 * q][j], v[j]);
        v[j] = fmaf(gq.y, t[4 * q + 1][j], v[j]);
        v[j] = fmaf(gq.z, t[4 * q + 2][j], v[j]);
        v[j] = fmaf(gq.w, t[4 * q + 3][j], v[j]);
      }
    }
    store_cols<CPT>(out0 + static_cast<int64_t>(n) * K, v);
    rg.refill(n, slot);  // after the row is consumed
    if (++slot == kFoldRing) slot = 0;
  }
  fold_cp_wait<0>();
}

// b_final = b + (b B) G for one map per block.
__global__ void __launch_bounds__(256) fold_b_kernel(const float* b, const float* __restrict__ Bm,
                                                     const float* __restrict__ Gm, float* bf,
                                                     int d_r, int rank) {
  __shared__ float part[256 / 32][kMaxRank];
  __shared__ float bB[kMaxRank];
  const int map = blockIdx.x;
  const float* bm = b + static_cast<int64_t>(map) * d_r;
  const float* B = Bm + static_cast<int64_t>(map) * d_r * rank;
  const float* G = Gm + static_cast<int64_t>(map) * rank * d_r;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int r = 0; r < rank; ++r) {
    float s = 0.f;
    for (int m = threadIdx.x; m < d_r; m += blockDim.x)
      s = fmaf(bm[m], B[static_cast<int64_t>(m) * rank + r], s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) part[warp][r] = s;
  }
  __syncthreads();
  if (threadIdx.x < rank) {
    float s = 0.f;
    for (int w = 0; w < 256 / 32; ++w) s += part[w][threadIdx.x];
    bB[threadIdx.x] = s;
  }
  __syncthreads();
  for (int n = threadIdx.x; n < d_r; n += blockDim.x) {
    float v = bm[n];
    for (int r = 0; r < rank; ++r) v = fmaf(bB[r], G[static_cast<int64_t>(r) * d_r + n], v);
    bf[static_cast<int64_t>(map) * d_r + n] = v;
  }
}

template <typename T, int R>
hf_status launch_fold_r(int n_maps, int d_r, int64_t K, const void* W, const float* B,
                        const float* G, void* Wf, int optin, cudaStream_t stream) {
  // four columns per thread where the accumulators fit (R <= 16), the column
  // groups tile K and shared memory allows; two otherwise
  constexpr int kWide = R <= 16 ? 4 : 2;
  const bool four = kWide == 4 && K % 4 == 0 &&
                    fold_smem_bytes<T>(d_r, R, 4) <= static_cast<size_t>(optin);
  const int cpt = four ? 4 : 2;
  const size_t smem = fold_smem_bytes<T>(d_r, R, cpt);
  if (smem > static_cast<size_t>(optin)) {
    set_error("hf_fold: unsupported: d_R x rank too large for one block's shared memory");
    return HF_ERR_UNSUPPORTED;
  }
  auto kern = four ? fold_kernel<T, R, kWide> : fold_kernel<T, R, 2>;
  HF_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(smem)),
              "hf_fold: shared memory size");
  const int64_t cols = 32 * cpt;
  const unsigned kblocks = static_cast<unsigned>((K + cols - 1) / cols);
  kern<<<dim3(kblocks, n_maps), kFoldThreads, smem, stream>>>(
      static_cast<const T*>(W), B, G, static_cast<T*>(Wf), d_r, K);
  HF_CUDA_TRY(cudaGetLastError(), "hf_fold: launch");
  return HF_OK;
}

template <typename T>
hf_status launch_fold(int n_maps, int d_r, int64_t K, int rank, const void* W, const float* b,
                      const float* B, const float* G, void* Wf, float* bf, cudaStream_t stream) {
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  hf_status s;
  switch (rank) {
    case 4: s = launch_fold_r<T, 4>(n_maps, d_r, K, W, B, G, Wf, optin, stream); break;
    case 8: s = launch_fold_r<T, 8>(n_maps, d_r, K, W, B, G, Wf, optin, stream); break;
    case 16: s = launch_fold_r<T, 16>(n_maps, d_r, K, W, B, G, Wf, optin, stream); break;
    case 32: s = launch_fold_r<T, 32>(n_maps, d_r, K, W, B, G, Wf, optin, stream); break;
    default:
      set_error("hf_fold: unsupported: rank must be 4, 8, 16 or 32");
      return HF_ERR_UNSUPPORTED;
  }
  if (s != HF_OK) return s;
  fold_b_kernel<<<n_maps, 256, 0, stream>>>(b, B, G, bf, d_r, rank);
  HF_CUDA_TRY(cudaGetLastError(), "hf_fold: bias launch");
  return HF_OK;
}

}  // namespace
}  // namespace hf

using namespace hf;

extern "C" hf_status hf_fold(hf_dtype dtype, int32_t n_maps, int32_t d_R, int64_t K, int32_t rank,
                             const void* d_W, const float* d_b, const float* d_B,
                             const float* d_G, void* d_W_final, float* d_b_final,
                             hf_stream_t stream_) {
  if (dtype != HF_BF16 && dtype != HF_F32) {
    set_error("hf_fold: unknown dtype");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (n_maps < 1 || n_maps > 65535 || d_R < 1 || K < 1 || rank < 1 || rank > kMaxRank) {
    set_error("hf_fold: n_maps in [1, 65535], d_R >= 1, K >= 1, rank in [1, 32]");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (!d_W || !d_b || !d_B || !d_G || !d_W_final || !d_b_final) {
    set_error("hf_fold: null pointer");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if ((reinterpret_cast<uintptr_t>(d_B) | reinterpret_cast<uintptr_t>(d_W) |
       reinterpret_cast<uintptr_t>(d_W_final)) & 15u || (K % 2)) {
    set_error("hf_fold: W, W_final and B must be 16-byte aligned and K even");
    return HF_ERR_INVALID_ARGUMENT;
  }
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  if (dtype == HF_BF16)
    return launch_fold<__nv_bfloat16>(n_maps, d_R, K, rank, d_W, d_b, d_B, d_G, d_W_final,
                                      d_b_final, stream);
  return launch_fold<float>(n_maps, d_R, K, rank, d_W, d_b, d_B, d_G, d_W_final, d_b_final,
                            stream);
}
