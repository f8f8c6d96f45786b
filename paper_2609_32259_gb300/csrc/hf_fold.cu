// hf_fold: folds the output-aware low-rank correction (Eq. 7) into the
// affine maps (Eq. 9): A_final = A (I + B G), b_final = b (I + B G).
// In the ABI's layout W = A^T ([d_R][K] per map), so
//   T = B^T W                      (rho x K)
//   W_final = W + G^T T            (element [n][k] += sum_r G[r][n] T[r][k])
//   b_final = b + (b B) G.
// A block reads its columns of W twice (the second time from L2) and
// writes them once (HBM-bound).  Plain CUDA-core
// arithmetic: a rank of 16 is far too thin for the tensor cores to matter.
#include <cuda_bf16.h>

#include <string>

#include "hf_internal.h"

namespace hf {
namespace {

constexpr int kMaxRank = 32;
constexpr int kFoldThreads = 256;

__device__ __forceinline__ void load2(const __nv_bfloat16* p, float* a, float* b) {
  const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
  *a = f.x;
  *b = f.y;
}
__device__ __forceinline__ void load2(const float* p, float* a, float* b) {
  const float2 f = *reinterpret_cast<const float2*>(p);
  *a = f.x;
  *b = f.y;
}
__device__ __forceinline__ void store2(__nv_bfloat16* p, float a, float b) {
  *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(a, b);
}
__device__ __forceinline__ void store2(float* p, float a, float b) {
  *reinterpret_cast<float2*>(p) = make_float2(a, b);
}

constexpr int kFoldPairs = 32;                 // column pairs per block (64 columns)
constexpr int kFoldSlices = kFoldThreads / kFoldPairs;  // row slices (8)

// One block folds columns [k0, k0 + 64) of one map:
//  pass 1: T = B^T W for the block's columns; thread (column pair, row slice)
//          accumulates rank x 2 products over rows n = slice (mod 8), reading
//          W with coalesced 4-byte loads (one 128-byte row segment per warp,
//          eight rows in flight) and B from shared memory; slices are summed
//          in smem;
//  pass 2: W_final = W + G^T T row by row (the rows come from L2 again), G^T
//          staged in smem with rows padded to rank + 4 floats (16-byte rows,
//          read as float4 broadcasts).
// Every element of the block's columns is read in pass 1 before any is
// written in pass 2, so W_final may alias W.
template <typename T, int R>
__global__ void __launch_bounds__(kFoldThreads) fold_kernel(const T* W, const float* __restrict__ Bm,
                                                            const float* __restrict__ Gm, T* Wf,
                                                            int d_r, int64_t K) {
  extern __shared__ __align__(16) float fsm[];
  constexpr int kGs = R + 4;                              // padded G^T row
  float* Gs = fsm;                                        // [d_r][kGs]; B [d_r][R] before
  float* Bs = fsm;
  float* Ps = Gs + static_cast<size_t>(d_r) * kGs;        // [slices][R][64]
  const int map = blockIdx.y;
  const int tid = threadIdx.x;
  const int cp = tid % kFoldPairs, sl = tid / kFoldPairs;
  const int64_t k = static_cast<int64_t>(blockIdx.x) * (2 * kFoldPairs) + 2 * cp;
  const bool live = k < K;  // K is even: both columns of a pair exist or neither
  const int64_t base = static_cast<int64_t>(map) * d_r * K + k;
  const float* B = Bm + static_cast<int64_t>(map) * d_r * R;
  const float* G = Gm + static_cast<int64_t>(map) * R * d_r;
  for (int i = tid; i < R * d_r / 4; i += kFoldThreads)
    reinterpret_cast<float4*>(Bs)[i] = __ldg(reinterpret_cast<const float4*>(B) + i);
  __syncthreads();
  // pass 1
  float acc[R][2];
#pragma unroll
  for (int r = 0; r < R; ++r) acc[r][0] = acc[r][1] = 0.f;
  if (live) {
#pragma unroll 8
    for (int n = sl; n < d_r; n += kFoldSlices) {
      float x0, x1;
      load2(W + base + static_cast<int64_t>(n) * K, &x0, &x1);
      const float4* bn = reinterpret_cast<const float4*>(Bs + n * R);
#pragma unroll
      for (int q = 0; q < R / 4; ++q) {
        const float4 b = bn[q];
        acc[4 * q][0] = fmaf(b.x, x0, acc[4 * q][0]);
        acc[4 * q][1] = fmaf(b.x, x1, acc[4 * q][1]);
        acc[4 * q + 1][0] = fmaf(b.y, x0, acc[4 * q + 1][0]);
        acc[4 * q + 1][1] = fmaf(b.y, x1, acc[4 * q + 1][1]);
        acc[4 * q + 2][0] = fmaf(b.z, x0, acc[4 * q + 2][0]);
        acc[4 * q + 2][1] = fmaf(b.z, x1, acc[4 * q + 2][1]);
        acc[4 * q + 3][0] = fmaf(b.w, x0, acc[4 * q + 3][0]);
        acc[4 * q + 3][1] = fmaf(b.w, x1, acc[4 * q + 3][1]);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < R; ++r)
    *reinterpret_cast<float2*>(Ps + (sl * R + r) * 64 + 2 * cp) = make_float2(acc[r][0], acc[r][1]);
  __syncthreads();
  float t0[R], t1[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    float a = 0.f, b = 0.f;
    for (int s2 = 0; s2 < kFoldSlices; ++s2) {
      const float2 v = *reinterpret_cast<const float2*>(Ps + (s2 * R + r) * 64 + 2 * cp);
      a += v.x;
      b += v.y;
    }
    t0[r] = a;
    t1[r] = b;
  }
  __syncthreads();  // B is no longer read: G^T takes its place
  for (int i = tid; i < R * d_r; i += kFoldThreads) {
    const int r = i / d_r, n = i - r * d_r;
    Gs[n * kGs + r] = __ldg(G + i);
  }
  __syncthreads();
  if (!live) return;
  // pass 2
#pragma unroll 8
  for (int n = sl; n < d_r; n += kFoldSlices) {
    float v0, v1;
    load2(W + base + static_cast<int64_t>(n) * K, &v0, &v1);
    const float4* g = reinterpret_cast<const float4*>(Gs + n * kGs);
#pragma unroll
    for (int q = 0; q < R / 4; ++q) {
      const float4 gq = g[q];
      v0 = fmaf(gq.x, t0[4 * q], v0);
      v1 = fmaf(gq.x, t1[4 * q], v1);
      v0 = fmaf(gq.y, t0[4 * q + 1], v0);
      v1 = fmaf(gq.y, t1[4 * q + 1], v1);
      v0 = fmaf(gq.z, t0[4 * q + 2], v0);
      v1 = fmaf(gq.z, t1[4 * q + 2], v1);
      v0 = fmaf(gq.w, t0[4 * q + 3], v0);
      v1 = fmaf(gq.w, t1[4 * q + 3], v1);
    }
    store2(Wf + base + static_cast<int64_t>(n) * K, v0, v1);
  }
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

size_t fold_smem(int d_r, int rank) {
  return (static_cast<size_t>(d_r) * (rank + 4) + static_cast<size_t>(kFoldSlices) * rank * 64) *
         sizeof(float);
}

template <typename T, int R>
hf_status launch_fold_r(int n_maps, int d_r, int64_t K, const void* W, const float* B,
                        const float* G, void* Wf, cudaStream_t stream) {
  auto kern = fold_kernel<T, R>;
  const size_t smem = fold_smem(d_r, R);
  HF_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(smem)),
              "hf_fold: shared memory size");
  const unsigned kblocks = static_cast<unsigned>((K + 2 * kFoldPairs - 1) / (2 * kFoldPairs));
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
  if (fold_smem(d_r, rank) > static_cast<size_t>(optin)) {
    set_error("hf_fold: unsupported: d_R x rank too large for one block's shared memory");
    return HF_ERR_UNSUPPORTED;
  }
  hf_status s;
  switch (rank) {
    case 4: s = launch_fold_r<T, 4>(n_maps, d_r, K, W, B, G, Wf, stream); break;
    case 8: s = launch_fold_r<T, 8>(n_maps, d_r, K, W, B, G, Wf, stream); break;
    case 16: s = launch_fold_r<T, 16>(n_maps, d_r, K, W, B, G, Wf, stream); break;
    case 32: s = launch_fold_r<T, 32>(n_maps, d_r, K, W, B, G, Wf, stream); break;
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
