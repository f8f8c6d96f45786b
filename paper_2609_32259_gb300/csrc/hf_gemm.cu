// fp32 matrix products on the tcgen05 tensor cores, for hf_recolor_fit's
// moments, Newton-Schulz roots and polar iterations (Section 3.2, Eq. 3-5).
//
// C = alpha op(A) op(B) + beta C_in + d I with fp32 accuracy from bf16
// products (C_in may be C itself; d I adds d on the diagonal).
// Every fp32 operand value x is split exactly into three bf16 parts,
// x0 = bf16(x), x1 = bf16(x - x0), x2 = x - x0 - x1 (what is left has at
// most 8 significant bits, so it is exact in bf16), and each part is stored
// K-major as a plane.  The product keeps the six terms a_i b_j with
// i + j <= 2, summed by the tensor core into one fp32 TMEM accumulator; the
// dropped terms are below 2^-23 of |a||b|, the size of fp32 rounding.
//
// The tensor core adds into its fp32 accumulator with truncation (measured
// on GB300: a sum of 4,096 positive products comes out 1e-5 low, 7.6e-5 at
// 16,384, where fp32 rounding to nearest is unbiased), so one accumulator
// never takes more than one 64-wide atom of K (24 MMAs, the smallest terms
// first): the epilogue drains each atom's accumulator into fp32 registers
// with rounding to nearest while the tensor core fills the other one.
//
// The kernel: persistent clusters of two CTAs (one per SM pair), pair tiles
// of 256 x 256 outputs (tcgen05.mma.cta_group::2, M = 256, N = 256,
// K = 16 bf16 per instruction), each CTA holding 128 rows of the A tile and
// 128 rows of the B tile.  A stage is one 128-byte atom (64 bf16) of K of
// one term's A plane and B plane, loaded by TMA (128-byte swizzle) and
// completing on the leader CTA's barrier.
//   warp 0      TMA producer
//   warp 1      TMEM allocator; in the leader CTA the thread issuing the MMAs
//               of one K atom into one of two 256-column accumulators
//   warps 2-17  epilogue: 4 warps per TMEM lane quarter, 64 columns each;
//               per K atom TMEM -> registers (running fp32 sums); per tile
//               alpha * sum + beta * C (or a split-K partial) -> global
// Small products are split along K so that every SM pair has work; a second
// kernel sums the partials.  Waits are bounded: a wait that runs out sets an
// error word and the CTA pair unwinds.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <string>

#include <cuda_bf16.h>

#include "hf_device.cuh"
#include "hf_internal.h"

namespace hf {
namespace {

constexpr int kGRows = 128;                 // rows of A (and of B) per CTA of a pair tile
constexpr int kGTile = 256;                 // pair tile: 256 x 256 outputs
constexpr int kGAtomBytes = kGRows * 128;   // one 128-byte atom of K for 128 rows
constexpr int kGStageBytes = 2 * kGAtomBytes;
constexpr int kGStages = 6;
constexpr int kGEpiWarps = 16;
constexpr int kGEpiCols = kGTile / (kGEpiWarps / 4);  // columns per epilogue thread
constexpr int kGThreads = 64 + 32 * kGEpiWarps;
constexpr int kGMaxTerms = 6;
constexpr int kGTmemCols = 512;

struct GemmParams {
  float* C;           // output, row-major with leading dimension ldc
  const float* Cin;   // beta term's matrix (same layout as C; may be C)
  float diag;         // added on the diagonal (row == column)
  int64_t ldc;
  float* partial;     // split-K partials [splits][M][N] (splits > 1)
  int32_t* err;       // error word (a wait ran out)
  int M, N;
  int Mp, Np;         // plane rows of A and B (multiples of 256)
  int n_kb;           // 128-byte atoms of K
  int tiles_m, tiles_n, splits, kb_per_split;
  int n_terms;
  int term_a[kGMaxTerms], term_b[kGMaxTerms];
  int vec;            // C rows can take 16-byte stores (ldc % 4 == 0, C 16-byte aligned)
  float alpha, beta;
};

__device__ __forceinline__ void gemm_decode(const GemmParams& P, int tile, int* m, int* n, int* sp) {
  *sp = tile % P.splits;
  const int rest = tile / P.splits;
  *m = rest % P.tiles_m;
  *n = rest / P.tiles_m;
}

__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void* map, int32_t x, int32_t y,
                                                 uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cta.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(map), "r"(x), "r"(y), "r"(bar_cluster)
      : "memory");
}

__global__ void __launch_bounds__(kGThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                const __grid_constant__ GemmParams P) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_addr(smem) & 1023u) {
    if (threadIdx.x == 0) atomicOr(P.err, 2);
    return;
  }
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int first = static_cast<int>(cluster_id_x());
  const int step = static_cast<int>(nclusters_x());
  const int total = P.tiles_m * P.tiles_n * P.splits;
  uint8_t* sA = smem;                                 // stage s: A atom at s * kGStageBytes
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kGStages * kGStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kGStages;
  uint64_t* tfull = bars + 2 * kGStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* sTmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* sAbort = reinterpret_cast<volatile int*>(sTmem + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(smem_addr(&full[s]), 2);   // one expect_tx per CTA + the TMA bytes
      mbar_init(smem_addr(&empty[s]), 1);  // the leader's multicast commit
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_addr(&tfull[a]), 1);
      mbar_init(smem_addr(&tempty[a]), 2 * kGEpiWarps);
    }
    mbar_init(smem_addr(drain), 1);
    *sAbort = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&tmap_a);
    tma_prefetch_map(&tmap_b);
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_addr(sTmem), kGTmemCols);
    tmem_relinquish_pair();
  }
  __syncthreads();
  cluster_sync();
  tc_fence_after_sync();
  const uint32_t tmem_base = *sTmem;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = first; tile < total && ok; tile += step) {
        int m, n, sp;
        gemm_decode(P, tile, &m, &n, &sp);
        const int kb0 = sp * P.kb_per_split, kb1 = min(P.n_kb, kb0 + P.kb_per_split);
        const int arow = m * kGTile + static_cast<int>(rank) * kGRows;
        const int brow = n * kGTile + static_cast<int>(rank) * kGRows;
        for (int kb = kb0; kb < kb1 && ok; ++kb) {
          for (int t = 0; t < P.n_terms; ++t) {
            if (!mbar_wait(smem_addr(&empty[stage]), phase ^ 1)) {
              atomicOr(P.err, 1);
              *sAbort = 1;
              ok = false;
              break;
            }
            const uint32_t fb = mapa_shared(smem_addr(&full[stage]), 0);
            mbar_arrive_expect_tx_cluster(fb, kGStageBytes);
            const uint32_t dst = smem_addr(sA + stage * kGStageBytes);
            tma_load_2d_pair(dst, &tmap_a, kb * 64, P.term_a[t] * P.Mp + arow, fb);
            tma_load_2d_pair(dst + kGAtomBytes, &tmap_b, kb * 64, P.term_b[t] * P.Np + brow, fb);
            if (++stage == kGStages) {
              stage = 0;
              phase ^= 1;
            }
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    if (lane == 0 && leader) {
      const uint32_t idesc = make_idesc(1u, kGTile, kGTile);
      const uint64_t desc0 = sw128_kmajor_desc(smem_addr(sA));
      const uint32_t step_s = kGStageBytes >> 4, atom = kGAtomBytes >> 4;
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = first; tile < total && ok; tile += step) {
        int m, n, sp;
        gemm_decode(P, tile, &m, &n, &sp);
        const int kb0 = sp * P.kb_per_split, kb1 = min(P.n_kb, kb0 + P.kb_per_split);
        for (int kb = kb0; kb < kb1 && ok; ++kb) {
          // one K atom per accumulator (the accumulator adds by truncation)
          if (!mbar_wait(smem_addr(&tempty[acc]), acc_phase ^ 1)) {
            atomicOr(P.err, 1);
            *sAbort = 1;
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * kGTile);
          uint32_t accumulate = 0;
          for (int t = 0; t < P.n_terms; ++t) {
            if (!mbar_wait(smem_addr(&full[stage]), phase)) {
              atomicOr(P.err, 1);
              *sAbort = 1;
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint64_t ad = desc0 + stage * step_s;
            const uint64_t bd = ad + atom;
            mma_bf16_pair(d_tmem, ad, bd, idesc, accumulate);
            mma_bf16_pair(d_tmem, ad + 2, bd + 2, idesc, 1);
            mma_bf16_pair(d_tmem, ad + 4, bd + 4, idesc, 1);
            mma_bf16_pair(d_tmem, ad + 6, bd + 6, idesc, 1);
            accumulate = 1;
            tc_commit_pair(smem_addr(&empty[stage]), 0x3);
            if (++stage == kGStages) {
              stage = 0;
              phase ^= 1;
            }
          }
          if (!ok) break;
          tc_commit_pair(smem_addr(&tfull[acc]), 0x3);
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1;
        }
      }
      tc_commit_pair(smem_addr(drain), 0x3);
    }
    if (lane == 0) {
      if (!mbar_wait(smem_addr(drain), 0)) {
        atomicOr(P.err, 1);
        *sAbort = 1;
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int e = warp - 2;       // 0..15
    const int q = warp & 3;       // TMEM lane quarter this warp may access
    const int cg = e >> 2;        // column group: columns cg * 64 .. + 63
    const int row_in = q * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    bool ok = true;
    for (int tile = first; tile < total && ok; tile += step) {
      int m, n, sp;
      gemm_decode(P, tile, &m, &n, &sp);
      const int kb0 = sp * P.kb_per_split, kb1 = min(P.n_kb, kb0 + P.kb_per_split);
      float sum[kGEpiCols];
#pragma unroll
      for (int i = 0; i < kGEpiCols; ++i) sum[i] = 0.f;
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait(smem_addr(&tfull[acc]), acc_phase)) {
          atomicOr(P.err, 1);
          *sAbort = 1;
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t ta = tmem_base + static_cast<uint32_t>(acc * kGTile + cg * kGEpiCols) +
                            (static_cast<uint32_t>(q * 32) << 16);
#pragma unroll
        for (int c0 = 0; c0 < kGEpiCols; c0 += 16) {
          uint32_t v[16];
          tmem_load_16(ta + static_cast<uint32_t>(c0), v);
#pragma unroll
          for (int i = 0; i < 16; ++i) sum[c0 + i] = __fadd_rn(sum[c0 + i], __uint_as_float(v[i]));
        }
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) {
          if (rank == 0)
            mbar_arrive_relaxed(smem_addr(&tempty[acc]));
          else
            mbar_arrive_cluster(mapa_shared(smem_addr(&tempty[acc]), 0));
        }
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
      if (!ok) break;
      const int row = m * kGTile + static_cast<int>(rank) * kGRows + row_in;
      const int col0 = n * kGTile + cg * kGEpiCols;
      if (row >= P.M) continue;
      if (P.splits > 1) {
        float* dst = P.partial + (static_cast<int64_t>(sp) * P.M + row) * P.N + col0;
        const bool v4 = (P.N % 4) == 0 && (reinterpret_cast<uintptr_t>(P.partial) & 15u) == 0;
#pragma unroll
        for (int i = 0; i < kGEpiCols; i += 4) {
          if (v4 && col0 + i + 4 <= P.N) {
            *reinterpret_cast<float4*>(dst + i) =
                make_float4(sum[i], sum[i + 1], sum[i + 2], sum[i + 3]);
          } else {
            for (int k = 0; k < 4; ++k)
              if (col0 + i + k < P.N) dst[i + k] = sum[i + k];
          }
        }
      } else {
        float* dst = P.C + static_cast<int64_t>(row) * P.ldc + col0;
        const float* cin = P.Cin + static_cast<int64_t>(row) * P.ldc + col0;
        const int dcol = row - col0;  // this row's diagonal element, if in range
#pragma unroll
        for (int i = 0; i < kGEpiCols; i += 4) {
          if (P.vec && col0 + i + 4 <= P.N) {
            float o[4] = {P.alpha * sum[i], P.alpha * sum[i + 1], P.alpha * sum[i + 2],
                          P.alpha * sum[i + 3]};
            if (P.beta != 0.f) {
              const float4 c = *reinterpret_cast<const float4*>(cin + i);
              o[0] = fmaf(P.beta, c.x, o[0]);
              o[1] = fmaf(P.beta, c.y, o[1]);
              o[2] = fmaf(P.beta, c.z, o[2]);
              o[3] = fmaf(P.beta, c.w, o[3]);
            }
#pragma unroll
            for (int k = 0; k < 4; ++k)
              if (dcol == i + k) o[k] += P.diag;
            *reinterpret_cast<float4*>(dst + i) = make_float4(o[0], o[1], o[2], o[3]);
          } else {
            for (int k = 0; k < 4; ++k) {
              if (col0 + i + k >= P.N) continue;
              float o = P.alpha * sum[i + k];
              if (P.beta != 0.f) o = fmaf(P.beta, cin[i + k], o);
              if (dcol == i + k) o += P.diag;
              dst[i + k] = o;
            }
          }
        }
      }
    }
  }

  __syncthreads();
  if (*sAbort) {
    // let copies that may still be in flight land before the CTA exits
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 200000ull) {
    }
  }
  cluster_sync();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc_pair(tmem_base, kGTmemCols);
  }
}

// C = alpha * sum_s partial[s] + beta * C_in + diag I.
__global__ void gemm_reduce_kernel(const float* partial, int splits, int M, int N, float* C,
                                   const float* Cin, int64_t ldc, float alpha, float beta,
                                   float diag) {
  const int64_t n_el = static_cast<int64_t>(M) * N;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_el;
       i += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += partial[k * n_el + i];
    const int64_t r = i / N, c = i - r * N;
    float o = alpha * s;
    if (beta != 0.f) o = fmaf(beta, Cin[r * ldc + c], o);
    if (r == c) o += diag;
    C[r * ldc + c] = o;
  }
}

// The three bf16 planes of an fp32 operand, K-major: plane p at
// out + p * rows_p * k_p, element (r, k) at r * k_p + k, for the view
// x(r, k) = src[r * s_r + k * s_k], r < R, k < K; zero outside.  A block
// handles 32 rows x 64 k through a shared-memory tile, read along whichever
// index is contiguous in the source and written along k.
__global__ void gemm_split_kernel(const float* src, int R, int K, int64_t s_r, int64_t s_k,
                                  __nv_bfloat16* out, int rows_p, int k_p) {
  __shared__ float tile[32][65];
  const int r0 = blockIdx.y * 32, k0 = blockIdx.x * 64;
  const int tid = threadIdx.x;  // 256 threads
  if (s_r == 1 && s_k != 1) {
    // contiguous along r: thread reads rows r0 + (tid & 31), k = k0 + (tid >> 5) + 8 i
    for (int i = 0; i < 8; ++i) {
      const int r = r0 + (tid & 31), k = k0 + (tid >> 5) + 8 * i;
      tile[tid & 31][(tid >> 5) + 8 * i] = (r < R && k < K) ? src[r + k * s_k] : 0.f;
    }
  } else {
    for (int i = 0; i < 8; ++i) {
      const int rr = (tid >> 6) + 4 * i, kk = tid & 63;
      const int r = r0 + rr, k = k0 + kk;
      tile[rr][kk] = (r < R && k < K) ? src[r * s_r + k * s_k] : 0.f;
    }
  }
  __syncthreads();
  const int64_t plane = static_cast<int64_t>(rows_p) * k_p;
  for (int i = 0; i < 4; ++i) {
    const int rr = (tid >> 5) + 8 * i, kk = 2 * (tid & 31);
    const int r = r0 + rr, k = k0 + kk;
    if (r >= rows_p || k >= k_p) continue;
    const float a = tile[rr][kk], b = tile[rr][kk + 1];
    const __nv_bfloat162 h0 = __floats2bfloat162_rn(a, b);
    const float2 f0 = __bfloat1622float2(h0);
    const float ra = a - f0.x, rb = b - f0.y;
    const __nv_bfloat162 h1 = __floats2bfloat162_rn(ra, rb);
    const float2 f1 = __bfloat1622float2(h1);
    const __nv_bfloat162 h2 = __floats2bfloat162_rn(ra - f1.x, rb - f1.y);
    __nv_bfloat162* o = reinterpret_cast<__nv_bfloat162*>(out + static_cast<int64_t>(r) * k_p + k);
    o[0] = h0;
    o[plane / 2] = h1;
    o[plane] = h2;
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn gemm_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// [rows][k_p] bf16 planes, box 128 rows x 64 k, 128-byte swizzle.
hf_status plane_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t k_p) {
  EncodeTiledFn fn = gemm_encode_fn();
  if (!fn) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return HF_ERR_CUDA;
  }
  const cuuint64_t dims[2] = {k_p, rows};
  const cuuint64_t strides[1] = {k_p * 2};
  const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(kGRows)};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (error " + std::to_string((int)r) + ")");
    return HF_ERR_CUDA;
  }
  return HF_OK;
}

int64_t round_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

size_t gemm_smem_bytes() {
  return static_cast<size_t>(kGStages) * kGStageBytes + (2 * kGStages + 5) * sizeof(uint64_t) + 8;
}

}  // namespace

size_t gemm_planes_bytes(int64_t rows, int64_t K) {
  return static_cast<size_t>(3 * round_up(rows, kGTile) * round_up(K, 64) * 2);
}

hf_status gemm_f32(cudaStream_t s, const GemmWork& wk, int M, int N, int K, float alpha,
                   const float* A, int64_t a_i, int64_t a_k, const float* B, int64_t b_k,
                   int64_t b_j, float beta, float* C, int64_t ldc, const float* Cin,
                   float diag) {
  if (Cin == nullptr) Cin = C;
  if (M <= 0 || N <= 0) return HF_OK;
  if (K <= 0) {
    set_error("hf_recolor_fit: internal error: a product with K = 0");
    return HF_ERR_INVALID_ARGUMENT;
  }
  const int64_t Mp = round_up(M, kGTile), Np = round_up(N, kGTile), Kp = round_up(K, 64);
  const size_t a_bytes = static_cast<size_t>(3 * Mp * Kp * 2);
  const size_t b_bytes = static_cast<size_t>(3 * Np * Kp * 2);
  // op(B)'s K-major plane is (j, k) -> B[k * b_k + j * b_j]; it is op(A)'s
  // when both views read the same matrix the same way (X^T X)
  const bool same = A == B && a_i == b_j && a_k == b_k && M == N;
  if (a_bytes > wk.planes_a_bytes || (!same && b_bytes > wk.planes_b_bytes)) {
    set_error("hf_recolor_fit: internal error: product planes exceed the workspace");
    return HF_ERR_INVALID_ARGUMENT;
  }
  __nv_bfloat16* pa = static_cast<__nv_bfloat16*>(wk.planes_a);
  __nv_bfloat16* pb = same ? pa : static_cast<__nv_bfloat16*>(wk.planes_b);
  {
    dim3 grid(static_cast<unsigned>(Kp / 64), static_cast<unsigned>(Mp / 32));
    gemm_split_kernel<<<grid, 256, 0, s>>>(A, M, K, a_i, a_k, pa, static_cast<int>(Mp),
                                           static_cast<int>(Kp));
  }
  if (!same) {
    dim3 grid(static_cast<unsigned>(Kp / 64), static_cast<unsigned>(Np / 32));
    gemm_split_kernel<<<grid, 256, 0, s>>>(B, N, K, b_j, b_k, pb, static_cast<int>(Np),
                                           static_cast<int>(Kp));
  }
  HF_CUDA_TRY(cudaGetLastError(), "hf_recolor_fit: operand split launch");
  CUtensorMap ma, mb;
  hf_status st = plane_map(&ma, pa, static_cast<uint64_t>(3 * Mp), static_cast<uint64_t>(Kp));
  if (st != HF_OK) return st;
  st = plane_map(&mb, pb, static_cast<uint64_t>(3 * Np), static_cast<uint64_t>(Kp));
  if (st != HF_OK) return st;

  GemmParams P;
  std::memset(&P, 0, sizeof(P));
  P.C = C;
  P.Cin = Cin;
  P.diag = diag;
  P.ldc = ldc;
  P.err = wk.err;
  P.M = M;
  P.N = N;
  P.Mp = static_cast<int>(Mp);
  P.Np = static_cast<int>(Np);
  P.n_kb = static_cast<int>(Kp / 64);
  P.tiles_m = static_cast<int>(Mp / kGTile);
  P.tiles_n = static_cast<int>(Np / kGTile);
  // terms a_i b_j with i + j <= 2, smallest first: an accumulator that
  // adds by truncation loses at most an ulp of its current magnitude per add
  const int ta[kGMaxTerms] = {2, 1, 0, 1, 0, 0}, tb[kGMaxTerms] = {0, 1, 2, 0, 1, 0};
  P.n_terms = kGMaxTerms;
  for (int t = 0; t < kGMaxTerms; ++t) {
    P.term_a[t] = ta[t];
    P.term_b[t] = tb[t];
  }
  P.vec = (ldc % 4 == 0 && ((reinterpret_cast<uintptr_t>(C) | reinterpret_cast<uintptr_t>(Cin)) &
                             15u) == 0)
              ? 1
              : 0;
  P.alpha = alpha;
  P.beta = beta;
  const int pairs = std::max(1, device_sm_count() / 2);
  const int tiles = P.tiles_m * P.tiles_n;
  // split K while the tiles leave SM pairs idle, keeping >= 4 atoms per split
  int splits = 1;
  while (tiles * splits * 2 <= pairs && P.n_kb / (splits * 2) >= 4 &&
         static_cast<size_t>(splits * 2) * M * N * 4 <= wk.partial_bytes)
    splits *= 2;
  // no split may be empty: its tile would be written from a stale accumulator
  P.kb_per_split = (P.n_kb + splits - 1) / splits;
  P.splits = (P.n_kb + P.kb_per_split - 1) / P.kb_per_split;
  splits = P.splits;
  P.partial = wk.partial;
  const size_t smem = gemm_smem_bytes();
  HF_CUDA_TRY(cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(smem)),
              "hf_recolor_fit: product shared memory");
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  const int clusters = std::max(1, std::min(pairs, tiles * splits));
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  cfg.blockDim = dim3(kGThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  HF_CUDA_TRY(cudaLaunchKernelEx(&cfg, gemm_kernel, ma, mb, P), "hf_recolor_fit: product launch");
  if (splits > 1) {
    const int64_t n_el = static_cast<int64_t>(M) * N;
    const int grid = static_cast<int>(std::min<int64_t>((n_el + 255) / 256, 4096));
    gemm_reduce_kernel<<<grid, 256, 0, s>>>(wk.partial, splits, M, N, C, Cin, ldc, alpha, beta,
                                            diag);
    HF_CUDA_TRY(cudaGetLastError(), "hf_recolor_fit: product reduce launch");
  }
  return HF_OK;
}

}  // namespace hf

using namespace hf;

namespace {

struct DebugGemmLayout {
  size_t planes_a, planes_b, partial, err, total, planes_bytes, partial_bytes;
};

DebugGemmLayout debug_gemm_layout(int M, int N, int K) {
  DebugGemmLayout L{};
  auto up = [](size_t x) { return (x + 255) / 256 * 256; };
  L.planes_bytes = gemm_planes_bytes(std::max(M, N), K);
  L.partial_bytes = static_cast<size_t>(2) * 96 * 65536 * sizeof(float);
  L.planes_a = 0;
  L.planes_b = up(L.planes_bytes);
  L.partial = L.planes_b + up(L.planes_bytes);
  L.err = L.partial + up(L.partial_bytes);
  L.total = L.err + 256;
  return L;
}

}  // namespace

extern "C" hf_status hf_debug_matmul_workspace_size(int32_t M, int32_t N, int32_t K,
                                                    size_t* bytes) {
  if (!bytes || M < 1 || N < 1 || K < 1) {
    set_error("hf_debug_matmul_workspace_size: need M, N, K >= 1");
    return HF_ERR_INVALID_ARGUMENT;
  }
  *bytes = debug_gemm_layout(M, N, K).total;
  return HF_OK;
}

extern "C" hf_status hf_debug_matmul_f32(int32_t M, int32_t N, int32_t K, float alpha,
                                         const float* d_A, int64_t a_i, int64_t a_k,
                                         const float* d_B, int64_t b_k, int64_t b_j, float beta,
                                         float* d_C, int64_t ldc, void* d_workspace,
                                         size_t workspace_bytes, int32_t* h_err,
                                         hf_stream_t stream) {
  if (M < 1 || N < 1 || K < 1 || !d_A || !d_B || !d_C || ldc < N) {
    set_error("hf_debug_matmul_f32: need M, N, K >= 1, non-null matrices and ldc >= N");
    return HF_ERR_INVALID_ARGUMENT;
  }
  const DebugGemmLayout L = debug_gemm_layout(M, N, K);
  if (!d_workspace || workspace_bytes < L.total ||
      (reinterpret_cast<uintptr_t>(d_workspace) & 255u)) {
    set_error("hf_debug_matmul_f32: workspace missing, too small or not 256-byte aligned");
    return HF_ERR_WORKSPACE;
  }
  char* ws = static_cast<char*>(d_workspace);
  GemmWork wk;
  wk.planes_a = ws + L.planes_a;
  wk.planes_b = ws + L.planes_b;
  wk.planes_a_bytes = wk.planes_b_bytes = L.planes_bytes;
  wk.partial = reinterpret_cast<float*>(ws + L.partial);
  wk.partial_bytes = L.partial_bytes;
  wk.err = reinterpret_cast<int32_t*>(ws + L.err);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  HF_CUDA_TRY(cudaMemsetAsync(wk.err, 0, sizeof(int32_t), s), "hf_debug_matmul_f32: clear");
  const hf_status st =
      gemm_f32(s, wk, M, N, K, alpha, d_A, a_i, a_k, d_B, b_k, b_j, beta, d_C, ldc, d_C, 0.f);
  if (st != HF_OK) return st;
  if (h_err) {
    HF_CUDA_TRY(cudaMemcpyAsync(h_err, wk.err, sizeof(int32_t), cudaMemcpyDeviceToHost, s),
                "hf_debug_matmul_f32: read back");
    HF_CUDA_TRY(cudaStreamSynchronize(s), "hf_debug_matmul_f32: synchronize");
  }
  return HF_OK;
}
