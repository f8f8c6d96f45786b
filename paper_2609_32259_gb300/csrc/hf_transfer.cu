// hf_transfer: the fused HeteroFold K/V map (Eq. 1-2 and Eq. 9).
//
// For receiver layer l and role c the receiver cache rows are
//   y_j = (x_j / r_{l,c}) A_final_{l,c} + b_final_{l,c},
//   x_j = [ pooled sender layer t1 || t2 || t3 ] at the alignment row of j,
// reshaped to receiver heads; keys then get the optional receiver key norm
// and RoPE at the receiver position of j.
//
// Receiver tokens whose alignment rows are identical have identical y
// before RoPE, so the contraction runs over the U distinct rows only; each
// distinct row covers a run of consecutive receiver rows [run_ptr[u],
// run_ptr[u+1]) at consecutive positions from upos[u], and the epilogue
// writes y (rotated per position for K) to every row of its run.
//
// One persistent CTA per SM walks tiles (l, c, 128 distinct rows, BN
// receiver columns) with warp-specialised roles:
//   warp 0      TMA producer of the map tile W[l][c][n0:n0+BN][k0:k0+BK]
//               (2-D tiled load, 128-byte swizzle);
//   warp 1      TMEM allocator and the single thread issuing tcgen05.mma
//               (M = 128, N = BN, K = 16 bf16 / 8 tf32 per instruction) into
//               one of two TMEM accumulators;
//   warps 2-9   epilogue, two groups of four warps (one per TMEM lane
//               quarter), each group owning half of the tile's columns;
//   warps 10-13 A tile builders.  When every map input row is one sender row
//               (Token Alignment with the three-layer neighbourhood) they copy
//               the 128 sender rows with cp.async, eight lanes per 128-byte
//               row; for pooled or blended rows they sum weighted sender rows
//               in fp32 registers and round once.  Both write the 128-byte
//               swizzled layout and fence it to the async proxy before
//               arriving on the stage barrier.
// Pipeline hand-offs use mbarriers with bounded waits; nothing traps.
#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>
#include <string>

#include "hf_device.cuh"
#include "hf_internal.h"

namespace hf {
namespace {

constexpr int kBM = 128;                 // distinct rows per tile (UMMA M)
constexpr int kThreads = 448;            // 14 warps
constexpr int kStageABytes = kBM * 128;  // 128 rows x 128 bytes
constexpr int kStgFloats = kBM * 32;     // epilogue staging per group
constexpr int kRunStride = 132;          // run starts / positions per group (129 used)
constexpr int kMaxStages = 8;
constexpr int kLag = 3;                  // cp.async groups in flight per loader thread
constexpr int kTmemCols = 512;           // two accumulators of up to 256 columns

struct XferParams {
  const void* sender;
  void* receiver;
  const float* bias;
  const float* inv_r;
  const LayerSegs* segs;
  const float* inv_freq;
  const float* knorm_w;
  const int32_t* row_ptr;
  const int32_t* col;
  const float* w;
  const int32_t* run_ptr;
  const int32_t* ucol;
  const int32_t* upos;
  const int32_t* dst_row;
  const int32_t* n_distinct;
  int32_t* status;
  int64_t T_s;        // sender rows per (layer, role)
  int64_t recv_rows;  // receiver rows per (layer, role) in receiver_kv
  int L_r, d_s, d_r, D_r;
  int n_kb, kb_per_seg, BN, n_tiles_n, groups, stages;
  int rope, paged, knorm;
  float knorm_eps;
  uint32_t idesc;
};

template <typename T>
struct Elem;
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kBK = 64;  // elements per 128-byte k-block
};
template <>
struct Elem<float> {
  static constexpr int kBK = 32;
};

__device__ __forceinline__ void store_pair(__nv_bfloat16* p, float a, float b) {
  *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(a, b);
}
__device__ __forceinline__ void store_pair(float* p, float a, float b) {
  *reinterpret_cast<float2*>(p) = make_float2(a, b);
}

__device__ __forceinline__ void decode_tile(int tile, int tiles_per_lc, int n_tiles_n, int* lc,
                                            int* m, int* n) {
  *lc = tile / tiles_per_lc;
  const int rem = tile - *lc * tiles_per_lc;
  *m = rem / n_tiles_n;
  *n = rem - *m * n_tiles_n;
}

__device__ __forceinline__ void raise_timeout(const XferParams& P, volatile int* abort_flag) {
  atomicOr(P.status, HF_CHECK_TIMEOUT);
  *abort_flag = 1;
}

// Accumulates w * (8 bf16 | 4 fp32 values) into acc.
__device__ __forceinline__ void accum16(const uint4& v, float wt, float* acc,
                                        const __nv_bfloat16*) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(h[i]);
    acc[2 * i] = fmaf(wt, f.x, acc[2 * i]);
    acc[2 * i + 1] = fmaf(wt, f.y, acc[2 * i + 1]);
  }
}
__device__ __forceinline__ void accum16(const uint4& v, float wt, float* acc, const float*) {
  acc[0] = fmaf(wt, __uint_as_float(v.x), acc[0]);
  acc[1] = fmaf(wt, __uint_as_float(v.y), acc[1]);
  acc[2] = fmaf(wt, __uint_as_float(v.z), acc[2]);
  acc[3] = fmaf(wt, __uint_as_float(v.w), acc[3]);
}
__device__ __forceinline__ uint4 pack16(const float* a, const __nv_bfloat16*) {
  uint4 r;
  __nv_bfloat162 h0 = __floats2bfloat162_rn(a[0], a[1]), h1 = __floats2bfloat162_rn(a[2], a[3]);
  __nv_bfloat162 h2 = __floats2bfloat162_rn(a[4], a[5]), h3 = __floats2bfloat162_rn(a[6], a[7]);
  r.x = *reinterpret_cast<uint32_t*>(&h0);
  r.y = *reinterpret_cast<uint32_t*>(&h1);
  r.z = *reinterpret_cast<uint32_t*>(&h2);
  r.w = *reinterpret_cast<uint32_t*>(&h3);
  return r;
}
__device__ __forceinline__ uint4 pack16(const float* a, const float*) {
  return make_uint4(__float_as_uint(a[0]), __float_as_uint(a[1]), __float_as_uint(a[2]),
                    __float_as_uint(a[3]));
}

// One chain of the epilogue's position walk: a lane's two rotation pairs at
// receiver row j (row u of the tile), with RoPE state carried from the
// chain's previous position four rows back.
struct Chain {
  int u;          // tile row holding the current position
  int expect;     // position this chain expects next (angle-addition valid)
  float cs0, sn0, cs1, sn1;
};

template <typename T>
__device__ __forceinline__ void walk_step(Chain& ch, int j, int it, const int32_t* srun,
                                          const int32_t* supos, const float* stg, int pl, int p0,
                                          bool do_rope, float f0, float f1, float C0, float S0,
                                          float C1, float S1, const XferParams& P, T* out_lc,
                                          int ocol, int q, int half) {
  const int drow = P.paged ? __ldg(P.dst_row + j) : j;
  while (srun[ch.u + 1] <= j) ++ch.u;
  const int u = ch.u;
  const float* urow = stg + u * 32;
  const int sw = u & 7;
  const float2 lo = *reinterpret_cast<const float2*>(urow + (((pl >> 1) ^ sw) << 2) + (p0 & 3));
  const float2 hi =
      *reinterpret_cast<const float2*>(urow + (((4 + (pl >> 1)) ^ sw) << 2) + (p0 & 3));
  float a0 = lo.x, a1 = lo.y, b0 = hi.x, b1 = hi.y;
  if (do_rope) {
    const int p = supos[u] + (j - srun[u]);
    if (p != ch.expect || (it & 15) == 0) {
      rope_sincos(p, f0, &ch.sn0, &ch.cs0);
      rope_sincos(p, f1, &ch.sn1, &ch.cs1);
    } else {  // advance the angle by four positions
      const float t0 = ch.cs0 * C0 - ch.sn0 * S0;
      ch.sn0 = ch.sn0 * C0 + ch.cs0 * S0;
      ch.cs0 = t0;
      const float t1 = ch.cs1 * C1 - ch.sn1 * S1;
      ch.sn1 = ch.sn1 * C1 + ch.cs1 * S1;
      ch.cs1 = t1;
    }
    ch.expect = p + 4;
    const float oa0 = a0 * ch.cs0 - b0 * ch.sn0, ob0 = b0 * ch.cs0 + a0 * ch.sn0;
    const float oa1 = a1 * ch.cs1 - b1 * ch.sn1, ob1 = b1 * ch.cs1 + a1 * ch.sn1;
    a0 = oa0;
    b0 = ob0;
    a1 = oa1;
    b1 = ob1;
  }
  if (drow >= 0) {
    T* o = out_lc + static_cast<int64_t>(drow) * P.d_r + ocol;
    store_pair(o + q + p0, a0, a1);
    store_pair(o + half + q + p0, b0, b1);
  }
}

// Last u in [0, nrows) with srun[u] <= j.
__device__ __forceinline__ int find_row(const int32_t* srun, int nrows, int j) {
  int lo = 0, hi = nrows - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (srun[mid] <= j) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <typename T, bool kGather>
__global__ void __launch_bounds__(kThreads, 1)
    transfer_kernel(const __grid_constant__ CUtensorMap tmap_w, const XferParams P) {
  constexpr int kBK = Elem<T>::kBK;
  constexpr int kPerChunk = 16 / sizeof(T);  // elements per 16-byte chunk
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_addr(smem) & 1023u) {  // the swizzled stages need 1024-byte alignment
    if (threadIdx.x == 0) atomicOr(P.status, HF_CHECK_INTERNAL);
    return;
  }
  const int stages = P.stages;
  const int stage_b_bytes = P.BN * 128;
  uint8_t* sA = smem;
  uint8_t* sB = sA + stages * kStageABytes;
  float* sStg = reinterpret_cast<float*>(sB + stages * stage_b_bytes);
  int32_t* sRun = reinterpret_cast<int32_t*>(sStg + 2 * kStgFloats);
  int32_t* sUpos = sRun + 2 * kRunStride;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sUpos + 2 * kRunStride);
  uint64_t* full = bars;
  uint64_t* empty = bars + kMaxStages;
  uint64_t* tfull = bars + 2 * kMaxStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* sTmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* sAbort = reinterpret_cast<volatile int*>(sTmem + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(smem_addr(&full[s]), 1 + kBM);  // TMA expect_tx + 128 A builders
      mbar_init(smem_addr(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_addr(&tfull[a]), 1);
      mbar_init(smem_addr(&tempty[a]), 8);  // one arrival per epilogue warp
    }
    mbar_init(smem_addr(drain), 1);
    *sAbort = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) tma_prefetch_map(&tmap_w);
  if (warp == 1) {
    tmem_alloc(smem_addr(sTmem), kTmemCols);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem_base = *sTmem;

  const int U = *P.n_distinct;
  const int m_tiles = (U + kBM - 1) / kBM;
  const int tiles_per_lc = m_tiles * P.n_tiles_n;
  const int total_tiles = 2 * P.L_r * tiles_per_lc;

  if (warp == 0) {
    // ------------------------------------------------------------ map tiles
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < total_tiles && ok; tile += gridDim.x) {
        int lc, m, n;
        decode_tile(tile, tiles_per_lc, P.n_tiles_n, &lc, &m, &n);
        for (int kb = 0; kb < P.n_kb; ++kb) {
          if (!mbar_wait(smem_addr(&empty[stage]), phase ^ 1)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          const uint32_t fb = smem_addr(&full[stage]);
          mbar_arrive_expect_tx(fb, stage_b_bytes);
          tma_load_2d(smem_addr(sB + stage * stage_b_bytes), &tmap_w, kb * kBK,
                      lc * P.d_r + n * P.BN, fb);
          if (++stage == stages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < total_tiles && ok; tile += gridDim.x) {
        if (!mbar_wait(smem_addr(&tempty[acc]), acc_phase ^ 1)) {
          raise_timeout(P, sAbort);
          break;
        }
        tc_fence_after_sync();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * 256);
        for (int kb = 0; kb < P.n_kb; ++kb) {
          if (!mbar_wait(smem_addr(&full[stage]), phase)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t a0 = smem_addr(sA + stage * kStageABytes);
          const uint32_t b0 = smem_addr(sB + stage * stage_b_bytes);
#pragma unroll
          for (int k = 0; k < 4; ++k) {  // four 32-byte K steps per 128-byte k-block
            const uint64_t ad = sw128_kmajor_desc(a0 + 32 * k);
            const uint64_t bd = sw128_kmajor_desc(b0 + 32 * k);
            if (sizeof(T) == 2)
              mma_bf16(d_tmem, ad, bd, P.idesc, (kb | k) != 0);
            else
              mma_tf32(d_tmem, ad, bd, P.idesc, (kb | k) != 0);
          }
          tc_commit(smem_addr(&empty[stage]));
          if (++stage == stages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(smem_addr(&tfull[acc]));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
      // every issued MMA has completed before TMEM is released
      tc_commit(smem_addr(drain));
      if (!mbar_wait(smem_addr(drain), 0)) raise_timeout(P, sAbort);
    }
    __syncwarp();
  } else if (warp < 10) {
    // ------------------------------------------------------------ epilogue
    const int g = (warp - 2) >> 2;
    const int sp = warp & 3;  // TMEM lane quarter this warp may access
    const int row = sp * 32 + lane;
    float* stg = sStg + g * kStgFloats;
    int32_t* srun = sRun + g * kRunStride;
    int32_t* supos = sUpos + g * kRunStride;
    const bool active = P.groups == 2 || g == 0;
    const int gcols = P.groups == 2 ? P.BN / 2 : P.BN;
    const int gcol0 = P.groups == 2 ? g * (P.BN / 2) : 0;
    const int D = P.D_r, half = P.D_r / 2;
    const int pg = lane >> 3, pl = lane & 7, p0 = 2 * pl;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
      int lc, m, n;
      decode_tile(tile, tiles_per_lc, P.n_tiles_n, &lc, &m, &n);
      const int c = lc & 1;
      if (!mbar_wait(smem_addr(&tfull[acc]), acc_phase)) {
        raise_timeout(P, sAbort);
        break;
      }
      tc_fence_after_sync();
      if (active) {
        const int u0 = m * kBM;
        const int nrows = min(kBM, U - u0);
        for (int i = row; i <= nrows; i += kBM) {
          srun[i] = P.run_ptr[u0 + i];
          supos[i] = i < nrows ? P.upos[u0 + i] : 0;
        }
        named_barrier_sync(1 + g, 128);
        // this warp's receiver rows [wjb, wje), walked as two chains
        const int jb = srun[0], je = srun[nrows];
        const int per = (je - jb + 3) >> 2;
        const int wjb = min(je, jb + sp * per), wje = min(je, wjb + per);
        const int hlen = (((wje - wjb + 1) >> 1) + 3) & ~3;  // chain A length, multiple of 4
        const int amid = min(wje, wjb + hlen);
        const int n_it = (hlen + 3) >> 2;
        const int ja0 = wjb + pg, jb0 = amid + pg;
        const int ua0 = ja0 < amid ? find_row(srun, nrows, ja0) : 0;
        const int ub0 = jb0 < wje ? find_row(srun, nrows, jb0) : 0;
        const float inv_r = P.inv_r[lc];
        const float* bias = P.bias + static_cast<int64_t>(lc) * P.d_r;
        const bool do_rope = P.rope && c == 0;
        const bool do_knorm = P.knorm && c == 0;
        const uint32_t ta = tmem_base + static_cast<uint32_t>(acc * 256) +
                            (static_cast<uint32_t>(sp * 32) << 16);
        T* const out_lc = reinterpret_cast<T*>(P.receiver) +
                          (static_cast<int64_t>(lc) * P.recv_rows) * P.d_r;
        for (int h0 = 0; h0 < gcols; h0 += D) {
          const int tcol = gcol0 + h0;       // accumulator column of the head
          const int ocol = n * P.BN + tcol;  // receiver feature index of the head
          float rn = 1.0f;
          if (do_knorm) {
            float ss = 0.0f;
            for (int q2 = 0; q2 < D; q2 += 16) {
              uint32_t v[16];
              tmem_load_16(ta + tcol + q2, v);
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const float y = fmaf(__uint_as_float(v[i]), inv_r, __ldg(bias + ocol + q2 + i));
                ss = fmaf(y, y, ss);
              }
            }
            rn = rsqrtf(ss / static_cast<float>(D) + P.knorm_eps);
          }
          for (int q = 0; q < half; q += 16) {
            // step 1: 16 rotation pairs (columns q.., half+q..) of every row -> smem
            uint32_t v[32];
            tmem_load_2x16(ta + tcol + q, ta + tcol + half + q, v);
            float bl[16], bh[16];
#pragma unroll
            for (int i = 0; i < 16; i += 4) {
              const float4 x = __ldg(reinterpret_cast<const float4*>(bias + ocol + q + i));
              const float4 z = __ldg(reinterpret_cast<const float4*>(bias + ocol + half + q + i));
              bl[i] = x.x; bl[i + 1] = x.y; bl[i + 2] = x.z; bl[i + 3] = x.w;
              bh[i] = z.x; bh[i + 1] = z.y; bh[i + 2] = z.z; bh[i + 3] = z.w;
            }
            float y[32];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              y[i] = fmaf(__uint_as_float(v[i]), inv_r, bl[i]);
              y[16 + i] = fmaf(__uint_as_float(v[16 + i]), inv_r, bh[i]);
            }
            if (do_knorm) {
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                y[i] *= rn * __ldg(P.knorm_w + q + i);
                y[16 + i] *= rn * __ldg(P.knorm_w + half + q + i);
              }
            }
            float* srow = stg + row * 32;
#pragma unroll
            for (int k = 0; k < 8; ++k)
              *reinterpret_cast<float4*>(srow + ((k ^ (row & 7)) << 2)) =
                  make_float4(y[4 * k], y[4 * k + 1], y[4 * k + 2], y[4 * k + 3]);
            named_barrier_sync(1 + g, 128);
            // step 2: lanes 8*pg .. 8*pg+7 own rows j = chain start + pg + 4*it
            // (two pairs each); a step advances the RoPE angle by four rows.
            float f0 = 0.f, f1 = 0.f, C0 = 1.f, S0 = 0.f, C1 = 1.f, S1 = 0.f;
            if (do_rope) {
              f0 = __ldg(P.inv_freq + q + p0);
              f1 = __ldg(P.inv_freq + q + p0 + 1);
              rope_sincos(4, f0, &S0, &C0);
              rope_sincos(4, f1, &S1, &C1);
            }
            Chain ca{ua0, INT_MIN, 1.f, 0.f, 1.f, 0.f};
            Chain cb{ub0, INT_MIN, 1.f, 0.f, 1.f, 0.f};
            for (int it = 0; it < n_it; ++it) {
              const int ja = ja0 + 4 * it, jbb = jb0 + 4 * it;
              if (ja < amid)
                walk_step<T>(ca, ja, it, srun, supos, stg, pl, p0, do_rope, f0, f1, C0, S0, C1,
                             S1, P, out_lc, ocol, q, half);
              if (jbb < wje)
                walk_step<T>(cb, jbb, it, srun, supos, stg, pl, p0, do_rope, f0, f1, C0, S0, C1,
                             S1, P, out_lc, ocol, q, half);
            }
            named_barrier_sync(1 + g, 128);
          }
        }
      }
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_addr(&tempty[acc]));
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1;
    }
  } else {
    // ------------------------------------------------------------ A builders
    const int t = threadIdx.x - 320;  // 0..127
    const T* sender = reinterpret_cast<const T*>(P.sender);
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    if (kGather) {
      // eight lanes per 128-byte row: lane -> (row 32*slab + 4*i + lane/8, chunk lane%8)
      const int slab = t >> 5, rsub = lane >> 3, ch = lane & 7;
      int pending = 0;  // committed groups whose stage arrival is still owed
      for (int tile = blockIdx.x; tile < total_tiles && ok; tile += gridDim.x) {
        int lc, m, n;
        decode_tile(tile, tiles_per_lc, P.n_tiles_n, &lc, &m, &n);
        const int l = lc >> 1, c = lc & 1;
        const LayerSegs* segs = P.segs + l;
        int64_t roff[8];
        uint32_t doff[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int r = slab * 32 + 4 * i + rsub;
          const int u = min(m * kBM + r, U - 1);
          roff[i] = static_cast<int64_t>(P.ucol[u]) * P.d_s + ch * kPerChunk;
          doff[i] = static_cast<uint32_t>(r * 128 + ((ch ^ (r & 7)) << 4));
        }
        for (int kb = 0; kb < P.n_kb; ++kb) {
          const int seg = kb / P.kb_per_seg;
          const int kin = kb - seg * P.kb_per_seg;
          if (!mbar_wait(smem_addr(&empty[stage]), phase ^ 1)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          const int tl = segs->layer[seg][0];
          const T* base = sender + (static_cast<int64_t>(tl * 2 + c) * P.T_s) * P.d_s + kin * kBK;
          const uint32_t sa = smem_addr(sA + stage * kStageABytes);
#pragma unroll
          for (int i = 0; i < 8; ++i) cp_async_16(sa + doff[i], base + roff[i]);
          cp_async_commit();
          if (pending == kLag) {
            // the group kLag k-blocks back has landed: publish its stage
            cp_async_wait<kLag>();
            fence_proxy_async_smem();
            const int s_old = (stage + stages - kLag) % stages;
            mbar_arrive(smem_addr(&full[s_old]));
          } else {
            ++pending;
          }
          if (++stage == stages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      cp_async_wait<0>();
      fence_proxy_async_smem();
      for (int k = pending; k >= 1; --k) mbar_arrive(smem_addr(&full[(stage + stages - k) % stages]));
    } else {
      // pooled CSR rows and/or blended sender layers: thread t owns tile row t
      for (int tile = blockIdx.x; tile < total_tiles && ok; tile += gridDim.x) {
        int lc, m, n;
        decode_tile(tile, tiles_per_lc, P.n_tiles_n, &lc, &m, &n);
        const int l = lc >> 1, c = lc & 1;
        const LayerSegs segs = P.segs[l];
        const int u = min(m * kBM + t, U - 1);
        const int j0 = P.run_ptr[u];
        const int e0 = P.row_ptr[j0], e1 = P.row_ptr[j0 + 1];
        for (int kb = 0; kb < P.n_kb; ++kb) {
          const int seg = kb / P.kb_per_seg;
          const int kin = kb - seg * P.kb_per_seg;
          if (!mbar_wait(smem_addr(&empty[stage]), phase ^ 1)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          float acc[kBK];
#pragma unroll
          for (int i = 0; i < kBK; ++i) acc[i] = 0.f;
          for (int ti = 0; ti < segs.n_terms[seg]; ++ti) {
            const int tl = segs.layer[seg][ti];
            const float om = segs.w[seg][ti];
            const T* base = sender + (static_cast<int64_t>(tl * 2 + c) * P.T_s) * P.d_s + kin * kBK;
            for (int e = e0; e < e1; ++e) {
              const int k = P.col[e];
              if (k < 0 || k >= P.T_s) continue;  // flagged at plan creation
              const float wt = om * P.w[e];
              const uint4* src =
                  reinterpret_cast<const uint4*>(base + static_cast<int64_t>(k) * P.d_s);
              uint4 x[8];
#pragma unroll
              for (int k2 = 0; k2 < 8; ++k2) x[k2] = __ldg(src + k2);
#pragma unroll
              for (int k2 = 0; k2 < 8; ++k2)
                accum16(x[k2], wt, acc + k2 * kPerChunk, (const T*)nullptr);
            }
          }
          uint8_t* dst = sA + stage * kStageABytes + t * 128;
#pragma unroll
          for (int k2 = 0; k2 < 8; ++k2)
            *reinterpret_cast<uint4*>(dst + ((k2 ^ (t & 7)) << 4)) =
                pack16(acc + k2 * kPerChunk, (const T*)nullptr);
          fence_proxy_async_smem();
          mbar_arrive(smem_addr(&full[stage]));
          if (++stage == stages) {
            stage = 0;
            phase ^= 1;
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
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
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

// 2-D row-major [rows][cols] tensor, box [box_rows][box_cols], 128B swizzle.
hf_status make_map(CUtensorMap* map, const void* base, bool f32, uint64_t rows, uint64_t cols,
                   uint32_t box_rows, uint32_t box_cols, CUtensorMapL2promotion promo) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) {
    set_error("cuTensorMapEncodeTiled is not available from the driver");
    return HF_ERR_CUDA;
  }
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * (f32 ? 4 : 2)};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                        2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, promo,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (error " + std::to_string((int)r) + ")");
    return HF_ERR_CUDA;
  }
  return HF_OK;
}

size_t smem_bytes(int BN, int stages) {
  return static_cast<size_t>(stages) * (kStageABytes + BN * 128) +
         2 * kStgFloats * sizeof(float) + 4 * kRunStride * sizeof(int32_t) +
         (2 * kMaxStages + 5) * sizeof(uint64_t) + 8;
}

int pick_stages(int BN) {
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  int s = 6;
  while (s > kLag + 1 && smem_bytes(BN, s) > static_cast<size_t>(optin)) --s;
  return s;
}

template <typename T, bool kGather>
hf_status launch_typed(const CUtensorMap& mw, const XferParams& P, int grid, size_t smem,
                       cudaStream_t stream) {
  auto kern = transfer_kernel<T, kGather>;
  HF_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(smem)),
              "set shared memory size");
  kern<<<grid, kThreads, smem, stream>>>(mw, P);
  HF_CUDA_TRY(cudaGetLastError(), "transfer kernel launch");
  return HF_OK;
}

}  // namespace

hf_status launch_transfer(hf_plan_s* p, const void* sender, void* receiver, cudaStream_t stream) {
  const hf_plan_desc& d = p->desc;
  if (p->T_r == 0) return HF_OK;
  const bool f32 = d.dtype == HF_F32;
  const int esize = f32 ? 4 : 2;
  const int bk = 128 / esize;
  CUtensorMap mw;
  hf_status s = make_map(&mw, d.d_W, f32, static_cast<uint64_t>(d.L_r) * 2 * p->d_r,
                         static_cast<uint64_t>(p->K), static_cast<uint32_t>(p->BN),
                         static_cast<uint32_t>(bk), CU_TENSOR_MAP_L2_PROMOTION_L2_256B);
  if (s != HF_OK) return s;
  XferParams P;
  std::memset(&P, 0, sizeof(P));
  char* ws = p->ws;
  P.sender = sender;
  P.receiver = receiver;
  P.bias = d.d_b;
  P.inv_r = reinterpret_cast<const float*>(ws + p->lay.inv_r);
  P.segs = reinterpret_cast<const LayerSegs*>(ws + p->lay.segs);
  P.inv_freq = reinterpret_cast<const float*>(ws + p->lay.inv_freq);
  P.knorm_w = d.d_knorm_w;
  P.row_ptr = d.d_row_ptr;
  P.col = d.d_col;
  P.w = d.d_w;
  P.run_ptr = reinterpret_cast<const int32_t*>(ws + p->lay.run_ptr);
  P.ucol = reinterpret_cast<const int32_t*>(ws + p->lay.ucol);
  P.upos = reinterpret_cast<const int32_t*>(ws + p->lay.upos);
  P.dst_row = reinterpret_cast<const int32_t*>(ws + p->lay.dst_row);
  P.n_distinct = reinterpret_cast<const int32_t*>(ws + p->lay.n_distinct);
  P.status = reinterpret_cast<int32_t*>(ws + p->lay.status);
  P.T_s = p->T_s;
  P.recv_rows = d.paged ? static_cast<int64_t>(d.n_blocks) * d.block_size : p->T_r;
  P.L_r = d.L_r;
  P.d_s = p->d_s;
  P.d_r = p->d_r;
  P.D_r = d.D_r;
  P.n_kb = p->K / bk;
  P.kb_per_seg = p->d_s / bk;
  P.BN = p->BN;
  P.n_tiles_n = p->d_r / p->BN;
  P.groups = p->groups;
  P.stages = pick_stages(p->BN);
  P.rope = d.theta_r > 0.0 ? 1 : 0;
  P.paged = d.paged ? 1 : 0;
  P.knorm = d.d_knorm_w ? 1 : 0;
  P.knorm_eps = d.knorm_eps;
  P.idesc = make_idesc(f32 ? 2u : 1u, kBM, p->BN);
  const size_t smem = smem_bytes(p->BN, P.stages);
  const int64_t max_tiles =
      2LL * d.L_r * ((p->T_r + kBM - 1) / kBM) * static_cast<int64_t>(P.n_tiles_n);
  const int grid = static_cast<int>(std::min<int64_t>(device_sm_count(), max_tiles));
  if (f32)
    return p->gather ? launch_typed<float, true>(mw, P, grid, smem, stream)
                     : launch_typed<float, false>(mw, P, grid, smem, stream);
  return p->gather ? launch_typed<__nv_bfloat16, true>(mw, P, grid, smem, stream)
                   : launch_typed<__nv_bfloat16, false>(mw, P, grid, smem, stream);
}

}  // namespace hf

extern "C" hf_status hf_transfer(hf_plan plan, const void* sender_kv, void* receiver_kv,
                                 hf_stream_t stream) {
  if (!plan) {
    hf::set_error("hf_transfer: null plan");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (plan->T_r > 0 && (!sender_kv || !receiver_kv)) {
    hf::set_error("hf_transfer: null cache pointer");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if ((reinterpret_cast<uintptr_t>(sender_kv) | reinterpret_cast<uintptr_t>(receiver_kv) |
       reinterpret_cast<uintptr_t>(plan->desc.d_W)) & 15u) {
    hf::set_error("hf_transfer: caches and maps must be 16-byte aligned");
    return HF_ERR_INVALID_ARGUMENT;
  }
  return hf::launch_transfer(plan, sender_kv, receiver_kv, reinterpret_cast<cudaStream_t>(stream));
}
