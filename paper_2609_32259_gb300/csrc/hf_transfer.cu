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
// Persistent clusters of two CTAs (one pair per SM pair) walk pair tiles
// (l, c, 256 distinct rows, BN receiver columns); each CTA owns 128 of the
// rows and half of the columns' map rows, with warp-specialised roles:
//   warp 0      TMA producer of this CTA's half of the map tile
//               W[l][c][n0:n0+BN][k0:k0+64 bf16] (2-D tiled load, 128-byte
//               swizzle), one 128-byte atom of K per B stage;
//   warp 1      TMEM allocator; in the leader CTA, the single thread issuing
//               tcgen05.mma.cta_group::2 (M = 256, N = BN, K = 16 bf16 /
//               8 tf32 per instruction) into one of two TMEM accumulators;
//   warps 2-11  epilogue of the CTA's 128 rows (warps 2-9 read TMEM);
//   warps 12-15 A tile builders, two atoms of K per A stage.  When every map
//               input row is one sender row (Token Alignment with the
//               three-layer neighbourhood) they copy the 128 sender rows with
//               cp.async, eight lanes per 128-byte row; for pooled or blended
//               rows they sum weighted sender rows in fp32 registers and round
//               once, or write the rounded row and its rounding residual as
//               two atoms (split operands).  Both write the 128-byte swizzled
//               layout and fence it to the async proxy before arriving on the
//               stage barrier.
// Overlap mean pooling is linear, so by default it follows the map: the
// tile rows of a CTA are a window of 128 consecutive aligned sender tokens
// and the epilogue pools the mapped rows of each receiver row's columns
// (pam_epilogue).  Plans whose rows the builders compute use wide tiles:
// two 256-column blocks per tile in the two accumulators, so each built A
// stage feeds twice the MMAs.
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

constexpr int kBM = 128;                 // distinct rows per CTA of a pair tile
constexpr int kPairRows = 2 * kBM;       // distinct rows per pair tile (UMMA M = 256)
constexpr int kEpiWarps = 10;            // epilogue: warps 2-11 (8 of them read TMEM)
constexpr int kBuilderWarps = 4;         // A tile builders: warps 12-15
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kThreads = 64 + kEpiThreads + 32 * kBuilderWarps;  // 16 warps
constexpr int kAtoms = 2;                // 128-byte swizzle atoms (k-blocks) per A stage (a B stage holds one)
constexpr int kAtomABytes = kBM * 128;   // 128 rows x 128 bytes
constexpr int kStageABytes = kAtoms * kAtomABytes;
constexpr int kStgFloats = kBM * 64;     // epilogue staging: 128 rows x 2 heads x 32
constexpr int kRunStride = 132;          // run starts / positions of a tile (129 used)
constexpr int kMaxStages = 8;
constexpr int kTmemCols = 512;           // two accumulators of up to 256 columns

struct XferParams {
  const void* sender;
  void* receiver;
  const float* bias;
  const float* inv_r;
  const LayerSegs* segs;
  const float* inv_freq;
  const float* inv_freq_s;  // sender RoPE (rotated sender keys)
  const int32_t* spos;      // sender position of every sender token (rotated sender keys)
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
  int64_t T_s;        // aligned sender tokens (CSR column range)
  int64_t s_rows;     // sender-cache rows per (layer, role)
  const int32_t* srow;  // cache row of each aligned sender token (message spans), or null
  int64_t recv_rows;  // receiver rows per (layer, role) in receiver_kv
  int L_r, d_s, d_r, D_r;
  int l0, n_l;  // receiver layers [l0, l0 + n_l) of this launch
  int n_kb, atoms_per_seg, last_atoms, BN, n_tiles_n, groups;  // n_kb: A stages per tile
  // split: each A stage holds one map atom of K as two bf16 atoms, the
  // rounded operand and its rounding residual, multiplied by the same B atom
  // (atoms_per_stage = 1); otherwise kAtoms atoms of K per A stage
  int split, atoms_per_stage, n_batoms;  // n_batoms: B atoms (map atoms of K) per tile
  int staged;  // split one-entry rows built by build_rows_staged
  // wide tiles (operand rows built by the loader warps, which bound those
  // paths): a tile covers two 256-column blocks, one per TMEM accumulator,
  // so every built A stage feeds twice the MMAs; the epilogue drains both
  // before the next tile's MMAs start
  int wide;
  // pooling after the map: the tile rows of CTA rank k in pair tile m are the
  // aligned sender tokens of window w = 2m + k, [w S, w S + 128) (S =
  // win_info[1]); the receiver rows [win_ptr[w], win_ptr[w+1]) are pooled
  // from them in the epilogue
  int pam;
  const int32_t* win_info;  // h, S, number of windows
  const int32_t* win_ptr;
  const int32_t* pos;       // RoPE position of every receiver row
  int stages_a, stages_b, lag;  // A ring (stages), B ring (atoms), loader groups in flight
  int rope, paged, knorm, unrot, D_s;
  int stall;  // test hook: the map producer withholds its first atom (hf_debug_transfer_stalled)
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

// Tiles of a launch over receiver layers [l0, l0 + n_l): a slot is (layer,
// 256-row pair block, column block), ordered layer-major so that the slots
// in flight share their Eq. 1 sender rows and maps in L2; tile = 2 * slot + c
// covers role c of the slot.  With at least two slots per CTA pair, a pair
// takes slots first, first + step, ... and both roles of each slot in turn,
// so that its key tiles (rotated epilogue) and value tiles (copy epilogue)
// alternate; with fewer, it takes tiles first, first + step, ... (the two
// roles of a slot on different pairs).  lc = 2 * l + c indexes the maps,
// biases and receiver cache.
// Slot order needs at least two slots per CTA pair, and is kept unless tile
// order fills the last round of tiles clearly better: a pair's share is
// whole slots (two tiles) in slot order, single tiles otherwise (at 1K
// receiver tokens, 256 slots over 76 pairs leave the last round 37% full,
// 512 tiles 74%).
__device__ __forceinline__ bool slot_order(int total_tiles, int tile_step) {
  if (total_tiles < 4 * tile_step) return false;
  const int slots = total_tiles >> 1;
  const float fill_slots =
      static_cast<float>(slots) / static_cast<float>(((slots + tile_step - 1) / tile_step) * tile_step);
  const float fill_tiles = static_cast<float>(total_tiles) /
                           static_cast<float>(((total_tiles + tile_step - 1) / tile_step) * tile_step);
  return fill_slots >= fill_tiles - 0.03f;
}
__device__ __forceinline__ int tile_of(int seq, int first, int step, bool by_slot) {
  return by_slot ? 2 * (first + (seq >> 1) * step) + (seq & 1) : first + seq * step;
}
__device__ __forceinline__ void decode_tile(int tile, int tiles_per_lc, int n_tiles_n, int l0,
                                            int* lc, int* m, int* n) {
  const int c = tile & 1;
  const int slot = tile >> 1;
  const int ol = slot / tiles_per_lc;
  const int rem = slot - ol * tiles_per_lc;
  *lc = 2 * (l0 + ol) + c;
  *m = rem / n_tiles_n;
  *n = rem - *m * n_tiles_n;
}

__device__ __forceinline__ void raise_timeout(const XferParams& P, volatile int* abort_flag) {
  atomicOr(P.status, HF_CHECK_TIMEOUT);
  *abort_flag = 1;
}

// Pooling after the map: the aligned sender token of row r (0..127) of the
// window of CTA row0 in pair tile m, w = 2m + row0/128, token w S + r (the
// last token past the end; those rows are never pooled).
__device__ __forceinline__ int pam_token(const XferParams& P, int m, int row0, int r) {
  const int w = (m * kPairRows + row0) >> 7;
  const int64_t k = static_cast<int64_t>(w) * __ldg(P.win_info + 1) + r;
  return static_cast<int>(k < P.T_s ? k : P.T_s - 1);
}

// Kernel variants fix pooling after the map at compile time (kPam 0: off,
// 1: on) so that neither path carries the other's registers; kPam 2 reads
// it from the parameters (fp32 and multi-direction launches).
template <int kPam>
__device__ __forceinline__ bool pam_on(const XferParams& P) {
  return kPam == 2 ? P.pam != 0 : kPam == 1;
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

// 8 fp32 values as bf16 (round to nearest) in *hi, and in *lo the bf16
// rounding of what that rounding lost (exact in fp32): hi + lo carries each
// value to about 16 mantissa bits.
__device__ __forceinline__ void pack16_split(const float* a, uint4* hi, uint4* lo) {
  uint32_t h[4], r[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat162 b = __floats2bfloat162_rn(a[2 * i], a[2 * i + 1]);
    const float2 bf = __bfloat1622float2(b);
    const __nv_bfloat162 d = __floats2bfloat162_rn(a[2 * i] - bf.x, a[2 * i + 1] - bf.y);
    h[i] = *reinterpret_cast<const uint32_t*>(&b);
    r[i] = *reinterpret_cast<const uint32_t*>(&d);
  }
  *hi = make_uint4(h[0], h[1], h[2], h[3]);
  *lo = make_uint4(r[0], r[1], r[2], r[3]);
}

// Writes 16 bytes of fp32 results of operand row t, chunk ch, into an A atom
// (rounded once), or into the value atom and the residual atom (split).
template <typename T>
__device__ __forceinline__ void put_chunk(const float* a, uint8_t* atom, uint8_t* lo_atom, int t,
                                          int ch) {
  const int off = t * 128 + ((ch ^ (t & 7)) << 4);
  if constexpr (sizeof(T) == 2) {
    if (lo_atom) {
      uint4 hi, lo;
      pack16_split(a, &hi, &lo);
      *reinterpret_cast<uint4*>(atom + off) = hi;
      *reinterpret_cast<uint4*>(lo_atom + off) = lo;
      return;
    }
  }
  *reinterpret_cast<uint4*>(atom + off) = pack16(a, (const T*)nullptr);
}

// Receiver-cache stores are streaming stores (st.global.cs, evict first):
// the output is written once and should not push map tiles and sender rows,
// which other tiles read again, out of L2.
__device__ __forceinline__ void store4(__nv_bfloat16* p, const float4& v) {
  const __nv_bfloat162 x = __floats2bfloat162_rn(v.x, v.y), y = __floats2bfloat162_rn(v.z, v.w);
  __stcs(reinterpret_cast<uint2*>(p),
         make_uint2(*reinterpret_cast<const uint32_t*>(&x), *reinterpret_cast<const uint32_t*>(&y)));
}
__device__ __forceinline__ void store4(float* p, const float4& v) {
  __stcs(reinterpret_cast<float4*>(p), v);
}

// Rotates the pairs (x[k], y[k]) by the angles with cosines c[k], sines s[k].
__device__ __forceinline__ void rotate4(float4& x, float4& y, const float* c, const float* s) {
  const float x0 = x.x * c[0] - y.x * s[0], y0 = y.x * c[0] + x.x * s[0];
  const float x1 = x.y * c[1] - y.y * s[1], y1 = y.y * c[1] + x.y * s[1];
  const float x2 = x.z * c[2] - y.z * s[2], y2 = y.z * c[2] + x.z * s[2];
  const float x3 = x.w * c[3] - y.w * s[3], y3 = y.w * c[3] + x.w * s[3];
  x = make_float4(x0, x1, x2, x3);
  y = make_float4(y0, y1, y2, y3);
}

// The epilogue's position walk for one lane: it owns four rotation pairs
// (columns q+4*qq .. +3 of the first half of each head and their partners
// half further on) of up to two heads, for the consecutive receiver rows
// [jb, je) of one slice.  Shared memory is slow to answer while the tensor
// core streams its operands, so the lane keeps the staged (unrotated) values
// of its current distinct row in registers and reads the next row's only
// when the walk enters its run; positions inside a run, and across runs of
// one request, are consecutive, so the angles advance by one position per
// row (re-anchored exactly every 16 rows and wherever the position jumps).
template <typename T>
__device__ __forceinline__ void walk_rows(int jb, int je, int u, const int32_t* srun,
                                          const int32_t* supos, const float* stg, int qq,
                                          bool two_heads, bool do_rope, const float* f,
                                          const float* C1, const float* S1, const XferParams& P,
                                          T* out_lc, int ocol, int q, int half) {
  if (jb >= je) return;
  float4 a0, b0, a1 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = a1;
  int uend = 0, pb = 0;  // end of the current run; position of row j is pb + j
  int expect = INT_MIN;  // position for which cs/sn are valid
  float cs[4] = {1.f, 1.f, 1.f, 1.f}, sn[4] = {0.f, 0.f, 0.f, 0.f};
  --u;
  int dnext = P.paged ? __ldg(P.dst_row + jb) : jb;  // destination of row j, read a row ahead
  for (int j = jb; j < je; ++j) {
    const int drow = dnext;
    if (P.paged) {
      if (j + 1 < je) dnext = __ldg(P.dst_row + j + 1);
    } else {
      dnext = j + 1;
    }
    if (j >= uend) {  // first row, or the first row of a later run
      do {
        ++u;
      } while (srun[u + 1] <= j);
      uend = srun[u + 1];
      pb = supos[u] - srun[u];
      const float* urow = stg + u * 64;
      const int sw = u & 7;
      a0 = *reinterpret_cast<const float4*>(urow + ((qq ^ sw) << 2));
      b0 = *reinterpret_cast<const float4*>(urow + (((4 + qq) ^ sw) << 2));
      if (two_heads) {
        a1 = *reinterpret_cast<const float4*>(urow + 32 + ((qq ^ sw) << 2));
        b1 = *reinterpret_cast<const float4*>(urow + 32 + (((4 + qq) ^ sw) << 2));
      }
    }
    float4 x0 = a0, y0 = b0, x1 = a1, y1 = b1;
    if (do_rope) {
      const int p = pb + j;
      if (p != expect || ((j - jb) & 15) == 0) {
#pragma unroll
        for (int k = 0; k < 4; ++k) rope_sincos(p, f[k], &sn[k], &cs[k]);
      } else {  // advance every angle by one position
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float t = cs[k] * C1[k] - sn[k] * S1[k];
          sn[k] = sn[k] * C1[k] + cs[k] * S1[k];
          cs[k] = t;
        }
      }
      expect = p + 1;
      rotate4(x0, y0, cs, sn);
      if (two_heads) rotate4(x1, y1, cs, sn);
    }
    if (drow >= 0) {
      T* o = out_lc + static_cast<int64_t>(drow) * P.d_r + ocol + q + 4 * qq;
      store4(o, x0);
      store4(o + half, y0);
      if (two_heads) {
        store4(o + 2 * half, x1);
        store4(o + 3 * half, y1);
      }
    }
  }
}

// Epilogue of a tile whose rows need no rotation (values; keys when RoPE and
// key norm are off): every receiver row of a run is the same row of
// y = acc / r + b, so each distinct row is converted once into the staging
// buffer and copied out whole.  Columns go in passes of 256 bytes per row
// (128 rows x 256 bytes of staging); in a pass, warp (g, sp) converts TMEM
// lane quarter sp, half g of the pass's columns, then warp e copies the runs
// of distinct rows e, e + 8, ...: 16 lanes x 16 bytes per receiver row, the
// two half-warps taking alternate receiver rows of the run.
template <typename T>
__device__ __forceinline__ void copy_epilogue(const XferParams& P, uint32_t ta,
                                              const float* bias_tile, float inv_r, int nrows,
                                              const int32_t* srun, uint8_t* stg, int g, int row,
                                              int e, int lane, T* out_lc, int ocol0) {
  constexpr int kPassCols = 256 / sizeof(T);  // 128 bf16 or 64 fp32 columns
  constexpr int kHalfCols = kPassCols / 2;
  constexpr int kPerChunk = 16 / sizeof(T);
  const int hw = lane >> 4, cidx = lane & 15;
  for (int pc0 = 0; pc0 < P.BN; pc0 += kPassCols) {
    uint8_t* srow = stg + row * 256;
#pragma unroll
    for (int k = 0; k < kHalfCols; k += 16) {
      if (e >= 8) break;  // the two extra warps only copy
      const int col = pc0 + g * kHalfCols + k;
      uint32_t v[16];
      tmem_load_16(ta + static_cast<uint32_t>(col), v);
      float y[16];
#pragma unroll
      for (int i = 0; i < 16; i += 4) {
        const float4 bb = __ldg(reinterpret_cast<const float4*>(bias_tile + col + i));
        y[i] = fmaf(__uint_as_float(v[i]), inv_r, bb.x);
        y[i + 1] = fmaf(__uint_as_float(v[i + 1]), inv_r, bb.y);
        y[i + 2] = fmaf(__uint_as_float(v[i + 2]), inv_r, bb.z);
        y[i + 3] = fmaf(__uint_as_float(v[i + 3]), inv_r, bb.w);
      }
#pragma unroll
      for (int h = 0; h < 16 / kPerChunk; ++h) {
        const int chunk = (col - pc0) / kPerChunk + h;  // 0..15 within the 256-byte row
        *reinterpret_cast<uint4*>(srow + ((chunk ^ (row & 7)) << 4)) =
            pack16(y + h * kPerChunk, (const T*)nullptr);
      }
    }
    named_barrier_sync(1, kEpiThreads);
    // the next distinct row's staged chunk and run bounds are read while this
    // row's receiver rows are stored (shared-memory reads are slow to answer
    // while the tensor core streams its operands)
    int u = e;
    uint4 val = make_uint4(0u, 0u, 0u, 0u);
    int js = 0, je = 0;
    if (u < nrows) {
      val = *reinterpret_cast<const uint4*>(stg + u * 256 + ((cidx ^ (u & 7)) << 4));
      js = srun[u];
      je = srun[u + 1];
    }
    while (u < nrows) {
      const int un = u + kEpiWarps;
      uint4 nval = val;
      int njs = 0, nje = 0;
      if (un < nrows) {
        nval = *reinterpret_cast<const uint4*>(stg + un * 256 + ((cidx ^ (un & 7)) << 4));
        njs = srun[un];
        nje = srun[un + 1];
      }
      for (int j = js + hw; j < je; j += 2) {
        const int drow = P.paged ? __ldg(P.dst_row + j) : j;
        if (drow >= 0)
          __stcs(reinterpret_cast<uint4*>(out_lc + static_cast<int64_t>(drow) * P.d_r + ocol0 +
                                          pc0 + cidx * kPerChunk),
                 val);
      }
      u = un;
      val = nval;
      js = njs;
      je = nje;
    }
    named_barrier_sync(1, kEpiThreads);
  }
}

// Pooling after the map, one lane's receiver rows [jb, je) of a window
// whose first aligned sender token is `base`: the staged rows hold
// z_i / r (i = token - base) for four rotation pairs of up to two heads, and
// y_j = sum_e w_e z_{col_e} / r + b, rotated at the receiver position of j
// for keys.  Positions of consecutive rows of a request are consecutive, so
// the angles advance by one position per row (re-anchored every 16 rows and
// wherever the position jumps).
template <typename T>
__device__ __forceinline__ void pam_walk(int jb, int je, int base, const float* stg, int qq,
                                         bool two_heads, bool do_rope, const float* f,
                                         const float* C1, const float* S1, const float4* bias4,
                                         const XferParams& P, T* out_lc, int ocol, int q,
                                         int half) {
  if (jb >= je) return;
  int expect = INT_MIN;  // position for which cs/sn are valid
  float cs[4] = {1.f, 1.f, 1.f, 1.f}, sn[4] = {0.f, 0.f, 0.f, 0.f};
  int e1 = __ldg(P.row_ptr + jb);
  for (int j = jb; j < je; ++j) {
    const int e0 = e1;
    e1 = __ldg(P.row_ptr + j + 1);
    float4 x0 = make_float4(0.f, 0.f, 0.f, 0.f), y0 = x0, x1 = x0, y1 = x0;
    for (int e = e0; e < e1; ++e) {
      const int loc = __ldg(P.col + e) - base;
      if (loc < 0 || loc >= kBM) continue;  // flagged at plan creation
      const float wt = __ldg(P.w + e);
      const float* urow = stg + loc * 64;
      const int sw = loc & 7;
      const float4 a = *reinterpret_cast<const float4*>(urow + ((qq ^ sw) << 2));
      const float4 b = *reinterpret_cast<const float4*>(urow + (((4 + qq) ^ sw) << 2));
      x0 = make_float4(fmaf(wt, a.x, x0.x), fmaf(wt, a.y, x0.y), fmaf(wt, a.z, x0.z),
                       fmaf(wt, a.w, x0.w));
      y0 = make_float4(fmaf(wt, b.x, y0.x), fmaf(wt, b.y, y0.y), fmaf(wt, b.z, y0.z),
                       fmaf(wt, b.w, y0.w));
      if (two_heads) {
        const float4 a1 = *reinterpret_cast<const float4*>(urow + 32 + ((qq ^ sw) << 2));
        const float4 b1 = *reinterpret_cast<const float4*>(urow + 32 + (((4 + qq) ^ sw) << 2));
        x1 = make_float4(fmaf(wt, a1.x, x1.x), fmaf(wt, a1.y, x1.y), fmaf(wt, a1.z, x1.z),
                         fmaf(wt, a1.w, x1.w));
        y1 = make_float4(fmaf(wt, b1.x, y1.x), fmaf(wt, b1.y, y1.y), fmaf(wt, b1.z, y1.z),
                         fmaf(wt, b1.w, y1.w));
      }
    }
    x0 = make_float4(x0.x + bias4[0].x, x0.y + bias4[0].y, x0.z + bias4[0].z, x0.w + bias4[0].w);
    y0 = make_float4(y0.x + bias4[1].x, y0.y + bias4[1].y, y0.z + bias4[1].z, y0.w + bias4[1].w);
    x1 = make_float4(x1.x + bias4[2].x, x1.y + bias4[2].y, x1.z + bias4[2].z, x1.w + bias4[2].w);
    y1 = make_float4(y1.x + bias4[3].x, y1.y + bias4[3].y, y1.z + bias4[3].z, y1.w + bias4[3].w);
    if (do_rope) {
      const int p = __ldg(P.pos + j);
      if (p != expect || ((j - jb) & 15) == 0) {
#pragma unroll
        for (int k = 0; k < 4; ++k) rope_sincos(p, f[k], &sn[k], &cs[k]);
      } else {  // advance every angle by one position
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float t = cs[k] * C1[k] - sn[k] * S1[k];
          sn[k] = sn[k] * C1[k] + cs[k] * S1[k];
          cs[k] = t;
        }
      }
      expect = p + 1;
      rotate4(x0, y0, cs, sn);
      if (two_heads) rotate4(x1, y1, cs, sn);
    }
    const int drow = P.paged ? __ldg(P.dst_row + j) : j;
    if (drow >= 0) {
      T* o = out_lc + static_cast<int64_t>(drow) * P.d_r + ocol + q + 4 * qq;
      store4(o, x0);
      store4(o + half, y0);
      if (two_heads) {
        store4(o + 2 * half, x1);
        store4(o + 3 * half, y1);
      }
    }
  }
}

// Epilogue of a tile with pooling after the map (both roles): TMEM row i of
// this CTA is the product of aligned sender token base + i; per 16 rotation
// pairs of a head pair, warp (g, sp), e < 8, stages z / r of TMEM lane
// quarter sp, head 2*hp+g, and the ten warps pool, rotate (keys) and store
// the window's receiver rows [jb, je), split into slices as in the rotated
// epilogue.
template <typename T>
__device__ __forceinline__ void pam_epilogue(const XferParams& P, uint32_t ta,
                                             const float* bias_tile, float inv_r, int base,
                                             int jb, int je, float* sStg, int e, int g, int row,
                                             int lane, bool do_rope, T* out_lc, int ocol0) {
  const int D = P.D_r, half = P.D_r / 2;
  const int n_heads = P.BN / D;
  const bool two_heads = n_heads >= 2;
  const int n_pairs = two_heads ? n_heads / 2 : 1;
  const bool stages_head = e < 8 && (g == 0 || two_heads);
  const int ps = lane >> 2, qq = lane & 3;
  const int per = (je - jb + kEpiWarps - 1) / kEpiWarps;
  const int wjb = min(je, jb + e * per), wje = min(je, wjb + per);
  const int per_slot = (wje - wjb + 7) >> 3;
  const int ljb = min(wje, wjb + ps * per_slot), lje = min(wje, ljb + per_slot);
  for (int hp = 0; hp < n_pairs; ++hp) {
    const int tcol = (2 * hp + g) * D;
    for (int q = 0; q < half; q += 16) {
      float f[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) f[k] = do_rope ? __ldg(P.inv_freq + q + 4 * qq + k) : 0.f;
      if (stages_head) {
        uint32_t v[32];
        tmem_load_2x16(ta + tcol + q, ta + tcol + half + q, v);
        float* srow = sStg + row * 64 + g * 32;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          *reinterpret_cast<float4*>(srow + ((k ^ (row & 7)) << 2)) = make_float4(
              __uint_as_float(v[4 * k]) * inv_r, __uint_as_float(v[4 * k + 1]) * inv_r,
              __uint_as_float(v[4 * k + 2]) * inv_r, __uint_as_float(v[4 * k + 3]) * inv_r);
      }
      named_barrier_sync(1, kEpiThreads);
      const float* bb = bias_tile + 2 * hp * D + q + 4 * qq;
      float4 bias4[4];
      bias4[0] = __ldg(reinterpret_cast<const float4*>(bb));
      bias4[1] = __ldg(reinterpret_cast<const float4*>(bb + half));
      bias4[2] = two_heads ? __ldg(reinterpret_cast<const float4*>(bb + D)) : make_float4(0.f, 0.f, 0.f, 0.f);
      bias4[3] = two_heads ? __ldg(reinterpret_cast<const float4*>(bb + D + half)) : make_float4(0.f, 0.f, 0.f, 0.f);
      float C1[4], S1[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        C1[k] = 1.f;
        S1[k] = 0.f;
        if (do_rope) rope_sincos(1, f[k], &S1[k], &C1[k]);  // one step = one row
      }
      pam_walk<T>(ljb, lje, base, sStg, qq, two_heads, do_rope, f, C1, S1, bias4, P, out_lc,
                  ocol0 + 2 * hp * D, q, half);
      named_barrier_sync(1, kEpiThreads);
    }
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

// One 128-byte atom of operand row t for the builder path: features
// [kin*kBK, (kin+1)*kBK) of segment `seg`, i.e. sum over the segment's
// sender layers (weight om) and the row's CSR entries (weight w) of the
// sender rows, accumulated in fp32 and written into the swizzled layout,
// rounded once, or as value + residual atoms when lo_atom is given.  With
// tok >= 0 the row is that one aligned sender token, weight 1 (pooling
// after the map), and the CSR range is not read.
template <typename T>
__device__ __forceinline__ void build_atom(const XferParams& P, const LayerSegs& segs, int seg,
                                           int kin, int c, int e0, int e1, int tok,
                                           uint8_t* atom, uint8_t* lo_atom, int t) {
  constexpr int kBK = Elem<T>::kBK;
  constexpr int kPerChunk = 16 / sizeof(T);
  const T* sender = reinterpret_cast<const T*>(P.sender);
  float acc[kBK];
#pragma unroll
  for (int i = 0; i < kBK; ++i) acc[i] = 0.f;
  for (int ti = 0; ti < segs.n_terms[seg]; ++ti) {
    const int tl = segs.layer[seg][ti];
    const float om = segs.w[seg][ti];
    const T* base = sender + (static_cast<int64_t>(tl * 2 + c) * P.s_rows) * P.d_s + kin * kBK;
    const int n_e = tok >= 0 ? 1 : e1 - e0;
    for (int ie = 0; ie < n_e; ++ie) {
      const int k = tok >= 0 ? tok : P.col[e0 + ie];
      if (k < 0 || k >= P.T_s) continue;  // flagged at plan creation
      const float wt = tok >= 0 ? om : om * P.w[e0 + ie];
      const int64_t kr = P.srow ? __ldg(P.srow + k) : k;
      const uint4* src = reinterpret_cast<const uint4*>(base + kr * P.d_s);
      uint4 x[8];
#pragma unroll
      for (int k2 = 0; k2 < 8; ++k2) x[k2] = __ldg(src + k2);
#pragma unroll
      for (int k2 = 0; k2 < 8; ++k2) accum16(x[k2], wt, acc + k2 * kPerChunk, (const T*)nullptr);
    }
  }
#pragma unroll
  for (int k2 = 0; k2 < 8; ++k2) put_chunk<T>(acc + k2 * kPerChunk, atom, lo_atom, t, k2);
}

// One atom of operand row t when the sender keys carry RoPE (split operands):
// each sender row is rotated back at its own sender position before the CSR
// and layer weights are applied.  Feature i of a head pairs with i + D_s/2
// (first half: x cos + y sin) or i - D_s/2 (second half: x cos - y sin), the
// angle pos * inv_freq_s_{i mod D_s/2}; a 16-byte chunk never straddles the
// halves (D_s/2 is a multiple of the chunk).  The angle uses the same
// exact-product reduction as the epilogue.
template <typename T>
__device__ __forceinline__ void build_atom_unrotated(const XferParams& P, const LayerSegs& segs,
                                                     int seg, int kin, int c, int e0, int e1,
                                                     uint8_t* atom, uint8_t* lo_atom, int t) {
  constexpr int kBK = Elem<T>::kBK;
  constexpr int kPerChunk = 16 / sizeof(T);
  const T* sender = reinterpret_cast<const T*>(P.sender);
  const int hs = P.D_s / 2;
#pragma unroll 1
  for (int ch = 0; ch < kBK / kPerChunk; ++ch) {
    const int el = kin * kBK + ch * kPerChunk;  // feature within the segment
    const int i = el % P.D_s;
    const bool first = i < hs;
    const int partner = first ? el + hs : el - hs;
    const int fi = first ? i : i - hs;
    float f[kPerChunk], acc[kPerChunk];
#pragma unroll
    for (int q = 0; q < kPerChunk; ++q) {
      f[q] = __ldg(P.inv_freq_s + fi + q);
      acc[q] = 0.f;
    }
    for (int ti = 0; ti < segs.n_terms[seg]; ++ti) {
      const int tl = segs.layer[seg][ti];
      const float om = segs.w[seg][ti];
      const T* base = sender + (static_cast<int64_t>(tl * 2 + c) * P.s_rows) * P.d_s;
      for (int e = e0; e < e1; ++e) {
        const int k = P.col[e];
        if (k < 0 || k >= P.T_s) continue;  // flagged at plan creation
        const float wt = om * P.w[e];
        const int64_t kr = P.srow ? __ldg(P.srow + k) : k;
        const T* row = base + kr * P.d_s;
        float x[kPerChunk], y[kPerChunk];
#pragma unroll
        for (int q = 0; q < kPerChunk; ++q) x[q] = y[q] = 0.f;
        accum16(__ldg(reinterpret_cast<const uint4*>(row + el)), 1.f, x, (const T*)nullptr);
        accum16(__ldg(reinterpret_cast<const uint4*>(row + partner)), 1.f, y, (const T*)nullptr);
        const int p = __ldg(P.spos + k);
#pragma unroll
        for (int q = 0; q < kPerChunk; ++q) {
          float sn, cs;
          rope_sincos(p, f[q], &sn, &cs);
          acc[q] = fmaf(wt, first ? fmaf(x[q], cs, y[q] * sn) : fmaf(x[q], cs, -y[q] * sn), acc[q]);
        }
      }
    }
    put_chunk<T>(acc, atom, lo_atom, t, ch);
  }
}

// One stage (kAtoms atoms = whole heads of one segment) of operand row t
// when the sender keys carry RoPE: every sender row is rotated back at its
// own sender position before the CSR and layer weights are applied, pair
// (i, i + D_s/2) of each head by the angle -pos * inv_freq_s_i:
// (x, y) -> (x cos + y sin, y cos - x sin).  Lanes take 16-byte chunks of
// pairs; the angle uses the same exact-product reduction as the epilogue.
template <typename T>
__device__ __forceinline__ void build_stage_unrotated(const XferParams& P, const LayerSegs& segs,
                                                      int seg, int kin, int c, int e0, int e1,
                                                      uint8_t* stage, int t) {
  constexpr int kBK = Elem<T>::kBK;
  constexpr int kPerChunk = 16 / sizeof(T);
  const T* sender = reinterpret_cast<const T*>(P.sender);
  const int hs = P.D_s / 2;
  const int elem0 = kin * kBK;  // the stage's first feature within the segment
  for (int pc = 0; pc < kBK / kPerChunk; ++pc) {
    const int pi = pc * kPerChunk;                 // first pair of the chunk, within the stage
    const int hh = pi / hs, i0 = pi - hh * hs;     // head within the stage, its frequency index
    const int ex = hh * P.D_s + i0, ey = ex + hs;  // stage features of the pair halves
    float f[kPerChunk], ax[kPerChunk], ay[kPerChunk];
#pragma unroll
    for (int i = 0; i < kPerChunk; ++i) {
      f[i] = __ldg(P.inv_freq_s + i0 + i);
      ax[i] = 0.f;
      ay[i] = 0.f;
    }
    for (int ti = 0; ti < segs.n_terms[seg]; ++ti) {
      const int tl = segs.layer[seg][ti];
      const float om = segs.w[seg][ti];
      const T* base = sender + (static_cast<int64_t>(tl * 2 + c) * P.s_rows) * P.d_s + elem0;
      for (int e = e0; e < e1; ++e) {
        const int k = P.col[e];
        if (k < 0 || k >= P.T_s) continue;  // flagged at plan creation
        const float wt = om * P.w[e];
        const int64_t kr = P.srow ? __ldg(P.srow + k) : k;
        const T* row = base + kr * P.d_s;
        float x[kPerChunk], y[kPerChunk];
#pragma unroll
        for (int i = 0; i < kPerChunk; ++i) x[i] = y[i] = 0.f;
        accum16(__ldg(reinterpret_cast<const uint4*>(row + ex)), 1.f, x, (const T*)nullptr);
        accum16(__ldg(reinterpret_cast<const uint4*>(row + ey)), 1.f, y, (const T*)nullptr);
        const int p = __ldg(P.spos + k);
#pragma unroll
        for (int i = 0; i < kPerChunk; ++i) {
          float sn, cs;
          rope_sincos(p, f[i], &sn, &cs);
          ax[i] = fmaf(wt, fmaf(x[i], cs, y[i] * sn), ax[i]);
          ay[i] = fmaf(wt, fmaf(y[i], cs, -x[i] * sn), ay[i]);
        }
      }
    }
    uint8_t* row_x = stage + (ex / kBK) * kAtomABytes + t * 128;
    uint8_t* row_y = stage + (ey / kBK) * kAtomABytes + t * 128;
    const int cx = (ex % kBK) / kPerChunk, cy = (ey % kBK) / kPerChunk;
    *reinterpret_cast<uint4*>(row_x + ((cx ^ (t & 7)) << 4)) = pack16(ax, (const T*)nullptr);
    *reinterpret_cast<uint4*>(row_y + ((cy ^ (t & 7)) << 4)) = pack16(ay, (const T*)nullptr);
  }
}

// Tiles of several transfer directions in one launch: direction d owns the
// launch's tiles [base[d], base[d + 1]) (2 x its slots, so a slot's two
// roles stay together), m_tiles[d] row blocks of U[d] distinct rows (with
// pooling after the map, 128 rows per window: one window per CTA of a pair
// tile).
template <int kDirs>
struct DirTable {
  int base[kDirs + 1];
  int m_tiles[kDirs];
  int U[kDirs];
};

template <int kDirs, int kPam>
__device__ __forceinline__ int build_dirs(const XferParams* Ps, int n_dir, DirTable<kDirs>* dt) {
  int total = 0;
  for (int d = 0; d < (kDirs == 1 ? 1 : n_dir); ++d) {
    const int U = pam_on<kPam>(Ps[d]) ? 128 * __ldg(Ps[d].win_info + 2) : *Ps[d].n_distinct;
    const int mt = (U + kPairRows - 1) / kPairRows;
    dt->U[d] = U;
    dt->m_tiles[d] = mt;
    dt->base[d] = total;
    total += 2 * Ps[d].n_l * mt * Ps[d].n_tiles_n;
  }
  dt->base[kDirs == 1 ? 1 : n_dir] = total;
  return total;
}

template <int kDirs>
__device__ __forceinline__ int dir_of(const DirTable<kDirs>& dt, int n_dir, int tile) {
  if (kDirs == 1) return 0;
  int d = 0;
  while (d + 1 < n_dir && tile >= dt.base[d + 1]) ++d;
  return d;
}

// Arrival on the leader CTA's copy of a pair barrier (`bar` is the local
// offset): a local arrive in the leader, a relaxed remote arrive in the
// follower.  What is announced is complete and visible before the call.
__device__ __forceinline__ void arrive_leader(uint32_t bar, int row0) {
  if (row0 == 0)
    mbar_arrive_relaxed(bar);
  else
    mbar_arrive_cluster(mapa_shared(bar, 0));
}

// A tile rows for one-entry alignment rows: this CTA's 128 sender rows of a
// tile are copied with cp.async, eight lanes per 128-byte row (lane -> row
// 32*slab + 4*i + lane/8, 16-byte chunk lane%8), into the 128-byte swizzled
// layout.  A thread keeps LAG groups in flight: after committing k-block i
// it waits for k-block i-LAG and fences it to the async proxy; then one lane
// per warp arrives on that stage's barrier in the leader CTA of the pair.
template <typename T, int LAG, int kDirs, int kPam>
__device__ __forceinline__ void gather_rows(const XferParams* Ps, const DirTable<kDirs>& dt,
                                            int n_dir, uint8_t* sA, uint64_t* full_a,
                                            uint64_t* empty_a, volatile int* sAbort, int t,
                                            int lane, int row0, int total_tiles, int first_tile,
                                            int tile_step) {
  constexpr int kBK = Elem<T>::kBK;
  const bool by_slot = slot_order(total_tiles, tile_step);
  constexpr int kPerChunk = 16 / sizeof(T);
  const int stages = Ps[0].stages_a;
  const int slab = t >> 5, rsub = lane >> 3, ch = lane & 7;
  int stage = 0;
  uint32_t phase = 0;
  int pending = 0;  // committed groups whose stage arrival is still owed
  bool ok = true;
  for (int seq = 0, tile = tile_of(0, first_tile, tile_step, by_slot); tile < total_tiles && ok;
       tile = tile_of(++seq, first_tile, tile_step, by_slot)) {
    const int dd = dir_of(dt, n_dir, tile);
    const XferParams& P = Ps[dd];
    const int U = dt.U[dd];
    const T* sender = reinterpret_cast<const T*>(P.sender);
    int lc, m, n;
    decode_tile(tile - dt.base[dd], dt.m_tiles[dd] * P.n_tiles_n, P.n_tiles_n, P.l0, &lc, &m, &n);
    const int l = lc >> 1, c = lc & 1;
    // element offset of segment s2's sender layer/role block; the current
    // segment's is in sbase and the next one's is loaded a segment ahead
    const LayerSegs* lsegs = P.segs + l;
    const int n_seg = __ldg(&lsegs->n_seg);
    auto seg_base = [&](int s2) -> int64_t {
      return (static_cast<int64_t>(__ldg(&lsegs->layer[s2][0]) * 2 + c) * P.s_rows) * P.d_s;
    };
    int64_t sbase = seg_base(0);
    int64_t snext = n_seg > 1 ? seg_base(1) : 0;
    int64_t roff[8];
    uint32_t doff[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = slab * 32 + 4 * i + rsub;
      int64_t kr;  // sender-cache row
      if (pam_on<kPam>(P)) {
        const int k = pam_token(P, m, row0, r);
        kr = P.srow ? __ldg(P.srow + k) : k;
      } else {
        kr = P.ucol[min(m * kPairRows + row0 + r, U - 1)];
      }
      roff[i] = kr * P.d_s + ch * kPerChunk;
      doff[i] = static_cast<uint32_t>(r * 128 + ((ch ^ (r & 7)) << 4));
    }
    int seg = 0, kin = 0;  // segment of the next atom, and the atom within it
    for (int kb = 0; kb < P.n_kb; ++kb) {
      if (!mbar_wait(smem_addr(&empty_a[stage]), phase ^ 1)) {
        raise_timeout(P, sAbort);
        ok = false;
        break;
      }
      const uint32_t sa = smem_addr(sA + stage * kStageABytes);
      const int na = kb == P.n_kb - 1 ? P.last_atoms : kAtoms;
#pragma unroll
      for (int a = 0; a < kAtoms; ++a) {
        if (a < na) {
          const T* base = sender + sbase + kin * kBK;
#pragma unroll
          for (int i = 0; i < 8; ++i) cp_async_16(sa + a * kAtomABytes + doff[i], base + roff[i]);
          if (++kin == P.atoms_per_seg) {
            kin = 0;
            ++seg;
            sbase = snext;
            if (seg + 1 < n_seg) snext = seg_base(seg + 1);
          }
        }
      }
      cp_async_commit();
      if (pending == LAG) {
        cp_async_wait<LAG>();
        fence_proxy_async_smem();
        __syncwarp();  // the warp's copies of that stage have landed
        if (lane == 0) arrive_leader(smem_addr(&full_a[(stage + stages - LAG) % stages]), row0);
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
  __syncwarp();
  if (lane == 0)
    for (int k = pending; k >= 1; --k)
      arrive_leader(smem_addr(&full_a[(stage + stages - k) % stages]), row0);
}

// Computed A rows in split mode without rotated keys (pooled rows, blended
// or weighted layers), staged: a stage is one map atom of K.  The loader
// copies the first two raw (term, entry) sender atoms of every row into the
// stage's two atom slots with cp.async, eight lanes per 128-byte row as in
// gather_rows, and keeps LAG stages in flight; once a stage's copies have
// landed, thread t of the warp finishes row 32 slab + t (finish_staged_row):
// it combines the two staged atoms and any further (term, entry) pairs
// (loaded directly) in fp32 with their weights, and overwrites the slots
// with the bf16 value and its rounding residual.  The first two pairs of a
// row are (term 0, entry 0) and (term 1, entry 0) for two-term segments,
// (term 0, entries 0 and 1) otherwise, so blended one-entry rows need no
// direct load.
struct StagedRow {
  int e0, e1;  // the finished row's CSR entries
  int tok;     // >= 0: the row is this aligned sender token, weight 1 (pooling after the map)
  int frow;    // its index among the CTA's 128 rows
};

template <typename T>
__device__ __forceinline__ void finish_staged_row(const XferParams& P, const LayerSegs* lsegs,
                                                  int c, const StagedRow& r, int kb,
                                                  uint8_t* slot0) {
  constexpr int kBK = Elem<T>::kBK;
  constexpr int kPerChunk = 16 / sizeof(T);
  const T* sender = reinterpret_cast<const T*>(P.sender);
  uint8_t* slot1 = slot0 + kAtomABytes;
  const int seg = kb / P.atoms_per_seg, kin = kb - seg * P.atoms_per_seg;
  const int n_t = __ldg(&lsegs->n_terms[seg]);
  const int la0 = __ldg(&lsegs->layer[seg][0]);
  const int la1 = n_t > 1 ? __ldg(&lsegs->layer[seg][1]) : la0;
  const float om0 = __ldg(&lsegs->w[seg][0]);
  const float om1 = n_t > 1 ? __ldg(&lsegs->w[seg][1]) : 0.f;
  const int64_t lrows = P.s_rows * P.d_s;
  const int frow = r.frow, sw = frow & 7;
  const bool one = r.tok >= 0;
  const int k0 = one ? r.tok : (r.e1 > r.e0 ? P.col[r.e0] : -1);
  const bool v0 = k0 >= 0 && k0 < P.T_s;
  int k1 = -1;
  if (!one && n_t == 1 && r.e1 > r.e0 + 1) k1 = P.col[r.e0 + 1];
  const bool v1 = n_t > 1 ? v0 : (k1 >= 0 && k1 < P.T_s);
  const float e_w0 = one ? 1.f : (v0 ? P.w[r.e0] : 0.f);
  const float w0 = v0 ? om0 * e_w0 : 0.f;
  const float w1 = !v1 ? 0.f : (n_t > 1 ? om1 * e_w0 : om0 * P.w[r.e0 + 1]);
  // two halves of four 16-byte chunks (fewer live registers)
#pragma unroll 1
  for (int h = 0; h < 2; ++h) {
    float acc[kBK / 2];
#pragma unroll
    for (int i = 0; i < kBK / 2; ++i) acc[i] = 0.f;
#pragma unroll
    for (int k2 = 0; k2 < 4; ++k2) {
      const int off = frow * 128 + (((4 * h + k2) ^ sw) << 4);
      if (v0)
        accum16(*reinterpret_cast<const uint4*>(slot0 + off), w0, acc + k2 * kPerChunk,
                (const T*)nullptr);
      if (v1)
        accum16(*reinterpret_cast<const uint4*>(slot1 + off), w1, acc + k2 * kPerChunk,
                (const T*)nullptr);
    }
    // the remaining (term, entry) pairs, loaded directly
    const int e_first = n_t > 1 ? r.e0 + 1 : r.e0 + 2;
    const int e_end = one ? e_first : r.e1;
    for (int e = e_first; e < e_end; ++e) {
      const int k = P.col[e];
      if (k < 0 || k >= P.T_s) continue;  // flagged at plan creation
      const int64_t kr = P.srow ? __ldg(P.srow + k) : k;
      for (int ti = 0; ti < n_t; ++ti) {
        const int la = ti == 0 ? la0 : la1;
        const float wt = (ti == 0 ? om0 : om1) * P.w[e];
        const uint4* src = reinterpret_cast<const uint4*>(
                               sender + static_cast<int64_t>(la * 2 + c) * lrows + kr * P.d_s +
                               kin * kBK) + 4 * h;
        uint4 x[4];
#pragma unroll
        for (int k2 = 0; k2 < 4; ++k2) x[k2] = __ldg(src + k2);
#pragma unroll
        for (int k2 = 0; k2 < 4; ++k2) accum16(x[k2], wt, acc + k2 * kPerChunk, (const T*)nullptr);
      }
    }
#pragma unroll
    for (int k2 = 0; k2 < 4; ++k2)
      put_chunk<T>(acc + k2 * kPerChunk, slot0, slot1, frow, 4 * h + k2);
  }
}

template <typename T, int LAG, int kDirs, int kPam>
__device__ __forceinline__ void build_rows_staged(const XferParams* Ps, const DirTable<kDirs>& dt,
                                                  int n_dir, uint8_t* sA, uint64_t* full_a,
                                                  uint64_t* empty_a, volatile int* sAbort, int t,
                                                  int lane, int row0, int total_tiles,
                                                  int first_tile, int tile_step) {
  constexpr int kBK = Elem<T>::kBK;
  constexpr int kPerChunk = 16 / sizeof(T);
  const bool by_slot = slot_order(total_tiles, tile_step);
  const int stages = Ps[0].stages_a;
  const int slab = t >> 5, rsub = lane >> 3, ch = lane & 7;
  int stage = 0;
  uint32_t phase = 0;
  bool ok = true;
  for (int seq = 0, tile = tile_of(0, first_tile, tile_step, by_slot); tile < total_tiles && ok;
       tile = tile_of(++seq, first_tile, tile_step, by_slot)) {
    const int dd = dir_of(dt, n_dir, tile);
    const XferParams& P = Ps[dd];
    const int U = dt.U[dd];
    const T* sender = reinterpret_cast<const T*>(P.sender);
    int lc, m, n;
    decode_tile(tile - dt.base[dd], dt.m_tiles[dd] * P.n_tiles_n, P.n_tiles_n, P.l0, &lc, &m, &n);
    const int l = lc >> 1, c = lc & 1;
    const LayerSegs* lsegs = P.segs + l;
    const int64_t lrows = P.s_rows * P.d_s;
    // cache rows of the first two entries of the eight rows this lane copies
    int32_t kr0[8], kr1[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      int k0, k1 = -1;
      if (pam_on<kPam>(P)) {
        k0 = pam_token(P, m, row0, slab * 32 + 4 * i + rsub);
      } else {
        const int u = min(m * kPairRows + row0 + slab * 32 + 4 * i + rsub, U - 1);
        const int j0 = P.run_ptr[u];
        const int e0 = P.row_ptr[j0], e1 = P.row_ptr[j0 + 1];
        k0 = e1 > e0 ? P.col[e0] : -1;
        k1 = e1 > e0 + 1 ? P.col[e0 + 1] : -1;
      }
      if (k0 >= P.T_s) k0 = -1;  // flagged at plan creation
      if (k1 >= P.T_s) k1 = -1;
      kr0[i] = k0 < 0 ? -1 : (P.srow ? __ldg(P.srow + k0) : k0);
      kr1[i] = k1 < 0 ? -1 : (P.srow ? __ldg(P.srow + k1) : k1);
    }
    StagedRow fr;
    fr.frow = slab * 32 + lane;
    fr.e0 = fr.e1 = 0;
    fr.tok = -1;
    if (pam_on<kPam>(P)) {
      fr.tok = pam_token(P, m, row0, fr.frow);
    } else {
      const int fu = min(m * kPairRows + row0 + fr.frow, U - 1);
      const int fj0 = P.run_ptr[fu];
      fr.e0 = P.row_ptr[fj0];
      fr.e1 = P.row_ptr[fj0 + 1];
    }
    int pending = 0;  // stages issued and not yet finished (<= LAG)
    for (int kb = 0; kb < P.n_kb; ++kb) {
      if (!mbar_wait(smem_addr(&empty_a[stage]), phase ^ 1)) {
        raise_timeout(P, sAbort);
        ok = false;
        break;
      }
      const int seg = kb / P.atoms_per_seg, kin = kb - seg * P.atoms_per_seg;
      const int n_t = __ldg(&lsegs->n_terms[seg]);
      const int la0 = __ldg(&lsegs->layer[seg][0]);
      const int la1 = n_t > 1 ? __ldg(&lsegs->layer[seg][1]) : la0;
      const T* b0 = sender + static_cast<int64_t>(la0 * 2 + c) * lrows + kin * kBK + ch * kPerChunk;
      const T* b1 = sender + static_cast<int64_t>(la1 * 2 + c) * lrows + kin * kBK + ch * kPerChunk;
      const uint32_t sa = smem_addr(sA + stage * kStageABytes);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int r = slab * 32 + 4 * i + rsub;
        const uint32_t doff = static_cast<uint32_t>(r * 128 + ((ch ^ (r & 7)) << 4));
        if (kr0[i] >= 0) {
          cp_async_16(sa + doff, b0 + static_cast<int64_t>(kr0[i]) * P.d_s);
          if (n_t > 1)
            cp_async_16(sa + kAtomABytes + doff, b1 + static_cast<int64_t>(kr0[i]) * P.d_s);
        }
        if (n_t == 1 && kr1[i] >= 0)
          cp_async_16(sa + kAtomABytes + doff, b0 + static_cast<int64_t>(kr1[i]) * P.d_s);
      }
      cp_async_commit();
      if (pending == LAG) {
        // stage kb - LAG (issued LAG stages ago) has landed for this thread;
        // after the warp barrier, for the whole warp
        cp_async_wait<LAG>();
        __syncwarp();
        const int st = (stage + stages - LAG) % stages;
        finish_staged_row<T>(P, lsegs, c, fr, kb - LAG, sA + st * kStageABytes);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) arrive_leader(smem_addr(&full_a[st]), row0);
      } else {
        ++pending;
      }
      if (++stage == stages) {
        stage = 0;
        phase ^= 1;
      }
    }
    if (!ok) break;
    // the tile's last `pending` stages: stage - pending .. stage - 1
    cp_async_wait<0>();
    __syncwarp();
    for (int q = pending; q >= 1; --q) {
      const int st = (stage + stages - q) % stages;
      finish_staged_row<T>(P, lsegs, c, fr, P.n_kb - q, sA + st * kStageABytes);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) arrive_leader(smem_addr(&full_a[st]), row0);
    }
  }
}

// The kernel body for one direction (kDirs = 1, the map and parameters are
// kernel parameters) or several (tiles of all directions in one launch;
// every role looks its tile's direction up and reads that direction's
// parameters).  All directions share the dtype, the operand path and the
// ring depths; a B stage is stage_b_stride bytes (the widest direction's).
template <typename T, bool kGather, int kDirs, int kPam>
__device__ __forceinline__ void transfer_body(const CUtensorMap* maps, const XferParams* Ps,
                                              int n_dir, int stage_b_stride) {
  constexpr int kBK = Elem<T>::kBK;
  const XferParams& P0 = Ps[0];
  extern __shared__ __align__(1024) uint8_t smem[];
  if (smem_addr(smem) & 1023u) {  // the swizzled stages need 1024-byte alignment
    if (threadIdx.x == 0) atomicOr(P0.status, HF_CHECK_INTERNAL);
    return;
  }
  const uint32_t rank = cluster_ctarank();  // 0: leader of the pair (issues the MMAs)
  const bool leader = rank == 0;
  const int first_tile = static_cast<int>(cluster_id_x());
  const int tile_step = static_cast<int>(nclusters_x());
  const int row0 = static_cast<int>(rank) * kBM;  // this CTA's rows within a pair tile
  const int stages_a = P0.stages_a, stages_b = P0.stages_b;
  const int stage_b_bytes = stage_b_stride;
  uint8_t* sA = smem;
  uint8_t* sB = sA + stages_a * kStageABytes;
  float* sStg = reinterpret_cast<float*>(sB + stages_b * stage_b_bytes);
  int32_t* sRun = reinterpret_cast<int32_t*>(sStg + kStgFloats);
  int32_t* sUpos = sRun + kRunStride;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sUpos + kRunStride);
  uint64_t* full_a = bars;
  uint64_t* empty_a = bars + kMaxStages;
  uint64_t* full_b = bars + 2 * kMaxStages;
  uint64_t* empty_b = bars + 3 * kMaxStages;
  uint64_t* tfull = bars + 4 * kMaxStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* sTmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* sAbort = reinterpret_cast<volatile int*>(sTmem + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    // full_a / full_b / tempty of the leader collect both CTAs' arrivals;
    // the follower's copies are unused.  empty_* / tfull / drain receive the
    // leader's multicast commits in both CTAs.
    for (int s = 0; s < stages_a; ++s) {
      mbar_init(smem_addr(&full_a[s]), 2 * kBuilderWarps);  // every A builder warp of the pair
      mbar_init(smem_addr(&empty_a[s]), 1);
    }
    for (int s = 0; s < stages_b; ++s) {
      mbar_init(smem_addr(&full_b[s]), 2);  // one expect_tx per CTA + the TMA bytes
      mbar_init(smem_addr(&empty_b[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_addr(&tfull[a]), 1);
      mbar_init(smem_addr(&tempty[a]), 2 * kEpiWarps);  // every epilogue warp of the pair
    }
    mbar_init(smem_addr(drain), 1);
    *sAbort = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0)
    for (int d = 0; d < (kDirs == 1 ? 1 : n_dir); ++d) tma_prefetch_map(&maps[d]);
  if (warp == 1) {
    tmem_alloc_pair(smem_addr(sTmem), kTmemCols);
    tmem_relinquish_pair();
  }
  __syncthreads();
  cluster_sync();  // the leader's barriers exist before any remote arrival
  tc_fence_after_sync();
  const uint32_t tmem_base = *sTmem;

  DirTable<kDirs> dt;
  const int total_tiles = build_dirs<kDirs, kPam>(Ps, n_dir, &dt);
  const bool by_slot = slot_order(total_tiles, tile_step);

  if (warp == 0) {
    // ------------------------------------------------------------ map tiles
    // this CTA's half of the B tile: receiver columns n0 + rank*BN/2 .. +BN/2
    if (lane == 0) {
      // a map tile is read by every row block of its layer: its lines are
      // kept in L2 ahead of the sender rows (13% fewer DRAM reads at 32K)
      const uint64_t pol_b = l2_policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int seq = 0, tile = tile_of(0, first_tile, tile_step, by_slot); tile < total_tiles && ok;
       tile = tile_of(++seq, first_tile, tile_step, by_slot)) {
        const int dd = dir_of(dt, n_dir, tile);
        const XferParams& P = Ps[dd];
        const CUtensorMap* tmap = &maps[dd];
        const int half_bn = P.BN / 2;  // B rows (receiver columns) per CTA
        const int atom_b_bytes = half_bn * 128;
        int lc, m, n;
        decode_tile(tile - dt.base[dd], dt.m_tiles[dd] * P.n_tiles_n, P.n_tiles_n, P.l0, &lc, &m,
                    &n);
        // a wide tile takes each map atom for its two column blocks in turn
        const int n_half = P.wide ? 2 : 1;
        const int n_loads = P.n_batoms * n_half;
        for (int ab = 0; ab < n_loads; ++ab) {
          const int at = ab / n_half, h = ab - at * n_half;
          if (!mbar_wait(smem_addr(&empty_b[stage]), phase ^ 1)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          const uint32_t fb = mapa_shared(smem_addr(&full_b[stage]), 0);
          if (!(P.stall && seq == 0 && ab == 0)) {  // the test hook leaves this stage empty
            mbar_arrive_expect_tx_cluster(fb, atom_b_bytes);
            tma_load_2d_pair_hint(smem_addr(sB + stage * stage_b_bytes), tmap, at * kBK,
                                  lc * P.d_r + (n * n_half + h) * P.BN +
                                      static_cast<int>(rank) * half_bn,
                                  fb, pol_b);
          }
          if (++stage == stages_b) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issue
    if (lane == 0 && leader) {
      // This single thread shares its scheduler with busy epilogue and
      // builder warps, so the loop keeps its instruction count low: barrier
      // addresses and descriptors advance by adds (a descriptor's start
      // address field is the smem byte address >> 4; it cannot carry out for
      // addresses below 256 KB).
      const uint32_t full_a0 = smem_addr(full_a), empty_a0 = smem_addr(empty_a);
      const uint32_t full_b0 = smem_addr(full_b), empty_b0 = smem_addr(empty_b);
      const uint64_t desc_a0 = sw128_kmajor_desc(smem_addr(sA));
      const uint64_t desc_b0 = sw128_kmajor_desc(smem_addr(sB));
      const uint32_t step_a = kStageABytes >> 4, step_b = static_cast<uint32_t>(stage_b_bytes) >> 4;
      const uint32_t atom_a = kAtomABytes >> 4;
      int sa = 0, sb = 0;
      uint32_t pa = 0, pb = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int seq = 0, tile = tile_of(0, first_tile, tile_step, by_slot); tile < total_tiles && ok;
       tile = tile_of(++seq, first_tile, tile_step, by_slot)) {
        const XferParams& P = Ps[dir_of(dt, n_dir, tile)];
        const uint32_t idesc = P.idesc;
        const int n_kb = P.n_kb, last_atoms = P.last_atoms, per_stage = P.atoms_per_stage;
        const bool split = P.split != 0;
        const bool wide = !kGather && P.wide != 0;  // both accumulators, one per column block
        const int n_half = wide ? 2 : 1;
        bool free_acc = mbar_wait(smem_addr(&tempty[wide ? 0 : acc]), acc_phase ^ 1);
        if (free_acc && wide) free_acc = mbar_wait(smem_addr(&tempty[1]), acc_phase ^ 1);
        if (!free_acc) {
          raise_timeout(P, sAbort);
          break;
        }
        tc_fence_after_sync();
        uint32_t accumulate = 0;
        for (int kb = 0; kb < n_kb && ok; ++kb) {
          if (!mbar_wait(full_a0 + 8 * sa, pa)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          const int na = kb == n_kb - 1 ? last_atoms : per_stage;
#pragma unroll
          for (int a = 0; a < kAtoms; ++a) {
            if (a >= na) break;
           for (int h = 0; h < n_half; ++h) {
            if (!mbar_wait(full_b0 + 8 * sb, pb)) {
              raise_timeout(P, sAbort);
              ok = false;
              break;
            }
            tc_fence_after_sync();
            const uint32_t d_tmem = tmem_base + static_cast<uint32_t>((wide ? h : acc) * 256);
            const uint64_t ad = desc_a0 + sa * step_a + a * atom_a;
            const uint64_t bd = desc_b0 + sb * step_b;
            // four 32-byte K steps per 128-byte atom (descriptor units of 16 bytes)
            if (sizeof(T) == 2) {
              mma_bf16_pair(d_tmem, ad, bd, idesc, accumulate);
              mma_bf16_pair(d_tmem, ad + 2, bd + 2, idesc, 1);
              mma_bf16_pair(d_tmem, ad + 4, bd + 4, idesc, 1);
              mma_bf16_pair(d_tmem, ad + 6, bd + 6, idesc, 1);
              if (split) {  // the residual atom against the same map atom
                const uint64_t lo = ad + atom_a;
                mma_bf16_pair(d_tmem, lo, bd, idesc, 1);
                mma_bf16_pair(d_tmem, lo + 2, bd + 2, idesc, 1);
                mma_bf16_pair(d_tmem, lo + 4, bd + 4, idesc, 1);
                mma_bf16_pair(d_tmem, lo + 6, bd + 6, idesc, 1);
              }
            } else {
              mma_tf32_pair(d_tmem, ad, bd, idesc, accumulate);
              mma_tf32_pair(d_tmem, ad + 2, bd + 2, idesc, 1);
              mma_tf32_pair(d_tmem, ad + 4, bd + 4, idesc, 1);
              mma_tf32_pair(d_tmem, ad + 6, bd + 6, idesc, 1);
            }
            tc_commit_pair(empty_b0 + 8 * sb, 0x3);
            if (++sb == stages_b) {
              sb = 0;
              pb ^= 1;
            }
           }
            if (!ok) break;
            accumulate = 1;
          }
          if (!ok) break;
          tc_commit_pair(empty_a0 + 8 * sa, 0x3);
          if (++sa == stages_a) {
            sa = 0;
            pa ^= 1;
          }
        }
        if (!ok) break;
        if (wide) {
          tc_commit_pair(smem_addr(&tfull[0]), 0x3);
          tc_commit_pair(smem_addr(&tfull[1]), 0x3);
          acc_phase ^= 1;
        } else {
          tc_commit_pair(smem_addr(&tfull[acc]), 0x3);
          acc ^= 1;
          if (acc == 0) acc_phase ^= 1;
        }
      }
      // every issued MMA has completed before TMEM is released
      tc_commit_pair(smem_addr(drain), 0x3);
    }
    if (lane == 0) {
      if (!mbar_wait(smem_addr(drain), 0)) raise_timeout(P0, sAbort);
    }
    __syncwarp();
  } else if (warp < 2 + kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    // Ten warps per CTA, for the CTA's 128 rows of the pair tile.  Step 1
    // (per 16 rotation pairs of a head pair): warp (g, sp), e < 8, reads TMEM
    // lane quarter sp of head 2*hp+g, applies 1/r, bias and key norm, and
    // stages fp32 rows in smem.  Step 2: the ten warps split the rows'
    // receiver positions and write both heads, rotated.
    const int e = warp - 2;   // 0..9: slice of the tile's receiver rows
    const int g = e >> 2;     // head of the pair this warp stages (e < 8)
    const int sp = warp & 3;  // TMEM lane quarter this warp may access
    const int row = sp * 32 + lane;
    const bool stager = e < 8;
    const int tid_e = threadIdx.x - 64;
    const int ps = lane >> 2, qq = lane & 3;  // row slot 0..7, pair quad 0..3
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int seq = 0, tile = tile_of(0, first_tile, tile_step, by_slot); tile < total_tiles;
       tile = tile_of(++seq, first_tile, tile_step, by_slot)) {
      const int dd = dir_of(dt, n_dir, tile);
      const XferParams& P = Ps[dd];
      const int U = dt.U[dd];
      const int D = P.D_r, half = P.D_r / 2;
      const int n_heads = P.BN / D;
      const bool two_heads = n_heads >= 2;
      const int n_pairs = two_heads ? n_heads / 2 : 1;
      int lc, m, n;
      decode_tile(tile - dt.base[dd], dt.m_tiles[dd] * P.n_tiles_n, P.n_tiles_n, P.l0, &lc, &m,
                  &n);
      const int c = lc & 1;
      // a wide tile's two column blocks are drained in turn, one per accumulator
      const bool wide = !kGather && P.wide != 0;
      const int n_half = wide ? 2 : 1;
      bool timed_out = false;
      for (int h = 0; h < n_half; ++h) {
      const int ac = wide ? h : acc;        // TMEM accumulator
      const int nb = wide ? 2 * n + h : n;  // 256-column block of the map and the receiver
      if (!mbar_wait(smem_addr(&tfull[ac]), acc_phase)) {
        raise_timeout(P, sAbort);
        timed_out = true;
        break;
      }
      tc_fence_after_sync();
      const int u0 = m * kPairRows + row0;
      const int nrows = min(kBM, U - u0);  // <= 0: this CTA has no rows in the tile
      if (nrows > 0 && pam_on<kPam>(P)) {
        const int w = u0 >> 7;  // this CTA's window
        const int base = w * __ldg(P.win_info + 1);
        const int jb = __ldg(P.win_ptr + w), je = __ldg(P.win_ptr + w + 1);
        T* const out_lc = reinterpret_cast<T*>(P.receiver) +
                          (static_cast<int64_t>(lc) * P.recv_rows) * P.d_r;
        pam_epilogue<T>(P,
                        tmem_base + static_cast<uint32_t>(ac * 256) +
                            (static_cast<uint32_t>(sp * 32) << 16),
                        P.bias + static_cast<int64_t>(lc) * P.d_r + nb * P.BN, P.inv_r[lc], base,
                        jb, je, sStg, e, g, row, lane, P.rope && c == 0, out_lc, nb * P.BN);
      } else if (nrows > 0) {
        for (int i = tid_e; i <= nrows; i += kEpiThreads) {
          sRun[i] = P.run_ptr[u0 + i];
          sUpos[i] = i < nrows ? P.upos[u0 + i] : 0;
        }
        named_barrier_sync(1, kEpiThreads);
        // this warp's receiver rows [wjb, wje); lane slot ps walks the
        // consecutive rows [ljb, lje) of them
        const int jb = sRun[0], je = sRun[nrows];
        const int per = (je - jb + kEpiWarps - 1) / kEpiWarps;
        const int wjb = min(je, jb + e * per), wje = min(je, wjb + per);
        const int per_slot = (wje - wjb + 7) >> 3;
        const int ljb = min(wje, wjb + ps * per_slot), lje = min(wje, ljb + per_slot);
        const int ustart = ljb < lje ? find_row(sRun, nrows, ljb) : 0;
        const float inv_r = P.inv_r[lc];
        const float* bias = P.bias + static_cast<int64_t>(lc) * P.d_r;
        const bool do_rope = P.rope && c == 0;
        const bool do_knorm = P.knorm && c == 0;
        const uint32_t ta = tmem_base + static_cast<uint32_t>(ac * 256) +
                            (static_cast<uint32_t>(sp * 32) << 16);
        T* const out_lc = reinterpret_cast<T*>(P.receiver) +
                          (static_cast<int64_t>(lc) * P.recv_rows) * P.d_r;
        if (c == 1 || (!P.rope && !P.knorm)) {
          copy_epilogue<T>(P, ta, bias + nb * P.BN, inv_r, nrows, sRun,
                           reinterpret_cast<uint8_t*>(sStg), g, row, e, lane, out_lc, nb * P.BN);
        } else
        for (int hp = 0; hp < n_pairs; ++hp) {
          const bool stages_head = stager && (g == 0 || two_heads);
          const int tcol = (2 * hp + g) * D;            // accumulator column of this warp's head
          const int ocol_pair = nb * P.BN + 2 * hp * D;  // receiver feature of the pair's first head
          float rn = 1.0f;
          if (do_knorm && stages_head) {
            float ss = 0.0f;
            for (int q2 = 0; q2 < D; q2 += 16) {
              uint32_t v[16];
              tmem_load_16(ta + tcol + q2, v);
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const float y = fmaf(__uint_as_float(v[i]), inv_r,
                                     __ldg(bias + nb * P.BN + tcol + q2 + i));
                ss = fmaf(y, y, ss);
              }
            }
            rn = rsqrtf(ss / static_cast<float>(D) + P.knorm_eps);
          }
          for (int q = 0; q < half; q += 16) {
            // this lane's four frequencies, loaded before step 1 so that the
            // global read overlaps the staging
            float f[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) f[k] = do_rope ? __ldg(P.inv_freq + q + 4 * qq + k) : 0.f;
            if (stages_head) {
              // step 1: pairs q..q+15 of head 2*hp+g for this warp's 32 rows
              uint32_t v[32];
              tmem_load_2x16(ta + tcol + q, ta + tcol + half + q, v);
              const float* bcol = bias + nb * P.BN + tcol;
              float y[32];
#pragma unroll
              for (int i = 0; i < 16; i += 4) {
                const float4 x = __ldg(reinterpret_cast<const float4*>(bcol + q + i));
                const float4 z = __ldg(reinterpret_cast<const float4*>(bcol + half + q + i));
                y[i] = fmaf(__uint_as_float(v[i]), inv_r, x.x);
                y[i + 1] = fmaf(__uint_as_float(v[i + 1]), inv_r, x.y);
                y[i + 2] = fmaf(__uint_as_float(v[i + 2]), inv_r, x.z);
                y[i + 3] = fmaf(__uint_as_float(v[i + 3]), inv_r, x.w);
                y[16 + i] = fmaf(__uint_as_float(v[16 + i]), inv_r, z.x);
                y[16 + i + 1] = fmaf(__uint_as_float(v[16 + i + 1]), inv_r, z.y);
                y[16 + i + 2] = fmaf(__uint_as_float(v[16 + i + 2]), inv_r, z.z);
                y[16 + i + 3] = fmaf(__uint_as_float(v[16 + i + 3]), inv_r, z.w);
              }
              if (do_knorm) {
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                  y[i] *= rn * __ldg(P.knorm_w + q + i);
                  y[16 + i] *= rn * __ldg(P.knorm_w + half + q + i);
                }
              }
              float* srow = sStg + row * 64 + g * 32;
#pragma unroll
              for (int k = 0; k < 8; ++k)
                *reinterpret_cast<float4*>(srow + ((k ^ (row & 7)) << 2)) =
                    make_float4(y[4 * k], y[4 * k + 1], y[4 * k + 2], y[4 * k + 3]);
            }
            named_barrier_sync(1, kEpiThreads);
            // step 2: rows of this warp's slice, both heads of the pair
            float C1[4], S1[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              C1[k] = 1.f;
              S1[k] = 0.f;
              if (do_rope) rope_sincos(1, f[k], &S1[k], &C1[k]);  // one step = one row
            }
            walk_rows<T>(ljb, lje, ustart, sRun, sUpos, sStg, qq, two_heads, do_rope, f, C1, S1, P,
                         out_lc, ocol_pair, q, half);
            named_barrier_sync(1, kEpiThreads);
          }
        }
      }
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) arrive_leader(smem_addr(&tempty[ac]), row0);
      }
      if (timed_out) break;
      if (wide) {
        acc_phase ^= 1;
      } else {
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
    }
  } else {
    // ------------------------------------------------------------ A builders
    const int t = threadIdx.x - 64 - kEpiThreads;  // 0..127
    if (kGather) {
      switch (P0.lag) {
        case 1: gather_rows<T, 1, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
        case 2: gather_rows<T, 2, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
        case 3: gather_rows<T, 3, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
        case 4: gather_rows<T, 4, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
        default: gather_rows<T, 5, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
      }
    } else if (P0.staged) {
      switch (P0.lag) {
        case 1: build_rows_staged<T, 1, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
        case 2: build_rows_staged<T, 2, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
        default: build_rows_staged<T, 3, kDirs, kPam>(Ps, dt, n_dir, sA, full_a, empty_a, sAbort, t, lane, row0, total_tiles, first_tile, tile_step); break;
      }
    } else {
      // pooled CSR rows, blended sender layers and/or rotated sender keys:
      // thread t owns tile row t
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int seq = 0, tile = tile_of(0, first_tile, tile_step, by_slot); tile < total_tiles && ok;
       tile = tile_of(++seq, first_tile, tile_step, by_slot)) {
        const int dd = dir_of(dt, n_dir, tile);
        const XferParams& P = Ps[dd];
        int lc, m, n;
        decode_tile(tile - dt.base[dd], dt.m_tiles[dd] * P.n_tiles_n, P.n_tiles_n, P.l0, &lc, &m,
                    &n);
        const int l = lc >> 1, c = lc & 1;
        const LayerSegs segs = P.segs[l];
        int e0 = 0, e1 = 0, tok = -1;
        if (pam_on<kPam>(P)) {  // sender token of this row of the CTA's window
          tok = pam_token(P, m, row0, t);
        } else {
          const int u = min(m * kPairRows + row0 + t, dt.U[dd] - 1);
          const int j0 = P.run_ptr[u];
          e0 = P.row_ptr[j0];
          e1 = P.row_ptr[j0 + 1];
        }
        const bool unrot_k = P.unrot && c == 0;
        int seg = 0, kin = 0;  // segment of the next atom, and the atom within it
        for (int kb = 0; kb < P.n_kb; ++kb) {
          if (!mbar_wait(smem_addr(&empty_a[stage]), phase ^ 1)) {
            raise_timeout(P, sAbort);
            ok = false;
            break;
          }
          uint8_t* st = sA + stage * kStageABytes;
          if (P.split) {
            // one map atom of K: the value atom and its residual atom
            if (unrot_k)
              build_atom_unrotated<T>(P, segs, seg, kin, c, e0, e1, st, st + kAtomABytes, t);
            else
              build_atom<T>(P, segs, seg, kin, c, e0, e1, tok, st, st + kAtomABytes, t);
            if (++kin == P.atoms_per_seg) {
              kin = 0;
              ++seg;
            }
          } else if (unrot_k) {
            // the stage is whole heads of one segment (checked at plan creation)
            build_stage_unrotated<T>(P, segs, seg, kin, c, e0, e1, st, t);
            kin += kAtoms;
            if (kin == P.atoms_per_seg) {
              kin = 0;
              ++seg;
            }
          } else {
            const int na = kb == P.n_kb - 1 ? P.last_atoms : kAtoms;
            for (int a = 0; a < na; ++a) {
              build_atom<T>(P, segs, seg, kin, c, e0, e1, tok, st + a * kAtomABytes, nullptr, t);
              if (++kin == P.atoms_per_seg) {
                kin = 0;
                ++seg;
              }
            }
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) arrive_leader(smem_addr(&full_a[stage]), row0);
          if (++stage == stages_a) {
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
  cluster_sync();  // neither CTA leaves while the pair's MMAs or arrivals may touch it
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

template <typename T, bool kGather, int kPam>
__global__ void __launch_bounds__(kThreads, 1)
    transfer_kernel(const __grid_constant__ CUtensorMap tmap_w,
                    const __grid_constant__ XferParams P) {
  transfer_body<T, kGather, 1, kPam>(&tmap_w, &P, 1, (P.BN / 2) * 128);
}

// Several directions in one launch (hf_transfer_batch).
struct BatchParams {
  CUtensorMap maps[kMaxBatch];
  XferParams P[kMaxBatch];
  int n_dir;
  int stage_b_stride;
};
static_assert(sizeof(BatchParams) < 32000, "BatchParams must fit the kernel parameter space");

template <typename T, bool kGather, int kPam>
__global__ void __launch_bounds__(kThreads, 1)
    transfer_batch_kernel(const __grid_constant__ BatchParams B) {
  transfer_body<T, kGather, kMaxBatch, kPam>(B.maps, B.P, B.n_dir, B.stage_b_stride);
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

size_t smem_bytes(int BN, int stages_a, int stages_b) {
  return static_cast<size_t>(stages_a) * kStageABytes +
         static_cast<size_t>(stages_b) * (BN / 2) * 128 + kStgFloats * sizeof(float) +
         2 * kRunStride * sizeof(int32_t) + (4 * kMaxStages + 5) * sizeof(uint64_t) + 8;
}

// Ring depths.  A B stage is one 128-byte atom of K of this CTA's map rows
// (16 KB at BN = 256), so the TMA producer refills the ring in fine steps;
// 96 KB of B stages, and the rest of shared memory in A stages (two atoms,
// 32 KB): three at BN = 256.  A loader waits for stage i - lag after issuing
// stage i, so it never blocks on a young group.  Measured on the 32K
// Llama -> Ministral-shaped transfer: three A stages and six one-atom B stages
// beat three two-atom B stages by 1%, and four A stages with four one-atom B
// stages lose 2-3% (deeper A rings do not pay; B depth does).
void pick_rings(int BN, int* stages_a, int* stages_b, int* lag) {
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  const int sb = std::min(kMaxStages, (96 * 1024) / ((BN / 2) * 128));
  int sa = kMaxStages;
  while (sa > 2 && smem_bytes(BN, sa, sb) > static_cast<size_t>(optin)) --sa;
  *stages_a = sa;
  *stages_b = sb;
  *lag = std::max(1, sa - 2);
}

// Launches `kern` with clusters of two CTAs: one CTA pair per co-resident
// cluster slot, at most one per pair tile.
template <typename Kern, typename... Args>
hf_status launch_pairs(Kern kern, int64_t max_pair_tiles, size_t smem, cudaStream_t stream,
                       Args... args) {
  HF_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(smem)),
              "set shared memory size");
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // one CTA pair per co-resident cluster slot, at most one per pair tile
  int clusters = device_sm_count() / 2;
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  int active = 0;
  if (cudaOccupancyMaxActiveClusters(&active, kern, &cfg) == cudaSuccess && active > 0)
    clusters = std::min(clusters, active);
  clusters = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(clusters, max_pair_tiles)));
  cfg.gridDim = dim3(2 * clusters, 1, 1);
  HF_CUDA_TRY(cudaLaunchKernelEx(&cfg, kern, args...), "transfer kernel launch");
  return HF_OK;
}

}  // namespace

namespace {

// The kernel parameters and map tile descriptor of one plan's launch over
// receiver layers [l_begin, l_end); *max_pair_tiles bounds its pair tiles.
hf_status make_xfer(hf_plan_s* p, const void* sender, void* receiver, int l_begin, int l_end,
                    XferParams* out, CUtensorMap* map_out, int64_t* max_pair_tiles) {
  const hf_plan_desc& d = p->desc;
  const bool f32 = d.dtype == HF_F32;
  const int esize = f32 ? 4 : 2;
  const int bk = 128 / esize;
  CUtensorMap& mw = *map_out;
  hf_status s = make_map(&mw, d.d_W, f32, static_cast<uint64_t>(d.L_r) * 2 * p->d_r,
                         static_cast<uint64_t>(p->K), static_cast<uint32_t>(p->BN / 2),
                         static_cast<uint32_t>(bk), CU_TENSOR_MAP_L2_PROMOTION_L2_256B);
  if (s != HF_OK) return s;
  XferParams& P = *out;
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
  P.s_rows = p->s_rows;
  P.srow = p->span ? reinterpret_cast<const int32_t*>(ws + p->lay.srow) : nullptr;
  P.recv_rows = d.paged ? static_cast<int64_t>(d.n_blocks) * d.block_size : p->T_r;
  P.L_r = d.L_r;
  P.l0 = l_begin;
  P.n_l = l_end - l_begin;
  P.d_s = p->d_s;
  P.d_r = p->d_r;
  P.D_r = d.D_r;
  const int n_atoms = p->K / bk;  // 128-byte k-blocks per output row
  P.split = p->split ? 1 : 0;
  P.staged = p->staged ? 1 : 0;
  P.pam = p->pam ? 1 : 0;
  P.win_info = reinterpret_cast<const int32_t*>(ws + p->lay.win_info);
  P.win_ptr = reinterpret_cast<const int32_t*>(ws + p->lay.win_ptr);
  P.pos = reinterpret_cast<const int32_t*>(ws + p->lay.pos);
  P.atoms_per_stage = p->split ? 1 : kAtoms;
  P.n_batoms = n_atoms;
  P.n_kb = (n_atoms + P.atoms_per_stage - 1) / P.atoms_per_stage;
  P.last_atoms = n_atoms - P.atoms_per_stage * (P.n_kb - 1);
  P.atoms_per_seg = p->d_s / bk;
  P.BN = p->BN;
  P.wide = p->wide ? 1 : 0;
  P.n_tiles_n = p->d_r / (p->BN * (p->wide ? 2 : 1));
  pick_rings(p->BN, &P.stages_a, &P.stages_b, &P.lag);
  P.rope = p->rope ? 1 : 0;
  P.unrot = p->unrot ? 1 : 0;
  P.D_s = d.D_s;
  P.inv_freq_s = reinterpret_cast<const float*>(ws + p->lay.inv_freq_s);
  P.spos = reinterpret_cast<const int32_t*>(ws + p->lay.spos);
  P.paged = d.paged ? 1 : 0;
  P.knorm = d.d_knorm_w ? 1 : 0;
  P.knorm_eps = d.knorm_eps;
  P.idesc = make_idesc(f32 ? 2u : 1u, kPairRows, p->BN);
  // pooling after the map: at most T_s windows (stride >= 1), two per pair tile
  const int64_t row_blocks = p->pam ? (p->T_s + 1) / 2 : (p->T_r + kPairRows - 1) / kPairRows;
  *max_pair_tiles = 2LL * P.n_l * row_blocks * static_cast<int64_t>(P.n_tiles_n);
  return HF_OK;
}

template <typename T, bool kGather, int kPam>
hf_status launch_batch_typed(const BatchParams& B, int64_t max_pair_tiles, size_t smem,
                             cudaStream_t stream) {
  return launch_pairs(transfer_batch_kernel<T, kGather, kPam>, max_pair_tiles, smem, stream, B);
}

}  // namespace

hf_status launch_transfer(hf_plan_s* p, const void* sender, void* receiver, cudaStream_t stream,
                          int l_begin, int l_end, bool stall) {
  const hf_plan_desc& d = p->desc;
  if (l_end < 0) l_end = d.L_r;
  if (p->T_r == 0 || l_end <= l_begin) return HF_OK;
  XferParams P;
  CUtensorMap mw;
  int64_t max_pair_tiles = 0;
  hf_status s = make_xfer(p, sender, receiver, l_begin, l_end, &P, &mw, &max_pair_tiles);
  if (s != HF_OK) return s;
  P.stall = stall ? 1 : 0;
  const size_t smem = smem_bytes(p->BN, P.stages_a, P.stages_b);
  if (d.dtype == HF_F32)
    return p->gather
               ? launch_pairs(transfer_kernel<float, true, 2>, max_pair_tiles, smem, stream, mw, P)
               : launch_pairs(transfer_kernel<float, false, 2>, max_pair_tiles, smem, stream, mw, P);
  if (p->pam)
    return p->gather
               ? launch_pairs(transfer_kernel<__nv_bfloat16, true, 1>, max_pair_tiles, smem, stream, mw, P)
               : launch_pairs(transfer_kernel<__nv_bfloat16, false, 1>, max_pair_tiles, smem, stream, mw, P);
  return p->gather
             ? launch_pairs(transfer_kernel<__nv_bfloat16, true, 0>, max_pair_tiles, smem, stream, mw, P)
             : launch_pairs(transfer_kernel<__nv_bfloat16, false, 0>, max_pair_tiles, smem, stream, mw, P);
}

bool batch_compatible(const hf_plan_s* const* plans, int n) {
  for (int i = 1; i < n; ++i)
    if (plans[i]->desc.dtype != plans[0]->desc.dtype || plans[i]->gather != plans[0]->gather ||
        plans[i]->split != plans[0]->split || plans[i]->staged != plans[0]->staged ||
        plans[i]->pam != plans[0]->pam || plans[i]->wide != plans[0]->wide)
      return false;
  return true;
}

hf_status launch_transfer_batch(hf_plan_s* const* plans, const void* const* senders,
                                void* const* receivers, int n, cudaStream_t stream) {
  BatchParams* B = new BatchParams();
  std::memset(B, 0, sizeof(*B));
  int64_t tiles = 0;
  int max_bn = 0, k = 0;
  for (int i = 0; i < n; ++i) {
    hf_plan_s* p = plans[i];
    if (p->T_r == 0) continue;
    int64_t mt = 0;
    const hf_status s = make_xfer(p, senders[i], receivers[i], 0, p->desc.L_r, &B->P[k],
                                  &B->maps[k], &mt);
    if (s != HF_OK) {
      delete B;
      return s;
    }
    tiles += mt;
    max_bn = std::max(max_bn, p->BN);
    ++k;
  }
  if (k == 0) {
    delete B;
    return HF_OK;
  }
  int sa = 0, sb = 0, lag = 0;
  pick_rings(max_bn, &sa, &sb, &lag);
  for (int i = 0; i < k; ++i) {
    B->P[i].stages_a = sa;
    B->P[i].stages_b = sb;
    B->P[i].lag = lag;
  }
  B->n_dir = k;
  B->stage_b_stride = (max_bn / 2) * 128;
  const size_t smem = smem_bytes(max_bn, sa, sb);
  hf_status s;
  if (plans[0]->desc.dtype == HF_F32)
    s = plans[0]->gather ? launch_batch_typed<float, true, 2>(*B, tiles, smem, stream)
                         : launch_batch_typed<float, false, 2>(*B, tiles, smem, stream);
  else if (plans[0]->pam)
    s = plans[0]->gather ? launch_batch_typed<__nv_bfloat16, true, 1>(*B, tiles, smem, stream)
                         : launch_batch_typed<__nv_bfloat16, false, 1>(*B, tiles, smem, stream);
  else
    s = plans[0]->gather ? launch_batch_typed<__nv_bfloat16, true, 0>(*B, tiles, smem, stream)
                         : launch_batch_typed<__nv_bfloat16, false, 0>(*B, tiles, smem, stream);
  delete B;
  return s;
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

extern "C" hf_status hf_debug_transfer_stalled(hf_plan plan, const void* sender_kv,
                                               void* receiver_kv, hf_stream_t stream) {
  if (!plan || plan->T_r == 0 || !sender_kv || !receiver_kv) {
    hf::set_error("hf_debug_transfer_stalled: needs a plan with receiver tokens and both caches");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if ((reinterpret_cast<uintptr_t>(sender_kv) | reinterpret_cast<uintptr_t>(receiver_kv) |
       reinterpret_cast<uintptr_t>(plan->desc.d_W)) & 15u) {
    hf::set_error("hf_debug_transfer_stalled: caches and maps must be 16-byte aligned");
    return HF_ERR_INVALID_ARGUMENT;
  }
  return hf::launch_transfer(plan, sender_kv, receiver_kv, reinterpret_cast<cudaStream_t>(stream),
                             0, -1, true);
}
