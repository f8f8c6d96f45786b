// Single-block in-place inclusive scans (sum or max) of int32 arrays, and
// small search helpers.  Used by the alignment builder (forward fill of the
// latest shared boundary, CSR row pointers) and the plan builder (numbering
// of distinct alignment rows).
#pragma once

#include <limits.h>
#include <stdint.h>

namespace hf {

constexpr int kScanThreads = 1024;
constexpr int kScanItems = 8;

struct ScanSum {
  static __device__ __forceinline__ int identity() { return 0; }
  __device__ __forceinline__ int operator()(int a, int b) const { return a + b; }
};

struct ScanMax {
  static __device__ __forceinline__ int identity() { return INT_MIN; }
  __device__ __forceinline__ int operator()(int a, int b) const { return a > b ? a : b; }
};

// Loads this thread's kScanItems consecutive items at i0 (identity past n):
// two 16-byte loads when the tile is whole and the array is 16-byte aligned.
template <typename Op>
__device__ __forceinline__ void scan_load(const int* data, int64_t n, int64_t i0, bool vec,
                                          int* v) {
  if (vec && i0 + kScanItems <= n) {
    const int4 a = *reinterpret_cast<const int4*>(data + i0);
    const int4 b = *reinterpret_cast<const int4*>(data + i0 + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  } else {
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) v[i] = (i0 + i < n) ? data[i0 + i] : Op::identity();
  }
}

// data[i] <- op(data[0..i]) for i < n, in tiles of 1024 x 8 items carried
// across tiles; the next tile's items are loaded while the current one is
// scanned.  *total (if not null) receives op over all n items (the identity
// when n == 0).  Launch with one block of kScanThreads threads.
template <typename Op>
__global__ void __launch_bounds__(kScanThreads) scan_inplace_kernel(int* data, int64_t n,
                                                                    int* total) {
  static_assert(kScanItems == 8, "scan_load reads two int4 per thread");
  __shared__ int warp_incl[kScanThreads / 32];
  const Op op;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool vec = (reinterpret_cast<uintptr_t>(data) & 15u) == 0;
  constexpr int64_t kTile = (int64_t)kScanThreads * kScanItems;
  int carry = Op::identity();
  int nv[kScanItems];
  if (n > 0) scan_load<Op>(data, n, (int64_t)tid * kScanItems, vec, nv);
  for (int64_t base = 0; base < n; base += kTile) {
    int v[kScanItems];
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) v[i] = nv[i];
    const int64_t i0 = base + (int64_t)tid * kScanItems;
    if (base + kTile < n) scan_load<Op>(data, n, i0 + kTile, vec, nv);
#pragma unroll
    for (int i = 1; i < kScanItems; ++i) v[i] = op(v[i - 1], v[i]);
    // inclusive scan of the per-thread totals within the warp
    int t = v[kScanItems - 1];
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, t, off);
      if (lane >= off) t = op(o, t);
    }
    int lane_excl = __shfl_up_sync(0xffffffffu, t, 1);
    if (lane == 0) lane_excl = Op::identity();
    if (lane == 31) warp_incl[warp] = t;
    __syncthreads();
    if (warp == 0) {
      int w = warp_incl[lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, w, off);
        if (lane >= off) w = op(o, w);
      }
      warp_incl[lane] = w;
    }
    __syncthreads();
    const int warp_excl = warp > 0 ? warp_incl[warp - 1] : Op::identity();
    const int excl = op(carry, op(warp_excl, lane_excl));
    if (vec && i0 + kScanItems <= n) {
      *reinterpret_cast<int4*>(data + i0) =
          make_int4(op(excl, v[0]), op(excl, v[1]), op(excl, v[2]), op(excl, v[3]));
      *reinterpret_cast<int4*>(data + i0 + 4) =
          make_int4(op(excl, v[4]), op(excl, v[5]), op(excl, v[6]), op(excl, v[7]));
    } else {
#pragma unroll
      for (int i = 0; i < kScanItems; ++i)
        if (i0 + i < n) data[i0 + i] = op(excl, v[i]);
    }
    carry = op(carry, warp_incl[31]);
    __syncthreads();
  }
  if (tid == 0 && total != nullptr) *total = carry;
}

// Index of the request owning global token j: the largest q with
// ptr[q] <= j (empty requests are skipped because a later equal pointer wins).
__device__ __forceinline__ int find_request(const int32_t* ptr, int n_req, int64_t j) {
  int lo = 0, hi = n_req - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (ptr[mid] <= j) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// First index k in [0, n) with a[k] >= x (n if none).
__device__ __forceinline__ int lower_bound_i32(const int32_t* a, int n, int32_t x) {
  int lo = 0, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (a[mid] < x) lo = mid + 1; else hi = mid;
  }
  return lo;
}

// First index k in [0, n) with a[k] > x (n if none).
__device__ __forceinline__ int upper_bound_i32(const int32_t* a, int n, int32_t x) {
  int lo = 0, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (a[mid] <= x) lo = mid + 1; else hi = mid;
  }
  return lo;
}

}  // namespace hf
