// Plan creation: descriptor validation, the layer table (Eq. 1, the
// interpolation reading or a caller-given table), RoPE inverse frequencies,
// and the per-transfer device metadata (receiver positions and destination
// rows, sender positions for rotated sender keys, runs of identical
// alignment rows).  Also the error-reporting helpers of the ABI.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>

#include "hf_device.cuh"
#include "hf_internal.h"
#include "hf_scan.cuh"

namespace hf {

namespace {
thread_local std::string g_last_error;
}

void set_error(const std::string& msg) { g_last_error = msg; }

hf_status cuda_fail(cudaError_t e, const char* what) {
  set_error(std::string(what) + ": " + cudaGetErrorString(e));
  return HF_ERR_CUDA;
}

int device_sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
    return 1;
  return n;
}

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

WorkspaceLayout workspace_layout(const hf_plan_desc& d) {
  const int L_r = d.L_r, D_r = d.D_r, D_s = d.D_s, n_req = d.n_req;
  const int64_t T_r = d.r_tok_ptr[n_req];
  const int64_t n_spos = d.sender_k_rotated ? d.s_tok_ptr[n_req] : 0;
  const int64_t n_srow = d.s_row0 ? d.s_tok_ptr[n_req] : 0;
  // pooling after the map may apply (the plan decides): window tables
  const bool pam = d.align_mode == HF_ALIGN_OVERLAP_MEAN && d.pool_before_map == 0;
  const int64_t n_key = pam ? T_r : 0;
  const int64_t n_win = pam ? d.s_tok_ptr[n_req] + 2 : 0;
  WorkspaceLayout w{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes, 256);
    return at;
  };
  w.status = take(sizeof(int32_t));
  w.n_distinct = take(sizeof(int32_t));
  w.segs = take(sizeof(LayerSegs) * (size_t)L_r);
  w.inv_r = take(sizeof(float) * 2 * (size_t)L_r);
  w.inv_freq = take(sizeof(float) * (size_t)(D_r / 2 > 0 ? D_r / 2 : 1));
  w.inv_freq_s = take(sizeof(float) * (size_t)(D_s / 2 > 0 ? D_s / 2 : 1));
  w.r_tok_ptr = take(sizeof(int32_t) * (size_t)(n_req + 1));
  w.r_pos0 = take(sizeof(int32_t) * (size_t)n_req);
  w.s_tok_ptr = take(sizeof(int32_t) * (size_t)(n_req + 1));
  w.s_pos0 = take(sizeof(int32_t) * (size_t)n_req);
  w.spos = take(sizeof(int32_t) * (size_t)(n_spos > 0 ? n_spos : 1));
  w.s_row0 = take(sizeof(int32_t) * (size_t)n_req);
  w.srow = take(sizeof(int32_t) * (size_t)(n_srow > 0 ? n_srow : 1));
  w.run_ptr = take(sizeof(int32_t) * (size_t)(T_r + 1));
  w.ucol = take(sizeof(int32_t) * (size_t)(T_r > 0 ? T_r : 1));
  w.upos = take(sizeof(int32_t) * (size_t)(T_r > 0 ? T_r : 1));
  w.pos = take(sizeof(int32_t) * (size_t)(T_r > 0 ? T_r : 1));
  w.dst_row = take(sizeof(int32_t) * (size_t)(T_r > 0 ? T_r : 1));
  w.new_flag = take(sizeof(int32_t) * (size_t)(T_r > 0 ? T_r : 1));
  w.win_info = take(sizeof(int32_t) * 4);
  w.row_key = take(sizeof(int32_t) * (size_t)(n_key > 0 ? n_key : 1));
  w.win_ptr = take(sizeof(int32_t) * (size_t)(n_win > 0 ? n_win : 1));
  w.total = off;
  return w;
}

namespace {

struct PlanDev {
  int32_t* status;
  int32_t* n_distinct;
  LayerSegs* segs;
  float* inv_r;
  float* inv_freq;
  float* inv_freq_s;
  int32_t* r_tok_ptr;
  int32_t* r_pos0;
  int32_t* s_tok_ptr;
  int32_t* s_pos0;
  int32_t* spos;
  int32_t* s_row0;
  int32_t* srow;
  int32_t* run_ptr;
  int32_t* ucol;
  int32_t* upos;
  int32_t* pos;
  int32_t* dst_row;
  int32_t* new_flag;
  int32_t* win_info;
  int32_t* row_key;
  int32_t* win_ptr;
};

PlanDev plan_dev(const hf_plan_s* p) {
  auto at = [&](size_t off) { return p->ws + off; };
  PlanDev d;
  d.status = reinterpret_cast<int32_t*>(at(p->lay.status));
  d.n_distinct = reinterpret_cast<int32_t*>(at(p->lay.n_distinct));
  d.segs = reinterpret_cast<LayerSegs*>(at(p->lay.segs));
  d.inv_r = reinterpret_cast<float*>(at(p->lay.inv_r));
  d.inv_freq = reinterpret_cast<float*>(at(p->lay.inv_freq));
  d.r_tok_ptr = reinterpret_cast<int32_t*>(at(p->lay.r_tok_ptr));
  d.r_pos0 = reinterpret_cast<int32_t*>(at(p->lay.r_pos0));
  d.inv_freq_s = reinterpret_cast<float*>(at(p->lay.inv_freq_s));
  d.s_tok_ptr = reinterpret_cast<int32_t*>(at(p->lay.s_tok_ptr));
  d.s_pos0 = reinterpret_cast<int32_t*>(at(p->lay.s_pos0));
  d.spos = reinterpret_cast<int32_t*>(at(p->lay.spos));
  d.s_row0 = reinterpret_cast<int32_t*>(at(p->lay.s_row0));
  d.srow = reinterpret_cast<int32_t*>(at(p->lay.srow));
  d.run_ptr = reinterpret_cast<int32_t*>(at(p->lay.run_ptr));
  d.ucol = reinterpret_cast<int32_t*>(at(p->lay.ucol));
  d.upos = reinterpret_cast<int32_t*>(at(p->lay.upos));
  d.pos = reinterpret_cast<int32_t*>(at(p->lay.pos));
  d.dst_row = reinterpret_cast<int32_t*>(at(p->lay.dst_row));
  d.new_flag = reinterpret_cast<int32_t*>(at(p->lay.new_flag));
  d.win_info = reinterpret_cast<int32_t*>(at(p->lay.win_info));
  d.row_key = reinterpret_cast<int32_t*>(at(p->lay.row_key));
  d.win_ptr = reinterpret_cast<int32_t*>(at(p->lay.win_ptr));
  return d;
}

// Copies the constant tables into the workspace and clears the counters.
// The tables stay in the kernel parameter space (__grid_constant__): indexing
// a by-value parameter with a thread-dependent index would make every
// thread copy the whole table to local memory first.
__global__ void plan_init_kernel(const __grid_constant__ PlanConsts t, PlanDev d) {
  const int tid = threadIdx.x;
  if (tid == 0) {
    *d.status = 0;
    *d.n_distinct = 0;
  }
  if (tid < 4) d.win_info[tid] = 0;
  for (int i = tid; i < 2 * t.L_r; i += blockDim.x) d.inv_r[i] = t.inv_r[i];
  for (int i = tid; i < t.D_r / 2; i += blockDim.x) d.inv_freq[i] = t.inv_freq[i];
  for (int i = tid; i <= t.n_req; i += blockDim.x) d.r_tok_ptr[i] = t.r_tok_ptr[i];
  for (int i = tid; i < t.n_req; i += blockDim.x) d.r_pos0[i] = t.r_pos0[i];
  for (int i = tid; i < t.D_s / 2; i += blockDim.x) d.inv_freq_s[i] = t.inv_freq_s[i];
  for (int i = tid; i <= t.n_req; i += blockDim.x) d.s_tok_ptr[i] = t.s_tok_ptr[i];
  for (int i = tid; i < t.n_req; i += blockDim.x) d.s_pos0[i] = t.s_pos0[i];
  for (int i = tid; i < t.n_req; i += blockDim.x) d.s_row0[i] = t.s_row0[i];
}

// Copies the layer table into the workspace, one 32-bit word per thread step.
__global__ void plan_segs_kernel(const __grid_constant__ SegTables t, LayerSegs* segs) {
  static_assert(sizeof(LayerSegs) % 4 == 0, "LayerSegs is copied as 32-bit words");
  const uint32_t* src = reinterpret_cast<const uint32_t*>(t.segs);
  uint32_t* dst = reinterpret_cast<uint32_t*>(segs);
  const int n = t.L_r * static_cast<int>(sizeof(LayerSegs) / 4);
  for (int i = threadIdx.x; i < n; i += blockDim.x) dst[i] = src[i];
}

// Per aligned sender token: its RoPE position (sender_k_rotated), the
// request's origin plus the token's index within the request; and its
// sender-cache row (message spans), the span's first row plus that index.
__global__ void plan_sender_kernel(PlanDev d, int64_t T_s, int n_req, int want_pos,
                                   int want_row) {
  for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < T_s;
       k += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(d.s_tok_ptr, n_req, k);
    const int32_t t = static_cast<int32_t>(k - d.s_tok_ptr[q]);
    if (want_pos) d.spos[k] = d.s_pos0[q] + t;
    if (want_row) d.srow[k] = d.s_row0[q] + t;
  }
}

struct RowArgs {
  PlanDev d;
  const int32_t* row_ptr;
  const int32_t* col;
  const float* w;
  const int32_t* block_table;
  int64_t T_r;
  int64_t T_s;
  int n_req;
  int paged, block_size, n_blocks, max_blocks;
  int single_entry;  // rows must be one entry of weight 1
  int span;          // map sender tokens to cache rows through d.srow
  int pam;           // pooling after the map: row keys and the widest column span
};

__device__ __forceinline__ void flag(int32_t* status, int bits) { atomicOr(status, bits); }

// Per receiver row: position, destination row, checks, and whether the row
// differs from the previous one (starts a new distinct row).
__global__ void plan_rows_kernel(RowArgs a) {
  const PlanDev& d = a.d;
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < a.T_r;
       j += (int64_t)gridDim.x * blockDim.x) {
    const int q = find_request(d.r_tok_ptr, a.n_req, j);
    const int32_t r0 = d.r_tok_ptr[q];
    const int32_t t = static_cast<int32_t>(j - r0);
    d.pos[j] = d.r_pos0[q] + t;
    int32_t dst = static_cast<int32_t>(j);
    if (a.paged) {
      const int bi = t / a.block_size;
      int32_t blk = -1;
      if (bi < a.max_blocks) blk = a.block_table[(int64_t)q * a.max_blocks + bi];
      if (blk < 0 || blk >= a.n_blocks) {
        flag(d.status, HF_CHECK_BAD_BLOCK);
        dst = -1;
      } else {
        dst = blk * a.block_size + t % a.block_size;
      }
    }
    d.dst_row[j] = dst;
    const int32_t e0 = a.row_ptr[j], e1 = a.row_ptr[j + 1];
    if (e1 <= e0) flag(d.status, HF_CHECK_BAD_ROW);
    if (a.single_entry && (e1 - e0 != 1 || a.w[e0] != 1.0f)) flag(d.status, HF_CHECK_BAD_ROW);
    int32_t kmin = INT_MAX, kmax = -1;
    for (int32_t e = e0; e < e1; ++e) {
      const int32_t k = a.col[e];
      if (k < 0 || k >= a.T_s) {
        flag(d.status, HF_CHECK_BAD_COLUMN);
      } else {
        kmin = min(kmin, k);
        kmax = max(kmax, k);
      }
    }
    if (a.pam) {
      // the row's first valid column (-1: none); made a running maximum by
      // a scan, it assigns the row to a window
      d.row_key[j] = kmax >= 0 ? kmin : -1;
      if (kmax >= 0) atomicMax(&d.win_info[0], kmax - kmin);
    }
    int is_new = (j == r0) ? 1 : 0;
    if (!is_new) {
      const int32_t p0 = a.row_ptr[j - 1];
      if (e1 - e0 != e0 - p0) {
        is_new = 1;
      } else {
        for (int32_t i = 0; i < e1 - e0; ++i) {
          if (a.col[e0 + i] != a.col[p0 + i] || a.w[e0 + i] != a.w[p0 + i]) {
            is_new = 1;
            break;
          }
        }
      }
    }
    d.new_flag[j] = is_new;
  }
}

// After the inclusive scan new_flag[j] = (index of j's distinct row) + 1.
__global__ void plan_runs_kernel(RowArgs a) {
  const PlanDev& d = a.d;
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < a.T_r;
       j += (int64_t)gridDim.x * blockDim.x) {
    const int32_t incl = d.new_flag[j];
    const bool starts = (j == 0) || (incl != d.new_flag[j - 1]);
    if (starts) {
      const int32_t u = incl - 1;
      d.run_ptr[u] = static_cast<int32_t>(j);
      // an empty row (flagged by plan_rows_kernel) has no column to read:
      // row_ptr[j] may be the end of the caller's col array
      const int32_t e0 = a.row_ptr[j];
      int32_t k = a.row_ptr[j + 1] > e0 ? a.col[e0] : 0;
      if (k < 0 || k >= a.T_s) k = 0;  // flagged by plan_rows_kernel
      d.ucol[u] = a.span ? d.srow[k] : k;  // the sender-cache row
      d.upos[u] = d.pos[j];
    }
    if (j == a.T_r - 1) {
      d.run_ptr[incl] = static_cast<int32_t>(a.T_r);
      *d.n_distinct = incl;
    }
  }
}

// Pooling after the map: window w holds the aligned sender tokens
// [w S, w S + 128), S = 128 - h with h the widest row's column span, so a
// row whose first column c satisfies w = floor(c / S) has every column in
// window w.  After the max-scan row_key[j] is the largest first column of
// rows 0..j (non-decreasing); window w takes the rows j with
// floor(row_key[j] / S) = w, win_ptr[w] the first of them.  A row whose
// columns leave its window (first columns that decrease, or h >= 128) is
// flagged.
__global__ void plan_windows_kernel(RowArgs a) {
  const PlanDev& d = a.d;
  const int32_t h = d.win_info[0];
  const bool too_wide = h >= 128;
  const int32_t S = too_wide ? 1 : 128 - h;
  const int32_t last = d.row_key[a.T_r - 1];
  const int32_t n_win = last < 0 ? 0 : last / S + 1;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    d.win_info[1] = S;
    d.win_info[2] = n_win;
    if (too_wide) flag(d.status, HF_CHECK_POOL_WINDOW);
  }
  const int64_t n = a.T_r > (int64_t)n_win + 1 ? a.T_r : (int64_t)n_win + 1;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    if (i < a.T_r) {
      const int32_t key = d.row_key[i];
      if (key >= 0) {
        const int64_t lo = (int64_t)(key / S) * S;
        for (int32_t e = a.row_ptr[i]; e < a.row_ptr[i + 1]; ++e) {
          const int32_t k = a.col[e];
          if (k >= 0 && k < a.T_s && (k < lo || k >= lo + 128)) flag(d.status, HF_CHECK_POOL_WINDOW);
        }
      }
    }
    if (i <= n_win) {
      const int64_t x = i * (int64_t)S;
      d.win_ptr[i] = x > INT_MAX ? static_cast<int32_t>(a.T_r)
                                 : lower_bound_i32(d.row_key, static_cast<int>(a.T_r),
                                                   static_cast<int32_t>(x));
    }
  }
}

// Eq. 1: pi(l) = 1 + round((l-1)(L_S-1)/(L_R-1)) (one-based), round half
// away from zero, computed exactly in integers.
int proportional_depth(int l1, int L_s, int L_r) {
  if (L_r == 1) return 1;
  const long long num = (long long)(l1 - 1) * (L_s - 1);
  const long long den = L_r - 1;
  return 1 + static_cast<int>((2 * num + den) / (2 * den));
}

void build_layer_table(const hf_plan_desc& d, LayerSegs* out) {
  for (int l = 0; l < d.L_r; ++l) {
    LayerSegs s;
    std::memset(&s, 0, sizeof(s));
    if (d.layer_mode == HF_LAYER_EXPLICIT) {
      s.n_seg = d.n_seg;
      for (int k = 0; k < d.n_seg; ++k) {
        s.n_terms[k] = d.n_terms;
        for (int t = 0; t < d.n_terms; ++t) {
          const size_t i = ((size_t)l * d.n_seg + k) * d.n_terms + t;
          s.layer[k][t] = d.h_seg_layer[i];
          s.w[k][t] = d.h_seg_w[i];
        }
      }
    } else if (d.layer_mode == HF_LAYER_PAPER3) {
      // N(l) = clip(pi - 4, pi, pi + 4) to [1, L_S], one segment each.
      const int pi = proportional_depth(l + 1, d.L_s, d.L_r);
      const int offs[3] = {-4, 0, 4};
      s.n_seg = 3;
      for (int k = 0; k < 3; ++k) {
        int t = pi + offs[k];
        t = t < 1 ? 1 : (t > d.L_s ? d.L_s : t);
        s.n_terms[k] = 1;
        s.layer[k][0] = t - 1;
        s.w[k][0] = 1.0f;
      }
    } else {
      // p = l (L_S - 1)/(L_R - 1); blend floor(p) and floor(p)+1 by (1-f, f).
      const double p = d.L_r > 1 ? (double)(l * (d.L_s - 1)) / (double)(d.L_r - 1) : 0.0;
      const int i0 = static_cast<int>(std::floor(p));
      const double f = p - i0;
      s.n_seg = 1;
      s.layer[0][0] = i0;
      s.w[0][0] = static_cast<float>(1.0 - f);
      s.n_terms[0] = 1;
      if (f > 0.0) {
        s.n_terms[0] = 2;
        s.layer[0][1] = i0 + 1 < d.L_s ? i0 + 1 : d.L_s - 1;
        s.w[0][1] = static_cast<float>(f);
      }
    }
    out[l] = s;
  }
}

hf_status validate(const hf_plan_desc* d) {
  auto bad = [](const char* m) {
    set_error(std::string("hf_plan_create: ") + m);
    return HF_ERR_INVALID_ARGUMENT;
  };
  auto unsup = [](const char* m) {
    set_error(std::string("hf_plan_create: unsupported: ") + m);
    return HF_ERR_UNSUPPORTED;
  };
  if (!d) return bad("null descriptor");
  if (d->L_s < 1 || d->H_s < 1 || d->D_s < 1 || d->L_r < 1 || d->H_r < 1 || d->D_r < 1)
    return bad("shapes must be positive");
  if (d->dtype != HF_BF16 && d->dtype != HF_F32) return bad("unknown dtype");
  if (d->layer_mode != HF_LAYER_PAPER3 && d->layer_mode != HF_LAYER_INTERP &&
      d->layer_mode != HF_LAYER_EXPLICIT)
    return bad("unknown layer mode");
  if (d->layer_mode == HF_LAYER_EXPLICIT) {
    if (d->n_seg < 1 || d->n_seg > kMaxSeg) return bad("explicit layer table: n_seg must be 1..8");
    if (d->n_terms < 1 || d->n_terms > kMaxTerms)
      return bad("explicit layer table: n_terms must be 1..2");
    if (!d->h_seg_layer || !d->h_seg_w) return bad("explicit layer table: null arrays");
    const size_t n = (size_t)d->L_r * d->n_seg * d->n_terms;
    for (size_t i = 0; i < n; ++i) {
      if (d->h_seg_layer[i] < 0 || d->h_seg_layer[i] >= d->L_s)
        return bad("explicit layer table: sender layer out of range");
      if (!std::isfinite(d->h_seg_w[i])) return bad("explicit layer table: weight not finite");
    }
  }
  if (d->align_mode != HF_ALIGN_TA && d->align_mode != HF_ALIGN_OVERLAP_MEAN &&
      d->align_mode != HF_ALIGN_SAME_INDEX)
    return bad("unknown align mode");
  if (d->n_req < 1 || d->n_req > kMaxReq) return bad("n_req must be in [1, 1024]");
  if (!d->s_tok_ptr || !d->r_tok_ptr) return bad("null token pointers");
  if (d->s_tok_ptr[0] != 0 || d->r_tok_ptr[0] != 0) return bad("token pointers must start at 0");
  for (int q = 0; q < d->n_req; ++q) {
    if (d->s_tok_ptr[q + 1] < d->s_tok_ptr[q] || d->r_tok_ptr[q + 1] < d->r_tok_ptr[q])
      return bad("token pointers must be non-decreasing");
    if (d->r_tok_ptr[q + 1] > d->r_tok_ptr[q] && d->s_tok_ptr[q + 1] == d->s_tok_ptr[q])
      return bad("a request has receiver tokens but no sender token");
  }
  if (!d->d_row_ptr || !d->d_W || !d->d_b || !d->h_r) return bad("null CSR or map pointer");
  if (d->r_tok_ptr[d->n_req] > 0 && (!d->d_col || !d->d_w)) return bad("null CSR arrays");
  for (int i = 0; i < 2 * d->L_r; ++i)
    if (!(d->h_r[i] > 0.0f) || !std::isfinite(d->h_r[i])) return bad("r must be positive");
  if (d->L_r > kMaxLayersR) return unsup("more than 128 receiver layers");
  const int esize = d->dtype == HF_BF16 ? 2 : 4;
  const int bke = 128 / esize;  // elements per 128-byte k-block
  const int d_s = d->H_s * d->D_s, d_r = d->H_r * d->D_r;
  if (d_s % bke) return unsup("d_S must be a multiple of 64 (bf16) or 32 (fp32)");
  if (d_r % 128) return unsup("d_R must be a multiple of 128");
  if (d->D_r % 32 || d->D_r > kMaxHeadDim) return unsup("D_r must be a multiple of 32, <= 256");
  const int BN = (d_r % 256 == 0) ? 256 : 128;
  if (BN % d->D_r) return unsup("a receiver head must fit one 128/256-column tile");
  if (d->h_inv_freq_r)
    for (int i = 0; i < d->D_r / 2; ++i)
      if (!std::isfinite(d->h_inv_freq_r[i])) return bad("h_inv_freq_r not finite");
  if (d->sender_k_rotated) {
    if (d->sender_k_rotated != 1) return bad("sender_k_rotated must be 0 or 1");
    if (!d->h_inv_freq_s && !(d->theta_s > 0.0))
      return bad("sender_k_rotated needs theta_s > 0 or h_inv_freq_s");
    if (d->h_inv_freq_s)
      for (int i = 0; i < d->D_s / 2; ++i)
        if (!std::isfinite(d->h_inv_freq_s[i])) return bad("h_inv_freq_s not finite");
    if (d->D_s > kMaxHeadDim) return unsup("sender_k_rotated: D_s above 256");
    const int chunk = 16 / esize;  // elements per 16-byte chunk
    if (d->D_s % 2 || (d->D_s / 2) % chunk || (2 * bke) % d->D_s || d_s % (2 * bke))
      return unsup("sender_k_rotated: D_s/2 must be a multiple of 8 (bf16) or 4 (fp32), D_s must "
                   "divide 128 (bf16) or 64 (fp32), d_S a multiple of 128 (bf16) or 64 (fp32)");
  }
  if (d->round_built_operands != 0 && d->round_built_operands != 1)
    return bad("round_built_operands must be 0 or 1");
  if (d->pool_before_map != 0 && d->pool_before_map != 1)
    return bad("pool_before_map must be 0 or 1");
  if (d->paged) {
    if (d->block_size < 1 || d->n_blocks < 1 || d->max_blocks_per_req < 1 || !d->d_block_table)
      return bad("paged layout needs block_size, n_blocks, max_blocks_per_req, d_block_table");
  }
  const int64_t T_s = d->s_tok_ptr[d->n_req];
  if (d->sender_rows < 0) return bad("sender_rows must be >= 0");
  const int64_t s_rows = d->sender_rows > 0 ? d->sender_rows : T_s;
  if (d->s_row0) {
    for (int q = 0; q < d->n_req; ++q) {
      const int64_t n_q = d->s_tok_ptr[q + 1] - d->s_tok_ptr[q];
      if (d->s_row0[q] < 0 || d->s_row0[q] + n_q > s_rows)
        return bad("a message span lies outside the sender cache (s_row0, sender_rows)");
    }
  } else if (s_rows < T_s) {
    return bad("sender_rows is smaller than the aligned sender tokens");
  }
  const long long rows = (long long)d->L_s * 2 * s_rows;
  if (rows >= (1LL << 31)) return unsup("sender cache has more than 2^31 rows");
  return HF_OK;
}

}  // namespace

hf_status launch_plan_kernels(hf_plan_s* p, const PlanTables& tables, cudaStream_t stream) {
  const PlanDev d = plan_dev(p);
  plan_init_kernel<<<1, 256, 0, stream>>>(tables.c, d);
  plan_segs_kernel<<<1, 128, 0, stream>>>(tables.s, d.segs);
  HF_CUDA_TRY(cudaGetLastError(), "plan init launch");
  if (p->T_r == 0) return HF_OK;
  RowArgs a;
  a.d = d;
  a.row_ptr = p->desc.d_row_ptr;
  a.col = p->desc.d_col;
  a.w = p->desc.d_w;
  a.block_table = p->desc.d_block_table;
  a.T_r = p->T_r;
  a.T_s = p->T_s;
  a.n_req = p->desc.n_req;
  a.paged = p->desc.paged;
  a.block_size = p->desc.block_size > 0 ? p->desc.block_size : 1;
  a.n_blocks = p->desc.n_blocks;
  a.max_blocks = p->desc.max_blocks_per_req;
  a.single_entry = p->desc.align_mode != HF_ALIGN_OVERLAP_MEAN;
  a.span = p->span ? 1 : 0;
  a.pam = p->pam ? 1 : 0;
  const int64_t want = (p->T_r + 255) / 256;
  const int grid = static_cast<int>(std::min<int64_t>(want, 8LL * device_sm_count()));
  plan_rows_kernel<<<grid, 256, 0, stream>>>(a);
  scan_inplace_kernel<ScanSum><<<1, kScanThreads, 0, stream>>>(d.new_flag, p->T_r, nullptr);
  if ((p->unrot || p->span) && p->T_s > 0) {
    const int64_t want_s = (p->T_s + 255) / 256;
    const int grid_s = static_cast<int>(std::min<int64_t>(want_s, 8LL * device_sm_count()));
    plan_sender_kernel<<<grid_s, 256, 0, stream>>>(d, p->T_s, p->desc.n_req, p->unrot ? 1 : 0,
                                                   p->span ? 1 : 0);
  }
  plan_runs_kernel<<<grid, 256, 0, stream>>>(a);
  if (p->pam) {
    scan_inplace_kernel<ScanMax><<<1, kScanThreads, 0, stream>>>(d.row_key, p->T_r, nullptr);
    const int64_t n_w = std::max<int64_t>(p->T_r, p->T_s + 2);
    const int grid_w = static_cast<int>(
        std::min<int64_t>((n_w + 255) / 256, 8LL * device_sm_count()));
    plan_windows_kernel<<<grid_w, 256, 0, stream>>>(a);
  }
  HF_CUDA_TRY(cudaGetLastError(), "plan kernels launch");
  return HF_OK;
}

}  // namespace hf

using namespace hf;

extern "C" hf_status hf_plan_workspace_size(const hf_plan_desc* desc, size_t* bytes) {
  if (!desc || !bytes || !desc->r_tok_ptr || !desc->s_tok_ptr || desc->n_req < 1 ||
      desc->n_req > kMaxReq) {
    set_error("hf_plan_workspace_size: invalid descriptor");
    return HF_ERR_INVALID_ARGUMENT;
  }
  *bytes = workspace_layout(*desc).total;
  return HF_OK;
}

namespace hf {

// Validates `desc`, fills `p` and `t`, and launches the plan kernels into
// the given workspace.  `p` and `t` belong to the caller.
hf_status plan_build(const hf_plan_desc* desc, void* d_workspace, size_t workspace_bytes,
                     cudaStream_t stream, hf_plan_s* p, PlanTables* t) {
  const hf_status v = validate(desc);
  if (v != HF_OK) return v;
  const WorkspaceLayout lay = workspace_layout(*desc);
  if (!d_workspace || workspace_bytes < lay.total ||
      (reinterpret_cast<uintptr_t>(d_workspace) & 255u)) {
    set_error("hf_plan_create: workspace missing, too small or not 256-byte aligned");
    return HF_ERR_WORKSPACE;
  }
  p->desc = *desc;
  p->d_s = desc->H_s * desc->D_s;
  p->d_r = desc->H_r * desc->D_r;
  p->n_seg = desc->layer_mode == HF_LAYER_PAPER3 ? 3
             : desc->layer_mode == HF_LAYER_EXPLICIT ? desc->n_seg : 1;
  p->K = p->n_seg * p->d_s;
  p->T_s = desc->s_tok_ptr[desc->n_req];
  p->span = desc->s_row0 != nullptr;
  p->s_rows = desc->sender_rows > 0 ? desc->sender_rows : p->T_s;
  p->T_r = desc->r_tok_ptr[desc->n_req];
  p->BN = (p->d_r % 256 == 0) ? 256 : 128;
  p->groups = ((p->BN / 2) % desc->D_r == 0) ? 2 : 1;
  // The copy-only operand path needs every segment to be one sender layer
  // with weight 1, one-entry rows and no rotation.
  bool one_layer_segments = desc->layer_mode == HF_LAYER_PAPER3;
  if (desc->layer_mode == HF_LAYER_EXPLICIT && desc->n_terms == 1) {
    one_layer_segments = true;
    for (int i = 0; i < desc->L_r * desc->n_seg; ++i)
      if (desc->h_seg_w[i] != 1.0f) one_layer_segments = false;
  }
  p->unrot = desc->sender_k_rotated == 1;
  p->rope = desc->theta_r > 0.0 || desc->h_inv_freq_r != nullptr;
  // overlap mean pooling commutes with the map (it is linear): unless the
  // pooled row itself is needed (key norm, sender keys rotated back per
  // position) or the caller asks otherwise, the map input rows are sender
  // rows and the epilogue pools the mapped rows
  p->pam = desc->align_mode == HF_ALIGN_OVERLAP_MEAN && desc->pool_before_map == 0 &&
           !p->unrot && desc->d_knorm_w == nullptr;
  const bool one_entry = desc->align_mode != HF_ALIGN_OVERLAP_MEAN || p->pam;
  p->gather = one_layer_segments && one_entry && !p->unrot;
  p->split = !p->gather && desc->dtype == HF_BF16 && desc->round_built_operands == 0;
  // one-entry rows (Token Alignment, same-index, sender rows of pooling
  // after the map) have at most two (term, entry) pairs per segment, both
  // staged by cp.async; pooled rows have more, whose direct loads stall the
  // warp anyway (measured slower staged)
  p->staged = p->split && !p->unrot && one_entry;
  // built operand rows bound their paths: a tile covering two 256-column
  // blocks (both TMEM accumulators) builds each A stage once for both
  p->wide = !p->gather && p->d_r % 512 == 0;
  p->ws = static_cast<char*>(d_workspace);
  p->ws_bytes = workspace_bytes;
  p->lay = lay;
  // host arrays are not kept
  p->desc.s_tok_ptr = nullptr;
  p->desc.r_tok_ptr = nullptr;
  p->desc.r_pos0 = nullptr;
  p->desc.h_r = nullptr;
  p->desc.h_inv_freq_r = nullptr;
  p->desc.h_inv_freq_s = nullptr;
  p->desc.s_pos0 = nullptr;
  p->desc.s_row0 = nullptr;
  p->desc.h_seg_layer = nullptr;
  p->desc.h_seg_w = nullptr;

  std::memset(t, 0, sizeof(*t));
  PlanConsts* c = &t->c;
  c->L_r = desc->L_r;
  c->D_r = desc->D_r;
  c->D_s = p->unrot ? desc->D_s : 0;
  c->n_req = desc->n_req;
  t->s.L_r = desc->L_r;
  build_layer_table(*desc, t->s.segs);
  for (int l = 0; l < desc->L_r; ++l) {
    const LayerSegs& sg = t->s.segs[l];
    int mx = 0;
    for (int k = 0; k < sg.n_seg; ++k)
      for (int i = 0; i < sg.n_terms[k]; ++i) mx = std::max(mx, sg.layer[k][i]);
    p->max_sender_layer[l] = mx;
  }
  for (int i = 0; i < 2 * desc->L_r; ++i) c->inv_r[i] = static_cast<float>(1.0 / desc->h_r[i]);
  // inv_freq_i = fp32(theta^(-2i/D)) evaluated in double precision
  // (or the caller's table)
  for (int i = 0; i < desc->D_r / 2; ++i)
    c->inv_freq[i] = desc->h_inv_freq_r ? desc->h_inv_freq_r[i]
                     : desc->theta_r > 0.0
                         ? static_cast<float>(std::pow(desc->theta_r, -(2.0 * i) / desc->D_r))
                         : 0.0f;
  if (p->unrot)
    for (int i = 0; i < desc->D_s / 2; ++i)
      c->inv_freq_s[i] = desc->h_inv_freq_s
                             ? desc->h_inv_freq_s[i]
                             : static_cast<float>(std::pow(desc->theta_s, -(2.0 * i) / desc->D_s));
  for (int q = 0; q <= desc->n_req; ++q) c->r_tok_ptr[q] = desc->r_tok_ptr[q];
  for (int q = 0; q < desc->n_req; ++q) c->r_pos0[q] = desc->r_pos0 ? desc->r_pos0[q] : 0;
  for (int q = 0; q <= desc->n_req; ++q) c->s_tok_ptr[q] = desc->s_tok_ptr[q];
  for (int q = 0; q < desc->n_req; ++q) c->s_pos0[q] = desc->s_pos0 ? desc->s_pos0[q] : 0;
  for (int q = 0; q < desc->n_req; ++q) c->s_row0[q] = desc->s_row0 ? desc->s_row0[q] : 0;
  return launch_plan_kernels(p, *t, stream);
}

}  // namespace hf

extern "C" hf_status hf_plan_create(const hf_plan_desc* desc, void* d_workspace,
                                    size_t workspace_bytes, hf_stream_t stream_, hf_plan* out) {
  if (!out) {
    set_error("hf_plan_create: null output handle");
    return HF_ERR_INVALID_ARGUMENT;
  }
  *out = nullptr;
  hf_plan_s* p = new hf_plan_s();
  PlanTables* t = new PlanTables();
  const hf_status s = plan_build(desc, d_workspace, workspace_bytes,
                                 reinterpret_cast<cudaStream_t>(stream_), p, t);
  delete t;
  if (s != HF_OK) {
    delete p;
    return s;
  }
  *out = p;
  return HF_OK;
}

extern "C" hf_status hf_plan_destroy(hf_plan plan) {
  if (plan && (plan->s_h2d || plan->events)) {
    int cur = 0;
    cudaGetDevice(&cur);
    cudaSetDevice(plan->aux_device);
    if (plan->s_h2d) cudaStreamDestroy(plan->s_h2d);
    if (plan->s_d2h) cudaStreamDestroy(plan->s_d2h);
    for (int i = 0; i < plan->n_events; ++i) cudaEventDestroy(plan->events[i]);
    delete[] plan->events;
    cudaSetDevice(cur);
  }
  delete plan;
  return HF_OK;
}

static hf_status read_word(hf_plan plan, hf_stream_t stream_, size_t off, int32_t* outv) {
  if (!plan || !outv) {
    set_error("null plan or output");
    return HF_ERR_INVALID_ARGUMENT;
  }
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  int32_t v = 0;
  HF_CUDA_TRY(cudaMemcpyAsync(&v, plan->ws + off, sizeof(v), cudaMemcpyDeviceToHost, stream),
              "read device word");
  HF_CUDA_TRY(cudaStreamSynchronize(stream), "stream synchronize");
  *outv = v;
  return HF_OK;
}

extern "C" hf_status hf_plan_device_status(hf_plan plan, hf_stream_t stream, int32_t* flags) {
  if (!plan) {
    set_error("null plan");
    return HF_ERR_INVALID_ARGUMENT;
  }
  const hf_status s = read_word(plan, stream, plan->lay.status, flags);
  if (s != HF_OK) return s;
  if (*flags != 0) {
    char buf[96];
    std::snprintf(buf, sizeof(buf), "device checks failed: status bits 0x%x", *flags);
    set_error(buf);
    return HF_ERR_DEVICE_CHECK;
  }
  return HF_OK;
}

extern "C" hf_status hf_plan_distinct_rows(hf_plan plan, hf_stream_t stream, int32_t* n_rows) {
  if (!plan) {
    set_error("null plan");
    return HF_ERR_INVALID_ARGUMENT;
  }
  return read_word(plan, stream, plan->lay.n_distinct, n_rows);
}

extern "C" const char* hf_status_string(hf_status s) {
  switch (s) {
    case HF_OK: return "ok";
    case HF_ERR_INVALID_ARGUMENT: return "invalid argument";
    case HF_ERR_UNSUPPORTED: return "unsupported";
    case HF_ERR_CUDA: return "CUDA error";
    case HF_ERR_DEVICE_CHECK: return "device check failed";
    case HF_ERR_WORKSPACE: return "bad workspace";
  }
  return "unknown status";
}

extern "C" const char* hf_last_error(void) { return g_last_error.c_str(); }
