// hf_recolor_fit: the Recolor initialisation of one map (Section 3.2,
// Eq. 3-5) on the GPU, from weighted aligned sample pairs (X, Y, w):
//   r = sqrt(sum w |x|^2 / (d_S sum w))                               (Eq. 3)
//   Z = X / r; weighted means and covariances of Z and Y
//   R* = polar factor of Sigma_Z^{-1/2} Sigma_ZY Sigma_Y^{-1/2}      (Eq. 4)
//   A = Sigma_Z^{-1/2} R* Sigma_Y^{1/2},  b = mu_Y - mu_Z A           (Eq. 5)
// Matrix square roots and the polar factor use Newton-Schulz iterations, so
// every step is a matrix product or an elementwise pass: the coupled
// iteration T = (3I - Z Y) / 2, Y <- Y T, Z <- T Z turns Y_0 = S / c,
// Z_0 = I into (S / c)^{1/2} and (S / c)^{-1/2}; X <- X (3I - X^T X) / 2
// turns X_0 = M / |M|_F into the orthogonal polar factor U Q^T of
// M = U Lambda Q^T (full column rank), which is the R* of Eq. 4.
// Offline (once per map, before folding).  The products are fp32 GEMMs on
// this library's tcgen05 kernel (hf_gemm.cu: each operand split exactly into
// three bf16 parts, six partial products in an fp32 accumulator: fp32
// accuracy); the statistics, centring and elementwise passes are this file's
// kernels.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <utility>

#include <cuda_bf16.h>

#include "hf_internal.h"

namespace hf {
namespace {

// The moments' products run over the samples in chunks of this many, so the
// bf16 planes of their operands stay a bounded part of the workspace.
constexpr int64_t kMomentChunk = 8192;
// Split-K partials: room for every SM pair's 256 x 256 tile twice over.
constexpr size_t kPartialBytes = static_cast<size_t>(2) * 96 * 65536 * sizeof(float);

hf_status sgemm(const GemmWork& h, cudaStream_t s, int M, int N, int K, float alpha,
                const float* A, int64_t a_i, int64_t a_k, const float* B, int64_t b_k,
                int64_t b_j, float beta, float* C, int64_t ldc, const float* Cin = nullptr,
                float diag = 0.f) {
  return gemm_f32(s, h, M, N, K, alpha, A, a_i, a_k, B, b_k, b_j, beta, C, ldc, Cin, diag);
}

// A product over the sample axis (K = N samples) in chunks of kMomentChunk:
// C = alpha sum_chunks op(A_c) op(B_c).
hf_status moment_product(const GemmWork& h, cudaStream_t s, int M, int N, int64_t K,
                         const float* A, int64_t a_i, int64_t a_k, const float* B, int64_t b_k,
                         int64_t b_j, float* C, int64_t ldc) {
  for (int64_t k0 = 0; k0 < K; k0 += kMomentChunk) {
    const int kc = static_cast<int>(std::min<int64_t>(kMomentChunk, K - k0));
    const hf_status st = sgemm(h, s, M, N, kc, 1.f, A + k0 * a_k, a_i, a_k, B + k0 * b_k, b_k,
                               b_j, k0 == 0 ? 0.f : 1.f, C, ldc);
    if (st != HF_OK) return st;
  }
  return HF_OK;
}

__device__ __forceinline__ float ld(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ float ld(const float* p) { return *p; }

// Column sums of w X and w Y, sum w, and sum w |x|^2.  A thread sums its
// column over the block's rows (at most a few hundred) in fp32; the partial
// sums meet in fp64 (GB300's fp64 rate is a small fraction of fp32's).
template <typename T>
__global__ void rc_stats_kernel(const T* X, const T* Y, const float* w, int64_t N, int dx,
                                int dy, double* sx, double* sy, double* sw_ss) {
  const int d = dx + dy;
  const int col = blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t rows = (N + gridDim.y - 1) / gridDim.y;
  const int64_t n0 = blockIdx.y * rows, n1 = min(N, n0 + rows);
  float s = 0.f, ssq = 0.f, swt = 0.f;
  if (col < d) {
    for (int64_t n = n0; n < n1; ++n) {
      const float wn = w[n];
      const float v = col < dx ? ld(X + n * dx + col) : ld(Y + n * dy + (col - dx));
      const float wv = wn * v;
      s += wv;
      if (col < dx) ssq = fmaf(wv, v, ssq);
      if (col == 0) swt += wn;
    }
    atomicAdd(col < dx ? sx + col : sy + (col - dx), static_cast<double>(s));
    if (col == 0) atomicAdd(sw_ss, static_cast<double>(swt));
  }
  // the shared sum of squares: every lane of the warp takes part (lanes
  // past the columns hold 0), one fp64 atomic per warp
  double q = ssq;
  for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  if ((threadIdx.x & 31) == 0 && q != 0.0) atomicAdd(sw_ss + 1, q);
}

// fp32 means mu_x (of X, not yet divided by r), mu_y, and [1 / W, 1 / r].
__global__ void rc_mean_kernel(const double* sx, const double* sy, const double* sw_ss, int dx,
                               int dy, float* mu, float* scal) {
  const double W = sw_ss[0];
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < dx + dy; c += gridDim.x * blockDim.x)
    mu[c] = static_cast<float>((c < dx ? sx[c] : sy[c - dx]) / W);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    scal[0] = static_cast<float>(1.0 / W);
    scal[1] = static_cast<float>(1.0 / sqrt(sw_ss[1] / (static_cast<double>(dx) * W)));
  }
}

// Xc = sqrt(w / W) (x - mu_x) / r and Yc = sqrt(w / W) (y - mu_y), fp32.
template <typename T>
__global__ void rc_center_kernel(const T* X, const T* Y, const float* w, int64_t N, int dx,
                                 int dy, const float* mu, const float* scal, float* Xc,
                                 float* Yc) {
  const int d = dx + dy;
  const float inv_w = scal[0], inv_r = scal[1];
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < N * d;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t n = i / d;
    const int c = static_cast<int>(i - n * d);
    const float sc = sqrtf(w[n] * inv_w);
    if (c < dx)
      Xc[n * dx + c] = sc * (ld(X + n * dx + c) - mu[c]) * inv_r;
    else
      Yc[n * dy + (c - dx)] = sc * (ld(Y + n * dy + (c - dx)) - mu[c]);
  }
}

// S += reg * trace(S) / d * I  (one block of 256 threads).
__global__ void rc_ridge_kernel(float* S, int d, float reg) {
  __shared__ double part[256];
  double t = 0.0;
  for (int i = threadIdx.x; i < d; i += blockDim.x) t += S[static_cast<int64_t>(i) * d + i];
  part[threadIdx.x] = t;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if (threadIdx.x < o) part[threadIdx.x] += part[threadIdx.x + o];
    __syncthreads();
  }
  const float add = reg * static_cast<float>(part[0] / d);
  for (int i = threadIdx.x; i < d; i += blockDim.x) S[static_cast<int64_t>(i) * d + i] += add;
}

// *out = trace(S) (one block of 256 threads).
__global__ void rc_trace_kernel(const float* S, int d, double* out) {
  __shared__ double part[256];
  double t = 0.0;
  for (int i = threadIdx.x; i < d; i += blockDim.x) t += S[static_cast<int64_t>(i) * d + i];
  part[threadIdx.x] = t;
  __syncthreads();
  for (int o = blockDim.x / 2; o > 0; o >>= 1) {
    if (threadIdx.x < o) part[threadIdx.x] += part[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = part[0];
}

// out = a * in + b * I (square, or the leading square of a d x e matrix when
// only scaling: b = 0).
__global__ void rc_affine_kernel(float* out, const float* in, int64_t n_el, int cols, float a,
                                 float b) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_el;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / cols, c = i - r * cols;
    out[i] = a * (in ? in[i] : 0.f) + (r == c ? b : 0.f);
  }
}

// sum of squares of x, or of (x - I) when minus_identity: fp32 per thread
// (a few dozen elements each), fp64 across threads.
__global__ void rc_sumsq_kernel(const float* x, int64_t n_el, int cols, int minus_identity,
                                double* out) {
  float s = 0.f;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_el;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / cols, c = i - r * cols;
    const float v = x[i] - (minus_identity && r == c ? 1.f : 0.f);
    s = fmaf(v, v, s);
  }
  double q = s;
  for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  if ((threadIdx.x & 31) == 0) atomicAdd(out, q);
}

// W_out = A^T in the output type: 32 x 32 tiles through shared memory, read
// and written along rows.
template <typename T>
__global__ void rc_transpose_kernel(const float* A, int dx, int dy, T* W_out) {
  __shared__ float tile[32][33];
  const int k0 = blockIdx.y * 32, j0 = blockIdx.x * 32;
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int k = k0 + i, j = j0 + threadIdx.x;
    if (k < dx && j < dy) tile[i][threadIdx.x] = A[static_cast<int64_t>(k) * dy + j];
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int j = j0 + i, k = k0 + threadIdx.x;
    if (k < dx && j < dy) W_out[static_cast<int64_t>(j) * dx + k] = T(tile[threadIdx.x][i]);
  }
}

// b = mu_y - mu_z A, mu_z = mu_x / r.  Block (j-tile of 32 columns, slice of
// 256 rows of A): thread (j, sub) sums 32 rows in fp64, the block combines its
// eight partial sums and adds them to bacc[j] (cleared before).
__global__ void rc_bias_partial_kernel(const float* A, int dx, int dy, const double* sx,
                                       const double* sw_ss, double* bacc) {
  __shared__ double part[8][33];
  const double W = sw_ss[0];
  const double inv = 1.0 / (W * sqrt(sw_ss[1] / (static_cast<double>(dx) * W)));
  const int j = blockIdx.x * 32 + threadIdx.x;
  const int kbase = blockIdx.y * 256 + threadIdx.y * 32;
  double s = 0.0;
  if (j < dy)
    for (int k = kbase; k < min(dx, kbase + 32); ++k)
      s = fma(sx[k] * inv, static_cast<double>(A[static_cast<int64_t>(k) * dy + j]), s);
  part[threadIdx.y][threadIdx.x] = s;
  __syncthreads();
  if (threadIdx.y == 0 && j < dy) {
    double t = 0.0;
    for (int q = 0; q < 8; ++q) t += part[q][threadIdx.x];
    atomicAdd(bacc + j, t);
  }
}

__global__ void rc_bias_final_kernel(const double* sy, const double* sw_ss, const double* bacc,
                                     int dy, float* b_out) {
  const double W = sw_ss[0];
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < dy; j += gridDim.x * blockDim.x)
    b_out[j] = static_cast<float>(sy[j] / W - bacc[j]);
}

struct Rc {
  size_t stats, bacc, mu, xc, yc, sz, sy, szy, p1, p2, p3, p4, sz_ih, sy_ih, sy_h, m, x1, x2, xtx, a,
      planes_a, planes_b, partial, err, total;
  size_t planes_bytes;
};

Rc rc_layout(int64_t N, int dx, int dy) {
  Rc L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = (off + bytes + 255) / 256 * 256;
    return at;
  };
  const size_t f = sizeof(float);
  const size_t dmax = static_cast<size_t>(dx > dy ? dx : dy);
  L.stats = take(sizeof(double) * (dx + dy + 4));
  L.bacc = take(sizeof(double) * dy);
  L.mu = take(f * (dx + dy + 2));
  L.xc = take(f * N * dx);
  L.yc = take(f * N * dy);
  L.sz = take(f * dx * dx);
  L.sy = take(f * dy * dy);
  L.szy = take(f * dx * dy);
  L.p1 = take(f * dmax * dmax);
  L.p2 = take(f * dmax * dmax);
  L.p3 = take(f * dmax * dmax);
  L.p4 = take(f * dmax * dmax);
  L.sz_ih = take(f * dx * dx);
  L.sy_ih = take(f * dy * dy);
  L.sy_h = take(f * dy * dy);
  L.m = take(f * dx * dy);
  L.x1 = take(f * dx * dy);
  L.x2 = take(f * dx * dy);
  L.xtx = take(f * dy * dy);
  L.a = take(f * dx * dy);
  // bf16 planes of the products' operands: rows up to max(d_S, d_R), K up
  // to max(d_S, one chunk of samples)
  const int64_t kmax = std::max<int64_t>(dx, std::min<int64_t>(N, kMomentChunk));
  L.planes_bytes = gemm_planes_bytes(static_cast<int64_t>(dmax), kmax);
  L.planes_a = take(L.planes_bytes);
  L.planes_b = take(L.planes_bytes);
  L.partial = take(kPartialBytes);
  L.err = take(sizeof(int32_t));
  L.total = off;
  return L;
}

hf_status read_double(cudaStream_t s, const double* d, double* h) {
  HF_CUDA_TRY(cudaMemcpyAsync(h, d, sizeof(double), cudaMemcpyDeviceToHost, s), "read back");
  HF_CUDA_TRY(cudaStreamSynchronize(s), "synchronize");
  return HF_OK;
}

constexpr int kMaxIter = 80;
constexpr double kTol = 2e-5;  // |X - I|_F / sqrt(d) at convergence

// Convergence test of an iteration's residual e (checked every 4 steps):
// below the tolerance, or no longer falling once small (the fp32 floor).
bool converged(double e, double* prev) {
  const bool done = e < kTol || (e < 1e-3 && e >= 0.5 * *prev);
  *prev = e;
  return done;
}

// Newton-Schulz square root and inverse square root of the SPD matrix S
// (d x d): root = S^{1/2} (when root is not null), inv_root = S^{-1/2}; Y, Z, T, U
// are d x d work buffers distinct from both.
// The coupled iteration Y <- Y T, Z <- T Z, T = (3I - Z Y) / 2 acts on each
// eigenvalue x^2 of Z Y (x the corresponding eigenvalue of (S/c)^{1/2}
// polynomials) as the cubic sign iteration x <- x (3 - x^2) / 2, which
// lifts small x by only 1.5 per step.  With a lower bound l <= x <= 1 (the
// ridge reg * trace / d bounds the smallest eigenvalue of S from below),
// each step first scales Y and Z by b = sqrt(3 / (l^2 + l + 1)), the factor
// for which the cubic maps [b l, b] onto [p(b l), 1] with p(b l) = p(b)
// (the scaled Newton-Schulz step that maximises the new lower bound): small
// x then grow by ~2.6 per step, and b -> 1 as l -> 1.  Scaling Y and Z
// together keeps Y = (S/c) Z, so the limits are unchanged.  With reg = 0
// there is no bound and the plain iteration runs.
hf_status ns_sqrt(cudaStream_t s, const GemmWork& h, const float* S, int d, float reg, float* Y, float* Z, float* T, float* U,
                  float* root, float* inv_root, double* dscr, int* iters) {
  const int64_t n_el = static_cast<int64_t>(d) * d;
  const int grid = 1024;
  double c2 = 0.0;
  HF_CUDA_TRY(cudaMemsetAsync(dscr, 0, sizeof(double), s), "clear");
  rc_sumsq_kernel<<<grid, 256, 0, s>>>(S, n_el, d, 0, dscr);
  hf_status st = read_double(s, dscr, &c2);
  if (st != HF_OK) return st;
  const double c = sqrt(c2);
  if (!(c > 0.0)) {
    set_error("hf_recolor_fit: a covariance is zero");
    return HF_ERR_INVALID_ARGUMENT;
  }
  double l = 0.0;  // lower bound of the eigenvalues x of (Z Y)^{1/2}
  if (reg > 0.f) {
    rc_trace_kernel<<<1, 256, 0, s>>>(S, d, dscr);
    double tr = 0.0;
    if ((st = read_double(s, dscr, &tr)) != HF_OK) return st;
    // S = S0 + reg tr(S0)/d I with S0 >= 0 and tr(S) = (1 + reg) tr(S0)
    const double lam_lo = reg * tr / (static_cast<double>(d) * (1.0 + reg));
    if (lam_lo > 0.0) l = std::min(1.0, sqrt(lam_lo / c));
  }
  rc_affine_kernel<<<grid, 256, 0, s>>>(Y, S, n_el, d, static_cast<float>(1.0 / c), 0.f);
  rc_affine_kernel<<<grid, 256, 0, s>>>(Z, nullptr, n_el, d, 0.f, 1.f);
  int it = 0;
  double prev = 1e30;
  for (; it < kMaxIter; ++it) {
    const double b = l > 0.0 ? sqrt(3.0 / (l * l + l + 1.0)) : 1.0;
    // T = 1.5 I - 0.5 b^2 Z Y
    if ((st = sgemm(h, s, d, d, d, static_cast<float>(-0.5 * b * b), Z, d, 1, Y, d, 1, 0.f, T,
                    d, nullptr, 1.5f)) != HF_OK)
      return st;
    // the residual |I - Z Y| = 2 |T - I| holds for unscaled steps
    if (it % 4 == 3 && b < 1.0 + 1e-6) {
      double e2 = 0.0;
      HF_CUDA_TRY(cudaMemsetAsync(dscr, 0, sizeof(double), s), "clear");
      // |I - Z Y| = 2 |T - I|
      rc_sumsq_kernel<<<grid, 256, 0, s>>>(T, n_el, d, 1, dscr);
      if ((st = read_double(s, dscr, &e2)) != HF_OK) return st;
      if (converged(2.0 * sqrt(e2 / d), &prev)) break;
    }
    const float bf = static_cast<float>(b);
    if ((st = sgemm(h, s, d, d, d, bf, Y, d, 1, T, d, 1, 0.f, U, d)) != HF_OK) return st;  // b Y T
    std::swap(Y, U);
    if ((st = sgemm(h, s, d, d, d, bf, T, d, 1, Z, d, 1, 0.f, U, d)) != HF_OK) return st;  // b T Z
    std::swap(Z, U);
    l = std::min(1.0, b * l * (3.0 - b * b * l * l) / 2.0);
  }
  *iters = it;
  // inv_root first: root may be null (not wanted), and neither may alias the
  // work buffers, which Y and Z rotate through
  rc_affine_kernel<<<grid, 256, 0, s>>>(inv_root, Z, n_el, d, static_cast<float>(1.0 / sqrt(c)),
                                        0.f);
  if (root)
    rc_affine_kernel<<<grid, 256, 0, s>>>(root, Y, n_el, d, static_cast<float>(sqrt(c)), 0.f);
  HF_CUDA_TRY(cudaGetLastError(), "hf_recolor_fit: iteration launch");
  return HF_OK;
}

// Orthogonal polar factor of M (dx x dy, dx >= dy, full column rank):
// X <- X (3I - X^T X) / 2 from X_0 = M / min(|M|_F, 1).  M is the whitened
// cross-covariance Sigma_Z^{-1/2} Sigma_ZY Sigma_Y^{-1/2} of one weighted
// sample set, so its singular values (canonical correlations; the ridges
// only lower them) are at most 1 (Cauchy-Schwarz), and the iteration needs
// no smaller scale: dividing by |M|_F = sqrt(sum of squared correlations)
// would only shrink them and add ~log_1.5 |M|_F steps.  Result in *out (one
// of the two buffers).
hf_status ns_polar(cudaStream_t s, const GemmWork& h, const float* M, int dx, int dy, float* X, float* X2,
                   float* P, double* dscr, float** out, int* iters) {
  const int64_t n_el = static_cast<int64_t>(dx) * dy, p_el = static_cast<int64_t>(dy) * dy;
  const int grid = 1024;
  double m2 = 0.0;
  HF_CUDA_TRY(cudaMemsetAsync(dscr, 0, sizeof(double), s), "clear");
  rc_sumsq_kernel<<<grid, 256, 0, s>>>(M, n_el, dy, 0, dscr);
  hf_status st = read_double(s, dscr, &m2);
  if (st != HF_OK) return st;
  if (!(m2 > 0.0)) {
    set_error("hf_recolor_fit: the cross-covariance is zero");
    return HF_ERR_INVALID_ARGUMENT;
  }
  rc_affine_kernel<<<grid, 256, 0, s>>>(X, M, n_el, dy,
                                        static_cast<float>(1.0 / std::min(sqrt(m2), 1.0)), 0.f);
  int it = 0;
  double prev = 1e30;
  for (; it < kMaxIter; ++it) {
    // P = X^T X
    if ((st = sgemm(h, s, dy, dy, dx, 1.f, X, 1, dy, X, dy, 1, 0.f, P, dy)) != HF_OK) return st;
    if (it % 4 == 3) {
      double e2 = 0.0;
      HF_CUDA_TRY(cudaMemsetAsync(dscr, 0, sizeof(double), s), "clear");
      rc_sumsq_kernel<<<grid, 256, 0, s>>>(P, p_el, dy, 1, dscr);
      if ((st = read_double(s, dscr, &e2)) != HF_OK) return st;
      if (converged(sqrt(e2 / dy), &prev)) break;
    }
    // X2 = 1.5 X - 0.5 X P
    if ((st = sgemm(h, s, dx, dy, dy, -0.5f, X, dy, 1, P, dy, 1, 1.5f, X2, dy, X)) != HF_OK)
      return st;
    std::swap(X, X2);
  }
  *iters = it;
  *out = X;
  HF_CUDA_TRY(cudaGetLastError(), "hf_recolor_fit: iteration launch");
  return HF_OK;
}

template <typename T>
hf_status recolor_typed(int64_t N, int dx, int dy, const void* Xv, const void* Yv, const float* w,
                        float reg, void* W_out, float* b_out, float* h_r, int32_t* h_iters,
                        char* ws, cudaStream_t s) {
  const Rc L = rc_layout(N, dx, dy);
  double* stats = reinterpret_cast<double*>(ws + L.stats);
  double* sx = stats;
  double* sy = sx + dx;
  double* sw_ss = sy + dy;    // [0] sum w, [1] sum w |x|^2
  double* dscr = sw_ss + 2;   // scratch scalar
  auto F = [&](size_t off) { return reinterpret_cast<float*>(ws + off); };
  const T* X = static_cast<const T*>(Xv);
  const T* Y = static_cast<const T*>(Yv);
  GemmWork h;
  h.planes_a = ws + L.planes_a;
  h.planes_b = ws + L.planes_b;
  h.planes_a_bytes = h.planes_b_bytes = L.planes_bytes;
  h.partial = F(L.partial);
  h.partial_bytes = kPartialBytes;
  h.err = reinterpret_cast<int32_t*>(ws + L.err);
  HF_CUDA_TRY(cudaMemsetAsync(h.err, 0, sizeof(int32_t), s), "clear");
  HF_CUDA_TRY(cudaMemsetAsync(stats, 0, sizeof(double) * (dx + dy + 4), s), "clear");
  const int d = dx + dy;
  // at most ~128 rows per thread, so the per-thread fp32 sums stay short
  dim3 sgrid((d + 255) / 256, static_cast<unsigned>(std::min<int64_t>((N + 127) / 128, 65535)));
  rc_stats_kernel<T><<<sgrid, 256, 0, s>>>(X, Y, w, N, dx, dy, sx, sy, sw_ss);
  float* mu = F(L.mu);
  rc_mean_kernel<<<(d + 255) / 256, 256, 0, s>>>(sx, sy, sw_ss, dx, dy, mu, mu + d);
  rc_center_kernel<T><<<2048, 256, 0, s>>>(X, Y, w, N, dx, dy, mu, mu + d, F(L.xc), F(L.yc));
  HF_CUDA_TRY(cudaGetLastError(), "hf_recolor_fit: moments launch");
  hf_status st;
  // Sigma_Z = Xc^T Xc, Sigma_Y = Yc^T Yc, Sigma_ZY = Xc^T Yc
  if ((st = moment_product(h, s, dx, dx, N, F(L.xc), 1, dx, F(L.xc), dx, 1, F(L.sz), dx)) != HF_OK)
    return st;
  if ((st = moment_product(h, s, dy, dy, N, F(L.yc), 1, dy, F(L.yc), dy, 1, F(L.sy), dy)) != HF_OK)
    return st;
  if ((st = moment_product(h, s, dx, dy, N, F(L.xc), 1, dx, F(L.yc), dy, 1, F(L.szy), dy)) != HF_OK)
    return st;
  if (reg > 0.f) {
    rc_ridge_kernel<<<1, 256, 0, s>>>(F(L.sz), dx, reg);
    rc_ridge_kernel<<<1, 256, 0, s>>>(F(L.sy), dy, reg);
  }
  int it1 = 0, it2 = 0, it3 = 0;
  if ((st = ns_sqrt(s, h, F(L.sz), dx, reg, F(L.p1), F(L.p2), F(L.p3), F(L.p4), nullptr,
                    F(L.sz_ih), dscr, &it1)) != HF_OK)
    return st;
  if ((st = ns_sqrt(s, h, F(L.sy), dy, reg, F(L.p1), F(L.p2), F(L.p3), F(L.p4), F(L.sy_h), F(L.sy_ih),
                    dscr, &it2)) != HF_OK)
    return st;
  // M = Sigma_Z^{-1/2} Sigma_ZY Sigma_Y^{-1/2}
  if ((st = sgemm(h, s, dx, dy, dx, 1.f, F(L.sz_ih), dx, 1, F(L.szy), dy, 1, 0.f, F(L.x2), dy)) != HF_OK)
    return st;
  if ((st = sgemm(h, s, dx, dy, dy, 1.f, F(L.x2), dy, 1, F(L.sy_ih), dy, 1, 0.f, F(L.m), dy)) != HF_OK)
    return st;
  float* R = nullptr;
  if ((st = ns_polar(s, h, F(L.m), dx, dy, F(L.x1), F(L.x2), F(L.xtx), dscr, &R, &it3)) != HF_OK)
    return st;
  // A = Sigma_Z^{-1/2} R* Sigma_Y^{1/2}
  float* tmp = R == F(L.x1) ? F(L.x2) : F(L.x1);
  if ((st = sgemm(h, s, dx, dy, dx, 1.f, F(L.sz_ih), dx, 1, R, dy, 1, 0.f, tmp, dy)) != HF_OK) return st;
  if ((st = sgemm(h, s, dx, dy, dy, 1.f, tmp, dy, 1, F(L.sy_h), dy, 1, 0.f, F(L.a), dy)) != HF_OK)
    return st;
  {
    double* bacc = reinterpret_cast<double*>(ws + L.bacc);
    HF_CUDA_TRY(cudaMemsetAsync(bacc, 0, sizeof(double) * dy, s), "clear");
    rc_transpose_kernel<T><<<dim3((dy + 31) / 32, (dx + 31) / 32), dim3(32, 8), 0, s>>>(
        F(L.a), dx, dy, static_cast<T*>(W_out));
    rc_bias_partial_kernel<<<dim3((dy + 31) / 32, (dx + 255) / 256), dim3(32, 8), 0, s>>>(
        F(L.a), dx, dy, sx, sw_ss, bacc);
    rc_bias_final_kernel<<<(dy + 255) / 256, 256, 0, s>>>(sy, sw_ss, bacc, dy, b_out);
  }
  HF_CUDA_TRY(cudaGetLastError(), "hf_recolor_fit: output launch");
  double hs[2];
  int32_t gemm_err = 0;
  HF_CUDA_TRY(cudaMemcpyAsync(hs, sw_ss, sizeof(hs), cudaMemcpyDeviceToHost, s), "read back");
  HF_CUDA_TRY(cudaMemcpyAsync(&gemm_err, h.err, sizeof(gemm_err), cudaMemcpyDeviceToHost, s),
              "read back");
  HF_CUDA_TRY(cudaStreamSynchronize(s), "synchronize");
  if (gemm_err != 0) {
    set_error("hf_recolor_fit: a product kernel's pipeline wait ran out (internal error)");
    return HF_ERR_DEVICE_CHECK;
  }
  if (h_r) *h_r = static_cast<float>(std::sqrt(hs[1] / (static_cast<double>(dx) * hs[0])));
  if (h_iters) {
    h_iters[0] = it1;
    h_iters[1] = it2;
    h_iters[2] = it3;
  }
  if (it1 >= kMaxIter || it2 >= kMaxIter || it3 >= kMaxIter) {
    set_error("hf_recolor_fit: an iteration did not converge (ill-conditioned covariances: "
              "raise reg)");
    return HF_ERR_DEVICE_CHECK;
  }
  return HF_OK;
}

}  // namespace
}  // namespace hf

using namespace hf;

extern "C" hf_status hf_recolor_workspace_size(int64_t N, int32_t d_S, int32_t d_R,
                                               size_t* bytes) {
  if (!bytes || N < 2 || d_S < 1 || d_R < 1 || d_S < d_R) {
    set_error("hf_recolor_workspace_size: need N >= 2 and d_S >= d_R >= 1");
    return HF_ERR_INVALID_ARGUMENT;
  }
  *bytes = rc_layout(N, d_S, d_R).total;
  return HF_OK;
}

extern "C" hf_status hf_recolor_fit(hf_dtype dtype, int64_t N, int32_t d_S, int32_t d_R,
                                    const void* d_X, const void* d_Y, const float* d_w, float reg,
                                    void* d_W_out, float* d_b_out, float* h_r_out,
                                    int32_t* h_iters_out, void* d_workspace,
                                    size_t workspace_bytes, hf_stream_t stream_) {
  if (dtype != HF_BF16 && dtype != HF_F32) {
    set_error("hf_recolor_fit: unknown dtype");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (N < 2 || d_S < 1 || d_R < 1 || d_S < d_R || N * static_cast<int64_t>(d_S) >= (1LL << 31)) {
    set_error("hf_recolor_fit: need N >= 2, d_S >= d_R >= 1 and N x d_S < 2^31");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (!d_X || !d_Y || !d_w || !d_W_out || !d_b_out || !(reg >= 0.f)) {
    set_error("hf_recolor_fit: null pointer or negative reg");
    return HF_ERR_INVALID_ARGUMENT;
  }
  if (!d_workspace || workspace_bytes < rc_layout(N, d_S, d_R).total ||
      (reinterpret_cast<uintptr_t>(d_workspace) & 255u)) {
    set_error("hf_recolor_fit: workspace missing, too small or not 256-byte aligned");
    return HF_ERR_WORKSPACE;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream_);
  char* ws = static_cast<char*>(d_workspace);
  if (dtype == HF_BF16)
    return recolor_typed<__nv_bfloat16>(N, d_S, d_R, d_X, d_Y, d_w, reg, d_W_out, d_b_out,
                                        h_r_out, h_iters_out, ws, s);
  return recolor_typed<float>(N, d_S, d_R, d_X, d_Y, d_w, reg, d_W_out, d_b_out, h_r_out,
                              h_iters_out, ws, s);
}
