/*
 * heterofold.h — C ABI of the GB300 (sm_103a) HeteroFold transfer library.
 *
 * HeteroFold (arxiv 2609.32259) turns a sender model's KV cache into a
 * receiver model's KV cache without receiver prefill.  At inference time it
 * applies, per receiver layer l and role c in {K, V}, one folded affine map
 * (Section 3.3 "Folding for inference", Eq. 9):
 *
 *     Phi_{l,c}(x_j) = (x_j / r_{l,c}) A_final_{l,c} + b_final_{l,c}
 *
 * to the concatenated features of three sender layers (Eq. 1-2) taken at
 * the sender token that Token Alignment pairs with receiver token j
 * (Section 3.1, Appendix B.1); the output is reshaped into the receiver's
 * KV heads, and keys get the receiver's key normalisation and RoPE at
 * receiver positions (Section 3 opening paragraph, Appendix B.1).
 *
 * Call sequence for one transfer:
 *   hf_align_build            character-end offsets -> alignment CSR (device)
 *   hf_plan_workspace_size    bytes of device workspace the plan needs
 *   hf_plan_create            validates, builds per-transfer metadata (device)
 *   hf_transfer               one kernel launch: receiver cache <- Phi(sender)
 *     (or hf_transfer_host    the same with both caches in host memory)
 *   hf_plan_destroy
 *
 * General rules:
 *  - Every pointer prefixed d_ is device memory; h_ or unprefixed arrays
 *    documented as "host" are host memory.  The library allocates no device
 *    memory: all device buffers belong to the caller, who keeps them alive
 *    and unchanged while work that uses them is in flight.
 *  - Every device-side function is asynchronous and stream-ordered on the
 *    given stream (NULL = the legacy default stream); none synchronises the
 *    host except hf_plan_device_status and hf_plan_distinct_rows.
 *  - Functions return an hf_status; HF_OK is 0.  On any other value
 *    hf_last_error() returns a message for the calling host thread.  Invalid
 *    arguments are caught on the host before any launch.
 *  - Data-dependent problems that only the device can see (unsorted
 *    offsets, out-of-range columns or blocks, a wait that timed out) set
 *    bits in a device status word; kernels skip the offending row or block
 *    and never trap.  hf_plan_device_status reads the word.
 *  - A plan may be used by one stream at a time.
 *  - Requires a GPU of compute capability 10.3 (GB300).
 */
#ifndef HETEROFOLD_H
#define HETEROFOLD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* hf_stream_t;

typedef enum {
  HF_OK = 0,
  HF_ERR_INVALID_ARGUMENT = 1, /* a host-visible argument is wrong; nothing launched */
  HF_ERR_UNSUPPORTED = 2,      /* valid but outside what the kernels handle */
  HF_ERR_CUDA = 3,             /* a CUDA runtime or driver call failed */
  HF_ERR_DEVICE_CHECK = 5,     /* the device status word has bits set */
  HF_ERR_WORKSPACE = 6         /* workspace too small or misaligned */
} hf_status;

/* Token alignment rules (rows of the alignment CSR). */
typedef enum {
  /* Token Alignment, Section 3.1 and Appendix B.1: one sender token per
     receiver token, weight 1: the sender token ending at the latest shared
     character-end boundary at or before the receiver token's end; the first
     sender token before the first shared boundary. */
  HF_ALIGN_TA = 0,
  /* Mean pooling over every sender token whose character span
     (end_{k-1}, end_k] overlaps the receiver token's span; weights are the
     fp32 rounding of 1/n. */
  HF_ALIGN_OVERLAP_MEAN = 1,
  /* Same-index pairing, Appendix A and B.1: a(j) = min(j, n_S), one-based. */
  HF_ALIGN_SAME_INDEX = 2
} hf_align_mode;

/* Layer alignment rules (map input segments per receiver layer). */
typedef enum {
  /* Eq. 1-2: three sender layers N(l) = clip(pi(l)-4, pi(l), pi(l)+4),
     pi(l) = 1 + round((l-1)(L_S-1)/(L_R-1)), concatenated: K = 3 d_S. */
  HF_LAYER_PAPER3 = 0,
  /* One segment: the linear interpolation of sender layers floor(p) and
     floor(p)+1 at p = l (L_S-1)/(L_R-1) (zero-based l): K = d_S. */
  HF_LAYER_INTERP = 1,
  /* A caller-given table with the structure of Eq. 2: n_seg (1 .. 8)
     segments per receiver layer, segment s = sum over its n_terms terms of
     h_seg_w * (sender layer h_seg_layer): K = n_seg d_S.  The KV Ridge
     comparison system (Appendix A baseline details, Appendix F mapper size)
     is this mode with its k = 8 selected sender layers as eight one-layer
     segments of weight 1, its per-head maps stacked into one dense
     [8 d_S, d_R] map per layer and role (each head's map reads all KV heads
     of the eight layers) and r = 1. */
  HF_LAYER_EXPLICIT = 2
} hf_layer_mode;

typedef enum {
  HF_BF16 = 0, /* bf16 K/V and maps; fp32 accumulation (tcgen05 kind::f16) */
  HF_F32 = 1   /* fp32 K/V and maps; tf32 products, fp32 accumulation */
} hf_dtype;

/* Bits of the device status word. */
#define HF_CHECK_BAD_OFFSETS   0x01 /* offsets not strictly increasing, or ends differ */
#define HF_CHECK_BAD_COLUMN    0x02 /* a CSR column outside the sender tokens */
#define HF_CHECK_BAD_ROW       0x04 /* an empty CSR row, or a row that is not one
                                       weight-1 entry where the align mode says so */
#define HF_CHECK_BAD_BLOCK     0x08 /* a block-table entry outside the pool */
#define HF_CHECK_CAPACITY      0x10 /* the CSR did not fit the given capacity */
#define HF_CHECK_TIMEOUT       0x20 /* a pipeline wait gave up (internal error) */
#define HF_CHECK_INTERNAL      0x40 /* a launch invariant did not hold (internal error) */
#define HF_CHECK_POOL_WINDOW   0x80 /* pooling after the map: a CSR row's columns do not
                                       fit its 128-token window (rows whose first
                                       columns decrease, or a row spanning 128 or more
                                       sender tokens); create the plan with
                                       pool_before_map = 1 */

/*
 * hf_align_build — alignment CSR from character-end offsets (Section 3.1,
 * Appendix B.1; mode as above).
 *
 * n_req      number of requests (1 .. 4096) concatenated in one call.
 * s_tok_ptr  host int32[n_req+1], non-decreasing, s_tok_ptr[0] = 0: request q
 *            owns sender tokens [s_tok_ptr[q], s_tok_ptr[q+1]).
 * r_tok_ptr  host int32[n_req+1], the same for receiver tokens.
 * d_s_end    device int32[T_s]: character-end offset of every sender token,
 *            restarting per request; strictly increasing and positive within
 *            a request (tokens are nonempty).
 * d_r_end    device int32[T_r]: the same for receiver tokens.  Within a
 *            request the last sender and receiver ends must be equal (both
 *            sides tokenise the same text); a request with receiver tokens
 *            needs at least one sender token.
 * d_row_ptr  device int32[T_r+1] out: CSR row pointers, global.
 * d_col      device int32[nnz_capacity] out: global sender token indices.
 * d_w        device float[nnz_capacity] out: pooling weights.
 * nnz_capacity  entries available in d_col/d_w; must be >= T_r for TA and
 *            same-index, >= T_r + T_s for overlap mean pooling.
 * d_info     device int32[2] out: [0] = nnz, [1] = status bits
 *            (HF_CHECK_BAD_OFFSETS, HF_CHECK_CAPACITY).
 * Rows are ordered like the receiver tokens; each row's columns ascend.
 */
hf_status hf_align_build(hf_align_mode mode, int32_t n_req, const int32_t* s_tok_ptr,
                         const int32_t* r_tok_ptr, const int32_t* d_s_end,
                         const int32_t* d_r_end, int32_t* d_row_ptr, int32_t* d_col,
                         float* d_w, int64_t nnz_capacity, int32_t* d_info,
                         hf_stream_t stream);

/* Everything a transfer needs besides the two caches. */
typedef struct {
  /* Shapes: layers, KV heads and head width of sender (s) and receiver (r).
     d_S = H_s * D_s and d_R = H_r * D_r are the flattened feature widths
     (head-major, index h * D + d). */
  int32_t L_s, H_s, D_s;
  int32_t L_r, H_r, D_r;
  hf_dtype dtype;          /* element type of both caches and of d_W */
  hf_layer_mode layer_mode;
  hf_align_mode align_mode; /* the rule the CSR was built with */

  /* Requests (host): as in hf_align_build. */
  int32_t n_req;
  const int32_t* s_tok_ptr;     /* host int32[n_req+1] */
  const int32_t* r_tok_ptr;     /* host int32[n_req+1] */
  const int32_t* r_pos0;        /* host int32[n_req] receiver position of each
                                   request's first token, or NULL for 0 */

  /* Alignment CSR (device, from hf_align_build or the caller). */
  const int32_t* d_row_ptr;     /* int32[T_r+1] */
  const int32_t* d_col;         /* int32[nnz] */
  const float* d_w;             /* float[nnz] */

  /* Folded maps (Eq. 9), device.  d_W is A_final transposed:
     [L_r][2][d_R][K] row-major in `dtype`, K = 3 d_S (PAPER3), d_S
     (INTERP) or n_seg d_S (EXPLICIT); row n of W[l][c] holds column n of
     A_final, and segment s of the map input occupies W columns
     [s d_S, (s+1) d_S). */
  const void* d_W;
  const float* d_b;             /* float[L_r][2][d_R], b_final */
  const float* h_r;             /* host float[L_r][2], Eq. 3's r (> 0) */

  /* Receiver key processing. */
  double theta_r;               /* RoPE base; <= 0 disables RoPE unless
                                   h_inv_freq_r is given */
  const float* d_knorm_w;       /* device float[D_r] key RMS-norm weight, or NULL */
  float knorm_eps;

  /* Receiver cache layout.  paged = 0: receiver_kv is
     [L_r][2][T_r][H_r][D_r].  paged = 1: receiver_kv is a block pool
     [L_r][2][n_blocks][block_size][H_r][D_r] and token t of request q goes
     to block d_block_table[q * max_blocks_per_req + t / block_size], slot
     t % block_size. */
  int32_t paged;
  int32_t block_size;
  int32_t n_blocks;
  int32_t max_blocks_per_req;
  const int32_t* d_block_table; /* device int32[n_req][max_blocks_per_req] */

  /* Optional fields below: a zero-initialised descriptor leaves them off. */

  /* Receiver RoPE inverse frequencies, host float[D_r/2] (for instance a
     scaled RoPE variant's table); NULL = fp32(theta_r^(-2i/D_r)).  When
     given, keys are rotated whatever theta_r is. */
  const float* h_inv_freq_r;

  /* Sender keys that already carry RoPE.  The paper maps keys captured
     before RoPE (Section 3 opening paragraph); with sender_k_rotated = 1
     the sender keys hold RoPE at sender positions and every sender key row
     is rotated back (rotate-half pairs (i, i + D_s/2), angle
     -pos * inv_freq_s_i) at its own sender position before pooling and
     blending; values are not touched.  The sender position of token t of
     request q is s_pos0[q] + t.  Requires D_s/2 a multiple of 8 (bf16) or
     4 (fp32), D_s dividing 128 (bf16) or 64 (fp32), and d_S a multiple of
     128 (bf16) or 64 (fp32); slower than the default path (the rotation
     runs in the operand builder). */
  int32_t sender_k_rotated;
  double theta_s;               /* sender RoPE base, used when h_inv_freq_s is NULL */
  const float* h_inv_freq_s;    /* host float[D_s/2], or NULL */
  const int32_t* s_pos0;        /* host int32[n_req], or NULL for 0 */

  /* Message spans (Appendix "HiddenBench Evaluation": only the K/V states
     of a message that follows a context are mapped).  s_row0 (host
     int32[n_req], or NULL): request q's sender tokens are the sender-cache
     rows s_row0[q] .. s_row0[q] + (s_tok_ptr[q+1] - s_tok_ptr[q]) - 1; the
     CSR columns still count the concatenated span tokens.  sender_rows:
     rows per (layer, role) in sender_kv (0: T_s = s_tok_ptr[n_req]); every
     span must lie inside it. */
  const int32_t* s_row0;
  int64_t sender_rows;

  /* HF_LAYER_EXPLICIT only: host arrays [L_r][n_seg][n_terms]. */
  int32_t n_seg;                /* 1 .. 8 segments per receiver layer */
  int32_t n_terms;              /* 1 .. 2 sender layers per segment */
  const int32_t* h_seg_layer;   /* zero-based sender layers, in [0, L_s) */
  const float* h_seg_w;         /* finite weights */

  /* bf16 plans whose map input rows are computed rather than copied
     (overlap mean pooling, blended layers, weighted explicit segments,
     rotated sender keys): 0 (default) carries each computed row to the
     tensor core as a pair of bf16 rows, the rounded value and its rounding
     residual, both against the same map rows, so the product sees ~16
     mantissa bits of the fp32 row (about twice the tensor-core work on
     those rows; the error is the output rounding alone); 1 rounds the row
     once to bf16 (faster; adds a relative error of about 2^-9 per input
     feature, which at 1e9 outputs can exceed 2e-2 absolute).  Ignored for
     copied rows and fp32 plans. */
  int32_t round_built_operands;

  /* Overlap mean pooling (HF_ALIGN_OVERLAP_MEAN) is linear, so the map
     commutes with it: y_j = (sum_e w_e x_{col_e} / r) A + b
                           = sum_e w_e (x_{col_e} A) / r + b.
     0 (default): plans in that mode without key norm or rotated sender keys
     map sender rows and pool the mapped rows in the epilogue (pooling after
     the map): the map input rows are sender rows (copied, or blended across
     layers), windows of 128 consecutive aligned sender tokens with a stride
     of 128 - h (h = the widest row's column span), and each receiver row is
     pooled from the window holding its columns.  Needs rows whose first
     columns do not decrease and that span fewer than 128 sender tokens
     (as hf_align_build makes them); otherwise HF_CHECK_POOL_WINDOW is set
     and the rows that do not fit are left incomplete (every access stays
     inside the caches).  1: pool before the map (map input rows computed
     per distinct CSR row), with no such limit. */
  int32_t pool_before_map;
} hf_plan_desc;

typedef struct hf_plan_s* hf_plan;

/* Bytes of device workspace hf_plan_create needs for this descriptor. */
hf_status hf_plan_workspace_size(const hf_plan_desc* desc, size_t* bytes);

/*
 * hf_plan_create — validate the descriptor and build the per-transfer
 * metadata on `stream`: the layer table (Eq. 1, interpolation or explicit),
 * RoPE inverse frequencies (fp32(theta^(-2i/D)) or the caller's tables), the
 * receiver position and destination row of every receiver token, the
 * sender position of every sender token (sender_k_rotated only), and the
 * runs of identical CSR rows (their map output is identical before RoPE).
 * d_workspace: device memory of hf_plan_workspace_size bytes, 256-byte
 * aligned, owned by the caller and reserved for this plan until
 * hf_plan_destroy.  The plan keeps pointers to d_row_ptr, d_col, d_w,
 * d_W, d_b, d_knorm_w and d_block_table; host arrays are copied.
 */
hf_status hf_plan_create(const hf_plan_desc* desc, void* d_workspace, size_t workspace_bytes,
                         hf_stream_t stream, hf_plan* out);

/*
 * hf_transfer — write the receiver cache (one kernel launch on `stream`).
 * sender_kv:   device [L_s][2][sender_rows][H_s][D_s] (sender_rows = T_s
 *              unless the plan maps message spans) in the plan's dtype, the
 *              sender's keys and values; keys pre-RoPE (Section 3: keys are
 *              mapped before key normalisation and RoPE) unless the plan
 *              says sender_k_rotated; 16-byte aligned.
 * receiver_kv: device, layout per desc.paged; 16-byte aligned.  Only the
 *              rows (contiguous) or block slots (paged) of the plan's
 *              receiver tokens are written.
 */
hf_status hf_transfer(hf_plan plan, const void* sender_kv, void* receiver_kv,
                      hf_stream_t stream);

/*
 * hf_transfer_host — the transfer for caches held in page-locked host
 * memory, with the host<->device copies overlapped with the computation.
 * The paper moves the sender payload GPU to GPU; this entry point serves
 * callers whose caches live on the host.
 * h_sender_kv:   page-locked host [L_s][2][sender_rows][H_s][D_s]
 *                (cudaHostAlloc or cudaHostRegister), the layout hf_transfer
 *                takes.
 * d_sender_kv:   device buffer of the same size: the sender layers are
 *                brought there (only layers 0 .. the highest one the layer
 *                table reads).  When every alignment row is one sender
 *                token (Token Alignment, same-index, no rotated keys), only
 *                the referenced rows are read, by a gather kernel through
 *                the mapped host memory; other rows of d_sender_kv are left
 *                as they were.  Otherwise whole layers are copied.
 * d_receiver_kv: device receiver cache, as for hf_transfer.
 * h_receiver_kv: page-locked host buffer of the receiver cache's size
 *                (contiguous or paged layout); every receiver layer is
 *                copied back whole (a paged pool's untouched blocks too).
 *                NULL: nothing is copied back (the receiver model reads its
 *                cache in device memory; only the sender comes from the
 *                host).
 * n_groups:      receiver layers are processed in n_groups consecutive
 *                groups (1 .. L_r; 0 = L_r, one per layer): group g's sender
 *                layers are copied in, its layers computed on `stream`,
 *                then copied out while later groups proceed.
 * The call is asynchronous: work starts after earlier work on `stream`, and
 * `stream` is ordered after the last copy out.  Copies run on two streams
 * the plan creates on first use (on the current device; released by
 * hf_plan_destroy).  One call at a time per plan.
 */
hf_status hf_transfer_host(hf_plan plan, const void* h_sender_kv, void* d_sender_kv,
                           void* d_receiver_kv, void* h_receiver_kv, int32_t n_groups,
                           hf_stream_t stream);

/*
 * hf_transfer_batch — several transfer directions in one call (a
 * multi-agent round sends each message to receivers of other model
 * families; Appendix "HiddenBench Evaluation").  Direction i is
 * hf_transfer(plans[i], sender_kv[i], receiver_kv[i]).  When all plans
 * share the dtype and the operand path (one-entry alignment rows with
 * one-layer segments, or not), the directions run in one launch of the
 * transfer kernel over all their tiles; otherwise each direction's kernel
 * runs on a stream of a per-device pool forked from `stream` (created on
 * the first such call on a device).  `stream` is ordered after all of them.
 * n in [0, 16]; a plan appears at most once; the receiver caches must not
 * overlap.  Asynchronous.
 */
hf_status hf_transfer_batch(const hf_plan* plans, const void* const* sender_kv,
                            void* const* receiver_kv, int32_t n, hf_stream_t stream);

/* Frees the plan's host memory and its copy streams.  Does not touch the
   workspace. */
hf_status hf_plan_destroy(hf_plan plan);

/* Synchronises `stream` and returns the plan's device status bits in
   *flags (0 = clean); HF_ERR_DEVICE_CHECK if any bit is set. */
hf_status hf_plan_device_status(hf_plan plan, hf_stream_t stream, int32_t* flags);

/* Synchronises `stream` and returns the number of distinct alignment rows. */
hf_status hf_plan_distinct_rows(hf_plan plan, hf_stream_t stream, int32_t* n_rows);

/*
 * hf_transfer_noalloc — hf_plan_create + hf_transfer + hf_plan_destroy in
 * one call that allocates no memory: the plan metadata goes to a device
 * array built into the library instead of a caller workspace.  The paper
 * has no counterpart; this is a convenience for callers that cannot
 * allocate device memory per call (a host framework or plugin that owns
 * every device allocation, or a fixed memory budget).
 *  - The built-in array holds 8 MiB per GPU (about 340K receiver tokens);
 *    every GPU that loads the library keeps it until the process exits.
 *    Larger transfers are rejected with HF_ERR_UNSUPPORTED and a message.
 *  - The first call on a device looks the array's device address up
 *    (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture.
 *  - Every call shares the array: calls that overlap on the GPU (different
 *    streams, or another thread) race and give wrong results.  Calls on one
 *    stream are ordered and safe.  The device status bits are not reported.
 *  - desc, sender_kv and receiver_kv are as for hf_plan_create and
 *    hf_transfer; the call is asynchronous on `stream`.
 */
hf_status hf_transfer_noalloc(const hf_plan_desc* desc, const void* sender_kv,
                              void* receiver_kv, hf_stream_t stream);

/*
 * hf_fold — folds the output-aware low-rank correction of Eq. 7,
 * y_hat = y0 + (y0 B) G, into the affine maps (Eq. 9):
 * A_final = A (I + B G), b_final = b (I + B G), for n_maps maps at once
 * (e.g. every receiver layer and role), in the layout hf_plan_desc takes.
 * Offline: run once per model pair, before plans that use the maps.
 * d_W:       device [n_maps][d_R][K] in `dtype`: W = A^T, as d_W of
 *            hf_plan_desc.
 * d_b:       device float[n_maps][d_R].
 * d_B:       device float[n_maps][d_R][rank]; d_G: float[n_maps][rank][d_R].
 * d_W_final: device, like d_W (may be d_W itself: folded in place);
 *            rounded once to `dtype`.
 * d_b_final: device float[n_maps][d_R] (may be d_b).
 * rank 4, 8, 16 or 32 (the paper uses 16); K even; d_W, d_W_final and
 * d_B 16-byte aligned.  Asynchronous on `stream`.
 */
hf_status hf_fold(hf_dtype dtype, int32_t n_maps, int32_t d_R, int64_t K, int32_t rank,
                  const void* d_W, const float* d_b, const float* d_B, const float* d_G,
                  void* d_W_final, float* d_b_final, hf_stream_t stream);

/*
 * hf_recolor_fit — the Recolor initialisation of one map (Section 3.2,
 * Eq. 3-5) from N weighted aligned sample pairs: r (Eq. 3), weighted means
 * and covariances of Z = X / r and Y, R* the orthogonal polar factor of
 * Sigma_Z^{-1/2} Sigma_ZY Sigma_Y^{-1/2} (the U Q^T of its thin SVD,
 * Eq. 4), A = Sigma_Z^{-1/2} R* Sigma_Y^{1/2} and b = mu_Y - mu_Z A (Eq. 5).
 * Offline (once per map before calibration and folding).
 * d_X:  device [N][d_S] in `dtype`: Eq. 2 concatenated sender features
 *       (d_S here is the map input width, 3 d_S of the plan in paper mode).
 * d_Y:  device [N][d_R] in `dtype`: receiver targets.
 * d_w:  device float[N], positive sample weights.
 * reg:  numerical stabilisation: reg * (mean eigenvalue) is added to each
 *       covariance's diagonal (0: none; the paper does not give its form).
 * d_W_out: device [d_R][d_S] in `dtype`: A^T, the layout of hf_plan_desc's
 *       d_W; d_b_out: device float[d_R]; h_r_out: host float, r (or NULL);
 *       h_iters_out: host int32[3] (or NULL), the iterations taken by the
 *       roots of Sigma_Z and Sigma_Y and by the polar factor.
 * d_workspace: hf_recolor_workspace_size bytes, 256-byte aligned.
 * Requires d_S >= d_R and N * d_S < 2^31.  Matrix roots and the polar
 * factor use Newton-Schulz iterations in fp32; the matrix products run on
 * this library's tcgen05 kernel in fp32 accuracy (each fp32 operand split
 * exactly into three bf16 parts, the six largest partial products summed in
 * an fp32 tensor-memory accumulator).  The call synchronises `stream`
 * (convergence checks) and returns HF_ERR_DEVICE_CHECK if an iteration does
 * not converge (raise reg) or a product kernel's wait ran out.
 */
hf_status hf_recolor_workspace_size(int64_t N, int32_t d_S, int32_t d_R, size_t* bytes);
hf_status hf_recolor_fit(hf_dtype dtype, int64_t N, int32_t d_S, int32_t d_R, const void* d_X,
                         const void* d_Y, const float* d_w, float reg, void* d_W_out,
                         float* d_b_out, float* h_r_out, int32_t* h_iters_out,
                         void* d_workspace, size_t workspace_bytes, hf_stream_t stream);

const char* hf_status_string(hf_status status);
const char* hf_last_error(void);

/*
 * Test hook for the kernel's bounded waits (not part of the method).
 * hf_debug_transfer_stalled launches hf_transfer's kernel with its map
 * producer withholding the first map atom, so the tensor-core issuer's wait
 * for it, and then every other role's wait, runs out: the launch ends after
 * a few seconds (each wait gives up after 2 s) with HF_CHECK_TIMEOUT set in
 * the plan's status word (hf_plan_device_status), instead of hanging, and
 * the CUDA context stays usable.  receiver_kv's contents are unspecified
 * afterwards; a plan created again starts with a clear status.  Arguments as
 * hf_transfer; HF_ERR_INVALID_ARGUMENT for a plan without receiver tokens.
 */
hf_status hf_debug_transfer_stalled(hf_plan plan, const void* sender_kv, void* receiver_kv,
                                    hf_stream_t stream);

/*
 * Test hook for the fp32 product kernel behind hf_recolor_fit (not part of
 * the method): C[M x N] = alpha op(A) op(B) + beta C on the tensor cores in
 * fp32 accuracy (each operand split exactly into three bf16 parts, the six
 * largest partial products summed in fp32).  Row-major C with leading
 * dimension ldc >= N; op(A)(i, k) = d_A[i * a_i + k * a_k] (i < M, k < K),
 * op(B)(k, j) = d_B[k * b_k + j * b_j] (j < N): strides express transposes.
 * d_workspace: hf_debug_matmul_workspace_size bytes, 256-byte aligned.
 * h_err (or NULL): synchronises `stream` and returns the kernel's error word
 * (0: clean; nonzero: a pipeline wait ran out).  Asynchronous otherwise.
 */
hf_status hf_debug_matmul_workspace_size(int32_t M, int32_t N, int32_t K, size_t* bytes);
hf_status hf_debug_matmul_f32(int32_t M, int32_t N, int32_t K, float alpha, const float* d_A,
                              int64_t a_i, int64_t a_k, const float* d_B, int64_t b_k,
                              int64_t b_j, float beta, float* d_C, int64_t ldc,
                              void* d_workspace, size_t workspace_bytes, int32_t* h_err,
                              hf_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* HETEROFOLD_H */
