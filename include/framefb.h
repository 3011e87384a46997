/*
 * framefb.h -- C ABI of the FrameFT adapter hot path on GB300 (sm_103a).
 *
 * FrameFT (arxiv 2608.26430) writes the update of a frozen weight
 * W in R^{m x n} as
 *
 *     dW = s * Phi_out * C * Phi_in^T,     s = alpha / sqrt(m n)      (Sec. 3.1)
 *
 * where Phi_in = P_n (n x K_n) and Phi_out = P_m (m x K_m) are the synthesis
 * matrices of tight fusion frames built by Spectral Tetris, modulation and
 * realification (Sec. 3.2, appendix example), shared by every layer of the
 * same dimension, and C (K_m x K_n) is sparse on a support shared by every
 * layer of a shape (Sec. 3.3).  Activations are row-major, one token per row:
 * X is N x n, Y and dY are N x m.
 *
 *   forward      Y  += X dW^T                         (Alg. 1 steps 5-6)
 *   backward dX  dX += dY dW
 *   grad coeff   dC  = s (Phi_out^T dY^T X Phi_in) sampled on supp(C)
 *                     (Lemma 1 proof, Appendix A: grad f(C) = P_m^T grad f(W) P_n)
 *   merge        W_t = W0 + dW(C_t)  for T tenants     (Alg. 1 step 6)
 *
 * Conventions for every entry point:
 *  - Plain pointers and sizes only.  "host" pointers are read during the call
 *    and may be freed when it returns; "device" pointers must stay valid until
 *    the work queued on `stream` has run.
 *  - The library never allocates device memory.  All device buffers (inputs,
 *    outputs, frames, plan image, workspace) belong to the caller.
 *  - Every argument is validated before any launch; a failed check returns a
 *    negative framefb_status and queues nothing.  The library never aborts
 *    and never prints.  Faults of queued kernels surface at the caller's next
 *    synchronisation of `stream`.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *  - Calls are stateless and may be made from several host threads.
 */
#ifndef FRAMEFB_H
#define FRAMEFB_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FRAMEFB_ABI_VERSION 2

/* Threads per CTA of the activation kernels; plans are cut for this count. */
#define FRAMEFB_THREADS 256

typedef enum {
  FRAMEFB_OK = 0,
  FRAMEFB_EINVAL = -1,        /* null pointer, bad size, misaligned pointer, inconsistent shapes */
  FRAMEFB_EUNSUPPORTED = -2,  /* Spectral Tetris / modulation infeasible, or no GPU path for these parameters */
  FRAMEFB_ENOMEM = -3,        /* host allocation failed */
  FRAMEFB_ECUDA = -4,         /* a CUDA runtime call (device query, attribute, launch) failed */
  FRAMEFB_EWORKSPACE = -5     /* workspace missing or smaller than framefb_workspace_size() */
} framefb_status;

typedef enum { FRAMEFB_F32 = 0, FRAMEFB_BF16 = 1 } framefb_dtype;

typedef enum {
  FRAMEFB_SUPPORT_UNIFORM = 0,    /* positions uniform over K_m x K_n */
  FRAMEFB_SUPPORT_ZIPF_ROWS = 1,  /* row r+1 drawn with probability ~ (r+1)^-s, column uniform */
  FRAMEFB_SUPPORT_BLOCKDIAG = 2   /* uniform inside the k diagonal blocks C_{l,i} (Sec. 3.1) */
} framefb_support_mode;

/* Human-readable name of a status code (static string, never NULL). */
const char* framefb_status_string(int32_t status);

/* FRAMEFB_ABI_VERSION of the loaded library. */
int32_t framefb_abi_version(void);

/* ------------------------------------------------------------------------ */
/* S1  frame construction (host)                                             */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t k;         /* number of subspaces */
  int32_t rho;       /* real dimension of each subspace; even, >= 2 (appendix discussion: realification doubles it) */
  int32_t parseval;  /* nonzero: scale by 1/sqrt(A) so that Phi Phi^T = I (Sec. 3.4 uses Parseval frames) */
} framefb_frame_params;

/*
 * Host-side frame storage.  All arrays are allocated by the library and owned
 * by the struct until framefb_frame_free().
 *
 * Column c = i*rho + 2r + s of Phi (d x ncols, ncols = k*rho) is the unit-norm
 * real vector of subspace i built from Spectral Tetris row r; s = 0 holds
 * (Re z_j, -Im z_j) on coordinates (2j, 2j+1), s = 1 holds (Im z_j, Re z_j),
 * z_j = F[r][j] omega^{(i j) mod k} / sqrt(d_c/rho_c), omega = exp(2 pi i/k)
 * (appendix: Spectral Tetris, Modulation; realification map x+iy -> [[x,-y],[y,x]]).
 * The full 2x2 block of every nonzero F[r][j] is stored, exact zeros included.
 */
typedef struct {
  int32_t d, k, rho, ncols;
  int64_t nnz;              /* stored entries */
  double A;                 /* frame bound of the unit-norm system: sum_i P_i P_i^T = A I, A = k*rho/d */
  double scale;             /* 1, or 1/sqrt(A) when Parseval was requested (already applied to the values) */
  int64_t* csc_colptr;      /* [ncols+1] */
  int32_t* csc_rowidx;      /* [nnz], ascending within a column */
  double*  csc_val;         /* [nnz] */
  int64_t* csr_rowptr;      /* [d+1] */
  int32_t* csr_colidx;      /* [nnz], ascending within a row */
  double*  csr_val;         /* [nnz] */
  int32_t  ngroups;         /* rho/2: one group per Spectral Tetris row */
  int32_t* grp_row0;        /* [ngroups] first coordinate of the group */
  int32_t* grp_nrows;       /* [ngroups] coordinates spanned by the group */
  int32_t  dft_groups;      /* 1 when k*rho == d: the groups are the disjoint coordinate blocks
                               [2kr, 2k(r+1)) and each carries the same realified DFT_k block */
} framefb_frame;

/*
 * Build the (k, rho, d) tight fusion frame (Sec. 3.2; appendix walk-through).
 * d: real dimension, even.  Returns FRAMEFB_EUNSUPPORTED when Spectral Tetris
 * cannot run (d/2 < rho) or the modulated system is not tight (k smaller than
 * the widest row support of F), FRAMEFB_EINVAL for bad arguments,
 * FRAMEFB_ENOMEM on allocation failure.  On error *out is zeroed.
 */
framefb_status framefb_frame_build(int32_t d, const framefb_frame_params* params, framefb_frame* out);
void framefb_frame_free(framefb_frame* f);

/*
 * Device view of a frame: fp32 copies of the CSC arrays uploaded by the
 * caller, and (for frames outside the structured kernels) the dense operand
 * image.
 *
 * Two device paths exist.  Frames with k = 16 and k*rho = d (dft_groups set:
 * rho/2 disjoint 32-coordinate groups, each a realified DFT_16 block) run on
 * the structured kernels, which read `val` only.  Every other frame the
 * builder produces -- the paper's own rho = 2 regime (k*rho = d with one
 * group: Phi is a dense realified DFT of size d/2) and redundant frames with
 * T blocks (k*rho > d) -- runs on the dense path, which treats Phi as a
 * dense d x ncols matrix and reads it from `dense`: a device copy, byte for
 * byte, of the image framefb_frame_dense_pack() writes (16-byte aligned).
 * `dense` may be NULL for structured frames.
 */
typedef struct {
  int32_t d, k, rho, ncols;
  int32_t dft_groups;
  int32_t pad_;
  const int64_t* colptr;    /* device [ncols+1] */
  const int32_t* rowidx;    /* device [nnz] */
  const float*   val;       /* device [nnz], fp32 */
  const void*    dense;     /* device dense operand image, or NULL (see above) */
} framefb_dev_frame;

/*
 * Dense operand image of a frame for the dense path (any frame; needed for
 * frames without dft_groups and k = 16).  framefb_frame_dense_bytes() gives
 * its size (0 for a NULL or empty frame); framefb_frame_dense_pack() writes
 * it into the caller's host buffer `out` of `bytes` bytes: Phi's columns as
 * bf16 hi + lo parts (the analysis operand) and Phi's rows rounded to tf32
 * (the synthesis operand), zero-padded rows.  The caller copies it verbatim
 * to the device and points framefb_dev_frame.dense at the copy.
 * FRAMEFB_EINVAL for a NULL argument or a buffer that is too small.
 */
size_t framefb_frame_dense_bytes(const framefb_frame* f);
framefb_status framefb_frame_dense_pack(const framefb_frame* f, void* out, size_t bytes);

/* ------------------------------------------------------------------------ */
/* S2  coefficient support (host)                                            */
/* ------------------------------------------------------------------------ */

/*
 * Draw nnz distinct positions (a, b) of C (rows x cols) from a splitmix64
 * stream seeded with `seed` (Sec. 3.3: random positions, shared across
 * layers).  mode: framefb_support_mode; zipf_s: exponent for ZIPF_ROWS;
 * k: number of diagonal blocks for BLOCKDIAG (must divide rows and cols).
 * Outputs (caller-owned host arrays): row[nnz], col[nnz] sorted row-major;
 * csr_rowptr[rows+1] (may be NULL); csc_perm[nnz] = entry indices ordered by
 * (col, row) (may be NULL).  FRAMEFB_EINVAL when nnz exceeds the positions
 * the mode can reach.
 */
framefb_status framefb_support_build(int32_t rows, int32_t cols, int64_t nnz, uint64_t seed,
                                     int32_t mode, double zipf_s, int32_t k,
                                     int32_t* row, int32_t* col, int64_t* csr_rowptr, int32_t* csc_perm);

/* ------------------------------------------------------------------------ */
/* Plan: the support of C re-indexed for the kernels (host, once per shape)   */
/* ------------------------------------------------------------------------ */

/*
 * A plan holds the support of C in the order the kernels walk it: the
 * frame columns re-indexed group-major, entries cut into FRAMEFB_THREADS
 * balanced chunks for the coefficient SpMM (by row) and its transpose (by
 * column), the fix-up list for rows split between chunks, per-group
 * occupancy masks, and the entry list of every 32 x 32 block for the merge.
 * Built once per (frame pair, support) -- the support is shared by all layers
 * of a shape (Sec. 3.3) -- and uploaded verbatim by the caller.
 *
 * fin, fout: host frames (Phi_in with d = n, Phi_out with d = m).
 * row, col: host, the support in sorted row-major order (as from
 * framefb_support_build); C values passed to the kernels follow this order.
 * C is K_m x K_n with K = the frame's ncols (= k*rho).  When both frames
 * have dft_groups and k = 16 the plan is cut for the structured kernels
 * (frame columns re-indexed group-major); otherwise for the dense path
 * (frame columns in the paper's order).  FRAMEFB_EUNSUPPORTED when a frame
 * has more than 32767 columns.  nnz may be 0.
 */
typedef struct framefb_plan framefb_plan;
framefb_status framefb_plan_build(const framefb_frame* fin, const framefb_frame* fout,
                                  const int32_t* row, const int32_t* col, int64_t nnz,
                                  framefb_plan** out);
/* Size and bytes of the position-independent device image; copy it to a
 * 16-byte aligned device buffer and pass that buffer as `plan_dev` below. */
size_t framefb_plan_bytes(const framefb_plan* plan);
const void* framefb_plan_data(const framefb_plan* plan);
void framefb_plan_free(framefb_plan* plan);

/*
 * Parts of a structured plan that the fused tcgen05 kernels cannot take
 * whole (more than 16 * FRAMEFB_THREADS entries, or an output frame of more
 * than 128 groups of 32 features: the LLaMA-3 shapes), for plans whose input
 * frame has at most 128 groups.  The support is cut into blocks of whole
 * groups of the output side (at most 128 groups, a multiple of 8) and, per
 * block, runs of at most 16 * FRAMEFB_THREADS entries in row-major order.
 * (Blocks of the input side would give every part a partial sum of each
 * row, and rounding the bf16 output once per part would exceed the bf16
 * tolerance on heavy-tailed supports: such plans have no parts.)  Every part is a plan of its own over its two blocks,
 * stored in the plan's device image after the whole plan, with the list of
 * its entries' indices into the caller's C values and dC (int32).  framefb_run
 * runs each part as a matrix of the fused kernels: ΔW is linear in C, so
 * Y and dX take the sum of the parts' contributions, and each part writes
 * its own entries of dC.  This restates the method exactly; it is the
 * library's own execution plan, with no counterpart in the paper.
 * framefb_plan_parts returns the number of parts (0 for plans the kernels
 * take whole) and fills up to max_parts descriptors (parts may be NULL).
 */
typedef struct {
  int64_t image_offset, image_bytes;  /* the part's plan image in the device image */
  int64_t q_offset;                   /* its int32 entry indices (nnz of them) in the device image */
  int32_t nnz;                        /* its entries */
  int32_t n0, m0;                     /* first input / output feature of its blocks */
  int32_t n, m;                       /* features of its blocks */
} framefb_plan_part;
int32_t framefb_plan_parts(const framefb_plan* plan, framefb_plan_part* parts, int32_t max_parts);

/* ------------------------------------------------------------------------ */
/* S3-S6  batched activation kernels (device)                                */
/* ------------------------------------------------------------------------ */

/*
 * One adapted matrix.  All pointers except fin/fout are device pointers.
 * X, dX: N x n row-major with leading dimension ldx elements (dX shares ldx).
 * dY, Y: N x m row-major with leading dimension ldy elements.
 * Element type: the dtype argument of the call (fp32 or bf16); rows must be
 * 16-byte aligned (pointer and ld * element size multiples of 16).
 * Pointers an operation does not use may be NULL (forward: X, Y;
 * backward_dx: dY, dX; grad_coeff: X, dY, dC).
 * fin, fout: HOST pointers to device frame views (d = n and d = m).
 * plan: HOST handle from framefb_plan_build (sizes and checks are taken from it).
 * plan_dev: device copy of framefb_plan_data(plan), byte for byte.
 * c_val: [nnz] fp32 coefficient values in the plan's support order.
 * dC: [nnz] fp32 output of grad_coeff (overwritten).
 * scale: s = alpha / sqrt(m n).
 * Y and dX accumulate (+=).  Different matrices of one call must not alias
 * their Y, dX or dC.
 */
typedef struct {
  int32_t N, n, m;
  int32_t pad_;
  const void* X;  void* dX;  int64_t ldx;
  const void* dY; void* Y;   int64_t ldy;
  const framefb_dev_frame* fin;
  const framefb_dev_frame* fout;
  const framefb_plan* plan;
  const void*  plan_dev;
  const float* c_val;
  float*       dC;
  float        scale;
  int32_t      pad2_;
} framefb_mat;

#define FRAMEFB_OP_FORWARD     1   /* Y  += X dW^T                                  */
#define FRAMEFB_OP_BACKWARD_DX 2   /* dX += dY dW                                   */
#define FRAMEFB_OP_GRAD_COEFF  4   /* dC  = s (Phi_out^T dY^T X Phi_in) on supp(C)   */

/* Device workspace (bytes) a call with `ops` over these matrices needs on the
 * current device; 0 when none.  Depends on the SM count of the current device. */
size_t framefb_workspace_size(const framefb_mat* mats, int32_t nmats, int32_t ops);

/*
 * Run `ops` (an OR of FRAMEFB_OP_*) over nmats matrices.  One launch covers
 * every matrix (a second, small launch reduces dC when GRAD_COEFF is set).
 * When several ops are requested, X and dY are read once for all of them.
 * ws: device workspace of at least framefb_workspace_size() bytes, 256-byte
 * aligned (may be NULL when that size is 0).
 */
framefb_status framefb_run(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype,
                           void* ws, size_t ws_bytes, void* stream);

/*
 * framefb_run without a caller-provided workspace.  The paper has no
 * counterpart: this entry point is for callers that cannot allocate device
 * memory where they call the library -- code that runs inside a fixed device
 * memory budget handed out by a host framework, or a latency-critical path
 * that must not call cudaMalloc because it can synchronise the device.
 * The dC partial sums go to a library-owned static device array of
 * FRAMEFB_STATIC_WS_BYTES (8 MiB) that every GPU which loads the library
 * holds until the process exits; nothing is allocated per call.  A call whose
 * workspace need (framefb_workspace_size) exceeds that size returns
 * FRAMEFB_EWORKSPACE and queues nothing.  The first call on a device looks up
 * the array's device address with cudaGetSymbolAddress and caches it with the
 * device's current context (a device reset or a new primary context makes
 * the next call look it up again): make that first call outside any stream
 * capture.  All calls on one device share
 * the array: calls whose kernels can overlap on the GPU (e.g. on unordered
 * streams) race on it and must be ordered by the caller.  Each call writes
 * every partial sum it reads, so no state carries over between calls.
 * Arguments and results are those of framefb_run.
 */
#define FRAMEFB_STATIC_WS_BYTES (8u << 20)
framefb_status framefb_run_static_ws(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype,
                                     void* stream);

/*
 * Names of the kernels framefb_run would launch for these arguments (no
 * launch, no device work beyond attribute queries): the distinct tile
 * kernels of its launch chunks, comma-separated, each with its op mask, e.g.
 * "tc2_tile_kernel<7>"; empty when no tile kernel runs (N = 0).  buf: host,
 * len bytes, always NUL-terminated.  The paper has no counterpart: this is a
 * query for benchmarks and tests.  Errors as framefb_run, and FRAMEFB_EINVAL
 * when buf is NULL or too short.
 */
framefb_status framefb_kernel_names(const framefb_mat* mats, int32_t nmats, int32_t ops, framefb_dtype dtype,
                                    char* buf, size_t len);

/* S3 -> S4 -> S5: Y += ((X Phi_in) C^T) Phi_out^T * s  (forward of Y = X W'^T). */
framefb_status framefb_forward(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                               void* ws, size_t ws_bytes, void* stream);
/* dX += ((dY Phi_out) C) Phi_in^T * s. */
framefb_status framefb_backward_dx(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                   void* ws, size_t ws_bytes, void* stream);
/* S6: dC_q = s sum_t (dY Phi_out)[t, a_q] (X Phi_in)[t, b_q]. */
framefb_status framefb_grad_coeff(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                  void* ws, size_t ws_bytes, void* stream);
/* backward_dx and grad_coeff in one pass over X and dY. */
framefb_status framefb_backward(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                void* ws, size_t ws_bytes, void* stream);
/* forward, backward_dx and grad_coeff in one pass over X and dY. */
framefb_status framefb_fused_fwd_bwd(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                     void* ws, size_t ws_bytes, void* stream);

/*
 * Mixed-tenant forward without merge (Sec. 3.4, multi-tenant serving): the
 * tokens of one batch belong to requests of different tenants, each with its
 * own coefficient values on the shared support:
 *   Y[t] += X[t] dW(C_{tenant(t)})^T  for every token t and matrix.
 * Tokens are grouped in nseg segments: segment i holds tokens
 * [seg_start[i], seg_start[i+1]) of tenant seg_tenant[i] (host arrays;
 * seg_start non-decreasing from 0 to N, empty segments allowed; tenants in
 * [0, ntenants)).  Each framefb_mat describes the whole batch (N = seg_start[nseg],
 * X and Y as for framefb_forward) and its c_val points to the tenants'
 * values, tenant-major: [ntenants][nnz] fp32 on the device.  For bf16
 * activations on the two-token tcgen05 kernels, and at most 256 segments,
 * the segment table travels in the kernel's launch parameters: each matrix's
 * units of work stay inside segments, and the coefficient SpMM loads a
 * tenant's values where the tenant changes (one launch per chunk of
 * matrices, as framefb_forward).  Otherwise every segment of every matrix
 * runs as its own matrix of framefb_forward (rows offset into X and Y, the
 * tenant's row of c_val).  Both give the same Y, bit for bit.  dX and dC are
 * not touched.
 * Errors as framefb_forward, and FRAMEFB_EINVAL for an inconsistent segment
 * table.
 */
framefb_status framefb_forward_tenants(const framefb_mat* mats, int32_t nmats, framefb_dtype dtype,
                                       const int32_t* seg_start, const int32_t* seg_tenant, int32_t nseg,
                                       int32_t ntenants, void* stream);

/* Number of waits on asynchronous row copies, since the library was loaded
 * on the current device, that gave up after their time limit (about one
 * second) instead of hanging; the CTA concerned stopped without finishing its
 * tiles, so the results of that call are incomplete.  0 in normal operation.
 * Synchronises with the device. */
framefb_status framefb_wait_timeouts(uint32_t* count);

/* ------------------------------------------------------------------------ */
/* S7  multi-tenant merge (device)                                           */
/* ------------------------------------------------------------------------ */

/*
 * W_t = W0 + s Phi_out C_t Phi_in^T for t < T (Alg. 1 step 6 per tenant).
 * W0: device, m x n row-major, leading dimension ldw elements, dtype elements.
 * Wout: device, T x m x n, tenant t at Wout + t*m*ldw elements, same ldw.
 * c_vals: device [T][nnz] fp32, tenant-major, plan support order (nnz from the plan).
 * fin, fout: host pointers to device frame views; plan: host handle;
 * plan_dev: its device copy.  Rows 16-byte aligned as for framefb_mat.
 * Wout must not overlap W0.
 */
framefb_status framefb_merge(const void* W0, framefb_dtype dtype, int32_t m, int32_t n, int64_t ldw,
                             const framefb_dev_frame* fin, const framefb_dev_frame* fout,
                             const framefb_plan* plan, const void* plan_dev, const float* c_vals,
                             int32_t T, float scale, void* Wout, void* stream);

/* ------------------------------------------------------------------------ */
/* Optimiser step on the coefficient values (device)                         */
/* ------------------------------------------------------------------------ */

/* AdamW hyperparameters (the paper's runs use AdamW with the stock defaults
 * beta1 0.9, beta2 0.999, eps 1e-8, weight decay 0.01 and the adapter
 * learning rates of its hyperparameter tables). */
typedef struct {
  float lr;            /* this step's learning rate, >= 0 */
  float beta1, beta2;  /* moment decay rates, in [0, 1) */
  float eps;           /* > 0 */
  float weight_decay;  /* decoupled weight decay, >= 0 */
} framefb_adamw_params;

/*
 * One AdamW step (Adam with decoupled weight decay; Appendix "Hyperparameters
 * used for the experiments": AdamW with a linear schedule with warmup) on n
 * fp32 coefficient values, elementwise and in place:
 *   p <- p (1 - lr wd);  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2;
 *   p <- p - lr (m / (1 - b1^step)) / (sqrt(v / (1 - b2^step)) + eps).
 * param, m, v: device fp32 [n], read and written; grad: device fp32 [n], read
 * (typically the dC of framefb_run, so n = matrices x nnz when the matrices'
 * C and dC are contiguous).  m and v are zero before step 1.  Pointers 4-byte
 * aligned (16-byte alignment of all four takes the vector path); the four
 * arrays must not overlap.  step: 1-based count of this step (bias
 * corrections, computed on the host in double precision).  n == 0 is a no-op.
 * Errors: FRAMEFB_EINVAL for n < 0, step < 1, a null or misaligned pointer or
 * hyperparameters outside the ranges above; FRAMEFB_ECUDA if the launch fails.
 * Asynchronous on `stream`.
 */
framefb_status framefb_adamw(float* param, const float* grad, float* m, float* v, int64_t n,
                             const framefb_adamw_params* hp, int64_t step, void* stream);

/* Learning rate of the step with 0-based index i under the linear schedule
 * with warmup over `total` steps, `warmup` of them warming up:
 * lr_max i / warmup for i < warmup, else lr_max max(0, (total - i) /
 * (total - warmup)); 0 for negative arguments.  Host only. */
double framefb_linear_warmup_lr(int64_t i, int64_t total, int64_t warmup, double lr_max);

#ifdef __cplusplus
}
#endif

#endif /* FRAMEFB_H */
