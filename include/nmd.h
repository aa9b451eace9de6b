/*
 * nmd.h -- C ABI of libnmd, a single-GPU (sm_103a) implementation of the
 * stochastic alternating least-squares sweep (SALSA) for subzero matrix
 * completion S ~ max(0, W H) of a sparse nonnegative m x n matrix S.
 *
 * The method (paper "Subzero matrix completion for sparse data analysis"):
 *   - auxiliary matrix, Sec. 3.2 eq. (updateZ): Z_ij = S_ij where S_ij > 0,
 *     otherwise min(0, L_ij), with L = W H = A B^T (eq. ABt; A = W, B = H^T);
 *   - factor updates, eqs. (lsqA)/(lsqB) in the Delta form of eqs.
 *     (spLsqA)/(spLsqB), restricted to a contiguous block of rows (parallel
 *     least squares, eq. lsqA_par) or to a mini-batch of columns with step
 *     size eta (stochastic least squares, eq. lsqA_sto) plus momentum
 *     (Sec. 4.1, after eq. lsqA_sto);
 *   - losses, Sec. 3.1: objective ||Z - L||_F/||S||_F (eq. auxCost, evaluated
 *     as eq. SLloss), RMSE (eq. RMSE), weighted Jaccard distance (eq. WJD).
 * Z is never stored: every kernel forms its tiles of L on chip.
 *
 * Conventions shared by every call:
 *   - Matrices are row-major, float32.  W is m x r, H is r x n.
 *   - Ownership: the caller owns every pointer it passes.  The library copies
 *     the CSR at nmd_create, keeps only the device workspace pointer it is
 *     given (and never frees it), and frees only its own host objects in
 *     nmd_destroy.  The library itself allocates no device memory.
 *   - Asynchrony: calls that take a handle enqueue their work on the CUDA
 *     stream given to nmd_create and return without waiting, except
 *     nmd_create (waits for its copies), nmd_get_factors, nmd_get_state,
 *     nmd_loss, nmd_sync and nmd_block_terms, which synchronise that stream.
 *   - Errors: every call returns an nmd_status.  A non-OK return leaves the
 *     handle usable; nmd_last_error() gives a one-line description.  Errors
 *     found on the device (a non-positive Cholesky pivot, a non-finite
 *     factor, a wait that ran out) are sticky: they are recorded in device
 *     memory, every later update becomes a no-op, and the next synchronising
 *     call returns the status and clears it.
 *   - Thread safety: none per handle; distinct handles are independent.
 */
#ifndef NMD_H
#define NMD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct nmd_handle nmd_handle;

typedef enum {
  NMD_OK = 0,
  NMD_ERR_INVALID = 1,     /* bad argument (size, index, option, null pointer) */
  NMD_ERR_CSR = 2,         /* malformed CSR: see nmd_create */
  NMD_ERR_NOT_SPD = 3,     /* a block Gram matrix had a non-positive pivot */
  NMD_ERR_DIVERGED = 4,    /* an update produced a non-finite factor entry */
  NMD_ERR_TIMEOUT = 5,     /* a bounded device-side wait ran out */
  NMD_ERR_CUDA = 6,        /* a CUDA runtime call failed */
  NMD_ERR_WORKSPACE = 7,   /* workspace too small or misaligned */
  NMD_ERR_UNSUPPORTED = 8  /* no kernel for this device / rank / precision */
} nmd_status;

typedef enum { NMD_ROW = 0, NMD_COL = 1 } nmd_side;
typedef enum { NMD_EXACT = 0, NMD_STOCH = 1 } nmd_kind;
typedef enum { NMD_ALTERNATE = 0, NMD_PHASED = 1 } nmd_order;

/* Arithmetic of a block step's least-squares problem (each factor is kept as
 * fp32 masters plus bf16 pieces hi = bf16(x), lo = bf16(x - hi),
 * lo2 = bf16(x - hi - lo), all rounded to nearest even):
 *   NMD_BF16 -- the step is set up on the bf16-rounded rows: the dense term
 *               (L = M_hi Q_hi^T and R = P Q_hi on the tcgen05 tensor cores,
 *               fp32 accumulation), the support term (on the hi pieces) and
 *               the Gram matrix G = Q_hi^T Q_hi all use them, so the rounding
 *               is not a coherent error between R and G; the solve X = (R +
 *               Rs) G^{-1} runs on the tensor cores with R + Rs and G^{-1} as
 *               hi + lo bf16 pieces (three products, fp32 accumulation), and
 *               the update is applied to the fp32 masters;
 *   NMD_FP32 -- fp32-accurate: L = M_hi Q_hi^T + M_hi Q_lo^T + M_lo Q_hi^T,
 *               P = P_hi + P_lo (two bf16 pieces), R = P_hi (Q_hi + Q_lo +
 *               Q_lo2) + P_lo Q_hi on the tensor cores; the support term and
 *               G from the fp32 masters;
 *   NMD_SIMT -- plain fp32 FMA on the CUDA cores (slow; reference path).
 * Gram matrices are formed in fp32, factored in fp32 (L D L^T Cholesky form),
 * updates are fp32 (the NMD_BF16 solve as above); loss reductions are fp64. */
typedef enum { NMD_BF16 = 0, NMD_FP32 = 1, NMD_SIMT = 2 } nmd_precision;

/* Form of the dense contraction (both give the same update, Sec. 3.2):
 *   NMD_EPI_Z     -- R = Z Q with the min(0, L) tile epilogue (eq. updateZ),
 *                    update M <- M + eta (R G^{-1} - M)         (eqs. lsqA/lsqB);
 *   NMD_EPI_DELTA -- R = Delta Q with the -max(0, L) tile epilogue (eq. updateD),
 *                    update M <- M + eta R G^{-1}                (eqs. spLsqA/spLsqB). */
typedef enum { NMD_EPI_Z = 0, NMD_EPI_DELTA = 1 } nmd_epilogue;

typedef struct {
  int64_t block_rows;   /* rows of S per row block  (>= 1) */
  int64_t block_cols;   /* columns of S per column block (>= 1) */
  int32_t schedule;     /* nmd_kind used by nmd_sweep */
  int32_t order;        /* nmd_order used by nmd_sweep for NMD_STOCH */
  double eta;           /* step size (> 0); Sec. 4.1 eq. lsqA_sto */
  double gamma;         /* momentum in [0, 1); used by NMD_STOCH updates only */
  double ridge;         /* lambda added to the Gram diagonal (>= 0; default 0) */
  int32_t precision;    /* nmd_precision */
  int32_t epilogue;     /* nmd_epilogue */
  uint64_t seed;        /* block-order seed */
  int32_t skip_zero_chunks;  /* nmd_skip_mode; Delta form only (ignored otherwise).  Default
                              * NMD_SKIP_NONE: the checks cost the dense kernel time when no
                              * chunk vanishes */
} nmd_options;

/* Chunk skipping in the Delta-form dense term -max(0, L) Q (Sec. 4.3: the
 * rectified matrix max(0, A B^T) is sparse when the model is mostly
 * negative).  A chunk is the product of a 128-row M tile with 64 or 128
 * Q-side rows (nmd_range_mask reports the count):
 *   NMD_SKIP_VOTE  -- the first product is computed, and the second is
 *                     skipped where max(0, L) is zero on the whole chunk;
 *   NMD_SKIP_RANGE -- before the dense kernel, a range search over the
 *                     normalised factor rows (eq. range-search: L_ij > 0
 *                     exactly when ||a_i/|a_i| - b_j/|b_j|||^2 < 2) clears the
 *                     chunks on which every L_ij <= 0, and both products are
 *                     skipped there.  The test bounds the distance of every
 *                     pair from below by that of the balls around the tile's
 *                     and the chunk's normalised rows, with a margin for the
 *                     rounding of the operands, so a cleared chunk adds
 *                     exactly zero and the results equal those without
 *                     skipping.
 * Both count the skipped chunks (nmd_skip_count). */
typedef enum { NMD_SKIP_NONE = 0, NMD_SKIP_VOTE = 1, NMD_SKIP_RANGE = 2 } nmd_skip_mode;

typedef struct {
  double obj;        /* ||Z - L||_F / ||S||_F  (eq. auxCost) */
  double rmse;       /* ||S - max(0, L)||_F / ||S||_F  (eq. RMSE) */
  double wjd;        /* 1 - sum min(S, Shat) / sum max(S, Shat)  (eq. WJD) */
  double s_fro;      /* ||S||_F */
  double sum_relu2;  /* sum over all (i, j) of max(0, L_ij)^2 */
  double sum_relu;   /* sum over all (i, j) of max(0, L_ij) */
} nmd_loss_out;

/* Library version string (static storage). */
const char* nmd_version(void);

/* Defaults: blocks of 4096, NMD_STOCH, NMD_ALTERNATE, eta = 1, gamma = 0.9
 * (the paper's defaults, Sec. 5.2 and Table "hyper"), ridge = 0, NMD_BF16,
 * NMD_EPI_Z, seed = 0. */
void nmd_default_options(nmd_options* opts);

/* Device workspace (bytes) nmd_create needs for this problem.  Validates the
 * CSR exactly as nmd_create does (the number of nonzeros is row_ptr[m]; the
 * size depends on the block panels, so the CSR itself is an argument).  The
 * workspace must be 256-byte aligned. */
nmd_status nmd_workspace_bytes(int64_t m, int64_t n, int32_t r, const int64_t* row_ptr,
                               const int32_t* col_idx, const float* vals,
                               const nmd_options* opts, size_t* bytes);

/* Create a solver for the m x n matrix S given as host CSR (row_ptr[m+1],
 * col_idx[nnz], vals[nnz]; the support of S is the set of stored entries
 * with value > 0, eq. updateZ -- stored zeros are dropped).
 * Rejected with NMD_ERR_CSR: row_ptr[0] != 0, decreasing row_ptr, column
 * index outside [0, n), columns not strictly increasing within a row,
 * negative or non-finite values.  Rejected with NMD_ERR_INVALID: m or n < 1
 * or >= 2^31, r < 1 or r > 256, block sizes < 1, eta <= 0, gamma outside
 * [0, 1), ridge < 0, unknown enum values.
 * d_workspace: device memory of at least nmd_workspace_bytes() bytes, owned
 * by the caller and kept until nmd_destroy.  stream: a cudaStream_t (NULL =
 * the legacy default stream).  The factors start at zero: call
 * nmd_set_factors before updating. */
nmd_status nmd_create(int64_t m, int64_t n, int32_t r, const int64_t* row_ptr,
                      const int32_t* col_idx, const float* vals, const nmd_options* opts,
                      void* d_workspace, size_t ws_bytes, void* stream, nmd_handle** out);

/* Set W (m x r, row-major) and H (r x n, row-major); host pointers if
 * on_device == 0, device pointers otherwise.  Resets both momentum buffers
 * to zero.  Asynchronous; host buffers must stay valid until the stream
 * reaches this point (the call waits for the host-to-device copies). */
nmd_status nmd_set_factors(nmd_handle* h, const float* W, const float* H, int on_device);

/* Copy W (m x r) and H (r x n) out, to host (on_device == 0) or device memory.
 * Synchronises the stream and reports any sticky device error. */
nmd_status nmd_get_factors(nmd_handle* h, float* W, float* H, int on_device);

/* One block update of one of four kinds (the M-side is the
 * factor updated, Q-side the rows contracted against):
 *   (NMD_ROW, NMD_EXACT, I): W_I <- least squares against all of H on S[I, :]
 *                            (eq. lsqA_par), W_I += eta (W_ls - W_I);
 *   (NMD_COL, NMD_EXACT, J): H_:J likewise on S[:, J];
 *   (NMD_COL, NMD_STOCH, J): all of W from the mini-batch H_:J on S[:, J]
 *                            (eq. lsqA_sto), with momentum;
 *   (NMD_ROW, NMD_STOCH, I): all of H from the mini-batch W_I on S[I, :].
 * Blocks are contiguous ranges [k b, min((k+1) b, N)) with b = block_rows
 * (row blocks, N = m) or block_cols (column blocks, N = n).  The block's Gram
 * matrix must be nonsingular (a block needs at least r rows with linearly
 * independent factor rows), else NMD_ERR_NOT_SPD is reported by the next
 * synchronising call and the update is skipped.  Asynchronous. */
nmd_status nmd_block_update(nmd_handle* h, int32_t side, int64_t block, int32_t kind);

/* One block update with combined row and column sub-sampling (Sec. 4.1, the
 * remark after eq. lsqA_sto: one update that subsamples both the rows and the
 * columns of Delta), for problems where even a block row of Z is too large:
 *   (NMD_ROW, I, J): W_I <- W_I + E, E = eta (X - W_I) + gamma E, with
 *                    X = argmin ||Z[I, J] - X H_:J|| (the least-squares
 *                    solution against the column block J on S[I, J]);
 *   (NMD_COL, I, J): H_:J likewise against W_I on S[I, J]^T.
 * Blocks as for nmd_block_update (row blocks of block_rows rows, column blocks
 * of block_cols columns); the momentum rows are those of the updated block.
 * The block's Gram matrix must be nonsingular (see nmd_block_update).  Not
 * used by nmd_sweep.  Asynchronous. */
nmd_status nmd_block_update_combined(nmd_handle* h, int32_t side, int64_t row_block, int64_t col_block);

/* One sweep: block orders are SplitMix64 + Fisher-Yates permutations of the
 * row blocks and column blocks for (seed, sweep index, side).  NMD_EXACT:
 * all row blocks, then all column blocks.  NMD_STOCH + NMD_ALTERNATE: for
 * t = 0 .. max(Kc, Kr)-1, column block perm_c[t] (if t < Kc) then row block
 * perm_r[t] (if t < Kr); NMD_PHASED: all column blocks, then all row blocks.
 * Every sweep visits each entry of Z twice.  Advances the sweep counter.
 * Asynchronous. */
nmd_status nmd_sweep(nmd_handle* h);

/* Block order of one sweep and side (perm must hold K = number of blocks of
 * that side; K is checked).  Pure host computation. */
nmd_status nmd_block_order(const nmd_handle* h, int64_t sweep, int32_t side, int64_t* perm,
                           int64_t K);

/* Losses of the current factors (eqs. auxCost/SLloss, RMSE, WJD): a dense
 * pass over all m x n entries of L plus a correction over the support of S,
 * reduced in a fixed order in fp64.  Synchronises the stream. */
nmd_status nmd_loss(nmd_handle* h, nmd_loss_out* out);

/* Waits for the stream and returns (then clears) any sticky device error. */
nmd_status nmd_sync(nmd_handle* h);

/* Verification hook: the right-hand side R = Z Q (NMD_EPI_Z) or Delta Q
 * (NMD_EPI_DELTA) for the M-side rows of one block update (rows x r,
 * row-major) and the Gram matrix G = Q^T Q (r x r), without updating
 * anything.  Host pointers; either may be NULL.  Synchronises. */
nmd_status nmd_block_terms(nmd_handle* h, int32_t side, int64_t block, int32_t kind, float* R,
                           float* G, int64_t* rows);

/* Verification hook: L = M Q^T, the first product of the tensor-core panel
 * kernel (eq. ABt restricted to one block), for the M-side rows and Q-side
 * rows of one block update, before any epilogue.  d_L: device memory of
 * rows x K floats (row-major), owned by the caller; rows and K are returned
 * in *rows and *cols when those are not NULL.  NMD_ERR_UNSUPPORTED for
 * NMD_SIMT.  Synchronises. */
nmd_status nmd_dense_products(nmd_handle* h, int32_t side, int64_t block, int32_t kind, float* d_L,
                              int64_t* rows, int64_t* cols);

/* Verification and timing hook: the support term of one block update alone
 * (the sparse correction of eqs. updateZ/updateD, Sec. 3.2): for every M-side
 * row i with support in the block's panel,
 *   Rs_i = sum over the panel's entries (i, k) of (S_ik - min(0, L_ik)) q_k,
 * with L_ik = m_i . q_k, and Rs_i = 0 on the other rows.  The step's own
 * operands are used: the bf16 pieces of both factors in the NMD_BF16 mode,
 * the fp32 masters otherwise.  d_R: caller-owned device memory of rows x
 * r_pad floats, row-major, r_pad = r rounded up to 16, 32, 64, 128 or 256;
 * *rows (if not NULL) receives the number of M-side rows.  Asynchronous on
 * the handle's stream (it first waits for any deferred update of a sweep),
 * so the caller can time it with events. */
nmd_status nmd_support_term(nmd_handle* h, int32_t side, int64_t block, int32_t kind, float* d_R, int64_t* rows);

/* Verification hook: the sparse traversal of one block update -- for every
 * M-side row with support in the block's panel, ascending, its entries in
 * ascending Q-side order.  Writes up to cap (row, q) index pairs to
 * rows_out/q_out (q relative to the block's first Q-side row) and the total
 * count to *count.  Pure host computation over the panel index. */
nmd_status nmd_panel_traversal(const nmd_handle* h, int32_t side, int64_t block, int32_t kind,
                               int64_t* rows_out, int64_t* q_out, int64_t cap, int64_t* count);

/* Checkpoint: factors W (m x r), H (r x n), momentum EW (m x r), EH (r x n)
 * and the sweep counter.  Host pointers.  nmd_get_state synchronises;
 * nmd_set_state is asynchronous (waits for its host copies). */
nmd_status nmd_get_state(nmd_handle* h, float* W, float* H, float* EW, float* EH,
                         int64_t* sweep_index);
nmd_status nmd_set_state(nmd_handle* h, const float* W, const float* H, const float* EW,
                         const float* EH, int64_t sweep_index);

/* Kernel timing with CUDA events recorded around each launch, on the stream
 * the launch goes to (inside nmd_sweep the library's own streams, which
 * overlap: class totals can add up to more than the elapsed time).
 * nmd_profile(h, 1) clears the totals and starts recording, nmd_profile(h, 0)
 * stops.  nmd_profile_read synchronises and returns the device time (ms) and
 * launch count accumulated for one kernel class: NMD_K_DENSE (the fused
 * Z-panel kernel), NMD_K_SPARSE (support correction), NMD_K_GRAM (Gram
 * matrix + inverse), NMD_K_UPDATE (least squares / momentum update),
 * NMD_K_LOSS (dense loss pass).  With the environment variable NMD_TRACE set
 * to a file name, the launches timed since the last read are also appended
 * to that file, one line "class start_ms end_ms" each, relative to the
 * first of them (a timeline across the streams). */
typedef enum { NMD_K_DENSE = 0, NMD_K_SPARSE = 1, NMD_K_GRAM = 2, NMD_K_UPDATE = 3, NMD_K_LOSS = 4 } nmd_kernel_class;
nmd_status nmd_profile(nmd_handle* h, int on);
nmd_status nmd_profile_read(nmd_handle* h, int32_t kernel_class, double* ms, int64_t* launches);

/* Gram matrix G = Q^T Q (r x r, row-major, written to d_G) of the K rows of a
 * caller's device matrix Q (row stride ld >= r floats), computed without any
 * device allocation and without a handle or workspace.  The paper has no
 * counterpart of this call; it exists for callers that cannot allocate
 * device memory at the point of the call -- code running inside a
 * framework or plugin that owns the whole device pool, or a real-time loop
 * that forbids cudaMalloc -- and so cannot provide the workspace that
 * nmd_create needs.  The partial sums go to a 2 MiB array in the library's
 * static device memory, which every GPU that loads the library holds until
 * the process exits.  Limits: r <= 128 (NMD_ERR_WORKSPACE beyond), K >= 1.
 * The first call on a device looks up that array's device address (with the
 * device current); make that first call before any stream capture.  All
 * calls share the array, so calls that overlap on the GPU (other streams,
 * other threads) race and must be serialised by the caller.  Asynchronous on
 * `stream` (a cudaStream_t, NULL = legacy default stream); the result equals
 * the Gram matrix of nmd_block_terms to fp32 rounding (summation order). */
nmd_status nmd_gram_noalloc(const float* d_Q, int64_t K, int32_t r, int64_t ld, float* d_G, void* stream);

/* Verification hook for failure detection: runs the bounded wait that every
 * pipeline wait of the tensor-core kernels uses (mbarrier polling with a
 * globaltimer limit, after which the kernel records NMD_ERR_TIMEOUT in the
 * sticky status, raises its abort flag and returns) on a barrier that nothing
 * arrives at, with a limit of limit_ns (1 us .. 1 s; the kernels use 2 s).
 * Synchronises; returns NMD_ERR_TIMEOUT when the wait gave up as designed
 * (the status is cleared, the handle stays usable), NMD_ERR_INVALID for a
 * limit out of range. */
nmd_status nmd_selftest_wait_timeout(nmd_handle* h, int64_t limit_ns);

/* Number of kernel launches this handle has issued (for launch accounting). */
int64_t nmd_launch_count(const nmd_handle* h);

/* Delta form (epilogue NMD_EPI_DELTA) with chunk skipping on: the number of
 * Q chunks (64 or 128 Q-side rows against a 128-row M tile) that the
 * tensor-core panel kernel skipped -- NMD_SKIP_VOTE: chunks whose second
 * product was skipped because max(0, L) was zero on the whole chunk;
 * NMD_SKIP_RANGE: chunks the range search cleared, both products skipped
 * (Sec. 4.3).  The first chunk of a tile is always computed under
 * NMD_SKIP_VOTE, and a tile with every chunk cleared computes its first
 * under NMD_SKIP_RANGE.  Counts since creation or the last reset;
 * synchronises; reset != 0 sets the count back to zero. */
nmd_status nmd_skip_count(nmd_handle* h, int64_t* skipped, int32_t reset);

/* Verification hook: the range-search mask of one block update (Sec. 4.3,
 * eq. range-search), computed from the current factors exactly as the step
 * would compute it under NMD_SKIP_RANGE, whatever the options say.  Writes
 * *ntiles (128-row M tiles), *words (32-bit words per tile), *chunk_rows
 * (Q-side rows per chunk) and, if mask != NULL and capacity >= ntiles x
 * words, the mask to host memory: word w of tile t at mask[t words + w],
 * bit c set = chunk 32 w + c is cleared (every L_ij of the tile's rows and
 * the chunk's rows is <= 0).  NMD_ERR_UNSUPPORTED for NMD_SIMT.
 * Synchronises. */
nmd_status nmd_range_mask(nmd_handle* h, int32_t side, int64_t block, int32_t kind, uint32_t* mask,
                          int64_t capacity, int64_t* ntiles, int64_t* words, int64_t* chunk_rows);

/* Cell embedding (Sec. 5.3, eqs. Lsvd and embed), for a square S (m = n:
 * rows and columns are the same cells) and r <= 128: with the model
 * L = W H = U Sigma V^T (its thin SVD, computed from the factors without
 * forming L), cell i is the unit vector
 *     xi_i = [u_i Sigma^{1/2}, v_i Sigma^{1/2}] / norm
 * of 2r elements (u_i, v_i the i-th rows of U and V; singular triples in
 * descending order; a triple is determined up to a common sign, which the
 * distances between cells do not see).  d_xi: device, n x 2r fp32 row-major,
 * caller-owned.  d_sigma: device, r fp32 (the singular values, descending) or
 * NULL.  Asynchronous on the handle's stream.  NMD_ERR_INVALID if m != n,
 * r > 128 or n < 6 r. */
nmd_status nmd_embed(nmd_handle* h, float* d_xi, float* d_sigma);

/* Device workspace (bytes) of nmd_nearest_neighbors for N points of d
 * coordinates (2 <= N < 2^31, 1 <= d <= 256). */
nmd_status nmd_nn_workspace_bytes(int64_t N, int32_t d, size_t* bytes);

/* Held-out one-nearest-neighbour search (Sec. 5.3): for each of the N points
 * (rows of d_x, N x d fp32 row-major, device), the other point j != i with the
 * largest inner product x_i . x_j -- for the unit vectors of nmd_embed the
 * nearest in Euclidean distance -- on the tensor cores (each coordinate as
 * three bf16 pieces, products accumulated in fp32: inner products good to
 * about 1e-5 of |x_i| |x_j|; ties and near-ties within that go to either
 * point, among exactly equal values to the smaller index).  d_nn: device,
 * N int32 (the neighbour); d_best: device, N fp32 (its inner product) or
 * NULL.  d_labels: device, N int32, or NULL; with labels and errors != NULL,
 * *errors = the number of points whose neighbour carries another label (the
 * 1-NN error count).  d_workspace: at least nmd_nn_workspace_bytes, 256-byte
 * aligned, caller-owned.  Synchronises the stream. */
nmd_status nmd_nearest_neighbors(const float* d_x, int64_t N, int32_t d, const int32_t* d_labels, int32_t* d_nn,
                                 float* d_best, int64_t* errors, void* d_workspace, size_t ws_bytes, void* stream);

const char* nmd_status_string(nmd_status s);
const char* nmd_last_error(const nmd_handle* h);
void nmd_destroy(nmd_handle* h);

#ifdef __cplusplus
}
#endif
#endif /* NMD_H */
