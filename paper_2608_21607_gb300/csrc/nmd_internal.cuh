// Internal declarations shared by the translation units of libnmd.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <atomic>
#include <string>
#include <vector>

#include "../../include/nmd.h"

namespace nmd {

typedef __nv_bfloat16 bf16;

// Kernel attributes (cudaFuncSetAttribute) and occupancy figures belong to a
// device, so the host code caches them per device ordinal: slot[d] holds the
// value f() returned with device d current (0 = not yet computed; f returns
// a positive value, or 0 when it failed and should run again next time).
constexpr int kMaxDevices = 64;
template <class F>
int per_device(std::atomic<int> (&slot)[kMaxDevices], F f) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return f();
  int v = slot[dev].load(std::memory_order_acquire);
  if (v == 0) {
    v = f();
    if (v > 0) slot[dev].store(v, std::memory_order_release);
  }
  return v;
}

// One row of a block's sparse panel: entries [beg, beg + len) of the CSR (or
// CSC) arrays, all belonging to M-side row `row` and lying in the block's
// Q-side range.  Rows are listed in ascending order.
struct PanelRow {
  int32_t row;
  int32_t len;
  int64_t beg;
};

// Panel rows of at most kShort entries go to the grouped short-row kernel (a
// few lanes per row).  Longer rows go to a kernel that puts the lanes over
// the entries, in segments of at most `seg` entries (chosen per block): a row
// of at most `seg` entries is one segment that writes its result directly; a
// longer row is cut into slices of `seg` entries, each slice's partial sum
// goes to a scratch slot and the slots of a row are added in a fixed order by
// a second pass.  `seg` is kSegMax when the block's long rows give enough
// segments to fill the GPU (rows of ~100 entries in a dense-ish panel), and
// shrinks to kSegMin otherwise (the few hubs of a power-law graph, each up to
// a whole block long, are then spread over many warps).
constexpr int kShort = 32;
constexpr int kSegMax = 128;
constexpr int kSegMin = 32;
constexpr int64_t kSegTarget = 4096;   // segments a block's long rows should give

// Per (side, kind): the panel lists of every block, concatenated.  For block k:
//   short rows    [row_ptr[k], row_ptr[k+1])   of `host`/`d`   (len <= kShort)
//   segments      [seg_ptr[k], seg_ptr[k+1])   of `seg`: first the segd[k]
//                 whole rows of kShort < len <= seg, then the slices of `seg`
//                 entries of the longer rows
//   split rows    [multi_ptr[k], multi_ptr[k+1]) of `multi`    (row, #segments,
//                 first slice relative to the block's slices)
// Rows are listed in ascending order.
struct PanelSet {
  std::vector<int64_t> row_ptr, seg_ptr, multi_ptr, segd;
  std::vector<PanelRow> host, seg, multi;
  PanelRow* d = nullptr;
  PanelRow* d_seg = nullptr;
  PanelRow* d_multi = nullptr;
  int64_t max_segments = 0;     // largest segment count of any block
  // per block, one byte per M-side row of the step: 1 if the row has support
  // entries in the panel (its row of Rs is written by the step), else 0
  std::vector<int64_t> flag_off;
  std::vector<uint8_t> flags;
  uint8_t* d_flags = nullptr;
};

// Device status word (sticky): [0] = nmd_status code of the first error,
// [1] = a detail (pivot column, row index), [2] = step counter at the error.
constexpr int kStatusWords = 4;

// One factor's device buffers (N rows, rp = padded rank columns).
struct Factor {
  int64_t rows = 0;
  float* master = nullptr;   // N x rp fp32, pad columns are zero
  bf16* hi = nullptr;        // N x rp, bf16(master)
  bf16* lo = nullptr;        // N x rp, bf16(master - hi)
  bf16* lo2 = nullptr;       // N x rp, bf16(master - hi - lo)
  float* E = nullptr;        // N x rp momentum (fp32)
};

// Operands of one dense panel contraction and one update, in device memory.
struct StepArgs {
  // M-side rows [m0, m0 + M) of factor fm, Q-side rows [q0, q0 + K) of fq
  const Factor* fm;
  const Factor* fq;
  int64_t m0, M, q0, K;
  int r, rp;
  int precision, epilogue;
  int num_sms = 152;         // streaming multiprocessors of the device (grid sizing)
  bool skip_zero = false;    // Delta form: skip chunks whose rectified tile is zero
  // Delta form, range search: per 128-row M tile, `rwords` words whose bit c
  // marks Q chunk c as all L <= 0 (both dense products skipped); or nullptr
  const uint32_t* rmask = nullptr;
  int64_t rwords = 0;
};

struct Workspace {
  size_t bytes = 0;
  // CSR of S and CSR of S^T (=CSC of S), support only
  int64_t* rowptr = nullptr;
  int32_t* col = nullptr;
  float* val = nullptr;
  int64_t* colptr = nullptr;
  int32_t* row = nullptr;
  float* valT = nullptr;
  // panel lists: [side][kind]
  PanelRow* panels = nullptr;
  // R, G and G^{-1} exist twice: step t uses copy t % 2, so that the tail of
  // step t's update can still read its copy while step t + 1 runs
  float* R = nullptr;          // max(m, n) x rp fp32 right-hand side / staging
  float* R2 = nullptr;         // second copy of R
  // the support term of R (sparse correction): written by the sparse kernels
  // on the rows with support in the step's panel (the others are not read),
  // added to R by the update; two copies like R
  float* Rs = nullptr;
  float* Rs2 = nullptr;
  float* gram_part = nullptr;  // kGramParts x rp x rp
  float* G = nullptr;          // rp x rp (Gram, for verification)
  float* Ginv = nullptr;       // rp x rp
  float* G2 = nullptr;
  float* Ginv2 = nullptr;
  float* Gc = nullptr;         // G and G^{-1} of an exact step's Q side (all of one factor),
  float* Ginvc = nullptr;      // kept while that factor is unchanged
  float* Gx = nullptr;         // rp x rp: the exact G of a bf16-mode step (verification hook)
  float* Tm = nullptr;         // rp x rp: scratch of the verification hook
  double* loss_part = nullptr; // kLossParts x 8
  double* loss_out = nullptr;  // 8
  int* status = nullptr;       // kStatusWords
  int* counters = nullptr;     // 64 ints; ints 0-1: skipped Delta-form chunks (u64)
  float* seg_partials = nullptr;  // max segments x rp (sparse correction of long rows)
  uint8_t* flags = nullptr;       // the panels' support-row flags, concatenated
  float* rpart = nullptr;         // kRpartRows x rp: partial R's of split-K steps
  // range search (Delta form): balls of the M tiles and Q chunks of a step
  // (centres rp floats each, radii) and the skip mask of its (tile, chunk) pairs
  float* ball_m = nullptr;        // ceil(max(m, n) / 128) x rp
  float* rad_m = nullptr;
  float* ball_q = nullptr;        // ceil(max(m, n) / 64) x rp
  float* rad_q = nullptr;
  uint32_t* rmask = nullptr;      // range_mask_words(m, n)
  // the bf16 pieces of G^{-1}, G2^{-1} and the cached G^{-1} of exact steps
  // (rp rows each), for the tensor-core update at r_pad = 256
  Factor gi[3];
  // the same three, transposed, for the update's tensor-core product at
  // r_pad <= 128 in the bf16 mode: hi then lo, rp rows of split_stride(rp)
  // each, written by the G^{-1} kernels
  bf16* gsplit[3] = {nullptr, nullptr, nullptr};
};

// row stride (bf16 elements) of a transposed, split G^{-1}: 8 past r_pad, so
// that the rows start 16-byte aligned and the fragment loads of a half warp
// fall in 16 different bank pairs
constexpr int split_stride(int rp) { return rp + 8; }

constexpr int kGramParts = 64;
constexpr int64_t kRpartRows = 256 * 128;   // splits x tiles x 128 rows never exceed 256 SMs' worth
constexpr int kLossParts = 2048;

}  // namespace nmd

struct nmd_handle {
  int64_t m = 0, n = 0, nnz = 0;
  int r = 0, rp = 0;
  nmd_options opt;
  cudaStream_t stream = nullptr;
  // the Gram chain (G, G^{-1}) and the support term run on two more streams,
  // forked from and joined back into `stream` around the dense kernel of
  // each step
  cudaStream_t side = nullptr, side2 = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr, ev_join2 = nullptr;
  // Within a sweep, the rows of a step's update that the next step does not
  // read are updated on `aux`, overlapping the next step.  pend[f] records,
  // for factor f (0 = W, 1 = B), the rows such an update may still be
  // writing and the event that marks its end.
  cudaStream_t aux = nullptr;   // lowest priority
  // a sweep runs on `hp` (highest priority, forked from and joined back into
  // `stream`), so that the next step's kernels are scheduled ahead of the
  // deferred updates; `cur` is the stream the current call issues to
  cudaStream_t hp = nullptr;
  cudaStream_t cur = nullptr;
  cudaEvent_t ev_in = nullptr, ev_out = nullptr;
  cudaEvent_t ev_prio = nullptr;
  struct Pending {
    bool active = false;
    int64_t step = 0;
    int64_t a0 = 0, a1 = 0, b0 = 0, b1 = 0;   // rows [a0, a1) and [b0, b1) in flight
    cudaEvent_t ev = nullptr;
  } pend[2];
  // version of each factor (0 = W, 1 = B), advanced by every write to it, and
  // the factor and version the cached exact-step Gram belongs to
  int64_t fver[2] = {0, 0};
  int gcache_f = -1;
  int64_t gcache_ver = -1;
  float* cur_R = nullptr;      // the copies of R, Rs and G the last step used
  float* cur_Rs = nullptr;
  const uint8_t* cur_flags = nullptr;   // the support-row flags of the last step
  float* cur_G = nullptr;
  float* cur_Ginv = nullptr;   // the inverse the last step's update applied
  nmd::Workspace ws;
  nmd::Factor W, B;            // A = W (m x r), B = H^T (n x r)
  nmd::PanelSet panels[2][2];  // [side][kind]
  double s_fro = 0.0;
  int64_t sweep_index = 0;
  int64_t step_index = 0;
  int64_t launches = 0;
  int num_sms = 0;
  int device = 0;
  int cc_major = 0, cc_minor = 0;
  std::string last_error;
  // kernel timing (nmd_profile): event pairs per launch, by kernel class
  bool profiling = false;
  std::vector<cudaEvent_t> event_pool;
  struct Timed { int cls; cudaEvent_t a, b; };  // a, b recorded on the stream the class runs on
  std::vector<Timed> timed;
  double prof_ms[5] = {0, 0, 0, 0, 0};
  int64_t prof_launches[5] = {0, 0, 0, 0, 0};
  ~nmd_handle();
};

namespace nmd {

// ---- launchers (kernels.cu) ----
void launch_pack(const float* src, bool src_is_rxN, int64_t N, int r, int rp, Factor& f,
                 cudaStream_t s);
void launch_unpack(const float* master, bool dst_is_rxN, int64_t N, int r, int rp, float* dst,
                   cudaStream_t s);
// G = Q^T Q of the Q-side rows [q0, q0 + K) (+ ridge on the diagonal) via
// nparts fixed-order partials of `chunk` rows; rounded: of their bf16 pieces
// (hi) instead of the fp32 masters.
void launch_gram(const Factor* fq, bool rounded, int64_t q0, int64_t K, int r, int rp, float* parts, int nparts,
                 int64_t chunk, float ridge, float* G, cudaStream_t s);
// Ginv = G^{-1} through the Cholesky (L D L^T) factorisation; NMD_ERR_NOT_SPD
// in the status words on failure
// G^{-1} (rp x rp, row-major); with gsplit also its hi and lo bf16 pieces,
// transposed (gsplit[n * split_stride(rp) + k] = hi(G^{-1}[k][n]), lo at
// gsplit + rp * split_stride(rp)), pad entries zero
void launch_chol_inv(const float* G, int r, int rp, float* Ginv, bf16* gsplit, int* status, cudaStream_t s);
// C = A B (row-major fp32, M x K times K x N, N and K <= 256)
void launch_small_gemm(const float* A, int64_t lda, const float* B, int64_t ldb, float* C, int64_t ldc, int64_t M,
                       int N, int K, cudaStream_t s);
// rows: short rows; whole: the whole rows of the long-row kernel; seg: the
// slices of the split rows, summed per row of `multi` into R
// (bf16 mode: the factors' hi pieces, else the fp32 masters)
// returns the number of kernels launched
int launch_sparse(const StepArgs& a, const PanelRow* rows, int64_t nrows, const PanelRow* whole,
                   int64_t nwhole, const PanelRow* seg, int64_t nseg, const PanelRow* multi, int64_t nmulti,
                   const int32_t* qidx, const float* vals, float* R, float* partials, int64_t seg_first,
                   cudaStream_t s);
// flags: one byte per row of the step (Rs is read only where it is nonzero)
// gsplit: G^{-1}'s pieces as written by launch_chol_inv (read by the bf16
// mode's tensor-core product at r_pad <= 128)
void launch_update(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags,
                   const float* Ginv, const bf16* gsplit, float eta, float gamma, bool momentum, int* status,
                   cudaStream_t s);
void launch_combine(float* R, const float* Rs, const uint8_t* flags, int64_t rows, int rp, cudaStream_t s);
// the bounded pipeline wait, run on a barrier that never completes
void launch_wait_selftest(int* status, uint64_t limit_ns, cudaStream_t s);
void launch_loss_sparse(const nmd_handle* h, double* parts, int nparts, cudaStream_t s);
void launch_loss_final(const double* dense_parts, int ndense, const double* sparse_parts,
                       int nsparse, double* out, cudaStream_t s);

// ---- dense contraction on the CUDA cores (panel_simt.cu) ----
void launch_panel_simt(const StepArgs& a, float* R, cudaStream_t s);
int launch_loss_dense_simt(const nmd_handle* h, double* parts, int maxparts, cudaStream_t s);

// ---- dense contraction on the tcgen05 tensor cores (panel_tc.cu) ----
// Returns NMD_OK, or NMD_ERR_UNSUPPORTED when no tensor-core kernel exists
// for this rank; `launches` is incremented by the number of kernels issued.
// rpart (rpart_rows x rp floats, or nullptr): scratch for the partial R's of
// a step whose K is split because it has fewer tiles than SMs
nmd_status launch_panel_tc(const StepArgs& a, float* R, int* status, int* counter,
                           int num_sms, cudaStream_t s, int64_t* launches, float* Lout = nullptr,
                           float* rpart = nullptr, int64_t rpart_rows = 0);
nmd_status launch_loss_dense_tc(const nmd_handle* h, double* parts, int maxparts, int* nparts,
                                int* status, cudaStream_t s, int64_t* launches);
bool tc_supported(int rp, int precision);
// The nearest-neighbour pass of the tensor-core kernel over one point set
// (rows [0, N) of f, all three bf16 pieces packed): per row the largest
// inner product with another row, as an orderable key (zeroed by the caller)
nmd_status launch_nearest_tc(const Factor& f, int64_t N, int rp, unsigned long long* keys, int* status,
                             int num_sms, cudaStream_t s);
// The cell embedding (Sec. 5.3): G_A = W^T W and G_B = B^T B into GA, GB,
// their eigendecompositions and the SVD of the r x r core (scratch: six
// r x r matrices), T_A, T_B (r x r), sigma (r) and the n x 2r rows xi.
int embed_max_rank();
nmd_status launch_embed(const Factor& W, const Factor& B, int64_t n, int r, int rp, float* gram_part, float* GA,
                        float* GB, float* scratch, float* TA, float* TB, float* sigma, float* xi, int num_sms,
                        cudaStream_t s, int64_t* launches);
// The update on the tensor cores (bf16 mode, r_pad = 256): X = (R + Rs)
// G^{-1} by the update pass of the dense kernel, R and G^{-1} in two bf16
// pieces each (gi: the pieces of G^{-1}, rp rows), the step applied to rows
// [a.m0, a.m0 + a.M) of a.fm in its epilogue
nmd_status launch_update_tc(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags,
                            const Factor& gi, float eta, float gamma, bool momentum, int* status, int num_sms,
                            cudaStream_t s);
// Q-side rows per chunk of the tensor-core dense kernel (64 or 128)
int panel_chunk_rows(int rp, int precision);
// balls of the 128-row M tiles of rows [m0, m0 + M) of Xm and of the bn-row
// Q chunks of rows [q0, q0 + K) of Xq (one launch)
void launch_range_balls(const float* Xm, int64_t m0, int64_t M, const float* Xq, int64_t q0, int64_t K, int bn,
                        int rp, float* cm, float* rm, float* cq, float* rq, cudaStream_t s);
void launch_range_mask(const float* cm, const float* rm, int64_t ntiles, const float* cq, const float* rq,
                       int64_t nchunks, int64_t words, int rp, uint32_t* mask, cudaStream_t s);

}  // namespace nmd
