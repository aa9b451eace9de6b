// Small kernels of the block step: operand packing, Gram matrix, Gram
// inverse, sparse support correction, least-squares/momentum update, and the
// support part and final reduction of the loss.
#include <float.h>
#include <math.h>

#include <algorithm>

#include "nmd_internal.cuh"

namespace nmd {

namespace {

__device__ __forceinline__ void set_status(int* status, int code, int detail, int step) {
  if (atomicCAS(status, 0, code) == 0) {
    status[1] = detail;
    status[2] = step;
  }
}

inline int grid_for(int64_t work, int threads, int cap = 152 * 16) {
  int64_t g = (work + threads - 1) / threads;
  if (g < 1) g = 1;
  return (int)std::min<int64_t>(g, cap);
}

// ---------------------------------------------------------------------------
// Packing: fp32 (N x r, or r x N) -> N x rp master plus bf16 hi/lo split
// (hi = bf16_rn(x), lo = bf16_rn(x - hi)); pad columns are zero.
// ---------------------------------------------------------------------------
__global__ void pack_kernel(const float* __restrict__ src, int src_is_rxN, int64_t N, int r, int rp,
                            float* __restrict__ master, bf16* __restrict__ hi, bf16* __restrict__ lo) {
  int64_t total = N * rp;
  for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t j = idx / rp;
    int c = (int)(idx - j * rp);
    float v = 0.f;
    if (c < r) v = src_is_rxN ? src[(int64_t)c * N + j] : src[j * r + c];
    master[idx] = v;
    if (hi) {
      bf16 h = __float2bfloat16_rn(v);
      hi[idx] = h;
      if (lo) lo[idx] = __float2bfloat16_rn(v - __bfloat162float(h));
    }
  }
}

__global__ void unpack_kernel(const float* __restrict__ master, int dst_is_rxN, int64_t N, int r,
                              int rp, float* __restrict__ dst) {
  int64_t total = N * r;
  for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t j, c;
    if (dst_is_rxN) { c = idx / N; j = idx - c * N; }
    else { j = idx / r; c = idx - j * r; }
    dst[idx] = master[j * rp + c];
  }
}

// ---------------------------------------------------------------------------
// Gram matrix G = Q^T Q over Q-side rows [q0, q0+K): grid (tiles, parts).
// Tile (ta, tb), ta >= tb, of 64 x 64 entries; part p sums the rows
// [p*chunk, (p+1)*chunk) in ascending order.  The partials are summed in a
// fixed order by the inverse kernel, so the result is deterministic.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) gram_kernel(const float* __restrict__ Q, int64_t q0, int64_t K,
                                                   int rp, float* __restrict__ parts, int64_t chunk) {
  __shared__ float Qa[32][65];
  __shared__ float Qb[32][65];
  int nt = (rp + 63) / 64;
  int t = blockIdx.x, ta = 0;
  while (t >= ta + 1) { t -= ta + 1; ++ta; }
  int tb = t;
  int p = blockIdx.y;
  int64_t k0 = (int64_t)p * chunk, k1 = min(K, k0 + chunk);
  int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  float acc[4][4] = {};
  int wa = min(64, rp - ta * 64), wb = min(64, rp - tb * 64);
  for (int64_t kb = k0; kb < k1; kb += 32) {
    for (int e = threadIdx.x; e < 32 * 64; e += 256) {
      int rr = e / 64, cc = e % 64;
      int64_t k = kb + rr;
      bool ok = k < k1;
      Qa[rr][cc] = (ok && cc < wa) ? Q[(q0 + k) * rp + ta * 64 + cc] : 0.f;
      Qb[rr][cc] = (ok && cc < wb) ? Q[(q0 + k) * rp + tb * 64 + cc] : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int rr = 0; rr < 32; ++rr) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = Qa[rr][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Qb[rr][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  (void)nt;
  float* out = parts + (size_t)p * rp * rp;
  for (int i = 0; i < 4; ++i)
    for (int j = 0; j < 4; ++j) {
      int a = ta * 64 + ty * 4 + i, b = tb * 64 + tx * 4 + j;
      if (a < rp && b < rp) out[(size_t)a * rp + b] = acc[i][j];
    }
}

// ---------------------------------------------------------------------------
// G^{-1} by the symmetric sweep operator (Gauss-Jordan without pivoting, valid
// for symmetric positive definite G): sweeping pivot k maps
//   a_kk -> -1/a_kk, a_ik -> a_ik/a_kk, a_kj -> a_kj/a_kk,
//   a_ij -> a_ij - a_ik a_kj / a_kk  (i, j != k);
// after all r pivots the matrix holds -G^{-1}.  The pivots are the Schur
// complements (the squared Cholesky pivots); one that is not positive
// relative to the diagonal marks G as not positive definite.
// One thread block; the r x r matrix lives in shared memory when it fits.
// ---------------------------------------------------------------------------
constexpr int kCholThreads = 1024;

__global__ void __launch_bounds__(kCholThreads) ginv_kernel(const float* __restrict__ parts, int nparts,
                                                            int r, int rp, float ridge,
                                                            float* __restrict__ Gout,
                                                            float* __restrict__ Ginv,
                                                            float* __restrict__ scratch,
                                                            int* __restrict__ status, int use_smem) {
  extern __shared__ float sm[];
  float* A = use_smem ? sm : scratch;             // r x r
  __shared__ float rowk[256];
  __shared__ float diag0[256];
  __shared__ int bad;
  if (threadIdx.x == 0) bad = 0;
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) {
    int i = e / r, j = e % r;
    int a = max(i, j), b = min(i, j);             // lower triangle holds the partials
    float s = 0.f;
    for (int p = 0; p < nparts; ++p) s += parts[(size_t)p * rp * rp + (size_t)a * rp + b];
    if (i == j) s += ridge;
    A[e] = s;
    if (i == j) diag0[i] = s;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < rp * rp; e += blockDim.x) {
    int i = e / rp, j = e % rp;
    Gout[e] = (i < r && j < r) ? A[i * r + j] : 0.f;
  }
  const float tol = 4.0f * (float)r * FLT_EPSILON;
  for (int k = 0; k < r; ++k) {
    float d = A[k * r + k];
    if (!(d > tol * diag0[k]) || !isfinite(d)) {
      if (threadIdx.x == 0) {
        bad = 1;
        set_status(status, NMD_ERR_NOT_SPD, k, 0);
      }
      break;   // uniform: every thread reads the same d
    }
    for (int j = threadIdx.x; j < r; j += blockDim.x) rowk[j] = A[k * r + j];
    __syncthreads();
    float inv = 1.0f / d;
    for (int e = threadIdx.x; e < r * r; e += blockDim.x) {
      int i = e / r, j = e % r;
      float v;
      if (i == k && j == k) v = -inv;
      else if (i == k) v = rowk[j] * inv;
      else if (j == k) v = rowk[i] * inv;                 // symmetric: a_ik = a_ki
      else v = A[e] - rowk[i] * rowk[j] * inv;
      A[e] = v;
    }
    __syncthreads();
  }
  __syncthreads();
  for (int e = threadIdx.x; e < rp * rp; e += blockDim.x) {
    int i = e / rp, j = e % rp;
    float v = 0.f;
    if (!bad && i < r && j < r) v = -0.5f * (A[i * r + j] + A[j * r + i]);   // symmetrise
    Ginv[e] = v;
  }
}

// ---------------------------------------------------------------------------
// Sparse correction: for every panel row i and entry (i, k) in the block,
// L_ik = m_i . q_k (the operands of the dense pass), c = S_ik - min(0, L_ik),
// R_i += c q_k.  One warp per light row; entries are visited in ascending k.
// ---------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ float ld(const T* p);
template <>
__device__ __forceinline__ float ld<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld<bf16>(const bf16* p) { return __bfloat162float(*p); }

template <typename T, int VPL>
__global__ void __launch_bounds__(256) sparse_light_kernel(const PanelRow* __restrict__ rows, int64_t nrows,
                                                           const T* __restrict__ Mop, int64_t m0,
                                                           const T* __restrict__ Qop,
                                                           const int32_t* __restrict__ qidx,
                                                           const float* __restrict__ vals,
                                                           float* __restrict__ R, int rp) {
  int lane = threadIdx.x & 31;
  int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (; w < nrows; w += nw) {
    PanelRow pr = rows[w];
    int64_t i = pr.row;
    float mv[VPL], acc[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      int c = lane + 32 * v;
      mv[v] = c < rp ? ld<T>(Mop + i * rp + c) : 0.f;
      acc[v] = 0.f;
    }
    for (int64_t e = pr.beg; e < pr.beg + pr.len; ++e) {
      int64_t k = qidx[e];
      float s = vals[e];
      float qv[VPL];
      float part = 0.f;
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        int c = lane + 32 * v;
        qv[v] = c < rp ? ld<T>(Qop + k * rp + c) : 0.f;
        part = fmaf(mv[v], qv[v], part);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      float cval = s - fminf(0.f, part);
#pragma unroll
      for (int v = 0; v < VPL; ++v) acc[v] = fmaf(cval, qv[v], acc[v]);
    }
    float* Ri = R + (i - m0) * rp;
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      int c = lane + 32 * v;
      if (c < rp) Ri[c] += acc[v];
    }
  }
}

// Heavy rows: one thread block (16 warps) per row; warp w takes entries
// beg + w, beg + w + 16, ...; the 16 partial sums are added in warp order.
template <typename T, int VPL>
__global__ void __launch_bounds__(512) sparse_heavy_kernel(const PanelRow* __restrict__ rows,
                                                           const T* __restrict__ Mop, int64_t m0,
                                                           const T* __restrict__ Qop,
                                                           const int32_t* __restrict__ qidx,
                                                           const float* __restrict__ vals,
                                                           float* __restrict__ R, int rp) {
  __shared__ float part_sm[16][256];
  int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  PanelRow pr = rows[blockIdx.x];
  int64_t i = pr.row;
  float mv[VPL], acc[VPL];
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    int c = lane + 32 * v;
    mv[v] = c < rp ? ld<T>(Mop + i * rp + c) : 0.f;
    acc[v] = 0.f;
  }
  for (int64_t e = pr.beg + wid; e < pr.beg + pr.len; e += 16) {
    int64_t k = qidx[e];
    float s = vals[e];
    float qv[VPL];
    float part = 0.f;
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      int c = lane + 32 * v;
      qv[v] = c < rp ? ld<T>(Qop + k * rp + c) : 0.f;
      part = fmaf(mv[v], qv[v], part);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    float cval = s - fminf(0.f, part);
#pragma unroll
    for (int v = 0; v < VPL; ++v) acc[v] = fmaf(cval, qv[v], acc[v]);
  }
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    int c = lane + 32 * v;
    if (c < 256) part_sm[wid][c] = acc[v];
  }
  __syncthreads();
  for (int c = threadIdx.x; c < rp; c += blockDim.x) {
    float s = 0.f;
    for (int w = 0; w < 16; ++w) s += part_sm[w][c];
    R[(i - m0) * rp + c] += s;
  }
}

// ---------------------------------------------------------------------------
// Update of the M-side rows: X = R G^{-1};
//   Z form:     U = eta (X - M)      (eqs. lsqA/lsqB with step size)
//   Delta form: U = eta X            (eqs. spLsqA/spLsqB)
// then E = U + gamma E (stochastic steps) and M += E, refreshing the bf16
// hi/lo copies.  Skipped entirely while a sticky error is set.
// ---------------------------------------------------------------------------
template <int RP>
__global__ void __launch_bounds__(256) update_kernel(float* __restrict__ M, bf16* __restrict__ Mhi,
                                                     bf16* __restrict__ Mlo, float* __restrict__ E,
                                                     int64_t m0, int64_t rows,
                                                     const float* __restrict__ R,
                                                     const float* __restrict__ Ginv, float eta,
                                                     float gamma, int momentum, int delta_form,
                                                     int* __restrict__ status) {
  static_assert(RP >= 16 && RP <= 256, "padded rank");
  constexpr bool kSmemG = RP <= 128;
  constexpr int ROWS = 256 / RP;                      // rows per pass; one (row, column) per thread
  __shared__ float Gs[kSmemG ? RP * RP : 1];
  __shared__ float Rs[ROWS][RP];
  if (*(volatile int*)status != 0) return;
  if (kSmemG)
    for (int e = threadIdx.x; e < RP * RP; e += blockDim.x) Gs[e] = Ginv[e];
  const int c = threadIdx.x % RP;
  const int rsub = threadIdx.x / RP;
  for (int64_t base = (int64_t)blockIdx.x * ROWS; base < rows; base += (int64_t)gridDim.x * ROWS) {
    __syncthreads();
    for (int e = threadIdx.x; e < ROWS * RP; e += blockDim.x) {
      int64_t li = base + e / RP;
      Rs[e / RP][e % RP] = li < rows ? R[li * RP + (e % RP)] : 0.f;
    }
    __syncthreads();
    int64_t li = base + rsub;
    if (li >= rows) continue;
    float x = 0.f;
#pragma unroll 8
    for (int k = 0; k < RP; ++k)
      x = fmaf(Rs[rsub][k], kSmemG ? Gs[k * RP + c] : __ldg(Ginv + k * RP + c), x);
    int64_t gi = (m0 + li) * RP + c;
    float mold = M[gi];
    float u = delta_form ? eta * x : eta * (x - mold);
    float e = momentum ? fmaf(gamma, E[gi], u) : u;
    if (momentum) E[gi] = e;
    float mnew = mold + e;
    if (!isfinite(mnew)) set_status(status, NMD_ERR_DIVERGED, (int)(m0 + li), 0);
    M[gi] = mnew;
    bf16 h = __float2bfloat16_rn(mnew);
    Mhi[gi] = h;
    Mlo[gi] = __float2bfloat16_rn(mnew - __bfloat162float(h));
  }
}

// ---------------------------------------------------------------------------
// Loss, support part: for every stored (i, j), with L = w_i . b_j and
// Shat = max(0, L):
//   a = (S - L)^2 - Shat^2          (objective correction, eq. SLloss)
//   b = (S - Shat)^2 - Shat^2       (RMSE correction)
//   mn = min(S, Shat), mx = max(S, Shat) - Shat   (WJD sums)
// One warp per row of S (fixed assignment), fp64 sums, per-block partials.
// ---------------------------------------------------------------------------
template <typename T, int VPL>
__global__ void __launch_bounds__(256) loss_sparse_kernel(const int64_t* __restrict__ rowptr,
                                                          const int32_t* __restrict__ col,
                                                          const float* __restrict__ val, int64_t m,
                                                          const T* __restrict__ Wop,
                                                          const T* __restrict__ Bop, int rp,
                                                          double* __restrict__ parts) {
  __shared__ double red[8][4];
  int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  double sa = 0, sb = 0, smn = 0, smx = 0;
  int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; i < m; i += nw) {
    float wv[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      int c = lane + 32 * v;
      wv[v] = c < rp ? ld<T>(Wop + i * rp + c) : 0.f;
    }
    for (int64_t e = rowptr[i]; e < rowptr[i + 1]; ++e) {
      int64_t j = col[e];
      float part = 0.f;
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        int c = lane + 32 * v;
        float b = c < rp ? ld<T>(Bop + j * rp + c) : 0.f;
        part = fmaf(wv[v], b, part);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      if (lane == 0) {
        double L = part, S = val[e];
        double sh = L > 0 ? L : 0.0;
        sa += (S - L) * (S - L) - sh * sh;
        sb += (S - sh) * (S - sh) - sh * sh;
        smn += S < sh ? S : sh;
        smx += (S > sh ? S : sh) - sh;
      }
    }
  }
  if (lane == 0) {
    red[wid][0] = sa; red[wid][1] = sb; red[wid][2] = smn; red[wid][3] = smx;
  }
  __syncthreads();
  if (threadIdx.x < 4) {
    double s = 0;
    for (int w = 0; w < 8; ++w) s += red[w][threadIdx.x];
    parts[(size_t)blockIdx.x * 8 + threadIdx.x] = s;
  }
}

// Fixed-order reduction of the loss partials:
// out = [sum relu^2, sum relu, sum a, sum b, sum mn, sum mx].
__global__ void loss_final_kernel(const double* __restrict__ dparts, int nd,
                                  const double* __restrict__ sparts, int ns, double* __restrict__ out) {
  __shared__ double red[256];
  for (int q = 0; q < 6; ++q) {
    const double* src = q < 2 ? dparts : sparts;
    int n = q < 2 ? nd : ns;
    int off = q < 2 ? q : q - 2;
    double s = 0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) s += src[(size_t)i * 8 + off];
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
      if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
      __syncthreads();
    }
    if (threadIdx.x == 0) out[q] = red[0];
    __syncthreads();
  }
}

}  // namespace

// ===========================================================================
// launchers
// ===========================================================================
void launch_pack(const float* src, bool src_is_rxN, int64_t N, int r, int rp, Factor& f, cudaStream_t s) {
  pack_kernel<<<grid_for(N * rp, 256), 256, 0, s>>>(src, src_is_rxN, N, r, rp, f.master, f.hi, f.lo);
}

void launch_unpack(const float* master, bool dst_is_rxN, int64_t N, int r, int rp, float* dst, cudaStream_t s) {
  unpack_kernel<<<grid_for(N * r, 256), 256, 0, s>>>(master, dst_is_rxN, N, r, rp, dst);
}

void launch_gram(const Factor& fq, int64_t q0, int64_t K, int r, int rp, float* parts, int nparts,
                 cudaStream_t s) {
  (void)r;
  int nt = (rp + 63) / 64;
  int64_t chunk = (K + nparts - 1) / nparts;
  chunk = (chunk + 31) / 32 * 32;
  dim3 grid(nt * (nt + 1) / 2, nparts);
  gram_kernel<<<grid, 256, 0, s>>>(fq.master, q0, K, rp, parts, chunk);
}

void launch_chol_inv(const float* parts, int nparts, int r, int rp, float ridge, float* G, float* Ginv,
                     float* scratch, int* status, cudaStream_t s) {
  size_t smem = (size_t)r * r * sizeof(float);
  int use_smem = smem <= 200 * 1024;
  if (use_smem && smem > 48 * 1024)
    cudaFuncSetAttribute(ginv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  ginv_kernel<<<1, kCholThreads, use_smem ? smem : 0, s>>>(parts, nparts, r, rp, ridge, G, Ginv, scratch,
                                                           status, use_smem);
}

template <typename T>
static void sparse_dispatch(const StepArgs& a, const T* Mop, const T* Qop, const PanelRow* light,
                            int64_t nlight, const PanelRow* heavy, int64_t nheavy, const int32_t* qidx,
                            const float* vals, float* R, cudaStream_t s) {
  // panel rows and qidx hold absolute M-side / Q-side row indices
  int g = grid_for(nlight * 32, 256, 152 * 64);
#define NMD_SP(V)                                                                                     \
  do {                                                                                                \
    if (nlight > 0)                                                                                   \
      sparse_light_kernel<T, V><<<g, 256, 0, s>>>(light, nlight, Mop, a.m0, Qop, qidx, vals, R, a.rp); \
    if (nheavy > 0)                                                                                   \
      sparse_heavy_kernel<T, V><<<(unsigned)nheavy, 512, 0, s>>>(heavy, Mop, a.m0, Qop, qidx, vals, R, \
                                                                  a.rp);                              \
  } while (0)
  switch (a.rp) {
    case 16: case 32: NMD_SP(1); break;
    case 64: NMD_SP(2); break;
    case 128: NMD_SP(4); break;
    default: NMD_SP(8); break;
  }
#undef NMD_SP
}

// The support correction always reads the fp32 masters, in every precision:
// on rows with few support entries the term S_ik q_k dominates R_i and is not
// averaged over many products, so rounding q_k to bf16 there would put its
// full relative error (up to 2^-9) into the update.
void launch_sparse(const StepArgs& a, const PanelRow* light, int64_t nlight, const PanelRow* heavy,
                   int64_t nheavy, const int32_t* qidx, const float* vals, float* R, cudaStream_t s) {
  sparse_dispatch<float>(a, a.fm->master, a.fq->master, light, nlight, heavy, nheavy, qidx, vals, R, s);
}

void launch_update(const StepArgs& a, const float* R, const float* Ginv, float eta, float gamma,
                   bool momentum, int* status, cudaStream_t s) {
  const Factor& f = *a.fm;
  int rows_per_pass = 256 / std::min(a.rp, 256);
  int g = grid_for(a.M, rows_per_pass, 152 * 8);
#define NMD_UP(RP)                                                                                   \
  update_kernel<RP><<<g, 256, 0, s>>>(f.master, f.hi, f.lo, f.E, a.m0, a.M, R, Ginv, eta, gamma,      \
                                      momentum, a.epilogue == NMD_EPI_DELTA, status)
  switch (a.rp) {
    case 16: NMD_UP(16); break;
    case 32: NMD_UP(32); break;
    case 64: NMD_UP(64); break;
    case 128: NMD_UP(128); break;
    default: NMD_UP(256); break;
  }
#undef NMD_UP
}

void launch_loss_sparse(const nmd_handle* h, double* parts, int nparts, cudaStream_t s) {
  bool bf = h->opt.precision == NMD_BF16;
#define NMD_LS(T, V, WP, BP) \
  loss_sparse_kernel<T, V><<<nparts, 256, 0, s>>>(h->ws.rowptr, h->ws.col, h->ws.val, h->m, WP, BP, h->rp, parts)
#define NMD_LSV(V)                                                   \
  do {                                                               \
    if (bf) NMD_LS(bf16, V, h->W.hi, h->B.hi);                       \
    else NMD_LS(float, V, h->W.master, h->B.master);                 \
  } while (0)
  switch (h->rp) {
    case 16: case 32: NMD_LSV(1); break;
    case 64: NMD_LSV(2); break;
    case 128: NMD_LSV(4); break;
    default: NMD_LSV(8); break;
  }
#undef NMD_LSV
#undef NMD_LS
}

void launch_loss_final(const double* dparts, int nd, const double* sparts, int ns, double* out, cudaStream_t s) {
  loss_final_kernel<<<1, 256, 0, s>>>(dparts, nd, sparts, ns, out);
}

}  // namespace nmd
