// Small kernels of the block step: operand packing, Gram matrix, Cholesky
// factor and inverse of the Gram matrix, sparse support correction,
// least-squares/momentum update, and the support part and final reduction of
// the loss.
#include <float.h>
#include <math.h>

#include <algorithm>
#include <atomic>

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
// Packing: fp32 (N x r, or r x N) -> N x rp master plus its bf16 pieces
// hi = bf16_rn(x), lo = bf16_rn(x - hi), lo2 = bf16_rn(x - hi - lo) (each
// difference is exact in fp32); pad columns are zero.
// ---------------------------------------------------------------------------
__global__ void pack_kernel(const float* __restrict__ src, int src_is_rxN, int64_t N, int r, int rp,
                            float* __restrict__ master, bf16* __restrict__ hi, bf16* __restrict__ lo,
                            bf16* __restrict__ lo2) {
  int64_t total = N * rp;
  for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    int64_t j = idx / rp;
    int c = (int)(idx - j * rp);
    float v = 0.f;
    if (c < r) v = src_is_rxN ? src[(int64_t)c * N + j] : src[j * r + c];
    master[idx] = v;
    if (hi) {
      const bf16 h = __float2bfloat16_rn(v);
      const float r1 = v - __bfloat162float(h);
      const bf16 l = __float2bfloat16_rn(r1);
      hi[idx] = h;
      lo[idx] = l;
      lo2[idx] = __float2bfloat16_rn(r1 - __bfloat162float(l));
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
// fixed order by gram_reduce_kernel, so the result is deterministic.  T is
// the element type of the rows read: float (the fp32 masters) or bf16 (the
// hi pieces, for the Gram matrix of the bf16-rounded rows).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }

template <typename T>
__global__ void __launch_bounds__(256, 4) gram_kernel(const T* __restrict__ Q, int64_t q0, int64_t K, int rp,
                                                      float* __restrict__ parts, int64_t chunk) {
  __shared__ float Qa[32][65];
  __shared__ float Qb[32][65];
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
      Qa[rr][cc] = (ok && cc < wa) ? to_f(Q[(q0 + k) * rp + ta * 64 + cc]) : 0.f;
      if (ta != tb) Qb[rr][cc] = (ok && cc < wb) ? to_f(Q[(q0 + k) * rp + tb * 64 + cc]) : 0.f;
    }
    __syncthreads();
    const float(*Qs)[65] = ta != tb ? Qb : Qa;   // a diagonal tile reads one copy
#pragma unroll 4
    for (int rr = 0; rr < 32; ++rr) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = Qa[rr][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Qs[rr][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* out = parts + (size_t)p * rp * rp;
  for (int i = 0; i < 4; ++i)
    for (int j = 0; j < 4; ++j) {
      int a = ta * 64 + ty * 4 + i, b = tb * 64 + tx * 4 + j;
      if (a < rp && b < rp) out[(size_t)a * rp + b] = acc[i][j];
    }
}

// G = the partials summed in part order (eight interleaved sums, added in a
// fixed tree), + ridge on the diagonal, written to both triangles from the
// lower one (the partials hold every entry whose 64-row tile is at or below
// its 64-column tile); pad rows and columns (>= r) are zero.  One thread per
// entry.
__global__ void __launch_bounds__(256) gram_reduce_kernel(const float* __restrict__ parts, int nparts, int r,
                                                          int rp, float ridge, float* __restrict__ G) {
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= rp * rp) return;
  const int i = e / rp, j = e - (e / rp) * rp;
  if (j > i) return;
  float sum = 0.f;
  if (i < r) {
    const float* src = parts + (size_t)i * rp + j;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    int p = 0;
    for (; p + 8 <= nparts; p += 8)
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] += __ldg(src + (size_t)(p + q) * rp * rp);
    for (; p < nparts; ++p) acc[0] += __ldg(src + (size_t)p * rp * rp);
    sum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
    if (i == j) sum += ridge;
  }
  G[(size_t)i * rp + j] = sum;
  G[(size_t)j * rp + i] = sum;
}

// C (M x N) = A (M x K) B (K x N), row-major fp32 with leading dimensions,
// for the small products of the Gram chain (T = G^{-1} Gt and Q' = Q T, both
// with N, K <= 256).  64 x 64 output tile per block of 16 x 16 threads, 4 x 4
// per thread, K in slices of 16 staged in shared memory; the order of every
// sum is fixed.
__global__ void __launch_bounds__(256) small_gemm_kernel(const float* __restrict__ A, int64_t lda,
                                                         const float* __restrict__ B, int64_t ldb,
                                                         float* __restrict__ Cm, int64_t ldc, int64_t M, int N,
                                                         int K) {
  __shared__ float As[16][64 + 4];
  __shared__ float Bs[16][64];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int64_t m0 = (int64_t)blockIdx.x * 64;
  const int n0 = blockIdx.y * 64;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int e = threadIdx.x; e < 64 * 16; e += 256) {
      const int rr = e / 16, kk = e % 16;
      const int64_t row = m0 + rr;
      As[kk][rr] = (row < M && k0 + kk < K) ? A[row * lda + k0 + kk] : 0.f;
      const int kb = e / 64, cc = e % 64;
      Bs[kb][cc] = (k0 + kb < K && n0 + cc < N) ? B[(int64_t)(k0 + kb) * ldb + n0 + cc] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t row = m0 + ty * 4 + i;
    if (row >= M) break;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int col = n0 + tx * 4 + j;
      if (col < N) Cm[row * ldc + col] = acc[i][j];
    }
  }
}

// ---------------------------------------------------------------------------
// G^{-1} through the Cholesky factorisation of G (the normal equations of
// eqs. lsqA/lsqB, Sec. 3.2), in its square-root-free form G = L D L^T (L unit
// lower triangular, D diagonal; the Cholesky factor is L D^{1/2}), then
// Y = L^{-1} and G^{-1} = Y^T D^{-1} Y, written to both triangles so that
// the result is exactly symmetric.  A pivot d_k <= 4 r eps g_kk (d_k is the
// Schur complement, the square of the Cholesky pivot) or a non-finite d_k
// marks G as not positive definite: NMD_ERR_NOT_SPD with detail k, and
// G^{-1} = 0.  One thread block; two forms below, by r_pad.
// ---------------------------------------------------------------------------

// Register-resident, blocked form for r_pad <= 32
// (the pad rows and columns >= r get a unit diagonal, so the padded matrix
// diag(G, I) is factored and inverted; its pad part is dropped at the end).
// Thread t owns row i = t / 4 and the CPT = r_pad / 4 contiguous columns
// c0 = (t % 4) CPT ... of it in registers; a warp holds 8 whole rows.  The
// columns are taken in panels of PB = min(8, CPT):
//  1. The PB x PB diagonal block lies in one warp: its rows factor it in
//     their registers, reading each other's entries by shuffles (pivot test
//     as above), and publish it.
//     Every row below then eliminates its own PB panel values against the
//     block (no communication) and publishes them; after a barrier every
//     row applies the rank-PB update a_ij -= sum_k a_ik a_jk / d_k to its
//     columns right of the panel.  Two barriers per panel.
//  2. Y = L^{-1} by panels of PB rows: inside the block's warp, forward
//     substitution with shuffles; the block's rows of Y go to shared memory
//     (two buffers) and every row below subtracts sum_k l_ik Y[k, :].  One
//     barrier per panel.
//  3. G^{-1} = Y^T D^{-1} Y from shared memory.
// entry (k, n) of G^{-1} as hi + lo bf16 pieces at row n, column k of the
// transposed split (hi rows first, then lo rows)
template <int RP>
__device__ __forceinline__ void store_split(bf16* gsplit, int n, int k, float v) {
  constexpr int SB = split_stride(RP);
  const bf16 hi = __float2bfloat16_rn(v);
  gsplit[n * SB + k] = hi;
  gsplit[RP * SB + n * SB + k] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

template <int RP>
__global__ void __launch_bounds__(RP * 4) ldlt_inv_reg_kernel(const float* __restrict__ G, int r,
                                                              float* __restrict__ Ginv, bf16* __restrict__ gsplit,
                                                              int* __restrict__ status) {
  constexpr int CPT = RP / 4, PB = CPT < 8 ? CPT : 8, LD = RP + 1;
  extern __shared__ __align__(16) float smr[];
  float* invd = smr;                 // RP: 1 / d_k
  float* diag0 = invd + RP;          // RP: the diagonal of G
  float* DB = diag0 + RP;            // PB x PB: the diagonal block being factored (64 floats)
  float* Pn = DB + 64;               // RP x PB: the panel's columns / 2 x PB x RP: rows of Y
  float* F = Pn + 2 * PB * RP;       // RP x LD: the factor, then Y
  __shared__ int bad;
  const int i = threadIdx.x / 4, s = threadIdx.x % 4, c0 = s * CPT, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) bad = 0;
  float a[CPT];
#pragma unroll
  for (int j = 0; j < CPT; j += 4) {
    const float4 v = *(const float4*)(G + (size_t)i * RP + c0 + j);
    a[j] = v.x; a[j + 1] = v.y; a[j + 2] = v.z; a[j + 3] = v.w;
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j)
    if (c0 + j == i) {
      if (i >= r) a[j] = 1.f;
      diag0[i] = a[j];
    }
  __syncthreads();
  const float tol = 4.0f * (float)r * FLT_EPSILON;
  // 1. G = L D L^T, a[] keeping a_ij = l_ij d_j (j < i) and d_i (j == i)
#pragma unroll
  for (int kb = 0; kb < RP; kb += PB) {
    const int sp = kb / CPT, jp = kb - (kb / CPT) * CPT;   // segment and offset of the panel's columns
    const bool in_block = i >= kb && i < kb + PB;
    if ((threadIdx.x >> 5) == (kb >> 3)) {
      // the block's rows kb + q are lanes 4 ((kb + q) % 8) + sp of this warp:
      // factor the block in their registers, one shuffle per entry read
      const bool mine = in_block && s == sp;
      const int qo = i - kb;
      float blk[PB];
#pragma unroll
      for (int k = 0; k < PB; ++k) blk[k] = a[jp + k];
#pragma unroll
      for (int k = 0; k < PB; ++k) {
        const int lk = ((kb + k) & 7) * 4 + sp;
        const float d = __shfl_sync(0xffffffffu, blk[k], lk);
        const float inv = 1.0f / d;
        if (lane == lk) {
          const int kk = kb + k;
          if (kk < r && (!(d > tol * diag0[kk]) || !isfinite(d))) {
            if (!bad) set_status(status, NMD_ERR_NOT_SPD, kk, 0);
            bad = 1;
          }
          invd[kk] = inv;
        }
        const float ajk = blk[k] * inv;
#pragma unroll
        for (int q = k + 1; q < PB; ++q) {
          const float aqk = __shfl_sync(0xffffffffu, blk[k], ((kb + q) & 7) * 4 + sp);
          if (mine && qo > k && q <= qo) blk[q] = fmaf(-ajk, aqk, blk[q]);
        }
      }
      if (mine)
#pragma unroll
        for (int k = 0; k < PB; ++k) {
          a[jp + k] = blk[k];
          DB[qo * PB + k] = blk[k];
        }
    }
    __syncthreads();
    if (bad) {   // uniform: every thread reads the flag after the barrier
#pragma unroll
      for (int j = 0; j < CPT; ++j) Ginv[(size_t)i * RP + c0 + j] = 0.f;
      return;
    }
    if (s == sp && i >= kb) {
      if (!in_block) {
#pragma unroll
        for (int k = 0; k < PB; ++k) {
          const float u = a[jp + k] * invd[kb + k];
#pragma unroll
          for (int q = k + 1; q < PB; ++q) a[jp + q] = fmaf(-u, DB[q * PB + k], a[jp + q]);
        }
      }
#pragma unroll
      for (int k = 0; k < PB; k += 4)
        *(float4*)(Pn + i * PB + k) = make_float4(a[jp + k], a[jp + k + 1], a[jp + k + 2], a[jp + k + 3]);
    }
    __syncthreads();
    if (i >= kb + PB) {
      float u[PB];
#pragma unroll
      for (int k = 0; k < PB; k += 4) {
        const float4 v = *(const float4*)(Pn + i * PB + k);
        u[k] = v.x * invd[kb + k]; u[k + 1] = v.y * invd[kb + k + 1];
        u[k + 2] = v.z * invd[kb + k + 2]; u[k + 3] = v.w * invd[kb + k + 3];
      }
#pragma unroll
      for (int jj = 0; jj < CPT; ++jj) {
        if (c0 + jj >= kb + PB) {
          float acc = a[jj];
#pragma unroll
          for (int k = 0; k < PB; k += 4) {
            const float4 v = *(const float4*)(Pn + (c0 + jj) * PB + k);
            acc = fmaf(-u[k], v.x, acc); acc = fmaf(-u[k + 1], v.y, acc);
            acc = fmaf(-u[k + 2], v.z, acc); acc = fmaf(-u[k + 3], v.w, acc);
          }
          a[jj] = acc;
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j) F[i * LD + c0 + j] = a[j];
  __syncthreads();
  // 2. Y = L^{-1} (a[] now holds row i of Y), l_ik = a_ik / d_k
#pragma unroll
  for (int j = 0; j < CPT; ++j) a[j] = c0 + j == i ? 1.f : 0.f;
#pragma unroll
  for (int kb = 0; kb < RP; kb += PB) {
    float* YP = Pn + ((kb / PB) & 1) * PB * RP;
    if ((threadIdx.x >> 5) == (kb >> 3)) {
      const int rl = i - kb;   // row within the block (outside [0, PB) for the warp's other rows)
#pragma unroll
      for (int k = 0; k + 1 < PB; ++k) {
        const int src = ((kb + k) & 7) * 4 + s;
        const float l = (rl > k && rl < PB) ? F[i * LD + kb + k] * invd[kb + k] : 0.f;
#pragma unroll
        for (int jj = 0; jj < CPT; ++jj) {
          const float yk = __shfl_sync(0xffffffffu, a[jj], src);
          a[jj] = fmaf(-l, yk, a[jj]);
        }
      }
      if (rl >= 0 && rl < PB)
#pragma unroll
        for (int jj = 0; jj < CPT; jj += 4)
          *(float4*)(YP + rl * RP + c0 + jj) = make_float4(a[jj], a[jj + 1], a[jj + 2], a[jj + 3]);
    }
    __syncthreads();
    if (i >= kb + PB) {
      float l[PB];
#pragma unroll
      for (int k = 0; k < PB; ++k) l[k] = F[i * LD + kb + k] * invd[kb + k];
#pragma unroll
      for (int jj = 0; jj < CPT; jj += 4) {
        float4 acc = make_float4(a[jj], a[jj + 1], a[jj + 2], a[jj + 3]);
#pragma unroll
        for (int k = 0; k < PB; ++k) {
          const float4 v = *(const float4*)(YP + k * RP + c0 + jj);
          acc.x = fmaf(-l[k], v.x, acc.x); acc.y = fmaf(-l[k], v.y, acc.y);
          acc.z = fmaf(-l[k], v.z, acc.z); acc.w = fmaf(-l[k], v.w, acc.w);
        }
        a[jj] = acc.x; a[jj + 1] = acc.y; a[jj + 2] = acc.z; a[jj + 3] = acc.w;
      }
    }
  }
  __syncthreads();   // every read of the factor is done
#pragma unroll
  for (int j = 0; j < CPT; ++j) F[i * LD + c0 + j] = a[j];
  __syncthreads();
  // 3. G^{-1}[i][j] = sum over k of Y[k][i] Y[k][j] / d_k (Y[k][j] = 0 for j > k)
#pragma unroll
  for (int j = 0; j < CPT; ++j) a[j] = 0.f;
  for (int k = i > c0 ? i : c0; k < RP; ++k) {
    const float w = F[k * LD + i] * invd[k];
#pragma unroll
    for (int j = 0; j < CPT; ++j) a[j] = fmaf(w, F[k * LD + c0 + j], a[j]);
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j) a[j] = (i < r && c0 + j < r) ? a[j] : 0.f;
#pragma unroll
  for (int j = 0; j < CPT; j += 4)
    *(float4*)(Ginv + (size_t)i * RP + c0 + j) = make_float4(a[j], a[j + 1], a[j + 2], a[j + 3]);
  if (gsplit)
#pragma unroll
    for (int j = 0; j < CPT; ++j) store_split<RP>(gsplit, c0 + j, i, a[j]);
}

inline size_t ldlt_reg_smem_bytes(int rp) {
  const size_t pb = rp / 4 < 8 ? rp / 4 : 8;
  return ((size_t)2 * rp + 64 + 2 * pb * rp + (size_t)rp * (rp + 1)) * sizeof(float);
}

// Tile-blocked form of the same factorisation for r_pad in {64, 128, 256}:
// the matrix is cut into 32 x 32 tiles and only the lower triangle of tiles
// is kept in shared memory (row stride 33, so a tile's rows and columns are
// both read without bank conflicts); pad rows and columns >= r get a unit
// diagonal, as in the register form.  For each tile column J:
//  1a. one warp factors the diagonal tile in registers (lane i holds row i;
//      every entry read by a shuffle), checks the pivots, and replaces the
//      tile by the inverse Yt of its unit lower factor (forward substitution
//      with shuffles), stored with its unit diagonal and zeros above;
//  1b. the tiles below: L_IJ = A_IJ Yt^T D_J^{-1}, one warp per row, lanes
//      over the 32 columns; the panel is also stored transposed in P;
//  1c. the trailing tiles: A_IK -= L_IJ D_J L_KJ^T, 4 x 4 outputs per thread
//      with float4 reads of the transposed panel.
// Three barriers per tile column (24 at r_pad = 256).  Then
//  2.  Y = L^{-1} by tile rows I: T_IJ = sum over K in [J, I) of L_IK Y_KJ
//      (Y_JJ is the diagonal tile's inverse), then Y_IJ = -Yt_I T_IJ over
//      L_IJ; two barriers per tile row;
//  3.  G^{-1} = Y^T D^{-1} Y from the tiles, 4 x 4 outputs per thread,
//      written to both triangles (exactly symmetric).
// The trailing update and the products in 2 and 3 are the r^3 part, spread
// over every thread; the serial part is the 32-step diagonal factorisation
// of each tile in one warp.
// ---------------------------------------------------------------------------
template <int RP>
struct TileChol {
  static constexpr int TB = 32, NT = RP / TB, LDT = TB + 1, TSZ = TB * LDT;
  static constexpr int NTILE = NT * (NT + 1) / 2;
  static constexpr int NTHR = RP * 4 > 1024 ? 1024 : RP * 4;
  static constexpr int PBUF = TB * RP;   // the transposed panel (32 x RP), or the T_IJ of one tile row
  static constexpr size_t SMEM = ((size_t)NTILE * TSZ + PBUF + 3 * RP) * sizeof(float);
  static_assert(RP % TB == 0 && NT >= 2, "tile form for r_pad >= 64");
};

__device__ __forceinline__ int tile_index(int I, int J) { return ((I * (I + 1)) >> 1) + J; }

// tile (I, J) of the lower triangle of tiles from its index q
__device__ __forceinline__ void tile_of(int q, int& I, int& J) {
  I = 0;
  while ((((I + 1) * (I + 2)) >> 1) <= q) ++I;
  J = q - ((I * (I + 1)) >> 1);
}

template <int RP>
__global__ void __launch_bounds__(TileChol<RP>::NTHR, 1) ldlt_inv_tile_kernel(const float* __restrict__ G, int r,
                                                                          float* __restrict__ Ginv,
                                                                          bf16* __restrict__ gsplit,
                                                                          int* __restrict__ status) {
  using C = TileChol<RP>;
  constexpr int TB = C::TB, NT = C::NT, LDT = C::LDT, TSZ = C::TSZ, NTHR = C::NTHR;
  extern __shared__ __align__(16) float smt[];
  float* A = smt;                        // NTILE tiles: the matrix, then L and Y
  float* P = A + C::NTILE * TSZ;         // PBUF
  float* dv = P + C::PBUF;               // RP: d_k
  float* invd = dv + RP;                 // RP: 1 / d_k
  float* diag0 = invd + RP;              // RP: the diagonal of G
  __shared__ int bad;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) bad = 0;
  for (int t = tid; t < C::NTILE * TB * TB; t += NTHR) {
    int I, J;
    tile_of(t / (TB * TB), I, J);
    const int e = t % (TB * TB), ii = e / TB, jj = e % TB, i = I * TB + ii, j = J * TB + jj;
    const float g = (i < r && j < r) ? G[(size_t)i * RP + j] : (i == j ? 1.f : 0.f);
    A[(t / (TB * TB)) * TSZ + ii * LDT + jj] = g;
    if (i == j) diag0[i] = g;
  }
  for (int e = tid; e < RP * RP; e += NTHR)
    if (e / RP >= r || e % RP >= r) {
      Ginv[e] = 0.f;
      if (gsplit) store_split<RP>(gsplit, e % RP, e / RP, 0.f);
    }
  __syncthreads();
  const float tol = 4.0f * (float)r * FLT_EPSILON;

  // 1. G = L D L^T, tile column by tile column
  for (int J = 0; J < NT; ++J) {
    if (warp == 0) {
      float* T = A + tile_index(J, J) * TSZ;
      float a[TB];
#pragma unroll
      for (int j = 0; j < TB; ++j) a[j] = T[lane * LDT + j];
      int badk = -1;
#pragma unroll
      for (int k = 0; k < TB; ++k) {
        const float d = __shfl_sync(0xffffffffu, a[k], k);
        const float inv = 1.0f / d;
        const int kk = J * TB + k;
        if (badk < 0 && kk < r && (!(d > tol * diag0[kk]) || !isfinite(d))) badk = kk;   // warp-uniform
        if (lane == k) {
          dv[kk] = d;
          invd[kk] = inv;
        }
        const float aik = a[k];
        const float l = aik * inv;
        if (lane > k) a[k] = l;
#pragma unroll
        for (int j = k + 1; j < TB; ++j) a[j] = fmaf(-aik, __shfl_sync(0xffffffffu, l, j), a[j]);
      }
      // the unit lower factor of the tile, then its inverse Yt in registers
#pragma unroll
      for (int j = 0; j < TB; ++j)
        if (j < lane) T[lane * LDT + j] = a[j];
      __syncwarp();
#pragma unroll
      for (int j = 0; j < TB; ++j) a[j] = j == lane ? 1.f : 0.f;
#pragma unroll
      for (int m = 0; m + 1 < TB; ++m) {
        const float lim = lane > m ? T[lane * LDT + m] : 0.f;
#pragma unroll
        for (int j = 0; j <= m; ++j) a[j] = fmaf(-lim, __shfl_sync(0xffffffffu, a[j], m), a[j]);
      }
      __syncwarp();
#pragma unroll
      for (int j = 0; j < TB; ++j) T[lane * LDT + j] = a[j];   // unit diagonal, zeros above
      if (lane == 0 && badk >= 0) {
        bad = 1;
        set_status(status, NMD_ERR_NOT_SPD, badk, 0);
      }
    }
    __syncthreads();
    if (bad) {   // uniform: every thread reads the flag after the barrier
      for (int e = tid; e < RP * RP; e += NTHR) Ginv[e] = 0.f;
      return;
    }
    // 1b. L_IJ = A_IJ Yt^T D_J^{-1} for the rows below the diagonal tile
    const float* Yt = A + tile_index(J, J) * TSZ;
    const int row0 = (J + 1) * TB;
    for (int i = row0 + warp; i < RP; i += NTHR / 32) {
      float* Ai = A + tile_index(i / TB, J) * TSZ + (i % TB) * LDT;
      float acc = 0.f;
#pragma unroll 8
      for (int m = 0; m < TB; ++m) acc = fmaf(Ai[m], Yt[lane * LDT + m], acc);
      acc *= invd[J * TB + lane];
      __syncwarp();
      Ai[lane] = acc;
      P[lane * RP + i] = acc;
    }
    __syncthreads();
    // 1c. A_IK -= L_IJ D_J L_KJ^T for J < K <= I (lower half of diagonal tiles)
    const int nt = NT - J - 1;
    for (int b = tid; b < (nt * (nt + 1) / 2) * 64; b += NTHR) {
      int I, K;
      tile_of(b / 64, I, K);
      I += J + 1;
      K += J + 1;
      const int u4 = (b % 64) / 8, v4 = b % 8;
      if (I == K && v4 > u4) continue;
      const int i0 = I * TB + 4 * u4, j0 = K * TB + 4 * v4;
      float acc[4][4] = {};
#pragma unroll 4
      for (int k = 0; k < TB; ++k) {
        const float dk = dv[J * TB + k];
        const float4 pa = *(const float4*)(P + k * RP + i0);
        const float4 pb = *(const float4*)(P + k * RP + j0);
        const float ya[4] = {pa.x * dk, pa.y * dk, pa.z * dk, pa.w * dk};
        const float yb[4] = {pb.x, pb.y, pb.z, pb.w};
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(ya[u], yb[v], acc[u][v]);
      }
      float* T = A + tile_index(I, K) * TSZ + 4 * u4 * LDT + 4 * v4;
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) T[u * LDT + v] -= acc[u][v];
    }
    __syncthreads();
  }

  // 2. Y = L^{-1} by tile rows; the diagonal tiles already hold their inverses
  for (int I = 1; I < NT; ++I) {
    for (int b = tid; b < I * 64; b += NTHR) {
      const int J = b / 64, u4 = (b % 64) / 8, v4 = b % 8;
      float acc[4][4] = {};
      for (int K = J; K < I; ++K) {
        const float* L = A + tile_index(I, K) * TSZ + 4 * u4 * LDT;
        const float* Y = A + tile_index(K, J) * TSZ + 4 * v4;
#pragma unroll 4
        for (int m = 0; m < TB; ++m) {
          float la[4], yb[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) la[u] = L[u * LDT + m];
#pragma unroll
          for (int v = 0; v < 4; ++v) yb[v] = Y[m * LDT + v];
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(la[u], yb[v], acc[u][v]);
        }
      }
      float* T = P + J * TB * TB + 4 * u4 * TB + 4 * v4;
#pragma unroll
      for (int u = 0; u < 4; ++u) *(float4*)(T + u * TB) = make_float4(acc[u][0], acc[u][1], acc[u][2], acc[u][3]);
    }
    __syncthreads();
    const float* Yd = A + tile_index(I, I) * TSZ;
    for (int b = tid; b < I * 64; b += NTHR) {
      const int J = b / 64, u4 = (b % 64) / 8, v4 = b % 8;
      const float* T = P + J * TB * TB + 4 * v4;
      float acc[4][4] = {};
#pragma unroll 4
      for (int m = 0; m < TB; ++m) {
        float ya[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) ya[u] = Yd[(4 * u4 + u) * LDT + m];
        const float4 t = *(const float4*)(T + m * TB);
        const float tb[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(ya[u], tb[v], acc[u][v]);
      }
      float* Y = A + tile_index(I, J) * TSZ + 4 * u4 * LDT + 4 * v4;
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) Y[u * LDT + v] = -acc[u][v];
    }
    __syncthreads();
  }

  // 3. G^{-1}[a][b] = sum over k of Y[k][a] Y[k][b] / d_k, tile rows K >= the tiles of a and b
  for (int b = tid; b < C::NTILE * 64; b += NTHR) {
    int I, J;
    tile_of(b / 64, I, J);
    const int u4 = (b % 64) / 8, v4 = b % 8;
    if (I == J && v4 > u4) continue;
    const int a0 = I * TB + 4 * u4, b0 = J * TB + 4 * v4;
    if (a0 >= r || b0 >= r) continue;
    float acc[4][4] = {};
    for (int K = I; K < NT; ++K) {
      const float* Ya = A + tile_index(K, I) * TSZ + 4 * u4;
      const float* Yb = A + tile_index(K, J) * TSZ + 4 * v4;
#pragma unroll 4
      for (int m = 0; m < TB; ++m) {
        const float w = invd[K * TB + m];
        float ya[4], yb[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) ya[u] = Ya[m * LDT + u] * w;
#pragma unroll
        for (int v = 0; v < 4; ++v) yb[v] = Yb[m * LDT + v];
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(ya[u], yb[v], acc[u][v]);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const int ga = a0 + u, gb = b0 + v;
        if (ga < r && gb < r && (a0 != b0 || v <= u)) {
          Ginv[(size_t)ga * RP + gb] = acc[u][v];
          Ginv[(size_t)gb * RP + ga] = acc[u][v];
          if (gsplit) {
            store_split<RP>(gsplit, gb, ga, acc[u][v]);
            store_split<RP>(gsplit, ga, gb, acc[u][v]);
          }
        }
      }
  }
}

// ---------------------------------------------------------------------------
// Sparse correction: for every panel row i and entry (i, k) in the block,
// L_ik = m_i . q_k, c = S_ik - min(0, L_ik), R_i += c q_k, on the step's
// operands (the bf16 pieces in the bf16 mode, else the fp32 masters).
// This kernel takes the rows with at most kShort entries in the panel (the
// connectome's panels average 1.3 entries per row): each row gets LPR lanes,
// one 16-byte load of its row segment each (8 bf16 or 4 fp32 values; two at
// r_pad = 256 in fp32), so a warp works on 32 / LPR rows at once and their
// loads are in flight together.  The lanes of a row first fetch the entries'
// indices and values (one entry per lane), then NE entries at a time are
// processed with their q rows in flight together; each dot product is summed
// over the row's lanes by a butterfly, and the accumulation over the entries
// stays in ascending order.  The result goes to Rs, the support term of R,
// one writer per row.  Rs is written only on the rows with support in the
// block's panel; a flag byte per row tells the update which rows of Rs to
// add, so the other rows are neither read nor cleared.  Longer rows:
// sparse_long_kernel below.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float ldv(const float* p) { return __ldg(p); }
__device__ __forceinline__ float ldv(const bf16* p) { return __bfloat162float(__ldg(p)); }

// 16 bytes of a factor row as floats: 8 bf16 or 4 fp32 values
__device__ __forceinline__ void load16(float* f, const bf16* p) {
  const uint4 u = __ldg((const uint4*)p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    f[2 * q] = __uint_as_float(w[q] << 16);
    f[2 * q + 1] = __uint_as_float(w[q] & 0xffff0000u);
  }
}
__device__ __forceinline__ void load16(float* f, const float* p) {
  const float4 v = __ldg((const float4*)p);
  f[0] = v.x; f[1] = v.y; f[2] = v.z; f[3] = v.w;
}

template <int RP, typename T>
__global__ void __launch_bounds__(256, 4) sparse_group_kernel(const PanelRow* __restrict__ rows, int64_t nrows,
                                                           const T* __restrict__ Mop, int64_t m0,
                                                           const T* __restrict__ Qop,
                                                           const int32_t* __restrict__ qidx,
                                                           const float* __restrict__ vals, float* __restrict__ R) {
  constexpr int E16 = 16 / (int)sizeof(T);               // elements per 16-byte load
  constexpr int LPR = RP / E16 < 32 ? RP / E16 : 32;     // lanes per row
  constexpr int CH = RP / (E16 * LPR);                   // 16-byte loads per lane and row
  constexpr int EPL = E16 * CH;                          // elements per lane
  constexpr int RPW = 32 / LPR;                          // rows per warp
  constexpr int NE = 2;                                  // entries whose q rows load together
  const int lane = threadIdx.x & 31, sub = lane % LPR, grp = lane / LPR;
  const int64_t wbase = ((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5) * RPW;
  if (wbase >= nrows) return;                            // warp-uniform
  const int64_t w = wbase + grp;
  const bool live_row = w < nrows;
  const PanelRow pr = live_row ? rows[w] : PanelRow{0, 0, 0};
  float mv[EPL], acc[EPL];
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    if (live_row) load16(mv + c * E16, Mop + (int64_t)pr.row * RP + (c * LPR + sub) * E16);
    else
#pragma unroll
      for (int q = 0; q < E16; ++q) mv[c * E16 + q] = 0.f;
  }
#pragma unroll
  for (int q = 0; q < EPL; ++q) acc[q] = 0.f;
  int maxlen = pr.len;                                   // longest row of the warp
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) maxlen = max(maxlen, __shfl_xor_sync(0xffffffffu, maxlen, o));
  for (int e0 = 0; e0 < maxlen; e0 += LPR) {
    int kl = -1;
    float sl = 0.f;
    if (e0 + sub < pr.len) {                             // lane sub holds entry e0 + sub of its row
      kl = __ldg(qidx + pr.beg + e0 + sub);
      sl = __ldg(vals + pr.beg + e0 + sub);
    }
    const int nb = min(LPR, maxlen - e0);                // warp-uniform
    for (int j0 = 0; j0 < nb; j0 += NE) {
      float qv[NE][EPL], part[NE], sv[NE];
#pragma unroll
      for (int j = 0; j < NE; ++j) {
        const int src = grp * LPR + ((j0 + j) & (LPR - 1));
        const int k = __shfl_sync(0xffffffffu, kl, src);
        sv[j] = __shfl_sync(0xffffffffu, sl, src);
        const bool live = j0 + j < nb && k >= 0;
#pragma unroll
        for (int c = 0; c < CH; ++c) {
          if (live) load16(qv[j] + c * E16, Qop + (int64_t)k * RP + (c * LPR + sub) * E16);
          else
#pragma unroll
            for (int q = 0; q < E16; ++q) qv[j][c * E16 + q] = 0.f;
        }
        part[j] = 0.f;
#pragma unroll
        for (int q = 0; q < EPL; ++q) part[j] = fmaf(mv[q], qv[j][q], part[j]);
      }
#pragma unroll
      for (int o = 1; o < LPR; o <<= 1)
#pragma unroll
        for (int j = 0; j < NE; ++j) part[j] += __shfl_xor_sync(0xffffffffu, part[j], o);
#pragma unroll
      for (int j = 0; j < NE; ++j) {
        const float cval = sv[j] - fminf(0.f, part[j]);   // zero for padding entries (s = 0, q = 0)
#pragma unroll
        for (int q = 0; q < EPL; ++q) acc[q] = fmaf(cval, qv[j][q], acc[q]);
      }
    }
  }
  if (live_row) {
    float* dst = R + (pr.row - m0) * RP;
#pragma unroll
    for (int c = 0; c < CH; ++c)
#pragma unroll
      for (int q = 0; q < E16; q += 4)
        *(float4*)(dst + (c * LPR + sub) * E16 + q) =
            make_float4(acc[c * E16 + q], acc[c * E16 + q + 1], acc[c * E16 + q + 2], acc[c * E16 + q + 3]);
  }
}

// Long rows (more than kShort entries in the panel): one warp per segment (a
// whole row, or a slice of a longer one), with the lanes over the entries.  LPE = rp / 32 lanes share an entry
// (lane sub = lane % LPE owns columns 32 sub ... 32 sub + 31; CPL = min(32, rp)
// of them are real), so a warp takes EPW = 32 / LPE entries at a time.  The
// q rows of those entries are first copied into a per-warp shared buffer with
// coalesced loads (whole 128-byte lines), as 32 chunks of 32 columns padded to
// 36 floats, chunk = lane that reads it, so that each lane's reads are free of
// bank conflicts.  Each lane then forms its part of L_ik = m_i . q_k, the LPE
// parts are added with shuffles, c = S_ik - min(0, L_ik), and the lane
// accumulates c q_k over its own entries; at the end the EPW entry slots are
// added with a butterfly (one reduction per row instead of one per entry).
// The order of every sum is fixed, so results are the same on every run.
// Stage 32 columns (one chunk) of a q row into 32 floats of shared memory,
// 16 bytes per load: 4 fp32 or 8 bf16 values.
__device__ __forceinline__ void stage16(float* dst, const float* src) {
  *(float4*)dst = __ldg((const float4*)src);
}
__device__ __forceinline__ void stage16(float* dst, const bf16* src) {
  const uint4 u = __ldg((const uint4*)src);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  float f[8];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    f[2 * q] = __uint_as_float(w[q] << 16);
    f[2 * q + 1] = __uint_as_float(w[q] & 0xffff0000u);
  }
  *(float4*)dst = make_float4(f[0], f[1], f[2], f[3]);
  *(float4*)(dst + 4) = make_float4(f[4], f[5], f[6], f[7]);
}

template <int LPE, int CPL, typename T>
__global__ void __launch_bounds__(256, 2) sparse_long_kernel(const PanelRow* __restrict__ segs, int64_t nseg,
                                                          const T* __restrict__ Mop, int64_t m0,
                                                          const T* __restrict__ Qop,
                                                          const int32_t* __restrict__ qidx,
                                                          const float* __restrict__ vals,
                                                          float* __restrict__ R, float* __restrict__ partials,
                                                          int rp) {
  constexpr int EPW = 32 / LPE;
  constexpr int CS = 36;                       // floats per staged chunk (32 + 4 padding)
  constexpr int NPF = 4;                       // entry iterations whose indices are fetched together
  constexpr int VEC = 16 / (int)sizeof(T);     // elements per 16-byte load
  constexpr int LPC = CPL / VEC;               // 16-byte loads per 32-column chunk
  __shared__ __align__(16) float stage[8][32 * CS];
  const int lane = threadIdx.x & 31;
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  if (w >= nseg) return;
  float* buf = stage[(threadIdx.x >> 5) & 7];
  const PanelRow pr = segs[w];
  const int sub = lane % LPE, slot = lane / LPE;
  const int64_t i = pr.row;
  float mv[CPL], acc[CPL];
#pragma unroll
  for (int c = 0; c < CPL; ++c) mv[c] = ldv(Mop + i * rp + 32 * sub + c);
#pragma unroll
  for (int c = 0; c < CPL; ++c) acc[c] = 0.f;
  for (int e00 = 0; e00 < pr.len; e00 += NPF * EPW) {
    int kk[NPF];
    float ss[NPF];
#pragma unroll
    for (int t = 0; t < NPF; ++t) {
      const int e = e00 + t * EPW + slot;
      const bool live = e < pr.len;
      kk[t] = live ? __ldg(qidx + pr.beg + e) : -1;
      ss[t] = live ? __ldg(vals + pr.beg + e) : 0.f;
    }
#pragma unroll
    for (int t = 0; t < NPF; ++t) {
      if (e00 + t * EPW >= pr.len) break;             // warp-uniform
      // stage: load f = lane + 32 u (u < LPC) of the 32 chunks; chunk f / LPC
      // is columns 32 (chunk % LPE) ... of entry slot chunk / LPE
#pragma unroll
      for (int u = 0; u < LPC; ++u) {
        const int f = lane + 32 * u;
        const int chunk = f / LPC, part = f % LPC;
        const int ke = __shfl_sync(0xffffffffu, kk[t], (chunk / LPE) * LPE);
        float* dst = buf + chunk * CS + VEC * part;
        if (ke >= 0) {
          stage16(dst, Qop + (int64_t)ke * rp + 32 * (chunk % LPE) + VEC * part);
        } else {
#pragma unroll
          for (int q = 0; q < VEC; q += 4) *(float4*)(dst + q) = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      __syncwarp();
      float q[CPL];
#pragma unroll
      for (int c = 0; c < CPL / 4; ++c) {
        const float4 v = *(const float4*)(buf + lane * CS + 4 * c);
        q[4 * c] = v.x; q[4 * c + 1] = v.y; q[4 * c + 2] = v.z; q[4 * c + 3] = v.w;
      }
      __syncwarp();                                   // the buffer is refilled next iteration
      float dot = 0.f;
#pragma unroll
      for (int c = 0; c < CPL; ++c) dot = fmaf(mv[c], q[c], dot);
#pragma unroll
      for (int o = 1; o < LPE; o <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
      const float cval = ss[t] - fminf(0.f, dot);    // zero for the padding slots (s = 0, q = 0)
#pragma unroll
      for (int c = 0; c < CPL; ++c) acc[c] = fmaf(cval, q[c], acc[c]);
    }
  }
#pragma unroll
  for (int o = LPE; o < 32; o <<= 1)
#pragma unroll
    for (int c = 0; c < CPL; ++c) acc[c] += __shfl_xor_sync(0xffffffffu, acc[c], o);
  if (slot == 0) {
    float* dst = (partials ? partials + w * rp : R + (i - m0) * rp) + 32 * sub;
#pragma unroll
    for (int c = 0; c < CPL / 4; ++c)
      *(float4*)(dst + 4 * c) = make_float4(acc[4 * c], acc[4 * c + 1], acc[4 * c + 2], acc[4 * c + 3]);
  }
}

// Rs_i = sum of the segment slots of row i.  One block per long row: thread
// t handles column t % RP of the slots g, g + G, g + 2G, ... (g = t / RP,
// G = 256 / RP groups) with eight loads in flight, and the G group sums are
// added in group order, so the result is the same on every run.
template <int RP>
__global__ void __launch_bounds__(256) sparse_reduce_kernel(const PanelRow* __restrict__ multi,
                                                            const float* __restrict__ partials,
                                                            float* __restrict__ R, int64_t m0) {
  constexpr int G = 256 / RP;
  __shared__ float gsum[256];
  const PanelRow mr = multi[blockIdx.x];
  const int c = threadIdx.x % RP, g = threadIdx.x / RP;
  const float* src = partials + mr.beg * RP + c;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  int q = g;
  for (; q + 7 * G < mr.len; q += 8 * G)
#pragma unroll
    for (int u = 0; u < 8; ++u) acc[u] += __ldg(src + (int64_t)(q + u * G) * RP);
  for (; q < mr.len; q += G) acc[0] += __ldg(src + (int64_t)q * RP);
  gsum[threadIdx.x] = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
  __syncthreads();
  if (g == 0) {
    float v = gsum[c];
#pragma unroll
    for (int k = 1; k < G; ++k) v += gsum[k * RP + c];
    R[(mr.row - m0) * RP + c] = v;
  }
}

// ---------------------------------------------------------------------------
// Update of the M-side rows: X = R G^{-1};
//   Z form:     U = eta (X - M)      (eqs. lsqA/lsqB with step size)
//   Delta form: U = eta X            (eqs. spLsqA/spLsqB)
// then E = U + gamma E (stochastic steps) and M += E, refreshing the bf16
// pieces: hi always, lo and lo2 only in the fp32-accurate mode (the only
// one whose dense kernel reads them).
// In the bf16 mode R and Ginv belong to the bf16-rounded Q-side rows (R = Z Qt,
// Ginv = (Qt^T Qt)^{-1}), so X is the least-squares solution for them.
// Skipped entirely while a sticky error is set.
// X = R G^{-1} is a small GEMM per tile of TR rows.  A block keeps CW columns
// of G^{-1} in shared memory; the tile's R rows (contiguous in global memory)
// are copied into a double buffer with cp.async one tile ahead, and each
// thread's M and E entries are loaded into registers before the product, so
// the memory latency of both overlaps the arithmetic.  Thread (ty, tx) owns
// rows 4 ty .. 4 ty + 3 and CPT columns: for CPT >= 4 the groups of four
// columns 4 tx + 4 TX g (g < CPT / 4), so that a quarter warp reads 128
// contiguous bytes of G^{-1} and a half warp writes whole 256-byte rows.
// ---------------------------------------------------------------------------
template <int RP, bool TC = false, int TRT = 64>
struct UpdCfg {
  static constexpr int CW = RP <= 128 ? RP : 128;   // output columns per block
  // rows per tile: on the tensor cores 64, or 32 for launches with fewer
  // 64-row tiles than SMs (the rows the next step reads: more blocks at once)
  static constexpr int TR = TC ? TRT : (RP <= 128 ? 64 : 32);
  static constexpr int TY = TR / 4;                  // row groups of four
  static constexpr int TX = 256 / TY;                // column groups
  static constexpr int CPT = CW / TX;                // columns per thread (1, 2, 4 or 8)
  // tensor-core product: the staged tile's rows padded to RP + 8 floats and
  // the two bf16 pieces of G^{-1} transposed, rows padded to RP + 8, so that
  // the fragment loads and stores of a half warp meet 16 different bank pairs;
  // one tile buffer (a block updates one tile)
  static constexpr int SR = TC ? RP + 8 : RP;        // row stride of a staged tile (floats)
  static constexpr int SB = split_stride(RP);        // row stride of a split G^{-1} (bf16)
  static constexpr size_t SMEM = TC ? (size_t)TR * SR * sizeof(float) + 2 * (size_t)RP * SB * sizeof(bf16)
                                    : ((size_t)RP * CW + 2 * (size_t)TR * RP) * sizeof(float);
  static_assert(CPT >= 1 && (CPT < 4 || CPT % 4 == 0), "column split");
  // tensor-core product: TR / 16 row groups of warps, each warp RP / (8 /
  // (TR / 16)) columns (at least one 8-column tile)
  static constexpr int RG = TR / 16, WC = TC ? RP / (8 / RG) : 8;
  static_assert(!TC || (CW == RP && (TR == 64 || TR == 32) && WC >= 8), "tensor-core product tiling");
};

template <int CPT, int TX>
__device__ __forceinline__ int upd_col(int tx, int j) {
  if (CPT >= 4) return (j / 4) * 4 * TX + 4 * tx + (j % 4);
  return CPT * tx + j;
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem_dst)),
               "l"(gsrc)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// D += A B on one 16 x 8 x 16 tile (bf16 operands, fp32 accumulation), the
// fragment layouts of the PTX ISA's mma.m16n8k16: a[0..3] hold A's (row g,
// columns 2c, 2c+1), (g+8, 2c..), (g, 2c+8..), (g+8, 2c+8..); b0, b1 hold B's
// (rows 2c, 2c+1; column g) and (2c+8, 2c+9; g); d holds (g, 2c), (g, 2c+1),
// (g+8, 2c), (g+8, 2c+1), with g = lane / 4 and c = lane % 4
__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// two fp32 values as hi + lo pieces (bf16, round to nearest), packed in pairs
__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - __low2float(h), x1 - __high2float(h));
  hi = reinterpret_cast<const uint32_t&>(h);
  lo = reinterpret_cast<const uint32_t&>(l);
}

// ---------------------------------------------------------------------------
// The support term with the step's whole Q-side block in shared memory (bf16
// mode, r_pad 16 or 32, the block's bf16 rows within kSparseQBytes: the
// planted and identity workloads, whose panels are dense enough that the q-row
// gathers, not the CSR stream, set the pace of the kernels above).  One CTA
// of 24 warps per SM copies the block's rows into shared memory once; then
// each warp takes work items -- the short rows, the whole long rows and the
// segments of split rows, the lists the other kernels take -- and splits each
// entry's row over NCH lanes, one 16-byte chunk (8 columns) each, so that a
// warp works on 32 / NCH entries at a time: each lane's partial dot product
// with m_i (packed fp32 FMAs, the even and odd columns summed apart) is added
// to the others' by a butterfly, c = S_ik - min(0, L_ik), and every lane adds
// c times its 8 columns of q_k to its own partial sums.  At the end of
// the item the partial sums of the entry slots are added by a butterfly over
// the slots and written once.  Each lane fetches one of every 32 entries'
// index and value (at most 128 entries per item: four), and they are passed
// to the lanes of their slot by shuffles; an item's indices, values and m_i
// are loaded while the previous item is computed, its descriptor two items
// ahead.  In shared memory, 16-byte chunk j of row k sits at chunk j ^ ((k >>
// 1) & (NCH - 1)).  Every index lies in [q0, q0 + K): the panel lists are
// built at create from the CSR cut to the block's columns (rows, for row
// steps), as for the kernels above.
// ---------------------------------------------------------------------------
constexpr size_t kSparseQBytes = 200 * 1024;

template <int RP>
struct SpSmem {
  static constexpr int NCH = RP * 2 / 16;   // 16-byte chunks per bf16 row = lanes per entry
  static constexpr int EPW = 32 / NCH;      // entries a warp works on at a time
  static constexpr int WARPS = 24;
};

// 8 floats from 16 bytes of bf16, as 4 pairs
__device__ __forceinline__ void unpack8(const uint4& u, float2* f) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) f[q] = make_float2(__uint_as_float(w[q] << 16), __uint_as_float(w[q] & 0xffff0000u));
}

// d = a b + c on a pair of floats (one packed fp32 FMA, each half rounded as fmaf)
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{.reg .b64 ra, rb, rc, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

template <int RP>
__global__ void __launch_bounds__(32 * SpSmem<RP>::WARPS, 1) sparse_smem_kernel(
    const PanelRow* __restrict__ rows, int64_t nrows, const PanelRow* __restrict__ whole, int64_t nwhole,
    const PanelRow* __restrict__ seg, int64_t nseg, const bf16* __restrict__ Mop, int64_t m0,
    const bf16* __restrict__ Qop, int64_t q0, int64_t K, const int32_t* __restrict__ qidx,
    const float* __restrict__ vals, float* __restrict__ R, float* __restrict__ partials) {
  using C = SpSmem<RP>;
  constexpr int NCH = C::NCH, EPW = C::EPW;
  static_assert(RP == 16 || RP == 32, "r_pad 16 or 32");
  extern __shared__ __align__(16) uint4 qs[];
  const uint4* qsrc = reinterpret_cast<const uint4*>(Qop + q0 * RP);
  for (int64_t e = threadIdx.x; e < K * NCH; e += blockDim.x) {
    const int64_t k = e / NCH;
    const int j = (int)(e % NCH);
    cp_async16(qs + k * NCH + (j ^ (int)((k >> 1) & (NCH - 1))), qsrc + e);
  }
  cp_async_commit();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ch = lane % NCH, slot = lane / NCH;
  const int64_t nlong = nrows + nwhole, nitems = nlong + nseg;
  const int64_t stride = (int64_t)gridDim.x * C::WARPS;
  auto desc = [&](int64_t x) -> PanelRow {
    if (x >= nitems) return PanelRow{0, 0, 0};
    return x < nrows ? rows[x] : x < nlong ? whole[x - nrows] : seg[x - nlong];
  };
  // an item's indices (relative to the block), values and this lane's chunk of m_i
  auto fetch = [&](const PanelRow& pr, int* k4, float* s4, uint4& mc) {
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int e = lane + 32 * t;
      const bool live = e < pr.len;
      k4[t] = live ? (int)(__ldg(qidx + pr.beg + e) - q0) : 0;
      s4[t] = live ? __ldg(vals + pr.beg + e) : 0.f;
    }
    mc = pr.len > 0 ? __ldg(reinterpret_cast<const uint4*>(Mop + (int64_t)pr.row * RP) + ch) : make_uint4(0, 0, 0, 0);
  };
  int64_t w = (int64_t)blockIdx.x * C::WARPS + warp;
  PanelRow cur = desc(w), nxt = desc(w + stride);
  int kk[4];
  float ss[4];
  uint4 mc;
  fetch(cur, kk, ss, mc);
  cp_async_wait_0();
  __syncthreads();
  for (; w < nitems; w += stride) {
    const PanelRow after = desc(w + 2 * stride);
    int kn[4];
    float sn[4];
    uint4 mn;
    fetch(nxt, kn, sn, mn);
    float2 mv[4], acc[4];
    unpack8(mc, mv);
#pragma unroll
    for (int q = 0; q < 4; ++q) acc[q] = make_float2(0.f, 0.f);
#pragma unroll
    for (int it = 0; it < 128 / EPW; ++it) {
      if (it * EPW >= cur.len) break;   // warp-uniform
      const int e = it * EPW + slot;
      constexpr int PER = 32 / EPW;       // iterations per batch of 32 entries
      const int k = __shfl_sync(0xffffffffu, kk[it / PER], e & 31);
      const float sv = __shfl_sync(0xffffffffu, ss[it / PER], e & 31);
      const bool live = e < cur.len;
      uint4 qc = make_uint4(0, 0, 0, 0);
      if (live) qc = qs[k * NCH + (ch ^ ((k >> 1) & (NCH - 1)))];
      float2 f[4];
      unpack8(qc, f);
      // the even and the odd columns' products summed separately, then added
      float2 d2 = make_float2(0.f, 0.f);
#pragma unroll
      for (int q = 0; q < 4; ++q) d2 = ffma2(mv[q], f[q], d2);
      float dot = d2.x + d2.y;
#pragma unroll
      for (int o = 1; o < NCH; o <<= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
      if (live) {
        const float cv = sv - fminf(0.f, dot);
        const float2 c2 = make_float2(cv, cv);
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[q] = ffma2(c2, f[q], acc[q]);
      }
    }
#pragma unroll
    for (int o = NCH; o < 32; o <<= 1)
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        acc[q].x += __shfl_xor_sync(0xffffffffu, acc[q].x, o);
        acc[q].y += __shfl_xor_sync(0xffffffffu, acc[q].y, o);
      }
    if (slot == 0) {
      float* out = (w < nlong ? R + ((int64_t)cur.row - m0) * RP : partials + (w - nlong) * RP) + 8 * ch;
      *(float4*)out = make_float4(acc[0].x, acc[0].y, acc[1].x, acc[1].y);
      *(float4*)(out + 4) = make_float4(acc[2].x, acc[2].y, acc[3].x, acc[3].y);
    }
    cur = nxt;
    nxt = after;
    mc = mn;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      kk[t] = kn[t];
      ss[t] = sn[t];
    }
  }
}

template <int RP, bool TC, int TRT>
__global__ void __launch_bounds__(256, (RP <= 64 ? 3 : 1)) update_kernel(float* __restrict__ M, bf16* __restrict__ Mhi,
                                                     bf16* __restrict__ Mlo, bf16* __restrict__ Mlo2,
                                                     float* __restrict__ E, int64_t m0, int64_t rows,
                                                     const float* __restrict__ R, const float* __restrict__ Rs,
                                                     const uint8_t* __restrict__ flags,
                                                     const float* __restrict__ Ginv,
                                                     const bf16* __restrict__ gsplit, float eta,
                                                     float gamma, int momentum, int delta_form, int write_lo,
                                                     int* __restrict__ status) {
  using C = UpdCfg<RP, TC, TRT>;
  constexpr int NV = C::TR * RP / 4 / 256;   // float4 of a tile per thread
  constexpr int CW = C::CW, TR = C::TR, TX = C::TX, CPT = C::CPT, SR = C::SR;
  extern __shared__ __align__(16) float sm[];
  // CUDA cores: G^{-1} (RP x CW) and two tile buffers (TR x RP, row-major
  // like R).  Tensor cores: one tile buffer (TR x SR) and G^{-1}'s bf16
  // pieces, transposed (RP x SB each).
  float* Gs = sm;
  float* Rb = TC ? sm : sm + RP * CW;
  bf16* GhT = reinterpret_cast<bf16*>(sm + TR * SR);
  bf16* GlT = GhT + RP * C::SB;
  if (*(volatile int*)status != 0) return;
  const int cw0 = blockIdx.y * CW;
  const int tx = threadIdx.x % TX, ty = threadIdx.x / TX;
  const int64_t ntiles = (rows + TR - 1) / TR;
  const int64_t total = rows * RP;              // floats of R in this step
  // float4 e of a tile sits at row 4e / RP, column 4e % RP of the staged tile
  auto soff = [](int e) { return ((4 * e) / RP) * SR + (4 * e) % RP; };
  auto issue = [&](int64_t tile, int buf) {
    const int64_t base = tile * TR * RP;
    float* dst = Rb + buf * TR * SR;
#pragma unroll
    for (int u = 0; u < NV; ++u) {
      const int e = threadIdx.x + 256 * u;
      if (base + 4 * e < total) cp_async16(dst + soff(e), R + base + 4 * e);
    }
  };
  int64_t t = blockIdx.x;
  if constexpr (TC) {
    // G^{-1}'s pieces, transposed (GhT[n][k] = hi(G^{-1}[k][n]): a B
    // fragment's pair of k values is one 32-bit load), and the first tile
    for (int e = threadIdx.x; e < RP * C::SB / 4; e += 256) cp_async16(GhT + 8 * e, gsplit + 8 * e);
    if (t < ntiles) issue(t, 0);
    cp_async_commit();
  } else {
    // G^{-1} (its CW columns) and the first tile of R in one copy group
    for (int e = threadIdx.x; e < RP * CW / 4; e += 256) {
      const int k = (4 * e) / CW, c = (4 * e) % CW;
      cp_async16(Gs + 4 * e, Ginv + k * RP + cw0 + c);
    }
    if (t < ntiles) issue(t, 0);
    cp_async_commit();
  }
  int buf = 0;
  for (; t < ntiles; t += gridDim.x, buf ^= (TC ? 0 : 1)) {
    if constexpr (TC) {
      // (the buffer was released by the barrier that ended the last tile)
      if (t != blockIdx.x) issue(t, 0);
    } else if (t + gridDim.x < ntiles) {
      issue(t + gridDim.x, buf ^ 1);
    }
    cp_async_commit();
    const int64_t base = t * TR;
    // the support term of this tile: Rs on the rows flagged as having
    // support in the step's panel (the other rows of Rs are stale)
    float4 sv[NV];
#pragma unroll
    for (int u = 0; u < NV; ++u) {
      const int64_t o = base * RP + 4 * (threadIdx.x + 256 * u);
      sv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (o < total && __ldg(flags + o / RP)) sv[u] = *(const float4*)(Rs + o);
    }
    // this thread's M and E entries, in flight during the product
    float mo[4][CPT], eo[4][CPT];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t li = base + 4 * ty + i;
      const bool live = li < rows;
      const float* mrow = M + (m0 + li) * RP + cw0;
      const float* erow = E + (m0 + li) * RP + cw0;
      if (CPT >= 4) {
#pragma unroll
        for (int j = 0; j < CPT; j += 4) {
          const int c = upd_col<CPT, TX>(tx, j);
          float4 v = make_float4(0.f, 0.f, 0.f, 0.f), w = v;
          if (live) {
            v = *(const float4*)(mrow + c);
            if (momentum) w = *(const float4*)(erow + c);
          }
          mo[i][j] = v.x; mo[i][j + 1] = v.y; mo[i][j + 2] = v.z; mo[i][j + 3] = v.w;
          eo[i][j] = w.x; eo[i][j + 1] = w.y; eo[i][j + 2] = w.z; eo[i][j + 3] = w.w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
          const int c = upd_col<CPT, TX>(tx, j);
          mo[i][j] = live ? mrow[c] : 0.f;
          eo[i][j] = (live && momentum) ? erow[c] : 0.f;
        }
      }
    }
    if constexpr (TC) cp_async_wait_0();
    else cp_async_wait_1();
    // add the support term to the entries this thread copied (its own copies
    // have landed), then publish the tile
#pragma unroll
    for (int u = 0; u < NV; ++u) {
      const int e = threadIdx.x + 256 * u;
      const int64_t o = base * RP + 4 * e;
      if (o < total) {
        float4* d = (float4*)(Rb + buf * TR * SR + soff(e));
        float4 v = *d;
        v.x += sv[u].x; v.y += sv[u].y; v.z += sv[u].z; v.w += sv[u].w;
        *d = v;
      }
    }
    __syncthreads();
    float x[4][CPT];
    if constexpr (TC) {
      // X = (R + Rs) G^{-1} on the tensor cores: both factors as hi + lo
      // bf16 pieces, three products (lo hi, hi lo, hi hi; lo lo dropped), fp32
      // accumulation.  Warp w takes rows 16 (w % RG) .. + 15 and columns
      // (w / RG) WC .. + WC - 1 of the tile's product.
      constexpr int RG = C::RG, WC = C::WC, NT = WC / 8;   // NT: 8-column tiles per warp
      float* Rt = Rb;
      const int lane = threadIdx.x % 32, warp = threadIdx.x / 32, g = lane / 4, c2 = 2 * (lane % 4);
      const int r0 = 16 * (warp % RG), n0 = (warp / RG) * WC;
      float acc[NT][4];
#pragma unroll
      for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < RP / 16; ++ks) {
        const int k0 = 16 * ks;
        uint32_t ah[4], al[4];
        const float2 v0 = *(const float2*)(Rt + (r0 + g) * SR + k0 + c2);
        const float2 v1 = *(const float2*)(Rt + (r0 + g + 8) * SR + k0 + c2);
        const float2 v2 = *(const float2*)(Rt + (r0 + g) * SR + k0 + 8 + c2);
        const float2 v3 = *(const float2*)(Rt + (r0 + g + 8) * SR + k0 + 8 + c2);
        split_pair(v0.x, v0.y, ah[0], al[0]);
        split_pair(v1.x, v1.y, ah[1], al[1]);
        split_pair(v2.x, v2.y, ah[2], al[2]);
        split_pair(v3.x, v3.y, ah[3], al[3]);
#pragma unroll
        for (int n = 0; n < NT; ++n) {
          const int row = (n0 + 8 * n + g) * C::SB + k0 + c2;
          const uint32_t bh0 = *reinterpret_cast<const uint32_t*>(GhT + row);
          const uint32_t bh1 = *reinterpret_cast<const uint32_t*>(GhT + row + 8);
          const uint32_t bl0 = *reinterpret_cast<const uint32_t*>(GlT + row);
          const uint32_t bl1 = *reinterpret_cast<const uint32_t*>(GlT + row + 8);
          mma_16816(acc[n], al, bh0, bh1);
          mma_16816(acc[n], ah, bl0, bl1);
          mma_16816(acc[n], ah, bh0, bh1);
        }
      }
      __syncthreads();   // every warp has read its rows of the tile: X replaces it
#pragma unroll
      for (int n = 0; n < NT; ++n) {
        float* o = Rt + (r0 + g) * SR + n0 + 8 * n + c2;
        *(float2*)o = make_float2(acc[n][0], acc[n][1]);
        *(float2*)(o + 8 * SR) = make_float2(acc[n][2], acc[n][3]);
      }
      __syncthreads();
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float* xr = Rt + (4 * ty + i) * SR;
        if (CPT >= 4) {
#pragma unroll
          for (int j = 0; j < CPT; j += 4) {
            const float4 v = *(const float4*)(xr + upd_col<CPT, TX>(tx, j));
            x[i][j] = v.x; x[i][j + 1] = v.y; x[i][j + 2] = v.z; x[i][j + 3] = v.w;
          }
        } else {
#pragma unroll
          for (int j = 0; j < CPT; ++j) x[i][j] = xr[upd_col<CPT, TX>(tx, j)];
        }
      }
    } else {
    const float* Rt = Rb + buf * TR * RP + (4 * ty) * RP;
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < CPT; ++j) x[i][j] = 0.f;
#pragma unroll 2
    for (int k = 0; k < RP; k += 4) {
      float4 a[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = *(const float4*)(Rt + i * RP + k);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        float b[CPT];
        const float* grow = Gs + (k + kk) * CW;
        if (CPT >= 4) {
#pragma unroll
          for (int j = 0; j < CPT; j += 4) {
            const float4 g = *(const float4*)(grow + upd_col<CPT, TX>(tx, j));
            b[j] = g.x; b[j + 1] = g.y; b[j + 2] = g.z; b[j + 3] = g.w;
          }
        } else {
#pragma unroll
          for (int j = 0; j < CPT; ++j) b[j] = grow[upd_col<CPT, TX>(tx, j)];
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float av = kk == 0 ? a[i].x : kk == 1 ? a[i].y : kk == 2 ? a[i].z : a[i].w;
#pragma unroll
          for (int j = 0; j < CPT; ++j) x[i][j] = fmaf(av, b[j], x[i][j]);
        }
      }
    }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t li = base + 4 * ty + i;
      if (li >= rows) continue;
      const int64_t g = (m0 + li) * RP + cw0;
      bool finite = true;
      float nv[CPT], ev[CPT];
#pragma unroll
      for (int j = 0; j < CPT; ++j) {
        const float u = delta_form ? eta * x[i][j] : eta * (x[i][j] - mo[i][j]);
        ev[j] = momentum ? fmaf(gamma, eo[i][j], u) : u;
        nv[j] = mo[i][j] + ev[j];
        finite = finite && isfinite(nv[j]);
      }
      uint32_t hw[CPT], lw[CPT], l2w[CPT];
#pragma unroll
      for (int j = 0; j < CPT; ++j) {
        const bf16 h = __float2bfloat16_rn(nv[j]);
        const float r1 = nv[j] - __bfloat162float(h);
        const bf16 l = __float2bfloat16_rn(r1);
        hw[j] = __bfloat16_as_ushort(h);
        lw[j] = __bfloat16_as_ushort(l);
        l2w[j] = __bfloat16_as_ushort(__float2bfloat16_rn(r1 - __bfloat162float(l)));
      }
      if (CPT >= 4) {
#pragma unroll
        for (int j = 0; j < CPT; j += 4) {
          const int c = upd_col<CPT, TX>(tx, j);
          *(float4*)(M + g + c) = make_float4(nv[j], nv[j + 1], nv[j + 2], nv[j + 3]);
          if (momentum) *(float4*)(E + g + c) = make_float4(ev[j], ev[j + 1], ev[j + 2], ev[j + 3]);
          *(uint2*)(Mhi + g + c) = make_uint2(hw[j] | (hw[j + 1] << 16), hw[j + 2] | (hw[j + 3] << 16));
          if (write_lo) {
            *(uint2*)(Mlo + g + c) = make_uint2(lw[j] | (lw[j + 1] << 16), lw[j + 2] | (lw[j + 3] << 16));
            *(uint2*)(Mlo2 + g + c) = make_uint2(l2w[j] | (l2w[j + 1] << 16), l2w[j + 2] | (l2w[j + 3] << 16));
          }
        }
      } else {
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
          const int c = upd_col<CPT, TX>(tx, j);
          M[g + c] = nv[j];
          if (momentum) E[g + c] = ev[j];
          Mhi[g + c] = __ushort_as_bfloat16((unsigned short)hw[j]);
          if (write_lo) {
            Mlo[g + c] = __ushort_as_bfloat16((unsigned short)lw[j]);
            Mlo2[g + c] = __ushort_as_bfloat16((unsigned short)l2w[j]);
          }
        }
      }
      if (!finite) set_status(status, NMD_ERR_DIVERGED, (int)(m0 + li), 0);
    }
    __syncthreads();   // the buffer read above is refilled by the next iteration's copy
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Loss, support part: for every stored (i, j), with L = w_i . b_j and
// Shat = max(0, L):
//   a = (S - L)^2,  b = (S - Shat)^2,  mn = min(S, Shat),  mx = max(S, Shat)
// (eqs. SLloss, RMSE, WJD on the support).  When the dense pass summed every
// entry (SUBTRACT: the CUDA-core loss pass), Shat^2 and Shat are subtracted
// again here, with L formed by the same sequential fma chain as that pass so
// the two cancel exactly.  The tensor-core loss pass skips support entries,
// and nothing is subtracted.  One warp per row of S, fp64 sums.
// ---------------------------------------------------------------------------
template <int VPL, bool SUBTRACT>
__global__ void __launch_bounds__(256) loss_sparse_kernel(const int64_t* __restrict__ rowptr,
                                                          const int32_t* __restrict__ col,
                                                          const float* __restrict__ val, int64_t m,
                                                          const float* __restrict__ Wop,
                                                          const float* __restrict__ Bop, int rp,
                                                          double* __restrict__ parts) {
  __shared__ double red[8][4];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  double sa = 0, sb = 0, smn = 0, smx = 0;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; i < m; i += nw) {
    float wv[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int c = lane + 32 * v;
      wv[v] = c < rp ? __ldg(Wop + i * rp + c) : 0.f;
    }
    for (int64_t e0 = rowptr[i]; e0 < rowptr[i + 1]; e0 += 32) {
      // lane l takes entry e0 + l
      const int64_t e = e0 + lane;
      const bool live = e < rowptr[i + 1];
      if (SUBTRACT) {
        if (live) {
          const int64_t j = col[e];
          float L = 0.f;
          for (int c = 0; c < rp; ++c) L = fmaf(__ldg(Wop + i * rp + c), __ldg(Bop + j * rp + c), L);
          const double Ld = L, S = val[e];
          const double sh = Ld > 0 ? Ld : 0.0;
          sa += (S - Ld) * (S - Ld) - sh * sh;
          sb += (S - sh) * (S - sh) - sh * sh;
          smn += S < sh ? S : sh;
          smx += (S > sh ? S : sh) - sh;
        }
      } else {
        const int64_t rem = rowptr[i + 1] - e0;
        const int cnt = rem < 32 ? (int)rem : 32;
        for (int q = 0; q < cnt; ++q) {
          const int64_t j = col[e0 + q];
          float part = 0.f;
#pragma unroll
          for (int v = 0; v < VPL; ++v) {
            const int c = lane + 32 * v;
            part = fmaf(wv[v], c < rp ? __ldg(Bop + j * rp + c) : 0.f, part);
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
          if (lane == q) {
            const double Ld = part, S = val[e0 + q];
            const double sh = Ld > 0 ? Ld : 0.0;
            sa += (S - Ld) * (S - Ld);
            sb += (S - sh) * (S - sh);
            smn += S < sh ? S : sh;
            smx += S > sh ? S : sh;
          }
        }
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sa += __shfl_xor_sync(0xffffffffu, sa, o);
    sb += __shfl_xor_sync(0xffffffffu, sb, o);
    smn += __shfl_xor_sync(0xffffffffu, smn, o);
    smx += __shfl_xor_sync(0xffffffffu, smx, o);
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
  pack_kernel<<<grid_for(N * rp, 256), 256, 0, s>>>(src, src_is_rxN, N, r, rp, f.master, f.hi, f.lo, f.lo2);
}

void launch_unpack(const float* master, bool dst_is_rxN, int64_t N, int r, int rp, float* dst, cudaStream_t s) {
  unpack_kernel<<<grid_for(N * r, 256), 256, 0, s>>>(master, dst_is_rxN, N, r, rp, dst);
}

void launch_gram(const Factor* fq, bool rounded, int64_t q0, int64_t K, int r, int rp, float* parts, int nparts,
                 int64_t chunk, float ridge, float* G, cudaStream_t s) {
  int nt = (rp + 63) / 64;
  dim3 grid(nt * (nt + 1) / 2, nparts);
  if (rounded)
    gram_kernel<bf16><<<grid, 256, 0, s>>>(fq->hi, q0, K, rp, parts, chunk);
  else
    gram_kernel<float><<<grid, 256, 0, s>>>(fq->master, q0, K, rp, parts, chunk);
  gram_reduce_kernel<<<(unsigned)((rp * rp + 255) / 256), 256, 0, s>>>(parts, nparts, r, rp, ridge, G);
}

void launch_small_gemm(const float* A, int64_t lda, const float* B, int64_t ldb, float* C, int64_t ldc, int64_t M,
                       int N, int K, cudaStream_t s) {
  if (M <= 0) return;
  dim3 grid((unsigned)((M + 63) / 64), (unsigned)((N + 63) / 64));
  small_gemm_kernel<<<grid, 256, 0, s>>>(A, lda, B, ldb, C, ldc, M, N, K);
}

void launch_chol_inv(const float* G, int r, int rp, float* Ginv, bf16* gsplit, int* status, cudaStream_t s) {
  switch (rp) {
    case 16: ldlt_inv_reg_kernel<16><<<1, 64, ldlt_reg_smem_bytes(16), s>>>(G, r, Ginv, gsplit, status); break;
    case 32: ldlt_inv_reg_kernel<32><<<1, 128, ldlt_reg_smem_bytes(32), s>>>(G, r, Ginv, gsplit, status); break;
    case 64:
      ldlt_inv_tile_kernel<64><<<1, TileChol<64>::NTHR, TileChol<64>::SMEM, s>>>(G, r, Ginv, gsplit, status);
      break;
    case 128: {
      static std::atomic<int> attr[kMaxDevices];
      per_device(attr, [] {
        return cudaFuncSetAttribute(ldlt_inv_tile_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)TileChol<128>::SMEM) == cudaSuccess ? 1 : 0;
      });
      ldlt_inv_tile_kernel<128><<<1, TileChol<128>::NTHR, TileChol<128>::SMEM, s>>>(G, r, Ginv, gsplit, status);
      break;
    }
    default: {
      static std::atomic<int> attr[kMaxDevices];
      per_device(attr, [] {
        return cudaFuncSetAttribute(ldlt_inv_tile_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)TileChol<256>::SMEM) == cudaSuccess ? 1 : 0;
      });
      ldlt_inv_tile_kernel<256><<<1, TileChol<256>::NTHR, TileChol<256>::SMEM, s>>>(G, r, Ginv, nullptr, status);
    }
  }
}

// ---------------------------------------------------------------------------
// Range search over the normalised factor rows (Sec. 4.3, eqs. nonzeros and
// range-search): L_ij > 0 exactly when ||a^_i - b^_j||^2 < 2, with a^ and b^
// the rows scaled to unit length.  A one-level spatial index: a ball (centre
// c, radius rho) around the normalised nonzero rows of every 128-row M tile
// and of every Q chunk of a step.  By the triangle inequality every pair of
// a tile and a chunk has
//     ||a^ - b^|| >= ||c_A - c_B|| - rho_A - rho_B;
// where that bound is at least sqrt(2 + 2 gamma), every pair has
// a^ . b^ <= -gamma, so L < 0 (or L = 0 for zero rows) on the whole (tile,
// chunk), and the Delta-form dense term -max(0, L) Q adds nothing there: the
// dense kernel skips both of its products for that chunk.
// gamma = 2^-7 covers the bf16 rounding of the operands that the dense
// kernel multiplies (its L differs from the masters' a . b by at most about
// 2^-8 |a| |b|) and its fp32 accumulation; the ball arithmetic is rounded
// outwards by 2^-12 relative plus 2^-14 (the fp32 normalisation of the rows
// is good to about 1e-6).  The balls come from the fp32 masters.
// ---------------------------------------------------------------------------
// Balls of groups of T consecutive rows: groups [0, g1) over the rows of the
// first set (the M tiles), groups [g1, gridDim.x) over the second (the Q
// chunks), in one launch.  Each row is read by RP / 8 lanes (8 columns each,
// two 16-byte loads), so a warp holds 256 / RP rows at once; two passes:
// the mean of the unit vectors of the nonzero rows, then the largest
// distance from it.
struct BallSet {
  const float* X;
  int64_t x0, N;
  int T;
  float* centre;
  float* radius;
};

template <int RP>
__global__ void __launch_bounds__(256) range_ball_kernel(BallSet a, int64_t g1, BallSet b) {
  constexpr int LPR = RP / 8;           // lanes per row
  constexpr int RPW = 32 / LPR;         // rows per warp at once
  __shared__ float part[8][RP];
  __shared__ float cs[RP];
  __shared__ float rmax[8];
  __shared__ int cnt[8];
  const bool first = blockIdx.x < g1;
  const BallSet& S = first ? a : b;
  const int64_t g = first ? blockIdx.x : blockIdx.x - g1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane % LPR, c0 = 8 * sub;   // this lane's 8 columns
  const int64_t r0 = g * S.T, r1 = r0 + S.T < S.N ? r0 + S.T : S.N;
  // the unit vector of row i (zero for a zero row or a row past the group)
  auto unit = [&](int64_t i, float (&v)[8]) {
    if (i < r1) {
      const float4* row = (const float4*)(S.X + (S.x0 + i) * RP + c0);
      const float4 p = __ldg(row), q = __ldg(row + 1);
      v[0] = p.x; v[1] = p.y; v[2] = p.z; v[3] = p.w; v[4] = q.x; v[5] = q.y; v[6] = q.z; v[7] = q.w;
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) v[k] = 0.f;
    }
    float ss = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) ss = fmaf(v[k], v[k], ss);
#pragma unroll
    for (int o = 1; o < LPR; o <<= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const float inv = ss > 0.f ? rsqrtf(ss) : 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] *= inv;
    return ss > 0.f;
  };
  float acc[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) acc[k] = 0.f;
  int n = 0;
  for (int64_t i0 = r0 + warp * RPW; i0 < r1; i0 += 8 * RPW) {
    float v[8];
    if (unit(i0 + lane / LPR, v)) {
      n += sub == 0;
#pragma unroll
      for (int k = 0; k < 8; ++k) acc[k] += v[k];
    }
  }
  // column sums over the warp's row slots, then over the warps
#pragma unroll
  for (int o = LPR; o < 32; o <<= 1) {
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[k] += __shfl_xor_sync(0xffffffffu, acc[k], o);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if (lane < LPR)
#pragma unroll
    for (int k = 0; k < 8; ++k) part[warp][c0 + k] = acc[k];
  if (lane == 0) cnt[warp] = n;
  __syncthreads();
  int ntot = 0;
#pragma unroll
  for (int w = 0; w < 8; ++w) ntot += cnt[w];
  for (int c = threadIdx.x; c < RP; c += 256) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) sum += part[w][c];
    cs[c] = ntot > 0 ? sum / (float)ntot : 0.f;
  }
  __syncthreads();
  float rm = 0.f;
  for (int64_t i0 = r0 + warp * RPW; i0 < r1; i0 += 8 * RPW) {
    float v[8];
    const bool nz = unit(i0 + lane / LPR, v);
    float d2 = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float e = v[k] - cs[c0 + k];
      d2 = fmaf(e, e, d2);
    }
#pragma unroll
    for (int o = 1; o < LPR; o <<= 1) d2 += __shfl_xor_sync(0xffffffffu, d2, o);
    if (nz) rm = fmaxf(rm, d2);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) rm = fmaxf(rm, __shfl_xor_sync(0xffffffffu, rm, o));
  if (lane == 0) rmax[warp] = rm;
  __syncthreads();
  for (int c = threadIdx.x; c < RP; c += 256) S.centre[g * RP + c] = cs[c];
  if (threadIdx.x == 0) {
    float m = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) m = fmaxf(m, rmax[w]);
    S.radius[g] = ntot > 0 ? sqrtf(m) : -1.f;   // -1: the group has no nonzero row
  }
}

// One block per M tile: bit c of word w of the tile's mask is set when the
// ball test clears Q chunk 32 w + c (every pair of the tile and the chunk has
// L <= 0).  A group without a nonzero row has L = 0 against everything.
// Warp w takes chunks w, w + 8, ...; its lanes read a chunk's centre
// together.
template <int RP>
__global__ void __launch_bounds__(256) range_mask_kernel(const float* __restrict__ cm, const float* __restrict__ rm,
                                                         const float* __restrict__ cq, const float* __restrict__ rq,
                                                         int64_t nchunks, int64_t words, uint32_t* __restrict__ mask) {
  constexpr float kOut = 1.0f + 1.0f / 4096.0f;
  constexpr float kIn = 1.0f - 1.0f / 4096.0f;
  constexpr float kThresh = 1.4201f;   // sqrt(2 + 2^-6) (1 + 2^-12) = 1.42007...
  constexpr int CPL = RP >= 32 ? RP / 32 : 1;
  __shared__ float ca[RP];
  __shared__ uint32_t bits[64];
  const int64_t t = blockIdx.x;
  for (int c = threadIdx.x; c < RP; c += 256) ca[c] = cm[t * RP + c];
  const float ra = rm[t];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int64_t w0 = 0; w0 < words; w0 += 64) {
    const int nw = (int)(words - w0 < 64 ? words - w0 : 64);
    __syncthreads();
    if (threadIdx.x < 64) bits[threadIdx.x] = 0u;
    __syncthreads();
    const int64_t cend = (w0 + nw) * 32 < nchunks ? (w0 + nw) * 32 : nchunks;
    for (int64_t c = w0 * 32 + warp; c < cend; c += 8) {
      const float rb = rq[c];
      bool skip;
      if (ra < 0.f || rb < 0.f) {
        skip = true;
      } else {
        float d2 = 0.f;
#pragma unroll
        for (int j = 0; j < CPL; ++j) {
          const int k = lane + 32 * j;
          const float e = k < RP ? ca[k] - cq[c * RP + k] : 0.f;
          d2 = fmaf(e, e, d2);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) d2 += __shfl_xor_sync(0xffffffffu, d2, o);
        const float lb = sqrtf(d2) * kIn - (ra + rb) * kOut - 1.0f / 16384.0f;
        skip = lb >= kThresh;
      }
      if (skip && lane == 0) atomicOr(&bits[(c >> 5) - w0], 1u << (c & 31));
    }
    __syncthreads();
    for (int w = threadIdx.x; w < nw; w += 256) mask[t * words + w0 + w] = bits[w];
  }
}

void launch_range_balls(const float* Xm, int64_t m0, int64_t M, const float* Xq, int64_t q0, int64_t K, int bn,
                        int rp, float* cm, float* rm, float* cq, float* rq, cudaStream_t s) {
  const int64_t g1 = (M + 127) / 128, g2 = (K + bn - 1) / bn;
  if (g1 + g2 == 0) return;
  const BallSet a{Xm, m0, M, 128, cm, rm}, b{Xq, q0, K, bn, cq, rq};
  const unsigned grid = (unsigned)(g1 + g2);
  switch (rp) {
    case 16: range_ball_kernel<16><<<grid, 256, 0, s>>>(a, g1, b); break;
    case 32: range_ball_kernel<32><<<grid, 256, 0, s>>>(a, g1, b); break;
    case 64: range_ball_kernel<64><<<grid, 256, 0, s>>>(a, g1, b); break;
    case 128: range_ball_kernel<128><<<grid, 256, 0, s>>>(a, g1, b); break;
    default: range_ball_kernel<256><<<grid, 256, 0, s>>>(a, g1, b); break;
  }
}

void launch_range_mask(const float* cm, const float* rm, int64_t ntiles, const float* cq, const float* rq,
                       int64_t nchunks, int64_t words, int rp, uint32_t* mask, cudaStream_t s) {
  if (ntiles == 0) return;
  const unsigned g = (unsigned)ntiles;
  switch (rp) {
    case 16: range_mask_kernel<16><<<g, 256, 0, s>>>(cm, rm, cq, rq, nchunks, words, mask); break;
    case 32: range_mask_kernel<32><<<g, 256, 0, s>>>(cm, rm, cq, rq, nchunks, words, mask); break;
    case 64: range_mask_kernel<64><<<g, 256, 0, s>>>(cm, rm, cq, rq, nchunks, words, mask); break;
    case 128: range_mask_kernel<128><<<g, 256, 0, s>>>(cm, rm, cq, rq, nchunks, words, mask); break;
    default: range_mask_kernel<256><<<g, 256, 0, s>>>(cm, rm, cq, rq, nchunks, words, mask); break;
  }
}

static void launch_reduce(const PanelRow* multi, int64_t nmulti, const float* partials, float* R, int64_t m0, int rp,
                          cudaStream_t s) {
  const unsigned grid = (unsigned)nmulti;
  switch (rp) {
    case 16: sparse_reduce_kernel<16><<<grid, 256, 0, s>>>(multi, partials, R, m0); break;
    case 32: sparse_reduce_kernel<32><<<grid, 256, 0, s>>>(multi, partials, R, m0); break;
    case 64: sparse_reduce_kernel<64><<<grid, 256, 0, s>>>(multi, partials, R, m0); break;
    case 128: sparse_reduce_kernel<128><<<grid, 256, 0, s>>>(multi, partials, R, m0); break;
    default: sparse_reduce_kernel<256><<<grid, 256, 0, s>>>(multi, partials, R, m0); break;
  }
}

template <int RP>
static bool launch_sparse_smem(const StepArgs& a, const PanelRow* rows, int64_t nrows, const PanelRow* whole,
                               int64_t nwhole, const PanelRow* seg, int64_t nseg, const int32_t* qidx,
                               const float* vals, float* R, float* partials, cudaStream_t s) {
  using C = SpSmem<RP>;
  static std::atomic<int> attr[kMaxDevices];
  if (!per_device(attr, [] {
        return cudaFuncSetAttribute(sparse_smem_kernel<RP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)kSparseQBytes) == cudaSuccess ? 1 : 0;
      }))
    return false;
  const int64_t nitems = nrows + nwhole + nseg;
  const int64_t grid = std::min<int64_t>(a.num_sms, (nitems + C::WARPS - 1) / C::WARPS);
  const size_t smem = (size_t)a.K * RP * sizeof(bf16);
  sparse_smem_kernel<RP><<<(unsigned)grid, 32 * C::WARPS, smem, s>>>(rows, nrows, whole, nwhole, seg, nseg, a.fm->hi,
                                                                    a.m0, a.fq->hi, a.q0, a.K, qidx, vals, R,
                                                                    partials);
  return true;
}

int launch_sparse(const StepArgs& a, const PanelRow* rows, int64_t nrows, const PanelRow* whole, int64_t nwhole,
                  const PanelRow* seg, int64_t nseg, const PanelRow* multi, int64_t nmulti, const int32_t* qidx,
                  const float* vals, float* R, float* partials, int64_t seg_first, cudaStream_t s) {
  // slice w of `seg` is slice seg_first + w of its block, whose partial slot
  // the reduction (multi[].beg, relative to the block) reads
  float* seg_partials = partials + seg_first * a.rp;
  // the Q-side block in shared memory where its bf16 rows fit
  if (a.precision == NMD_BF16 && (a.rp == 16 || a.rp == 32) && a.K * a.rp * 2 <= (int64_t)kSparseQBytes &&
      nrows + nwhole + nseg > 0) {
    const bool ok = a.rp == 16 ? launch_sparse_smem<16>(a, rows, nrows, whole, nwhole, seg, nseg, qidx, vals, R,
                                                        seg_partials, s)
                               : launch_sparse_smem<32>(a, rows, nrows, whole, nwhole, seg, nseg, qidx, vals, R,
                                                        seg_partials, s);
    if (ok) {
      if (nseg > 0) launch_reduce(multi, nmulti, partials, R, a.m0, a.rp, s);
      return 1 + (nseg > 0);
    }
  }
  // The support term reads the same factor values as the rest of the step's
  // least-squares problem: the bf16 pieces in the bf16 mode (whose dense term
  // and Gram matrix are formed from them), the fp32 masters otherwise.
#define NMD_SP(RPV, LPE, CPL, TT, MOP, QOP)                                                                  \
  do {                                                                                                       \
    if (nrows > 0) {                                                                                         \
      constexpr int rpw = 32 / ((RPV) / (16 / (int)sizeof(TT)) < 32 ? (RPV) / (16 / (int)sizeof(TT)) : 32);  \
      const int64_t nb = (nrows + 8 * rpw - 1) / (8 * rpw);                                                  \
      sparse_group_kernel<RPV, TT><<<(unsigned)nb, 256, 0, s>>>(rows, nrows, MOP, a.m0, QOP, qidx, vals, R); \
    }                                                                                                        \
    if (nwhole > 0)                                                                                          \
      sparse_long_kernel<LPE, CPL, TT><<<(unsigned)((nwhole + 7) / 8), 256, 0, s>>>(                          \
          whole, nwhole, MOP, a.m0, QOP, qidx, vals, R, nullptr, a.rp);                                      \
    if (nseg > 0) {                                                                                          \
      sparse_long_kernel<LPE, CPL, TT><<<(unsigned)((nseg + 7) / 8), 256, 0, s>>>(                            \
          seg, nseg, MOP, a.m0, QOP, qidx, vals, R, seg_partials, a.rp);                                     \
      launch_reduce(multi, nmulti, partials, R, a.m0, a.rp, s);                                              \
    }                                                                                                        \
  } while (0)
#define NMD_SP2(RPV, LPE, CPL)                                                              \
  do {                                                                                      \
    if (a.precision == NMD_BF16) NMD_SP(RPV, LPE, CPL, bf16, a.fm->hi, a.fq->hi);           \
    else NMD_SP(RPV, LPE, CPL, float, a.fm->master, a.fq->master);                          \
  } while (0)
  switch (a.rp) {
    case 16: NMD_SP2(16, 1, 16); break;
    case 32: NMD_SP2(32, 1, 32); break;
    case 64: NMD_SP2(64, 2, 32); break;
    case 128: NMD_SP2(128, 4, 32); break;
    default: NMD_SP2(256, 8, 32); break;
  }
#undef NMD_SP2
#undef NMD_SP
  return (nrows > 0) + (nwhole > 0) + 2 * (nseg > 0);
}

template <int RP, bool TC, int TRT = 64>
static void update_rp(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags, const float* Ginv,
                      const bf16* gsplit, float eta, float gamma, bool momentum, int* status, cudaStream_t s) {
  using C = UpdCfg<RP, TC, TRT>;
  // the attribute and the occupancy belong to the current device
  static std::atomic<int> cache[kMaxDevices];
  const int per_sm = per_device(cache, [] {
    int n = 0;
    cudaFuncSetAttribute(update_kernel<RP, TC, TRT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    // at r_pad <= 64 the largest shared-memory configuration, like the dense
    // kernel's, so that an SM running update blocks can take a dense CTA and
    // vice versa
    if (RP <= 64) cudaFuncSetAttribute(update_kernel<RP, TC, TRT>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, update_kernel<RP, TC, TRT>, 256, C::SMEM) != cudaSuccess ||
        n < 1)
      n = 1;
    return n;
  });
  // one tile per block: blocks retire every few microseconds, so that the
  // higher-priority streams' kernels (the dense kernel, the next step's Gram
  // chain and support term) get SM slots while a deferred update runs.  (One
  // persistent block per SM instead slowed the dense kernel beside it.)
  // per_sm only bounds the grid when the tiles exceed 65,535 waves' worth
  const int64_t tiles = (a.M + C::TR - 1) / C::TR;
  dim3 grid((unsigned)std::min<int64_t>(tiles, (int64_t)a.num_sms * per_sm * 65535), RP / C::CW);
  const Factor& f = *a.fm;
  update_kernel<RP, TC, TRT><<<grid, 256, C::SMEM, s>>>(f.master, f.hi, f.lo, f.lo2, f.E, a.m0, a.M, R, Rs, flags, Ginv,
                                                   gsplit, eta, gamma, momentum, a.epilogue == NMD_EPI_DELTA,
                                                   a.precision == NMD_FP32, status);
}

// X = (R + Rs) G^{-1}: in the bf16 mode on the tensor cores (two bf16 pieces
// per factor, three products, fp32 accumulation: mma.sync, since the SMs the
// deferred update shares with the dense kernel have no tensor memory free),
// in the other modes on the CUDA cores in fp32
void launch_update(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags, const float* Ginv,
                   const bf16* gsplit, float eta, float gamma, bool momentum, int* status, cudaStream_t s) {
  const bool tc = a.precision == NMD_BF16 && gsplit != nullptr;
  // 32-row tiles where the rows fill fewer 64-row tiles than there are SMs
  const bool small = a.M < (int64_t)a.num_sms * 64;
  switch (a.rp) {
#define NMD_UPD(RPV)                                                                                          \
  (!tc ? update_rp<RPV, false>(a, R, Rs, flags, Ginv, gsplit, eta, gamma, momentum, status, s)                 \
       : (small && RPV >= 32) ? update_rp<RPV, true, (RPV >= 32 ? 32 : 64)>(a, R, Rs, flags, Ginv, gsplit, eta, \
                                                                            gamma, momentum, status, s)        \
                              : update_rp<RPV, true>(a, R, Rs, flags, Ginv, gsplit, eta, gamma, momentum, status, s))
    case 16: NMD_UPD(16); break;
    case 32: NMD_UPD(32); break;
    case 64: NMD_UPD(64); break;
    case 128: NMD_UPD(128); break;
    default: update_rp<256, false>(a, R, Rs, flags, Ginv, gsplit, eta, gamma, momentum, status, s); break;
#undef NMD_UPD
  }
}

// R += Rs on the flagged rows (the terms of a step without update)
__global__ void combine_kernel(float* __restrict__ R, const float* __restrict__ Rs,
                               const uint8_t* __restrict__ flags, int64_t n, int rp) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    if (flags[i / rp]) R[i] += Rs[i];
}

void launch_combine(float* R, const float* Rs, const uint8_t* flags, int64_t rows, int rp, cudaStream_t s) {
  combine_kernel<<<grid_for(rows * rp, 256), 256, 0, s>>>(R, Rs, flags, rows * rp, rp);
}

void launch_loss_sparse(const nmd_handle* h, double* parts, int nparts, cudaStream_t s) {
  // fp32 masters in every precision, like the support correction of the update
  const bool subtract = h->opt.precision == NMD_SIMT;
#define NMD_LS(V)                                                                                          \
  do {                                                                                                     \
    if (subtract)                                                                                          \
      loss_sparse_kernel<V, true><<<nparts, 256, 0, s>>>(h->ws.rowptr, h->ws.col, h->ws.val, h->m,           \
                                                        h->W.master, h->B.master, h->rp, parts);           \
    else                                                                                                   \
      loss_sparse_kernel<V, false><<<nparts, 256, 0, s>>>(h->ws.rowptr, h->ws.col, h->ws.val, h->m,          \
                                                         h->W.master, h->B.master, h->rp, parts);          \
  } while (0)
  switch (h->rp) {
    case 16: case 32: NMD_LS(1); break;
    case 64: NMD_LS(2); break;
    case 128: NMD_LS(4); break;
    default: NMD_LS(8); break;
  }
#undef NMD_LS
}

void launch_loss_final(const double* dparts, int nd, const double* sparts, int ns, double* out, cudaStream_t s) {
  loss_final_kernel<<<1, 256, 0, s>>>(dparts, nd, sparts, ns, out);
}

}  // namespace nmd
