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
      if (ta != tb) Qb[rr][cc] = (ok && cc < wb) ? Q[(q0 + k) * rp + tb * 64 + cc] : 0.f;
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
// Thread (ty, tx) of a T x T block owns the entries (ty + T a, tx + T b).
template <int T>
__global__ void __launch_bounds__(T * T) ginv_kernel(const float* __restrict__ parts, int nparts, int r, int rp,
                                                     float ridge, float* __restrict__ Gout,
                                                     float* __restrict__ Ginv, float* __restrict__ scratch,
                                                     int* __restrict__ status, int use_smem) {
  extern __shared__ float sm[];
  float* A = use_smem ? sm : scratch;             // r x r
  __shared__ float rowk[256];
  __shared__ float diag0[256];
  __shared__ int bad;
  const int tx = threadIdx.x % T, ty = threadIdx.x / T;
  if (threadIdx.x == 0) bad = 0;
  for (int i = ty; i < r; i += T)
    for (int j = tx; j < r; j += T) {
      const int a = max(i, j), b = min(i, j);     // the partials hold the lower triangle
      const float* src = parts + (size_t)a * rp + b;
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      int p = 0;
      for (; p + 8 <= nparts; p += 8)
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] += __ldg(src + (size_t)(p + q) * rp * rp);
      for (; p < nparts; ++p) acc[0] += __ldg(src + (size_t)p * rp * rp);
      float sum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
      if (i == j) {
        sum += ridge;
        diag0[i] = sum;
      }
      A[i * r + j] = sum;
    }
  __syncthreads();
  for (int i = ty; i < rp; i += T)
    for (int j = tx; j < rp; j += T) Gout[i * rp + j] = (i < r && j < r) ? A[i * r + j] : 0.f;
  const float tol = 4.0f * (float)r * FLT_EPSILON;
  for (int k = 0; k < r; ++k) {
    const float d = A[k * r + k];
    if (!(d > tol * diag0[k]) || !isfinite(d)) {
      if (threadIdx.x == 0) {
        bad = 1;
        set_status(status, NMD_ERR_NOT_SPD, k, 0);
      }
      break;   // uniform: every thread read the same d
    }
    for (int j = threadIdx.x; j < r; j += T * T) rowk[j] = A[k * r + j];
    __syncthreads();
    const float inv = 1.0f / d;
    for (int i = ty; i < r; i += T) {
      const float ri = rowk[i] * inv;
      for (int j = tx; j < r; j += T) {
        float v;
        if (i == k && j == k) v = -inv;
        else if (i == k) v = rowk[j] * inv;
        else if (j == k) v = ri;                  // symmetric: a_ik = a_ki
        else v = A[i * r + j] - ri * rowk[j];
        A[i * r + j] = v;
      }
    }
    __syncthreads();
  }
  __syncthreads();
  for (int i = ty; i < rp; i += T)
    for (int j = tx; j < rp; j += T) {
      float v = 0.f;
      if (!bad && i < r && j < r) v = -0.5f * (A[i * r + j] + A[j * r + i]);   // symmetrise
      Ginv[i * rp + j] = v;
    }
}

// Register-resident variant for rp <= 128: thread t owns row t / 4 and the
// rp / 4 contiguous columns (t % 4) rp / 4 ... of it.  Before pivot k the
// owners of row k publish it to shared memory (two alternating buffers, one
// barrier per pivot); every thread then updates its own entries from that
// row alone, using the symmetry a_ik = a_ki.  Each update is written so that
// (i, j) and (j, i) round identically (the product a_ik a_kj is formed
// before the division), so the matrix stays exactly symmetric.  The partial
// Gram matrices are summed in part order first.
template <int RP>
__global__ void __launch_bounds__(RP * 4) ginv_reg_kernel(const float* __restrict__ parts, int nparts, int r,
                                                          float ridge, float* __restrict__ Gout,
                                                          float* __restrict__ Ginv, int* __restrict__ status) {
  constexpr int CPT = RP / 4;
  __shared__ __align__(16) float rk[2][RP];
  __shared__ float diag0[RP];
  const int i = threadIdx.x / 4, c0 = (threadIdx.x % 4) * CPT;
  // the partials hold the entries whose 64-row tile is >= their 64-column tile
  const bool direct = (i / 64) >= (c0 / 64);
  float a[CPT];
#pragma unroll
  for (int j = 0; j < CPT; ++j) a[j] = 0.f;
#pragma unroll 4
  for (int p = 0; p < nparts; ++p) {
    const float* src = parts + (size_t)p * RP * RP;
    if (direct) {
#pragma unroll
      for (int j = 0; j < CPT; j += 4) {
        const float4 v = __ldg((const float4*)(src + i * RP + c0 + j));
        a[j] += v.x; a[j + 1] += v.y; a[j + 2] += v.z; a[j + 3] += v.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < CPT; ++j) a[j] += __ldg(src + (c0 + j) * RP + i);
    }
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j)
    if (c0 + j == i && i < r) {
      a[j] += ridge;
      diag0[i] = a[j];
    }
#pragma unroll
  for (int j = 0; j < CPT; ++j) Gout[i * RP + c0 + j] = (i < r && c0 + j < r) ? a[j] : 0.f;
  const float tol = 4.0f * (float)r * FLT_EPSILON;
  bool bad = false;
  for (int k = 0; k < r; ++k) {
    float* rb = rk[k & 1];
    if (i == k) {
#pragma unroll
      for (int j = 0; j < CPT; j += 4) *(float4*)(rb + c0 + j) = make_float4(a[j], a[j + 1], a[j + 2], a[j + 3]);
    }
    __syncthreads();
    const float d = rb[k];
    if (!(d > tol * diag0[k]) || !isfinite(d)) {   // uniform: every thread read the same d
      bad = true;
      if (threadIdx.x == 0) set_status(status, NMD_ERR_NOT_SPD, k, 0);
      break;
    }
    const float inv = 1.0f / d;
    if (i == k) {
#pragma unroll
      for (int j = 0; j < CPT; ++j) a[j] = (c0 + j == k) ? -inv : a[j] * inv;
    } else {
      const float ri = rb[i];
#pragma unroll
      for (int j = 0; j < CPT; ++j) {
        const float rj = rb[c0 + j];
        a[j] = (c0 + j == k) ? ri * inv : fmaf(-(ri * rj), inv, a[j]);
      }
    }
  }
#pragma unroll
  for (int j = 0; j < CPT; ++j) Ginv[i * RP + c0 + j] = (!bad && i < r && c0 + j < r) ? -a[j] : 0.f;
}

// ---------------------------------------------------------------------------
// Sparse correction: for every panel row i and entry (i, k) in the block,
// L_ik = m_i . q_k, c = S_ik - min(0, L_ik), R_i += c q_k (fp32 masters).
// This kernel takes the rows with at most kShort entries in the panel: one
// warp per row; the lanes first fetch the entries' indices and values (one
// per lane), then NE entries at a time are processed with their q rows in
// flight together, lanes over the r columns; the accumulation order over
// the entries stays ascending.  The result goes to Rs, the support term of
// R, one writer per row (or to a partial slot when `partials` is given).
// Rs is written only on the rows with support in the block's panel; a flag
// byte per row tells the update which rows of Rs to add, so the other rows
// are neither read nor cleared.  Longer rows: sparse_long_kernel below.
// ---------------------------------------------------------------------------
template <int VPL, int NE>
__global__ void __launch_bounds__(256) sparse_rows_kernel(const PanelRow* __restrict__ rows, int64_t nrows,
                                                          const float* __restrict__ Mop, int64_t m0,
                                                          const float* __restrict__ Qop,
                                                          const int32_t* __restrict__ qidx,
                                                          const float* __restrict__ vals,
                                                          float* __restrict__ R, float* __restrict__ partials,
                                                          int rp) {
  const int lane = threadIdx.x & 31;
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  if (w >= nrows) return;
  const PanelRow pr = rows[w];
  const int64_t i = pr.row;
  int kl = 0;
  float sl = 0.f;
  if (lane < pr.len) {
    kl = qidx[pr.beg + lane];
    sl = vals[pr.beg + lane];
  }
  float mv[VPL], acc[VPL];
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane + 32 * v;
    mv[v] = c < rp ? __ldg(Mop + i * rp + c) : 0.f;
    acc[v] = 0.f;
  }
  for (int e = 0; e < pr.len; e += NE) {
    float qv[NE][VPL], part[NE];
    float sv[NE];
#pragma unroll
    for (int j = 0; j < NE; ++j) {
      const int k = __shfl_sync(0xffffffffu, kl, (e + j) & 31);
      sv[j] = __shfl_sync(0xffffffffu, sl, (e + j) & 31);
      const bool live = e + j < pr.len;
      part[j] = 0.f;
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int c = lane + 32 * v;
        qv[j][v] = (live && c < rp) ? __ldg(Qop + (int64_t)k * rp + c) : 0.f;
        part[j] = fmaf(mv[v], qv[j][v], part[j]);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int j = 0; j < NE; ++j) part[j] += __shfl_xor_sync(0xffffffffu, part[j], o);
#pragma unroll
    for (int j = 0; j < NE; ++j) {
      const float cval = sv[j] - fminf(0.f, part[j]);        // zero for the padding entries (q = 0)
#pragma unroll
      for (int v = 0; v < VPL; ++v) acc[v] = fmaf(cval, qv[j][v], acc[v]);
    }
  }
  float* dst = partials ? partials + w * rp : R + (i - m0) * rp;
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int c = lane + 32 * v;
    if (c < rp) dst[c] = acc[v];
  }
}

// Long rows (more than kShort entries in the panel): one warp per row or kSeg
// slice with the lanes over the entries.  LPE = rp / 32 lanes share an entry
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
template <int LPE, int CPL>
__global__ void __launch_bounds__(256, 2) sparse_long_kernel(const PanelRow* __restrict__ segs, int64_t nseg,
                                                          const float* __restrict__ Mop, int64_t m0,
                                                          const float* __restrict__ Qop,
                                                          const int32_t* __restrict__ qidx,
                                                          const float* __restrict__ vals,
                                                          float* __restrict__ R, float* __restrict__ partials,
                                                          int rp) {
  constexpr int EPW = 32 / LPE;
  constexpr int CS = 36;                       // floats per staged chunk (32 + 4 padding)
  constexpr int NPF = 4;                       // entry iterations whose indices are fetched together
  __shared__ __align__(16) float stage[8][32 * CS];
  const int lane = threadIdx.x & 31;
  const int64_t w = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  if (w >= nseg) return;
  float* buf = stage[(threadIdx.x >> 5) & 7];
  const PanelRow pr = segs[w];
  const int sub = lane % LPE, slot = lane / LPE;
  const int64_t i = pr.row;
  float mv[CPL], acc[CPL];
  {
    const float4* m4 = (const float4*)(Mop + i * rp + 32 * sub);
#pragma unroll
    for (int c = 0; c < CPL / 4; ++c) {
      const float4 v = __ldg(m4 + c);
      mv[4 * c] = v.x; mv[4 * c + 1] = v.y; mv[4 * c + 2] = v.z; mv[4 * c + 3] = v.w;
    }
  }
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
      // stage: float4 f = lane + 32 u (u < CPL / 4) of the 32 chunks; chunk
      // f / 8 is columns 32 (chunk % LPE) ... of entry slot chunk / LPE
#pragma unroll
      for (int u = 0; u < CPL / 4; ++u) {
        const int f = lane + 32 * u;
        const int chunk = f / (CPL / 4), part = f % (CPL / 4);
        const int ke = __shfl_sync(0xffffffffu, kk[t], (chunk / LPE) * LPE);
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (ke >= 0) v = __ldg((const float4*)(Qop + (int64_t)ke * rp + 32 * (chunk % LPE)) + part);
        *(float4*)(buf + chunk * CS + 4 * part) = v;
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
// pieces (the third piece only where the fp32-accurate mode reads it).
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
template <int RP>
struct UpdCfg {
  static constexpr int CW = RP <= 128 ? RP : 128;   // output columns per block
  static constexpr int TR = RP <= 128 ? 64 : 32;    // rows per tile
  static constexpr int TY = TR / 4;                  // row groups of four
  static constexpr int TX = 256 / TY;                // column groups
  static constexpr int CPT = CW / TX;                // columns per thread (1, 2, 4 or 8)
  static constexpr size_t SMEM = ((size_t)RP * CW + 2 * (size_t)TR * RP) * sizeof(float);
  static_assert(CPT >= 1 && (CPT < 4 || CPT % 4 == 0), "column split");
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

template <int RP>
__global__ void __launch_bounds__(256, (RP <= 64 ? 3 : 1)) update_kernel(float* __restrict__ M, bf16* __restrict__ Mhi,
                                                     bf16* __restrict__ Mlo, bf16* __restrict__ Mlo2,
                                                     float* __restrict__ E, int64_t m0, int64_t rows,
                                                     const float* __restrict__ R, const float* __restrict__ Rs,
                                                     const uint8_t* __restrict__ flags,
                                                     const float* __restrict__ Ginv, float eta,
                                                     float gamma, int momentum, int delta_form, int write_lo2,
                                                     int* __restrict__ status) {
  using C = UpdCfg<RP>;
  constexpr int NV = C::TR * RP / 4 / 256;   // float4 of a tile per thread
  constexpr int CW = C::CW, TR = C::TR, TX = C::TX, CPT = C::CPT;
  extern __shared__ __align__(16) float sm[];
  float* Gs = sm;                               // RP x CW
  float* Rb = sm + RP * CW;                     // 2 x TR x RP, row-major like R
  if (*(volatile int*)status != 0) return;
  const int cw0 = blockIdx.y * CW;
  const int tx = threadIdx.x % TX, ty = threadIdx.x / TX;
  const int64_t ntiles = (rows + TR - 1) / TR;
  const int64_t total = rows * RP;              // floats of R in this step
  auto issue = [&](int64_t tile, int buf) {
    const int64_t base = tile * TR * RP;
    float* dst = Rb + buf * TR * RP;
#pragma unroll
    for (int u = 0; u < NV; ++u) {
      const int e = threadIdx.x + 256 * u;
      if (base + 4 * e < total) cp_async16(dst + 4 * e, R + base + 4 * e);
    }
  };
  int64_t t = blockIdx.x;
  // G^{-1} (its CW columns) and the first tile of R in one copy group
  for (int e = threadIdx.x; e < RP * CW / 4; e += 256) {
    const int k = (4 * e) / CW, c = (4 * e) % CW;
    cp_async16(Gs + 4 * e, Ginv + k * RP + cw0 + c);
  }
  if (t < ntiles) issue(t, 0);
  cp_async_commit();
  int buf = 0;
  for (; t < ntiles; t += gridDim.x, buf ^= 1) {
    if (t + gridDim.x < ntiles) issue(t + gridDim.x, buf ^ 1);
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
    cp_async_wait_1();
    // add the support term to the entries this thread copied (its own copies
    // have landed), then publish the tile
#pragma unroll
    for (int u = 0; u < NV; ++u) {
      const int e = threadIdx.x + 256 * u;
      const int64_t o = base * RP + 4 * e;
      if (o < total) {
        float4* d = (float4*)(Rb + buf * TR * RP + 4 * e);
        float4 v = *d;
        v.x += sv[u].x; v.y += sv[u].y; v.z += sv[u].z; v.w += sv[u].w;
        *d = v;
      }
    }
    __syncthreads();
    const float* Rt = Rb + buf * TR * RP + (4 * ty) * RP;
    float x[4][CPT];
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
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t li = base + 4 * ty + i;
      if (li >= rows) break;
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
          *(uint2*)(Mlo + g + c) = make_uint2(lw[j] | (lw[j + 1] << 16), lw[j + 2] | (lw[j + 3] << 16));
          if (write_lo2)
            *(uint2*)(Mlo2 + g + c) = make_uint2(l2w[j] | (l2w[j + 1] << 16), l2w[j + 2] | (l2w[j + 3] << 16));
        }
      } else {
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
          const int c = upd_col<CPT, TX>(tx, j);
          M[g + c] = nv[j];
          if (momentum) E[g + c] = ev[j];
          Mhi[g + c] = __ushort_as_bfloat16((unsigned short)hw[j]);
          Mlo[g + c] = __ushort_as_bfloat16((unsigned short)lw[j]);
          if (write_lo2) Mlo2[g + c] = __ushort_as_bfloat16((unsigned short)l2w[j]);
        }
      }
      if (!finite) set_status(status, NMD_ERR_DIVERGED, (int)(m0 + li), 0);
    }
    __syncthreads();   // the buffer read above is refilled by the next iteration's copy
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
}

template <typename T>
__device__ __forceinline__ float ld(const T* p);
template <>
__device__ __forceinline__ float ld<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld<bf16>(const bf16* p) { return __bfloat162float(*p); }

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
  const size_t smem = (size_t)r * r * sizeof(float);
  const int use_smem = smem <= 200 * 1024;
  if (rp <= 128) {
    switch (rp) {
      case 16: ginv_reg_kernel<16><<<1, 64, 0, s>>>(parts, nparts, r, ridge, G, Ginv, status); break;
      case 32: ginv_reg_kernel<32><<<1, 128, 0, s>>>(parts, nparts, r, ridge, G, Ginv, status); break;
      case 64: ginv_reg_kernel<64><<<1, 256, 0, s>>>(parts, nparts, r, ridge, G, Ginv, status); break;
      default: ginv_reg_kernel<128><<<1, 512, 0, s>>>(parts, nparts, r, ridge, G, Ginv, status); break;
    }
  } else {
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(ginv_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
      attr = true;
    }
    ginv_kernel<32><<<1, 1024, use_smem ? smem : 0, s>>>(parts, nparts, r, rp, ridge, G, Ginv, scratch, status,
                                                         use_smem);
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

void launch_sparse(const StepArgs& a, const PanelRow* rows, int64_t nrows, const PanelRow* whole, int64_t nwhole,
                   const PanelRow* seg, int64_t nseg, const PanelRow* multi, int64_t nmulti, const int32_t* qidx,
                   const float* vals, float* R, float* partials, cudaStream_t s) {
  // The support correction always reads the fp32 masters, in every precision:
  // on rows with few support entries the term S_ik q_k dominates R_i and is
  // not averaged over many products, so rounding q_k to bf16 there would put
  // its full relative error (up to 2^-9) into the update.
  const float* Mop = a.fm->master;
  const float* Qop = a.fq->master;
#define NMD_SP(V, LPE, CPL)                                                                                  \
  do {                                                                                                       \
    if (nrows > 0)                                                                                           \
      sparse_rows_kernel<V, 4><<<(unsigned)((nrows + 7) / 8), 256, 0, s>>>(rows, nrows, Mop, a.m0, Qop, qidx, \
                                                                           vals, R, nullptr, a.rp);         \
    if (nwhole > 0)                                                                                          \
      sparse_long_kernel<LPE, CPL><<<(unsigned)((nwhole + 7) / 8), 256, 0, s>>>(whole, nwhole, Mop, a.m0, Qop, \
                                                                                qidx, vals, R, nullptr, a.rp); \
    if (nseg > 0) {                                                                                          \
      sparse_long_kernel<LPE, CPL><<<(unsigned)((nseg + 7) / 8), 256, 0, s>>>(seg, nseg, Mop, a.m0, Qop, qidx, \
                                                                              vals, R, partials, a.rp);      \
      launch_reduce(multi, nmulti, partials, R, a.m0, a.rp, s);                                              \
    }                                                                                                        \
  } while (0)
  switch (a.rp) {
    case 16: NMD_SP(1, 1, 16); break;
    case 32: NMD_SP(1, 1, 32); break;
    case 64: NMD_SP(2, 2, 32); break;
    case 128: NMD_SP(4, 4, 32); break;
    default: NMD_SP(8, 8, 32); break;
  }
#undef NMD_SP
}

template <int RP>
static void update_rp(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags, const float* Ginv,
                      float eta, float gamma, bool momentum, int* status, cudaStream_t s) {
  using C = UpdCfg<RP>;
  static int per_sm = 0;
  if (per_sm == 0) {
    cudaFuncSetAttribute(update_kernel<RP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, update_kernel<RP>, 256, C::SMEM) != cudaSuccess ||
        per_sm < 1)
      per_sm = 1;
  }
  const int64_t tiles = (a.M + C::TR - 1) / C::TR;
  dim3 grid((unsigned)std::min<int64_t>(tiles, (int64_t)a.num_sms * per_sm), RP / C::CW);
  const Factor& f = *a.fm;
  update_kernel<RP><<<grid, 256, C::SMEM, s>>>(f.master, f.hi, f.lo, f.lo2, f.E, a.m0, a.M, R, Rs, flags, Ginv, eta,
                                               gamma,
                                               momentum, a.epilogue == NMD_EPI_DELTA,
                                               a.precision == NMD_FP32, status);
}

void launch_update(const StepArgs& a, const float* R, const float* Rs, const uint8_t* flags, const float* Ginv,
                   float eta, float gamma, bool momentum, int* status, cudaStream_t s) {
  switch (a.rp) {
    case 16: update_rp<16>(a, R, Rs, flags, Ginv, eta, gamma, momentum, status, s); break;
    case 32: update_rp<32>(a, R, Rs, flags, Ginv, eta, gamma, momentum, status, s); break;
    case 64: update_rp<64>(a, R, Rs, flags, Ginv, eta, gamma, momentum, status, s); break;
    case 128: update_rp<128>(a, R, Rs, flags, Ginv, eta, gamma, momentum, status, s); break;
    default: update_rp<256>(a, R, Rs, flags, Ginv, eta, gamma, momentum, status, s); break;
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
