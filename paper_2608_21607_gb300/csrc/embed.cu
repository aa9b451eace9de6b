// The cell embedding and the nearest-neighbour search of Sec. 5.3.
//
// Embedding (eqs. Lsvd and embed): for a square S the rank-r model
// L = A B^T (A = W, B = H^T, both n x r) has the SVD L = U Sigma V^T, and cell
// i is the unit vector xi_i ~ [u_i, v_i] Sigma^{1/2}.  L itself is never
// formed:
//   G_A = A^T A = P_A Lambda_A P_A^T,  G_B = B^T B = P_B Lambda_B P_B^T
//   (eigendecompositions, so that R_A = Lambda_A^{1/2} P_A^T satisfies
//   R_A^T R_A = G_A and A = Q_A R_A with Q_A = A R_A^{-1} orthonormal),
//   C = R_A R_B^T = U' Sigma V'^T  (r x r SVD), so L = (Q_A U') Sigma (Q_B V')^T,
//   u_i Sigma^{1/2} = a_i R_A^{-1} U' Sigma^{1/2} = a_i T_A with
//   T_A = R_B^T V' Sigma^{-1/2} = P_B Lambda_B^{1/2} V' Sigma^{-1/2}
//   (from U' Sigma = R_A R_B^T V'), and likewise
//   v_i Sigma^{1/2} = b_i T_B, T_B = P_A Lambda_A^{1/2} U' Sigma^{-1/2}.
// The Gram matrices come from the solver's Gram kernel; the three r x r
// decompositions run in one thread block (one-sided Jacobi); one more kernel
// forms and normalises the n rows.
//
// Nearest neighbours: the tensor-core kernel's nearest-neighbour pass over
// the points (three bf16 pieces per coordinate, as in the fp32-accurate
// mode), then one kernel decodes the per-row keys and counts the label
// disagreements of the held-out 1-NN error.
#include <cfloat>
#include <cstdio>

#include "nmd_internal.cuh"

namespace nmd {
namespace {

constexpr int kEmbedMaxRank = 128;   // xi has 2r <= 256 coordinates (the kernels' largest r_pad)

// One-sided Jacobi (Hestenes): the columns of X (n x n, column k at X + k n)
// are rotated in pairs until every pair is orthogonal to working precision
// (|x_p . x_q| <= 2 n eps |x_p| |x_q|, at most 60 sweeps); V (same layout)
// accumulates the rotations, so that on return X = X_in V.  In each of the
// n2 - 1 steps of a sweep (n2 = n rounded up to even) the round-robin
// ordering gives n2 / 2 disjoint pairs, one warp per pair; a rotation with
// t = tan(theta) = sign(zeta) / (|zeta| + sqrt(1 + zeta^2)),
// zeta = (|x_q|^2 - |x_p|^2) / (2 x_p . x_q), makes the pair orthogonal.
__device__ void jacobi(float* X, float* V, int n, volatile int* changed) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const int n2 = n + (n & 1);
  const float tol = 2.0f * (float)n * FLT_EPSILON;
  for (int e = threadIdx.x; e < n * n; e += blockDim.x) V[e] = (e / n == e % n) ? 1.f : 0.f;
  __syncthreads();
  for (int sweep = 0; sweep < 60; ++sweep) {
    if (threadIdx.x == 0) *changed = 0;
    __syncthreads();
    for (int step = 0; step + 1 < n2; ++step) {
      for (int k = warp; k < n2 / 2; k += nw) {
        const int b = n2 - 1 - k;   // >= n2 / 2 >= 1
        const int p = k == 0 ? 0 : (k - 1 + step) % (n2 - 1) + 1;
        const int q = (b - 1 + step) % (n2 - 1) + 1;
        if (p >= n || q >= n) continue;
        float* xp = X + (size_t)p * n;
        float* xq = X + (size_t)q * n;
        float al = 0.f, be = 0.f, ga = 0.f;
        for (int i = lane; i < n; i += 32) {
          const float u = xp[i], v = xq[i];
          al = fmaf(u, u, al);
          be = fmaf(v, v, be);
          ga = fmaf(u, v, ga);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          al += __shfl_xor_sync(0xffffffffu, al, o);
          be += __shfl_xor_sync(0xffffffffu, be, o);
          ga += __shfl_xor_sync(0xffffffffu, ga, o);
        }
        if (ga != 0.f && fabsf(ga) > tol * sqrtf(al * be)) {   // warp-uniform
          const float zeta = (be - al) / (2.f * ga);
          const float t = copysignf(1.f, zeta) / (fabsf(zeta) + sqrtf(fmaf(zeta, zeta, 1.f)));
          const float c = 1.f / sqrtf(fmaf(t, t, 1.f)), s = c * t;
          float* vp = V + (size_t)p * n;
          float* vq = V + (size_t)q * n;
          for (int i = lane; i < n; i += 32) {
            const float u = xp[i], v = xq[i];
            xp[i] = c * u - s * v;
            xq[i] = s * u + c * v;
            const float g = vp[i], h = vq[i];
            vp[i] = c * g - s * h;
            vq[i] = s * g + c * h;
          }
          if (lane == 0) *changed = 1;
        }
      }
      __syncthreads();
    }
    const bool done = *changed == 0;   // every thread reads it after the barrier
    __syncthreads();
    if (done) break;
  }
}

// column norms of X (n x n, column-major) into out[0, n): one warp per column
__device__ void column_norms(const float* X, int n, float* out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  for (int k = warp; k < n; k += nw) {
    float ss = 0.f;
    for (int i = lane; i < n; i += 32) ss = fmaf(X[(size_t)k * n + i], X[(size_t)k * n + i], ss);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if (lane == 0) out[k] = sqrtf(ss);
  }
}

// T_A, T_B (r x r, row-major, columns in descending order of sigma) and sigma
// from G_A, G_B (rp-strided rows; only the r x r part is read).  scr holds
// six r x r matrices.
__global__ void __launch_bounds__(1024) embed_core_kernel(const float* __restrict__ GA,
                                                          const float* __restrict__ GB, int r, int rp,
                                                          float* __restrict__ scr, float* __restrict__ TA,
                                                          float* __restrict__ TB, float* __restrict__ sigma) {
  __shared__ int changed;
  __shared__ float la[kEmbedMaxRank], lb[kEmbedMaxRank], sg[kEmbedMaxRank];
  __shared__ int rank[kEmbedMaxRank];
  const size_t rr = (size_t)r * r;
  float* XA = scr;
  float* VA = XA + rr;
  float* XB = VA + rr;
  float* VB = XB + rr;
  float* C = VB + rr;
  float* VC = C + rr;
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) {   // symmetric: column-major = row-major
    XA[e] = GA[(size_t)(e / r) * rp + e % r];
    XB[e] = GB[(size_t)(e / r) * rp + e % r];
  }
  __syncthreads();
  // G = P Lambda P^T: for a positive semi-definite G, G V has columns lambda_k p_k with V = P
  jacobi(XA, VA, r, &changed);
  jacobi(XB, VB, r, &changed);
  column_norms(XA, r, la);
  column_norms(XB, r, lb);
  __syncthreads();
  // C = Lambda_A^{1/2} P_A^T P_B Lambda_B^{1/2}, column-major
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) {
    const int j = e / r, i = e % r;
    float acc = 0.f;
    for (int k = 0; k < r; ++k) acc = fmaf(VA[(size_t)i * r + k], VB[(size_t)j * r + k], acc);
    C[e] = sqrtf(la[i]) * acc * sqrtf(lb[j]);
  }
  __syncthreads();
  // C V' = U' Sigma
  jacobi(C, VC, r, &changed);
  column_norms(C, r, sg);
  __syncthreads();
  float smax = 0.f;
  for (int k = 0; k < r; ++k) smax = fmaxf(smax, sg[k]);
  // descending order of sigma (ties by index)
  for (int k = threadIdx.x; k < r; k += blockDim.x) {
    int rk = 0;
    for (int j = 0; j < r; ++j) rk += sg[j] > sg[k] || (sg[j] == sg[k] && j < k);
    rank[k] = rk;
  }
  __syncthreads();
  const float cut = smax * (float)r * FLT_EPSILON;   // singular values below this carry no direction
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) {
    const int i = e / r, k = e % r;
    float ta = 0.f, tb = 0.f;
    if (sg[k] > cut) {
      const float inv = 1.f / sqrtf(sg[k]);
      for (int j = 0; j < r; ++j) {
        ta = fmaf(VB[(size_t)j * r + i] * sqrtf(lb[j]), VC[(size_t)k * r + j], ta);
        tb = fmaf(VA[(size_t)j * r + i] * sqrtf(la[j]), C[(size_t)k * r + j] / sg[k], tb);
      }
      ta *= inv;
      tb *= inv;
    }
    TA[(size_t)i * r + rank[k]] = ta;
    TB[(size_t)i * r + rank[k]] = tb;
  }
  for (int k = threadIdx.x; k < r; k += blockDim.x) sigma[rank[k]] = sg[k];
}

// xi_i = [a_i T_A, b_i T_B] / norm, one warp per row; T_A and T_B in shared memory
__global__ void __launch_bounds__(256) embed_rows_kernel(const float* __restrict__ A, const float* __restrict__ B,
                                                         int64_t n, int r, int rp, const float* __restrict__ TA,
                                                         const float* __restrict__ TB, float* __restrict__ xi) {
  extern __shared__ __align__(16) float smt[];
  float* sa = smt;
  float* sb = smt + (size_t)r * r;
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) {
    sa[e] = TA[e];
    sb[e] = TB[e];
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int64_t i = (int64_t)blockIdx.x * 8 + warp; i < n; i += (int64_t)gridDim.x * 8) {
    float x[kEmbedMaxRank / 32], y[kEmbedMaxRank / 32];
#pragma unroll
    for (int j = 0; j < kEmbedMaxRank / 32; ++j) x[j] = y[j] = 0.f;
    for (int kb = 0; kb < r; kb += 32) {
      const float av = kb + lane < r ? A[i * rp + kb + lane] : 0.f;
      const float bv = kb + lane < r ? B[i * rp + kb + lane] : 0.f;
      const int kn = r - kb < 32 ? r - kb : 32;
      for (int kk = 0; kk < kn; ++kk) {
        const float ak = __shfl_sync(0xffffffffu, av, kk), bk = __shfl_sync(0xffffffffu, bv, kk);
        const float* ta = sa + (size_t)(kb + kk) * r;
        const float* tb = sb + (size_t)(kb + kk) * r;
#pragma unroll
        for (int j = 0; j < kEmbedMaxRank / 32; ++j) {
          const int c = lane + 32 * j;
          if (c < r) {
            x[j] = fmaf(ak, ta[c], x[j]);
            y[j] = fmaf(bk, tb[c], y[j]);
          }
        }
      }
    }
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < kEmbedMaxRank / 32; ++j) ss = fmaf(x[j], x[j], fmaf(y[j], y[j], ss));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
    float* out = xi + i * 2 * r;
#pragma unroll
    for (int j = 0; j < kEmbedMaxRank / 32; ++j) {
      const int c = lane + 32 * j;
      if (c < r) {
        out[c] = x[j] * inv;
        out[r + c] = y[j] * inv;
      }
    }
  }
}

// keys -> (nearest index, its inner product); label disagreements counted
__global__ void nn_decode_kernel(const unsigned long long* __restrict__ key, int64_t N, int32_t* __restrict__ nn,
                                 float* __restrict__ best, const int32_t* __restrict__ labels,
                                 unsigned long long* __restrict__ errors) {
  unsigned long long mine = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < N; i += (int64_t)gridDim.x * blockDim.x) {
    const unsigned long long k = key[i];
    int32_t j = -1;
    float v = -INFINITY;
    if (k != 0ull) {
      const uint32_t ord = (uint32_t)(k >> 32);
      const uint32_t bits = (ord & 0x80000000u) ? (ord & 0x7fffffffu) : ~ord;
      v = __uint_as_float(bits);
      j = (int32_t)(~(uint32_t)(k & 0xffffffffull));
    }
    nn[i] = j;
    if (best) best[i] = v;
    if (labels && j >= 0 && labels[j] != labels[i]) ++mine;
  }
  if (errors) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mine += __shfl_xor_sync(0xffffffffu, mine, o);
    if ((threadIdx.x & 31) == 0 && mine) atomicAdd(errors, mine);
  }
}

int pad_dim(int d) {
  return d <= 16 ? 16 : d <= 32 ? 32 : d <= 64 ? 64 : d <= 128 ? 128 : 256;
}

// workspace of nmd_nearest_neighbors: master, three pieces, keys, status, count
struct NnLayout {
  size_t master, hi, lo, lo2, keys, status, count, total;
};

NnLayout nn_layout(int64_t N, int dp) {
  NnLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    off = (off + 255) & ~size_t(255);
    const size_t at = off;
    off += bytes;
    return at;
  };
  L.master = take((size_t)N * dp * sizeof(float));
  L.hi = take((size_t)N * dp * sizeof(bf16));
  L.lo = take((size_t)N * dp * sizeof(bf16));
  L.lo2 = take((size_t)N * dp * sizeof(bf16));
  L.keys = take((size_t)N * sizeof(unsigned long long));
  L.status = take(kStatusWords * sizeof(int));
  L.count = take(sizeof(unsigned long long));
  L.total = (off + 255) & ~size_t(255);
  return L;
}

}  // namespace

int embed_max_rank() { return kEmbedMaxRank; }

nmd_status launch_embed(const Factor& W, const Factor& B, int64_t n, int r, int rp, float* gram_part, float* GA,
                        float* GB, float* scratch, float* TA, float* TB, float* sigma, float* xi, int num_sms,
                        cudaStream_t s, int64_t* launches) {
  const int64_t chunk = ((n + kGramParts - 1) / kGramParts + 31) / 32 * 32;
  launch_gram(&W, false, 0, n, r, rp, gram_part, kGramParts, chunk, 0.f, GA, s);
  launch_gram(&B, false, 0, n, r, rp, gram_part, kGramParts, chunk, 0.f, GB, s);
  embed_core_kernel<<<1, 1024, 0, s>>>(GA, GB, r, rp, scratch, TA, TB, sigma);
  static std::atomic<int> attr[kMaxDevices];
  if (!per_device(attr, [] {
        return cudaFuncSetAttribute(embed_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)(2 * kEmbedMaxRank * kEmbedMaxRank * sizeof(float))) == cudaSuccess ? 1 : 0;
      }))
    return NMD_ERR_CUDA;
  const size_t smem = (size_t)2 * r * r * sizeof(float);
  const unsigned grid = (unsigned)std::min<int64_t>((n + 7) / 8, (int64_t)num_sms * 4);
  embed_rows_kernel<<<grid, 256, smem, s>>>(W.master, B.master, n, r, rp, TA, TB, xi);
  *launches += 6;
  return NMD_OK;
}

}  // namespace nmd

using namespace nmd;

extern "C" {

nmd_status nmd_nn_workspace_bytes(int64_t N, int32_t d, size_t* bytes) {
  if (N < 2 || d < 1 || d > 256 || !bytes) return NMD_ERR_INVALID;
  *bytes = nn_layout(N, pad_dim(d)).total;
  return NMD_OK;
}

nmd_status nmd_nearest_neighbors(const float* d_x, int64_t N, int32_t d, const int32_t* d_labels, int32_t* d_nn,
                                 float* d_best, int64_t* errors, void* d_workspace, size_t ws_bytes, void* stream) {
  if (!d_x || !d_nn || !d_workspace || N < 2 || N >= (int64_t(1) << 31) || d < 1 || d > 256)
    return NMD_ERR_INVALID;
  const int dp = pad_dim(d);
  const NnLayout L = nn_layout(N, dp);
  if (ws_bytes < L.total || ((uintptr_t)d_workspace & 255u)) return NMD_ERR_WORKSPACE;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return NMD_ERR_CUDA;
  cudaStream_t s = (cudaStream_t)stream;
  char* w = (char*)d_workspace;
  Factor f;
  f.rows = N;
  f.master = (float*)(w + L.master);
  f.hi = (bf16*)(w + L.hi);
  f.lo = (bf16*)(w + L.lo);
  f.lo2 = (bf16*)(w + L.lo2);
  unsigned long long* keys = (unsigned long long*)(w + L.keys);
  int* status = (int*)(w + L.status);
  unsigned long long* count = (unsigned long long*)(w + L.count);
  if (cudaMemsetAsync(keys, 0, (size_t)N * sizeof(unsigned long long), s) != cudaSuccess ||
      cudaMemsetAsync(status, 0, kStatusWords * sizeof(int), s) != cudaSuccess ||
      cudaMemsetAsync(count, 0, sizeof(unsigned long long), s) != cudaSuccess)
    return NMD_ERR_CUDA;
  launch_pack(d_x, false, N, d, dp, f, s);
  nmd_status st = launch_nearest_tc(f, N, dp, keys, status, sms, s);
  if (st != NMD_OK) return st;
  const unsigned grid = (unsigned)std::min<int64_t>((N + 255) / 256, (int64_t)sms * 8);
  nn_decode_kernel<<<grid, 256, 0, s>>>(keys, N, d_nn, d_best, d_labels, count);
  if (cudaGetLastError() != cudaSuccess) return NMD_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return NMD_ERR_CUDA;
  int hs[2] = {0, 0};
  if (cudaMemcpy(hs, status, sizeof hs, cudaMemcpyDeviceToHost) != cudaSuccess) return NMD_ERR_CUDA;
  if (hs[0] != 0) {
    fprintf(stderr, "nmd_nearest_neighbors: device status %d (detail %d)\n", hs[0], hs[1]);
    return (nmd_status)hs[0];
  }
  if (errors) {
    unsigned long long c = 0;
    if (cudaMemcpy(&c, count, sizeof c, cudaMemcpyDeviceToHost) != cudaSuccess) return NMD_ERR_CUDA;
    *errors = (int64_t)c;
  }
  return NMD_OK;
}

}  // extern "C"
