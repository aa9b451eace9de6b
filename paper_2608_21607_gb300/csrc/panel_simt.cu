// Dense Z-panel contraction and dense loss pass on the CUDA cores (fp32 FMA).
// This is the NMD_SIMT path: exact fp32 arithmetic, no tensor cores.  It
// computes the same quantities as the tcgen05 kernels of panel_tc.cu:
//   R_i = sum_k P(L_ik) q_k,  L_ik = m_i . q_k,
//   P = min(0, .)  (Z form, eq. updateZ)  or  -max(0, .)  (Delta form, eq. updateD);
// and for the loss, sum max(0, L)^2 and sum max(0, L) over all of L = W H.
#include <algorithm>

#include "nmd_internal.cuh"

namespace nmd {
namespace {

constexpr int TM = 32;   // M-side rows per thread block
constexpr int TK = 32;   // Q-side rows per chunk

template <int RP>
__device__ __forceinline__ void load_rows(float* dst, const float* __restrict__ src, int64_t r0, int64_t nrows,
                                          int64_t limit) {
  for (int e = threadIdx.x; e < nrows * RP; e += blockDim.x) {
    int rr = e / RP, c = e % RP;
    int64_t g = r0 + rr;
    dst[rr * (RP + 1) + c] = g < limit ? src[g * RP + c] : 0.f;
  }
}

template <int RP, int EPI>
__global__ void __launch_bounds__(256) panel_simt_kernel(const float* __restrict__ M, int64_t m0, int64_t Mrows,
                                                         const float* __restrict__ Q, int64_t q0, int64_t K,
                                                         float* __restrict__ R) {
  extern __shared__ float sm[];
  float* Ms = sm;                          // TM x (RP+1)
  float* Qs = Ms + TM * (RP + 1);          // TK x (RP+1)
  float* Ps = Qs + TK * (RP + 1);          // TM x (TK+1)
  constexpr int NACC = TM * RP / 256;
  constexpr int RSTEP = 256 / RP > 0 ? 256 / RP : 1;
  const int64_t i0 = (int64_t)blockIdx.x * TM;
  load_rows<RP>(Ms, M + m0 * RP, i0, TM, Mrows);
  const int lk = threadIdx.x % TK, li = threadIdx.x / TK;   // L entries (li + 8j, lk)
  const int c = threadIdx.x % RP, rr0 = threadIdx.x / RP;   // R entries (rr0 + RSTEP j, c)
  float acc[NACC];
#pragma unroll
  for (int j = 0; j < NACC; ++j) acc[j] = 0.f;
  for (int64_t k0 = 0; k0 < K; k0 += TK) {
    __syncthreads();
    load_rows<RP>(Qs, Q + q0 * RP, k0, TK, K);
    __syncthreads();
#pragma unroll
    for (int j = 0; j < TM / 8; ++j) {
      int i = li + 8 * j;
      float l = 0.f;
#pragma unroll 8
      for (int cc = 0; cc < RP; ++cc) l = fmaf(Ms[i * (RP + 1) + cc], Qs[lk * (RP + 1) + cc], l);
      float p = EPI == 0 ? fminf(0.f, l) : -fmaxf(0.f, l);
      Ps[i * (TK + 1) + lk] = (k0 + lk < K) ? p : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < NACC; ++j) {
      int i = rr0 + RSTEP * j;
      float a = acc[j];
#pragma unroll 8
      for (int k = 0; k < TK; ++k) a = fmaf(Ps[i * (TK + 1) + k], Qs[k * (RP + 1) + c], a);
      acc[j] = a;
    }
  }
#pragma unroll
  for (int j = 0; j < NACC; ++j) {
    int64_t i = i0 + rr0 + RSTEP * j;
    if (i < Mrows) R[i * RP + c] = acc[j];
  }
}

// Dense loss: thread block b sums tiles b, b + grid, ... of TM rows of W
// against all of B; per-thread chunk sums in fp32 are accumulated in fp64.
template <int RP>
__global__ void __launch_bounds__(256) loss_dense_simt_kernel(const float* __restrict__ W, int64_t m,
                                                              const float* __restrict__ B, int64_t n,
                                                              double* __restrict__ parts) {
  extern __shared__ float sm[];
  float* Ms = sm;
  float* Qs = Ms + TM * (RP + 1);
  __shared__ double red[2][256];
  const int lk = threadIdx.x % TK, li = threadIdx.x / TK;
  double s2 = 0.0, s1 = 0.0;
  for (int64_t t = blockIdx.x; t * TM < m; t += gridDim.x) {
    __syncthreads();
    load_rows<RP>(Ms, W, t * TM, TM, m);
    for (int64_t k0 = 0; k0 < n; k0 += TK) {
      __syncthreads();
      load_rows<RP>(Qs, B, k0, TK, n);
      __syncthreads();
      float c2 = 0.f, c1 = 0.f;
#pragma unroll
      for (int j = 0; j < TM / 8; ++j) {
        int i = li + 8 * j;
        float l = 0.f;
#pragma unroll 8
        for (int cc = 0; cc < RP; ++cc) l = fmaf(Ms[i * (RP + 1) + cc], Qs[lk * (RP + 1) + cc], l);
        float p = fmaxf(0.f, l);
        c2 = fmaf(p, p, c2);
        c1 += p;
      }
      s2 += c2;
      s1 += c1;
    }
  }
  red[0][threadIdx.x] = s2;
  red[1][threadIdx.x] = s1;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      red[0][threadIdx.x] += red[0][threadIdx.x + w];
      red[1][threadIdx.x] += red[1][threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    parts[(size_t)blockIdx.x * 8 + 0] = red[0][0];
    parts[(size_t)blockIdx.x * 8 + 1] = red[1][0];
  }
}

template <int RP>
void panel_simt_rp(const StepArgs& a, float* R, cudaStream_t s) {
  size_t smem = ((size_t)(TM + TK) * (RP + 1) + TM * (TK + 1)) * sizeof(float);
  int grid = (int)((a.M + TM - 1) / TM);
  if (a.epilogue == NMD_EPI_DELTA) {
    cudaFuncSetAttribute(panel_simt_kernel<RP, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    panel_simt_kernel<RP, 1><<<grid, 256, smem, s>>>(a.fm->master, a.m0, a.M, a.fq->master, a.q0, a.K, R);
  } else {
    cudaFuncSetAttribute(panel_simt_kernel<RP, 0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    panel_simt_kernel<RP, 0><<<grid, 256, smem, s>>>(a.fm->master, a.m0, a.M, a.fq->master, a.q0, a.K, R);
  }
}

template <int RP>
int loss_simt_rp(const nmd_handle* h, double* parts, int maxparts, cudaStream_t s) {
  size_t smem = (size_t)(TM + TK) * (RP + 1) * sizeof(float);
  int grid = (int)std::min<int64_t>((h->m + TM - 1) / TM, maxparts);
  cudaFuncSetAttribute(loss_dense_simt_kernel<RP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  loss_dense_simt_kernel<RP><<<grid, 256, smem, s>>>(h->W.master, h->m, h->B.master, h->n, parts);
  return grid;
}

}  // namespace

void launch_panel_simt(const StepArgs& a, float* R, cudaStream_t s) {
  switch (a.rp) {
    case 16: panel_simt_rp<16>(a, R, s); break;
    case 32: panel_simt_rp<32>(a, R, s); break;
    case 64: panel_simt_rp<64>(a, R, s); break;
    case 128: panel_simt_rp<128>(a, R, s); break;
    default: panel_simt_rp<256>(a, R, s); break;
  }
}

int launch_loss_dense_simt(const nmd_handle* h, double* parts, int maxparts, cudaStream_t s) {
  switch (h->rp) {
    case 16: return loss_simt_rp<16>(h, parts, maxparts, s);
    case 32: return loss_simt_rp<32>(h, parts, maxparts, s);
    case 64: return loss_simt_rp<64>(h, parts, maxparts, s);
    case 128: return loss_simt_rp<128>(h, parts, maxparts, s);
    default: return loss_simt_rp<256>(h, parts, maxparts, s);
  }
}

}  // namespace nmd
