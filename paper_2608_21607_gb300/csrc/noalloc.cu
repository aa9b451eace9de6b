// Gram matrix of a caller's device matrix with no device allocation: the
// partial sums live in a file-scope device array instead of a workspace.
#include <stdio.h>

#include <mutex>

#include "nmd_internal.cuh"

namespace nmd {
namespace {

// Scratch for the partial Gram matrices: nparts x r x r floats, at most
// kNoAllocScratchFloats (2 MiB).  Every GPU that loads the library holds one
// copy of this array until the process exits.
constexpr int64_t kNoAllocScratchFloats = 512 * 1024;
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

constexpr int kNoAllocMaxDevices = 64;
constexpr int kNoAllocMaxRank = 128;

// Device address of the array, looked up once per device with that device
// current (a host-side reference to the symbol is not a device address).
nmd_status scratch_address(float** out, std::string* why) {
  static std::mutex mu;
  static float* addr[kNoAllocMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    *why = std::string("cudaGetDevice: ") + cudaGetErrorString(e);
    return NMD_ERR_CUDA;
  }
  if (dev < 0 || dev >= kNoAllocMaxDevices) {
    *why = "device ordinal out of range";
    return NMD_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> g(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p) {
      *why = std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e);
      return NMD_ERR_CUDA;
    }
    addr[dev] = (float*)p;
  }
  *out = addr[dev];
  return NMD_OK;
}

// Part p sums rows [p chunk, (p+1) chunk) of Q (row stride ld, r <= 128
// columns) into the r x r partial p; 16 x 16 threads, each owning the entries
// (ty + 16 a, tx + 16 b).
__global__ void __launch_bounds__(256) gram_noalloc_kernel(const float* __restrict__ Q, int64_t ld, int64_t K,
                                                           int r, int64_t chunk, float* __restrict__ parts) {
  __shared__ float tile[32][129];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int64_t k0 = (int64_t)blockIdx.x * chunk, k1 = min(K, k0 + chunk);
  float acc[8][8];
  const int na = (r + 15) / 16;
#pragma unroll
  for (int a = 0; a < 8; ++a)
#pragma unroll
    for (int b = 0; b < 8; ++b) acc[a][b] = 0.f;
  for (int64_t kb = k0; kb < k1; kb += 32) {
    __syncthreads();
    for (int e = threadIdx.x; e < 32 * r; e += 256) {
      const int rr = e / r, c = e % r;
      tile[rr][c] = kb + rr < k1 ? Q[(kb + rr) * ld + c] : 0.f;
    }
    __syncthreads();
    for (int rr = 0; rr < 32; ++rr) {
#pragma unroll
      for (int a = 0; a < 8; ++a) {
        if (a >= na) break;
        const float qa = ty + 16 * a < r ? tile[rr][ty + 16 * a] : 0.f;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
          if (b >= na) break;
          const float qb = tx + 16 * b < r ? tile[rr][tx + 16 * b] : 0.f;
          acc[a][b] = fmaf(qa, qb, acc[a][b]);
        }
      }
    }
  }
  float* out = parts + (int64_t)blockIdx.x * r * r;
#pragma unroll
  for (int a = 0; a < 8; ++a)
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const int i = ty + 16 * a, j = tx + 16 * b;
      if (a < na && b < na && i < r && j < r) out[i * r + j] = acc[a][b];
    }
}

// G = sum of the partials in part order.
__global__ void gram_noalloc_reduce(const float* __restrict__ parts, int nparts, int r, float* __restrict__ G) {
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < r * r; e += gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int p = 0; p < nparts; ++p) s += parts[(int64_t)p * r * r + e];
    G[e] = s;
  }
}

}  // namespace
}  // namespace nmd

extern "C" nmd_status nmd_gram_noalloc(const float* d_Q, int64_t K, int32_t r, int64_t ld, float* d_G,
                                       void* stream) {
  using namespace nmd;
  if (!d_Q || !d_G || K < 1 || r < 1 || ld < r) return NMD_ERR_INVALID;
  if (r > kNoAllocMaxRank) {
    fprintf(stderr, "nmd_gram_noalloc: r = %d exceeds the maximum rank %d of the static scratch\n", r,
            kNoAllocMaxRank);
    return NMD_ERR_WORKSPACE;
  }
  // the largest part count whose partials fit the static array
  const int64_t max_parts = kNoAllocScratchFloats / ((int64_t)r * r);
  const int64_t want_parts = (K + 255) / 256;
  const int nparts = (int)(want_parts < max_parts ? want_parts : max_parts);
  const int64_t chunk = (K + nparts - 1) / nparts;
  float* scratch = nullptr;
  std::string why;
  nmd_status st = scratch_address(&scratch, &why);
  if (st != NMD_OK) {
    fprintf(stderr, "nmd_gram_noalloc: %s\n", why.c_str());
    return st;
  }
  cudaStream_t s = (cudaStream_t)stream;
  gram_noalloc_kernel<<<nparts, 256, 0, s>>>(d_Q, ld, K, r, chunk, scratch);
  gram_noalloc_reduce<<<(r * r + 255) / 256, 256, 0, s>>>(scratch, nparts, r, d_G);
  return cudaGetLastError() == cudaSuccess ? NMD_OK : NMD_ERR_CUDA;
}
