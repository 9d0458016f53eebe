// Bulk fills of the counter-based random contract (the integer Philox stream
// and its Gaussian transform).  The other kernels draw Z_i^(k) and Omega inline
// with the same device functions; these fills expose the stream itself.
#include "zo_kernels.h"

namespace zo {
namespace {

__global__ void philox_fill_kernel(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3,
                                   uint32_t* __restrict__ out, int64_t n_words) {
  const int64_t n_ctr = (n_words + 3) / 4;
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < n_ctr;
       c += (int64_t)gridDim.x * blockDim.x) {
    const uint4 w = philox4x32_10(make_uint4((uint32_t)c, x1, x2, x3), (uint32_t)seed,
                                  (uint32_t)(seed >> 32));
    const int64_t e = 4 * c;
    if (e + 3 < n_words) {
      out[e] = w.x; out[e + 1] = w.y; out[e + 2] = w.z; out[e + 3] = w.w;
    } else {
      const uint32_t v[4] = {w.x, w.y, w.z, w.w};
      for (int l = 0; l < 4 && e + l < n_words; ++l) out[e + l] = v[l];
    }
  }
}

__global__ void normal_fill_kernel(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3,
                                   float* __restrict__ out, int64_t n) {
  const int64_t n_ctr = (n + 3) / 4;
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < n_ctr;
       c += (int64_t)gridDim.x * blockDim.x) {
    const float4 z = normal4(seed, (uint32_t)c, x1, x2, x3);
    const int64_t e = 4 * c;
    if (e + 3 < n) {
      out[e] = z.x; out[e + 1] = z.y; out[e + 2] = z.z; out[e + 3] = z.w;
    } else {
      const float v[4] = {z.x, z.y, z.z, z.w};
      for (int l = 0; l < 4 && e + l < n; ++l) out[e + l] = v[l];
    }
  }
}

int grid_for(int64_t n_ctr) {
  const int64_t blocks = (n_ctr + 255) / 256;
  return (int)(blocks < 152 * 16 ? (blocks > 0 ? blocks : 1) : 152 * 16);
}

}  // namespace

cudaError_t launch_philox_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, uint32_t* out,
                               int64_t n_words, cudaStream_t s) {
  if (n_words <= 0) return cudaSuccess;
  // the counter word c is 32 bits: at most 2^32 counters (2^34 words)
  philox_fill_kernel<<<grid_for((n_words + 3) / 4), 256, 0, s>>>(seed, x1, x2, x3, out, n_words);
  return cudaGetLastError();
}

cudaError_t launch_normal_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, float* out,
                               int64_t n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  normal_fill_kernel<<<grid_for((n + 3) / 4), 256, 0, s>>>(seed, x1, x2, x3, out, n);
  return cudaGetLastError();
}

}  // namespace zo
