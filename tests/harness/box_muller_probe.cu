// Exhaustive check of the GPU's Box-Muller transform (zo_device.cuh: box_muller) over
// every uniform the counter contract can produce, u = j 2^-24 for j = 1 .. 2^24, against
// the host's double precision:
//   radius: box_muller(x_j, x_1) with ub = 1 (cos 2 pi = 1, sin 2 pi = 0 exactly) is
//           (rad(u_j), 0), rad(u) = sqrt(-2 ln u);
//   angle:  box_muller(x_0, x_j) with ua = 2^-24 (the largest radius, 5.77) is
//           rad(2^-24) (cos 2 pi u_j, sin 2 pi u_j), each product rounded once.
// Prints the largest absolute errors of both sweeps; run by tests/test_gpu_box_muller.py.
#include <cmath>
#include <cstdio>
#include <vector>

#include "zo_device.cuh"

__global__ void probe(float* rad, float* zc, float* zs, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint32_t xj = (uint32_t)i << 8;                   // u01(xj) = (i + 1) 2^-24
  const uint32_t x_one = 0xFFFFFF00u;                     // u01 = 1
  const uint32_t x_min = 0u;                              // u01 = 2^-24
  rad[i] = zo::box_muller(xj, x_one).x;
  const float2 z = zo::box_muller(x_min, xj);
  zc[i] = z.x;
  zs[i] = z.y;
}

int main() {
  const int n = 1 << 24;
  float *d_rad, *d_c, *d_s;
  if (cudaMalloc(&d_rad, n * 4) != cudaSuccess || cudaMalloc(&d_c, n * 4) != cudaSuccess ||
      cudaMalloc(&d_s, n * 4) != cudaSuccess) {
    std::printf("ERROR cudaMalloc\n");
    return 1;
  }
  probe<<<(n + 255) / 256, 256>>>(d_rad, d_c, d_s, n);
  if (cudaDeviceSynchronize() != cudaSuccess) {
    std::printf("ERROR kernel\n");
    return 1;
  }
  std::vector<float> rad(n), c(n), s(n);
  cudaMemcpy(rad.data(), d_rad, n * 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(c.data(), d_c, n * 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(s.data(), d_s, n * 4, cudaMemcpyDeviceToHost);
  const double two_pi = 6.283185307179586476925286766559;
  const double r_max = std::sqrt(-2.0 * std::log(5.9604644775390625e-08));
  double e_rad = 0, e_c = 0, e_s = 0, u_rad = 0, u_c = 0, u_s = 0;
  for (int i = 0; i < n; ++i) {
    const double u = (double)(i + 1) * 5.9604644775390625e-08;
    const double dr = std::fabs((double)rad[i] - std::sqrt(-2.0 * std::log(u)));
    if (dr > e_rad) { e_rad = dr; u_rad = u; }
    const double dc = std::fabs((double)c[i] - r_max * std::cos(two_pi * u));
    if (dc > e_c) { e_c = dc; u_c = u; }
    const double ds = std::fabs((double)s[i] - r_max * std::sin(two_pi * u));
    if (ds > e_s) { e_s = ds; u_s = u; }
  }
  std::printf("radius %.6e at %.9g\nzcos %.6e at %.9g\nzsin %.6e at %.9g\n", e_rad, u_rad, e_c,
              u_c, e_s, u_s);
  return 0;
}
