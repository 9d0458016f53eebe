// Pieces shared by the two perturbed-linear GEMM files (zo_linear.cu: single-CTA tiles and
// the S = X P^T kernel; zo_linear_pair.cu: SM-pair tiles with S computed in-kernel).
#pragma once

#include <cuda_bf16.h>
#include <cstdint>

#include "zo_tc_common.cuh"

namespace zo {
namespace lin {

// S_HL row: [hi | lo] of the R sums in chunks of 8, then zero chunks up to 64 elements.
template <int R>
__device__ __forceinline__ void write_s_row(__nv_bfloat16* s_hl, int row, const float (&x)[R]) {
  constexpr int kGroups = R / 8;
  uint4* out = reinterpret_cast<uint4*>(s_hl + (int64_t)row * 64);
#pragma unroll
  for (int g = 0; g < kGroups; ++g) {
    float c[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) c[e] = x[8 * g + e];
    uint4 hi, lo;
    tc::split8(c, hi, lo);
    out[g] = hi;
    out[kGroups + g] = lo;
  }
#pragma unroll
  for (int z = 2 * kGroups; z < 8; ++z) out[z] = make_uint4(0u, 0u, 0u, 0u);
}

}  // namespace lin
}  // namespace zo
