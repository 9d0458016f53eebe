// Pieces shared by the two perturbed-linear GEMM files (zo_linear.cu: single-CTA tiles and
// the S = X P^T kernel; zo_linear_pair.cu: SM-pair tiles with S computed in-kernel).
#pragma once

#include <cuda_bf16.h>
#include <cstdint>

#include "zo_tc_common.cuh"

namespace zo {
namespace lin {

// An S_HL row holds hl_width(R) bf16: [hi | lo] of the R sums in groups of 8, then zeros
// (R = 16).  write_s_chunk: the hi and lo groups of sums kC j .. kC j + kC - 1, kC =
// min(R, 32).
template <int R>
__device__ __forceinline__ void write_s_chunk(__nv_bfloat16* s_hl, int row, int j,
                                              const float (&x)[R < 32 ? R : 32]) {
  constexpr int kC = R < 32 ? R : 32;
  uint4* out = reinterpret_cast<uint4*>(s_hl + (int64_t)row * tc::hl_width(R));
#pragma unroll
  for (int g = 0; g < kC / 8; ++g) {
    float c[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) c[e] = x[8 * g + e];
    uint4 hi, lo;
    tc::split8(c, hi, lo);
    out[kC / 8 * j + g] = hi;
    out[R / 8 + kC / 8 * j + g] = lo;
  }
}

// the zero groups of an S_HL row past 2R
template <int R>
__device__ __forceinline__ void zero_s_pad(__nv_bfloat16* s_hl, int row) {
  uint4* out = reinterpret_cast<uint4*>(s_hl + (int64_t)row * tc::hl_width(R));
#pragma unroll
  for (int z = R / 4; z < tc::hl_width(R) / 8; ++z) out[z] = make_uint4(0u, 0u, 0u, 0u);
}

// a whole S_HL row, R <= 32
template <int R>
__device__ __forceinline__ void write_s_row(__nv_bfloat16* s_hl, int row, const float (&x)[R]) {
  static_assert(R <= 32, "one chunk per row");
  write_s_chunk<R>(s_hl, row, 0, x);
  zero_s_pad<R>(s_hl, row);
}

}  // namespace lin
}  // namespace zo
