// The U operand of the r <= 32 tensor-core weight pass (zo_wpass_tc.cu): rows
// [hi(U s) | lo(U s) | 0 ...] in fp16 with s = 2^kUVScaleExp (zo_tc_common.cuh), formed once
// per refresh, stacked per matrix in 128-row blocks and read by TMA.  The perturbed-linear
// route (zo_linear.cu, zo_linear_pair.cu; every r) reads rows of the same layout as a bf16
// pair, hi = bf16(x), lo = bf16(x - hi), unscaled, from a buffer of its own: there U meets
// the bf16 X and W in one accumulator.
// Also the dispatch of the split by rank (r >= 64: the chunk-major U of zo_wpass_tmem.cu).
// P^T = V C^T, the other operand, comes from the tensor-core projection (zo_project_tc.cu).
#include "zo_kernels.h"
#include "zo_tc_common.cuh"

namespace zo {
namespace {

using namespace tc;

// The split kernel below (U rows; r <= 32 for the weight pass, every r for the
// perturbed-linear route) handles 128 consecutive rows of one matrix
// per CTA: each thread splits one row into 16-byte chunks of hi and lo, staged
// in shared memory with the chunk index XOR (row & 7) so a quarter-warp's stores hit
// distinct banks; the CTA then writes its rows, which are contiguous in the stacked
// operand, with coalesced 16-byte stores.  Padding columns of a row stay at the zero they
// were set to.
template <int R>
__device__ __forceinline__ void write_rows(const uint4* Os, uint16_t* dst_rows, int rows) {
  constexpr int kVecPerRow = hl_width(R) * 2 / 16;   // 8 or 16 chunks per row
  uint4* dst = reinterpret_cast<uint4*>(dst_rows);
  for (int e = threadIdx.x; e < rows * kVecPerRow; e += blockDim.x) {
    const int row = e / kVecPerRow, c = e % kVecPerRow;
    if (c * 8 < 2 * R) dst[e] = Os[row * kVecPerRow + (c ^ (row & 7))];
  }
}

// dst[u_row0 + i] = [hi | lo | 0 ...] of row i of U (row width hl_width(R)): the fp16 pair
// of U 2^kUVScaleExp (kF16) or the bf16 pair of U.
template <int R, bool kF16>
__global__ void __launch_bounds__(128)
split_u_kernel(const MatDesc* __restrict__ mats, const TcMat* __restrict__ tcm,
               const int2* __restrict__ units, uint16_t* __restrict__ dst) {
  constexpr int kVecPerRow = hl_width(R) * 2 / 16;
  extern __shared__ uint4 su_smem[];
  uint4* Os = su_smem;                                     // 128 x kVecPerRow
  const int2 u = units[blockIdx.x];
  const MatDesc md = mats[u.x];
  const int tid = threadIdx.x;
  const int64_t i0 = u.y;
  const int rows = (int)(md.m - i0 < 128 ? md.m - i0 : 128);
  if (tid < rows) {
    const float4* src = reinterpret_cast<const float4*>(md.U + (i0 + tid) * R);
    uint4* orow = Os + tid * kVecPerRow;
#pragma unroll
    for (int g = 0; g < R / 8; ++g) {
      const float4 a = src[2 * g], b = src[2 * g + 1];
      const float x[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
      uint4 hi, lo;
      if constexpr (kF16) split8_f16(x, exp2i(kUVScaleExp), hi, lo);
      else split8(x, hi, lo);
      orow[g ^ (tid & 7)] = hi;
      orow[(R / 8 + g) ^ (tid & 7)] = lo;
    }
  }
  __syncthreads();
  write_rows<R>(Os, dst + ((int64_t)tcm[u.x].u_row0 + i0) * hl_width(R), rows);
}

template <int R, bool kF16>
cudaError_t launch_split_u_r(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                             int32_t n_units, uint16_t* dst, cudaStream_t s) {
  const size_t smem = 128 * (size_t)hl_width(R) * 2;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(split_u_kernel<R, kF16>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  split_u_kernel<R, kF16><<<n_units, 128, smem, s>>>(d_mats, d_tc, d_units, dst);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_split_u(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                           int32_t n_units, int32_t r, void* u_op, cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 16: return launch_split_u_r<16, true>(d_mats, d_tc, d_units, n_units, static_cast<uint16_t*>(u_op), s);
    case 32: return launch_split_u_r<32, true>(d_mats, d_tc, d_units, n_units, static_cast<uint16_t*>(u_op), s);
    case 64:
    case 128: return launch_split_u_chunks(d_mats, d_tc, d_units, n_units, r, static_cast<uint4*>(u_op), s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_split_u_bf16(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                                int32_t n_units, int32_t r, __nv_bfloat16* u_lin, cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 16: return launch_split_u_r<16, false>(d_mats, d_tc, d_units, n_units, reinterpret_cast<uint16_t*>(u_lin), s);
    case 32: return launch_split_u_r<32, false>(d_mats, d_tc, d_units, n_units, reinterpret_cast<uint16_t*>(u_lin), s);
    case 64: return launch_split_u_r<64, false>(d_mats, d_tc, d_units, n_units, reinterpret_cast<uint16_t*>(u_lin), s);
    case 128: return launch_split_u_r<128, false>(d_mats, d_tc, d_units, n_units, reinterpret_cast<uint16_t*>(u_lin), s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
