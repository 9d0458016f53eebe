// Device-side definitions shared by the kernels of the SubZero+ weight path.
//
// The random-number contract (Philox4x32-10 + uniform + Box-Muller) is written
// here from its published definitions (Salmon et al., SC'11; Box & Muller 1958)
// and is the only source of Z_i^(k) (Sec. 4.1, Eq. (4); App. A.1 seed trick) and
// of Omega_U / Omega_V (Alg. 1) on the GPU.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

namespace zo {

// ---------------------------------------------------------------------------
// Status words written by kernels (read back by zo_sync_status).
// ---------------------------------------------------------------------------
enum DeviceStatus : uint32_t {
  kDevOk = 0,
  kDevTimeout = 1,   // a bounded mbarrier / flag wait gave up
  kDevBounds = 2,    // an internal bound check failed; the access was skipped
  kDevNotPosDef = 4, // refresh: a Gram matrix had a non-positive Cholesky pivot
};

// ---------------------------------------------------------------------------
// Counter contract
// ---------------------------------------------------------------------------
constexpr uint32_t kTagZ = 1;
constexpr uint32_t kTagOmegaU = 2;
constexpr uint32_t kTagOmegaV = 3;

__host__ __device__ constexpr uint32_t query_word(uint32_t tag, uint32_t k) {
  return (tag << 24) | (k & 0xFFFFFFu);
}

// Philox4x32 with ten rounds.  Round: (x0,x1,x2,x3) -> (hi(B*x2)^x1^k0, lo(B*x2),
// hi(A*x0)^x3^k1, lo(A*x0)) with A = 0xD2511F53, B = 0xCD9E8D57; the key is
// advanced by the Weyl constants (0x9E3779B9, 0xBB67AE85) between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int rnd = 0; rnd < 10; ++rnd) {
    if (rnd > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t hi_a = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo_a = 0xD2511F53u * c.x;
    const uint32_t hi_b = __umulhi(0xCD9E8D57u, c.z);
    const uint32_t lo_b = 0xCD9E8D57u * c.z;
    c = make_uint4(hi_b ^ c.y ^ k0, lo_b, hi_a ^ c.w ^ k1, lo_a);
  }
  return c;
}

// u = ((x >> 8) + 1) * 2^-24 in (0, 1]; the integer fits 24 bits, so exact in fp32.
__device__ __forceinline__ float u01(uint32_t x) {
  return __uint2float_rn((x >> 8) + 1u) * 5.9604644775390625e-08f;
}

// Box-Muller on one pair of uniforms: (rad cos(2 pi ub), rad sin(2 pi ub)).
__device__ __forceinline__ float2 box_muller(uint32_t xa, uint32_t xb) {
  const float ua = u01(xa);
  const float ub = u01(xb);
  const float rad = sqrtf(-2.0f * logf(ua));
  float s, c;
  sincospif(2.0f * ub, &s, &c);
  return make_float2(rad * c, rad * s);
}

// Four normals of counter word `c4` of the stream (seed, x1, x2, x3).
__device__ __forceinline__ float4 normal4(uint64_t seed, uint32_t c4, uint32_t x1, uint32_t x2,
                                          uint32_t x3) {
  const uint4 w = philox4x32_10(make_uint4(c4, x1, x2, x3), static_cast<uint32_t>(seed),
                                static_cast<uint32_t>(seed >> 32));
  const float2 a = box_muller(w.x, w.y);
  const float2 b = box_muller(w.z, w.w);
  return make_float4(a.x, a.y, b.x, b.y);
}

// ---------------------------------------------------------------------------
// Matrix descriptor as seen by the kernels (built by the host runtime).
// ---------------------------------------------------------------------------
struct MatDesc {
  void* W;          // m x n, leading dimension ldw (elements)
  int64_t m, n, ldw;
  int32_t dtype;    // 0 = fp32, 1 = bf16
  uint32_t gidx;    // global Philox matrix index
  float* U;         // m x r
  float* V;         // n x r
  float* M;         // r x r first moment
  float* Vm;        // r x r second moment
  float* C;         // r x r coefficient of the current pass (workspace)
  float* P;         // FMA path: r x n, P = C V^T (workspace)
  int64_t tile0;    // first weight-pass tile of this matrix (FMA path)
};

// Per-matrix record of the tensor-core weight pass (128 x 128 tiles).
struct TcMat {
  int64_t m, n;
  int64_t tile0;     // first tile of this matrix
  int32_t tiles_n;   // column tiles
  int32_t u_row0;    // first row of this matrix in the stacked hi/lo U operand
  int32_t p_row0;    // first row of this matrix in the stacked hi/lo P^T operand
  int32_t pad;
};

// One block of the batched TSQR used by the refresh (see zo_qr.cu).
struct QrBlock {
  float* rows;         // storage of this block's rows (R floats per row)
  const float* s_in;   // down pass: the R x R block of the parent's Q for this block
  float* r_out;        // up pass: where this block's R x R triangular factor goes
  float* tau;          // R Householder scalars of this block
  int64_t row0;        // level 0: first panel row of the block (element addressing of Omega)
  int32_t n_real;      // rows of real data in the block (the rest is zero padding)
  int32_t flags;       // kQrTop | kQrLevel0
  uint32_t gidx;       // matrix index for Omega
  uint32_t tag;        // kTagOmegaU or kTagOmegaV
};
constexpr int32_t kQrTop = 1;
constexpr int32_t kQrLevel0 = 2;

}  // namespace zo
