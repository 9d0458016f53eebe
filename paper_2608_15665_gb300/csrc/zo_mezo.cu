// Full-space SPSA perturbation of MeZO, Eq. (1): W_i <- rnd(W_i + coef * Z_i) with
// Z_i[row, col] ~ N(0, 1) drawn per element from the counter contract:
//   counter = (row * ceil(n_i / 4) + col / 4, matrix index, t, 5 << 24), lane col % 4.
// coef = +eps / -2 eps / +eps gives the two evaluations of Eq. (1) and the restore;
// coef = eps - eta * rho fuses the restore with MeZO's SGD update.
//
// Unlike the subspace pass, every weight needs its own Gaussian: one Philox4x32-10
// call and two Box-Muller transforms per 4 weights, so the pass is bound by the ALU
// (integer multiplies, log / sqrt / sincos), not by HBM.  Tiles are the FMA pass's
// 32 rows x (32 lanes x 16 bytes): a warp reads and writes 512 contiguous bytes of
// a row, each thread draws the 2 (bf16) or 1 (fp32) counter words of its 16 bytes.
#include "zo_kernels.h"

namespace zo {
namespace {

constexpr uint32_t kTagMezo = 5;

// The Philox round keys of one seed: (k0, k1) = (seed_lo, seed_hi) advanced by the Weyl
// constants (0x9E3779B9, 0xBB67AE85) once per round -- the key schedule of zo_device.cuh's
// philox4x32_10, formed once on the host.  Passed as a kernel parameter, each key is read
// from the constant bank by the round's XOR: the eight Philox calls of a thread spend no
// instructions and no registers on it.
struct RoundKeys {
  uint32_t k0[10], k1[10];
};

RoundKeys round_keys(uint64_t seed) {
  RoundKeys k;
  k.k0[0] = (uint32_t)seed;
  k.k1[0] = (uint32_t)(seed >> 32);
  for (int r = 1; r < 10; ++r) {
    k.k0[r] = k.k0[r - 1] + 0x9E3779B9u;
    k.k1[r] = k.k1[r - 1] + 0xBB67AE85u;
  }
  return k;
}

// philox4x32_10 and normal4 of zo_device.cuh with the round keys given.
__device__ __forceinline__ float4 normal4_keyed(const RoundKeys& k, uint32_t c4, uint32_t x1,
                                                uint32_t x2, uint32_t x3) {
  uint4 c = make_uint4(c4, x1, x2, x3);
#pragma unroll
  for (int rnd = 0; rnd < 10; ++rnd) {
    const uint32_t hi_a = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo_a = 0xD2511F53u * c.x;
    const uint32_t hi_b = __umulhi(0xCD9E8D57u, c.z);
    const uint32_t lo_b = 0xCD9E8D57u * c.z;
    c = make_uint4(hi_b ^ c.y ^ k.k0[rnd], lo_b, hi_a ^ c.w ^ k.k1[rnd], lo_a);
  }
  const float2 a = box_muller(c.x, c.y);
  const float2 b = box_muller(c.z, c.w);
  return make_float4(a.x, a.y, b.x, b.y);
}

__device__ __forceinline__ int find_matrix_tile(const int64_t* __restrict__ prefix, int n_mats,
                                                int64_t tile) {
  int lo = 0, hi = n_mats - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(prefix + mid) <= tile) lo = mid; else hi = mid - 1;
  }
  return lo;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

__global__ void __launch_bounds__(256)
mezo_kernel(const MatDesc* __restrict__ mats, int n_mats, const int64_t* __restrict__ prefix,
            const __grid_constant__ RoundKeys keys, uint32_t t, float coef) {
  const int64_t tile = blockIdx.x;
  const MatDesc md = mats[find_matrix_tile(prefix, n_mats, tile)];
  const int bf16 = md.dtype == 1;
  const int vec = bf16 ? 8 : 4;                       // elements per 16 bytes
  const int64_t tn = 32 * vec;                        // tile columns
  const int64_t local = tile - md.tile0;
  const int64_t tiles_n = (md.n + tn - 1) / tn;
  const int64_t row0 = (local / tiles_n) * kFmaTileRows;
  const int64_t col = (local % tiles_n) * tn + (threadIdx.x & 31) * vec;
  const uint32_t n4 = (uint32_t)((md.n + 3) / 4);
  const uint32_t x3 = query_word(kTagMezo, 0);
  if (col >= md.n) return;
  const bool full = col + vec <= md.n;
  for (int rr = threadIdx.x >> 5; rr < kFmaTileRows; rr += 8) {
    const int64_t row = row0 + rr;
    if (row >= md.m) break;
    const uint32_t c0 = (uint32_t)(row * n4 + col / 4);
    float z[8];
    const float4 za = normal4_keyed(keys, c0, md.gidx, t, x3);
    z[0] = za.x; z[1] = za.y; z[2] = za.z; z[3] = za.w;
    if (bf16) {
      const float4 zb = normal4_keyed(keys, c0 + 1, md.gidx, t, x3);
      z[4] = zb.x; z[5] = zb.y; z[6] = zb.z; z[7] = zb.w;
    }
    if (bf16) {
      __nv_bfloat16* w = reinterpret_cast<__nv_bfloat16*>(md.W) + row * md.ldw + col;
      if (full) {
        const uint4 raw = *reinterpret_cast<const uint4*>(w);
        const uint32_t v[4] = {raw.x, raw.y, raw.z, raw.w};
        uint32_t o[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float lo = fmaf(coef, z[2 * k], __uint_as_float(v[k] << 16));
          const float hi = fmaf(coef, z[2 * k + 1], __uint_as_float(v[k] & 0xFFFF0000u));
          o[k] = pack_bf16x2(lo, hi);
        }
        *reinterpret_cast<uint4*>(w) = make_uint4(o[0], o[1], o[2], o[3]);
      } else {
        for (int k = 0; k < 8 && col + k < md.n; ++k)
          w[k] = __float2bfloat16_rn(fmaf(coef, z[k], __bfloat162float(w[k])));
      }
    } else {
      float* w = reinterpret_cast<float*>(md.W) + row * md.ldw + col;
      if (full) {
        float4 x = *reinterpret_cast<const float4*>(w);
        x.x = fmaf(coef, z[0], x.x); x.y = fmaf(coef, z[1], x.y);
        x.z = fmaf(coef, z[2], x.z); x.w = fmaf(coef, z[3], x.w);
        *reinterpret_cast<float4*>(w) = x;
      } else {
        for (int k = 0; k < 4 && col + k < md.n; ++k) w[k] = fmaf(coef, z[k], w[k]);
      }
    }
  }
}

}  // namespace

cudaError_t launch_mezo(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_tile_prefix,
                        int64_t n_tiles, uint64_t seed, uint32_t t, float coef, cudaStream_t s) {
  if (n_tiles <= 0) return cudaSuccess;
  if (n_tiles > 0x7FFFFFFF) return cudaErrorInvalidValue;
  mezo_kernel<<<(unsigned)n_tiles, 256, 0, s>>>(d_mats, n_mats, d_tile_prefix, round_keys(seed), t,
                                                coef);
  return cudaGetLastError();
}

}  // namespace zo
