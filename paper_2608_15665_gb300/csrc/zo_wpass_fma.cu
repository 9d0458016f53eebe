// Weight pass, fp32-FMA path: W_i <- rnd(W_i + U_i P_i) for every matrix in one
// launch, with P_i = C_i V_i^T precomputed (r x n fp32).  This is the fused
// form of Alg. 2's "W_i <- W_i + eps U_i Z_i V_i^T" (Eq. (4)) and of the update
// of Eq. (10): the r-term contraction is done in fp32 FMAs and W is rounded once.
//
// Tiling: a CTA owns a 32-row x TN-column tile of one W_i (TN = 32 lanes x 16 B).
// Each thread keeps a 4-row x (16 B of W) register tile; W is read and written
// with 16-byte coalesced vector accesses (a warp covers 512 contiguous bytes of
// a row), U and P tiles are staged through shared memory.  HBM traffic per
// element is one read and one write of W; U and P tiles come from L2.
#include "zo_kernels.h"

namespace zo {
namespace {

constexpr int kRows = kFmaTileRows;   // 32
constexpr int kRowsPerThread = kRows / 8;   // 8 warps stacked over the tile rows

template <typename T> struct Vec;
template <> struct Vec<float> { static constexpr int N = 4; };
template <> struct Vec<__nv_bfloat16> { static constexpr int N = 8; };

__device__ __forceinline__ void unpack(const uint4& raw, float (&w)[4], float) {
  w[0] = __uint_as_float(raw.x); w[1] = __uint_as_float(raw.y);
  w[2] = __uint_as_float(raw.z); w[3] = __uint_as_float(raw.w);
}
__device__ __forceinline__ uint4 pack(const float (&w)[4], float) {
  return make_uint4(__float_as_uint(w[0]), __float_as_uint(w[1]), __float_as_uint(w[2]),
                    __float_as_uint(w[3]));
}
__device__ __forceinline__ void unpack(const uint4& raw, float (&w)[8], __nv_bfloat16) {
  const uint32_t v[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    w[2 * i] = __uint_as_float(v[i] << 16);
    w[2 * i + 1] = __uint_as_float(v[i] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ uint32_t pack2_bf16(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);   // RNE, lo in the low half
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ uint4 pack(const float (&w)[8], __nv_bfloat16) {
  return make_uint4(pack2_bf16(w[0], w[1]), pack2_bf16(w[2], w[3]), pack2_bf16(w[4], w[5]),
                    pack2_bf16(w[6], w[7]));
}

template <typename T>
__device__ __forceinline__ float load_scalar(const T* p);
template <>
__device__ __forceinline__ float load_scalar<float>(const float* p) { return *p; }
template <>
__device__ __forceinline__ float load_scalar<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}
template <typename T>
__device__ __forceinline__ void store_scalar(T* p, float x);
template <>
__device__ __forceinline__ void store_scalar<float>(float* p, float x) { *p = x; }
template <>
__device__ __forceinline__ void store_scalar<__nv_bfloat16>(__nv_bfloat16* p, float x) {
  *p = __float2bfloat16_rn(x);
}

__device__ __forceinline__ int find_matrix(const int64_t* __restrict__ prefix, int n_mats,
                                           int64_t tile) {
  int lo = 0, hi = n_mats - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(prefix + mid) <= tile) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// With kFused, P's columns of this tile are formed here from C (already in shared memory,
// Cs) and V, in the projection kernel's order (sum over b ascending, one fmaf per term),
// instead of being read from md.P.
template <int R, typename T, bool kFused>
__device__ __forceinline__ void wpass_tile(const MatDesc& md, int64_t local, float* Us, float* Ps,
                                           const float* Cs) {
  constexpr int VEC = Vec<T>::N;
  constexpr int TN = 32 * VEC;
  const int tid = threadIdx.x;
  const int tx = tid & 31, ty = tid >> 5;
  const int64_t tiles_n = (md.n + TN - 1) / TN;
  const int64_t row0 = (local / tiles_n) * kRows;
  const int64_t col0 = (local % tiles_n) * TN;
  T* W = reinterpret_cast<T*>(md.W);

  // prefetch this thread's W vectors (4 rows x 16 B)
  uint4 wraw[kRowsPerThread];
  const int64_t col = col0 + tx * VEC;
  const bool full_vec = col + VEC <= md.n;
#pragma unroll
  for (int rho = 0; rho < kRowsPerThread; ++rho) {
    const int64_t row = row0 + ty * kRowsPerThread + rho;
    wraw[rho] = make_uint4(0u, 0u, 0u, 0u);
    if (row < md.m && full_vec)
      wraw[rho] = *reinterpret_cast<const uint4*>(W + row * md.ldw + col);
  }

  // stage U rows [row0, row0+64) and P columns [col0, col0+TN) in shared memory
  {
    const float4* U4 = reinterpret_cast<const float4*>(md.U);
    float4* Us4 = reinterpret_cast<float4*>(Us);
    for (int idx = tid; idx < kRows * R / 4; idx += blockDim.x) {
      const int64_t row = row0 + idx / (R / 4);
      Us4[idx] = row < md.m ? U4[row0 * (R / 4) + idx] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    // layout [k][c % VEC / 4][c / VEC][c % 4]: a thread's 16-B chunks are contiguous across lanes
    if constexpr (kFused) {
      for (int c = tid; c < TN; c += blockDim.x) {
        const int64_t gc = col0 + c;
        const int lane = c / VEC, part = (c % VEC) / 4, l4 = c % 4;
        float v[R];
#pragma unroll
        for (int b = 0; b < R; ++b) v[b] = gc < md.n ? md.V[gc * R + b] : 0.f;
#pragma unroll
        for (int k = 0; k < R; ++k) {
          float acc = 0.f;
#pragma unroll
          for (int b = 0; b < R; ++b) acc = fmaf(Cs[k * R + b], v[b], acc);
          Ps[k * TN + part * 128 + lane * 4 + l4] = gc < md.n ? acc : 0.f;
        }
      }
    } else {
      for (int idx = tid; idx < R * TN; idx += blockDim.x) {
        const int k = idx / TN, c = idx % TN;
        const int64_t gc = col0 + c;
        const float pv = gc < md.n ? md.P[(int64_t)k * md.n + gc] : 0.f;
        const int lane = c / VEC, part = (c % VEC) / 4, l4 = c % 4;
        Ps[k * TN + part * 128 + lane * 4 + l4] = pv;
      }
    }
  }
  __syncthreads();

  float acc[kRowsPerThread][VEC];
#pragma unroll
  for (int rho = 0; rho < kRowsPerThread; ++rho)
#pragma unroll
    for (int v = 0; v < VEC; ++v) acc[rho][v] = 0.f;

  const float4* Us4 = reinterpret_cast<const float4*>(Us);
  const float4* Ps4 = reinterpret_cast<const float4*>(Ps);
#pragma unroll 2
  for (int k4 = 0; k4 < R / 4; ++k4) {
    float4 u[kRowsPerThread];
#pragma unroll
    for (int rho = 0; rho < kRowsPerThread; ++rho)
      u[rho] = Us4[(ty * kRowsPerThread + rho) * (R / 4) + k4];
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const int k = 4 * k4 + kk;
      float p[VEC];
#pragma unroll
      for (int part = 0; part < VEC / 4; ++part) {
        const float4 t = Ps4[(k * TN + part * 128) / 4 + tx];
        p[4 * part] = t.x; p[4 * part + 1] = t.y; p[4 * part + 2] = t.z; p[4 * part + 3] = t.w;
      }
#pragma unroll
      for (int rho = 0; rho < kRowsPerThread; ++rho) {
        const float uk = kk == 0 ? u[rho].x : kk == 1 ? u[rho].y : kk == 2 ? u[rho].z : u[rho].w;
#pragma unroll
        for (int v = 0; v < VEC; ++v) acc[rho][v] = fmaf(uk, p[v], acc[rho][v]);
      }
    }
  }

#pragma unroll
  for (int rho = 0; rho < kRowsPerThread; ++rho) {
    const int64_t row = row0 + ty * kRowsPerThread + rho;
    if (row >= md.m) continue;
    T* wrow = W + row * md.ldw;
    if (full_vec) {
      float w[VEC];
      unpack(wraw[rho], w, T());
#pragma unroll
      for (int v = 0; v < VEC; ++v) w[v] += acc[rho][v];
      *reinterpret_cast<uint4*>(wrow + col) = pack(w, T());
    } else {
#pragma unroll
      for (int v = 0; v < VEC; ++v)
        if (col + v < md.n) store_scalar<T>(wrow + col + v, load_scalar<T>(wrow + col + v) + acc[rho][v]);
    }
  }
}

template <int R>
__global__ void __launch_bounds__(256, 2)
wpass_fma_kernel(const MatDesc* __restrict__ mats, int n_mats, const int64_t* __restrict__ prefix) {
  extern __shared__ float4 smem4[];
  float* Us = reinterpret_cast<float*>(smem4);
  float* Ps = Us + kRows * R;
  const int64_t tile = blockIdx.x;
  const int i = find_matrix(prefix, n_mats, tile);
  const MatDesc md = mats[i];
  const int64_t local = tile - md.tile0;
  if (md.dtype == 1)
    wpass_tile<R, __nv_bfloat16, false>(md, local, Us, Ps, nullptr);
  else
    wpass_tile<R, float, false>(md, local, Us, Ps, nullptr);
}

// One launch per perturbation pass at small r: every CTA forms its matrix's C = eps (ca
// Z_qa + cb Z_qb) in shared memory -- r^2 Gaussians, the coefficient kernel's arithmetic --
// and the P columns of its tile, then updates the tile.  For the L2-resident sets the pass
// is launch-bound, and one launch replaces three.
template <int R>
__global__ void __launch_bounds__(256, 2)
wpass_fma_fused_kernel(const MatDesc* __restrict__ mats, int n_mats,
                       const int64_t* __restrict__ prefix, CoeffParams p) {
  extern __shared__ float4 smem4[];
  float* Us = reinterpret_cast<float*>(smem4);
  float* Ps = Us + kRows * R;
  float* Cs = Ps + R * 256;
  const int64_t tile = blockIdx.x;
  const int i = find_matrix(prefix, n_mats, tile);
  const MatDesc md = mats[i];
  for (int c = threadIdx.x; c < R * R / 4; c += blockDim.x) {
    const float4 za = normal4(p.seed, (uint32_t)c, md.gidx, p.t, query_word(kTagZ, (uint32_t)p.qa));
    float4 acc = make_float4(p.ca * za.x, p.ca * za.y, p.ca * za.z, p.ca * za.w);
    if (p.qb >= 0) {
      const float4 zb = normal4(p.seed, (uint32_t)c, md.gidx, p.t, query_word(kTagZ, (uint32_t)p.qb));
      acc = make_float4(fmaf(p.cb, zb.x, acc.x), fmaf(p.cb, zb.y, acc.y), fmaf(p.cb, zb.z, acc.z),
                        fmaf(p.cb, zb.w, acc.w));
    }
    reinterpret_cast<float4*>(Cs)[c] =
        make_float4(p.eps * acc.x, p.eps * acc.y, p.eps * acc.z, p.eps * acc.w);
  }
  __syncthreads();
  const int64_t local = tile - md.tile0;
  if (md.dtype == 1)
    wpass_tile<R, __nv_bfloat16, true>(md, local, Us, Ps, Cs);
  else
    wpass_tile<R, float, true>(md, local, Us, Ps, Cs);
}

template <int R>
cudaError_t launch_r(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_prefix,
                     int64_t n_tiles, cudaStream_t s) {
  const size_t smem = sizeof(float) * (size_t)(kRows * R + R * 256);
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(wpass_fma_kernel<R>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  wpass_fma_kernel<R><<<(unsigned)n_tiles, 256, smem, s>>>(d_mats, n_mats, d_prefix);
  return cudaGetLastError();
}

template <int R>
cudaError_t launch_fused_r(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_prefix,
                           int64_t n_tiles, const CoeffParams& p, cudaStream_t s) {
  const size_t smem = sizeof(float) * (size_t)(kRows * R + R * 256 + R * R);
  wpass_fma_fused_kernel<R><<<(unsigned)n_tiles, 256, smem, s>>>(d_mats, n_mats, d_prefix, p);
  return cudaGetLastError();
}

}  // namespace

bool wpass_fma_fused_supported(int32_t r) { return r == 4 || r == 8; }

cudaError_t launch_wpass_fma_fused(const MatDesc* d_mats, int32_t n_mats,
                                   const int64_t* d_tile_prefix, int64_t n_tiles,
                                   const CoeffParams& p, cudaStream_t s) {
  if (n_tiles <= 0) return cudaSuccess;
  if (n_tiles > 0x7FFFFFFF) return cudaErrorInvalidValue;
  switch (p.r) {
    case 4: return launch_fused_r<4>(d_mats, n_mats, d_tile_prefix, n_tiles, p, s);
    case 8: return launch_fused_r<8>(d_mats, n_mats, d_tile_prefix, n_tiles, p, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_wpass_fma(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_tile_prefix,
                             int64_t n_tiles, int32_t r, cudaStream_t s) {
  if (n_tiles <= 0) return cudaSuccess;
  if (n_tiles > 0x7FFFFFFF) return cudaErrorInvalidValue;
  switch (r) {
    case 4: return launch_r<4>(d_mats, n_mats, d_tile_prefix, n_tiles, s);
    case 8: return launch_r<8>(d_mats, n_mats, d_tile_prefix, n_tiles, s);
    case 16: return launch_r<16>(d_mats, n_mats, d_tile_prefix, n_tiles, s);
    case 32: return launch_r<32>(d_mats, n_mats, d_tile_prefix, n_tiles, s);
    case 64: return launch_r<64>(d_mats, n_mats, d_tile_prefix, n_tiles, s);
    case 128: return launch_r<128>(d_mats, n_mats, d_tile_prefix, n_tiles, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
