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
#include <algorithm>
#include <atomic>

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

// C = eps (ca Z_qa + cb Z_qb) of one matrix into shared memory, with the coefficient
// kernel's arithmetic (so that every path forms the same C).
template <int R>
__device__ __forceinline__ void draw_perturb_c(const MatDesc& md, const CoeffParams& p, float* Cs) {
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
  draw_perturb_c<R>(md, p, Cs);
  __syncthreads();
  const int64_t local = tile - md.tile0;
  if (md.dtype == 1)
    wpass_tile<R, __nv_bfloat16, true>(md, local, Us, Ps, Cs);
  else
    wpass_tile<R, float, true>(md, local, Us, Ps, Cs);
}

// The dynamic shared-memory limit of a kernel belongs to each device's context: raise it
// once per device (bit d of `done`), before the kernel's first launch there.
template <typename Kernel>
cudaError_t allow_smem(Kernel kernel, int bytes, std::atomic<uint64_t>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
  if (bit && (done.load(std::memory_order_relaxed) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done.fetch_or(bit, std::memory_order_relaxed);
  return e;
}

template <int R>
cudaError_t launch_r(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_prefix,
                     int64_t n_tiles, cudaStream_t s) {
  const size_t smem = sizeof(float) * (size_t)(kRows * R + R * 256);
  static std::atomic<uint64_t> done{0};
  cudaError_t e = allow_smem(wpass_fma_kernel<R>, (int)smem, done);
  if (e != cudaSuccess) return e;
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


// Narrow tiles.  On thin matrices -- the r_L x n and m x r_L factors of a LoRA adapter --
// the 32 x TN tile above is mostly empty (8 of its 32 rows, or 8 of its 128 columns), and a
// set of them becomes tens of thousands of nearly idle CTAs.  Here each matrix has a tile
// shape of its own, `rows` x `chunks` 16-byte column chunks filling up to kNarrowChunks
// chunks, and thread t updates chunks t, t + 256, ... of the tile in row-major order, so
// a warp still reads and writes contiguous bytes of W.  The CTA forms C (drawn, or read
// from the coefficient kernel's output) and the P columns of its tile, and stages the U
// rows.  These sets fit in L2 and the pass is latency-bound, so a CTA puts its loads out
// first -- U rows by cp.async straight into shared memory, then the V rows of its P
// columns and its W chunks into registers -- and draws C while they are in flight.  The
// arithmetic and its order are the tiled kernel's (P[k][c] and the update sum each by fmaf
// from zero in ascending index, one add and one rounding into W), so both tilings give
// bit-identical weights.
constexpr int kNarrowThreads = 256;
constexpr int kNarrowIters = kNarrowChunks / kNarrowThreads;       // W chunks per thread
constexpr int kNarrowColIters = kNarrowMaxCols / kNarrowThreads;   // P columns per thread

__device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

// Row and chunk of cell f of a tile `chunks` chunks wide: f / chunks as one fp32 product.
// With f < kNarrowChunks and chunks <= kNarrowChunks the fraction of (f + 1/2) / chunks
// stays >= 1/(2 chunks) away from an integer, far above the product's rounding error
// (< 2^-22 x 1024), so the truncation is exact.
__device__ __forceinline__ void split_cell(int f, int chunks, float inv, int& rl, int& cl) {
  rl = (int)__fmul_rn(__fadd_rn((float)f, 0.5f), inv);
  cl = f - rl * chunks;
}

template <int R, typename T, bool kDraw>
__device__ __forceinline__ void narrow_tile(const MatDesc& md, const NarrowMat& g, int64_t row0,
                                            int64_t ch0, const CoeffParams& p, float* Cs,
                                            float* Ps, float* Us) {
  constexpr int VEC = Vec<T>::N;
  const int tid = threadIdx.x;
  const int rows = g.rows, chunks = g.chunks, cols = chunks * VEC, cells = rows * chunks;
  const float inv = __frcp_rn((float)chunks);
  const int64_t cpr = (md.n + VEC - 1) / VEC;   // chunks per row of W
  const int64_t col0 = ch0 * VEC;
  const int row_end = (int)min64(rows, md.m - row0);     // live rows of the tile
  const int ch_end = (int)min64(chunks, cpr - ch0);       // live chunks of the tile
  const int full_end = (int)min64(chunks, md.n / VEC - ch0);  // chunks without a tail
  T* Wt = reinterpret_cast<T*>(md.W) + row0 * md.ldw + col0;

  // U rows of the tile: asynchronous copies into shared memory, issued first (zero-filled
  // past the last row)
  {
    const float* U0 = md.U + row0 * R;
    for (int idx = tid; idx < rows * (R / 4); idx += kNarrowThreads) {
      const bool live = idx < row_end * (R / 4);
      const uint32_t dst = (uint32_t)__cvta_generic_to_shared(Us + 4 * idx);
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst),
                   "l"(live ? U0 + 4 * idx : U0), "r"(live ? 16 : 0) : "memory");
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
  }
  // V rows of the P columns this thread forms
  const int col_end = (int)min64(cols, md.n - col0);     // live columns of the tile
  float v[kNarrowColIters][R];
#pragma unroll
  for (int j = 0; j < kNarrowColIters; ++j) {
    const int c = tid + kNarrowThreads * j;
    const float4* vrow = reinterpret_cast<const float4*>(md.V + (col0 + (c < col_end ? c : 0)) * R);
#pragma unroll
    for (int b4 = 0; b4 < R / 4; ++b4) {
      const float4 t = c < col_end ? vrow[b4] : make_float4(0.f, 0.f, 0.f, 0.f);
      v[j][4 * b4] = t.x; v[j][4 * b4 + 1] = t.y; v[j][4 * b4 + 2] = t.z; v[j][4 * b4 + 3] = t.w;
    }
  }
  // this thread's W chunks (needed last, in the update)
  uint4 wraw[kNarrowIters];
#pragma unroll
  for (int j = 0; j < kNarrowIters; ++j) {
    const int f = tid + kNarrowThreads * j;
    wraw[j] = make_uint4(0u, 0u, 0u, 0u);
    if (f < cells) {
      int rl, cl;
      split_cell(f, chunks, inv, rl, cl);
      if (rl < row_end && cl < full_end)
        wraw[j] = *reinterpret_cast<const uint4*>(Wt + (int64_t)rl * md.ldw + cl * VEC);
    }
  }
  // C while the loads are in flight
  if constexpr (kDraw) {
    draw_perturb_c<R>(md, p, Cs);
  } else {
    for (int e = tid; e < R * R / 4; e += kNarrowThreads)
      reinterpret_cast<float4*>(Cs)[e] = reinterpret_cast<const float4*>(md.C)[e];
  }
  asm volatile("cp.async.wait_all;\n" ::: "memory");
  __syncthreads();

  // P[k][c] = sum_b C[k][b] V[col0 + c][b] for the tile's columns (zero past n)
#pragma unroll
  for (int j = 0; j < kNarrowColIters; ++j) {
    const int c = tid + kNarrowThreads * j;
    if (c >= cols) break;
#pragma unroll
    for (int k = 0; k < R; ++k) {
      float acc = 0.f;
#pragma unroll
      for (int b = 0; b < R; ++b) acc = fmaf(Cs[k * R + b], v[j][b], acc);
      Ps[k * cols + c] = c < col_end ? acc : 0.f;
    }
  }
  __syncthreads();

  const float4* Us4 = reinterpret_cast<const float4*>(Us);
  const float4* Ps4 = reinterpret_cast<const float4*>(Ps);
#pragma unroll
  for (int j = 0; j < kNarrowIters; ++j) {
    const int f = tid + kNarrowThreads * j;
    if (f >= cells) break;
    int rl, cl;
    split_cell(f, chunks, inv, rl, cl);
    if (rl >= row_end || cl >= ch_end) continue;
    float acc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e) acc[e] = 0.f;
#pragma unroll
    for (int k4 = 0; k4 < R / 4; ++k4) {
      const float4 u = Us4[rl * (R / 4) + k4];
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const int k = 4 * k4 + kk;
        const float uk = kk == 0 ? u.x : kk == 1 ? u.y : kk == 2 ? u.z : u.w;
#pragma unroll
        for (int part = 0; part < VEC / 4; ++part) {
          const float4 t = Ps4[(k * cols + cl * VEC) / 4 + part];
          acc[4 * part] = fmaf(uk, t.x, acc[4 * part]);
          acc[4 * part + 1] = fmaf(uk, t.y, acc[4 * part + 1]);
          acc[4 * part + 2] = fmaf(uk, t.z, acc[4 * part + 2]);
          acc[4 * part + 3] = fmaf(uk, t.w, acc[4 * part + 3]);
        }
      }
    }
    T* wp = Wt + (int64_t)rl * md.ldw + cl * VEC;
    if (cl < full_end) {
      float w[VEC];
      unpack(wraw[j], w, T());
#pragma unroll
      for (int e = 0; e < VEC; ++e) w[e] += acc[e];
      *reinterpret_cast<uint4*>(wp) = pack(w, T());
    } else {
      const int left = col_end - cl * VEC;   // elements of the ragged last chunk
#pragma unroll
      for (int e = 0; e < VEC; ++e)
        if (e < left) store_scalar<T>(wp + e, load_scalar<T>(wp + e) + acc[e]);
    }
  }
}

// Shared memory: C (R x R), then the P part (p_floats), then the U part.
template <int R, bool kDraw>
__global__ void __launch_bounds__(kNarrowThreads, R <= 4 ? 4 : 3)
wpass_narrow_kernel(const MatDesc* __restrict__ mats, const NarrowMat* __restrict__ narrow,
                    const int4* __restrict__ tiles, CoeffParams p, int32_t p_floats) {
  extern __shared__ float4 smem4[];
  float* Cs = reinterpret_cast<float*>(smem4);
  float* Ps = Cs + R * R;
  float* Us = Ps + p_floats;
  // (matrix, first row, first chunk) of this tile, laid out by the host
  const int4 td = __ldg(tiles + blockIdx.x);
  const MatDesc md = mats[td.x];
  const NarrowMat g = narrow[td.x];
  if (md.dtype == 1)
    narrow_tile<R, __nv_bfloat16, kDraw>(md, g, td.y, td.z, p, Cs, Ps, Us);
  else
    narrow_tile<R, float, kDraw>(md, g, td.y, td.z, p, Cs, Ps, Us);
}

template <int R, bool kDraw>
cudaError_t launch_narrow_r(const MatDesc* d_mats, const NarrowMat* d_narrow,
                            const int4* d_tiles, int64_t n_tiles, const CoeffParams& p,
                            int64_t p_floats, int64_t u_floats, cudaStream_t s) {
  const size_t smem = sizeof(float) * (size_t)(R * R + p_floats + u_floats);
  // the largest shape narrow_tile_shape can give: kNarrowMaxCols P columns, or
  // kNarrowChunks rows of U
  static std::atomic<uint64_t> done{0};
  const int most = (int)(sizeof(float) * (R * R + R * kNarrowMaxCols + R * kNarrowChunks));
  cudaError_t e = allow_smem(wpass_narrow_kernel<R, kDraw>, most, done);
  if (e != cudaSuccess) return e;
  wpass_narrow_kernel<R, kDraw><<<(unsigned)n_tiles, kNarrowThreads, smem, s>>>(
      d_mats, d_narrow, d_tiles, p, (int32_t)p_floats);
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

bool wpass_narrow_supported(int32_t r) { return r == 4 || r == 8; }

void narrow_tile_shape(int64_t m, int64_t n, int32_t dtype, int32_t* rows, int32_t* chunks) {
  const int64_t vec = dtype == 1 ? 8 : 4;
  const int64_t cpr = (n + vec - 1) / vec;
  const int64_t max_chunks = kNarrowMaxCols / vec;
  int64_t ch = std::min<int64_t>({cpr, 128, max_chunks});
  const int64_t rw = std::max<int64_t>(1, std::min<int64_t>(m, kNarrowChunks / ch));
  // a short matrix takes its whole height and widens the tile instead
  ch = std::max<int64_t>(1, std::min<int64_t>({cpr, kNarrowChunks / rw, max_chunks}));
  *rows = (int32_t)rw;
  *chunks = (int32_t)ch;
}

int64_t narrow_p_floats(int32_t r, int32_t chunks, int32_t dtype) {
  return (int64_t)r * chunks * (dtype == 1 ? 8 : 4);
}
int64_t narrow_u_floats(int32_t r, int32_t rows) { return (int64_t)r * rows; }

cudaError_t launch_wpass_narrow(const MatDesc* d_mats, const NarrowMat* d_narrow,
                                const int4* d_tiles, int64_t n_tiles, const CoeffParams& p,
                                int64_t p_floats, int64_t u_floats, cudaStream_t s) {
  if (n_tiles <= 0) return cudaSuccess;
  if (n_tiles > 0x7FFFFFFF || p_floats < 0 || u_floats < 0 ||
      p_floats > (int64_t)p.r * kNarrowMaxCols || u_floats > (int64_t)p.r * kNarrowChunks)
    return cudaErrorInvalidValue;
  const bool draw = p.mode == kCoeffPerturb;
  switch (p.r) {
    case 4:
      return draw ? launch_narrow_r<4, true>(d_mats, d_narrow, d_tiles, n_tiles, p, p_floats, u_floats, s)
                  : launch_narrow_r<4, false>(d_mats, d_narrow, d_tiles, n_tiles, p, p_floats, u_floats, s);
    case 8:
      return draw ? launch_narrow_r<8, true>(d_mats, d_narrow, d_tiles, n_tiles, p, p_floats, u_floats, s)
                  : launch_narrow_r<8, false>(d_mats, d_narrow, d_tiles, n_tiles, p, p_floats, u_floats, s);
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
