// Subspace refresh for tall panels at r = 16 ... 128: Alg. 1's Haar factor by
// CholeskyQR2 (Fukaya, Nakatsukasa, Yanagisawa and Yamamoto, 2014).
//
// Alg. 1 wants Q of the QR factorisation of a Gaussian panel Omega (rows x r) with the
// signs fixed so that diag(R) > 0 (Eq. (11)).  That Q is unique, and it is also
// Omega R^-1 with R^T R = Omega^T Omega the Cholesky factorisation (whose diagonal is
// positive by construction).  One Cholesky QR in fp32 leaves Q orthogonal only to about
// kappa(Omega)^2 u; applied a second time to its own output it reaches O(u) when
// kappa(Omega)^2 u << 1 -- for a tall Gaussian panel (rows >= 4r), kappa <= ~3.  So per
// panel:
//   G1 = Omega^T Omega,  L1 L1^T = G1,  Q1 = Omega L1^-T,
//   G2 = Q1^T Q1,        L2 L2^T = G2,  Q  = Q1 L2^-T        (Q = Omega (L2^T L1^T)^-1),
// and Q lands in U (or V).  Every step but the two r x r Cholesky factorisations is a
// batched product over rows, so the refresh runs at the speed of those products instead
// of r dependent Householder steps per block.  Omega is drawn in the kernels from the
// counter contract (tags 2 / 3, element e = row * r + col at counter e / 4, lane e % 4),
// exactly as the TSQR of zo_qr.cu draws it; panels shorter than 4r, and every panel at
// r = 4 and 8, keep the TSQR.
//
// Launches per refresh: gram(Omega), chol, apply(Omega -> Q1), gram(Q1), chol,
// apply(Q1 -> Q).  Sums over rows are fixed-order (per 1024-row chunk, then chunk by
// chunk), so a refresh is bit-reproducible.
#include "zo_kernels.h"

namespace zo {
namespace {

constexpr int kCqThreads = 256;
constexpr int kGramSub = 32;     // rows staged per step of the Gram kernel
constexpr int kApplySub = 64;    // rows per tile of the apply kernel

// Rows r0 .. r0 + n - 1 of a panel into shared memory (row-major, `ld` floats per row):
// drawn from the counter contract, or read from the panel's output buffer.
template <int R, bool kOmega>
__device__ __forceinline__ void stage_rows(const CqPanel& pn, int64_t r0, int n, float* dst, int ld,
                                           uint64_t seed, uint32_t refresh_idx) {
  constexpr int kW = R / 4;                      // 4-float words per row
  for (int w = threadIdx.x; w < n * kW; w += blockDim.x) {
    const int i = w / kW, c4 = w % kW;
    float4 z;
    if constexpr (kOmega) {
      const uint32_t c = (uint32_t)((((r0 + i) * R) >> 2) + c4);
      z = normal4(seed, c, pn.gidx, refresh_idx, query_word(pn.tag, 0));
    } else {
      z = reinterpret_cast<const float4*>(pn.out + (r0 + i) * R)[c4];
    }
    *reinterpret_cast<float4*>(dst + i * ld + 4 * c4) = z;
  }
}

// T consecutive floats (T = 1, 2, 4 or 8) from shared memory, and the same to global memory.
template <int T>
__device__ __forceinline__ void load_t(const float* p, float (&v)[T]) {
  if constexpr (T >= 4) {
#pragma unroll
    for (int q = 0; q < T / 4; ++q) {
      const float4 a = reinterpret_cast<const float4*>(p)[q];
      v[4 * q] = a.x; v[4 * q + 1] = a.y; v[4 * q + 2] = a.z; v[4 * q + 3] = a.w;
    }
  } else if constexpr (T == 2) {
    const float2 a = *reinterpret_cast<const float2*>(p);
    v[0] = a.x; v[1] = a.y;
  } else {
    v[0] = p[0];
  }
}
template <int T>
__device__ __forceinline__ void store_t(float* p, const float (&v)[T]) {
  if constexpr (T >= 4) {
#pragma unroll
    for (int q = 0; q < T / 4; ++q)
      reinterpret_cast<float4*>(p)[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
  } else if constexpr (T == 2) {
    *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
  } else {
    p[0] = v[0];
  }
}

// Partial Gram matrix X^T X of one chunk (<= kCqChunkRows rows of one panel).  Thread
// (ty, tx) of a 16 x 16 grid accumulates the T x T block rows ty*T.., columns tx*T..,
// T = R / 16, over the chunk's rows.
template <int R, bool kOmega>
__global__ void __launch_bounds__(kCqThreads)
cq_gram_kernel(const CqPanel* __restrict__ panels, const CqChunk* __restrict__ chunks,
               float* __restrict__ partial, uint64_t seed, uint32_t refresh_idx) {
  constexpr int T = R / 16;
  constexpr int kLd = R + 4;
  __shared__ __align__(16) float X[kGramSub * kLd];
  const CqChunk ch = chunks[blockIdx.x];
  const CqPanel pn = panels[ch.panel];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[T][T];
#pragma unroll
  for (int a = 0; a < T; ++a)
#pragma unroll
    for (int b = 0; b < T; ++b) acc[a][b] = 0.f;
  for (int s0 = 0; s0 < ch.nrows; s0 += kGramSub) {
    const int n = ch.nrows - s0 < kGramSub ? ch.nrows - s0 : kGramSub;
    __syncthreads();
    stage_rows<R, kOmega>(pn, ch.row0 + s0, n, X, kLd, seed, refresh_idx);
    __syncthreads();
    for (int k = 0; k < n; ++k) {
      float xa[T], xb[T];
      load_t<T>(X + k * kLd + ty * T, xa);
      load_t<T>(X + k * kLd + tx * T, xb);
#pragma unroll
      for (int a = 0; a < T; ++a)
#pragma unroll
        for (int b = 0; b < T; ++b) acc[a][b] = fmaf(xa[a], xb[b], acc[a][b]);
    }
  }
  float* out = partial + (int64_t)blockIdx.x * R * R;
#pragma unroll
  for (int a = 0; a < T; ++a)
#pragma unroll
    for (int b = 0; b < T; ++b) out[(ty * T + a) * R + tx * T + b] = acc[a][b];
}

// One CTA per panel: G = sum of the panel's chunk partials (chunk order), then the
// Cholesky factor L (G = L L^T, right-looking, in shared memory) and its inverse; writes
// L^-1 (lower triangular, zeros above) to linv[panel].  A non-positive pivot -- not
// expected for a tall Gaussian panel -- sets kDevNotPosDef and leaves L^-1 = 0.
template <int R>
__global__ void __launch_bounds__(kCqThreads)
cq_chol_kernel(const CqPanel* __restrict__ panels, const float* __restrict__ partial,
               float* __restrict__ linv, uint32_t* __restrict__ status) {
  constexpr int kLd = R + 1;
  extern __shared__ float cq_smem[];
  float* G = cq_smem;                            // R x kLd: G, then L in its lower triangle
  float* Y = cq_smem + R * kLd;                  // R x kLd: L^-1
  __shared__ int bad;
  const CqPanel pn = panels[blockIdx.x];
  const int tid = threadIdx.x;
  for (int e = tid; e < R * R; e += kCqThreads) {
    float g = 0.f;
    for (int c = 0; c < pn.n_chunks; ++c) g += partial[(int64_t)(pn.chunk0 + c) * R * R + e];
    G[(e / R) * kLd + e % R] = g;
  }
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int k = 0; k < R; ++k) {
    if (tid == 0) {
      const float d = G[k * kLd + k];
      if (!(d > 0.f)) bad = 1;
      G[k * kLd + k] = d > 0.f ? sqrtf(d) : 1.f;
    }
    __syncthreads();
    const float inv = 1.f / G[k * kLd + k];
    for (int i = k + 1 + tid; i < R; i += kCqThreads) G[i * kLd + k] *= inv;
    __syncthreads();
    // trailing update of the lower triangle: G[i][j] -= L[i][k] L[j][k], k < j <= i
    const int m = R - k - 1;
    for (int e = tid; e < m * m; e += kCqThreads) {
      const int i = k + 1 + e / m, j = k + 1 + e % m;
      if (j <= i) G[i * kLd + j] = fmaf(-G[i * kLd + k], G[j * kLd + k], G[i * kLd + j]);
    }
    __syncthreads();
  }
  // L Y = I: thread t < R solves column t by forward substitution
  if (tid < R) {
    const int t = tid;
    for (int i = 0; i < t; ++i) Y[i * kLd + t] = 0.f;
    Y[t * kLd + t] = 1.f / G[t * kLd + t];
    for (int i = t + 1; i < R; ++i) {
      float s = 0.f;
      for (int k = t; k < i; ++k) s = fmaf(G[i * kLd + k], Y[k * kLd + t], s);
      Y[i * kLd + t] = -s / G[i * kLd + i];
    }
  }
  __syncthreads();
  float* out = linv + (int64_t)blockIdx.x * R * R;
  for (int e = tid; e < R * R; e += kCqThreads) out[e] = bad ? 0.f : Y[(e / R) * kLd + e % R];
  if (tid == 0 && bad) atomicOr(status, (uint32_t)kDevNotPosDef);
}

// Q rows = X rows L^-T over one chunk, in tiles of kApplySub rows: out[j][a] =
// sum_{b <= a} X[j][b] Linv[a][b].  X is staged b-major (XT[b][j]) and Linv as its
// transpose LT[b][a], so one 16-byte load feeds 4 rows or 4 columns; thread (ty, tx) of
// a 16 x 16 grid owns rows 4 ty .. + 3 and columns tx * T .. + T - 1, T = R / 16.
// Writes Q over the panel's rows (in place when X was read from them: a tile is fully
// staged before any of its rows is written).
template <int R, bool kOmega>
__global__ void __launch_bounds__(kCqThreads)
cq_apply_kernel(const CqPanel* __restrict__ panels, const CqChunk* __restrict__ chunks,
                const float* __restrict__ linv, uint64_t seed, uint32_t refresh_idx) {
  constexpr int T = R / 16;
  constexpr int kLdX = kApplySub + 4;            // XT row pitch (floats)
  constexpr int kLdL = R + 4;                    // LT row pitch
  extern __shared__ float cq_smem[];
  float* XT = cq_smem;                           // R x kLdX
  float* LT = cq_smem + R * kLdX;                // R x kLdL
  float* Xs = LT + R * kLdL;                     // kApplySub x (R + 4), staging
  const CqChunk ch = chunks[blockIdx.x];
  const CqPanel pn = panels[ch.panel];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const float* L = linv + (int64_t)ch.panel * R * R;
  for (int e = threadIdx.x; e < R * R; e += kCqThreads) LT[(e % R) * kLdL + e / R] = L[e];
  for (int s0 = 0; s0 < ch.nrows; s0 += kApplySub) {
    const int n = ch.nrows - s0 < kApplySub ? ch.nrows - s0 : kApplySub;
    __syncthreads();
    stage_rows<R, kOmega>(pn, ch.row0 + s0, n, Xs, R + 4, seed, refresh_idx);
    __syncthreads();
    for (int e = threadIdx.x; e < kApplySub * R; e += kCqThreads) {
      const int j = e % kApplySub, b = e / kApplySub;
      XT[b * kLdX + j] = j < n ? Xs[j * (R + 4) + b] : 0.f;
    }
    __syncthreads();
    float acc[4][T];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int c = 0; c < T; ++c) acc[i][c] = 0.f;
    for (int b = 0; b < R; ++b) {
      const float4 x4 = *reinterpret_cast<const float4*>(XT + b * kLdX + 4 * ty);
      const float x[4] = {x4.x, x4.y, x4.z, x4.w};
      float l[T];
      load_t<T>(LT + b * kLdL + tx * T, l);
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int c = 0; c < T; ++c) acc[i][c] = fmaf(x[i], l[c], acc[i][c]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int j = 4 * ty + i;
      if (j >= n) continue;
      store_t<T>(pn.out + (ch.row0 + s0 + j) * R + tx * T, acc[i]);
    }
  }
}

template <int R>
size_t chol_smem() { return sizeof(float) * 2 * R * (R + 1); }
template <int R>
size_t apply_smem() {
  return sizeof(float) * ((size_t)R * (kApplySub + 4) + (size_t)R * (R + 4) + (size_t)kApplySub * (R + 4));
}

template <int R>
cudaError_t run_cholqr_r(const CqPanel* d_panels, int32_t n_panels, const CqChunk* d_chunks,
                         int32_t n_chunks, float* d_partial, float* d_linv, uint64_t seed,
                         uint32_t refresh_idx, uint32_t* d_status, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(cq_chol_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)chol_smem<R>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(cq_apply_kernel<R, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)apply_smem<R>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(cq_apply_kernel<R, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)apply_smem<R>());
  if (e != cudaSuccess) return e;
  // first Cholesky QR: Omega -> Q1 (written to the panels)
  cq_gram_kernel<R, true><<<n_chunks, kCqThreads, 0, s>>>(d_panels, d_chunks, d_partial, seed, refresh_idx);
  cq_chol_kernel<R><<<n_panels, kCqThreads, chol_smem<R>(), s>>>(d_panels, d_partial, d_linv, d_status);
  cq_apply_kernel<R, true><<<n_chunks, kCqThreads, apply_smem<R>(), s>>>(d_panels, d_chunks, d_linv,
                                                                         seed, refresh_idx);
  // second: Q1 -> Q, in place
  cq_gram_kernel<R, false><<<n_chunks, kCqThreads, 0, s>>>(d_panels, d_chunks, d_partial, seed, refresh_idx);
  cq_chol_kernel<R><<<n_panels, kCqThreads, chol_smem<R>(), s>>>(d_panels, d_partial, d_linv, d_status);
  cq_apply_kernel<R, false><<<n_chunks, kCqThreads, apply_smem<R>(), s>>>(d_panels, d_chunks, d_linv,
                                                                          seed, refresh_idx);
  return cudaGetLastError();
}

}  // namespace

bool cholqr_supported(int32_t r) { return r == 16 || r == 32 || r == 64 || r == 128; }

cudaError_t launch_cholqr(const CqPanel* d_panels, int32_t n_panels, const CqChunk* d_chunks,
                          int32_t n_chunks, float* d_partial, float* d_linv, int32_t r,
                          uint64_t seed, uint32_t refresh_idx, uint32_t* d_status, cudaStream_t s) {
  if (n_panels <= 0) return cudaSuccess;
  switch (r) {
    case 16: return run_cholqr_r<16>(d_panels, n_panels, d_chunks, n_chunks, d_partial, d_linv, seed, refresh_idx, d_status, s);
    case 32: return run_cholqr_r<32>(d_panels, n_panels, d_chunks, n_chunks, d_partial, d_linv, seed, refresh_idx, d_status, s);
    case 64: return run_cholqr_r<64>(d_panels, n_panels, d_chunks, n_chunks, d_partial, d_linv, seed, refresh_idx, d_status, s);
    case 128: return run_cholqr_r<128>(d_panels, n_panels, d_chunks, n_chunks, d_partial, d_linv, seed, refresh_idx, d_status, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
