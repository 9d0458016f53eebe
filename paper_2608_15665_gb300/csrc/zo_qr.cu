// Subspace refresh: Alg. 1 (the Haar-distributed bases U, V) for every matrix in a few launches.
//
// For each panel (Omega_U, m x r and Omega_V, n x r) we need the thin QR factor
// with a positive diagonal of R (Eq. (11)).  Panels are tall and skinny (m up to
// 25600, r <= 128) and there are up to ~900 of them, so the factorisation is a
// batched TSQR (communication-avoiding QR, Demmel et al. 2012):
//
//   up pass, level 0:  each block of B rows draws its Omega rows from the
//                      counter contract, factors them by Householder reflections
//                      held in registers (one or more rows per thread), stores
//                      the reflectors over its rows and its r x r R factor into
//                      the next level's stack.
//   up pass, level l:  the stacked R factors are factored the same way.
//   top block:         once a panel's stack fits in one block, that block forms
//                      Q_top = H_0 ... H_(r-1) [diag(sgn R_cc); 0] directly -- the sign
//                      correction of Eq. (11) folded into the start of Q -- and
//                      writes it over its stack.
//   down pass:         every other block applies its reflectors to [S; 0], S the
//                      r x r block of its parent's Q that multiplies its R, giving
//                      its rows of Q; at level 0 those are the rows of U (or V).
//
// Householder convention (Golub & Van Loan, Sec. 5.1): for x = A[j:, j],
// beta = -sign(x_0) ||x||, v = x / (x_0 - beta) with v_0 = 1, tau = (beta - x_0)/beta.
// Blocks with fewer real rows than B are padded with zero rows, which leaves the
// factorisation of the real rows unchanged and produces zero rows of Q there.
#include "zo_kernels.h"

namespace zo {
namespace {

constexpr int kQrThreads = 256;
constexpr int kQrWarps = kQrThreads / 32;

template <int R>
struct QrShape {
  static constexpr int kRPT = R >= 64 ? 1 : 64 / R;   // rows per thread
  static constexpr int kB = kQrThreads * kRPT;        // rows per block
  static constexpr int kLd = R + 1;                   // padded row stride of the reflector copy
};

// Shared scratch of one QR block.
template <int R>
struct QrSmem {
  float red[2][kQrWarps][R];   // per-warp partial sums, double-buffered by step parity
  float wbuf[2][R];            // reduced vector of the current step
  float rowj[2][R];            // row j of the panel (owner's copy)
  float scal[2][2];            // tau, 1/(alpha - beta) of the current step
  float diag[R];               // beta_j = R_jj
  float tau[R];
};

// Recursive-halving reduction of R per-lane values across a warp.  Afterwards
// lane l holds the warp sum of element c = l * (R/32) + k (k < R/32) when R >= 32,
// or of element c = l / (32/R) (in p[0]) when R < 32.
template <int R>
__device__ __forceinline__ void warp_reduce_scatter(float (&p)[R], int lane) {
#pragma unroll
  for (int s = 0; s < 5; ++s) {
    const int o = 16 >> s;
    const int size = R >> s;
    if (size >= 2) {
      const int half = size >> 1;
      const bool upper = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < R / 2; ++i) {
        if (i < half) {
          const float send = upper ? p[i] : p[i + half];
          const float keep = upper ? p[i + half] : p[i];
          p[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
      }
    } else {
      p[0] += __shfl_xor_sync(0xffffffffu, p[0], o);
    }
  }
}

// Block-wide sum of H per-thread values (columns off .. off+H-1) into
// red[warp][off + c] (one partial per warp).
template <int H>
__device__ __forceinline__ void block_partials(float (&p)[H], float* red_buf, int row_len,
                                               int off) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float* red = red_buf + warp * row_len + off;
  warp_reduce_scatter<H>(p, lane);
  if (H >= 32) {
    constexpr int kKeep = H >= 32 ? H / 32 : 1;
#pragma unroll
    for (int k = 0; k < kKeep; ++k) red[lane * kKeep + k] = p[k];
  } else {
    constexpr int kStride = H >= 32 ? 1 : 32 / H;
    if (lane % kStride == 0) red[lane / kStride] = p[0];
  }
}

// Columns are reduced in groups of at most 64 so that R = 128 fits in registers.
template <int R>
struct QrHalves {
  static constexpr int kH = R > 64 ? 64 : R;
  static constexpr int kN = R / kH;
  static constexpr int kC32 = (R + 31) / 32;       // 32-column groups handled by warp 0
};

// a[j] for a runtime j without indexing the register array dynamically.
template <int R>
__device__ __forceinline__ float pick(const float (&row)[R], int j) {
  float x = 0.f;
#pragma unroll
  for (int c = 0; c < R; ++c)
    if (c == j) x = row[c];
  return x;
}

// Householder factorisation of the block held in registers (row i = rho*256 + tid).
template <int R>
__device__ void factor_block(float (&a)[QrShape<R>::kRPT][R], QrSmem<R>& sm) {
  constexpr int RPT = QrShape<R>::kRPT;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  using Hv = QrHalves<R>;
  for (int j = 0; j < R; ++j) {
    const int buf = j & 1;
#pragma unroll
    for (int hh = 0; hh < Hv::kN; ++hh) {
      float p[Hv::kH];
#pragma unroll
      for (int c = 0; c < Hv::kH; ++c) p[c] = 0.f;
#pragma unroll
      for (int rho = 0; rho < RPT; ++rho) {
        const int i = rho * kQrThreads + tid;
        if (i > j) {
          const float x = pick<R>(a[rho], j);
#pragma unroll
          for (int c = 0; c < Hv::kH; ++c)
            if (hh * Hv::kH + c >= j) p[c] = fmaf(x, a[rho][hh * Hv::kH + c], p[c]);
        }
      }
      block_partials<Hv::kH>(p, &sm.red[buf][0][0], R, hh * Hv::kH);
    }
    if (tid == j) {
#pragma unroll
      for (int c = 0; c < R; ++c) sm.rowj[buf][c] = a[0][c];
    }
    __syncthreads();
    if (warp == 0) {
      float sk[Hv::kC32];
#pragma unroll
      for (int k = 0; k < Hv::kC32; ++k) {
        const int c = lane + 32 * k;
        sk[k] = 0.f;
        if (c < R) {
#pragma unroll
          for (int w = 0; w < kQrWarps; ++w) sk[k] += sm.red[buf][w][c];
        }
      }
      float sel = 0.f;
#pragma unroll
      for (int k = 0; k < Hv::kC32; ++k)
        if (k == (j >> 5)) sel = sk[k];
      const float s_j = __shfl_sync(0xffffffffu, sel, j & 31);
      const float alpha = sm.rowj[buf][j];
      float tau = 0.f, beta = alpha, scale = 0.f;
      if (s_j != 0.f) {
        beta = -copysignf(sqrtf(fmaf(alpha, alpha, s_j)), alpha);
        tau = (beta - alpha) / beta;
        scale = 1.0f / (alpha - beta);
      }
#pragma unroll
      for (int k = 0; k < Hv::kC32; ++k) {
        const int c = lane + 32 * k;
        if (c < R && c > j) sm.wbuf[buf][c] = fmaf(scale, sk[k], sm.rowj[buf][c]);
      }
      if (lane == 0) {
        sm.scal[buf][0] = tau;
        sm.scal[buf][1] = scale;
        sm.diag[j] = beta;
        sm.tau[j] = tau;
      }
    }
    __syncthreads();
    const float tau = sm.scal[buf][0], scale = sm.scal[buf][1];
#pragma unroll
    for (int rho = 0; rho < RPT; ++rho) {
      const int i = rho * kQrThreads + tid;
      if (i > j) {
        const float v = pick<R>(a[rho], j) * scale;
        const float tv = -tau * v;
#pragma unroll
        for (int c = 0; c < R; ++c) {
          if (c > j) a[rho][c] = fmaf(tv, sm.wbuf[buf][c], a[rho][c]);
          if (c == j) a[rho][c] = v;
        }
      } else if (i == j) {
        const float beta = sm.diag[j];
#pragma unroll
        for (int c = 0; c < R; ++c) {
          if (c > j) a[rho][c] = fmaf(-tau, sm.wbuf[buf][c], a[rho][c]);
          if (c == j) a[rho][c] = beta;
        }
      }
    }
  }
}

// Y <- H_0 H_1 ... H_(R-1) Y with the reflectors in refl (padded stride kLd).
template <int R>
__device__ void apply_reflectors_backward(float (&a)[QrShape<R>::kRPT][R], const float* refl,
                                          QrSmem<R>& sm) {
  constexpr int RPT = QrShape<R>::kRPT;
  constexpr int LD = QrShape<R>::kLd;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  using Hv = QrHalves<R>;
  for (int j = R - 1; j >= 0; --j) {
    const int buf = j & 1;
#pragma unroll
    for (int hh = 0; hh < Hv::kN; ++hh) {
      float p[Hv::kH];
#pragma unroll
      for (int c = 0; c < Hv::kH; ++c) p[c] = 0.f;
#pragma unroll
      for (int rho = 0; rho < RPT; ++rho) {
        const int i = rho * kQrThreads + tid;
        if (i >= j) {
          const float v = (i == j) ? 1.0f : refl[i * LD + j];
#pragma unroll
          for (int c = 0; c < Hv::kH; ++c) p[c] = fmaf(v, a[rho][hh * Hv::kH + c], p[c]);
        }
      }
      block_partials<Hv::kH>(p, &sm.red[buf][0][0], R, hh * Hv::kH);
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
      for (int h = 0; h < (R + 31) / 32; ++h) {
        const int c = lane + 32 * h;
        if (c < R) {
          float s = 0.f;
#pragma unroll
          for (int w = 0; w < kQrWarps; ++w) s += sm.red[buf][w][c];
          sm.wbuf[buf][c] = s;
        }
      }
    }
    __syncthreads();
    const float tau = sm.tau[j];
#pragma unroll
    for (int rho = 0; rho < RPT; ++rho) {
      const int i = rho * kQrThreads + tid;
      if (i >= j) {
        const float v = (i == j) ? 1.0f : refl[i * LD + j];
        const float tv = -tau * v;
#pragma unroll
        for (int c = 0; c < R; ++c) a[rho][c] = fmaf(tv, sm.wbuf[buf][c], a[rho][c]);
      }
    }
  }
}

template <int R>
__device__ __forceinline__ void store_rows(const float (&a)[QrShape<R>::kRPT][R], float* dst,
                                           int n_real) {
  constexpr int RPT = QrShape<R>::kRPT;
#pragma unroll
  for (int rho = 0; rho < RPT; ++rho) {
    const int i = rho * kQrThreads + threadIdx.x;
    if (i < n_real) {
      float4* d4 = reinterpret_cast<float4*>(dst + (int64_t)i * R);
#pragma unroll
      for (int c4 = 0; c4 < R / 4; ++c4)
        d4[c4] = make_float4(a[rho][4 * c4], a[rho][4 * c4 + 1], a[rho][4 * c4 + 2],
                             a[rho][4 * c4 + 3]);
    }
  }
}

template <int R>
__device__ __forceinline__ void regs_to_refl(const float (&a)[QrShape<R>::kRPT][R], float* refl) {
  constexpr int RPT = QrShape<R>::kRPT;
  constexpr int LD = QrShape<R>::kLd;
#pragma unroll
  for (int rho = 0; rho < RPT; ++rho) {
    const int i = rho * kQrThreads + threadIdx.x;
#pragma unroll
    for (int c = 0; c < R; ++c) refl[i * LD + c] = a[rho][c];
  }
}

template <int R>
__global__ void __launch_bounds__(kQrThreads)
qr_up_kernel(const QrBlock* __restrict__ blocks, uint64_t seed, uint32_t refresh_idx) {
  constexpr int RPT = QrShape<R>::kRPT;
  extern __shared__ float4 qr_smem4[];
  QrSmem<R>& sm = *reinterpret_cast<QrSmem<R>*>(qr_smem4);
  float* refl = reinterpret_cast<float*>(qr_smem4) + (sizeof(QrSmem<R>) + 15) / 16 * 4;
  const QrBlock blk = blocks[blockIdx.x];
  const int tid = threadIdx.x;

  float a[RPT][R];
#pragma unroll
  for (int rho = 0; rho < RPT; ++rho) {
    const int i = rho * kQrThreads + tid;
    if (i < blk.n_real) {
      if (blk.flags & kQrLevel0) {
        // element e = (row0 + i) * R + c of the panel uses counter e / 4, lane e % 4
        const uint32_t c0 = (uint32_t)(((blk.row0 + i) * R) >> 2);
#pragma unroll
        for (int c4 = 0; c4 < R / 4; ++c4) {
          const float4 z = normal4(seed, c0 + c4, blk.gidx, refresh_idx, query_word(blk.tag, 0));
          a[rho][4 * c4] = z.x; a[rho][4 * c4 + 1] = z.y;
          a[rho][4 * c4 + 2] = z.z; a[rho][4 * c4 + 3] = z.w;
        }
      } else {
        const float4* s4 = reinterpret_cast<const float4*>(blk.rows + (int64_t)i * R);
#pragma unroll
        for (int c4 = 0; c4 < R / 4; ++c4) {
          const float4 z = s4[c4];
          a[rho][4 * c4] = z.x; a[rho][4 * c4 + 1] = z.y;
          a[rho][4 * c4 + 2] = z.z; a[rho][4 * c4 + 3] = z.w;
        }
      }
    } else {
#pragma unroll
      for (int c = 0; c < R; ++c) a[rho][c] = 0.f;
    }
  }

  factor_block<R>(a, sm);

  if (blk.flags & kQrTop) {
    regs_to_refl<R>(a, refl);
    __syncthreads();
    // Q = H_0 ... H_(R-1) [diag(sgn R_cc); 0]  (Eq. (11), sgn(0) = +1)
#pragma unroll
    for (int rho = 0; rho < RPT; ++rho) {
      const int i = rho * kQrThreads + tid;
#pragma unroll
      for (int c = 0; c < R; ++c) a[rho][c] = (i == c) ? (sm.diag[c] < 0.f ? -1.f : 1.f) : 0.f;
    }
    apply_reflectors_backward<R>(a, refl, sm);
    store_rows<R>(a, blk.rows, blk.n_real);
  } else {
    store_rows<R>(a, blk.rows, blk.n_real);
    if (tid < R) {
      // R factor row `tid` (upper triangle of the block's first R rows)
      float4* d4 = reinterpret_cast<float4*>(blk.r_out + tid * R);
#pragma unroll
      for (int c4 = 0; c4 < R / 4; ++c4) {
        float v[4];
#pragma unroll
        for (int l = 0; l < 4; ++l) v[l] = (4 * c4 + l >= tid) ? a[0][4 * c4 + l] : 0.f;
        d4[c4] = make_float4(v[0], v[1], v[2], v[3]);
      }
      blk.tau[tid] = sm.tau[tid];
    }
  }
}

template <int R>
__global__ void __launch_bounds__(kQrThreads) qr_down_kernel(const QrBlock* __restrict__ blocks) {
  constexpr int RPT = QrShape<R>::kRPT;
  constexpr int LD = QrShape<R>::kLd;
  extern __shared__ float4 qr_smem4[];
  QrSmem<R>& sm = *reinterpret_cast<QrSmem<R>*>(qr_smem4);
  float* refl = reinterpret_cast<float*>(qr_smem4) + (sizeof(QrSmem<R>) + 15) / 16 * 4;
  const QrBlock blk = blocks[blockIdx.x];
  const int tid = threadIdx.x;

  float a[RPT][R];
#pragma unroll
  for (int rho = 0; rho < RPT; ++rho) {
    const int i = rho * kQrThreads + tid;
    if (i < blk.n_real) {
      const float4* s4 = reinterpret_cast<const float4*>(blk.rows + (int64_t)i * R);
#pragma unroll
      for (int c4 = 0; c4 < R / 4; ++c4) {
        const float4 z = s4[c4];
        refl[i * LD + 4 * c4] = z.x; refl[i * LD + 4 * c4 + 1] = z.y;
        refl[i * LD + 4 * c4 + 2] = z.z; refl[i * LD + 4 * c4 + 3] = z.w;
      }
    } else {
#pragma unroll
      for (int c = 0; c < R; ++c) refl[i * LD + c] = 0.f;
    }
    // Y = [S; 0]
#pragma unroll
    for (int c = 0; c < R; ++c) a[rho][c] = (i < R) ? blk.s_in[i * R + c] : 0.f;
  }
  if (tid < R) sm.tau[tid] = blk.tau[tid];
  __syncthreads();
  apply_reflectors_backward<R>(a, refl, sm);
  store_rows<R>(a, blk.rows, blk.n_real);
}

template <int R>
size_t qr_smem_bytes() {
  return (sizeof(QrSmem<R>) + 15) / 16 * 16 +
         sizeof(float) * (size_t)QrShape<R>::kB * QrShape<R>::kLd;
}

template <int R>
cudaError_t launch_up_r(const QrBlock* d_blocks, int32_t n_blocks, uint64_t seed, uint32_t j,
                        cudaStream_t s) {
  const size_t smem = qr_smem_bytes<R>();
  cudaError_t e = cudaFuncSetAttribute(qr_up_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  qr_up_kernel<R><<<n_blocks, kQrThreads, smem, s>>>(d_blocks, seed, j);
  return cudaGetLastError();
}

template <int R>
cudaError_t launch_down_r(const QrBlock* d_blocks, int32_t n_blocks, cudaStream_t s) {
  const size_t smem = qr_smem_bytes<R>();
  cudaError_t e = cudaFuncSetAttribute(qr_down_kernel<R>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  qr_down_kernel<R><<<n_blocks, kQrThreads, smem, s>>>(d_blocks);
  return cudaGetLastError();
}

__global__ void zero_moments_kernel(const MatDesc* __restrict__ mats, int r) {
  const MatDesc md = mats[blockIdx.x];
  for (int e = threadIdx.x; e < r * r; e += blockDim.x) {
    md.M[e] = 0.f;
    md.Vm[e] = 0.f;
  }
}

}  // namespace

int32_t qr_block_rows(int32_t r) {
  switch (r) {
    case 4: return QrShape<4>::kB;
    case 8: return QrShape<8>::kB;
    case 16: return QrShape<16>::kB;
    case 32: return QrShape<32>::kB;
    case 64: return QrShape<64>::kB;
    case 128: return QrShape<128>::kB;
    default: return 0;
  }
}

cudaError_t launch_qr_up(const QrBlock* d_blocks, int32_t n_blocks, int32_t r, uint64_t seed,
                         uint32_t refresh_idx, uint32_t* /*d_status*/, cudaStream_t s) {
  if (n_blocks <= 0) return cudaSuccess;
  switch (r) {
    case 4: return launch_up_r<4>(d_blocks, n_blocks, seed, refresh_idx, s);
    case 8: return launch_up_r<8>(d_blocks, n_blocks, seed, refresh_idx, s);
    case 16: return launch_up_r<16>(d_blocks, n_blocks, seed, refresh_idx, s);
    case 32: return launch_up_r<32>(d_blocks, n_blocks, seed, refresh_idx, s);
    case 64: return launch_up_r<64>(d_blocks, n_blocks, seed, refresh_idx, s);
    case 128: return launch_up_r<128>(d_blocks, n_blocks, seed, refresh_idx, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_qr_down(const QrBlock* d_blocks, int32_t n_blocks, int32_t r,
                           uint32_t* /*d_status*/, cudaStream_t s) {
  if (n_blocks <= 0) return cudaSuccess;
  switch (r) {
    case 4: return launch_down_r<4>(d_blocks, n_blocks, s);
    case 8: return launch_down_r<8>(d_blocks, n_blocks, s);
    case 16: return launch_down_r<16>(d_blocks, n_blocks, s);
    case 32: return launch_down_r<32>(d_blocks, n_blocks, s);
    case 64: return launch_down_r<64>(d_blocks, n_blocks, s);
    case 128: return launch_down_r<128>(d_blocks, n_blocks, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_zero_moments(const MatDesc* d_mats, int32_t n_mats, int32_t r, cudaStream_t s) {
  if (n_mats <= 0) return cudaSuccess;
  zero_moments_kernel<<<n_mats, 256, 0, s>>>(d_mats, r);
  return cudaGetLastError();
}

}  // namespace zo
