// One linear layer of the loss evaluation at the perturbed weights, without a weight pass:
//   Y = X (W_i + U_i C_i V_i^T)^T = X W_i^T + S U_i^T,  S = X P_i^T,  P_i = C_i V_i^T,
// the forward of Alg. 3 at W' = W + eps U Z V^T (Eq. (4) form) with W left as it is.
// X (T x n) and Y (T x m) are bf16 activations of the caller; W_i is the context's bf16
// matrix (nn.Linear layout, m x n).
//
// Two tcgen05 GEMMs with one kernel template (both operands K-major in shared memory,
// 128-byte swizzle, loaded by TMA; fp32 accumulators in TMEM; persistent CTAs over
// output tiles of 128 rows of X):
//   kModeS  S = X P^T with B = [P_hi ; P_lo] (2r rows, K-major, from P_K): N = 2r; the
//           epilogue sums the two halves, S = D[:, :r] + D[:, r:], and writes S as bf16
//           hi/lo rows [S_hi | S_lo | 0] of 64 elements (S_HL), the layout of the U
//           operand.
//   kModeY  Y = X W^T over K = n (single bf16 products, both operands exact in bf16)
//           followed by one more K step from S_HL and the U operand, with the weight
//           pass's three products S_hi U_hi + S_hi U_lo + S_lo U_hi (relative error
//           ~2^-16 of the rank-r term); N = 256 columns of Y per tile; the epilogue
//           rounds to bf16 and TMA-stores Y.
// P_K is P_HL (the projection's rows [P_hi(j, :) | P_lo(j, :)], j < n) transposed by
// transpose_p_kernel.  Ragged edges: TMA zero-fills loads past T, n and m and clips
// stores.
//
// Roles of the 192 threads of a CTA:
//   warp 0, lane 0: TMA producer -- per K step one X box (64 x 128 rows) and the B rows
//                   (W: N/32 boxes of 64 x 32; P_K: one box of 64 x 2r), into a ring
//                   of kStages slots; kModeY ends each tile with the extension step.
//   warp 1, lane 0: MMA issuer (4 x K = 16 per K step, 3r/16 for the extension) into
//                   one of two TMEM accumulators; warp 1 also owns TMEM.
//   warps 2..5:     epilogue -- warp w owns rows 32 (w % 4) .. + 31 of the tile (its
//                   TMEM lane group) and stores them 64 columns at a time through two
//                   staged 32 x 64 boxes.
// Every mbarrier wait is bounded; on expiry the kernel records kDevTimeout in the status
// word, lets the other roles stop, drains its copies and frees TMEM.
#include <cuda.h>

#include "zo_kernels.h"
#include "zo_sm100.cuh"
#include "zo_tc_common.cuh"

namespace zo {
namespace {

using namespace sm100;
using namespace tc;

constexpr int kLinThreads = 192;
constexpr int kModeS = 0;
constexpr int kModeY = 1;

template <int kMode, int R>
struct LinCfg {
  static_assert(R == 16 || R == 32, "the U operand rows [hi | lo | 0] exist for r <= 32");
  static constexpr int kN = kMode == kModeY ? 256 : 2 * R;          // tile columns
  static constexpr int kStages = 4;
  static constexpr int kABytes = kBM * 128;                          // 128 rows x 64 bf16
  static constexpr int kBBytes = kN * 128;                           // kN rows x 64 bf16
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kBoxBytes = 32 * 128;                         // 32 rows x 64 bf16
  static constexpr int kOutBytes = 4 * 2 * kBoxBytes;                // two boxes per warp
  static constexpr int kTmemCols = kN * 2 <= 32 ? 32 : kN * 2;       // two accumulators
  static constexpr size_t kSmem = (size_t)kStages * kStageBytes + kOutBytes + 1024 + 1024;
  static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
  static_assert(kTmemCols <= 512, "TMEM columns");
};

struct LinShared {
  uint64_t full[4], empty[4];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t drain;      // one commit after the MMA thread's last MMA
  uint32_t tmem_base;
  int abort_flag;
};

__device__ __forceinline__ void lin_give_up(LinShared& sh, uint32_t* status) {
  atomicOr(status, (uint32_t)kDevTimeout);
  *reinterpret_cast<volatile int*>(&sh.abort_flag) = 1;
}

// tm_a: X (box 64 x 128).  kModeS: tm_b = P_K (box 64 x 2r), tm_o = S_HL (box 64 x 32).
// kModeY: w_map = W_i (box 64 x 32), tm_s = S_HL (box 64 x 128), tm_u = U operand (box
// 64 x 128) with this matrix's rows from u_row0, tm_o = Y (box 64 x 32).
template <int kMode, int R>
__global__ void __launch_bounds__(kLinThreads, 1)
linear_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
              const CUtensorMap* __restrict__ w_map, const __grid_constant__ CUtensorMap tm_s,
              const __grid_constant__ CUtensorMap tm_u, const __grid_constant__ CUtensorMap tm_o,
              int rows, int cols, int k_steps, int u_row0, uint32_t* __restrict__ status,
              long long wait_cycles) {
  using Cfg = LinCfg<kMode, R>;
  static_assert(sizeof(LinShared) <= 1024, "barrier block");
  constexpr int kN = Cfg::kN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* st_smem = smem;                                          // stages: [A | B]
  uint8_t* o_smem = st_smem + Cfg::kStages * Cfg::kStageBytes;      // epilogue boxes
  LinShared& sh = *reinterpret_cast<LinShared*>(o_smem + Cfg::kOutBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles_m = (cols + kN - 1) / kN;
  const int n_tiles = ((rows + kBM - 1) / kBM) * tiles_m;
  const int steps = k_steps + (kMode == kModeY ? 1 : 0);           // + the extension
  const volatile int* abort = &sh.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::kStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sh.acc_full[s], 1);
      mbar_init(&sh.acc_empty[s], 4);
    }
    mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_a);
    prefetch_tmap(&tm_o);
    if constexpr (kMode == kModeS) {
      prefetch_tmap(&tm_b);
    } else {
      prefetch_tmap(w_map);
      prefetch_tmap(&tm_s);
      prefetch_tmap(&tm_u);
    }
  }
  if (warp == 1) {
    tmem_alloc(&sh.tmem_base, Cfg::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    int64_t n_st = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x) {
      const int tb = tile / tiles_m, nb = tile % tiles_m;
      for (int k = 0; k < steps; ++k) {
        const int s = (int)(n_st % Cfg::kStages);
        if (!mbar_wait_bounded(&sh.empty[s], (uint32_t)(((n_st / Cfg::kStages) & 1) ^ 1), abort,
                               wait_cycles)) {
          ok = false;
          break;
        }
        uint8_t* a_dst = st_smem + s * Cfg::kStageBytes;
        uint8_t* b_dst = a_dst + Cfg::kABytes;
        mbar_arrive_expect_tx(&sh.full[s], Cfg::kStageBytes);
        if (kMode == kModeY && k == k_steps) {
          // the extension: S_HL rows of the token block, U operand rows of the W block
          tma_load_2d(a_dst, &tm_s, 0, tb * kBM, &sh.full[s]);
          for (int h = 0; h < kN / kBM; ++h)
            tma_load_2d(b_dst + h * kPanelBytes, &tm_u, 0, u_row0 + nb * kN + h * kBM, &sh.full[s]);
        } else {
          tma_load_2d(a_dst, &tm_a, 64 * k, tb * kBM, &sh.full[s]);
          if constexpr (kMode == kModeS) {
            tma_load_2d(b_dst, &tm_b, 64 * k, 0, &sh.full[s]);
          } else {
            for (int h = 0; h < kN / 32; ++h)
              tma_load_2d(b_dst + h * Cfg::kBoxBytes, w_map, 64 * k, nb * kN + 32 * h, &sh.full[s]);
          }
        }
        ++n_st;
      }
    }
    if (!ok) lin_give_up(sh, status);
    for (int s = 0; s < Cfg::kStages; ++s) {
      const int64_t k = last_in_slot(n_st, s, Cfg::kStages);
      if (k >= 0)
        mbar_wait_bounded(&sh.full[s], (uint32_t)((k / Cfg::kStages) & 1), nullptr, wait_cycles);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc = idesc_bf16_f32(kBM, kN);
    int64_t n_st = 0, it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < n_tiles && ok; tile += gridDim.x, ++it) {
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_empty[acc], (uint32_t)(((it >> 1) & 1) ^ 1), abort,
                             wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(acc * kN);
      for (int k = 0; k < steps; ++k) {
        const int s = (int)(n_st % Cfg::kStages);
        if (!mbar_wait_bounded(&sh.full[s], (uint32_t)((n_st / Cfg::kStages) & 1), abort,
                               wait_cycles)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = smem_u32(st_smem + s * Cfg::kStageBytes);
        const uint32_t b_base = a_base + Cfg::kABytes;
        if (kMode == kModeY && k == k_steps) {
          // hi chunk kk at element 16 kk of an operand row, lo chunk at R + 16 kk
#pragma unroll
          for (int kk = 0; kk < R / 16; ++kk) {
            const uint32_t hi = (uint32_t)(16 * kk * 2), lo = (uint32_t)((R + 16 * kk) * 2);
            mma_bf16(d, sdesc_k_sw128(a_base + hi), sdesc_k_sw128(b_base + hi), idesc, 1u);
            mma_bf16(d, sdesc_k_sw128(a_base + hi), sdesc_k_sw128(b_base + lo), idesc, 1u);
            mma_bf16(d, sdesc_k_sw128(a_base + lo), sdesc_k_sw128(b_base + hi), idesc, 1u);
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_bf16(d, sdesc_k_sw128(a_base + 32 * kk), sdesc_k_sw128(b_base + 32 * kk), idesc,
                     (k > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&sh.empty[s]);
        ++n_st;
      }
      if (!ok) break;
      mma_commit(&sh.acc_full[acc]);
    }
    if (!ok) lin_give_up(sh, status);
    if (n_st > 0) {
      // every MMA issued by this thread -- a tile left half-way included -- has completed
      // before TMEM is released
      mma_commit(&sh.drain);
      mbar_wait_bounded(&sh.drain, 0u, nullptr, wait_cycles);
    }
  } else if (warp >= 2 && warp <= 5) {
    // ------------------------------------------------------------ epilogue
    const int g = warp & 3;                      // TMEM lane group == rows 32 g .. + 31
    const uint32_t lane_base = (uint32_t)(g * 32) << 16;
    uint8_t* obox = o_smem + g * 2 * Cfg::kBoxBytes;
    int64_t it = 0, n_box = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++it) {
      const int tb = tile / tiles_m, nb = tile % tiles_m;
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_full[acc], (uint32_t)((it >> 1) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int y = tb * kBM + 32 * g;
      if constexpr (kMode == kModeS) {
        // S = D[:, :R] + D[:, R:2R]; row [S_hi | S_lo | 0] of 64 elements
        uint32_t v[2 * R];
        if constexpr (R == 32) {
          uint32_t a[32], b[32];
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kN), a);
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kN + 32), b);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) { v[e] = a[e]; v[32 + e] = b[e]; }
        } else {
          uint32_t a[32];
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kN), a);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = a[e];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.acc_empty[acc]);
        if (lane == 0) bulk_wait_read_all();    // the previous tile's box has been stored
        __syncwarp();
#pragma unroll
        for (int j = 0; j < R / 8; ++j) {
          float x[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            x[e] = __uint_as_float(v[8 * j + e]) + __uint_as_float(v[R + 8 * j + e]);
          uint4 hi, lo;
          split8(x, hi, lo);
          *reinterpret_cast<uint4*>(obox + lane * 128 + ((j ^ (lane & 7)) << 4)) = hi;
          *reinterpret_cast<uint4*>(obox + lane * 128 + (((R / 8 + j) ^ (lane & 7)) << 4)) = lo;
        }
#pragma unroll
        for (int j = 2 * R / 8; j < 8; ++j)
          *reinterpret_cast<uint4*>(obox + lane * 128 + ((j ^ (lane & 7)) << 4)) =
              make_uint4(0u, 0u, 0u, 0u);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (y < rows) tma_store_2d(&tm_o, 0, y, obox);
          bulk_commit();
        }
        __syncwarp();
      } else {
        // 64 columns of Y at a time, alternating between the warp's two boxes
#pragma unroll 1
        for (int h = 0; h < kN / 64; ++h) {
          uint32_t v[2][32];
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kN + 64 * h), v[0]);
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kN + 64 * h + 32), v[1]);
          tmem_ld_wait();
          if (h == kN / 64 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.acc_empty[acc]);
          }
          uint8_t* box = obox + (int)(n_box & 1) * Cfg::kBoxBytes;
          if (lane == 0) bulk_wait_read_1();     // the store that used this box has read it
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const __nv_bfloat162 b2 =
                  __floats2bfloat162_rn(__uint_as_float(v[j >> 2][(j & 3) * 8 + 2 * e]),
                                        __uint_as_float(v[j >> 2][(j & 3) * 8 + 2 * e + 1]));
              w[e] = *reinterpret_cast<const uint32_t*>(&b2);
            }
            *reinterpret_cast<uint4*>(box + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                make_uint4(w[0], w[1], w[2], w[3]);
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            const int x = nb * kN + 64 * h;
            if (y < rows && x < cols) tma_store_2d(&tm_o, x, y, box);
            bulk_commit();
          }
          __syncwarp();
          ++n_box;
        }
      }
    }
    if (!ok && lane == 0) lin_give_up(sh, status);
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

// P_K[k][j] = P_HL[p_row0 + j][k] for k < 2r (rows [P_hi ; P_lo]), j < n: a 64 x 64 tile
// per CTA through shared memory.
__global__ void __launch_bounds__(256)
transpose_p_kernel(const __nv_bfloat16* __restrict__ p_hl, int64_t p_row0, int hl_width, int n,
                   int r2, __nv_bfloat16* __restrict__ p_k, int64_t ld_k) {
  __shared__ __nv_bfloat16 t[64][66];
  const int j0 = blockIdx.x * 64;
  for (int e = threadIdx.x; e < 64 * 64; e += blockDim.x) {
    const int jj = e / 64, k = e % 64;
    t[jj][k] = (j0 + jj < n && k < r2) ? p_hl[(p_row0 + j0 + jj) * hl_width + k]
                                       : __float2bfloat16_rn(0.f);
  }
  __syncthreads();
  for (int e = threadIdx.x; e < 64 * 64; e += blockDim.x) {
    const int k = e / 64, jj = e % 64;
    if (k < r2 && j0 + jj < n) p_k[(int64_t)k * ld_k + j0 + jj] = t[jj][k];
  }
}

template <int kMode, int R>
cudaError_t launch_linear_r(const CUtensorMap& tm_a, const CUtensorMap& tm_b,
                            const CUtensorMap* w_map, const CUtensorMap& tm_s,
                            const CUtensorMap& tm_u, const CUtensorMap& tm_o, int rows, int cols,
                            int k_steps, int u_row0, int grid, uint32_t* d_status,
                            cudaStream_t s) {
  using Cfg = LinCfg<kMode, R>;
  cudaError_t e = cudaFuncSetAttribute(linear_kernel<kMode, R>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)Cfg::kSmem);
  if (e != cudaSuccess) return e;
  linear_kernel<kMode, R><<<grid, kLinThreads, Cfg::kSmem, s>>>(
      tm_a, tm_b, w_map, tm_s, tm_u, tm_o, rows, cols, k_steps, u_row0, d_status, kWaitCycles);
  return cudaGetLastError();
}

}  // namespace

bool linear_supported(int32_t r) { return r == 16 || r == 32; }

int32_t linear_tiles(int64_t rows, int64_t cols, bool s_gemm, int32_t r) {
  const int64_t n = s_gemm ? 2 * r : 256;
  return (int32_t)(((rows + kBM - 1) / kBM) * ((cols + n - 1) / n));
}

cudaError_t launch_transpose_p(const __nv_bfloat16* p_hl, int64_t p_row0, int32_t hl_width,
                               int64_t n, int32_t r, __nv_bfloat16* p_k, int64_t ld_k,
                               cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  transpose_p_kernel<<<(unsigned)((n + 63) / 64), 256, 0, s>>>(p_hl, p_row0, hl_width, (int)n,
                                                              2 * r, p_k, ld_k);
  return cudaGetLastError();
}

cudaError_t launch_linear_s(const CUtensorMap& tm_x, const CUtensorMap& tm_pk,
                            const CUtensorMap& tm_s_out, int64_t T, int64_t n, int32_t r,
                            int32_t grid, uint32_t* d_status, cudaStream_t s) {
  const int k_steps = (int)((n + 63) / 64);
  switch (r) {
    case 16: return launch_linear_r<kModeS, 16>(tm_x, tm_pk, nullptr, tm_x, tm_x, tm_s_out, (int)T, 32, k_steps, 0, grid, d_status, s);
    case 32: return launch_linear_r<kModeS, 32>(tm_x, tm_pk, nullptr, tm_x, tm_x, tm_s_out, (int)T, 64, k_steps, 0, grid, d_status, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_linear_y(const CUtensorMap& tm_x, const CUtensorMap* d_w_map,
                            const CUtensorMap& tm_s_in, const CUtensorMap& tm_u,
                            const CUtensorMap& tm_y, int64_t T, int64_t m, int64_t n,
                            int32_t u_row0, int32_t r, int32_t grid, uint32_t* d_status,
                            cudaStream_t s) {
  const int k_steps = (int)((n + 63) / 64);
  switch (r) {
    case 16: return launch_linear_r<kModeY, 16>(tm_x, tm_x, d_w_map, tm_s_in, tm_u, tm_y, (int)T, (int)m, k_steps, u_row0, grid, d_status, s);
    case 32: return launch_linear_r<kModeY, 32>(tm_x, tm_x, d_w_map, tm_s_in, tm_u, tm_y, (int)T, (int)m, k_steps, u_row0, grid, d_status, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
