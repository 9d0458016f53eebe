// Projection P_i^T = V_i C_i^T on the 5th-generation tensor cores, r >= 16: the
// prologue of every weight pass (Eq. (4) and Eq. (10) need U_i C_i V_i^T; the weight
// pass takes P_i = C_i V_i^T as its second operand).
//
// At r = 128 the projection is an r^2-deep contraction per column of P -- 2 r^2 flops
// per row of V, 37 GFLOP per pass on the LLaMA-7B set -- so it runs as a GEMM on
// tcgen05.mma: D (128 rows of V x r columns) = V_tile . C^T with M = 128, N = K = r.
// Both operands are scaled fp16 pairs like the weight pass's operands (V 2^kUVScaleExp,
// C_i 2^(e_C,i); zo_tc_common.cuh) and the products hi.hi + hi.lo + lo.hi accumulate in
// fp32 in Tensor Memory (relative error ~2^-21 against the summed terms); the epilogue
// rescales D to P_i 2^(e_P,i) and splits it into the fp16 hi/lo rows of P_HL.  V_HL
// ([hi | lo] rows of V) is formed once per refresh, C_HL and e_C,i once per pass.
//
// Roles of the 192 threads of a CTA (one CTA per SM, each over a contiguous range of
// 128-row units, so C_HL is reloaded only when the matrix changes):
//   warp 0, lane 0: TMA producer -- the C_HL tile of a new matrix (r rows), the V_HL
//                   tile of every unit (128 rows) into a ring of 2-4 stages, so the
//                   loads of later units overlap the MMAs and the epilogue.
//   warp 1, lane 0: MMA issuer -- 3 * r/16 tcgen05.mma (M=128, N=r, K=16) per unit into
//                   one of two TMEM accumulators; warp 1 also owns the TMEM allocation.
//   warps 2..5:     epilogue -- warp w owns 32 rows (its TMEM lane group): tcgen05.ld
//                   the fp32 row of D, scale and split it into fp16 hi/lo, write them as 32 x 64
//                   boxes of P_HL into shared memory (128-byte swizzle) and TMA-store
//                   them, 64 columns of D at a time (one hi and one lo box staged).
//                   For the perturbed-linear route (kPK) it writes instead the
//                   K-major bf16 pair [P_hi ; P_lo] of P (P_K): the exact fp32 P of D (a
//                   power-of-two rescale) split into bf16 hi = bf16(P), lo = bf16(P - hi),
//                   row k of P_K taking column j from lane j (64 contiguous bytes a warp).
// Every mbarrier wait is bounded; on expiry the kernel records kDevTimeout in the
// status word, lets the other roles stop, drains its copies and frees TMEM.
#include <cuda.h>

#include "zo_kernels.h"
#include "zo_sm100.cuh"
#include "zo_tc_common.cuh"

namespace zo {
namespace {

using namespace sm100;
using namespace tc;

constexpr int kProjThreads = 192;

// 32 lanes x 16 consecutive 32-bit columns of Tensor Memory (the R = 16 accumulator).
__device__ __forceinline__ void tmem_ld_32x32b_x16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15])
      : "r"(taddr));
}

template <int R>
struct ProjCfg {
  static_assert(R == 16 || R == 32 || R == 64 || R == 128,
                "the tensor-core projection covers r = 16 ... 128");
  static constexpr int kHLW = hl_width(R);                 // bf16 per operand row (2R, or
                                                           // 64 with zeros past 2R at R = 16)
  static constexpr int kPanels = kHLW / 64;                // 128-byte panels per row
  static constexpr int kVBytes = kPanels * kPanelBytes;    // V tile: 128 rows
  static constexpr int kCPanelBytes = R * 128;             // C panel: R rows x 128 bytes
  static constexpr int kCBytes = kPanels * kCPanelBytes;
  static constexpr int kOutBoxBytes = 32 * 128;            // 32 rows x 64 bf16
  // each epilogue warp stages one hi and one lo box (R <= 32: one box holds both) and
  // stores them 64 columns of D at a time
  static constexpr int kWarpOutBytes = (R <= 32 ? 1 : 2) * kOutBoxBytes;
  static constexpr int kOutBytes = 4 * kWarpOutBytes;
  static constexpr int kKC = R / 16;                       // K chunks of 16
  static constexpr int kTmemCols = 2 * R;                  // two accumulators
  // V ring: a unit's V tile is loaded while earlier units are multiplied
  static constexpr int kVStages = R == 128 ? 2 : R == 64 ? 3 : 4;
  // R = 128: 2 x 64 + 64 + 32 KB; R = 64: 3 x 32 + 16 + 32 KB; R = 32: 4 x 16 + 4 + 16 KB;
  // R = 16: 4 x 16 + 2 + 16 KB
  static constexpr size_t kSmem =
      (size_t)kVStages * kVBytes + kCBytes + kOutBytes + 1024 + 1024;
};

struct ProjShared {
  uint64_t v_full[4], v_empty[4], c_full, c_empty;
  uint64_t acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int abort_flag;
};

__device__ __forceinline__ void proj_give_up(ProjShared& sh, uint32_t* status) {
  atomicOr(status, (uint32_t)kDevTimeout);
  *reinterpret_cast<volatile int*>(&sh.abort_flag) = 1;
}

// kPK: write P_K at p_k + pk_off[i] (rows of n_i rounded up to 64) from pinv (2^-(e_P,i),
// written by the C split) instead of P_HL.
template <int R, bool kPK>
__global__ void __launch_bounds__(kProjThreads, 1)
project_tc_kernel(const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_c,
                  const __grid_constant__ CUtensorMap tm_p, const TcMat* __restrict__ mats,
                  const int2* __restrict__ units, int n_units, uint32_t* __restrict__ status,
                  long long wait_cycles, __nv_bfloat16* __restrict__ p_k,
                  const int64_t* __restrict__ pk_off, const float* __restrict__ pinv) {
  using Cfg = ProjCfg<R>;
  static_assert(sizeof(ProjShared) <= 1024, "barrier block");
  static_assert(Cfg::kSmem <= 227 * 1024, "shared memory per CTA");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* v_smem = smem;
  uint8_t* c_smem = v_smem + Cfg::kVStages * Cfg::kVBytes;
  uint8_t* o_smem = c_smem + Cfg::kCBytes;
  ProjShared& sh = *reinterpret_cast<ProjShared*>(o_smem + Cfg::kOutBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int u_begin = (int)((int64_t)n_units * blockIdx.x / gridDim.x);
  const int u_end = (int)((int64_t)n_units * (blockIdx.x + 1) / gridDim.x);
  const volatile int* abort = &sh.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::kVStages; ++s) {
      mbar_init(&sh.v_full[s], 1);
      mbar_init(&sh.v_empty[s], 1);
    }
    mbar_init(&sh.c_full, 1);
    mbar_init(&sh.c_empty, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sh.acc_full[s], 1);
      mbar_init(&sh.acc_empty[s], 4);
    }
    sh.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_v);
    prefetch_tmap(&tm_c);
    prefetch_tmap(&tm_p);
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
    int64_t n_v = 0, n_c = 0;                     // tiles issued into the V ring and C slot
    int prev_i = -1;
    bool ok = true;
    for (int u = u_begin; u < u_end; ++u) {
      const int2 un = units[u];
      if (un.x != prev_i) {
        if (!mbar_wait_bounded(&sh.c_empty, (uint32_t)((n_c & 1) ^ 1), abort, wait_cycles)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&sh.c_full, Cfg::kCBytes);
        for (int p = 0; p < Cfg::kPanels; ++p)
          tma_load_2d(c_smem + p * Cfg::kCPanelBytes, &tm_c, 64 * p, un.x * R, &sh.c_full);
        ++n_c;
        prev_i = un.x;
      }
      const int vs = (int)(n_v % Cfg::kVStages);
      if (!mbar_wait_bounded(&sh.v_empty[vs], (uint32_t)(((n_v / Cfg::kVStages) & 1) ^ 1), abort,
                             wait_cycles)) {
        ok = false;
        break;
      }
      mbar_arrive_expect_tx(&sh.v_full[vs], Cfg::kVBytes);
      for (int p = 0; p < Cfg::kPanels; ++p)
        tma_load_2d(v_smem + vs * Cfg::kVBytes + p * kPanelBytes, &tm_v, 64 * p,
                    mats[un.x].p_row0 + un.y, &sh.v_full[vs]);
      ++n_v;
    }
    if (!ok) proj_give_up(sh, status);
    // drain: the last copy issued into each slot has landed before the CTA exits
    if (n_c > 0) mbar_wait_bounded(&sh.c_full, (uint32_t)((n_c - 1) & 1), nullptr, wait_cycles);
    for (int vs = 0; vs < Cfg::kVStages; ++vs) {
      const int64_t k = last_in_slot(n_v, vs, Cfg::kVStages);
      if (k >= 0)
        mbar_wait_bounded(&sh.v_full[vs], (uint32_t)((k / Cfg::kVStages) & 1), nullptr, wait_cycles);
    }
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc = idesc_f16_f32(kBM, R);
    int64_t it = 0, n_c = 0;
    int prev_i = -1;
    bool ok = true;
    for (int u = u_begin; u < u_end; ++u, ++it) {
      const int2 un = units[u];
      const bool new_c = un.x != prev_i;
      const bool last_c = u + 1 >= u_end || units[u + 1].x != un.x;
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_empty[acc], (uint32_t)(((it >> 1) & 1) ^ 1), abort,
                             wait_cycles)) { ok = false; break; }
      if (new_c) {
        if (!mbar_wait_bounded(&sh.c_full, (uint32_t)(n_c & 1), abort, wait_cycles)) {
          ok = false;
          break;
        }
        ++n_c;
        prev_i = un.x;
      }
      const int vs = (int)(it % Cfg::kVStages);
      if (!mbar_wait_bounded(&sh.v_full[vs], (uint32_t)((it / Cfg::kVStages) & 1), abort,
                             wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(acc * R);
      const uint32_t a_base = smem_u32(v_smem + vs * Cfg::kVBytes), b_base = smem_u32(c_smem);
      // hi.lo and lo.hi first, hi.hi last (see zo_wpass_tc.cu)
#pragma unroll
      for (int pass = 0; pass < 3; ++pass) {
#pragma unroll
        for (int kk = 0; kk < Cfg::kKC; ++kk) {
          // hi chunk kk at element 16 kk of an operand row, lo chunk at R + 16 kk
          const int e_a = (pass == 1 ? R : 0) + 16 * kk, e_b = (pass == 0 ? R : 0) + 16 * kk;
          const uint64_t a_d = sdesc_k_sw128(a_base + (e_a / 64) * kPanelBytes + (e_a % 64) * 2);
          const uint64_t b_d =
              sdesc_k_sw128(b_base + (e_b / 64) * Cfg::kCPanelBytes + (e_b % 64) * 2);
          mma_f16(d, a_d, b_d, idesc, (pass | kk) != 0 ? 1u : 0u);
        }
      }
      mma_commit(&sh.v_empty[vs]);
      if (last_c) mma_commit(&sh.c_empty);
      mma_commit(&sh.acc_full[acc]);
    }
    if (!ok) proj_give_up(sh, status);
    if (it > 0) {
      // every MMA issued by this thread has completed before TMEM is released
      const int64_t last = it - 1;
      mbar_wait_bounded(&sh.acc_full[last & 1], (uint32_t)((last >> 1) & 1), nullptr, wait_cycles);
    }
  } else if (warp >= 2 && warp <= 5) {
    // ------------------------------------------------------------ epilogue
    const int g = warp & 3;                      // TMEM lane group == rows 32 g .. + 31
    const uint32_t lane_base = (uint32_t)(g * 32) << 16;
    uint8_t* obox = o_smem + g * Cfg::kWarpOutBytes;   // this warp's boxes
    // D = 2^(kUVScaleExp + e_C) P^T; P_HL holds P 2^(e_C + p_scale_offset(R))
    const float p_scale = exp2i(p_scale_offset(R) - kUVScaleExp);
    int64_t it = 0;
    bool ok = true;
    for (int u = u_begin; u < u_end; ++u, ++it) {
      const int2 un = units[u];
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_full[acc], (uint32_t)((it >> 1) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int y = mats[un.x].p_row0 + un.y + 32 * g;
      // the previous unit's stores have finished reading this warp's boxes
      if (lane == 0) bulk_wait_read_all();
      __syncwarp();
      if constexpr (kPK) {
        // D 2^-(kUVScaleExp + e_C,i) = P exactly (both factors powers of two); kC columns
        // of D at a time
        constexpr int kC = R < 32 ? R : 32;
        const float unscale = p_scale * pinv[un.x];
        const int64_t n = mats[un.x].n;
        const int64_t ld = (n + 63) / 64 * 64;
        const int64_t j = un.y + 32 * g + lane;
        __nv_bfloat16* dst = p_k + pk_off[un.x] + j;
#pragma unroll 1
        for (int c = 0; c < R / kC; ++c) {
          uint32_t v[kC];
          if constexpr (kC == 32)
            tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * R + 32 * c), v);
          else
            tmem_ld_32x32b_x16(tmem + lane_base + (uint32_t)(acc * R), v);
          tmem_ld_wait();
          if (j < n) {
#pragma unroll
            for (int k = 0; k < kC; ++k) {
              const float x = __uint_as_float(v[k]) * unscale;
              const __nv_bfloat16 hi = __float2bfloat16_rn(x);
              dst[(kC * c + k) * ld] = hi;
              dst[(R + kC * c + k) * ld] = __float2bfloat16_rn(x - __bfloat162float(hi));
            }
          }
        }
      } else if constexpr (R <= 32) {
        // one 64-wide box per row: hi at columns 8 j, lo at R + 8 j, zeros past 2R
        uint32_t v[R];
        if constexpr (R == 32)
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * R), v);
        else
          tmem_ld_32x32b_x16(tmem + lane_base + (uint32_t)(acc * R), v);
        tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < R / 8; ++j) {
          float x[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) x[e] = __uint_as_float(v[8 * j + e]);
          uint4 hi, lo;
          split8_f16(x, p_scale, hi, lo);
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
          tma_store_2d(&tm_p, 0, y, obox);
          bulk_commit();
        }
      } else {
#pragma unroll
        for (int h = 0; h < R / 64; ++h) {       // 64 columns of D: one hi and one lo box
          if (h > 0) {
            // the stores of the previous 64 columns have read the two boxes
            if (lane == 0) bulk_wait_read_all();
            __syncwarp();
          }
          uint32_t v[2][32];
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * R + 64 * h), v[0]);
          tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * R + 64 * h + 32), v[1]);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 8; ++j) {          // columns 64 h + 8 j .. + 7
            float x[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) x[e] = __uint_as_float(v[j >> 2][(j & 3) * 8 + e]);
            uint4 hi, lo;
            split8_f16(x, p_scale, hi, lo);
            const int sw = (j ^ (lane & 7)) << 4;
            *reinterpret_cast<uint4*>(obox + lane * 128 + sw) = hi;
            *reinterpret_cast<uint4*>(obox + Cfg::kOutBoxBytes + lane * 128 + sw) = lo;
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            // hi to P_HL columns 64 h .. + 63, lo to R + 64 h .. + 63
            tma_store_2d(&tm_p, 64 * h, y, obox);
            tma_store_2d(&tm_p, R + 64 * h, y, obox + Cfg::kOutBoxBytes);
            bulk_commit();
          }
          __syncwarp();
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.acc_empty[acc]);
      __syncwarp();
    }
    if (!ok && lane == 0) proj_give_up(sh, status);
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

// Rows [hi | lo] of the scaled fp16 pair of V (units = (matrix, first row) x 128 rows, into
// V_HL at p_row0; scale 2^kUVScaleExp) or of C (one CTA per matrix, r rows into C_HL at
// matrix * r; scale 2^(e_C,i) from the coefficient kernel's max |C_i| = amax[i], with
// pinv[i] = 2^-(e_P,i) written for the weight pass).  Each thread splits one row;
// the rows are staged in shared memory with the 16-byte chunk index XOR (row & 7) and
// written with coalesced 16-byte stores.
template <int R, bool kC>
__global__ void __launch_bounds__(128)
split_rows_kernel(const MatDesc* __restrict__ mats, const TcMat* __restrict__ tcm,
                  const int2* __restrict__ units, const float* __restrict__ amax_in,
                  uint16_t* __restrict__ dst, float* __restrict__ pinv) {
  constexpr int kVecPerRow = 2 * R * 2 / 16;     // 16-byte chunks of [hi | lo]
  constexpr int kSw = kVecPerRow >= 8 ? 7 : kVecPerRow - 1;   // chunk swizzle within a row
  constexpr int kStride = hl_width(R) / 8;       // chunks per row of V_HL / C_HL
  extern __shared__ uint4 Os[];                  // 128 x kVecPerRow
  const int tid = threadIdx.x;
  int i, rows;
  int64_t row0, dst_row0;
  const float* src;
  if constexpr (kC) {
    i = blockIdx.x;
    row0 = 0;
    rows = R;
    src = mats[i].C;
    dst_row0 = (int64_t)i * R;
  } else {
    const int2 u = units[blockIdx.x];
    i = u.x;
    row0 = u.y;
    rows = (int)(mats[i].n - row0 < 128 ? mats[i].n - row0 : 128);
    src = mats[i].V;
    dst_row0 = (int64_t)tcm[i].p_row0 + row0;
  }
  float scale = exp2i(kUVScaleExp);
  if constexpr (kC) {
    const int e_c = coeff_scale_exp(amax_in[i]);
    scale = exp2i(e_c);
    if (tid == 0) pinv[i] = exp2i(-(e_c + p_scale_offset(R)));
  }
  if (tid < rows) {
    const float4* s4 = reinterpret_cast<const float4*>(src + (row0 + tid) * R);
    uint4* orow = Os + tid * kVecPerRow;
#pragma unroll
    for (int g = 0; g < R / 8; ++g) {
      const float4 a = s4[2 * g], b = s4[2 * g + 1];
      const float x[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
      uint4 hi, lo;
      split8_f16(x, scale, hi, lo);
      orow[g ^ (tid & kSw)] = hi;
      orow[(R / 8 + g) ^ (tid & kSw)] = lo;
    }
  }
  __syncthreads();
  // rows are hl_width(R) wide; at R = 16 the chunks past [hi | lo] keep their zeros
  uint4* d4 = reinterpret_cast<uint4*>(dst + dst_row0 * hl_width(R));
  for (int e = tid; e < rows * kVecPerRow; e += 128) {
    const int row = e / kVecPerRow, c = e % kVecPerRow;
    d4[row * kStride + c] = Os[row * kVecPerRow + (c ^ (row & kSw))];
  }
}

template <int R, bool kPK>
cudaError_t launch_project_tc_r(const CUtensorMap& tm_v, const CUtensorMap& tm_c,
                                const CUtensorMap& tm_p, const TcMat* d_tc, const int2* d_units,
                                int32_t n_units, int32_t grid, uint32_t* d_status, cudaStream_t s,
                                __nv_bfloat16* p_k = nullptr, const int64_t* pk_off = nullptr,
                                const float* pinv = nullptr) {
  const size_t smem = ProjCfg<R>::kSmem;
  cudaError_t e = cudaFuncSetAttribute(project_tc_kernel<R, kPK>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  project_tc_kernel<R, kPK><<<grid, kProjThreads, smem, s>>>(tm_v, tm_c, tm_p, d_tc, d_units,
                                                             n_units, d_status, kWaitCycles, p_k,
                                                             pk_off, pinv);
  return cudaGetLastError();
}

template <int R, bool kC>
cudaError_t launch_split_rows_r(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                                int32_t n_blocks, const float* amax, uint16_t* dst, float* pinv,
                                cudaStream_t s) {
  constexpr size_t smem = 128 * (size_t)(2 * R * 2);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(split_rows_kernel<R, kC>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  split_rows_kernel<R, kC><<<n_blocks, 128, smem, s>>>(d_mats, d_tc, d_units, amax, dst, pinv);
  return cudaGetLastError();
}

}  // namespace

bool project_tc_supported(int32_t r) { return r == 16 || r == 32 || r == 64 || r == 128; }

cudaError_t launch_split_v(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                           int32_t n_units, int32_t r, uint16_t* v_hl, cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 16: return launch_split_rows_r<16, false>(d_mats, d_tc, d_units, n_units, nullptr, v_hl, nullptr, s);
    case 32: return launch_split_rows_r<32, false>(d_mats, d_tc, d_units, n_units, nullptr, v_hl, nullptr, s);
    case 64: return launch_split_rows_r<64, false>(d_mats, d_tc, d_units, n_units, nullptr, v_hl, nullptr, s);
    case 128: return launch_split_rows_r<128, false>(d_mats, d_tc, d_units, n_units, nullptr, v_hl, nullptr, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_split_c(const MatDesc* d_mats, int32_t n_mats, int32_t r, const float* amax,
                           uint16_t* c_hl, float* pinv, cudaStream_t s) {
  if (n_mats <= 0) return cudaSuccess;
  switch (r) {
    case 16: return launch_split_rows_r<16, true>(d_mats, nullptr, nullptr, n_mats, amax, c_hl, pinv, s);
    case 32: return launch_split_rows_r<32, true>(d_mats, nullptr, nullptr, n_mats, amax, c_hl, pinv, s);
    case 64: return launch_split_rows_r<64, true>(d_mats, nullptr, nullptr, n_mats, amax, c_hl, pinv, s);
    case 128: return launch_split_rows_r<128, true>(d_mats, nullptr, nullptr, n_mats, amax, c_hl, pinv, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_project_tc(const CUtensorMap& tm_v, const CUtensorMap& tm_c,
                              const CUtensorMap& tm_p, const TcMat* d_tc, const int2* d_units,
                              int32_t n_units, int32_t grid, int32_t r, uint32_t* d_status,
                              cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 16: return launch_project_tc_r<16, false>(tm_v, tm_c, tm_p, d_tc, d_units, n_units, grid, d_status, s);
    case 32: return launch_project_tc_r<32, false>(tm_v, tm_c, tm_p, d_tc, d_units, n_units, grid, d_status, s);
    case 64: return launch_project_tc_r<64, false>(tm_v, tm_c, tm_p, d_tc, d_units, n_units, grid, d_status, s);
    case 128: return launch_project_tc_r<128, false>(tm_v, tm_c, tm_p, d_tc, d_units, n_units, grid, d_status, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_project_tc_pk(const CUtensorMap& tm_v, const CUtensorMap& tm_c,
                                 const TcMat* d_tc, const int2* d_units, int32_t n_units,
                                 int32_t grid, int32_t r, const float* pinv, const int64_t* pk_off,
                                 __nv_bfloat16* p_k, uint32_t* d_status, cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 16: return launch_project_tc_r<16, true>(tm_v, tm_c, tm_v, d_tc, d_units, n_units, grid, d_status, s, p_k, pk_off, pinv);
    case 32: return launch_project_tc_r<32, true>(tm_v, tm_c, tm_v, d_tc, d_units, n_units, grid, d_status, s, p_k, pk_off, pinv);
    case 64: return launch_project_tc_r<64, true>(tm_v, tm_c, tm_v, d_tc, d_units, n_units, grid, d_status, s, p_k, pk_off, pinv);
    case 128: return launch_project_tc_r<128, true>(tm_v, tm_c, tm_v, d_tc, d_units, n_units, grid, d_status, s, p_k, pk_off, pinv);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
