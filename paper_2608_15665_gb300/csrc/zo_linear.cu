// One linear layer of the loss evaluation at the perturbed weights, without a weight pass:
//   Y = X (W_i + U_i C_i V_i^T)^T = X W_i^T + S U_i^T,  S = X P_i^T,  P_i = C_i V_i^T,
// the forward of Alg. 3 at W' = W + eps U Z V^T (Eq. (4) form) with W left as it is.
// X (T x n) and Y (T x m) are bf16 activations of the caller; W_i is the context's bf16
// matrix (nn.Linear layout, m x n).
//
// Two tcgen05 GEMMs with one kernel template (both operands K-major in shared memory,
// 128-byte swizzle, loaded by TMA; fp32 accumulators in TMEM; persistent CTAs over
// output tiles of 128 rows of X):
//   kModeS  partial S = X P^T over a range of K with B = [P_hi ; P_lo] (2r rows, K-major,
//           from P_K): N = 2r, tiles = (128 rows of X) x (K range) so that a few row
//           blocks still fill the SMs; the epilogue sums the two halves, D[:, :r] +
//           D[:, r:], and writes the fp32 partial rows.  S leaves as bf16 hi/lo rows
//           [S_hi | S_lo | 0] of 64 elements (S_HL), the layout of the U operand: with a
//           single K range the epilogue writes S_HL directly; with up to kFusedSplits
//           ranges the warp that finishes a 32-row group last (a counter per group,
//           atomicInc wrapping back to 0) adds the group's partials in K-range order;
//           with more, reduce_s_kernel does (one warp reading 32 x k_split partial rows
//           would take k_split L2 round trips).
//   kModeY  Y = X W^T over K = n (single bf16 products, both operands exact in bf16)
//           followed by one more K step from S_HL and the U operand, with the weight
//           pass's three products S_hi U_hi + S_hi U_lo + S_lo U_hi (relative error
//           ~2^-16 of the rank-r term); N = 256 columns of Y per tile; the epilogue
//           rounds to bf16 and TMA-stores Y.
//   kModeY2 the same over 256 x 256 tiles: two M = 128 halves of X rows share each
//           stage's W rows, so a stage (64 KB) carries twice the MMA work of a kModeY
//           stage (48 KB) -- the operand bytes an SM takes in per flop fall by a third,
//           and the 3-stage ring covers 1.5x the load latency.  Both halves'
//           accumulators fill TMEM (2 x 256 columns), so the epilogue of a tile (eight
//           warps) is not overlapped with the next tile's MMAs.
//   kModeY2N the same over 256 x 224 tiles (halves 256 TMEM columns apart; Y stored 32
//           columns at a time through 64-byte-swizzled boxes): 4096 columns make 19 of
//           them, so 16 or 8 row blocks make exactly two or one wave on 152 SMs.
//           linear_y_tiling picks the tiling with the fewest waves of tile work.
// P_K, the K-major bf16 pair [P_hi ; P_lo] of P, is written by the tensor-core projection
// (zo_project_tc.cu) for every matrix once per loss evaluation (zo_linear_prepare).
// Ragged edges: TMA zero-fills loads past T, n and m; Y's stores are clipped to T rows and
// m columns (m a multiple of 8, so that no 16-byte chunk reaches past Y's columns).
//
// Roles of the threads of a CTA (192; kModeY2 320):
//   warp 0, lane 0: TMA producer -- per K step one X box (64 x 128 rows) per half and
//                   the B rows (W: N/32 boxes of 64 x 32; P_K: one box of 64 x 2r), into
//                   a ring of kStages slots; the Y modes end each tile with the extension
//                   step.
//   warp 1, lane 0: MMA issuer (4 x K = 16 per K step and half, 3r/16 for the extension)
//                   into one of two TMEM accumulators (kModeY2: the single pair of
//                   halves); warp 1 also owns TMEM.
//   warps 2..:      epilogue -- warp w owns rows 32 (w % 4) .. + 31 of a half (its TMEM
//                   lane group; kModeY2 has eight warps, four per half); the Y modes store
//                   them 64 columns at a time through staged 32 x 64 boxes (TMA), kModeS
//                   writes its fp32 partial rows.
// Every mbarrier wait is bounded; on expiry the kernel records kDevTimeout in the status
// word, lets the other roles stop, drains its copies and frees TMEM.
#include <algorithm>

#include <cuda.h>

#include "zo_kernels.h"
#include "zo_linear_common.cuh"
#include "zo_sm100.cuh"
#include "zo_tc_common.cuh"

namespace zo {
namespace {

using namespace sm100;
using namespace tc;
using namespace lin;

constexpr int kFusedSplits = 4;   // most K ranges whose S partials the S kernel sums itself
constexpr int kModeS = 0;
constexpr int kModeY = 1;
constexpr int kModeY2 = 2;
constexpr int kModeY2N = 3;

template <int kMode, int R>
struct LinCfg {
  static_assert(R == 16 || R == 32, "the U operand rows [hi | lo | 0] exist for r <= 32");
  static constexpr bool kY = kMode != kModeS;
  static constexpr bool kWide = kMode == kModeY2 || kMode == kModeY2N;
  static constexpr int kHalves = kWide ? 2 : 1;                      // 128-row halves per tile
  static constexpr int kTileRows = kHalves * kBM;
  static constexpr int kN = kMode == kModeY2N ? 224 : kY ? 256 : 2 * R;   // tile columns
  static constexpr int kHalfCols = kMode == kModeY2N ? 256 : kN;     // TMEM columns per half
  static constexpr int kStages = kWide ? 3 : 4;
  static constexpr int kAccs = kWide ? 1 : 2;                        // accumulator buffers
  static constexpr int kAccCols = kHalves * kHalfCols;               // TMEM columns of one
  static constexpr int kEpiWarps = kWide ? 8 : 4;
  static constexpr int kThreads = 64 + 32 * kEpiWarps;
  static constexpr int kABytes = kTileRows * 128;                    // rows x 64 bf16
  // B rows of a slot: the Y modes' extension step loads 256 U operand rows (two boxes)
  static constexpr int kBRows = kY ? 256 : kN;
  static constexpr int kBBytes = kBRows * 128;                       // 64 bf16 per row
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kMainTx = kABytes + kN * 128;            // bytes of a K step
  static constexpr int kCW = kN % 64 == 0 ? 64 : 32;                 // Y columns per store
  static constexpr int kBoxBytes = 32 * kCW * 2;                     // 32 rows x kCW bf16
  static constexpr int kBoxesPerWarp = kMode == kModeY2 ? 1 : 2;
  static constexpr int kOutBytes = kEpiWarps * kBoxesPerWarp * kBoxBytes;
  static constexpr int kTmemCols = kAccs * kAccCols <= 32 ? 32 : kAccs * kAccCols;
  static constexpr size_t kSmem = (size_t)kStages * kStageBytes + kOutBytes + 1024 + 1024;
  static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
  static_assert(kTmemCols <= 512, "TMEM columns");
  static_assert(kABytes == kHalves * kPanelBytes, "one 128-row panel per half");
  static_assert(kN % 32 == 0 && kN <= kBRows && kN <= kHalfCols, "tile columns");
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

// tm_a: X (box 64 x 128).  kModeS: tm_b = P_K (box 64 x 2r); K split into k_split
// ranges of k_chunk steps; fp32 partials to part[(k range) x rows x R], S_HL rows to
// s_out, s_count = one zeroed counter per 32 rows (null: partials only, for
// reduce_s_kernel).
// kModeY: w_map = W_i (box 64 x 32), tm_s = S_HL (box 64 x 128), tm_u = U operand (box
// 64 x 128) with this matrix's rows from u_row0, tm_o = Y (box 64 x 32).
template <int kMode, int R>
__global__ void __launch_bounds__(LinCfg<kMode, R>::kThreads, 1)
linear_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
              const CUtensorMap* __restrict__ w_map, const __grid_constant__ CUtensorMap tm_s,
              const __grid_constant__ CUtensorMap tm_u, const __grid_constant__ CUtensorMap tm_o,
              int rows, int cols, int k_steps, int k_split, int k_chunk, int u_row0,
              float* __restrict__ part, __nv_bfloat16* __restrict__ s_out,
              uint32_t* __restrict__ s_count, uint32_t* __restrict__ status,
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
  // Y modes: tile = (row block, column block), K = all steps + the extension;
  // kModeS: tile = (row block, K range)
  const int tiles_m = Cfg::kY ? (cols + kN - 1) / kN : k_split;
  const int n_tiles = ((rows + Cfg::kTileRows - 1) / Cfg::kTileRows) * tiles_m;
  auto k_range = [&](int nb, int& kb, int& ke) {
    if (Cfg::kY) {
      kb = 0;
      ke = k_steps + 1;                                             // + the extension
    } else {
      kb = nb * k_chunk;
      ke = min(k_steps, kb + k_chunk);
    }
  };
  const volatile int* abort = &sh.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::kStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], 1);
    }
    for (int s = 0; s < Cfg::kAccs; ++s) {
      mbar_init(&sh.acc_full[s], 1);
      mbar_init(&sh.acc_empty[s], Cfg::kEpiWarps);
    }
    mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_a);
    if constexpr (kMode == kModeS) {
      prefetch_tmap(&tm_b);
    } else {
      prefetch_tmap(&tm_o);
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
      int kb, ke;
      k_range(nb, kb, ke);
      for (int k = kb; k < ke; ++k) {
        const int s = (int)(n_st % Cfg::kStages);
        if (!mbar_wait_bounded(&sh.empty[s], (uint32_t)(((n_st / Cfg::kStages) & 1) ^ 1), abort,
                               wait_cycles)) {
          ok = false;
          break;
        }
        uint8_t* a_dst = st_smem + s * Cfg::kStageBytes;
        uint8_t* b_dst = a_dst + Cfg::kABytes;
        mbar_arrive_expect_tx(&sh.full[s], (Cfg::kY && k == k_steps) ? (uint32_t)Cfg::kStageBytes
                                                                     : Cfg::kMainTx);
        if (Cfg::kY && k == k_steps) {
          // the extension: S_HL rows of the token block, U operand rows of the W block
          for (int h = 0; h < Cfg::kHalves; ++h)
            tma_load_2d(a_dst + h * kPanelBytes, &tm_s, 0, tb * Cfg::kTileRows + h * kBM,
                        &sh.full[s]);
          for (int h = 0; h < Cfg::kBRows / kBM; ++h)
            tma_load_2d(b_dst + h * kPanelBytes, &tm_u, 0, u_row0 + nb * kN + h * kBM, &sh.full[s]);
        } else {
          for (int h = 0; h < Cfg::kHalves; ++h)
            tma_load_2d(a_dst + h * kPanelBytes, &tm_a, 64 * k, tb * Cfg::kTileRows + h * kBM,
                        &sh.full[s]);
          if constexpr (kMode == kModeS) {
            tma_load_2d(b_dst, &tm_b, 64 * k, 0, &sh.full[s]);
          } else {
            for (int h = 0; h < kN / 32; ++h)
              tma_load_2d(b_dst + h * 4096, w_map, 64 * k, nb * kN + 32 * h, &sh.full[s]);
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
      const int acc = (int)(it % Cfg::kAccs);
      const int64_t use = it / Cfg::kAccs;
      if (!mbar_wait_bounded(&sh.acc_empty[acc], (uint32_t)((use & 1) ^ 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d0 = tmem + (uint32_t)(acc * Cfg::kAccCols);
      int kb, ke;
      k_range(tile % tiles_m, kb, ke);
      for (int k = kb; k < ke; ++k) {
        const int s = (int)(n_st % Cfg::kStages);
        if (!mbar_wait_bounded(&sh.full[s], (uint32_t)((n_st / Cfg::kStages) & 1), abort,
                               wait_cycles)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t st_base = smem_u32(st_smem + s * Cfg::kStageBytes);
        const uint32_t b_base = st_base + Cfg::kABytes;
#pragma unroll
        for (int h = 0; h < Cfg::kHalves; ++h) {
          const uint32_t d = d0 + (uint32_t)(h * Cfg::kHalfCols);
          const uint32_t a_base = st_base + (uint32_t)(h * kPanelBytes);
          if (Cfg::kY && k == k_steps) {
            // hi chunk kk at element 16 kk of an operand row, lo chunk at R + 16 kk
#pragma unroll
            for (int kk = 0; kk < R / 16; ++kk) {
              const uint32_t hi = (uint32_t)(16 * kk * 2), lo = (uint32_t)((R + 16 * kk) * 2);
              mma_f16(d, sdesc_k_sw128(a_base + hi), sdesc_k_sw128(b_base + hi), idesc, 1u);
              mma_f16(d, sdesc_k_sw128(a_base + hi), sdesc_k_sw128(b_base + lo), idesc, 1u);
              mma_f16(d, sdesc_k_sw128(a_base + lo), sdesc_k_sw128(b_base + hi), idesc, 1u);
            }
          } else {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_f16(d, sdesc_k_sw128(a_base + 32 * kk), sdesc_k_sw128(b_base + 32 * kk), idesc,
                       (k > kb || kk > 0) ? 1u : 0u);
          }
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
  } else if (warp >= 2 && warp < 2 + Cfg::kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    const int g = warp & 3;                      // TMEM lane group == rows 32 g .. + 31
    const int half = (warp - 2) / 4;             // of the tile's 128-row halves
    const uint32_t lane_base = (uint32_t)(g * 32) << 16;
    uint8_t* obox = o_smem + (warp - 2) * Cfg::kBoxesPerWarp * Cfg::kBoxBytes;
    int64_t it = 0, n_box = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < n_tiles; tile += gridDim.x, ++it) {
      const int tb = tile / tiles_m, nb = tile % tiles_m;   // kModeS: nb = the K range
      const int acc = (int)(it % Cfg::kAccs);
      const int64_t use = it / Cfg::kAccs;
      if (!mbar_wait_bounded(&sh.acc_full[acc], (uint32_t)(use & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int y = tb * Cfg::kTileRows + half * kBM + 32 * g;
      const uint32_t t_base =
          tmem + lane_base + (uint32_t)(acc * Cfg::kAccCols + half * Cfg::kHalfCols);
      if constexpr (kMode == kModeS) {
        // partial S over this K range: D[:, :R] + D[:, R:2R], fp32, this lane's row
        uint32_t v[2 * R];
        if constexpr (R == 32) {
          uint32_t a[32], b[32];
          tmem_ld_32x32b_x32(t_base, a);
          tmem_ld_32x32b_x32(t_base + 32u, b);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) { v[e] = a[e]; v[32 + e] = b[e]; }
        } else {
          uint32_t a[32];
          tmem_ld_32x32b_x32(t_base, a);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = a[e];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.acc_empty[acc]);
        const int row = y + lane;
        float x[R];
#pragma unroll
        for (int e = 0; e < R; ++e) x[e] = __uint_as_float(v[e]) + __uint_as_float(v[R + e]);
        if (k_split == 1) {
          if (row < rows) {
#pragma unroll
            for (int e = 0; e < R; ++e) x[e] = 0.f + x[e];     // as the sum over one range
            write_s_row<R>(s_out, row, x);
          }
        } else {
          if (row < rows) {
            float4* dst = reinterpret_cast<float4*>(part + ((int64_t)nb * rows + row) * R);
#pragma unroll
            for (int j = 0; j < R / 4; ++j)
              dst[j] = make_float4(x[4 * j], x[4 * j + 1], x[4 * j + 2], x[4 * j + 3]);
          }
          // the last of the k_split warps to finish this 32-row group sums its partials
          if (s_count != nullptr) {
            __threadfence();
            __syncwarp();
            uint32_t old = 0;
            if (lane == 0) old = atomicInc(&s_count[tb * 4 + g], (uint32_t)(k_split - 1));
            old = __shfl_sync(0xffffffffu, old, 0);
            if (old == (uint32_t)(k_split - 1)) {
              __threadfence();
              if (row < rows) {
#pragma unroll
                for (int e = 0; e < R; ++e) x[e] = 0.f;
                for (int ks = 0; ks < k_split; ++ks) {
                  const float4* src =
                      reinterpret_cast<const float4*>(part + ((int64_t)ks * rows + row) * R);
#pragma unroll
                  for (int j = 0; j < R / 4; ++j) {
                    const float4 q = __ldcg(src + j);
                    x[4 * j] += q.x;
                    x[4 * j + 1] += q.y;
                    x[4 * j + 2] += q.z;
                    x[4 * j + 3] += q.w;
                  }
                }
                write_s_row<R>(s_out, row, x);
              }
            }
          }
        }
      } else {
        // kCW columns of Y at a time, through the warp's box(es) in turn
        constexpr int kCW = Cfg::kCW;
#pragma unroll 1
        for (int c = 0; c < kN / kCW; ++c) {
          uint32_t v[2][32];
          tmem_ld_32x32b_x32(t_base + (uint32_t)(kCW * c), v[0]);
          if constexpr (kCW == 64) tmem_ld_32x32b_x32(t_base + (uint32_t)(kCW * c + 32), v[1]);
          tmem_ld_wait();
          if (c == kN / kCW - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh.acc_empty[acc]);
          }
          uint8_t* box = obox + (int)(n_box % Cfg::kBoxesPerWarp) * Cfg::kBoxBytes;
          if (lane == 0) {                       // the store that used this box has read it
            if constexpr (Cfg::kBoxesPerWarp == 2)
              bulk_wait_read_1();
            else
              bulk_wait_read_all();
          }
          __syncwarp();
          // 16-byte chunk j of row `lane`: 128-byte swizzle (chunk ^ row % 8) for 64
          // columns, 64-byte swizzle (chunk ^ (row / 2) % 4) for 32
#pragma unroll
          for (int j = 0; j < kCW / 8; ++j) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const __nv_bfloat162 b2 =
                  __floats2bfloat162_rn(__uint_as_float(v[j >> 2][(j & 3) * 8 + 2 * e]),
                                        __uint_as_float(v[j >> 2][(j & 3) * 8 + 2 * e + 1]));
              w[e] = *reinterpret_cast<const uint32_t*>(&b2);
            }
            const int off = kCW == 64 ? lane * 128 + ((j ^ (lane & 7)) << 4)
                                      : lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4);
            *reinterpret_cast<uint4*>(box + off) = make_uint4(w[0], w[1], w[2], w[3]);
          }
          fence_async_smem();
          __syncwarp();
          if (lane == 0) {
            const int x = nb * kN + kCW * c;
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

// S_HL[row] = [hi | lo | 0] of the sum over the K ranges of the fp32 partial rows of S
// (k_split > kFusedSplits): thread (row, g) adds columns 8 g .. 8 g + 7 in K-range order.
template <int R>
__global__ void __launch_bounds__(128)
reduce_s_kernel(const float* __restrict__ part, int rows, int k_split,
                __nv_bfloat16* __restrict__ s_hl) {
  constexpr int kGroups = R / 8;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)rows * kGroups) return;
  const int row = (int)(idx / kGroups), g = (int)(idx % kGroups);
  float x[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) x[e] = 0.f;
  for (int ks = 0; ks < k_split; ++ks) {
    const float4* src = reinterpret_cast<const float4*>(part + ((int64_t)ks * rows + row) * R + 8 * g);
    const float4 a = src[0], b = src[1];
    x[0] += a.x; x[1] += a.y; x[2] += a.z; x[3] += a.w;
    x[4] += b.x; x[5] += b.y; x[6] += b.z; x[7] += b.w;
  }
  uint4 hi, lo;
  split8(x, hi, lo);
  uint4* out = reinterpret_cast<uint4*>(s_hl + (int64_t)row * 64);
  out[g] = hi;
  out[kGroups + g] = lo;
  if (g == 0)
    for (int z = 2 * kGroups; z < 8; ++z) out[z] = make_uint4(0u, 0u, 0u, 0u);
}

template <int kMode, int R>
cudaError_t launch_linear_r(const CUtensorMap& tm_a, const CUtensorMap& tm_b,
                            const CUtensorMap* w_map, const CUtensorMap& tm_s,
                            const CUtensorMap& tm_u, const CUtensorMap& tm_o, int rows, int cols,
                            int k_steps, int k_split, int k_chunk, int u_row0, float* part,
                            __nv_bfloat16* s_out, uint32_t* s_count, int grid,
                            uint32_t* d_status, cudaStream_t s) {
  using Cfg = LinCfg<kMode, R>;
  cudaError_t e = cudaFuncSetAttribute(linear_kernel<kMode, R>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)Cfg::kSmem);
  if (e != cudaSuccess) return e;
  linear_kernel<kMode, R><<<grid, Cfg::kThreads, Cfg::kSmem, s>>>(
      tm_a, tm_b, w_map, tm_s, tm_u, tm_o, rows, cols, k_steps, k_split, k_chunk, u_row0, part,
      s_out, s_count, d_status, kWaitCycles);
  return cudaGetLastError();
}

}  // namespace

bool linear_supported(int32_t r) { return r == 16 || r == 32 || r == 64 || r == 128; }
bool linear_single_cta_supported(int32_t r) { return r == 16 || r == 32; }

void linear_s_split(int64_t T, int64_t n, int32_t sms, int32_t* k_split, int32_t* k_chunk) {
  const int64_t k_steps = (n + 63) / 64;
  const int64_t blocks = (T + kBM - 1) / kBM;
  // at most one wave of tiles: a second, partial wave would double the kernel's time
  int64_t want = std::max<int64_t>(1, std::min<int64_t>(k_steps, sms / blocks));
  const int64_t chunk = (k_steps + want - 1) / want;
  *k_chunk = (int32_t)chunk;
  *k_split = (int32_t)((k_steps + chunk - 1) / chunk);   // every K range non-empty
}

int32_t linear_y_tiling(int64_t T, int64_t m, int32_t sms, int32_t option) {
  if (option >= 1 && option <= 3) return option;
  // waves of tiles x the time of one tile, relative to 256 x 256 (1000): 128 x 256 tiles
  // run at ~1/1.6 of it, 256 x 224 tiles at ~0.9
  auto cost = [&](int rows, int cols, int64_t per_tile) {
    const int64_t tiles = (T + rows - 1) / rows * ((m + cols - 1) / cols);
    return (tiles + sms - 1) / sms * per_tile;
  };
  int32_t best = 2;
  int64_t c_best = cost(256, 256, 1000);
  const int64_t c3 = cost(256, 224, 900), c1 = cost(128, 256, 625);
  if (c3 < c_best) { best = 3; c_best = c3; }
  if (c1 < c_best) best = 1;
  return best;
}

int32_t linear_y_tile_rows(int32_t tiling) { return tiling == 1 ? 128 : 256; }
int32_t linear_y_tile_cols(int32_t tiling) { return tiling == 3 ? 224 : 256; }

int64_t linear_pk_elems(int64_t n, int32_t r) { return 2 * (int64_t)r * ((n + 63) / 64 * 64); }

cudaError_t launch_linear_s(const CUtensorMap& tm_x, const CUtensorMap& tm_pk, int64_t T,
                            int64_t n, int32_t r, int32_t k_split, int32_t k_chunk, float* part,
                            __nv_bfloat16* s_hl, uint32_t* s_count, int32_t sms,
                            uint32_t* d_status, cudaStream_t s) {
  const int k_steps = (int)((n + 63) / 64);
  const int tiles = (int)((T + kBM - 1) / kBM) * k_split;
  const int grid = std::min<int>(tiles, sms);
  const bool fused = k_split <= kFusedSplits;
  uint32_t* count = fused ? s_count : nullptr;
  cudaError_t e;
  switch (r) {
    case 16:
      e = launch_linear_r<kModeS, 16>(tm_x, tm_pk, nullptr, tm_x, tm_x, tm_x, (int)T, 32, k_steps,
                                      k_split, k_chunk, 0, part, s_hl, count, grid, d_status, s);
      if (e == cudaSuccess && !fused)
        reduce_s_kernel<16><<<(unsigned)((T * 2 + 127) / 128), 128, 0, s>>>(part, (int)T, k_split, s_hl);
      break;
    case 32:
      e = launch_linear_r<kModeS, 32>(tm_x, tm_pk, nullptr, tm_x, tm_x, tm_x, (int)T, 64, k_steps,
                                      k_split, k_chunk, 0, part, s_hl, count, grid, d_status, s);
      if (e == cudaSuccess && !fused)
        reduce_s_kernel<32><<<(unsigned)((T * 4 + 127) / 128), 128, 0, s>>>(part, (int)T, k_split, s_hl);
      break;
    default: return cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

int32_t linear_s_launches(int32_t k_split) { return k_split <= kFusedSplits ? 1 : 2; }

cudaError_t launch_linear_y(const CUtensorMap& tm_x, const CUtensorMap* d_w_map,
                            const CUtensorMap& tm_s_in, const CUtensorMap& tm_u,
                            const CUtensorMap& tm_y, int64_t T, int64_t m, int64_t n,
                            int32_t u_row0, int32_t r, int32_t tiling, int32_t sms,
                            uint32_t* d_status, cudaStream_t s) {
  if (tiling < 1 || tiling > 3) return cudaErrorInvalidValue;
  const int k_steps = (int)((n + 63) / 64);
  const int64_t rows = linear_y_tile_rows(tiling), cols = linear_y_tile_cols(tiling);
  const int64_t tiles = (T + rows - 1) / rows * ((m + cols - 1) / cols);
  const int grid = (int)std::min<int64_t>(tiles, sms);
#define ZO_LINEAR_Y(MODE, RR)                                                                  \
  launch_linear_r<MODE, RR>(tm_x, tm_x, d_w_map, tm_s_in, tm_u, tm_y, (int)T, (int)m, k_steps, \
                            1, k_steps, u_row0, nullptr, nullptr, nullptr, grid, d_status, s)
  switch (r * 4 + tiling) {
    case 16 * 4 + 1: return ZO_LINEAR_Y(kModeY, 16);
    case 16 * 4 + 2: return ZO_LINEAR_Y(kModeY2, 16);
    case 16 * 4 + 3: return ZO_LINEAR_Y(kModeY2N, 16);
    case 32 * 4 + 1: return ZO_LINEAR_Y(kModeY, 32);
    case 32 * 4 + 2: return ZO_LINEAR_Y(kModeY2, 32);
    case 32 * 4 + 3: return ZO_LINEAR_Y(kModeY2N, 32);
    default: return cudaErrorInvalidValue;
  }
#undef ZO_LINEAR_Y
}

}  // namespace zo
