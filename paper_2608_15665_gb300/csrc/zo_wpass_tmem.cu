// Weight pass on the 5th-generation tensor cores for r >= 64, with the U operand in
// Tensor Memory: W_i <- rnd_bf16(W_i + U_i P_i) for every bf16 matrix in one persistent
// launch (the fused form of Alg. 2's "W_i <- W_i + eps U_i Z_i V_i^T", Eq. (4), and of
// the update of Eq. (10)).  The r <= 32 kernel, with both operands in shared memory, and
// the operand split (scaled fp16 pairs, hi.hi + hi.lo + lo.hi in fp32) are described in
// zo_wpass_tc.cu.
//
// Why Tensor Memory for U: at r = 64 and 128 the 3r/16 MMAs of a 128 x 128 tile (12 and
// 24) read their operands at up to 128 B/clk from shared memory, the SM's whole shared-
// memory bandwidth, while the epilogue and the TMA copies need the same bandwidth for
// the W tile.  tcgen05.mma with A in TMEM reads only P from shared memory, and the
// 64 KB of shared memory a U tile would take holds P stages instead (3 at r = 64).
//
// Roles of the 480 threads of a CTA (one CTA per SM, persistent over chunks of tiles):
//   warp 0, lane 0:  TMA producer of W -- each tile as 8 boxes of 32 rows x 64
//                    columns, 128-byte swizzle, as far ahead as the W ring allows.
//   warp 1, lane 0:  MMA issuer -- 3 * r/16 tcgen05.mma (M=128, N=128, K=16, A in TMEM)
//                    per tile into one of two TMEM accumulators; warp 1 also owns the
//                    TMEM allocation (2 x 128 accumulator + 2 x r U columns).
//   warps 2..9:      epilogue -- warp w owns rows 32 (w % 4) .. + 31 (its TMEM lane
//                    group) of one column half, a 32 x 64 W box: tcgen05.ld the fp32
//                    update, add it to the W rows in shared memory, round to bf16 in
//                    place, TMA-store the box.  Eight warps, two per lane group: the
//                    epilogue of four warps alone is the bottleneck at r >= 64.
//   warp 10, lane 0: TMA producer of the P tile of every tile (2-3 stages).
//   warps 11..14:    U loaders -- when the row block changes, copy the tile's 128 rows
//                    of U_T into one of two TMEM U buffers (tcgen05.st; warp w writes
//                    lanes 32 (w % 4) .. + 31).
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

constexpr int kEpiWarp0 = 2;       // first epilogue warp
constexpr int kTmemCols = 512;     // two accumulators + two U tiles (R columns each)

template <int R>
struct TmemCfg {
  static_assert(R == 64 || R == 128, "the TMEM-operand kernel covers r = 64 and r = 128");
  static constexpr int kHLW = hl_width(R);
  static constexpr int kPanels = kHLW / 64;
  static constexpr int kOpBytes = kPanels * kPanelBytes;        // one P tile (hi + lo)
  static constexpr int kACols = R;                              // TMEM columns of one U tile
  // W stages of 32 KB and P stages of 32 / 64 KB (R = 64: 4 x 32 + 3 x 32 KB, R = 128:
  // 3 x 32 + 2 x 64 KB; with the barriers 226 KB of the 227 KB a CTA may hold)
  static constexpr int kWStages = R >= 128 ? 3 : 4;
  static constexpr int kBStages = R >= 128 ? 2 : 3;
  static constexpr int kKC = R / 16;                            // K chunks of 16
  // eight epilogue warps (one 32 x 64 W box each), one P producer, four U loaders
  static constexpr int kEpiWarps = 8;
  static constexpr int kBoxesPerWarp = 8 / kEpiWarps;
  static constexpr int kPWarp = kEpiWarp0 + kEpiWarps;
  static constexpr int kUWarp0 = kPWarp + 1;
  static constexpr int kThreads = 32 * (kUWarp0 + 4);
  // R = 64: a W stage is released one tile late, once the next tile's store is issued,
  // so a store's shared-memory reads overlap the next tile's epilogue (measured +4%);
  // at R = 128 the 3-stage W ring cannot spare the stage (-1%)
  static constexpr bool kDeferRelease = R == 64;
  static constexpr size_t kSmem = (size_t)kWStages * kWStageBytes + (size_t)kBStages * kOpBytes +
                                  1024 /*barriers*/ + 1024 /*align*/;
};

template <int R>
__global__ void __launch_bounds__(TmemCfg<R>::kThreads, 1)
wpass_tmem_kernel(const uint4* __restrict__ u_t, const __grid_constant__ CUtensorMap tm_b,
                const CUtensorMap* __restrict__ w_maps, const TcMat* __restrict__ mats,
                const float* __restrict__ pinv, int n_mats, int64_t n_tiles,
                uint32_t* __restrict__ status, long long wait_cycles, int inject_wait) {
  using Cfg = TmemCfg<R>;
  static_assert(Cfg::kWStages >= 2 && Cfg::kWStages <= 4, "W ring must fit Shared::w_full");
  static_assert(Cfg::kBStages >= 2 && Cfg::kBStages <= 4, "P ring must fit Shared::b_full");
  static_assert(2 * kBN + 2 * Cfg::kACols <= kTmemCols, "accumulators + U buffers in TMEM");
  static_assert(sizeof(Shared) <= 1024, "barrier block");
  static_assert(Cfg::kSmem <= 227 * 1024, "shared memory per CTA");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* w_smem = smem;
  uint8_t* b_smem = w_smem + Cfg::kWStages * kWStageBytes;
  Shared& sh = *reinterpret_cast<Shared*>(b_smem + Cfg::kBStages * Cfg::kOpBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Interleaved walk: CTA b takes the chunks of kTileChunk tiles b, b + G, b + 2G, ...
  // At any moment the G CTAs work on neighbouring tiles -- the same row blocks of one
  // matrix -- so the DRAM sees one moving front of nearby rows instead of G scattered
  // streams (LLaMA-7B set: 6.35 TB/s against 5.03 TB/s for contiguous per-CTA ranges);
  // the U tile is reused within a chunk.
  const int64_t G = gridDim.x;
  const int64_t t_begin = (int64_t)blockIdx.x * kTileChunk;
  const int64_t t_end = n_tiles;
  const int64_t t_stride = G * kTileChunk;
  const volatile int* abort = &sh.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::kWStages; ++s) {
      mbar_init(&sh.w_full[s], 1);
      mbar_init(&sh.w_empty[s], Cfg::kEpiWarps);
    }
    for (int s = 0; s < Cfg::kBStages; ++s) {
      mbar_init(&sh.b_full[s], 1);
      mbar_init(&sh.b_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sh.a_full[s], 4);      // the four U-loader warps
      mbar_init(&sh.a_empty[s], 1);
      mbar_init(&sh.acc_full[s], 1);
      mbar_init(&sh.acc_empty[s], Cfg::kEpiWarps);
    }
    mbar_init(&sh.never, 1);
    sh.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_b);
  }
  if (warp == 1) {
    tmem_alloc(&sh.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer: W tiles
    int64_t n_w = 0;                              // copies issued into the W ring
    bool ok = true;
    TileIter ti;
    ti.init(mats, n_mats, t_begin, t_end, t_stride);
    ti.chunk = kTileChunk;
    for (; ti.valid(); ti.next()) {
      const CUtensorMap* wmap = w_maps + ti.i;
      // W tile: 4 row groups x 2 column halves
      const int s = (int)(n_w % Cfg::kWStages);
      const uint32_t ph = (uint32_t)((n_w / Cfg::kWStages) & 1);
      if (!mbar_wait_bounded(&sh.w_empty[s], ph ^ 1u, abort, wait_cycles)) { ok = false; break; }
      // the tile's scale rides with its W stage (see zo_wpass_tc.cu)
      sh.w_scale[s] = pinv[ti.i] * exp2i(-kUVScaleExp);
      mbar_arrive_expect_tx(&sh.w_full[s], kWStageBytes);
      uint8_t* dst = w_smem + s * kWStageBytes;
      for (int g = 0; g < 4; ++g)
        for (int h = 0; h < 2; ++h)
          tma_load_2d(dst + (g * 2 + h) * kWBoxBytes, wmap, (int)(ti.cb * kBN + 64 * h),
                      (int)(ti.rb * kBM + 32 * g), &sh.w_full[s]);
      ++n_w;
    }
    if (!ok) give_up(sh, status);
    // drain: the last copy issued into every slot has landed before the CTA exits
    for (int s = 0; s < Cfg::kWStages; ++s) {
      const int64_t k = last_in_slot(n_w, s, Cfg::kWStages);
      if (k >= 0) mbar_wait_bounded(&sh.w_full[s], (uint32_t)((k / Cfg::kWStages) & 1), nullptr, wait_cycles);
    }
  } else if (warp == Cfg::kPWarp && lane == 0) {
    // ------------------------------------------------------------ TMA producer: P tiles
    int64_t n_b = 0;                              // P tiles issued into the ring
    bool ok = true;
    TileIter ti;
    ti.init(mats, n_mats, t_begin, t_end, t_stride);
    ti.chunk = kTileChunk;
    for (; ti.valid(); ti.next()) {
      const TcMat& mt = mats[ti.i];
      const int s = (int)(n_b % Cfg::kBStages);
      const uint32_t ph = (uint32_t)((n_b / Cfg::kBStages) & 1);
      if (!mbar_wait_bounded(&sh.b_empty[s], ph ^ 1u, abort, wait_cycles)) { ok = false; break; }
      mbar_arrive_expect_tx(&sh.b_full[s], Cfg::kOpBytes);
      for (int p = 0; p < Cfg::kPanels; ++p)
        tma_load_2d(b_smem + s * Cfg::kOpBytes + p * kPanelBytes, &tm_b, 64 * p,
                    (int)(mt.p_row0 + ti.cb * kBN), &sh.b_full[s]);
      ++n_b;
    }
    if (!ok) give_up(sh, status);
    for (int s = 0; s < Cfg::kBStages; ++s) {
      const int64_t k = last_in_slot(n_b, s, Cfg::kBStages);
      if (k >= 0) mbar_wait_bounded(&sh.b_full[s], (uint32_t)((k / Cfg::kBStages) & 1), nullptr, wait_cycles);
    }
  } else if (warp >= Cfg::kUWarp0) {
    // ------------------------------------------------------------ U tiles into TMEM
    // Warp w may address TMEM lanes 32 (w % 4) .. + 31 only, so the four loader warps
    // cover the tile's 128 rows; lane t writes row 32 (w % 4) + t: its R words of
    // [hi | lo] (two fp16 per 32-bit column, lower half first).  U_T keeps chunk j of
    // the block's 128 rows contiguous, so each 16-byte load of the warp is one 512-byte
    // access.
    const int q = warp & 3;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    int64_t n_a = 0;
    int prev_i = -1;
    int64_t prev_rb = -1;
    bool ok = true;
    TileIter ti;
    ti.init(mats, n_mats, t_begin, t_end, t_stride);
    ti.chunk = kTileChunk;
    for (; ti.valid(); ti.next()) {
      if (ti.i == prev_i && ti.rb == prev_rb) continue;
      prev_i = ti.i;
      prev_rb = ti.rb;
      const int s = (int)(n_a & 1);
      const uint32_t ph = (uint32_t)((n_a >> 1) & 1);
      int got = 1;
      if (lane == 0) got = mbar_wait_bounded(&sh.a_empty[s], ph ^ 1u, abort, wait_cycles) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, got, 0)) { ok = false; break; }
      tc_fence_after();
      const int64_t block = mats[ti.i].u_row0 / kBM + ti.rb;
      const uint4* src = u_t + block * (R / 4) * kBM + 32 * q + lane;
      const uint32_t col0 = (uint32_t)(2 * kBN + s * Cfg::kACols);
      if constexpr (Cfg::kACols >= 32) {
        constexpr int kPieces = Cfg::kACols / 32;
#pragma unroll
        for (int p0 = 0; p0 < kPieces; p0 += 2) {
          // the loads of two 32-column pieces in flight before their stores
          uint32_t v[2][32];
#pragma unroll
          for (int pp = 0; pp < 2; ++pp) {
            if (p0 + pp >= kPieces) break;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const uint4 t4 = __ldg(src + ((p0 + pp) * 8 + j) * kBM);
              v[pp][4 * j] = t4.x; v[pp][4 * j + 1] = t4.y; v[pp][4 * j + 2] = t4.z; v[pp][4 * j + 3] = t4.w;
            }
          }
#pragma unroll
          for (int pp = 0; pp < 2; ++pp)
            if (p0 + pp < kPieces) tmem_st_32x32b_x32(tmem + lane_base + col0 + 32 * (p0 + pp), v[pp]);
        }
      } else {
        uint32_t v[16];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint4 t4 = __ldg(src + j * kBM);
          v[4 * j] = t4.x; v[4 * j + 1] = t4.y; v[4 * j + 2] = t4.z; v[4 * j + 3] = t4.w;
        }
        tmem_st_32x32b_x16(tmem + lane_base + col0, v);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.a_full[s]);
      ++n_a;
    }
    if (!ok && lane == 0) give_up(sh, status);
  } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc = idesc_f16_f32(kBM, kBN);
    int64_t it = 0, a_it = 0;
    int prev_i = -1;
    int64_t prev_rb = -1;
    int sa = 0;
    bool ok = true;
    TileIter ti, nx;                            // nx runs one tile ahead of ti
    ti.init(mats, n_mats, t_begin, t_end, t_stride);
    ti.chunk = kTileChunk;
    nx = ti;
    nx.next();
    for (; ti.valid(); ti = nx, nx.next(), ++it) {
      const bool new_a = ti.i != prev_i || ti.rb != prev_rb;
      if (new_a) {
        sa = (int)(a_it & 1);
        if (!mbar_wait_bounded(&sh.a_full[sa], (uint32_t)((a_it >> 1) & 1), abort, wait_cycles)) {
          ok = false;
          break;
        }
        ++a_it;
        prev_i = ti.i;
        prev_rb = ti.rb;
      }
      // the U buffer is released after its last tile: the next tile starts another row
      // block (or there is none)
      const bool last_a = !nx.valid() || nx.i != ti.i || nx.rb != ti.rb;
      const int sb = (int)(it % Cfg::kBStages);
      if (!mbar_wait_bounded(&sh.b_full[sb], (uint32_t)((it / Cfg::kBStages) & 1), abort,
                             wait_cycles)) { ok = false; break; }
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_empty[acc], (uint32_t)(((it >> 1) & 1) ^ 1), abort,
                             wait_cycles)) { ok = false; break; }
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(acc * kBN);
      const uint32_t a_base = tmem + (uint32_t)(2 * kBN + sa * Cfg::kACols);
      const uint32_t b_base = smem_u32(b_smem + sb * Cfg::kOpBytes);
      // hi.lo and lo.hi first, hi.hi last (see zo_wpass_tc.cu): only the r/16 hi.hi MMAs
      // round at the update's full size
#pragma unroll
      for (int pass = 0; pass < 3; ++pass) {
#pragma unroll
        for (int kk = 0; kk < Cfg::kKC; ++kk) {
          // U: hi chunk kk at column 8 kk of the buffer, lo chunk at R/2 + 8 kk;
          // P: hi chunk kk at element 16 kk of the operand row, lo chunk at R + 16 kk
          const uint32_t a_t = a_base + (uint32_t)((pass == 1 ? R / 2 : 0) + 8 * kk);
          const int e_b = (pass == 0 ? R : 0) + 16 * kk;
          const uint64_t b_d =
              sdesc_k_sw128(b_base + (uint32_t)((e_b / 64) * kPanelBytes + (e_b % 64) * 2));
          mma_f16_ts(d, a_t, b_d, idesc, (pass | kk) != 0 ? 1u : 0u);
        }
      }
      mma_commit(&sh.b_empty[sb]);
      if (last_a) mma_commit(&sh.a_empty[sa]);
      mma_commit(&sh.acc_full[acc]);
    }
    if (!ok) give_up(sh, status);
    if (it > 0) {
      // every MMA issued by this thread has completed before TMEM is released
      const int64_t last = it - 1;
      mbar_wait_bounded(&sh.acc_full[last & 1], (uint32_t)((last >> 1) & 1), nullptr, wait_cycles);
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + Cfg::kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    // Warp w owns rows 32 (w % 4) .. + 31 of the tile (its TMEM lane group) and
    // kBoxesPerWarp of the two column halves -- 32 x 64 W boxes.
    const int g = warp & 3;                      // TMEM lane group == tile row group
    const int h0 = (warp - kEpiWarp0) >> 2;      // first column half
    const uint32_t lane_base = (uint32_t)(g * 32) << 16;
    int s_prev = -1;                             // stage whose release is deferred
    int64_t it = 0;
    bool ok = true;
    TileIter ti;
    ti.init(mats, n_mats, t_begin, t_end, t_stride);
    ti.chunk = kTileChunk;
    for (; ti.valid(); ti.next(), ++it) {
      const TcMat& mt = mats[ti.i];
      const int acc = (int)(it & 1);
      // test hook (zo_set_option ZO_OPTION_TEST_WAIT_TIMEOUT): CTA 0's epilogue first waits
      // on a barrier that nothing arrives on, so its bounded wait runs out
      if (inject_wait && blockIdx.x == 0 && it == 0 &&
          !mbar_wait_bounded(&sh.never, 0u, abort, wait_cycles)) {
        ok = false;
        break;
      }
      if (!mbar_wait_bounded(&sh.acc_full[acc], (uint32_t)((it >> 1) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int s = (int)(it % Cfg::kWStages);
      if (!mbar_wait_bounded(&sh.w_full[s], (uint32_t)((it / Cfg::kWStages) & 1), abort,
                             wait_cycles)) {
        ok = false;
        break;
      }
      uint8_t* stage = w_smem + s * kWStageBytes;
      // the accumulator holds 2^(kUVScaleExp + e_P,i) U P: back to U P in the add
      const uint64_t wscale2 = splat2(sh.w_scale[s]);
#pragma unroll
      for (int hh = 0; hh < Cfg::kBoxesPerWarp; ++hh) {
        const int h = h0 + hh;
        // both 32-column loads of the box in flight before the one wait
        uint32_t v[2][32];
        tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kBN + 64 * h), v[0]);
        tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kBN + 64 * h + 32), v[1]);
        tmem_ld_wait();
        uint8_t* box = stage + (g * 2 + h) * kWBoxBytes + lane * 128;
#pragma unroll
        for (int j = 0; j < 8; ++j) {              // logical 16-byte chunk of the row
          uint4* p = reinterpret_cast<uint4*>(box + ((j ^ (lane & 7)) << 4));
          uint4 raw = *p;
          uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
          for (int e = 0; e < 4; ++e)
            wv[e] = bf16x2_add_scaled(wv[e], v[j >> 2][(j & 3) * 8 + 2 * e],
                                      v[j >> 2][(j & 3) * 8 + 2 * e + 1], wscale2);
          *p = make_uint4(wv[0], wv[1], wv[2], wv[3]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.acc_empty[acc]);
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int64_t y = ti.rb * kBM + 32 * g;
        for (int hh = 0; hh < Cfg::kBoxesPerWarp; ++hh) {
          const int h = h0 + hh;
          const int64_t x = ti.cb * kBN + 64 * h;
          if (y < mt.m && x < mt.n)
            tma_store_2d(w_maps + ti.i, (int)x, (int)y, stage + (g * 2 + h) * kWBoxBytes);
        }
        bulk_commit();
        if constexpr (Cfg::kDeferRelease) {
          if (s_prev >= 0) {
            bulk_wait_read_1();                  // the previous tile's store has read its stage
            mbar_arrive(&sh.w_empty[s_prev]);
          }
          s_prev = s;
        } else {
          bulk_wait_read_all();
          mbar_arrive(&sh.w_empty[s]);
        }
      }
      __syncwarp();
    }
    if (lane == 0 && s_prev >= 0) {
      bulk_wait_read_all();
      mbar_arrive(&sh.w_empty[s_prev]);
    }
    if (!ok && lane == 0) give_up(sh, status);
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// U_T: the U operand in the layout the TMEM loaders read.  Row i of the stacked operand
// is [hi | lo] of the fp16 pair of U[i, :] 2^kUVScaleExp = R 32-bit words = R/4 chunks of
// 16 bytes;
// within each 128-row block chunk j of all 128 rows is contiguous:
//   U_T[(block * (R/4) + j) * 128 + (i % 128)] = chunk j of row i,
// so one warp reads 512 contiguous bytes per chunk (one row per lane), and this kernel
// (one thread per row) writes 128 consecutive chunks per store instruction.
template <int R>
__global__ void __launch_bounds__(128)
split_u_chunks_kernel(const MatDesc* __restrict__ mats, const TcMat* __restrict__ tcm,
               const int2* __restrict__ units, uint4* __restrict__ u_t) {
  const int2 u = units[blockIdx.x];
  const MatDesc md = mats[u.x];
  const int tid = threadIdx.x;
  const int64_t i0 = u.y;
  const int rows = (int)(md.m - i0 < 128 ? md.m - i0 : 128);
  if (tid >= rows) return;                  // rows past m stay at the zero they were set to
  const int64_t block = (tcm[u.x].u_row0 + i0) / 128;
  uint4* dst = u_t + block * (R / 4) * 128 + tid;
  const float4* src = reinterpret_cast<const float4*>(md.U + (i0 + tid) * R);
#pragma unroll
  for (int g = 0; g < R / 8; ++g) {
    const float4 a = src[2 * g], b = src[2 * g + 1];
    const float x[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    uint4 hi, lo;
    split8_f16(x, exp2i(kUVScaleExp), hi, lo);
    dst[(int64_t)g * 128] = hi;
    dst[(int64_t)(R / 8 + g) * 128] = lo;
  }
}

template <int R>
cudaError_t launch_tmem_r(const uint4* u_t, const CUtensorMap& tm_b, const CUtensorMap* w_maps,
                          const TcMat* mats, const float* pinv, int n_mats, int64_t n_tiles, int grid,
                          uint32_t* status, bool inject_wait, cudaStream_t s) {
  const size_t smem = TmemCfg<R>::kSmem;
  cudaError_t e = cudaFuncSetAttribute(wpass_tmem_kernel<R>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const long long wait = inject_wait ? kTestWaitCycles : kWaitCycles;
  wpass_tmem_kernel<R><<<grid, TmemCfg<R>::kThreads, smem, s>>>(u_t, tm_b, w_maps, mats, pinv,
                                                                 n_mats, n_tiles, status, wait,
                                                                 inject_wait ? 1 : 0);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_split_u_chunks(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                                  int32_t n_units, int32_t r, uint4* u_t, cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 64: split_u_chunks_kernel<64><<<n_units, 128, 0, s>>>(d_mats, d_tc, d_units, u_t); break;
    case 128: split_u_chunks_kernel<128><<<n_units, 128, 0, s>>>(d_mats, d_tc, d_units, u_t); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_wpass_tmem(const uint4* u_t, const CUtensorMap& tm_b,
                              const CUtensorMap* d_w_maps, const TcMat* d_tc, const float* d_pinv,
                              int32_t n_mats, int64_t n_tiles, int32_t grid, int32_t r,
                              uint32_t* d_status, bool inject_wait, cudaStream_t s) {
  if (n_tiles <= 0) return cudaSuccess;
  switch (r) {
    case 64: return launch_tmem_r<64>(u_t, tm_b, d_w_maps, d_tc, d_pinv, n_mats, n_tiles, grid, d_status, inject_wait, s);
    case 128: return launch_tmem_r<128>(u_t, tm_b, d_w_maps, d_tc, d_pinv, n_mats, n_tiles, grid, d_status, inject_wait, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
