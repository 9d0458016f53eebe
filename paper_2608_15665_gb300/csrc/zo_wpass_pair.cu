// Weight pass at r = 128 on SM pairs: W_i <- rnd_bf16(W_i + U_i P_i) for every bf16 matrix
// in one persistent launch (the fused form of Alg. 2's "W_i <- W_i + eps U_i Z_i V_i^T",
// Eq. (4), and of the update of Eq. (10)), with the contraction issued as M = 256 MMAs
// across the two SMs of a cluster (tcgen05.mma.cta_group::2).
//
// Why pairs at r = 128: the 3 r / 16 = 24 MMAs of a 128 x 128 tile read their B operand
// (the P tile) from shared memory, 96 KB per tile, on top of 128 KB of W traffic (TMA load,
// the epilogue's read and write, the TMA store) and the 64 KB P tile itself: 288 KB per tile
// against the ~2600 cycles of HBM time a tile has, at 128 B/clk.  An M = 256 MMA of the pair
// computes a 256 x 128 tile -- 128 rows in each SM's Tensor Memory -- reading the A operand
// (U) from each SM's own Tensor Memory and the B operand (the P tile) half from each SM's
// shared memory.  Each SM then moves 128 KB of W, 32 KB of P loads and 48 KB of MMA reads
// per 128 x 128 tile of its own: 208 KB.
//
// Pair tile = 256 rows x 128 columns of one W_i; CTA c of the cluster owns rows 128 c ..
// 128 c + 127 (its W boxes, its U rows in its Tensor Memory, its accumulator lanes) and
// rows 64 c .. 64 c + 63 of the P tile (P_HL rows = W columns).  Both CTAs walk the same
// pair tiles (chunks of kTileChunk consecutive pair tiles, interleaved over the pairs), so
// their loops and barrier sequences run in lockstep.
//
// Roles (480 threads per CTA, one CTA per SM):
//   warp 0, lane 0:   W producer (this CTA's 128 rows of the tile), 4 stages; it stores
//                     the tile's per-matrix scale beside the stage.
//   warp 1:           Tensor Memory allocation (.cta_group::2, in both CTAs); in the even
//                     CTA (the leader) lane 0 issues every MMA of the pair.
//   warps 2..9:       epilogue of this CTA's 128 rows, one 32 x 64 box per warp.
//   warp 10, lane 0:  producer of this CTA's half of the P tile, 3 stages of 32 KB; both
//                     halves complete their bytes on the leader's b_full (the TMA's
//                     .cta_group::2 form), which the leader's producer arms for both.
//   warps 11..14:     U loaders: this CTA's 128 rows of U into one of two TMEM buffers.
// Barriers: local to each CTA -- w_full, w_empty, and b_empty, a_empty, acc_full (arrived in
// both CTAs by the leader's multicast commits); in the leader only -- b_full (the P halves'
// bytes), a_full (the eight U-loader warps), acc_empty (the sixteen epilogue warps), arrived
// from the peer through its shared::cluster address.  The arrivals and waits keep the
// default (CTA-scope) semantics: what they order is Tensor Memory and shared memory that the
// tensor cores and TMA reach through the tcgen05 fences and the async proxy.  Every wait is
// bounded; a give-up sets the abort flag of both CTAs and the status word.  Before the
// closing cluster barrier the producers wait for the leader's release of every stage they
// filled, so no commit or copy of the pair arrives in a CTA that has gone.
#include <cuda.h>

#include "zo_kernels.h"
#include "zo_cluster.cuh"
#include "zo_sm100.cuh"
#include "zo_tc_common.cuh"

namespace zo {
namespace {

using namespace sm100;
using namespace tc;
using namespace cta2;

constexpr int kR = 128;
constexpr int kPM = 256;                                   // pair tile rows
constexpr int kHLW = hl_width(kR);                         // 256 per P_HL row: [hi | lo]
constexpr int kPanels = kHLW / 64;                         // 4 panels of 128-byte rows
constexpr int kHalfRows = kBN / 2;                         // 64 P_HL rows per CTA
constexpr int kHalfPanelBytes = kHalfRows * 128;           // 8 KB
constexpr int kHalfOpBytes = kPanels * kHalfPanelBytes;    // 32 KB: this CTA's half P tile
// half P tiles leave room for the W ring of the r = 64 kernel: 4 W + 3 P stages (224 KB), a W
// stage released one tile late so the store's shared-memory reads overlap the next tile
constexpr int kWStages = 4;
constexpr int kBStages = 3;
constexpr bool kDeferRelease = true;
constexpr int kKC = kR / 16;                               // K chunks of 16
constexpr int kACols = kR;                                 // TMEM columns of one U tile
constexpr int kTmemCols = 512;                             // 2 accumulators + 2 U tiles
constexpr int kEpiWarp0 = 2, kEpiWarps = 8;
constexpr int kPWarp = kEpiWarp0 + kEpiWarps;              // lane 0 loads the P half
constexpr int kUWarp0 = kPWarp + 1;
constexpr int kThreads = 32 * (kUWarp0 + 4);
constexpr size_t kSmem = (size_t)kWStages * kWStageBytes + (size_t)kBStages * kHalfOpBytes +
                         1024 /*barriers*/ + 1024 /*align*/;

struct PairShared {
  float w_scale[kWStages];       // scale of the tile in W stage s (see zo_wpass_tc.cu)
  int abort_flag;
  uint64_t w_full[kWStages], w_empty[kWStages];
  uint64_t b_full[kBStages], b_empty[kBStages];
  uint64_t a_full[2], a_empty[2];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t never;                // test hook: a barrier no thread ever arrives on
  uint32_t tmem_base;
};

__device__ __forceinline__ void give_up_pair(PairShared& sh, uint32_t* status) {
  atomicOr(status, (uint32_t)kDevTimeout);
  *reinterpret_cast<volatile int*>(&sh.abort_flag) = 1;
  store_peer(&sh.abort_flag, 1);
}

// The pair tiles of one pair: chunks of kTileChunk consecutive pair tiles b, b + G, ...
// (G pairs); tiles are numbered matrix by matrix, pair row block by pair row block.
struct PairIter {
  const TcMat* mats;
  int n_mats;
  int64_t t, t_end, stride, in_chunk = 0;
  int i;
  int64_t rb, cb;                              // pair row block (256 rows), column block
  __device__ void init(const TcMat* m, int nm, int64_t t0, int64_t t1, int64_t step) {
    mats = m;
    n_mats = nm;
    t = t0;
    t_end = t1;
    stride = step;
    int lo = 0, hi = nm - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (mats[mid].tile0 <= t0) lo = mid; else hi = mid - 1;
    }
    i = lo;
    set_local();
  }
  __device__ void set_local() {
    if (t >= t_end) return;
    const int64_t local = t - mats[i].tile0;
    rb = local / mats[i].tiles_n;
    cb = local % mats[i].tiles_n;
  }
  __device__ bool valid() const { return t < t_end; }
  __device__ void next() {
    if (++in_chunk < kTileChunk) {
      t += 1;
    } else {
      in_chunk = 0;
      t += stride - (kTileChunk - 1);
    }
    if (t >= t_end) return;
    while (i + 1 < n_mats && mats[i + 1].tile0 <= t) ++i;
    set_local();
  }
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
wpass_pair_kernel(const uint4* __restrict__ u_t, const __grid_constant__ CUtensorMap tm_b64,
                  const CUtensorMap* __restrict__ w_maps, const TcMat* __restrict__ mats,
                  const float* __restrict__ pinv, int n_mats, int64_t n_pair_tiles,
                  uint32_t* __restrict__ status, long long wait_cycles, int inject_wait) {
  static_assert(sizeof(PairShared) <= 1024, "barrier block");
  static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
  static_assert(2 * kBN + 2 * kACols <= kTmemCols, "accumulators + U buffers in TMEM");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* w_smem = smem;
  uint8_t* b_smem = w_smem + kWStages * kWStageBytes;
  PairShared& sh = *reinterpret_cast<PairShared*>(b_smem + kBStages * kHalfOpBytes);
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int64_t t_begin = pair * kTileChunk;
  const int64_t t_stride = n_pairs * kTileChunk;
  const volatile int* abort = &sh.abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kWStages; ++s) {
      mbar_init(&sh.w_full[s], 1);
      mbar_init(&sh.w_empty[s], kEpiWarps);
    }
    for (int s = 0; s < kBStages; ++s) {
      mbar_init(&sh.b_full[s], 1);            // the leader's producer (bytes of both halves)
      mbar_init(&sh.b_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sh.a_full[s], 8);            // four U-loader warps in each CTA
      mbar_init(&sh.a_empty[s], 1);
      mbar_init(&sh.acc_full[s], 1);
      mbar_init(&sh.acc_empty[s], 2 * kEpiWarps);
    }
    mbar_init(&sh.never, 1);
    sh.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_b64);
  }
  if (warp == 1) tmem_alloc_pair(&sh.tmem_base, kTmemCols);
  tc_fence_before();
  cluster_sync_all();                          // both CTAs' barriers and TMEM exist
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;

  if (warp == 0 && lane == 0) {
    // ---------------------------------------------------------------- W tiles (this CTA)
    int64_t n_w = 0;
    bool ok = true;
    PairIter ti;
    ti.init(mats, n_mats, t_begin, n_pair_tiles, t_stride);
    for (; ti.valid(); ti.next()) {
      const int s = (int)(n_w % kWStages);
      const uint32_t ph = (uint32_t)((n_w / kWStages) & 1);
      if (!mbar_wait_bounded(&sh.w_empty[s], ph ^ 1u, abort, wait_cycles)) { ok = false; break; }
      sh.w_scale[s] = pinv[ti.i] * exp2i(-kUVScaleExp);
      mbar_arrive_expect_tx(&sh.w_full[s], kWStageBytes);
      uint8_t* dst = w_smem + s * kWStageBytes;
      const int64_t row0 = ti.rb * kPM + kBM * rank;
      for (int g = 0; g < 4; ++g)
        for (int h = 0; h < 2; ++h)
          tma_load_2d(dst + (g * 2 + h) * kWBoxBytes, w_maps + ti.i, (int)(ti.cb * kBN + 64 * h),
                      (int)(row0 + 32 * g), &sh.w_full[s]);
      ++n_w;
    }
    if (!ok) give_up_pair(sh, status);
    for (int s = 0; s < kWStages; ++s) {
      const int64_t k = last_in_slot(n_w, s, kWStages);
      if (k >= 0) mbar_wait_bounded(&sh.w_full[s], (uint32_t)((k / kWStages) & 1), nullptr, wait_cycles);
    }
  } else if (warp == kPWarp && lane == 0) {
    // ---------------------------------------------------------------- P half tiles
    int64_t n_b = 0;
    bool ok = true;
    PairIter ti;
    ti.init(mats, n_mats, t_begin, n_pair_tiles, t_stride);
    for (; ti.valid(); ti.next()) {
      const int s = (int)(n_b % kBStages);
      const uint32_t ph = (uint32_t)((n_b / kBStages) & 1);
      // b_empty is arrived in both CTAs by the leader's commit once the MMAs read the stage
      if (!mbar_wait_bounded(&sh.b_empty[s], ph ^ 1u, abort, wait_cycles)) { ok = false; break; }
      // the leader arms its b_full for both halves; each half's bytes complete there
      if (leader) mbar_arrive_expect_tx(&sh.b_full[s], 2 * kHalfOpBytes);
      const int y = (int)(mats[ti.i].p_row0 + ti.cb * kBN + kHalfRows * rank);
      for (int p = 0; p < kPanels; ++p)
        tma_load_2d_to_leader(b_smem + s * kHalfOpBytes + p * kHalfPanelBytes, &tm_b64, 64 * p, y,
                              &sh.b_full[s]);
      ++n_b;
    }
    if (!ok) give_up_pair(sh, status);
    // tail: the leader's MMAs have released every stage this CTA filled (their commits
    // arrive here, after the copies into it landed)
    for (int s = 0; s < kBStages; ++s) {
      const int64_t k = last_in_slot(n_b, s, kBStages);
      if (k >= 0)
        mbar_wait_bounded(&sh.b_empty[s], (uint32_t)((k / kBStages) & 1), nullptr, wait_cycles);
    }
  } else if (warp >= kUWarp0) {
    // ---------------------------------------------------------------- U rows into TMEM
    // warp w writes TMEM lanes 32 (w % 4) .. + 31 of this CTA's 128-row U block; U_T keeps
    // chunk j of a block's 128 rows contiguous (zo_wpass_tmem.cu) and is padded to 256-row
    // blocks per matrix, so the pair's two blocks are 2 rb and 2 rb + 1
    const int q = warp & 3;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    int64_t n_a = 0;
    int prev_i = -1;
    int64_t prev_rb = -1;
    bool ok = true;
    PairIter ti;
    ti.init(mats, n_mats, t_begin, n_pair_tiles, t_stride);
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
      const int64_t block = mats[ti.i].u_row0 / kBM + 2 * ti.rb + rank;
      const uint4* src = u_t + block * (kR / 4) * kBM + 32 * q + lane;
      const uint32_t col0 = (uint32_t)(2 * kBN + s * kACols);
#pragma unroll
      for (int p0 = 0; p0 < kACols / 32; p0 += 2) {
        // the loads of two 32-column pieces in flight before their stores
        uint32_t v[2][32];
#pragma unroll
        for (int pp = 0; pp < 2; ++pp)
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const uint4 t4 = __ldg(src + ((p0 + pp) * 8 + j) * kBM);
            v[pp][4 * j] = t4.x; v[pp][4 * j + 1] = t4.y; v[pp][4 * j + 2] = t4.z; v[pp][4 * j + 3] = t4.w;
          }
#pragma unroll
        for (int pp = 0; pp < 2; ++pp)
          tmem_st_32x32b_x32(tmem + lane_base + col0 + 32 * (p0 + pp), v[pp]);
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) arrive_leader(&sh.a_full[s]);
      ++n_a;
    }
    if (!ok && lane == 0) give_up_pair(sh, status);
    // tail: the leader's MMAs have released both U buffers this CTA filled
    if (lane == 0)
      for (int s = 0; s < 2; ++s) {
        const int64_t k = last_in_slot(n_a, s, 2);
        if (k >= 0) mbar_wait_bounded(&sh.a_empty[s], (uint32_t)((k >> 1) & 1), nullptr, wait_cycles);
      }
  } else if (warp == 1 && lane == 0 && leader) {
    // ---------------------------------------------------------------- MMA issuer (leader)
    constexpr uint32_t idesc = idesc_f16_f32(kPM, kBN);
    int64_t it = 0, a_it = 0;
    int prev_i = -1;
    int64_t prev_rb = -1;
    int sa = 0;
    bool ok = true;
    PairIter ti, nx;                            // nx runs one tile ahead of ti
    ti.init(mats, n_mats, t_begin, n_pair_tiles, t_stride);
    nx = ti;
    nx.next();
    for (; ti.valid(); ti = nx, nx.next(), ++it) {
      if (ti.i != prev_i || ti.rb != prev_rb) {
        sa = (int)(a_it & 1);
        if (!mbar_wait_bounded(&sh.a_full[sa], (uint32_t)((a_it >> 1) & 1), abort, wait_cycles)) {
          ok = false;
          break;
        }
        ++a_it;
        prev_i = ti.i;
        prev_rb = ti.rb;
      }
      const bool last_a = !nx.valid() || nx.i != ti.i || nx.rb != ti.rb;
      const int sb = (int)(it % kBStages);
      if (!mbar_wait_bounded(&sh.b_full[sb], (uint32_t)((it / kBStages) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_empty[acc], (uint32_t)(((it >> 1) & 1) ^ 1), abort,
                                wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(acc * kBN);
      const uint32_t a_base = tmem + (uint32_t)(2 * kBN + sa * kACols);
      const uint32_t b_base = smem_u32(b_smem + sb * kHalfOpBytes);
      // hi.lo and lo.hi first, hi.hi last (see zo_wpass_tc.cu)
#pragma unroll
      for (int pass = 0; pass < 3; ++pass) {
#pragma unroll
        for (int kk = 0; kk < kKC; ++kk) {
          // U: hi chunk kk at column 8 kk of the buffer, lo chunk at R/2 + 8 kk;
          // P: hi chunk kk at element 16 kk of the operand row, lo chunk at R + 16 kk
          const uint32_t a_t = a_base + (uint32_t)((pass == 1 ? kR / 2 : 0) + 8 * kk);
          const int e_b = (pass == 0 ? kR : 0) + 16 * kk;
          const uint64_t b_d =
              sdesc_k_sw128(b_base + (uint32_t)((e_b / 64) * kHalfPanelBytes + (e_b % 64) * 2));
          mma_pair_ts(d, a_t, b_d, idesc, (pass | kk) != 0 ? 1u : 0u);
        }
      }
      commit_both(&sh.b_empty[sb]);
      if (last_a) commit_both(&sh.a_empty[sa]);
      commit_both(&sh.acc_full[acc]);
    }
    if (!ok) give_up_pair(sh, status);
    if (it > 0) {
      // every MMA of the pair has completed before TMEM is released
      const int64_t last = it - 1;
      mbar_wait_bounded(&sh.acc_full[last & 1], (uint32_t)((last >> 1) & 1), nullptr, wait_cycles);
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ---------------------------------------------------------------- epilogue (each CTA)
    const int g = warp & 3;                      // TMEM lane group == tile row group
    const int h = (warp - kEpiWarp0) >> 2;       // column half
    const uint32_t lane_base = (uint32_t)(g * 32) << 16;
    int s_prev = -1;                             // stage whose release is deferred
    int64_t it = 0;
    bool ok = true;
    PairIter ti;
    ti.init(mats, n_mats, t_begin, n_pair_tiles, t_stride);
    for (; ti.valid(); ti.next(), ++it) {
      const TcMat& mt = mats[ti.i];
      const int acc = (int)(it & 1);
      // test hook (zo_set_option ZO_OPTION_TEST_WAIT_TIMEOUT): CTA 0's epilogue first waits
      // on a barrier that nothing arrives on; the expired wait is reported in the status
      // word and the pass then goes on (the pair's other roles are not stopped)
      if (inject_wait && blockIdx.x == 0 && it == 0 && lane == 0 &&
          !mbar_wait_bounded(&sh.never, 0u, nullptr, wait_cycles))
        atomicOr(status, (uint32_t)kDevTimeout);
      __syncwarp();
      if (!mbar_wait_bounded(&sh.acc_full[acc], (uint32_t)((it >> 1) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int s = (int)(it % kWStages);
      if (!mbar_wait_bounded(&sh.w_full[s], (uint32_t)((it / kWStages) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      uint8_t* stage = w_smem + s * kWStageBytes;
      // the accumulator holds 2^(kUVScaleExp + e_P,i) U P: back to U P in the add
      const uint64_t wscale2 = splat2(sh.w_scale[s]);
      uint32_t v[2][32];
      tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kBN + 64 * h), v[0]);
      tmem_ld_32x32b_x32(tmem + lane_base + (uint32_t)(acc * kBN + 64 * h + 32), v[1]);
      tmem_ld_wait();
      uint8_t* box = stage + (g * 2 + h) * kWBoxBytes;
#pragma unroll
      for (int j = 0; j < 8; ++j) {              // logical 16-byte chunk of the row
        uint4* p = reinterpret_cast<uint4*>(box + lane * 128 + ((j ^ (lane & 7)) << 4));
        uint4 raw = *p;
        uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
        for (int e = 0; e < 4; ++e)
          wv[e] = bf16x2_add_scaled(wv[e], v[j >> 2][(j & 3) * 8 + 2 * e],
                                    v[j >> 2][(j & 3) * 8 + 2 * e + 1], wscale2);
        *p = make_uint4(wv[0], wv[1], wv[2], wv[3]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) arrive_leader(&sh.acc_empty[acc]);
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int64_t y = ti.rb * kPM + kBM * rank + 32 * g;
        const int64_t x = ti.cb * kBN + 64 * h;
        if (y < mt.m && x < mt.n) tma_store_2d(w_maps + ti.i, (int)x, (int)y, box);
        bulk_commit();
        if constexpr (kDeferRelease) {
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
    if (!ok && lane == 0) give_up_pair(sh, status);
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  cluster_sync_all();                          // neither CTA frees TMEM or exits early
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
}

}  // namespace

bool wpass_pair_supported(int32_t r) { return r == kR; }
int32_t pair_tile_rows() { return kPM; }

cudaError_t launch_wpass_pair(const uint4* u_t, const CUtensorMap& tm_b64,
                              const CUtensorMap* d_w_maps, const TcMat* d_tc, const float* d_pinv,
                              int32_t n_mats, int64_t n_pair_tiles, int32_t n_pairs,
                              uint32_t* d_status, bool inject_wait, cudaStream_t s) {
  if (n_pair_tiles <= 0) return cudaSuccess;
  if (n_pairs <= 0) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(wpass_pair_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  if (e != cudaSuccess) return e;
  const long long wait = inject_wait ? kTestWaitCycles : kWaitCycles;
  wpass_pair_kernel<<<2 * n_pairs, kThreads, kSmem, s>>>(u_t, tm_b64, d_w_maps, d_tc, d_pinv,
                                                         n_mats, n_pair_tiles, d_status, wait,
                                                         inject_wait ? 1 : 0);
  return cudaGetLastError();
}

int32_t wpass_pair_max_pairs() {
  // clusters of the pair kernel that fit on the device at once (each pair is persistent
  // over its share of the tiles, so every pair must be resident)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 2;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  if (cudaFuncSetAttribute(wpass_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)kSmem) != cudaSuccess)
    return 0;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, wpass_pair_kernel, &cfg) != cudaSuccess) return 0;
  return clusters;
}

}  // namespace zo
