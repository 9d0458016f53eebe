// The Y GEMM of the perturbed linear layer (Y = X W_i^T + S U_i^T, the forward of Alg. 3
// at W' = W + eps U Z V^T, Eq. (4) form, with W left as it is) on SM pairs: M = 256
// tcgen05.mma.cta_group::2 across the two SMs of a cluster.
//
// Pair tile = 256 rows of X (tokens) x N columns of Y (rows of W_i); CTA c of the cluster
// holds rows 128 c .. 128 c + 127 of the tile (its half of the A operand, its accumulator
// lanes) and rows N/2 c .. N/2 c + N/2 - 1 of the B operand (W rows, then U operand rows);
// the leader's MMAs read both halves of B.  Each SM then stages 128 x 64 + N/2 x 64 bf16
// per 64 elements of K for 128 x N x 64 multiply-adds (two such panels per operand stage,
// three stages), and holds a 128 x N fp32 accumulator -- two of them fit its Tensor Memory
// (N <= 256), so a tile's epilogue runs while the MMAs of the pair's next tile accumulate
// into the other one.
//
// K steps: n / 64 steps of X and W (single bf16 products, both operands exact in bf16),
// then the rank-r term from S_HL = [S_hi | S_lo | 0] (A) and the U operand
// [U_hi | U_lo | 0] (B) with the three products S_hi U_hi + S_hi U_lo + S_lo U_hi.  For
// r <= 32 that is one operand stage holding one 64-wide panel of each, the same MMAs, in
// the same order, as the single-CTA kernels of zo_linear.cu, so each 128-row half of a
// pair tile gets the bits those kernels give; r = 64 takes one stage of two panels (hi,
// lo), r = 128 three stages of two panels (S_hi U_hi, S_hi U_lo, S_lo U_hi).
// S = X P^T comes from S tiles or from contributor tiles in the same launch (see the
// kernel's comment), its rows published through per-writer ready flags.  N (256, 240,
// 224, 192 or 128) is chosen by the host by simulating the launch's schedule
// (linear_pair_tiling).
//
// Roles (320 threads per CTA, one CTA per SM):
//   warp 0, lane 0: TMA producer of this CTA's halves, kStages stages; both halves of a
//                   stage complete their bytes on the leader's full barrier (the TMA's
//                   .cta_group::2 form), which the leader's producer arms for both.
//   warp 1:         Tensor Memory (.cta_group::2, in both CTAs); in the leader lane 0
//                   issues every MMA of the pair into one of two accumulators.
//   warps 2..9:     epilogue of this CTA's 128 rows: warp w reads TMEM lanes 32 (w % 4) ..
//                   + 31, every other 16-column chunk, rounds to bf16 and stores 32 x 16
//                   boxes of Y (32-byte swizzle) by TMA.
// Barriers: in each CTA empty[s], acc_full[a] and s_full[a] (a contributor's S columns;
// arrived in both CTAs by the leader's multicast commits); in the leader full[s] (bytes
// of both halves) and acc_empty[a] (the sixteen epilogue warps of the pair, the peer's
// through its shared::cluster address).
// Every wait is bounded; a give-up sets the abort flag of both CTAs and kDevTimeout in
// the status word, the producers wait (bounded) for the leader's release of every stage
// they filled, the MMA thread for its last MMAs, and TMEM is freed after a cluster barrier.
#include <algorithm>
#include <vector>

#include <cuda.h>

#include "zo_cluster.cuh"
#include "zo_kernels.h"
#include "zo_linear_common.cuh"
#include "zo_sm100.cuh"
#include "zo_tc_common.cuh"

namespace zo {
namespace {

using namespace sm100;
using namespace tc;
using namespace cta2;
using namespace lin;

constexpr int kPairRows = 2 * kBM;   // 256 rows of X per pair tile

template <int N>
struct PairLin {
  static_assert(N % 16 == 0 && N >= 128 && N <= 256, "pair tile columns");
  static constexpr int kHalfN = N / 2;                        // B rows per CTA (multiple of 8)
  static constexpr int kPanels = 2;                           // 64-element K panels per stage
  static constexpr int kAPanel = kBM * 128;                   // 128 rows x 64 bf16
  // a contributor's slice rows per CTA: as many as the accumulator's spare TMEM columns
  // hold (N + 2 x rows <= 256), at most 32
  static constexpr int kSliceRows = (256 - N) / 2 < 32 ? (256 - N) / 2 : 32;
  // B rows per CTA and panel: N/2 rows of W (or of the U operand), then room for a
  // contributor tile's slice of P_K rows, so that one MMA of N + s_cols columns covers both
  static constexpr int kBPanel = (kHalfN + kSliceRows) * 128;
  static constexpr int kABytes = kPanels * kAPanel;
  static constexpr int kStageBytes = kPanels * (kAPanel + kBPanel);  // a multiple of 1024
  static constexpr int kCoreBytes = kPanels * (kAPanel + kHalfN * 128);  // without slices
  static constexpr int kEpiWarps = 8;
  static constexpr int kBoxBytes = 32 * 16 * 2;               // 32 rows x 16 bf16 of Y
  static constexpr int kOutBytes = kEpiWarps * kBoxBytes;
  static constexpr int kStagesFit = (227 * 1024 - kOutBytes - 2048) / kStageBytes;
  static constexpr int kStages = kStagesFit < 8 ? kStagesFit : 8;
  static constexpr int kThreads = 64 + 32 * kEpiWarps;
  static constexpr int kAccStride = 256;                      // TMEM columns between the two
  static constexpr int kTmemCols = 512;
  static constexpr int kChunks = N / 16;                      // 16-column chunks of a row
  static constexpr size_t kSmem = (size_t)kStages * kStageBytes + kOutBytes + 1024 + 1024;
  // an S tile's stage: as many 64-element panels of X and of P_K's r rows as fit a stage,
  // at most 4 (its stages are fewer than a Y tile's, so that it ends before the Y tiles
  // need S)
  template <int R>
  static constexpr int s_panels() {
    return kStageBytes / (kAPanel + R * 128) < 4 ? kStageBytes / (kAPanel + R * 128) : 4;
  }
  // operand stages of a Y tile's rank-r step
  template <int R>
  static constexpr int ext_stages() { return R == 128 ? 3 : 1; }
  static_assert(kStages >= 3, "operand ring");
  static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
  static_assert(kAccStride + N <= kTmemCols, "two accumulators in TMEM");
};

struct LinPairShared {
  uint64_t full[8], empty[8];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t s_full[2];      // a contributor tile's S columns are complete (leader's commit)
  uint64_t drain;          // one commit after the leader's last MMA
  uint32_t tmem_base;
  int abort_flag;
};

// S's flags and counters, kLinearPairCounters words per row block:
//  * [0, 32) ready flags, one per writer of S_HL rows (a warp writing one 32-row group of
//    one slice: flag 8 c + 4 rank + g for contributor c, or 4 rank + g for the row block's S
//    tiles), each set to the call's epoch by a release store once its rows are written.
//    The Y tiles wait until every writer's flag holds their epoch.  No atomics: with a
//    shared counter the writers' compare-and-swap retries serialised (32 of them per row
//    block with four contributors), stalling the Y tiles' rank-r step.
//  * [32 + 4 rank + g] the K ranges of 32-row group g of CTA rank whose fp32 partial rows an
//    S tile has written (s_split > 1), as (call epoch << kCountBits) | count: call e moves
//    it to (e, count + 1), or to (e, 1) from an older call's value, by an acquire-release
//    compare-and-swap at GPU scope (the release publishes the caller's partial row, the
//    acquire shows the others' to the one that completes the group).
// Calls whose T covers fewer row blocks leave other words behind, which the epoch makes
// harmless.
constexpr int kCountBits = 6;
constexpr int kPartialCounter0 = 32;
__device__ __forceinline__ uint32_t count_epoch(uint32_t* f, uint32_t epoch) {
  uint32_t cur;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(cur) : "l"(f) : "memory");
  for (;;) {
    const uint32_t want =
        (cur >> kCountBits) == epoch ? cur + 1 : (epoch << kCountBits) + 1;
    uint32_t prev;
    asm volatile("atom.acq_rel.gpu.global.cas.b32 %0, [%1], %2, %3;"
                 : "=r"(prev) : "l"(f), "r"(cur), "r"(want) : "memory");
    if (prev == cur) return want & ((1u << kCountBits) - 1);
    cur = prev;
  }
}
__device__ __forceinline__ void set_ready(uint32_t* f, uint32_t epoch) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(f), "r"(epoch) : "memory");
}
// every one of the n (<= 32) flags at f holds epoch (bounded; false on abort or timeout).
// Each poll issues the n loads together (relaxed, independent, so they overlap in one L2
// round trip -- acquire loads would complete one after another); once all match, one
// acquire-release fence gives the acquire.
__device__ __forceinline__ bool wait_s_rows(const uint32_t* f, int n, uint32_t epoch,
                                            const volatile int* abort, long long limit_cycles) {
  const long long t0 = clock64();
  for (;;) {
    uint32_t v[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      v[j] = epoch;
      if (j < n)
        asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v[j]) : "l"(f + j) : "memory");
    }
    bool all = true;
#pragma unroll
    for (int j = 0; j < 32; ++j) all = all && v[j] == epoch;
    if (all) {
      asm volatile("fence.acq_rel.gpu;" ::: "memory");
      return true;
    }
    if (*abort) return false;
    if (clock64() - t0 > limit_cycles) return false;
    __nanosleep(64);
  }
}
// generic-proxy global writes <-> later async-proxy (TMA) reads
__device__ __forceinline__ void fence_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ void lp_give_up(LinPairShared& sh, uint32_t* status) {
  atomicOr(status, (uint32_t)kDevTimeout);
  *reinterpret_cast<volatile int*>(&sh.abort_flag) = 1;
  store_peer(&sh.abort_flag, 1);
}

// 32 lanes x 16 consecutive 32-bit columns: thread t gets lane (base lane + t)
__device__ __forceinline__ void tmem_ld_32x32b_x16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15])
      : "r"(taddr));
}

// Columns kC j .. kC j + kC - 1 of S for this thread's row (kC = min(R, 32)): the sum of
// the accumulator's X P_hi^T and X P_lo^T columns.  Warp-collective.
template <int R>
__device__ __forceinline__ void load_s_chunk(uint32_t t_base, int j, float (&x)[R < 32 ? R : 32]) {
  uint32_t v[32];
  tmem_ld_32x32b_x32(t_base + (uint32_t)(32 * j), v);
  if constexpr (R == 16) {
    tmem_ld_wait();
#pragma unroll
    for (int q = 0; q < 16; ++q) x[q] = __uint_as_float(v[q]) + __uint_as_float(v[16 + q]);
  } else {
    uint32_t w[32];
    tmem_ld_32x32b_x32(t_base + (uint32_t)(R + 32 * j), w);
    tmem_ld_wait();
#pragma unroll
    for (int q = 0; q < 32; ++q) x[q] = __uint_as_float(v[q]) + __uint_as_float(w[q]);
  }
}

// A contributor's S slice for this thread's row: S's columns half_s nb .. + half_s - 1
// (half_s = 16 or 32) are the sums of the accumulator's columns t_hi + j (X P_hi^T) and
// t_lo + j (X P_lo^T); their hi and lo groups go to the S_HL row (the zero groups past 2R
// with the first slice).  Warp-collective.
template <int R>
__device__ __forceinline__ void write_s_slice(uint32_t t_hi, uint32_t t_lo, int half_s, int nb,
                                              __nv_bfloat16* s_hl, int row, bool valid) {
  float x[32];
  if (half_s == 16) {
    uint32_t v[16], w[16];
    tmem_ld_32x32b_x16(t_hi, v);
    tmem_ld_32x32b_x16(t_lo, w);
    tmem_ld_wait();
#pragma unroll
    for (int j = 0; j < 16; ++j) x[j] = __uint_as_float(v[j]) + __uint_as_float(w[j]);
  } else {
    uint32_t v[32], w[32];
    tmem_ld_32x32b_x32(t_hi, v);
    tmem_ld_32x32b_x32(t_lo, w);
    tmem_ld_wait();
#pragma unroll
    for (int j = 0; j < 32; ++j) x[j] = __uint_as_float(v[j]) + __uint_as_float(w[j]);
  }
  if (!valid) return;
  uint4* out = reinterpret_cast<uint4*>(s_hl + (int64_t)row * hl_width(R));
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    if (8 * g < half_s) {
      float c[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) c[e] = 0.f + x[8 * g + e];
      uint4 hi, lo;
      split8(c, hi, lo);
      out[(nb * half_s) / 8 + g] = hi;
      out[(R + nb * half_s) / 8 + g] = lo;
    }
  }
  if (nb == 0) zero_s_pad<R>(s_hl, row);
}

// Pair tile t -> (row block tb, column block nb): column stripes of `group` column blocks,
// each walked row block by row block (group = the column blocks: plain row-major order).
// Stripes about one wave of tiles wide keep the wave's W rows few enough to stay in L2
// while every row block of X passes them.
struct StripeOrder {
  int tiles_n, row_blocks, group;
  __device__ void decode(int64_t t, int& tb, int& nb) const {
    const int64_t per = (int64_t)row_blocks * group;
    const int full = tiles_n / group;
    if (t < (int64_t)full * per) {
      const int stripe = (int)(t / per), rem = (int)(t % per);
      tb = rem / group;
      nb = stripe * group + rem % group;
    } else {
      const int rem = (int)(t - (int64_t)full * per);
      const int last = tiles_n - full * group;
      tb = rem / last;
      nb = full * group + rem % last;
    }
  }
};

// The launch's tiles: first s_split S tiles per row block (S = X P^T for its 256 rows over
// one of s_split K ranges: with one range its S_HL rows directly, else fp32 partial rows
// that the last range of each 32-row group sums), then the Y tiles in stripe order.
struct PairTiles {
  int row_blocks, s_split;
  StripeOrder order;
  // true: an S tile of row block tb over K range nb
  __device__ bool decode(int64_t t, int& tb, int& nb) const {
    const int64_t n_s = (int64_t)row_blocks * s_split;
    if (t < n_s) {
      tb = (int)(t % row_blocks);
      nb = (int)(t / row_blocks);
      return true;
    }
    order.decode(t - n_s, tb, nb);
    return false;
  }
};

// tm_x: X (box 64 x 128), tm_w: W_i (box 64 x N/2), tm_s: S_HL (box 64 x 128), tm_u: the
// route's U operand (box 64 x N/2; this matrix's rows from u_row0), tm_y: Y (box 16 x 32,
// 32-byte swizzle), tm_pk: P_K = [P_hi ; P_lo] (box 64 x R: CTA c loads rows R c ..),
// tm_ps: P_K in boxes of s_cols / 2 rows (the contributor tiles' slices).  rows = T, cols =
// m, k_steps = ceil(n / 64).  S comes one of two ways:
//  * n_contrib > 0 (contributor tiles; s_split = 0): the Y tiles of column blocks
//    0 .. n_contrib - 1 of each row block (consecutive in the tile order, the first of their
//    stripe) also compute S's columns s_cols/2 nb .. + s_cols/2 - 1 over all of K, in the
//    same MMAs as their dense product: each CTA's B rows are its N/2 rows of W followed by
//    s_cols / 2 rows of P_hi (CTA 0) or P_lo (CTA 1), and the MMAs are N + s_cols wide (a
//    separate narrow MMA per K step cost far more than its columns).  Their epilogues
//    write those S_HL columns and set their ready flags (n_contrib x 8 complete a row
//    block's S); their Y columns from N/2 on sit s_cols / 2 accumulator columns further.
//  * else S tiles first: s_split per row block over K ranges of s_chunk 64-element panels
//    each (one range at r <= 64, so that every pair tiling sums S in the contributors'
//    order; at r = 128 the same ranges for every N), then the Y tiles in stripe order.
// s_hl: the S_HL rows; s_part: s_split x rows x R fp32 partial rows (s_split > 1); s_count:
// kLinearPairCounters flags and counters per row block; epoch: this call's (1 .. 2^26 - 1),
// which S's writers count with; wait_epoch: the one its Y tiles wait for (= epoch; the test
// hook passes one that never comes, so that every Y tile's bounded wait runs out).
template <int N, int R>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PairLin<N>::kThreads, 1)
linear_pair_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                   const __grid_constant__ CUtensorMap tm_s, const __grid_constant__ CUtensorMap tm_u,
                   const __grid_constant__ CUtensorMap tm_y, const __grid_constant__ CUtensorMap tm_pk,
                   const __grid_constant__ CUtensorMap tm_ps,
                   int rows, int cols, int k_steps, int u_row0, int group, int s_split,
                   int s_chunk, int n_contrib, int s_cols,
                   __nv_bfloat16* __restrict__ s_hl, float* __restrict__ s_part,
                   uint32_t* __restrict__ s_count,
                   uint32_t epoch, uint32_t wait_epoch, uint32_t* __restrict__ status,
                   long long wait_cycles) {
  using Cfg = PairLin<N>;
  constexpr int S = Cfg::kStages;
  constexpr int kSP = Cfg::template s_panels<R>();            // panels per S-tile stage
  constexpr int kExt = Cfg::template ext_stages<R>();         // stages of the rank-r step
  static_assert(R == 16 || R == 32 || R == 64 || R == 128, "rank");
  static_assert(kSP >= 1, "S-tile stage");
  static_assert(2 * R <= Cfg::kAccStride, "an S tile's 2 r accumulator columns");
  static_assert(sizeof(LinPairShared) <= 1024, "barrier block");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* st_smem = smem;                                    // stages: [A | B | slice]
  uint8_t* o_smem = st_smem + S * Cfg::kStageBytes;           // one Y box per epilogue warp
  LinPairShared& sh = *reinterpret_cast<LinPairShared*>(o_smem + Cfg::kOutBytes);

  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int tiles_n = (cols + N - 1) / N;
  const int row_blocks = (rows + kPairRows - 1) / kPairRows;
  const int64_t n_tiles = (int64_t)row_blocks * (tiles_n + s_split);
  const PairTiles tiles{row_blocks, s_split,
                        StripeOrder{tiles_n, row_blocks, group < 1 || group > tiles_n ? tiles_n : group}};
  const volatile int* abort = &sh.abort_flag;
  // S's writers per row block: 8 32-row groups from each contributor, or from its S tiles
  const int s_writers = (int)kLinearPairCountsPerCall * (n_contrib > 0 ? n_contrib : 1);
  const int half_s = s_cols / 2;                              // a slice's P_K rows per CTA
  // a contributor tile: one of the first n_contrib column blocks of its row block
  auto contributor = [&](bool s_tile, int nb) { return !s_tile && nb < n_contrib; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&sh.full[s], 1);              // the leader's producer (bytes of both halves)
      mbar_init(&sh.empty[s], 1);             // the leader's commit
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sh.acc_full[a], 1);
      mbar_init(&sh.acc_empty[a], 2 * Cfg::kEpiWarps);
      mbar_init(&sh.s_full[a], 1);
    }
    mbar_init(&sh.drain, 1);
    sh.abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_x);
    prefetch_tmap(&tm_w);
    prefetch_tmap(&tm_s);
    prefetch_tmap(&tm_u);
    prefetch_tmap(&tm_y);
    prefetch_tmap(&tm_pk);
    prefetch_tmap(&tm_ps);
  }
  if (warp == 1) tmem_alloc_pair(&sh.tmem_base, Cfg::kTmemCols);
  tc_fence_before();
  cluster_sync_all();                         // both CTAs' barriers and TMEM exist
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;
  // launched as a programmatic dependent of the stream's previous kernel: the prologue
  // above overlaps that kernel's tail; everything below reads or writes memory it may use
  // (X, S_HL, the flags, Y), so wait for its completion.  Then let the stream's next
  // kernel be scheduled as SMs free up (it waits the same way).
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer (each CTA)
    int s = 0;
    uint32_t ph = 0;
    int64_t n_st = 0;
    bool ok = true;
    const int k_stages = (k_steps + Cfg::kPanels - 1) / Cfg::kPanels;
    for (int64_t tile = pair; tile < n_tiles && ok; tile += n_pairs) {
      int tb, nb;
      const bool s_tile = tiles.decode(tile, tb, nb);
      const int y_a = tb * kPairRows + kBM * (int)rank;
      const int y_b = nb * N + Cfg::kHalfN * (int)rank;
      // an S tile's K range (nb = the range; stages of up to kSP panels) or a Y tile's K
      // steps and its rank-r step
      const int p_lo = s_tile ? nb * s_chunk : 0;
      const int p_hi = s_tile ? min(k_steps, p_lo + s_chunk) : 0;
      const int n_k = s_tile ? (p_hi - p_lo + kSP - 1) / kSP : k_stages + kExt;
      for (int k = 0; k < n_k; ++k) {
        if (!mbar_wait_bounded(&sh.empty[s], ph ^ 1u, abort, wait_cycles)) {
          ok = false;
          break;
        }
        uint8_t* a_dst = st_smem + s * Cfg::kStageBytes;
        uint8_t* b_dst = a_dst + Cfg::kABytes;
        if (s_tile) {
          // kSP panels of X, then this CTA's R rows of P_K for each (P_hi in CTA 0, P_lo in
          // CTA 1); panels past n read TMA's zero fill
          const int pb = p_lo + kSP * k, np = min(kSP, p_hi - pb);
          if (leader) mbar_arrive_expect_tx(&sh.full[s], 2u * np * (Cfg::kAPanel + R * 128));
          for (int p = 0; p < np; ++p) {
            const int x = 64 * (pb + p);
            tma_load_2d_to_leader(a_dst + p * Cfg::kAPanel, &tm_x, x, y_a, &sh.full[s]);
            tma_load_2d_to_leader(a_dst + kSP * Cfg::kAPanel + p * R * 128, &tm_pk, x, R * (int)rank,
                                  &sh.full[s]);
          }
        } else if (k < k_stages) {
          // panels past n read TMA's zero fill; a contributor also loads its S slice's
          // P_K rows (P_hi rows in CTA 0, P_lo rows in CTA 1)
          const bool contrib = contributor(s_tile, nb);
          if (leader)
            mbar_arrive_expect_tx(&sh.full[s], 2u * (Cfg::kCoreBytes +
                                                     (contrib ? Cfg::kPanels * half_s * 128 : 0)));
#pragma unroll
          for (int p = 0; p < Cfg::kPanels; ++p) {
            const int x = 64 * (Cfg::kPanels * k + p);
            tma_load_2d_to_leader(a_dst + p * Cfg::kAPanel, &tm_x, x, y_a, &sh.full[s]);
            tma_load_2d_to_leader(b_dst + p * Cfg::kBPanel, &tm_w, x, y_b, &sh.full[s]);
            if (contrib)
              tma_load_2d_to_leader(b_dst + p * Cfg::kBPanel + Cfg::kHalfN * 128, &tm_ps, x,
                                    R * (int)rank + nb * half_s, &sh.full[s]);
          }
        } else {                               // the rank-r step: S_HL rows, U operand rows
          const int j = k - k_stages;
          if (j == 0) {
            // this row block's S rows: written by its S tile (both CTAs' epilogues) earlier
            // in this launch
            if (!wait_s_rows(s_count + (int64_t)tb * kLinearPairCounters, s_writers, wait_epoch,
                             abort, wait_cycles)) {
              ok = false;
              break;
            }
            fence_async_global();
          }
          if constexpr (R <= 32) {
            // one 64-wide panel of each: [hi | lo | 0]
            if (leader) mbar_arrive_expect_tx(&sh.full[s], 2u * (Cfg::kAPanel + Cfg::kHalfN * 128));
            tma_load_2d_to_leader(a_dst, &tm_s, 0, y_a, &sh.full[s]);
            tma_load_2d_to_leader(b_dst, &tm_u, 0, u_row0 + y_b, &sh.full[s]);
          } else {
            // two panels of each, from S_HL columns sx, sx + 64 and U columns ux, ux + 64:
            // r = 64 the hi and the lo panel of both; r = 128 the hi panels (stage 0), the
            // hi panels of S and the lo ones of U (stage 1), the lo ones of S and the hi ones
            // of U (stage 2)
            const int sx = j == 2 ? R : 0, ux = j == 1 ? R : 0;
            if (leader) mbar_arrive_expect_tx(&sh.full[s], 2u * Cfg::kCoreBytes);
#pragma unroll
            for (int p = 0; p < 2; ++p) {
              tma_load_2d_to_leader(a_dst + p * Cfg::kAPanel, &tm_s, sx + 64 * p, y_a, &sh.full[s]);
              tma_load_2d_to_leader(b_dst + p * Cfg::kBPanel, &tm_u, ux + 64 * p, u_row0 + y_b,
                                    &sh.full[s]);
            }
          }
        }
        ++n_st;
        if (++s == S) { s = 0; ph ^= 1u; }
      }
    }
    if (!ok) lp_give_up(sh, status);
    // tail: the leader's MMAs have released every stage this CTA filled
    for (int q = 0; q < S; ++q) {
      const int64_t k = last_in_slot(n_st, q, S);
      if (k >= 0) mbar_wait_bounded(&sh.empty[q], (uint32_t)((k / S) & 1), nullptr, wait_cycles);
    }
  } else if (warp == 1 && lane == 0 && leader) {
    // ------------------------------------------------------------ MMA issuer (leader)
    constexpr uint32_t idesc_s = idesc_bf16_f32(kPairRows, 2 * R);
    // a Y tile's MMAs: N columns, a contributor's N + s_cols (its B rows per CTA: N/2 of W
    // or U, then half_s slice rows; D's columns [0, N/2) W rows of CTA 0, [N/2, N/2 +
    // half_s) its P_hi slice, [N/2 + half_s, N + half_s) W rows of CTA 1, then its P_lo
    // slice)
    const uint32_t idesc_y = idesc_bf16_f32(kPairRows, N);
    const uint32_t idesc_c = idesc_bf16_f32(kPairRows, N + (s_cols > 0 ? s_cols : 0));
    // descriptors advance by their 16-byte address units: 32 bytes per K = 16 step, one
    // panel per 64 elements of K
    constexpr uint64_t kStepK = 32 >> 4, kPanelA = Cfg::kAPanel >> 4, kPanelB = Cfg::kBPanel >> 4;
    const int k_stages = (k_steps + Cfg::kPanels - 1) / Cfg::kPanels;
    int s = 0;
    uint32_t ph = 0;
    int64_t n_st = 0, it = 0;
    bool ok = true;
    for (int64_t tile = pair; tile < n_tiles && ok; tile += n_pairs, ++it) {
      int tb, nb;
      const bool s_tile = tiles.decode(tile, tb, nb);
      const int acc = (int)(it & 1);
      if (!mbar_wait_bounded(&sh.acc_empty[acc], (uint32_t)(((it >> 1) & 1) ^ 1), abort,
                             wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();                          // the epilogue's reads of this accumulator
      const uint32_t d = tmem + (uint32_t)(acc * Cfg::kAccStride);
      const int p_lo = s_tile ? nb * s_chunk : 0;
      const int p_hi = s_tile ? min(k_steps, p_lo + s_chunk) : 0;
      const int n_k = s_tile ? (p_hi - p_lo + kSP - 1) / kSP : k_stages + kExt;
      const bool contrib = contributor(s_tile, nb);
      const uint32_t idesc = contrib ? idesc_c : idesc_y;
      for (int k = 0; k < n_k; ++k) {
        // the operands arrive by TMA on this barrier: its wait orders the MMAs' reads
        if (!mbar_wait_bounded(&sh.full[s], ph, abort, wait_cycles)) {
          ok = false;
          break;
        }
        // a contributor's rank-r step adds into the columns of its slice too (garbage
        // there, read no more): its epilogue has read them before the S rows it waited for
        // were ready, which this stage's operands waited for
        if (contrib && k == k_stages) tc_fence_after();
        const uint64_t a0 = sdesc_k_sw128(smem_u32(st_smem + s * Cfg::kStageBytes));
        const uint64_t b0 = sdesc_k_sw128(smem_u32(st_smem + s * Cfg::kStageBytes + Cfg::kABytes));
        if (s_tile) {
          // D[:, :R] = X P_hi^T, D[:, R:2R] = X P_lo^T; the P_K panels follow the kSP X panels
          const uint64_t bs = a0 + kSP * kPanelA;
          const int np = min(kSP, p_hi - (p_lo + kSP * k));
          for (int p = 0; p < np; ++p)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_pair_ss(d, a0 + p * kPanelA + kk * kStepK, bs + p * (R * 128 >> 4) + kk * kStepK,
                          idesc_s, (k > 0 || p > 0 || kk > 0) ? 1u : 0u);
        } else if (k < k_stages) {
#pragma unroll
          for (int p = 0; p < Cfg::kPanels; ++p)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_pair_ss(d, a0 + p * kPanelA + kk * kStepK, b0 + p * kPanelB + kk * kStepK, idesc,
                          (k > 0 || p > 0 || kk > 0) ? 1u : 0u);
        } else if constexpr (R <= 32) {
          // hi chunk kk at element 16 kk of an operand row, lo chunk at R + 16 kk
#pragma unroll
          for (int kk = 0; kk < R / 16; ++kk) {
            const uint64_t hi = kk * kStepK, lo = (R / 16 + kk) * kStepK;
            mma_pair_ss(d, a0 + hi, b0 + hi, idesc, 1u);
            mma_pair_ss(d, a0 + hi, b0 + lo, idesc, 1u);
            mma_pair_ss(d, a0 + lo, b0 + hi, idesc, 1u);
          }
        } else if constexpr (R == 64) {
          // panel 0 holds the hi chunks, panel 1 the lo ones
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t st = kk * kStepK;
            mma_pair_ss(d, a0 + st, b0 + st, idesc, 1u);
            mma_pair_ss(d, a0 + st, b0 + kPanelB + st, idesc, 1u);
            mma_pair_ss(d, a0 + kPanelA + st, b0 + st, idesc, 1u);
          }
        } else {
          // one of the three products over its 128 elements of K
#pragma unroll
          for (int p = 0; p < 2; ++p)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_pair_ss(d, a0 + p * kPanelA + kk * kStepK, b0 + p * kPanelB + kk * kStepK,
                          idesc, 1u);
        }
        commit_both(&sh.empty[s]);
        // a contributor's S columns are complete after its last dense K step
        if (contrib && k == k_stages - 1) commit_both(&sh.s_full[acc]);
        ++n_st;
        if (++s == S) { s = 0; ph ^= 1u; }
      }
      if (!ok) break;
      commit_both(&sh.acc_full[acc]);
    }
    if (!ok) lp_give_up(sh, status);
    if (n_st > 0) {
      // every MMA of the pair -- a tile left half-way included -- has completed before
      // TMEM is released
      commit_both(&sh.drain);
      mbar_wait_bounded(&sh.drain, 0u, nullptr, wait_cycles);
    }
  } else if (warp >= 2 && warp < 2 + Cfg::kEpiWarps) {
    // ------------------------------------------------------------ epilogue (each CTA)
    const int e = warp - 2;
    const int g = warp & 3;                      // TMEM lane group == rows 32 g .. + 31
    const int h = e >> 2;                        // chunks h, h + 2, ...
    const uint32_t lane_base = (uint32_t)(g * 32) << 16;
    uint8_t* box = o_smem + e * Cfg::kBoxBytes;
    int64_t it = 0;
    uint32_t sfull_ph = 0;                       // bit a: s_full[a]'s next phase parity
    bool ok = true;
    for (int64_t tile = pair; tile < n_tiles; tile += n_pairs, ++it) {
      int tb, nb;
      const bool s_tile = tiles.decode(tile, tb, nb);
      const int acc = (int)(it & 1);
      const int y = tb * kPairRows + kBM * (int)rank + 32 * g;
      const uint32_t t_base = tmem + lane_base + (uint32_t)(acc * Cfg::kAccStride);
      if (contributor(s_tile, nb) && h == 0) {
        // this tile's S slice, before its rank-r step (which waits for every slice of the
        // row block): four warps per CTA, one per TMEM lane group
        if (!mbar_wait_bounded(&sh.s_full[acc], (sfull_ph >> acc) & 1u, abort, wait_cycles)) {
          ok = false;
          break;
        }
        sfull_ph ^= 1u << acc;
        tc_fence_after();
        write_s_slice<R>(t_base + (uint32_t)(N / 2), t_base + (uint32_t)(N + half_s), half_s, nb,
                         s_hl, y + lane, y + lane < rows);
        tc_fence_before();                       // before the rank-r step's MMAs
        fence_async_global();
        __threadfence();
        __syncwarp();
        if (lane == 0)
          set_ready(s_count + (int64_t)tb * kLinearPairCounters + 8 * nb + 4 * (int)rank + g, epoch);
      }
      if (!mbar_wait_bounded(&sh.acc_full[acc], (uint32_t)((it >> 1) & 1), abort, wait_cycles)) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (s_tile) {
        // this K range's S = D[:, :R] + D[:, R:2R] for this lane's row; four warps per CTA
        // (one per TMEM lane group).  One range: the S_HL row directly.  Several: the fp32
        // partial row, and the warp that completes its 32-row group's ranges sums them in
        // range order and writes the S_HL rows.  Then the group's ready flag is set.
        if (h == 0) {
          // kC columns of S at a time (D[:, kC j ..] + D[:, R + kC j ..])
          constexpr int kC = R < 32 ? R : 32;
          const int row = y + lane;
          uint32_t* cnt = s_count + (int64_t)tb * kLinearPairCounters;
          float* part_row = s_part + ((int64_t)nb * rows + row) * R;
#pragma unroll 1
          for (int j = 0; j < R / kC; ++j) {
            float x[kC];
            load_s_chunk<R>(t_base, j, x);
            if (j == R / kC - 1) {                   // this warp's last read of the accumulator
              tc_fence_before();
              __syncwarp();
              if (lane == 0) arrive_leader(&sh.acc_empty[acc]);
            }
            if (row < rows) {
              if (s_split > 1) {
                float4* dst = reinterpret_cast<float4*>(part_row + kC * j);
#pragma unroll
                for (int q = 0; q < kC / 4; ++q)
                  dst[q] = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
              } else {
#pragma unroll
                for (int q = 0; q < kC; ++q) x[q] = 0.f + x[q];
                write_s_chunk<R>(s_hl, row, j, x);
              }
            }
          }
          bool last = true;
          if (s_split > 1) {
            __threadfence();
            __syncwarp();
            uint32_t n_done = 0;
            if (lane == 0) n_done = count_epoch(cnt + kPartialCounter0 + 4 * (int)rank + g, epoch);
            n_done = __shfl_sync(0xffffffffu, n_done, 0);
            last = n_done == (uint32_t)s_split;
            if (last && row < rows) {
#pragma unroll 1
              for (int j = 0; j < R / kC; ++j) {
                float x[kC];
#pragma unroll
                for (int q = 0; q < kC; ++q) x[q] = 0.f;
                for (int ks = 0; ks < s_split; ++ks) {
                  const float4* src = reinterpret_cast<const float4*>(
                      s_part + ((int64_t)ks * rows + row) * R + kC * j);
#pragma unroll
                  for (int q = 0; q < kC / 4; ++q) {
                    const float4 p4 = __ldcg(src + q);
                    x[4 * q] += p4.x;
                    x[4 * q + 1] += p4.y;
                    x[4 * q + 2] += p4.z;
                    x[4 * q + 3] += p4.w;
                  }
                }
                write_s_chunk<R>(s_hl, row, j, x);
              }
            }
          }
          if (last) {
            if (row < rows) zero_s_pad<R>(s_hl, row);
            fence_async_global();
            __threadfence();
            __syncwarp();
            if (lane == 0) set_ready(cnt + 4 * (int)rank + g, epoch);
          }
        } else {
          __syncwarp();
          if (lane == 0) arrive_leader(&sh.acc_empty[acc]);
        }
        continue;
      }
      // a contributor's Y columns from N/2 on sit half_s columns further (after its P_hi
      // slice)
      const int shift = contributor(s_tile, nb) ? half_s : 0;
#pragma unroll 1
      for (int c = h; c < Cfg::kChunks; c += 2) {
        uint32_t v[16];
        tmem_ld_32x32b_x16(t_base + (uint32_t)(16 * c + (16 * c >= Cfg::kHalfN ? shift : 0)), v);
        tmem_ld_wait();
        if (c + 2 >= Cfg::kChunks) {             // this warp's last read of the accumulator
          tc_fence_before();
          __syncwarp();
          if (lane == 0) arrive_leader(&sh.acc_empty[acc]);
        }
        if (lane == 0) bulk_wait_read_all();     // the box's previous store has read it
        __syncwarp();
        uint32_t w[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const __nv_bfloat162 b2 =
              __floats2bfloat162_rn(__uint_as_float(v[2 * q]), __uint_as_float(v[2 * q + 1]));
          w[q] = *reinterpret_cast<const uint32_t*>(&b2);
        }
        // 16-byte chunk j of row `lane` (32-byte rows): 32-byte swizzle, chunk ^ (row / 4) % 2
#pragma unroll
        for (int j = 0; j < 2; ++j)
          *reinterpret_cast<uint4*>(box + lane * 32 + ((j ^ ((lane >> 2) & 1)) << 4)) =
              make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
        fence_async_smem();
        __syncwarp();
        if (lane == 0) {
          const int x = nb * N + 16 * c;
          if (y < rows && x < cols) tma_store_2d(&tm_y, x, y, box);
          bulk_commit();
        }
        __syncwarp();
      }
    }
    if (!ok && lane == 0) lp_give_up(sh, status);
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  cluster_sync_all();                          // neither CTA frees TMEM or exits early
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, Cfg::kTmemCols);
  }
}

template <int N, int R>
cudaError_t launch_pair_nr(const CUtensorMap& tm_x, const CUtensorMap& tm_w,
                           const CUtensorMap& tm_s, const CUtensorMap& tm_u,
                           const CUtensorMap& tm_y, const CUtensorMap& tm_pk,
                           const CUtensorMap& tm_ps, int rows, int cols, int k_steps, int u_row0,
                           const LinearPairPlan& plan, __nv_bfloat16* s_hl, float* s_part,
                           uint32_t* s_count, uint32_t epoch, bool inject_wait,
                           uint32_t* d_status, cudaStream_t s) {
  using Cfg = PairLin<N>;
  // a contributor's TMEM reads stay aligned to their widths: slices of 16 or 32 rows per
  // CTA, N/2 a multiple of the slice rows
  if (plan.n_contrib > 0 && (plan.s_cols / 2 > Cfg::kSliceRows ||
                             (plan.s_cols != 32 && plan.s_cols != 64) ||
                             Cfg::kHalfN % (plan.s_cols / 2) != 0))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(linear_pair_kernel<N, R>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)Cfg::kSmem);
  if (e != cudaSuccess) return e;
  // a programmatic dependent launch: the kernel's prologue may start before the stream's
  // previous kernel ends (the kernel waits for it before touching memory)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * plan.pairs, 1, 1);
  cfg.blockDim = dim3(Cfg::kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const uint32_t wait_epoch = inject_wait ? epoch + 1 : epoch;
  const long long wait_limit = inject_wait ? kTestWaitCycles : kWaitCycles;
  e = cudaLaunchKernelEx(&cfg, linear_pair_kernel<N, R>, tm_x, tm_w, tm_s, tm_u, tm_y, tm_pk,
                         tm_ps, rows, cols, k_steps, u_row0, (int)plan.group, (int)plan.s_split,
                         (int)plan.s_chunk, (int)plan.n_contrib, (int)plan.s_cols, s_hl, s_part,
                         s_count, epoch, wait_epoch, d_status, wait_limit);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int N>
int max_pairs_n() {
  using Cfg = PairLin<N>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2, 1, 1);
  cfg.blockDim = dim3(Cfg::kThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 2;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  if (cudaFuncSetAttribute(linear_pair_kernel<N, 32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)Cfg::kSmem) != cudaSuccess)
    return 0;
  int clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&clusters, linear_pair_kernel<N, 32>, &cfg) != cudaSuccess)
    return 0;
  return clusters;
}

constexpr int kPairCols[] = {256, 240, 224, 192, 128};

}  // namespace

int32_t linear_pair_cols(int32_t tiling) {
  return tiling >= kLinearPairTiling0 && tiling < kLinearPairTiling0 + 5
             ? kPairCols[tiling - kLinearPairTiling0]
             : 0;
}

int32_t linear_pair_max_pairs() {
  // every N has the same threads and (within a stage) the same shared-memory class: one
  // CTA per SM; the smallest count over the tilings is the safe one
  int p = max_pairs_n<256>();
  p = std::min(p, max_pairs_n<240>());
  p = std::min(p, max_pairs_n<224>());
  p = std::min(p, max_pairs_n<192>());
  p = std::min(p, max_pairs_n<128>());
  return p;
}

namespace {
int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
// PairLin<N>'s slice rows, stage bytes and S-tile panels per stage, on the host
int64_t slice_rows_host(int64_t N) { return std::min<int64_t>(32, (256 - N) / 2); }
int64_t core_bytes_host(int64_t N) { return 2 * (kBM * 128 + N / 2 * 128); }
int s_panels_host(int64_t N, int32_t r) {
  const int64_t stage = core_bytes_host(N) + 2 * slice_rows_host(N) * 128;
  return (int)std::min<int64_t>(4, stage / (kBM * 128 + (int64_t)r * 128));
}
}  // namespace

LinearPairPlan linear_pair_plan(int64_t T, int64_t m, int64_t n, int32_t r, int32_t tiling,
                                int32_t n_pairs) {
  LinearPairPlan pl{};
  const int64_t N = linear_pair_cols(tiling);
  if (N == 0 || n_pairs <= 0 || T <= 0 || m <= 0 || n <= 0) return pl;
  const int64_t panels = ceil_div(n, 64);
  const int64_t row_blocks = ceil_div(T, kPairRows);
  const int64_t tiles_n = ceil_div(m, N);
  const int64_t y_tiles = row_blocks * tiles_n;
  if (r <= 64) {
    // contributors: n_contrib column blocks per row block, each S's 2r / n_contrib = 32 or
    // 64 columns (16 or 32 slice rows per CTA, within the accumulator's spare columns, N/2
    // a multiple of them so that the epilogue's TMEM reads stay aligned); as many as the
    // row block's column blocks allow, up to 4 (the slices' extra MMA time falls on more
    // tiles but less on each).  The launch's pair count is a multiple of n_contrib unless
    // every tile runs at once, so that no row block's contributors straddle two waves.
    const int64_t pairs = std::min<int64_t>(y_tiles, n_pairs);
    for (int nc : {4, 2, 1}) {
      const int sc = 2 * r / nc;
      if ((sc != 32 && sc != 64) || sc / 2 > slice_rows_host(N) || (N / 2) % (sc / 2) != 0 ||
          nc > tiles_n)
        continue;
      if (pairs < y_tiles && pairs % nc != 0) continue;
      pl.n_contrib = nc;
      pl.s_cols = sc;
      break;
    }
    // else S tiles over one K range: S summed in the contributors' order, so that every
    // pair tiling of a call gives the same S
    pl.s_split = pl.n_contrib > 0 ? 0 : 1;
    pl.s_chunk = (int32_t)panels;
  } else {
    // S tiles: about one per pair, K ranges of s_chunk 64-element panels (a multiple of 6,
    // so that stages of 2 or 3 panels divide them, where K allows), every range non-empty,
    // at most 15 (the partial counters' count field); the same for every tile width
    const int64_t want =
        std::max<int64_t>(1, std::min<int64_t>({n_pairs / row_blocks, panels, 15}));
    int64_t chunk = ceil_div(panels, want);
    if (chunk > 6) chunk = ceil_div(chunk, 6) * 6;
    pl.s_chunk = (int32_t)chunk;
    pl.s_split = (int32_t)ceil_div(panels, chunk);
  }
  const int64_t tiles = row_blocks * (tiles_n + pl.s_split);
  pl.pairs = (int32_t)std::min<int64_t>(tiles, n_pairs);
  // column stripes as wide as one wave of pairs spread over every row block: a wave then
  // shares its few W rows across all of X (measured on the LLaMA-7B shapes: 4 column blocks
  // per stripe at 4096 tokens beat row-major order by 4% (4096 x 4096), 15% (11008 x 4096)
  // and 2% (4096 x 11008)); with contributors a multiple of n_contrib, so that a row
  // block's contributors are consecutive tiles
  int64_t group = std::max<int64_t>(1, pl.pairs / row_blocks);
  if (pl.n_contrib > 0) group = std::max<int64_t>(pl.n_contrib, group / pl.n_contrib * pl.n_contrib);
  pl.group = (int32_t)group;
  return pl;
}

int32_t linear_pair_tiling(int64_t T, int64_t m, int64_t n, int32_t r, int32_t n_pairs) {
  // The tiling whose simulated launch ends first.  Each pair runs its tiles in the launch's
  // order (t, t + pairs, ...); a Y tile costs its operand stages at the bytes each brings
  // into the SM (the rate that bounds these tiles, ~64 B per cycle: per 128 elements of K
  // 32 KB of X plus N/2 rows of W, plus a contributor's slice rows), an S tile its stages
  // at a Y stage's cost (they run at about that pace, whatever their bytes); a Y tile's
  // rank-r step waits until its row block's S is written, kSWait Y stages after the last S
  // tile or contributor's K loop ends.  Checked against the measured best tiling of the
  // LLaMA-7B shapes at r = 32, 64 and 128 (4096 tokens): 8 of 9 picked, the ninth within 1%.
  constexpr int64_t kSWait = 6;
  int32_t best = kLinearPairTiling0;
  int64_t c_best = -1;
  const int64_t row_blocks = ceil_div(T, kPairRows);
  const int64_t k_stages = ceil_div(ceil_div(n, 64), 2);
  const int64_t ext = r == 128 ? 3 : 1;
  std::vector<int64_t> fin, ready;
  for (int i = 0; i < 5; ++i) {
    const int64_t N = kPairCols[i];
    const LinearPairPlan pl = linear_pair_plan(T, m, n, r, kLinearPairTiling0 + i, n_pairs);
    if (pl.pairs <= 0) continue;
    const int64_t tiles_n = ceil_div(m, N);
    const int64_t n_s = row_blocks * pl.s_split;
    const int64_t total = n_s + row_blocks * tiles_n;
    const int64_t P = pl.pairs;
    const int64_t y_stage = core_bytes_host(N);
    const int64_t c_stage = y_stage + (int64_t)pl.s_cols * 128;
    const int64_t s_cost = ceil_div(pl.s_chunk, s_panels_host(N, r)) * y_stage;
    const int64_t g = std::min<int64_t>(pl.group, tiles_n);   // the kernel's stripe width
    fin.assign((size_t)total, 0);
    ready.assign((size_t)row_blocks, -1);
    auto start_of = [&](int64_t t) { return t >= P ? fin[(size_t)(t - P)] : int64_t(0); };
    for (int64_t t = 0; t < n_s; ++t) {                       // S tiles: no waits
      fin[(size_t)t] = start_of(t) + s_cost;
      const int64_t tb = t % row_blocks;
      ready[(size_t)tb] = std::max(ready[(size_t)tb], fin[(size_t)t] + kSWait * y_stage);
    }
    for (int64_t t = n_s; t < total; ++t) {
      // the stripe order's (row block, column block) of Y tile j
      const int64_t j = t - n_s, per = row_blocks * g, full = tiles_n / g;
      int64_t tb, nb;
      if (j < full * per) {
        tb = (j % per) / g;
        nb = (j / per) * g + (j % per) % g;
      } else {
        const int64_t last = tiles_n - full * g, rem = j - full * per;
        tb = rem / last;
        nb = full * g + rem % last;
      }
      if (ready[(size_t)tb] < 0) {
        // contributors are stripe 0's tiles n_s + tb g + 0 .. n_contrib - 1; each starts
        // after its pair's previous tile, which comes before every tile of this row block
        int64_t rd = 0;
        for (int64_t c = 0; c < pl.n_contrib; ++c)
          rd = std::max(rd, start_of(n_s + tb * g + c) + k_stages * c_stage + kSWait * y_stage);
        ready[(size_t)tb] = rd;
      }
      const int64_t st = nb < pl.n_contrib ? c_stage : y_stage;
      const int64_t k_done = start_of(t) + k_stages * st;
      fin[(size_t)t] = std::max(k_done, ready[(size_t)tb]) + ext * st;
    }
    int64_t c = 0;
    for (int64_t t = 0; t < total; ++t) c = std::max(c, fin[(size_t)t]);
    if (c_best < 0 || c < c_best) {
      c_best = c;
      best = kLinearPairTiling0 + i;
    }
  }
  return best;
}

cudaError_t launch_linear_pair(const CUtensorMap& tm_x, const CUtensorMap& tm_w,
                               const CUtensorMap& tm_s, const CUtensorMap& tm_u,
                               const CUtensorMap& tm_y, const CUtensorMap& tm_pk,
                               const CUtensorMap& tm_ps, int64_t T, int64_t m, int64_t n,
                               int32_t u_row0, int32_t r, int32_t tiling,
                               const LinearPairPlan& plan, __nv_bfloat16* s_hl, float* s_part,
                               uint32_t* s_count, uint32_t epoch, bool inject_wait,
                               uint32_t* d_status, cudaStream_t s) {
  const int32_t N = linear_pair_cols(tiling);
  if (N == 0 || plan.pairs <= 0 || plan.group <= 0 || (r != 16 && r != 32 && r != 64 && r != 128))
    return cudaErrorInvalidValue;
  if (plan.n_contrib > 0 ? (plan.s_split != 0 || plan.n_contrib > 4 ||
                            plan.s_cols * plan.n_contrib != 2 * r)
                         : (plan.s_split < 1 || plan.s_split > 15 || plan.s_chunk < 1))
    return cudaErrorInvalidValue;
  const int k_steps = (int)ceil_div(n, 64);
#define ZO_PAIR_Y(NN, RR)                                                                     \
  launch_pair_nr<NN, RR>(tm_x, tm_w, tm_s, tm_u, tm_y, tm_pk, tm_ps, (int)T, (int)m, k_steps,  \
                         u_row0, plan, s_hl, s_part, s_count, epoch, inject_wait, d_status, s)
#define ZO_PAIR_RANKS(NN)                                 \
  case NN * 256 + 16: return ZO_PAIR_Y(NN, 16);           \
  case NN * 256 + 32: return ZO_PAIR_Y(NN, 32);           \
  case NN * 256 + 64: return ZO_PAIR_Y(NN, 64);           \
  case NN * 256 + 128: return ZO_PAIR_Y(NN, 128);
  switch (N * 256 + r) {
    ZO_PAIR_RANKS(256)
    ZO_PAIR_RANKS(240)
    ZO_PAIR_RANKS(224)
    ZO_PAIR_RANKS(192)
    ZO_PAIR_RANKS(128)
    default: return cudaErrorInvalidValue;
  }
#undef ZO_PAIR_RANKS
#undef ZO_PAIR_Y
}

}  // namespace zo
