// Pieces shared by the two tensor-core weight-pass kernels (zo_wpass_tc.cu: the U
// operand in shared memory, r <= 32; zo_wpass_tmem.cu: the U operand in Tensor Memory,
// r >= 64): tile geometry, the barrier block, the interleaved tile walk and the hi/lo
// split of the operands.
#pragma once

#include <cuda_bf16.h>
#include <cstdint>

#include "zo_kernels.h"

namespace zo {
namespace tc {

constexpr int kBM = 128;                         // tile rows (TMEM lanes)
constexpr int kBN = 128;                         // tile columns (TMEM columns per accumulator)
constexpr int kWBoxBytes = 32 * 64 * 2;          // one TMA box of W: 32 rows x 64 bf16
constexpr int kWStageBytes = kBM * kBN * 2;      // 32 KB
constexpr int kPanelBytes = kBM * 64 * 2;        // 128 rows x 128 bytes = 16 KB
constexpr long long kWaitCycles = 4000000000LL;  // default wait limit, ~2 s at 2 GHz
constexpr long long kTestWaitCycles = 200000000LL;  // with the test hook armed, ~0.1 s
constexpr int kTileChunk = 4;                    // consecutive tiles per CTA visit (U reuse)

// Width in bf16 of a stacked operand row [hi(r) | lo(r) | 0 ...]: at least one 128-byte
// swizzle row.
__host__ __device__ constexpr int hl_width(int r) { return 2 * r > 64 ? 2 * r : 64; }

struct Shared {
  uint64_t w_full[4], w_empty[4];
  uint64_t a_full[2], a_empty[2];
  uint64_t b_full[4], b_empty[4];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t never;          // test hook: a barrier no thread ever arrives on
  uint32_t tmem_base;
  int abort_flag;
};

// Walks this CTA's tiles t0, t0 + stride, ... (< t_end), each decoded into (matrix, row
// block, column block); tiles are numbered matrix by matrix, row block by row block.
// With chunk > 1 it takes `chunk` consecutive tiles, then jumps by the stride.
struct TileIter {
  const TcMat* mats;
  int n_mats;
  int64_t t, t_end, stride;
  int i;
  int64_t rb, cb, tiles_m;
  int64_t chunk = 1, in_chunk = 0;
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
    tiles_m = (mats[i].m + kBM - 1) / kBM;
  }
  __device__ bool valid() const { return t < t_end; }
  __device__ void next() {
    if (stride != 1) {
      if (++in_chunk < chunk) {
        t += 1;
      } else {
        in_chunk = 0;
        t += stride - (chunk - 1);
      }
      if (t >= t_end) return;
      while (i + 1 < n_mats && mats[i + 1].tile0 <= t) ++i;
      set_local();
      return;
    }
    ++t;
    if (t >= t_end) return;
    if (++cb == mats[i].tiles_n) {
      cb = 0;
      if (++rb == tiles_m) {
        ++i;
        rb = 0;
        tiles_m = (mats[i].m + kBM - 1) / kBM;
      }
    }
  }
};

// index of the last of n_issued ring entries that went into slot s (ring of S slots), or -1
__device__ __forceinline__ int64_t last_in_slot(int64_t n_issued, int s, int S) {
  if (n_issued <= s) return -1;
  return s + (int64_t)S * ((n_issued - 1 - s) / S);
}

__device__ __forceinline__ void give_up(Shared& sh, uint32_t* status) {
  atomicOr(status, (uint32_t)kDevTimeout);
  *reinterpret_cast<volatile int*>(&sh.abort_flag) = 1;
}

// x = hi + lo for 8 consecutive fp32 values: hi = bf16(x), lo = bf16(x - hi), packed two
// per 32-bit word (lower half = first element).
__device__ __forceinline__ void split8(const float (&x)[8], uint4& hi, uint4& lo) {
  uint32_t hw[4], lw[4];
#pragma unroll
  for (int pr = 0; pr < 4; ++pr) {
    const __nv_bfloat162 h2 = __floats2bfloat162_rn(x[2 * pr], x[2 * pr + 1]);
    const __nv_bfloat162 l2 =
        __floats2bfloat162_rn(x[2 * pr] - __low2float(h2), x[2 * pr + 1] - __high2float(h2));
    hw[pr] = *reinterpret_cast<const uint32_t*>(&h2);
    lw[pr] = *reinterpret_cast<const uint32_t*>(&l2);
  }
  hi = make_uint4(hw[0], hw[1], hw[2], hw[3]);
  lo = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

}  // namespace tc
}  // namespace zo
