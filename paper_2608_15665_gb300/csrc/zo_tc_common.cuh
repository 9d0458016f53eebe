// Pieces shared by the two tensor-core weight-pass kernels (zo_wpass_tc.cu: the U
// operand in shared memory, r <= 32; zo_wpass_tmem.cu: the U operand in Tensor Memory,
// r >= 64): tile geometry, the barrier block, the interleaved tile walk and the hi/lo
// split of the operands.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
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
  // scale of the tile in W stage s (written by the W producer before it arms w_full[s],
  // read by the epilogue after its wait on w_full[s])
  float w_scale[4];
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

// ---- fp16 operands of the weight pass and the projection -------------------------------
// The tensor-core operands U, P = C V^T (and, in the projection, V and C) are held as
// pairs of fp16 values, x s = hi + lo with hi = f16(x s), lo = f16(x s - hi), where s is a
// power of two that puts x s into fp16's normal range.  fp16 carries an 11-bit
// significand, so hi + lo keeps ~22 bits of x (relative representation error <= 2^-22,
// against 2^-17 for a bf16 pair) and the three products hi.hi + hi.lo + lo.hi that the
// MMAs accumulate in fp32 drop only lo.lo (~2^-22): the update U P then errs by ~2^-21 of
// sum |U| |P|, the grade of an fp32 evaluation, at the MMA count of the bf16 pair.
// Scales (all exact powers of two, undone in fp32 by the consumer):
//   U, V:  2^kUVScaleExp  (|U|, |V| <= 1 for column-orthonormal bases)
//   C_i:   2^(e_C,i) with e_C,i = 14 - E, max |C_i| < 2^E (from the maximum the coefficient
//          kernel writes), so |C_i s| < 2^14
//   P_i:   2^(e_P,i), e_P,i = e_C,i + p_scale_offset(r): |P_kj| <= ||C_k,:|| ||V_j,:|| <=
//          sqrt(r) max |C_i|, so |P_i s| <= 2^15 (fp16 holds up to 65504)
// The weight pass multiplies its accumulator by pinv_i 2^-kUVScaleExp, pinv_i = 2^-(e_P,i).
// Each matrix's scale depends on its own C alone, so a set split over several contexts (or
// ranks) gets the same bits as one context over the whole set.
constexpr int kUVScaleExp = 14;
__host__ __device__ constexpr int p_scale_offset(int r) {   // 1 - ceil(log2(r) / 2)
  return r <= 16 ? -1 : r <= 64 ? -2 : -3;
}
constexpr int kScaleExpMax = 100;   // |e_C| bound: keeps every scale a normal fp32 value

// 2^e as an fp32 value, -126 <= e <= 127 (exact).
__device__ __forceinline__ float exp2i(int e) { return __int_as_float((e + 127) << 23); }

// e_C of a coefficient matrix whose largest magnitude is amax (>= 0): 14 - E with
// amax < 2^E; a zero or fp32-subnormal amax takes the largest exponent, a non-finite one 0.
__device__ __forceinline__ int coeff_scale_exp(float amax) {
  const int biased = (__float_as_int(amax) >> 23) & 0xFF;
  if (biased == 0) return kScaleExpMax;
  if (biased == 0xFF) return 0;
  const int e = 14 - (biased - 126);
  return e > kScaleExpMax ? kScaleExpMax : e < -kScaleExpMax ? -kScaleExpMax : e;
}

// s x = hi + lo in fp16 for 8 consecutive fp32 values, packed two per 32-bit word (lower
// half = first element).  s x - hi is exact in fp32.
__device__ __forceinline__ void split8_f16(const float (&x)[8], float s, uint4& hi, uint4& lo) {
  uint32_t hw[4], lw[4];
#pragma unroll
  for (int pr = 0; pr < 4; ++pr) {
    const float a = x[2 * pr] * s, b = x[2 * pr + 1] * s;
    const __half2 h2 = __floats2half2_rn(a, b);
    const float2 hf = __half22float2(h2);
    const __half2 l2 = __floats2half2_rn(a - hf.x, b - hf.y);
    hw[pr] = *reinterpret_cast<const uint32_t*>(&h2);
    lw[pr] = *reinterpret_cast<const uint32_t*>(&l2);
  }
  hi = make_uint4(hw[0], hw[1], hw[2], hw[3]);
  lo = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

// The weight-pass epilogue's arithmetic for two neighbouring bf16 weights w (packed, lower
// half = first) and their fp32 updates a, b: rnd_bf16(w + s a), rnd_bf16(w' + s b), as one
// packed fp32 multiply-add (fma.rn.f32x2: each lane an IEEE fp32 fma, round to nearest)
// and one packed conversion.  s2 holds {s, s}.
__device__ __forceinline__ uint64_t splat2(float s) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %1};" : "=l"(r) : "f"(s));
  return r;
}
__device__ __forceinline__ uint32_t bf16x2_add_scaled(uint32_t w, uint32_t a, uint32_t b, uint64_t s2) {
  uint32_t out;
  asm("{\n\t.reg .b64 x, c, d;\n\t.reg .b32 l, h;\n\t"
      "mov.b64 x, {%1, %2};\n\t"
      "shl.b32 l, %3, 16;\n\t"
      "and.b32 h, %3, 0xFFFF0000;\n\t"
      "mov.b64 c, {l, h};\n\t"
      "fma.rn.f32x2 d, x, %4, c;\n\t"
      "mov.b64 {l, h}, d;\n\t"
      "cvt.rn.bf16x2.f32 %0, h, l;\n\t}"
      : "=r"(out)
      : "r"(a), "r"(b), "r"(w), "l"(s2));
  return out;
}

// x = hi + lo for 8 consecutive fp32 values: hi = bf16(x), lo = bf16(x - hi), packed two
// per 32-bit word (lower half = first element).  (The perturbed-linear route's operands,
// which meet the bf16 X and W in the same accumulator.)
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
