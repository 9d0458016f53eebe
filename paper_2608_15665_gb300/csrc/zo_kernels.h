// Host-side launchers of the SubZero+ kernels (internal to the library).
#pragma once

#include <cstdint>
#include <string>
#include <cuda.h>
#include <cuda_runtime.h>

#include "zo_device.cuh"

namespace zo {

// Text returned by zo_last_error (zo_api.cu); thread-local.
void set_last_error(const char* msg);
inline void set_last_error(const std::string& msg) { set_last_error(msg.c_str()); }

// ---- counter-based Gaussian contract (zo_rng.cu) ---------------------------
cudaError_t launch_philox_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, uint32_t* out,
                               int64_t n_words, cudaStream_t s);
cudaError_t launch_normal_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, float* out,
                               int64_t n, cudaStream_t s);

// ---- per-pass coefficient C_i and projection P_i (zo_coeff.cu) ---------------
enum CoeffMode : int32_t { kCoeffPerturb = 0, kCoeffStep = 1 };

struct CoeffParams {
  int32_t mode;
  uint64_t seed;
  uint32_t t;
  int32_t r, q;
  // perturb: C = eps (ca Z_qa + cb Z_qb)
  int32_t qa, qb;
  float ca, cb, eps;
  // step: rho from losses, G, optimizer, C = -lr D + restore_coef eps Z_restore
  const float* losses;
  int32_t n_losses, scheme, optimizer;
  float lr, beta1, beta2, eps_adam;
  float inv_bc1, inv_bc2;   // 1 / (1 - beta^adam_t), formed on the host in double
  int32_t restore_query;
  float restore_coef;
  float* gamma_out;
  // tensor-core path: max |C_i| of every matrix (null: not written), for the one
  // exponent of the pass's fp16 operand scales (zo_tc_common.cuh)
  float* amax;
};

cudaError_t launch_coeff(const MatDesc* d_mats, int32_t n_mats, const CoeffParams& p,
                         cudaStream_t s);

// P_i = C_i V_i^T (r x n, fp32) for the FMA weight pass.  Work units are
// (matrix, first column) pairs of 128 columns.
cudaError_t launch_project_fma(const MatDesc* d_mats, const int2* d_units, int32_t n_units,
                               int32_t r, cudaStream_t s);


// ---- weight pass, fp32 FMA path (zo_wpass_fma.cu) ---------------------------
constexpr int kFmaTileRows = 32;
__host__ __device__ constexpr int fma_tile_cols(int32_t dtype) { return dtype == 1 ? 256 : 128; }

cudaError_t launch_wpass_fma(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_tile_prefix,
                             int64_t n_tiles, int32_t r, cudaStream_t s);

// One-launch perturbation pass of the FMA path at r in {4, 8}: each CTA forms C from p
// (mode kCoeffPerturb) and its tile's P columns itself (zo_wpass_fma.cu).
bool wpass_fma_fused_supported(int32_t r);
cudaError_t launch_wpass_fma_fused(const MatDesc* d_mats, int32_t n_mats,
                                   const int64_t* d_tile_prefix, int64_t n_tiles,
                                   const CoeffParams& p, cudaStream_t s);

// Narrow-tile FMA pass at r in {4, 8} for thin matrices (LoRA factors and the like):
// matrix i is cut into tiles of `rows` rows x `chunks` 16-byte column chunks
// (rows x chunks <= kNarrowChunks, chunks x elements-per-chunk <= kNarrowMaxCols), numbered
// from tile0 on.  Each CTA forms C (drawn from p.mode == kCoeffPerturb, or read from
// MatDesc::C with kCoeffStep) and its tile's P columns itself (zo_wpass_fma.cu).
struct NarrowMat {
  int64_t tile0;
  int32_t rows;
  int32_t chunks;
};
constexpr int kNarrowChunks = 1024;
constexpr int kNarrowMaxCols = 512;
bool wpass_narrow_supported(int32_t r);
// Tile shape of an m x n matrix of the given dtype (0 = fp32, 1 = bf16).
void narrow_tile_shape(int64_t m, int64_t n, int32_t dtype, int32_t* rows, int32_t* chunks);
// Shared-memory floats of the P and U parts of one tile of this shape.
int64_t narrow_p_floats(int32_t r, int32_t chunks, int32_t dtype);
int64_t narrow_u_floats(int32_t r, int32_t rows);
// d_tiles[t] = (matrix, first row, first 16-byte chunk, 0) of tile t; p_floats / u_floats:
// the largest P and U parts over the set's tiles.
cudaError_t launch_wpass_narrow(const MatDesc* d_mats, const NarrowMat* d_narrow,
                                const int4* d_tiles, int64_t n_tiles, const CoeffParams& p,
                                int64_t p_floats, int64_t u_floats, cudaStream_t s);

// ---- full-space SPSA perturbation of Eq. (1) (zo_mezo.cu) -------------------------
// W_i <- rnd(W_i + coef Z_i), Z_i per element from the counter contract (tag 5), on the
// FMA pass's tiles (d_tile_prefix / MatDesc::tile0).
cudaError_t launch_mezo(const MatDesc* d_mats, int32_t n_mats, const int64_t* d_tile_prefix,
                        int64_t n_tiles, uint64_t seed, uint32_t t, float coef, cudaStream_t s);

// ---- weight pass, tcgen05 path (zo_wpass_tc.cu: r <= 32, zo_wpass_tmem.cu: r >= 64) -----
bool wpass_tc_supported(int32_t r);
bool wpass_tc_u_in_tmem(int32_t r);   // the U operand is read from Tensor Memory (r >= 64)
int32_t tc_hl_width(int32_t r);       // 16-bit elements per hi/lo operand row
int32_t tc_tile_rows();
int32_t tc_tile_cols();
// Bytes of the stacked U operand for `rows` rows (both layouts below fit).
int64_t tc_u_operand_bytes(int32_t r, int64_t rows);
// The U operand of every matrix from U (after a refresh): the fp16 pair of U 2^kUVScaleExp
// (zo_tc_common.cuh); units = (matrix, first row) x 128 rows.  r <= 32: rows [hi | lo | 0]
// of tc_hl_width(r) fp16, read by TMA (tm_a); r >= 64: chunk-major per 128-row block, read
// into Tensor Memory (zo_wpass_tmem.cu).
cudaError_t launch_split_u(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                           int32_t n_units, int32_t r, void* u_op, cudaStream_t s);
// The perturbed-linear route's U operand (r in {16, 32, 64, 128}): rows [hi | lo | 0] of
// the bf16 pair of U, unscaled, tc_hl_width(r) elements per row, rows as the r <= 32 U
// operand above.
cudaError_t launch_split_u_bf16(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                                int32_t n_units, int32_t r, __nv_bfloat16* u_lin, cudaStream_t s);
// tm_a is used for r <= 32, u_op for r >= 64; d_pinv[i] = 2^-(e_P,i) from launch_split_c.
cudaError_t launch_wpass_tc(const CUtensorMap& tm_a, const void* u_op, const CUtensorMap& tm_b,
                            const CUtensorMap* d_w_maps, const TcMat* d_tc, const float* d_pinv,
                            int32_t n_mats, int64_t n_tiles, int32_t grid, int32_t r,
                            uint32_t* d_status, bool inject_wait, cudaStream_t s);
// r >= 64 (zo_wpass_tmem.cu)
cudaError_t launch_split_u_chunks(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                                  int32_t n_units, int32_t r, uint4* u_t, cudaStream_t s);
cudaError_t launch_wpass_tmem(const uint4* u_t, const CUtensorMap& tm_b,
                              const CUtensorMap* d_w_maps, const TcMat* d_tc, const float* d_pinv,
                              int32_t n_mats, int64_t n_tiles, int32_t grid, int32_t r,
                              uint32_t* d_status, bool inject_wait, cudaStream_t s);

// r = 128 on SM pairs (zo_wpass_pair.cu): tiles of 256 rows (pair_tile_rows()) numbered in
// d_tc's tile0 / tiles_n, the U operand padded to 256-row blocks per matrix, tm_b64 over
// P_HL with 64 x 64 boxes; 2 n_pairs CTAs in clusters of two.
bool wpass_pair_supported(int32_t r);
int32_t pair_tile_rows();
int32_t wpass_pair_max_pairs();   // co-resident clusters of the kernel (0 if unknown)
cudaError_t launch_wpass_pair(const uint4* u_t, const CUtensorMap& tm_b64,
                              const CUtensorMap* d_w_maps, const TcMat* d_tc, const float* d_pinv,
                              int32_t n_mats, int64_t n_pair_tiles, int32_t n_pairs,
                              uint32_t* d_status, bool inject_wait, cudaStream_t s);

// ---- projection P = C V^T on the tensor cores, r >= 16 (zo_project_tc.cu) ---------
bool project_tc_supported(int32_t r);
// V_HL rows [hi | lo] of the fp16 pair of V 2^kUVScaleExp (after a refresh); units = the
// projection units (matrix, first row)
cudaError_t launch_split_v(const MatDesc* d_mats, const TcMat* d_tc, const int2* d_units,
                           int32_t n_units, int32_t r, uint16_t* v_hl, cudaStream_t s);
// C_HL rows [hi | lo] of the fp16 pair of C_i 2^(e_C,i) (every pass), r rows per matrix at
// matrix * r, with e_C,i from amax[i] = max |C_i| (the coefficient kernel's), and
// pinv[i] = 2^-(e_P,i), e_P,i = e_C,i + p_scale_offset(r)
cudaError_t launch_split_c(const MatDesc* d_mats, int32_t n_mats, int32_t r, const float* amax,
                           uint16_t* c_hl, float* pinv, cudaStream_t s);
// P_HL = [hi | lo] of the fp16 pair of (V C^T) 2^(e_P,i): tm_v over V_HL (box 64 x 128),
// tm_c over C_HL (box 64 x r), tm_p over P_HL (box 64 x 32)
cudaError_t launch_project_tc(const CUtensorMap& tm_v, const CUtensorMap& tm_c,
                              const CUtensorMap& tm_p, const TcMat* d_tc, const int2* d_units,
                              int32_t n_units, int32_t grid, int32_t r, uint32_t* d_status,
                              cudaStream_t s);
// The same projection writing, instead of P_HL, P_K = the K-major bf16 pair [P_hi ; P_lo]
// of P_i at p_k + pk_off[i] (rows of n_i rounded up to 64; r in {16, 32, 64, 128}), from pinv.
cudaError_t launch_project_tc_pk(const CUtensorMap& tm_v, const CUtensorMap& tm_c,
                                 const TcMat* d_tc, const int2* d_units, int32_t n_units,
                                 int32_t grid, int32_t r, const float* pinv, const int64_t* pk_off,
                                 __nv_bfloat16* p_k, uint32_t* d_status, cudaStream_t s);

// ---- a linear layer at the perturbed weights, without a weight pass (zo_linear.cu) -----
// Y = X (W + U C V^T)^T = X W^T + S U^T, S = X P^T, for bf16 contexts at r in
// {16, 32, 64, 128}; the single-CTA tilings (this file) at r in {16, 32}, the SM-pair ones
// (zo_linear_pair.cu) at every r.
bool linear_supported(int32_t r);
bool linear_single_cta_supported(int32_t r);
// The S GEMM's split of K = n into k_split ranges of k_chunk steps of 64 (~ one wave).
void linear_s_split(int64_t T, int64_t n, int32_t sms, int32_t* k_split, int32_t* k_chunk);
// Tiling of the Y GEMM: 1 = 128 x 256, 2 = 256 x 256, 3 = 256 x 224 (rows of X x columns
// of Y).  Option 1..3 forces one; 0 takes the one with the least tile work per SM (waves
// of tiles x a tile's relative time).
int32_t linear_y_tiling(int64_t T, int64_t m, int32_t sms, int32_t option);
int32_t linear_y_tile_rows(int32_t tiling);
int32_t linear_y_tile_cols(int32_t tiling);
// Elements of matrix i's P_K: 2r rows of n rounded up to 64.
int64_t linear_pk_elems(int64_t n, int32_t r);
// Kernels launch_linear_s launches for a split of k_split K ranges (1, or 2 with the
// separate reduction).
int32_t linear_s_launches(int32_t k_split);
// S_HL rows [S_hi | S_lo | 0] of S = X P^T: tm_x over X (box 64 x 128), tm_pk over P_K
// (box 64 x 2r); part = k_split x T x r fp32 workspace; s_count = one counter per 32 rows
// of X, zero before the launch and zero again after it (a launch cut short by a wait
// timeout can leave counts behind: zero them before the next).
cudaError_t launch_linear_s(const CUtensorMap& tm_x, const CUtensorMap& tm_pk, int64_t T,
                            int64_t n, int32_t r, int32_t k_split, int32_t k_chunk, float* part,
                            __nv_bfloat16* s_hl, uint32_t* s_count, int32_t sms,
                            uint32_t* d_status, cudaStream_t s);
// Y = X W^T + S U^T: d_w_map = W's descriptor (box 64 x 32), tm_s_in over S_HL (box
// 64 x 128), tm_u over the bf16 U operand (box 64 x 128; W's rows from u_row0), tm_y over Y
// (box 64 x 32, 128-byte swizzle; tiling 3: box 32 x 32, 64-byte swizzle).
cudaError_t launch_linear_y(const CUtensorMap& tm_x, const CUtensorMap* d_w_map,
                            const CUtensorMap& tm_s_in, const CUtensorMap& tm_u,
                            const CUtensorMap& tm_y, int64_t T, int64_t m, int64_t n,
                            int32_t u_row0, int32_t r, int32_t tiling, int32_t sms,
                            uint32_t* d_status, cudaStream_t s);

// The Y GEMM on SM pairs (zo_linear_pair.cu): 256 x N tiles (rows of X x columns of Y),
// M = 256 MMAs across a 2-CTA cluster, two accumulators per SM.  Tilings
// kLinearPairTiling0 + 0 .. 4 are N = 256, 240, 224, 192, 128.
constexpr int32_t kLinearPairTiling0 = 4;
int32_t linear_pair_cols(int32_t tiling);        // N of a pair tiling, 0 for the others
int32_t linear_pair_max_pairs();                 // co-resident clusters (0 if unknown)
// How one call computes S = X P^T and walks its tiles: n_contrib > 0 -- the first n_contrib
// Y tiles (column blocks) of each row block also compute s_cols / 2 of S's columns each
// (r <= 64, where the accumulator has spare columns); else s_split S tiles per row block
// over K ranges of s_chunk 64-element panels (one range at r <= 64, about one S tile per
// pair at r = 128; at most 15).  pairs: clusters launched; group: column blocks per stripe
// of the tile order.  pairs = 0: no plan (bad arguments).
struct LinearPairPlan {
  int32_t pairs, group, n_contrib, s_cols, s_split, s_chunk;
};
LinearPairPlan linear_pair_plan(int64_t T, int64_t m, int64_t n, int32_t r, int32_t tiling,
                                int32_t n_pairs);
// The pair tiling whose busiest pair has the least work (tiles dealt round-robin).
int32_t linear_pair_tiling(int64_t T, int64_t m, int64_t n, int32_t r, int32_t n_pairs);
// One launch computes S (written to s_hl as S_HL rows of tc_hl_width(r)) and Y = X W^T +
// S U^T, r in {16, 32, 64, 128}, as plan (linear_pair_plan) says.  tm_x over X (box
// 64 x 128), tm_w over W_i (box 64 x N/2), tm_s over s_hl (box 64 x 128), tm_u over the
// bf16 U operand (box 64 x N/2; W_i's rows from u_row0), tm_y over Y (box 16 x 32, 32-byte
// swizzle), tm_pk over P_K (box 64 x r), tm_ps over P_K (box 64 x s_cols / 2; any box when
// n_contrib = 0).  s_part: s_split x T x r floats (s_split > 1).  s_count:
// kLinearPairCounters counters per 256 rows of X (zero before the first call), epoch:
// 1 .. kLinearPairEpochs - 1, a new one per call (the counters of a launch cut short by a
// wait timeout must be zeroed before the epochs start again).  inject_wait (test hook):
// the Y tiles wait for a count that never comes, with the short test limit; the launch
// then reports kDevTimeout.
cudaError_t launch_linear_pair(const CUtensorMap& tm_x, const CUtensorMap& tm_w,
                               const CUtensorMap& tm_s, const CUtensorMap& tm_u,
                               const CUtensorMap& tm_y, const CUtensorMap& tm_pk,
                               const CUtensorMap& tm_ps, int64_t T, int64_t m, int64_t n,
                               int32_t u_row0, int32_t r, int32_t tiling,
                               const LinearPairPlan& plan, __nv_bfloat16* s_hl, float* s_part,
                               uint32_t* s_count, uint32_t epoch, bool inject_wait,
                               uint32_t* d_status, cudaStream_t s);
constexpr uint32_t kLinearPairCountsPerCall = 8;   // 32-row groups of a 256-row block
                                                   // (S_HL writes per S slice)
constexpr int32_t kLinearPairCounters = 40;        // flags and counters per 256-row block
constexpr uint32_t kLinearPairEpochs = 1u << 26;

// ---- refresh of tall panels at r = 16 ... 128: CholeskyQR2 (zo_cholqr.cu) ----------
constexpr int32_t kCqChunkRows = 1024;   // rows per partial Gram matrix
struct CqPanel {
  float* out;          // U_i or V_i: rows x r, row-major; receives Q
  int64_t rows;
  uint32_t gidx;       // matrix index for Omega
  uint32_t tag;        // kTagOmegaU or kTagOmegaV
  int32_t chunk0;      // first chunk of this panel
  int32_t n_chunks;
};
struct CqChunk {
  int64_t row0;        // first panel row of the chunk
  int32_t panel;
  int32_t nrows;       // <= kCqChunkRows
};
bool cholqr_supported(int32_t r);
// Six launches: Gram, Cholesky + inverse, apply; twice.  d_partial: n_chunks x r x r
// floats, d_linv: n_panels x r x r floats.
cudaError_t launch_cholqr(const CqPanel* d_panels, int32_t n_panels, const CqChunk* d_chunks,
                          int32_t n_chunks, float* d_partial, float* d_linv, int32_t r,
                          uint64_t seed, uint32_t refresh_idx, uint32_t* d_status, cudaStream_t s);

// ---- refresh: batched TSQR + sign correction (zo_qr.cu) ------------------------
int32_t qr_block_rows(int32_t r);
cudaError_t launch_qr_up(const QrBlock* d_blocks, int32_t n_blocks, int32_t r, uint64_t seed,
                         uint32_t refresh_idx, uint32_t* d_status, cudaStream_t s);
cudaError_t launch_qr_down(const QrBlock* d_blocks, int32_t n_blocks, int32_t r,
                           uint32_t* d_status, cudaStream_t s);
cudaError_t launch_zero_moments(const MatDesc* d_mats, int32_t n_mats, int32_t r, cudaStream_t s);

}  // namespace zo
