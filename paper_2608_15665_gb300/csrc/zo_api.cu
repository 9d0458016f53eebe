// Host runtime and C ABI of the SubZero+ weight path (declared in include/zo.h).
//
// The context owns: a device copy of the matrix table, the per-pass coefficient
// C_i (r x r) and projection P_i (r x n_i) buffers, the TSQR workspace of the
// refresh, a loss staging buffer and a device status word.  Every call validates
// its arguments on the host, then launches on the context's stream.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <cudaTypedefs.h>

#include "../../include/zo.h"
#include "zo_kernels.h"

namespace {

thread_local std::string g_last_error;

zo_status cuda_fail(cudaError_t e, const char* what) {
  g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
  return ZO_ERR_CUDA;
}

#define ZO_CUDA(call, what)                                   \
  do {                                                        \
    cudaError_t _e = (call);                                  \
    if (_e != cudaSuccess) return cuda_fail(_e, what);        \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool supported_rank(int32_t r) {
  return r == 4 || r == 8 || r == 16 || r == 32 || r == 64 || r == 128;
}

struct QrLevel {
  std::vector<zo::QrBlock> up;    // all blocks of this level (tops included)
  std::vector<zo::QrBlock> down;  // non-top blocks of this level
};

}  // namespace

void zo::set_last_error(const char* msg) { g_last_error = msg; }

namespace {

// Makes a context's device current for the length of a call and gives the caller's back:
// every kernel of a context runs on the device it was created on, whatever device the
// calling thread has selected since.
struct DeviceGuard {
  int prev = -1;
  bool switched = false;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev && cudaSetDevice(dev) == cudaSuccess)
      switched = true;
  }
  ~DeviceGuard() {
    if (switched) cudaSetDevice(prev);
  }
};

}  // namespace


struct zo_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  int32_t n_mats = 0, r = 0, q = 0;
  uint64_t seed = 0;
  uint32_t base = 0;
  std::vector<zo::MatDesc> h_mats;
  zo::MatDesc* d_mats = nullptr;
  int64_t* d_tile_prefix = nullptr;
  int64_t n_tiles = 0;
  // narrow tiles of the FMA path (r in {4, 8}); chosen automatically when they need at
  // most half the CTAs of the 32-row tiles
  zo::NarrowMat* d_narrow = nullptr;
  int4* d_narrow_tiles = nullptr;          // (matrix, first row, first chunk) of each tile
  int64_t n_narrow_tiles = 0, narrow_p = 0, narrow_u = 0;
  bool narrow_ok = false, narrow_auto = false;
  int2* d_proj_units = nullptr;
  int32_t n_proj_units = 0;
  float* d_coeff_ws = nullptr;   // C_i and P_i
  float* d_losses = nullptr;
  int32_t max_losses = 0;
  float* d_qr_ws = nullptr;      // TSQR stacks and tau
  zo::QrBlock* d_qr_blocks = nullptr;
  // tall panels at r = 16 ... 128 are refreshed by CholeskyQR2 instead of the TSQR
  zo::CqPanel* d_cq_panels = nullptr;
  zo::CqChunk* d_cq_chunks = nullptr;
  float* d_cq_partial = nullptr;
  float* d_cq_linv = nullptr;
  int32_t n_cq_panels = 0, n_cq_chunks = 0;
  std::vector<int64_t> up_off, up_cnt, down_off, down_cnt;   // per level, into d_qr_blocks
  uint32_t* d_status = nullptr;
  int path_option = 0;
  int last_path = 0;
  bool inject_wait = false;      // test hook armed for the next tensor-core pass
  int64_t launches = 0;          // kernels launched by this context
  // tensor-core weight pass (all matrices bf16, r in {16, 32, 64, 128})
  bool tc_ok = false;
  bool tc_failed = false;            // the set qualifies, but its setup failed (zo_last_error
                                     // at zo_create); the automatic path then refuses to run
  std::string tc_fail_msg;
  bool proj_tc = false;              // the projection's descriptors are in place
  int sms = 0;
  void* d_u_op = nullptr;            // stacked U operand of every U_i, 128-row padded: the fp16
                                     // pair of U 2^14 (rows [hi | lo | 0] for r <= 32,
                                     // chunk-major for r >= 64)
  uint16_t* d_p_hl = nullptr;        // stacked [hi | lo] fp16 rows of every P_i^T 2^(e_P,i),
                                     // 128-row padded
  float* d_amax = nullptr;           // max |C_i| of the current pass, one per matrix
  float* d_pinv = nullptr;           // 2^-(e_P,i) of the current pass, one per matrix
  zo::TcMat* d_tc = nullptr;
  std::vector<zo::TcMat> h_tc;       // host copy (operand rows of each matrix)
  // zo_linear_prepare / zo_linear_perturbed: P_K of every matrix ([P_hi ; P_lo] rows,
  // K-major) at element offsets pk_off, S_HL and the partial sums of S (T rows each)
  __nv_bfloat16* d_pk = nullptr;
  int64_t* d_pk_off = nullptr;
  std::vector<int64_t> h_pk_off;
  bool linear_ready = false;
  __nv_bfloat16* d_u_lin = nullptr;  // the U operand as a bf16 pair (rows as d_u_op at r <= 32)
  CUtensorMap tm_u_lin{};
  bool u_lin_valid = false;          // d_u_lin holds the current U (cleared by every refresh)
  int64_t u_rows = 0;                // rows of the stacked U operand
  int linear_tile = 0;           // ZO_OPTION_LINEAR_TILE
  int last_linear_tiling = 0;    // tiling of the last Y GEMM (1..3, or a pair tiling)
  int linear_pairs = -1;         // co-resident clusters of the pair Y GEMM (-1: not asked)
  __nv_bfloat16* d_s_hl = nullptr;
  float* d_s_part = nullptr;
  uint32_t* d_s_count = nullptr;   // one counter per 32 rows of S_HL's capacity
  // the SM-pair route's row-block counters (one per 256 rows of S_HL's capacity) and the
  // epoch of its last call
  uint32_t* d_s_flags = nullptr;
  uint32_t lin_epoch = 0;
  int64_t s_cap = 0, part_cap = 0;
  int64_t tc_tiles = 0;
  // r = 128: the weight pass on SM pairs (256-row tiles numbered in d_tc_pair), unless
  // ZO_OPTION_PAIR_MMA = 0 selects the single-SM kernel
  bool pair_ok = false;
  int pair_option = 1;
  zo::TcMat* d_tc_pair = nullptr;
  int64_t pair_tiles = 0;
  int32_t n_pairs = 0;
  CUtensorMap tm_b64{};              // P_HL in 64 x 64 boxes (one SM's half of a P tile)
  CUtensorMap* d_w_maps = nullptr;   // one TMA descriptor per W_i (device memory)
  CUtensorMap tm_a{}, tm_b{};        // descriptors of the stacked operands (kernel parameters)
  int2* d_u_units = nullptr;
  int32_t n_u_units = 0;
  uint16_t* d_v_hl = nullptr;        // fp16 [hi | lo] rows of every V_i 2^14, rows as P_HL
  uint16_t* d_c_hl = nullptr;        // fp16 [hi | lo] rows of every C_i 2^(e_C,i), r rows each
  CUtensorMap tm_v{}, tm_c{}, tm_p{};  // V_HL, C_HL, and P_HL in 32-row boxes
  bool timing = false;
  std::vector<cudaEvent_t> ev_start, ev_stop;
  size_t ev_used = 0;
  double timing_ms = 0.0;
  int64_t timing_launches = 0;
};

namespace {

void free_ctx(zo_ctx* c) {
  if (!c) return;
  cudaFree(c->d_mats);
  cudaFree(c->d_tile_prefix);
  cudaFree(c->d_narrow);
  cudaFree(c->d_narrow_tiles);
  cudaFree(c->d_proj_units);
  cudaFree(c->d_coeff_ws);
  cudaFree(c->d_losses);
  cudaFree(c->d_qr_ws);
  cudaFree(c->d_qr_blocks);
  cudaFree(c->d_cq_panels);
  cudaFree(c->d_cq_chunks);
  cudaFree(c->d_cq_partial);
  cudaFree(c->d_cq_linv);
  cudaFree(c->d_status);
  cudaFree(c->d_u_op);
  cudaFree(c->d_p_hl);
  cudaFree(c->d_tc);
  cudaFree(c->d_tc_pair);
  cudaFree(c->d_pk);
  cudaFree(c->d_pk_off);
  cudaFree(c->d_s_hl);
  cudaFree(c->d_s_part);
  cudaFree(c->d_s_count);
  cudaFree(c->d_s_flags);
  cudaFree(c->d_w_maps);
  cudaFree(c->d_u_units);
  cudaFree(c->d_v_hl);
  cudaFree(c->d_c_hl);
  cudaFree(c->d_pinv);
  cudaFree(c->d_amax);
  cudaFree(c->d_u_lin);
  for (auto e : c->ev_start) cudaEventDestroy(e);
  for (auto e : c->ev_stop) cudaEventDestroy(e);
  delete c;
}

zo_status validate_matrix(const zo_matrix& mt, int32_t r) {
  if (!mt.W || !mt.U || !mt.V || !mt.M || !mt.Vm) {
    g_last_error = "null buffer in zo_matrix";
    return ZO_ERR_INVALID_ARG;
  }
  if (mt.dtype != ZO_F32 && mt.dtype != ZO_BF16) {
    g_last_error = "unknown dtype";
    return ZO_ERR_DTYPE;
  }
  if (mt.m < r || mt.n < r || mt.ldw < mt.n) {
    g_last_error = "need r <= min(m, n) and ldw >= n";
    return ZO_ERR_SHAPE;
  }
  // the Philox counter word addresses e / 4 of an m x r (or n x r) buffer in 32 bits
  if (mt.m * (int64_t)r >= (int64_t(1) << 34) || mt.n * (int64_t)r >= (int64_t(1) << 34)) {
    g_last_error = "matrix too large for the 32-bit counter word";
    return ZO_ERR_SHAPE;
  }
  const int64_t esize = mt.dtype == ZO_BF16 ? 2 : 4;
  if (!aligned16(mt.W) || (mt.ldw * esize) % 16 != 0 || !aligned16(mt.U) || !aligned16(mt.V) ||
      !aligned16(mt.M) || !aligned16(mt.Vm)) {
    g_last_error = "buffers must be 16-byte aligned and ldw*sizeof(dtype) a multiple of 16";
    return ZO_ERR_ALIGN;
  }
  return ZO_OK;
}

// TSQR plan of one panel (rows x r) stored at `panel`; appends blocks per level and
// returns the floats of workspace it needs (stacks + tau), assigning offsets from *ws.
void plan_panel(float* panel, int64_t rows, int32_t r, uint32_t gidx, uint32_t tag, int32_t B,
                std::vector<QrLevel>& levels, float* ws_base, int64_t* ws_off) {
  float* storage = panel;
  int64_t level_rows = rows;
  for (int level = 0;; ++level) {
    if ((int)levels.size() <= level) levels.emplace_back();
    const int64_t nb = (level_rows + B - 1) / B;
    float* stack = nullptr;
    if (nb > 1) {
      stack = ws_base ? ws_base + *ws_off : nullptr;
      *ws_off += nb * (int64_t)r * r;
    }
    for (int64_t b = 0; b < nb; ++b) {
      zo::QrBlock blk{};
      blk.rows = storage ? storage + b * (int64_t)B * r : nullptr;
      blk.n_real = (int32_t)std::min<int64_t>(B, level_rows - b * B);
      blk.row0 = b * B;
      blk.flags = (level == 0 ? zo::kQrLevel0 : 0) | (nb == 1 ? zo::kQrTop : 0);
      blk.gidx = gidx;
      blk.tag = tag;
      blk.tau = ws_base ? ws_base + *ws_off : nullptr;
      *ws_off += (r + 3) / 4 * 4;
      if (nb > 1) {
        blk.r_out = stack ? stack + b * (int64_t)r * r : nullptr;
        blk.s_in = blk.r_out;
      }
      levels[level].up.push_back(blk);
      if (nb > 1) levels[level].down.push_back(blk);
    }
    if (nb == 1) break;
    storage = stack;
    level_rows = nb * r;
  }
}

zo_status record_start(zo_ctx* c) {
  if (!c->timing) return ZO_OK;
  if (c->ev_used == c->ev_start.size()) {
    cudaEvent_t a, b;
    ZO_CUDA(cudaEventCreate(&a), "cudaEventCreate");
    ZO_CUDA(cudaEventCreate(&b), "cudaEventCreate");
    c->ev_start.push_back(a);
    c->ev_stop.push_back(b);
  }
  ZO_CUDA(cudaEventRecord(c->ev_start[c->ev_used], c->stream), "cudaEventRecord");
  return ZO_OK;
}

zo_status record_stop(zo_ctx* c) {
  if (!c->timing) return ZO_OK;
  ZO_CUDA(cudaEventRecord(c->ev_stop[c->ev_used], c->stream), "cudaEventRecord");
  ++c->ev_used;
  return ZO_OK;
}

bool tc_path(const zo_ctx* c) { return c->tc_ok && (c->path_option == 0 || c->path_option == 2); }
// The automatic path on a set that qualifies for the tensor cores but could not be set up
// for them: refused (ZO_ERR_UNSUPPORTED) instead of running the FMA pass unasked.
bool tc_refused(const zo_ctx* c) { return c->tc_failed && c->path_option == 0; }
zo_status refuse_tc(const zo_ctx* c) {
  g_last_error = c->tc_fail_msg;
  return ZO_ERR_UNSUPPORTED;
}
bool narrow_path(const zo_ctx* c) {
  return c->narrow_ok && (c->path_option == 3 || (c->path_option == 0 && c->narrow_auto));
}

// Projection of C_i onto V_i and the weight pass, shared by zo_perturb and zo_step.
zo_status run_weight_pass(zo_ctx* c) {
  const bool use_tc = tc_path(c);
  if (!use_tc && narrow_path(c)) {
    // C_i is the coefficient kernel's output; P columns are formed in the pass
    zo::CoeffParams p{};
    p.mode = zo::kCoeffStep;
    p.r = c->r;
    zo_status st = record_start(c);
    if (st != ZO_OK) return st;
    ZO_CUDA(zo::launch_wpass_narrow(c->d_mats, c->d_narrow, c->d_narrow_tiles,
                                    c->n_narrow_tiles, p, c->narrow_p, c->narrow_u, c->stream),
            "narrow-tile weight-pass kernel");
    c->last_path = 3;
    ++c->launches;
    return record_stop(c);
  }
  if (use_tc) {
    // setup_tc keeps tc_ok only with the projection's descriptors in place (proj_tc)
    ZO_CUDA(zo::launch_split_c(c->d_mats, c->n_mats, c->r, c->d_amax, c->d_c_hl, c->d_pinv,
                               c->stream),
            "split C");
    ++c->launches;
    const int grid = std::min<int>(c->n_proj_units, c->sms);
    ZO_CUDA(zo::launch_project_tc(c->tm_v, c->tm_c, c->tm_p, c->d_tc, c->d_proj_units,
                                  c->n_proj_units, grid, c->r, c->d_status, c->stream),
            "tensor-core projection kernel");
  } else {
    ZO_CUDA(zo::launch_project_fma(c->d_mats, c->d_proj_units, c->n_proj_units, c->r, c->stream),
            "projection kernel");
  }
  ++c->launches;
  zo_status st = record_start(c);
  if (st != ZO_OK) return st;
  if (use_tc) {
    const int grid = (int)std::min<int64_t>(c->tc_tiles, c->sms);
    const bool inject = c->inject_wait;
    c->inject_wait = false;
    if (c->pair_ok && c->pair_option == 1) {
      ZO_CUDA(zo::launch_wpass_pair(static_cast<const uint4*>(c->d_u_op), c->tm_b64, c->d_w_maps,
                                    c->d_tc_pair, c->d_pinv, c->n_mats, c->pair_tiles,
                                    (int32_t)std::min<int64_t>(c->pair_tiles, c->n_pairs),
                                    c->d_status, inject, c->stream),
              "tensor-core weight-pass kernel (SM pairs)");
    } else {
      ZO_CUDA(zo::launch_wpass_tc(c->tm_a, c->d_u_op, c->tm_b, c->d_w_maps, c->d_tc, c->d_pinv,
                                  c->n_mats, c->tc_tiles, grid, c->r, c->d_status, inject,
                                  c->stream),
              "tensor-core weight-pass kernel");
    }
    c->last_path = 2;
  } else {
    ZO_CUDA(zo::launch_wpass_fma(c->d_mats, c->n_mats, c->d_tile_prefix, c->n_tiles, c->r,
                                 c->stream),
            "weight-pass kernel");
    c->last_path = 1;
  }
  ++c->launches;
  return record_stop(c);
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D tensor map of 16-bit elements (bf16, or fp16 with f16 = true): `cols` contiguous
// elements per row, `rows` rows `row_bytes` apart, boxes of box_cols x box_rows with the
// 128-byte swizzle.
bool encode_16b_2d(CUtensorMap* tm, void* base, uint64_t cols, uint64_t rows, uint64_t row_bytes,
                   uint32_t box_cols, uint32_t box_rows, bool f16,
                   CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {row_bytes};
  const cuuint32_t box[2] = {box_cols, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return enc(tm, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base,
             dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
bool encode_bf16_2d(CUtensorMap* tm, void* base, uint64_t cols, uint64_t rows, uint64_t row_bytes,
                    uint32_t box_cols, uint32_t box_rows,
                    CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  return encode_16b_2d(tm, base, cols, rows, row_bytes, box_cols, box_rows, false, swizzle);
}
bool encode_f16_2d(CUtensorMap* tm, void* base, uint64_t cols, uint64_t rows, uint64_t row_bytes,
                   uint32_t box_cols, uint32_t box_rows) {
  return encode_16b_2d(tm, base, cols, rows, row_bytes, box_cols, box_rows, true);
}

// Tile table of the narrow-tile FMA pass (r in {4, 8}).
zo_status setup_narrow(zo_ctx* c, const zo_matrix* mats) {
  if (!zo::wpass_narrow_supported(c->r)) return ZO_OK;
  std::vector<zo::NarrowMat> nm(c->n_mats);
  int64_t tiles = 0;
  for (int32_t i = 0; i < c->n_mats; ++i) {
    int32_t rows = 1, chunks = 1;
    zo::narrow_tile_shape(mats[i].m, mats[i].n, mats[i].dtype, &rows, &chunks);
    const int64_t vec = mats[i].dtype == ZO_BF16 ? 8 : 4;
    const int64_t cpr = (mats[i].n + vec - 1) / vec;
    nm[i] = {tiles, rows, chunks};
    tiles += ((mats[i].m + rows - 1) / rows) * ((cpr + chunks - 1) / chunks);
    c->narrow_p = std::max(c->narrow_p, zo::narrow_p_floats(c->r, chunks, mats[i].dtype));
    c->narrow_u = std::max(c->narrow_u, zo::narrow_u_floats(c->r, rows));
  }
  c->n_narrow_tiles = tiles;
  if (tiles > 0x7FFFFFFF) return ZO_OK;   // beyond one grid: the 32-row tiles only
  std::vector<int4> tab((size_t)tiles);
  for (int32_t i = 0; i < c->n_mats; ++i) {
    const int64_t vec = mats[i].dtype == ZO_BF16 ? 8 : 4;
    const int64_t cpr = (mats[i].n + vec - 1) / vec;
    if (mats[i].m > 0x7FFFFFFF || cpr > 0x7FFFFFFF) return ZO_OK;   // rows, chunks as int
    const int64_t tiles_c = (cpr + nm[i].chunks - 1) / nm[i].chunks;
    const int64_t end = i + 1 < c->n_mats ? nm[i + 1].tile0 : tiles;
    for (int64_t t = nm[i].tile0; t < end; ++t) {
      const int64_t local = t - nm[i].tile0;
      tab[(size_t)t] = make_int4(i, (int)((local / tiles_c) * nm[i].rows),
                                 (int)((local % tiles_c) * nm[i].chunks), 0);
    }
  }
  cudaError_t e = cudaMalloc(&c->d_narrow, sizeof(zo::NarrowMat) * c->n_mats);
  if (e == cudaSuccess) e = cudaMalloc(&c->d_narrow_tiles, sizeof(int4) * std::max<int64_t>(tiles, 1));
  if (e == cudaSuccess)
    e = cudaMemcpy(c->d_narrow, nm.data(), sizeof(zo::NarrowMat) * c->n_mats, cudaMemcpyHostToDevice);
  if (e == cudaSuccess && tiles > 0)
    e = cudaMemcpy(c->d_narrow_tiles, tab.data(), sizeof(int4) * tiles, cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    cuda_fail(e, "narrow-tile table");
    return e == cudaErrorMemoryAllocation ? ZO_ERR_NOMEM : ZO_ERR_CUDA;
  }
  c->narrow_ok = true;
  // chosen automatically for sets that need at most half the CTAs of the 32-row tiles
  c->narrow_auto = 2 * tiles <= c->n_tiles;
  return ZO_OK;
}

// Buffers and descriptors of the tensor-core weight pass; leaves tc_ok false when
// the context does not qualify: an fp32 matrix, r outside {16, 32, 64, 128}, or a
// width n not a multiple of 8 -- TMA stores write whole 16-byte chunks, and the chunk
// that holds a row's last element would also overwrite the caller's elements past n.
// A set that qualifies but whose descriptors or row counts the tensor-core pass cannot
// take gets tc_failed instead: the automatic path then returns ZO_ERR_UNSUPPORTED rather
// than running the FMA pass in its place; ZO_OPTION_WPASS_PATH = 1 selects that pass.
zo_status setup_tc(zo_ctx* c, const zo_matrix* mats) {
  if (!zo::wpass_tc_supported(c->r)) return ZO_OK;
  for (int32_t i = 0; i < c->n_mats; ++i)
    if (mats[i].dtype != ZO_BF16 || mats[i].n % 8 != 0) return ZO_OK;
  auto refuse = [&](const char* why) {
    c->tc_failed = true;
    c->tc_fail_msg = std::string("the tensor-core weight pass could not be set up (") + why +
                     "); set ZO_OPTION_WPASS_PATH = 1 to run the FMA pass instead";
    g_last_error = c->tc_fail_msg;
    return ZO_OK;
  };
  const int64_t BM = zo::tc_tile_rows(), BN = zo::tc_tile_cols();
  const int64_t HLW = zo::tc_hl_width(c->r);
  // at r = 128 the U operand is padded to the SM pair's 256-row tiles (the second 128-row
  // block of a ragged pair tile reads zeros), which the single-SM kernel reads as well
  const bool pair = zo::wpass_pair_supported(c->r);
  const int64_t UPAD = pair ? zo::pair_tile_rows() : BM;
  std::vector<zo::TcMat> tc(c->n_mats), tcp;
  std::vector<int2> uunits;
  int64_t urows = 0, prows = 0, tiles = 0, ptiles = 0;
  for (int32_t i = 0; i < c->n_mats; ++i) {
    const int64_t m = mats[i].m, n = mats[i].n;
    tc[i].m = m;
    tc[i].n = n;
    tc[i].tile0 = tiles;
    tc[i].tiles_n = (int32_t)((n + BN - 1) / BN);
    tc[i].u_row0 = (int32_t)urows;
    tc[i].p_row0 = (int32_t)prows;
    tc[i].pad = 0;
    tiles += ((m + BM - 1) / BM) * tc[i].tiles_n;
    if (pair) {
      zo::TcMat tp = tc[i];
      tp.tile0 = ptiles;
      ptiles += ((m + UPAD - 1) / UPAD) * tp.tiles_n;
      tcp.push_back(tp);
    }
    urows += (m + UPAD - 1) / UPAD * UPAD;
    prows += (n + BN - 1) / BN * BN;
    for (int64_t r0 = 0; r0 < m; r0 += 128) uunits.push_back(make_int2(i, (int)r0));
  }
  if (urows >= (int64_t(1) << 31) || prows >= (int64_t(1) << 31))
    return refuse("more than 2^31 stacked operand rows");
  c->h_tc = tc;
  c->u_rows = urows;
  ZO_CUDA(cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, c->device), "SM count");
  const int64_t u_bytes = zo::tc_u_operand_bytes(c->r, urows);
  ZO_CUDA(cudaMalloc(&c->d_u_op, u_bytes), "cudaMalloc(U hi/lo)");
  ZO_CUDA(cudaMalloc(&c->d_p_hl, sizeof(uint16_t) * prows * HLW), "cudaMalloc(P hi/lo)");
  ZO_CUDA(cudaMemset(c->d_u_op, 0, u_bytes), "memset");
  ZO_CUDA(cudaMemset(c->d_p_hl, 0, sizeof(uint16_t) * prows * HLW), "memset");
  ZO_CUDA(cudaMalloc(&c->d_pinv, sizeof(float) * c->n_mats), "cudaMalloc(P scales)");
  ZO_CUDA(cudaMemset(c->d_pinv, 0, sizeof(float) * c->n_mats), "memset");
  ZO_CUDA(cudaMalloc(&c->d_amax, sizeof(float) * c->n_mats), "cudaMalloc(C maxima)");
  ZO_CUDA(cudaMemset(c->d_amax, 0, sizeof(float) * c->n_mats), "memset");
  ZO_CUDA(cudaMalloc(&c->d_tc, sizeof(zo::TcMat) * c->n_mats), "cudaMalloc(tile table)");
  ZO_CUDA(cudaMemcpy(c->d_tc, tc.data(), sizeof(zo::TcMat) * c->n_mats, cudaMemcpyHostToDevice),
          "upload tile table");
  if (pair) {
    ZO_CUDA(cudaMalloc(&c->d_tc_pair, sizeof(zo::TcMat) * c->n_mats), "cudaMalloc(pair tile table)");
    ZO_CUDA(cudaMemcpy(c->d_tc_pair, tcp.data(), sizeof(zo::TcMat) * c->n_mats,
                       cudaMemcpyHostToDevice),
            "upload pair tile table");
  }
  ZO_CUDA(cudaMalloc(&c->d_u_units, sizeof(int2) * uunits.size()), "cudaMalloc(units)");
  ZO_CUDA(cudaMemcpy(c->d_u_units, uunits.data(), sizeof(int2) * uunits.size(),
                     cudaMemcpyHostToDevice),
          "upload units");
  c->n_u_units = (int32_t)uunits.size();
  std::vector<CUtensorMap> wmaps(c->n_mats);
  bool ok = encode_f16_2d(&c->tm_b, c->d_p_hl, HLW, prows, HLW * 2, 64, 128);
  if (ok && !zo::wpass_tc_u_in_tmem(c->r))   // r <= 32: U rows read by TMA
    ok = encode_f16_2d(&c->tm_a, c->d_u_op, HLW, urows, HLW * 2, 64, 128);
  int32_t bad_w = -1;
  for (int32_t i = 0; ok && i < c->n_mats; ++i) {
    ok = encode_bf16_2d(&wmaps[i], mats[i].W, mats[i].n, mats[i].m, mats[i].ldw * 2, 64, 32);
    if (!ok) bad_w = i;
  }
  if (!ok) {
    const std::string why = bad_w >= 0 ? "cuTensorMapEncodeTiled rejected the descriptor of W_" +
                                             std::to_string(bad_w)
                                       : std::string("cuTensorMapEncodeTiled unavailable or "
                                                     "rejected an operand descriptor");
    return refuse(why.c_str());
  }
  ZO_CUDA(cudaMalloc(&c->d_w_maps, sizeof(CUtensorMap) * c->n_mats), "cudaMalloc(tensor maps)");
  ZO_CUDA(cudaMemcpy(c->d_w_maps, wmaps.data(), sizeof(CUtensorMap) * c->n_mats,
                     cudaMemcpyHostToDevice),
          "upload tensor maps");
  c->tc_tiles = tiles;
  c->tc_ok = true;
  if (pair) {
    // every pair is persistent over its share of the tiles: launch only as many pairs as
    // fit on the device at once
    c->n_pairs = zo::wpass_pair_max_pairs();
    c->pair_tiles = ptiles;
    c->pair_ok = c->n_pairs > 0 && encode_f16_2d(&c->tm_b64, c->d_p_hl, HLW, prows, HLW * 2, 64, 64);
    if (!c->pair_ok) return refuse("the SM-pair weight pass could not be set up");
  }
  // the projection P = C V^T on the tensor cores (every tensor-core rank): V_HL, C_HL
  const int64_t crows = (int64_t)c->n_mats * c->r;
  ZO_CUDA(cudaMalloc(&c->d_v_hl, sizeof(uint16_t) * prows * HLW), "cudaMalloc(V hi/lo)");
  ZO_CUDA(cudaMemset(c->d_v_hl, 0, sizeof(uint16_t) * prows * HLW), "memset");
  ZO_CUDA(cudaMalloc(&c->d_c_hl, sizeof(uint16_t) * crows * HLW), "cudaMalloc(C hi/lo)");
  ZO_CUDA(cudaMemset(c->d_c_hl, 0, sizeof(uint16_t) * crows * HLW), "memset");
  c->proj_tc = zo::project_tc_supported(c->r) &&
               encode_f16_2d(&c->tm_v, c->d_v_hl, HLW, prows, HLW * 2, 64, 128) &&
               encode_f16_2d(&c->tm_c, c->d_c_hl, HLW, crows, HLW * 2, 64, (uint32_t)c->r) &&
               encode_f16_2d(&c->tm_p, c->d_p_hl, HLW, prows, HLW * 2, 64, 32);
  if (!c->proj_tc) {
    c->tc_ok = false;
    return refuse("cuTensorMapEncodeTiled rejected a projection descriptor");
  }
  return ZO_OK;
}

}  // namespace

extern "C" {

const char* zo_status_string(int32_t s) {
  switch (s) {
    case ZO_OK: return "ok";
    case ZO_ERR_INVALID_ARG: return "invalid argument";
    case ZO_ERR_SHAPE: return "unsupported or inconsistent shape";
    case ZO_ERR_ALIGN: return "misaligned buffer";
    case ZO_ERR_DTYPE: return "unknown dtype";
    case ZO_ERR_CUDA: return "CUDA error";
    case ZO_ERR_TIMEOUT: return "device-side wait timed out";
    case ZO_ERR_UNSUPPORTED: return "unsupported request";
    case ZO_ERR_NOMEM: return "out of device memory";
    default: return "unknown status";
  }
}

const char* zo_last_error(void) { return g_last_error.c_str(); }

zo_status zo_create(zo_ctx** out, const zo_matrix* mats, int32_t n_mats, int32_t r, int32_t q,
                    uint64_t seed, uint32_t matrix_index_base, void* stream) {
  if (!out) return ZO_ERR_INVALID_ARG;
  *out = nullptr;
  if (!mats || n_mats <= 0) {
    g_last_error = "need at least one matrix";
    return ZO_ERR_INVALID_ARG;
  }
  if (!supported_rank(r)) {
    g_last_error = "rank r must be one of 4, 8, 16, 32, 64, 128";
    return ZO_ERR_SHAPE;
  }
  if (q < 1 || q > 4096) {
    g_last_error = "q must be in [1, 4096]";
    return ZO_ERR_INVALID_ARG;
  }
  for (int32_t i = 0; i < n_mats; ++i) {
    zo_status st = validate_matrix(mats[i], r);
    if (st != ZO_OK) return st;
  }
  int dev = 0;
  ZO_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  cudaDeviceProp prop;
  ZO_CUDA(cudaGetDeviceProperties(&prop, dev), "cudaGetDeviceProperties");
  if (!(prop.major == 10 && prop.minor == 3)) {
    g_last_error = "this library is built for sm_103a (GB300) only; found sm_" +
                   std::to_string(prop.major) + std::to_string(prop.minor);
    return ZO_ERR_CUDA;
  }

  zo_ctx* c = new zo_ctx();
  c->device = dev;
  c->sms = prop.multiProcessorCount;
  c->stream = reinterpret_cast<cudaStream_t>(stream);
  c->n_mats = n_mats;
  c->r = r;
  c->q = q;
  c->seed = seed;
  c->base = matrix_index_base;

  // coefficient workspace: C_i (r*r) then P_i (r*n_i) per matrix
  int64_t coeff_floats = 0;
  std::vector<int64_t> c_off(n_mats), p_off(n_mats);
  for (int32_t i = 0; i < n_mats; ++i) {
    c_off[i] = coeff_floats;
    coeff_floats += (int64_t)r * r;
    p_off[i] = coeff_floats;
    coeff_floats += ((int64_t)r * mats[i].n + 3) / 4 * 4;
  }
  auto fail = [&](zo_status st) {
    free_ctx(c);
    return st;
  };
  cudaError_t e = cudaMalloc(&c->d_coeff_ws, sizeof(float) * coeff_floats);
  if (e != cudaSuccess) {
    cuda_fail(e, "cudaMalloc(coefficient workspace)");
    return fail(ZO_ERR_NOMEM);
  }

  // weight-pass tiles and projection units
  std::vector<int64_t> prefix(n_mats + 1, 0);
  std::vector<int2> units;
  c->h_mats.resize(n_mats);
  for (int32_t i = 0; i < n_mats; ++i) {
    const zo_matrix& mt = mats[i];
    zo::MatDesc d{};
    d.W = mt.W;
    d.m = mt.m;
    d.n = mt.n;
    d.ldw = mt.ldw;
    d.dtype = mt.dtype;
    d.gidx = matrix_index_base + (uint32_t)i;
    d.U = mt.U;
    d.V = mt.V;
    d.M = mt.M;
    d.Vm = mt.Vm;
    d.C = c->d_coeff_ws + c_off[i];
    d.P = c->d_coeff_ws + p_off[i];
    const int tn = zo::fma_tile_cols(mt.dtype);
    const int64_t tiles = ((mt.m + zo::kFmaTileRows - 1) / zo::kFmaTileRows) * ((mt.n + tn - 1) / tn);
    d.tile0 = prefix[i];
    prefix[i + 1] = prefix[i] + tiles;
    for (int64_t j0 = 0; j0 < mt.n; j0 += 128) units.push_back(make_int2(i, (int)j0));
    c->h_mats[i] = d;
  }
  c->n_tiles = prefix[n_mats];
  c->n_proj_units = (int32_t)units.size();
  if (c->n_tiles > 0x7FFFFFFF) {
    g_last_error = "too many weight-pass tiles";
    return fail(ZO_ERR_SHAPE);
  }

  // refresh plan (dry run for sizes, then the real pass with pointers)
  const int32_t B = zo::qr_block_rows(r);
  int64_t qr_floats = 0;
  // a panel with rows >= 4r has kappa(Omega) <= ~3, well inside CholeskyQR2's range
  auto use_cholqr = [&](int64_t rows) { return zo::cholqr_supported(r) && rows >= 4 * (int64_t)r; };
  {
    std::vector<QrLevel> dry;
    for (int32_t i = 0; i < n_mats; ++i) {
      if (!use_cholqr(mats[i].m)) plan_panel(nullptr, mats[i].m, r, 0, zo::kTagOmegaU, B, dry, nullptr, &qr_floats);
      if (!use_cholqr(mats[i].n)) plan_panel(nullptr, mats[i].n, r, 0, zo::kTagOmegaV, B, dry, nullptr, &qr_floats);
    }
  }
  e = cudaMalloc(&c->d_qr_ws, sizeof(float) * std::max<int64_t>(qr_floats, 4));
  if (e != cudaSuccess) {
    cuda_fail(e, "cudaMalloc(refresh workspace)");
    return fail(ZO_ERR_NOMEM);
  }
  std::vector<QrLevel> levels;
  int64_t off = 0;
  std::vector<zo::CqPanel> cq_panels;
  std::vector<zo::CqChunk> cq_chunks;
  auto add_cholqr = [&](float* out, int64_t rows, uint32_t gidx, uint32_t tag) {
    zo::CqPanel p{out, rows, gidx, tag, (int32_t)cq_chunks.size(), 0};
    for (int64_t r0 = 0; r0 < rows; r0 += zo::kCqChunkRows) {
      cq_chunks.push_back({r0, (int32_t)cq_panels.size(),
                           (int32_t)std::min<int64_t>(zo::kCqChunkRows, rows - r0)});
      ++p.n_chunks;
    }
    cq_panels.push_back(p);
  };
  for (int32_t i = 0; i < n_mats; ++i) {
    const uint32_t gidx = matrix_index_base + (uint32_t)i;
    if (use_cholqr(mats[i].m)) add_cholqr(mats[i].U, mats[i].m, gidx, zo::kTagOmegaU);
    else plan_panel(mats[i].U, mats[i].m, r, gidx, zo::kTagOmegaU, B, levels, c->d_qr_ws, &off);
    if (use_cholqr(mats[i].n)) add_cholqr(mats[i].V, mats[i].n, gidx, zo::kTagOmegaV);
    else plan_panel(mats[i].V, mats[i].n, r, gidx, zo::kTagOmegaV, B, levels, c->d_qr_ws, &off);
  }
  c->n_cq_panels = (int32_t)cq_panels.size();
  c->n_cq_chunks = (int32_t)cq_chunks.size();
  std::vector<zo::QrBlock> all_blocks;
  for (auto& lv : levels) {
    c->up_off.push_back((int64_t)all_blocks.size());
    c->up_cnt.push_back((int64_t)lv.up.size());
    all_blocks.insert(all_blocks.end(), lv.up.begin(), lv.up.end());
    c->down_off.push_back((int64_t)all_blocks.size());
    c->down_cnt.push_back((int64_t)lv.down.size());
    all_blocks.insert(all_blocks.end(), lv.down.begin(), lv.down.end());
  }

  c->max_losses = std::max(2 * q, q + 1);
  e = cudaMalloc(&c->d_losses, sizeof(float) * c->max_losses);
  if (e == cudaSuccess) e = cudaMalloc(&c->d_mats, sizeof(zo::MatDesc) * n_mats);
  if (e == cudaSuccess) e = cudaMalloc(&c->d_tile_prefix, sizeof(int64_t) * (n_mats + 1));
  if (e == cudaSuccess) e = cudaMalloc(&c->d_proj_units, sizeof(int2) * std::max<size_t>(units.size(), 1));
  if (e == cudaSuccess) e = cudaMalloc(&c->d_qr_blocks, sizeof(zo::QrBlock) * std::max<size_t>(all_blocks.size(), 1));
  if (e == cudaSuccess) e = cudaMalloc(&c->d_status, sizeof(uint32_t));
  if (e == cudaSuccess && c->n_cq_panels > 0) {
    e = cudaMalloc(&c->d_cq_panels, sizeof(zo::CqPanel) * cq_panels.size());
    if (e == cudaSuccess) e = cudaMalloc(&c->d_cq_chunks, sizeof(zo::CqChunk) * cq_chunks.size());
    if (e == cudaSuccess)
      e = cudaMalloc(&c->d_cq_partial, sizeof(float) * (size_t)cq_chunks.size() * r * r);
    if (e == cudaSuccess)
      e = cudaMalloc(&c->d_cq_linv, sizeof(float) * (size_t)cq_panels.size() * r * r);
  }
  if (e != cudaSuccess) {
    cuda_fail(e, "cudaMalloc(context tables)");
    return fail(ZO_ERR_NOMEM);
  }
  e = cudaMemcpy(c->d_mats, c->h_mats.data(), sizeof(zo::MatDesc) * n_mats, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(c->d_tile_prefix, prefix.data(), sizeof(int64_t) * (n_mats + 1), cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !units.empty())
    e = cudaMemcpy(c->d_proj_units, units.data(), sizeof(int2) * units.size(), cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !all_blocks.empty())
    e = cudaMemcpy(c->d_qr_blocks, all_blocks.data(), sizeof(zo::QrBlock) * all_blocks.size(),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess && c->n_cq_panels > 0)
    e = cudaMemcpy(c->d_cq_panels, cq_panels.data(), sizeof(zo::CqPanel) * cq_panels.size(),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess && c->n_cq_panels > 0)
    e = cudaMemcpy(c->d_cq_chunks, cq_chunks.data(), sizeof(zo::CqChunk) * cq_chunks.size(),
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(c->d_status, 0, sizeof(uint32_t));
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cuda_fail(e, "zo_create upload");
    return fail(ZO_ERR_CUDA);
  }
  zo_status st = setup_tc(c, mats);
  if (st != ZO_OK) return fail(st);
  st = setup_narrow(c, mats);
  if (st != ZO_OK) return fail(st);
  e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cuda_fail(e, "zo_create tensor-core setup");
    return fail(ZO_ERR_CUDA);
  }
  *out = c;
  return ZO_OK;
}

zo_status zo_destroy(zo_ctx* c) {
  if (!c) return ZO_OK;
  DeviceGuard guard(c->device);
  cudaError_t e = cudaStreamSynchronize(c->stream);
  free_ctx(c);
  if (e != cudaSuccess) return cuda_fail(e, "zo_destroy");
  return ZO_OK;
}

zo_status zo_refresh(zo_ctx* c, uint32_t refresh_idx, int32_t reset_moments) {
  if (!c) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  c->linear_ready = false;   // a prepared P_K belongs to the old V
  const int n_levels = (int)c->up_off.size();
  for (int lv = 0; lv < n_levels; ++lv) {
    if (c->up_cnt[lv] == 0) continue;
    ZO_CUDA(zo::launch_qr_up(c->d_qr_blocks + c->up_off[lv], (int32_t)c->up_cnt[lv], c->r, c->seed,
                             refresh_idx, c->d_status, c->stream),
            "refresh up-pass kernel");
    ++c->launches;
  }
  for (int lv = n_levels - 1; lv >= 0; --lv) {
    if (c->down_cnt[lv] == 0) continue;
    ZO_CUDA(zo::launch_qr_down(c->d_qr_blocks + c->down_off[lv], (int32_t)c->down_cnt[lv], c->r,
                               c->d_status, c->stream),
            "refresh down-pass kernel");
    ++c->launches;
  }
  if (c->n_cq_panels > 0) {
    ZO_CUDA(zo::launch_cholqr(c->d_cq_panels, c->n_cq_panels, c->d_cq_chunks, c->n_cq_chunks,
                              c->d_cq_partial, c->d_cq_linv, c->r, c->seed, refresh_idx,
                              c->d_status, c->stream),
            "refresh CholeskyQR2 kernels");
    c->launches += 6;
  }
  if (reset_moments) {
    ZO_CUDA(zo::launch_zero_moments(c->d_mats, c->n_mats, c->r, c->stream), "zero moments");
    ++c->launches;
  }
  c->u_lin_valid = false;   // the linear route's bf16 U operand belongs to the old U
  if (c->tc_ok) {
    ZO_CUDA(zo::launch_split_u(c->d_mats, c->d_tc, c->d_u_units, c->n_u_units, c->r, c->d_u_op,
                               c->stream),
            "split U into hi/lo");
    ++c->launches;
    if (c->proj_tc) {
      ZO_CUDA(zo::launch_split_v(c->d_mats, c->d_tc, c->d_proj_units, c->n_proj_units, c->r,
                                 c->d_v_hl, c->stream),
              "split V into hi/lo");
      ++c->launches;
    }
  }
  return ZO_OK;
}

zo_status zo_init_subspace(zo_ctx* c, uint32_t refresh_idx) {
  return zo_refresh(c, refresh_idx, 1);
}

zo_status zo_perturb(zo_ctx* c, uint32_t t, int32_t qa, float ca, int32_t qb, float cb, float eps) {
  if (!c) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  if (qa < 0 || qa >= c->q || qb < -1 || qb >= c->q || !std::isfinite(ca) || !std::isfinite(cb) ||
      !std::isfinite(eps)) {
    g_last_error = "zo_perturb: query index out of range or non-finite scalar";
    return ZO_ERR_INVALID_ARG;
  }
  if (tc_refused(c)) return refuse_tc(c);
  zo::CoeffParams p{};
  p.mode = zo::kCoeffPerturb;
  p.seed = c->seed;
  p.t = t;
  p.r = c->r;
  p.q = c->q;
  p.qa = qa;
  p.qb = qb;
  p.ca = ca;
  p.cb = cb;
  p.eps = eps;
  const bool use_tc = tc_path(c);
  p.amax = use_tc ? c->d_amax : nullptr;
  if (!use_tc && narrow_path(c)) {
    zo_status st = record_start(c);
    if (st != ZO_OK) return st;
    ZO_CUDA(zo::launch_wpass_narrow(c->d_mats, c->d_narrow, c->d_narrow_tiles,
                                    c->n_narrow_tiles, p, c->narrow_p, c->narrow_u, c->stream),
            "narrow-tile weight-pass kernel");
    c->last_path = 3;
    ++c->launches;
    return record_stop(c);
  }
  if (!use_tc && zo::wpass_fma_fused_supported(c->r) && c->n_tiles <= 4 * (int64_t)c->sms) {
    // small r on the FMA path and a pass of a few waves at most (launch-bound, as for
    // sets that fit in L2): C, P and the weight update in one launch.  On larger passes
    // every CTA drawing C again costs more than the two launches it saves.
    zo_status st = record_start(c);
    if (st != ZO_OK) return st;
    ZO_CUDA(zo::launch_wpass_fma_fused(c->d_mats, c->n_mats, c->d_tile_prefix, c->n_tiles, p,
                                       c->stream),
            "fused weight-pass kernel");
    c->last_path = 1;
    ++c->launches;
    return record_stop(c);
  }
  ZO_CUDA(zo::launch_coeff(c->d_mats, c->n_mats, p, c->stream), "coefficient kernel");
  ++c->launches;
  return run_weight_pass(c);
}

zo_status zo_step(zo_ctx* c, uint32_t t, int32_t adam_t, const float* losses, int32_t n_losses,
                  int32_t losses_on_host, int32_t scheme, int32_t optimizer, float eps, float lr,
                  float beta1, float beta2, float eps_adam, int32_t restore_query,
                  float restore_coef, float* gamma_out) {
  if (!c || !losses) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  int32_t want = -1;
  if (scheme == ZO_SCHEME_CENTRAL) want = 2 * c->q;
  else if (scheme == ZO_SCHEME_FORWARD) want = c->q + 1;
  else if (scheme == ZO_SCHEME_DIRECT) want = c->q;
  if (want < 0 || n_losses != want) {
    g_last_error = "zo_step: unknown scheme or wrong number of losses";
    return ZO_ERR_INVALID_ARG;
  }
  if (optimizer != ZO_OPT_ADAM && optimizer != ZO_OPT_SGD) {
    g_last_error = "zo_step: unknown optimizer";
    return ZO_ERR_INVALID_ARG;
  }
  if (restore_query < -1 || restore_query >= c->q || !std::isfinite(eps) || !std::isfinite(lr) ||
      !std::isfinite(restore_coef) || (scheme != ZO_SCHEME_DIRECT && eps == 0.0f)) {
    g_last_error = "zo_step: restore query out of range or bad scalar";
    return ZO_ERR_INVALID_ARG;
  }
  double inv_bc1 = 1.0, inv_bc2 = 1.0;
  if (optimizer == ZO_OPT_ADAM) {
    if (adam_t < 1 || !(beta1 >= 0.0f && beta1 < 1.0f) || !(beta2 >= 0.0f && beta2 < 1.0f) ||
        !(eps_adam >= 0.0f)) {
      g_last_error = "zo_step: need adam_t >= 1, betas in [0, 1), eps_adam >= 0";
      return ZO_ERR_INVALID_ARG;
    }
    inv_bc1 = 1.0 / (1.0 - std::pow((double)beta1, (double)adam_t));
    inv_bc2 = 1.0 / (1.0 - std::pow((double)beta2, (double)adam_t));
  }
  if (tc_refused(c)) return refuse_tc(c);
  const float* d_losses = losses;
  if (losses_on_host) {
    ZO_CUDA(cudaMemcpyAsync(c->d_losses, losses, sizeof(float) * n_losses, cudaMemcpyHostToDevice,
                            c->stream),
            "copy losses to device");
    d_losses = c->d_losses;
  }
  zo::CoeffParams p{};
  p.mode = zo::kCoeffStep;
  p.seed = c->seed;
  p.t = t;
  p.r = c->r;
  p.q = c->q;
  p.eps = eps;
  p.losses = d_losses;
  p.n_losses = n_losses;
  p.scheme = scheme;
  p.optimizer = optimizer;
  p.lr = lr;
  p.beta1 = beta1;
  p.beta2 = beta2;
  p.eps_adam = eps_adam;
  p.inv_bc1 = (float)inv_bc1;
  p.inv_bc2 = (float)inv_bc2;
  p.restore_query = restore_query;
  p.restore_coef = restore_coef;
  p.gamma_out = gamma_out;
  p.amax = tc_path(c) ? c->d_amax : nullptr;
  ZO_CUDA(zo::launch_coeff(c->d_mats, c->n_mats, p, c->stream), "coefficient kernel");
  ++c->launches;
  return run_weight_pass(c);
}

zo_status zo_linear_prepare(zo_ctx* c, uint32_t t, int32_t qa, float ca, int32_t qb, float cb,
                            float eps) {
  if (!c) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  if (!c->tc_ok || !zo::linear_supported(c->r)) {
    g_last_error = "zo_linear_prepare needs the tensor-core path with r in {16, 32, 64, 128}";
    return ZO_ERR_UNSUPPORTED;
  }
  if (qa < 0 || qa >= c->q || qb < -1 || qb >= c->q || !std::isfinite(ca) || !std::isfinite(cb) ||
      !std::isfinite(eps)) {
    g_last_error = "zo_linear_prepare: query index out of range or non-finite scalar";
    return ZO_ERR_INVALID_ARG;
  }
  const int32_t r = c->r;
  if (!c->d_pk) {
    c->h_pk_off.assign(c->n_mats, 0);
    int64_t total = 0;
    for (int32_t i = 0; i < c->n_mats; ++i) {
      c->h_pk_off[i] = total;
      total += zo::linear_pk_elems(c->h_mats[i].n, r);
    }
    __nv_bfloat16* pk = nullptr;
    int64_t* pk_off = nullptr;
    cudaError_t e = cudaMalloc(&pk, sizeof(__nv_bfloat16) * total);
    if (e == cudaSuccess) e = cudaMalloc(&pk_off, sizeof(int64_t) * c->n_mats);
    // on the context's stream, ahead of the kernels that read it (the host copy stays)
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(pk_off, c->h_pk_off.data(), sizeof(int64_t) * c->n_mats,
                          cudaMemcpyHostToDevice, c->stream);
    if (e != cudaSuccess) {
      cudaFree(pk);
      cudaFree(pk_off);
      return cuda_fail(e, "P_K workspace");
    }
    c->d_pk = pk;
    c->d_pk_off = pk_off;
  }
  if (!c->d_u_lin) {
    // the route's U operand: the bf16 pair of U in rows of tc_hl_width(r), stacked like
    // d_u_op's at r <= 32
    const int64_t HLW = zo::tc_hl_width(r);
    const size_t bytes = sizeof(__nv_bfloat16) * (size_t)c->u_rows * HLW;
    __nv_bfloat16* u_lin = nullptr;
    cudaError_t e = cudaMalloc(&u_lin, bytes);
    // padding rows and columns stay zero; on the context's stream, before the split
    if (e == cudaSuccess) e = cudaMemsetAsync(u_lin, 0, bytes, c->stream);
    if (e != cudaSuccess) {
      cudaFree(u_lin);
      return cuda_fail(e, "linear U operand");
    }
    if (!encode_bf16_2d(&c->tm_u_lin, u_lin, HLW, c->u_rows, HLW * 2, 64, 128)) {
      cudaFree(u_lin);
      g_last_error = "zo_linear_prepare: cuTensorMapEncodeTiled rejected the U operand descriptor";
      return ZO_ERR_CUDA;
    }
    c->d_u_lin = u_lin;
    c->u_lin_valid = false;
  }
  if (!c->u_lin_valid) {
    ZO_CUDA(zo::launch_split_u_bf16(c->d_mats, c->d_tc, c->d_u_units, c->n_u_units, r, c->d_u_lin,
                                    c->stream),
            "split U into a bf16 pair");
    ++c->launches;
    c->u_lin_valid = true;
  }
  // C_i = eps (ca Z_qa + cb Z_qb) for every matrix, P_i = C_i V_i^T, P_K = [P_hi ; P_lo]
  zo::CoeffParams p{};
  p.mode = zo::kCoeffPerturb;
  p.seed = c->seed;
  p.t = t;
  p.r = r;
  p.q = c->q;
  p.qa = qa;
  p.qb = qb;
  p.ca = ca;
  p.cb = cb;
  p.eps = eps;
  p.amax = c->d_amax;
  ZO_CUDA(zo::launch_coeff(c->d_mats, c->n_mats, p, c->stream), "coefficient kernel");
  ZO_CUDA(zo::launch_split_c(c->d_mats, c->n_mats, r, c->d_amax, c->d_c_hl, c->d_pinv, c->stream),
          "split C");
  ZO_CUDA(zo::launch_project_tc_pk(c->tm_v, c->tm_c, c->d_tc, c->d_proj_units, c->n_proj_units,
                                   std::min<int32_t>(c->n_proj_units, c->sms), r, c->d_pinv,
                                   c->d_pk_off, c->d_pk, c->d_status, c->stream),
          "tensor-core projection kernel (P_K)");
  c->launches += 3;
  c->linear_ready = true;
  return ZO_OK;
}

zo_status zo_linear_perturbed(zo_ctx* c, int32_t mat, const void* X, int64_t T, int64_t ldx,
                              void* Y, int64_t ldy) {
  if (!c || !X || !Y) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  if (!c->linear_ready) {
    g_last_error = "zo_linear_perturbed: call zo_linear_prepare first";
    return ZO_ERR_INVALID_ARG;
  }
  if (mat < 0 || mat >= c->n_mats) {
    g_last_error = "zo_linear_perturbed: matrix index out of range";
    return ZO_ERR_INVALID_ARG;
  }
  const zo::MatDesc& md = c->h_mats[mat];
  const int64_t m = md.m, n = md.n;
  if (T < 1 || T >= (int64_t(1) << 31) || ldx < n || ldy < m || m % 8 != 0) {
    // (Y's rows are written by TMA in 16-byte chunks: m % 8 keeps them inside Y's columns)
    g_last_error = "zo_linear_perturbed: need 1 <= T < 2^31, ldx >= n, ldy >= m, m % 8 == 0";
    return ZO_ERR_SHAPE;
  }
  if (!aligned16(X) || !aligned16(Y) || (ldx * 2) % 16 != 0 || (ldy * 2) % 16 != 0) {
    g_last_error = "zo_linear_perturbed: X, Y and their row strides must be 16-byte aligned";
    return ZO_ERR_ALIGN;
  }
  const int32_t r = c->r;
  const int64_t HLW = zo::tc_hl_width(r);
  // the Y GEMM's tiling: automatic = the pair tiling whose busiest pair has the least
  // operand traffic (the single-CTA tilings if no cluster of the pair kernel fits), or the
  // one ZO_OPTION_LINEAR_TILE names
  if (c->linear_pairs < 0) c->linear_pairs = std::max(0, (int)zo::linear_pair_max_pairs());
  int32_t tiling = c->linear_tile;
  if (tiling == 0)
    tiling = c->linear_pairs > 0 || !zo::linear_single_cta_supported(r)
                 ? zo::linear_pair_tiling(T, m, n, r, c->linear_pairs)
                 : zo::linear_y_tiling(T, m, c->sms, 0);
  const int32_t pair_n = zo::linear_pair_cols(tiling);
  if (pair_n > 0 && c->linear_pairs <= 0) {
    g_last_error = "zo_linear_perturbed: no cluster of the SM-pair GEMM fits on this device";
    return ZO_ERR_UNSUPPORTED;
  }
  if (pair_n == 0 && !zo::linear_single_cta_supported(r)) {
    g_last_error = "zo_linear_perturbed: the single-CTA tilings 1..3 take r in {16, 32}";
    return ZO_ERR_UNSUPPORTED;
  }
  // S's K split: the single-CTA route's S kernel, or the pair launch's plan (contributor
  // tiles, or S tiles); each split writes k_split x T x r fp32 partials
  int32_t k_split = 1, k_chunk = 1;
  zo::LinearPairPlan plan{};
  if (pair_n > 0) {
    plan = zo::linear_pair_plan(T, m, n, r, tiling, c->linear_pairs);
    if (plan.pairs <= 0) {
      g_last_error = "zo_linear_perturbed: no SM-pair plan for this shape";
      return ZO_ERR_UNSUPPORTED;
    }
    k_split = std::max<int32_t>(1, plan.s_split);
  } else {
    zo::linear_s_split(T, n, c->sms, &k_split, &k_chunk);
  }
  const int64_t part = (int64_t)k_split * T * r;
  if (T > c->s_cap || part > c->part_cap) {
    ZO_CUDA(cudaStreamSynchronize(c->stream), "stream synchronize");
    if (T > c->s_cap) {
      cudaFree(c->d_s_hl);
      cudaFree(c->d_s_count);
      cudaFree(c->d_s_flags);
      c->d_s_hl = nullptr;
      c->d_s_count = nullptr;
      c->d_s_flags = nullptr;
      c->s_cap = 0;
      const int64_t cap = (T + 127) / 128 * 128;
      const int64_t n_flags = (cap / 256 + 1) * zo::kLinearPairCounters;
      ZO_CUDA(cudaMalloc(&c->d_s_hl, sizeof(__nv_bfloat16) * cap * HLW), "cudaMalloc(S_HL)");
      ZO_CUDA(cudaMalloc(&c->d_s_count, sizeof(uint32_t) * (cap / 32)), "cudaMalloc(S counters)");
      ZO_CUDA(cudaMalloc(&c->d_s_flags, sizeof(uint32_t) * n_flags),
              "cudaMalloc(S row-block counters)");
      // on the context's stream: a plain cudaMemset runs on the legacy default stream,
      // which a non-blocking stream's kernels are not ordered after
      ZO_CUDA(cudaMemsetAsync(c->d_s_count, 0, sizeof(uint32_t) * (cap / 32), c->stream),
              "zero S counters");
      ZO_CUDA(cudaMemsetAsync(c->d_s_flags, 0, sizeof(uint32_t) * n_flags, c->stream),
              "zero S row-block counters");
      c->lin_epoch = 0;
      c->s_cap = cap;
    }
    if (part > c->part_cap) {
      cudaFree(c->d_s_part);
      c->d_s_part = nullptr;
      c->part_cap = 0;
      ZO_CUDA(cudaMalloc(&c->d_s_part, sizeof(float) * part), "cudaMalloc(partial S)");
      c->part_cap = part;
    }
  }
  const bool narrow_y = pair_n == 0 && zo::linear_y_tile_cols(tiling) % 64 != 0;
  CUtensorMap tm_x{}, tm_pk{}, tm_s{}, tm_y{}, tm_w{}, tm_u{}, tm_pk_half{}, tm_ps{};
  bool enc =
      encode_bf16_2d(&tm_x, const_cast<void*>(X), n, T, ldx * 2, 64, 128) &&
      encode_bf16_2d(&tm_pk, c->d_pk + c->h_pk_off[mat], n, 2 * r, (n + 63) / 64 * 64 * 2, 64,
                     (uint32_t)(2 * r)) &&
      encode_bf16_2d(&tm_s, c->d_s_hl, HLW, T, HLW * 2, 64, 128);
  if (pair_n > 0) {
    // W_i and the U operand in boxes of N/2 rows (each CTA of a pair loads half of the
    // tile's B rows), Y in 32 x 16 boxes
    enc = enc && encode_bf16_2d(&tm_w, md.W, n, m, md.ldw * 2, 64, (uint32_t)(pair_n / 2)) &&
          encode_bf16_2d(&tm_u, c->d_u_lin, HLW, c->u_rows, HLW * 2, 64, (uint32_t)(pair_n / 2)) &&
          encode_bf16_2d(&tm_y, Y, m, T, ldy * 2, 16, 32, CU_TENSOR_MAP_SWIZZLE_32B) &&
          // P_K in boxes of r rows: CTA 0 of a pair loads P_hi, CTA 1 P_lo; and in boxes of a
          // contributor's slice rows
          encode_bf16_2d(&tm_pk_half, c->d_pk + c->h_pk_off[mat], n, 2 * r, (n + 63) / 64 * 64 * 2,
                         64, (uint32_t)r) &&
          encode_bf16_2d(&tm_ps, c->d_pk + c->h_pk_off[mat], n, 2 * r, (n + 63) / 64 * 64 * 2,
                         64, (uint32_t)(plan.n_contrib > 0 ? plan.s_cols / 2 : r));
  } else {
    enc = enc && (narrow_y ? encode_bf16_2d(&tm_y, Y, m, T, ldy * 2, 32, 32,
                                            CU_TENSOR_MAP_SWIZZLE_64B)
                           : encode_bf16_2d(&tm_y, Y, m, T, ldy * 2, 64, 32));
  }
  if (!enc) {
    g_last_error = "zo_linear_perturbed: cuTensorMapEncodeTiled rejected a descriptor";
    return ZO_ERR_CUDA;
  }
  if (pair_n > 0) {
    // one launch: S = X P^T (in contributor tiles or S tiles) and Y = X W^T + S U^T
    if (c->lin_epoch + 1 >= zo::kLinearPairEpochs) {
      // the epochs start again: no counter may hold an old call's complete count
      ZO_CUDA(cudaMemsetAsync(c->d_s_flags, 0,
                              sizeof(uint32_t) * (c->s_cap / 256 + 1) * zo::kLinearPairCounters,
                              c->stream),
              "zero S row-block counters");
      c->lin_epoch = 0;
    }
    ++c->lin_epoch;
    const bool inject = c->inject_wait;    // the test hook is one-shot
    c->inject_wait = false;
    ZO_CUDA(zo::launch_linear_pair(tm_x, tm_w, tm_s, tm_u, tm_y, tm_pk_half, tm_ps, T, m, n,
                                   c->h_tc[mat].u_row0, r, tiling, plan, c->d_s_hl, c->d_s_part,
                                   c->d_s_flags, c->lin_epoch, inject, c->d_status, c->stream),
            "perturbed linear kernel (SM pairs)");
    c->launches += 1;
  } else {
    // S = X P^T (split K, the partial sums reduced into S_HL), Y = X W^T + S U^T
    ZO_CUDA(zo::launch_linear_s(tm_x, tm_pk, T, n, r, k_split, k_chunk, c->d_s_part, c->d_s_hl,
                                c->d_s_count, c->sms, c->d_status, c->stream),
            "S = X P^T kernels");
    ZO_CUDA(zo::launch_linear_y(tm_x, c->d_w_maps + mat, tm_s, c->tm_u_lin, tm_y, T, m, n,
                                c->h_tc[mat].u_row0, r, tiling, c->sms, c->d_status, c->stream),
            "perturbed linear kernel");
    c->launches += 1 + zo::linear_s_launches(k_split);
  }
  c->last_linear_tiling = tiling;
  return ZO_OK;
}

zo_status zo_mezo_perturb(zo_ctx* c, uint32_t t, float coef) {
  if (!c) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  if (!std::isfinite(coef)) {
    g_last_error = "zo_mezo_perturb: non-finite coefficient";
    return ZO_ERR_INVALID_ARG;
  }
  for (const auto& d : c->h_mats) {
    if (d.m * ((d.n + 3) / 4) >= (int64_t(1) << 32)) {
      g_last_error = "zo_mezo_perturb: matrix too large for the 32-bit counter word";
      return ZO_ERR_SHAPE;
    }
  }
  zo_status st = record_start(c);
  if (st != ZO_OK) return st;
  ZO_CUDA(zo::launch_mezo(c->d_mats, c->n_mats, c->d_tile_prefix, c->n_tiles, c->seed, t, coef,
                          c->stream),
          "full-space perturbation kernel");
  ++c->launches;
  return record_stop(c);
}

zo_status zo_sync_status(zo_ctx* c) {
  if (!c) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  ZO_CUDA(cudaStreamSynchronize(c->stream), "stream synchronize");
  uint32_t s = 0;
  ZO_CUDA(cudaMemcpy(&s, c->d_status, sizeof(s), cudaMemcpyDeviceToHost), "read status");
  if (s != 0) {
    // cleared on the context's stream (ordered before its next kernels) and waited for
    ZO_CUDA(cudaMemsetAsync(c->d_status, 0, sizeof(uint32_t), c->stream), "clear status");
    // a perturbed-linear S kernel cut short can leave its group counters part-counted, and
    // an SM-pair launch its row-block counters
    if ((s & zo::kDevTimeout) && c->d_s_count)
      ZO_CUDA(cudaMemsetAsync(c->d_s_count, 0, sizeof(uint32_t) * (c->s_cap / 32), c->stream),
              "zero S counters");
    if ((s & zo::kDevTimeout) && c->d_s_flags) {
      ZO_CUDA(cudaMemsetAsync(c->d_s_flags, 0,
                              sizeof(uint32_t) * (c->s_cap / 256 + 1) * zo::kLinearPairCounters,
                              c->stream),
              "zero S row-block counters");
      c->lin_epoch = 0;
    }
    ZO_CUDA(cudaStreamSynchronize(c->stream), "stream synchronize");
    if (s & zo::kDevTimeout) {
      g_last_error = "a device-side wait ran out";
      return ZO_ERR_TIMEOUT;
    }
    g_last_error = (s & zo::kDevNotPosDef)
                       ? "refresh: a Gram matrix of a panel was not positive definite"
                       : "a device-side bound check failed";
    return ZO_ERR_CUDA;
  }
  return ZO_OK;
}

zo_status zo_set_option(zo_ctx* c, int32_t option, int64_t value) {
  if (!c) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  if (option == ZO_OPTION_WPASS_PATH) {
    if (value < 0 || value > 3) return ZO_ERR_INVALID_ARG;
    if (value == 2 && !c->tc_ok) {
      g_last_error = "the tensor-core weight pass needs every W in bf16 with n a multiple of 8, "
                     "and r in {16, 32, 64, 128}";
      return ZO_ERR_UNSUPPORTED;
    }
    if (value == 3 && !c->narrow_ok) {
      g_last_error = "the narrow-tile weight pass needs r in {4, 8}";
      return ZO_ERR_UNSUPPORTED;
    }
    c->path_option = (int)value;
    return ZO_OK;
  }
  if (option == ZO_OPTION_TEST_WAIT_TIMEOUT) {
    if (value != 0 && value != 1) return ZO_ERR_INVALID_ARG;
    if (value == 1 && !c->tc_ok) {
      g_last_error = "the wait-timeout test hook needs the tensor-core weight pass";
      return ZO_ERR_UNSUPPORTED;
    }
    c->inject_wait = value != 0;
    return ZO_OK;
  }
  if (option == ZO_OPTION_LINEAR_TILE) {
    if (value < 0 || value >= zo::kLinearPairTiling0 + 5) return ZO_ERR_INVALID_ARG;
    c->linear_tile = (int)value;
    return ZO_OK;
  }
  if (option == ZO_OPTION_PAIR_MMA) {
    if (value != 0 && value != 1) return ZO_ERR_INVALID_ARG;
    if (value == 1 && !c->pair_ok) {
      g_last_error = "the SM-pair weight pass needs the tensor-core path at r = 128";
      return ZO_ERR_UNSUPPORTED;
    }
    c->pair_option = (int)value;
    return ZO_OK;
  }
  if (option == ZO_OPTION_TIMING) {
    if (value != 0 && value != 1) return ZO_ERR_INVALID_ARG;
    ZO_CUDA(cudaStreamSynchronize(c->stream), "stream synchronize");
    c->timing = value != 0;
    c->ev_used = 0;
    c->timing_ms = 0.0;
    c->timing_launches = 0;
    return ZO_OK;
  }
  return ZO_ERR_INVALID_ARG;
}

zo_status zo_get_timing(zo_ctx* c, double* total_ms, int64_t* launches) {
  if (!c || !total_ms || !launches) return ZO_ERR_INVALID_ARG;
  DeviceGuard guard(c->device);
  ZO_CUDA(cudaStreamSynchronize(c->stream), "stream synchronize");
  for (size_t k = 0; k < c->ev_used; ++k) {
    float ms = 0.f;
    ZO_CUDA(cudaEventElapsedTime(&ms, c->ev_start[k], c->ev_stop[k]), "cudaEventElapsedTime");
    c->timing_ms += ms;
    ++c->timing_launches;
  }
  c->ev_used = 0;
  *total_ms = c->timing_ms;
  *launches = c->timing_launches;
  return ZO_OK;
}

int32_t zo_wpass_path(const zo_ctx* c) { return c ? c->last_path : 0; }

int32_t zo_linear_tiling(const zo_ctx* c) { return c ? c->last_linear_tiling : 0; }

int64_t zo_kernel_launches(const zo_ctx* c) { return c ? c->launches : 0; }

zo_status zo_philox_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, uint32_t* out,
                         int64_t n_words, void* stream) {
  if (n_words < 0 || (n_words > 0 && !out) || (n_words + 3) / 4 > (int64_t(1) << 32)) {
    g_last_error = "zo_philox_fill: bad output or size";
    return ZO_ERR_INVALID_ARG;
  }
  ZO_CUDA(zo::launch_philox_fill(seed, x1, x2, x3, out, n_words,
                                 reinterpret_cast<cudaStream_t>(stream)),
          "philox fill kernel");
  return ZO_OK;
}

zo_status zo_normal_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, float* out,
                         int64_t n, void* stream) {
  if (n < 0 || (n > 0 && !out) || (n + 3) / 4 > (int64_t(1) << 32)) {
    g_last_error = "zo_normal_fill: bad output or size";
    return ZO_ERR_INVALID_ARG;
  }
  ZO_CUDA(zo::launch_normal_fill(seed, x1, x2, x3, out, n, reinterpret_cast<cudaStream_t>(stream)),
          "normal fill kernel");
  return ZO_OK;
}

}  // extern "C"
