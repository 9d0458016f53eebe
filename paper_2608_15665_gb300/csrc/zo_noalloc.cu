// zo_perturb_noalloc: one perturbation pass on one matrix without any device
// allocation.  The paper has no counterpart; this entry point exists for callers
// that cannot call cudaMalloc themselves or let a library do it: code whose device
// memory is owned by another allocator (a framework's caching pool that has
// reserved the GPU's memory, where a stray cudaMalloc fails or fragments it), or
// latency-critical loops where cudaMalloc / cudaFree would synchronise the device.
//
// It runs the same kernels as the FMA path of zo_perturb (coefficient C, projection
// P = C V^T, weight pass) on one matrix, with every piece of scratch -- the one-entry
// matrix table, the tile prefix, the projection work list, C and P -- placed in the
// file-scope array below.  That array is a fixed 8 MiB that every GPU which loads
// this library keeps until the process exits.  The tables are written by a small kernel
// that takes them as launch parameters, so a call makes no host-to-device copy: it is
// four kernel launches on the caller's stream and nothing else.
#include <algorithm>
#include <cmath>
#include <mutex>
#include <string>

#include "../../include/zo.h"
#include "zo_kernels.h"

namespace {

// 2^21 floats = 8 MiB, 256-byte aligned; holds the table, C (r*r) and P (r*n).
constexpr int64_t kScratchFloats = int64_t(1) << 21;
static __device__ __align__(256) float g_noalloc_scratch[kScratchFloats];

// Device addresses of the array, one per device, resolved on first use.
constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
float* g_scratch_ptr[kMaxDevices] = {nullptr};

// Offsets (in floats) of the pieces inside the scratch array for a matrix with
// n columns and rank r; returns the total.
struct Layout {
  int64_t desc, prefix, units, C, P, total;
};
Layout layout_for(int64_t n, int32_t r) {
  auto up64 = [](int64_t x) { return (x + 63) / 64 * 64; };   // 256-byte granules
  Layout L{};
  L.desc = 0;
  L.prefix = up64((int64_t)(sizeof(zo::MatDesc) + 3) / 4);
  L.units = L.prefix + 64;                                     // two int64
  const int64_t n_units = (n + 127) / 128;
  L.C = L.units + up64(2 * n_units);                           // int2 per unit
  L.P = L.C + up64((int64_t)r * r);
  L.total = L.P + (int64_t)r * n;
  return L;
}

zo_status fail(zo_status st, const std::string& msg) {
  zo::set_last_error(msg);
  return st;
}

// Writes the one-entry matrix table, the tile prefix (0, tiles) and the projection work
// list (matrix 0, first column 128 u) for u < n_units into the scratch array.
__global__ void __launch_bounds__(256)
noalloc_tables_kernel(zo::MatDesc d, int64_t tiles, int32_t n_units, zo::MatDesc* __restrict__ desc,
                      int64_t* __restrict__ prefix, int2* __restrict__ units) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (tid == 0) {
    *desc = d;
    prefix[0] = 0;
    prefix[1] = tiles;
  }
  for (int64_t u = tid; u < n_units; u += (int64_t)gridDim.x * blockDim.x)
    units[u] = make_int2(0, (int)(u * 128));
}

}  // namespace

extern "C" ZO_API zo_status zo_perturb_noalloc(void* W, int64_t m, int64_t n, int64_t ldw,
                                              int32_t dtype, const float* U, const float* V,
                                              int32_t r, uint64_t seed, uint32_t matrix_index,
                                              uint32_t t, int32_t qa, float ca, int32_t qb,
                                              float cb, float eps, void* stream) {
  if (!W || !U || !V) return fail(ZO_ERR_INVALID_ARG, "null W, U or V");
  if (dtype != ZO_F32 && dtype != ZO_BF16) return fail(ZO_ERR_DTYPE, "unknown dtype");
  if (!(r == 4 || r == 8 || r == 16 || r == 32 || r == 64))
    return fail(ZO_ERR_SHAPE, "rank r must be one of 4, 8, 16, 32, 64");
  if (m < r || n < r || ldw < n) return fail(ZO_ERR_SHAPE, "need r <= min(m, n) and ldw >= n");
  if (qa < 0 || qa > 0xFFFFFF || qb < -1 || qb > 0xFFFFFF)
    return fail(ZO_ERR_INVALID_ARG, "query index out of range");
  if (!std::isfinite(ca) || !std::isfinite(cb) || !std::isfinite(eps))
    return fail(ZO_ERR_INVALID_ARG, "non-finite scalar");
  const int64_t esize = dtype == ZO_BF16 ? 2 : 4;
  if ((reinterpret_cast<uintptr_t>(W) & 15u) || (ldw * esize) % 16 ||
      (reinterpret_cast<uintptr_t>(U) & 15u) || (reinterpret_cast<uintptr_t>(V) & 15u))
    return fail(ZO_ERR_ALIGN, "W, U, V must be 16-byte aligned and ldw*sizeof(dtype) a multiple of 16");
  const Layout L = layout_for(n, r);
  if (L.total > kScratchFloats)
    return fail(ZO_ERR_SHAPE, "zo_perturb_noalloc needs " + std::to_string(L.total) +
                                  " floats of scratch (r*n + r*r + tables); its static scratch holds " +
                                  std::to_string(kScratchFloats) + " floats (8 MiB)");
  const int64_t tiles = ((m + zo::kFmaTileRows - 1) / zo::kFmaTileRows) *
                        ((n + zo::fma_tile_cols(dtype) - 1) / zo::fma_tile_cols(dtype));
  if (tiles > 0x7FFFFFFF) return fail(ZO_ERR_SHAPE, "too many weight-pass tiles");

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(ZO_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return fail(ZO_ERR_CUDA, "device ordinal out of range");
  float* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_ptr[dev]) {
      cudaDeviceProp prop;
      e = cudaGetDeviceProperties(&prop, dev);
      if (e != cudaSuccess)
        return fail(ZO_ERR_CUDA, std::string("cudaGetDeviceProperties: ") + cudaGetErrorString(e));
      if (!(prop.major == 10 && prop.minor == 3))
        return fail(ZO_ERR_CUDA, "this library is built for sm_103a (GB300) only");
      // the array's name in host code is only a handle; its device address comes from here
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (e != cudaSuccess)
        return fail(ZO_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      g_scratch_ptr[dev] = static_cast<float*>(p);
    }
    scratch = g_scratch_ptr[dev];
  }

  // one-entry table, tile prefix and projection work list, written into the scratch by
  // the first of the call's kernels
  zo::MatDesc d{};
  d.W = W;
  d.m = m;
  d.n = n;
  d.ldw = ldw;
  d.dtype = dtype;
  d.gidx = matrix_index;
  d.U = const_cast<float*>(U);
  d.V = const_cast<float*>(V);
  d.C = scratch + L.C;
  d.P = scratch + L.P;
  d.tile0 = 0;
  const int64_t n_units = (n + 127) / 128;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  zo::MatDesc* d_desc = reinterpret_cast<zo::MatDesc*>(scratch + L.desc);
  int64_t* d_prefix = reinterpret_cast<int64_t*>(scratch + L.prefix);
  int2* d_units = reinterpret_cast<int2*>(scratch + L.units);
  const int table_blocks = (int)std::min<int64_t>((n_units + 255) / 256, 64);
  noalloc_tables_kernel<<<table_blocks, 256, 0, s>>>(d, tiles, (int32_t)n_units, d_desc, d_prefix,
                                                      d_units);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(ZO_ERR_CUDA, std::string("table kernel: ") + cudaGetErrorString(e));

  zo::CoeffParams p{};
  p.mode = zo::kCoeffPerturb;
  p.seed = seed;
  p.t = t;
  p.r = r;
  p.q = 1;
  p.qa = qa;
  p.qb = qb;
  p.ca = ca;
  p.cb = cb;
  p.eps = eps;
  e = zo::launch_coeff(d_desc, 1, p, s);
  if (e == cudaSuccess) e = zo::launch_project_fma(d_desc, d_units, (int32_t)n_units, r, s);
  if (e == cudaSuccess) e = zo::launch_wpass_fma(d_desc, 1, d_prefix, tiles, r, s);
  if (e != cudaSuccess) return fail(ZO_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
  return ZO_OK;
}
