// Per-pass r x r coefficient C_i and its projection P_i = C_i V_i^T.
//
// Every weight pass of the library has the form W_i <- rnd(W_i + U_i C_i V_i^T)
// (Alg. 2 / Eq. (4), with consecutive updates fused).  C_i is formed here, one
// CTA per matrix, from the Gaussian Z_i^(k) of the counter contract:
//   perturb: C_i = eps (ca Z_i^(qa) + cb Z_i^(qb))
//   step:    rho_k from the losses (Eq. (3) central / Eq. (6) forward),
//            G_i = (1/q) sum_k rho_k Z_i^(k)                       (Eq. (6), Alg. 3)
//            Adam: M <- b1 M + (1-b1) G, Vm <- b2 Vm + (1-b2) G.G  (Eqs. (7), (8))
//                  D = (M / (1-b1^t)) / (sqrt(Vm / (1-b2^t)) + eps_adam)  (Eqs. (9), (10))
//            SGD:  D = G                                              (Sec. 3)
//            C_i = -lr D + restore_coef eps Z_i^(restore_query)
// P_i = C_i V_i^T (r x n) then feeds the weight pass.  For the tensor-core path the kernel
// also writes max |C_i| (p.amax), from which the pass's operand scale is chosen.
#include "zo_kernels.h"

namespace zo {
namespace {

constexpr int kMaxQ = 4096;

__device__ __forceinline__ float4 f4_axpy(float a, float4 x, float4 y) {  // a*x + y
  return make_float4(fmaf(a, x.x, y.x), fmaf(a, x.y, y.y), fmaf(a, x.z, y.z), fmaf(a, x.w, y.w));
}
__device__ __forceinline__ float4 f4_scale(float a, float4 x) {
  return make_float4(a * x.x, a * x.y, a * x.z, a * x.w);
}

__global__ void __launch_bounds__(256) coeff_kernel(const MatDesc* __restrict__ mats,
                                                    CoeffParams p) {
  __shared__ float rho_s[kMaxQ];
  __shared__ float red_s[8];
  __shared__ float max_s[8];
  const MatDesc md = mats[blockIdx.x];
  const int r = p.r;
  const int rr = r * r;          // r is a multiple of 4, so rr is a multiple of 16
  const int n_ctr = rr / 4;
  const int tid = threadIdx.x;

  if (p.mode == kCoeffStep) {
    for (int k = tid; k < p.q; k += blockDim.x) {
      float rho;
      if (p.scheme == 0) {          // central: (L+_k - L-_k) / (2 eps)
        rho = (p.losses[2 * k] - p.losses[2 * k + 1]) / (2.0f * p.eps);
      } else if (p.scheme == 1) {   // forward: (l_(k+1) - l_0) / eps
        rho = (p.losses[k + 1] - p.losses[0]) / p.eps;
      } else {                      // rho given directly
        rho = p.losses[k];
      }
      rho_s[k] = rho;
    }
    __syncthreads();
  }

  float gsq = 0.0f;
  float cmax = 0.0f;
  float4* C4 = reinterpret_cast<float4*>(md.C);
  for (int c = tid; c < n_ctr; c += blockDim.x) {
    float4 out;
    if (p.mode == kCoeffPerturb) {
      float4 acc = f4_scale(p.ca, normal4(p.seed, (uint32_t)c, md.gidx, p.t,
                                          query_word(kTagZ, (uint32_t)p.qa)));
      if (p.qb >= 0)
        acc = f4_axpy(p.cb, normal4(p.seed, (uint32_t)c, md.gidx, p.t,
                                    query_word(kTagZ, (uint32_t)p.qb)), acc);
      out = f4_scale(p.eps, acc);
    } else {
      // G: accumulate in query order, then divide by q (Alg. 3)
      float4 g = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int k = 0; k < p.q; ++k)
        g = f4_axpy(rho_s[k], normal4(p.seed, (uint32_t)c, md.gidx, p.t,
                                      query_word(kTagZ, (uint32_t)k)), g);
      const float fq = (float)p.q;
      g = make_float4(g.x / fq, g.y / fq, g.z / fq, g.w / fq);
      gsq += g.x * g.x + g.y * g.y + g.z * g.z + g.w * g.w;
      float4 d;
      if (p.optimizer == 0) {
        float4* M4 = reinterpret_cast<float4*>(md.M);
        float4* V4 = reinterpret_cast<float4*>(md.Vm);
        float4 m = M4[c], v = V4[c];
        const float b1 = p.beta1, b2 = p.beta2;
        const float a1 = 1.0f - b1, a2 = 1.0f - b2;
        m = make_float4(b1 * m.x + a1 * g.x, b1 * m.y + a1 * g.y, b1 * m.z + a1 * g.z,
                        b1 * m.w + a1 * g.w);
        v = make_float4(b2 * v.x + a2 * (g.x * g.x), b2 * v.y + a2 * (g.y * g.y),
                        b2 * v.z + a2 * (g.z * g.z), b2 * v.w + a2 * (g.w * g.w));
        M4[c] = m;
        V4[c] = v;
        d.x = (m.x * p.inv_bc1) / (sqrtf(v.x * p.inv_bc2) + p.eps_adam);
        d.y = (m.y * p.inv_bc1) / (sqrtf(v.y * p.inv_bc2) + p.eps_adam);
        d.z = (m.z * p.inv_bc1) / (sqrtf(v.z * p.inv_bc2) + p.eps_adam);
        d.w = (m.w * p.inv_bc1) / (sqrtf(v.w * p.inv_bc2) + p.eps_adam);
      } else {
        d = g;
      }
      out = f4_scale(-p.lr, d);
      if (p.restore_query >= 0) {
        const float4 z = normal4(p.seed, (uint32_t)c, md.gidx, p.t,
                                 query_word(kTagZ, (uint32_t)p.restore_query));
        out = f4_axpy(p.restore_coef * p.eps, z, out);
      }
    }
    C4[c] = out;
    cmax = fmaxf(cmax, fmaxf(fmaxf(fabsf(out.x), fabsf(out.y)), fmaxf(fabsf(out.z), fabsf(out.w))));
  }

  if (p.amax != nullptr) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(0xffffffffu, cmax, o));
    if ((tid & 31) == 0) max_s[tid >> 5] = cmax;
    __syncthreads();
    if (tid == 0) {
      float m = 0.f;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = fmaxf(m, max_s[w]);
      p.amax[blockIdx.x] = m;
    }
  }

  if (p.mode == kCoeffStep && p.gamma_out != nullptr) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) gsq += __shfl_xor_sync(0xffffffffu, gsq, o);
    if ((tid & 31) == 0) red_s[tid >> 5] = gsq;
    __syncthreads();
    if (tid == 0) {
      float s = 0.f;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red_s[w];
      p.gamma_out[blockIdx.x] = sqrtf(s);
    }
  }
}

// P[a][j] = sum_b C[a][b] V[j][b]; one thread per column j, rows a split over ty.
template <int R>
__global__ void __launch_bounds__(256) project_fma_kernel(const MatDesc* __restrict__ mats,
                                                          const int2* __restrict__ units) {
  extern __shared__ float Cs[];   // R x R
  const int2 u = units[blockIdx.x];
  const MatDesc md = mats[u.x];
  const int tid = threadIdx.x;
  for (int e = tid; e < R * R; e += blockDim.x) Cs[e] = md.C[e];
  __syncthreads();
  const int64_t j = (int64_t)u.y + (tid & 127);
  if (j >= md.n) return;
  float v[R];
  const float4* vrow = reinterpret_cast<const float4*>(md.V + j * R);
#pragma unroll
  for (int b = 0; b < R / 4; ++b) {
    const float4 t = vrow[b];
    v[4 * b] = t.x; v[4 * b + 1] = t.y; v[4 * b + 2] = t.z; v[4 * b + 3] = t.w;
  }
  for (int a = tid >> 7; a < R; a += 2) {
    const float4* crow = reinterpret_cast<const float4*>(Cs + a * R);
    float acc = 0.f;
#pragma unroll
    for (int b4 = 0; b4 < R / 4; ++b4) {
      const float4 c4 = crow[b4];
      acc = fmaf(c4.x, v[4 * b4], acc);
      acc = fmaf(c4.y, v[4 * b4 + 1], acc);
      acc = fmaf(c4.z, v[4 * b4 + 2], acc);
      acc = fmaf(c4.w, v[4 * b4 + 3], acc);
    }
    md.P[(int64_t)a * md.n + j] = acc;
  }
}

template <int R>
cudaError_t launch_project_fma_r(const MatDesc* d_mats, const int2* d_units, int32_t n_units,
                                 cudaStream_t s) {
  const size_t smem = sizeof(float) * R * R;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(project_fma_kernel<R>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  project_fma_kernel<R><<<n_units, 256, smem, s>>>(d_mats, d_units);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_coeff(const MatDesc* d_mats, int32_t n_mats, const CoeffParams& p,
                         cudaStream_t s) {
  if (n_mats <= 0) return cudaSuccess;
  if (p.q > kMaxQ) return cudaErrorInvalidValue;
  coeff_kernel<<<n_mats, 256, 0, s>>>(d_mats, p);
  return cudaGetLastError();
}

cudaError_t launch_project_fma(const MatDesc* d_mats, const int2* d_units, int32_t n_units,
                               int32_t r, cudaStream_t s) {
  if (n_units <= 0) return cudaSuccess;
  switch (r) {
    case 4: return launch_project_fma_r<4>(d_mats, d_units, n_units, s);
    case 8: return launch_project_fma_r<8>(d_mats, d_units, n_units, s);
    case 16: return launch_project_fma_r<16>(d_mats, d_units, n_units, s);
    case 32: return launch_project_fma_r<32>(d_mats, d_units, n_units, s);
    case 64: return launch_project_fma_r<64>(d_mats, d_units, n_units, s);
    case 128: return launch_project_fma_r<128>(d_mats, d_units, n_units, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace zo
