/*
 * zo.h -- C ABI of the SubZero+ subspace zeroth-order weight path on GB300 (sm_103a).
 *
 * SubZero+ (arXiv 2608.15665) fine-tunes every trainable matrix W_i (m_i x n_i)
 * of a model with perturbations confined to a per-matrix subspace:
 *   W_i <- W_i + eps * U_i Z_i V_i^T                      (Sec. 4.1, Eq. (4); Alg. 2)
 * where U_i (m_i x r) and V_i (n_i x r) are Haar-distributed column-orthonormal
 * bases refreshed every F steps (Sec. 4.3, Eq. (11); Alg. 1) and Z_i is an r x r
 * Gaussian regenerated from a seed (App. A.1).  The q query losses give
 *   Zbar_i = (1/q) sum_k rho_k Z_i^(k)                    (Eq. (6); Alg. 3)
 * which drives an Adam optimizer on r x r moments       (Sec. 4.2, Eqs. (7)-(10))
 * whose update W_i <- W_i - eta U_i D_i V_i^T is applied in the same pass as the
 * restore of the last query.  The forward passes that produce the losses are the
 * caller's; the losses enter this ABI as fp32 arrays.
 *
 * Conventions for every entry point
 * ---------------------------------
 * - All tensors (W, U, V, M, Vm, losses, gamma) are CALLER-OWNED device memory
 *   unless an argument says "host".  The library allocates only its context:
 *   a device copy of the matrix table, per-call coefficient/projection buffers
 *   (O(sum_i r*(r + m_i + n_i)) floats) and the refresh workspace.  All are freed
 *   by zo_destroy.
 * - Every call is asynchronous on the stream given to zo_create (a cudaStream_t
 *   passed as void*; NULL = legacy default stream).  Arguments are validated on the
 *   host before anything is launched; a rejected call launches nothing and
 *   leaves all buffers untouched.
 * - A context belongs to the device that was current at zo_create; each call on it
 *   makes that device current for its duration and restores the caller's device.
 * - Kernels that detect a problem at run time (an mbarrier wait that ran out of
 *   iterations, an internal bound check) write a code to a device status word;
 *   zo_sync_status() synchronises the stream and returns and clears it.
 * - There is no CPU fallback: without a usable sm_103 device zo_create fails with
 *   ZO_ERR_CUDA.
 * - Layouts are row-major.  W_i has leading dimension ldw >= n (in elements);
 *   U_i is m x r and V_i is n x r, both contiguous fp32; M_i and Vm_i are r x r
 *   contiguous fp32.
 * - Random numbers follow one counter-based contract shared by nothing but its
 *   definition: Philox4x32-10 (Salmon et al., SC'11), key = (seed lo, seed hi),
 *   counter = (e / 4, matrix index, t or refresh index j, tag << 24 | query k),
 *   lane e % 4 for element e of a row-major buffer; u = ((x >> 8) + 1) * 2^-24;
 *   Box-Muller on lane pairs (0,1), (2,3): z_a = sqrt(-2 ln u_a) cos(2 pi u_b),
 *   z_b = sqrt(-2 ln u_a) sin(2 pi u_b).  Tags: 1 = Z, 2 = Omega_U, 3 = Omega_V.
 */
#ifndef SUBZERO_GB300_ZO_H
#define SUBZERO_GB300_ZO_H

#include <stdint.h>

#if defined(__GNUC__)
#define ZO_API __attribute__((visibility("default")))
#else
#define ZO_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum zo_status {
  ZO_OK = 0,
  ZO_ERR_INVALID_ARG = 1,   /* null pointer, bad enum, negative size, bad scalar */
  ZO_ERR_SHAPE = 2,         /* r > min(m, n), r unsupported, ldw < n, sizes too large */
  ZO_ERR_ALIGN = 3,         /* a buffer is not 16-byte aligned */
  ZO_ERR_DTYPE = 4,         /* unknown weight dtype */
  ZO_ERR_CUDA = 5,          /* a CUDA runtime call failed (message: zo_last_error) */
  ZO_ERR_TIMEOUT = 6,       /* a bounded device-side wait ran out (zo_sync_status) */
  ZO_ERR_UNSUPPORTED = 7,   /* valid request the library does not implement */
  ZO_ERR_NOMEM = 8          /* workspace allocation failed */
} zo_status;

/* Weight storage dtypes. */
enum { ZO_F32 = 0, ZO_BF16 = 1 };

/* How zo_step turns the losses into rho_k. */
enum {
  ZO_SCHEME_CENTRAL = 0,  /* losses = [L+_0, L-_0, ..., L+_(q-1), L-_(q-1)]: rho_k = (L+_k - L-_k)/(2 eps), Eq. (3) */
  ZO_SCHEME_FORWARD = 1,  /* losses = [l_0, l_1, ..., l_q]: rho_k = (l_(k+1) - l_0)/eps, Eq. (6), Alg. 3 */
  ZO_SCHEME_DIRECT = 2    /* losses = [rho_0, ..., rho_(q-1)] given directly */
};

/* Optimizer applied in the subspace by zo_step. */
enum {
  ZO_OPT_ADAM = 0,        /* subspace Adam, Eqs. (7)-(10) */
  ZO_OPT_SGD = 1          /* SubZero's subspace SGD (Sec. 3): D = Zbar, moments untouched */
};

/* Options for zo_set_option. */
enum {
  ZO_OPTION_WPASS_PATH = 0, /* 0 = automatic: tcgen05 when every W is bf16 with n a
                                   multiple of 8 (its TMA stores write 16-byte chunks) and
                                   r >= 16 -- if such a set's tensor-core descriptors
                                   cannot be built (cuTensorMapEncodeTiled rejects one, e.g.
                                   a W row stride of 2^40 bytes or more), zo_perturb and
                                   zo_step return ZO_ERR_UNSUPPORTED instead of running
                                   another pass, and value 1 selects the FMA pass;
                                   else, at r in {4, 8}, the narrow-tile FMA pass when its
                                   tiles number at most half of the 32-row tiles (sets of
                                   thin matrices such as LoRA factors); else the FMA pass,
                               1 = FMA path on 32-row tiles, 2 = tcgen05 path,
                               3 = FMA path on narrow tiles (r in {4, 8}).  All FMA
                               tilings give bit-identical weights. */
  ZO_OPTION_TIMING = 1,     /* 1 = record CUDA events around every weight-pass launch */
  ZO_OPTION_TEST_WAIT_TIMEOUT = 2, /* test hook: 1 = in the next tensor-core weight pass, one
                                     CTA first waits on a barrier nothing arrives on, so its
                                     bounded wait (~0.1 s) runs out; that pass then reports
                                     ZO_ERR_TIMEOUT via zo_sync_status and leaves W partly
                                     updated.  If an SM-pair zo_linear_perturbed call comes
                                     first, it takes the hook instead: its Y tiles wait for
                                     S rows that are never counted as written, give up after
                                     ~0.1 s and leave Y partly written.  Nothing faults; the
                                     context stays usable. */
  ZO_OPTION_LINEAR_TILE = 3, /* tiles (rows of X x columns of Y) of zo_linear_perturbed's
                               Y = X W^T + S U^T GEMM: 0 = automatic (the SM-pair tiling
                               whose busiest pair has the least operand traffic; the
                               single-CTA ones if no 2-CTA cluster fits), 1 = 128 x 256,
                               2 = 256 x 256, 3 = 256 x 224 on single CTAs (S = X P^T by a
                               separate split-K kernel), 4 .. 8 = 256 x 256, 240, 224, 192,
                               128 on SM pairs (M = 256 MMAs across a 2-CTA cluster, S in
                               the same launch).  The tilings of one family give
                               bit-identical Y; the two families may differ in the last
                               bits of S (each splits S's K in ranges of its own).  At
                               r in {64, 128} only the SM-pair tilings exist: a call with
                               1 .. 3 set returns ZO_ERR_UNSUPPORTED. */
  ZO_OPTION_PAIR_MMA = 4    /* tensor-core weight pass at r = 128: 1 (default) = M = 256 MMAs
                               across the two SMs of a cluster (each SM holds and reads half
                               of every P tile), 0 = the single-SM kernel.  Both give
                               bit-identical weights. */
};

/* One trainable matrix W_i with its projection bases and Adam moments. */
typedef struct zo_matrix {
  void* W;        /* device; m x n, row-major, leading dimension ldw elements, dtype below */
  int64_t m;      /* rows (nn.Linear out_features) */
  int64_t n;      /* columns (nn.Linear in_features) */
  int64_t ldw;    /* leading dimension of W in elements, >= n */
  int32_t dtype;  /* ZO_F32 or ZO_BF16 */
  int32_t reserved;
  float* U;       /* device; m x r fp32, written by zo_refresh / zo_init_subspace */
  float* V;       /* device; n x r fp32, written by zo_refresh / zo_init_subspace */
  float* M;       /* device; r x r fp32 first moment (Eq. (7)) */
  float* Vm;      /* device; r x r fp32 second moment (Eq. (8)); named Vm to keep V for the basis */
} zo_matrix;

typedef struct zo_ctx zo_ctx;

/*
 * zo_create -- bind the caller's matrices into a context (Alg. 3 "Require" line).
 *   mats[n_mats]: copied; the pointers inside must stay valid until zo_destroy.
 *   r: subspace rank, 1 <= r <= min(m_i, n_i); the library supports r in {4, 8, 16, 32, 64, 128}.
 *   q: queries per step (K in the paper), 1 <= q <= 4096.
 *   seed: 64-bit base seed of the Philox key.
 *   matrix_index_base: matrix i of this table uses Philox matrix index base + i
 *     (lets several contexts or ranks share one global numbering).
 *   stream: cudaStream_t (void*) every later call launches on.
 * Validates every matrix (non-null, 16-byte aligned, shapes, dtype), allocates
 * the workspace and uploads the table.  On failure *out is NULL.
 */
ZO_API zo_status zo_create(zo_ctx** out, const zo_matrix* mats, int32_t n_mats, int32_t r, int32_t q,
                    uint64_t seed, uint32_t matrix_index_base, void* stream);

/* zo_destroy -- synchronise the stream, free the context and its workspace.  NULL is a no-op. */
ZO_API zo_status zo_destroy(zo_ctx* ctx);

/*
 * zo_refresh -- Alg. 1 (Haar-distributed bases) for every matrix at refresh index j
 * (Alg. 3 calls it when t mod F == 0; j = t / F).  Draws Omega_U (m x r, tag 2)
 * and Omega_V (n x r, tag 3) from the counter contract and writes into U_i and V_i
 * the Q of their thin QR factorisation with diag(R) > 0, i.e. Q with column c
 * multiplied by sgn(R_cc) (Eq. (11), sgn(0) = +1).  That factor is unique; panels
 * with at least 4r rows at r >= 16 reach it by CholeskyQR2 (two rounds of Cholesky
 * of the Gram matrix and a triangular solve), the others by a batched Householder
 * TSQR with the sign fix.  A Gram matrix without a positive pivot (not expected for
 * such panels) makes the next zo_sync_status return ZO_ERR_CUDA.  reset_moments != 0
 * also zeroes M_i and Vm_i.
 */
ZO_API zo_status zo_refresh(zo_ctx* ctx, uint32_t refresh_idx, int32_t reset_moments);

/* zo_init_subspace -- the first lines of Alg. 3: M_i = Vm_i = 0 and U_i, V_i from
 * Alg. 1 at refresh index refresh_idx (normally 0). */
ZO_API zo_status zo_init_subspace(zo_ctx* ctx, uint32_t refresh_idx);

/*
 * zo_perturb -- one fused weight pass of Alg. 2 (the in-place perturbation) over all matrices:
 *   W_i <- rnd(W_i + eps * U_i (ca Z_i^(qa) + cb Z_i^(qb)) V_i^T)
 * with Z_i^(k) the step-t Gaussian of query k (tag 1).  qb = -1 drops the second
 * term.  Two terms fuse the restore of one query with the perturbation of the
 * next (e.g. ca = +1, cb = -1 gives W += eps U (Z_(k+1) - Z_k) V^T); the sum is
 * formed in fp32 and W is rounded once (RNE) to its dtype.
 * 0 <= qa, qb < q.
 * The update U C V^T is evaluated to fp32 grade on either path: the FMA pass in fp32;
 * the tensor-core pass with U, P = C V^T (and, in the projection, V and C) held as
 * power-of-two-scaled fp16 pairs hi + lo (~22 significant bits) and three products
 * accumulated in fp32, which errs by ~2^-21 of sum |U| |C| |V|^T.
 */
ZO_API zo_status zo_perturb(zo_ctx* ctx, uint32_t t, int32_t qa, float ca, int32_t qb, float cb,
                     float eps);

/*
 * zo_step -- the update of Alg. 3 for all matrices, fused with the final restore:
 *   rho_k from the losses per `scheme` (Eq. (3) or Eq. (6)),
 *   G_i = (1/q) sum_k rho_k Z_i^(k)                       (Eq. (6), Alg. 3)
 *   ZO_OPT_ADAM: M_i, Vm_i updated in place (Eqs. (7)-(8)); with
 *     bias corrections 1 - beta^adam_t (Eq. (9), adam_t >= 1 counts Adam updates
 *     since the moments were zeroed), D_i = Mhat / (sqrt(Vhat) + eps_adam);
 *   ZO_OPT_SGD: D_i = G_i (moments untouched; adam_t, betas ignored);
 *   W_i <- rnd(W_i + U_i (-lr D_i + restore_coef * eps * Z_i^(restore_query)) V_i^T)
 *     (Eq. (10) plus the restore; restore_query = -1 drops the restore term).
 * losses: n_losses fp32 values (2q central, q+1 forward, q direct); device memory
 *   unless losses_on_host != 0, in which case they are copied from host memory on the
 *   context's stream before the launch.  A pageable host buffer may be reused as soon
 *   as the call returns (the runtime stages it before returning); a page-locked one is
 *   read only when the stream reaches the copy, so it must stay unchanged until then.
 * gamma_out: NULL or device array of n_mats floats receiving ||G_i||_F (Sec. 4.1).
 */
ZO_API zo_status zo_step(zo_ctx* ctx, uint32_t t, int32_t adam_t, const float* losses, int32_t n_losses,
                  int32_t losses_on_host, int32_t scheme, int32_t optimizer, float eps, float lr,
                  float beta1, float beta2, float eps_adam, int32_t restore_query,
                  float restore_coef, float* gamma_out);

/*
 * zo_mezo_perturb -- the full-space SPSA perturbation of Sec. 3, Eq. (1) (MeZO, the
 * paper's comparison baseline), for every matrix of the context:
 *   W_i <- rnd(W_i + coef * Z_i),  Z_i[row, col] ~ N(0, 1) i.i.d., regenerated from the seed
 * with counter = (row * ceil(n_i / 4) + col / 4, matrix index, t, 5 << 24), lane col % 4
 * (each row starts on a fresh counter word).  coef = +eps, -2 eps, +eps give the two
 * evaluations of Eq. (1) and the restore; coef = eps - lr * rho fuses the restore with
 * MeZO's SGD update (rho = (L+ - L-) / (2 eps)).  U, V and the moments are not touched.
 * Each weight costs one quarter of a Philox call plus half a Box-Muller transform, so
 * this pass is bound by the ALU rather than HBM.  Timed like the weight passes when
 * ZO_OPTION_TIMING is on.
 */
ZO_API zo_status zo_mezo_perturb(zo_ctx* ctx, uint32_t t, float coef);

/*
 * Linear layers at the perturbed weights WITHOUT a weight pass: the forward of a loss
 * evaluation of Alg. 3 at W_i' = W_i + U_i C_i V_i^T (Eq. (4) form) with every W_i left as
 * it is, for contexts on the tensor-core path (every W bf16, n a multiple of 8) with r in
 * {16, 32, 64, 128}; otherwise ZO_ERR_UNSUPPORTED.
 *
 * zo_linear_prepare -- once per loss evaluation: C_i = eps (ca Z_i^(qa) + cb Z_i^(qb)) at
 *   step t (qb = -1: one term) for every matrix -- the coefficient zo_perturb(ctx, t, qa,
 *   ca, qb, cb, eps) would add to W_i -- and P_i = C_i V_i^T, kept for the calls below
 *   until the next zo_linear_prepare; zo_refresh (new U, V) discards it, and
 *   zo_linear_perturbed then returns ZO_ERR_INVALID_ARG until the next prepare.
 * zo_linear_perturbed -- one layer: Y = X (W_i + U_i C_i V_i^T)^T = X W_i^T +
 *   (X V_i C_i^T) U_i^T.  X: T x n_i bf16, row stride ldx elements; Y: T x m_i bf16, row
 *   stride ldy (device, caller-owned, 16-byte aligned, strides multiples of 8; m_i a
 *   multiple of 8, else ZO_ERR_SHAPE).  The dense product is exact in bf16 with fp32
 *   accumulation; the rank-r term carries the bf16 hi/lo split's ~2^-16 relative error;
 *   Y is rounded to bf16 once.  W_i is read, never written.  Asynchronous; device errors
 *   go to the status word.  The GEMM's tiling follows ZO_OPTION_LINEAR_TILE (the tilings
 *   of one family give the same Y bits); the context keeps an S workspace sized for the most tokens
 *   seen so far, and a call with more synchronises the stream to grow it.
 */
ZO_API zo_status zo_linear_prepare(zo_ctx* ctx, uint32_t t, int32_t qa, float ca, int32_t qb,
                                   float cb, float eps);
ZO_API zo_status zo_linear_perturbed(zo_ctx* ctx, int32_t i, const void* X, int64_t T,
                                     int64_t ldx, void* Y, int64_t ldy);

/* zo_sync_status -- synchronise the stream; return (and clear) the device status word. */
ZO_API zo_status zo_sync_status(zo_ctx* ctx);

/* zo_set_option -- see ZO_OPTION_*; returns ZO_ERR_INVALID_ARG for unknown options/values. */
ZO_API zo_status zo_set_option(zo_ctx* ctx, int32_t option, int64_t value);

/*
 * zo_get_timing -- with ZO_OPTION_TIMING on, the summed device time (ms) and count of
 * weight-pass kernel launches since the option was last set.  Synchronises the stream.
 * The context holds a pair of CUDA events per timed launch until this call folds them
 * into the totals (and reuses them), so long timed runs should call it now and then.
 */
ZO_API zo_status zo_get_timing(zo_ctx* ctx, double* total_ms, int64_t* launches);

/* zo_wpass_path -- the weight-pass path the last zo_perturb / zo_step launched
   (1 = FMA on 32-row tiles, 2 = tcgen05, 3 = FMA on narrow tiles). */
ZO_API int32_t zo_wpass_path(const zo_ctx* ctx);

/* zo_linear_tiling -- the tiling (1 .. 8, as ZO_OPTION_LINEAR_TILE) of the Y GEMM that
 * the last zo_linear_perturbed launched; 0 before the first call or for a null ctx. */
ZO_API int32_t zo_linear_tiling(const zo_ctx* ctx);

/* zo_kernel_launches -- number of kernels this context has launched since zo_create. */
ZO_API int64_t zo_kernel_launches(const zo_ctx* ctx);

/*
 * zo_philox_fill -- the raw integer stream of the counter contract:
 *   out[4c + l] = Philox4x32-10(counter = (c, x1, x2, x3), key = seed)[l], 0 <= 4c + l < n_words.
 * out: device uint32 array.  Asynchronous on `stream` (void* cudaStream_t).
 */
ZO_API zo_status zo_philox_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, uint32_t* out,
                         int64_t n_words, void* stream);

/*
 * zo_normal_fill -- the Gaussian stream of the contract (uniform + Box-Muller on
 * lane pairs), elements 0..n-1, fp32, into device memory.  This is exactly how
 * Z_i^(k) (x1 = i, x2 = t, x3 = 1 << 24 | k) and Omega (x2 = j, x3 = tag << 24)
 * are drawn inside the other calls.
 */
ZO_API zo_status zo_normal_fill(uint64_t seed, uint32_t x1, uint32_t x2, uint32_t x3, float* out,
                         int64_t n, void* stream);

/*
 * zo_perturb_noalloc -- one perturbation pass on a single matrix that allocates no
 * device memory.  The paper has no counterpart; it is for callers that cannot
 * allocate: code whose GPU memory is already reserved by another allocator (a
 * framework's caching pool), where a cudaMalloc would fail or fragment that pool,
 * and loops that cannot afford the device synchronisation cudaMalloc/cudaFree may
 * cause.  It computes what zo_perturb computes for one matrix on the fp32-FMA path:
 *   W <- rnd(W + eps * U (ca Z^(qa) + cb Z^(qb)) V^T)   (qb = -1 drops the second term)
 * with Z^(k) drawn for matrix index `matrix_index` at step t from `seed`
 * (the counter contract above).  W (m x n, ldw, dtype), U (m x r) and V (n x r) are
 * caller-owned device buffers; r in {4, 8, 16, 32, 64}.
 * Scratch (the coefficient C, the projection C V^T and small work tables) lives in a
 * fixed 8 MiB array inside the library (2^21 floats), which every GPU that loads the
 * library holds until the process exits.  A request needing more -- about r * n + r * r
 * floats -- is rejected with ZO_ERR_SHAPE before anything is launched.
 * The first call on a device looks up that array's device address (cudaGetSymbolAddress)
 * with the device current; make that first call before capturing any stream.
 * A call copies nothing from the host: it launches four kernels on `stream` (the first
 * writes the call's small tables into the array from its launch parameters).
 * All calls share the one array and rewrite everything they read from it before
 * reading it, so nothing needs clearing between calls -- but two calls whose work
 * overlaps on the GPU (different streams, or different host threads) race on it.
 * U must hold m x r and V n x r contiguous fp32 values: the C ABI cannot check the sizes
 * of the buffers behind the pointers.
 * Asynchronous on `stream` (void* cudaStream_t); errors as for zo_perturb.
 */
ZO_API zo_status zo_perturb_noalloc(void* W, int64_t m, int64_t n, int64_t ldw, int32_t dtype,
                                    const float* U, const float* V, int32_t r, uint64_t seed,
                                    uint32_t matrix_index, uint32_t t, int32_t qa, float ca,
                                    int32_t qb, float cb, float eps, void* stream);

/* zo_status_string -- static description of a status code. */
ZO_API const char* zo_status_string(int32_t status);

/* zo_last_error -- last CUDA error text seen by this thread (static storage). */
ZO_API const char* zo_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SUBZERO_GB300_ZO_H */
