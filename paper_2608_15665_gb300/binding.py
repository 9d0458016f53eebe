"""ctypes binding of the C ABI in include/zo.h (argument marshalling only).

Every function here has the name of the C entry point it calls and does nothing
but convert arguments (torch tensors -> device pointers, Python scalars -> C
types) and turn a non-zero status into ``ZoError``.  All computation runs in
the CUDA library ``libsubzero_zo.so``; if that library is missing, importing
this module fails -- there is no fallback.
"""

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libsubzero_zo.so")

ZO_OK = 0
ZO_ERR_INVALID_ARG = 1
ZO_ERR_SHAPE = 2
ZO_ERR_ALIGN = 3
ZO_ERR_DTYPE = 4
ZO_ERR_CUDA = 5
ZO_ERR_TIMEOUT = 6
ZO_ERR_UNSUPPORTED = 7
ZO_ERR_NOMEM = 8

ZO_F32 = 0
ZO_BF16 = 1

ZO_SCHEME_CENTRAL = 0
ZO_SCHEME_FORWARD = 1
ZO_SCHEME_DIRECT = 2

ZO_OPT_ADAM = 0
ZO_OPT_SGD = 1

ZO_OPTION_WPASS_PATH = 0
ZO_OPTION_TIMING = 1
ZO_OPTION_TEST_WAIT_TIMEOUT = 2
ZO_OPTION_LINEAR_TILE = 3
ZO_OPTION_PAIR_MMA = 4


class ZoError(RuntimeError):
    def __init__(self, status, where, detail=""):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status}) {detail}".rstrip())


class zo_matrix(ctypes.Structure):
    _fields_ = [
        ("W", ctypes.c_void_p),
        ("m", ctypes.c_int64),
        ("n", ctypes.c_int64),
        ("ldw", ctypes.c_int64),
        ("dtype", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
        ("U", ctypes.c_void_p),
        ("V", ctypes.c_void_p),
        ("M", ctypes.c_void_p),
        ("Vm", ctypes.c_void_p),
    ]


_c = ctypes
_SIGNATURES = {
    "zo_create": (_c.c_int32, [_c.POINTER(_c.c_void_p), _c.POINTER(zo_matrix), _c.c_int32,
                               _c.c_int32, _c.c_int32, _c.c_uint64, _c.c_uint32, _c.c_void_p]),
    "zo_destroy": (_c.c_int32, [_c.c_void_p]),
    "zo_refresh": (_c.c_int32, [_c.c_void_p, _c.c_uint32, _c.c_int32]),
    "zo_init_subspace": (_c.c_int32, [_c.c_void_p, _c.c_uint32]),
    "zo_perturb": (_c.c_int32, [_c.c_void_p, _c.c_uint32, _c.c_int32, _c.c_float, _c.c_int32,
                                _c.c_float, _c.c_float]),
    "zo_step": (_c.c_int32, [_c.c_void_p, _c.c_uint32, _c.c_int32, _c.c_void_p, _c.c_int32,
                             _c.c_int32, _c.c_int32, _c.c_int32, _c.c_float, _c.c_float,
                             _c.c_float, _c.c_float, _c.c_float, _c.c_int32, _c.c_float,
                             _c.c_void_p]),
    "zo_mezo_perturb": (_c.c_int32, [_c.c_void_p, _c.c_uint32, _c.c_float]),
    "zo_linear_prepare": (_c.c_int32, [_c.c_void_p, _c.c_uint32, _c.c_int32, _c.c_float,
                                       _c.c_int32, _c.c_float, _c.c_float]),
    "zo_linear_perturbed": (_c.c_int32, [_c.c_void_p, _c.c_int32, _c.c_void_p, _c.c_int64,
                                         _c.c_int64, _c.c_void_p, _c.c_int64]),
    "zo_sync_status": (_c.c_int32, [_c.c_void_p]),
    "zo_set_option": (_c.c_int32, [_c.c_void_p, _c.c_int32, _c.c_int64]),
    "zo_get_timing": (_c.c_int32, [_c.c_void_p, _c.POINTER(_c.c_double), _c.POINTER(_c.c_int64)]),
    "zo_wpass_path": (_c.c_int32, [_c.c_void_p]),
    "zo_linear_tiling": (_c.c_int32, [_c.c_void_p]),
    "zo_kernel_launches": (_c.c_int64, [_c.c_void_p]),
    "zo_philox_fill": (_c.c_int32, [_c.c_uint64, _c.c_uint32, _c.c_uint32, _c.c_uint32,
                                    _c.c_void_p, _c.c_int64, _c.c_void_p]),
    "zo_normal_fill": (_c.c_int32, [_c.c_uint64, _c.c_uint32, _c.c_uint32, _c.c_uint32,
                                    _c.c_void_p, _c.c_int64, _c.c_void_p]),
    "zo_perturb_noalloc": (_c.c_int32, [_c.c_void_p, _c.c_int64, _c.c_int64, _c.c_int64,
                                        _c.c_int32, _c.c_void_p, _c.c_void_p, _c.c_int32,
                                        _c.c_uint64, _c.c_uint32, _c.c_uint32, _c.c_int32,
                                        _c.c_float, _c.c_int32, _c.c_float, _c.c_float,
                                        _c.c_void_p]),
    "zo_status_string": (_c.c_char_p, [_c.c_int32]),
    "zo_last_error": (_c.c_char_p, []),
}


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is missing: build it with paper_2608_15665_gb300.build.build() "
            "(nvcc, sm_103a). There is no CPU fallback.")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


LIB = _load()


def status_string(status):
    return LIB.zo_status_string(int(status)).decode()


def zo_last_error():
    return LIB.zo_last_error().decode()


def _check(status, where):
    if status != ZO_OK:
        raise ZoError(status, where, zo_last_error())


def _ptr(t):
    """Device pointer of a tensor (or an int address, or None -> NULL)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream_handle(stream):
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_matrix(W, U, V, M, Vm):
    """zo_matrix for torch tensors: W (m x n, bf16/fp32, row stride ldw), U (m x r),
    V (n x r), M and Vm (r x r), all fp32 except W."""
    import torch
    if W.dtype == torch.bfloat16:
        dt = ZO_BF16
    elif W.dtype == torch.float32:
        dt = ZO_F32
    else:
        raise ZoError(ZO_ERR_DTYPE, "make_matrix", str(W.dtype))
    if W.dim() != 2 or W.stride(1) != 1:
        raise ZoError(ZO_ERR_SHAPE, "make_matrix", "W must be 2-D with unit column stride")
    for name, t in (("U", U), ("V", V), ("M", M), ("Vm", Vm)):
        if t.dtype != torch.float32 or not t.is_contiguous():
            raise ZoError(ZO_ERR_DTYPE, "make_matrix", f"{name} must be contiguous fp32")
    return zo_matrix(_ptr(W), W.shape[0], W.shape[1], W.stride(0), dt, 0, _ptr(U), _ptr(V),
                     _ptr(M), _ptr(Vm))


def zo_create(mats, r, q, seed, matrix_index_base=0, stream=None):
    arr = (zo_matrix * len(mats))(*mats)
    ctx = ctypes.c_void_p()
    _check(LIB.zo_create(ctypes.byref(ctx), arr, len(mats), int(r), int(q), int(seed) & (2**64 - 1),
                         int(matrix_index_base), _stream_handle(stream)), "zo_create")
    return ctx


def zo_destroy(ctx):
    _check(LIB.zo_destroy(ctx), "zo_destroy")


def zo_refresh(ctx, refresh_idx, reset_moments=False):
    _check(LIB.zo_refresh(ctx, int(refresh_idx), int(bool(reset_moments))), "zo_refresh")


def zo_init_subspace(ctx, refresh_idx=0):
    _check(LIB.zo_init_subspace(ctx, int(refresh_idx)), "zo_init_subspace")


def zo_perturb(ctx, t, qa, ca, qb, cb, eps):
    _check(LIB.zo_perturb(ctx, int(t), int(qa), float(ca), int(qb), float(cb), float(eps)),
           "zo_perturb")


def zo_step(ctx, t, adam_t, losses, scheme, eps, lr, beta1, beta2, eps_adam, restore_query,
            restore_coef, optimizer=ZO_OPT_ADAM, gamma_out=None):
    """losses: a CUDA fp32 tensor, or a CPU fp32 tensor / numpy array (copied by the library
    on the context's stream; a page-locked CPU tensor is read only when the stream reaches
    that copy, so keep it alive and unchanged until then)."""
    import numpy as np
    keep = None
    if hasattr(losses, "is_cuda") and losses.is_cuda:
        ptr, n, on_host = _ptr(losses), losses.numel(), 0
    else:
        keep = np.ascontiguousarray(np.asarray(losses, dtype=np.float32))
        ptr, n, on_host = keep.ctypes.data, keep.size, 1
    _check(LIB.zo_step(ctx, int(t), int(adam_t), ptr, int(n), on_host, int(scheme), int(optimizer),
                       float(eps), float(lr), float(beta1), float(beta2), float(eps_adam),
                       int(restore_query), float(restore_coef), _ptr(gamma_out)), "zo_step")
    del keep


def zo_mezo_perturb(ctx, t, coef):
    _check(LIB.zo_mezo_perturb(ctx, int(t), float(coef)), "zo_mezo_perturb")


def zo_linear_prepare(ctx, t, qa, ca, qb, cb, eps):
    """C_i = eps (ca Z_qa + cb Z_qb) at step t and P_i = C_i V_i^T for every matrix, for the
    zo_linear_perturbed calls of one loss evaluation."""
    _check(LIB.zo_linear_prepare(ctx, int(t), int(qa), float(ca), int(qb), float(cb),
                                 float(eps)), "zo_linear_prepare")


def zo_linear_perturbed(ctx, i, X, Y):
    """Y = X (W_i + U_i C_i V_i^T)^T with the prepared C_i; X (T x n) and Y (T x m) bf16
    CUDA tensors with unit column stride."""
    if X.dim() != 2 or Y.dim() != 2 or X.stride(1) != 1 or Y.stride(1) != 1 or X.shape[0] != Y.shape[0]:
        raise ValueError("X and Y must be 2-D, row-major (unit column stride), with the same rows")
    _check(LIB.zo_linear_perturbed(ctx, int(i), _ptr(X), int(X.shape[0]), int(X.stride(0)),
                                   _ptr(Y), int(Y.stride(0))), "zo_linear_perturbed")


def zo_sync_status(ctx):
    _check(LIB.zo_sync_status(ctx), "zo_sync_status")


def zo_set_option(ctx, option, value):
    _check(LIB.zo_set_option(ctx, int(option), int(value)), "zo_set_option")


def zo_get_timing(ctx):
    ms = ctypes.c_double()
    n = ctypes.c_int64()
    _check(LIB.zo_get_timing(ctx, ctypes.byref(ms), ctypes.byref(n)), "zo_get_timing")
    return ms.value, n.value


def zo_wpass_path(ctx):
    return int(LIB.zo_wpass_path(ctx))


def zo_linear_tiling(ctx):
    return int(LIB.zo_linear_tiling(ctx))


def zo_kernel_launches(ctx):
    return int(LIB.zo_kernel_launches(ctx))


def zo_perturb_noalloc(W, U, V, r, seed, matrix_index, t, qa, ca, qb, cb, eps, stream=None):
    """One perturbation pass on one matrix with no device allocation (see include/zo.h).
    W: m x n bf16/fp32 with unit column stride; U (m x r) and V (n x r) contiguous fp32 --
    checked here, since the C ABI cannot see the sizes behind its pointers."""
    import torch
    if W.dtype == torch.bfloat16:
        dt = ZO_BF16
    elif W.dtype == torch.float32:
        dt = ZO_F32
    else:
        raise ZoError(ZO_ERR_DTYPE, "zo_perturb_noalloc", str(W.dtype))
    if W.dim() != 2 or W.stride(1) != 1:
        raise ZoError(ZO_ERR_SHAPE, "zo_perturb_noalloc", "W must be 2-D with unit column stride")
    for name, t_, rows in (("U", U, W.shape[0]), ("V", V, W.shape[1])):
        if t_.dtype != torch.float32 or not t_.is_contiguous():
            raise ZoError(ZO_ERR_DTYPE, "zo_perturb_noalloc", f"{name} must be contiguous fp32")
        if tuple(t_.shape) != (rows, int(r)):
            raise ZoError(ZO_ERR_SHAPE, "zo_perturb_noalloc",
                          f"{name} has shape {tuple(t_.shape)}, expected {(rows, int(r))}")
    _check(LIB.zo_perturb_noalloc(_ptr(W), W.shape[0], W.shape[1], W.stride(0), dt, _ptr(U),
                                  _ptr(V), int(r), int(seed) & (2**64 - 1), int(matrix_index),
                                  int(t), int(qa), float(ca), int(qb), float(cb), float(eps),
                                  _stream_handle(stream)), "zo_perturb_noalloc")


def zo_philox_fill(seed, x1, x2, x3, out, stream=None):
    _check(LIB.zo_philox_fill(int(seed) & (2**64 - 1), int(x1), int(x2), int(x3), _ptr(out),
                              out.numel(), _stream_handle(stream)), "zo_philox_fill")


def zo_normal_fill(seed, x1, x2, x3, out, stream=None):
    _check(LIB.zo_normal_fill(int(seed) & (2**64 - 1), int(x1), int(x2), int(x3), _ptr(out),
                              out.numel(), _stream_handle(stream)), "zo_normal_fill")
