"""The C-ABI library loads, exports what include/zo.h declares, and validates
arguments on the host (no GPU: nothing here reaches a kernel launch)."""

import ctypes
import os
import re

import pytest

from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "zo.h")


def declared_functions():
    text = open(HEADER).read()
    return re.findall(r"^ZO_API\s+[\w\s\*]+?\b(zo_\w+)\s*\(", text, flags=re.M)


def test_header_declares_the_paper_entry_points():
    names = set(declared_functions())
    for want in ("zo_create", "zo_destroy", "zo_init_subspace", "zo_refresh", "zo_perturb",
                 "zo_step", "zo_sync_status", "zo_philox_fill", "zo_normal_fill"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    so = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(so, n)]
    assert not missing, missing


def test_binding_covers_every_declared_symbol(lib):
    assert set(declared_functions()) <= set(lib._SIGNATURES)


def test_status_strings(lib):
    assert lib.status_string(lib.ZO_OK) == "ok"
    assert "align" in lib.status_string(lib.ZO_ERR_ALIGN)
    assert lib.status_string(99) == "unknown status"


def _mat(lib, W=0x1000, m=64, n=64, ldw=64, dtype=1, U=0x2000, V=0x3000, M=0x4000, Vm=0x5000):
    return lib.zo_matrix(W, m, n, ldw, dtype, 0, U, V, M, Vm)


def _create_status(lib, mats, r=8, q=2):
    arr = (lib.zo_matrix * len(mats))(*mats)
    ctx = ctypes.c_void_p()
    st = lib.LIB.zo_create(ctypes.byref(ctx), arr, len(mats), r, q, 1, 0, None)
    return st, ctx


@pytest.mark.parametrize("kw,status", [
    (dict(W=0), 1), (dict(U=0), 1), (dict(Vm=0), 1),          # null buffers
    (dict(dtype=7), 4),                                         # unknown dtype
    (dict(m=4), 2), (dict(n=4), 2), (dict(ldw=32), 2),          # r > min(m, n), ldw < n
    (dict(W=0x1008), 3), (dict(U=0x2004), 3), (dict(ldw=68, dtype=1), 3),  # alignment
])
def test_create_rejects_bad_matrices_before_touching_the_device(lib, kw, status):
    st, ctx = _create_status(lib, [_mat(lib, **kw)])
    assert st == status and not ctx.value


@pytest.mark.parametrize("r,q,status", [(5, 2, 2), (128, 2, 2), (0, 2, 2), (8, 0, 1), (8, 5000, 1)])
def test_create_rejects_bad_rank_and_query_count(lib, r, q, status):
    st, _ = _create_status(lib, [_mat(lib)], r=r, q=q)
    assert st == status


def test_calls_on_null_context_are_rejected(lib):
    L = lib.LIB
    assert L.zo_perturb(None, 0, 0, 1.0, -1, 0.0, 1e-3) == lib.ZO_ERR_INVALID_ARG
    assert L.zo_refresh(None, 0, 0) == lib.ZO_ERR_INVALID_ARG
    assert L.zo_sync_status(None) == lib.ZO_ERR_INVALID_ARG
    assert L.zo_destroy(None) == lib.ZO_OK
    assert L.zo_wpass_path(None) == 0
    assert L.zo_linear_tiling(None) == 0


def test_rng_fills_validate_sizes(lib):
    L = lib.LIB
    assert L.zo_philox_fill(1, 0, 0, 0, None, -1, None) == lib.ZO_ERR_INVALID_ARG
    assert L.zo_normal_fill(1, 0, 0, 0, None, 16, None) == lib.ZO_ERR_INVALID_ARG
    assert L.zo_philox_fill(1, 0, 0, 0, None, 0, None) == lib.ZO_OK   # empty: nothing launched


def test_create_rejects_an_empty_set_and_a_null_output(lib):
    arr = (lib.zo_matrix * 1)(_mat(lib))
    ctx = ctypes.c_void_p(0x1234)
    assert lib.LIB.zo_create(ctypes.byref(ctx), arr, 0, 8, 2, 1, 0, None) == lib.ZO_ERR_INVALID_ARG
    assert not ctx.value                                       # *out cleared on failure
    assert lib.LIB.zo_create(ctypes.byref(ctx), None, 1, 8, 2, 1, 0, None) == lib.ZO_ERR_INVALID_ARG
    assert lib.LIB.zo_create(None, arr, 1, 8, 2, 1, 0, None) == lib.ZO_ERR_INVALID_ARG


def test_create_without_a_device_fails_instead_of_falling_back(lib):
    # a valid request on a machine with no visible GPU: the library has no CPU path, so the
    # context is refused with ZO_ERR_CUDA (on a GPU machine the same call would build a
    # context over the fake pointers, so it is not made there)
    from conftest import cuda_available
    if cuda_available():
        pytest.skip("a GPU is visible")
    st, ctx = _create_status(lib, [_mat(lib)])
    assert st == lib.ZO_ERR_CUDA and not ctx.value
    assert lib.LIB.zo_last_error()


def _noalloc(lib, W=0x1000, m=64, n=64, ldw=64, dtype=0, U=0x2000, V=0x3000, r=8, qa=0, qb=-1,
             ca=1.0, cb=0.0, eps=1e-3):
    return lib.LIB.zo_perturb_noalloc(W, m, n, ldw, dtype, U, V, r, 1, 0, 0, qa, ca, qb, cb, eps,
                                      None)


@pytest.mark.parametrize("kw,status", [
    (dict(W=0), 1), (dict(U=0), 1), (dict(V=0), 1),               # null buffers
    (dict(dtype=3), 4),                                           # unknown dtype
    (dict(r=128), 2), (dict(r=5), 2),                             # ranks outside {4 ... 64}
    (dict(m=4), 2), (dict(ldw=32), 2),                            # r > m, ldw < n
    (dict(qa=-1), 1), (dict(qb=-2), 1), (dict(eps=float("inf")), 1),
    (dict(W=0x1008), 3), (dict(ldw=66, dtype=1), 3),              # alignment
    (dict(n=40000, ldw=40000, r=64), 2),                          # beyond the 8 MiB scratch
])
def test_noalloc_validates_on_the_host(lib, kw, status):
    # every one of these is refused before any CUDA call, so it needs no device
    assert _noalloc(lib, **kw) == status


@pytest.mark.parametrize("what", ["U rows", "V rank", "U dtype", "V strided", "W strided",
                                  "W dtype"])
def test_noalloc_binding_checks_shapes_before_the_call(lib, what):
    # the C ABI cannot see the sizes behind U and V; the binding refuses a U or V that does
    # not hold m x r / n x r contiguous fp32 values, and a W without unit column stride,
    # before the library is called (CPU tensors: nothing reaches a device)
    import torch
    m, n, r = 64, 96, 8
    W = torch.zeros(m, n)
    U = torch.zeros(m, r)
    V = torch.zeros(n, r)
    if what == "U rows":
        U = torch.zeros(m - 1, r)
    elif what == "V rank":
        V = torch.zeros(n, 2 * r)
    elif what == "U dtype":
        U = U.double()
    elif what == "V strided":
        V = torch.zeros(n, 2 * r)[:, ::2]
    elif what == "W strided":
        W = torch.zeros(n, m).t()
    else:
        W = W.half()
    with pytest.raises(lib.ZoError) as e:
        lib.zo_perturb_noalloc(W, U, V, r, 1, 0, 0, 0, 1.0, -1, 0.0, 1e-3)
    assert e.value.status in (lib.ZO_ERR_SHAPE, lib.ZO_ERR_DTYPE)
