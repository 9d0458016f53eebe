"""Shared set-up for the GPU parity tests: weights on the device, snapshots to fp64."""

import numpy as np
import torch

from oracle import subzero
from parity import to_f64, update_terms


def make_weight(m, n, dtype, seed, device, ldw=None, scale=0.02):
    """N(0, scale^2) weight from torch's CPU generator, copied to the device.
    With ldw > n the tensor is a column slice of an m x ldw buffer (row stride ldw)."""
    g = torch.Generator().manual_seed(seed)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    w = (torch.randn(m, n, generator=g, dtype=torch.float32) * scale).to(dt)
    if ldw is None or ldw == n:
        return w.to(device)
    buf = torch.zeros(m, ldw, dtype=dt)
    buf[:, :n] = w
    return buf.to(device)[:, :n]


def snapshot(z):
    torch.cuda.synchronize()
    return {
        "W": [to_f64(W) for W in z.weights],
        "U": [to_f64(U) for U in z.U],
        "V": [to_f64(V) for V in z.V],
        "M": [to_f64(M) for M in z.M],
        "Vm": [to_f64(Vm) for Vm in z.Vm],
    }


def dtype_of(W):
    return "bf16" if W.dtype == torch.bfloat16 else "f32"


def f32(x):
    """The fp32 value a Python float becomes at the C boundary."""
    return float(np.float32(x))


def oracle_perturb(before, i, dtype, seed, gidx, t, r, terms, eps):
    """Expected W after a perturbation pass, and the (T, TZ) operand scale of the update."""
    C = subzero.perturb_coeff(seed, gidx, t, r, terms, f32(eps))
    W = subzero.apply_pass(before["W"][i], dtype, before["U"][i], before["V"][i], C)
    zc = abs(f32(eps)) * sum(abs(c) for _, c in terms)
    return W, update_terms(before["U"][i], C, before["V"][i], zc)


def oracle_step(before, i, dtype, seed, gidx, t, r, q, losses, scheme, eps, lr, beta1, beta2,
                eps_adam, adam_t, restore_terms, optimizer="adam"):
    rho = subzero.rho_from_losses(np.asarray(losses, np.float32), scheme, f32(eps), q)
    G = subzero.grad_G(seed, gidx, t, r, rho)
    if optimizer == "adam":
        M, Vm, D, _, _ = subzero.adam(before["M"][i], before["Vm"][i], G, f32(beta1), f32(beta2),
                                      f32(eps_adam), adam_t)
    else:
        M, Vm, D = before["M"][i], before["Vm"][i], subzero.sgd_direction(G)
    C = subzero.step_coeff(D, f32(lr), f32(eps), restore_terms, seed, gidx, t, r)
    W = subzero.apply_pass(before["W"][i], dtype, before["U"][i], before["V"][i], C)
    zc = abs(f32(eps)) * sum(abs(c) for _, c in restore_terms)
    return W, M, Vm, G, update_terms(before["U"][i], C, before["V"][i], zc)
