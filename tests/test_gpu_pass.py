"""Per-call GPU parity of the weight passes (zo_perturb, zo_step) against the oracle.

Each test reads the library's state before a call (W, U, V, M, Vm), lets the
oracle compute the call exactly in fp64 from that state, and compares:
bf16 weights within 1 ulp of the oracle's rounded result, fp32 weights and the
Adam moments within relative 1e-5, both at the scale of the operands (tests/parity.py).
"""

import numpy as np
import pytest
import torch

from gpu_util import dtype_of, f32, make_weight, oracle_perturb, oracle_step, snapshot
from oracle import rounding, subzero
from parity import assert_moments, assert_weights, gabs, to_f64

pytestmark = pytest.mark.gpu

# (r, [(m, n, dtype, ldw)]) -- several tiles in both directions plus ragged tails
CASES = {
    "r4": (4, [(300, 520, "bf16", None), (64, 1000, "f32", None), (8, 5120, "f32", None),
               (5120, 8, "f32", None)]),
    "r8": (8, [(300, 520, "bf16", None), (1030, 72, "bf16", None), (256, 256, "f32", None)]),
    "r16": (16, [(300, 520, "bf16", 528), (130, 1000, "bf16", None), (100, 96, "f32", 100)]),
    "r32": (32, [(300, 520, "bf16", None), (1030, 72, "bf16", 80), (64, 2048, "f32", None)]),
    "r64": (64, [(300, 520, "bf16", None), (130, 1000, "bf16", None), (1030, 72, "f32", None)]),
    "r128": (128, [(300, 520, "bf16", None), (130, 1000, "f32", None)]),
}


def _build(gpu, case, seed, base=3):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    r, spec = CASES[case]
    weights = [make_weight(m, n, dt, 100 + k, gpu, ldw) for k, (m, n, dt, ldw) in enumerate(spec)]
    z = SubZeroPlus(weights, r, 4, seed, matrix_index_base=base)
    z.init_subspace(0)
    return z, base


@pytest.mark.parametrize("case", list(CASES))
@pytest.mark.parametrize("eps", [1e-3, 1e-1])
def test_perturb_pass_matches_oracle(lib, gpu, case, eps):
    z, base = _build(gpu, case, seed=555)
    calls = [(0, 1.0, -1, 0.0), (0, -2.0, -1, 0.0), (0, 1.0, 1, 1.0), (3, 1.0, 2, -1.0)]
    for t, (qa, ca, qb, cb) in zip((0, 0, 7, 123456), calls):
        before = snapshot(z)
        z.perturb(t, qa, ca, qb, cb, eps)
        after = snapshot(z)
        terms = [(qa, ca)] + ([(qb, cb)] if qb >= 0 else [])
        for i, W in enumerate(z.weights):
            want, T = oracle_perturb(before, i, dtype_of(W), z.seed, base + i, t, z.r, terms, eps)
            assert_weights(after["W"][i], want, dtype_of(W), f"{case} matrix {i} t={t}",
                           before=before["W"][i], terms=T)
    z.sync()
    z.close()


@pytest.mark.parametrize("case", ["r4", "r8", "r16", "r32", "r64", "r128"])
@pytest.mark.parametrize("scheme", ["central", "forward", "direct"])
def test_step_matches_oracle(lib, gpu, case, scheme):
    z, base = _build(gpu, case, seed=777)
    q, eps, lr, b1, b2, ea = z.q, 1e-3, 1e-2, 0.9, 0.95, 1e-8
    n_losses = {"central": 2 * q, "forward": q + 1, "direct": q}[scheme]
    restore = {"central": (q - 1, 1.0), "forward": (q - 1, -1.0), "direct": (-1, 0.0)}[scheme]
    rs = np.random.default_rng(5)
    gamma = torch.zeros(len(z.weights), dtype=torch.float32, device=gpu)
    for step, t in enumerate((0, 1, 2)):
        if scheme == "direct":
            losses = (rs.standard_normal(n_losses) * 7.0).astype(np.float32)
        else:
            losses = (2.0 + 0.01 * rs.standard_normal(n_losses)).astype(np.float32)
        before = snapshot(z)
        z.step(t, step + 1, losses, scheme, eps, lr, b1, b2, ea, restore[0], restore[1],
               gamma_out=gamma)
        after = snapshot(z)
        g = gamma.cpu().double().numpy()
        rterms = [restore] if restore[0] >= 0 else []
        rho = subzero.rho_from_losses(losses, scheme, f32(eps), q)
        for i, W in enumerate(z.weights):
            Wo, Mo, Vmo, G, T = oracle_step(before, i, dtype_of(W), z.seed, base + i, t, z.r, q,
                                            losses, scheme, eps, lr, b1, b2, ea, step + 1, rterms)
            ga = gabs(z.seed, base + i, t, z.r, rho)
            assert_moments(after["M"][i], after["Vm"][i], Mo, Vmo, before["M"][i],
                           before["Vm"][i], ga, b1, b2, f"{case} {i}")
            assert_weights(after["W"][i], Wo, dtype_of(W), f"W {case} {i} step {step}",
                           before=before["W"][i], terms=T)
            assert abs(g[i] - np.linalg.norm(G)) <= 1e-5 * np.linalg.norm(ga)
    z.close()


def test_sgd_step_matches_oracle_and_leaves_moments(lib, gpu):
    z, base = _build(gpu, "r8", seed=31)
    z.M[0].fill_(0.25)
    losses = (2.0 + 0.01 * np.random.default_rng(1).standard_normal(2 * z.q)).astype(np.float32)
    before = snapshot(z)
    from paper_2608_15665_gb300 import binding as zb
    z.step(4, 1, losses, "central", 1e-3, 1e-4, 0.9, 0.95, 1e-8, z.q - 1, 1.0,
           optimizer=zb.ZO_OPT_SGD)
    after = snapshot(z)
    for i, W in enumerate(z.weights):
        Wo, _, _, _, T = oracle_step(before, i, dtype_of(W), z.seed, base + i, 4, z.r, z.q, losses,
                                     "central", 1e-3, 1e-4, 0.9, 0.95, 1e-8, 1, [(z.q - 1, 1.0)],
                                     optimizer="sgd")
        assert_weights(after["W"][i], Wo, dtype_of(W), f"sgd W {i}", before=before["W"][i],
                       terms=T)
        assert np.array_equal(after["M"][i], before["M"][i])
    z.close()


def test_losses_from_device_memory(lib, gpu):
    z, base = _build(gpu, "r16", seed=9)
    losses = (2.0 + 0.01 * np.random.default_rng(2).standard_normal(2 * z.q)).astype(np.float32)
    before = snapshot(z)
    z.step(0, 1, torch.from_numpy(losses).to(gpu), "central", 1e-3, 1e-3, 0.9, 0.95, 1e-8,
           z.q - 1, 1.0)
    after = snapshot(z)
    Wo, Mo, Vmo, _, T = oracle_step(before, 0, "bf16", z.seed, base, 0, z.r, z.q, losses,
                                    "central", 1e-3, 1e-3, 0.9, 0.95, 1e-8, 1, [(z.q - 1, 1.0)])
    ga = gabs(z.seed, base, 0, z.r, subzero.rho_from_losses(losses, "central", f32(1e-3), z.q))
    assert_moments(after["M"][0], after["Vm"][0], Mo, Vmo, before["M"][0], before["Vm"][0], ga,
                   0.9, 0.95, "device losses")
    assert_weights(after["W"][0], Wo, "bf16", "W", before=before["W"][0], terms=T)
    z.close()


def test_same_calls_give_bit_identical_weights(lib, gpu):
    outs = []
    for _ in range(2):
        z, _ = _build(gpu, "r32", seed=2024)
        z.perturb(3, 0, 1.0, -1, 0.0, 1e-1)
        z.perturb(3, 0, 1.0, 1, 1.0, 1e-1)
        z.step(3, 1, np.full(2 * z.q, 2.0, np.float32) + np.arange(2 * z.q, dtype=np.float32) * 1e-3,
               "central", 1e-1, 1e-2, 0.9, 0.95, 1e-8, z.q - 1, 1.0)
        torch.cuda.synchronize()
        outs.append([W.clone() for W in z.weights])
        z.close()
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_padding_columns_beyond_n_are_untouched(lib, gpu):
    # ldw > n: the bytes between n and ldw belong to the caller and must not change
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    buf = make_weight(200, 272, "bf16", 3, gpu)
    view = buf[:, :264]
    z = SubZeroPlus([view], 8, 2, 1)
    z.init_subspace(0)
    pad = buf[:, 264:].clone()
    z.perturb(0, 0, 1.0, -1, 0.0, 1e-1)
    torch.cuda.synchronize()
    assert torch.equal(buf[:, 264:], pad)
    z.close()


def test_rejected_calls_launch_nothing(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    z, _ = _build(gpu, "r8", seed=4)
    before = snapshot(z)
    with pytest.raises(zb.ZoError) as e:
        z.perturb(0, 4, 1.0, -1, 0.0, 1e-3)          # qa == q
    assert e.value.status == zb.ZO_ERR_INVALID_ARG
    with pytest.raises(zb.ZoError):
        z.step(0, 1, np.zeros(3, np.float32), "central", 1e-3, 1e-3, 0.9, 0.95, 1e-8, 3, 1.0)
    with pytest.raises(zb.ZoError):
        z.step(0, 0, np.zeros(8, np.float32), "central", 1e-3, 1e-3, 0.9, 0.95, 1e-8, 3, 1.0)
    after = snapshot(z)
    for k in ("W", "M", "Vm"):
        for a, b in zip(before[k], after[k]):
            assert np.array_equal(a, b)
    z.sync()
    z.close()


# bf16-only contexts with r in {16, 32, 64} run the tensor-core weight pass:
# tiles of 128 x 128 with ragged rows and columns, and a padded row stride.
TC_CASES = {
    "tc16": (16, [(300, 520, None), (130, 1000, 1008), (1030, 72, None), (128, 128, None)]),
    "tc32": (32, [(300, 520, 528), (1030, 72, 80), (257, 2048, None)]),
    "tc64": (64, [(300, 520, None), (130, 1000, None), (1030, 72, 72), (2048, 384, None)]),
    "tc128": (128, [(300, 520, None), (130, 1000, 1008), (1030, 136, None)]),
}


def _build_tc(gpu, case, seed, base=11):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    r, spec = TC_CASES[case]
    weights = [make_weight(m, n, "bf16", 200 + k, gpu, ldw) for k, (m, n, ldw) in enumerate(spec)]
    z = SubZeroPlus(weights, r, 4, seed, matrix_index_base=base)
    z.init_subspace(0)
    return z, base


@pytest.mark.parametrize("case", list(TC_CASES))
@pytest.mark.parametrize("eps", [1e-3, 1e-1])
def test_tensor_core_pass_matches_oracle(lib, gpu, case, eps):
    from paper_2608_15665_gb300 import binding as zb
    z, base = _build_tc(gpu, case, seed=909)
    calls = [(0, 1.0, -1, 0.0), (0, -2.0, -1, 0.0), (0, 1.0, 1, 1.0), (3, 1.0, 2, -1.0)]
    for t, (qa, ca, qb, cb) in zip((0, 0, 7, 99), calls):
        before = snapshot(z)
        z.perturb(t, qa, ca, qb, cb, eps)
        after = snapshot(z)
        assert zb.zo_wpass_path(z.ctx) == 2
        terms = [(qa, ca)] + ([(qb, cb)] if qb >= 0 else [])
        for i in range(len(z.weights)):
            want, T = oracle_perturb(before, i, "bf16", z.seed, base + i, t, z.r, terms, eps)
            assert_weights(after["W"][i], want, "bf16", f"{case} matrix {i} t={t}",
                           before=before["W"][i], terms=T)
    z.sync()
    z.close()


@pytest.mark.parametrize("case", list(TC_CASES))
def test_tensor_core_step_matches_oracle(lib, gpu, case):
    z, base = _build_tc(gpu, case, seed=313)
    q, eps, lr, b1, b2, ea = z.q, 1e-2, 1e-2, 0.9, 0.95, 1e-8
    rs = np.random.default_rng(8)
    for step in range(2):
        losses = (2.0 + 0.01 * rs.standard_normal(2 * q)).astype(np.float32)
        before = snapshot(z)
        z.step(step, step + 1, losses, "central", eps, lr, b1, b2, ea, q - 1, 1.0)
        after = snapshot(z)
        rho = subzero.rho_from_losses(losses, "central", f32(eps), q)
        for i in range(len(z.weights)):
            Wo, Mo, Vmo, _, T = oracle_step(before, i, "bf16", z.seed, base + i, step, z.r, q,
                                            losses, "central", eps, lr, b1, b2, ea, step + 1,
                                            [(q - 1, 1.0)])
            assert_moments(after["M"][i], after["Vm"][i], Mo, Vmo, before["M"][i],
                           before["Vm"][i], gabs(z.seed, base + i, step, z.r, rho), b1, b2,
                           f"{case} {i}")
            assert_weights(after["W"][i], Wo, "bf16", f"W {case} {i} step {step}",
                           before=before["W"][i], terms=T)
    z.sync()
    z.close()


@pytest.mark.parametrize("r", [16, 32, 64, 128])
def test_tensor_core_rings_wrap(lib, gpu, r):
    # 1280 + 15 tiles over 152 CTAs in chunks of 4: some CTAs take 3 chunks, so their U
    # operand ring (two stages / two TMEM buffers) is reused and every barrier phase
    # wraps; checked element by element for one pass and one step.
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    base = 40
    weights = [make_weight(m, n, "bf16", 600 + k, gpu, None)
               for k, (m, n) in enumerate([(4096, 5120), (300, 520)])]
    z = SubZeroPlus(weights, r, 2, 2024, matrix_index_base=base)
    z.init_subspace(0)
    before = snapshot(z)
    z.perturb(0, 0, 1.0, 1, -1.0, 1e-1)
    after = snapshot(z)
    assert zb.zo_wpass_path(z.ctx) == 2
    for i in range(2):
        want, T = oracle_perturb(before, i, "bf16", z.seed, base + i, 0, r, [(0, 1.0), (1, -1.0)],
                                 1e-1)
        assert_weights(after["W"][i], want, "bf16", f"r{r} matrix {i} pass", before=before["W"][i],
                       terms=T)
    losses = np.array([2.01, 1.99, 2.0, 2.02], np.float32)
    before = after
    z.step(0, 1, losses, "central", 1e-1, 1e-2, 0.9, 0.95, 1e-8, 1, 1.0)
    after = snapshot(z)
    for i in range(2):
        Wo, _, _, _, T = oracle_step(before, i, "bf16", z.seed, base + i, 0, r, 2, losses, "central",
                                     1e-1, 1e-2, 0.9, 0.95, 1e-8, 1, [(1, 1.0)])
        assert_weights(after["W"][i], Wo, "bf16", f"r{r} matrix {i} step", before=before["W"][i],
                       terms=T)
    z.sync()
    z.close()


@pytest.mark.parametrize("shapes", [
    [(300, 520, None), (130, 1000, 1008), (1030, 136, None)],
    # a pair tile's second 128 rows empty (m = 128), exactly full (m = 256), one row into the
    # second pair tile (m = 257), and 200 rows of a single column block
    [(128, 256, None), (256, 384, None), (257, 136, 144), (200, 128, None)],
], ids=["ragged", "edges"])
def test_sm_pair_and_single_sm_passes_are_bit_identical(lib, gpu, shapes):
    # r = 128: the weight pass as M = 256 MMAs across an SM pair (the default) and as the
    # single-SM kernel sum the same products in the same order: a pass and a step give the
    # same bits (both are also checked against the oracle above)
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    out = {}
    for option in (1, 0):
        weights = [make_weight(m, n, "bf16", 700 + k, gpu, ldw) for k, (m, n, ldw) in enumerate(shapes)]
        z = SubZeroPlus(weights, 128, 4, 5151, matrix_index_base=3)
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_PAIR_MMA, option)
        z.init_subspace(0)
        z.perturb(0, 0, 1.0, 1, -1.0, 1e-1)
        z.step(0, 1, np.array([2.01, 1.99, 2.0, 2.02, 1.98, 2.0, 2.03, 2.01], np.float32),
               "central", 1e-1, 1e-2, 0.9, 0.95, 1e-8, 3, 1.0)
        z.sync()
        assert zb.zo_wpass_path(z.ctx) == 2
        out[option] = [W.clone() for W in z.weights]
        z.close()
    for i, (a, b) in enumerate(zip(out[1], out[0])):
        assert torch.equal(a, b), f"matrix {i}: SM-pair and single-SM weight passes differ"


@pytest.mark.parametrize("case", list(TC_CASES))
def test_tensor_core_and_fma_paths_agree(lib, gpu, case):
    # one pass from the same state on both paths: each is within 1 ulp (at the operand
    # scale) of the exact result, so they differ by at most 2 such ulps, and rarely at all
    from paper_2608_15665_gb300 import binding as zb
    out = {}
    for path in (1, 2):
        z, base = _build_tc(gpu, case, seed=4321)
        before = snapshot(z)
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_WPASS_PATH, path)
        z.perturb(0, 0, 1.0, 1, -1.0, 1e-1)
        assert zb.zo_wpass_path(z.ctx) == path
        out[path] = [to_f64(W) for W in z.weights]
        z.close()
    for i, (a, b) in enumerate(zip(out[1], out[2])):
        _, (T, TZ) = oracle_perturb(before, i, "bf16", 4321, base + i, 0, TC_CASES[case][0],
                                    [(0, 1.0), (1, -1.0)], 1e-1)
        scale = np.maximum.reduce([np.abs(a), np.abs(b), np.abs(before["W"][i]), T])
        d = np.abs(a - b)
        assert np.all(d <= 2 * rounding.bf16_ulp(scale) + 2 * TZ)
        assert (d > 0).mean() < 1e-2


# Sets of thin matrices at r in {4, 8}: LoRA-like factors in both orientations, ragged
# widths, padded rows, a tall matrix of a single 16-byte chunk per row.
NARROW_CASES = {
    "lora4": (4, [(8, 1000, "f32", 1004), (1000, 8, "f32", None), (8, 520, "bf16", None),
                  (520, 8, "bf16", 16), (5, 77, "f32", 80), (3000, 4, "f32", None)]),
    "lora8": (8, [(8, 5120, "f32", None), (5120, 8, "f32", None), (16, 1030, "bf16", 1032),
                  (1030, 12, "bf16", 16)]),
    "r4": CASES["r4"],
    "r8": CASES["r8"],
}


def _build_narrow(gpu, case, seed, base=21):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    r, spec = NARROW_CASES[case]
    weights = [make_weight(m, n, dt, 300 + k, gpu, ldw) for k, (m, n, dt, ldw) in enumerate(spec)]
    z = SubZeroPlus(weights, r, 4, seed, matrix_index_base=base)
    z.init_subspace(0)
    return z, base


@pytest.mark.parametrize("case", list(NARROW_CASES))
def test_narrow_tile_pass_and_step_match_oracle(lib, gpu, case):
    from paper_2608_15665_gb300 import binding as zb
    z, base = _build_narrow(gpu, case, seed=2468)
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_WPASS_PATH, 3)
    calls = [(0, 1.0, -1, 0.0), (0, -2.0, 1, 1.0), (3, 1.0, 2, -1.0)]
    for t, (qa, ca, qb, cb) in zip((0, 0, 5), calls):
        before = snapshot(z)
        z.perturb(t, qa, ca, qb, cb, 1e-1)
        after = snapshot(z)
        assert zb.zo_wpass_path(z.ctx) == 3
        terms = [(qa, ca)] + ([(qb, cb)] if qb >= 0 else [])
        for i, W in enumerate(z.weights):
            want, T = oracle_perturb(before, i, dtype_of(W), z.seed, base + i, t, z.r, terms, 1e-1)
            assert_weights(after["W"][i], want, dtype_of(W), f"{case} matrix {i} t={t}",
                           before=before["W"][i], terms=T)
    q, eps, lr, b1, b2, ea = z.q, 1e-2, 1e-2, 0.9, 0.95, 1e-8
    losses = np.array([2.01, 1.99, 2.0, 2.02, 1.97, 2.0, 2.03, 1.98], np.float32)
    before = snapshot(z)
    z.step(5, 1, losses, "central", eps, lr, b1, b2, ea, q - 1, 1.0)
    after = snapshot(z)
    assert zb.zo_wpass_path(z.ctx) == 3
    rho = subzero.rho_from_losses(losses, "central", f32(eps), q)
    for i, W in enumerate(z.weights):
        Wo, Mo, Vmo, _, T = oracle_step(before, i, dtype_of(W), z.seed, base + i, 5, z.r, q, losses,
                                        "central", eps, lr, b1, b2, ea, 1, [(q - 1, 1.0)])
        assert_moments(after["M"][i], after["Vm"][i], Mo, Vmo, before["M"][i], before["Vm"][i],
                       gabs(z.seed, base + i, 5, z.r, rho), b1, b2, f"{case} {i}")
        assert_weights(after["W"][i], Wo, dtype_of(W), f"W {case} {i} step",
                       before=before["W"][i], terms=T)
    z.sync()
    z.close()


@pytest.mark.parametrize("case", list(NARROW_CASES))
def test_narrow_and_32_row_tiles_are_bit_identical(lib, gpu, case):
    # the two FMA tilings share C, the order of P's sum and of the update's sum, and the one
    # rounding: every weight must come out bit for bit the same, pass after pass
    from paper_2608_15665_gb300 import binding as zb
    out = {}
    losses = np.array([2.01, 1.99, 2.0, 2.02, 1.97, 2.0, 2.03, 1.98], np.float32)
    for path in (1, 3):
        z, _ = _build_narrow(gpu, case, seed=1357)
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_WPASS_PATH, path)
        z.perturb(0, 0, 1.0, -1, 0.0, 1e-1)
        z.perturb(0, 0, -2.0, 1, 1.0, 1e-1)
        z.step(0, 1, losses, "central", 1e-1, 1e-2, 0.9, 0.95, 1e-8, z.q - 1, 1.0)
        assert zb.zo_wpass_path(z.ctx) == path
        z.sync()
        out[path] = [W.detach().cpu().contiguous() for W in z.weights]
        z.close()
    for i, (a, b) in enumerate(zip(out[1], out[3])):
        assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a.view(torch.int32),
                           b.view(torch.int16) if b.dtype == torch.bfloat16 else b.view(torch.int32)), \
            f"{case} matrix {i}"


def test_narrow_tiles_are_chosen_for_thin_sets(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    z, _ = _build_narrow(gpu, "lora4", seed=11)
    z.perturb(0, 0, 1.0, -1, 0.0, 1e-3)
    assert zb.zo_wpass_path(z.ctx) == 3           # automatic: thin set -> narrow tiles
    z.close()
    z, _ = _build(gpu, "r8", seed=11)
    z.perturb(0, 0, 1.0, -1, 0.0, 1e-3)
    assert zb.zo_wpass_path(z.ctx) == 1           # 256 x 256 etc.: the 32-row tiles
    z.close()
    z, _ = _build_tc(gpu, "tc32", seed=11)
    with pytest.raises(RuntimeError):
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_WPASS_PATH, 3)   # r = 32: no narrow tiles
    z.close()


@pytest.mark.parametrize("r", [16, 32, 64, 128])
@pytest.mark.parametrize("widths,path", [((512, 136), 2), ((517, 133), 1)], ids=["n%8=0", "odd-n"])
def test_row_padding_past_n_is_untouched(lib, gpu, r, widths, path):
    # W is a column slice of a wider buffer (ldw > n): the elements past n in each row
    # belong to the caller and keep their (NaN) contents.  TMA stores write whole 16-byte
    # chunks, so a set with a width that is not a multiple of 8 takes the FMA path.
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    shapes = [(300, widths[0], 528), (259, widths[1], 144)]
    bufs, weights = [], []
    for k, (m, n, ldw) in enumerate(shapes):
        g = torch.Generator().manual_seed(900 + k)
        buf = torch.full((m, ldw), float("nan"), dtype=torch.bfloat16)
        buf[:, :n] = (torch.randn(m, n, generator=g) * 0.02).to(torch.bfloat16)
        buf = buf.to(gpu)
        bufs.append(buf)
        weights.append(buf[:, :n])
    z = SubZeroPlus(weights, r, 2, 77)
    z.init_subspace(0)
    before = snapshot(z)
    z.perturb(0, 0, 1.0, 1, -1.0, 1e-1)
    assert zb.zo_wpass_path(z.ctx) == path
    after = snapshot(z)
    for i in range(2):
        want, T = oracle_perturb(before, i, "bf16", z.seed, i, 0, r, [(0, 1.0), (1, -1.0)], 1e-1)
        assert_weights(after["W"][i], want, "bf16", f"r{r} matrix {i}", before=before["W"][i],
                       terms=T)
    z.step(0, 1, np.array([2.01, 1.99, 2.0, 2.02], np.float32), "central", 1e-1, 1e-2, 0.9, 0.95,
           1e-8, 1, 1.0)
    z.sync()
    for (m, n, ldw), buf in zip(shapes, bufs):
        assert torch.isnan(buf[:, n:].float()).all(), f"row padding of a {m}x{n} matrix written"
        assert not torch.isnan(buf[:, :n].float()).any()
    z.close()
