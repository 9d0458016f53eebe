"""A linear layer at the perturbed weights without a weight pass (zo_linear_perturbed)
against the oracle: Y = X (W + U C V^T)^T with C = eps (ca Z_qa + cb Z_qb), W untouched.

The GPU sums X W^T in fp32 from exact bf16 products, adds the rank-r term S U^T with the
bf16 hi/lo split, and rounds Y to bf16 once; the oracle rounds the fp64 value once.  The
two differ by at most one bf16 ulp of the output plus the fp32 accumulation bound
(n 2^-24 sum |X||W|), the split's 2^-14 of sum |X||V||C||U| and the fp32 Gaussians'
allowance (tests/parity.py NORMAL_ABS) carried through |X||V| and |U|.
"""

import numpy as np
import pytest
import torch

from gpu_util import f32, make_weight, snapshot
from oracle import rounding, subzero
from parity import NORMAL_ABS, to_f64

pytestmark = pytest.mark.gpu

# ZO_OPTION_LINEAR_TILE values: 1..3 single-CTA tiles (with the separate S = X P^T
# kernel; r <= 32), 4..8 SM-pair tiles (N = 256, 240, 224, 192, 128 columns of Y; S in the
# same launch; every r)
TILINGS = (1, 2, 3, 4, 5, 6, 7, 8)
PAIR_TILINGS = (4, 5, 6, 7, 8)

# (r, [(m, n, ldw)], token counts).  r = 64 and 128 (the paper's rank): the rank-r step in
# one operand stage of two panels and in three, S tiles with 128 and 256 accumulator
# columns and one or two K panels per stage; ragged row blocks, column blocks and K panels.
# S comes from S tiles or from contributor tiles depending on the tiling (every pair tiling
# must give the same bits); 2000 and 3000 tokens put several row blocks' contributors in
# one wave of tiles.
LINEAR_CASES = {
    "r32": (32, [(304, 520, None), (264, 2048, None), (1032, 72, 80)], (1, 130, 300, 2000)),
    "r16": (16, [(304, 520, 528), (136, 1000, 1008), (64, 136, None)], (7, 257)),
    "r64": (64, [(392, 648, None), (136, 2056, 2064)], (5, 300, 3000)),
    "r128": (128, [(520, 1032, None), (264, 264, 272)], (3, 513)),
}


def _tilings(r):
    return TILINGS if r <= 32 else PAIR_TILINGS


def _context(gpu, case, seed, base=31):
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    r, spec, _ = LINEAR_CASES[case]
    weights = [make_weight(m, n, "bf16", 700 + k, gpu, ldw) for k, (m, n, ldw) in enumerate(spec)]
    z = SubZeroPlus(weights, r, 4, seed, matrix_index_base=base)
    z.init_subspace(0)
    return z, base


def _tokens(T, n, seed, gpu):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(T, n, generator=g).to(torch.bfloat16).to(gpu)


def _check(Y, X, W, U, V, C, zc, what):
    Xd, Wd = to_f64(X), np.asarray(W, np.float64)
    want = subzero.perturbed_linear(Xd, Wd, U, V, C, "bf16")
    got = to_f64(Y)
    aX = np.abs(Xd)
    a_w = aX @ np.abs(Wd).T
    a_s = aX @ (np.abs(V) @ np.abs(C).T) @ np.abs(U).T
    a_z = zc * NORMAL_ABS * np.outer(aX @ np.abs(V).sum(axis=1), np.abs(U).sum(axis=1))
    n = Wd.shape[1]
    tol = (rounding.bf16_ulp(np.maximum(np.abs(want), np.abs(got)))
           + 2.0 * (n * 2.0 ** -24 * a_w + 2.0 ** -14 * a_s + a_z))
    d = np.abs(got - want)
    bad = d > tol
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {d.size} outside the bound, worst "
                           f"{float((d - tol).max()):.3g} over")
    return want


@pytest.mark.parametrize("case", list(LINEAR_CASES))
@pytest.mark.parametrize("eps", [1e-3, 1e-1])
def test_perturbed_linear_matches_oracle_and_leaves_W(lib, gpu, case, eps):
    from paper_2608_15665_gb300 import binding as zb
    z, base = _context(gpu, case, seed=4242)
    r, spec, tokens = LINEAR_CASES[case]
    before = snapshot(z)
    W_bits = [W.detach().clone() for W in z.weights]
    terms = [(1, 1.0), (2, -1.0)]
    zb.zo_linear_prepare(z.ctx, 5, 1, 1.0, 2, -1.0, eps)
    for i, (m, n, _) in enumerate(spec):
        for T in tokens:
            X = _tokens(T, n, 17 * T + i, gpu)
            ldy = (m + 7) // 8 * 8
            out = {}
            # 128x256, 256x256, 256x224 on single CTAs; 256 x (256, 240, 224, 192, 128) on SM pairs
            for tiling in _tilings(r):
                zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, tiling)
                Ybuf = torch.full((T, ldy), float("nan"), dtype=torch.bfloat16, device=gpu)
                zb.zo_linear_perturbed(z.ctx, i, X, Ybuf[:, :m])
                z.sync()
                assert zb.zo_linear_tiling(z.ctx) == tiling
                # the padding columns of Y's rows are not written
                assert torch.isnan(Ybuf[:, m:].float()).all()
                out[tiling] = Ybuf[:, :m]
            # the tilings of one family sum each output in the same order: the single-CTA
            # ones take S from the split-K S kernel, the SM-pair ones from their own S tiles
            # (K ranges of 64-element panels, the same for every pair tiling), so the two
            # families may differ in S's last bits
            for tiling in _tilings(r):
                ref = 2 if tiling <= 3 else 6
                assert torch.equal(out[tiling].view(torch.int16), out[ref].view(torch.int16)), tiling
            C = subzero.perturb_coeff(z.seed, base + i, 5, r, terms, f32(eps))
            zc = abs(f32(eps)) * 2.0
            for Y in [out[k] for k in (3, 6) if k in out]:
                want = _check(Y, X, before["W"][i], before["U"][i], before["V"][i], C, zc,
                              f"{case} matrix {i} T={T} eps={eps}")
            if eps == 1e-1:
                # the perturbation is visible: most outputs differ from the plain layer's
                plain = rounding.round_to_bf16(to_f64(X) @ before["W"][i].T)
                assert (plain != want).mean() > 0.5
    if r > 32:
        # the single-CTA tilings take r <= 32; the automatic choice is an SM-pair one
        m, n, _ = spec[0]
        X = _tokens(8, n, 1, gpu)
        Y = torch.empty((8, m), dtype=torch.bfloat16, device=gpu)
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, 2)
        with pytest.raises(RuntimeError):
            zb.zo_linear_perturbed(z.ctx, 0, X, Y)
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, 0)
        zb.zo_linear_perturbed(z.ctx, 0, X, Y)
        z.sync()
        assert zb.zo_linear_tiling(z.ctx) >= 4
    for W, Wb in zip(z.weights, W_bits):
        assert torch.equal(W.view(torch.int16), Wb.view(torch.int16))
    z.close()


def test_perturbed_linear_single_query_and_repeat(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    z, base = _context(gpu, "r32", seed=99)
    r, spec, _ = LINEAR_CASES["r32"]
    m, n, _ = spec[1]
    X = _tokens(64, n, 3, gpu)
    Y1 = torch.empty((64, m), dtype=torch.bfloat16, device=gpu)
    Y2 = torch.empty_like(Y1)
    zb.zo_linear_prepare(z.ctx, 0, 3, -2.0, -1, 0.0, 1e-2)
    # a weight pass after the prepare rewrites W and the pass's own C / P workspace; the
    # prepared coefficient stays, and the layer sees the new W
    z.perturb(7, 0, 1.0, -1, 0.0, 1e-3)
    z.sync()
    before = snapshot(z)
    zb.zo_linear_perturbed(z.ctx, 1, X, Y1)
    zb.zo_linear_perturbed(z.ctx, 1, X, Y2)
    z.sync()
    assert torch.equal(Y1.view(torch.int16), Y2.view(torch.int16))   # deterministic
    assert zb.zo_linear_tiling(z.ctx) >= 4        # the automatic choice runs on SM pairs
    C = subzero.perturb_coeff(z.seed, base + 1, 0, r, [(3, -2.0)], f32(1e-2))
    _check(Y1, X, before["W"][1], before["U"][1], before["V"][1], C, 2.0 * f32(1e-2),
           "single query")
    z.close()


def test_perturbed_linear_back_to_back_calls_read_each_others_output(lib, gpu):
    """Two calls on the context's stream with no synchronisation between them, the second
    reading the first's Y as its X: each pair launch starts as a programmatic dependent of
    the stream's previous kernel and must wait for it before touching memory.  Y1 starts
    as NaN, so a second launch that read it early would not match the oracle."""
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    base = 5
    w = [make_weight(520, 520, "bf16", 910, gpu)]
    z = SubZeroPlus(w, 32, 4, 77, matrix_index_base=base)
    z.init_subspace(0)
    zb.zo_linear_prepare(z.ctx, 2, 3, 1.0, -1, 0.0, 1e-2)
    before = snapshot(z)
    C = subzero.perturb_coeff(z.seed, base, 2, 32, [(3, 1.0)], f32(1e-2))
    X = _tokens(600, 520, 8, gpu)
    Y1 = torch.full((600, 520), float("nan"), dtype=torch.bfloat16, device=gpu)
    Y2 = torch.empty_like(Y1)
    torch.cuda.synchronize()
    for _ in range(3):
        zb.zo_linear_perturbed(z.ctx, 0, X, Y1)
        zb.zo_linear_perturbed(z.ctx, 0, Y1, Y2)
        z.sync()
        assert torch.isfinite(Y2.float()).all()
        _check(Y1, X, before["W"][0], before["U"][0], before["V"][0], C, 2.0 * f32(1e-2), "first")
        _check(Y2, Y1, before["W"][0], before["U"][0], before["V"][0], C, 2.0 * f32(1e-2),
               "second, reading the first's output")
        Y1.fill_(float("nan"))
        torch.cuda.synchronize()
    z.close()


def test_perturbed_linear_long_token_block(lib, gpu):
    """S = X P^T's three ways to S_HL: 257 and 300 tokens split K over many ranges (a
    separate reduction kernel); 5000 tokens (40 row blocks) over 3 ranges, which the S
    kernel sums itself through its per-group counters; 19500 tokens (more row blocks than
    SMs) not at all, the epilogue writing S_HL directly while CTAs take several tiles.
    The calls run in turn on one context, so the counters must come back to zero."""
    from paper_2608_15665_gb300 import binding as zb
    z, base = _context(gpu, "r16", seed=2024)
    r, spec, _ = LINEAR_CASES["r16"]
    m, n, _ = spec[2]
    zb.zo_linear_prepare(z.ctx, 2, 0, 1.0, 3, -0.5, 1e-2)
    before = snapshot(z)
    C = subzero.perturb_coeff(z.seed, base + 2, 2, r, [(0, 1.0), (3, -0.5)], f32(1e-2))
    for T in (257, 5000, 19500, 5000, 300):
        X = _tokens(T, n, T, gpu)
        Y = torch.empty((T, m), dtype=torch.bfloat16, device=gpu)
        zb.zo_linear_perturbed(z.ctx, 2, X, Y)
        z.sync()
        _check(Y, X, before["W"][2], before["U"][2], before["V"][2], C, 2.0 * f32(1e-2),
               f"long token block T={T}")
    z.close()


def test_perturbed_linear_rejections(lib, gpu):
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    z, _ = _context(gpu, "r32", seed=5)
    X = _tokens(8, 520, 1, gpu)
    Y = torch.empty((8, 304), dtype=torch.bfloat16, device=gpu)
    with pytest.raises(RuntimeError):
        zb.zo_linear_perturbed(z.ctx, 0, X, Y)                                     # not prepared
    with pytest.raises(RuntimeError):
        zb.zo_linear_prepare(z.ctx, 0, 4, 1.0, -1, 0.0, 1e-3)                      # query 4 of 4
    zb.zo_linear_prepare(z.ctx, 0, 0, 1.0, -1, 0.0, 1e-3)
    with pytest.raises(RuntimeError):
        zb.zo_linear_perturbed(z.ctx, 3, X, Y)                                     # no matrix 3
    with pytest.raises(RuntimeError):
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, 9)                       # no tiling 9
    z.refresh(1)                                                                   # new U, V
    with pytest.raises(RuntimeError):
        zb.zo_linear_perturbed(z.ctx, 0, X, Y)                                     # stale P
    zb.zo_linear_prepare(z.ctx, 0, 0, 1.0, -1, 0.0, 1e-3)
    Ybad = torch.empty((8, 312), dtype=torch.bfloat16, device=gpu)[:, 1:305]       # misaligned
    with pytest.raises(RuntimeError):
        zb.zo_linear_perturbed(z.ctx, 0, X, Ybad)
    z.close()
    # an output width that is not a multiple of 8 (TMA stores write 16-byte chunks)
    w = [make_weight(300, 520, "bf16", 2, gpu)]
    zo = SubZeroPlus(w, 32, 4, 1)
    zo.init_subspace(0)
    zb.zo_linear_prepare(zo.ctx, 0, 0, 1.0, -1, 0.0, 1e-3)
    with pytest.raises(RuntimeError):
        zb.zo_linear_perturbed(zo.ctx, 0, X, Y[:, :300])
    zo.close()
    w = [make_weight(304, 520, "f32", 1, gpu)]
    zf = SubZeroPlus(w, 32, 4, 1)
    zf.init_subspace(0)
    with pytest.raises(RuntimeError):                                             # FMA path
        zb.zo_linear_prepare(zf.ctx, 0, 0, 1.0, -1, 0.0, 1e-3)
    zf.close()


@pytest.mark.parametrize("scheme,case", [("central", "r32"), ("forward", "r32"),
                                         ("central", "r128")])
def test_linear_route_step_matches_oracle(lib, gpu, scheme, case):
    """One whole Alg. 3 step on the perturbed-linear route (SubZeroPlus.run_step_linear):
    every loss comes from zo_linear_perturbed outputs while W stays as it is; each
    evaluation's Y matches the oracle's layer, element by element, at the point the scheme
    defines (Eq. (3): W + eps Z_k, W - eps Z_k; Eq. (6): W, then W + eps Z_k; eps large
    enough that most outputs move); and zo_step (nothing to restore) leaves W and the
    moments at the oracle's single update from the losses."""
    from gpu_util import oracle_step
    from parity import assert_moments, assert_weights, gabs
    z, base = _context(gpu, case, seed=777)
    r, spec, _ = LINEAR_CASES[case]
    eps, lr, b1, b2, ea, t = 0.5, 1e-3, 0.9, 0.95, 1e-8, 3
    T = 48
    X = [_tokens(T, n, 100 + i, gpu) for i, (m, n, _) in enumerate(spec)]
    gw = [torch.randn(T, m, generator=torch.Generator().manual_seed(200 + i)).double().numpy()
          for i, (m, n, _) in enumerate(spec)]
    if scheme == "central":
        points = [(k, c) for k in range(z.q) for c in (1.0, -1.0)]
    else:
        points = [(0, 0.0)] + [(k, 1.0) for k in range(z.q)]
    before = snapshot(z)
    W_bits = [W.detach().clone() for W in z.weights]

    def loss_fn(t_, idx):
        for W, Wb in zip(z.weights, W_bits):           # the evaluations never write W
            assert torch.equal(W.view(torch.int16), Wb.view(torch.int16))
        k, c = points[idx]
        loss = 2.0
        for i in range(len(spec)):
            Y = z.linear_perturbed(i, X[i])
            z.sync()
            # element by element at the point the scheme defines (the bound of _check)
            C = subzero.perturb_coeff(z.seed, base + i, t_, r, [(k, c)], f32(eps))
            want = _check(Y, X[i], before["W"][i], before["U"][i], before["V"][i], C,
                          abs(f32(eps) * c), f"{scheme} evaluation {idx}, matrix {i}")
            if c != 0.0:                                # the perturbation is visible
                plain = rounding.round_to_bf16(to_f64(X[i]) @ before["W"][i].T)
                assert (plain != want).mean() > 0.5
            loss += float((to_f64(Y) * gw[i]).mean())
        return loss

    losses = z.run_step_linear(t, 1, loss_fn, scheme, eps, lr, b1, b2, ea)
    assert len(losses) == len(points)
    after = snapshot(z)
    z.sync()
    rho = subzero.rho_from_losses(np.asarray(losses, np.float32), scheme, f32(eps), z.q)
    for i in range(len(spec)):
        Wo, Mo, Vmo, G, Tm = oracle_step(before, i, "bf16", z.seed, base + i, t, r, z.q, losses,
                                         scheme, eps, lr, b1, b2, ea, 1, [])
        assert_moments(after["M"][i], after["Vm"][i], Mo, Vmo, before["M"][i], before["Vm"][i],
                       gabs(z.seed, base + i, t, r, rho), b1, b2, f"linear route {i}")
        assert_weights(after["W"][i], Wo, "bf16", f"linear-route step, matrix {i}",
                       before=before["W"][i], terms=Tm)
    z.close()
