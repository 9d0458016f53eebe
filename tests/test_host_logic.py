"""Host-side logic that needs no GPU: workload shapes, input generators, call plan."""

import numpy as np
import pytest

from oracle import subzero
from paper_2608_15665_gb300 import workloads


@pytest.mark.parametrize("name,params,n_mats,r,q", [
    ("single256_f32_r8", 65_536, 1, 8, 4),
    ("opt1.3b_bf16_r16", 1_207_959_552, 144, 16, 4),
    ("llama7b_bf16_r32", 6_476_005_376, 224, 32, 4),
    ("lora_opt13b_f32_r4", 6_553_600, 160, 4, 8),
    ("dense32b_bf16_r64", 31_205_621_760, 448, 64, 8),
    ("llama7b_bf16_r128_q99", 6_476_005_376, 224, 128, 99),
    ("llama13b_bf16_r128_q99", 12_687_769_600, 280, 128, 99),
])
def test_workload_shapes(name, params, n_mats, r, q):
    wl = workloads.get(name)
    assert wl.params == params and wl.n_mats == n_mats and wl.r == r and wl.q == q
    assert all(min(m, n) >= r for m, n in wl.shapes)


def test_bytes_per_pass_llama7b():
    wl = workloads.get("llama7b_bf16_r32")
    assert wl.bytes_per_pass() == 4 * 6_476_005_376


def test_loss_table_is_seeded_and_windowed():
    wl = workloads.get("single256_f32_r8")
    full = workloads.loss_table(wl, "central")
    assert full.shape == (10, 8) and full.dtype == np.float32
    assert np.array_equal(workloads.loss_table(wl, "central", steps=3, start=4), full[4:7])
    assert abs(full.mean() - 2.0) < 0.01 and 0.003 < full.std() < 0.03
    assert workloads.loss_table(wl, "forward").shape == (10, 5)


def test_init_weights_on_cpu():
    wl = workloads.get("lora_opt13b_f32_r4")
    A = workloads.init_weight(wl, 0)
    B = workloads.init_weight(wl, 1)
    assert A.shape == (8, 5120) and B.shape == (5120, 8)
    assert float(B.abs().max()) == 0.0 and 0.015 < float(A.std()) < 0.025


@pytest.mark.parametrize("q", [1, 3, 4, 8])
@pytest.mark.parametrize("scheme", ["central", "forward"])
def test_call_plan_matches_the_oracle_plan(lib, scheme, q):
    from paper_2608_15665_gb300.schedule import step_plan
    calls, restore = step_plan(scheme, q)
    passes, orestore = subzero.pass_plan(scheme, q)
    assert len(calls) == len(passes)
    for ((qa, ca), second), terms in zip(calls, passes):
        mine = [(qa, ca)] + ([second] if second is not None else [])
        assert sorted(mine) == sorted(terms)
    assert [restore] == orestore


@pytest.mark.parametrize("q", [1, 2, 5])
def test_linear_plan_visits_the_scheme_points(lib, q):
    # the perturbed-linear route evaluates each loss at an absolute point: Eq. (3) pairs
    # W + eps Z_k, W - eps Z_k; Eq. (6) W itself, then W + eps Z_k -- the same points the
    # weight-pass plan reaches by accumulating its passes
    from paper_2608_15665_gb300.schedule import linear_plan, step_plan
    for scheme in ("central", "forward"):
        pts = [(k, c) for (k, c), second in linear_plan(scheme, q) if second is None]
        assert len(pts) == len(linear_plan(scheme, q))
        calls, _ = step_plan(scheme, q)
        acc, visited = {}, [] if scheme == "central" else [{}]
        for (qa, ca), second in calls:
            for kk, cc in [(qa, ca)] + ([second] if second else []):
                acc[kk] = acc.get(kk, 0.0) + cc
            visited.append({k: c for k, c in acc.items() if c != 0.0})
        want = [{k: c} if c != 0.0 else {} for k, c in pts]
        assert visited == want, scheme
    with pytest.raises(ValueError):
        linear_plan("direct", q)
