"""The SM-pair perturbed-linear planner (linear_pair_plan / linear_pair_tiling in
zo_linear_pair.cu), built into a host probe with nvcc and run on the CPU: every plan it
makes for a grid of shapes, ranks and pair counts keeps the kernel's preconditions, and
its tile order, run as the kernel runs it (each pair's tiles in order; a Y tile's rank-r
step waits until all of its row block's S writers -- its S tiles or its contributor tiles'
K loops -- are done), finishes: no tile waits on one that can only start after it.  The
automatic tiling at the LLaMA-7B shapes is the one measured fastest (r = 32, 4096 tokens,
76 pairs: 256 x 240 for all three)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_15665_gb300", "csrc")


def _cd(a, b):
    return -(-a // b)


@pytest.fixture(scope="module")
def plans(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not available")
    d = tmp_path_factory.mktemp("plan")
    exe = str(d / "probe")
    cmd = [nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-std=c++17",
           "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include"), "-I", CSRC,
           os.path.join(ROOT, "tests", "harness", "linear_plan_probe.cu"),
           os.path.join(CSRC, "zo_linear_pair.cu"), "-o", exe]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    rows = []
    for line in out.splitlines():
        v = [int(x) for x in line.split()]
        rows.append(dict(zip(["T", "m", "n", "r", "np", "tiling", "N", "pairs", "group",
                              "nc", "sc", "ss", "ch", "auto"], v)))
    return rows


def _decode(t, n_s, rb, tn, group):
    """The kernel's tile order: S tiles first (row block t % rb), then the Y tiles in
    column stripes of `group` column blocks (the kernel clamps group to [1, tiles_n])."""
    if t < n_s:
        return t % rb, t // rb, True
    j = t - n_s
    g = tn if (group < 1 or group > tn) else group
    per, full = rb * g, tn // g
    if j < full * per:
        return (j % per) // g, (j // per) * g + (j % per) % g, False
    rem, last = j - full * per, tn - full * g
    return rem // last, full * g + rem % last, False


def _finishes(p):
    rb, tn = _cd(p["T"], 256), _cd(p["m"], p["N"])
    n_s = rb * p["ss"]
    total = n_s + rb * tn
    P = p["pairs"]
    order = [_decode(t, n_s, rb, tn, p["group"]) for t in range(total)]
    queues = [list(range(q, total, P)) for q in range(P)]
    pos, k_done = [0] * P, [False] * P
    writers = {}                       # row block -> S writers done (S tiles or contributors)
    need = p["ss"] if p["nc"] == 0 else min(p["nc"], tn)
    progress = True
    while progress:
        progress = False
        for q in range(P):
            if pos[q] >= len(queues[q]):
                continue
            tb, nb, s_tile = order[queues[q][pos[q]]]
            if s_tile:
                writers[tb] = writers.get(tb, 0) + 1
                pos[q] += 1
                progress = True
                continue
            if not k_done[q]:
                if nb < p["nc"]:
                    writers[tb] = writers.get(tb, 0) + 1
                k_done[q] = True
                progress = True
            if writers.get(tb, 0) >= need:
                pos[q] += 1
                k_done[q] = False
                progress = True
    return all(pos[q] >= len(queues[q]) for q in range(P))


def test_every_plan_keeps_the_kernels_preconditions(plans):
    assert plans
    for p in plans:
        assert 1 <= p["pairs"] <= p["np"], p
        assert 4 <= p["auto"] <= 8, p
        panels = _cd(p["n"], 64)
        if p["nc"]:
            # contributors: r <= 64, slices of 16 or 32 rows per CTA within the spare TMEM
            # columns, aligned TMEM reads, <= 32 ready flags, consecutive in stripe 0
            assert p["r"] <= 64 and p["ss"] == 0, p
            assert p["nc"] in (1, 2, 4) and p["sc"] in (32, 64), p
            assert p["sc"] * p["nc"] == 2 * p["r"], p
            assert p["sc"] // 2 <= min(32, (256 - p["N"]) // 2), p
            assert (p["N"] // 2) % (p["sc"] // 2) == 0, p
            assert p["nc"] <= _cd(p["m"], p["N"]) and p["group"] % p["nc"] == 0, p
        else:
            assert 1 <= p["ss"] <= 15 and p["ch"] >= 1, p
            assert (p["ss"] - 1) * p["ch"] < panels <= p["ss"] * p["ch"], p   # no empty range
            if p["r"] <= 64:
                assert p["ss"] == 1, p      # one K range: S summed like the contributors'


def test_every_plans_tile_order_finishes(plans):
    # the small token counts cover the waits; the large ones only the order's arithmetic
    checked = 0
    for p in plans:
        if _cd(p["T"], 256) * (_cd(p["m"], p["N"]) + p["ss"]) > 4000:
            continue
        assert _finishes(p), p
        checked += 1
    assert checked > 1000


def test_automatic_tiling_at_the_llama7b_shapes(plans):
    want = {(4096, 4096): 5, (11008, 4096): 5, (4096, 11008): 5}
    got = {(p["m"], p["n"]): p["auto"] for p in plans
           if p["T"] == 4096 and p["r"] == 32 and p["np"] == 76 and (p["m"], p["n"]) in want}
    assert got == want
