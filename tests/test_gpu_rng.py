"""GPU parity of the counter-based random contract (bit-exact integers, fp32 normals)."""

import numpy as np
import pytest
import torch

from oracle import rng
from parity import NORMAL_ABS

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed,x1,x2,x3,n", [
    (0, 0, 0, 0, 4099),
    ((7 << 32) | 123, 5, 9, (1 << 24) | 3, 100_003),
    (2 ** 64 - 1, 2 ** 32 - 1, 2 ** 32 - 1, 2 ** 32 - 1, 1021),
    (1003, 17, 25, 2 << 24, 1_000_000),
])
def test_philox_stream_is_bit_exact(lib, gpu, seed, x1, x2, x3, n):
    out = torch.zeros(n, dtype=torch.int32, device=gpu)
    lib.zo_philox_fill(seed, x1, x2, x3, out)
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint32).astype(np.uint64)
    assert np.array_equal(got, rng.philox_block(seed, x1, x2, x3, n))


def test_philox_known_answer_on_device(lib, gpu, golden):
    row = [int(x, 16) for x in golden("philox4x32_10_kat.txt")[0]]
    assert row[:6] == [0] * 6
    out = torch.zeros(4, dtype=torch.int32, device=gpu)
    lib.zo_philox_fill(0, 0, 0, 0, out)
    assert [int(v) for v in out.cpu().numpy().view(np.uint32)] == row[6:10]


@pytest.mark.parametrize("n", [1, 3, 4, 4097, 1_000_003])
def test_normals_match_oracle(lib, gpu, n):
    x3 = rng.query_counter_word(rng.TAG_Z, 2)
    out = torch.zeros(n, dtype=torch.float32, device=gpu)
    lib.zo_normal_fill(2026, 3, 7, x3, out)
    got = out.cpu().double().numpy()
    want = rng.normals(2026, 3, 7, x3, n)
    assert np.max(np.abs(got - want)) <= NORMAL_ABS


def test_perturbation_and_omega_streams(lib, gpu):
    # Z_i^(k) at step t and Omega_U at refresh j, addressed exactly as the kernels do
    r = 16
    out = torch.zeros(r * r, dtype=torch.float32, device=gpu)
    lib.zo_normal_fill(99, 4, 11, rng.query_counter_word(rng.TAG_Z, 5), out)
    assert np.max(np.abs(out.cpu().double().numpy().reshape(r, r) - rng.gen_Z(99, 4, 11, 5, r))) <= NORMAL_ABS
    out = torch.zeros(300 * r, dtype=torch.float32, device=gpu)
    lib.zo_normal_fill(99, 4, 2, rng.query_counter_word(rng.TAG_OMEGA_U, 0), out)
    want = rng.gen_omega(99, 4, 2, "U", 300, r)
    assert np.max(np.abs(out.cpu().double().numpy().reshape(300, r) - want)) <= NORMAL_ABS
