"""Pins of the oracle's counter-based Gaussian contract (no GPU)."""

import numpy as np
import pytest
from scipy import stats

from oracle import rng


def test_philox_known_answers(golden):
    rows = golden("philox4x32_10_kat.txt")
    assert len(rows) == 3
    for row in rows:
        v = [int(x, 16) for x in row]
        ctr, key, want = v[0:4], v[4:6], v[6:10]
        out = rng.philox4x32_10(np.array([ctr], np.uint64), np.array([key], np.uint64))[0]
        assert [int(x) for x in out] == want


def test_philox_block_layout_matches_single_calls():
    seed = (7 << 32) | 123
    words = rng.philox_block(seed, 5, 9, rng.query_counter_word(rng.TAG_Z, 3), 4 * 6)
    for c in range(6):
        one = rng.philox4x32_10(np.array([[c, 5, 9, (1 << 24) | 3]], np.uint64),
                                np.array([[123, 7]], np.uint64))[0]
        assert [int(x) for x in words[4 * c:4 * c + 4]] == [int(x) for x in one]


def test_uniform_exact_and_in_range():
    x = np.array([0, 255, 256, 0x7FFFFFFF, 0xFFFFFF00, 0xFFFFFFFF], np.uint64)
    u = rng.uniform_from_u32(x)
    assert u[0] == 2.0 ** -24 and u[1] == 2.0 ** -24 and u[2] == 2.0 ** -23
    assert u[4] == 1.0 and u[5] == 1.0
    # every value is exactly representable in fp32
    xs = rng.philox_block(1, 2, 3, 4, 1 << 16)
    us = rng.uniform_from_u32(xs)
    assert np.all(us.astype(np.float32).astype(np.float64) == us)
    assert np.all((us > 0) & (us <= 1))


def test_normals_moments_and_ks():
    z = rng.normals(2026, 1, 2, 3, 1_000_000)
    n = z.size
    assert abs(z.mean()) < 5 / np.sqrt(n)
    assert abs(z.var() - 1.0) < 5 * np.sqrt(2.0 / n)
    assert abs(np.mean(z ** 4) - 3.0) < 5 * np.sqrt(96.0 / n)
    assert stats.kstest(z, "norm").pvalue > 1e-3
    # the four lanes of one counter are uncorrelated
    lanes = z[: n // 4 * 4].reshape(-1, 4)
    c = np.corrcoef(lanes.T)
    assert np.max(np.abs(c - np.eye(4))) < 5 / np.sqrt(lanes.shape[0])


def test_box_muller_pairs_follow_the_definition():
    words = rng.philox_block(99, 0, 0, 0, 8).reshape(-1, 4)
    u = rng.uniform_from_u32(words)
    z = rng.normals(99, 0, 0, 0, 8).reshape(-1, 4)
    rad = np.sqrt(-2 * np.log(u[:, 0]))
    assert np.allclose(z[:, 0], rad * np.cos(2 * np.pi * u[:, 1]), rtol=0, atol=1e-15)
    assert np.allclose(z[:, 1], rad * np.sin(2 * np.pi * u[:, 1]), rtol=0, atol=1e-15)
    # radius of each pair is sqrt(-2 ln u_a)
    rad2 = np.sqrt(-2 * np.log(u[:, 2]))
    assert np.allclose(np.hypot(z[:, 2], z[:, 3]), rad2, rtol=1e-14)


def test_counter_fields_select_independent_streams():
    base = rng.gen_Z(5, 0, 0, 0, 8)
    for args in [(5, 1, 0, 0), (5, 0, 1, 0), (5, 0, 0, 1), (6, 0, 0, 0)]:
        other = rng.gen_Z(*args, 8)
        assert not np.allclose(base, other)
    # Omega_U and Omega_V of the same (matrix, refresh) differ, and a prefix of
    # a longer Omega is the shorter one (row-major element addressing)
    ou = rng.gen_omega(5, 3, 1, "U", 10, 4)
    ov = rng.gen_omega(5, 3, 1, "V", 10, 4)
    assert not np.allclose(ou, ov)
    assert np.array_equal(rng.gen_omega(5, 3, 1, "U", 6, 4), ou[:6])


@pytest.mark.parametrize("seed", [0, 1, (1 << 40) + 17])
def test_seed_splits_into_key_words(seed):
    k0, k1 = rng.key_of_seed(seed)
    assert k0 == seed & 0xFFFFFFFF and k1 == seed >> 32
