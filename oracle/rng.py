"""Counter-based Gaussian contract of the oracle (test infrastructure only).

The paper draws every random matrix from a seed: Alg. 2 reseeds the generator
and then draws i.i.d. N(0,1) entries for Z_i; Alg. 3 takes a fresh seed for each
query of each step; App. A.1 keeps only the seeds and regenerates each Z when
needed; Alg. 1 draws the Gaussian Omega_U, Omega_V.  The paper does not say which generator.  The
contract fixed here (and implemented independently by the CUDA library) is:

* generator: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random
  numbers: as easy as 1, 2, 3", SC'11): a 4x32-bit counter, a 2x32-bit key,
  ten rounds of two 32x32->64 multiplies with a Weyl key schedule.
* key    = (seed mod 2^32, seed div 2^32)
* counter= (c, matrix index i, step t or refresh index j (mod 2^32),
            tag << 24 | query k)
  tag 1 = Z (perturbation), 2 = Omega_U, 3 = Omega_V.
* element e of a row-major buffer takes counter word c = e // 4, lane e % 4.
* uniform   u = ((x >> 8) + 1) * 2^-24  in (0, 1]  (exact in fp32 and fp64)
* Box-Muller: lanes (0,1) and (2,3) are pairs (u_a, u_b);
  rad = sqrt(-2 ln u_a); z_a = rad cos(2 pi u_b); z_b = rad sin(2 pi u_b).

Parity: the integer stream is bit-exact between the two sides; the normals
differ only by the fp32 rounding of log/sqrt/sin/cos on the GPU.
"""

import numpy as np

# Philox4x32 round multipliers and Weyl key increments (Salmon et al. 2011).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
MASK32 = 0xFFFFFFFF

TAG_Z = 1
TAG_OMEGA_U = 2
TAG_OMEGA_V = 3


def _u32(a):
    return np.asarray(a, dtype=np.uint64) & np.uint64(MASK32)


def philox4x32_10(ctr, key):
    """Philox4x32 with 10 rounds.

    ctr: array (..., 4) of uint32-valued integers; key: array (..., 2).
    Returns an array (..., 4) of uint64 holding the 32-bit outputs.

    One round maps (x0, x1, x2, x3) with key (k0, k1) to
      (hi(M1*x2) ^ x1 ^ k0,  lo(M1*x2),  hi(M0*x0) ^ x3 ^ k1,  lo(M0*x0)),
    and the key is bumped by (W0, W1) between rounds.
    """
    ctr = _u32(ctr)
    key = _u32(key)
    x0, x1, x2, x3 = (ctr[..., 0], ctr[..., 1], ctr[..., 2], ctr[..., 3])
    k0, k1 = key[..., 0], key[..., 1]
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    s32 = np.uint64(32)
    msk = np.uint64(MASK32)
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + np.uint64(PHILOX_W0)) & msk
            k1 = (k1 + np.uint64(PHILOX_W1)) & msk
        p0 = m0 * x0          # < 2^64: exact in uint64
        p1 = m1 * x2
        hi0, lo0 = p0 >> s32, p0 & msk
        hi1, lo1 = p1 >> s32, p1 & msk
        x0, x1, x2, x3 = hi1 ^ x1 ^ k0, lo1, hi0 ^ x3 ^ k1, lo0
    return np.stack([x0, x1, x2, x3], axis=-1)


def key_of_seed(seed):
    seed = int(seed)
    return (seed & MASK32, (seed >> 32) & MASK32)


def philox_block(seed, x1, x2, x3, n_words):
    """The uint32 words 0..n_words-1 of the stream (c = 0, 1, ...; 4 lanes each)."""
    n_ctr = (int(n_words) + 3) // 4
    c = np.arange(n_ctr, dtype=np.uint64)
    ctr = np.stack([c,
                    np.full(n_ctr, int(x1) & MASK32, dtype=np.uint64),
                    np.full(n_ctr, int(x2) & MASK32, dtype=np.uint64),
                    np.full(n_ctr, int(x3) & MASK32, dtype=np.uint64)], axis=-1)
    k0, k1 = key_of_seed(seed)
    key = np.broadcast_to(np.array([k0, k1], dtype=np.uint64), (n_ctr, 2))
    return philox4x32_10(ctr, key).reshape(-1)[:n_words]


def uniform_from_u32(x):
    """u = ((x >> 8) + 1) * 2^-24, in (0, 1]."""
    x = np.asarray(x, dtype=np.uint64)
    return ((x >> np.uint64(8)).astype(np.float64) + 1.0) * 2.0 ** -24


def normals(seed, x1, x2, x3, n):
    """n i.i.d. N(0,1) values (fp64) of the stream addressed by (x1, x2, x3)."""
    n = int(n)
    n4 = (n + 3) // 4 * 4
    words = philox_block(seed, x1, x2, x3, n4).reshape(-1, 4)
    u = uniform_from_u32(words)
    out = np.empty_like(u)
    for a, b in ((0, 1), (2, 3)):
        rad = np.sqrt(-2.0 * np.log(u[:, a]))
        ang = 2.0 * np.pi * u[:, b]
        out[:, a] = rad * np.cos(ang)
        out[:, b] = rad * np.sin(ang)
    return out.reshape(-1)[:n]


def query_counter_word(tag, k):
    return ((int(tag) & 0xFF) << 24) | (int(k) & 0xFFFFFF)


def gen_Z(seed, i, t, k, r):
    """Z_i^(k) at step t: r x r, row-major, i.i.d. N(0,1) (Eq. (4), Alg. 2)."""
    z = normals(seed, i, t, query_counter_word(TAG_Z, k), r * r)
    return z.reshape(r, r)


def gen_omega(seed, i, j, which, rows, r):
    """Omega_U (which='U', m x r) or Omega_V (which='V', n x r) at refresh j (Alg. 1)."""
    tag = TAG_OMEGA_U if which == "U" else TAG_OMEGA_V
    w = normals(seed, i, j, query_counter_word(tag, 0), rows * r)
    return w.reshape(rows, r)
