"""Pins for the oracle's random streams: Philox4x32-10 against cuRAND's host
generator (a library, run on the CPU), the word->uniform map, Box-Muller
normals against the normal distribution, the reset polynomials against numpy's
sine and cosine, and bf16 rounding against torch's conversion."""
import ctypes
import glob
import math
import os

import numpy as np
import pytest


def _curand():
    cands = []
    for root in ("/usr/local/cuda/lib64", "/usr/local/cuda/targets/sbsa-linux/lib",
                 "/usr/local/cuda/targets/x86_64-linux/lib"):
        cands += sorted(glob.glob(os.path.join(root, "libcurand.so*")))
    for c in cands:
        try:
            return ctypes.CDLL(c)
        except OSError:
            continue
    return None


def _curand_philox_stream(seed: int, n_words: int) -> np.ndarray:
    lib = _curand()
    if lib is None:
        pytest.skip("libcurand not found")
    gen = ctypes.c_void_p()
    CURAND_RNG_PSEUDO_PHILOX4_32_10 = 161  # curand.h enum value
    assert lib.curandCreateGeneratorHost(ctypes.byref(gen), CURAND_RNG_PSEUDO_PHILOX4_32_10) == 0
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        out = np.zeros(n_words, dtype=np.uint32)
        assert lib.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p),
                                  ctypes.c_size_t(n_words)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    return out


@pytest.mark.parametrize("seed", [0, 1234, 0x123456789ABC, 0xFFFFFFFFFFFFFFFF])
def test_philox_matches_curand_host_generator(oracle, seed):
    """cuRAND's host Philox4_32_10 generator emits block j as
    Philox(key = (seed lo, seed hi), counter = (j / 65536, 0, j % 65536, 0)).
    Checking blocks across both counter words the layout touches and both key
    words pins the round function, the multipliers and the key schedule."""
    n_blocks = 65536 + 300
    stream = _curand_philox_stream(seed, 4 * n_blocks).reshape(-1, 4)
    k0, k1 = seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF
    rng = np.random.default_rng(5)
    blocks = list(range(0, 40)) + list(rng.integers(0, n_blocks, 200)) + [65535, 65536, 65537]
    for j in blocks:
        ctr = [j // 65536, 0, j % 65536, 0]
        got = oracle.philox(k0, k1, ctr)
        assert np.array_equal(got, stream[j]), (j, got, stream[j])


def test_philox_counter_words_are_all_live(oracle):
    """Every counter word and key word changes the output (no word dropped)."""
    base = oracle.philox(3, 5, [7, 11, 13, 17])
    for w in range(4):
        c = [7, 11, 13, 17]
        c[w] ^= 1
        assert not np.array_equal(oracle.philox(3, 5, c), base)
    assert not np.array_equal(oracle.philox(2, 5, [7, 11, 13, 17]), base)
    assert not np.array_equal(oracle.philox(3, 4, [7, 11, 13, 17]), base)


def test_word_to_uniform_exact_endpoints(oracle):
    L = oracle.lib()
    assert L.oracle_word_to_uniform(0) == 2.0 ** -24
    assert L.oracle_word_to_uniform(0xFFFFFFFF) == 1.0 - 2.0 ** -24
    assert L.oracle_word_to_uniform(0x80000000) == 0.5 + 2.0 ** -24
    # 512 consecutive words share one cell (top 23 bits)
    assert L.oracle_word_to_uniform(0x1FF) == L.oracle_word_to_uniform(0)
    assert L.oracle_word_to_uniform(0x200) == 3 * 2.0 ** -24


def test_box_muller_normals_distribution(oracle):
    """Normals drawn for 4000 (env, step) pairs (32000 samples): mean 0, var 1,
    Kolmogorov-Smirnov against N(0, 1), no correlation between paired outputs."""
    stats = pytest.importorskip("scipy.stats")
    eps = np.array([oracle.normals(e, 0, t) for e in range(40) for t in range(100)])
    x = eps.reshape(-1)
    assert abs(x.mean()) < 0.03
    assert abs(x.var() - 1.0) < 0.04
    assert stats.kstest(x, "norm").pvalue > 1e-3
    c = np.corrcoef(eps[:, 0], eps[:, 1])[0, 1]
    assert abs(c) < 0.05
    # independent streams for different seeds and steps
    assert not np.allclose(oracle.normals(0, 0, 0), oracle.normals(0, 1, 0))
    assert not np.allclose(oracle.normals(0, 0, 0), oracle.normals(0, 0, 1))


def test_box_muller_pair_radius(oracle):
    """Each pair (eps_2k, eps_2k+1) has radius^2 = -2 ln u_2k, with u from the
    action stream (counter word 2 = 0)."""
    L = oracle.lib()
    env, seed, t_g = 17, 3, (1 << 33) + 5
    eps = oracle.normals(env, seed, t_g)
    words = np.concatenate([oracle.philox(env, seed, [t_g & 0xFFFFFFFF, t_g >> 32, 0, b])
                            for b in range(2)])
    u = np.array([L.oracle_word_to_uniform(int(w)) for w in words], dtype=np.float64)
    for k in range(4):
        r2 = eps[2 * k] ** 2 + eps[2 * k + 1] ** 2
        assert math.isclose(r2, -2 * math.log(u[2 * k]), rel_tol=1e-12)
        ang = math.atan2(eps[2 * k + 1], eps[2 * k]) % (2 * math.pi)
        assert math.isclose(ang, (2 * math.pi * u[2 * k + 1]) % (2 * math.pi), abs_tol=1e-9)


def test_taylor_half_angle_polynomials(oracle):
    """Reset sine/cosine polynomials on [-pi/2, pi/2] (the widest half-angle
    drawn): sine within 4 ulps of the true value; cosine within 2 ulps of 1.0
    absolute (its Horner sum of O(1) terms cancels near pi/2)."""
    L = oracle.lib()
    xs = np.linspace(-math.pi / 2, math.pi / 2, 2001).astype(np.float32)
    for x in xs:
        s = L.oracle_taylor_sin(float(x))
        c = L.oracle_taylor_cos(float(x))
        ulp_s = np.spacing(np.float32(abs(math.sin(float(x))) + 1e-30))
        ulp_c = np.spacing(np.float32(abs(math.cos(float(x)))))
        assert abs(s - math.sin(float(x))) <= 4 * ulp_s + 1e-30
        assert abs(c - math.cos(float(x))) <= 4 * ulp_c + 2 * 1.2e-7


def test_bf16_rounding_matches_torch(oracle):
    torch = pytest.importorskip("torch")
    L = oracle.lib()
    rng = np.random.default_rng(0)
    xs = np.concatenate([rng.standard_normal(3000).astype(np.float32),
                         (rng.standard_normal(1000) * 1e-3).astype(np.float32)])
    # exact ties: bf16 value + half ulp, both parities
    ties = []
    for base in (1.0, 1.0078125, -3.0, 0.5 + 2 ** -8):
        b = np.float32(base)
        ulp = np.float32(2.0 ** (math.floor(math.log2(abs(base))) - 7))
        ties.append(np.float32(b + ulp / 2))
    xs = np.concatenate([xs, np.array(ties, dtype=np.float32), np.float32([0.0, -0.0])])
    ref = torch.from_numpy(xs).to(torch.bfloat16).to(torch.float32).numpy()
    got = np.array([L.oracle_to_bf16(float(x)) for x in xs], dtype=np.float32)
    assert np.array_equal(got, ref)


def test_bf16_rounding_of_double_is_single_rounding(oracle):
    """A double just below a bf16 tie rounds down even though it rounds to the
    tie in float (no double rounding)."""
    L = oracle.lib()
    tie = 1.0 + 2.0 ** -8          # halfway between 1 and 1 + 2^-7
    below = tie - 2.0 ** -40       # rounds to `tie` in float
    assert float(np.float32(below)) == tie
    assert L.oracle_to_bf16(below) == 1.0
    assert L.oracle_to_bf16(tie + 2.0 ** -40) == 1.0 + 2.0 ** -7
