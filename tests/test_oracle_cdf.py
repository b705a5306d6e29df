"""Pins of the oracle's integer CDF (the coder input of the Torchac-based coder, Sec. 5.1; the
paper does not say how probabilities were made integer, so the quantiser is a reading pinned by
exact table checks, closed forms, invariants and agreement with the softmax it approximates)."""
import math

import numpy as np
import pytest

import oracle as O
from oracle import gen_exp2_tables


def test_exp2_tables_exact():
    H, L = O.exp2_tables()
    gH, gL = gen_exp2_tables.tables()  # exact big-integer bracketing and an independent series
    assert H.tolist() == gH and L.tolist() == gL
    # and against binary64 evaluation (every entry is far from a rounding tie)
    for i in range(256):
        assert H[i] == round(2 ** 31 * 2 ** (-i / 256))
        assert L[i] == round(2 ** 31 * 2 ** (-i / 65536))


def test_exp2_fixed_close_to_exp2():
    rng = np.random.default_rng(0)
    for a in list(range(0, 70000, 997)) + rng.integers(0, 40 * 65536, 3000).tolist():
        e = O.exp2_fixed(int(a))
        ref = 2 ** 31 * 2 ** (-a / 65536)
        # two rounded table entries and one rounded product: a few units of 2^-31 relative, plus
        # the final right shift's truncation
        assert abs(e - ref) <= ref * 2 ** -29 + 1.0, a
    assert O.exp2_fixed(0) == 2 ** 31
    assert O.exp2_fixed(40 * 65536) == 0
    assert O.exp2_fixed(10 ** 9) == 0  # clamped


def check_cdf(cdf, V, P):
    assert cdf.shape[-1] == V + 1
    assert np.all(cdf[..., 0] == 0) and np.all(cdf[..., -1] == 2 ** P)
    assert np.all(np.diff(cdf.astype(np.int64), axis=-1) >= 1)


@pytest.mark.parametrize("V,P", [(32, 16), (1000, 20), (32000, 24)])
def test_invariants_random_rows(V, P):
    rng = np.random.default_rng(V)
    z = (rng.normal(size=(6, V)) * rng.uniform(0.1, 8, size=(6, 1))).astype(np.float32)
    cdf = O.quantize_cdf(z, P)
    check_cdf(cdf, V, P)
    # the quantised probabilities follow the softmax: the floor of 1 per symbol and the
    # floor/residual rounding cost at most (V + 1) / T of mass each; exp2 error 2^-28 relative
    T = 2.0 ** P
    zz = z.astype(np.float64)
    sm = np.exp(zz - zz.max(1, keepdims=True))
    sm /= sm.sum(1, keepdims=True)
    q = np.diff(cdf.astype(np.int64), axis=1) / T
    assert np.max(np.abs(q - sm * (T - V) / T - 1 / T)) <= (V + 2) / T + 1e-6


def test_uniform_closed_form():
    cdf = O.quantize_cdf(np.zeros((1, 32), np.float32), 16)[0]
    assert cdf.tolist() == [2048 * j for j in range(33)]
    cdf = O.quantize_cdf(np.full((1, 32), -3.25, np.float32), 16)[0]
    assert cdf.tolist() == [2048 * j for j in range(33)]


def test_one_hot_dominant():
    for V, P, hot in [(32, 16, 7), (32000, 24, 31999), (100, 12, 0)]:
        z = np.zeros(V, np.float32)
        z[hot] = 100.0
        f = np.diff(O.quantize_cdf(z, P)[0].astype(np.int64))
        assert f[hot] == 2 ** P - V + 1
        assert np.all(np.delete(f, hot) == 1)


def test_shift_invariance_integer_logits():
    rng = np.random.default_rng(9)
    z = rng.integers(-20, 20, size=(5, 500)).astype(np.float32)
    a = O.quantize_cdf(z, 20)
    b = O.quantize_cdf(z + np.float32(1024.0), 20)
    assert np.array_equal(a, b)


def test_residual_goes_to_lowest_argmax():
    z = np.zeros(5, np.float32)
    z[1] = z[3] = 2.0
    f = np.diff(O.quantize_cdf(z, 10)[0].astype(np.int64))
    e = [O.exp2_fixed(int(-np.rint(np.float32(np.float32(v - 2.0) * np.float32(65536 * math.log2(math.e))))))
         for v in z]
    S = sum(e)
    M = 1024 - 5
    g = [ei * M // S for ei in e]
    resid = M - sum(g)
    assert resid > 0
    assert f.tolist() == [1 + g[0], 1 + g[1] + resid, 1 + g[2], 1 + g[3], 1 + g[4]]


def test_cdf_pair_matches_cdf():
    rng = np.random.default_rng(2)
    z = rng.normal(size=(40, 32)).astype(np.float32)
    sym = rng.integers(0, 32, 40)
    st, fr = O.cdf_pairs(z, sym, 16)
    cdf = O.quantize_cdf(z, 16)
    assert np.array_equal(st, cdf[np.arange(40), sym])
    assert np.array_equal(fr, cdf[np.arange(40), sym + 1] - st)


def test_huge_logit_gaps_clamp():
    """Gaps far beyond the 40 * 2^16 cap (e.g. -1e30) clamp to e = 0, i.e. freq 1."""
    for gap in [-1e30, -3.0e38, -1e6, -27.8]:
        z = np.full(10, np.float32(gap), np.float32)
        z[3] = 0.0
        f = np.diff(O.quantize_cdf(z, 16)[0].astype(np.int64))
        assert f[3] == 2 ** 16 - 9 and np.all(np.delete(f, 3) == 1), gap
