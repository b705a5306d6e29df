"""The error terms of the three-pass TF32 form that fp32 models' contractions use on the tensor
cores (gemm_tf32.cu, attn_tf32.cu), checked in exact arithmetic on the CPU: x = hi + lo with hi
= x with its low 13 bits cleared, a product a b taken as lo_a hi_b + hi_a lo_b + hi_a hi_b where
the tensor core reads only the top 19 bits of each operand (so lo is truncated, or rounded, to
10 mantissa bits). The GPU tests bound the whole contraction by 2^-17 sum |a b|: 2^-19 for the
fp32 accumulation (as for the fp16 kernel) plus the split's terms checked here, each below
2^-20 |a b|."""
import numpy as np


def tf32_trunc(x: np.ndarray) -> np.ndarray:
    return (x.view(np.uint32) & np.uint32(0xFFFFE000)).view(np.float32)


def tf32_round(x: np.ndarray) -> np.ndarray:
    # to nearest, ties away from zero, on the 13 dropped bits
    u = x.view(np.uint32).astype(np.uint64)
    u = ((u + 0x1000) & 0xFFFFE000).astype(np.uint32)
    return u.view(np.float32)


def split(x: np.ndarray):
    hi = tf32_trunc(x)
    lo = (x - hi).astype(np.float32)  # exact: x and hi share the exponent and the top bits
    return hi, lo


def test_split_is_exact_and_lo_small():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(200_000) * np.exp2(rng.integers(-20, 20, 200_000))).astype(np.float32)
    hi, lo = split(x)
    assert np.array_equal(hi.astype(np.float64) + lo.astype(np.float64), x.astype(np.float64))
    assert np.all(np.abs(lo) <= np.abs(x) * 2.0 ** -10)
    assert np.all(hi.view(np.uint32) & 0x1FFF == 0)


def test_three_pass_product_error_below_three_times_2_pow_minus_20():
    rng = np.random.default_rng(1)
    n = 200_000
    a = (rng.standard_normal(n) * np.exp2(rng.integers(-8, 8, n))).astype(np.float32)
    b = (rng.standard_normal(n) * np.exp2(rng.integers(-8, 8, n))).astype(np.float32)
    ha, la = split(a)
    hb, lb = split(b)
    exact = a.astype(np.float64) * b.astype(np.float64)
    for read in (tf32_trunc, tf32_round):  # however the tensor core reads the low parts
        got = (read(la).astype(np.float64) * hb + ha.astype(np.float64) * read(lb) +
               ha.astype(np.float64) * hb.astype(np.float64))
        err = np.abs(got - exact)
        assert np.all(err <= 3 * 2.0 ** -20 * np.abs(exact) + 1e-45)
        # and the sum of such products keeps the relative bound of sum |a b|
        k = 500
        e_sum = np.abs((got - exact).reshape(-1, k).sum(axis=1))
        ref = np.abs(exact).reshape(-1, k).sum(axis=1)
        assert np.all(e_sum <= 3 * 2.0 ** -20 * ref)
