"""Pins of the oracle's arithmetic coder (Sec. 3 "Arithmetic coding" and its worked example):
the paper's AAAB intervals and code, the entropy bound, the uniform closed form, brute force on
tiny alphabets, and bit-equality with the arbitrary-precision restatement."""
import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as O
from oracle import coder_spec as spec

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_aaab_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "aaab_example.json")))
    probs = [Fraction(p) for p in g["probs"]]
    iv = spec.interval_code(g["message"], probs)
    assert [(float(a), float(b)) for a, b in iv] == [(float(a), float(b)) for a, b in
                                                     [(Fraction(x), Fraction(y)) for x, y in g["intervals"]]]
    lo, hi = iv[-1]
    mid = (lo + hi) / 2
    assert mid == Fraction(g["midpoint"])
    assert spec.binary_digits(mid, 8) == g["binary"]
    code = Fraction(int(g["binary"], 2), 2 ** 8)
    assert lo <= code < hi


@pytest.mark.parametrize("P", [8, 16, 20, 24])
def test_integer_coder_code_lies_in_exact_interval(P):
    """The integer coder's code, read as a binary fraction, lies in the real interval of the
    recursion of Sec. 3 computed with the same (quantised) probabilities."""
    T = 2 ** P
    fA = round(0.8 * T)
    starts, freqs = [0, 0, 0, fA], [fA, fA, fA, T - fA]
    data, nbits = O.range_encode(np.array(starts), np.array(freqs), P)
    x = Fraction(int.from_bytes(data, "big"), 2 ** (8 * len(data)))
    lo, hi = spec.interval_code([0, 0, 0, 1], [Fraction(fA, T), Fraction(T - fA, T)])[-1]
    assert lo <= x < hi
    # -log2(0.8^3 * 0.2) = 3.29 bits; the code costs between J + 1 and J + 2 bits
    J = -math.log2((fA / T) ** 3 * (1 - fA / T))
    assert J + 1 - 1e-6 < nbits <= J + 2 + 1e-6


def random_stream(rng, n, V, P):
    T = 2 ** P
    cdfs = []
    st, fr, sym = [], [], []
    for _ in range(n):
        w = rng.exponential(size=V) ** 3
        f = 1 + np.floor(w / w.sum() * (T - V)).astype(np.int64)
        f[np.argmax(f)] += T - f.sum()
        c = np.concatenate([[0], np.cumsum(f)])
        s = int(rng.integers(0, V))
        cdfs.append(c)
        st.append(int(c[s]))
        fr.append(int(f[s]))
        sym.append(s)
    return st, fr, sym, cdfs


@pytest.mark.parametrize("P", [4, 12, 16, 24, 31])
def test_matches_bigint_spec_and_bound(P):
    rng = np.random.default_rng(P)
    for trial in range(60):
        n = int(rng.choice([0, 1, 2, 5, 50, 300, 2048])) if trial % 3 else int(rng.integers(0, 40))
        V = int(rng.integers(2, min(64, 2 ** P - 1) + 1))
        st, fr, sym, cdfs = random_stream(rng, n, V, P)
        data, nbits = O.range_encode(np.array(st, dtype=np.uint32), np.array(fr, dtype=np.uint32), P)
        code, nb = spec.encode(st, fr, P)
        assert nb == nbits and data == spec.code_bytes(code, nb)
        # entropy bound of Sec. 3 in its textbook form: J + 1 - eps < l <= J + 2 + eps
        J = -sum(math.log2(f / 2 ** P) for f in fr)
        eps = n * 2.0 ** (P - 60) * 1.45 + 1e-9
        assert J + 1 - eps < nbits <= J + 2 + eps
        # decode with both decoders
        assert spec.decode(code, nb, cdfs, P) == sym
        dec = O.Decoder(data, nbits)
        assert [dec.step(c, P) for c in cdfs] == sym


def test_ten_thousand_windows_against_bigint_spec():
    """10^4 independent short windows with random P in 1..31, random lengths (empty included) and
    random pairs drawn directly (any start in [0, T - freq], freq in [1, T], with runs of
    probability-one tokens and of the smallest freq): each window's code from the C coder equals
    the arbitrary-precision restatement bit for bit."""
    rng = np.random.default_rng(2409)
    for w in range(10_000):
        P = int(rng.integers(1, 32))
        T = 2 ** P
        n = int(rng.integers(0, 24))
        kind = w % 4
        if kind == 0:
            fr = rng.integers(1, T + 1, n)
        elif kind == 1:  # long runs of the smallest freq: one renormalisation step per token
            fr = np.ones(n, dtype=np.int64)
        elif kind == 2:  # probability-one tokens mixed in
            fr = np.where(rng.random(n) < 0.5, T, rng.integers(1, T + 1, n))
        else:  # freq near T, start at the top of the range (the carry-heavy case)
            fr = np.maximum(1, T - rng.integers(0, 4, n))
        st = np.array([int(rng.integers(0, T - f + 1)) if kind != 3 else T - int(f) for f in fr], dtype=np.int64)
        data, nbits = O.range_encode(st.astype(np.uint32), fr.astype(np.uint32), P)
        code, nb = spec.encode(st.tolist(), fr.tolist(), P)
        assert nb == nbits and data == spec.code_bytes(code, nb), (w, P, n)


def test_uniform_closed_form():
    """V = 32 equiprobable symbols at P = 16: l = 5n + 1 and the first 5n bits are the
    symbols' 5-bit binary codes, concatenated."""
    rng = np.random.default_rng(3)
    for n in [1, 2, 7, 100, 256]:
        sym = rng.integers(0, 32, n)
        data, nbits = O.range_encode(sym * 2048, np.full(n, 2048), 16)
        assert nbits == 5 * n + 1
        bits = "".join(f"{b:08b}" for b in data)
        assert bits[: 5 * n] == "".join(f"{s:05b}" for s in sym)


def test_brute_force_tiny_alphabets():
    rng = np.random.default_rng(11)
    for V, P in [(3, 4), (4, 6), (3, 8)]:
        T = 2 ** P
        f = 1 + rng.multinomial(T - V, rng.dirichlet(np.ones(V)))
        cdf = np.concatenate([[0], np.cumsum(f)])
        for n in range(1, 6):
            codes = {}
            for seq in itertools.product(range(V), repeat=n):
                st = [int(cdf[s]) for s in seq]
                fr = [int(f[s]) for s in seq]
                data, nbits = O.range_encode(np.array(st), np.array(fr), P)
                bits = "".join(f"{b:08b}" for b in data)[:nbits]
                dec = O.Decoder(data, nbits)
                assert tuple(dec.step(cdf, P) for _ in range(n)) == seq
                codes[seq] = bits
            vals = list(codes.values())
            assert len(set(vals)) == len(vals)  # distinct
            for a in vals:  # prefix-free within a fixed n
                for b in vals:
                    assert a == b or not b.startswith(a)


def test_corrupt_codes_do_not_crash():
    rng = np.random.default_rng(5)
    cdf = np.array([0, 3, 10, 1000, 1024])
    for _ in range(300):
        data = rng.integers(0, 256, 8, dtype=np.uint8).tobytes()
        dec = O.Decoder(data, 64)
        for _ in range(20):
            s = dec.step(cdf, 10)
            assert -1 <= s < 4
            if s < 0:
                break


def test_empty_stream():
    data, nbits = O.range_encode(np.zeros(0, np.uint32), np.zeros(0, np.uint32), 16)
    assert nbits == 2 and data == b"\x00"
