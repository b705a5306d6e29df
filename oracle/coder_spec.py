"""Arbitrary-precision restatements of the arithmetic coder (test infrastructure only).

* `interval_code` -- the real-interval recursion of Sec. 3 "Arithmetic coding" in exact
  rationals: start from [0, 1), give each symbol the sub-interval of its cumulative
  probability (symbol order low to high) and keep the chosen one; any number of the final
  interval represents the message. Used for the paper's worked example (a message "AAAB"
  with P(A) = 0.8, P(B) = 0.2).
* `encode` / `decode` -- the exact integer form the oracle and the CUDA coder implement,
  written with Python integers so that L is held as one unbounded integer:
      R = 2^62, L = 0, B = 0; per symbol: r = R >> P; L += r*s; R = r*f;
      k = max(0, 62 - bitlen(R)); R <<= k; L <<= k; B += k
  and the code is the top B+2 bits of v = ceil(L / 2^60) * 2^60.
"""
from __future__ import annotations

from fractions import Fraction

W_C = 62


def interval_code(message: list[int], probs: list[Fraction]) -> list[tuple[Fraction, Fraction]]:
    """Intervals [low, high) after each symbol of the real-interval recursion (Sec. 3)."""
    cum = [Fraction(0)]
    for p in probs:
        cum.append(cum[-1] + p)
    low, high = Fraction(0), Fraction(1)
    out = []
    for s in message:
        width = high - low
        low, high = low + width * cum[s], low + width * cum[s + 1]
        out.append((low, high))
    return out


def binary_digits(x: Fraction, n: int) -> str:
    """First n binary digits of x in [0, 1) (truncated)."""
    bits = []
    for _ in range(n):
        x *= 2
        b = int(x >= 1)
        bits.append(str(b))
        x -= b
    return "".join(bits)


def encode(start: list[int], freq: list[int], P: int) -> tuple[int, int]:
    """Returns (code as an integer of `nbits` bits, nbits)."""
    R, L, B = 1 << W_C, 0, 0
    for s, f in zip(start, freq):
        r = R >> P
        L += r * s
        R = r * f
        k = max(0, W_C - R.bit_length())
        R <<= k
        L <<= k
        B += k
    v = -(-L // (1 << 60)) * (1 << 60)
    nbits = B + 2
    return v >> 60, nbits


def code_bytes(code: int, nbits: int) -> bytes:
    nbytes = (nbits + 7) // 8
    return (code << (8 * nbytes - nbits)).to_bytes(nbytes, "big") if nbytes else b""


def decode(code: int, nbits: int, cdfs, P: int) -> list[int]:
    """Decode len(cdfs) symbols; cdfs[i] is the CDF (length V+1) used at step i, or a callable
    taking the symbols decoded so far and returning it."""
    def bit(i):
        return (code >> (nbits - 1 - i)) & 1 if i < nbits else 0

    pos = 0
    D = 0
    for _ in range(W_C):
        D = (D << 1) | bit(pos)
        pos += 1
    R = 1 << W_C
    out: list[int] = []
    for i in range(len(cdfs)):
        cdf = cdfs[i](out) if callable(cdfs[i]) else cdfs[i]
        cdf = [int(c) for c in cdf]
        r = R >> P
        t = D // r
        if t >= (1 << P):
            raise ValueError("corrupt code")
        s = next(j for j in range(len(cdf) - 1) if cdf[j] <= t < cdf[j + 1])
        D -= r * cdf[s]
        R = r * (cdf[s + 1] - cdf[s])
        k = max(0, W_C - R.bit_length())
        for _ in range(k):
            D = (D << 1) | bit(pos)
            pos += 1
        R <<= k
        out.append(s)
    return out
