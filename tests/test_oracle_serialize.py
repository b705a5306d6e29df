"""Pins of the oracle's serialisation (Sec. 3 "Serialization", Fig. 1) against IEEE-754 closed
forms, Python's struct/hex library routines, and a round-trip sweep of fp32 bit patterns."""
import json
import os
import struct

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
SEPS = {0: [16], 1: [17], 2: [17, 16], 3: [18], 4: []}


def hex_tokens(h: str):
    return [int(c, 16) for c in h]


def test_ieee754_closed_forms():
    cases = json.load(open(os.path.join(GOLDEN, "ieee754_hex.json")))["cases"]
    vals = np.array([float(c["value"]) for c in cases], dtype=np.float32)
    tok = O.serialize(vals, 0).reshape(len(cases), 9)
    for row, c in zip(tok, cases):
        assert list(row[:8]) == hex_tokens(c["hex"]), c
        assert row[8] == 16


@pytest.mark.parametrize("sep_mode", [0, 1, 2, 3, 4])
def test_against_struct_hex(sep_mode):
    rng = np.random.default_rng(1)
    bits = rng.integers(0, 2 ** 32, 5000, dtype=np.uint64).astype(np.uint32)
    vals = bits.view(np.float32)
    tok = O.serialize(vals, sep_mode)
    expect = []
    for b in bits:
        h = struct.pack(">I", int(b)).hex()  # big-endian hex = most significant nibble first
        expect += hex_tokens(h) + SEPS[sep_mode]
    assert tok.tolist() == expect


def test_uint8_codes_all():
    codes = np.arange(256, dtype=np.uint8)
    tok = O.serialize(codes, 0).reshape(256, 3)
    for c, row in zip(range(256), tok):
        assert list(row) == hex_tokens(f"{c:02x}") + [16]
    assert np.array_equal(O.deserialize(tok.reshape(-1), 1, 0), codes)


def test_round_trip_sampled_sweep():
    """Every 256th fp32 bit pattern (2^24 patterns) plus NaN payloads, +-0, +-inf, subnormals."""
    special = np.array([0, 0x80000000, 0x7F800000, 0xFF800000, 0x7FC00000, 0x7FA00001, 0xFFFFFFFF,
                        0x00000001, 0x007FFFFF, 0x80000001, 0x7F7FFFFF], dtype=np.uint32)
    for chunk in range(16):
        base = np.arange(chunk * (1 << 20), (chunk + 1) * (1 << 20), dtype=np.uint64) * 256 + 255 * (chunk % 2)
        bits = np.concatenate([base.astype(np.uint32), special])
        tok = O.serialize(bits.view(np.float32), 0)
        back = O.deserialize(tok, 0, 0).view(np.uint32)
        assert np.array_equal(back, bits)


def test_malformed_rejected():
    tok = O.serialize(np.array([1.5], np.float32), 0)
    bad = tok.copy()
    bad[8] = 17
    with pytest.raises(ValueError):
        O.deserialize(bad, 0, 0)
    bad = tok.copy()
    bad[3] = 16
    with pytest.raises(ValueError):
        O.deserialize(bad, 0, 0)
    with pytest.raises(ValueError):
        O.deserialize(tok[:-1], 0, 0)


def test_tokens_per_value():
    assert O.tokens_per_value(0, 0) == 9
    assert O.tokens_per_value(0, 2) == 10
    assert O.tokens_per_value(0, 4) == 8
    assert O.tokens_per_value(1, 0) == 3
