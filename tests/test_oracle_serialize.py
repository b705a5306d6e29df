"""Pins of the oracle's serialisation (Sec. 4 "Serialization", Fig. 1) against IEEE-754 closed
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


# ---- byte grouping (Sec. 5.3 "Byte grouping": bytes per group BPG in {1, 2, 3, 4, 8}) ----

def grouped_by_hex_string(vals: np.ndarray, sep_mode: int, group: int, order: int):
    """The definition through Python's bytes.hex(): the byte stream (each fp32 big- or
    little-endian, uint8 codes as is), two hex characters per byte, the separator after every
    `group` bytes and after a final partial group."""
    if vals.dtype == np.float32:
        data = vals.astype(">f4" if order == 0 else "<f4").tobytes()
    else:
        data = vals.tobytes()
    out = []
    for k in range(0, len(data), group):
        out += hex_tokens(data[k:k + group].hex()) + SEPS[sep_mode]
    return out


def test_grouped_worked_examples():
    # 1.0f = 3f800000, -2.0f = c0000000
    v = np.array([1.0, -2.0], dtype=np.float32)
    assert O.serialize(v[:1], 0, 1, 0).tolist() == [3, 15, 16, 8, 0, 16, 0, 0, 16, 0, 0, 16]
    assert O.serialize(v[:1], 0, 1, 1).tolist() == [0, 0, 16, 0, 0, 16, 8, 0, 16, 3, 15, 16]
    # BPG 3 crosses the value boundary; the last group (2 bytes) is partial and still separated
    assert O.serialize(v, 3, 3, 0).tolist() == [3, 15, 8, 0, 0, 0, 18, 0, 0, 12, 0, 0, 0, 18, 0, 0, 0, 0, 18]
    # BPG 8: one separator per two values; H_{c+s} separators are two tokens
    assert O.serialize(v, 2, 8, 0).tolist() == [3, 15, 8, 0, 0, 0, 0, 0, 12, 0, 0, 0, 0, 0, 0, 0, 17, 16]
    assert O.serial_tokens(0, 2, 3, 8, 0) == 3 * 8 + 2 * 2


def test_grouped_default_group_is_one_value():
    # the paper's default BPG = 4 for fp32 (and 1 for uint8 codes) is the one-group-per-value layout
    rng = np.random.default_rng(7)
    vals = rng.integers(0, 2 ** 32, 3000, dtype=np.uint64).astype(np.uint32).view(np.float32)
    codes = rng.integers(0, 256, 3000).astype(np.uint8)
    for sep in range(5):
        assert np.array_equal(O.serialize(vals, sep, 4, 0), O.serialize(vals, sep))
        assert np.array_equal(O.serialize(codes, sep, 1, 0), O.serialize(codes, sep))


@pytest.mark.parametrize("group", [1, 2, 3, 4, 8])
@pytest.mark.parametrize("order", [0, 1])
@pytest.mark.parametrize("sep_mode", [0, 2, 4])
def test_grouped_against_hex_string_and_round_trip(group, order, sep_mode):
    rng = np.random.default_rng(100 * group + 10 * order + sep_mode)
    for n in (1, 2, 3, 5, 8, 333):
        vals = rng.integers(0, 2 ** 32, n, dtype=np.uint64).astype(np.uint32).view(np.float32)
        tok = O.serialize(vals, sep_mode, group, order)
        assert tok.tolist() == grouped_by_hex_string(vals, sep_mode, group, order), n
        assert tok.size == O.serial_tokens(0, sep_mode, n, group, order)
        back = O.deserialize(tok, 0, sep_mode, group, order)
        assert back.view(np.uint32).tolist() == vals.view(np.uint32).tolist()
        codes = rng.integers(0, 256, n).astype(np.uint8)
        tc = O.serialize(codes, sep_mode, group, 0)
        assert tc.tolist() == grouped_by_hex_string(codes, sep_mode, group, 0)
        assert np.array_equal(O.deserialize(tc, 1, sep_mode, group, 0), codes)


def test_grouped_rejects_malformed_streams():
    vals = np.array([1.0, -2.0, 3.5], dtype=np.float32)
    tok = O.serialize(vals, 0, 3, 0)
    with pytest.raises(ValueError):
        O.deserialize(tok[:-1], 0, 0, 3, 0)  # no value count gives this length
    bad = tok.copy()
    bad[6] = 5  # a digit where the separator belongs
    with pytest.raises(ValueError):
        O.deserialize(bad, 0, 0, 3, 0)
    bad = tok.copy()
    bad[0] = 16  # a separator where a digit belongs
    with pytest.raises(ValueError):
        O.deserialize(bad, 0, 0, 3, 0)
