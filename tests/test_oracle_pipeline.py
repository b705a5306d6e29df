"""Oracle end to end (Sec. 4): serialise -> windows with BOS -> LM -> integer CDF -> one code per
window -> container; decoding each window token by token (KV-cached, Sec. 4 "Compression")
must return the serialised tokens, and deserialising must return the input bits (lossless)."""
import zlib

import numpy as np
import pytest

import oracle as O
from paper_2409_17836_gb300 import inputs as I


def small_cfg(**kw):
    base = dict(n_layers=2, d_model=32, n_heads=2, n_kv_heads=1, d_ffn=64, vocab=32, bf16=False, window=50,
                cdf_bits=16, weight_seed=3, init_std=0.3)
    base.update(kw)
    return O.OracleConfig(**base)


@pytest.mark.parametrize("sep_mode,kind", [(0, 0), (2, 0), (4, 0), (0, 1)])
def test_round_trip(sep_mode, kind):
    c = small_cfg(sep_mode=sep_mode, input_kind=kind)
    if kind == 0:
        vals = I.tiny_gradient(1)[:23]
    else:
        vals = I.lossy_codes(I.tiny_gradient(1), keep=0.05)
    buf = O.encode(c, vals, n_par=4)
    h = O.parse_container(buf)
    tok = O.serialize(vals, sep_mode)
    assert h["n_tok"] == tok.size and h["n_values"] == vals.size and h["n_win"] == -(-tok.size // 50)
    assert h["model_crc"] == O.model_crc(c)
    out = []
    for w in range(h["n_win"]):
        n = min(50, tok.size - 50 * w)
        code = buf[h["offsets"][w]: h["offsets"][w + 1]]
        out.append(O.decode_window(c, code, int(h["bitlen"][w]), n))
        assert h["crc_tok"][w] == O.crc32(out[-1].astype("<u2").tobytes())
    out = np.concatenate(out)
    assert np.array_equal(out, tok)
    back = O.deserialize(out, kind, sep_mode)
    assert back.tobytes() == vals.tobytes()
    assert abs(O.compression_rate(len(buf), vals.size, 4 if kind == 0 else 1) - 100 * len(buf) /
               (vals.size * (4 if kind == 0 else 1))) < 1e-12


def test_window_codes_are_independent():
    c = small_cfg()
    tok = O.serialize(I.tiny_gradient(2)[:30], 0)
    all_codes = O.encode_windows(c, tok, 0, 5, n_par=2)
    for w in (0, 3):
        assert O.encode_windows(c, tok, w, 1)[0] == all_codes[w]


def test_header_crc_detects_corruption():
    c = small_cfg()
    buf = bytearray(O.encode(c, I.tiny_gradient(3)[:10]))
    buf[9] ^= 1
    with pytest.raises(ValueError):
        O.parse_container(bytes(buf))


def test_config1_sample_windows_round_trip():
    """The 4,096-value configuration (2 layers, d 128, 4 heads, FFN 512, V 32, fp32, W 256,
    P 16): first, middle and last windows."""
    c = O.OracleConfig(n_layers=2, d_model=128, n_heads=4, n_kv_heads=4, d_ffn=512, vocab=32, bf16=False,
                       window=256, cdf_bits=16, weight_seed=0)
    tok = O.serialize(I.tiny_gradient(0), 0)
    assert tok.size == 36864
    for w in (0, 71, 143):
        (code, nbits), = O.encode_windows(c, tok, w, 1)
        dec = O.decode_window(c, code, nbits, 256)
        assert np.array_equal(dec, tok[w * 256:(w + 1) * 256])
        # random-init weights: the prior is weak, so a code costs more than 4 bits per token
        assert nbits > 4 * 256


def test_crc32_check_value_and_library():
    """The container's CRC-32 (IEEE 802.3, reflected polynomial 0xEDB88320): the published check
    value of the nine ASCII digits, and agreement with zlib on random buffers and lengths."""
    assert O.crc32(b"123456789") == 0xCBF43926
    assert O.crc32(b"") == 0
    rng = np.random.default_rng(7)
    for n in (1, 2, 3, 17, 4096, 10001):
        b = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
        assert O.crc32(b) == zlib.crc32(b)


def test_window_crc_table_matches_tokens():
    c = small_cfg()
    vals = I.tiny_gradient(5)[:19]
    buf = O.encode(c, vals)
    h = O.parse_container(buf)
    tok = O.serialize(vals, 0).astype("<u2")
    for w in range(h["n_win"]):
        assert h["crc_tok"][w] == zlib.crc32(tok[50 * w: 50 * (w + 1)].tobytes())
    # a flipped bit in the table is caught by comparing against the decoded tokens
    bad = bytearray(buf)
    bad[64 + 4 * h["n_win"]] ^= 1
    assert O.parse_container(bytes(bad))["crc_tok"][0] != h["crc_tok"][0]
