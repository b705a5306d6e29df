"""Restricted-alphabet coding (a variant the paper does not describe: the integer CDF of each
position is taken over the ids the serialisation can emit -- 16 hex digits and the separator
ids -- and the coded symbol is the token's index among them). Pinned by closed forms on a
model with zero weights, whose logits are all zero."""
import numpy as np
import pytest

import oracle as O


def tiny_cfg(**kw):
    base = dict(n_layers=1, d_model=64, n_heads=2, n_kv_heads=2, d_ffn=128, vocab=32, bf16=False, window=40,
                cdf_bits=16, weight_seed=3, init_std=0.02)
    base.update(kw)
    return O.OracleConfig(**base)


def test_alphabet_ids():
    assert O.alphabet_ids(0) == list(range(16)) + [16]
    assert O.alphabet_ids(2) == list(range(16)) + [16, 17]
    assert O.alphabet_ids(3) == list(range(16)) + [18]
    assert O.alphabet_ids(4) == list(range(16))


def test_zero_model_gives_uniform_restricted_cdf():
    # zero weights -> zero logits -> every e = 2^31; with V' = 17 ids and T = 2^16:
    # g = floor(2^31 (T - 17) / (17 * 2^31)) = 3854, freq = 3855, and the remainder
    # (T - 17) - 17 * 3854 = 1 goes to index 0 (the lowest index of the largest e)
    cfg = tiny_cfg(init_std=0.0, alphabet=1)
    tok = np.array([3, 16, 0, 15, 16, 9], dtype=np.uint16)
    st, fr, lg = O.window_pairs(cfg, tok, tok.size)
    assert np.all(lg == 0.0)
    idx = np.array([3, 16, 0, 15, 16, 9])
    freq = np.where(idx == 0, 3856, 3855)
    start = np.where(idx == 0, 0, 3856 + (idx - 1) * 3855)
    assert fr.tolist() == freq.tolist() and st.tolist() == start.tolist()
    # the whole vocabulary (32 ids) on the same model: freq = 1 + floor((T - 32) / 32) = 2048
    st32, fr32, _ = O.window_pairs(tiny_cfg(init_std=0.0), tok, tok.size)
    assert fr32.tolist() == [2048] * tok.size and st32.tolist() == (tok.astype(int) * 2048).tolist()


@pytest.mark.parametrize("sep_mode", [0, 2, 4])
def test_restricted_alphabet_round_trip(sep_mode):
    cfg = tiny_cfg(alphabet=1, sep_mode=sep_mode)
    vals = np.random.default_rng(sep_mode).normal(0, 1e-2, 11).astype(np.float32)
    tok = O.serialize(vals, sep_mode)
    W = cfg.window
    n_win = -(-tok.size // W)
    codes = O.encode_windows(cfg, tok, 0, n_win)
    for w, (code, nbits) in enumerate(codes):
        n = min(W, tok.size - w * W)
        assert np.array_equal(O.decode_window(cfg, code, nbits, n), tok[w * W: w * W + n])
    # a token outside the alphabet cannot be coded
    with pytest.raises(RuntimeError):
        O.window_pairs(cfg, np.array([19 if sep_mode != 4 else 16, 1], dtype=np.uint16), 2)
