"""The whole encode path on the GPU (lmgc_encode) against the oracle, and the KV-cached decode
(lmgc_decode) as its exact inverse: lossless round trips, CDF and bitstream parity given the
GPU's own logits and pairs, and container size within 0.5% of the oracle's."""
import struct

import numpy as np
import pytest
import torch

import oracle as O
from paper_2409_17836_gb300 import configs, inputs as I, lmgc as L
from tests._util import cpu_threads, oracle_config

pytestmark = pytest.mark.gpu


def parse(buf: bytes):
    return O.parse_container(buf)


def encode(ctx, vals):
    d = torch.from_numpy(vals.view(np.int32) if vals.dtype == np.float32 else vals).cuda()
    return L.lmgc_encode(ctx, d).cpu().numpy().tobytes()


def decode_all(ctx, buf, ids):
    dbuf = torch.from_numpy(np.frombuffer(buf, np.uint8).copy()).cuda()
    return L.lmgc_decode(ctx, dbuf, ids).cpu().numpy().view(np.uint16)


def test_tiny_full_encode_decode_and_oracle_size():
    cfg = configs.TINY
    ctx = L.Context(cfg)
    vals = I.tiny_gradient(0)
    buf = encode(ctx, vals)
    h = parse(buf)
    assert h["n_win"] == 144 and h["n_tok"] == 36864 and h["model_crc"] == O.model_crc(oracle_config(cfg))
    # full decode of every window: lossless
    toks = decode_all(ctx, buf, list(range(144)))
    tok_ref = O.serialize(vals, 0)
    assert np.array_equal(toks.reshape(-1), tok_ref)
    back = O.deserialize(toks.reshape(-1), 0, 0)
    assert back.tobytes() == vals.tobytes()
    # oracle encode of the same input: container size within 0.5%
    ref = O.encode(oracle_config(cfg), vals, n_par=cpu_threads())
    assert abs(len(buf) - len(ref)) <= 0.005 * len(ref), (len(buf), len(ref))
    ctx.close()


def test_fp32_gqa_hd64_round_trip():
    """An fp32 model with head dim 64 and grouped-query heads (the other shape of the TF32
    attention): encode then decode of every window is lossless, the decoder's one-row steps
    (keys and values from the cache) reproducing the encoder's logits; 14 windows of 200 tokens
    (the last partial) in batches of 4."""
    cfg = L.ModelConfig(n_layers=2, d_model=128, n_heads=2, n_kv_heads=1, d_ffn=256, vocab=32, dtype=L.F32,
                        window=200, cdf_bits=16, batch_windows=4, init_std=0.1)
    ctx = L.Context(cfg)
    vals = I.tiny_gradient(0)[:300]  # 2700 tokens
    buf = encode(ctx, vals)
    h = parse(buf)
    assert h["n_win"] == 14
    toks = decode_all(ctx, buf, list(range(14)))
    assert np.array_equal(toks.reshape(-1)[:2700], O.serialize(vals, 0))
    ctx.close()


def test_decode_batch_windows():
    """The decode batch query: at least one window, at most one workspace row per window, and a
    batch that covers the KV cache the context already holds after a decode."""
    cfg = configs.TINY
    ctx = L.Context(cfg)
    n = L.lmgc_decode_batch_windows(ctx)
    assert 1 <= n <= cfg.batch_windows * cfg.window
    vals = I.tiny_gradient(0)[:200]  # 1800 tokens: 8 windows of 256 (the last partial)
    buf = encode(ctx, vals)
    toks = decode_all(ctx, buf, list(range(8)))
    assert np.array_equal(toks.reshape(-1)[:1800], O.serialize(vals, 0))
    assert L.lmgc_decode_batch_windows(ctx) >= min(8, n)
    ctx.close()


def test_tiny_pairs_and_codes_given_gpu_logits():
    """CDF pairs bit-exact given the GPU's logits; codes bit-exact given those pairs."""
    cfg = configs.TINY
    ctx = L.Context(configs.with_(cfg, batch_windows=8))
    vals = I.tiny_gradient(0)[:2000]
    tok = O.serialize(vals, 0)
    W = cfg.window
    n_win = -(-tok.size // W)
    lg = L.lmgc_lm_probs(ctx, torch.from_numpy(tok.view(np.int16)).cuda(), 0, n_win).cpu().numpy()
    buf = encode(ctx, vals)
    h = parse(buf)
    for w in range(n_win):
        n = min(W, tok.size - w * W)
        st, fr = O.cdf_pairs(lg[w, :n], tok[w * W: w * W + n], cfg.cdf_bits)
        code, nbits = O.range_encode(st, fr, cfg.cdf_bits)
        assert h["bitlen"][w] == nbits and buf[h["offsets"][w]: h["offsets"][w + 1]] == code, w
    ctx.close()


def test_tinyllama_shape_pairs_and_codes_given_gpu_logits():
    """The tensor-core path (bf16, vocab 32000, P = 24, RMSNorm in the GEMMs, each row's maximum
    taken in the vocabulary GEMM's epilogue): every window's code of lmgc_encode is bit-exact with
    the oracle's CDF pairs and coder applied to the GPU's own logits of the same windows. One
    layer keeps it short; three windows, the last partial, in two batches."""
    cfg = configs.with_(configs.TINYLLAMA, n_layers=1, batch_windows=2)
    ctx = L.Context(cfg)
    W = cfg.window
    vals = I.convnet_gradient(0)[: (2 * W + 700) // 9]
    tok = O.serialize(vals, 0)
    n_win = -(-tok.size // W)
    assert n_win == 3
    buf = encode(ctx, vals)
    h = parse(buf)
    dtok = torch.from_numpy(tok.view(np.int16)).cuda()
    for w in range(n_win):
        n = min(W, tok.size - w * W)
        lg = L.lmgc_lm_probs(ctx, dtok, w, 1)[0, :n].cpu().numpy()
        st, fr = O.cdf_pairs(lg, tok[w * W: w * W + n], cfg.cdf_bits)
        code, nbits = O.range_encode(st, fr, cfg.cdf_bits)
        assert h["bitlen"][w] == nbits and buf[h["offsets"][w]: h["offsets"][w + 1]] == code, w
    ctx.close()


@pytest.mark.parametrize("group,order", [(3, 1), (8, 0), (1, 0)])
def test_byte_grouped_encode_decode_and_codes(group, order):
    """Byte grouping (Sec. 5.3) through the whole path: the container records the layout, every
    window's code is bit-exact with the oracle's pairs and coder on the GPU's logits of the
    oracle's token stream, and decoding restores the tokens and the values."""
    cfg = configs.with_(configs.TINY, sep_mode=1, byte_group=group, byte_order=order, batch_windows=4)
    ctx = L.Context(cfg)
    vals = I.tiny_gradient(3)[:1111]
    tok = O.serialize(vals, 1, group, order)
    buf = encode(ctx, vals)
    h = parse(buf)
    assert (h["sep_mode"], h["byte_group"], h["byte_order"]) == (1, group, order)
    assert h["n_tok"] == tok.size and h["n_values"] == vals.size
    W = cfg.window
    n_win = h["n_win"]
    lg = L.lmgc_lm_probs(ctx, torch.from_numpy(tok.view(np.int16)).cuda(), 0, n_win).cpu().numpy()
    for w in range(n_win):
        n = min(W, tok.size - w * W)
        st, fr = O.cdf_pairs(lg[w, :n], tok[w * W: w * W + n], cfg.cdf_bits)
        code, nbits = O.range_encode(st, fr, cfg.cdf_bits)
        assert h["bitlen"][w] == nbits and buf[h["offsets"][w]: h["offsets"][w + 1]] == code, w
    toks = decode_all(ctx, buf, list(range(n_win)))
    flat = np.concatenate([toks[w, :min(W, tok.size - w * W)] for w in range(n_win)])
    assert np.array_equal(flat, tok)
    back = torch.zeros(vals.size, dtype=torch.int32, device="cuda")
    assert L.lmgc_deserialize(ctx, torch.from_numpy(flat.view(np.int16)).cuda(), back) == vals.size
    assert back.cpu().numpy().tobytes() == vals.tobytes()
    # a context with the default layout rejects this container
    other = L.Context(configs.with_(configs.TINY, sep_mode=1, batch_windows=4))
    with pytest.raises(L.LmgcError) as e:
        decode_all(other, buf, [0])
    assert e.value.status == L.ERR_CORRUPT
    other.close()
    ctx.close()


@pytest.mark.parametrize("sep,group", [(0, 0), (2, 0), (4, 2)])
def test_alphabet_encode_decode_and_codes(sep, group):
    """Restricted-alphabet coding through the whole path: the container word carries the flag,
    every window's code is bit-exact with the oracle's pairs over the alphabet columns of the
    GPU's logits and its coder, decoding restores the tokens and values, the container is
    within 0.5% of the oracle's own encode, no larger than the full-vocabulary container, and a
    full-vocabulary context rejects it."""
    cfg = configs.with_(configs.TINY, sep_mode=sep, byte_group=group, alphabet=1, batch_windows=4)
    ctx = L.Context(cfg)
    vals = I.tiny_gradient(6)[:1500]
    tok = O.serialize(vals, sep, group, 0)
    A = np.array(O.alphabet_ids(sep))
    index = np.full(32, -1)
    index[A] = np.arange(A.size)
    buf = encode(ctx, vals)
    h = parse(buf)
    assert h["alphabet"] == 1 and h["sep_mode"] == sep and h["n_tok"] == tok.size
    W = cfg.window
    n_win = h["n_win"]
    lg = L.lmgc_lm_probs(ctx, torch.from_numpy(tok.view(np.int16)).cuda(), 0, n_win).cpu().numpy()
    for w in range(n_win):
        n = min(W, tok.size - w * W)
        t = tok[w * W: w * W + n]
        st, fr = O.cdf_pairs(np.ascontiguousarray(lg[w, :n][:, A]), index[t].astype(np.uint16), cfg.cdf_bits)
        code, nbits = O.range_encode(st, fr, cfg.cdf_bits)
        assert h["bitlen"][w] == nbits and buf[h["offsets"][w]: h["offsets"][w + 1]] == code, w
    toks = decode_all(ctx, buf, list(range(n_win)))
    flat = np.concatenate([toks[w, :min(W, tok.size - w * W)] for w in range(n_win)])
    assert np.array_equal(flat, tok)
    assert O.deserialize(flat, 0, sep, group, 0).tobytes() == vals.tobytes()
    ref = O.encode(oracle_config(cfg), vals, n_par=cpu_threads())
    assert abs(len(buf) - len(ref)) <= 0.005 * len(ref), (len(buf), len(ref))
    full = L.Context(configs.with_(cfg, alphabet=0))
    assert len(buf) <= len(encode(full, vals))
    with pytest.raises(L.LmgcError) as e:
        decode_all(full, buf, [0])
    assert e.value.status == L.ERR_CORRUPT
    full.close()
    ctx.close()


def test_tinyllama_shape_alphabet_narrow_head():
    """Restricted alphabet on the tensor-core path: encode and decode project onto the alphabet's
    17 rows of the vocabulary weight only (a 32-column GEMM), and every window's code is
    bit-exact with the oracle's pairs over those columns of the full 32,000-column logits of
    lmgc_lm_probs, so the narrow projection reproduces the full one's columns exactly. The
    partial last window decodes back to its tokens."""
    cfg = configs.with_(configs.TINYLLAMA, n_layers=1, batch_windows=2, alphabet=1)
    ctx = L.Context(cfg)
    W = cfg.window
    vals = I.convnet_gradient(1)[: (2 * W + 700) // 9]
    tok = O.serialize(vals, 0)
    n_win = -(-tok.size // W)
    A = np.array(O.alphabet_ids(0))
    index = np.full(32, -1)
    index[A] = np.arange(A.size)
    buf = encode(ctx, vals)
    h = parse(buf)
    assert h["alphabet"] == 1 and h["n_win"] == n_win == 3
    dtok = torch.from_numpy(tok.view(np.int16)).cuda()
    for w in range(n_win):
        n = min(W, tok.size - w * W)
        lg = L.lmgc_lm_probs(ctx, dtok, w, 1)[0, :n].cpu().numpy()
        t = tok[w * W: w * W + n]
        st, fr = O.cdf_pairs(np.ascontiguousarray(lg[:, A]), index[t].astype(np.uint16), cfg.cdf_bits)
        code, nbits = O.range_encode(st, fr, cfg.cdf_bits)
        assert h["bitlen"][w] == nbits and buf[h["offsets"][w]: h["offsets"][w + 1]] == code, w
    last = decode_all(ctx, buf, [n_win - 1])[0, : tok.size - (n_win - 1) * W]
    assert np.array_equal(last, tok[(n_win - 1) * W:])
    ctx.close()


@pytest.mark.parametrize("setting", ["quant16", "quant1", "sparse50", "sparse25"])
def test_compatibility_inputs_round_trip(setting):
    """Sec. 5.4 compatibility inputs one at a time through the whole path: Eq. 4 indices of every
    value (16 bits as big-endian byte pairs in 2-byte groups, 1 bit as bytes) or the top 50% /
    25% of |v| kept as fp32. The restored tokens equal the oracle's serialisation of the same
    input, the values come back exactly, and the container's size is within 0.5% of the
    oracle's encode."""
    g = I.tiny_gradient(4)
    if setting.startswith("quant"):
        vals, group = I.code_bytes(I.quantized_codes(g, 16 if setting == "quant16" else 1))
        cfg = configs.with_(configs.TINY, input_kind=L.IN_U8, byte_group=group, batch_windows=8)
        kind = 1
    else:
        vals, group = I.sparsified(g, 0.5 if setting == "sparse50" else 0.25), 0
        cfg = configs.with_(configs.TINY, batch_windows=8)
        kind = 0
    ctx = L.Context(cfg)
    buf = encode(ctx, vals)
    h = parse(buf)
    tok = O.serialize(vals, 0, group, 0)
    assert h["n_tok"] == tok.size and h["byte_group"] == group
    toks = decode_all(ctx, buf, list(range(h["n_win"])))
    W = cfg.window
    flat = np.concatenate([toks[w, :min(W, tok.size - w * W)] for w in range(h["n_win"])])
    assert np.array_equal(flat, tok)
    assert O.deserialize(flat, kind, 0, group, 0).tobytes() == vals.tobytes()
    ref = O.encode(oracle_config(cfg), vals, n_par=cpu_threads())
    assert abs(len(buf) - len(ref)) <= 0.005 * len(ref), (len(buf), len(ref))
    ctx.close()


@pytest.mark.parametrize("n,sep,kind", [(1, 0, 0), (29, 2, 0), (1000, 4, 0), (777, 0, 1)])
def test_tiny_edge_sizes_round_trip(n, sep, kind):
    cfg = configs.with_(configs.TINY, sep_mode=sep, input_kind=kind, batch_windows=3)
    ctx = L.Context(cfg)
    if kind == 0:
        vals = I.tiny_gradient(5)[:n]
    else:
        vals = I.lossy_codes(I.tiny_gradient(5), keep=n / 4096)
    buf = encode(ctx, vals)
    h = parse(buf)
    toks = decode_all(ctx, buf, list(range(h["n_win"])))
    tpv = O.tokens_per_value(kind, sep)
    flat = np.concatenate([toks[w, :min(cfg.window, h["n_tok"] - w * cfg.window)] for w in range(h["n_win"])])
    assert np.array_equal(flat, O.serialize(vals, sep))
    assert O.deserialize(flat, kind, sep).tobytes() == vals.tobytes()
    assert h["n_tok"] == vals.size * tpv
    ctx.close()


def test_corrupt_container_rejected():
    ctx = L.Context(configs.with_(configs.TINY, batch_windows=2))
    buf = bytearray(encode(ctx, I.tiny_gradient(1)[:100]))
    bad = bytearray(buf)
    bad[20] ^= 0xFF
    with pytest.raises(L.LmgcError) as e:
        decode_all(ctx, bytes(bad), [0])
    assert e.value.status == L.ERR_CORRUPT
    with pytest.raises(L.LmgcError):
        decode_all(ctx, bytes(buf[:70]), [0])
    other = L.Context(configs.with_(configs.TINY, batch_windows=2, weight_seed=9))
    with pytest.raises(L.LmgcError) as e:
        decode_all(other, bytes(buf), [0])
    assert e.value.status == L.ERR_CORRUPT
    with pytest.raises(L.LmgcError):
        decode_all(ctx, bytes(buf), [10 ** 6])
    # the token checksum table: it equals the oracle's, a flipped checksum bit fails the window it
    # covers, and a flipped payload bit (which the coder alone would decode into other tokens)
    # fails too, while the untouched window still decodes
    h = parse(bytes(buf))
    assert np.array_equal(h["crc_tok"], O.window_crcs(O.serialize(I.tiny_gradient(1)[:100], 0), 256))
    bad = bytearray(buf)
    bad[64 + 4 * h["n_win"] + 1] ^= 0x10
    with pytest.raises(L.LmgcError) as e:
        decode_all(ctx, bytes(bad), [0])
    assert e.value.status == L.ERR_CORRUPT
    decode_all(ctx, bytes(bad), [1])
    bad = bytearray(buf)
    bad[h["offsets"][1] + 5] ^= 0x04
    with pytest.raises(L.LmgcError) as e:
        decode_all(ctx, bytes(bad), [1])
    assert e.value.status == L.ERR_CORRUPT
    decode_all(ctx, bytes(bad), [0])
    ctx.close()
    other.close()


def test_host_buffer_encode_matches_device():
    ctx = L.Context(configs.with_(configs.TINY, batch_windows=8))
    vals = I.tiny_gradient(2)
    dev = encode(ctx, vals)
    hin = torch.from_numpy(vals.view(np.int32).copy()).pin_memory()
    hout = torch.empty(L.lmgc_encode_bound(ctx, vals.size), dtype=torch.uint8).pin_memory()
    nb = L.lmgc_encode_host(ctx, hin, hout)
    assert hout[:nb].numpy().tobytes() == dev
    ctx.close()


def test_tinyllama_shape_sampled_round_trip():
    """TinyLlama shape (bf16, 22 layers, GQA, vocab 32000, P = 24) on ConvNet gradients: the
    first windows are encoded and decoded (KV-cached) back to the exact input bits; the ideal code
    length -sum log2(freq / T) of the first 16 tokens under the GPU's logits is within 0.5% of the
    same length under the oracle's (both through the oracle's quantiser)."""
    cfg = configs.with_(configs.TINYLLAMA, batch_windows=2)
    ctx = L.Context(cfg)
    g = I.convnet_gradient(0)
    vals = g[: (2 * 2048 - 300) // 9]  # a full window and a partial one
    buf = encode(ctx, vals)
    h = parse(buf)
    assert h["n_win"] == 2
    toks = decode_all(ctx, buf, [0, 1])
    flat = np.concatenate([toks[0], toks[1, : h["n_tok"] - 2048]])
    assert O.deserialize(flat, 0, 0).tobytes() == vals.tobytes()
    tok = O.serialize(vals, 0)
    lg = L.lmgc_lm_probs(ctx, torch.from_numpy(tok.view(np.int16)).cuda(), 0, 1)[0, :16].cpu().numpy()
    ctx.close()
    st_g, fr_g = O.cdf_pairs(lg, tok[:16], 24)
    st_o, fr_o, _ = O.window_pairs(oracle_config(cfg, n_threads=cpu_threads()), tok, 16)
    jg = -np.log2(fr_g / 2.0 ** 24).sum()
    jo = -np.log2(fr_o / 2.0 ** 24).sum()
    assert abs(jg - jo) <= 0.005 * jo, (jg, jo)


def test_window_ranges_assemble_to_the_container():
    """lmgc_encode_windows on two window ranges (as two GPUs would) plus lmgc_container_header,
    assembled, equal lmgc_encode's container byte for byte."""
    from paper_2409_17836_gb300 import shard

    ctx = L.Context(configs.with_(configs.TINY, batch_windows=5))
    vals = I.tiny_gradient(4)[:1000]
    d = torch.from_numpy(vals.view(np.int32).copy()).cuda()
    ref = L.lmgc_encode(ctx, d).cpu().numpy().tobytes()
    n_win = -(-vals.size * 9 // 256)
    parts = []
    for first, count in shard.window_ranges(n_win, 2):
        pay, bl, crc = L.lmgc_encode_windows(ctx, d, first, count)
        parts.append((bl.cpu().numpy().view(np.uint32), crc.cpu().numpy().view(np.uint32), pay.cpu().numpy().tobytes()))
    got = shard.assemble(L.lmgc_container_header(ctx, vals.size), [p[0] for p in parts], [p[1] for p in parts],
                         [p[2] for p in parts])
    assert got == ref
    ctx.close()
