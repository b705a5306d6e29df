"""GPU parity of the integer stages against the oracle, through the C ABI:
serialisation (Sec. 4), integer CDF given identical logits, and the arithmetic coder (Sec. 3)
given identical (start, freq) pairs -- all bit-exact."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2409_17836_gb300 import configs, lmgc as L
from tests._util import random_pairs, to_pair_tiles

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx_tiny():
    c = L.Context(configs.with_(configs.TINY, batch_windows=4))
    yield c
    c.close()


def ctx_for(**kw):
    return L.Context(configs.with_(configs.TINY, batch_windows=1, **kw))


SPECIAL = np.array([0, 0x80000000, 0x7F800000, 0xFF800000, 0x7FC00000, 0x7FA00001, 0xFFFFFFFF, 1, 0x007FFFFF,
                    0x3F800000], dtype=np.uint32)


@pytest.mark.parametrize("sep_mode", [0, 1, 2, 3, 4])
@pytest.mark.parametrize("n", [1, 7, 1023, 1024, 1025, 4096, 100003])
def test_serialize_bit_exact(sep_mode, n):
    ctx = ctx_for(sep_mode=sep_mode)
    rng = np.random.default_rng(n + sep_mode)
    bits = rng.integers(0, 2 ** 32, n, dtype=np.uint64).astype(np.uint32)
    bits[: min(n, SPECIAL.size)] = SPECIAL[: min(n, SPECIAL.size)]
    vals = bits.view(np.float32)
    d = torch.from_numpy(bits.view(np.int32).copy()).cuda()
    tok = L.lmgc_serialize(ctx, d)
    ref = O.serialize(vals, sep_mode)
    assert np.array_equal(tok.cpu().numpy().view(np.uint16), ref)
    back = torch.empty(n, dtype=torch.int32, device="cuda")
    assert L.lmgc_deserialize(ctx, tok, back) == n
    assert np.array_equal(back.cpu().numpy().view(np.uint32), bits)
    ctx.close()


def test_serialize_unaligned_input_and_u8():
    ctx = ctx_for()
    rng = np.random.default_rng(3)
    bits = rng.integers(0, 2 ** 32, 5001, dtype=np.uint64).astype(np.uint32)
    d = torch.from_numpy(bits.view(np.int32).copy()).cuda()
    tok = L.lmgc_serialize(ctx, d[1:])  # 4-byte aligned, not 16
    assert np.array_equal(tok.cpu().numpy().view(np.uint16), O.serialize(bits[1:].view(np.float32), 0))
    ctx.close()
    ctx = ctx_for(input_kind=L.IN_U8)
    codes = rng.integers(0, 256, 3001).astype(np.uint8)
    tok = L.lmgc_serialize(ctx, torch.from_numpy(codes).cuda())
    assert np.array_equal(tok.cpu().numpy().view(np.uint16), O.serialize(codes, 0))
    out = torch.empty(3001, dtype=torch.uint8, device="cuda")
    L.lmgc_deserialize(ctx, tok, out)
    assert np.array_equal(out.cpu().numpy(), codes)
    ctx.close()


@pytest.mark.parametrize("group,order", [(1, 0), (2, 1), (3, 0), (3, 1), (4, 1), (5, 1), (6, 0), (7, 1), (8, 0),
                                         (8, 1)])
@pytest.mark.parametrize("sep_mode", [0, 2, 4])
def test_serialize_byte_groups_bit_exact(group, order, sep_mode):
    """Byte grouping (Sec. 5.3): tokens bit-exact with the oracle for fp32 values (either byte
    order) and uint8 codes, ragged counts whose last group is partial; round trip; the token
    count through lmgc_serial_tokens. The counts span whole tiles of word-aligned units (the
    unit kernel, one instantiation per group width) and the rest (the per-group kernel)."""
    ctx = ctx_for(sep_mode=sep_mode, byte_group=group, byte_order=order)
    rng = np.random.default_rng(10 * group + order + sep_mode)
    for n in (1, 2, 3, 1001, 65537):
        bits = rng.integers(0, 2 ** 32, n, dtype=np.uint64).astype(np.uint32)
        bits[: min(n, SPECIAL.size)] = SPECIAL[: min(n, SPECIAL.size)]
        d = torch.from_numpy(bits.view(np.int32).copy()).cuda()
        tok = L.lmgc_serialize(ctx, d)
        ref = O.serialize(bits.view(np.float32), sep_mode, group, order)
        assert L.lmgc_serial_tokens(ctx, n) == ref.size
        assert np.array_equal(tok.cpu().numpy().view(np.uint16), ref), n
        back = torch.zeros(n, dtype=torch.int32, device="cuda")
        assert L.lmgc_deserialize(ctx, tok, back) == n
        assert np.array_equal(back.cpu().numpy().view(np.uint32), bits), n
    # a per-value token count exists unless groups cross values and carry separators
    assert (ctx.tpv is None) == (group in (3, 5, 6, 7, 8) and sep_mode != 4)
    ctx.close()
    ctx = ctx_for(sep_mode=sep_mode, byte_group=group, input_kind=L.IN_U8)
    codes = rng.integers(0, 256, 4099).astype(np.uint8)
    tok = L.lmgc_serialize(ctx, torch.from_numpy(codes).cuda())
    assert np.array_equal(tok.cpu().numpy().view(np.uint16), O.serialize(codes, sep_mode, group, 0))
    out = torch.empty(4099, dtype=torch.uint8, device="cuda")
    assert L.lmgc_deserialize(ctx, tok, out) == 4099
    assert np.array_equal(out.cpu().numpy(), codes)
    ctx.close()


def test_deserialize_byte_groups_rejects_malformed():
    ctx = ctx_for(byte_group=3)
    tok = L.lmgc_serialize(ctx, torch.ones(10, dtype=torch.float32, device="cuda"))
    assert tok.numel() == 2 * 40 + 14
    bad = tok.clone()
    bad[6] = 5  # a digit where the first group's separator belongs
    with pytest.raises(L.LmgcError) as e:
        L.lmgc_deserialize(ctx, bad, torch.empty(10, device="cuda"))
    assert e.value.status == L.ERR_CORRUPT
    with pytest.raises(L.LmgcError) as e:
        L.lmgc_deserialize(ctx, tok[:-1], torch.empty(10, device="cuda"))  # no count gives 93 tokens
    assert e.value.status == L.ERR_CORRUPT
    ctx.close()


def test_deserialize_rejects_malformed(ctx_tiny):
    tok = L.lmgc_serialize(ctx_tiny, torch.ones(10, dtype=torch.float32, device="cuda"))
    bad = tok.clone()
    bad[8] = 17
    with pytest.raises(L.LmgcError) as e:
        L.lmgc_deserialize(ctx_tiny, bad, torch.empty(10, device="cuda"))
    assert e.value.status == L.ERR_CORRUPT
    with pytest.raises(L.LmgcError):
        L.lmgc_deserialize(ctx_tiny, tok[:-1], torch.empty(10, device="cuda"))


def logit_rows(rng, rows, V):
    z = rng.normal(size=(rows, V)) * rng.uniform(0.05, 12, size=(rows, 1))
    z = z.astype(np.float32)
    z[0] = 0.0                      # uniform
    z[1] = -7.5
    z[1, V // 3] = 100.0            # one-hot dominant (others clamp to e = 0)
    z[2] = np.round(z[2])           # many ties
    z[3, :] = -1e30                 # huge negative values
    z[3, 5] = 3.0
    z[4] = z[4] * 1e-6              # nearly uniform, ties in a
    return z


@pytest.mark.parametrize("V,P,rows", [(32, 16, 3000), (1000, 20, 300), (32000, 24, 64)])
def test_cdf_bit_exact(V, P, rows):
    ctx = L.Context(configs.with_(configs.TINY, vocab=V, cdf_bits=P, batch_windows=1))
    rng = np.random.default_rng(V)
    z = logit_rows(rng, rows, V)
    dz = torch.from_numpy(z).cuda()
    cdf = L.lmgc_quantize_cdf(ctx, dz).cpu().numpy().view(np.uint32)
    ref = O.quantize_cdf(z, P)
    assert np.array_equal(cdf, ref)
    sym = rng.integers(0, V, rows).astype(np.uint16)
    sym[1] = V // 3
    st, fr = L.lmgc_cdf_pairs(ctx, dz, torch.from_numpy(sym.view(np.int16)).cuda())
    rs, rf = O.cdf_pairs(z, sym, P)
    assert np.array_equal(st.cpu().numpy().view(np.uint32), rs)
    assert np.array_equal(fr.cpu().numpy().view(np.uint32), rf)
    ctx.close()


def coder(start, freq, P, n_win, W, lens, layout):
    """The GPU coder on [n_win][W] pairs passed in the given layout: row-major and position-major
    through lmgc_range_encode's strides, window tiles through lmgc_range_encode_tiled, checked
    ("tile") or vouched for as the encode path does ("tile-trusted")."""
    wl = torch.from_numpy(lens.view(np.int32)).cuda() if lens is not None else None
    if layout in ("tile", "tile-trusted"):
        st, fr = to_pair_tiles(start), to_pair_tiles(freq)
        assert st.size == L.lmgc_pair_tile_elems(n_win, W)
        return L.lmgc_range_encode_tiled(torch.from_numpy(st.view(np.int32)).cuda(),
                                         torch.from_numpy(fr.view(np.int32)).cuda(), P, n_win, W, wl,
                                         validate=layout == "tile")
    if layout == "row":
        s_dev, f_dev, sw, sp = start, freq, W, 1
    else:
        s_dev, f_dev, sw, sp = start.T.copy(), freq.T.copy(), 1, n_win
    return L.lmgc_range_encode(torch.from_numpy(s_dev.view(np.int32)).cuda(),
                               torch.from_numpy(f_dev.view(np.int32)).cuda(), P, n_win, W, wl, sw, sp)


def check_codes(out, bitlen, start, freq, P, lens):
    payload = out.cpu().numpy().tobytes()
    bl = bitlen.cpu().numpy()
    off = 0
    for w in range(start.shape[0]):
        code, nbits = O.range_encode(start[w, :lens[w]], freq[w, :lens[w]], P)
        assert bl[w] == nbits, w
        assert payload[off: off + len(code)] == code, w
        off += len(code)
    assert off == len(payload)


@pytest.mark.parametrize("P,layout", [(16, "row"), (24, "pos"), (24, "row"), (30, "pos"), (16, "tile"), (24, "tile"),
                                      (30, "tile"), (7, "tile"), (16, "tile-trusted"), (24, "tile-trusted"),
                                      (30, "tile-trusted"), (7, "tile-trusted")])
def test_range_encode_bit_exact(P, layout):
    """Ragged windows (lengths 1..300, one of 17) over random integer CDFs, 70 windows (two full
    32-window blocks and a partial one), W = 300 (not a multiple of the 8-position tile group).
    Every freq is below 2^P (at least V symbols share the range), so the unchecked form applies."""
    rng = np.random.default_rng(P)
    n_win, W = 70, 300
    V = 32 if P <= 16 else 1000
    if P == 7:
        V = 100
    start, freq, lens = random_pairs(rng, n_win, W, P, V=V)
    lens = rng.integers(1, W + 1, n_win).astype(np.uint32)
    lens[0], lens[1], lens[-1] = W, 1, 17
    out, bitlen = coder(start, freq, P, n_win, W, lens, layout)
    check_codes(out, bitlen, start, freq, P, lens)


@pytest.mark.parametrize("layout", ["tile", "tile-trusted", "pos"])
@pytest.mark.parametrize("P", [16, 24])
def test_range_encode_carry_heavy(P, layout):
    """Streams built to carry: mostly tokens at the top of the range (start = T - freq) with small
    freq, so L's low bits fill with ones and additions carry into already completed words, some
    through whole words of ones; plus probability-one tokens (freq = T), which shift nothing."""
    rng = np.random.default_rng(100 + P)
    T = 1 << P
    n_win, W = 64, 512
    freq = rng.integers(1, 6, (n_win, W)).astype(np.int64)
    start = T - freq - rng.integers(0, 2, (n_win, W))
    low = rng.random((n_win, W)) < 0.08  # an occasional low symbol
    start = np.where(low, rng.integers(0, T // 2, (n_win, W)), start)
    one = rng.random((n_win, W)) < 0.05
    freq = np.where(one, T, freq)
    start = np.where(one, 0, np.clip(start, 0, T - freq))
    start, freq = start.astype(np.uint32), freq.astype(np.uint32)
    lens = np.full(n_win, W, np.uint32)
    out, bitlen = coder(start, freq, P, n_win, W, lens, layout)
    check_codes(out, bitlen, start, freq, P, lens)


def test_range_encode_many_windows_sampled():
    """A coder-only batch in the position-major layout: 8192 windows x 2048 tokens over
    vocab 32000 at P = 24; sampled windows are compared with the oracle."""
    rng = np.random.default_rng(11)
    n_win, W, P = 8192, 2048, 24
    start, freq, _ = random_pairs(rng, n_win, W, P)
    out, bitlen = L.lmgc_range_encode(torch.from_numpy(start.T.copy().view(np.int32)).cuda(),
                                      torch.from_numpy(freq.T.copy().view(np.int32)).cuda(), P, n_win, W, None, 1,
                                      n_win)
    bl = bitlen.cpu().numpy().astype(np.int64)
    offs = np.concatenate([[0], np.cumsum((bl + 7) // 8)])
    payload = out.cpu().numpy()
    assert offs[-1] == payload.size
    for w in [0, 1, 31, 32, 4095, 8191] + rng.integers(0, n_win, 10).tolist():
        code, nbits = O.range_encode(start[w], freq[w], P)
        assert bl[w] == nbits and payload[offs[w]:offs[w + 1]].tobytes() == code, w


def test_range_encode_rejects_bad_pairs():
    s = torch.zeros(4, dtype=torch.int32, device="cuda")
    f = torch.zeros(4, dtype=torch.int32, device="cuda")  # freq 0 is invalid
    with pytest.raises(L.LmgcError):
        L.lmgc_range_encode(s, f, 16, 1, 4, None, 4, 1)
    # window tiles: freq 0, freq above T, start + freq above T, each in its own window of a block
    T = 1 << 16
    for bad in [(0, 0), (0, T + 1), (T - 3, 4), (0xFFFFFFFF, 2)]:
        st = np.zeros((3, 20), np.uint32)
        fr = np.full((3, 20), 2, np.uint32)
        st[1, 13], fr[1, 13] = bad
        with pytest.raises(L.LmgcError) as e:
            L.lmgc_range_encode_tiled(torch.from_numpy(to_pair_tiles(st).view(np.int32)).cuda(),
                                      torch.from_numpy(to_pair_tiles(fr).view(np.int32)).cuda(), 16, 3, 20, None)
        assert e.value.status == L.ERR_INVALID, bad


def test_range_encode_tiled_rejects_misaligned_pairs():
    """The tiles are staged by bulk copies, whose sources must be 16-byte aligned: a pair array
    that starts 4 bytes into an allocation is refused on the host (INVALID), before any launch."""
    st = np.zeros((32, 8), np.uint32)
    fr = np.full((32, 8), 2, np.uint32)
    s = torch.from_numpy(np.concatenate([[0], to_pair_tiles(st)]).astype(np.uint32).view(np.int32)).cuda()
    f = torch.from_numpy(np.concatenate([[0], to_pair_tiles(fr)]).astype(np.uint32).view(np.int32)).cuda()
    for validate in (True, False):
        with pytest.raises(L.LmgcError) as e:
            L.lmgc_range_encode_tiled(s[1:], f[1:], 16, 32, 8, None, validate=validate)
        assert e.value.status == L.ERR_INVALID
    out, bitlen = L.lmgc_range_encode_tiled(s[1:].clone(), f[1:].clone(), 16, 32, 8, None)
    check_codes(out, bitlen, st, fr, 16, np.full(32, 8, np.uint32))


@pytest.mark.parametrize("sep_mode,V,P", [(0, 32, 16), (2, 1000, 20), (4, 32000, 24)])
def test_cdf_pairs_alphabet_bit_exact(sep_mode, V, P):
    """Restricted-alphabet pairs: the quantiser over each row's alphabet logits (ascending ids)
    and the token's index among them, bit-exact with the oracle's full quantiser applied to the
    gathered columns; a token outside the alphabet is CORRUPT."""
    ctx = L.Context(configs.with_(configs.TINY, vocab=V, cdf_bits=P, sep_mode=sep_mode, alphabet=1, batch_windows=1))
    A = np.array(O.alphabet_ids(sep_mode))
    rng = np.random.default_rng(V + sep_mode)
    rows = 2000
    z = logit_rows(rng, rows, V)
    z[5, A[3]] = 50.0            # the alphabet's own maximum far above the rest of it
    z[6, :] = -3.0
    z[6, A[-1]] = 9.0            # ... at its last id
    idx = rng.integers(0, A.size, rows)
    idx[6] = A.size - 1
    sym = A[idx].astype(np.uint16)
    dz = torch.from_numpy(z).cuda()
    st, fr = L.lmgc_cdf_pairs(ctx, dz, torch.from_numpy(sym.view(np.int16)).cuda())
    rs, rf = O.cdf_pairs(np.ascontiguousarray(z[:, A]), idx.astype(np.uint16), P)
    assert np.array_equal(st.cpu().numpy().view(np.uint32), rs)
    assert np.array_equal(fr.cpu().numpy().view(np.uint32), rf)
    bad = sym.copy()
    bad[7] = 19  # BOS is context only, never coded
    with pytest.raises(L.LmgcError) as e:
        L.lmgc_cdf_pairs(ctx, dz, torch.from_numpy(bad.view(np.int16)).cuda())
    assert e.value.status == L.ERR_CORRUPT
    ctx.close()
