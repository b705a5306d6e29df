"""Edge cases and the largest configurations, through the C ABI:

* empty inputs at every entry point that takes a count;
* degenerate coder windows of 0, 1 and 2 tokens against the oracle (Sec. 3 coder);
* the 64M-value Laplace configuration: its serialisation sampled against the oracle, and
  windows at the start, middle and end of its 294,912-window stream coded in place and matched
  against a standalone encode of the same tokens, then decoded back (lossless);
* the coder at the size of the coder-only benchmark (2^20 windows x 2048 tokens, vocabulary
  32000, P = 24): sampled windows bit-exact against the oracle, and every window's length within
  the Sec. 3 bound J + 1 - eps < l <= J + 2 + eps."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2409_17836_gb300 import configs, inputs as I, lmgc as L
from tests._util import random_pairs, to_pair_tiles

pytestmark = pytest.mark.gpu


def test_empty_inputs():
    ctx = L.Context(configs.with_(configs.TINY, batch_windows=2))
    empty = torch.empty(0, dtype=torch.int32, device="cuda")
    assert L.lmgc_serialize(ctx, empty).numel() == 0
    with pytest.raises(L.LmgcError) as e:
        L.lmgc_encode(ctx, empty)
    assert e.value.status == L.ERR_INVALID
    # a coder call with no windows writes nothing
    out, bl = L.lmgc_range_encode(empty, empty, 16, 0, 256, None, 1, 0)
    assert out.numel() == 0 and bl.numel() == 0
    # CDF pairs of zero rows, and a decode of no windows from a valid container
    z = torch.empty((0, 32), dtype=torch.float32, device="cuda")
    st, fr = L.lmgc_cdf_pairs(ctx, z, torch.empty(0, dtype=torch.int16, device="cuda"))
    assert st.numel() == 0 and fr.numel() == 0
    vals = I.tiny_gradient(0)[:50]
    buf = L.lmgc_encode(ctx, torch.from_numpy(vals.view(np.int32).copy()).cuda())
    assert L.lmgc_decode(ctx, buf, []).shape[0] == 0
    ctx.close()


@pytest.mark.parametrize("tiled", [False, True])
@pytest.mark.parametrize("P", [16, 24])
def test_degenerate_window_lengths(P, tiled):
    """Windows of 0, 1, 2, 7, 8, 9 and W tokens in one call (row-major strides, or window tiles
    whose 8-position groups end mid-window): each code equals the oracle's code of the same prefix
    (a window of no tokens codes to the 2 termination bits)."""
    rng = np.random.default_rng(P)
    W = 64
    lens = np.array([0, 1, 2, W, 1, 0, 7, 8, 9], dtype=np.uint32)
    start, freq, _ = random_pairs(rng, lens.size, W, P, V=32 if P == 16 else 32000, layout="row")
    wl = torch.from_numpy(lens.view(np.int32)).cuda()
    if tiled:
        out, bitlen = L.lmgc_range_encode_tiled(torch.from_numpy(to_pair_tiles(start).view(np.int32)).cuda(),
                                                torch.from_numpy(to_pair_tiles(freq).view(np.int32)).cuda(), P,
                                                lens.size, W, wl)
    else:
        out, bitlen = L.lmgc_range_encode(torch.from_numpy(start.view(np.int32)).cuda(),
                                          torch.from_numpy(freq.view(np.int32)).cuda(), P, lens.size, W, wl, W, 1)
    bl = bitlen.cpu().numpy().astype(np.int64)
    payload = out.cpu().numpy().tobytes()
    off = 0
    for w, n in enumerate(lens):
        code, nbits = O.range_encode(start[w, :n], freq[w, :n], P)
        assert bl[w] == nbits, (w, n)
        assert payload[off:off + len(code)] == code, (w, n)
        off += len(code)
    assert off == len(payload)
    assert bl[0] == 2 and bl[5] == 2


@pytest.fixture(scope="module")
def laplace():
    return I.laplace_gradient()


def test_laplace_64m_serialise_sampled(laplace):
    vals = laplace
    ctx = L.Context(configs.with_(configs.TINYLLAMA, n_layers=1, batch_windows=1))
    d = torch.from_numpy(vals.view(np.int32)).cuda()
    tok = L.lmgc_serialize(ctx, d)
    assert tok.numel() == 9 * vals.size == 603_979_776
    rng = np.random.default_rng(64)
    idx = np.unique(np.concatenate([[0, 1, vals.size - 1], rng.integers(0, vals.size, 20000)]))
    got = tok.view(-1, 9)[torch.from_numpy(idx).cuda()].cpu().numpy().view(np.uint16)
    ref = O.serialize(vals[idx], 0).reshape(-1, 9)
    assert np.array_equal(got, ref)
    ctx.close()


def test_laplace_64m_windows_in_place_and_round_trip(laplace):
    """Windows w, w+1 for w at the start, middle and end of the 64M-value stream (multiples of 9,
    so that they start on a value): coded in place from the whole stream they equal the codes of
    a standalone encode of the values they cover, which decodes back to those tokens."""
    vals = laplace
    cfg = configs.with_(configs.TINYLLAMA, batch_windows=2)
    ctx = L.Context(cfg)
    W = cfg.window
    n_win = 9 * vals.size // W
    assert n_win == 294_912
    d = torch.from_numpy(vals.view(np.int32)).cuda()
    for w in (0, 9 * (n_win // 18), 9 * ((n_win - 2) // 9)):
        pay, bl, crc = L.lmgc_encode_windows(ctx, d, w, 2)
        v0 = w * W // 9
        sub = vals[v0: v0 + 2 * W // 9 + 1]  # the values of windows w and w + 1 (and one more token run)
        ds = torch.from_numpy(sub.view(np.int32).copy()).cuda()
        buf = L.lmgc_encode(ctx, ds)
        h = O.parse_container(buf.cpu().numpy().tobytes())
        assert np.array_equal(h["bitlen"][:2], bl.cpu().numpy().astype(np.int64)), w
        assert np.array_equal(h["crc_tok"][:2], crc.cpu().numpy().view(np.uint32)), w
        raw = buf.cpu().numpy().tobytes()
        assert raw[h["offsets"][0]: h["offsets"][2]] == pay.cpu().numpy().tobytes(), w
        toks = L.lmgc_decode(ctx, buf, [0, 1]).cpu().numpy().view(np.uint16).reshape(-1)
        assert np.array_equal(toks, O.serialize(sub, 0)[: 2 * W]), w
    ctx.close()


def test_range_encode_coder_benchmark_size():
    """2^20 windows x 2048 tokens (2^31 tokens) over 256 random integer CDFs of vocabulary 32000
    at P = 24, in the window tiles the encode path and the coder microbenchmark use: sampled
    windows bit-exact against the oracle, and every window's bit length within the coding bound of
    its own (start, freq) stream."""
    n_win, W, P, V = 1 << 20, 2048, 24, 32000
    T = 1 << P
    G, NB = W // 8, n_win // 32
    rng = np.random.default_rng(2048)
    cdfs = []
    for _ in range(256):
        w = rng.exponential(size=V) ** 2
        f = 1 + np.floor(w / w.sum() * (T - V)).astype(np.int64)
        f[np.argmax(f)] += T - f.sum()
        cdfs.append(np.concatenate([[0], np.cumsum(f)]))
    cdf = torch.from_numpy(np.array(cdfs, dtype=np.int32)).cuda()  # [256][V + 1]
    g = torch.Generator(device="cuda").manual_seed(2048)
    # tiles as [window block][position group][window in block][position in group]
    start = torch.empty((NB, G, 32, 8), dtype=torch.int32, device="cuda")
    freq = torch.empty((NB, G, 32, 8), dtype=torch.int32, device="cuda")
    assert start.numel() == L.lmgc_pair_tile_elems(n_win, W)
    flat = cdf.view(-1)
    for g0 in range(0, G, 16):  # 128 positions at a time keep the temporaries small
        row = torch.randint(0, 256, (128, n_win), device="cuda", generator=g)
        sym = torch.randint(0, V, (128, n_win), device="cuda", generator=g)
        lo = flat[row * (V + 1) + sym]
        fr = flat[row * (V + 1) + sym + 1] - lo
        # [position][window] -> [block][group][window in block][position in group]
        start[:, g0:g0 + 16] = lo.view(16, 8, NB, 32).permute(2, 0, 3, 1)
        freq[:, g0:g0 + 16] = fr.view(16, 8, NB, 32).permute(2, 0, 3, 1)
        del row, sym, lo, fr
    out, bitlen = L.lmgc_range_encode_tiled(start, freq, P, n_win, W, None)
    bl = bitlen.cpu().numpy().astype(np.int64)
    # the bound for every window: J = -sum log2(freq / T), eps <= n 2^(P-60) 1.45
    J = torch.zeros((NB, 32), dtype=torch.float64, device="cuda")
    for g0 in range(0, G, 16):
        J -= torch.log2(freq[:, g0:g0 + 16].double() / T).sum(dim=(1, 3))
    J = J.view(-1).cpu().numpy()
    eps = W * 2.0 ** (P - 60) * 1.45
    assert np.all(bl > J + 1 - eps) and np.all(bl <= J + 2 + eps)
    offs = np.concatenate([[0], np.cumsum((bl + 7) // 8)])
    assert offs[-1] == out.numel()
    for w in [0, 1, 31, 32, n_win // 2, n_win - 1] + rng.integers(0, n_win, 8).tolist():
        s = start[w // 32, :, w % 32, :].reshape(-1).cpu().numpy().view(np.uint32)
        f = freq[w // 32, :, w % 32, :].reshape(-1).cpu().numpy().view(np.uint32)
        code, nbits = O.range_encode(s, f, P)
        assert bl[w] == nbits, w
        assert out[offs[w]: offs[w + 1]].cpu().numpy().tobytes() == code, w
