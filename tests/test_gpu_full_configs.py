"""Parity at the workloads' full sizes, in the launch configuration the bench times (sampled
outputs the oracle can compute one by one, plus lossless round trips on sampled windows).

* TinyLlama shape, 64 windows per batch (the bench's batch): logits of sampled positions of a
  window in the middle of the batch against the fp64 oracle (<= 5e-2).
* Llama-2-7B shape (32 layers, d 4096, MHA, head dim 128, vocab 32000, 4096-token windows):
  sampled logits, and a KV-cached decode round trip of a partial window.
* The 8-bit lossy input (Eq. 4 codes of the top-10% ConvNet gradient) with 128 windows per
  batch: the whole input is encoded, sampled windows decoded.
* The whole ConvNet gradient (1,314 windows): encoded in 21 batches; the first, a middle and the
  last (partial) window decoded back; code lengths of sampled prefixes compared with the ideal
  length -sum log2(freq / T) under the oracle's own CDFs (within 0.5%).
* Full-width single layers over whole windows (every position, every one of the 32,000 logits,
  so every 64-key attention block and block boundary at the real head layouts): TinyLlama width
  (d 2048, 32/4 GQA heads, head dim 64) over a full 2048-token window and a partial one, with the
  container's size against the oracle's own encode of the same input (within 0.5%); Llama-2-7B
  width (d 4096, 32 heads MHA, head dim 128) over the first 1,024 positions of a 4096-token window."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2409_17836_gb300 import configs, inputs as I, lmgc as L
from tests._util import cpu_threads, oracle_config

pytestmark = pytest.mark.gpu


def dev(a):
    return torch.from_numpy(a.view(np.int32) if a.dtype == np.float32 else a.view(np.int16) if a.dtype == np.uint16
                            else a).cuda()


def decode(ctx, buf, ids):
    return L.lmgc_decode(ctx, torch.from_numpy(np.frombuffer(buf, np.uint8).copy()).cuda(), ids).cpu().numpy().view(
        np.uint16)


def test_tinyllama_bench_batch_sampled_logits():
    cfg = configs.TINYLLAMA  # batch_windows = 64, as timed by the bench
    ctx = L.Context(cfg)
    vals = I.convnet_gradient(0)
    tok = O.serialize(vals, 0)
    lg = L.lmgc_lm_probs(ctx, dev(tok), 0, 64)  # one full batch
    oc = oracle_config(cfg, n_threads=cpu_threads())
    for w in (37, 63):
        ref = O.window_logits(oc, tok[w * 2048:(w + 1) * 2048], 6)
        err = np.abs(lg[w, :6].cpu().numpy().astype(np.float64) - ref).max()
        assert err <= 5e-2, (w, err)
    ctx.close()


def test_llama2_7b_shape_sampled_logits_and_round_trip():
    cfg = configs.with_(configs.LLAMA2_7B, batch_windows=1)
    ctx = L.Context(cfg)
    vals = I.convnet_gradient(0)[:111]  # 999 tokens: one partial 4096-token window
    tok = O.serialize(vals, 0)
    lg = L.lmgc_lm_probs(ctx, dev(tok), 0, 1)[0, :4].cpu().numpy()
    ref = O.window_logits(oracle_config(cfg, n_threads=cpu_threads()), tok, 4)
    assert np.abs(lg.astype(np.float64) - ref).max() <= 5e-2
    buf = L.lmgc_encode(ctx, dev(vals)).cpu().numpy().tobytes()
    out = decode(ctx, buf, [0])[0, :tok.size]
    assert O.deserialize(out, 0, 0).tobytes() == vals.tobytes()
    ctx.close()


def test_lossy_full_input_round_trip():
    cfg = configs.TINYLLAMA_LOSSY
    ctx = L.Context(cfg)
    codes = I.lossy_codes(I.convnet_gradient(0))
    assert codes.size == 29895
    buf = L.lmgc_encode(ctx, torch.from_numpy(codes).cuda()).cpu().numpy().tobytes()
    h = O.parse_container(buf)
    assert h["n_win"] == 44 and h["n_tok"] == 3 * 29895
    tok = O.serialize(codes, 0)
    ids = [0, 21, 43]
    out = decode(ctx, buf, ids)
    for i, w in enumerate(ids):
        n = min(2048, tok.size - w * 2048)
        assert np.array_equal(out[i, :n], tok[w * 2048: w * 2048 + n]), w
    ctx.close()


def test_convnet_gradient_whole_encode_and_sampled_decode():
    cfg = configs.TINYLLAMA
    ctx = L.Context(cfg)
    vals = I.convnet_gradient(0)
    buf = L.lmgc_encode(ctx, dev(vals)).cpu().numpy().tobytes()
    h = O.parse_container(buf)
    assert h["n_win"] == 1314 and h["n_tok"] == 9 * vals.size
    tok = O.serialize(vals, 0)
    ids = [0, 657, 1313]
    out = decode(ctx, buf, ids)
    for i, w in enumerate(ids):
        n = min(2048, tok.size - w * 2048)
        assert np.array_equal(out[i, :n], tok[w * 2048: w * 2048 + n]), w
    # ideal code length of sampled prefixes: GPU logits vs oracle logits, each through the oracle
    # quantiser (the GPU's own quantiser is bit-exact with it given the same logits)
    oc = oracle_config(cfg, n_threads=cpu_threads())
    lg = L.lmgc_lm_probs(ctx, dev(tok), 657, 1)[0, :8].cpu().numpy()
    seg = tok[657 * 2048: 657 * 2048 + 8]
    st_g, fr_g = O.cdf_pairs(lg, seg, 24)
    st_o, fr_o, _ = O.window_pairs(oc, tok[657 * 2048:], 8)
    jg = -np.log2(fr_g / 2.0 ** 24).sum()
    jo = -np.log2(fr_o / 2.0 ** 24).sum()
    assert abs(jg - jo) <= 0.005 * jo, (jg, jo)
    ctx.close()


def test_tinyllama_width_whole_windows_logits_and_container_size():
    """One layer at TinyLlama width over a full 2048-token window and a 1,741-token partial one:
    every logit of every position within 5e-2 of the oracle (whose fp32-rounded logits drive its
    own quantiser), and the GPU container within 0.5% of the size of the oracle's container for
    the same input (Eq. 3's rate to within 0.5%)."""
    cfg = configs.with_(configs.TINYLLAMA, n_layers=1, batch_windows=2)
    ctx = L.Context(cfg)
    vals = I.convnet_gradient(0)[:421]  # 3,789 tokens: windows of 2048 and 1741
    tok = O.serialize(vals, 0)
    W = cfg.window
    lg = L.lmgc_lm_probs(ctx, dev(tok), 0, 2).cpu().numpy()
    gpu = L.lmgc_encode(ctx, dev(vals)).cpu().numpy().tobytes()
    ctx.close()
    oc = oracle_config(cfg, n_threads=cpu_threads())
    codes = []
    for w in range(2):
        seg = tok[w * W:(w + 1) * W]
        st, fr, lo = O.window_pairs(oc, seg, seg.size)
        err = np.abs(lg[w, :seg.size].astype(np.float64) - lo.astype(np.float64)).max(axis=1)
        assert err.max() <= 5e-2, (w, int(err.argmax()), float(err.max()))
        codes.append(O.range_encode(st, fr, cfg.cdf_bits))
    orc = O.build_container(oc, vals.size, tok.size, codes, O.window_crcs(tok, W))
    hg, ho = O.parse_container(gpu), O.parse_container(orc)
    for w in range(2):
        assert abs(int(hg["bitlen"][w]) - int(ho["bitlen"][w])) <= 0.005 * int(ho["bitlen"][w]), w
    assert abs(len(gpu) - len(orc)) <= 0.005 * len(orc), (len(gpu), len(orc))


def test_llama2_7b_width_first_1024_positions():
    """One layer at Llama-2-7B width (MHA, head dim 128) in a 4096-token window: every logit of the
    first 1,024 positions (16 key blocks) within 5e-2 of the fp64 oracle."""
    cfg = configs.with_(configs.LLAMA2_7B, n_layers=1, batch_windows=1)
    ctx = L.Context(cfg)
    tok = O.serialize(I.convnet_gradient(0)[:1000], 0)  # 9,000 tokens: windows 0, 1 and part of 2
    lg = L.lmgc_lm_probs(ctx, dev(tok), 1, 1)[0, :1024].cpu().numpy()
    ctx.close()
    ref = O.window_logits(oracle_config(cfg, n_threads=cpu_threads()), tok[4096:8192], 1024)
    err = np.abs(lg.astype(np.float64) - ref).max(axis=1)
    assert err.max() <= 5e-2, (int(err.argmax()), float(err.max()))
