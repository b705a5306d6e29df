"""Pins of the oracle LM prior (Eq. 1 / Eq. 2 with a Llama-family decoder, Sec. 5.1).

The paper prints no logits, so the oracle is pinned by: the published splitmix64 test vector;
torch library routines (rms_norm, scaled_dot_product_attention, silu, linear, embedding) in
fp64; RoPE's closed-form angles and its relative-position property; causality; zero weights;
and KV-cached feeding equal to the one-shot forward."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O

TINY = dict(n_layers=2, d_model=64, n_heads=4, n_kv_heads=2, d_ffn=96, vocab=24, window=40, cdf_bits=16)


def cfg(**kw):
    base = dict(TINY, bf16=False, weight_seed=7, init_std=0.02)
    base.update(kw)
    return O.OracleConfig(**base)


def test_splitmix64_published_vector():
    # Vigna's splitmix64 reference: seeded with 1234567 the first five outputs are these
    # (the state advances by 0x9E3779B97F4A7C15 before each mix).
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423, 4593380528125082431,
              16408922859458223821]
    s = 1234567
    for e in expect:
        assert O.splitmix64(s) == e
        s = (s + 0x9E3779B97F4A7C15) % (1 << 64)


def test_weights_distribution_and_bf16():
    w = O.weight_tensor(3, 5, 200000, 0.02, False)
    a = np.float32(0.02 * math.sqrt(3.0))
    assert np.abs(w).max() <= a
    assert abs(w.mean()) < 2e-4
    assert abs(w.std() - 0.02) < 2e-4
    wb = O.weight_tensor(3, 5, 200000, 0.02, True)
    # round-to-nearest-even to bf16 equals torch's conversion
    ref = torch.from_numpy(w).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(wb, ref)
    # different tensor ids and seeds give different streams
    assert not np.array_equal(w[:100], O.weight_tensor(3, 6, 100, 0.02, False))
    assert not np.array_equal(w[:100], O.weight_tensor(4, 5, 100, 0.02, False))
    assert np.all(O.weight_tensor(3, 5, 100, 0.0, False) == 0)


def test_rmsnorm_vs_torch():
    x = np.random.default_rng(0).normal(size=(7, 33)) * 3
    y = O.rmsnorm(x, 1e-5)
    ref = F.rms_norm(torch.from_numpy(x), (33,), eps=1e-5).numpy()
    np.testing.assert_allclose(y, ref, rtol=1e-13, atol=1e-14)


def test_attention_vs_torch_sdpa():
    rng = np.random.default_rng(1)
    n, nq, nkv, hd = 19, 4, 2, 8
    q = rng.normal(size=(n, nq * hd))
    k = rng.normal(size=(n, nkv * hd))
    v = rng.normal(size=(n, nkv * hd))
    o = O.attention(q, k, v, nq, nkv)
    tq = torch.from_numpy(q).view(n, nq, hd).transpose(0, 1)
    tk = torch.from_numpy(k).view(n, nkv, hd).repeat_interleave(nq // nkv, dim=1).transpose(0, 1)
    tv = torch.from_numpy(v).view(n, nkv, hd).repeat_interleave(nq // nkv, dim=1).transpose(0, 1)
    ref = F.scaled_dot_product_attention(tq[None], tk[None], tv[None], is_causal=True)[0]
    np.testing.assert_allclose(o, ref.transpose(0, 1).reshape(n, nq * hd).numpy(), rtol=1e-12, atol=1e-12)
    # rows fed later (p0 > 0) see the same keys as in one shot
    o2 = O.attention(q[10:], k, v, nq, nkv, p0=10)
    np.testing.assert_array_equal(o2, o[10:])


def test_rope_closed_forms_and_relative_property():
    theta = 10000.0
    # hd = 2: one pair rotated by pos radians
    x = np.array([[1.0, 0.0]] * 3)
    y = O.rope(x, np.array([0, 1, 5]), 1, theta)
    np.testing.assert_allclose(y, [[1, 0], [math.cos(1), math.sin(1)], [math.cos(5), math.sin(5)]], atol=1e-15)
    # hd = 4: pair (0, 2) at angle pos, pair (1, 3) at angle pos * theta^(-1/2)
    x = np.array([[1.0, 1.0, 0.0, 0.0]])
    y = O.rope(x, np.array([3]), 1, theta)
    np.testing.assert_allclose(y[0], [math.cos(3), math.cos(0.03), math.sin(3), math.sin(0.03)], atol=1e-15)
    # relative position: <R(m) q, R(n) k> depends on m - n only; norms preserved
    rng = np.random.default_rng(2)
    hd = 16
    q, k = rng.normal(size=(1, hd)), rng.normal(size=(1, hd))
    dots = []
    for m, nn in [(5, 2), (9, 6), (103, 100)]:
        dots.append(float((O.rope(q, np.array([m]), 1, theta) @ O.rope(k, np.array([nn]), 1, theta).T)[0, 0]))
    np.testing.assert_allclose(dots, dots[0], rtol=1e-10)
    np.testing.assert_allclose(np.linalg.norm(O.rope(q, np.array([77]), 1, theta)), np.linalg.norm(q))


def test_swiglu_vs_torch():
    rng = np.random.default_rng(3)
    g, u = rng.normal(size=50) * 4, rng.normal(size=50)
    ref = (F.silu(torch.from_numpy(g)) * torch.from_numpy(u)).numpy()
    np.testing.assert_allclose(O.swiglu(g, u), ref, rtol=1e-13, atol=1e-15)


def torch_forward(c: O.OracleConfig, tok_in: np.ndarray) -> np.ndarray:
    """The same Llama decoder composed from torch library routines in fp64 (RoPE as complex
    multiplication), weights from the oracle's generator."""
    d, nq, nkv, Fd, V = c.d_model, c.n_heads, c.n_kv_heads, c.d_ffn, c.vocab
    hd = d // nq
    n = tok_in.size

    def W(tid, shape):
        w = O.weight_tensor(c.weight_seed, tid, int(np.prod(shape)), c.init_std, c.bf16)
        return torch.from_numpy(w.astype(np.float64)).reshape(shape)

    def rope(x, heads):
        x = x.view(n, heads, hd)
        z = torch.complex(x[..., : hd // 2], x[..., hd // 2:])
        freq = c.rope_theta ** (-2.0 * torch.arange(hd // 2, dtype=torch.float64) / hd)
        ang = torch.arange(n, dtype=torch.float64)[:, None] * freq[None, :]
        z = z * torch.polar(torch.ones_like(ang), ang)[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    x = F.embedding(torch.from_numpy(tok_in.astype(np.int64)), W(0, (V, d)))
    for l in range(c.n_layers):
        t = 1 + 7 * l
        h = F.rms_norm(x, (d,), eps=c.rms_eps)
        q = rope(F.linear(h, W(t, (nq * hd, d))), nq)
        k = rope(F.linear(h, W(t + 1, (nkv * hd, d))), nkv)
        v = F.linear(h, W(t + 2, (nkv * hd, d))).view(n, nkv, hd)
        g = nq // nkv
        o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.repeat_interleave(g, 1).transpose(0, 1)[None],
                                           v.repeat_interleave(g, 1).transpose(0, 1)[None], is_causal=True)[0]
        x = x + F.linear(o.transpose(0, 1).reshape(n, d), W(t + 3, (d, nq * hd)))
        h = F.rms_norm(x, (d,), eps=c.rms_eps)
        a = F.silu(F.linear(h, W(t + 4, (Fd, d)))) * F.linear(h, W(t + 5, (Fd, d)))
        x = x + F.linear(a, W(t + 6, (d, Fd)))
    h = F.rms_norm(x, (d,), eps=c.rms_eps)
    return F.linear(h, W(1 + 7 * c.n_layers, (V, d))).numpy()


@pytest.mark.parametrize("bf16", [False, True])
def test_forward_vs_torch_composition(bf16):
    c = cfg(bf16=bf16, init_std=0.2)
    rng = np.random.default_rng(4)
    win = rng.integers(0, 20, 30).astype(np.uint16)
    lg = O.window_logits(c, win, 30)
    ref = torch_forward(c, np.concatenate([[O.TOK_BOS], win[:29]]))
    np.testing.assert_allclose(lg, ref, rtol=1e-9, atol=1e-11)
    assert np.abs(lg).max() > 0.1


def test_causality_and_kv_cache():
    c = cfg()
    rng = np.random.default_rng(5)
    win = rng.integers(0, 20, 25).astype(np.uint16)
    lg = O.window_logits(c, win, 25)
    win2 = win.copy()
    win2[12] = (win2[12] + 1) % 20
    lg2 = O.window_logits(c, win2, 25)
    # position i reads input tokens BOS, t_0..t_{i-1}: changing t_12 leaves positions <= 12 equal
    assert np.array_equal(lg[:13], lg2[:13])
    assert not np.allclose(lg[13:], lg2[13:])
    # feeding one position at a time through the KV cache equals the one-shot forward
    m = O.OracleLM(c, 25)
    inp = np.concatenate([[O.TOK_BOS], win[:24]]).astype(np.uint16)
    step = np.concatenate([m.feed(inp[:7])] + [m.feed(inp[i:i + 1]) for i in range(7, 25)])
    np.testing.assert_array_equal(step, lg)


def test_zero_weights_give_zero_logits():
    c = cfg(init_std=0.0)
    lg = O.window_logits(c, np.arange(10, dtype=np.uint16), 10)
    assert np.all(lg == 0.0)


def test_one_layer_one_head_two_positions_by_hand():
    """A 1-layer, 1-head, W = 2 model written out scalar by scalar (plain Python floats, no
    library routine): position 0 sees only itself, so its attention output is v_0; position 1
    mixes v_0 and v_1 with the softmax of its two scaled scores; RoPE turns the pairs (i, i + hd/2)
    of position 1 by 1 * theta^(-2i/hd) radians and leaves position 0 as it is."""
    d, hd, Fd, V = 4, 4, 3, 20
    c = cfg(n_layers=1, d_model=d, n_heads=1, n_kv_heads=1, d_ffn=Fd, vocab=V, window=2, init_std=0.5)
    t0, t1 = 7, 3

    def W(tid, rows, cols):
        w = O.weight_tensor(c.weight_seed, tid, rows * cols, c.init_std, False).astype(np.float64).tolist()
        return [w[r * cols:(r + 1) * cols] for r in range(rows)]

    def matvec(M, x):
        return [sum(M[r][j] * x[j] for j in range(len(x))) for r in range(len(M))]

    def norm(x):
        s = 1.0 / math.sqrt(sum(v * v for v in x) / len(x) + c.rms_eps)
        return [v * s for v in x]

    def rope(x, pos):
        out = list(x)
        for i in range(hd // 2):
            ang = pos * c.rope_theta ** (-2.0 * i / hd)
            a, b = x[i], x[i + hd // 2]
            out[i] = a * math.cos(ang) - b * math.sin(ang)
            out[i + hd // 2] = b * math.cos(ang) + a * math.sin(ang)
        return out

    E, Wq, Wk, Wv, Wo = W(0, V, d), W(1, hd, d), W(2, hd, d), W(3, hd, d), W(4, d, hd)
    Wg, Wu, Wd, Wh = W(5, Fd, d), W(6, Fd, d), W(7, d, Fd), W(8, V, d)
    xs = [list(E[O.TOK_BOS]), list(E[t0])]  # inputs: BOS, then the window's first token
    ns = [norm(x) for x in xs]
    q = [rope(matvec(Wq, ns[p]), p) for p in range(2)]
    k = [rope(matvec(Wk, ns[p]), p) for p in range(2)]
    v = [matvec(Wv, ns[p]) for p in range(2)]
    s0 = sum(q[1][i] * k[0][i] for i in range(hd)) / math.sqrt(hd)
    s1 = sum(q[1][i] * k[1][i] for i in range(hd)) / math.sqrt(hd)
    w0 = 1.0 / (1.0 + math.exp(s1 - s0))
    att = [v[0], [w0 * v[0][i] + (1.0 - w0) * v[1][i] for i in range(hd)]]
    logits = []
    for p in range(2):
        x = [xs[p][i] + o for i, o in enumerate(matvec(Wo, att[p]))]
        n2 = norm(x)
        g, u = matvec(Wg, n2), matvec(Wu, n2)
        a = [g[j] / (1.0 + math.exp(-g[j])) * u[j] for j in range(Fd)]
        x = [x[i] + o for i, o in enumerate(matvec(Wd, a))]
        logits.append(matvec(Wh, norm(x)))
    lg = O.window_logits(c, np.array([t0, t1], dtype=np.uint16), 2)
    # fp64 on both sides, different operation order: agreement to rounding (logits are O(1))
    np.testing.assert_allclose(lg, np.array(logits), rtol=1e-10, atol=1e-12)
    assert np.abs(lg).max() > 0.1
