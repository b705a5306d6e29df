"""The model's dense contraction (lmgc_gemm): C = A . B^T for the linear layers and the
vocabulary projection of the Eq. 2 model, compared with the fp64 definition. A bf16-weight model
computes with fp16 operands on the tcgen05 kernel (its bf16 weight values are exact in fp16); an
fp32 model with fp32 operands on the tcgen05 kernel in three-pass TF32 form. Bound per element:
accumulation error <= 2^-19 * sum_k |a_k b_k| on the tensor cores (their fp32 accumulation aligns
products with truncation, measured at up to 1.4 x 2^-22 * sum |a b|); for the TF32 form also the
split's terms (see test_gemm_fp32_tf32x3); plus one fp16 rounding of the output for epilogues 0
and 3: 2^-11 relative (2^-10 allowed), and below 2^-14 the fixed 2^-24 spacing of fp16
subnormals (2^-25 absolute)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2409_17836_gb300 import configs, lmgc as L

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx_f16():
    c = L.Context(L.ModelConfig(n_layers=1, d_model=64, n_heads=1, n_kv_heads=1, d_ffn=64, vocab=32, dtype=L.BF16,
                                window=64, cdf_bits=16))
    yield c
    c.close()


def run(ctx, M, N, K, epi, seed=0, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    a = (torch.randn(M, K, generator=g) * scale).to(torch.float16)
    b = (torch.randn(N, K, generator=g) * scale).to(torch.float16)
    c0 = torch.randn(M, N, generator=g)
    if epi == 0:
        c = torch.empty(M, N, dtype=torch.float16, device="cuda")
    else:
        c = c0.clone().cuda()
    L.lmgc_gemm(ctx, a.cuda(), b.cuda(), c, epi)
    af, bf = a.float().numpy(), b.float().numpy()
    ref = O.gemm_nt(af, bf)
    bound = 2.0 ** -19 * O.gemm_nt(np.abs(af), np.abs(bf)) + 1e-30
    if epi in (1, 5):
        ref = ref + c0.numpy().astype(np.float64)
        bound += 2.0 ** -23 * np.abs(ref)
    got = c.float().cpu().numpy().astype(np.float64)
    if epi == 0:
        bound += 2.0 ** -10 * np.abs(ref) + 2.0 ** -25
    err = np.abs(got - ref)
    assert np.all(err <= bound), float((err / bound).max())
    return c


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (300, 520, 136), (1, 256, 2048), (7, 2560, 2048),
                                   (1000, 2048, 5632), (2048, 32000, 2048)])
@pytest.mark.parametrize("epi", [0, 1, 2])
def test_gemm_tc_shapes(ctx_f16, M, N, K, epi):
    if M * N > 2048 * 32000 // 2 and epi != 2:
        pytest.skip("the vocabulary shape is checked with the fp32 epilogue only")
    run(ctx_f16, M, N, K, epi, seed=M + N + K)


@pytest.mark.parametrize("M,N,K", [(300, 520, 136), (7, 2560, 2048), (1000, 2048, 2048)])
def test_gemm_tc_wide_residual_epilogue(ctx_f16, M, N, K):
    """epi 5 (the residual add through 8 epilogue warps) meets the epi 1 bound and equals epi 1
    bit for bit: the same products accumulate in the same order, one fp32 add per element."""
    c5 = run(ctx_f16, M, N, K, 5, seed=M + N + K)
    c1 = run(ctx_f16, M, N, K, 1, seed=M + N + K)
    assert torch.equal(c1, c5)


def test_gemm_tc_row_invariance(ctx_f16):
    """A row's result does not depend on M or on the row's place in a tile (the decoder relies on
    this): rows computed alone equal the same rows inside a 1000-row product, bit for bit."""
    g = torch.Generator().manual_seed(5)
    a = torch.randn(1000, 2048, generator=g).to(torch.float16).cuda()
    b = torch.randn(2560, 2048, generator=g).to(torch.float16).cuda()
    full = torch.empty(1000, 2560, device="cuda")
    L.lmgc_gemm(ctx_f16, a, b, full, 2)
    for r in [0, 1, 127, 128, 517, 999]:
        one = torch.empty(1, 2560, device="cuda")
        L.lmgc_gemm(ctx_f16, a[r:r + 1].contiguous(), b, one, 2)
        assert torch.equal(one[0], full[r]), r
    part = torch.empty(3, 2560, device="cuda")
    L.lmgc_gemm(ctx_f16, a[517:520].contiguous(), b, part, 2)
    assert torch.equal(part, full[517:520])


@pytest.fixture(scope="module")
def ctx_f32():
    c = L.Context(configs.with_(configs.TINY, batch_windows=1))
    yield c
    c.close()


@pytest.mark.parametrize("M,N,K", [(300, 520, 136), (128, 128, 32), (1, 384, 128), (36864 // 9, 1024, 128),
                                   (257, 32, 512), (5, 17, 8), (1000, 130, 520)])
@pytest.mark.parametrize("epi", [0, 1, 2])
def test_gemm_fp32_tf32x3(ctx_f32, M, N, K, epi):
    """An fp32 model's contraction on the tcgen05 TF32 kernel in three passes (lo_A hi_B + hi_A lo_B
    + hi_A hi_B, hi = x with its low 13 bits cleared). Bound per element: the dropped lo_A lo_B
    term (< 2^-20 |a b|), the truncation of each lo to TF32 in the two cross terms (< 2^-20 |a b|
    each) and the tensor cores' fp32 accumulation (2^-19 sum |a b|, as for the fp16 kernel):
    2^-19 + 3 2^-20 < 2^-17 of sum_k |a_k b_k|, plus one fp32 rounding of C += for epilogue 1.
    Shapes with ragged M and N tiles, N <= 32 (the narrow tile), K not a multiple of the 32-wide K
    step, and M = 1 (a decode step)."""
    g = torch.Generator().manual_seed(M + N + K + epi)
    a = torch.randn(M, K, generator=g)
    b = torch.randn(N, K, generator=g)
    c0 = torch.randn(M, N, generator=g)
    c = c0.clone().cuda() if epi == 1 else torch.full((M, N), float("nan"), device="cuda")
    L.lmgc_gemm(ctx_f32, a.cuda(), b.cuda(), c, epi)
    an, bn = a.numpy().astype(np.float64), b.numpy().astype(np.float64)
    ref = O.gemm_nt(an, bn)
    bound = 2.0 ** -17 * O.gemm_nt(np.abs(an), np.abs(bn)) + 1e-30
    if epi == 1:
        ref = ref + c0.numpy().astype(np.float64)
        bound += 2.0 ** -23 * np.abs(ref)
    got = c.cpu().numpy().astype(np.float64)
    err = np.abs(got - ref)
    assert np.all(err <= bound), float((err / bound).max())


def test_gemm_fp32_rows_independent_of_m(ctx_f32):
    """Each row of C is the same whatever M and the row's place in a tile (the decoder's one-row
    steps reproduce the encoder's logits bit for bit)."""
    g = torch.Generator().manual_seed(7)
    a = torch.randn(700, 128, generator=g).cuda()
    b = torch.randn(384, 128, generator=g).cuda()
    full = torch.empty(700, 384, device="cuda")
    L.lmgc_gemm(ctx_f32, a, b, full, 2)
    for r in (0, 127, 128, 333, 699):
        one = torch.empty(1, 384, device="cuda")
        L.lmgc_gemm(ctx_f32, a[r:r + 1].contiguous(), b, one, 2)
        assert torch.equal(one[0], full[r])
    part = torch.empty(3, 384, device="cuda")
    L.lmgc_gemm(ctx_f32, a[517:520].contiguous(), b, part, 2)
    assert torch.equal(part, full[517:520])


def test_gemm_rejects_misaligned_operands(ctx_f32):
    """TMA reads A and B and the epilogues store C with 16-byte vectors: an operand 4 bytes off a
    16-byte boundary is refused (INVALID) before any launch."""
    a = torch.randn(9, 64, device="cuda")
    b = torch.randn(32, 64, device="cuda")
    c = torch.zeros(8 * 32 + 1, device="cuda")
    for args in ((a.view(-1)[1:1 + 8 * 64].view(8, 64), b[:32], c[:256].view(8, 32)),
                 (a[:8], b.view(-1)[1:1 + 31 * 64].view(31, 64), c[:248].view(8, 31)),
                 (a[:8], b, c[1:].view(8, 32))):
        with pytest.raises(L.LmgcError) as e:
            L.lmgc_gemm(ctx_f32, *args, 2)
        assert e.value.status == L.ERR_INVALID


def test_gemm_rejects_bad_k(ctx_f16):
    a = torch.zeros(4, 12, dtype=torch.float16, device="cuda")
    with pytest.raises(L.LmgcError):
        L.lmgc_gemm(ctx_f16, a, a, torch.zeros(4, 4, device="cuda"), 2)


@pytest.mark.parametrize("M,F,K", [(300, 512, 136), (1, 5632, 2048), (1000, 1408, 2048)])
def test_gemm_tc_swiglu_epilogue(ctx_f16, M, F, K):
    """Epilogue 3: gate/up rows interleaved in 128-row blocks, C = silu(gate) * up in fp16."""
    g = torch.Generator().manual_seed(F + M)
    a = torch.randn(M, K, generator=g).to(torch.float16)
    wg = (torch.randn(F, K, generator=g) * 0.05).to(torch.float16)
    wu = (torch.randn(F, K, generator=g) * 0.05).to(torch.float16)
    inter = torch.empty(2 * F, K, dtype=torch.float16)
    for t in range(F // 128):
        inter[256 * t: 256 * t + 128] = wg[128 * t: 128 * t + 128]
        inter[256 * t + 128: 256 * t + 256] = wu[128 * t: 128 * t + 128]
    c = torch.empty(M, F, dtype=torch.float16, device="cuda")
    L.lmgc_gemm(ctx_f16, a.cuda(), inter.cuda(), c, 3)
    af = a.float().numpy()
    gr = O.gemm_nt(af, wg.float().numpy())
    ur = O.gemm_nt(af, wu.float().numpy())
    ref = O.swiglu(gr, ur)
    eg = 2.0 ** -19 * O.gemm_nt(np.abs(af), np.abs(wg.float().numpy()))
    eu = 2.0 ** -19 * O.gemm_nt(np.abs(af), np.abs(wu.float().numpy()))
    silu = gr / (1 + np.exp(-gr))
    bound = 1.1 * np.abs(ur) * eg + np.abs(silu) * eu + 2.0 ** -10 * np.abs(ref) + 2.0 ** -25
    err = np.abs(c.float().cpu().numpy() - ref)
    assert np.all(err <= bound), float((err / bound).max())
