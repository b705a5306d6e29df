"""The Sec. 5.4 compatibility inputs one at a time (the f3 sweep): Eq. 4 quantisation to 16, 8 and
1 bits over every value, magnitude sparsification that keeps fp32 values, and the byte stream
that carries 16-bit indices (4 hex digits per index through 2-byte groups). Worked by hand."""
import numpy as np

import oracle as O
from paper_2409_17836_gb300 import inputs as I


def test_eq4_worked_examples():
    v = np.array([-1.0, 0.0, 3.0], dtype=np.float32)
    # (v - min) / (max - min) * (2^n - 1): 0, 0.25, 1 of the range
    assert I.quantized_codes(v, 16).tolist() == [0, 16384, 65535]  # 16383.75 rounds up
    assert I.quantized_codes(v, 8).tolist() == [0, 64, 255]        # 63.75
    assert I.quantized_codes(v, 16).dtype == np.uint16 and I.quantized_codes(v, 8).dtype == np.uint8
    w = np.array([-2.0, 0.5, 3.0], dtype=np.float32)
    assert I.quantized_codes(w, 1).tolist() == [0, 0, 1]             # 0.5 rounds to even


def test_sparsified_keeps_largest_in_index_order():
    g = np.array([0.1, -5.0, 2.0, 2.0, -2.0, 0.0, 7.0, -0.2], dtype=np.float32)
    # |v| ranks: 7 (idx 6), 5 (idx 1), then the tie 2.0 / 2.0 / -2.0 at indices 2, 3, 4
    assert I.sparsified(g, 0.5).tolist() == [-5.0, 2.0, 2.0, 7.0]   # keeps indices 1, 2, 3, 6
    assert I.sparsified(g, 0.25).tolist() == [-5.0, 7.0]
    assert I.sparsified(g, 0.5).dtype == np.float32


def test_16bit_codes_as_byte_pairs():
    b, group = I.code_bytes(np.array([0x1234, 0xABCD, 0x0007], dtype=np.uint16))
    assert group == 2 and b.tolist() == [0x12, 0x34, 0xAB, 0xCD, 0x00, 0x07]
    tok = O.serialize(b, 0, group, 0)
    assert tok.tolist() == [1, 2, 3, 4, 16, 10, 11, 12, 13, 16, 0, 0, 0, 7, 16]
    assert np.array_equal(O.deserialize(tok, 1, 0, group, 0), b)
    c, g8 = I.code_bytes(np.array([5, 250], dtype=np.uint8))
    assert g8 == 0 and c.tolist() == [5, 250]


def test_lossy_codes_top_k_and_eq4_ends():
    """The lossy input (top 10% by magnitude, then 8-bit Eq. 4 over the kept values): the kept
    values stay in index order, a magnitude tie goes to the lower index, the kept minimum codes to
    0 and the maximum to 255, and a value in between to rint of its place in the range."""
    g = np.zeros(40, dtype=np.float32)
    g[[3, 9, 17, 25, 31]] = [-4.0, 1.0, 6.0, -1.0, 2.0]  # |1.0| ties at indices 9 and 25
    # k = floor(0.1 * 40) = 4: -4, 6, 2 and the lower-index 1.0 (index 9)
    codes = I.lossy_codes(g, keep=0.1)
    assert codes.dtype == np.uint8 and codes.tolist() == [0, 128, 255, 153]
    # (1 + 4) / 10 * 255 = 127.5 -> 128 after rint (ties to even), (2 + 4) / 10 * 255 = 153
    assert round((1 + 4) / 10 * 255) == 128 and np.rint(5 / 10 * 255) == 128
    big = I.lossy_codes(I.convnet_gradient(0))
    assert big.size == 29895 and big.min() == 0 and big.max() == 255
