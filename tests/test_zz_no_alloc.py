"""The allocation-free coder entry point, lmgc_range_encode_noalloc.

It exists for callers that cannot allocate device memory -- for example a process whose device
memory is already held entirely by another allocator, or a latency-critical path where
cudaMalloc / cudaFree (which may synchronise the device) are not allowed. Instead of allocating
per call, it keeps its scratch in one fixed 64 MiB device array inside the library.

Its codes must equal those of lmgc_range_encode (the allocating entry point) bit for bit, on two
calls in a row: the array keeps the previous call's contents, so the second call checks that
nothing left behind leaks into its output. This file is collected last so that a run stopping at
the first failure has already run every other test; it also passes on its own.
"""
import numpy as np
import pytest
import torch

from paper_2409_17836_gb300 import lmgc as L
from tests._util import random_pairs

pytestmark = pytest.mark.gpu


def _both(start, freq, P, n_win, W, lens, sw, sp):
    s = torch.from_numpy(start.view(np.int32)).cuda()
    f = torch.from_numpy(freq.view(np.int32)).cuda()
    wl = torch.from_numpy(lens.view(np.int32)).cuda() if lens is not None else None
    ref_out, ref_bl = L.lmgc_range_encode(s, f, P, n_win, W, wl, sw, sp)
    out = torch.full((ref_out.numel() + 64,), 0xA5, dtype=torch.uint8, device="cuda")
    bitlen = torch.full((n_win,), -1, dtype=torch.int32, device="cuda")
    nbytes = L.lmgc_range_encode_noalloc(s, f, P, n_win, W, wl, sw, sp, out, bitlen)
    assert nbytes == ref_out.numel()
    assert torch.equal(bitlen, ref_bl)
    assert torch.equal(out[:nbytes], ref_out)
    return nbytes


def test_noalloc_matches_allocating_coder_twice():
    rng = np.random.default_rng(2024)
    # first call: 300 windows of 2048 tokens over vocab 32000 at P = 24, position-major layout
    n_win, W, P = 300, 2048, 24
    start, freq, _ = random_pairs(rng, n_win, W, P)
    n1 = _both(start.T.copy(), freq.T.copy(), P, n_win, W, None, 1, n_win)
    # second call, different shape and layout: 97 ragged windows (row-major) at P = 16; the
    # array still holds the first call's codes
    n_win2, W2, P2 = 97, 256, 16
    start2, freq2, _ = random_pairs(rng, n_win2, W2, P2, V=32)
    lens = rng.integers(1, W2 + 1, n_win2).astype(np.uint32)
    n2 = _both(start2, freq2, P2, n_win2, W2, lens, W2, 1)
    assert n1 > 0 and n2 > 0


def test_noalloc_rejects_more_than_its_fixed_scratch():
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    out = torch.zeros(16, dtype=torch.uint8, device="cuda")
    # 20,000 windows of 2048 tokens at P = 24 need about 123 MB of scratch (> 64 MiB)
    with pytest.raises(L.LmgcError) as e:
        L.lmgc_range_encode_noalloc(dummy, dummy, 24, 20000, 2048, None, 1, 20000, out, dummy)
    assert e.value.status == L.ERR_INVALID
    assert "fixed maximum" in str(e.value)


def test_noalloc_runs_with_device_memory_exhausted():
    """The point of the entry point: it still works when the caller has left it no device memory
    to allocate. Torch claims all but a small margin of the free device memory (after one call has
    loaded the module and found the array), then the call must succeed and reproduce the codes
    computed beforehand. A version that quietly fell back to cudaMalloc for its 20 MB of slots
    would fail here."""
    rng = np.random.default_rng(77)
    n_win, W, P = 3000, 2048, 24
    start, freq, _ = random_pairs(rng, n_win, W, P)
    s = torch.from_numpy(start.T.copy().view(np.int32)).cuda()
    f = torch.from_numpy(freq.T.copy().view(np.int32)).cuda()
    ref_out, ref_bl = L.lmgc_range_encode(s, f, P, n_win, W, None, 1, n_win)
    out = torch.zeros(ref_out.numel() + 64, dtype=torch.uint8, device="cuda")
    bitlen = torch.zeros(n_win, dtype=torch.int32, device="cuda")
    L.lmgc_range_encode_noalloc(s, f, P, n_win, W, None, 1, n_win, out, bitlen)  # set-up call
    out.zero_()
    bitlen.zero_()
    torch.cuda.synchronize()
    margin = 16 << 20
    hold = []
    try:
        while True:
            free, _ = torch.cuda.mem_get_info()
            if free <= 2 * margin:
                break
            try:
                hold.append(torch.empty(min(free - margin, 1 << 30), dtype=torch.uint8, device="cuda"))
            except torch.OutOfMemoryError:
                break
        free, _ = torch.cuda.mem_get_info()
        assert free < 64 << 20, free  # less than the 64 MiB array itself: no room for a second one
        nbytes = L.lmgc_range_encode_noalloc(s, f, P, n_win, W, None, 1, n_win, out, bitlen)
        assert nbytes == ref_out.numel()
        assert torch.equal(bitlen, ref_bl)
        assert torch.equal(out[:nbytes], ref_out)
    finally:
        del hold
        torch.cuda.empty_cache()


def test_noalloc_rejects_windows_beyond_its_scratch():
    """A window whose slot alone exceeds the array is refused before any size arithmetic that
    could wrap."""
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    out = torch.zeros(16, dtype=torch.uint8, device="cuda")
    for W in [(1 << 29) // 24 + 1, 1 << 62]:
        with pytest.raises(L.LmgcError) as e:
            L.lmgc_range_encode_noalloc(dummy, dummy, 24, 1, W, None, 1, 1, out, dummy)
        assert e.value.status == L.ERR_INVALID
        assert "fixed maximum" in str(e.value)
