"""Seeded synthetic inputs shaped like the paper's workloads (no datasets or checkpoints here).

This module holds input generators only (no step of the encode path). Both the CUDA path's
tests and the oracle's tests draw their inputs from here.

The paper compresses gradients of networks trained on MNIST / CIFAR-10 / TinyImageNet
(Sec. 5.1 "Datasets and models", "Evaluation protocols"). Those datasets and training runs are
not available, so seeded stand-ins of the same kind are used:

* `tiny_gradient`      4,096 values = 4 tensors x 1,024, N(0, s_l^2), s_l = 10^(-3 + 2l/3).
* `convnet_gradient`   the gradient of one cross-entropy step of a seeded random-init
                       4-layer ConvNet (298,954 parameters) on Gaussian 3x32x32 inputs.
* `lossy_codes`        Sec. 5.4 "Compatibility": top-10% magnitude sparsification followed by
                       8-bit linear quantisation (Eq. 4) of the kept values.
* `laplace_gradient`   a 200-tensor Laplace mixture with log-uniform scales (throughput sweep).
* `sparsified`, `quantized_codes`, `code_bytes`   the Sec. 5.4 compatibility inputs one at a time
                     (sparsification 50/25/10% as fp32; 16/8/1-bit Eq. 4 indices).
"""
from __future__ import annotations

import numpy as np


def tiny_gradient(seed: int = 0) -> np.ndarray:
    rng = np.random.default_rng(seed)
    parts = [rng.normal(0.0, 10.0 ** (-3.0 + 2.0 * l / 3.0), 1024) for l in range(4)]
    return np.concatenate(parts).astype(np.float32)


def convnet_gradient(seed: int = 0, batch: int = 64) -> np.ndarray:
    """Gradient of a ConvNet: conv3x3(3->64)-ReLU-pool2, conv3x3(64->128)-ReLU-pool2,
    conv3x3(128->192)-ReLU-pool2, global average pool, fc(192->10); mean cross-entropy on
    x ~ N(0, 1) [batch, 3, 32, 32] and uniform labels. Flattened in parameters() order."""
    import torch
    import torch.nn as nn

    g = torch.Generator().manual_seed(seed)
    with torch.random.fork_rng(devices=[]):
        torch.manual_seed(seed)
        net = nn.Sequential(
            nn.Conv2d(3, 64, 3, padding=1), nn.ReLU(), nn.MaxPool2d(2),
            nn.Conv2d(64, 128, 3, padding=1), nn.ReLU(), nn.MaxPool2d(2),
            nn.Conv2d(128, 192, 3, padding=1), nn.ReLU(), nn.MaxPool2d(2),
            nn.AdaptiveAvgPool2d(1), nn.Flatten(), nn.Linear(192, 10),
        )
    x = torch.randn(batch, 3, 32, 32, generator=g)
    y = torch.randint(0, 10, (batch,), generator=g)
    loss = nn.functional.cross_entropy(net(x), y)
    loss.backward()
    grad = torch.cat([p.grad.reshape(-1) for p in net.parameters()])
    return grad.detach().numpy().astype(np.float32)


def sparsified(grad: np.ndarray, keep: float) -> np.ndarray:
    """Sec. 5.4 sparsification alone: the floor(keep*N) largest |v| (ties to the lower index) in
    index order, still fp32 (the paper: sparsified gradients stay 32-bit floats)."""
    g = np.asarray(grad, dtype=np.float32)
    k = int(np.floor(keep * g.size))
    order = np.lexsort((np.arange(g.size), -np.abs(g.astype(np.float64))))
    return g[np.sort(order[:k])].copy()


def quantized_codes(grad: np.ndarray, bits: int) -> np.ndarray:
    """Sec. 5.4 quantisation alone: Eq. 4 over every value (n = 16, 8 or 1 bits; 1 bit is SignSGD's
    setting); the indices are what is coded."""
    return lossy_codes(grad, keep=1.0, bits=bits)


def code_bytes(codes: np.ndarray) -> tuple[np.ndarray, int]:
    """The byte stream of integer codes for the uint8 input kind, and the byte group that keeps one
    code per separator group: uint16 codes as big-endian byte pairs (4 hex digits, most
    significant first, then the separator: byte_group 2); uint8 codes as they are (group 0)."""
    if codes.dtype == np.uint16:
        return np.ascontiguousarray(codes.astype(">u2")).view(np.uint8), 2
    return np.ascontiguousarray(codes, dtype=np.uint8), 0


def lossy_codes(grad: np.ndarray, keep: float = 0.1, bits: int = 8) -> np.ndarray:
    """Sec. 5.4: keep the floor(keep*N) largest |v| (ties to the lower index) in index order,
    then v_bar = (v - min v) / (max v - min v) * (2^bits - 1) (Eq. 4) over the kept values,
    rounded to nearest and clamped; the codes are what would be transmitted."""
    g = np.asarray(grad, dtype=np.float32)
    k = int(np.floor(keep * g.size))
    order = np.lexsort((np.arange(g.size), -np.abs(g.astype(np.float64))))
    kept_idx = np.sort(order[:k])
    v = g[kept_idx].astype(np.float64)
    lo, hi = v.min(), v.max()
    q = np.rint((v - lo) / (hi - lo) * (2 ** bits - 1)) if hi > lo else np.zeros_like(v)
    q = np.clip(q, 0, 2 ** bits - 1)
    return q.astype(np.uint8 if bits <= 8 else np.uint16)


def laplace_gradient(n: int = 64 * 1024 * 1024, n_tensors: int = 200, seed: int = 5) -> np.ndarray:
    rng = np.random.default_rng(seed)
    base = n // n_tensors
    sizes = [base] * (n_tensors - 1) + [n - base * (n_tensors - 1)]
    out = np.empty(n, dtype=np.float32)
    o = 0
    for s in sizes:
        b = 10.0 ** rng.uniform(-5.0, -2.0)
        out[o:o + s] = rng.laplace(0.0, b, s).astype(np.float32)
        o += s
    return out


def token_windows(n_tok: int, window: int) -> int:
    return (n_tok + window - 1) // window
