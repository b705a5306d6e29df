"""Shared helpers of the tests (CPU and GPU)."""
import os

import numpy as np

import oracle as O


def oracle_config(cfg, n_threads: int = 1) -> O.OracleConfig:
    """The oracle's description of the model a ModelConfig names."""
    return O.OracleConfig(n_layers=cfg.n_layers, d_model=cfg.d_model, n_heads=cfg.n_heads, n_kv_heads=cfg.n_kv_heads,
                          d_ffn=cfg.d_ffn, vocab=cfg.vocab, bf16=cfg.dtype == 1, window=cfg.window,
                          cdf_bits=cfg.cdf_bits, weight_seed=cfg.weight_seed, init_std=cfg.init_std,
                          rms_eps=cfg.rms_eps, rope_theta=cfg.rope_theta, sep_mode=cfg.sep_mode,
                          input_kind=cfg.input_kind, n_threads=n_threads, byte_group=cfg.byte_group,
                          byte_order=cfg.byte_order, alphabet=cfg.alphabet)


def cpu_threads() -> int:
    return max(1, len(os.sched_getaffinity(0)))


def random_pairs(rng, n_win, W, P, lens=None, V=32000, layout="pos"):
    """Seeded random (start, freq) streams from random integer CDFs; returns arrays in the
    requested layout plus per-window lists for the oracle."""
    T = 1 << P
    n_rows = 64
    cdfs = []
    for _ in range(n_rows):
        w = rng.exponential(size=V) ** 2
        f = 1 + np.floor(w / w.sum() * (T - V)).astype(np.int64)
        f[np.argmax(f)] += T - f.sum()
        cdfs.append(np.concatenate([[0], np.cumsum(f)]))
    cdfs = np.array(cdfs)
    row = rng.integers(0, n_rows, (n_win, W))
    sym = rng.integers(0, V, (n_win, W))
    # bias symbols toward likely ones half of the time
    likely = np.argmax(np.diff(cdfs, axis=1), axis=1)
    pick = rng.random((n_win, W)) < 0.5
    sym = np.where(pick, likely[row], sym)
    start = cdfs[row, sym].astype(np.uint32)
    freq = (cdfs[row, sym + 1] - cdfs[row, sym]).astype(np.uint32)
    if lens is None:
        lens = np.full(n_win, W, dtype=np.uint32)
    return start, freq, lens


def to_pair_tiles(a: np.ndarray) -> np.ndarray:
    """A [n_win][W] (window-major) pair array in the coder's window tiles: 32 windows x 8 positions
    per 256-element tile, tiles by window block then by position group, padding zero."""
    n_win, W = a.shape
    nb, G = -(-n_win // 32), -(-W // 8)
    pad = np.zeros((nb * 32, G * 8), dtype=a.dtype)
    pad[:n_win, :W] = a
    return np.ascontiguousarray(pad.reshape(nb, 32, G, 8).transpose(0, 2, 1, 3)).reshape(-1)
