"""Model and coder shapes of the workloads (the paper's LLMs, Sec. 5.1, with random-init weights).

* TINY        2 layers, d 128, 4 heads, FFN 512, vocab 32, fp32, 256-token windows, P = 16
* TINYLLAMA   TinyLlama-1.1B shape: 22 layers, d 2048, 32 Q / 4 KV heads, SwiGLU 5632, vocab 32000,
              bf16, 2048-token windows (the paper's default window, Sec. 5.1), P = 24
* LLAMA2_7B   Llama-2-7B shape: 32 layers, d 4096, 32 heads (MHA), FFN 11008, vocab 32000, bf16,
              4096-token windows, P = 24
P = 24 for vocab 32000 because at P = 16 the floor of one count per symbol would take 32000 of
65536 counts (half the probability mass).
"""
from __future__ import annotations

import dataclasses

from .lmgc import BF16, F32, IN_F32, IN_U8, ModelConfig

TINY = ModelConfig(n_layers=2, d_model=128, n_heads=4, n_kv_heads=4, d_ffn=512, vocab=32, dtype=F32, window=256,
                   cdf_bits=16, batch_windows=144)
TINYLLAMA = ModelConfig(n_layers=22, d_model=2048, n_heads=32, n_kv_heads=4, d_ffn=5632, vocab=32000, dtype=BF16,
                        window=2048, cdf_bits=24, batch_windows=64)
LLAMA2_7B = ModelConfig(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=32, d_ffn=11008, vocab=32000, dtype=BF16,
                        window=4096, cdf_bits=24, batch_windows=32)
TINYLLAMA_LOSSY = dataclasses.replace(TINYLLAMA, input_kind=IN_U8, batch_windows=128)


def with_(cfg: ModelConfig, **kw) -> ModelConfig:
    return dataclasses.replace(cfg, **kw)
