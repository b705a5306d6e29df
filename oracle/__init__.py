"""CPU oracle of the LM-GC encode path (arXiv 2409.17836) -- TEST INFRASTRUCTURE ONLY.

Only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` may import
this package. The CUDA path never imports it and shares none of its code.

This module wraps the plain C oracle (`lmgc_oracle.c`, built with gcc) through ctypes and adds
the container layout in plain Python. Every function names the passage it follows:

* `serialize` / `deserialize`      Sec. 4 "Serialization", Fig. 1 (hex digits + separators)
* `OracleLM`, `window_logits`      Eq. 1 / Eq. 2 (next-token distributions after BOS), fp64
* `quantize_cdf`, `cdf_pair`       integer CDF for the Torchac-style coder of Sec. 5.1
* `range_encode`, `Decoder`        Sec. 3 "Arithmetic coding" in exact integer form
* `encode`, `decode_window`        Sec. 4 "Compression" (independent windows, BOS not coded)
* `compression_rate`               Eq. 3

Parity unpinned: the bit-level values of the LM logits (the paper prints none; they are pinned
by invariants and by torch library routines only).
"""
from __future__ import annotations

import ctypes as C
import dataclasses
import os
import struct

import numpy as np

from . import build as _build

_lib = None


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = C.CDLL(path)
        i64, i32, u64, u32, f32, vp = C.c_int64, C.c_int32, C.c_uint64, C.c_uint32, C.c_float, C.c_void_p
        sig = {
            "orc_tokens_per_value": (i64, [i32, i32]),
            "orc_serialize": (i64, [i32, i32, vp, i64, vp]),
            "orc_deserialize": (i64, [i32, i32, vp, i64, vp]),
            "orc_serial_tokens": (i64, [i32, i32, i32, i32, i64]),
            "orc_serialize_grouped": (i64, [i32, i32, i32, i32, vp, i64, vp]),
            "orc_deserialize_grouped": (i64, [i32, i32, i32, i32, vp, i64, vp]),
            "orc_splitmix64": (u64, [u64]),
            "orc_bf16_round": (f32, [f32]),
            "orc_weight": (f32, [u64, u32, u64, f32, i32]),
            "orc_weight_tensor": (None, [u64, u32, u64, f32, i32, vp]),
            "orc_rmsnorm": (None, [vp, i64, i32, C.c_double, vp]),
            "orc_rope": (None, [vp, i64, vp, i32, i32, C.c_double]),
            "orc_attention": (None, [vp, vp, vp, i64, i64, i32, i32, i32, vp]),
            "orc_swiglu": (None, [vp, vp, i64, vp]),
            "orc_lm_new": (vp, [vp, i64]),
            "orc_lm_free": (None, [vp]),
            "orc_lm_feed": (i32, [vp, vp, i64, vp]),
            "orc_lm_window_logits": (i32, [vp, vp, i64, vp]),
            "orc_exp2_tables": (None, [vp, vp]),
            "orc_exp2_fixed": (u32, [i64]),
            "orc_quantize_cdf": (i32, [vp, i32, i32, vp]),
            "orc_cdf_pair": (i32, [vp, i32, i32, i32, vp, vp]),
            "orc_range_encode": (i64, [vp, vp, i64, i32, vp, i64]),
            "orc_dec_size": (i64, []),
            "orc_dec_init": (None, [vp, vp, i64]),
            "orc_dec_step": (i32, [vp, vp, i32, i32]),
            "orc_window_pairs": (i32, [vp, i32, vp, i64, vp, vp, vp]),
            "orc_encode_windows": (i32, [vp, i32, vp, i64, i64, i64, vp, i64, vp, i32]),
            "orc_decode_window": (i32, [vp, i32, vp, i64, i64, vp]),
            "orc_crc32": (u32, [vp, i64]),
            "orc_num_threads": (i32, []),
            "orc_cfg_layout": (C.c_size_t, [vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        # the C struct this binding copies: its size and every field's offset but the last array
        off = (C.c_size_t * 14)()
        size = L.orc_cfg_layout(off)
        names = [f for f, _ in _Cfg._fields_]
        if size != C.sizeof(_Cfg) or [getattr(_Cfg, f).offset for f in names[:14]] != list(off):
            raise RuntimeError("oracle: the binding's _Cfg does not match orc_cfg")
        _lib = L
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(C.c_void_p)


# ------------------------------------------------------------------------------------------
# Serialisation (Sec. 4, Fig. 1). Token ids: hex digit -> 0..15, ' ' 16, ',' 17, ';' 18, BOS 19.
# sep_mode: 0 H_s (space), 1 H_c (comma), 2 H_{c+s}, 3 H_semi, 4 H_n (none). input_kind 0 = fp32,
# 1 = uint8 codes (Eq. 4 indices).
# ------------------------------------------------------------------------------------------
TOK_SPACE, TOK_COMMA, TOK_SEMI, TOK_BOS = 16, 17, 18, 19


def tokens_per_value(input_kind: int, sep_mode: int) -> int:
    return int(lib().orc_tokens_per_value(input_kind, sep_mode))


def serial_tokens(input_kind: int, sep_mode: int, n: int, byte_group: int = 0, byte_order: int = 0) -> int:
    """Token count of n values (Sec. 4; byte grouping of Sec. 5.3)."""
    return int(lib().orc_serial_tokens(input_kind, sep_mode, byte_group, byte_order, n))


def serialize(values: np.ndarray, sep_mode: int = 0, byte_group: int = 0, byte_order: int = 0) -> np.ndarray:
    """byte_group 0 and byte_order 0: one group per value, each value's nibbles most significant
    first (Sec. 4). Otherwise the byte-grouped form (Sec. 5.3 "Byte grouping"): bytes in order
    (fp32 most or least significant first), two digits each, a separator every byte_group bytes."""
    kind = 0 if values.dtype == np.float32 else 1
    if kind == 1 and values.dtype != np.uint8:
        raise TypeError("values must be float32 or uint8")
    v = np.ascontiguousarray(values)
    nt = serial_tokens(kind, sep_mode, v.size, byte_group, byte_order)
    if nt < 0:
        raise ValueError("bad serialisation arguments")
    out = np.empty(max(nt, 1), dtype=np.uint16)
    if byte_group == 0 and byte_order == 0:
        n = lib().orc_serialize(kind, sep_mode, _p(v), v.size, _p(out))
    else:
        n = lib().orc_serialize_grouped(kind, sep_mode, byte_group, byte_order, _p(v), v.size, _p(out))
    if n < 0:
        raise ValueError("bad serialisation arguments")
    return out[:n]


def deserialize(tokens: np.ndarray, input_kind: int, sep_mode: int = 0, byte_group: int = 0,
                byte_order: int = 0) -> np.ndarray:
    t = np.ascontiguousarray(tokens, dtype=np.uint16)
    out = np.empty(max(t.size // 2, 1), dtype=np.float32 if input_kind == 0 else np.uint8)
    if byte_group == 0 and byte_order == 0:
        n = lib().orc_deserialize(input_kind, sep_mode, _p(t), t.size, _p(out))
    else:
        n = lib().orc_deserialize_grouped(input_kind, sep_mode, byte_group, byte_order, _p(t), t.size, _p(out))
    if n < 0:
        raise ValueError("malformed token stream")
    return out[:n]


# ------------------------------------------------------------------------------------------
# Weights and the LM (Eq. 1 / Eq. 2).
# ------------------------------------------------------------------------------------------
def splitmix64(x: int) -> int:
    return int(lib().orc_splitmix64(x))


def weight_tensor(seed: int, tid: int, n: int, init_std: float, bf16: bool) -> np.ndarray:
    out = np.empty(n, dtype=np.float32)
    lib().orc_weight_tensor(seed, tid, n, init_std, int(bf16), _p(out))
    return out


def alphabet_ids(sep_mode: int) -> list[int]:
    """The ids a serialisation can emit (restricted-alphabet coding, a variant the paper does not
    describe): the 16 hex digits and the separator ids of sep_mode, ascending."""
    seps = {0: [TOK_SPACE], 1: [TOK_COMMA], 2: [TOK_COMMA, TOK_SPACE], 3: [TOK_SEMI], 4: []}[sep_mode]
    return list(range(16)) + sorted(seps)


class _Cfg(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("d_ffn", C.c_int32), ("vocab", C.c_int32),
                ("bf16", C.c_int32), ("window", C.c_int32), ("weight_seed", C.c_uint64),
                ("init_std", C.c_float), ("rms_eps", C.c_float), ("rope_theta", C.c_float),
                ("n_threads", C.c_int32), ("n_alpha", C.c_int32), ("alpha", C.c_uint16 * 32)]


@dataclasses.dataclass
class OracleConfig:
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    d_ffn: int
    vocab: int
    bf16: bool
    window: int
    cdf_bits: int
    weight_seed: int = 0
    init_std: float = 0.02
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0
    sep_mode: int = 0
    input_kind: int = 0
    n_threads: int = 1
    byte_group: int = 0  # bytes per separator group (Sec. 5.3); 0 = one group per value
    byte_order: int = 0  # fp32 bytes most (0) or least (1) significant first
    alphabet: int = 0    # 1: code over the ids the serialisation can emit (alphabet_ids) only

    def c(self) -> _Cfg:
        ids = alphabet_ids(self.sep_mode) if self.alphabet else []
        arr = (C.c_uint16 * 32)(*ids)
        return _Cfg(self.n_layers, self.d_model, self.n_heads, self.n_kv_heads, self.d_ffn, self.vocab,
                    int(self.bf16), self.window, self.weight_seed, self.init_std, self.rms_eps,
                    self.rope_theta, self.n_threads, len(ids), arr)


class OracleLM:
    """Incremental forward of one window with a KV cache: `feed(tokens)` appends positions and
    returns their next-token logits (fp64)."""

    def __init__(self, cfg: OracleConfig, max_pos: int):
        self.cfg = cfg
        self._c = cfg.c()
        self._h = lib().orc_lm_new(C.byref(self._c), max_pos)
        if not self._h:
            raise MemoryError("oracle LM allocation failed")

    def feed(self, tokens) -> np.ndarray:
        t = np.ascontiguousarray(np.asarray(tokens, dtype=np.uint16).reshape(-1))
        out = np.empty((t.size, self.cfg.vocab), dtype=np.float64)
        if lib().orc_lm_feed(self._h, _p(t), t.size, _p(out)) != 0:
            raise ValueError("feed past max_pos")
        return out

    def __del__(self):
        if getattr(self, "_h", None):
            lib().orc_lm_free(self._h)
            self._h = None


def window_logits(cfg: OracleConfig, win_tok: np.ndarray, n_pos: int) -> np.ndarray:
    """Logits [n_pos][V] for model input [BOS, win_tok[0], ..., win_tok[n_pos-2]] (Eq. 2)."""
    t = np.ascontiguousarray(win_tok, dtype=np.uint16)
    if t.size < n_pos - 1:
        raise ValueError("not enough window tokens")
    out = np.empty((n_pos, cfg.vocab), dtype=np.float64)
    c = cfg.c()
    if lib().orc_lm_window_logits(C.byref(c), _p(t), n_pos, _p(out)) != 0:
        raise RuntimeError("oracle forward failed")
    return out


def rmsnorm(x: np.ndarray, eps: float) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty_like(x)
    lib().orc_rmsnorm(_p(x), x.shape[0], x.shape[1], eps, _p(y))
    return y


def rope(x: np.ndarray, pos: np.ndarray, n_heads: int, theta: float) -> np.ndarray:
    y = np.array(x, dtype=np.float64, order="C", copy=True)
    p = np.ascontiguousarray(pos, dtype=np.int64)
    lib().orc_rope(_p(y), y.shape[0], _p(p), n_heads, y.shape[1] // n_heads, theta)
    return y


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, nq: int, nkv: int, p0: int = 0) -> np.ndarray:
    """Causal GQA attention of rows at positions p0.. (q [n][nq*hd], k/v [p0+n][nkv*hd])."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    out = np.empty_like(q)
    lib().orc_attention(_p(q), _p(k), _p(v), p0, q.shape[0], nq, nkv, q.shape[1] // nq, _p(out))
    return out


def swiglu(g: np.ndarray, u: np.ndarray) -> np.ndarray:
    g = np.ascontiguousarray(g, dtype=np.float64)
    u = np.ascontiguousarray(u, dtype=np.float64)
    out = np.empty_like(g)
    lib().orc_swiglu(_p(g), _p(u), g.size, _p(out))
    return out


# ------------------------------------------------------------------------------------------
# Integer CDF (Torchac-style coder input, Sec. 5.1) and the arithmetic coder (Sec. 3).
# ------------------------------------------------------------------------------------------
def exp2_tables() -> tuple[np.ndarray, np.ndarray]:
    H = np.empty(256, dtype=np.uint32)
    L = np.empty(256, dtype=np.uint32)
    lib().orc_exp2_tables(_p(H), _p(L))
    return H, L


def exp2_fixed(a: int) -> int:
    return int(lib().orc_exp2_fixed(a))


def quantize_cdf(z: np.ndarray, P: int) -> np.ndarray:
    """Integer CDF rows [rows][V+1] (cdf[0] = 0, cdf[V] = 2^P) from fp32 logit rows."""
    z = np.ascontiguousarray(np.atleast_2d(z), dtype=np.float32)
    rows, V = z.shape
    out = np.empty((rows, V + 1), dtype=np.uint32)
    for r in range(rows):
        if lib().orc_quantize_cdf(_p(z[r]), V, P, _p(out[r])) != 0:
            raise ValueError("bad (V, P)")
    return out


def cdf_pairs(z: np.ndarray, sym: np.ndarray, P: int) -> tuple[np.ndarray, np.ndarray]:
    cdf = quantize_cdf(z, P)
    s = np.asarray(sym, dtype=np.int64).reshape(-1)
    idx = np.arange(s.size)
    start = cdf[idx, s]
    return start.astype(np.uint32), (cdf[idx, s + 1] - start).astype(np.uint32)


def range_encode(start: np.ndarray, freq: np.ndarray, P: int) -> tuple[bytes, int]:
    """Code of one stream: (bytes MSB-first zero padded, bit length)."""
    s = np.ascontiguousarray(start, dtype=np.uint32)
    f = np.ascontiguousarray(freq, dtype=np.uint32)
    cap = (s.size * P + 2 + 7) // 8 + 8
    out = np.zeros(cap, dtype=np.uint8)
    n = lib().orc_range_encode(_p(s), _p(f), s.size, P, _p(out), cap)
    if n < 0:
        raise ValueError("bad coder input")
    return out[: (n + 7) // 8].tobytes(), int(n)


class Decoder:
    def __init__(self, code: bytes, nbits: int):
        self._buf = np.frombuffer(code, dtype=np.uint8).copy() if len(code) else np.zeros(1, np.uint8)
        self._st = (C.c_uint8 * int(lib().orc_dec_size()))()
        lib().orc_dec_init(C.byref(self._st), _p(self._buf), nbits)

    def step(self, cdf: np.ndarray, P: int) -> int:
        c = np.ascontiguousarray(cdf, dtype=np.uint32)
        return int(lib().orc_dec_step(C.byref(self._st), _p(c), c.size - 1, P))


def window_pairs(cfg: OracleConfig, win_tok: np.ndarray, n: int):
    """(start, freq, fp32 logits) of one window's first n tokens under the oracle LM."""
    t = np.ascontiguousarray(win_tok, dtype=np.uint16)
    st = np.empty(n, np.uint32)
    fr = np.empty(n, np.uint32)
    lg = np.empty((n, cfg.vocab), np.float32)
    c = cfg.c()
    if lib().orc_window_pairs(C.byref(c), cfg.cdf_bits, _p(t), n, _p(st), _p(fr), _p(lg)) != 0:
        raise RuntimeError("oracle window failed")
    return st, fr, lg


def encode_windows(cfg: OracleConfig, tok: np.ndarray, w0: int, nw: int, n_par: int = 1):
    """Codes of windows [w0, w0+nw): list of (bytes, bitlen)."""
    t = np.ascontiguousarray(tok, dtype=np.uint16)
    capw = (cfg.window * cfg.cdf_bits + 2 + 7) // 8 + 8
    out = np.zeros(nw * capw, dtype=np.uint8)
    bl = np.zeros(nw, dtype=np.int64)
    c = cfg.c()
    rc = lib().orc_encode_windows(C.byref(c), cfg.cdf_bits, _p(t), t.size, w0, nw, _p(out), capw, _p(bl), n_par)
    if rc != 0:
        raise RuntimeError("oracle encode failed")
    return [(out[i * capw: i * capw + (int(bl[i]) + 7) // 8].tobytes(), int(bl[i])) for i in range(nw)]


def decode_window(cfg: OracleConfig, code: bytes, nbits: int, n: int) -> np.ndarray:
    buf = np.frombuffer(code, dtype=np.uint8).copy() if len(code) else np.zeros(1, np.uint8)
    out = np.empty(n, dtype=np.uint16)
    c = cfg.c()
    if lib().orc_decode_window(C.byref(c), cfg.cdf_bits, _p(buf), nbits, n, _p(out)) != 0:
        raise ValueError("corrupt code")
    return out


def crc32(b: bytes) -> int:
    a = np.frombuffer(b, dtype=np.uint8).copy() if len(b) else np.zeros(1, np.uint8)
    return int(lib().orc_crc32(_p(a), len(b)))


# ------------------------------------------------------------------------------------------
# Container (a build choice; the paper stores one code per window without a format).
#   0  "LMGC"            4  u32 version (2)      8  u64 n_values       16 u64 n_tok
#   24 u32 window        28 u32 cdf_bits         32 u32 input_kind     36 u32 serialisation
#   40 u32 vocab         44 u32 n_win            48 u64 weight_seed    56 u32 model crc
#   60 u32 crc32 of bytes [0, 60)
#   64 u32 bitlen[n_win] | u32 crc_tok[n_win] | each window's code, ceil(bitlen/8) bytes, in
#   window order. crc_tok[w] = crc32 of window w's token ids as little-endian u16 (its own
#   length: W, or fewer for the last window), so that a decoder can check each window it restores.
# serialisation = sep_mode | byte_group << 8 | byte_order << 16 | alphabet << 24 (0 in the upper
# bits: the default one group per value, most significant byte first, the whole vocabulary).
# model crc = crc32 of '<7i3f' (n_layers, d_model, n_heads, n_kv_heads, d_ffn, vocab, bf16,
# init_std, rms_eps, rope_theta).
# ------------------------------------------------------------------------------------------
HEADER_BYTES = 64


def model_crc(cfg: OracleConfig) -> int:
    return crc32(struct.pack("<7i3f", cfg.n_layers, cfg.d_model, cfg.n_heads, cfg.n_kv_heads, cfg.d_ffn,
                             cfg.vocab, int(cfg.bf16), cfg.init_std, cfg.rms_eps, cfg.rope_theta))


CONTAINER_VERSION = 2


def window_crcs(tok: np.ndarray, window: int, first: int = 0, count: int | None = None) -> np.ndarray:
    """crc_tok of windows [first, first + count): crc32 of each window's ids as little-endian u16."""
    t = np.ascontiguousarray(tok, dtype="<u2")
    n_win = -(-t.size // window)
    count = n_win - first if count is None else count
    return np.array([crc32(t[w * window: (w + 1) * window].tobytes()) for w in range(first, first + count)],
                    dtype=np.uint32)


def serial_word(cfg: OracleConfig) -> int:
    return cfg.sep_mode | cfg.byte_group << 8 | cfg.byte_order << 16 | cfg.alphabet << 24


def build_container(cfg: OracleConfig, n_values: int, n_tok: int, codes: list[tuple[bytes, int]],
                    crcs: np.ndarray) -> bytes:
    head = struct.pack("<4sIQQIIIIIIQI", b"LMGC", CONTAINER_VERSION, n_values, n_tok, cfg.window, cfg.cdf_bits,
                       cfg.input_kind, serial_word(cfg), cfg.vocab, len(codes), cfg.weight_seed, model_crc(cfg))
    head += struct.pack("<I", crc32(head))
    assert len(head) == HEADER_BYTES and len(crcs) == len(codes)
    table = np.array([bl for _, bl in codes], dtype="<u4").tobytes() + np.asarray(crcs, dtype="<u4").tobytes()
    return head + table + b"".join(c for c, _ in codes)


def parse_container(buf: bytes) -> dict:
    if len(buf) < HEADER_BYTES or buf[:4] != b"LMGC":
        raise ValueError("not a container")
    f = struct.unpack("<4sIQQIIIIIIQI", buf[:60])
    (crc,) = struct.unpack("<I", buf[60:64])
    if crc != crc32(buf[:60]):
        raise ValueError("header crc mismatch")
    if f[1] != CONTAINER_VERSION:
        raise ValueError("unknown container version")
    n_win = f[9]
    if len(buf) < 64 + 8 * n_win:
        raise ValueError("window table truncated")
    bl = np.frombuffer(buf[64: 64 + 4 * n_win], dtype="<u4").astype(np.int64)
    crc_tok = np.frombuffer(buf[64 + 4 * n_win: 64 + 8 * n_win], dtype="<u4").astype(np.uint32)
    offs = np.concatenate([[0], np.cumsum((bl + 7) // 8)]) + 64 + 8 * n_win
    return dict(version=f[1], n_values=f[2], n_tok=f[3], window=f[4], cdf_bits=f[5], input_kind=f[6],
                sep_mode=f[7] & 0xFF, byte_group=(f[7] >> 8) & 0xFF, byte_order=(f[7] >> 16) & 0xFF,
                alphabet=(f[7] >> 24) & 0xFF, vocab=f[8], n_win=n_win, weight_seed=f[10], model_crc=f[11], bitlen=bl,
                crc_tok=crc_tok, offsets=offs)


def encode(cfg: OracleConfig, values: np.ndarray, n_par: int = 1) -> bytes:
    """Full oracle encode of a gradient vector into the container (Sec. 4)."""
    tok = serialize(values, cfg.sep_mode, cfg.byte_group, cfg.byte_order)
    W = cfg.window
    n_win = (tok.size + W - 1) // W
    codes = encode_windows(cfg, tok, 0, n_win, n_par)
    return build_container(cfg, values.size, tok.size, codes, window_crcs(tok, W))


def compression_rate(container_bytes: int, n_values: int, bytes_per_value: int = 4) -> float:
    """Eq. 3: 100 * compressed size / original size."""
    return 100.0 * container_bytes / (bytes_per_value * n_values)


def gemm_nt(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """C = A . B^T in fp64 (the plain definition of the model's linear layers; a library matmul
    serves as the step)."""
    return np.asarray(a, dtype=np.float64) @ np.asarray(b, dtype=np.float64).T
