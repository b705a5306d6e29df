"""Python binding of liblmgc.so (include/lmgc.h): argument marshalling only.

Every function has the name of the C entry point it calls and takes torch CUDA tensors for the
device buffers; all computation happens in the library's CUDA kernels. There is no CPU fallback:
if the library is missing or cannot load, `load()` raises.
"""
from __future__ import annotations

import ctypes as C
import dataclasses
import os

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblmgc.so")

OK, ERR_INVALID, ERR_NO_SPACE, ERR_CUDA, ERR_CORRUPT, ERR_LIMIT, ERR_NOMEM = 0, -1, -2, -3, -4, -5, -6
F32, BF16 = 0, 1
SEP_SPACE, SEP_COMMA, SEP_COMMA_SPACE, SEP_SEMI, SEP_NONE = 0, 1, 2, 3, 4
IN_F32, IN_U8 = 0, 1
KERNEL_CLASSES = ["gemm", "attention", "cdf_pairs", "range_encode", "serialize", "norm_rope_act", "other"]


class LmgcError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"lmgc status {status}: {msg}")
        self.status = status


class Config(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("d_ffn", C.c_int32), ("vocab", C.c_int32), ("dtype", C.c_int32),
                ("window", C.c_int32), ("cdf_bits", C.c_int32), ("sep_mode", C.c_int32),
                ("input_kind", C.c_int32), ("batch_windows", C.c_int32), ("weight_seed", C.c_uint64),
                ("init_std", C.c_float), ("rms_eps", C.c_float), ("rope_theta", C.c_float),
                ("byte_group", C.c_int32), ("byte_order", C.c_int32), ("alphabet", C.c_int32)]


@dataclasses.dataclass
class ModelConfig:
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    d_ffn: int
    vocab: int
    dtype: int
    window: int
    cdf_bits: int
    batch_windows: int = 1
    sep_mode: int = SEP_SPACE
    input_kind: int = IN_F32
    weight_seed: int = 0
    init_std: float = 0.02
    rms_eps: float = 1e-5
    rope_theta: float = 10000.0
    byte_group: int = 0  # bytes per separator group (Sec. 5.3 byte grouping); 0 = one group per value
    byte_order: int = 0  # fp32 bytes most (0) or least (1) significant first
    alphabet: int = 0  # 1: integer CDFs over the ids the serialisation can emit only

    def c(self) -> Config:
        return Config(self.n_layers, self.d_model, self.n_heads, self.n_kv_heads, self.d_ffn, self.vocab, self.dtype,
                      self.window, self.cdf_bits, self.sep_mode, self.input_kind, self.batch_windows,
                      self.weight_seed, self.init_std, self.rms_eps, self.rope_theta, self.byte_group,
                      self.byte_order, self.alphabet)


_lib = None

SYMBOLS = {
    "lmgc_create": (C.c_int, [C.c_void_p, C.c_void_p]),
    "lmgc_destroy": (C.c_int, [C.c_void_p]),
    "lmgc_last_error": (C.c_int, [C.c_void_p, C.c_char_p, C.c_size_t]),
    "lmgc_tokens_per_value": (C.c_int, [C.c_void_p, C.c_void_p]),
    "lmgc_serial_tokens": (C.c_int, [C.c_void_p, C.c_size_t, C.c_void_p]),
    "lmgc_serialize": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p]),
    "lmgc_deserialize": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p,
                                   C.c_void_p]),
    "lmgc_lm_probs": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_size_t, C.c_size_t, C.c_void_p, C.c_void_p]),
    "lmgc_quantize_cdf": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p]),
    "lmgc_gemm": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t, C.c_size_t, C.c_size_t, C.c_int,
                            C.c_void_p]),
    "lmgc_cdf_pairs": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "lmgc_range_encode": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int, C.c_size_t, C.c_size_t, C.c_void_p, C.c_size_t,
                                    C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p, C.c_void_p]),
    "lmgc_range_encode_tiled": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int, C.c_size_t, C.c_size_t, C.c_void_p,
                                          C.c_int, C.c_void_p, C.c_size_t, C.POINTER(C.c_size_t), C.c_void_p,
                                          C.c_void_p]),
    "lmgc_pair_tile_elems": (C.c_int, [C.c_size_t, C.c_size_t, C.POINTER(C.c_size_t)]),
    "lmgc_range_encode_noalloc": (C.c_int, [C.c_void_p, C.c_void_p, C.c_int, C.c_size_t, C.c_size_t, C.c_void_p,
                                            C.c_size_t, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p,
                                            C.c_void_p]),
    "lmgc_encode_bound": (C.c_int, [C.c_void_p, C.c_size_t, C.c_void_p]),
    "lmgc_encode": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p]),
    "lmgc_encode_windows": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_size_t, C.c_size_t, C.c_void_p,
                                      C.c_size_t, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "lmgc_container_header": (C.c_int, [C.c_void_p, C.c_size_t, C.c_void_p]),
    "lmgc_encode_host": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p,
                                   C.c_void_p]),
    "lmgc_decode": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p, C.c_size_t,
                              C.c_void_p]),
    "lmgc_decode_batch_windows": (C.c_int, [C.c_void_p, C.POINTER(C.c_size_t)]),
    "lmgc_stage_times": (C.c_int, [C.c_void_p, C.c_void_p, C.c_size_t]),
    "lmgc_launch_count": (C.c_int, [C.c_void_p]),
    "lmgc_profile": (C.c_int, [C.c_void_p, C.c_int]),
    "lmgc_kernel_stats": (C.c_int, [C.c_void_p, C.c_int, C.c_char_p, C.c_size_t, C.c_void_p, C.c_void_p,
                                    C.c_void_p]),
}


def load(path: str = LIB_PATH):
    """Load liblmgc.so (raises if it is missing: there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise FileNotFoundError(f"{path} not built: run __graft_entry__.build()")
        L = C.CDLL(path)
        for name, (res, args) in SYMBOLS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        return t.data_ptr()
    return t


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def _check(ctx, st: int):
    if st != OK:
        buf = C.create_string_buffer(512)
        load().lmgc_last_error(ctx.handle if ctx is not None else None, buf, 512)
        raise LmgcError(st, buf.value.decode(errors="replace"))


class Context:
    """Owns an lmgc_ctx (device weights + workspace) on the current CUDA device."""

    def __init__(self, cfg: ModelConfig):
        if not torch.cuda.is_available():
            raise RuntimeError("liblmgc needs a CUDA device")
        self.cfg = cfg
        self._c = cfg.c()
        h = C.c_void_p()
        st = load().lmgc_create(C.byref(self._c), C.byref(h))
        if st != OK:
            buf = C.create_string_buffer(512)
            load().lmgc_last_error(None, buf, 512)
            raise LmgcError(st, buf.value.decode(errors="replace"))
        self.handle = h

    def close(self):
        if getattr(self, "handle", None):
            load().lmgc_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def tpv(self) -> int | None:
        """Tokens per value, or None when byte groups cross values (byte_group 3 or 8)."""
        v = C.c_size_t()
        return v.value if load().lmgc_tokens_per_value(self.handle, C.byref(v)) == OK else None


# ---- entry points (same names as the C ABI) ----

def lmgc_tokens_per_value(ctx: Context) -> int:
    v = C.c_size_t()
    _check(ctx, load().lmgc_tokens_per_value(ctx.handle, C.byref(v)))
    return v.value


def lmgc_serial_tokens(ctx: Context, n: int) -> int:
    v = C.c_size_t()
    _check(ctx, load().lmgc_serial_tokens(ctx.handle, n, C.byref(v)))
    return v.value


def lmgc_serialize(ctx: Context, values: torch.Tensor, tokens: torch.Tensor | None = None, stream=None):
    n = values.numel()
    if tokens is None:
        tokens = torch.empty(lmgc_serial_tokens(ctx, n), dtype=torch.int16, device=values.device)
    n_tok = C.c_size_t()
    _check(ctx, load().lmgc_serialize(ctx.handle, _ptr(values), n, _ptr(tokens), tokens.numel(), C.byref(n_tok),
                                      _stream(stream)))
    return tokens[: n_tok.value]


def lmgc_deserialize(ctx: Context, tokens: torch.Tensor, out: torch.Tensor, stream=None) -> int:
    nv = C.c_size_t()
    _check(ctx, load().lmgc_deserialize(ctx.handle, _ptr(tokens), tokens.numel(), _ptr(out), out.numel(),
                                        C.byref(nv), _stream(stream)))
    return nv.value


def lmgc_lm_probs(ctx: Context, tokens: torch.Tensor, first_win: int, n_win: int, logits: torch.Tensor | None = None,
                  stream=None) -> torch.Tensor:
    W, V = ctx.cfg.window, ctx.cfg.vocab
    if logits is None:
        logits = torch.empty((n_win, W, V), dtype=torch.float32, device=tokens.device)
    _check(ctx, load().lmgc_lm_probs(ctx.handle, _ptr(tokens), tokens.numel(), first_win, n_win, _ptr(logits),
                                     _stream(stream)))
    return logits


def lmgc_gemm(ctx: Context, a: torch.Tensor, b: torch.Tensor, c: torch.Tensor, epi: int, stream=None) -> torch.Tensor:
    """c (op)= a @ b.T; a [M][K], b [N][K] in the context's dtype; c per epi (0: dtype, 1/2: fp32)."""
    M, K = a.shape
    N = b.shape[0]
    _check(ctx, load().lmgc_gemm(ctx.handle, _ptr(a), _ptr(b), _ptr(c), M, N, K, epi, _stream(stream)))
    return c


def lmgc_quantize_cdf(ctx: Context, logits: torch.Tensor, stream=None) -> torch.Tensor:
    rows = logits.numel() // ctx.cfg.vocab
    cdf = torch.empty((rows, ctx.cfg.vocab + 1), dtype=torch.int32, device=logits.device)
    _check(ctx, load().lmgc_quantize_cdf(ctx.handle, _ptr(logits), rows, _ptr(cdf), _stream(stream)))
    return cdf


def lmgc_cdf_pairs(ctx: Context, logits: torch.Tensor, sym: torch.Tensor, stream=None):
    rows = logits.numel() // ctx.cfg.vocab
    start = torch.empty(rows, dtype=torch.int32, device=logits.device)
    freq = torch.empty(rows, dtype=torch.int32, device=logits.device)
    _check(ctx, load().lmgc_cdf_pairs(ctx.handle, _ptr(logits), rows, _ptr(sym), _ptr(start), _ptr(freq),
                                      _stream(stream)))
    return start, freq


def lmgc_range_encode(start: torch.Tensor, freq: torch.Tensor, cdf_bits: int, n_win: int, win_tokens: int,
                      win_len: torch.Tensor | None, stride_win: int, stride_pos: int, out: torch.Tensor | None = None,
                      stream=None):
    """Returns (payload bytes tensor view, bitlen tensor)."""
    bitlen = torch.empty(max(n_win, 1), dtype=torch.int32, device=start.device)
    nbytes = C.c_size_t()
    if out is None:
        # a first call with no output learns the size (NO_SPACE), a second writes
        st = load().lmgc_range_encode(_ptr(start), _ptr(freq), cdf_bits, n_win, win_tokens, _ptr(win_len),
                                      stride_win, stride_pos, None, 0, C.byref(nbytes), _ptr(bitlen),
                                      _stream(stream))
        if st not in (OK, ERR_NO_SPACE):
            _check(None, st)
        out = torch.empty(max(nbytes.value, 1), dtype=torch.uint8, device=start.device)
    st = load().lmgc_range_encode(_ptr(start), _ptr(freq), cdf_bits, n_win, win_tokens, _ptr(win_len), stride_win,
                                  stride_pos, _ptr(out), out.numel(), C.byref(nbytes), _ptr(bitlen), _stream(stream))
    _check(None, st)
    return out[: nbytes.value], bitlen[:n_win]


def lmgc_pair_tile_elems(n_win: int, win_tokens: int) -> int:
    n = C.c_size_t()
    _check(None, load().lmgc_pair_tile_elems(n_win, win_tokens, C.byref(n)))
    return n.value


def lmgc_range_encode_tiled(start: torch.Tensor, freq: torch.Tensor, cdf_bits: int, n_win: int, win_tokens: int,
                            win_len: torch.Tensor | None, out: torch.Tensor | None = None, stream=None,
                            validate: bool = True):
    """The coder over pairs in window tiles (lmgc_pair_tile_elems elements per array); returns
    (payload bytes, bitlen). validate=False skips the per-pair check, as the encode path does for
    its own pairs (the caller vouches for 0 < freq < 2^cdf_bits and start + freq <= 2^cdf_bits)."""
    bitlen = torch.empty(max(n_win, 1), dtype=torch.int32, device=start.device)
    nbytes = C.c_size_t()
    v = 1 if validate else 0
    if out is None:
        st = load().lmgc_range_encode_tiled(_ptr(start), _ptr(freq), cdf_bits, n_win, win_tokens, _ptr(win_len), v,
                                            None, 0, C.byref(nbytes), _ptr(bitlen), _stream(stream))
        if st not in (OK, ERR_NO_SPACE):
            _check(None, st)
        out = torch.empty(max(nbytes.value, 1), dtype=torch.uint8, device=start.device)
    st = load().lmgc_range_encode_tiled(_ptr(start), _ptr(freq), cdf_bits, n_win, win_tokens, _ptr(win_len), v,
                                        _ptr(out), out.numel(), C.byref(nbytes), _ptr(bitlen), _stream(stream))
    _check(None, st)
    return out[: nbytes.value], bitlen[:n_win]


def lmgc_range_encode_noalloc(start: torch.Tensor, freq: torch.Tensor, cdf_bits: int, n_win: int, win_tokens: int,
                              win_len: torch.Tensor | None, stride_win: int, stride_pos: int, out: torch.Tensor,
                              bitlen: torch.Tensor, stream=None) -> int:
    """The allocation-free coder: writes the codes into `out` and the bit lengths into `bitlen`
    (both caller-owned device tensors); returns the payload bytes."""
    nbytes = C.c_size_t()
    st = load().lmgc_range_encode_noalloc(_ptr(start), _ptr(freq), cdf_bits, n_win, win_tokens, _ptr(win_len),
                                          stride_win, stride_pos, _ptr(out), out.numel(), C.byref(nbytes),
                                          _ptr(bitlen), _stream(stream))
    _check(None, st)
    return nbytes.value


def lmgc_encode_bound(ctx: Context, n: int) -> int:
    b = C.c_size_t()
    _check(ctx, load().lmgc_encode_bound(ctx.handle, n, C.byref(b)))
    return b.value


def lmgc_encode(ctx: Context, values: torch.Tensor, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    n = values.numel()
    if out is None:
        out = torch.empty(lmgc_encode_bound(ctx, n), dtype=torch.uint8, device=values.device)
    nb = C.c_size_t()
    _check(ctx, load().lmgc_encode(ctx.handle, _ptr(values), n, _ptr(out), out.numel(), C.byref(nb),
                                   _stream(stream)))
    return out[: nb.value]


def lmgc_encode_windows(ctx: Context, values: torch.Tensor, first_win: int, n_win: int, stream=None):
    """Codes of windows [first_win, first_win + n_win): (payload uint8 tensor, bitlen int32 tensor,
    token checksum int32 tensor)."""
    bitlen = torch.empty(max(n_win, 1), dtype=torch.int32, device=values.device)
    crc = torch.empty(max(n_win, 1), dtype=torch.int32, device=values.device)
    nb = C.c_size_t()
    st = load().lmgc_encode_windows(ctx.handle, _ptr(values), values.numel(), first_win, n_win, None, 0, C.byref(nb),
                                    _ptr(bitlen), _ptr(crc), _stream(stream))
    if st != ERR_NO_SPACE:
        _check(ctx, st)
    out = torch.empty(max(nb.value, 1), dtype=torch.uint8, device=values.device)
    _check(ctx, load().lmgc_encode_windows(ctx.handle, _ptr(values), values.numel(), first_win, n_win, _ptr(out),
                                           out.numel(), C.byref(nb), _ptr(bitlen), _ptr(crc), _stream(stream)))
    return out[: nb.value], bitlen[:n_win], crc[:n_win]


def lmgc_container_header(ctx: Context, n: int) -> bytes:
    buf = (C.c_uint8 * 64)()
    _check(ctx, load().lmgc_container_header(ctx.handle, n, buf))
    return bytes(buf)


def lmgc_encode_host(ctx: Context, values: torch.Tensor, out: torch.Tensor, stream=None) -> int:
    """values and out are CPU tensors (pinned for asynchronous copies); returns container bytes."""
    nb = C.c_size_t()
    _check(ctx, load().lmgc_encode_host(ctx.handle, _ptr(values), values.numel(), _ptr(out), out.numel(),
                                        C.byref(nb), _stream(stream)))
    return nb.value


def lmgc_decode_batch_windows(ctx: Context) -> int:
    """Windows lmgc_decode would take per batch with the device memory free now."""
    n = C.c_size_t()
    _check(ctx, load().lmgc_decode_batch_windows(ctx.handle, C.byref(n)))
    return n.value


def lmgc_decode(ctx: Context, container: torch.Tensor, win_ids, out: torch.Tensor | None = None,
                stream=None) -> torch.Tensor:
    ids = (C.c_uint32 * max(len(win_ids), 1))(*[int(w) for w in win_ids])
    W = ctx.cfg.window
    if out is None:
        out = torch.zeros((len(win_ids), W), dtype=torch.int16, device=container.device)
    _check(ctx, load().lmgc_decode(ctx.handle, _ptr(container), container.numel(), ids, len(win_ids), _ptr(out),
                                   out.numel(), _stream(stream)))
    return out


def lmgc_stage_times(ctx: Context) -> list[float]:
    ms = (C.c_float * 5)()
    _check(ctx, load().lmgc_stage_times(ctx.handle, ms, 5))
    return list(ms)


def lmgc_launch_count() -> int:
    n = C.c_uint64()
    _check(None, load().lmgc_launch_count(C.byref(n)))
    return n.value


def lmgc_profile(ctx: Context | None, enable: bool) -> None:
    """ctx None: the process-wide counters of the context-free entry points."""
    _check(ctx, load().lmgc_profile(ctx.handle if ctx is not None else None, int(enable)))


def lmgc_kernel_stats(ctx: Context | None) -> dict:
    out = {}
    for cls in range(len(KERNEL_CLASSES)):
        name = C.create_string_buffer(32)
        launches, ms, work = C.c_int(), C.c_float(), C.c_double()
        _check(ctx, load().lmgc_kernel_stats(ctx.handle if ctx is not None else None, cls, name, 32,
                                             C.byref(launches), C.byref(ms), C.byref(work)))
        out[name.value.decode()] = dict(launches=launches.value, ms=ms.value, work=work.value)
    return out


def lmgc_create(cfg: ModelConfig) -> Context:
    return Context(cfg)


def lmgc_destroy(ctx: Context) -> None:
    ctx.close()


def lmgc_last_error(ctx: Context | None) -> str:
    buf = C.create_string_buffer(512)
    load().lmgc_last_error(ctx.handle if ctx is not None else None, buf, 512)
    return buf.value.decode(errors="replace")
