"""The C ABI: liblmgc.so builds for sm_103a and exports every entry point include/lmgc.h
declares (no GPU needed; nothing is computed)."""
import ctypes
import os
import re

from paper_2409_17836_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "lmgc.h")).read()
    return sorted(set(re.findall(r"^lmgc_status\s+(lmgc_\w+)\s*\(", text, flags=re.M)))


def test_library_exports_every_declared_symbol():
    path = B.build()
    lib = ctypes.CDLL(path)
    syms = declared_symbols()
    assert len(syms) >= 16
    missing = [s for s in syms if not hasattr(lib, s)]
    assert not missing, missing


def test_binding_names_match_header():
    from paper_2409_17836_gb300 import lmgc
    assert sorted(lmgc.SYMBOLS) == declared_symbols()
    for s in declared_symbols():
        assert callable(getattr(lmgc, s)), s


def test_config_layout_and_constants_match_header(tmp_path):
    """The binding's lmgc_config matches the header's struct field by field (offsets, size), and
    its status, dtype, separator and input-kind constants equal the header's enums: a C program
    compiled against include/lmgc.h prints them."""
    import subprocess

    from paper_2409_17836_gb300 import lmgc as L

    fields = [f for f, _ in L.Config._fields_]
    consts = {"OK": "LMGC_OK", "ERR_INVALID": "LMGC_ERR_INVALID", "ERR_NO_SPACE": "LMGC_ERR_NO_SPACE",
              "ERR_CUDA": "LMGC_ERR_CUDA", "ERR_CORRUPT": "LMGC_ERR_CORRUPT", "ERR_LIMIT": "LMGC_ERR_LIMIT",
              "ERR_NOMEM": "LMGC_ERR_NOMEM", "F32": "LMGC_F32", "BF16": "LMGC_BF16", "SEP_SPACE": "LMGC_SEP_SPACE",
              "SEP_COMMA": "LMGC_SEP_COMMA", "SEP_COMMA_SPACE": "LMGC_SEP_COMMA_SPACE", "SEP_SEMI": "LMGC_SEP_SEMI",
              "SEP_NONE": "LMGC_SEP_NONE", "IN_F32": "LMGC_IN_F32", "IN_U8": "LMGC_IN_U8"}
    src = ["#include <stdio.h>", "#include <stddef.h>", '#include "lmgc.h"', "int main(void) {",
           '  printf("size %zu\\n", sizeof(lmgc_config));']
    src += [f'  printf("off {f} %zu\\n", offsetof(lmgc_config, {f}));' for f in fields]
    src += [f'  printf("const {k} %d\\n", (int){v});' for k, v in consts.items()]
    src += ["  return 0;", "}"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src) + "\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {}
    for line in out:
        if line:
            kind, *rest = line.split()
            got[(kind, rest[0]) if kind != "size" else ("size",)] = int(rest[-1])
    assert got[("size",)] == ctypes.sizeof(L.Config)
    for f in fields:
        assert got[("off", f)] == getattr(L.Config, f).offset, f
    for k in consts:
        assert got[("const", k)] == getattr(L, k), k


def test_create_rejects_bad_configs_before_any_cuda_call():
    """lmgc_create validates the configuration before it touches the device, so every rejection
    is checkable without a GPU: INVALID and a message naming the problem."""
    from paper_2409_17836_gb300 import configs
    from paper_2409_17836_gb300 import lmgc as L

    lib = L.load()
    cases = [
        (dict(vocab=19), "bad model shape"),                              # the 20 reserved ids
        (dict(n_heads=3), "bad model shape"),                             # d_model % n_heads
        (dict(n_heads=4, n_kv_heads=3), "bad model shape"),               # n_heads % n_kv_heads
        (dict(d_model=96, n_heads=2, n_kv_heads=2), "head dim"),          # hd 48
        (dict(dtype=1), "head dim of a bf16 model"),                      # hd 32: no tcgen05 attention
        (dict(cdf_bits=31), "cdf_bits"),
        (dict(vocab=70000, cdf_bits=16), "cdf_bits"),                     # 2^P must exceed V
        (dict(dtype=7), "dtype"),
        (dict(sep_mode=5), "separator mode"),
        (dict(input_kind=2), "input kind"),
        (dict(byte_group=9), "byte_group"),
        (dict(byte_order=2), "byte_order"),
        (dict(alphabet=2), "alphabet"),
    ]
    for kw, fragment in cases:
        c = configs.with_(configs.TINY, **kw).c()
        h = ctypes.c_void_p()
        st = lib.lmgc_create(ctypes.byref(c), ctypes.byref(h))
        assert st == L.ERR_INVALID and not h.value, (kw, st)
        buf = ctypes.create_string_buffer(512)
        lib.lmgc_last_error(None, buf, 512)
        assert fragment in buf.value.decode(), (kw, buf.value)
