"""CPU checks of the C ABI: the library builds, loads and exports every entry point that
include/crvq.h declares; host-only functions agree with the oracle; argument validation
rejects bad calls before anything reaches a GPU. No GPU needed."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import crvq_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2412_09282_gb300 import build
    build.build()
    from paper_2412_09282_gb300 import _lib
    return _lib.load()


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "crvq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(crvq_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_entry_points():
    names = _declared_symbols()
    for required in ["crvq_hessian", "crvq_select_reorder_channels", "crvq_kmeans_init",
                     "crvq_encode_beam", "crvq_update_codebook", "crvq_reconstruct_error"]:
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    from paper_2412_09282_gb300 import _lib
    for name in _declared_symbols():
        assert hasattr(lib, name), name
        assert name in _lib.SIGNATURES, f"{name} has no ctypes signature"


def test_avg_bits_and_crit_groups_match_oracle(lib):
    import paper_2412_09282_gb300 as P
    for e, d, m, lam in [(8, 8, 1, 0.0), (8, 8, 4, 0.02), (10, 8, 2, 0.05), (12, 16, 3, 0.1)]:
        for M, N in [(4096, 4096), (11008, 4096), (512, 512)]:
            for ip in (False, True):
                assert P.crvq_avg_bits(e, d, m, lam, M, N, ip) == pytest.approx(
                    O.avg_bits(e, d, m, lam, M, N, ip), rel=1e-12)
                for nb in (1, 2, 3):
                    assert P.crvq_avg_bits_bases(e, d, nb, m - 1, lam, M, N, ip) == \
                        pytest.approx(O.avg_bits(e, d, m, lam, M, N, ip, n_base=nb), rel=1e-12)
    assert np.isnan(P.crvq_avg_bits_bases(8, 8, 0, 1, 0.02))
    assert np.isnan(P.crvq_avg_bits_bases(8, 8, 1, -1, 0.02))
    for N, d, lam in [(512, 8, 0.02), (4096, 8, 0.02), (11008, 8, 0.01), (8192, 8, 0.05),
                      (64, 8, 0.0), (64, 8, 1.0), (64, 8, 0.125), (8, 8, 0.5)]:
        assert P.crvq_n_crit_groups(N, d, lam) == O.n_crit_groups(N, d, lam)


def test_validation_rejects_before_launch(lib):
    c = ctypes
    # d other than 8 is unsupported; NULL pointers are invalid
    assert lib.crvq_hessian(None, 1, 8, 16, 0.0, None, None, None, None, None) == -2
    assert lib.crvq_hessian(None, 1, 8, 8, 0.0, None, None, None, None, None) == -1
    assert b"NULL" in lib.crvq_last_error()
    dummy = c.c_void_p(16)
    # N not a multiple of d
    assert lib.crvq_hessian(dummy, 4, 12, 8, 0.0, dummy, dummy, None, None, None) == -1
    # negative damping
    assert lib.crvq_hessian(dummy, 4, 16, 8, -1.0, dummy, dummy, None, None, None) == -1
    # blocks-only Hessian: same rules, H_blocks required
    assert lib.crvq_hessian_blocks(None, 1, 8, 16, 0.0, None, None, None, None, None) == -2
    assert lib.crvq_hessian_blocks(dummy, 4, 16, 8, 0.0, None, None, None, None, None) == -1
    assert lib.crvq_hessian_blocks(dummy, 4, 12, 8, 0.0, None, None, None, dummy, None) == -1
    assert lib.crvq_hessian_blocks(dummy, 0, 16, 8, 0.0, None, None, None, dummy, None) == -1
    # beam width beyond the implemented maximum
    from paper_2412_09282_gb300 import _lib
    cb = (_lib.crvq_codebook * 1)()
    cb[0] = _lib.crvq_codebook(16, 4, 0, 32, 2, 2)
    assert lib.crvq_encode_beam(dummy, 16, 2, 2, 8, dummy, cb, 1, 0, 17, 0, None, None) == -2
    assert lib.crvq_encode_beam(dummy, 16, 2, 2, 8, dummy, cb, 1, 0, 0, 0, None, None) == -1
    # n_fixed must leave a searched codebook
    assert lib.crvq_encode_beam(dummy, 16, 2, 2, 8, dummy, cb, 1, 1, 1, 0, None, None) == -1
    # ldT too small for the set
    assert lib.crvq_encode_beam(dummy, 8, 2, 2, 8, dummy, cb, 1, 0, 1, 0, None, None) == -1
    # more groups than a grid row per group allows
    big = 65536
    cb[0] = _lib.crvq_codebook(16, 4, 0, 32, big, big)
    assert lib.crvq_encode_beam(dummy, 8 * big, 1, big, 8, dummy, cb, 1, 0, 2, 0, None,
                                None) == -2
    assert b"65535 groups" in lib.crvq_last_error()
    cb[0] = _lib.crvq_codebook(16, 4, 0, 32, 2, 2)
    # codebook coverage beyond the set
    cb[0] = _lib.crvq_codebook(16, 4, 0, 32, 4, 3)
    assert lib.crvq_update_codebook(dummy, 16, 2, 2, 8, dummy, cb, 1, 0, dummy, None,
                                    None) == -1
    # K larger than the number of vectors for k-means init
    assert lib.crvq_kmeans_init(dummy, 16, 2, 2, 8, None, 0, 5, 0, dummy, None) == -1
    # crit_frac outside [0, 1]
    gc = c.c_int64(0)
    assert lib.crvq_select_reorder_channels(dummy, 2, 16, 8, dummy, dummy, dummy, 1.5, 0, 0,
                                            dummy, None, dummy, dummy, c.byref(gc), None) == -1
    # inference product: more than 8 inputs unsupported; row strides below the sizes invalid
    cb[0] = _lib.crvq_codebook(16, 4, 0, 32, 2, 2)
    assert lib.crvq_lut_matvec(dummy, 16, 9, 16, 8, None, cb, 1, 2, dummy, 2, None) == -2
    assert lib.crvq_lut_matvec(dummy, 8, 1, 16, 8, None, cb, 1, 2, dummy, 2, None) == -1
    assert lib.crvq_lut_matvec(dummy, 16, 1, 16, 8, None, cb, 1, 2, dummy, 1, None) == -1
    assert lib.crvq_lut_matvec(dummy, 16, 1, 12, 8, None, cb, 1, 2, dummy, 2, None) == -1
    # unknown importance mode
    assert lib.crvq_select_reorder_channels(dummy, 2, 16, 8, dummy, dummy, dummy, 0.5, 7, 0,
                                            dummy, None, dummy, dummy, c.byref(gc), None) == -1


def test_step_calls_refuse_host_memory_before_launch(lib):
    """Valid shapes and options but host pointers: every step call returns
    CRVQ_ERR_INVALID_ARG naming the array, instead of handing the pointer to a kernel."""
    from paper_2412_09282_gb300 import _lib
    c = ctypes
    buf = (c.c_float * 4096)()
    host = c.c_void_p((c.addressof(buf) + 15) // 16 * 16)       # 16-byte aligned host memory
    cb = (_lib.crvq_codebook * 1)()
    cb[0] = _lib.crvq_codebook(host.value, 4, 0, host.value, 2, 2)
    gc = c.c_int64(0)
    calls = [
        lambda: lib.crvq_hessian(host, 4, 16, 8, 0.0, host, host, None, None, None),
        lambda: lib.crvq_hessian_blocks(host, 4, 16, 8, 0.0, None, None, None, host, None),
        lambda: lib.crvq_select_reorder_channels(host, 2, 16, 8, host, host, host, 0.5, 0, 0,
                                                 host, None, host, host, c.byref(gc), None),
        lambda: lib.crvq_kmeans_init(host, 16, 2, 2, 8, None, 0, 2, 0, host, None),
        lambda: lib.crvq_encode_beam(host, 16, 2, 2, 8, host, cb, 1, 0, 1, 0, None, None),
        lambda: lib.crvq_update_codebook(host, 16, 2, 2, 8, host, cb, 1, 0, host, None, None),
        lambda: lib.crvq_update_codebook_noalloc(host, 16, 2, 2, 8, host, cb, 1, 0, host, None,
                                                 None),
        lambda: lib.crvq_lut_matvec(host, 16, 1, 16, 8, None, cb, 1, 2, host, 2, None),
        lambda: lib.crvq_reconstruct_error(host, 2, 16, 8, host, None, cb, 1, 0, None, 0, 0.0,
                                           None, (c.c_double * 3)(), None),
    ]
    for call in calls:
        assert call() == -1
        assert b"not device memory" in lib.crvq_last_error()


def test_quantize_layer_rejects_bad_shapes_and_options_before_launch(lib):
    """crvq_quantize_layer validates its shapes and configuration before any CUDA call."""
    from paper_2412_09282_gb300 import _lib
    c = ctypes
    dummy = c.c_void_p(16)
    outs = _lib.crvq_layer_outputs(dummy, dummy, dummy, dummy, dummy, None, None)
    rep = _lib.crvq_layer_report()

    def cfg(**kw):
        base = dict(d=8, K_base=256, n_ext=1, K_ext=256, crit_frac=0.02, B=8, kmeans_iters=10,
                    refine_rounds=1, eps_rel=1e-3, damp_rel=0.01, importance_mode=0, seed=0)
        base.update(kw)
        return _lib.crvq_config(**base)

    def call(M=512, N=512, n_tok=64, **kw):
        cf = cfg(**kw)
        return lib.crvq_quantize_layer(dummy, dummy, M, N, n_tok, c.byref(cf), c.byref(outs),
                                       c.byref(rep), None)

    assert call(d=16) == -2                       # only d = 8 is implemented
    assert call(N=500) == -1                      # N % d != 0
    assert call(N=49160) == -1                    # beyond the channel limit
    assert call(M=0) == -1
    assert call(n_tok=0) == -1
    assert call(K_base=0) == -1
    assert call(M=4, N=64, K_base=64) == -1       # K_base > M * G (32 vectors)
    assert call(n_ext=8) == -1                    # at most 7 extended codebooks
    assert call(n_base=-1) == -1
    assert call(n_base=2, n_ext=7) == -1          # at most 8 codebooks in all
    assert call(n_base=2**31 - 1) == -1
    assert b"n_base" in lib.crvq_last_error()
    assert call(crit_frac=1.5) == -1
    assert call(B=17) == -1
    assert call(kmeans_iters=-1) == -1
    assert call(importance_mode=4) == -1
    assert call(damp_rel=-1.0) == -1
    assert call(crit_frac=0.0) == -1              # extended codebooks need a critical group
    assert b"critical" in lib.crvq_last_error()
    # a NULL required pointer
    assert lib.crvq_quantize_layer(None, dummy, 512, 512, 64, c.byref(cfg()), c.byref(outs),
                                   c.byref(rep), None) == -1


_STRUCTS = ["crvq_codebook", "crvq_kernel_stat", "crvq_config", "crvq_layer_outputs",
            "crvq_layer_report"]


def _header_fields(struct):
    """Field names of `struct` as declared in include/crvq.h (comments removed)."""
    src = open(os.path.join(ROOT, "include", "crvq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = re.search(r"typedef struct " + struct + r"\s*\{(.*?)\}\s*" + struct + ";", src,
                     flags=re.S).group(1)
    return [re.search(r"\**\s*(\w+)\s*(\[\d+\])?$", decl.strip()).group(1)
            for decl in body.split(";") if decl.strip()]


def test_ctypes_structs_match_the_header_layout(tmp_path):
    """sizeof / offsetof of every struct of the ABI, as gcc lays out include/crvq.h, against the
    binding's ctypes declarations (field names in the same order)."""
    import shutil
    import subprocess
    from paper_2412_09282_gb300 import _lib
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "crvq.h"', 'int main(void) {']
    for s in _STRUCTS:
        lines.append(f'  printf("{s} size %zu\\n", sizeof({s}));')
        for f in _header_fields(s):
            lines.append(f'  printf("{s} {f} %zu\\n", offsetof({s}, {f}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o",
                    str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
    got = {tuple(l.split()[:-1]): int(l.split()[-1]) for l in out.splitlines()}
    for s in _STRUCTS:
        cls = getattr(_lib, s)
        assert [n for n, _ in cls._fields_] == _header_fields(s), s
        assert ctypes.sizeof(cls) == got[(s, "size")], s
        for n, _ in cls._fields_:
            assert getattr(cls, n).offset == got[(s, n)], (s, n)


def test_binding_raises_when_the_library_is_missing(tmp_path):
    """No CPU fallback: with the shared library absent, the first call raises ImportError."""
    import subprocess
    import sys
    code = (
        "import sys; sys.path.insert(0, %r)\n"
        "from paper_2412_09282_gb300 import _lib\n"
        "_lib.LIB_PATH = %r; _lib._lib = None\n"
        "try:\n"
        "    _lib.load()\n"
        "except ImportError as e:\n"
        "    print('raised', 'no CPU fallback' in str(e))\n"
        "else:\n"
        "    print('loaded')\n" % (ROOT, str(tmp_path / "libcrvq.so")))
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True,
                         timeout=300)
    assert out.stdout.strip() == "raised True", out.stdout + out.stderr
