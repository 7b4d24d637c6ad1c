"""The C-ABI library builds, loads without a GPU, and exports what the header declares."""
import ctypes
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mlkv_gpu.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mlkv_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    if not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2504_01506_gb300 import build

    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_interface():
    names = declared_functions()
    for must in ("mlkv_open", "mlkv_close", "mlkv_get", "mlkv_put", "mlkv_apply_grad", "mlkv_lookahead",
                 "mlkv_insert", "mlkv_find", "mlkv_export", "mlkv_dedup", "mlkv_sync"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_lists_every_symbol():
    from paper_2504_01506_gb300 import _lib

    assert sorted(_lib.EXPORTED) == declared_functions()


def test_config_layout_matches_header(tmp_path):
    """The ctypes Config mirrors struct mlkv_config field by field."""
    from paper_2504_01506_gb300._lib import Config

    fields = [f for f, _ in Config._fields_]
    prog = tmp_path / "layout.c"
    body = "".join(f'printf("{f} %zu\\n", offsetof(mlkv_config, {f}));' for f in fields)
    prog.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "mlkv_gpu.h"\n'
                    f'int main(void){{printf("size %zu\\n", sizeof(mlkv_config));{body}return 0;}}\n')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.dirname(HEADER), str(prog), "-o", str(exe)], check=True)
    out = dict(ln.split() for ln in subprocess.run([str(exe)], capture_output=True, text=True,
                                                   check=True).stdout.splitlines())
    assert int(out["size"]) == ctypes.sizeof(Config)
    for f in fields:
        assert int(out[f]) == getattr(Config, f).offset, f


def test_status_strings_without_gpu(lib):
    lib.mlkv_status_string.restype = ctypes.c_char_p
    assert lib.mlkv_status_string(5) == b"table full"
    assert lib.mlkv_status_string(0) == b"ok"


def test_null_and_bad_arguments_without_gpu(lib):
    """Host-side checks return at once, before any CUDA call."""
    lib.mlkv_get.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]
    assert lib.mlkv_get(None, None, 0, None, None) == 1
    assert lib.mlkv_open(None, None) == 1
    assert lib.mlkv_close(None) == 0


def test_binding_argument_counts_match_header(lib):
    """Every declared function takes as many arguments in the ctypes binding as
    the header declares (a dropped or extra parameter would pass pointers into
    the wrong places)."""
    from paper_2504_01506_gb300 import _lib

    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    arity = {}
    for m in re.finditer(r"\b(mlkv_[a-z_]+)\s*\(([^)]*)\)\s*;", src, flags=re.S):
        params = " ".join(m.group(2).split())
        arity[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    assert sorted(arity) == declared_functions()
    bound = _lib.load()
    for name, n in arity.items():
        assert len(getattr(bound, name).argtypes) == n, name


def test_binding_constants_match_header():
    """Status codes, kernel ids, flags and limits in the binding equal the header's."""
    from paper_2504_01506_gb300 import _lib

    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    defines = {m.group(1): int(m.group(2)) for m in re.finditer(r"#define MLKV_(\w+) (\d+)u?\b", src)}
    checked = 0
    for name, value in defines.items():
        if hasattr(_lib, name):
            assert getattr(_lib, name) == value, name
            checked += 1
    assert checked >= 20  # status codes, kernel ids, flags and limits
    assert re.search(r"#define MLKV_STALENESS_ASYNC INT64_MAX\b", src) and _lib.STALENESS_ASYNC == 2**63 - 1


def test_open_validates_its_config_without_gpu(lib):
    """mlkv_open checks every field before its first CUDA call: each bad config
    returns its status here, where no GPU is present."""
    from paper_2504_01506_gb300 import _lib

    bound = _lib.load()
    good = dict(dim=8, capacity=100, max_batch=10, lr=0.01, eps=1e-8, state_init=0.0, init_lo=-0.01,
                init_hi=0.01, seed=1, insert_on_miss=1, staleness_bound=0, hbm_cache_rows=0, flags=0, reserved=0)
    cases = [
        (dict(dim=0), _lib.ERR_INVALID), (dict(dim=1025), _lib.ERR_INVALID), (dict(dim=258), _lib.ERR_INVALID),
        (dict(capacity=0), _lib.ERR_INVALID), (dict(capacity=2**31 - 2), _lib.ERR_INVALID),
        (dict(max_batch=0), _lib.ERR_INVALID), (dict(max_batch=2**30), _lib.ERR_INVALID),
        (dict(reserved=1), _lib.ERR_INVALID), (dict(flags=1), _lib.ERR_INVALID),
        (dict(init_lo=0.5, init_hi=0.1), _lib.ERR_INVALID), (dict(init_lo=float("nan")), _lib.ERR_INVALID),
        (dict(staleness_bound=-1), _lib.ERR_INVALID),
        (dict(staleness_bound=1, hbm_cache_rows=1000), _lib.ERR_UNSUPPORTED),
        (dict(staleness_bound=_lib.STALENESS_ASYNC, hbm_cache_rows=1000), _lib.ERR_UNSUPPORTED),
        (dict(hbm_cache_rows=-1), _lib.ERR_INVALID),
        (dict(hbm_cache_rows=2 * 10 + 63), _lib.ERR_INVALID),  # below two batches and 64 lines
    ]
    for over, code in cases:
        cfg = _lib.Config(**dict(good, **over))
        h = ctypes.c_void_p()
        assert bound.mlkv_open(ctypes.byref(cfg), ctypes.byref(h)) == code, over
        assert not h.value, over


def test_fault_injection_arguments_without_gpu(lib):
    """mlkv_debug_fail only sets a host-side countdown: it works with no GPU and
    rejects an unknown kind or a negative count."""
    from paper_2504_01506_gb300 import _lib

    bound = _lib.load()
    assert bound.mlkv_debug_fail(99, 1) == _lib.ERR_INVALID
    assert bound.mlkv_debug_fail(_lib.FAULT_ALLOC, -1) == _lib.ERR_INVALID
    assert bound.mlkv_debug_fail(_lib.FAULT_ALLOC, 3) == _lib.OK
    assert bound.mlkv_debug_fail(_lib.FAULT_ALLOC, 0) == _lib.OK
    assert bound.mlkv_debug_fail(_lib.FAULT_COPY, 0) == _lib.OK
    assert bound.mlkv_debug_fail(_lib.FAULT_WAIT, 0) == _lib.OK
