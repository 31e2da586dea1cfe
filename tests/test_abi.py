"""The C-ABI library builds for sm_103a, loads, and exports every declared entry point.

No compute call is made here (no GPU is needed).
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h")]


def _declared():
    names = []
    for h in HEADERS:
        text = open(h).read()
        names += re.findall(r"^LR_API\s+[\w\s\*]+?\b(lr_\w+)\s*\(", text, flags=re.M)
    return names


@pytest.fixture(scope="module")
def lib():
    from paper_2607_18253_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_entry_points():
    names = _declared()
    assert len(names) == len(set(names))
    for must in ("lr_create", "lr_load_state", "lr_estimate_ttft", "lr_route", "lr_status"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_binding_covers_the_header():
    from paper_2607_18253_gb300 import router
    assert set(_declared()) == set(router.EXPORTED_SYMBOLS)


def test_strerror_without_gpu(lib):
    lib.lr_strerror.restype = ctypes.c_char_p
    lib.lr_strerror.argtypes = [ctypes.c_int]
    assert lib.lr_strerror(0) == b"ok"
    assert b"max_iters" in lib.lr_strerror(5)
    assert lib.lr_strerror(99) == b"unknown error"


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_2607_18253_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "from oracle" not in text, f
                assert "sfs_oracle" not in text, f


def test_workload_generator_is_deterministic():
    import numpy as np
    from paper_2607_18253_gb300 import workloads as W
    a = W.make_workload("pool64", num_queries=50)
    b = W.make_workload("pool64", num_queries=80)
    for name in ("n_run", "run_ctx", "run_dec", "n_wait", "wait_pre", "wait_dec"):
        assert np.array_equal(getattr(a, name), getattr(b, name))
    assert np.array_equal(a.prompt_len, b.prompt_len[:50])
    assert np.all(a.n_run <= a.max_seqs)
    assert a.run_ctx.shape == (64, a.cap_running)


def _prototypes():
    protos = {}
    for h in HEADERS:
        text = open(h).read()
        for m in re.finditer(r"^LR_API\s+[\w\s\*]+?\b(lr_\w+)\s*\((.*?)\);", text, flags=re.M | re.S):
            args = m.group(2).strip()
            protos[m.group(1)] = [" ".join(a.split()) for a in args.split(",")] if args not in ("", "void") else []
    return protos


def test_binding_argtypes_match_the_header(lib):
    # every parameter of every prototype against the binding's ctypes declaration:
    # a pointer for a pointer, the same width and kind for a scalar
    from paper_2607_18253_gb300 import router
    bound = router.load_library()
    scalar = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "float": ctypes.c_float,
              "double": ctypes.c_double, "int": ctypes.c_int}
    protos = _prototypes()
    assert set(protos) == set(_declared())
    for name, params in protos.items():
        at = getattr(bound, name).argtypes
        assert at is not None and len(at) == len(params), (name, params, at)
        for p, t in zip(params, at):
            if "*" in p:
                assert t in (ctypes.c_void_p, ctypes.c_char_p) or issubclass(t, ctypes._Pointer), (name, p, t)
            else:
                ctype = p.replace("const ", "").split()[0]
                assert ctypes.sizeof(t) == ctypes.sizeof(scalar[ctype]), (name, p, t)
                assert (t in (ctypes.c_float, ctypes.c_double)) == (ctype in ("float", "double")), (name, p, t)
