"""The C-ABI library builds, loads without a GPU, exports every symbol the
header declares, and rejects bad arguments before launching anything (CPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def htam():
    from paper_2605_29734_gb300 import build

    build.build()
    from paper_2605_29734_gb300 import htam as mod

    return mod


def _declared_functions():
    text = open(os.path.join(ROOT, "include", "htam.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(htam_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("htam_build_memory", "htam_append_transitions", "htam_query"):
        assert required in names


def test_every_declared_symbol_is_exported(htam):
    lib = htam.lib()
    for name in _declared_functions():
        assert hasattr(lib, name), f"{name} declared in include/htam.h but not exported"
    assert set(htam.EXPORTS) == set(_declared_functions())


def test_status_strings(htam):
    for code in range(7):
        assert htam.lib().htam_status_string(code).startswith(b"HTAM_")


def _build(htam, **kw):
    args = dict(entries=16, gids=16, n=4, d=16, g=2, dtype=htam.HTAM_BF16, cap=8)
    args.update(kw)
    out = ctypes.c_void_p(123)
    rc = htam.lib().htam_build_memory(ctypes.c_void_p(args["entries"]), ctypes.c_void_p(args["gids"]),
                                      args["n"], args["d"], args["g"], args["dtype"], args["cap"],
                                      ctypes.c_void_p(0), ctypes.byref(out))
    return rc, out


@pytest.mark.parametrize("kw", [
    dict(d=12),              # not a multiple of 8
    dict(d=0),
    dict(d=32768),           # above the limit
    dict(g=0),
    dict(g=70000),
    dict(n=-1),
    dict(cap=2),             # capacity below n
    dict(cap=1 << 31),
    dict(dtype=7),
    dict(entries=0),         # null with n > 0
    dict(gids=0),
    dict(entries=8),         # misaligned
    dict(gids=4),
])
def test_build_rejects_bad_arguments_before_any_launch(htam, kw):
    rc, out = _build(htam, **kw)
    assert rc == htam.HTAM_EINVAL
    assert not out.value


def test_build_without_device_reports_no_device(htam):
    import torch

    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    rc, out = _build(htam)
    assert rc == htam.HTAM_ENODEV
    assert not out.value


def test_null_memory_is_rejected(htam):
    lib = htam.lib()
    p = htam.QueryParams(1, 1, 1.0, 0.0)
    z = ctypes.c_void_p(0)
    assert lib.htam_query(z, z, 0, ctypes.byref(p), z, z, z, z, z, z, z) == htam.HTAM_EINVAL
    assert lib.htam_query_host(z, z, 0, ctypes.byref(p), z, z, z, z, z, z, z) == htam.HTAM_EINVAL
    assert lib.htam_append_transitions(z, z, z, 1, z) == htam.HTAM_EINVAL
    assert lib.htam_memory_info(z, z, z, z, z) == htam.HTAM_EINVAL
    assert lib.htam_memory_group_counts(z, z) == htam.HTAM_EINVAL
    assert lib.htam_device_status(z, z) == htam.HTAM_EINVAL
    lib.htam_free_memory(z)  # no-op


def test_binding_without_the_library_fails_loudly(tmp_path):
    """No CPU fallback: a binding whose library is absent refuses to import."""
    import importlib.util
    import shutil

    pkg = tmp_path / "htam_copy"
    pkg.mkdir()
    shutil.copy(os.path.join(ROOT, "paper_2605_29734_gb300", "htam.py"), pkg / "htam.py")
    spec = importlib.util.spec_from_file_location("htam_copy_binding", pkg / "htam.py")
    module = importlib.util.module_from_spec(spec)
    with pytest.raises(ImportError, match="libhtam.so is missing"):
        spec.loader.exec_module(module)


def test_product_package_never_reaches_the_oracle():
    """The oracle is test infrastructure: nothing in the package imports it
    or names its library (the shared input generators only mention it)."""
    pkg = os.path.join(ROOT, "paper_2605_29734_gb300")
    for dirpath, _, files in os.walk(pkg):
        if "_build" in dirpath or "__pycache__" in dirpath:
            continue
        for name in files:
            if name.endswith((".py", ".cu", ".cuh", ".h", ".c")):
                text = open(os.path.join(dirpath, name)).read()
                assert not re.search(r"(import\s+oracle|from\s+oracle|htam_oracle)", text), os.path.join(dirpath, name)
