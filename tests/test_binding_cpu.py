"""The C ABI library builds for sm_103a and exports every entry point that
include/f2gpu.h declares (no compute calls: no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    inc = os.path.join(ROOT, "include")
    for h in sorted(os.listdir(inc)):
        if h.endswith(".h"):
            with open(os.path.join(inc, h)) as f:
                text = re.sub(r"/\*.*?\*/", "", f.read(), flags=re.S)
            names |= set(re.findall(r"\b(f2_[a-z0-9_]+)\s*\(", text))
    return sorted(names)


@pytest.fixture(scope="module")
def libpath():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2608_20532_gb300 import binding

    return binding.library_path()


def test_header_declares_the_boundary():
    names = _declared()
    for required in ("f2_create", "f2_learn_batched", "f2_get_basis", "f2_solve_affine", "f2_encode_batched",
                     "f2_store_export", "f2_store_import", "f2_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    for name in _declared():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (f2_[a-z0-9_]+)", out))
    assert set(_declared()) <= exported


def test_binding_covers_every_symbol(libpath):
    from paper_2608_20532_gb300 import binding

    assert set(binding.EXPORTS) == set(_declared())
    lib = binding.load_library()
    assert lib.f2_status_string(0).decode() == "ok"
    assert "out of range" in lib.f2_status_string(3).decode()


def test_missing_library_fails_loudly(tmp_path):
    from paper_2608_20532_gb300 import binding

    with pytest.raises(RuntimeError):
        binding.load_library(str(tmp_path / "nope.so"))


def _header_constants():
    """Every F2_* enumerator and numeric #define of the headers, by value."""
    consts = {}
    inc = os.path.join(ROOT, "include")
    for h in sorted(os.listdir(inc)):
        if not h.endswith(".h"):
            continue
        with open(os.path.join(inc, h)) as f:
            text = re.sub(r"/\*.*?\*/", "", f.read(), flags=re.S)
        for name, val in re.findall(r"\b(F2_[A-Z0-9_]+)\s*=\s*(-?\d+)", text):
            consts[name] = int(val)
        for name, val in re.findall(r"#define\s+(F2_[A-Z0-9_]+)\s+(\d+)u?\b", text):
            consts[name] = int(val)
    return consts


def test_binding_constants_match_the_header():
    """The binding's status codes, flags and option numbers are the header's."""
    from paper_2608_20532_gb300 import binding

    consts = _header_constants()
    for prefix in ("F2_OK", "F2_ERR_", "F2_FLAG_", "F2_OPT_"):
        names = [n for n in consts if n.startswith(prefix)]
        assert names, prefix
        for n in names:
            assert getattr(binding, n, None) == consts[n], n
    ours = [n for n in dir(binding) if n.startswith(("F2_OPT_", "F2_ERR_", "F2_FLAG_"))]
    assert set(ours) <= set(consts), set(ours) - set(consts)
