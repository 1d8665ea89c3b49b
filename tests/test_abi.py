"""The C ABI without a GPU: the library loads, exports every entry point that the public
headers declare, and rejects invalid arguments on the host before any CUDA call."""
import ctypes as C
import re

import pytest

from conftest import ROOT
from paper_1805_08469_gb300 import _lib
from paper_1805_08469_gb300._build import build_library


def _declared():
    names = []
    for h in sorted((ROOT / "include").glob("*.h")):
        text = re.sub(r"/\*.*?\*/", "", h.read_text(), flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(gem_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def L():
    build_library()
    return _lib.lib()


def test_headers_declare_the_boundary():
    names = _declared()
    for must in ("gem_create", "gem_pull", "gem_commit", "gem_commit_batch", "gem_destroy",
                 "gem_set_theta", "gem_theta", "gem_set_stream", "gem_sync"):
        assert must in names


def test_every_declared_symbol_is_exported(L):
    missing = [n for n in _declared() if not hasattr(L, n)]
    assert not missing, missing


def test_host_side_argument_checks(L):
    h = C.c_void_p()
    assert L.gem_create(0, 4, 0.01, 0.9, 1e-8, C.byref(h)) == -1      # P = 0
    assert L.gem_create(10, 0, 0.01, 0.9, 1e-8, C.byref(h)) == -1     # n = 0
    assert L.gem_create(10, 4, 0.0, 0.9, 1e-8, C.byref(h)) == -1      # eta <= 0
    assert L.gem_create(10, 4, 0.01, 1.0, 1e-8, C.byref(h)) == -1     # mu >= 1
    assert L.gem_create(10, 4, 0.01, 0.9, 0.0, C.byref(h)) == -1      # eps <= 0
    assert L.gem_create(10, 4, 0.01, 0.9, float("nan"), C.byref(h)) == -1
    assert L.gem_create(10, 4, 0.01, 0.9, 1e-8, None) == -1
    assert L.gem_commit(None, 0, None) == -1
    assert L.gem_commit_batch(None, None, None, 0) == -1
    assert L.gem_sync(None) == -1
    L.gem_destroy(None)
    assert L.gem_launch_count(None) == 0
    assert L.gem_status_string(-3).decode().startswith("GEM_ECUDA")


def test_oracle_is_not_imported_by_the_product():
    pkg = ROOT / "paper_1805_08469_gb300"
    for f in list(pkg.rglob("*.py")) + list(pkg.rglob("*.cu")) + list(pkg.rglob("*.h")) + list(pkg.rglob("*.cpp")):
        text = f.read_text()
        assert "import oracle" not in text and "from oracle" not in text and "oracle/" not in text, f
