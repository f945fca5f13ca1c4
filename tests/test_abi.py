"""The C-ABI library loads and exports every entry point the headers declare (no GPU needed)."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = re.sub(r"//[^\n]*", "", src)
        names |= set(re.findall(r"\b(zl_\w+)\s*\(", src))
    return names


@pytest.fixture(scope="module")
def lib():
    import paper_2608_07974_gb300 as pkg
    path = pkg.build()
    return ctypes.CDLL(path)


def test_library_exports_every_declared_symbol(lib):
    names = declared_symbols()
    assert len(names) >= 20
    for n in sorted(names):
        assert hasattr(lib, n), n


def test_binding_lists_every_declared_symbol():
    from paper_2608_07974_gb300 import binding
    assert set(binding.EXPORTS) == declared_symbols()


def test_bad_arguments_are_rejected_on_the_host(lib):
    """zl_create validates its arguments before touching the device."""
    from paper_2608_07974_gb300 import binding as b
    dims = b.zl_model_dims(0, 0, 4, 128, 4, 4, 344, 512, 64, 1e-5, 1e4)
    cfg = b.zl_train_cfg(0.5, 0, 1, 1e-3, 0.9, 0.999, 1e-8, 0.01, 1, 0, 0, 1.0, 0, 0, 1.0, 0)
    for bounds, K in ([[0, 3, 2], 2], [[0, 2, 5], 2], [[1, 4], 1], [[0, 4], 0]):
        with pytest.raises(b.ZLError) as e:
            b.zl_create(dims, K, bounds, cfg)
        assert e.value.status == b.ZL_ERR_ARG
    bad = b.zl_train_cfg(1.5, 0, 1, 1e-3, 0.9, 0.999, 1e-8, 0.01, 1, 0, 0, 1.0, 0, 0, 1.0, 0)
    with pytest.raises(b.ZLError):
        b.zl_create(dims, 2, [0, 2, 4], bad)
    odd = b.zl_model_dims(0, 0, 4, 130, 4, 4, 344, 512, 64, 1e-5, 1e4)
    with pytest.raises(b.ZLError):
        b.zl_create(odd, 2, [0, 2, 4], cfg)
    assert "zl_create" in b.last_error()
