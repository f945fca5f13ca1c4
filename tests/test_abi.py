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


def _header_struct_fields(name):
    """(field, C type) pairs, in order, of `typedef struct { ... } name;` in include/zerolock.h."""
    src = open(os.path.join(ROOT, "include", "zerolock.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = re.search(r"typedef struct \{([^{}]*)\}\s*" + name + r"\s*;", src, flags=re.S).group(1)
    fields = []
    for decl in body.split(";"):
        decl = decl.strip()
        if decl:
            ctype, rest = decl.split(None, 1)
            fields += [(v.strip(), ctype) for v in rest.split(",")]
    return fields


@pytest.mark.parametrize("name", ["zl_model_dims", "zl_train_cfg"])
def test_binding_structs_match_the_header_layout(name):
    """The ctypes structures list the header's fields in the header's order, with C int / float types
    matching the declarations (a drift here would shift every later field across the ABI)."""
    from paper_2608_07974_gb300 import binding
    want = {"int": ctypes.c_int, "float": ctypes.c_float, "unsigned": ctypes.c_uint}
    fields = _header_struct_fields(name)
    st = getattr(binding, name)
    assert [f for f, _ in st._fields_] == [f for f, _ in fields]
    for (f, t), (_, ct) in zip(st._fields_, fields):
        assert t is want[ct], (f, ct, t)
    assert ctypes.sizeof(st) == 4 * len(fields)


def test_product_path_never_imports_the_oracle():
    """Nothing in the package or its CUDA sources refers to the oracle or the tests: the only way to
    compute is the library."""
    import ast
    pkg = os.path.join(ROOT, "paper_2608_07974_gb300")
    for py in glob.glob(os.path.join(pkg, "*.py")):
        tree = ast.parse(open(py).read())
        for node in ast.walk(tree):
            mods = []
            if isinstance(node, ast.Import):
                mods = [a.name for a in node.names]
            elif isinstance(node, ast.ImportFrom):
                mods = [node.module or ""]
            for mod in mods:
                assert not mod.split(".")[0] in ("oracle", "tests"), (py, mod)
    for src in glob.glob(os.path.join(pkg, "csrc", "*")):
        assert "oracle" not in open(src).read().lower(), src


def test_binding_refuses_to_load_without_the_library(monkeypatch):
    """With libzerolock.so absent the binding raises ImportError: there is no CPU fallback."""
    import importlib
    import sys
    from paper_2608_07974_gb300 import binding
    real = os.path.exists
    monkeypatch.setattr(os.path, "exists", lambda p: False if p == binding.LIB_PATH else real(p))
    saved = sys.modules.pop("paper_2608_07974_gb300.binding")
    try:
        with pytest.raises(ImportError):
            importlib.import_module("paper_2608_07974_gb300.binding")
    finally:
        sys.modules["paper_2608_07974_gb300.binding"] = saved


def _header_prototypes():
    """name -> list of parameter kinds ('ptr', 'int', 'float', 'size_t') for every zl_ function."""
    src = open(os.path.join(ROOT, "include", "zerolock.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    protos = {}
    for name, args in re.findall(r"\b(zl_\w+)\s*\(([^)]*)\)\s*;", src, flags=re.S):
        kinds = []
        for a in args.split(","):
            a = " ".join(a.split())
            if not a or a == "void":
                continue
            if "*" in a:
                kinds.append("ptr")
            elif a.startswith("size_t"):
                kinds.append("size_t")
            elif a.startswith("float"):
                kinds.append("float")
            else:
                assert a.startswith("int"), a
                kinds.append("int")
        protos[name] = kinds
    return protos


def test_binding_argument_types_match_the_header_prototypes():
    """Every entry point is called with the header's arity and argument kinds (pointer, int, float,
    size_t): a mismatch would pass garbage across the ABI without any error."""
    from paper_2608_07974_gb300 import binding
    kind = {ctypes.c_int: "int", ctypes.c_float: "float", ctypes.c_size_t: "size_t",
            ctypes.c_void_p: "ptr", ctypes.c_char_p: "ptr"}
    protos = _header_prototypes()
    assert set(protos) == set(binding.EXPORTS)
    for name, want in protos.items():
        got = getattr(binding._lib, name).argtypes
        assert got is not None, name
        got = [kind.get(t, "ptr" if hasattr(t, "contents") or issubclass(t, ctypes._Pointer) else repr(t))
               for t in got]
        assert got == want, (name, got, want)


# Argument checks that every single-kernel entry point makes before it touches the device. The
# non-NULL pointers below are placeholders that must never be dereferenced; the test runs only where
# no GPU is present, so even a wrongly accepted call cannot reach a kernel.
@pytest.mark.skipif(__import__("torch").cuda.is_available(), reason="placeholder pointers: host-only check")
def test_single_kernel_entry_points_reject_bad_arguments_on_the_host():
    from paper_2608_07974_gb300 import binding as b
    L = b._lib
    P = 256   # placeholder device address
    cases = [
        ("zl_op_local_loss", (1, None, None, P, 4, 8, 8, 1.0, 0, P, P, P, None)),        # z NULL
        ("zl_op_local_loss", (2, P, None, P, 4, 8, 8, 1.0, 0, P, P, P, None)),           # dtype
        ("zl_op_local_loss", (1, P, None, P, 0, 8, 8, 1.0, 0, P, P, P, None)),           # N = 0
        ("zl_op_local_loss", (1, P, None, P, 4, 8, 12, 1.0, 0, P, P, P, None)),          # ldz % 8
        ("zl_op_local_loss", (1, P, None, P, 4, 8, 8, 0.5, 0, P, P, P, None)),           # alpha < 1 without t
        ("zl_op_local_loss", (1, P, P, P, 4, 8, 8, 1.5, 0, P, P, P, None)),              # alpha > 1
        ("zl_op_local_loss", (1, P, P, P, 4, 8, 8, 0.5, 2, P, P, P, None)),              # kl_dir
        ("zl_op_local_loss", (1, P, None, P, (1 << 24) + 1, 8, 8, 1.0, 0, P, P, P, None)),  # N above 2^24
        ("zl_op_local_loss_noalloc", (1, P, None, P, 65537, 8, 8, 1.0, 0, P, P, None)),  # beyond the scratch
        ("zl_op_attention", (1, P, P, P, 2, 64, 4, 3, 64, None)),                        # H % Hkv
        ("zl_op_attention", (1, P, P, P, 2, 64, 4, 4, 130, None)),                       # hd > 128
        ("zl_op_attention", (1, P, P, P, 2, 64, 4, 4, 63, None)),                        # hd odd
        ("zl_op_attention_bwd", (1, P, P, P, P, None, 2, 64, 4, 4, 64, None)),           # dqkv NULL
        ("zl_op_gemm", (1, 3, 8, 8, 8, P, P, P, None)),                                  # mode
        ("zl_op_gemm", (1, 0, -1, 8, 8, P, P, P, None)),                                 # M < 0
        ("zl_op_gemm_ex", (1, 0, 8, 8, 8, P, P, P, None, None, 1, None)),                # r_mode 1 without R
        ("zl_op_gemm_ex", (1, 2, 8, 8, 8, P, P, P, None, P, 0, None)),                   # mode 2 with R
        ("zl_op_gemm_ex", (1, 2, 12, 8, 8, P, P, P, P, None, 0, None)),                  # column sums, M % 8
    ]
    for name, args in cases:
        assert getattr(L, name)(*args) == b.ZL_ERR_ARG, (name, args)
        assert b.last_error(), name
    assert L.zl_kernel_launches(None) == b.ZL_ERR_ARG
    for name in ("zl_step", "zl_bp_step", "zl_eval_global_loss"):
        assert getattr(L, name)(None, P, P, 1, 1, None) == b.ZL_ERR_ARG, name
    assert L.zl_synchronize(None, 0) == b.ZL_ERR_ARG
    L.zl_free(None)   # NULL-safe


def test_loss_bindings_reject_undersized_tensors_before_the_call():
    """The loss bindings check every tensor against the sizes the call reads or writes (N * ldz for z,
    t and dz; N for labels and per-row losses) and raise before any pointer reaches the library (CPU
    tensors stand in: a wrongly accepted call would fail on the host pointers, not pass)."""
    import torch
    from paper_2608_07974_gb300 import binding as b
    N, V, ldz = 4, 8, 8
    z, dz = torch.zeros(N * ldz), torch.zeros(N * ldz)
    lab, rl, loss = torch.zeros(N, dtype=torch.int32), torch.zeros(N), torch.zeros(1)
    short = torch.zeros(N * ldz - 1)
    cases = [dict(z=short), dict(dz=short), dict(t=short), dict(labels=torch.zeros(N - 1, dtype=torch.int32)),
             dict(row_loss=torch.zeros(N - 1)), dict(loss=torch.zeros(0))]
    for bad in cases:
        a = dict(z=z, t=None, labels=lab, dz=dz, row_loss=rl, loss=loss)
        a.update(bad)
        alpha = 0.5 if "t" in bad else 1.0
        with pytest.raises(b.ZLError) as e:
            b.zl_op_local_loss(b.ZL_DTYPE_F32, a["z"], a["t"], a["labels"], N, V, ldz, alpha, 0, a["dz"],
                               a["row_loss"], a["loss"])
        assert e.value.status == b.ZL_ERR_ARG, bad
        if "row_loss" not in bad:
            with pytest.raises(b.ZLError) as e:
                b.zl_op_local_loss_noalloc(b.ZL_DTYPE_F32, a["z"], a["t"], a["labels"], N, V, ldz, alpha, 0, a["dz"],
                                           a["loss"])
            assert e.value.status == b.ZL_ERR_ARG, bad
