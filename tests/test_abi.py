"""The C-ABI library: it loads, exports every symbol include/rpd.h declares, and its host
side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rpd.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(rpd_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def rpd():
    import paper_2609_36452_gb300 as m
    return m


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("rpd_create", "rpd_set_head", "rpd_step", "rpd_destroy", "rpd_step_batched",
              "rpd_step_host", "rpd_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(rpd):
    lib = ctypes.CDLL(rpd.lib_path)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_names_match_header(rpd):
    for n in declared_functions():
        assert callable(getattr(rpd, n)), n


def test_version_and_error_strings(rpd):
    assert b"sm_103a" in rpd.rpd_version()
    assert isinstance(rpd.rpd_last_error(), bytes)


@pytest.mark.parametrize("d,V,K,eps", [(60, 4096, 3, 1e-6), (4100, 4096, 3, 1e-6), (256, 100, 3, 1e-6),
                                       (256, 4096, 0, 1e-6), (256, 4096, 65, 1e-6),
                                       (256, 4096, 3, -1.0)])
def test_create_rejects_bad_shapes(rpd, d, V, K, eps):
    h = rpd.rpd_create(d, V, K, ctypes.c_float(eps))
    assert not h
    assert rpd.rpd_last_error() != b""


def test_null_context_is_rejected(rpd):
    stats = ctypes.c_void_p()
    rc = rpd.rpd_step(None, None, None, 4, ctypes.c_float(0.9), ctypes.c_float(1.0), None, None, stats)
    assert rc == rpd.RPD_ERR_INVALID_ARGUMENT
    assert rpd.rpd_set_rule(None, None) == rpd.RPD_ERR_INVALID_ARGUMENT
    assert rpd.rpd_set_head(None, None, None) == rpd.RPD_ERR_INVALID_ARGUMENT
    rpd.rpd_destroy(None)


def test_create_without_gpu_fails_cleanly(rpd):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = rpd.rpd_create(256, 4096, 3, ctypes.c_float(1e-6))
    assert not h
    assert rpd.rpd_last_error() != b""


def test_header_is_plain_c_and_links(rpd, tmp_path):
    """A C99 program that includes rpd.h, takes the address of every declared function and
    calls the ones that need no GPU compiles with gcc and links against the library."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    names = declared_functions()
    src = tmp_path / "use_rpd.c"
    src.write_text(
        "#include <stdio.h>\n#include \"rpd.h\"\n"
        "typedef void (*any_fn)(void);\n"
        "int main(void) {\n"
        "  any_fn fns[] = {" + ", ".join(f"(any_fn){n}" for n in names) + "};\n"
        "  rpd_rule r = {0.6f, 3.5f, 15.0f, 6, 32, 0};\n"
        "  int rc = rpd_set_rule(NULL, &r);\n"
        "  printf(\"%d %d %s\\n\", (int)(sizeof(fns) / sizeof(fns[0])), rc, rpd_version());\n"
        "  return rc == RPD_ERR_INVALID_ARGUMENT ? 0 : 1;\n"
        "}\n")
    exe = tmp_path / "use_rpd"
    libdir = os.path.dirname(rpd.lib_path)
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-pedantic-errors", "-I",
                        os.path.join(ROOT, "include"), str(src), "-o", str(exe), "-L", libdir,
                        "-lrpd", f"-Wl,-rpath,{libdir}"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True)
    assert run.returncode == 0, run.stdout + run.stderr
    assert run.stdout.split()[0] == str(len(names))


def test_binding_refuses_tensors_the_abi_would_misread(rpd):
    """The Python binding checks side (host/device), element type, contiguity and size of
    every tensor before calling the C ABI, so a wrong tensor is an error, not a kernel
    reading the wrong memory."""
    import torch
    ok = torch.zeros(6, dtype=torch.int32)
    assert rpd._arg(ok, "x", "int32", 6, cuda=False) is not None
    bad = [
        (torch.zeros(6, dtype=torch.int32), dict(dtype="int32", numel=6, cuda=True)),     # host, not CUDA
        (torch.zeros(6, dtype=torch.int64), dict(dtype="int32", numel=6, cuda=False)),    # element type
        (torch.zeros(6, 2, dtype=torch.int32)[:, 0], dict(dtype="int32", numel=6, cuda=False)),  # strided
        (torch.zeros(5, dtype=torch.int32), dict(dtype="int32", numel=6, cuda=False)),    # size
        (None, dict(dtype="int32", numel=6, cuda=False)),
    ]
    for t, kw in bad:
        with pytest.raises(rpd.RpdError) as e:
            rpd._arg(t, "x", kw["dtype"], kw["numel"], cuda=kw["cuda"])
        assert e.value.code == rpd.RPD_ERR_INVALID_ARGUMENT
