"""C ABI checks that need no GPU: the library builds and loads, exports every
function include/*.h declares, and rejects invalid arguments on the host
before any device work (no pointer below is ever dereferenced)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in sorted(os.listdir(os.path.join(ROOT, "include")))
           if f.endswith(".h")]


@pytest.fixture(scope="module")
def lib():
    from paper_2506_20194_gb300.build import build_library
    build_library()
    from paper_2506_20194_gb300 import duo
    return duo.load_library()


def _declared_functions():
    txt = "\n".join(open(h).read() for h in HEADERS)
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(duo_\w+)\s*\(", txt, flags=re.M)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for n in ("duo_pack", "duo_sparsify", "duo_spmspv", "duo_spmspv_multi", "duo_free",
              "duo_strerror", "duo_packed_query", "duo_packed_export", "duo_device_status",
              "duo_abi_version", "duo_sparsify_threshold", "duo_spmspv_threshold",
              "duo_calib_create", "duo_calib_precompute", "duo_calib_status", "duo_calib_query",
              "duo_calib_export", "duo_calib_score", "duo_calib_free", "duo_calib_prune"):
        assert n in names


def test_binding_types_every_declared_function(lib):
    """The Python binding sets argument and result types for every function
    include/*.h declares (no call goes through ctypes' int defaults)."""
    for n in _declared_functions():
        f = getattr(lib, n)
        assert f.argtypes is not None, f"{n}: no argtypes in the binding"
        assert f.restype is not None, f"{n}: no restype in the binding"


def test_calib_info_mirror_matches_header():
    """duo.py's ctypes mirror of duo_calib_info lists the header's fields in
    the header's order."""
    from paper_2506_20194_gb300 import duo
    txt = open(os.path.join(ROOT, "include", "duo_calib.h")).read()
    body = re.search(r"typedef struct duo_calib_info \{(.*?)\} duo_calib_info;", txt, flags=re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    fields = re.findall(r"(\w+)\s*[,;]", body)
    assert fields == [name for name, _ in duo._CalibInfo._fields_]


def test_library_exports_every_declared_symbol(lib):
    for n in _declared_functions():
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"


def test_abi_version_and_strerror(lib):
    assert lib.duo_abi_version() == 1
    from paper_2506_20194_gb300 import duo
    for code in (0, -1, -2, -3, -4, -5, -6):
        assert duo.duo_strerror(code) and duo.duo_strerror(code) != "unknown status code"
    assert duo.duo_strerror(-99) == "unknown status code"


FAKE = 0x10000   # never dereferenced: validation rejects every call first


def test_pack_argument_validation(lib):
    h = ctypes.c_void_p()
    EINVAL, ERANGE = -1, -4
    assert lib.duo_pack(None, 4, 4, 4, 1, None, ctypes.byref(h)) == EINVAL
    assert lib.duo_pack(FAKE, 4, 4, 4, 1, None, None) == EINVAL
    assert lib.duo_pack(FAKE, 0, 4, 4, 1, None, ctypes.byref(h)) == EINVAL
    assert lib.duo_pack(FAKE, 4, 0, 4, 1, None, ctypes.byref(h)) == EINVAL
    assert lib.duo_pack(FAKE, 4, 8, 4, 1, None, ctypes.byref(h)) == EINVAL     # ldw < in
    assert lib.duo_pack(FAKE, 4, 4, 4, 7, None, ctypes.byref(h)) == EINVAL     # fmt
    assert lib.duo_pack(FAKE + 1, 4, 4, 4, 1, None, ctypes.byref(h)) == EINVAL  # alignment
    assert lib.duo_pack(FAKE, 4, 65536, 65536, 1, None, ctypes.byref(h)) == ERANGE
    assert lib.duo_pack(FAKE, 70000, 4, 4, 0, None, ctypes.byref(h)) == ERANGE  # IDX16 rows
    assert h.value is None
    # Passes host validation; without a GPU (or with a non-device pointer)
    # the call still fails cleanly.
    assert lib.duo_pack(FAKE, 4, 4, 4, 1, None, ctypes.byref(h)) in (-1, -3)
    assert h.value is None


def test_sparsify_argument_validation(lib):
    EINVAL = -1
    assert lib.duo_sparsify(None, 8, 2, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify(FAKE, 0, 0, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify(FAKE, 65536, 2, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify(FAKE, 8, 9, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify(FAKE, 8, -1, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify(FAKE, 8, 2, None, FAKE, None) == EINVAL
    assert lib.duo_sparsify(FAKE + 1, 8, 2, FAKE, FAKE, None) == EINVAL


def test_spmspv_rejects_dead_or_fake_handles(lib):
    EINVAL = -1
    assert lib.duo_spmspv(None, FAKE, None, None, 2, FAKE, None) == EINVAL
    assert lib.duo_spmspv(FAKE, FAKE, None, None, 2, FAKE, None) == EINVAL   # not a live handle
    assert lib.duo_spmspv(FAKE, FAKE, FAKE, None, 2, FAKE, None) == EINVAL   # half a kept list
    arr = (ctypes.c_void_p * 5)(FAKE, FAKE, FAKE, FAKE, FAKE)
    assert lib.duo_spmspv_multi(arr, 5, FAKE, None, None, 2, arr, None) == EINVAL   # n > 4
    assert lib.duo_spmspv_multi(arr, 0, FAKE, None, None, 2, arr, None) == EINVAL


def test_threshold_entry_points_validate_before_launch(lib):
    EINVAL = -1
    arr = (ctypes.c_void_p * 5)(FAKE, FAKE, FAKE, FAKE, FAKE)
    assert lib.duo_spmspv_threshold(arr, 5, FAKE, 0x3800, arr, None) == EINVAL   # n > 4
    assert lib.duo_spmspv_threshold(arr, 0, FAKE, 0x3800, arr, None) == EINVAL
    assert lib.duo_spmspv_threshold(arr, 1, None, 0x3800, arr, None) == EINVAL   # no x
    assert lib.duo_spmspv_threshold(arr, 1, FAKE, 0x3800, arr, None) == EINVAL   # not a live handle
    assert lib.duo_sparsify_threshold(None, 16, 0x3800, FAKE, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify_threshold(FAKE, 0, 0x3800, FAKE, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify_threshold(FAKE, 65536, 0x3800, FAKE, FAKE, FAKE, None) == EINVAL
    assert lib.duo_sparsify_threshold(FAKE, 16, 0x3800, FAKE, FAKE, None, None) == EINVAL   # no count
    assert lib.duo_sparsify_threshold(FAKE + 1, 16, 0x3800, FAKE, FAKE, FAKE, None) == EINVAL   # misaligned


def test_free_and_query_reject_non_handles(lib):
    assert lib.duo_free(None) == 0
    assert lib.duo_free(FAKE) == -1
    from paper_2506_20194_gb300 import duo
    info = duo._Info()
    assert lib.duo_packed_query(FAKE, ctypes.byref(info)) == -1
    assert lib.duo_packed_export(FAKE, 0, FAKE, 16) == -1


def test_binding_fails_loudly_without_library(tmp_path):
    import paper_2506_20194_gb300.duo as duo
    saved = duo._lib
    try:
        duo._lib = None
        with pytest.raises(RuntimeError):
            duo.load_library(str(tmp_path / "missing.so"))
    finally:
        duo._lib = saved


def test_calib_argument_validation(lib):
    EINVAL = -1
    vp, i64 = ctypes.c_void_p, ctypes.c_int64
    lib.duo_calib_create.argtypes = [i64, i64, vp, ctypes.POINTER(vp)]
    lib.duo_calib_precompute.argtypes = [vp, vp, i64, ctypes.c_float, ctypes.c_int, vp]
    lib.duo_calib_score.argtypes = [vp, vp, i64, i64, vp, vp]
    lib.duo_calib_free.argtypes = [vp]
    lib.duo_calib_status.argtypes = [vp, vp]
    lib.duo_calib_export.argtypes = [vp, ctypes.c_int, vp, i64, vp]
    h = ctypes.c_void_p()
    assert lib.duo_calib_create(0, 8, None, ctypes.byref(h)) == EINVAL
    assert lib.duo_calib_create(8, 0, None, ctypes.byref(h)) == EINVAL
    assert lib.duo_calib_create(40000, 8, None, ctypes.byref(h)) == EINVAL
    assert lib.duo_calib_create(8, 8, None, None) == EINVAL
    assert h.value is None
    # an unknown handle is rejected before it is dereferenced
    assert lib.duo_calib_precompute(FAKE, FAKE, 1, 0.1, 1, None) == EINVAL
    assert lib.duo_calib_precompute(None, FAKE, 1, 0.1, 1, None) == EINVAL
    assert lib.duo_calib_score(FAKE, FAKE, 4, 8, FAKE, None) == EINVAL
    assert lib.duo_calib_status(FAKE, None) == EINVAL
    assert lib.duo_calib_export(FAKE, 0, FAKE, 32, None) == EINVAL
    lib.duo_calib_prune.argtypes = [vp, vp, i64, i64, ctypes.c_int, ctypes.c_int, vp, vp, vp]
    assert lib.duo_calib_prune(FAKE, FAKE, 4, 8, 50, 128, FAKE, None, None) == EINVAL
    assert lib.duo_calib_prune(None, FAKE, 4, 8, 50, 128, FAKE, None, None) == EINVAL
    assert lib.duo_calib_free(FAKE) == EINVAL
    assert lib.duo_calib_free(None) == 0


def test_copy_argument_validation(lib):
    """duo_copy rejects NULL ends and negative sizes before touching the
    GPU, accepts an empty copy at once; an unknown address is refused (EINVAL where CUDA can classify it,
    ECUDA where no device is present), never copied."""
    vp, i64 = ctypes.c_void_p, ctypes.c_int64
    lib.duo_copy.argtypes = [vp, vp, i64, vp]
    EINVAL, ECUDA = -1, -3
    assert lib.duo_copy(None, FAKE, 16, None) == EINVAL
    assert lib.duo_copy(FAKE, None, 16, None) == EINVAL
    assert lib.duo_copy(FAKE, FAKE, -1, None) == EINVAL
    assert lib.duo_copy(None, None, 0, None) == 0
    assert lib.duo_copy(FAKE, FAKE, 16, None) in (EINVAL, ECUDA)


@pytest.mark.parametrize("cname,pyname,header", [("duo_packed_info", "_Info", "duo.h"),
                                                  ("duo_calib_info", "_CalibInfo", "duo_calib.h")])
def test_struct_mirrors_match_the_c_layout(tmp_path, cname, pyname, header):
    """The ctypes mirrors have the C compiler's size and field offsets
    (a small C program prints them; gcc, no GPU)."""
    import shutil
    import subprocess
    from paper_2506_20194_gb300 import duo
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    mirror = getattr(duo, pyname)
    cfields = {"inp": "in"}   # Python keyword renamed in the mirror
    lines = [f'printf("%zu\\n", sizeof({cname}));']
    for name, _ in mirror._fields_:
        lines.append(f'printf("%zu\\n", offsetof({cname}, {cfields.get(name, name)}));')
    src = tmp_path / "layout.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "%s"\nint main(void) {\n%s\nreturn 0;\n}\n'
                   % (header, "\n".join(lines)))
    exe = tmp_path / "layout"
    subprocess.run([cc, "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    want = [ctypes.sizeof(mirror)] + [getattr(mirror, name).offset for name, _ in mirror._fields_]
    assert got == want

