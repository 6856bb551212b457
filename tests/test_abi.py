"""The C-ABI library loads and exports every entry point include/mds.h
declares; host-side argument validation (no device work)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mds.h")
LIB = os.path.join(ROOT, "paper_2410_18234_gb300", "_lib", "libmds.so")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mds_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(LIB):
        from paper_2410_18234_gb300 import build
        build.build()
    return ctypes.CDLL(LIB)


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("mds_create", "mds_verify", "mds_verify_host", "mds_status", "mds_destroy"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_binding_mirrors_the_abi():
    from paper_2410_18234_gb300 import mds
    assert set(mds.EXPORTS) == set(_declared())
    for name in _declared():
        assert callable(getattr(mds, name, None)) or name in ("mds_error_string",), name


def test_error_strings(lib):
    lib.mds_error_string.restype = ctypes.c_char_p
    for code in (0, -1, -2, -3, -4, -5):
        assert lib.mds_error_string(code)
    assert b"unknown" in lib.mds_error_string(-99)


def test_create_rejects_bad_config_before_touching_a_device():
    from paper_2410_18234_gb300 import mds
    cases = [dict(max_B=0, K=2, L=4, V=100), dict(max_B=1, K=0, L=4, V=100), dict(max_B=1, K=17, L=4, V=100),
             dict(max_B=1, K=2, L=0, V=100), dict(max_B=1, K=2, L=65, V=100), dict(max_B=1, K=2, L=4, V=0),
             dict(max_B=1, K=2, L=4, V=(1 << 24) + 1)]
    for c in cases:
        with pytest.raises(mds.MdsError) as e:
            mds.mds_create(**c)
        assert e.value.code == mds.MDS_ESHAPE
    for c in (dict(wis_s=9), dict(is_h=-1.0), dict(cluster=3), dict(dtype=7), dict(omega0=-2),
              dict(omega0=mds.MDS_MAX_OMEGA0 + 1), dict(acc_prob=2), dict(acc_prob=-1), dict(top_k=-1),
              dict(top_k=mds.MDS_MAX_TOPK + 1)):
        with pytest.raises(mds.MdsError) as e:
            mds.mds_create(4, 2, 4, 100, **c)
        assert e.value.code == mds.MDS_EINVAL


def test_verify_rejects_null_context(lib):
    lib.mds_verify.restype = ctypes.c_int
    rc = lib.mds_verify(None, None, None, None, None, None, 0, ctypes.c_uint64(0), None, None, None, 1, None)
    assert rc == -1
    lib.mds_status.restype = ctypes.c_int
    assert lib.mds_status(None, None) == -1
    lib.mds_destroy(None)


def test_binding_config_matches_the_header():
    """The ctypes mirror of mds_config has the header's fields in order, and
    the scheme ids and limits agree."""
    from paper_2410_18234_gb300 import mds
    text = open(HEADER).read()
    body = re.search(r"typedef struct \{(.*?)\} mds_config;", text, flags=re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    fields = re.findall(r"\b(\w+)\s*;", body)
    assert [f[0] for f in mds.MdsConfig._fields_] == fields
    enum = re.search(r"typedef enum \{([^}]*)\} mds_scheme;", text).group(1)
    ids = dict((k, int(v)) for k, v in re.findall(r"(MDS_\w+)\s*=\s*(\d+)", enum))
    for name, sid in mds.SCHEMES.items():
        assert ids["MDS_" + name.upper()] == sid
    assert int(re.search(r"#define MDS_MAX_OMEGA0 (\d+)", text).group(1)) == mds.MDS_MAX_OMEGA0
    assert int(re.search(r"#define MDS_ST_OMEGA0 (\d+)u", text).group(1)) == mds.MDS_ST_OMEGA0
    assert int(re.search(r"#define MDS_MAX_TOPK (\d+)", text).group(1)) == mds.MDS_MAX_TOPK


def test_header_compiles_as_c_and_matches_the_binding_layout(tmp_path):
    """include/mds.h is plain C (C99), and mds_config's size and field
    offsets as a C compiler lays them out equal the ctypes mirror's."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    from paper_2410_18234_gb300 import mds
    fields = [f[0] for f in mds.MdsConfig._fields_]
    prints = "".join(f'printf("%zu\\n", offsetof(mds_config, {f}));' for f in fields)
    src = tmp_path / "layout.c"
    src.write_text('#include <stddef.h>\n#include <stdio.h>\n#include "mds.h"\n'
                   'int main(void) { printf("%zu\\n", sizeof(mds_config)); ' + prints + " return 0; }\n")
    exe = tmp_path / "layout"
    subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src), "-o",
                    str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    assert got[0] == ctypes.sizeof(mds.MdsConfig)
    assert got[1:] == [getattr(mds.MdsConfig, f).offset for f in fields]
