"""The binding matches the C header in include/regioncache.h: its ctypes
structures have every field's name, order and offset and the structure's
size as a C compiler (gcc, no GPU) lays them out, and every function's
argument and return types are those of its prototype."""
import ctypes
import os
import re
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "regioncache.h")
STRUCTS = ("rc_dims", "rc_layer_weights", "rc_global_weights", "rc_batch_item")


def header_fields(name):
    """Field names of `typedef struct name { ... } name;` in declaration order."""
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = re.search(r"typedef struct %s \{(.*?)\} %s;" % (name, name), src, flags=re.S).group(1)
    names = []
    for decl in body.split(";"):
        decl = decl.strip()
        if not decl:
            continue
        # "int a, b" / "const void* W" / "const int32_t* dirty_idx"
        head, *rest = decl.split(",")
        names.append(re.split(r"[\s*]+", head.strip())[-1])
        names += [r.strip().lstrip("*").strip() for r in rest]
    return names


@pytest.fixture(scope="module")
def c_layout():
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "regioncache.h"',
             "int main(void) {"]
    for s in STRUCTS:
        lines.append('printf("%s size %%zu\\n", sizeof(%s));' % (s, s))
        for f in header_fields(s):
            lines.append('printf("%s %s %%zu\\n", offsetof(%s, %s));' % (s, f, s, f))
    lines += ["return 0;", "}"]
    with tempfile.TemporaryDirectory(dir=os.path.join(ROOT, "tests")) as tmp:
        c_path, exe = os.path.join(tmp, "layout.c"), os.path.join(tmp, "layout")
        with open(c_path, "w") as fh:
            fh.write("\n".join(lines))
        subprocess.run([cc, "-std=c11", "-I", os.path.join(ROOT, "include"), c_path, "-o", exe],
                       check=True)
        out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    lay = {}
    for ln in out.splitlines():
        s, f, v = ln.split()
        lay.setdefault(s, {})[f] = int(v)
    return lay


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def test_ctypes_structures_match_the_header(R, c_layout):
    for s in STRUCTS:
        py = getattr(R, s)
        names = [n for n, _ in py._fields_]
        assert names == header_fields(s), s
        for n in names:
            assert getattr(py, n).offset == c_layout[s][n], f"{s}.{n}"
        assert ctypes.sizeof(py) == c_layout[s]["size"], s


def header_prototypes():
    """{name: (return kind, [parameter kinds])} of every function the header
    declares, kinds being ptr / int / float / double / u64 / none."""
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"#.*", "", src)

    def kind(decl):
        decl = decl.strip()
        if "*" in decl or decl.split()[0] == "rc_stream" or " rc_stream " in f" {decl} ":
            return "ptr"
        words = [w for w in re.split(r"\s+", decl) if w != "const"]
        t = words[0]
        return {"int": "int", "rc_status": "int", "int32_t": "int", "float": "float",
                "double": "double", "size_t": "u64", "uint64_t": "u64", "void": "none"}[t]

    out = {}
    for m in re.finditer(r"([A-Za-z_][\w\s\*]*?)\b(rc_\w+)\s*\(([^)]*)\)\s*;", src):
        ret, name, params = m.group(1), m.group(2), m.group(3).strip()
        ps = [] if params in ("", "void") else [kind(p) for p in params.split(",")]
        out[name] = (kind(ret + " x"), ps)
    return out


def ctypes_kind(t):
    if t is None:
        return "none"
    if t in (ctypes.c_void_p, ctypes.c_char_p) or hasattr(t, "_type_") and isinstance(
            t._type_, type):
        return "ptr"
    return {ctypes.c_int: "int", ctypes.c_float: "float", ctypes.c_double: "double",
            ctypes.c_size_t: "u64", ctypes.c_uint64: "u64"}[t]


def test_binding_signatures_match_the_header(R):
    protos = header_prototypes()
    assert set(protos) == set(R.header_symbols())
    for name, (ret, params) in protos.items():
        f = getattr(R._lib, name)
        assert f.argtypes is not None, f"{name}: no argtypes in the binding"
        got = [ctypes_kind(a) for a in f.argtypes]
        assert got == params, f"{name}: binding {got} vs header {params}"
        assert ctypes_kind(f.restype) == ret, f"{name}: return {f.restype} vs {ret}"
