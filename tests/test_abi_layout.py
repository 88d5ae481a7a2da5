"""The binding's ctypes structures have the C header's layout: every field's
name, order, offset and the structure's size, as a C compiler lays them out
from include/regioncache.h (gcc, no GPU)."""
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
