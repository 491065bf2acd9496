"""The ctypes mirror of domino_head_weights has the C layout of include/domino.h (CPU): a small C
program compiled against the header prints sizeof and every field's offset, and the binding's
structure must agree field by field (a reordered or missing field would otherwise pass garbage
pointers to the library without any error)."""
import ctypes
import os
import shutil
import subprocess
import tempfile

import pytest

from paper_2605_29707_gb300 import binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FIELDS = [name for name, _ in binding.domino_head_weights._fields_]


def test_head_weights_layout_matches_the_header():
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lines = ["#include <stddef.h>", "#include <stdio.h>", '#include "domino.h"', "int main(void) {",
             '  printf("sizeof %zu\\n", sizeof(domino_head_weights));']
    lines += [f'  printf("{f} %zu\\n", offsetof(domino_head_weights, {f}));' for f in FIELDS]
    lines += ["  return 0;", "}"]
    with tempfile.TemporaryDirectory() as d:
        src, exe = os.path.join(d, "layout.c"), os.path.join(d, "layout")
        with open(src, "w") as f:
            f.write("\n".join(lines) + "\n")
        subprocess.run([cc, "-I", os.path.join(ROOT, "include"), src, "-o", exe], check=True, capture_output=True)
        out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    c = dict((k, int(v)) for k, v in (line.split() for line in out.splitlines()))
    assert c["sizeof"] == ctypes.sizeof(binding.domino_head_weights)
    for f in FIELDS:
        assert c[f] == getattr(binding.domino_head_weights, f).offset, f


def _prototypes():
    """{entry point: number of parameters} from the header's DOMINO_API declarations."""
    import re
    with open(os.path.join(ROOT, "include", "domino.h")) as f:
        text = re.sub(r"/\*.*?\*/", " ", f.read(), flags=re.S)  # drop comments
    out = {}
    for m in re.finditer(r"DOMINO_API\s+[\w\s\*]+?\b(domino_\w+)\s*\(([^)]*)\)\s*;", text):
        params = m.group(2).strip()
        out[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_binding_argument_counts_match_the_prototypes():
    """Every entry point the binding declares takes as many arguments as its C prototype."""
    protos = _prototypes()
    assert sorted(protos) == sorted(binding.SYMBOLS)
    lib = binding.load()
    for name, n in protos.items():
        argtypes = getattr(lib, name).argtypes
        assert argtypes is not None, name
        assert len(argtypes) == n, (name, len(argtypes), n)
