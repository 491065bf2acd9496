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
