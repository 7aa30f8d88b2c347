"""The binding's ctypes mirrors of the C-ABI structs against the headers themselves.

A C program compiled from the headers in ``include/`` prints ``sizeof`` and the
``offsetof`` of every field the Python mirror names; a field added on one side
only, or in a different place, changes an offset or the size.
"""
import ctypes
import shutil
import subprocess
from pathlib import Path

import pytest

from paper_2606_15615_gb300 import moeca as M

ROOT = Path(__file__).resolve().parents[1]
STRUCTS = [(n, getattr(M, n)) for n in (
    "moeca_config", "moeca_layer_weights", "moeca_step_args", "moeca_stats", "moeca_layer_state",
    "moeca_layer_trace", "moeca_shard", "moeca_kernel_times", "moeca_route_args", "moeca_ddpm_args")]


def test_struct_layouts_match_the_header(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "moeca.h"', "int main(void) {"]
    expect = []
    for cname, py in STRUCTS:
        lines.append(f'  printf("%zu\\n", sizeof({cname}));')
        expect.append(ctypes.sizeof(py))
        for field, _ in py._fields_:
            lines.append(f'  printf("%zu\\n", offsetof({cname}, {field}));')
            expect.append(getattr(py, field).offset)
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-std=c11", f"-I{ROOT / 'include'}", str(src), "-o", str(exe)], check=True)
    got = [int(v) for v in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    assert got == expect
