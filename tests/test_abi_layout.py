"""The ctypes structures of the library binding (include/vlac.h) and of the
oracle's wrapper (oracle/orc.h) match their C headers field by field: the
size of every struct and the offset of every member, as a C compiler lays
them out (gcc on the host; no GPU)."""
import ctypes as C
import os
import shutil
import subprocess

import pytest

import oracle
from paper_2608_10824_gb300 import vlac

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
# header directory, header, {C struct: ctypes structure}; each header is
# compiled in a program of its own
HEADERS = [
    ("include", "vlac.h", {"vlac_dims": vlac.Dims, "vlac_weights": vlac.Weights, "vlac_rational": vlac.Rational,
                           "vlac_step_opts": vlac.StepOpts, "vlac_step_out": vlac.StepOut}),
    ("oracle", "orc.h", {"orc_dims": oracle._Dims, "orc_weights": oracle._Weights, "orc_opts": oracle._Opts,
                         "orc_out": oracle._Out}),
]
CASES = [(h, cname, py) for _, h, structs in HEADERS for cname, py in structs.items()]


@pytest.fixture(scope="module")
def c_layout(tmp_path_factory):
    if shutil.which("gcc") is None:
        pytest.skip("no host C compiler")
    table = {}
    d = tmp_path_factory.mktemp("abi")
    for inc, header, structs in HEADERS:
        lines = ["#include <stdio.h>", "#include <stddef.h>", f'#include "{header}"', "int main(void) {"]
        for cname, py in structs.items():
            lines.append(f'  printf("{cname} sizeof %zu\\n", sizeof({cname}));')
            for fname, _ in py._fields_:
                lines.append(f'  printf("{cname} {fname} %zu\\n", offsetof({cname}, {fname}));')
        lines += ["  return 0;", "}"]
        src, exe = d / f"{header}.c", d / f"{header}.layout"
        src.write_text("\n".join(lines) + "\n")
        subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, inc), "-o", str(exe), str(src)], check=True)
        out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout
        for line in out.splitlines():
            s, f, v = line.split()
            table[(s, f)] = int(v)
    return table


@pytest.mark.parametrize("header,cname,py", CASES, ids=[c for _, c, _ in CASES])
def test_struct_matches_header(c_layout, header, cname, py):
    assert C.sizeof(py) == c_layout[(cname, "sizeof")], f"{header}: {cname}"
    for fname, _ in py._fields_:
        assert getattr(py, fname).offset == c_layout[(cname, fname)], f"{header}: {cname}.{fname}"
