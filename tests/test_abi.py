"""The C ABI without a GPU: the library builds, loads, exports every function
declared in include/*.h, and the binding's struct layouts match the header's
as compiled by the host C compiler.  No compute call is made."""
import ctypes as C
import glob
import os
import re
import subprocess

import pytest

from paper_2606_17081_gb300 import build as B
from paper_2606_17081_gb300 import routesim as rs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libpath():
    return B.build()


def _declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*[A-Za-z_][\w\s\*]*?\b([a-z_][a-z0-9_]*)\s*\(", text, flags=re.M):
            if m.group(1) not in ("if", "while", "for", "return", "sizeof"):
                names.add(m.group(1))
    return names


def test_every_declared_symbol_is_exported(libpath):
    declared = _declared_functions()
    assert set(rs.EXPORTS) <= declared
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True,
                         text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    missing = declared - exported
    assert not missing, missing
    L = C.CDLL(libpath)
    for name in declared:
        getattr(L, name)
    assert rs.lib() is not None


def test_struct_layout_matches_header(tmp_path, libpath):
    structs = {"rs_config": rs.rs_config, "rs_trace": rs.rs_trace,
               "rs_replica_params": rs.rs_replica_params,
               "rs_replica_result": rs.rs_replica_result, "rs_records": rs.rs_records,
               "rs_timing": rs.rs_timing}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "routesim.h"', 'int main(void){']
    for sname, cls in structs.items():
        lines.append(f'printf("{sname} %zu\\n", sizeof({sname}));')
        for f, _ in cls._fields_:
            lines.append(f'printf("{sname}.{f} %zu\\n", offsetof({sname}, {f}));')
    lines.append("return 0;}")
    src = tmp_path / "probe.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    got = dict(line.split() for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                       check=True).stdout.splitlines())
    for sname, cls in structs.items():
        assert int(got[sname]) == C.sizeof(cls), sname
        for f, _ in cls._fields_:
            assert int(got[f"{sname}.{f}"]) == getattr(cls, f).offset, (sname, f)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(rs, "LIB_PATH", str(tmp_path / "absent.so"))
    monkeypatch.setattr(rs, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        rs.lib()


def test_default_config_is_the_papers(libpath):
    c = rs.rs_config_default()
    assert (c.block_size, c.cap, c.hyst_k) == (16, 64, 3)
    assert (c.lat_a, c.lat_b, c.lat_d, c.w_c) == (0.005, 0.020, 0.010, 0.015)
    assert (c.dt, c.alpha, c.theta1, c.theta2, c.eps_frac) == (5.0, 0.3, 0.3, 2.0, 0.1)
    assert list(c.regime_tau)[1:] == [pytest.approx(0.7), pytest.approx(0.8)]
    assert list(c.regime_omega)[1:] == [1.0, pytest.approx(0.1)]
