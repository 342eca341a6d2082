"""The C-ABI library builds, loads and exports what include/isjl_sim.h declares
(no compute calls: these run without a GPU)."""
import ctypes
import os
import re
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "isjl_sim.h")


@pytest.fixture(scope="module")
def built_lib():
    from paper_2608_02244_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]+?\b(isjl_\w+)\s*\(", text, re.M)))


def test_header_declares_expected_entry_points():
    from paper_2608_02244_gb300 import sim
    assert set(declared_functions()) == set(sim.EXPORTS)


def test_library_exports_every_declared_symbol(built_lib):
    for name in declared_functions():
        assert hasattr(built_lib, name), name


def test_binding_loads_and_status_strings(built_lib):
    from paper_2608_02244_gb300 import sim
    assert sim.lib() is not None
    assert sim.isjl_status_string(0) == "ok"
    assert "step limit" in sim.isjl_status_string(5)


def test_probe_rejects_bad_arguments_without_a_gpu(built_lib):
    """Argument checks come before any CUDA call."""
    from paper_2608_02244_gb300 import sim
    n, ms = ctypes.c_double(), ctypes.c_float()
    L = sim.lib()
    assert L.isjl_probe_int_rate(2, 10, None, ctypes.byref(n), ctypes.byref(ms)) == sim.ISJL_ERR_INVALID_ARG
    assert L.isjl_probe_int_rate(0, 0, None, ctypes.byref(n), ctypes.byref(ms)) == sim.ISJL_ERR_INVALID_ARG
    assert L.isjl_probe_int_rate(1, 10, None, None, ctypes.byref(ms)) == sim.ISJL_ERR_INVALID_ARG
    assert "internal" in sim.isjl_status_string(sim.ISJL_ERR_INTERNAL)


def test_ctypes_layout_matches_header():
    """Compile the header with gcc and compare sizes/offsets with the binding."""
    from paper_2608_02244_gb300 import sim
    prog = r"""
#include <stdio.h>
#include <stddef.h>
#include "isjl_sim.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu\n", sizeof(isjl_config), sizeof(isjl_instances), sizeof(isjl_outputs),
         sizeof(isjl_record), sizeof(isjl_summary));
  printf("%zu %zu %zu %zu\n", offsetof(isjl_record, status), offsetof(isjl_record, c_T),
         offsetof(isjl_summary, T_make), offsetof(isjl_summary, c_T));
  printf("%zu %zu\n", offsetof(isjl_config, c), offsetof(isjl_config, flags));
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        open(src, "w").write(prog)
        subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), src, "-o", exe], check=True)
        lines = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split("\n")
    sizes = [int(x) for x in lines[0].split()]
    assert sizes == [ctypes.sizeof(sim.isjl_config), ctypes.sizeof(sim.isjl_instances),
                     ctypes.sizeof(sim.isjl_outputs), ctypes.sizeof(sim.isjl_record),
                     ctypes.sizeof(sim.isjl_summary)]
    offs = [int(x) for x in lines[1].split()]
    assert offs == [sim.isjl_record.status.offset, sim.isjl_record.c_T.offset,
                    sim.isjl_summary.T_make.offset, sim.isjl_summary.c_T.offset]
    offs2 = [int(x) for x in lines[2].split()]
    assert offs2 == [sim.isjl_config.c.offset, sim.isjl_config.flags.offset]
    assert sim.RECORD_DTYPE.itemsize == sizes[3]


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    from paper_2608_02244_gb300 import sim
    monkeypatch.setattr(sim, "_lib", None)
    monkeypatch.setattr(sim, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        sim.lib()
