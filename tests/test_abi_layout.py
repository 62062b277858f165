"""The C ABI's structs seen from C: include/mtsim.h compiles as strict C99
and C++11, and every field's offset and the struct sizes that a C compiler
gives agree with the binding's numpy dtypes and ctypes structures."""
import ctypes
import os
import shutil
import subprocess

import pytest

from paper_2608_16336_gb300 import _build, mtsim

HEADER = os.path.join(_build.INCLUDE, "mtsim.h")

MIRRORS = {
    "sim_request_result_t": mtsim.RESULT_DTYPE,
    "sim_replica_stats_t": mtsim.STATS_DTYPE,
    "sim_migration_event_t": mtsim.EVENT_DTYPE,
    "sim_latency_stats_t": mtsim.LATENCY_DTYPE,
    "sim_cluster_t": mtsim.sim_cluster_t,
    "sim_tier_table_t": mtsim.sim_tier_table_t,
    "sim_policy_t": mtsim.sim_policy_t,
    "sim_launch_info_t": mtsim.sim_launch_info_t,
}


def _fields(mirror):
    """[(name, offset)] and the size of a numpy dtype or ctypes structure."""
    if isinstance(mirror, type) and issubclass(mirror, ctypes.Structure):
        return [(n, getattr(mirror, n).offset) for n, _ in mirror._fields_], ctypes.sizeof(mirror)
    return [(n, mirror.fields[n][1]) for n in mirror.names], mirror.itemsize


@pytest.fixture(scope="module")
def gcc():
    cc = shutil.which("gcc")
    if cc is None:
        pytest.skip("no C compiler")
    return cc


@pytest.mark.parametrize("std", ["c99", "c11"])
def test_header_is_strict_c(gcc, std):
    subprocess.run([gcc, "-std=" + std, "-Wall", "-Wextra", "-pedantic", "-Werror", "-fsyntax-only", "-x", "c",
                    HEADER], check=True)


def test_header_is_cxx(gcc):
    cxx = shutil.which("g++")
    if cxx is None:
        pytest.skip("no C++ compiler")
    subprocess.run([cxx, "-std=c++11", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-x", "c++", HEADER],
                   check=True)


def test_struct_layout_matches_binding(gcc, tmp_path):
    lines = ["#include <stddef.h>", "#include <stdio.h>", '#include "mtsim.h"', "int main(void) {"]
    for st, mirror in MIRRORS.items():
        names, _ = _fields(mirror)
        lines.append('    printf("%s size %%zu\\n", sizeof(%s));' % (st, st))
        for n, _ in names:
            lines.append('    printf("%s %s %%zu\\n", offsetof(%s, %s));' % (st, n, st, n))
    lines += ["    return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-I", _build.INCLUDE, str(src), "-o", str(exe)], check=True)
    got = {}
    for ln in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines():
        st, field, val = ln.split()
        got[(st, field)] = int(val)
    for st, mirror in MIRRORS.items():
        names, size = _fields(mirror)
        assert got[(st, "size")] == size, st
        for n, off in names:
            assert got[(st, n)] == off, (st, n)
