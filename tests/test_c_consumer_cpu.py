"""The C ABI from plain C: a C99 program that includes include/isam.h, links
libisam.so and calls the entry points that need no GPU (version, the
host-side planners, argument errors).  It checks that the header compiles
as C, that the exported symbols link by name, and that results reach a C
caller unchanged."""
import os
import subprocess

import pytest

from paper_1810_09958_gb300 import build, isam

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "isam.h"

int main(void) {
    int g[8], r[7], d[4];
    const int caps[3] = {76, 38, 19};
    if (isam_version() != 100) return 10;
    if (isam_gemm_plan_for(8192, 8192, 8192, 0, 0, 1.0f, 152, 232448, caps, g) != ISAM_OK) return 11;
    if (isam_gru_plan_for(1, 32, 1024, 0, 152, 232448, r) != ISAM_OK) return 12;
    if (isam_dwsep_plan_for(56, 128, 256, 232448, d) != ISAM_OK) return 13;
    if (isam_gru_plan_for(1, 1, 80, 0, 152, 232448, r) != ISAM_ERR_UNSUPPORTED) return 14;
    if (strlen(isam_last_error_string()) == 0) return 15;
    if (isam_gemm(0, 4, 4, 0, 0, 1.0f, NULL, NULL, 0.0f, NULL) != ISAM_ERR_INVALID_ARG) return 16;
    if (isam_gru_plan_for(1, 32, 1024, 0, 152, 232448, r) != ISAM_OK) return 17;
    printf("gemm %d %d %d %d %d %d %d %d\n", g[0], g[1], g[2], g[3], g[4], g[5], g[6], g[7]);
    printf("gru %d %d %d %d %d %d %d\n", r[0], r[1], r[2], r[3], r[4], r[5], r[6]);
    printf("dwsep %d %d %d %d\n", d[0], d[1], d[2], d[3]);
    return 0;
}
"""


@pytest.fixture(scope="module")
def lib_dir():
    build.build()
    return os.path.dirname(isam.LIB_PATH)


def test_c_program_links_and_gets_the_python_plans(tmp_path, lib_dir):
    src = tmp_path / "consumer.c"
    exe = tmp_path / "consumer"
    src.write_text(PROGRAM)
    cc = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(src),
                         "-L", lib_dir, "-lisam", "-Wl,-rpath," + lib_dir, "-o", str(exe)],
                        capture_output=True, text=True, timeout=120)
    assert cc.returncode == 0, cc.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert run.returncode == 0, (run.returncode, run.stdout, run.stderr)
    got = {line.split()[0]: [int(v) for v in line.split()[1:]] for line in run.stdout.splitlines()}
    py_gemm = isam.gemm_plan(8192, 8192, 8192, 0, 0, 1.0, num_sms=152, smem_optin=232448, cluster_caps=[76, 38, 19])
    py_gru = isam.gru_plan(1, 32, 1024, False, num_sms=152, smem_optin=232448)
    py_dw = isam.dwsep_plan(56, 128, 256, smem_optin=232448)
    assert got["gemm"] == list(py_gemm.values())
    assert got["gru"] == list(py_gru.values())
    assert got["dwsep"] == list(py_dw.values())
