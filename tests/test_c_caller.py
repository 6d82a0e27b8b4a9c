"""The public headers are plain C: a C99 program that includes all of them
compiles with warnings as errors, links against libsky_slice.so and runs
without a GPU (argument rejection and the host-side layer allocator).  The
sizes and field offsets it prints for every public struct must equal those of
the ctypes structures of the Python binding."""
import ctypes as C
import os
import shutil
import subprocess

import pytest

from paper_2202_11836_gb300 import _lib as L

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_c99_program_builds_and_runs(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    if not os.path.exists(L.LIB_PATH):
        from paper_2202_11836_gb300 import build
        build.build()
    libdir = os.path.dirname(L.LIB_PATH)
    exe = tmp_path / "abi_host"
    cmd = [cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic",
           "-I", os.path.join(ROOT, "include"), os.path.join(ROOT, "tests", "c", "abi_host.c"),
           "-L", libdir, "-lsky_slice", "-Wl,-rpath," + libdir, "-o", str(exe)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stderr
    out = r.stdout.strip().splitlines()
    lines = dict(line.split(" ", 1) for line in out if not line.startswith("layout "))
    layouts = {ln.split()[1]: list(map(int, ln.split()[2:])) for ln in out
               if ln.startswith("layout ")}
    structs = {"sky_slice_config": L.SkySliceConfig, "sky_layer_cost": L.SkyLayerCost,
               "sky_kernel_stat": L.SkyKernelStat, "sky_optimizer_config": L.SkyOptimizerConfig,
               "sky_alloc_problem": L.SkyAllocProblem}
    assert set(layouts) == set(structs)
    for cname, py in structs.items():
        want = [C.sizeof(py)] + [getattr(py, f).offset for f, _ in py._fields_]
        assert layouts[cname] == want, (cname, layouts[cname], want)
    assert lines["create"] == "SKY_ERR_INVALID_ARG 1"
    # Sec. IV-A even split of 9 layers on 3 devices
    assert lines["even"] == "SKY_OK 0 3 6 9"
    # the three times slower middle device ends with no more layers than the others
    st, *pi = lines["heuristic"].split()
    pi = list(map(int, pi))
    assert st == "SKY_OK" and pi[0] == 0 and pi[3] == 9
    assert pi[2] - pi[1] <= min(pi[1] - pi[0], pi[3] - pi[2]) and pi[2] - pi[1] < 3
    assert lines["launches"] == "0"
