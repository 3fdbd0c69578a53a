"""include/selkv.h from plain C: a C11 program (tests/c/consumer.c) compiles against the header,
links libselkv.so and runs its host-side checks (no GPU needed: no call reaches a launch)."""
import os
import shutil
import subprocess

import pytest

import paper_2607_16213_gb300 as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("gcc") is None, reason="no C compiler")
def test_header_compiles_as_c_and_links(tmp_path):
    from paper_2607_16213_gb300 import build as b
    b.build()
    lib = S.library_path()
    exe = tmp_path / "consumer"
    cc = subprocess.run(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
                         os.path.join(ROOT, "tests", "c", "consumer.c"), "-o", str(exe),
                         "-L", os.path.dirname(lib), "-l:" + os.path.basename(lib),
                         "-Wl,-rpath," + os.path.dirname(lib)], capture_output=True, text=True)
    assert cc.returncode == 0, cc.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert run.returncode == 0, run.stdout + run.stderr
    assert run.stdout.strip().endswith("done"), run.stdout
