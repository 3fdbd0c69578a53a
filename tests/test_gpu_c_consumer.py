"""The compensated decode through the C ABI from plain C on a GPU (tests/c/decode_gpu.c): caches,
queries and bias in cudaMalloc'd memory, one bf16 and one fp32 decode, compared in the program
with a double-precision host softmax over the same rounded inputs."""
import os
import shutil
import subprocess

import pytest

import paper_2607_16213_gb300 as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


@pytest.mark.gpu
@pytest.mark.skipif(shutil.which("gcc") is None, reason="no C compiler")
def test_decode_from_c(tmp_path):
    from paper_2607_16213_gb300 import build as b
    b.build()
    lib = S.library_path()
    exe = tmp_path / "decode_gpu"
    libdirs = [d for d in (os.path.join(CUDA, "lib64"), os.path.join(CUDA, "lib")) if os.path.isdir(d)]
    cc = subprocess.run(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"),
                         "-I", os.path.join(CUDA, "include"), os.path.join(ROOT, "tests", "c", "decode_gpu.c"),
                         "-o", str(exe), "-L", os.path.dirname(lib), "-l:" + os.path.basename(lib),
                         *["-L" + d for d in libdirs], "-lcudart", "-lm",
                         "-Wl,-rpath," + ":".join([os.path.dirname(lib), *libdirs])],
                        capture_output=True, text=True)
    assert cc.returncode == 0, cc.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300)
    print(run.stdout)
    assert run.returncode == 0, run.stdout + run.stderr
    assert run.stdout.strip().endswith("done"), run.stdout
