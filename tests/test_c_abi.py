"""The boundary from plain C: the header and a C caller compile as strict
C99 (no GPU needed), and on a GPU the caller links against the library and
runs a small decode/evict loop through the C ABI alone."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "abi_smoke.c")
CUDA_HOME = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _cc():
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc:
        pytest.skip("no C compiler")
    if not os.path.exists(os.path.join(CUDA_HOME, "include", "cuda_runtime_api.h")):
        pytest.skip("no CUDA headers")
    return cc


def test_header_and_c_caller_compile_as_c99():
    cc = _cc()
    cmd = [cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-fsyntax-only",
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA_HOME, "include"), SRC]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


@pytest.mark.gpu
def test_c_caller_runs_a_decode_evict_loop(tmp_path):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():  # pragma: no cover
        pytest.skip("needs a CUDA GPU")
    from paper_2607_10582_gb300 import build as mdbuild
    mdbuild.build()
    cc = _cc()
    libdir = os.path.join(ROOT, "paper_2607_10582_gb300")
    cudalib = os.path.join(CUDA_HOME, "lib64")
    exe = str(tmp_path / "abi_smoke")
    cmd = [cc, "-std=c99", "-O2", SRC, "-o", exe, "-I", os.path.join(ROOT, "include"),
           "-I", os.path.join(CUDA_HOME, "include"), "-L", libdir, "-lmemdecay", "-L", cudalib, "-lcudart",
           "-lm", f"-Wl,-rpath,{libdir}", f"-Wl,-rpath,{cudalib}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == "ok", (r.stdout, r.stderr)


def test_binding_constants_match_the_header():
    """Every limit and enumerator the Python binding mirrors has the header's
    value (the header is the boundary's definition)."""
    import re

    import paper_2607_10582_gb300 as md
    text = open(os.path.join(ROOT, "include", "memdecay.h")).read()
    defines = dict(re.findall(r"#define\s+(MD_\w+)\s+(-?\d+)\b", text))
    enums = dict(re.findall(r"\b(MD_\w+)\s*=\s*(-?\d+)\s*[,}\n/]", text))
    values = {**enums, **defines}
    for name in ("MD_MAX_BATCH", "MD_HEAD_DIM", "MD_MAX_GROUP", "MD_MAX_CHUNKS", "MD_MAX_CHUNK_TOKENS",
                 "MD_CALIB_BUCKETS", "MD_CALIB_BUCKET_WIDTH", "MD_OK", "MD_ERR_DEVICE_TIMEOUT"):
        assert name in values, name
    mirrored = [n for n in values if hasattr(md, n)]
    assert len(mirrored) >= 30
    for n in mirrored:
        assert getattr(md, n) == int(values[n]), n
