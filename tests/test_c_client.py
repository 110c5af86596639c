"""The C ABI used from plain C: the header compiles as strict C99, and (on a GPU) a C client that
allocates with cudaMalloc and calls only libdtp reproduces the Python binding bit for bit, and its
bf16 pass through the allocation-free entry point equals the workspace entry point's."""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "dtp_c_client.c")
OUT = os.path.join(ROOT, "_build", "c_client")          # git-ignored
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _have_cuda_headers():
    return os.path.exists(os.path.join(CUDA, "include", "cuda_runtime.h"))


@pytest.mark.skipif(shutil.which("gcc") is None or not _have_cuda_headers(), reason="gcc or CUDA headers missing")
def test_header_and_client_compile_as_c99():
    os.makedirs(OUT, exist_ok=True)
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-Wno-long-long",
                        "-I", os.path.join(ROOT, "include"), "-isystem", os.path.join(CUDA, "include"),
                        "-c", SRC, "-o", os.path.join(OUT, "client.o")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


@pytest.mark.gpu
def test_c_client_matches_the_binding():
    import torch

    import oracle
    from paper_2609_13846_gb300 import build, dtp, synth
    lib = build.build()
    os.makedirs(OUT, exist_ok=True)
    exe = os.path.join(OUT, "client")
    r = subprocess.run(["gcc", "-std=c99", "-O2", "-I", os.path.join(ROOT, "include"), "-isystem",
                        os.path.join(CUDA, "include"), SRC, "-o", exe, "-L", os.path.dirname(lib), "-ldtp",
                        f"-Wl,-rpath,{os.path.dirname(lib)}", "-L", os.path.join(CUDA, "lib64"), "-lcudart",
                        f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}"], capture_output=True, text=True)
    if r.returncode != 0 and "ldtp" in r.stderr:
        # the library file is libdtp.so in the package directory; link it by path instead
        r = subprocess.run(["gcc", "-std=c99", "-O2", "-I", os.path.join(ROOT, "include"), "-isystem",
                            os.path.join(CUDA, "include"), SRC, "-o", exe, lib,
                            f"-Wl,-rpath,{os.path.dirname(lib)}", "-L", os.path.join(CUDA, "lib64"), "-lcudart",
                            f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    T, d, H, N, D = 300, 64, 4, 192, 2
    L = synth.make_layer(d, H, N, T, seed=21, dtype="f32", outliers=True)
    inp = os.path.join(OUT, "in.bin")
    outp = os.path.join(OUT, "out.bin")
    np.concatenate([L[k].numpy().ravel() for k in ("X", "C", "W_gate", "W_up")]).astype(np.float32).tofile(inp)
    run = subprocess.run([exe, inp, outp, str(T), str(d), str(H), str(N), str(D)], capture_output=True, text=True)
    assert run.returncode == 0, run.stderr
    raw = open(outp, "rb").read()
    A_c = np.frombuffer(raw[:H * N * 4], np.float32).reshape(H, N)
    h_c = np.frombuffer(raw[H * N * 4:H * N * 4 + H * 4], np.int32)
    nu_c = np.frombuffer(raw[H * N * 4 + H * 4:H * N * 4 + H * 4 + N * 4], np.int32)
    sq_c = int(np.frombuffer(raw[-8:], np.int64)[0])
    g = {k: v.to("cuda:0") for k, v in L.items()}
    A_py = dtp.affinity_accumulate(g["X"], g["C"], g["W_gate"], g["W_up"])
    lay = dtp.search_layout(A_py, D, 10)
    np.testing.assert_array_equal(A_c, A_py.cpu().numpy())
    np.testing.assert_array_equal(h_c, lay["h"].cpu().numpy())
    np.testing.assert_array_equal(nu_c, lay["nu"].cpu().numpy())
    assert sq_c == int(lay["score_q"])
    ref = oracle.affinity_fo(*(L[k].double().numpy() for k in ("X", "C", "W_gate", "W_up")))
    assert np.linalg.norm(A_c - ref) / np.linalg.norm(ref) <= 1e-5
    # bf16 through plain C: the allocation-free entry point equals the workspace one bit for bit and
    # its status reader reports DTP_OK
    assert "noalloc_equal 1 status 0" in run.stdout, run.stdout
