"""The C ABI used from C: tests/c/abi_step.c includes include/geocache.h,
links libgeocache.so and drives one correspondence build (Sec. 3.2,
correspondence operator), one anchor rotation and one cached step with DDIM
reconstruction (Eq. 1, closed-form conversion) with device memory from the
CUDA runtime.  On the CPU the program is compiled and linked (the header is
valid C11 and every call it makes resolves); on the GPU it runs and its
outputs are compared with the oracle."""
import os
import subprocess

import numpy as np
import pytest

import oracle
from paper_2608_13255_gb300 import build as gbuild
from paper_2608_13255_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "abi_step.c")


def _cuda_root():
    return os.path.dirname(os.path.dirname(gbuild.nvcc()))


def _compile(out_dir):
    lib = gbuild.build()
    exe = os.path.join(out_dir, "abi_step")
    cuda = _cuda_root()
    cmd = ["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-O1", "-I", os.path.join(ROOT, "include"),
           "-I", os.path.join(cuda, "include"), SRC, lib, "-L", os.path.join(cuda, "lib64"), "-lcudart",
           "-Wl,-rpath," + os.path.dirname(lib) + ":" + os.path.join(cuda, "lib64"), "-o", exe]
    res = subprocess.run(cmd, capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    return exe


def test_c_caller_compiles_and_links(tmp_path):
    exe = _compile(str(tmp_path))
    assert os.access(exe, os.X_OK)


@pytest.mark.gpu
def test_c_caller_matches_oracle(tmp_path):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    exe = _compile(str(tmp_path))
    w = synth.make_workload("tiny")
    rng = np.random.default_rng(31)
    shp = (w.B, w.N, w.C, w.H, w.W)
    x0_prev = rng.standard_normal(shp, dtype=np.float32)
    x_t = rng.standard_normal(shp, dtype=np.float32)
    delta = (0.1 * rng.standard_normal(shp)).astype(np.float32)
    inp, outp = str(tmp_path / "in.bin"), str(tmp_path / "out.bin")
    with open(inp, "wb") as f:
        f.write(np.array([w.B, w.N, w.H, w.W, w.C], np.int32).tobytes())
        for a, dt in ((w.pos, np.float32), (w.valid, np.uint8), (w.cams, np.float32), (x0_prev, np.float32),
                      (x_t, np.float32), (delta, np.float32)):
            f.write(np.ascontiguousarray(a, dtype=dt).tobytes())
    res = subprocess.run([exe, inp, outp], capture_output=True, text=True, timeout=120)
    assert res.returncode == 0, res.stderr + res.stdout
    raw = open(outp, "rb").read()
    anchors = list(np.frombuffer(raw[:8], np.int32))
    sched = {"kind": "single_cached"}
    assert anchors == oracle.rotate_anchors(w.N, 2, oracle.cached_ordinal(1, 2, sched)) == [0, 3]
    n = int(np.prod(shp))
    tau = np.frombuffer(raw[8:8 + 4 * w.B], np.float32)
    x0_out = np.frombuffer(raw[8 + 4 * w.B:8 + 4 * w.B + 4 * n], np.float32).reshape(shp)
    x_next = np.frombuffer(raw[8 + 4 * w.B + 4 * n:], np.float32).reshape(shp)
    t_ref = oracle.tau(w.pos, w.valid)
    np.testing.assert_array_equal(tau, t_ref)
    x0_new = x0_prev[:, anchors] + delta[:, anchors]
    ref_x0, ref_xn, _ = oracle.transport_step(anchors, x0_new, x0_prev, geom=(w.pos, w.valid, w.cams, t_ref),
                                              x_t=x_t, recon=dict(sampler=oracle.DDIM, a_t=0.5, a_prev=0.6))
    for got, ref, scale in ((x0_out, ref_x0, 1.0), (x_next, ref_xn, 2.0)):
        err = np.abs(got.astype(np.float64) - ref) / np.maximum(np.abs(ref), 1.0)
        assert err.max() <= 1e-5 * scale
    assert np.abs(ref_x0 - x0_prev).max() > 1e-3
