"""The decode path called from plain C on the GPU (tests/c/abi_decode_check.c:
CUDA runtime for memory and a stream, libmilo for the plan and the calls, no
Python or torch on the path).  Its seeded inputs and both outputs (with a
workspace and with the built-in scratch) are compared here with the oracle."""
import os
import shutil
import subprocess

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def test_c_caller_decodes_like_the_oracle(tmp_path, oracle):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    from paper_2609_29913_gb300 import build, milo
    build.build()
    libdir = os.path.dirname(milo.LIB_PATH)
    exe = str(tmp_path / "abi_decode_check")
    cudalib = next((p for p in (os.path.join(CUDA, "lib64"), os.path.join(CUDA, "lib")) if os.path.isdir(p)))
    cmd = [gcc, "-std=c99", "-Wall", "-Werror", "-O1", os.path.join(ROOT, "tests", "c", "abi_decode_check.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"),
           "-L", libdir, "-l:libmilo.so", "-L", cudalib, "-lcudart",
           f"-Wl,-rpath,{libdir}", f"-Wl,-rpath,{cudalib}", "-o", exe]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    run = subprocess.run([exe, str(tmp_path)], capture_output=True, text=True)
    assert run.returncode == 0, run.stderr
    assert run.stdout.split() == ["path", "0", "kernels", "2"]
    rd = lambda name, dt: np.fromfile(tmp_path / name, dtype=dt)
    nb, hkv, g, d, batch = 3, 2, 7, 128, 2
    off = rd("off.i64", np.int64).reshape(4, nb * hkv)
    ref = oracle.attention(num_kv_heads=hkv, head_dim=d, block_len=rd("block_len.i32", np.int32),
                           rank_k=rd("rank_k.i32", np.int32), rank_v=rd("rank_v.i32", np.int32),
                           off_ck=off[0], off_pk=off[1], off_cv=off[2], off_pv=off[3],
                           arena=rd("arena.u16", np.uint16), q=rd("q.u16", np.uint16).reshape(batch, hkv * g, d),
                           tail_k=rd("tail_k.u16", np.uint16).reshape(-1, hkv, d),
                           tail_v=rd("tail_v.u16", np.uint16).reshape(-1, hkv, d),
                           tail_offsets=rd("tail_offsets.i64", np.int64))
    for name in ("out.f32", "out_static.f32"):
        got = rd(name, np.float32).reshape(batch, hkv * g, d).astype(np.float64)
        assert np.isfinite(got).all(), name
        assert np.abs(got - ref).max() <= 1e-2, name
        assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 2e-3, name
