"""The C ABI from plain C (no GPU): tests/c/abi_host_check.c is compiled
with gcc against include/milo.h and linked with libmilo.so; its host-only
results (validation, packed layout, chunk list, partition, error codes)
must equal what the ctypes binding computes for the same table."""
import os
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def milo():
    from paper_2609_29913_gb300 import build, milo
    build.build()
    milo.lib()
    return milo


def run_c(tmp_path, milo):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    exe = str(tmp_path / "abi_host_check")
    libdir = os.path.dirname(milo.LIB_PATH)
    cmd = [gcc, "-std=c99", "-Wall", "-Werror", "-O1", os.path.join(ROOT, "tests", "c", "abi_host_check.c"),
           "-I", os.path.join(ROOT, "include"), "-L", libdir, "-l:libmilo.so", f"-Wl,-rpath,{libdir}", "-o", exe]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    res = {}
    for line in out.splitlines():
        k, *v = line.split()
        res[k] = v
    return res


def test_c_caller_agrees_with_the_binding(tmp_path, milo):
    res = run_c(tmp_path, milo)
    # the same table through ctypes
    bl = np.array([33, 512], np.int32)
    rk = np.array([8, 13, 64, 0], np.int32)
    rv = np.array([5, 16, 32, 64], np.int32)
    off = np.zeros((4, 4), np.int64)
    cur = 0
    for e in range(4):
        n = int(bl[e // 2])
        for f, sz in enumerate((n * rk[e], rk[e] * 64, n * rv[e], rv[e] * 64)):
            off[f, e] = cur
            cur += (int(sz) + 7) // 8 * 8
    arena = np.zeros(1 << 17, np.uint16)
    t = milo.HostTable(num_kv_heads=2, head_dim=64, block_len=bl, rank_k=rk, rank_v=rv, off_ck=off[0],
                       off_pk=off[1], off_cv=off[2], off_pv=off[3], arena_ptr=arena.ctypes.data, arena_elems=cur)
    assert int(res["version"][0]) == int(milo.lib().milo_version())
    assert res["validate"] == ["0"] and milo.milo_validate_table(t) == 0
    _, total = milo.milo_packed_layout(t)
    assert res["layout"] == ["0"] and int(res["packed_total"][0]) == total
    assert res["chunks_status"] == ["0"] and int(res["chunks"][0]) == len(milo.milo_chunk_prefix(t)["entry"])
    part = milo.milo_partition_prefix(t, 3)
    assert res["partition_status"] == ["0"]
    assert int(res["segments"][0]) == len(part["entry"]) and int(res["slots"][0]) == part["num_slots"]
    assert res["bad_rank"] == ["2"] and res["odd_offset"] == ["3"] and res["null_plan"] == ["1"]
    assert " ".join(res["status_string"]) == milo.lib().milo_status_string(2).decode()
