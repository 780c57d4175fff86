"""The C ABI from C. A C11 program including include/cm.h and include/cm_testing.h
compiles with -Wall -Werror, links against libcm.so and runs (argument validation
only; no GPU needed); and, on a GPU, a C program runs a whole merge (ingest into two
replicas, union, render) whose results are checked against the CPU oracle."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_01308_gb300")


def test_c_program_compiles_links_and_runs(tmp_path):
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    if not os.path.exists(os.path.join(PKG, "libcm.so")):
        pytest.skip("libcm.so not built")
    exe = str(tmp_path / "abi_smoke")
    subprocess.run([cc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-pedantic",
                    "-I" + os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "c_abi", "abi_smoke.c"),
                    "-L" + PKG, "-lcm", "-Wl,-rpath," + PKG, "-o", exe], check=True)
    r = subprocess.run([exe], capture_output=True, text=True)
    assert r.returncode == 0, (r.returncode, r.stdout, r.stderr)
    assert r.stdout.startswith("ok")


def _cuda_home():
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return "/usr/local/cuda"


@pytest.mark.gpu
def test_merge_through_the_c_abi_from_c_matches_the_oracle(tmp_path):
    """tests/c_abi/merge_from_c.c ingests the tiny workload's deliveries into two
    replicas (fragment 0 re-delivered to replica 0), unions and renders, all from C;
    its ids, absorptions, order and rendered bytes must equal the oracle's."""
    import numpy as np
    import torch

    import oracle
    import synthetic
    from parity_util import THETA, assert_k_parity
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    cuda = _cuda_home()
    libdirs = [d for d in (os.path.join(cuda, "lib64"), os.path.join(cuda, "lib")) if os.path.isdir(d)]
    exe = str(tmp_path / "merge_from_c")
    cmd = [cc, "-std=c11", "-Wall", "-Wextra", "-Werror", "-I" + os.path.join(ROOT, "include"),
           "-I" + os.path.join(cuda, "include"), os.path.join(ROOT, "tests", "c_abi", "merge_from_c.c"),
           "-L" + PKG, "-lcm", "-Wl,-rpath," + PKG]
    for d in libdirs:
        cmd += ["-L" + d, "-Wl,-rpath," + d]
    subprocess.run(cmd + ["-lcudart", "-o", exe], check=True)

    w = synthetic.WORKLOADS["tiny"]
    specs = synthetic.fragment_specs(w)
    bits = [synthetic.make_fragment_bits(s, w.num_layers, w.num_kv_heads, w.head_dim) for s in specs]
    plan = [(0, 0), (1, 1), (0, 0)]          # (replica, fragment): fragment 0 re-delivered
    args = [exe, str(w.num_layers), str(w.num_kv_heads), str(w.head_dim),
            str(tmp_path / "out_k.bin"), str(tmp_path / "out_v.bin")]
    for i, (r, f) in enumerate(plan):
        K, V = bits[f]
        kp, vp = tmp_path / f"k{i}.bin", tmp_path / f"v{i}.bin"
        K.tofile(kp)
        V.tofile(vp)
        args += [str(r), str(K.shape[2]), str(kp), str(vp)]
    res = subprocess.run(args, capture_output=True, text=True)
    assert res.returncode == 0, (res.stdout, res.stderr)
    lines = res.stdout.split("\n")
    ref = [oracle.make_fragment(K, V) for K, V in bits]
    for i, (r, f) in enumerate(plan):
        _, idx, fid, absorbed = lines[i].split()
        assert int(idx) == i and fid == ref[f].fid.hex()
        assert absorbed == ("1" if i == 2 else "0")
    S = oracle.from_deliveries(ref)
    K_ref, V_ref, order = oracle.render(S, THETA)
    assert lines[3] == "size 2"
    assert lines[4] == f"seq_len {K_ref.shape[2]}"
    assert lines[5].split()[1:] == [f.fid.hex() for f in order]
    shape = K_ref.shape
    k_out = np.fromfile(tmp_path / "out_k.bin", dtype=np.uint16).reshape(shape)
    v_out = np.fromfile(tmp_path / "out_v.bin", dtype=np.uint16).reshape(shape)
    assert np.array_equal(v_out, V_ref)
    assert assert_k_parity(k_out, K_ref) == 0
