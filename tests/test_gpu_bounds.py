"""The bounds-checked testing build (build.py --bounds, libcm_bounds.so; a stand-in for a
device memory checker): the parity cases of tests/bounds_cases.py run against it in a
separate process, with every global access of the render and content-address kernels
checked against the buffer it belongs to. No access may fall outside, the results must
be the oracle's, and a negative block-table entry (an input the host does not check) must
be counted."""
import json
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def test_bounds_checked_build_sees_no_access_outside_its_buffers():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sys.path.insert(0, os.path.dirname(HERE))
    from paper_2607_01308_gb300 import build as cm_build
    lib = cm_build.build(bounds=True)
    env = dict(os.environ, CM_LIBRARY=lib)
    r = subprocess.run([sys.executable, os.path.join(HERE, "bounds_cases.py")], env=env,
                       stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:]
    res = json.loads(r.stdout.strip().splitlines()[-1])
    assert res["enabled"]
    assert res["cases"] >= 35
    assert res["violations"] == 0
    assert res["negative_table_entry_violations"] > 0
    assert res["violations_after"] == 0


def test_normal_build_reports_no_checks():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_01308_gb300 as cm
    if os.environ.get("CM_LIBRARY"):
        pytest.skip("another build of the library is loaded")
    count, enabled = cm.cm_testing_bounds_violations(0)
    assert not enabled and count == 0
