"""The allocation-free content address, cm_fragment_id_static.

Some callers cannot allocate device memory (a serving engine whose KV-cache pool
already owns nearly all of the GPU, or a host that routes every device allocation
through its own allocator), so this entry point keeps its scratch in a static
device array instead of calling cudaMalloc. This file is named to be collected
last: it calls the entry point through the C ABI, twice in a row, and checks its
id and norm key against cm_fragment_id bit for bit (the tolerance of every id
and key test in this suite), and checks that a fragment beyond its 1 GiB limit is
refused before any GPU work.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


def _fragment(shape, seed):
    g = torch.Generator(device="cuda:0").manual_seed(seed)
    K = (torch.randn(shape, generator=g, device="cuda:0") * 1.1).to(torch.bfloat16)
    V = torch.randn(shape, generator=g, device="cuda:0").to(torch.bfloat16)
    return K, V


def test_static_scratch_id_matches_cm_fragment_id_on_two_calls_in_a_row():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ctx = cm.Context(0, 1.0e6)
    stream = torch.cuda.current_stream()
    shapes = [(28, 8, 300, 128), (4, 2, 37, 64)]
    for call, shape in enumerate(shapes):
        K, V = _fragment(shape, 100 + call)
        ref_id, ref_q = ctx.fragment_id(K, V)
        id_out = torch.full((16,), 0xAB, dtype=torch.uint8, device="cuda:0")
        q_out = torch.full((shape[2],), -1, dtype=torch.int64, device="cuda:0")
        frag = cm.fragment_from_tensors(K, V)
        st = cm.lib.cm_fragment_id_static(ctypes.byref(frag), -1, stream.cuda_stream or None,
                                          id_out.data_ptr(),
                                          ctypes.cast(q_out.data_ptr(), ctypes.POINTER(ctypes.c_uint64)))
        assert st == cm.Status.OK, cm.cm_last_error_message()
        torch.cuda.synchronize()
        assert bytes(id_out.cpu().numpy().tobytes()) == ref_id
        assert np.array_equal(q_out.cpu().numpy().view(np.uint64), np.array(ref_q, dtype=np.uint64))
    ctx.close()


def test_static_scratch_refuses_fragments_beyond_its_limit():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    K, V = _fragment((1, 1, 16, 128), 7)
    ids = torch.empty(16, dtype=torch.uint8, device="cuda:0")
    q = torch.empty(16, dtype=torch.int64, device="cuda:0")
    # 64 x 64 x 4096 x 128 x 2 x 2 bytes = 8 GiB > 1 GiB; rejected before any access
    big = cm.cm_fragment(64, 64, 4096, 128, K.data_ptr(), V.data_ptr())
    st = cm.lib.cm_fragment_id_static(ctypes.byref(big), -1, None, ids.data_ptr(),
                                      ctypes.cast(q.data_ptr(), ctypes.POINTER(ctypes.c_uint64)))
    assert st == cm.Status.ERR_UNSUPPORTED
    assert "1 GiB" in cm.cm_last_error_message()
