"""The allocation-free content address, cm_fragment_id_static.

Some callers cannot allocate device memory (a serving engine whose KV-cache pool
already owns nearly all of the GPU, or a host that routes every device allocation
through its own allocator), so this entry point keeps its scratch in a static
device array instead of calling cudaMalloc. This file is named to be collected
last: it calls the entry point through the C ABI, twice in a row, and checks its
id and norm key against cm_fragment_id bit for bit (the tolerance of every id
and key test in this suite), also with an explicit routing layer, for a one-leaf
tree and for a fragment that fills the static scratch's largest layout (exactly
1 GiB of K and V, 2^20 leaves); and it checks that fragments beyond that limit are
refused before any GPU work.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


def _static_call(K, V, routing_layer, stream=None):
    """cm_fragment_id_static through the C ABI into device buffers; (status, id, key)."""
    T = K.shape[2]
    id_out = torch.full((16,), 0xAB, dtype=torch.uint8, device="cuda:0")
    q_out = torch.full((T,), -1, dtype=torch.int64, device="cuda:0")
    frag = cm.fragment_from_tensors(K, V)
    handle = stream.cuda_stream if stream is not None else torch.cuda.current_stream().cuda_stream
    st = cm.lib.cm_fragment_id_static(ctypes.byref(frag), routing_layer, handle or None,
                                      id_out.data_ptr(),
                                      ctypes.cast(q_out.data_ptr(), ctypes.POINTER(ctypes.c_uint64)))
    torch.cuda.synchronize()
    return st, bytes(id_out.cpu().numpy().tobytes()), q_out.cpu().numpy().view(np.uint64)


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


@pytest.mark.parametrize("layer", [0, 3])
def test_static_scratch_with_an_explicit_routing_layer(layer):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    K, V = _fragment((4, 2, 70, 64), 40 + layer)
    ctx = cm.Context(0, 1.0e6, routing_layer=layer)
    ref_id, ref_q = ctx.fragment_id(K, V)
    for _ in range(2):
        st, fid, q = _static_call(K, V, layer)
        assert st == cm.Status.OK, cm.cm_last_error_message()
        assert fid == ref_id
        assert np.array_equal(q, np.array(ref_q, dtype=np.uint64))
    ctx.close()


@pytest.mark.parametrize("shape", [(1, 1, 1, 256), (1, 1, 2, 16)])
def test_static_scratch_one_leaf_tree(shape):
    # 1024 and 128 bytes of K and V: one leaf, the root an inner node over one child
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    K, V = _fragment(shape, 50)
    ctx = cm.Context(0, 1.0e6)
    ref_id, ref_q = ctx.fragment_id(K, V)
    for _ in range(2):
        st, fid, q = _static_call(K, V, -1)
        assert st == cm.Status.OK, cm.cm_last_error_message()
        assert fid == ref_id and np.array_equal(q, np.array(ref_q, dtype=np.uint64))
    ctx.close()


def test_static_scratch_at_its_limit_and_one_row_beyond():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    # 4 x 8 x 65536 x 128 bf16 = 256 Mi elements: K and V hold exactly 1 GiB, 2^20 leaves
    K, V = _fragment((4, 8, 65536, 128), 60)
    ctx = cm.Context(0, 1.0e6)
    ref_id, ref_q = ctx.fragment_id(K, V)
    for _ in range(2):
        st, fid, q = _static_call(K, V, -1)
        assert st == cm.Status.OK, cm.cm_last_error_message()
        assert fid == ref_id and np.array_equal(q, np.array(ref_q, dtype=np.uint64))
    ctx.close()
    # one more token: 16 KiB past the limit, refused before any access
    del K, V
    K2, V2 = _fragment((1, 1, 16, 128), 61)
    over = cm.cm_fragment(4, 8, 65537, 128, K2.data_ptr(), V2.data_ptr())
    ids = torch.empty(16, dtype=torch.uint8, device="cuda:0")
    q = torch.empty(16, dtype=torch.int64, device="cuda:0")
    st = cm.lib.cm_fragment_id_static(ctypes.byref(over), -1, None, ids.data_ptr(),
                                      ctypes.cast(q.data_ptr(), ctypes.POINTER(ctypes.c_uint64)))
    assert st == cm.Status.ERR_UNSUPPORTED
    assert "1 GiB" in cm.cm_last_error_message()
