"""Failure detection on the GPU without a fault: every wait of the half-SM render
kernel on its own TMA copies is bounded (about one second); when one runs out, the
warp records the failure in the context and returns. A test-only hook withholds one
copy so that the wait runs out (the hook always runs that kernel: the full-SM render
loads into registers and has no waits); the host must read CM_ERR_TIMEOUT and the
context must stay usable, with either render width set. Re-delivery (the paper's fault model, Section 5.9) is covered by
the absorption tests."""
import numpy as np
import pytest
import torch

import oracle
import synthetic
from parity_util import THETA, assert_k_parity, empty_out, gpu_fragments, oracle_fragment

pytestmark = pytest.mark.gpu

cm = pytest.importorskip("paper_2607_01308_gb300")


@pytest.mark.parametrize("warps", [16, 8])
def test_withheld_copy_times_out_and_the_context_recovers(warps):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ctx = cm.Context(0, THETA)
    cm.cm_context_set_render_warps(ctx.handle, warps)
    w, frags, _ = gpu_fragments("tiny")
    S = cm.FragmentSet(ctx)
    S.ingest_batch(frags)
    k_out, v_out = empty_out(w.num_layers, w.num_kv_heads, S.seq_len(), w.head_dim)
    stream = torch.cuda.current_stream()
    st = cm.lib.cm_testing_render_withheld_load(S.handle, k_out.data_ptr(), v_out.data_ptr(),
                                                S.seq_len(), stream.cuda_stream or None)
    assert st == cm.Status.OK
    with pytest.raises(cm.CMError) as e:
        ctx.check()
    assert e.value.status == cm.Status.ERR_TIMEOUT
    ctx.check()   # reported once, then cleared
    # the context still works: a normal render matches the oracle
    n, order = S.render(k_out, v_out)
    ctx.check()
    ref = oracle.from_deliveries([oracle_fragment(K, V) for K, V in frags])
    K_ref, V_ref, o_order = oracle.render(ref, THETA)
    assert order == [f.fid for f in o_order]
    assert np.array_equal(synthetic.to_bits(v_out), V_ref)
    assert assert_k_parity(synthetic.to_bits(k_out), K_ref) == 0
    S.close()
    ctx.close()
