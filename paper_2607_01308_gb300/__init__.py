"""GB300-native CanonicalMerge / LatentFragmentSet (arxiv 2607.01308).

The compute path is libcm.so: hand-written CUDA for sm_103a behind the C ABI of
include/cm.h. This package is its Python binding (ctypes). Importing it fails
loudly if the library has not been built; nothing here computes on the CPU.

    import paper_2607_01308_gb300 as cm
    ctx = cm.Context(device=0, rope_theta=1e6)
    S = cm.FragmentSet(ctx)
    fid, absorbed = S.ingest(K, V)          # Algorithm 2, Ingest
    n, order = S.render(k_out, v_out)       # Algorithm 2, Render (= Algorithm 1)
"""
from ._binding import (  # noqa: F401
    CMError, Status, cm_id, cm_fragment, lib, LIB_PATH, EXPORTED,
    cm_abi_version, cm_status_string, cm_last_error_message,
    cm_context_create, cm_context_destroy, cm_context_check, cm_testing_bounds_violations,
    cm_set_create, cm_set_destroy,
    cm_fragment_id, cm_fragment_id_static, cm_ingest, cm_ingest_batch, cm_ingest_many,
    cm_render_many, cm_ingest_render, cm_render_job, cm_set_contains, cm_set_leq, ingest_many, render_many,
    cm_measure_int_alu, cm_context_set_render_warps, cm_context_set_overlap, cm_context_set_dedup_by_bytes,
    cm_context_set_timing, cm_context_kernel_times, cm_kernel_times, cm_union, cm_set_size, cm_set_seq_len, cm_set_ids,
    cm_render, cm_render_incremental, cm_render_paged, cm_paged_cache, cm_bagmerge,
    fragment_from_tensors, Context, FragmentSet,
)
