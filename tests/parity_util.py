"""Helpers shared by the GPU parity tests: seeded fragments on the GPU, the same
bytes handed to the CPU oracle, and comparison of bf16 bit arrays."""
import numpy as np
import torch

import oracle
import synthetic
from oracle.bf16 import is_nan_bits, ulp_distance

THETA = synthetic.ROPE_THETA


def gpu_fragments(name, request=0, device="cuda:0"):
    """Distinct fragments of a workload as bf16 CUDA tensors, and its delivery schedule."""
    w = synthetic.WORKLOADS[name]
    specs = synthetic.fragment_specs(w, request)
    frags = [synthetic.make_fragment_torch(s, w.num_layers, w.num_kv_heads, w.head_dim, device)
             for s in specs]
    return w, frags, synthetic.delivery_schedule(w, request)


def oracle_fragment(K, V, routing_layer=-1):
    return oracle.make_fragment(synthetic.to_bits(K), synthetic.to_bits(V), routing_layer)


def assert_k_parity(gpu_bits, ref_bits, what="K"):
    """K: within 1 bf16 ulp per element (NaN on both sides counts as equal); returns the
    number of elements that are not bit-exact."""
    g = np.asarray(gpu_bits)
    r = np.asarray(ref_bits)
    assert g.shape == r.shape, (g.shape, r.shape)
    gn, rn = is_nan_bits(g), is_nan_bits(r)
    assert np.array_equal(gn, rn), f"{what}: NaN positions differ"
    ok = ~gn
    ulps = ulp_distance(g[ok], r[ok])
    worst = int(ulps.max()) if ulps.size else 0
    assert worst <= 1, f"{what}: {int((ulps > 1).sum())} elements beyond 1 ulp (max {worst})"
    return int((ulps != 0).sum())


def empty_out(L, H, cap, d, device="cuda:0", fill=None):
    k = torch.empty((L, H, cap, d), dtype=torch.bfloat16, device=device)
    v = torch.empty_like(k)
    if fill is not None:
        k.view(torch.int16).fill_(fill)
        v.view(torch.int16).fill_(fill)
    return k, v
