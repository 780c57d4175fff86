"""CPU oracle for the CanonicalMerge / LatentFragmentSet hot path.

TEST INFRASTRUCTURE ONLY. This package is a plain, slow, fp64 restatement of
what the paper defines (Sections 4.2-4.5, Algorithms 1 and 2, Eq. rho, Eq.
bagmerge-k/v, Eq. setunion). It exists to check the CUDA library. Only the test
suite, the package smoke check and the benchmark's CPU-baseline leg may import
it; the library never does, and the two share no code.

Modules:
  bf16             exact bf16 decode, direct fp64 -> bf16 round-half-even
  content_address  Id(C): BLAKE2s-128 tree hash of the canonical byte stream
  norm             per-row fp64 K-norms at the routing layer -> integer key Q[t]
  fragment_set     LatentFragmentSet: ingest (absorbing) and union
  merge            canonical order, BagMerge with delta RoPE re-encoding, Render

Parity status: every function above is pinned by the `-m "not gpu"` tests
(hashlib / RFC 7693 vectors and an independent pure-Python BLAKE2s for the
tree, closed forms for the norm key, brute force for the order and the set
algebra, rotation composition and the offset-0 identity for the render, an
exact-rational check of the bf16 rounding).
"""
from .bf16 import bits_to_f64, f64_to_bits, ulp_distance, is_nan_bits
from .content_address import fragment_id, fragment_stream, tree_levels, id_as_int
from .norm import norm_key, rho_fp64, tail_sum, default_routing_layer
from .fragment_set import Fragment, FragmentSet, make_fragment, ingest, union, from_deliveries
from .merge import (canonical_order, offsets, delta_cos_sin, rotate_pairs_f64, rotate_k, bagmerge,
                     canonical_merge, render, naive_multiset_render)
