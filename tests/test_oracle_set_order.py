"""Pins for the oracle's LatentFragmentSet algebra (Eq. setunion, Algorithm 2)
and canonical order (Algorithm 1) (CPU only): brute force over small sets and
all input orders."""
import itertools

import numpy as np
import pytest

import oracle
from oracle.content_address import id_as_int
from oracle.norm import rho_fp64
from synthetic import random_bits


def _pool(n, T=(6, 9, 7, 11, 8), L=3, H=2, d=16, seed=0):
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n):
        K = random_bits(rng, (L, H, T[i % len(T)], d), scale=0.5 + 0.25 * i)
        V = random_bits(rng, (L, H, T[i % len(T)], d))
        out.append(oracle.make_fragment(K, V))
    return out


def _subsets(pool, k_max=4):
    for k in range(0, k_max + 1):
        for combo in itertools.combinations(pool, k):
            yield oracle.from_deliveries(combo)


def test_union_is_a_join_semilattice():
    pool = _pool(4)
    sets = list(_subsets(pool))
    for A in sets:
        assert oracle.union(A, A) == A
        for B in sets:
            AB = oracle.union(A, B)
            assert AB == oracle.union(B, A)
            assert A.leq(AB) and B.leq(AB)
            # least upper bound: any C above both is above A u B
            for C in sets:
                if A.leq(C) and B.leq(C):
                    assert AB.leq(C)
    for A, B, C in itertools.product(sets[::3], repeat=3):
        assert oracle.union(oracle.union(A, B), C) == oracle.union(A, oracle.union(B, C))


def test_ingest_absorbs_byte_identical_redelivery_only():
    (a, b) = _pool(2)
    copy = oracle.make_fragment(a.K.copy(), a.V.copy())
    S = oracle.from_deliveries([a, b, copy, b])
    assert len(S) == 2 and S.ids() == sorted([a.fid, b.fid])
    # one flipped bit is a different fragment (absorption is syntactic)
    V2 = a.V.copy()
    V2[0, 0, 0, 0] ^= 1
    S2 = oracle.ingest(S, oracle.make_fragment(a.K, V2))
    assert len(S2) == 3


def test_canonical_order_is_a_function_of_the_set():
    for n in range(1, 6):
        pool = _pool(n, seed=n)
        ref_order, _ = oracle.canonical_order(pool)
        for perm in itertools.permutations(pool):
            order, _ = oracle.canonical_order(list(perm))
            assert [f.fid for f in order] == [f.fid for f in ref_order]


def test_order_by_integer_key_matches_order_by_fp64_rho():
    pool = _pool(5, seed=9)
    order, S = oracle.canonical_order(pool)
    t_star = min(f.seq_len for f in pool)
    rho = [rho_fp64(f.K, 1, t_star) for f in order]
    assert rho == sorted(rho, reverse=True)
    assert S == sorted(S, reverse=True)


def test_exact_ties_break_by_descending_big_endian_id():
    rng = np.random.default_rng(12)
    K = random_bits(rng, (3, 2, 6, 16))
    frags = []
    for i in range(4):
        V = random_bits(rng, (3, 2, 6, 16))   # same K, different V: equal keys, distinct ids
        frags.append(oracle.make_fragment(K, V))
    order, S = oracle.canonical_order(frags)
    assert len(set(S)) == 1
    ids = [id_as_int(f.fid) for f in order]
    assert ids == sorted(ids, reverse=True)


def test_offsets_are_exclusive_prefix_sums():
    pool = _pool(4, seed=3)
    order, _ = oracle.canonical_order(pool)
    offs = oracle.offsets(order)
    assert offs[0] == 0
    for i in range(1, 4):
        assert offs[i] == offs[i - 1] + order[i - 1].seq_len
