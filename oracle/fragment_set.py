"""LatentFragmentSet state (test infrastructure only).

Section 4.4, Eq. setunion and Algorithm 2: the replicated state is a set of
(Id, unshifted fragment) pairs. Ingest inserts a delivery keyed by its Id, so a
byte-identical re-delivery is absorbed; Merge is set union, which is
commutative, associative, idempotent and absorbing; the partial order is
inclusion over ids. Absorption is syntactic (Section 4.4, last paragraph):
equal bytes give equal ids, and nothing else is merged.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Iterable, List

import numpy as np

from .content_address import fragment_id
from .norm import default_routing_layer, norm_key


@dataclasses.dataclass(frozen=True)
class Fragment:
    K: np.ndarray          # uint16 [L, H, T, d]
    V: np.ndarray          # uint16 [L, H, T, d]
    fid: bytes             # 16-byte content address
    Q: np.ndarray          # uint64 [T] norm key at the routing layer

    @property
    def shape(self):
        return self.K.shape

    @property
    def seq_len(self) -> int:
        return self.K.shape[2]


def make_fragment(K: np.ndarray, V: np.ndarray, routing_layer: int = -1) -> Fragment:
    """Id and norm key of one delivery (what cm_ingest computes)."""
    L = K.shape[0]
    rl = default_routing_layer(L) if routing_layer < 0 else routing_layer
    return Fragment(K, V, fragment_id(K, V), norm_key(K, rl))


class FragmentSet:
    """Immutable set of fragments keyed by Id."""

    def __init__(self, items: Dict[bytes, Fragment] = None):
        self._items: Dict[bytes, Fragment] = dict(items or {})

    def ids(self) -> List[bytes]:
        """Ids in ascending (big-endian) order."""
        return sorted(self._items)

    def fragments(self) -> List[Fragment]:
        return [self._items[k] for k in self.ids()]

    def __len__(self) -> int:
        return len(self._items)

    def __contains__(self, fid: bytes) -> bool:
        return fid in self._items

    def __eq__(self, other) -> bool:
        return isinstance(other, FragmentSet) and set(self._items) == set(other._items)

    def leq(self, other: "FragmentSet") -> bool:
        """S <= T iff every id of S is in T (the semilattice order)."""
        return set(self._items) <= set(other._items)


def ingest(S: FragmentSet, C: Fragment) -> FragmentSet:
    """Algorithm 2, Ingest: S u {(Id(C), C)}; an existing id keeps its record."""
    items = dict(S._items)
    items.setdefault(C.fid, C)
    return FragmentSet(items)


def union(S1: FragmentSet, S2: FragmentSet) -> FragmentSet:
    """Algorithm 2, Merge (Eq. setunion): S1 u S2; S1's record wins on equal ids."""
    items = dict(S2._items)
    items.update(S1._items)
    return FragmentSet(items)


def from_deliveries(deliveries: Iterable[Fragment]) -> FragmentSet:
    S = FragmentSet()
    for C in deliveries:
        S = ingest(S, C)
    return S
