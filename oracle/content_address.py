"""Content address Id(C) of a fragment (test infrastructure only).

Section 4.3 and Algorithm 2 (function Id): the identity of a fragment is a
collision-resistant hash over its shapes, dtype and the raw bytes of every
layer's unshifted K and V, in the order K^1, V^1, ..., K^L, V^L. The paper does
not name the hash. Reading used here: BLAKE2s (RFC 7693) in its tree mode
(BLAKE2 paper, Section 2.10), 16-byte digests, computed with hashlib.blake2s.

Byte stream:   K[0] V[0] K[1] V[1] ... K[L-1] V[L-1], each [H][T][d] bf16, little endian
Every node:    digest_size=16, no key, fanout=16, depth=255, leaf_size=1024,
               inner_size=16, salt = <L,H,d,1> as four little-endian uint16
               (1 = bf16), person = <T> as a little-endian uint64
Level 0:       leaf j hashes stream bytes [1024 j, 1024 (j+1)), node_offset=j,
               node_depth=0, last_node set on the final leaf
Level k >= 1:  node j hashes the concatenated 16-byte digests of children
               [16 j, 16 j + 16) of level k-1, node_offset=j, node_depth=k,
               last_node set on the final node of the level
Root:          the digest of the first level k >= 1 that has a single node.
"""
from __future__ import annotations

import hashlib
import struct
from typing import List, Tuple

import numpy as np

DIGEST_SIZE = 16
LEAF_SIZE = 1024
FANOUT = 16
DEPTH = 255
DTYPE_CODE_BF16 = 1


def tree_salt(L: int, H: int, d: int) -> bytes:
    return struct.pack("<HHHH", L, H, d, DTYPE_CODE_BF16)


def tree_person(T: int) -> bytes:
    return struct.pack("<Q", T)


def node_digest(data: bytes, *, salt: bytes, person: bytes, node_offset: int,
                node_depth: int, last_node: bool) -> bytes:
    return hashlib.blake2s(
        data, digest_size=DIGEST_SIZE, salt=salt, person=person, fanout=FANOUT,
        depth=DEPTH, leaf_size=LEAF_SIZE, node_offset=node_offset,
        node_depth=node_depth, inner_size=DIGEST_SIZE, last_node=last_node).digest()


def fragment_stream(K: np.ndarray, V: np.ndarray) -> bytes:
    """The canonical byte string of Algorithm 2: K and V of each layer in turn."""
    assert K.dtype == np.uint16 and V.dtype == np.uint16 and K.shape == V.shape
    parts = []
    for l in range(K.shape[0]):
        parts.append(np.ascontiguousarray(K[l]).astype("<u2").tobytes())
        parts.append(np.ascontiguousarray(V[l]).astype("<u2").tobytes())
    return b"".join(parts)


def tree_levels(stream: bytes, salt: bytes, person: bytes) -> List[List[bytes]]:
    """All levels of the hash tree, level 0 (leaves) first, root level last."""
    n = len(stream)
    n_leaves = max(1, -(-n // LEAF_SIZE))
    level = [node_digest(stream[j * LEAF_SIZE:(j + 1) * LEAF_SIZE], salt=salt, person=person,
                         node_offset=j, node_depth=0, last_node=(j == n_leaves - 1))
             for j in range(n_leaves)]
    levels = [level]
    depth = 0
    while depth == 0 or len(level) > 1:
        depth += 1
        prev = level
        n_nodes = -(-len(prev) // FANOUT)
        level = [node_digest(b"".join(prev[j * FANOUT:(j + 1) * FANOUT]), salt=salt,
                             person=person, node_offset=j, node_depth=depth,
                             last_node=(j == n_nodes - 1))
                 for j in range(n_nodes)]
        levels.append(level)
    return levels


def fragment_id(K: np.ndarray, V: np.ndarray) -> bytes:
    """Id(C): the 16-byte root digest (Algorithm 2, function Id)."""
    L, H, T, d = K.shape
    levels = tree_levels(fragment_stream(K, V), tree_salt(L, H, d), tree_person(T))
    return levels[-1][0]


def id_as_int(fid: bytes) -> int:
    """The id read as a big-endian unsigned integer (the order of the tie-break)."""
    return int.from_bytes(fid, "big")


def level_sizes(n_bytes: int) -> Tuple[int, ...]:
    """Number of nodes of each level for a stream of n_bytes."""
    sizes = [max(1, -(-n_bytes // LEAF_SIZE))]
    while len(sizes) == 1 or sizes[-1] > 1:
        sizes.append(-(-sizes[-1] // FANOUT))
    return tuple(sizes)
