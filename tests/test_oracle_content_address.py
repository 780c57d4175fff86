"""Pins for the oracle's content address Id(C) (CPU only).

hashlib.blake2s is pinned to the RFC 7693 test vector; the tree-mode parameters
the oracle passes to it are pinned to an independent pure-Python BLAKE2s built
from RFC 7693 and the BLAKE2 parameter block; whole small trees are rebuilt
node by node with that implementation and compared with the oracle's root.
"""
import hashlib
import json
import os
import struct

import numpy as np
import pytest

import blake2s_rfc7693 as ref
from oracle import content_address as ca
from synthetic import random_bits

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_hashlib_matches_rfc7693_vector():
    g = json.load(open(os.path.join(GOLDEN, "blake2s_rfc7693.json")))
    msg = bytes.fromhex(g["message_hex"])
    assert hashlib.blake2s(msg, digest_size=g["digest_size"]).hexdigest() == g["digest_hex"]
    assert ref.blake2s(msg, digest_size=g["digest_size"]).hex() == g["digest_hex"]


@pytest.mark.parametrize("n", [0, 1, 63, 64, 65, 128, 1000, 1024, 2048 + 5])
def test_tree_node_parameters_match_independent_blake2s(n):
    rng = np.random.default_rng(n)
    data = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
    salt = ca.tree_salt(int(rng.integers(1, 99)), int(rng.integers(1, 64)), 128)
    person = ca.tree_person(int(rng.integers(1, 1 << 40)))
    for node_offset, node_depth, last in [(0, 0, False), (5, 0, True), ((1 << 47) + 3, 2, False),
                                          (77, 1, True)]:
        got = ca.node_digest(data, salt=salt, person=person, node_offset=node_offset,
                             node_depth=node_depth, last_node=last)
        want = ref.blake2s(data, digest_size=16, last_node=last, fanout=ca.FANOUT,
                           depth=ca.DEPTH, leaf_size=ca.LEAF_SIZE, node_offset=node_offset,
                           node_depth=node_depth, inner_size=16, salt=salt, person=person)
        assert got == want


def _brute_force_root(stream: bytes, salt: bytes, person: bytes) -> bytes:
    """Level by level with the independent implementation; stop at one node, depth >= 1."""
    def node(data, off, depth, last):
        return ref.blake2s(data, digest_size=16, last_node=last, fanout=ca.FANOUT, depth=255,
                           leaf_size=1024, node_offset=off, node_depth=depth, inner_size=16,
                           salt=salt, person=person)
    chunks = [stream[i:i + 1024] for i in range(0, max(len(stream), 1), 1024)] or [b""]
    level = [node(c, j, 0, j == len(chunks) - 1) for j, c in enumerate(chunks)]
    depth = 0
    while True:
        depth += 1
        groups = [level[i:i + ca.FANOUT] for i in range(0, len(level), ca.FANOUT)]
        level = [node(b"".join(g), j, depth, j == len(groups) - 1) for j, g in enumerate(groups)]
        if len(level) == 1:
            return level[0]


@pytest.mark.parametrize("shape", [(1, 1, 1, 16), (2, 1, 3, 64), (4, 2, 37, 64), (1, 1, 513, 128)])
def test_fragment_id_matches_brute_force_tree(shape):
    rng = np.random.default_rng(sum(shape))
    K = random_bits(rng, shape)
    V = random_bits(rng, shape)
    L, H, T, d = shape
    stream = ca.fragment_stream(K, V)
    assert len(stream) == 2 * L * H * T * d * 2
    want = _brute_force_root(stream, ca.tree_salt(L, H, d), ca.tree_person(T))
    assert ca.fragment_id(K, V) == want


def test_stream_order_is_k_then_v_per_layer():
    rng = np.random.default_rng(3)
    K = random_bits(rng, (3, 2, 5, 16))
    V = random_bits(rng, (3, 2, 5, 16))
    s = ca.fragment_stream(K, V)
    P = 2 * 5 * 16 * 2
    for l in range(3):
        assert s[2 * l * P:(2 * l + 1) * P] == K[l].astype("<u2").tobytes()
        assert s[(2 * l + 1) * P:(2 * l + 2) * P] == V[l].astype("<u2").tobytes()


def test_level_sizes():
    assert ca.FANOUT == 16
    assert ca.level_sizes(1) == (1, 1)
    assert ca.level_sizes(1024) == (1, 1)
    assert ca.level_sizes(1025) == (2, 1)
    assert ca.level_sizes(16 * 1024) == (16, 1)
    assert ca.level_sizes(16 * 1024 + 1) == (17, 2, 1)
    # Qwen3-4B-shaped fragment, T = 4096: 604 MB -> 589 824 leaves
    n = 36 * 8 * 4096 * 128 * 2 * 2
    assert ca.level_sizes(n) == (589824, 36864, 2304, 144, 9, 1)


def test_id_sensitive_to_every_byte_and_to_shape():
    rng = np.random.default_rng(5)
    K = random_bits(rng, (2, 2, 9, 32))
    V = random_bits(rng, (2, 2, 9, 32))
    base = ca.fragment_id(K, V)
    for arr in (K, V):
        for _ in range(20):
            idx = tuple(int(rng.integers(0, s)) for s in arr.shape)
            bit = np.uint16(1 << int(rng.integers(0, 16)))
            arr[idx] ^= bit
            assert ca.fragment_id(K, V) != base
            arr[idx] ^= bit
    assert ca.fragment_id(K, V) == base
    # same byte stream under another shape is another fragment (shapes are hashed)
    assert ca.fragment_id(K.reshape(2, 1, 18, 32), V.reshape(2, 1, 18, 32)) != base
    assert ca.fragment_id(K.reshape(2, 2, 18, 16), V.reshape(2, 2, 18, 16)) != base


def test_id_as_int_is_big_endian():
    assert ca.id_as_int(bytes([1] + [0] * 15)) == 1 << 120
    assert ca.id_as_int(bytes([0] * 15 + [1])) == 1


def test_salt_and_personalisation_byte_layout():
    # salt = (L, H, d, dtype code 1 = bf16) as four little-endian uint16; person = T as a
    # little-endian uint64 (the documented parameter layout of every tree node)
    assert ca.tree_salt(28, 8, 128) == bytes([28, 0, 8, 0, 128, 0, 1, 0])
    assert ca.tree_salt(300, 2, 64) == bytes([0x2C, 0x01, 2, 0, 64, 0, 1, 0])
    assert ca.tree_person(4096) == bytes([0, 0x10, 0, 0, 0, 0, 0, 0])
    assert ca.tree_person((1 << 40) + 3) == bytes([3, 0, 0, 0, 0, 1, 0, 0])
    # and the parameter block the nodes are hashed with carries them at bytes 16..31
    pb = ref.param_block(16, fanout=ca.FANOUT, depth=ca.DEPTH, leaf_size=ca.LEAF_SIZE,
                         node_offset=5, node_depth=2, inner_size=16,
                         salt=ca.tree_salt(28, 8, 128), person=ca.tree_person(4096))
    assert pb[0:4] == bytes([16, 0, 16, 255]) and pb[4:8] == (1024).to_bytes(4, "little")
    assert pb[8:14] == (5).to_bytes(6, "little") and pb[14:16] == bytes([2, 16])
    assert pb[16:24] == bytes([28, 0, 8, 0, 128, 0, 1, 0])
    assert pb[24:32] == bytes([0, 0x10, 0, 0, 0, 0, 0, 0])


def _golden_ids():
    import importlib.util
    import json
    import os
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    spec = importlib.util.spec_from_file_location("_golden_ca", os.path.join(here, "content_address_ids.py"))
    gen = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(gen)
    with open(os.path.join(here, "content_address_ids.json")) as fh:
        return gen, json.load(fh)["fragments"]


def test_content_address_is_frozen_on_golden_fragments():
    # the ids recorded when the address's definition was fixed: any change to the leaf
    # size, fanout, parameter block or byte stream changes them
    from oracle.content_address import fragment_id
    gen, rows = _golden_ids()
    assert len(rows) == 3
    for row in rows:
        K, V = gen.fragment_bits(row["shape"], row["seed"])
        assert fragment_id(K, V).hex() == row["id_hex"], row["name"]
