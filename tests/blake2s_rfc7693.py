"""An independent pure-Python BLAKE2s, written from RFC 7693 and the tree-mode
parameter block of the BLAKE2 paper (Aumasson et al., 2013, Section 2.8 / 2.10).

Test helper only: it pins the oracle's use of hashlib.blake2s (digest size,
fanout, depth, leaf size, node offset, node depth, inner size, salt,
personalisation, last-node flag) against a second implementation, and rebuilds
small hash trees node by node. Slow; use on a few KiB at most.
"""
import struct

IV = (0x6A09E667, 0xBB67AE85, 0x3C6EF372, 0xA54FF53A,
      0x510E527F, 0x9B05688C, 0x1F83D9AB, 0x5BE0CD19)

SIGMA = (
    (0, 1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15),
    (14, 10, 4, 8, 9, 15, 13, 6, 1, 12, 0, 2, 11, 7, 5, 3),
    (11, 8, 12, 0, 5, 2, 15, 13, 10, 14, 3, 6, 7, 1, 9, 4),
    (7, 9, 3, 1, 13, 12, 11, 14, 2, 6, 5, 10, 4, 0, 15, 8),
    (9, 0, 5, 7, 2, 4, 10, 15, 14, 1, 11, 12, 6, 8, 3, 13),
    (2, 12, 6, 10, 0, 11, 8, 3, 4, 13, 7, 5, 15, 14, 1, 9),
    (12, 5, 1, 15, 14, 13, 4, 10, 0, 7, 6, 3, 9, 2, 8, 11),
    (13, 11, 7, 14, 12, 1, 3, 9, 5, 0, 15, 4, 8, 6, 2, 10),
    (6, 15, 14, 9, 11, 3, 0, 8, 12, 2, 13, 7, 1, 4, 10, 5),
    (10, 2, 8, 4, 7, 6, 1, 5, 15, 11, 9, 14, 3, 12, 13, 0),
)

M32 = 0xFFFFFFFF


def _rotr(x, n):
    return ((x >> n) | (x << (32 - n))) & M32


def _mix(v, a, b, c, d, x, y):
    v[a] = (v[a] + v[b] + x) & M32
    v[d] = _rotr(v[d] ^ v[a], 16)
    v[c] = (v[c] + v[d]) & M32
    v[b] = _rotr(v[b] ^ v[c], 12)
    v[a] = (v[a] + v[b] + y) & M32
    v[d] = _rotr(v[d] ^ v[a], 8)
    v[c] = (v[c] + v[d]) & M32
    v[b] = _rotr(v[b] ^ v[c], 7)


def compress(h, block, t, last_block, last_node):
    m = struct.unpack("<16I", block)
    v = list(h) + list(IV)
    v[12] ^= t & M32
    v[13] ^= (t >> 32) & M32
    if last_block:
        v[14] ^= M32
        if last_node:
            v[15] ^= M32
    for r in range(10):
        s = SIGMA[r]
        _mix(v, 0, 4, 8, 12, m[s[0]], m[s[1]])
        _mix(v, 1, 5, 9, 13, m[s[2]], m[s[3]])
        _mix(v, 2, 6, 10, 14, m[s[4]], m[s[5]])
        _mix(v, 3, 7, 11, 15, m[s[6]], m[s[7]])
        _mix(v, 0, 5, 10, 15, m[s[8]], m[s[9]])
        _mix(v, 1, 6, 11, 12, m[s[10]], m[s[11]])
        _mix(v, 2, 7, 8, 13, m[s[12]], m[s[13]])
        _mix(v, 3, 4, 9, 14, m[s[14]], m[s[15]])
    return [h[i] ^ v[i] ^ v[i + 8] for i in range(8)]


def param_block(digest_size, key_size=0, fanout=1, depth=1, leaf_size=0, node_offset=0,
                node_depth=0, inner_size=0, salt=b"\0" * 8, person=b"\0" * 8):
    """The 32-byte BLAKE2s parameter block (little-endian fields)."""
    assert len(salt) == 8 and len(person) == 8
    p = bytes([digest_size, key_size, fanout, depth]) + struct.pack("<I", leaf_size)
    p += struct.pack("<Q", node_offset)[:6] + bytes([node_depth, inner_size]) + salt + person
    assert len(p) == 32
    return p


def blake2s(data, digest_size=32, last_node=False, **params):
    p = param_block(digest_size, **params)
    h = [IV[i] ^ w for i, w in enumerate(struct.unpack("<8I", p))]
    n = len(data)
    if n == 0:
        h = compress(h, b"\0" * 64, 0, True, last_node)
    else:
        off = 0
        while n - off > 64:
            off += 64
            h = compress(h, data[off - 64:off], off, False, last_node)
        tail = data[off:]
        h = compress(h, tail + b"\0" * (64 - len(tail)), n, True, last_node)
    return struct.pack("<8I", *h)[:digest_size]
