"""Writes content_address_ids.json next to this file: the content address (Section 4.3;
Algorithm 2, Id) the oracle gives three fragments whose bytes come from a fixed
counter-mode SHA-256 stream. The ids freeze the address's definition (BLAKE2s tree,
1 KiB leaves, fanout 16, the parameter block, the byte stream K[0] V[0] ... K[L-1]
V[L-1]): a later change to any of it fails the CPU test that recomputes them with the
oracle and the GPU test that recomputes them with the library. Calls only oracle/.

    python tests/golden/content_address_ids.py
"""
import hashlib
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))

FRAGMENTS = [
    {"name": "tiny-shaped: 4 layers, 2 KV heads, 37 tokens, head_dim 64 (74 leaves, root at level 2)",
     "shape": [4, 2, 37, 64], "seed": "cm-golden-1"},
    {"name": "Qwen3-1.7B-shaped at 64 tokens: 28 layers, 8 KV heads, head_dim 128 "
             "(7168 leaves, root at level 4)",
     "shape": [28, 8, 64, 128], "seed": "cm-golden-2"},
    {"name": "one leaf: 1 layer, 1 KV head, 2 tokens, head_dim 128 (1024 bytes of K and V, "
             "the root an inner node over one child)",
     "shape": [1, 1, 2, 128], "seed": "cm-golden-3"},
]


def fragment_bits(shape, seed):
    """(K, V) as uint16 arrays of `shape`: the bytes SHA-256(seed ':' i) for i = 0, 1, ...,
    concatenated and read as little-endian uint16, K first, then V."""
    count = int(np.prod(shape))
    need = 2 * count * 2
    out = bytearray()
    i = 0
    while len(out) < need:
        out += hashlib.sha256(f"{seed}:{i}".encode()).digest()
        i += 1
    words = np.frombuffer(bytes(out[:need]), dtype="<u2")
    return (words[:count].reshape(shape).astype(np.uint16),
            words[count:].reshape(shape).astype(np.uint16))


def main():
    sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))
    from oracle.content_address import fragment_id
    rows = []
    for f in FRAGMENTS:
        K, V = fragment_bits(f["shape"], f["seed"])
        rows.append(dict(f, id_hex=fragment_id(K, V).hex()))
    doc = {"source": "Section 4.3 (the address is a collision-resistant hash over shapes, dtypes "
                     "and raw bytes); the hash is this library's reading of it, computed by the "
                     "oracle (oracle/content_address.py) on the bytes fragment_bits() generates",
           "fragments": rows}
    with open(os.path.join(HERE, "content_address_ids.json"), "w") as fh:
        json.dump(doc, fh, indent=1)
        fh.write("\n")


if __name__ == "__main__":
    main()
