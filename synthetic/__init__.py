"""Seeded synthetic KV-cache fragments and delivery schedules.

This module only *makes inputs*. It holds none of the merge arithmetic
(content address, norm key, canonical order, delta rotation); both the CPU
oracle and the CUDA library are fed from here and compared against each other.

A fragment is one thinker's legacy KV cache (Section 4.1): per layer a K and a V
tensor of shape [H, T, d] (the batch dimension of 1 is dropped), bf16. K is
stored *post-rotation*: the key at position t has been rotated by R(t). The
pre-rotation below uses the rotate-half pairing (j, j + d/2) with inverse
frequencies theta^(-2j/d) evaluated in fp32, the way a bf16 model runtime
produces its cache; it only shapes the synthetic bytes; the bytes are the input.

Workloads (shapes of the paper's Qwen3-1.7B / Qwen3-4B caches, Section 5.8):
  tiny       L=4,  H=2, d=64,  T=37,53; K scaled 0.8 / 1.2, V unscaled;
             fragment 0 re-delivered once as a byte copy (3 deliveries)
  q17_n2     L=28, H=8, d=128, N=2 x T=512, K and V scaled per fragment U(0.5,1.5)
  q17_arity  L=28, H=8, d=128, N=5, T ~ U{256..2048}, 8 deliveries (3 duplicates)
  q4b        L=36, H=8, d=128, N=4 x T=4096, scale U(0.5,1.5)
  q4b_t512   the q4b shape with T=512 per fragment (302 MB of inputs): profiling case
  q4b_t2048  the q4b shape with T=2048 per fragment (1.2 GB of inputs): profiling case
             large enough for the two-kernel tree top (73,728 level-1 nodes)
  serve      q4b shape, 64 requests x N=3, T ~ U{512..4096}, each delivery
             re-sent with probability 0.1, shuffled per request

Seeds: fragment i of request r draws its length and scale from
numpy.random.default_rng(42 + 1000 r + i) and its values from a torch generator
seeded with the same number; the delivery schedule of request r (duplicates and
order) comes from numpy.random.default_rng(42 + 1000 r + 999).
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np

ROPE_THETA = 1.0e6
BASE_SEED = 42


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    num_layers: int
    num_kv_heads: int
    head_dim: int
    num_fragments: int
    # fixed lengths (one per fragment) or an inclusive [lo, hi] range to draw from
    lengths: Optional[Sequence[int]] = None
    length_range: Optional[Sequence[int]] = None
    # fixed K scales (tiny) or None for U(0.5, 1.5) on both K and V
    k_scales: Optional[Sequence[float]] = None
    scale_v: bool = True
    num_requests: int = 1
    # explicit duplicate schedule (indices of fragments re-sent once), or a
    # re-send probability per delivery, or a fixed number of duplicates
    dup_indices: Optional[Sequence[int]] = None
    dup_prob: float = 0.0
    num_dups: int = 0

    @property
    def bytes_per_token(self) -> int:
        return self.num_layers * self.num_kv_heads * self.head_dim * 2 * 2


WORKLOADS = {
    "tiny": Workload("tiny", 4, 2, 64, 2, lengths=(37, 53), k_scales=(0.8, 1.2),
                     scale_v=False, dup_indices=(0,)),
    "q17_n2": Workload("q17_n2", 28, 8, 128, 2, lengths=(512, 512)),
    "q17_arity": Workload("q17_arity", 28, 8, 128, 5, length_range=(256, 2048), num_dups=3),
    "q4b": Workload("q4b", 36, 8, 128, 4, lengths=(4096, 4096, 4096, 4096)),
    "q4b_t512": Workload("q4b_t512", 36, 8, 128, 4, lengths=(512, 512, 512, 512)),
    "q4b_t2048": Workload("q4b_t2048", 36, 8, 128, 4, lengths=(2048, 2048, 2048, 2048)),
    "serve": Workload("serve", 36, 8, 128, 3, length_range=(512, 4096), num_requests=64,
                      dup_prob=0.1),
}


@dataclasses.dataclass(frozen=True)
class FragmentSpec:
    seed: int
    seq_len: int
    k_scale: float
    v_scale: float


def fragment_specs(w: Workload, request: int = 0) -> List[FragmentSpec]:
    """Length, scales and data seed of each distinct fragment of one request."""
    specs = []
    for i in range(w.num_fragments):
        seed = BASE_SEED + 1000 * request + i
        rng = np.random.default_rng(seed)
        if w.lengths is not None:
            T = int(w.lengths[i])
        else:
            lo, hi = w.length_range
            T = int(rng.integers(lo, hi + 1))
        if w.k_scales is not None:
            ks, vs = float(w.k_scales[i]), 1.0
        else:
            sc = float(rng.uniform(0.5, 1.5))
            ks, vs = sc, (sc if w.scale_v else 1.0)
        specs.append(FragmentSpec(seed, T, ks, vs))
    return specs


def delivery_schedule(w: Workload, request: int = 0) -> List[int]:
    """Fragment index of each delivery, duplicates included, in delivery order."""
    rng = np.random.default_rng(BASE_SEED + 1000 * request + 999)
    msgs = list(range(w.num_fragments))
    if w.dup_indices is not None:
        msgs += list(w.dup_indices)
    if w.num_dups:
        msgs += [int(x) for x in rng.choice(w.num_fragments, size=w.num_dups, replace=True)]
    if w.dup_prob > 0.0:
        msgs += [i for i in range(w.num_fragments) if rng.random() < w.dup_prob]
    if w.dup_indices is None:
        rng.shuffle(msgs)
    return msgs


def _torch():
    import torch
    return torch


def _rope_tables(torch, T: int, d: int, theta: float, device):
    half = d // 2
    inv_freq = 1.0 / (theta ** (torch.arange(0, half, device=device, dtype=torch.float32) * 2.0 / d))
    pos = torch.arange(T, device=device, dtype=torch.float32)
    ang = pos[:, None] * inv_freq[None, :]
    return torch.cos(ang), torch.sin(ang)


def make_fragment_torch(spec: FragmentSpec, L: int, H: int, d: int, device="cpu",
                        theta: float = ROPE_THETA):
    """(K, V) as bf16 torch tensors [L, H, T, d] on `device`, from spec.seed.

    Values are N(0,1) fp32, scaled, K rotated by R(t) at positions 0..T-1, then
    rounded to bf16 by torch. Generated one layer at a time to bound fp32 scratch.
    """
    torch = _torch()
    T = spec.seq_len
    gen = torch.Generator(device=device)
    gen.manual_seed(spec.seed)
    K = torch.empty((L, H, T, d), dtype=torch.bfloat16, device=device)
    V = torch.empty((L, H, T, d), dtype=torch.bfloat16, device=device)
    cos, sin = _rope_tables(torch, T, d, theta, device)
    half = d // 2
    for l in range(L):
        k = torch.randn((H, T, d), generator=gen, device=device, dtype=torch.float32) * spec.k_scale
        v = torch.randn((H, T, d), generator=gen, device=device, dtype=torch.float32) * spec.v_scale
        k1, k2 = k[..., :half], k[..., half:]
        kr = torch.cat([k1 * cos - k2 * sin, k2 * cos + k1 * sin], dim=-1)
        K[l] = kr.to(torch.bfloat16)
        V[l] = v.to(torch.bfloat16)
    return K, V


def to_bits(t) -> np.ndarray:
    """bf16 torch tensor (any device) -> numpy uint16 array of its raw bits."""
    torch = _torch()
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def make_fragment_bits(spec: FragmentSpec, L: int, H: int, d: int, theta: float = ROPE_THETA):
    """(K, V) as numpy uint16 bit arrays [L, H, T, d], generated on the CPU."""
    K, V = make_fragment_torch(spec, L, H, d, "cpu", theta)
    return to_bits(K), to_bits(V)


def random_bits(rng: np.random.Generator, shape, scale: float = 1.0) -> np.ndarray:
    """Gaussian values rounded to bf16 (by torch), as uint16 bits; for small tests."""
    torch = _torch()
    x = torch.from_numpy(rng.standard_normal(size=shape).astype(np.float32) * np.float32(scale))
    return to_bits(x.to(torch.bfloat16))
