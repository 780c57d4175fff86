"""ctypes binding of libcm.so (include/cm.h): argument marshalling only.

Every function of the C ABI is exposed under its own name, taking plain ints for
pointers and handles and raising CMError when the call returns a status other
than CM_OK. Context / FragmentSet wrap the handles for use with torch CUDA
tensors (torch is used for device memory and streams only).
"""
from __future__ import annotations

import ctypes
import enum
import os
from typing import List, Optional, Sequence, Tuple

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
# CM_LIBRARY names another build of the same library (the bounds-checked testing build,
# libcm_bounds.so); by default the in-tree libcm.so
LIB_PATH = os.environ.get("CM_LIBRARY") or os.path.join(PKG_DIR, "libcm.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is not built: run `python -c \"import __graft_entry__ as g; "
                      f"g.build()\"` (nvcc, sm_103a) first; there is no fallback implementation")

lib = ctypes.CDLL(LIB_PATH)


class Status(enum.IntEnum):
    OK = 0
    ERR_INVALID_ARG = 1
    ERR_SHAPE_MISMATCH = 2
    ERR_CAPACITY = 3
    ERR_ALIGNMENT = 4
    ERR_COLLISION = 5
    ERR_CUDA = 6
    ERR_OOM = 7
    ERR_TIMEOUT = 8
    ERR_UNSUPPORTED = 9


class CMError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = Status(status) if status in Status._value2member_map_ else status
        super().__init__(f"{cm_status_string(status)}: {message}")


class cm_id(ctypes.Structure):
    _fields_ = [("b", ctypes.c_uint8 * 16)]

    def to_bytes(self) -> bytes:
        return bytes(self.b)


class cm_fragment(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("seq_len", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("k", ctypes.c_void_p), ("v", ctypes.c_void_p)]


class cm_kernel_times(ctypes.Structure):
    _fields_ = [("leaf_hash_ms", ctypes.c_double), ("leaf_hash_launches", ctypes.c_int64),
                ("inner_hash_ms", ctypes.c_double), ("inner_hash_launches", ctypes.c_int64),
                ("render_ms", ctypes.c_double), ("render_launches", ctypes.c_int64),
                ("leaf_hash_fragments", ctypes.c_int64), ("aux_launches", ctypes.c_int64)]

    def as_dict(self) -> dict:
        return {name: getattr(self, name) for name, _ in self._fields_}


class cm_paged_cache(ctypes.Structure):
    _fields_ = [("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p),
                ("block_table", ctypes.c_void_p), ("table_entries", ctypes.c_int64),
                ("block_size", ctypes.c_int64), ("stride_block", ctypes.c_int64),
                ("stride_layer", ctypes.c_int64), ("stride_head", ctypes.c_int64),
                ("stride_token", ctypes.c_int64)]


class cm_render_job(ctypes.Structure):
    _fields_ = [("set", ctypes.c_void_p), ("k_out", ctypes.c_void_p), ("v_out", ctypes.c_void_p),
                ("capacity_tokens", ctypes.c_int64)]


_c = ctypes
_P = ctypes.c_void_p
_SIGS = {
    "cm_abi_version": (_c.c_int32, []),
    "cm_status_string": (_c.c_char_p, [_c.c_int]),
    "cm_last_error_message": (_c.c_char_p, []),
    "cm_context_create": (_c.c_int, [_c.c_int32, _c.c_double, _c.c_int32, _c.c_int32,
                                     _c.POINTER(_P)]),
    "cm_context_destroy": (_c.c_int, [_P]),
    "cm_set_create": (_c.c_int, [_P, _c.POINTER(_P)]),
    "cm_set_destroy": (_c.c_int, [_P]),
    "cm_fragment_id": (_c.c_int, [_P, _c.POINTER(cm_fragment), _P, _c.POINTER(cm_id),
                                  _c.POINTER(_c.c_uint64)]),
    "cm_ingest": (_c.c_int, [_P, _c.POINTER(cm_fragment), _P, _c.POINTER(cm_id),
                             _c.POINTER(_c.c_int32)]),
    "cm_fragment_id_static": (_c.c_int, [_c.POINTER(cm_fragment), _c.c_int32, _P, _P,
                                         _c.POINTER(_c.c_uint64)]),
    "cm_ingest_batch": (_c.c_int, [_P, _c.POINTER(cm_fragment), _c.c_int32, _P,
                                   _c.POINTER(cm_id), _c.POINTER(_c.c_int32)]),
    "cm_ingest_many": (_c.c_int, [_c.POINTER(_P), _c.POINTER(cm_fragment), _c.c_int32, _P,
                                  _c.POINTER(cm_id), _c.POINTER(_c.c_int32)]),
    "cm_render_many": (_c.c_int, [_c.POINTER(cm_render_job), _c.c_int32, _P,
                                  _c.POINTER(_c.c_int64)]),
    "cm_ingest_render": (_c.c_int, [_c.POINTER(_P), _c.POINTER(cm_fragment), _c.c_int32, _P, _P, _P,
                                    _c.c_int64, _P, _c.POINTER(cm_id), _c.POINTER(_c.c_int32),
                                    _c.POINTER(_c.c_int64), _c.POINTER(cm_id), _c.POINTER(_c.c_int32)]),
    "cm_set_contains": (_c.c_int, [_P, _c.POINTER(cm_id), _c.c_int64, _c.POINTER(_c.c_uint8)]),
    "cm_set_leq": (_c.c_int, [_P, _P, _c.POINTER(_c.c_int32)]),
    "cm_measure_int_alu": (_c.c_int, [_c.c_int32, _c.POINTER(_c.c_double), _c.POINTER(_c.c_double)]),
    "cm_context_set_render_warps": (_c.c_int, [_P, _c.c_int32]),
    "cm_context_set_overlap": (_c.c_int, [_P, _c.c_int32]),
    "cm_context_set_dedup_by_bytes": (_c.c_int, [_P, _c.c_int32]),
    "cm_context_set_timing": (_c.c_int, [_P, _c.c_int32]),
    "cm_context_kernel_times": (_c.c_int, [_P, _c.POINTER(cm_kernel_times), _c.c_int32]),
    "cm_union": (_c.c_int, [_P, _P]),
    "cm_context_check": (_c.c_int, [_P, _P]),
    "cm_set_size": (_c.c_int, [_P, _c.POINTER(_c.c_int64)]),
    "cm_set_seq_len": (_c.c_int, [_P, _c.POINTER(_c.c_int64)]),
    "cm_set_ids": (_c.c_int, [_P, _c.POINTER(cm_id), _c.c_int64]),
    "cm_render": (_c.c_int, [_P, _P, _P, _c.c_int64, _P, _c.POINTER(_c.c_int64),
                             _c.POINTER(cm_id)]),
    "cm_bagmerge": (_c.c_int, [_P, _c.POINTER(cm_fragment), _c.c_int32, _P, _P, _c.c_int64, _P,
                               _c.POINTER(_c.c_int64)]),
    "cm_testing_render_withheld_load": (_c.c_int, [_P, _P, _P, _c.c_int64, _P]),
    "cm_testing_bounds_violations": (_c.c_int, [_c.c_int32, _c.POINTER(_c.c_uint64),
                                                _c.POINTER(_c.c_int32)]),
    "cm_render_paged": (_c.c_int, [_P, _c.POINTER(cm_paged_cache), _P, _c.POINTER(_c.c_int64),
                                   _c.POINTER(cm_id)]),
    "cm_render_incremental": (_c.c_int, [_P, _P, _P, _c.c_int64, _c.POINTER(cm_id), _c.c_int64, _P,
                                         _c.POINTER(_c.c_int64), _c.POINTER(cm_id),
                                         _c.POINTER(_c.c_int64)]),
}
for _name, (_res, _args) in _SIGS.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args

EXPORTED = tuple(_SIGS)


def cm_abi_version() -> int:
    return lib.cm_abi_version()


def cm_status_string(status: int) -> str:
    return lib.cm_status_string(int(status)).decode()


def cm_last_error_message() -> str:
    return lib.cm_last_error_message().decode()


def _check(status: int) -> None:
    if status != 0:
        raise CMError(status, cm_last_error_message())


def _stream_handle(stream) -> Optional[int]:
    """None -> torch's current stream if torch is loaded with CUDA, else the legacy default."""
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream or None
        except ImportError:
            pass
        return None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


def cm_context_create(device: int = 0, rope_theta: float = 1.0e6, routing_layer: int = -1,
                      verify_bytes_on_hit: bool = False) -> int:
    out = _P()
    _check(lib.cm_context_create(device, rope_theta, routing_layer, int(verify_bytes_on_hit),
                                 ctypes.byref(out)))
    return out.value


def cm_context_destroy(ctx: Optional[int]) -> None:
    _check(lib.cm_context_destroy(ctx))


def cm_context_check(ctx: int, stream=None) -> None:
    _check(lib.cm_context_check(ctx, _stream_handle(stream)))


def cm_testing_bounds_violations(device: int = 0) -> Tuple[int, bool]:
    """(count, enabled): out-of-buffer accesses counted by a bounds-checked build since the
    previous call (the device is synchronised), and whether this library is such a build."""
    n, en = ctypes.c_uint64(), ctypes.c_int32()
    _check(lib.cm_testing_bounds_violations(device, ctypes.byref(n), ctypes.byref(en)))
    return n.value, bool(en.value)


def cm_set_create(ctx: int) -> int:
    out = _P()
    _check(lib.cm_set_create(ctx, ctypes.byref(out)))
    return out.value


def cm_set_destroy(s: Optional[int]) -> None:
    _check(lib.cm_set_destroy(s))


def cm_fragment_id(ctx: int, frag: cm_fragment, stream=None,
                   want_norm_key: bool = True) -> Tuple[bytes, Optional[List[int]]]:
    out = cm_id()
    q = (ctypes.c_uint64 * frag.seq_len)() if want_norm_key else None
    _check(lib.cm_fragment_id(ctx, ctypes.byref(frag), _stream_handle(stream), ctypes.byref(out),
                              q))
    return out.to_bytes(), (list(q) if q is not None else None)


def cm_fragment_id_static(frag: cm_fragment, id_out: int, norm_key_out: int,
                          routing_layer: int = -1, stream=None) -> None:
    """Allocation-free id + norm key into caller-owned device buffers (asynchronous)."""
    _check(lib.cm_fragment_id_static(ctypes.byref(frag), routing_layer, _stream_handle(stream),
                                     id_out, ctypes.cast(norm_key_out, ctypes.POINTER(ctypes.c_uint64))))


def cm_ingest(s: int, frag: cm_fragment, stream=None) -> Tuple[bytes, bool]:
    out = cm_id()
    absorbed = ctypes.c_int32(0)
    _check(lib.cm_ingest(s, ctypes.byref(frag), _stream_handle(stream), ctypes.byref(out),
                         ctypes.byref(absorbed)))
    return out.to_bytes(), bool(absorbed.value)


def cm_ingest_batch(s: int, frags: Sequence[cm_fragment], stream=None) -> List[Tuple[bytes, bool]]:
    n = len(frags)
    arr = (cm_fragment * max(n, 1))(*frags)
    ids = (cm_id * max(n, 1))()
    absorbed = (ctypes.c_int32 * max(n, 1))()
    _check(lib.cm_ingest_batch(s, arr, n, _stream_handle(stream), ids, absorbed))
    return [(ids[i].to_bytes(), bool(absorbed[i])) for i in range(n)]


def cm_ingest_many(sets: Sequence[int], frags: Sequence[cm_fragment],
                   stream=None) -> List[Tuple[bytes, bool]]:
    n = len(frags)
    if len(sets) != n:
        raise ValueError("one set per delivery")
    set_arr = (_P * max(n, 1))(*sets)
    arr = (cm_fragment * max(n, 1))(*frags)
    ids = (cm_id * max(n, 1))()
    absorbed = (ctypes.c_int32 * max(n, 1))()
    _check(lib.cm_ingest_many(set_arr, arr, n, _stream_handle(stream), ids, absorbed))
    return [(ids[i].to_bytes(), bool(absorbed[i])) for i in range(n)]


def cm_ingest_render(sets: Sequence[int], frags: Sequence[cm_fragment], target: int, k_out: int,
                     v_out: int, capacity_tokens: int, stream=None):
    """cm_ingest_render: returns ([(id, absorbed)] per delivery, rendered length, canonical
    order as a list of ids, overlapped flag)."""
    n = len(frags)
    if len(sets) != n:
        raise ValueError("one set per delivery")
    set_arr = (_P * max(n, 1))(*sets)
    arr = (cm_fragment * max(n, 1))(*frags)
    ids = (cm_id * max(n, 1))()
    absorbed = (ctypes.c_int32 * max(n, 1))()
    seq = ctypes.c_int64()
    cap_order = n + 64
    order = (cm_id * cap_order)()
    ovl = ctypes.c_int32()
    # the order array must hold the target's final size: at most its current size plus
    # every other set's and every delivery's
    members = cm_set_size(target) + n + sum(cm_set_size(s) for s in set(sets) if s != target)
    if members > cap_order:
        order = (cm_id * members)()
    _check(lib.cm_ingest_render(set_arr, arr, n, target, k_out, v_out, capacity_tokens,
                                _stream_handle(stream), ids, absorbed, ctypes.byref(seq), order,
                                ctypes.byref(ovl)))
    size = cm_set_size(target)
    return ([(ids[i].to_bytes(), bool(absorbed[i])) for i in range(n)], seq.value,
            [order[i].to_bytes() for i in range(size)], bool(ovl.value))


def cm_render_many(jobs: Sequence[cm_render_job], stream=None) -> List[int]:
    n = len(jobs)
    arr = (cm_render_job * max(n, 1))(*jobs)
    seq = (ctypes.c_int64 * max(n, 1))()
    _check(lib.cm_render_many(arr, n, _stream_handle(stream), seq))
    return [seq[i] for i in range(n)]


def cm_set_contains(s: int, ids: Sequence[bytes]) -> List[bool]:
    n = len(ids)
    arr = (cm_id * max(n, 1))()
    for i, fid in enumerate(ids):
        arr[i].b[:] = list(fid)
    out = (ctypes.c_uint8 * max(n, 1))()
    _check(lib.cm_set_contains(s, arr, n, out))
    return [bool(out[i]) for i in range(n)]


def cm_set_leq(a: int, b: int) -> bool:
    out = ctypes.c_int32()
    _check(lib.cm_set_leq(a, b, ctypes.byref(out)))
    return bool(out.value)


def cm_measure_int_alu(device: int = 0) -> Tuple[float, float]:
    """(xor3_tops, compress_tops): register-only integer-ALU throughput of the device."""
    x, c = ctypes.c_double(), ctypes.c_double()
    _check(lib.cm_measure_int_alu(device, ctypes.byref(x), ctypes.byref(c)))
    return x.value, c.value


def cm_context_set_dedup_by_bytes(ctx: int, enable: bool) -> None:
    _check(lib.cm_context_set_dedup_by_bytes(ctx, int(enable)))


def cm_context_set_overlap(ctx: int, mode: int) -> None:
    _check(lib.cm_context_set_overlap(ctx, mode))


def cm_context_set_render_warps(ctx: int, warps: int) -> None:
    _check(lib.cm_context_set_render_warps(ctx, warps))


def cm_context_set_timing(ctx: int, enable: bool) -> None:
    _check(lib.cm_context_set_timing(ctx, int(enable)))


def cm_context_kernel_times(ctx: int, reset: bool = False) -> dict:
    out = cm_kernel_times()
    _check(lib.cm_context_kernel_times(ctx, ctypes.byref(out), int(reset)))
    return out.as_dict()


def cm_union(dst: int, src: int) -> None:
    _check(lib.cm_union(dst, src))


def cm_set_size(s: int) -> int:
    out = ctypes.c_int64()
    _check(lib.cm_set_size(s, ctypes.byref(out)))
    return out.value


def cm_set_seq_len(s: int) -> int:
    out = ctypes.c_int64()
    _check(lib.cm_set_seq_len(s, ctypes.byref(out)))
    return out.value


def cm_set_ids(s: int) -> List[bytes]:
    n = cm_set_size(s)
    arr = (cm_id * max(n, 1))()
    _check(lib.cm_set_ids(s, arr, n))
    return [arr[i].to_bytes() for i in range(n)]


def cm_render(s: int, k_out: int, v_out: int, capacity_tokens: int,
              stream=None, want_order: bool = True) -> Tuple[int, Optional[List[bytes]]]:
    """(rendered length, canonical order); the order is None when want_order is False."""
    seq = ctypes.c_int64()
    if not want_order:
        _check(lib.cm_render(s, k_out, v_out, capacity_tokens, _stream_handle(stream),
                             ctypes.byref(seq), None))
        return seq.value, None
    n = cm_set_size(s)
    order = (cm_id * max(n, 1))()
    _check(lib.cm_render(s, k_out, v_out, capacity_tokens, _stream_handle(stream),
                         ctypes.byref(seq), order))
    return seq.value, [order[i].to_bytes() for i in range(n)]


def cm_render_incremental(s: int, k_out: int, v_out: int, capacity_tokens: int,
                          prev_order: Sequence[bytes], stream=None) -> Tuple[int, List[bytes], int]:
    n = cm_set_size(s)
    order = (cm_id * max(n, 1))()
    prev = (cm_id * max(len(prev_order), 1))()
    for i, fid in enumerate(prev_order):
        prev[i].b[:] = list(fid)
    seq = ctypes.c_int64()
    reused = ctypes.c_int64()
    _check(lib.cm_render_incremental(s, k_out, v_out, capacity_tokens, prev, len(prev_order),
                                     _stream_handle(stream), ctypes.byref(seq), order,
                                     ctypes.byref(reused)))
    return seq.value, [order[i].to_bytes() for i in range(n)], reused.value


def cm_render_paged(s: int, cache: cm_paged_cache, stream=None) -> Tuple[int, List[bytes]]:
    n = cm_set_size(s)
    order = (cm_id * max(n, 1))()
    seq = ctypes.c_int64()
    _check(lib.cm_render_paged(s, ctypes.byref(cache), _stream_handle(stream), ctypes.byref(seq),
                               order))
    return seq.value, [order[i].to_bytes() for i in range(n)]


def cm_bagmerge(ctx: int, frags: Sequence[cm_fragment], k_out: int, v_out: int,
                capacity_tokens: int, stream=None) -> int:
    arr = (cm_fragment * max(len(frags), 1))(*frags)
    seq = ctypes.c_int64()
    _check(lib.cm_bagmerge(ctx, arr, len(frags), k_out, v_out, capacity_tokens,
                           _stream_handle(stream), ctypes.byref(seq)))
    return seq.value


# ---------------------------------------------------------------- torch-facing helpers

def fragment_from_tensors(K, V) -> cm_fragment:
    """Descriptor of a fragment held in two bf16 CUDA tensors [L, H, T, d] (contiguous)."""
    import torch
    if K.shape != V.shape or K.dim() != 4:
        raise ValueError("K and V must both be [layers, kv_heads, seq_len, head_dim]")
    for t in (K, V):
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
            raise ValueError("K and V must be contiguous bf16 CUDA tensors")
    L, H, T, d = K.shape
    return cm_fragment(L, H, T, d, K.data_ptr(), V.data_ptr())


class Context:
    """A libcm context on one CUDA device."""

    def __init__(self, device: int = 0, rope_theta: float = 1.0e6, routing_layer: int = -1,
                 verify_bytes_on_hit: bool = False):
        self.handle = cm_context_create(device, rope_theta, routing_layer, verify_bytes_on_hit)
        self.device = device
        self.rope_theta = rope_theta

    def close(self):
        if self.handle:
            cm_context_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def check(self, stream=None) -> None:
        cm_context_check(self.handle, stream)

    def fragment_id(self, K, V, stream=None):
        return cm_fragment_id(self.handle, fragment_from_tensors(K, V), stream)

    def bagmerge(self, fragments, k_out, v_out, stream=None) -> int:
        """BagMerge in the given order; fragments = [(K, V), ...] tensors."""
        frags = [fragment_from_tensors(K, V) for K, V in fragments]
        return cm_bagmerge(self.handle, frags, k_out.data_ptr(), v_out.data_ptr(),
                           k_out.shape[2], stream)


class FragmentSet:
    """A LatentFragmentSet. Holds a reference to every ingested tensor pair it keeps,
    because the library borrows fragment memory."""

    def __init__(self, ctx: Context):
        self.ctx = ctx
        self.handle = cm_set_create(ctx.handle)
        self._keep = {}
        self._held = []   # tensors of failed batch calls, some of which the set may hold

    def close(self):
        if self.handle:
            cm_set_destroy(self.handle)
            self.handle = None
            self._keep.clear()
            self._held.clear()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def ingest_batch(self, pairs, stream=None) -> List[Tuple[bytes, bool]]:
        """Ingest [(K, V), ...] in order with one synchronisation."""
        pairs = list(pairs)
        try:
            res = cm_ingest_batch(self.handle, [fragment_from_tensors(K, V) for K, V in pairs],
                                  stream)
        except CMError:
            # the deliveries before a failing one (CM_ERR_COLLISION) are in the set
            self._held.extend(pairs)
            raise
        for (fid, absorbed), kv in zip(res, pairs):
            if not absorbed:
                self._keep.setdefault(fid, kv)
        return res

    def ingest(self, K, V, stream=None) -> Tuple[bytes, bool]:
        fid, absorbed = cm_ingest(self.handle, fragment_from_tensors(K, V), stream)
        if not absorbed:
            self._keep[fid] = (K, V)
        return fid, absorbed

    def union(self, other: "FragmentSet") -> None:
        cm_union(self.handle, other.handle)
        for fid, kv in other._keep.items():
            self._keep.setdefault(fid, kv)
        self._held.extend(other._held)

    def __len__(self) -> int:
        return cm_set_size(self.handle)

    def contains(self, ids: Sequence[bytes]) -> List[bool]:
        """Membership of each id (for replica exchange: ship only what the other lacks)."""
        return cm_set_contains(self.handle, ids)

    def __le__(self, other: "FragmentSet") -> bool:
        """The inclusion order of Section 4.4: every id of self is in other."""
        return cm_set_leq(self.handle, other.handle)

    def ids(self) -> List[bytes]:
        return cm_set_ids(self.handle)

    def seq_len(self) -> int:
        return cm_set_seq_len(self.handle)

    def render_incremental(self, k_out, v_out, prev_order, stream=None):
        """(seq_len, order, reused_tokens): re-render only what changed since prev_order."""
        return cm_render_incremental(self.handle, k_out.data_ptr(), v_out.data_ptr(),
                                     k_out.shape[2], prev_order, stream)

    def render(self, k_out, v_out, stream=None) -> Tuple[int, List[bytes]]:
        return cm_render(self.handle, k_out.data_ptr() if k_out is not None else 0,
                         v_out.data_ptr() if v_out is not None else 0,
                         k_out.shape[2] if k_out is not None else 0, stream)


def ingest_many(deliveries, stream=None) -> List[Tuple[bytes, bool]]:
    """Ingest [(FragmentSet, K, V), ...] in order, one GPU pass and one synchronisation
    for all of them; deliveries may go to different sets."""
    deliveries = list(deliveries)
    try:
        res = cm_ingest_many([S.handle for S, _, _ in deliveries],
                             [fragment_from_tensors(K, V) for _, K, V in deliveries], stream)
    except CMError:
        # the deliveries before a failing one (CM_ERR_COLLISION) are in their sets
        for S, K, V in deliveries:
            S._held.append((K, V))
        raise
    for (fid, absorbed), (S, K, V) in zip(res, deliveries):
        if not absorbed:
            S._keep.setdefault(fid, (K, V))
    return res


def render_many(jobs, stream=None) -> List[int]:
    """Render [(FragmentSet, k_out, v_out), ...] in shared launches; returns the lengths."""
    return cm_render_many([cm_render_job(S.handle, k.data_ptr() if k is not None else 0,
                                         v.data_ptr() if v is not None else 0,
                                         k.shape[2] if k is not None else 0)
                           for S, k, v in jobs], stream)
