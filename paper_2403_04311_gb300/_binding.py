"""ctypes binding of the alto_agg C ABI (include/alto_agg.h).

Argument marshalling only: every step of the aggregation runs in the CUDA
library.  PyTorch supplies device memory (its caching allocator, through the
ABI's allocator callbacks) and streams.  Loading fails loudly when the
compiled library is missing -- there is no other implementation to fall back
to.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import _build

MAX_DEPTH = 8
OK, EINVAL, ENOMEM, ENOSPC, EDUP, ELAST, EINCONSIST, ECLOSED, ETIMEOUT, ECUDA = (
    0, -1, -2, -3, -4, -5, -6, -7, -8, -9)
STATUS_NAMES = {OK: "OK", EINVAL: "EINVAL", ENOMEM: "ENOMEM", ENOSPC: "ENOSPC", EDUP: "EDUP",
                ELAST: "ELAST", EINCONSIST: "EINCONSIST", ECLOSED: "ECLOSED",
                ETIMEOUT: "ETIMEOUT", ECUDA: "ECUDA"}
PAYLOAD_NONE, PAYLOAD_CONCAT = 0, 1
SCORE_NONE, SCORE_MAX, SCORE_TOPK = 0, 1, 2
FLAG_STREAM_RELEASE = 1
FLAG_DOUBLE_RING = 2
FLAG_TEST_STALL = 4
FLAG_DIRECT_LAUNCH = 8
OPS_PARTIAL = 0x80

RECORD_DTYPE = np.dtype([
    ("completion_seq", "<u8"), ("payload_off", "<u8"), ("payload_len", "<u8"),
    ("topk_off", "<u8"), ("parent_id", "<u4"), ("n_children", "<u4"),
    ("level", "u1"), ("ops", "u1"), ("topk_n", "<u2"), ("score", "<f4"),
])
PAIR_DTYPE = np.dtype([("child_index", "<u4"), ("score", "<f4")])


class alto_agg_config(ctypes.Structure):
    _fields_ = [
        ("depth", ctypes.c_int32),
        ("payload_op", ctypes.c_int32 * MAX_DEPTH),
        ("score_op", ctypes.c_int32 * MAX_DEPTH),
        ("topk_k", ctypes.c_int32 * MAX_DEPTH),
        ("max_batch_fragments", ctypes.c_int64),
        ("max_batch_payload", ctypes.c_int64),
        ("max_open_groups", ctypes.c_int64),
        ("arena_elems", ctypes.c_int64),
        ("out_records", ctypes.c_int64),
        ("out_payload_elems", ctypes.c_int64),
        ("out_topk", ctypes.c_int64),
        ("max_emit_children", ctypes.c_int64),
        ("spin_limit", ctypes.c_int64),
        ("flags", ctypes.c_int64),
    ]


ALLOC_FN = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)
FREE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p)


class alto_allocator(ctypes.Structure):
    _fields_ = [("ctx", ctypes.c_void_p), ("alloc", ALLOC_FN), ("free", FREE_FN)]


class alto_batch(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_int64), ("depth", ctypes.c_int32), ("reserved", ctypes.c_int32),
        ("tags", ctypes.c_void_p), ("payload_off", ctypes.c_void_p),
        ("n_payload", ctypes.c_int64), ("payload", ctypes.c_void_p), ("score", ctypes.c_void_p),
    ]


class alto_drain(ctypes.Structure):
    _fields_ = [
        ("n_records", ctypes.c_int64), ("records", ctypes.c_void_p),
        ("n_payload", ctypes.c_int64), ("payload", ctypes.c_void_p),
        ("n_topk", ctypes.c_int64), ("topk", ctypes.c_void_p),
        ("first_batch", ctypes.c_uint64), ("n_batches", ctypes.c_uint64),
    ]


NUM_STAGES = 10
STAGE_NAMES = ("ingest", "leaf_sort", "leaf_accumulate", "leaf_finalize", "upper_levels",
               "emit_order", "carry_over", "dense_place", "gather", "records")


class alto_profile(ctypes.Structure):
    _fields_ = [("pushes", ctypes.c_int64), ("launches", ctypes.c_int64),
                ("stage_ms", ctypes.c_double * NUM_STAGES),
                ("stage_launches", ctypes.c_int64 * NUM_STAGES)]


MAX_DELIMS = 32


class alto_split_args(ctypes.Structure):
    _fields_ = [("n_src", ctypes.c_int64), ("n_tokens", ctypes.c_int64),
                ("depth_in", ctypes.c_int32), ("n_delims", ctypes.c_int32),
                ("delims", ctypes.c_int32 * MAX_DELIMS),
                ("src_tags", ctypes.c_void_p), ("src_id", ctypes.c_void_p),
                ("tok_off", ctypes.c_void_p), ("tokens", ctypes.c_void_p),
                ("cap_frag", ctypes.c_int64), ("out_tags", ctypes.c_void_p),
                ("out_off", ctypes.c_void_p), ("out_counts", ctypes.c_void_p),
                ("scratch", ctypes.c_void_p), ("scratch_bytes", ctypes.c_int64)]


ROUTE_HASH, ROUTE_LEAST_LOADED = 0, 1


class alto_router_config(ctypes.Structure):
    _fields_ = [("depth", ctypes.c_int32), ("level", ctypes.c_int32), ("n_replicas", ctypes.c_int32),
                ("policy", ctypes.c_int32), ("max_batch_fragments", ctypes.c_int64),
                ("max_batch_payload", ctypes.c_int64), ("max_flows", ctypes.c_int64),
                ("with_score", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class alto_routed(ctypes.Structure):
    _fields_ = [("replica", ctypes.c_void_p), ("perm", ctypes.c_void_p), ("frag_off", ctypes.c_void_p),
                ("pay_off", ctypes.c_void_p), ("tags", ctypes.c_void_p), ("payload_off", ctypes.c_void_p),
                ("payload", ctypes.c_void_p), ("score", ctypes.c_void_p)]


EXPORTS = ("alto_agg_create", "alto_agg_push_batch", "alto_agg_drain", "alto_agg_stats",
           "alto_agg_profile", "alto_agg_profile_read", "alto_agg_oneshot_noalloc",
           "alto_agg_destroy", "alto_split_scratch_bytes", "alto_split_text",
           "alto_router_create", "alto_router_route", "alto_router_counts", "alto_router_release",
           "alto_router_destroy")

_lib = None


def load_library(build: bool = True):
    """Load (building first if needed) libalto_agg.so."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.build() if build else _build.LIB
    if not os.path.exists(path):
        raise RuntimeError(f"alto_agg CUDA library missing at {path}; run the package build")
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    lib.alto_agg_create.restype = ctypes.c_int
    lib.alto_agg_create.argtypes = [ctypes.POINTER(alto_agg_config), ctypes.POINTER(alto_allocator),
                                    P, ctypes.POINTER(P)]
    lib.alto_agg_push_batch.restype = ctypes.c_int
    lib.alto_agg_push_batch.argtypes = [P, ctypes.POINTER(alto_batch), P]
    lib.alto_agg_drain.restype = ctypes.c_int
    lib.alto_agg_drain.argtypes = [P, P, ctypes.POINTER(alto_drain)]
    lib.alto_agg_stats.restype = ctypes.c_int
    lib.alto_agg_stats.argtypes = [P, P, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
    lib.alto_agg_destroy.restype = ctypes.c_int
    lib.alto_agg_destroy.argtypes = [P]
    lib.alto_agg_profile.restype = ctypes.c_int
    lib.alto_agg_profile.argtypes = [P, ctypes.c_int]
    lib.alto_agg_profile_read.restype = ctypes.c_int
    lib.alto_agg_profile_read.argtypes = [P, ctypes.POINTER(alto_profile)]
    lib.alto_agg_oneshot_noalloc.restype = ctypes.c_int
    lib.alto_agg_oneshot_noalloc.argtypes = [
        ctypes.POINTER(alto_agg_config), ctypes.POINTER(alto_batch), P, ctypes.c_int64, P,
        ctypes.c_int64, P, ctypes.c_int64, P, P]
    lib.alto_split_scratch_bytes.restype = ctypes.c_int64
    lib.alto_split_scratch_bytes.argtypes = [ctypes.c_int64, ctypes.c_int64]
    lib.alto_split_text.restype = ctypes.c_int
    lib.alto_split_text.argtypes = [ctypes.POINTER(alto_split_args), P]
    lib.alto_router_create.restype = ctypes.c_int
    lib.alto_router_create.argtypes = [ctypes.POINTER(alto_router_config), ctypes.POINTER(alto_allocator), P,
                                       ctypes.POINTER(P)]
    lib.alto_router_route.restype = ctypes.c_int
    lib.alto_router_route.argtypes = [P, ctypes.POINTER(alto_batch), P, ctypes.POINTER(alto_routed)]
    lib.alto_router_counts.restype = ctypes.c_int
    lib.alto_router_counts.argtypes = [P, P, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
    lib.alto_router_release.restype = ctypes.c_int
    lib.alto_router_release.argtypes = [P, P, ctypes.c_int64, P]
    lib.alto_router_destroy.restype = ctypes.c_int
    lib.alto_router_destroy.argtypes = [P]
    _lib = lib
    return lib


def make_config(depth, payload_op, score_op, topk_k=None, *, max_batch_fragments,
                max_batch_payload, max_open_groups=0, arena_elems=0, out_records=0,
                out_payload_elems=0, out_topk=0, max_emit_children=0, spin_limit=0,
                stream_release=False, double_ring=False, test_stall=False, direct_launch=False):
    c = alto_agg_config()
    c.depth = depth
    topk_k = topk_k or [0] * depth
    for l in range(min(depth, MAX_DEPTH)):
        c.payload_op[l] = int(payload_op[l])
        c.score_op[l] = int(score_op[l])
        c.topk_k[l] = int(topk_k[l])
    c.max_batch_fragments = int(max_batch_fragments)
    c.max_batch_payload = int(max_batch_payload)
    c.max_open_groups = int(max_open_groups)
    c.arena_elems = int(arena_elems)
    c.out_records = int(out_records)
    c.out_payload_elems = int(out_payload_elems)
    c.out_topk = int(out_topk)
    c.max_emit_children = int(max_emit_children)
    c.spin_limit = int(spin_limit)
    c.flags = ((FLAG_STREAM_RELEASE if stream_release else 0) | (FLAG_DOUBLE_RING if double_ring else 0) |
               (FLAG_TEST_STALL if test_stall else 0) | (FLAG_DIRECT_LAUNCH if direct_launch else 0))
    return c


class _TorchAllocator:
    """The ABI allocator callbacks backed by PyTorch's caching allocator."""

    def __init__(self, device):
        import torch
        self._torch = torch
        self._device = device

        def _alloc(_ctx, nbytes, stream):
            return self._torch.cuda.caching_allocator_alloc(int(nbytes), self._device,
                                                            int(stream or 0))

        def _free(_ctx, ptr, _stream):
            if ptr:
                self._torch.cuda.caching_allocator_delete(int(ptr))

        self._alloc = ALLOC_FN(_alloc)
        self._free = FREE_FN(_free)
        self.struct = alto_allocator(None, self._alloc, self._free)


def alto_agg_create(cfg: alto_agg_config, allocator=None, stream=0):
    """Returns (status, handle).  ``allocator`` is an alto_allocator struct,
    a _TorchAllocator, or None (library uses cudaMallocAsync)."""
    lib = load_library()
    h = ctypes.c_void_p()
    a = allocator.struct if isinstance(allocator, _TorchAllocator) else allocator
    st = lib.alto_agg_create(ctypes.byref(cfg), ctypes.byref(a) if a is not None else None,
                             ctypes.c_void_p(stream), ctypes.byref(h))
    return st, h


def alto_agg_push_batch(h, batch: alto_batch, stream=0) -> int:
    return load_library().alto_agg_push_batch(h, ctypes.byref(batch), ctypes.c_void_p(stream))


def alto_agg_drain(h, stream=0):
    d = alto_drain()
    st = load_library().alto_agg_drain(h, ctypes.c_void_p(stream), ctypes.byref(d))
    return st, d


def alto_agg_stats(h, stream=0):
    og, au = ctypes.c_int64(), ctypes.c_int64()
    st = load_library().alto_agg_stats(h, ctypes.c_void_p(stream), ctypes.byref(og), ctypes.byref(au))
    return st, og.value, au.value


def alto_agg_destroy(h) -> int:
    return load_library().alto_agg_destroy(h)


def alto_agg_oneshot_noalloc(cfg, batch, out_records, cap_records, out_payload, cap_payload,
                             out_topk, cap_topk, out_counts, stream=0) -> int:
    """All pointers are device addresses (ints); the call allocates nothing."""
    return load_library().alto_agg_oneshot_noalloc(
        ctypes.byref(cfg), ctypes.byref(batch), ctypes.c_void_p(out_records), cap_records,
        ctypes.c_void_p(out_payload), cap_payload, ctypes.c_void_p(out_topk), cap_topk,
        ctypes.c_void_p(out_counts), ctypes.c_void_p(stream))


PROFILE_OFF, PROFILE_STAGES, PROFILE_HOT = 0, 1, 2


def alto_agg_profile(h, enable) -> int:
    """enable: False/0 off, True/1 every stage boundary, 2 the leaf accumulate
    and gather stages only."""
    mode = PROFILE_STAGES if enable is True else int(enable)
    return load_library().alto_agg_profile(h, mode)


def alto_split_scratch_bytes(n_src: int, n_tokens: int) -> int:
    return load_library().alto_split_scratch_bytes(n_src, n_tokens)


def alto_split_text(args, stream=0) -> int:
    return load_library().alto_split_text(ctypes.byref(args), ctypes.c_void_p(stream))


def split_text(src_tags, src_id, tok_off, tokens, delims, cap_frag=None, stream=None):
    """Device tensors in (src_tags uint64 [depth_in, n_src] or None, src_id
    int32/uint32 [n_src], tok_off int32 [n_src + 1], tokens int32), device
    tensors out: (status, n_frag, tags [depth_in + 1, n_frag] as int64 bits,
    off [n_frag + 1] as int32).  Allocation only; every step runs in the
    library's kernels."""
    import torch
    n_src = int(src_id.numel())
    n_tokens = int(tokens.numel())
    depth_in = 0 if src_tags is None else int(src_tags.shape[0])
    cap = int(cap_frag) if cap_frag is not None else n_tokens + n_src
    dev = tokens.device
    stream = stream or torch.cuda.current_stream()
    out_tags = torch.empty((depth_in + 1) * max(cap, 1), dtype=torch.int64, device=dev)
    out_off = torch.empty(cap + 1, dtype=torch.int32, device=dev)
    counts = torch.zeros(2, dtype=torch.int64, device=dev)
    nbytes = alto_split_scratch_bytes(n_src, n_tokens)
    scratch = torch.empty(max(nbytes, 256) + 256, dtype=torch.uint8, device=dev)
    base = (scratch.data_ptr() + 255) & ~255
    a = alto_split_args()
    a.n_src, a.n_tokens, a.depth_in, a.n_delims = n_src, n_tokens, depth_in, len(delims)
    for k, x in enumerate(delims):
        a.delims[k] = int(x)
    a.src_tags = src_tags.data_ptr() if src_tags is not None else None
    a.src_id, a.tok_off = src_id.data_ptr(), tok_off.data_ptr()
    a.tokens = tokens.data_ptr() if n_tokens else None
    a.cap_frag = cap
    a.out_tags, a.out_off, a.out_counts = out_tags.data_ptr(), out_off.data_ptr(), counts.data_ptr()
    a.scratch, a.scratch_bytes = base, nbytes
    st = alto_split_text(a, stream.cuda_stream)
    if st != OK:
        return st, 0, None, None
    torch.cuda.current_stream().synchronize() if stream is None else stream.synchronize()
    status, n_frag = (int(x) for x in counts.cpu().tolist())
    if status != OK:
        return status, n_frag, None, None
    tags = out_tags[:(depth_in + 1) * n_frag].view(depth_in + 1, n_frag)
    return status, n_frag, tags, out_off[:n_frag + 1]


def alto_agg_profile_read(h):
    p = alto_profile()
    st = load_library().alto_agg_profile_read(h, ctypes.byref(p))
    return st, dict(pushes=p.pushes, launches=p.launches,
                    stage_ms={STAGE_NAMES[i]: p.stage_ms[i] for i in range(NUM_STAGES)},
                    stage_launches={STAGE_NAMES[i]: p.stage_launches[i] for i in range(NUM_STAGES)})


class _DevView:
    """A raw device buffer exposed through __cuda_array_interface__."""

    def __init__(self, ptr, nbytes):
        self.__cuda_array_interface__ = {
            "shape": (int(nbytes),), "typestr": "|u1", "data": (int(ptr), False), "version": 3,
        }


class Drain:
    """What one drain returned: status, the batch range, and device views of
    the records (uint8, 48 bytes each), payload (int32) and top-k pairs (uint8,
    8 bytes each).  The views are made on first access (they are only valid
    until the next push, drain or destroy, like the pointers behind them)."""

    __slots__ = ("status", "first_batch", "n_batches", "n_records", "n_payload", "n_topk", "_ptrs", "_views")

    def __init__(self, status, raw=None):
        self.status = int(status)
        self.first_batch = int(raw.first_batch) if raw is not None else 0
        self.n_batches = int(raw.n_batches) if raw is not None else 0
        ok = raw is not None and self.status == OK
        self.n_records = int(raw.n_records) if ok else 0
        self.n_payload = int(raw.n_payload) if ok else 0
        self.n_topk = int(raw.n_topk) if ok else 0
        self._ptrs = (raw.records, raw.payload, raw.topk) if ok else None
        self._views = {}

    def _view(self, k):
        if self._ptrs is None:
            return None
        v = self._views.get(k)
        if v is None:
            import torch
            ptr = self._ptrs[k]
            nbytes = (self.n_records * 48, self.n_payload * 4, self.n_topk * 8)[k]
            if not ptr or nbytes == 0:
                v = torch.zeros(0, dtype=torch.uint8, device="cuda")
            else:
                v = torch.as_tensor(_DevView(ptr, nbytes), device="cuda")
            if k == 1:
                v = v.view(torch.int32)
            self._views[k] = v
        return v

    @property
    def records(self):
        return self._view(0)

    @property
    def payload(self):
        return self._view(1)

    @property
    def topk(self):
        return self._view(2)

    def host(self):
        """(records as RECORD_DTYPE, payload int32, topk as PAIR_DTYPE) numpy copies."""
        rec = self.records.cpu().numpy().view(RECORD_DTYPE) if self.records is not None else \
            np.zeros(0, RECORD_DTYPE)
        pay = self.payload.cpu().numpy() if self.payload is not None else np.zeros(0, np.int32)
        tk = self.topk.cpu().numpy().view(PAIR_DTYPE) if self.topk is not None else \
            np.zeros(0, PAIR_DTYPE)
        return rec, pay, tk


class Aggregator:
    """Owning wrapper around one alto_agg handle on the current CUDA device."""

    def __init__(self, depth, payload_op, score_op, topk_k=None, *, max_batch_fragments,
                 max_batch_payload, stream=None, use_torch_allocator=True, **caps):
        import torch
        self._torch = torch
        self.depth = depth
        self.has_score = any(s != SCORE_NONE for s in score_op)
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self._alloc = _TorchAllocator(torch.cuda.current_device()) if use_torch_allocator else None
        self.cfg = make_config(depth, payload_op, score_op, topk_k,
                               max_batch_fragments=max_batch_fragments,
                               max_batch_payload=max_batch_payload, **caps)
        st, self._h = alto_agg_create(self.cfg, self._alloc, self.stream.cuda_stream)
        if st != OK:
            raise RuntimeError(f"alto_agg_create failed: {STATUS_NAMES.get(st, st)}")

    def push(self, tags, off, payload, score=None, n=None) -> int:
        """tags: uint64-valued int64 CUDA tensor (D, n) contiguous; off: int32
        (n+1,) holding u32 offsets; payload: int32; score: float32 or None."""
        b = alto_batch()
        b.n = int(tags.shape[-1]) if n is None else int(n)
        b.depth = self.depth
        b.tags = tags.data_ptr()
        b.payload_off = off.data_ptr()
        b.n_payload = int(payload.numel())
        b.payload = payload.data_ptr() if payload.numel() else None
        b.score = score.data_ptr() if score is not None else None
        return alto_agg_push_batch(self._h, b, self.stream.cuda_stream)

    def drain(self) -> Drain:
        st, d = alto_agg_drain(self._h, self.stream.cuda_stream)
        return Drain(st, d)

    def stats(self):
        return alto_agg_stats(self._h, self.stream.cuda_stream)

    def profile(self, enable) -> int:
        return alto_agg_profile(self._h, enable)

    def profile_read(self):
        return alto_agg_profile_read(self._h)

    def close(self):
        if getattr(self, "_h", None):
            alto_agg_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Router:
    """Owning wrapper around one alto_router handle: routes device batches to
    R replicas and exposes each replica's sub-batch as device tensors."""

    def __init__(self, depth, level, n_replicas, policy, *, max_batch_fragments, max_batch_payload,
                 max_flows=0, with_score=False, stream=None, use_torch_allocator=True):
        import torch
        self._torch = torch
        self.depth, self.level, self.R = depth, level, n_replicas
        self.with_score = bool(with_score)
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self._alloc = _TorchAllocator(torch.cuda.current_device()) if use_torch_allocator else None
        c = alto_router_config()
        c.depth, c.level, c.n_replicas, c.policy = depth, level, n_replicas, policy
        c.max_batch_fragments, c.max_batch_payload, c.max_flows = max_batch_fragments, max_batch_payload, max_flows
        c.with_score = 1 if with_score else 0
        h = ctypes.c_void_p()
        a = self._alloc.struct if self._alloc is not None else None
        st = load_library().alto_router_create(ctypes.byref(c), ctypes.byref(a) if a is not None else None,
                                               ctypes.c_void_p(self.stream.cuda_stream), ctypes.byref(h))
        if st != OK:
            raise RuntimeError(f"alto_router_create failed: {STATUS_NAMES.get(st, st)}")
        self._h = h
        self.routed = alto_routed()

    def route(self, tags, off, payload, score=None, n=None) -> int:
        b = alto_batch()
        b.n = int(tags.shape[-1]) if n is None else int(n)
        b.depth = self.depth
        b.tags = tags.data_ptr()
        b.payload_off = off.data_ptr()
        b.n_payload = int(payload.numel())
        b.payload = payload.data_ptr() if payload.numel() else None
        b.score = score.data_ptr() if score is not None else None
        self._n = b.n
        return load_library().alto_router_route(self._h, ctypes.byref(b), ctypes.c_void_p(self.stream.cuda_stream),
                                                ctypes.byref(self.routed))

    def counts(self):
        """Synchronise; (status, frag_off [R+1], pay_off [R+1]) as numpy int64."""
        import numpy as np
        fo = (ctypes.c_int64 * (self.R + 1))()
        po = (ctypes.c_int64 * (self.R + 1))()
        st = load_library().alto_router_counts(self._h, ctypes.c_void_p(self.stream.cuda_stream), fo, po)
        return st, np.frombuffer(fo, dtype=np.int64).copy(), np.frombuffer(po, dtype=np.int64).copy()

    def outputs(self, frag_off, pay_off):
        """Device views of the last routing: (replica, perm, [per replica (tags
        (D, n_r), payload_off (n_r + 1), payload, score or None)])."""
        torch = self._torch
        r = self.routed
        n = int(frag_off[-1])

        def view(ptr, count, dtype, esize):
            if count == 0 or not ptr:
                return torch.zeros(0, dtype=dtype, device="cuda")
            return torch.as_tensor(_DevView(ptr, count * esize), device="cuda").view(dtype)

        replica = view(r.replica, n, torch.int32, 4)
        perm = view(r.perm, n, torch.int32, 4)
        tags = view(r.tags, self.depth * n, torch.int64, 8)
        poff = view(r.payload_off, n + self.R, torch.int32, 4)
        pay = view(r.payload, int(pay_off[-1]), torch.int32, 4)
        score = view(r.score, n, torch.float32, 4) if self.with_score else None
        parts = []
        for k in range(self.R):
            a, b = int(frag_off[k]), int(frag_off[k + 1])
            nr = b - a
            parts.append((tags[self.depth * a:self.depth * b].view(self.depth, nr),
                          poff[a + k:b + k + 1], pay[int(pay_off[k]):int(pay_off[k + 1])],
                          None if score is None else score[a:b]))
        return replica, perm, parts

    def all_outputs(self, n, n_payload):
        """Device views of the last routing's whole partition, every replica's
        batch in turn: tags (D * n, each replica's block level-major), payload
        offsets (n + R: each replica's n_r + 1), payload (n_payload)."""
        torch = self._torch
        r = self.routed

        def view(ptr, count, dtype, esize):
            if count == 0 or not ptr:
                return torch.zeros(0, dtype=dtype, device="cuda")
            return torch.as_tensor(_DevView(ptr, count * esize), device="cuda").view(dtype)

        return (view(r.tags, self.depth * int(n), torch.int64, 8),
                view(r.payload_off, int(n) + self.R, torch.int32, 4),
                view(r.payload, int(n_payload), torch.int32, 4))

    def release(self, records_ptr, n_records) -> int:
        return load_library().alto_router_release(self._h, ctypes.c_void_p(records_ptr), int(n_records),
                                                  ctypes.c_void_p(self.stream.cuda_stream))

    def close(self):
        if getattr(self, "_h", None):
            load_library().alto_router_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
