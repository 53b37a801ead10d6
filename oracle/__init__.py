"""CPU oracle for nested-ancestry re-aggregation -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg may import this package.  The CUDA library never does, and the two share
no code.  ``alto_oracle.cpp`` holds the definition (see its header for the
paper passages it follows); this module compiles it with the host compiler and
wraps it with ctypes, with an API shaped like the library's
(create / push / drain / destroy) but operating on host arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

from .route import HASH, LEAST_LOADED, RouterOracle, splitmix64_mix  # noqa: F401
from .split_text import split_pieces, split_text  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "alto_oracle.cpp")
_LIB = os.path.join(_HERE, "liboracle.so")

# status codes of the oracle (same numeric values as the public interface)
OK, EINVAL, ENOMEM, ENOSPC, EDUP, ELAST, EINCONSIST, ECLOSED = 0, -1, -2, -3, -4, -5, -6, -7

RECORD_DTYPE = np.dtype([
    ("completion_seq", "<u8"), ("payload_off", "<u8"), ("payload_len", "<u8"),
    ("topk_off", "<u8"), ("parent_id", "<u4"), ("n_children", "<u4"),
    ("level", "u1"), ("ops", "u1"), ("topk_n", "<u2"), ("score", "<f4"),
])
PAIR_DTYPE = np.dtype([("child_index", "<u4"), ("score", "<f4")])
assert RECORD_DTYPE.itemsize == 48 and PAIR_DTYPE.itemsize == 8


class _Drain(ctypes.Structure):
    _fields_ = [
        ("n_records", ctypes.c_int64), ("records", ctypes.c_void_p),
        ("n_payload", ctypes.c_int64), ("payload", ctypes.c_void_p),
        ("n_topk", ctypes.c_int64), ("topk", ctypes.c_void_p),
        ("first_batch", ctypes.c_uint64), ("n_batches", ctypes.c_uint64),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle with the host C++ compiler (plain -O2, one thread)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["g++", "-O2", "-std=c++17", "-shared", "-fPIC", _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.orc_create.restype = ctypes.c_void_p
        lib.orc_create.argtypes = [ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        lib.orc_push.restype = ctypes.c_int
        lib.orc_push.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p,
                                 ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]
        lib.orc_drain.restype = ctypes.c_int
        lib.orc_drain.argtypes = [ctypes.c_void_p, ctypes.POINTER(_Drain)]
        lib.orc_set_stream_release.restype = ctypes.c_int
        lib.orc_set_stream_release.argtypes = [ctypes.c_void_p, ctypes.c_int]
        lib.orc_open_groups.restype = ctypes.c_int64
        lib.orc_open_groups.argtypes = [ctypes.c_void_p]
        lib.orc_destroy.restype = None
        lib.orc_destroy.argtypes = [ctypes.c_void_p]
        _lib = lib
    return _lib


@dataclass
class Drain:
    status: int
    records: np.ndarray   # RECORD_DTYPE
    payload: np.ndarray   # int32
    topk: np.ndarray      # PAIR_DTYPE
    first_batch: int
    n_batches: int


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


class Oracle:
    """Arrival-order reference aggregator over host arrays."""

    def __init__(self, depth, payload_op, score_op, topk_k, stream_release=False):
        lib = _load()
        self.depth = int(depth)
        po = np.asarray(list(payload_op) + [0] * (8 - len(payload_op)), dtype=np.int32)
        so = np.asarray(list(score_op) + [0] * (8 - len(score_op)), dtype=np.int32)
        kk = np.asarray(list(topk_k) + [0] * (8 - len(topk_k)), dtype=np.int32)
        self._h = lib.orc_create(self.depth, _ptr(po), _ptr(so), _ptr(kk))
        if not self._h:
            raise ValueError("invalid aggregation config")
        if stream_release and lib.orc_set_stream_release(self._h, 1) != 0:
            self.close()
            raise ValueError("streaming release needs a CONCAT level")

    @classmethod
    def for_stream(cls, stream, stream_release=False):
        return cls(stream.depth, stream.payload_op, stream.score_op, stream.topk_k, stream_release)

    def push(self, tags, off, payload, score=None, depth=None) -> int:
        tags = np.ascontiguousarray(tags, dtype=np.uint64)
        n = tags.shape[-1] if tags.ndim == 2 else (tags.size // self.depth)
        off = np.ascontiguousarray(off, dtype=np.uint32)
        payload = np.ascontiguousarray(payload, dtype=np.int32)
        if score is not None:
            score = np.ascontiguousarray(score, dtype=np.float32)
        return _load().orc_push(self._h, n, self.depth if depth is None else depth,
                                _ptr(tags), _ptr(off), payload.size, _ptr(payload), _ptr(score))

    def push_batch(self, b: dict) -> int:
        return self.push(b["tags"], b["off"], b["payload"], b["score"])

    def drain(self) -> Drain:
        d = _Drain()
        st = _load().orc_drain(self._h, ctypes.byref(d))

        def grab(ptr, n, dt):
            if n == 0:
                return np.zeros(0, dtype=dt)
            buf = (ctypes.c_char * (n * dt.itemsize)).from_address(ptr)
            return np.frombuffer(bytes(buf), dtype=dt).copy()

        return Drain(st, grab(d.records, d.n_records, RECORD_DTYPE),
                     grab(d.payload, d.n_payload, np.dtype(np.int32)),
                     grab(d.topk, d.n_topk, PAIR_DTYPE), int(d.first_batch), int(d.n_batches))

    def open_groups(self) -> int:
        return int(_load().orc_open_groups(self._h))

    def close(self):
        if getattr(self, "_h", None):
            _load().orc_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def run_stream(stream, drain_every: int = 1, stream_release: bool = False):
    """Push every batch of a generated stream and drain every
    ``drain_every`` batches (and at the end); returns the list of drains."""
    o = Oracle.for_stream(stream, stream_release)
    out = []
    for b in range(stream.n_batches):
        o.push_batch(stream.batch(b))
        if (b + 1) % drain_every == 0 or b == stream.n_batches - 1:
            out.append(o.drain())
    o.close()
    return out
