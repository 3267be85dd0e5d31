"""ctypes wrapper of the plain C fp64 oracle (oracle.c).

TEST INFRASTRUCTURE ONLY: the tests, `__graft_entry__.smoke()` and the CPU-baseline leg
of `bench.py` use it.  The product path (the CUDA library and its binding) never imports
this package.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None

EINVAL, EPAGE, ECAPACITY = -1, -2, -3
POS_SLOT, POS_TOKEN = 0, 1


def build(force: bool = False) -> str:
    """Compile oracle.c with gcc (OpenMP when available, no FMA contraction)."""
    if not force and os.path.exists(_LIB_PATH) and \
            os.path.getmtime(_LIB_PATH) >= max(os.path.getmtime(_SRC),
                                               os.path.getmtime(os.path.join(_HERE, "oracle.h"))):
        return _LIB_PATH
    base = ["gcc", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-std=c11",
            "-o", _LIB_PATH + ".tmp", _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True, text=True)
    os.replace(_LIB_PATH + ".tmp", _LIB_PATH)
    return _LIB_PATH


class _Cache(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("page_slots", ctypes.c_int32), ("max_pages", ctypes.c_int32),
        ("pool_pages", ctypes.c_int64), ("max_slots", ctypes.c_int64),
        ("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p),
        ("slot_pos", ctypes.c_void_p), ("slot_ntok", ctypes.c_void_p),
        ("page_table", ctypes.c_void_p), ("num_slots", ctypes.c_void_p),
        ("num_tokens", ctypes.c_void_p),
    ]


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB_PATH)
        P = ctypes.POINTER(_Cache)
        vp, i32, i64, f64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        sig = {
            "oracle_bf16_to_f64": (f64, [ctypes.c_uint16]),
            "oracle_f64_to_bf16": (ctypes.c_uint16, [f64]),
            "oracle_rope_f64": (None, [vp, vp, i32, i64, f64]),
            "oracle_rope_bf16": (None, [vp, vp, i32, i32, i64, f64]),
            "oracle_gather": (ctypes.c_int, [P, i32, i32, vp, vp]),
            "oracle_fill": (ctypes.c_int, [P, vp, vp, vp, vp, vp, i32]),
            "oracle_decode_attn": (ctypes.c_int, [P, vp, vp, i32]),
            "oracle_attn_weights": (ctypes.c_int, [P, vp, i32, i32, vp]),
            "oracle_append": (ctypes.c_int, [P, vp, vp, vp, vp, vp, i32, f64]),
            "oracle_prefill": (ctypes.c_int, [P, vp, vp, vp, vp, vp, vp, i32, f64, vp, vp, i32]),
            "oracle_max_threads": (ctypes.c_int, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype, fn.argtypes = res, args
        _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data


class OracleError(RuntimeError):
    pass


def _check(rc, what):
    if rc != 0:
        raise OracleError(f"{what} failed with code {rc}")


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    f = np.vectorize(lib().oracle_bf16_to_f64, otypes=[np.float64])
    return f(np.asarray(bits, dtype=np.uint16))


def f64_to_bf16(x: np.ndarray) -> np.ndarray:
    f = np.vectorize(lib().oracle_f64_to_bf16, otypes=[np.uint16])
    return f(np.asarray(x, dtype=np.float64))


def rope_f64(x_bits: np.ndarray, pos: int, base: float = 10000.0) -> np.ndarray:
    x = np.ascontiguousarray(x_bits, dtype=np.uint16)
    y = np.empty(x.shape, dtype=np.float64)
    lib().oracle_rope_f64(_ptr(x), _ptr(y), x.shape[-1], int(pos), float(base))
    return y


def rope_bf16(x_bits: np.ndarray, pos: int, base: float = 10000.0) -> np.ndarray:
    x = np.ascontiguousarray(x_bits, dtype=np.uint16)
    y = np.empty_like(x)
    d = x.shape[-1]
    lib().oracle_rope_bf16(_ptr(x), _ptr(y), x.size // d, d, int(pos), float(base))
    return y


def max_threads() -> int:
    return int(lib().oracle_max_threads())


class OracleCache:
    """Host copy of one layer of the paged smashed-KV cache, driven by the C oracle."""

    def __init__(self, batch, n_q_heads, n_kv_heads, head_dim, page_slots, page_table,
                 pool_pages, max_slots):
        self.page_table = np.ascontiguousarray(page_table, dtype=np.int32)
        assert self.page_table.shape[0] == batch
        self.shape = dict(batch=batch, n_q_heads=n_q_heads, n_kv_heads=n_kv_heads,
                          head_dim=head_dim, page_slots=page_slots)
        self.k_pool = np.zeros((pool_pages, n_kv_heads, page_slots, head_dim), np.uint16)
        self.v_pool = np.zeros_like(self.k_pool)
        self.slot_pos = np.zeros((pool_pages, page_slots), np.int32)
        self.slot_ntok = np.zeros((pool_pages, page_slots), np.int32)
        self.num_slots = np.zeros(batch, np.int32)
        self.num_tokens = np.zeros(batch, np.int64)
        self._c = _Cache(batch, n_q_heads, n_kv_heads, head_dim, page_slots,
                         self.page_table.shape[1], pool_pages, max_slots,
                         _ptr(self.k_pool), _ptr(self.v_pool), _ptr(self.slot_pos),
                         _ptr(self.slot_ntok), _ptr(self.page_table), _ptr(self.num_slots),
                         _ptr(self.num_tokens))

    @classmethod
    def from_case(cls, case, fill: bool = True):
        w = case.w
        c = cls(w.batch, w.n_q_heads, w.n_kv_heads, w.head_dim, w.page_slots,
                case.page_table, case.pool_pages, case.max_slots)
        if fill:
            c.fill(case.k, case.v, case.slot_pos, case.slot_ntok, case.num_slots)
        return c

    def fill(self, k_log, v_log, pos, ntok, counts):
        k_log = np.ascontiguousarray(k_log, np.uint16)
        v_log = np.ascontiguousarray(v_log, np.uint16)
        pos = np.ascontiguousarray(pos, np.int32)
        ntok = np.ascontiguousarray(ntok, np.int32)
        counts = np.ascontiguousarray(counts, np.int32)
        _check(lib().oracle_fill(ctypes.byref(self._c), _ptr(k_log), _ptr(v_log), _ptr(pos),
                                 _ptr(ntok), _ptr(counts), k_log.shape[1]), "oracle_fill")

    def gather(self, b, g):
        L = int(self.num_slots[b])
        d = self.shape["head_dim"]
        k = np.empty((L, d), np.float64)
        v = np.empty((L, d), np.float64)
        _check(lib().oracle_gather(ctypes.byref(self._c), b, g, _ptr(k), _ptr(v)),
               "oracle_gather")
        return k, v

    def decode_attn(self, q_bits, n_threads: int = 0):
        q = np.ascontiguousarray(q_bits, np.uint16)
        s = self.shape
        assert q.shape == (s["batch"], s["n_q_heads"], s["head_dim"])
        out = np.empty(q.shape, np.float64)
        _check(lib().oracle_decode_attn(ctypes.byref(self._c), _ptr(q), _ptr(out),
                                        int(n_threads)), "oracle_decode_attn")
        return out

    def attn_weights(self, q_bits, b, h):
        q = np.ascontiguousarray(q_bits, np.uint16)
        w = np.empty(max(int(self.num_slots[b]), 1), np.float64)
        _check(lib().oracle_attn_weights(ctypes.byref(self._c), _ptr(q), b, h, _ptr(w)),
               "oracle_attn_weights")
        return w[: int(self.num_slots[b])]

    def append(self, k_new, v_new, ntok, q_inout=None, pos=None, pos_mode=POS_SLOT,
               rope_base=10000.0):
        k_new = np.ascontiguousarray(k_new, np.uint16)
        v_new = np.ascontiguousarray(v_new, np.uint16)
        ntok = np.ascontiguousarray(ntok, np.int32)
        if pos is not None:
            pos = np.ascontiguousarray(pos, np.int32)
        if q_inout is not None:
            assert q_inout.dtype == np.uint16 and q_inout.flags.c_contiguous
        return lib().oracle_append(ctypes.byref(self._c), _ptr(k_new), _ptr(v_new),
                                   _ptr(q_inout), _ptr(pos), _ptr(ntok), int(pos_mode),
                                   float(rope_base))

    def prefill(self, q, k_new, v_new, offsets, ntok=None, pos=None, pos_mode=POS_SLOT,
                rope_base=10000.0, want=None, n_threads: int = 0):
        """Chunked prefill (oracle_prefill).  q [T][n_q_heads][d] bf16 bits is rotated in place
        (must be C-contiguous uint16); want: optional bool [T], the rows to attend (the others
        are appended, their out rows 0).  Returns (status, out [T][n_q_heads][d] fp64)."""
        assert q.dtype == np.uint16 and q.flags.c_contiguous
        k_new = np.ascontiguousarray(k_new, np.uint16)
        v_new = np.ascontiguousarray(v_new, np.uint16)
        offsets = np.ascontiguousarray(offsets, np.int32)
        T = int(offsets[-1])
        ntok = np.ones(T, np.int32) if ntok is None else np.ascontiguousarray(ntok, np.int32)
        if pos is not None:
            pos = np.ascontiguousarray(pos, np.int32)
        if want is not None:
            want = np.ascontiguousarray(want, np.uint8)
        out = np.empty(q.shape, np.float64)
        rc = lib().oracle_prefill(ctypes.byref(self._c), _ptr(q), _ptr(k_new), _ptr(v_new),
                                  _ptr(offsets), _ptr(pos), _ptr(ntok), int(pos_mode),
                                  float(rope_base), _ptr(out), _ptr(want), int(n_threads))
        return rc, out
