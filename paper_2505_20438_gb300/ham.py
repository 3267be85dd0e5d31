"""Python binding of libham.so (include/ham.h): the same names, argument marshalling only.

Tensors are torch tensors in device memory (the library never sees torch types: it gets
data pointers and the raw cudaStream_t).  Every step of the decode path runs in the
library's CUDA kernels; there is no fallback.  If libham.so is missing or cannot load, every
call raises.

Shapes are checked here because the C ABI receives bare pointers and cannot.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libham.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "ham.h")

HAM_OK, HAM_EINVAL, HAM_ENOMEM, HAM_ECAPACITY, HAM_ECUDA, HAM_EDEVICE, HAM_EUNSUPPORTED = range(7)
STATUS_NAMES = {0: "HAM_OK", 1: "HAM_EINVAL", 2: "HAM_ENOMEM", 3: "HAM_ECAPACITY",
                4: "HAM_ECUDA", 5: "HAM_EDEVICE", 6: "HAM_EUNSUPPORTED"}
(HAM_DEVERR_NONE, HAM_DEVERR_CAPACITY, HAM_DEVERR_NTOK, HAM_DEVERR_PAGE, HAM_DEVERR_SLOTS,
 HAM_DEVERR_TIMEOUT) = range(6)
HAM_POS_SLOT, HAM_POS_TOKEN = 0, 1
HAM_DTYPE_BF16, HAM_DTYPE_F32 = 0, 1
HAM_KV_BF16, HAM_KV_E4M3 = 0, 1


class HamError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class ham_config(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_int32), ("batch", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_slots", ctypes.c_int32),
                ("max_slots_per_seq", ctypes.c_int32), ("pos_mode", ctypes.c_int32),
                ("pool_pages", ctypes.c_int64), ("rope_base", ctypes.c_double),
                ("page_seed", ctypes.c_uint64), ("kv_dtype", ctypes.c_int32)]


class ham_attn_args(ctypes.Structure):
    _fields_ = [("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p),
                ("page_table", ctypes.c_void_p), ("num_slots", ctypes.c_void_p),
                ("q", ctypes.c_void_p), ("out", ctypes.c_void_p), ("err", ctypes.c_void_p),
                ("pool_pages", ctypes.c_int64), ("batch", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_slots", ctypes.c_int32),
                ("max_pages", ctypes.c_int32), ("max_slots", ctypes.c_int32),
                ("ctas", ctypes.c_int32), ("out_dtype", ctypes.c_int32)]


class ham_kv_info(ctypes.Structure):
    _fields_ = [("cfg", ham_config), ("max_pages_per_seq", ctypes.c_int32),
                ("attn_ctas", ctypes.c_int32), ("num_sms", ctypes.c_int32),
                ("device", ctypes.c_int32), ("pool_bytes", ctypes.c_int64),
                ("scratch_bytes", ctypes.c_int64)]


class ham_embed_config(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("max_batch", ctypes.c_int32), ("max_patch", ctypes.c_int32)]


_vp, _i32, _i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
_SIGNATURES = {
    "ham_embedder_alloc": [ctypes.POINTER(ham_embed_config), _vp, _vp, _vp, _vp, _vp,
                           ctypes.POINTER(_vp)],
    "ham_embedder_free": [_vp],
    "ham_embed": [_vp, _vp, _vp, _i32, _i32, _vp, _vp],
    "ham_embedder_status": [_vp, _vp, ctypes.POINTER(_i32)],
    "ham_embedder_set_vocab": [_vp, _vp, _i32],
    "ham_embed_tokens": [_vp, _vp, _vp, _i32, _i32, _vp, _vp],
    "ham_kv_alloc": [ctypes.POINTER(ham_config), ctypes.POINTER(_vp)],
    "ham_kv_free": [_vp],
    "ham_kv_append": [_vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp],
    "ham_decode_attn": [_vp, _i32, _vp, _vp, _vp],
    "ham_slot_lengths": [_vp, _vp, _vp, _vp],
    "ham_kv_get_info": [_vp, ctypes.POINTER(ham_kv_info)],
    "ham_decode_attn_ex": [_vp, _i32, _vp, _vp, _i32, _vp],
    "ham_kv_layer_lengths": [_vp, _i32, _vp, _vp, _vp],
    "ham_kv_status": [_vp, _vp, ctypes.POINTER(_i32)],
    "ham_kv_set_page_table": [_vp, _vp],
    "ham_kv_get_page_table": [_vp, _vp],
    "ham_kv_fill": [_vp, _i32, _vp, _vp, _vp, _vp, _vp, _i32, _vp],
    "ham_kv_export": [_vp, _i32, _vp, _vp, _vp, _vp, _vp],
    "ham_kv_export_scales": [_vp, _i32, _vp, _vp],
    "ham_kv_reset": [_vp, _vp],
    "ham_kv_set_lengths": [_vp, _i32, _vp, _vp, _vp],
    "ham_kv_set_attn_ctas": [_vp, _i32],
    "ham_kv_set_wait_limit_ns": [_vp, ctypes.c_uint64],
    "ham_split_plan": [_i32, _i32, _vp, _i32, _vp, _vp, _vp],
    "ham_decode_attn_noalloc": [ctypes.c_void_p, _vp],
    "ham_decode_step": [_vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _vp],
    "ham_prefill": [_vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _vp, _i32, _vp],
    "ham_qkv_append": [_vp, _i32, _vp, _vp, _i32, _vp, _vp, _vp, _vp],
    "ham_micro_step": [_vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _vp],
}
_lib = None


def lib() -> ctypes.CDLL:
    """Load libham.so (built by __graft_entry__.build() / paper_2505_20438_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        for name, args in _SIGNATURES.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        L.ham_last_error.argtypes = []
        L.ham_last_error.restype = ctypes.c_char_p
        _lib = L
    return _lib


def header_functions(path: str = HEADER):
    """Names of the functions include/ham.h declares."""
    text = open(path).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(ham_\w+)\s*\(", text, re.M)))


def _check(rc: int):
    if rc != HAM_OK:
        raise HamError(rc, lib().ham_last_error().decode(errors="replace"))


def ham_last_error() -> str:
    return lib().ham_last_error().decode(errors="replace")


# ---------------------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------------------

def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _dev(t, shape, dtype_name, what, nullable=False):
    if t is None:
        if nullable:
            return None
        raise ValueError(f"{what} is required")
    import torch
    dtype = {"bf16": torch.bfloat16, "f32": torch.float32, "i32": torch.int32,
             "i64": torch.int64}[dtype_name]
    if not t.is_cuda:
        raise ValueError(f"{what} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{what} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{what} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    return t.data_ptr()


class KV:
    """Owning handle of one paged smashed-KV cache (ham_kv*)."""

    def __init__(self, ptr: int):
        self.ptr = ptr
        self.info = ham_kv_get_info(self)
        c = self.info.cfg
        self.layers, self.batch = c.layers, c.batch
        self.n_q_heads, self.n_kv_heads, self.head_dim = c.n_q_heads, c.n_kv_heads, c.head_dim
        self.page_slots, self.max_slots = c.page_slots, c.max_slots_per_seq
        self.pool_pages = c.pool_pages
        self.kv_dtype = c.kv_dtype
        self.max_pages = self.info.max_pages_per_seq

    @property
    def _as_parameter_(self):
        return ctypes.c_void_p(self.ptr)

    def close(self):
        if self.ptr:
            ham_kv_free(self)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ---------------------------------------------------------------------------------------
# the C ABI, one function each
# ---------------------------------------------------------------------------------------

def ham_kv_alloc(layers, batch, n_q_heads, n_kv_heads, head_dim, page_slots,
                 max_slots_per_seq, pos_mode=HAM_POS_SLOT, pool_pages=0, rope_base=10000.0,
                 page_seed=0, kv_dtype=0) -> KV:
    cfg = ham_config(layers, batch, n_q_heads, n_kv_heads, head_dim, page_slots,
                     max_slots_per_seq, pos_mode, pool_pages, rope_base, page_seed, kv_dtype)
    out = ctypes.c_void_p()
    _check(lib().ham_kv_alloc(ctypes.byref(cfg), ctypes.byref(out)))
    return KV(out.value)


def ham_kv_free(kv: KV):
    ptr, kv.ptr = kv.ptr, 0
    _check(lib().ham_kv_free(ctypes.c_void_p(ptr)))


def ham_kv_get_info(kv: KV) -> ham_kv_info:
    info = ham_kv_info()
    _check(lib().ham_kv_get_info(ctypes.c_void_p(kv.ptr), ctypes.byref(info)))
    return info


def ham_kv_append(kv: KV, layer, q_inout, k_new, v_new, pos, ntok, stream=None):
    B, Hq, Hkv, d = kv.batch, kv.n_q_heads, kv.n_kv_heads, kv.head_dim
    _check(lib().ham_kv_append(
        kv, layer, _dev(q_inout, (B, Hq, d), "bf16", "q_inout", nullable=True),
        _dev(k_new, (B, Hkv, d), "bf16", "k_new"), _dev(v_new, (B, Hkv, d), "bf16", "v_new"),
        _dev(pos, (B,), "i32", "pos", nullable=True), _dev(ntok, (B,), "i32", "ntok"),
        _stream_ptr(stream)))


def ham_decode_attn(kv: KV, layer, q, out, stream=None):
    B, Hq, d = kv.batch, kv.n_q_heads, kv.head_dim
    _check(lib().ham_decode_attn(kv, layer, _dev(q, (B, Hq, d), "bf16", "q"),
                                 _dev(out, (B, Hq, d), "bf16", "out"), _stream_ptr(stream)))


def ham_decode_attn_ex(kv: KV, layer, q, out, stream=None):
    """Output dtype follows `out` (bf16 or fp32)."""
    import torch
    B, Hq, d = kv.batch, kv.n_q_heads, kv.head_dim
    f32 = out is not None and out.dtype == torch.float32
    _check(lib().ham_decode_attn_ex(
        kv, layer, _dev(q, (B, Hq, d), "bf16", "q"),
        _dev(out, (B, Hq, d), "f32" if f32 else "bf16", "out"),
        HAM_DTYPE_F32 if f32 else HAM_DTYPE_BF16, _stream_ptr(stream)))


def ham_decode_step(kv: KV, layer, q, k_new, v_new, pos, ntok, out, q_rot=None, stream=None):
    """Fused append + attention of one layer.  q is the unrotated query (not written);
    q_rot (optional) receives RoPE(q).  Output dtype follows `out` (bf16 or fp32)."""
    import torch
    B, Hq, Hkv, d = kv.batch, kv.n_q_heads, kv.n_kv_heads, kv.head_dim
    f32 = out is not None and out.dtype == torch.float32
    _check(lib().ham_decode_step(
        kv, layer, _dev(q, (B, Hq, d), "bf16", "q"),
        _dev(q_rot, (B, Hq, d), "bf16", "q_rot", nullable=True),
        _dev(k_new, (B, Hkv, d), "bf16", "k_new"), _dev(v_new, (B, Hkv, d), "bf16", "v_new"),
        _dev(pos, (B,), "i32", "pos", nullable=True), _dev(ntok, (B,), "i32", "ntok"),
        _dev(out, (B, Hq, d), "f32" if f32 else "bf16", "out"),
        HAM_DTYPE_F32 if f32 else HAM_DTYPE_BF16, _stream_ptr(stream)))


def ham_micro_step(kv: KV, layer, q, k_new, v_new, pos, ntok, out, q_rot=None, stream=None):
    """ham_decode_step for caches of at most 16 slots per sequence (the micro-step decoder's
    local context), in one launch.  Output dtype follows `out` (bf16 or fp32)."""
    import torch
    B, Hq, Hkv, d = kv.batch, kv.n_q_heads, kv.n_kv_heads, kv.head_dim
    f32 = out is not None and out.dtype == torch.float32
    _check(lib().ham_micro_step(
        kv, layer, _dev(q, (B, Hq, d), "bf16", "q"),
        _dev(q_rot, (B, Hq, d), "bf16", "q_rot", nullable=True),
        _dev(k_new, (B, Hkv, d), "bf16", "k_new"), _dev(v_new, (B, Hkv, d), "bf16", "v_new"),
        _dev(pos, (B,), "i32", "pos", nullable=True), _dev(ntok, (B,), "i32", "ntok"),
        _dev(out, (B, Hq, d), "f32" if f32 else "bf16", "out"),
        HAM_DTYPE_F32 if f32 else HAM_DTYPE_BF16, _stream_ptr(stream)))


def ham_prefill(kv: KV, layer, q, k_new, v_new, offsets, out, pos=None, ntok=None,
                stream=None):
    """Chunked prefill of one layer: sequence b's new rows are offsets[b] .. offsets[b+1]-1 of
    q [T][n_q_heads][d] (rotated in place), k_new, v_new [T][n_kv_heads][d]; each becomes one
    slot and attends causally.  pos, ntok: optional int32 [T].  Output dtype follows `out`."""
    import torch
    Hq, Hkv, d = kv.n_q_heads, kv.n_kv_heads, kv.head_dim
    T = q.shape[0] if q is not None and q.dim() == 3 else 0
    f32 = out is not None and out.dtype == torch.float32
    _check(lib().ham_prefill(
        kv, layer, _dev(q, (T, Hq, d), "bf16", "q"), _dev(k_new, (T, Hkv, d), "bf16", "k_new"),
        _dev(v_new, (T, Hkv, d), "bf16", "v_new"),
        _dev(offsets, (kv.batch + 1,), "i32", "offsets"),
        _dev(pos, (T,), "i32", "pos", nullable=True), _dev(ntok, (T,), "i32", "ntok", nullable=True),
        T, _dev(out, (T, Hq, d), "f32" if f32 else "bf16", "out"),
        HAM_DTYPE_F32 if f32 else HAM_DTYPE_BF16, _stream_ptr(stream)))


def ham_qkv_append(kv: KV, layer, x, w_qkv, ntok, q_rot, pos=None, stream=None):
    """Layer front of one macro-step: project x [B][H] with the fused weight
    w_qkv [(Hq + 2 Hkv) d][H], rotate q and k at the new slot's position, append k and v, write
    the rotated queries to q_rot [B][Hq][d]."""
    B, Hq, Hkv, d = kv.batch, kv.n_q_heads, kv.n_kv_heads, kv.head_dim
    H = x.shape[1] if x is not None and x.dim() == 2 else 0
    _check(lib().ham_qkv_append(
        kv, layer, _dev(x, (B, H), "bf16", "x"),
        _dev(w_qkv, ((Hq + 2 * Hkv) * d, H), "bf16", "w_qkv"), H,
        _dev(pos, (B,), "i32", "pos", nullable=True), _dev(ntok, (B,), "i32", "ntok"),
        _dev(q_rot, (B, Hq, d), "bf16", "q_rot"), _stream_ptr(stream)))


def ham_slot_lengths(kv: KV, stream=None):
    slots = np.zeros(kv.batch, np.int32)
    tokens = np.zeros(kv.batch, np.int64)
    _check(lib().ham_slot_lengths(kv, slots.ctypes.data, tokens.ctypes.data, _stream_ptr(stream)))
    return slots, tokens


def ham_kv_layer_lengths(kv: KV, layer, stream=None):
    slots = np.zeros(kv.batch, np.int32)
    tokens = np.zeros(kv.batch, np.int64)
    _check(lib().ham_kv_layer_lengths(kv, layer, slots.ctypes.data, tokens.ctypes.data,
                                      _stream_ptr(stream)))
    return slots, tokens


def ham_kv_status(kv: KV, stream=None) -> int:
    """Device error code (HAM_DEVERR_*), read and cleared; does not raise on HAM_EDEVICE."""
    code = ctypes.c_int32(0)
    rc = lib().ham_kv_status(kv, _stream_ptr(stream), ctypes.byref(code))
    if rc not in (HAM_OK, HAM_EDEVICE):
        _check(rc)
    return code.value


def ham_kv_set_page_table(kv: KV, page_table: np.ndarray):
    pt = np.ascontiguousarray(page_table, np.int32)
    if pt.shape != (kv.batch, kv.max_pages):
        raise ValueError(f"page table must have shape {(kv.batch, kv.max_pages)}")
    _check(lib().ham_kv_set_page_table(kv, pt.ctypes.data))


def ham_kv_get_page_table(kv: KV) -> np.ndarray:
    pt = np.zeros((kv.batch, kv.max_pages), np.int32)
    _check(lib().ham_kv_get_page_table(kv, pt.ctypes.data))
    return pt


def ham_kv_fill(kv: KV, layer, k_log, v_log, counts, pos=None, ntok=None, stream=None):
    B, Hkv, d = kv.batch, kv.n_kv_heads, kv.head_dim
    lmax = int(k_log.shape[1]) if k_log is not None else 0
    _check(lib().ham_kv_fill(
        kv, layer, _dev(k_log, (B, lmax, Hkv, d), "bf16", "k_log", nullable=lmax == 0),
        _dev(v_log, (B, lmax, Hkv, d), "bf16", "v_log", nullable=lmax == 0),
        _dev(pos, (B, lmax), "i32", "pos", nullable=True),
        _dev(ntok, (B, lmax), "i32", "ntok", nullable=True),
        _dev(counts, (B,), "i32", "counts"), lmax, _stream_ptr(stream)))


def ham_kv_export(kv: KV, layer, stream=None):
    """Copy one layer's raw pools and slot metadata into new device tensors (FP8 pools: uint8
    codes, K [pages][Hkv][P][d] and V [pages][Hkv][d][P])."""
    import torch
    shape = (kv.pool_pages, kv.n_kv_heads, kv.page_slots, kv.head_dim)
    if kv.kv_dtype == HAM_KV_E4M3:
        k = torch.empty(shape, dtype=torch.uint8, device="cuda")
        v = torch.empty((kv.pool_pages, kv.n_kv_heads, kv.head_dim, kv.page_slots),
                        dtype=torch.uint8, device="cuda")
    else:
        k = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
        v = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    pos = torch.empty((kv.pool_pages, kv.page_slots), dtype=torch.int32, device="cuda")
    ntok = torch.empty_like(pos)
    _check(lib().ham_kv_export(kv, layer, k.data_ptr(), v.data_ptr(), pos.data_ptr(),
                               ntok.data_ptr(), _stream_ptr(stream)))
    return k, v, pos, ntok


def ham_kv_export_scales(kv: KV, layer, stream=None):
    """One layer's exponent array of an FP8 cache: int8 [pages][Hkv][P/16][2][16]."""
    import torch
    e = torch.empty((kv.pool_pages, kv.n_kv_heads, kv.page_slots // 16, 2, 16),
                    dtype=torch.int8, device="cuda")
    _check(lib().ham_kv_export_scales(kv, layer, e.data_ptr(), _stream_ptr(stream)))
    return e


def ham_kv_set_lengths(kv: KV, layer, num_slots, num_tokens=None, stream=None):
    B = kv.batch
    _check(lib().ham_kv_set_lengths(
        kv, layer, _dev(num_slots, (B,), "i32", "num_slots"),
        _dev(num_tokens, (B,), "i64", "num_tokens", nullable=True), _stream_ptr(stream)))


def ham_kv_reset(kv: KV, stream=None):
    _check(lib().ham_kv_reset(kv, _stream_ptr(stream)))


def ham_kv_set_attn_ctas(kv: KV, ctas: int):
    _check(lib().ham_kv_set_attn_ctas(kv, int(ctas)))
    kv.info = ham_kv_get_info(kv)


def ham_kv_set_wait_limit_ns(kv: KV, ns: int):
    """Limit of the attention and prefill kernels' data waits (0: the default 2 s); a testing aid
    for the failure path."""
    _check(lib().ham_kv_set_wait_limit_ns(kv, int(ns)))


def ham_split_plan(num_slots, n_kv_heads: int, ctas: int):
    """Host evaluation of the attention split plan: (cta_begin, seg_first_cta, seg_last_cta)."""
    ns = np.ascontiguousarray(num_slots, np.int32)
    B = ns.shape[0]
    begin = np.zeros(ctas + 1, np.int64)
    first = np.zeros(B * n_kv_heads, np.int32)
    last = np.zeros(B * n_kv_heads, np.int32)
    _check(lib().ham_split_plan(B, n_kv_heads, ns.ctypes.data, ctas, begin.ctypes.data,
                                first.ctypes.data, last.ctypes.data))
    return begin, first, last


def ham_decode_attn_noalloc(k_pool, v_pool, page_table, num_slots, q, out, max_slots,
                            ctas=0, err=None, stream=None):
    """Decode attention over caller-owned buffers; the library allocates nothing (its
    scratch is a static device array shared by all calls)."""
    import torch
    P, Hkv, S, d = (int(x) for x in k_pool.shape)
    B, Hq = int(q.shape[0]), int(q.shape[1])
    max_pages = int(page_table.shape[1])
    f32 = out.dtype == torch.float32
    args = ham_attn_args(
        _dev(k_pool, (P, Hkv, S, d), "bf16", "k_pool"), _dev(v_pool, (P, Hkv, S, d), "bf16", "v_pool"),
        _dev(page_table, (B, max_pages), "i32", "page_table"), _dev(num_slots, (B,), "i32", "num_slots"),
        _dev(q, (B, Hq, d), "bf16", "q"), _dev(out, (B, Hq, d), "f32" if f32 else "bf16", "out"),
        _dev(err, (1,), "i32", "err", nullable=True), P, B, Hq, Hkv, d, S, max_pages,
        int(max_slots), int(ctas), HAM_DTYPE_F32 if f32 else HAM_DTYPE_BF16)
    _check(lib().ham_decode_attn_noalloc(ctypes.byref(args), _stream_ptr(stream)))


# ---------------------------------------------------------------------------------------
# compositional embedder
# ---------------------------------------------------------------------------------------

class Embedder:
    """Owning handle of one compositional embedder (ham_embedder*)."""

    def __init__(self, ptr: int, cfg: ham_embed_config):
        self.ptr = ptr
        self.hidden, self.n_heads = cfg.hidden, cfg.n_heads
        self.max_batch, self.max_patch = cfg.max_batch, cfg.max_patch

    @property
    def _as_parameter_(self):
        return ctypes.c_void_p(self.ptr)

    def close(self):
        if self.ptr:
            ham_embedder_free(self)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def ham_embedder_alloc(hidden, n_heads, max_batch, max_patch, wq, wk, wv, wo, pos) -> Embedder:
    """Weights: CUDA bf16 tensors, wq/wk/wv/wo [hidden][hidden] ([out][in]), pos
    [max_patch][hidden].  The handle keeps its own copies."""
    cfg = ham_embed_config(hidden, n_heads, max_batch, max_patch)
    H = hidden
    out = ctypes.c_void_p()
    _check(lib().ham_embedder_alloc(
        ctypes.byref(cfg), _dev(wq, (H, H), "bf16", "wq"), _dev(wk, (H, H), "bf16", "wk"),
        _dev(wv, (H, H), "bf16", "wv"), _dev(wo, (H, H), "bf16", "wo"),
        _dev(pos, (max_patch, H), "bf16", "pos"), ctypes.byref(out)))
    return Embedder(out.value, cfg)


def ham_embedder_free(e: Embedder):
    ptr, e.ptr = e.ptr, 0
    _check(lib().ham_embedder_free(ctypes.c_void_p(ptr)))


def ham_embed(e: Embedder, x, offsets, out, stream=None):
    """x: CUDA bf16 [total_tokens][hidden]; offsets: CUDA int32 [batch + 1]; out: CUDA bf16
    [batch][hidden]."""
    B = out.shape[0] if out is not None else 0
    T = x.shape[0] if x is not None else 0
    _check(lib().ham_embed(e, _dev(x, (T, e.hidden), "bf16", "x"),
                           _dev(offsets, (B + 1,), "i32", "offsets"), B, T,
                           _dev(out, (B, e.hidden), "bf16", "out"), _stream_ptr(stream)))


def ham_embedder_set_vocab(e: Embedder, table):
    """table: CUDA bf16 [vocab][hidden], the token embeddings (copied; the projections of every
    entry are tabulated on the handle, synchronously)."""
    V = table.shape[0] if table is not None and table.dim() == 2 else 0
    _check(lib().ham_embedder_set_vocab(e, _dev(table, (V, e.hidden), "bf16", "table"), V))


def ham_embed_tokens(e: Embedder, ids, offsets, out, stream=None):
    """ids: CUDA int32 [total_tokens] (token ids); offsets: CUDA int32 [batch + 1]; out: CUDA
    bf16 [batch][hidden]."""
    B = out.shape[0] if out is not None else 0
    T = ids.shape[0] if ids is not None else 0
    _check(lib().ham_embed_tokens(e, _dev(ids, (T,), "i32", "ids"),
                                  _dev(offsets, (B + 1,), "i32", "offsets"), B, T,
                                  _dev(out, (B, e.hidden), "bf16", "out"), _stream_ptr(stream)))


def ham_embedder_status(e: Embedder, stream=None) -> int:
    """Device error code (HAM_DEVERR_*), read and cleared; does not raise on HAM_EDEVICE."""
    code = ctypes.c_int32(0)
    rc = lib().ham_embedder_status(e, _stream_ptr(stream), ctypes.byref(code))
    if rc not in (HAM_OK, HAM_EDEVICE):
        _check(rc)
    return code.value
