"""FP8 (e4m3) smashed-KV rows: encoding, per-row power-of-two scale, decoding; plain numpy.

TEST INFRASTRUCTURE ONLY: the tests, `__graft_entry__.smoke()` and the CPU-baseline leg of
`bench.py` may use it; the product path never imports this package.

Why: decoding reads every stored key and value each step and is bound by memory bandwidth
(Sec. 2.3; Sec. 3.7: the KV cache is what HAMburger shrinks), so storing a slot's rows in 8 bits
instead of 16 roughly halves the bytes a step reads.  The paper itself keeps the base model's
precision; this is a storage format of this library, specified here so that the CUDA path can be
checked against it bit for bit.

Format (readings Q1-Q4 of the paper's silence on any 8-bit cache format, taken here):
  Q1  e4m3 codes (1 sign bit, 4 exponent bits with bias 7, 3 mantissa bits; no infinities;
      S.1111.111 is NaN; largest finite 448 = 1.75 * 2^8; subnormals are multiples of 2^-9);
  Q2  one scale per stored row (one slot of one KV head), a power of two 2^e, e an int8: a row is
      appended once and never rewritten, so a page-wide scale would have to be fixed before the
      page's later rows are known, and rescaling would change rows already stored;
  Q3  e is chosen from the row's largest magnitude a = m 2^E (0.5 <= m < 1) as e = E - 8, so
      that a 2^-e lies in [128, 256): below 448, with every element scaled exactly (a power of
      two) and rounded once, to nearest with ties to even, onto the e4m3 grid; a row of zeros
      gets e = 0 and zero codes.  e is then clamped to [-124, 119] so that every decoded value
      is a finite bf16 value: the finest step of the e4m3 grid is 2^-9 and that of bf16 is 2^-133
      (its smallest subnormal), hence e >= -124; a row maximum just below 2^128 (E = 128) would
      round up to 256 * 2^120 = 2^128, past the largest bf16 value, hence e <= 119 (such a row's
      largest elements then saturate at 448 * 2^119).  Rows must be finite;
  Q4  the key is rotated first (the bf16 row ham_kv_append would store), then encoded; the value
      row is encoded as given.  A decoded element code * 2^e has at most 4 significant bits and
      is therefore exact in bf16, so attention over an FP8 pool is attention over those exact
      bf16 values.
"""
from __future__ import annotations

import numpy as np

E4M3_MAX = 448.0
E4M3_NAN_CODES = (0x7F, 0xFF)


def e4m3_value(code) -> np.ndarray:
    """Exact value of e4m3 codes (uint8), NaN for the two NaN codes (reading Q1: the OCP e4m3
    "fn" format; the paper keeps the base model's precision and fixes no 8-bit format)."""
    c = np.asarray(code, dtype=np.int64)
    sign = np.where(c & 0x80, -1.0, 1.0)
    exp = (c >> 3) & 0xF
    man = (c & 0x7).astype(np.float64)
    normal = np.ldexp(1.0 + man / 8.0, (exp - 7).astype(np.int32))
    sub = np.ldexp(man / 8.0, -6)
    v = sign * np.where(exp == 0, sub, normal)
    return np.where((c & 0x7F) == 0x7F, np.nan, v)


def _grid() -> np.ndarray:
    """The non-negative finite e4m3 values in increasing order (codes 0x00 .. 0x7E)."""
    return e4m3_value(np.arange(0x7F))


def e4m3_encode(x) -> np.ndarray:
    """Round finite values to the nearest e4m3 value, ties to the even code, magnitudes above 448
    saturating to 448, the sign kept (a negative value that rounds to zero gives -0, 0x80);
    returns uint8 codes.  Brute force over the 127 non-negative values: the
    grid is increasing in the code, so the even-code tie rule is the even-mantissa rule."""
    x = np.asarray(x, dtype=np.float64)
    a = np.minimum(np.abs(x), E4M3_MAX)
    grid = _grid()
    hi = np.searchsorted(grid, a, side="left")            # first grid value >= a
    hi = np.minimum(hi, len(grid) - 1)
    lo = np.maximum(hi - 1, 0)
    d_lo, d_hi = a - grid[lo], grid[hi] - a
    pick_hi = (d_hi < d_lo) | ((d_hi == d_lo) & (hi % 2 == 0))
    code = np.where(grid[hi] == a, hi, np.where(pick_hi, hi, lo)).astype(np.int64)
    code = np.where(np.signbit(x), code | 0x80, code)    # the sign survives, zero included
    return code.astype(np.uint8)


E_MIN, E_MAX = -124, 119   # Q3: the decoded values code * 2^e stay finite and exact in bf16


def row_exponent(values) -> int:
    """Scale exponent e of one row (Q3): e = E - 8 for the largest magnitude m 2^E, clamped to
    [E_MIN, E_MAX]; 0 if all zero."""
    a = float(np.max(np.abs(np.asarray(values, dtype=np.float64)))) if np.size(values) else 0.0
    if a == 0.0:
        return 0
    _, E = np.frexp(a)
    return int(min(max(int(E) - 8, E_MIN), E_MAX))


def encode_row(values):
    """(codes uint8 [n], e int) of one row of exact values (bf16 values given as float): one
    power-of-two scale per stored row (Q2, Q3), each element rounded once (Q1)."""
    v = np.asarray(values, dtype=np.float64)
    e = row_exponent(v)
    return e4m3_encode(np.ldexp(v, -e)), e


def decode_row(codes, e) -> np.ndarray:
    """Exact values code * 2^e of one row (Q4: what attention over an FP8 pool reads)."""
    return np.ldexp(e4m3_value(codes), int(e))


def encode_rows(rows):
    """Every row of an [..., d] array: (codes [..., d] uint8, e [...] int8); encode_row applied
    to all rows at once (the same steps, vectorised over the rows)."""
    r = np.asarray(rows, dtype=np.float64)
    a = np.max(np.abs(r), axis=-1) if r.shape[-1] else np.zeros(r.shape[:-1])
    _, E = np.frexp(a)
    e = np.where(a == 0.0, 0, np.clip(E.astype(np.int64) - 8, E_MIN, E_MAX))
    codes = e4m3_encode(np.ldexp(r, -e[..., None].astype(np.int32)))
    return codes, e.astype(np.int8)


def decode_rows(codes, es) -> np.ndarray:
    c = np.asarray(codes)
    return np.ldexp(e4m3_value(c), np.asarray(es, dtype=np.int32)[..., None])


def decoded_bf16_bits(codes, es) -> np.ndarray:
    """bf16 bit patterns of the decoded rows (exact, Q4): attention over an FP8 pool is the
    attention oracle run on these bits."""
    v = decode_rows(codes, es)
    b = v.astype(np.float32).view(np.uint32) >> np.uint32(16)   # exact values: truncation is exact
    return b.astype(np.uint16)
