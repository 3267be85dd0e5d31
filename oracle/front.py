"""Macro-step layer front of HAMburger: q/k/v projection, RoPE and append, plain fp64 numpy.

TEST INFRASTRUCTURE ONLY: the tests, `__graft_entry__.smoke()` and the CPU-baseline leg of
`bench.py` use it; the product path never imports this package.

What it computes.  A macro-step is one forward of the base model (Sec. 3.1), which stores one
key/value set for the whole group of tokens it fused.  Each attention layer of the base model
(Llama-3.2, Sec. 4.1) first projects the layer's normalised input x of width H into queries,
keys and values with bias-free linear maps, turns queries and keys by the rotary embedding at
the macro-step's position (Sec. 3.2: the merged embedding enters at an offset position) and
stores the key and value as the sequence's new slot.  For sequence b:

    y      = W x_b                                    (W = [W_q; W_k; W_v], [out][in])
    q_h    = y[h d : (h+1) d]                          h < Hq
    k_g    = y[(Hq + g) d : ...],  v_g = y[(Hq + Hkv + g) d : ...]
    RoPE at p: pairs (i, i + d/2), theta_i = p * base^(-2i/d),
               (a, c) -> (a cos - c sin, c cos + a sin)
    slot n = num_slots[b]:  K row <- bf16(RoPE(k_g)),  V row <- bf16(v_g),
                            slot_pos = p, slot_ntok = ntok[b];  counters advance
    q_rot[b, h] = bf16(RoPE(q_h))

Readings where the paper leaves details open, taken here:
  F1  the projections are the base model's bias-free q/k/v linear maps, one fused weight with
      the rows of W_q, then W_k, then W_v;
  F2  the rotation acts on the exact projection, and each stored value is rounded once to
      bf16 (nearest, ties to even); no intermediate rounding of q/k before the rotation;
  F3  the position p is pos[b] if given, else the slot index n (slot mode) or the tokens
      already in the sequence (token mode), as for the plain append;
  F4  a sequence whose append cannot happen (token count < 1, no room, a page id outside the
      pool) gets no slot and no counter change; its q_rot row is the unrotated projection.

Weights and inputs are bf16 bit patterns (uint16); products of two bf16 values are exact in
fp64 and the sums are fp64.
"""
from __future__ import annotations

import numpy as np

POS_SLOT, POS_TOKEN = 0, 1
ECAPACITY, EPAGE, EINVAL = -3, -2, -1


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact value of bf16 bit patterns (the upper half of an fp32)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x) -> np.ndarray:
    """Round fp64 values to bf16, nearest with ties to even (finite inputs).

    Exact: with a = m 2^e (0.5 <= m < 1) the bf16 quantum of a is 2^(e-8) (8 significant
    bits; 2^-133 below the normal range), a / quantum is an exact scaling, and its fraction
    decides the rounding."""
    x = np.asarray(x, dtype=np.float64)
    a = np.abs(x)
    _, e = np.frexp(a)
    quantum = np.where(e - 1 < -126, 2.0 ** -133, np.ldexp(1.0, (e - 8).astype(np.int32)))
    q = a / quantum
    lo = np.floor(q)
    rest = q - lo
    up = (rest > 0.5) | ((rest == 0.5) & (np.fmod(lo, 2.0) == 1.0))
    r = (lo + up) * quantum
    bits = (r.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)
    sign = np.where(np.signbit(x), np.uint16(0x8000), np.uint16(0))
    return (bits | sign).astype(np.uint16)


def project(x_bits, w_bits) -> np.ndarray:
    """y[b, o] = sum_k W[o, k] x[b, k] in fp64 (the linear map of F1: the base model's q/k/v
    projections, Sec. 4.1, fused into one weight)."""
    x = bf16_bits_to_f64(x_bits)
    w = bf16_bits_to_f64(w_bits)
    return x @ w.T


def rope_values(y, pos: int, base: float = 10000.0) -> np.ndarray:
    """Rotate-half RoPE of fp64 rows y [..., d] at integer position pos (fp64 throughout): the
    base model's rotary embedding (Sec. 4.1) at the macro-step's offset position (Sec. 3.2)."""
    y = np.asarray(y, dtype=np.float64)
    d = y.shape[-1]
    half = d // 2
    i = np.arange(half, dtype=np.float64)
    theta = float(pos) * np.power(float(base), -(2.0 * i) / float(d))
    c, s = np.cos(theta), np.sin(theta)
    a, b = y[..., :half], y[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def qkv_append(cache, x_bits, w_bits, ntok, pos=None, pos_mode=POS_SLOT, rope_base=10000.0):
    """One layer front of one macro-step on an oracle.OracleCache (its arrays are edited): the
    macro-step's one forward stores one key/value set (Sec. 3.1), projected, rotated at the
    offset position (Sec. 3.2) and appended as the append oracle appends it.

    x_bits [B][H], w_bits [(Hq + 2 Hkv) d][H] bf16 bits; ntok [B]; pos nullable [B].
    Returns (status, q_rot bits [B][Hq][d], y fp64 [B][(Hq + 2 Hkv) d]): status 0, or the
    first failure code of a sequence that was skipped (F4)."""
    s = cache.shape
    B, Hq, Hkv, d, P = s["batch"], s["n_q_heads"], s["n_kv_heads"], s["head_dim"], s["page_slots"]
    y = project(x_bits, w_bits)
    assert y.shape == (B, (Hq + 2 * Hkv) * d)
    q = y[:, : Hq * d].reshape(B, Hq, d)
    k = y[:, Hq * d: (Hq + Hkv) * d].reshape(B, Hkv, d)
    v = y[:, (Hq + Hkv) * d:].reshape(B, Hkv, d)
    q_rot = np.empty((B, Hq, d), np.uint16)
    status = 0
    max_slots = cache._c.max_slots
    pool_pages = cache._c.pool_pages
    for b in range(B):
        n = int(cache.num_slots[b])
        t = int(ntok[b])
        code = 0
        if t < 1:
            code = EINVAL
        elif n < 0 or n >= max_slots:
            code = ECAPACITY
        else:
            page = int(cache.page_table[b, n // P])
            if page < 0 or page >= pool_pages:
                code = EPAGE
        if code:
            status = status or code
            q_rot[b] = f64_to_bf16_bits(q[b])
            continue
        p = int(pos[b]) if pos is not None else (n if pos_mode == POS_SLOT
                                                 else int(cache.num_tokens[b]))
        row = n % P
        cache.k_pool[page, :, row, :] = f64_to_bf16_bits(rope_values(k[b], p, rope_base))
        cache.v_pool[page, :, row, :] = f64_to_bf16_bits(v[b])
        cache.slot_pos[page, row] = p
        cache.slot_ntok[page, row] = t
        cache.num_slots[b] = n + 1
        cache.num_tokens[b] += t
        q_rot[b] = f64_to_bf16_bits(rope_values(q[b], p, rope_base))
    return status, q_rot, y
