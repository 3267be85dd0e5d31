"""Pins of the layer-front oracle (q/k/v projection, RoPE, append) to things other than itself.

The projection is pinned by exact brute force on tiny inputs and by one-hot weights (which
make it an exact selection); the rotation, the head layout of the fused weight, the slot
placement and the counters by the plain append oracle (itself pinned elsewhere), reached
through one-hot weights; the rounding by the C oracle's rounding; the failure cases by the
definition (no slot, counters unchanged, unrotated q).
"""
import math
from fractions import Fraction

import numpy as np
import pytest

from paper_2505_20438_gb300 import workload as wl

pytestmark = pytest.mark.usefixtures("oracle_lib")


def _oracle():
    import oracle
    return oracle


def _front():
    from oracle import front
    return front


def _cache(batch, hq, hkv, d, page, counts, seed, max_slots=64):
    w = wl.Workload(f"front_s{seed}", batch=batch, n_q_heads=hq, n_kv_heads=hkv, head_dim=d,
                    page_slots=page, layers=1, seed=seed, pool_factor=1.5)
    case = wl.make_case(w, num_slots=np.array(counts, np.int32),
                        extra_slots=max_slots - max(counts))
    return case


def test_rounding_matches_c_oracle_including_ties():
    rng = np.random.default_rng(5)
    x = rng.standard_normal(5000) * np.exp(rng.uniform(-40, 40, 5000))
    b = rng.integers(0, 0x7F00, 1000).astype(np.uint16)
    lo = _front().bf16_bits_to_f64(b)
    hi = _front().bf16_bits_to_f64(b + 1)
    x = np.concatenate([x, (lo + hi) / 2, -(lo + hi) / 2, [0.0, -0.0, 2.0 ** -134, 3e-39]])
    assert np.array_equal(_front().f64_to_bf16_bits(x), _oracle().f64_to_bf16(x))


def test_projection_is_exact_brute_force():
    """Every entry against the exact rational sum of the products (tiny sizes)."""
    w = wl.front_workload(2, hidden=48, n_q_heads=2, n_kv_heads=1, head_dim=8, seed=1)
    x, W = wl.front_inputs(w)
    y = _front().project(x, W)
    xf = _front().bf16_bits_to_f64(x)
    Wf = _front().bf16_bits_to_f64(W)
    for b in range(w.batch):
        for o in range(w.out_rows):
            exact = sum(Fraction(float(Wf[o, k])) * Fraction(float(xf[b, k]))
                        for k in range(w.hidden))
            assert abs(Fraction(float(y[b, o])) - exact) <= Fraction(1, 2 ** 40) * (
                sum(abs(Fraction(float(Wf[o, k])) * Fraction(float(xf[b, k])))
                    for k in range(w.hidden)) + Fraction(1, 2 ** 100))


def test_rope_matches_c_oracle_and_is_a_relative_rotation():
    rng = wl.rng_for(3, 0)
    d = 64
    a = wl.normal_bf16(rng, (d,))
    b = wl.normal_bf16(rng, (d,))
    for p in (0, 1, 17, 4095, 262143):
        ref = _oracle().rope_f64(a, p)
        got = _front().rope_values(_front().bf16_bits_to_f64(a), p)
        # theta = p * base^(-2i/d): a last-bit difference between two pow implementations
        # grows with p, so the bar does too
        assert np.allclose(got, ref, rtol=0, atol=4e-16 * (p + 1) * np.abs(got).max())
    af, bf = _front().bf16_bits_to_f64(a), _front().bf16_bits_to_f64(b)
    assert np.array_equal(_front().rope_values(af, 0), af)         # position 0 is identity
    r = _front().rope_values(af, 1234)
    assert np.allclose(r[:32] ** 2 + r[32:] ** 2, af[:32] ** 2 + af[32:] ** 2, rtol=1e-13)
    # q.k depends only on the difference of the positions
    dot = [float(_front().rope_values(af, p + 7) @ _front().rope_values(bf, p)) for p in
           (0, 100, 5000)]
    assert max(dot) - min(dot) < 1e-11


@pytest.mark.parametrize("pos_mode,explicit", [(0, False), (1, False), (0, True)])
def test_one_hot_weights_reduce_to_the_append_oracle(pos_mode, explicit):
    """With one-hot rows the projection selects input entries exactly, so the front must equal
    the plain append of the selected bf16 values, bit for bit: keys rotated, values copied,
    q rotated, metadata and counters."""
    oracle = _oracle()
    B, hq, hkv, d, H = 3, 8, 2, 64, 96
    case = _cache(B, hq, hkv, d, 16, (15, 16, 40), seed=4)
    rng = wl.rng_for(4, 11)
    cols = rng.integers(0, H, (hq + 2 * hkv) * d)
    W = np.zeros(((hq + 2 * hkv) * d, H), np.uint16)
    W[np.arange(W.shape[0]), cols] = 0x3F80                    # 1.0
    a = oracle.OracleCache.from_case(case)
    b = oracle.OracleCache.from_case(case)
    for step in range(3):                                      # crosses a page edge
        x = wl.normal_bf16(rng, (B, H))
        ntok = wl.ntok_capped_geometric(rng, (B,))
        pos = rng.integers(0, 300000, B).astype(np.int32) if explicit else None
        sel = x[:, cols]                                       # exact projection
        q = np.ascontiguousarray(sel[:, : hq * d].reshape(B, hq, d))
        k = sel[:, hq * d: (hq + hkv) * d].reshape(B, hkv, d)
        v = sel[:, (hq + hkv) * d:].reshape(B, hkv, d)
        assert a.append(k, v, ntok, q_inout=q, pos=pos, pos_mode=pos_mode) == 0
        st, q_rot, _ = _front().qkv_append(b, x, W, ntok, pos=pos, pos_mode=pos_mode)
        assert st == 0
        assert np.array_equal(q_rot, q)
    assert np.array_equal(a.k_pool, b.k_pool) and np.array_equal(a.v_pool, b.v_pool)
    assert np.array_equal(a.slot_pos, b.slot_pos) and np.array_equal(a.slot_ntok, b.slot_ntok)
    assert np.array_equal(a.num_slots, b.num_slots)
    assert np.array_equal(a.num_tokens, b.num_tokens)


def test_dense_front_rounds_once():
    """General weights: each stored value is the projection (rotated for q, k) rounded once,
    so it lies within half a bf16 ulp of the fp64 value, and values are the plain projection."""
    oracle = _oracle()
    w = wl.front_workload(2, hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64, seed=6)
    x, W = wl.front_inputs(w)
    case = _cache(2, 4, 2, 64, 16, (5, 33), seed=6)
    c = oracle.OracleCache.from_case(case)
    n0 = c.num_slots.copy()
    st, q_rot, y = _front().qkv_append(c, x, W, np.array([2, 1], np.int32))
    assert st == 0
    front = _front()
    for b in range(2):
        n = int(n0[b])
        page, row = case.page_table[b, n // 16], n % 16
        kexact = front.rope_values(y[b, 4 * 64: 6 * 64].reshape(2, 64), n)
        vexact = y[b, 6 * 64:].reshape(2, 64)
        for got, exact in ((c.k_pool[page, :, row], kexact), (c.v_pool[page, :, row], vexact),
                           (q_rot[b], front.rope_values(y[b, :4 * 64].reshape(4, 64), n))):
            g = front.bf16_bits_to_f64(got)
            ulp = np.ldexp(1.0, np.frexp(np.abs(exact))[1] - 8)
            assert np.all(np.abs(g - exact) <= ulp / 2)
    assert list(c.num_slots) == [int(n0[0]) + 1, int(n0[1]) + 1]
    assert list(c.num_tokens) == [int(case.slot_ntok[0].sum()) + 2, int(case.slot_ntok[1].sum()) + 1]


def test_failed_sequences_are_left_alone():
    oracle = _oracle()
    w = wl.front_workload(3, hidden=128, n_q_heads=4, n_kv_heads=2, head_dim=64, seed=7)
    x, W = wl.front_inputs(w)
    case = _cache(3, 4, 2, 64, 16, (3, 8, 8), seed=7, max_slots=8)   # sequences 1, 2 full
    c = oracle.OracleCache.from_case(case)
    k0, v0, n0, t0 = c.k_pool.copy(), c.v_pool.copy(), c.num_slots.copy(), c.num_tokens.copy()
    st, q_rot, y = _front().qkv_append(c, x, W, np.array([0, 1, 1], np.int32))  # seq 0: ntok 0
    assert st != 0
    assert np.array_equal(c.k_pool, k0) and np.array_equal(c.v_pool, v0)
    assert np.array_equal(c.num_slots, n0) and np.array_equal(c.num_tokens, t0)
    for b in range(3):   # unrotated projection
        assert np.array_equal(q_rot[b], _front().f64_to_bf16_bits(y[b, :256].reshape(4, 64)))


def test_front_then_attention_equals_attention_over_the_logical_list():
    """The appended slot is the last element of the logical list the attention oracle reads."""
    oracle = _oracle()
    w = wl.front_workload(2, hidden=128, n_q_heads=8, n_kv_heads=2, head_dim=64, seed=8)
    x, W = wl.front_inputs(w)
    case = _cache(2, 8, 2, 64, 16, (31, 2), seed=8)
    c = oracle.OracleCache.from_case(case)
    st, q_rot, y = _front().qkv_append(c, x, W, np.array([1, 3], np.int32))
    assert st == 0
    out = c.decode_attn(q_rot)
    for b in range(2):
        L = int(c.num_slots[b])
        for g in range(2):
            kl, vl = c.gather(b, g)
            assert kl.shape[0] == L
            kexact = _front().rope_values(y[b, (8 + g) * 64: (9 + g) * 64], L - 1)
            assert np.array_equal(_front().f64_to_bf16_bits(kl[-1]), _front().f64_to_bf16_bits(kexact))
            for h in range(4 * g, 4 * g + 4):
                qf = _front().bf16_bits_to_f64(q_rot[b, h])
                s = kl @ qf / math.sqrt(64)
                p = np.exp(s - s.max())
                assert np.allclose(out[b, h], (p / p.sum()) @ vl, atol=1e-12)
