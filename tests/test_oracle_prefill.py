"""Pins of the chunked-prefill oracle (prompt ingestion: one slot per prompt token, causal
attention of the chunk over the cache and itself) against things other than itself: torch's
scaled-dot-product attention with a causal / offset mask, the complex-exponential form of
RoPE, the sequence of single-slot decode steps it must equal, closed forms and invariants."""
import math

import numpy as np
import pytest
import torch

from paper_2505_20438_gb300 import workload as wl

pytestmark = pytest.mark.usefixtures("oracle_lib")


def _o():
    import oracle
    return oracle


def _w(batch=2, hq=8, hkv=2, d=64, page=16, seed=0, scale=1.0):
    return wl.Workload("pin_prefill", batch=batch, n_q_heads=hq, n_kv_heads=hkv, head_dim=d,
                       page_slots=page, layers=1, value_scale=scale, seed=seed, pool_factor=1.5)


def _run(case, q=None, pos_mode=0, pos=None, want=None, headroom=0):
    """Oracle prefill of `case` on a cache filled with case.base; returns (cache, q, status, out)."""
    o = _o()
    oc = o.OracleCache.from_case(case.base)
    qq = np.ascontiguousarray(case.q if q is None else q).copy()
    rc, out = oc.prefill(qq, case.k_new, case.v_new, case.offsets, ntok=case.ntok, pos=pos,
                         pos_mode=pos_mode, want=want)
    return oc, qq, rc, out


def _f64(bits):
    return wl.bf16_bits_to_f32(bits).astype(np.float64)


def _rope_complex(x_bits, pos, base=10000.0):
    x = _f64(x_bits)
    d = x.shape[-1]
    half = d // 2
    w = base ** (-(np.arange(half) * 2.0) / d)
    z = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * pos * w)
    return np.concatenate([z.real, z.imag], axis=-1)


def _masked_sdpa(oc, case, q_rot, b):
    """torch SDPA of sequence b's rotated rows over its stored slots with the mask
    slot <= L + j (the causal attention over the cache and the chunk)."""
    w = case.w
    L, n, a = int(case.base.num_slots[b]), int(case.rows[b]), int(case.offsets[b])
    ks, vs = zip(*(oc.gather(b, g) for g in range(w.n_kv_heads)))
    k = torch.from_numpy(np.stack(ks))[None]          # [1][Hkv][L+n][d]
    v = torch.from_numpy(np.stack(vs))[None]
    q = torch.from_numpy(_f64(q_rot[a:a + n])).permute(1, 0, 2)[None]   # [1][Hq][n][d]
    mask = torch.arange(L + n)[None, :] <= (L + torch.arange(n))[:, None]
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=mask,
                                                           enable_gqa=True)
    return ref[0].permute(1, 0, 2).numpy()             # [n][Hq][d]


def test_fresh_prompt_matches_causal_sdpa():
    case = wl.make_prefill_case(_w(seed=1), [40, 23], cached=np.array([0, 0], np.int32))
    oc, q_rot, rc, out = _run(case)
    assert rc == 0
    for b in range(2):
        a, n = int(case.offsets[b]), int(case.rows[b])
        ref = _masked_sdpa(oc, case, q_rot, b)
        np.testing.assert_allclose(out[a:a + n], ref, rtol=1e-10, atol=1e-12)


def test_chunk_over_cached_slots_matches_offset_mask():
    case = wl.make_prefill_case(_w(batch=3, seed=2), [20, 33, 5],
                                cached=np.array([37, 0, 80], np.int32))
    oc, q_rot, rc, out = _run(case)
    assert rc == 0
    assert list(oc.num_slots) == [57, 33, 85]
    for b in range(3):
        a, n = int(case.offsets[b]), int(case.rows[b])
        np.testing.assert_allclose(out[a:a + n], _masked_sdpa(oc, case, q_rot, b),
                                   rtol=1e-10, atol=1e-12)


def test_rotations_match_the_complex_form():
    """q rows and stored keys: the complex-exponential RoPE at the slot index, to bf16
    rounding (half an ulp, which is at most 2^-9 of the value)."""
    case = wl.make_prefill_case(_w(seed=3), [9, 14], cached=np.array([5, 30], np.int32))
    oc, q_rot, rc, _ = _run(case)
    assert rc == 0
    for b in range(2):
        L, a = int(case.base.num_slots[b]), int(case.offsets[b])
        k_all, _ = oc.gather(b, 1)
        for j in range(int(case.rows[b])):
            for got, x in ((_f64(q_rot[a + j]), case.q[a + j]), (k_all[L + j], case.k_new[a + j, 1])):
                ref = _rope_complex(x, L + j)
                assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0 ** -8 + 1e-30)


def test_equals_sequential_single_slot_decode_steps():
    """The chunk is the same as appending its rows one at a time and decoding after each."""
    o = _o()
    case = wl.make_prefill_case(_w(batch=1, seed=4), [25], cached=np.array([19], np.int32))
    _, _, rc, out = _run(case)
    assert rc == 0
    seq = o.OracleCache.from_case(case.base)
    for j in range(25):
        q = case.q[j][None].copy()
        assert seq.append(case.k_new[j][None], case.v_new[j][None], case.ntok[j:j + 1],
                          q_inout=q) == 0
        np.testing.assert_array_equal(seq.decode_attn(q)[0], out[j])


def test_split_chunks_give_the_same_result():
    o = _o()
    case = wl.make_prefill_case(_w(batch=2, seed=5), [30, 12], cached=np.array([3, 40], np.int32))
    oc, q_rot, rc, out = _run(case)
    assert rc == 0
    two = o.OracleCache.from_case(case.base)
    split = [0, 17]  # rows of the first call per sequence; the rest in the second
    first = np.array([min(s, int(r)) for s, r in zip(split, case.rows)], np.int32)
    outs = np.zeros_like(out)
    qq = case.q.copy()
    for part in (0, 1):
        sel = [np.arange(case.offsets[b], case.offsets[b] + first[b]) if part == 0 else
               np.arange(case.offsets[b] + first[b], case.offsets[b + 1]) for b in range(2)]
        idx = np.concatenate(sel).astype(np.int64)
        offs = np.concatenate([[0], np.cumsum([len(s) for s in sel])]).astype(np.int32)
        qp = np.ascontiguousarray(qq[idx])
        rc2, op = two.prefill(qp, case.k_new[idx], case.v_new[idx], offs, ntok=case.ntok[idx])
        assert rc2 == 0
        outs[idx] = op
        qq[idx] = qp
    np.testing.assert_array_equal(outs, out)
    np.testing.assert_array_equal(qq, q_rot)
    np.testing.assert_array_equal(two.k_pool, oc.k_pool)
    np.testing.assert_array_equal(two.v_pool, oc.v_pool)


def test_token_positions_follow_the_running_count():
    o = _o()
    rng = wl.rng_for(6, 1)
    ntok = rng.integers(1, 5, 18).astype(np.int32)
    case = wl.make_prefill_case(_w(batch=1, seed=6), [18], cached=np.array([7], np.int32),
                                ntok=ntok)
    t0 = int(case.base.slot_ntok[0, :7].sum())
    oc, q_rot, rc, _ = _run(case, pos_mode=o.POS_TOKEN)
    assert rc == 0
    want = t0 + np.concatenate([[0], np.cumsum(ntok)[:-1]])
    pt = case.base.page_table[0]
    got = [oc.slot_pos[pt[(7 + j) // 16], (7 + j) % 16] for j in range(18)]
    assert list(got) == list(want)
    assert int(oc.num_tokens[0]) == t0 + int(ntok.sum())
    for j in range(18):
        np.testing.assert_array_equal(q_rot[j], o.rope_bf16(case.q[j], int(want[j])))


def test_first_row_of_an_empty_sequence_attends_only_itself():
    case = wl.make_prefill_case(_w(seed=7), [4, 1], cached=np.array([0, 0], np.int32))
    _, _, rc, out = _run(case)
    assert rc == 0
    G = case.w.group
    for b in range(2):
        a = int(case.offsets[b])
        for h in range(case.w.n_q_heads):
            np.testing.assert_array_equal(out[a, h], _f64(case.v_new[a, h // G]))


def test_rows_that_do_not_fit_leave_the_sequence_untouched():
    o = _o()
    case = wl.make_prefill_case(_w(seed=8), [6, 9], cached=np.array([10, 20], np.int32))
    # capacity = 20 + 9: shrink it so that sequence 1 no longer fits
    case.base.max_slots = 25
    oc, q_rot, rc, out = _run(case)
    assert rc == o.ECAPACITY
    assert list(oc.num_slots) == [16, 20]
    a = int(case.offsets[1])
    assert np.all(out[a:] == 0)
    np.testing.assert_array_equal(q_rot[a:], case.q[a:])
    ok = wl.make_prefill_case(_w(seed=8), [6, 0], cached=np.array([10, 20], np.int32))
    _, _, rc0, out0 = _run(ok)
    assert rc0 == 0
    np.testing.assert_array_equal(out[:6], out0[:6])
    bad = wl.make_prefill_case(_w(seed=8), [6, 9], cached=np.array([10, 20], np.int32),
                               ntok=np.array([1] * 6 + [1, 0] + [1] * 7, np.int32))
    oc2, _, rc2, out2 = _run(bad)
    assert rc2 == o.EINVAL and list(oc2.num_slots) == [16, 20] and np.all(out2[6:] == 0)


def test_capacity_boundary_is_exact():
    # a chunk that fills the sequence to its capacity is stored; one row more is refused whole
    o = _o()
    for cap, fits in ((29, True), (28, False)):
        case = wl.make_prefill_case(_w(seed=8), [6, 9], cached=np.array([10, 20], np.int32))
        case.base.max_slots = cap
        oc, _, rc, out = _run(case)
        if fits:
            assert rc == 0 and list(oc.num_slots) == [16, 29]
        else:
            assert rc == o.ECAPACITY and list(oc.num_slots) == [16, 20]
            assert np.all(out[int(case.offsets[1]):] == 0)


def test_row_mask_only_skips_attention():
    case = wl.make_prefill_case(_w(seed=9), [12, 7], cached=np.array([4, 0], np.int32))
    oc_all, q_all, _, out_all = _run(case)
    want = np.zeros(19, bool)
    want[[0, 5, 11, 12, 18]] = True
    oc, q, rc, out = _run(case, want=want)
    assert rc == 0
    np.testing.assert_array_equal(out[want], out_all[want])
    assert np.all(out[~want] == 0)
    np.testing.assert_array_equal(oc.k_pool, oc_all.k_pool)
    np.testing.assert_array_equal(q, q_all)


def test_scale_is_one_over_sqrt_head_dim():
    """A zero cached slot and one new slot at position 0 (RoPE is the identity there) with
    k = e_0, v = e_1, q = 3 e_0: the new slot's weight is w / (1 + w), w = exp(3 / sqrt(d))."""
    o = _o()
    d = 64
    case = wl.make_prefill_case(_w(batch=1, hq=1, hkv=1, d=d, seed=10), [1],
                                cached=np.array([1], np.int32))
    oc = o.OracleCache.from_case(case.base)
    oc.k_pool[:] = 0
    oc.v_pool[:] = 0

    def bits(x):
        return int(wl.f32_to_bf16_bits(np.array([x], np.float32))[0])

    k1 = np.zeros((1, 1, d), np.uint16)
    v1 = np.zeros((1, 1, d), np.uint16)
    q = np.zeros((1, 1, d), np.uint16)
    k1[0, 0, 0], v1[0, 0, 1], q[0, 0, 0] = bits(1.0), bits(1.0), bits(3.0)
    rc, out = oc.prefill(q, k1, v1, np.array([0, 1], np.int32), pos=np.array([0], np.int32))
    assert rc == 0
    w1 = math.exp(3.0 / math.sqrt(d))
    assert abs(out[0, 0, 1] - w1 / (1.0 + w1)) < 1e-12
    assert np.all(out[0, 0, [0] + list(range(2, d))] == 0)
