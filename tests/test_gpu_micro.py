"""GPU: the micro-step attention (ham_micro_step) against the oracle and against ham_decode_step.

The micro-step decoder's cache holds its context entries and the micro-tokens of the current
macro-step (at most 16 slots).  Every stored bit (keys rotated in fp64, values, metadata,
counters) and the rotated queries are exact; the attention output meets the decode parity bar
in bf16 and a tight bar in fp32 (the kernel's dot products, softmax and sums are fp32 over at
most 16 entries, so its error is a few fp32 roundings).
"""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import assert_parity, dev_bf16, dev_i32, gpu_cache, host_bits, small_case

pytestmark = pytest.mark.gpu

F32_MAX_ABS = 2e-5      # fp32 output: a few fp32 roundings of values of size ~1
F32_MEAN_ABS = 2e-6


def _export(kv, layer=0):
    k, v, pos, ntok = ham.ham_kv_export(kv, layer)
    return host_bits(k), host_bits(v), pos.cpu().numpy(), ntok.cpu().numpy()


def _step(kv, oc, q, k_new, v_new, ntok, f32, pos=None, pos_mode=ham.HAM_POS_SLOT):
    import torch
    B, Hq, d = q.shape
    q_ref = q.copy()
    st = oc.append(k_new, v_new, ntok, q_inout=q_ref, pos=pos, pos_mode=pos_mode)
    ref = oc.decode_attn(q_ref)
    out = torch.full((B, Hq, d), float("nan"), dtype=torch.float32 if f32 else torch.bfloat16,
                     device="cuda")
    q_rot = torch.full((B, Hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    ham.ham_micro_step(kv, 0, dev_bf16(q), dev_bf16(k_new), dev_bf16(v_new),
                       None if pos is None else dev_i32(pos), dev_i32(ntok), out, q_rot=q_rot)
    torch.cuda.synchronize()
    return st, ref, q_ref, out.float().cpu().numpy().astype(np.float64), host_bits(q_rot)


@pytest.mark.parametrize("hq,hkv,d,counts,cap", [
    (32, 8, 64, (4, 4, 4, 4, 4, 4, 4, 4), 8),      # Llama-3.2-1B heads, 4 context entries
    (32, 8, 128, (0, 5, 11), 16),                  # an empty sequence; up to a full chunk
    (8, 8, 64, (3, 1, 7, 2), 12),                  # group 1
    (16, 2, 128, (6, 9), 14),                      # group 8
])
@pytest.mark.parametrize("f32", [False, True])
def test_micro_step_matches_oracle(hq, hkv, d, counts, cap, f32):
    case = small_case(batch=len(counts), hq=hq, hkv=hkv, d=d, page=16, counts=counts,
                      seed=hq + d + cap, extra_slots=cap - max(counts))
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    rng = wl.rng_for(hq + d, 5)
    B = len(counts)
    for step in range(cap - max(counts)):            # micro-steps until the cache is full
        q = wl.normal_bf16(rng, (B, hq, d))
        k_new = wl.normal_bf16(rng, (B, hkv, d))
        v_new = wl.normal_bf16(rng, (B, hkv, d))
        ntok = np.ones(B, np.int32)
        st, ref, q_ref, got, q_rot = _step(kv, oc, q, k_new, v_new, ntok, f32)
        assert st == 0
        assert np.array_equal(q_rot, q_ref), f"step {step}: rotated queries"
        if f32:
            assert_parity(got, ref, F32_MAX_ABS, F32_MEAN_ABS, what=f"step {step} (fp32)")
        else:
            assert_parity(got, ref, what=f"step {step}")
    k, v, p, n = _export(kv)
    assert np.array_equal(k, oc.k_pool) and np.array_equal(v, oc.v_pool)
    assert np.array_equal(p, oc.slot_pos) and np.array_equal(n, oc.slot_ntok)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_first_entry_of_an_empty_cache_is_its_value():
    """One slot: the softmax weight is 1 and the output is the new value (fp32 exact)."""
    import torch
    case = small_case(batch=2, hq=8, hkv=2, d=64, page=16, counts=(0, 0), seed=3, extra_slots=4)
    kv = gpu_cache(case)
    out = torch.empty((2, 8, 64), dtype=torch.float32, device="cuda")
    ham.ham_micro_step(kv, 0, dev_bf16(case.q), dev_bf16(case.k_new), dev_bf16(case.v_new), None,
                       dev_i32(case.ntok_new), out)
    got = out.cpu().numpy()
    vals = wl.bf16_bits_to_f32(case.v_new)                  # [B][Hkv][d]
    for h in range(8):
        assert np.array_equal(got[:, h], vals[:, h // 4])


@pytest.mark.parametrize("pos_mode,explicit", [(ham.HAM_POS_TOKEN, False), (ham.HAM_POS_SLOT, True)])
def test_micro_step_positions(pos_mode, explicit):
    case = small_case(batch=3, hq=32, hkv=8, d=64, page=16, counts=(4, 4, 2), seed=6,
                      extra_slots=4)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case, pos_mode=pos_mode)
    rng = wl.rng_for(6, 9)
    for step in range(3):
        q = wl.normal_bf16(rng, (3, 32, 64))
        k_new = wl.normal_bf16(rng, (3, 8, 64))
        v_new = wl.normal_bf16(rng, (3, 8, 64))
        ntok = wl.ntok_capped_geometric(rng, (3,))
        pos = rng.integers(0, 300000, 3).astype(np.int32) if explicit else None
        st, ref, q_ref, got, q_rot = _step(kv, oc, q, k_new, v_new, ntok, False, pos=pos,
                                           pos_mode=pos_mode)
        assert st == 0 and np.array_equal(q_rot, q_ref)
        assert_parity(got, ref, what=f"step {step}")
    k, v, p, n = _export(kv)
    assert np.array_equal(k, oc.k_pool) and np.array_equal(p, oc.slot_pos)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)


def test_micro_step_equals_decode_step():
    """Same inputs through both entry points: identical cache bits and rotated queries, outputs
    within the parity bar of each other."""
    import torch
    case = small_case(batch=8, hq=32, hkv=8, d=64, page=16, counts=(4,) * 8, seed=12,
                      extra_slots=4)
    kv_a, kv_b = gpu_cache(case), gpu_cache(case)
    rng = wl.rng_for(12, 1)
    for step in range(4):
        q = dev_bf16(wl.normal_bf16(rng, (8, 32, 64)))
        k_new = dev_bf16(wl.normal_bf16(rng, (8, 8, 64)))
        v_new = dev_bf16(wl.normal_bf16(rng, (8, 8, 64)))
        ntok = dev_i32(wl.ntok_capped_geometric(rng, (8,)))
        outs, rots = [], []
        for kv, fn in ((kv_a, ham.ham_micro_step), (kv_b, ham.ham_decode_step)):
            out = torch.empty((8, 32, 64), dtype=torch.float32, device="cuda")
            q_rot = torch.empty((8, 32, 64), dtype=torch.bfloat16, device="cuda")
            fn(kv, 0, q, k_new, v_new, None, ntok, out, q_rot=q_rot)
            outs.append(out.cpu().numpy().astype(np.float64))
            rots.append(host_bits(q_rot))
        assert np.array_equal(rots[0], rots[1])
        assert_parity(outs[0], outs[1], what=f"step {step}")
    ea, eb = _export(kv_a), _export(kv_b)
    for x, y in zip(ea, eb):
        assert np.array_equal(x, y)


def test_micro_step_failures():
    """A full sequence and ntok < 1: no slot, the error word set, attention with the unrotated
    query over the old slots; the other sequences proceed."""
    case = small_case(batch=3, hq=8, hkv=2, d=64, page=16, counts=(16, 3, 5), seed=13,
                      extra_slots=0)                        # capacity 16: sequence 0 is full
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    q = case.q.copy()
    ntok = np.array([1, 0, 2], np.int32)
    st, ref, q_ref, got, q_rot = _step(kv, oc, q, case.k_new, case.v_new, ntok, True)
    assert st != 0
    assert ham.ham_kv_status(kv) in (ham.HAM_DEVERR_CAPACITY, ham.HAM_DEVERR_NTOK)
    assert_parity(got, ref, F32_MAX_ABS, F32_MEAN_ABS, what="failed sequences")
    slots, _ = ham.ham_slot_lengths(kv)
    assert list(slots) == [16, 3, 6]
    k, v, p, n = _export(kv)
    assert np.array_equal(k, oc.k_pool) and np.array_equal(v, oc.v_pool)


def test_micro_step_rejects_large_caches():
    import torch
    case = small_case(batch=2, hq=8, hkv=2, d=64, page=16, counts=(3, 4), seed=14,
                      extra_slots=14)                       # 18 slots per sequence
    kv = gpu_cache(case)
    out = torch.empty((2, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ham.HamError) as e:
        ham.ham_micro_step(kv, 0, dev_bf16(case.q), dev_bf16(case.k_new), dev_bf16(case.v_new),
                           None, dev_i32(case.ntok_new), out)
    assert e.value.status == ham.HAM_EUNSUPPORTED
