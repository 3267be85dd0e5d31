"""GPU: fill, fused RoPE + append and slot bookkeeping are bit-exact against the oracle."""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import dev_bf16, dev_i32, gpu_cache, host_bits, small_case

pytestmark = pytest.mark.gpu


def _export_host(kv, layer=0):
    k, v, pos, ntok = ham.ham_kv_export(kv, layer)
    return host_bits(k), host_bits(v), pos.cpu().numpy(), ntok.cpu().numpy()


@pytest.mark.parametrize("d,page,counts", [(64, 16, (37, 80)), (128, 32, (0, 100, 7)),
                                           (128, 128, (255,))])
def test_fill_is_bit_exact(d, page, counts):
    case = small_case(batch=len(counts), hq=8, hkv=2, d=d, page=page, counts=counts, seed=1)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    k, v, pos, ntok = _export_host(kv)
    assert np.array_equal(k, oc.k_pool) and np.array_equal(v, oc.v_pool)
    assert np.array_equal(pos, oc.slot_pos) and np.array_equal(ntok, oc.slot_ntok)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)


@pytest.mark.parametrize("pos_mode", [ham.HAM_POS_SLOT, ham.HAM_POS_TOKEN])
@pytest.mark.parametrize("d,hq,hkv", [(64, 8, 2), (128, 32, 8), (128, 8, 8)])
def test_append_is_bit_exact(pos_mode, d, hq, hkv):
    case = small_case(batch=3, hq=hq, hkv=hkv, d=d, page=16, counts=(15, 16, 200), seed=2,
                      extra_slots=8)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case, pos_mode=pos_mode)
    q_host = case.q.copy()
    q_dev = dev_bf16(case.q)
    rng = wl.rng_for(2, 50)
    for step in range(3):                      # several macro-steps, crossing a page edge
        k_new = wl.normal_bf16(rng, case.k_new.shape)
        v_new = wl.normal_bf16(rng, case.v_new.shape)
        ntok = wl.ntok_capped_geometric(rng, (case.w.batch,))
        assert oc.append(k_new, v_new, ntok, q_inout=q_host, pos_mode=pos_mode) == 0
        ham.ham_kv_append(kv, 0, q_dev, dev_bf16(k_new), dev_bf16(v_new), None, dev_i32(ntok))
    k, v, pos, ntok_arr = _export_host(kv)
    assert np.array_equal(v, oc.v_pool)
    assert np.array_equal(k, oc.k_pool)                     # RoPE'd keys, bit for bit
    assert np.array_equal(pos, oc.slot_pos) and np.array_equal(ntok_arr, oc.slot_ntok)
    assert np.array_equal(host_bits(q_dev), q_host)         # q turned in place
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_append_explicit_large_positions_bit_exact():
    """Explicit positions up to ~2.6e5 (long context at 4 tokens per slot)."""
    case = small_case(batch=4, hq=32, hkv=8, d=128, page=16, counts=(3, 3, 3, 3), seed=3)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    pos = np.array([0, 4095, 131071, 262143], np.int32)
    q_host = case.q.copy()
    q_dev = dev_bf16(case.q)
    assert oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q_host, pos=pos) == 0
    ham.ham_kv_append(kv, 0, q_dev, dev_bf16(case.k_new), dev_bf16(case.v_new), dev_i32(pos),
                      dev_i32(case.ntok_new))
    k, v, p, _ = _export_host(kv)
    assert np.array_equal(k, oc.k_pool) and np.array_equal(v, oc.v_pool)
    assert np.array_equal(p, oc.slot_pos)
    assert np.array_equal(host_bits(q_dev), q_host)


def test_append_touches_only_its_rows():
    case = small_case(batch=2, d=64, page=16, counts=(31, 64), seed=4)
    kv = gpu_cache(case)
    k0, v0, p0, n0 = _export_host(kv)
    ham.ham_kv_append(kv, 0, None, dev_bf16(case.k_new), dev_bf16(case.v_new), None,
                      dev_i32(case.ntok_new))
    k1, v1, p1, n1 = _export_host(kv)
    rows = {(int(case.page_table[b, n // 16]), n % 16) for b, n in enumerate((31, 64))}
    changed = np.argwhere((k1 != k0).any(-1) | (v1 != v0).any(-1))
    assert {(int(p), int(r)) for p, _, r in changed} <= rows
    assert len(np.argwhere((p1 != p0) | (n1 != n0))) <= 2


def test_append_device_errors_skip_the_write():
    case = small_case(batch=2, d=64, page=16, counts=(5, 6), seed=5, extra_slots=1)
    kv = gpu_cache(case)
    k0, v0, _, _ = _export_host(kv)
    # ntok < 1 for sequence 0, sequence 1 fine
    ham.ham_kv_append(kv, 0, None, dev_bf16(case.k_new), dev_bf16(case.v_new), None,
                      dev_i32(np.array([0, 2], np.int32)))
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NTOK
    slots, _ = ham.ham_kv_layer_lengths(kv, 0)
    assert list(slots) == [5, 7]
    # sequence 1 is now full (capacity 7): its append is refused on the device
    ham.ham_kv_append(kv, 0, None, dev_bf16(case.k_new), dev_bf16(case.v_new), None,
                      dev_i32(np.array([1, 1], np.int32)))
    with pytest.raises(ham.HamError) as e:
        ham.ham_slot_lengths(kv)
    assert e.value.status == ham.HAM_EDEVICE
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_CAPACITY
    slots, _ = ham.ham_kv_layer_lengths(kv, 0)
    assert list(slots) == [6, 7]
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_host_side_errors_launch_nothing():
    case = small_case(batch=2, d=64, page=16, counts=(5, 6), seed=6)
    kv = gpu_cache(case)
    t = __import__("torch")
    bad = t.zeros(10, dtype=t.bfloat16, device="cuda")
    with pytest.raises(ValueError):
        ham.ham_kv_append(kv, 0, None, bad, bad, None, dev_i32(case.ntok_new))
    with pytest.raises(ham.HamError) as e:
        ham.ham_kv_append(kv, 3, None, dev_bf16(case.k_new), dev_bf16(case.v_new), None,
                          dev_i32(case.ntok_new))
    assert e.value.status == ham.HAM_EINVAL
    pt = ham.ham_kv_get_page_table(kv)
    assert np.array_equal(pt, case.page_table)
    bad_pt = pt.copy()
    bad_pt[0, 0] = bad_pt[1, 0]                  # page used twice
    with pytest.raises(ham.HamError):
        ham.ham_kv_set_page_table(kv, bad_pt)
    bad_pt = pt.copy()
    bad_pt[0, 0] = case.pool_pages               # outside the pool
    with pytest.raises(ham.HamError):
        ham.ham_kv_set_page_table(kv, bad_pt)
    assert np.array_equal(ham.ham_kv_get_page_table(kv), case.page_table)
    slots, _ = ham.ham_slot_lengths(kv)
    assert list(slots) == [5, 6]


def test_layers_keep_separate_pools_and_counters():
    case = small_case(batch=2, d=64, page=16, counts=(9, 20), seed=7)
    kv = gpu_cache(case, layers=3)
    rng = wl.rng_for(7, 3)
    news = []
    for layer in range(3):
        k_new = wl.normal_bf16(rng, case.k_new.shape)
        news.append(k_new)
        ham.ham_kv_append(kv, layer, None, dev_bf16(k_new), dev_bf16(case.v_new), None,
                          dev_i32(np.array([1, 1], np.int32)))
    for layer in range(3):
        slots, _ = ham.ham_kv_layer_lengths(kv, layer)
        assert list(slots) == [10, 21]
        k, _, _, _ = _export_host(kv, layer)
        page, row = case.page_table[0, 9 // 16], 9 % 16
        assert np.array_equal(k[page, :, row], oracle.rope_bf16(news[layer][0], 9))
    ham.ham_kv_reset(kv)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert list(slots) == [0, 0] and list(tokens) == [0, 0]
