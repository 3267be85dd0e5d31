"""GPU: decode attention for callers that cannot allocate device memory.

Some callers own all their device memory up front (a host framework's arena, an inference
server plugin) or must not allocate where attention runs.  ham_decode_attn_noalloc takes
every input and output from them and uses a static scratch array compiled into libham.so.
This file is collected last so that a run stopping at its first failure has run the rest.
"""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham

from gpu_helpers import MAX_ABS, MEAN_ABS, assert_parity, dev_bf16, gpu_cache, small_case

pytestmark = pytest.mark.gpu


def _caller_owned_copy(kv):
    """The cache as the caller would hold it: its own pool, page table and counts."""
    import torch
    k_pool, v_pool, _, _ = ham.ham_kv_export(kv, 0)
    page_table = torch.from_numpy(ham.ham_kv_get_page_table(kv)).cuda()
    slots, _ = ham.ham_slot_lengths(kv)
    return k_pool, v_pool, page_table, torch.from_numpy(slots).cuda()


@pytest.mark.parametrize("hq,hkv,d,counts", [(32, 8, 128, (2000, 35, 901)),
                                             (8, 2, 64, (0, 300))])
def test_noalloc_matches_decode_attn_on_two_calls(hq, hkv, d, counts):
    import torch
    case = small_case(batch=len(counts), hq=hq, hkv=hkv, d=d, page=16, counts=counts, seed=21)
    kv = gpu_cache(case)
    q = dev_bf16(case.q)
    ref = torch.full(q.shape, float("nan"), dtype=torch.float32, device="cuda")
    ham.ham_decode_attn_ex(kv, 0, q, ref)
    ref = ref.cpu().numpy().astype(np.float64)
    k_pool, v_pool, page_table, num_slots = _caller_owned_copy(kv)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    for dtype in (torch.float32, torch.bfloat16):        # two calls in a row
        out = torch.full(q.shape, float("nan"), dtype=dtype, device="cuda")
        ham.ham_decode_attn_noalloc(k_pool, v_pool, page_table, num_slots, q, out,
                                    kv.max_slots, err=err)
        torch.cuda.synchronize()
        got = out.float().cpu().numpy().astype(np.float64)
        assert_parity(got, ref, MAX_ABS, MEAN_ABS, what=f"noalloc vs ham_decode_attn {dtype}")
        assert int(err.item()) == 0
    # and against the oracle directly
    assert_parity(got, oracle.OracleCache.from_case(case).decode_attn(case.q), what="oracle")


def test_noalloc_rejects_configurations_beyond_its_scratch():
    import torch
    case = small_case(batch=2, hq=32, hkv=8, d=128, page=16, counts=(100, 100), seed=22)
    kv = gpu_cache(case)
    q = dev_bf16(case.q)
    out = torch.zeros(q.shape, dtype=torch.bfloat16, device="cuda")
    k_pool, v_pool, page_table, num_slots = _caller_owned_copy(kv)
    with pytest.raises(ham.HamError) as e:
        ham.ham_decode_attn_noalloc(k_pool, v_pool, page_table, num_slots, q, out,
                                    kv.max_slots, ctas=8000)
    assert e.value.status == ham.HAM_EINVAL and "scratch" in str(e.value)
    assert float(out.abs().sum()) == 0.0                   # nothing ran
