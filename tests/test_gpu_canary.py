"""GPU: no stray writes into pool pages a cache does not map.

Canary pages: the pool is first filled to capacity through one page table, whose pages then
hold a known pattern of rows and slot metadata; the page table is switched to a disjoint set
of pages and the cache is driven through fill, appends, decode attention, fused decode steps
and (bf16 pools) a chunked prefill.  Every byte of the canary pages (K and V rows, slot
positions and token counts, and for FP8 pools the codes' exponents) must come back unchanged:
a write through a wrong page id, a wrong row or a wrong stride would land there.
"""
import numpy as np
import pytest

from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import dev_bf16, dev_i32, small_case, torch

pytestmark = pytest.mark.gpu


def _snapshot(kv, fp8):
    t = torch()
    k, v, pos, ntok = ham.ham_kv_export(kv, 0)
    bits = (lambda x: x) if fp8 else (lambda x: x.view(t.int16))  # compare raw bits
    out = [bits(k).cpu().numpy(), bits(v).cpu().numpy(), pos.cpu().numpy(), ntok.cpu().numpy()]
    if fp8:
        out.append(ham.ham_kv_export_scales(kv, 0).cpu().numpy())
    return out


@pytest.mark.parametrize("fp8,page", [(False, 16), (False, 32), (True, 16), (True, 32)])
def test_unmapped_pages_are_never_written(fp8, page):
    t = torch()
    counts = (37, 100, 5)
    case = small_case(batch=3, hq=32, hkv=8, d=128, page=page, counts=counts, seed=61,
                      pool_factor=2.5, extra_slots=12)
    w = case.w
    B, max_pages = w.batch, case.page_table.shape[1]
    assert case.pool_pages >= 2 * B * max_pages
    perm = wl.rng_for(61, 11).permutation(case.pool_pages).astype(np.int32)
    canary_pt = perm[:B * max_pages].reshape(B, max_pages)
    work_pt = perm[B * max_pages:2 * B * max_pages].reshape(B, max_pages)
    canary = np.unique(canary_pt)

    kv = ham.ham_kv_alloc(1, B, w.n_q_heads, w.n_kv_heads, w.head_dim, page, case.max_slots,
                          pool_pages=case.pool_pages,
                          kv_dtype=ham.HAM_KV_E4M3 if fp8 else ham.HAM_KV_BF16)
    # 1. the canary pages, every slot written (rows, positions and token counts)
    ham.ham_kv_set_page_table(kv, canary_pt)
    rng = wl.rng_for(61, 12)
    cap = case.max_slots
    kc = wl.normal_bf16(rng, (B, cap, w.n_kv_heads, w.head_dim))
    vc = wl.normal_bf16(rng, (B, cap, w.n_kv_heads, w.head_dim))
    pos_c = rng.integers(1000, 2000, size=(B, cap)).astype(np.int32)
    ntok_c = rng.integers(1, 5, size=(B, cap)).astype(np.int32)
    ham.ham_kv_fill(kv, 0, dev_bf16(kc), dev_bf16(vc), dev_i32(np.full(B, cap, np.int32)),
                    pos=dev_i32(pos_c), ntok=dev_i32(ntok_c))
    t.cuda.synchronize()
    before = _snapshot(kv, fp8)

    # 2. the working pages: the cache's own life
    ham.ham_kv_set_page_table(kv, work_pt)
    ham.ham_kv_set_lengths(kv, 0, dev_i32(np.zeros(B, np.int32)),
                           t.zeros(B, dtype=t.int64, device="cuda"))
    ham.ham_kv_fill(kv, 0, dev_bf16(case.k), dev_bf16(case.v), dev_i32(case.num_slots),
                    pos=dev_i32(case.slot_pos), ntok=dev_i32(case.slot_ntok))
    q = dev_bf16(case.q)
    out = t.empty(q.shape, dtype=t.bfloat16, device="cuda")
    for step in range(2):
        k_new = dev_bf16(wl.normal_bf16(rng, case.k_new.shape))
        v_new = dev_bf16(wl.normal_bf16(rng, case.v_new.shape))
        ntok = dev_i32(wl.ntok_capped_geometric(rng, (B,)))
        ham.ham_kv_append(kv, 0, q, k_new, v_new, None, ntok)
        ham.ham_decode_attn_ex(kv, 0, q, out)
        ham.ham_decode_step(kv, 0, q, k_new, v_new, None, ntok, out)
    if not fp8:  # chunked prefill: 3, 0 and 2 new rows
        rows = np.array([3, 0, 2], np.int32)
        T = int(rows.sum())
        offsets = np.concatenate([[0], np.cumsum(rows)]).astype(np.int32)
        qp = dev_bf16(wl.normal_bf16(rng, (T, w.n_q_heads, w.head_dim)))
        kp = dev_bf16(wl.normal_bf16(rng, (T, w.n_kv_heads, w.head_dim)))
        vp = dev_bf16(wl.normal_bf16(rng, (T, w.n_kv_heads, w.head_dim)))
        outp = t.empty((T, w.n_q_heads, w.head_dim), dtype=t.bfloat16, device="cuda")
        ham.ham_prefill(kv, 0, qp, kp, vp, dev_i32(offsets), outp)
    t.cuda.synchronize()
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    slots, _ = ham.ham_slot_lengths(kv)
    assert list(slots) == [c + 4 + (r if not fp8 else 0) for c, r in zip(counts, (3, 0, 2))]

    # 3. the canary pages, byte for byte
    after = _snapshot(kv, fp8)
    names = ["K", "V", "slot_pos", "slot_ntok", "exponents"]
    for name, a, b in zip(names, before, after):
        assert np.array_equal(a[canary], b[canary]), f"{name} of a canary page changed"
    # and the working pages did change (the operations ran on them)
    work = np.unique(work_pt)
    assert not np.array_equal(before[0][work], after[0][work])
    ham.ham_kv_free(kv)
