"""GPU: a bounded wait that runs out is reported through the device error word, and the handle
keeps working afterwards.

Every wait of the attention and prefill kernels on their shared-memory ring is bounded; one
that runs out records HAM_DEVERR_TIMEOUT, stops its CTA's work, lets the copies the CTA issued
land and returns, so the GPU context stays usable.  Here the waits are made to run out on a
healthy GPU by shortening their limit to a nanosecond (ham_kv_set_wait_limit_ns): a chunk that
has not landed by the first poll ends the wait.  One CTA streams the whole cache through its
ring, so such a chunk is certain.  After the limit is restored, the same handle gives oracle
parity again.  No fault, trap or endless loop is involved.
"""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import assert_parity, dev_bf16, dev_i32, gpu_cache, gpu_decode, small_case, torch

pytestmark = pytest.mark.gpu


def test_decode_attention_wait_runs_out_then_recovers():
    t = torch()
    case = small_case(batch=1, hq=32, hkv=8, d=128, page=16, counts=(8192,), seed=41)
    kv = gpu_cache(case)
    ham.ham_kv_set_attn_ctas(kv, 1)          # one CTA: 4096 chunks through one 4-stage ring
    ham.ham_kv_set_wait_limit_ns(kv, 1)
    q = dev_bf16(case.q)
    out = t.zeros(q.shape, dtype=t.float32, device="cuda")
    ham.ham_decode_attn_ex(kv, 0, q, out)
    t.cuda.synchronize()
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_TIMEOUT
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE     # read and cleared
    ham.ham_kv_set_wait_limit_ns(kv, 0)                      # the default again
    ref = oracle.OracleCache.from_case(case).decode_attn(case.q)
    assert_parity(gpu_decode(kv, case.q), ref, what="after the timeout, one CTA")
    ham.ham_kv_set_attn_ctas(kv, 0)
    assert_parity(gpu_decode(kv, case.q), ref, what="after the timeout, default CTAs")
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_fp8_decode_attention_wait_runs_out_then_recovers():
    """The FP8 pass (tcgen05 over 128-slot tiles): its ring, product and four-warp waits give up
    on the shortened limit; the copies and products in flight are waited for, the tensor memory
    freed, and the handle decodes at parity afterwards."""
    from test_gpu_fp8 import fp8_cache, _reference, _decode
    t = torch()
    case = small_case(batch=1, hq=32, hkv=8, d=128, page=16, counts=(8192,), seed=45)
    kv = fp8_cache(case)
    ham.ham_kv_set_attn_ctas(kv, 1)          # one CTA: 512 chunks through one 3-tile ring
    ham.ham_kv_set_wait_limit_ns(kv, 1)
    q = dev_bf16(case.q)
    out = t.zeros(q.shape, dtype=t.float32, device="cuda")
    ham.ham_decode_attn_ex(kv, 0, q, out)
    t.cuda.synchronize()
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_TIMEOUT
    ham.ham_kv_set_wait_limit_ns(kv, 0)
    ref = _reference(case).decode_attn(case.q)
    assert_parity(_decode(kv, case.q, f32=True), ref, max_abs=3e-3, mean_abs=3e-4,
                  what="FP8 after the timeout, one CTA")
    ham.ham_kv_set_attn_ctas(kv, 0)
    assert_parity(_decode(kv, case.q), ref, what="FP8 after the timeout, default CTAs")
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_prefill_wait_runs_out_then_recovers():
    t = torch()
    w = wl.Workload("prefill_timeout", batch=1, n_q_heads=32, n_kv_heads=8, head_dim=128,
                    page_slots=16, layers=1, value_scale=1.0, seed=43, pool_factor=1.5)
    case = wl.make_prefill_case(w, (2048,), cached=np.array([1024], np.int32))
    kv = gpu_cache(case.base)
    before, before_tok = ham.ham_kv_layer_lengths(kv, 0)
    offsets = dev_i32(case.offsets)

    def run():
        q = dev_bf16(case.q)
        out = t.full(q.shape, float("nan"), dtype=t.float32, device="cuda")
        ham.ham_prefill(kv, 0, q, dev_bf16(case.k_new), dev_bf16(case.v_new), offsets, out,
                        ntok=dev_i32(case.ntok))
        t.cuda.synchronize()
        return out

    ham.ham_kv_set_wait_limit_ns(kv, 1)
    run()
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_TIMEOUT
    # the rows were stored before the attention ran: roll the counters back, restore the
    # limit and ingest the chunk again
    ham.ham_kv_set_lengths(kv, 0, dev_i32(before),
                           t.from_numpy(np.ascontiguousarray(before_tok, np.int64)).cuda())
    ham.ham_kv_set_wait_limit_ns(kv, 0)
    out = run()
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    oc = oracle.OracleCache.from_case(case.base)
    rc, ref = oc.prefill(case.q.copy(), case.k_new, case.v_new, case.offsets, ntok=case.ntok)
    assert rc == 0
    assert_parity(out.cpu().numpy().astype(np.float64), ref, what="prefill after the timeout")


def test_wait_limit_above_the_default_is_rejected():
    case = small_case(batch=1, counts=(16,), seed=44)
    kv = gpu_cache(case)
    with pytest.raises(ham.HamError) as e:
        ham.ham_kv_set_wait_limit_ns(kv, 3_000_000_000)
    assert e.value.status == ham.HAM_EINVAL
