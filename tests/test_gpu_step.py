"""GPU: the fused decode step (append + attention in one pass over the cache).

The cache, the counters and the rotated q it reports (q_rot) are compared bit for bit with
the oracle's append; its attention output with the oracle's attention over the n + 1 slots.
The query it is given is never written.
"""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import (MAX_ABS, MEAN_ABS, assert_parity, dev_bf16, dev_i32, gpu_cache,
                         host_bits, small_case, torch)

pytestmark = pytest.mark.gpu

# Against the oracle: the tensor-core pass rounds each softmax weight to bf16 (relative
# error <= 2^-8, bf16's unit roundoff), which moves an output by sum_i dw_i (v_i - out) /
# sum(w): errors of random sign, about 2^-8 |v| / sqrt(slots) typically, but on sequences of a
# few slots nothing averages them out, so the bar is the bf16 one (MAX_ABS, MEAN_ABS) even
# with fp32 output.  GPU against GPU with the same split:
# the stored slots' weights are rounded the same way; what differs is the appended slot,
# whose weight the fused step keeps in fp32 (the two calls round it to bf16 in the MMA), and a
# rare one-ulp difference of an fp32-rotated q element.  That moves an output by at most
# 2^-8 * w_new / sum(w) * |v|, small against the bf16 bar.
SAME_SPLIT_MAX, SAME_SPLIT_MEAN = 2e-3, 1e-4
Q_ROT_UNWRITTEN = 0x7FC1  # a bf16 NaN pattern no rotation produces


def _export_host(kv, layer=0):
    k, v, pos, ntok = ham.ham_kv_export(kv, layer)
    return host_bits(k), host_bits(v), pos.cpu().numpy(), ntok.cpu().numpy()


def _assert_cache_equal(kv, oc, layer=0):
    k, v, pos, ntok = _export_host(kv, layer)
    assert np.array_equal(v, oc.v_pool), "V pool"
    assert np.array_equal(k, oc.k_pool), "K pool (RoPE'd keys)"
    assert np.array_equal(pos, oc.slot_pos) and np.array_equal(ntok, oc.slot_ntok)
    slots, tokens = ham.ham_kv_layer_lengths(kv, layer)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)


def _step(kv, q_bits, k_new, v_new, ntok, pos=None, f32=True, layer=0):
    """One fused step; returns (out as float64, q_rot bits).  Checks that q is untouched."""
    t = torch()
    q_dev = dev_bf16(q_bits)
    q_rot = dev_bf16(np.full(q_bits.shape, Q_ROT_UNWRITTEN, np.uint16))
    out = t.full(q_dev.shape, float("nan"), dtype=t.float32 if f32 else t.bfloat16,
                 device="cuda")
    ham.ham_decode_step(kv, layer, q_dev, dev_bf16(k_new), dev_bf16(v_new),
                        None if pos is None else dev_i32(pos), dev_i32(ntok), out, q_rot=q_rot)
    t.cuda.synchronize()
    assert np.array_equal(host_bits(q_dev), q_bits), "q was written"
    return out.float().cpu().numpy().astype(np.float64), host_bits(q_rot)


@pytest.mark.parametrize("pos_mode", [ham.HAM_POS_SLOT, ham.HAM_POS_TOKEN])
@pytest.mark.parametrize("d,hq,hkv,page,counts", [
    (64, 8, 2, 16, (15, 16, 0, 47)),       # new slot ends chunk 0 / opens chunk 1 / first
    (128, 32, 8, 32, (31, 200, 5)),        # page edge; Llama-3 8B head layout
    (128, 8, 8, 16, (1, 64)),              # group 1
    (64, 16, 2, 128, (127, 300)),          # group 8
])
def test_step_matches_oracle(pos_mode, d, hq, hkv, page, counts):
    case = small_case(batch=len(counts), hq=hq, hkv=hkv, d=d, page=page, counts=counts,
                      seed=11, extra_slots=8)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case, pos_mode=pos_mode)
    q = case.q.copy()
    rng = wl.rng_for(11, 60)
    for step in range(3):
        k_new = wl.normal_bf16(rng, case.k_new.shape)
        v_new = wl.normal_bf16(rng, case.v_new.shape)
        ntok = wl.ntok_capped_geometric(rng, (case.w.batch,))
        q_ref = q.copy()
        assert oc.append(k_new, v_new, ntok, q_inout=q_ref, pos_mode=pos_mode) == 0
        ref = oc.decode_attn(q_ref)
        got, q_rot = _step(kv, q, k_new, v_new, ntok)
        assert np.array_equal(q_rot, q_ref), f"q_rot after step {step}"
        assert_parity(got, ref, MAX_ABS, MEAN_ABS, what=f"step {step}")
        q = wl.normal_bf16(rng, case.q.shape)        # next macro-step's fresh queries
    _assert_cache_equal(kv, oc)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_step_batch_above_128():
    """More than 128 sequences: the combine reads the stored CTA ranges; a few long sequences
    span many CTAs, some sequences are empty (the appended slot alone)."""
    rng = np.random.default_rng(9)
    counts = rng.integers(0, 70, size=260)
    counts[rng.choice(260, 6, replace=False)] = 0
    counts[rng.choice(260, 5, replace=False)] = rng.integers(600, 1500, size=5)
    case = small_case(batch=260, hq=16, hkv=2, d=128, page=32, counts=tuple(int(c) for c in counts),
                      seed=9, extra_slots=4)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    rng2 = wl.rng_for(9, 61)
    q = case.q.copy()
    for step in range(2):
        k_new = wl.normal_bf16(rng2, case.k_new.shape)
        v_new = wl.normal_bf16(rng2, case.v_new.shape)
        ntok = wl.ntok_capped_geometric(rng2, (case.w.batch,))
        q_ref = q.copy()
        assert oc.append(k_new, v_new, ntok, q_inout=q_ref) == 0
        ref = oc.decode_attn(q_ref)
        got, q_rot = _step(kv, q, k_new, v_new, ntok)
        assert np.array_equal(q_rot, q_ref), f"q_rot after step {step}"
        assert_parity(got, ref, MAX_ABS, MEAN_ABS, what=f"B260 step {step}")
        q = wl.normal_bf16(rng2, case.q.shape)
    _assert_cache_equal(kv, oc)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_step_equals_append_then_attend_on_gpu():
    """Same cache bits and rotated q bits as the two separate calls; outputs agree closely."""
    case = small_case(batch=3, hq=32, hkv=8, d=128, page=16, counts=(100, 17, 640), seed=12)
    kv1, kv2 = gpu_cache(case), gpu_cache(case)
    for kv in (kv1, kv2):
        ham.ham_kv_set_attn_ctas(kv, 300)          # the same split for both paths
    q1 = dev_bf16(case.q)
    t = torch()
    out1 = t.empty(q1.shape, dtype=t.float32, device="cuda")
    ham.ham_kv_append(kv1, 0, q1, dev_bf16(case.k_new), dev_bf16(case.v_new), None,
                      dev_i32(case.ntok_new))
    ham.ham_decode_attn_ex(kv1, 0, q1, out1)
    out2, q_rot = _step(kv2, case.q, case.k_new, case.v_new, case.ntok_new)
    assert np.array_equal(host_bits(q1), q_rot)
    a, b = _export_host(kv1), _export_host(kv2)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    assert_parity(out2, out1.cpu().numpy().astype(np.float64), SAME_SPLIT_MAX, SAME_SPLIT_MEAN,
                  what="2-call")


def test_step_positions_beyond_the_rope_table():
    """Explicit positions up to ~2.6e5 take the sincos path in both kernels."""
    case = small_case(batch=4, hq=32, hkv=8, d=128, page=16, counts=(3, 40, 0, 16), seed=13)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    pos = np.array([0, 4095, 131071, 262143], np.int32)
    q_ref = case.q.copy()
    assert oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q_ref, pos=pos) == 0
    ref = oc.decode_attn(q_ref)
    got, q_rot = _step(kv, case.q, case.k_new, case.v_new, case.ntok_new, pos=pos)
    assert np.array_equal(q_rot, q_ref)
    assert_parity(got, ref, MAX_ABS, MEAN_ABS, what="large positions")
    _assert_cache_equal(kv, oc)


@pytest.mark.parametrize("ctas", [1, 5, 37, 600])
def test_step_split_counts(ctas):
    """Any CTA count: identical cache and q_rot, attention within tolerance."""
    case = small_case(batch=3, hq=8, hkv=2, d=64, page=16, counts=(0, 333, 48), seed=14)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    ham.ham_kv_set_attn_ctas(kv, ctas)
    q_ref = case.q.copy()
    assert oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q_ref) == 0
    got, q_rot = _step(kv, case.q, case.k_new, case.v_new, case.ntok_new)
    assert np.array_equal(q_rot, q_ref)
    assert_parity(got, oc.decode_attn(q_ref), MAX_ABS, MEAN_ABS, what=f"ctas={ctas}")
    _assert_cache_equal(kv, oc)


def test_step_failed_appends_behave_like_the_two_calls():
    """A full sequence and ntok = 0 (one of them on an empty sequence): no append, unrotated
    q attends over the old slots (none: output 0), the error is recorded and q_rot rows of
    those sequences are left alone."""
    case = small_case(batch=4, hq=8, hkv=2, d=64, page=16, counts=(20, 37, 9, 0), seed=15,
                      extra_slots=0)
    oc = oracle.OracleCache.from_case(case)
    assert case.max_slots == 37                    # sequence 1 is full
    kv = gpu_cache(case)
    ntok = np.array([2, 1, 0, 0], np.int32)        # sequences 2 and 3 give ntok = 0
    q_ref = case.q.copy()
    assert oc.append(case.k_new, case.v_new, ntok, q_inout=q_ref) != 0
    ref = oc.decode_attn(q_ref)
    got, q_rot = _step(kv, case.q, case.k_new, case.v_new, ntok)
    assert np.array_equal(q_rot[0], q_ref[0])
    assert np.all(q_rot[1:] == Q_ROT_UNWRITTEN)
    assert np.array_equal(q_ref[1:], case.q[1:])   # the oracle left them unrotated too
    assert_parity(got, ref, MAX_ABS, MEAN_ABS, what="failed appends")
    assert np.all(got[3] == 0.0)                   # nothing to attend to
    # read (and clear) the error word first: the counter read-back refuses while it is set
    assert ham.ham_kv_status(kv) in (ham.HAM_DEVERR_CAPACITY, ham.HAM_DEVERR_NTOK)
    _assert_cache_equal(kv, oc)


def test_step_alternating_caches():
    """Steps alternating between two caches on one stream: each launch may plan and start its
    first copies before the previous one (other cache) has finished.  Every step is checked."""
    cases = [small_case(batch=3, hq=32, hkv=8, d=128, page=16, counts=c, seed=s)
             for c, s in (((300, 17, 64), 19), ((5, 250, 0), 20))]
    ocs = [oracle.OracleCache.from_case(c) for c in cases]
    kvs = [gpu_cache(c) for c in cases]
    rng = wl.rng_for(19, 61)
    for step in range(3):
        for case, oc, kv in zip(cases, ocs, kvs):
            q = wl.normal_bf16(rng, case.q.shape)
            k_new = wl.normal_bf16(rng, case.k_new.shape)
            v_new = wl.normal_bf16(rng, case.v_new.shape)
            ntok = wl.ntok_capped_geometric(rng, (case.w.batch,))
            q_ref = q.copy()
            assert oc.append(k_new, v_new, ntok, q_inout=q_ref) == 0
            got, q_rot = _step(kv, q, k_new, v_new, ntok)
            assert np.array_equal(q_rot, q_ref)
            assert_parity(got, oc.decode_attn(q_ref), MAX_ABS, MEAN_ABS, what=f"step {step}")
    for oc, kv in zip(ocs, kvs):
        _assert_cache_equal(kv, oc)


def test_step_host_errors():
    case = small_case(batch=2, counts=(3, 4), seed=16)
    kv = gpu_cache(case)
    t = torch()
    q = dev_bf16(case.q)
    k, v, n = dev_bf16(case.k_new), dev_bf16(case.v_new), dev_i32(case.ntok_new)
    out = t.empty(q.shape, dtype=t.bfloat16, device="cuda")
    with pytest.raises(ham.HamError):
        ham.ham_decode_step(kv, 1, q, k, v, None, n, out)          # layer out of range
    with pytest.raises(ham.HamError):
        ham.ham_decode_step(kv, 0, q, k, v, None, n, q)             # out aliases q
    with pytest.raises(ham.HamError):
        ham.ham_decode_step(kv, 0, q, k, v, None, n, out, q_rot=out)  # q_rot aliases out
    rc = ham.lib().ham_decode_step(kv, 0, q.data_ptr() + 2, None, k.data_ptr(), v.data_ptr(),
                                   None, n.data_ptr(), out.data_ptr(), ham.HAM_DTYPE_BF16, None)
    assert rc == ham.HAM_EINVAL
    t.cuda.synchronize()
    slots, _ = ham.ham_slot_lengths(kv)
    assert list(slots) == [3, 4]                   # nothing launched


def test_step_then_attention_sees_the_slot():
    """After a step, plain attention with the rotated q reproduces the step's output."""
    case = small_case(batch=2, hq=32, hkv=8, d=128, page=32, counts=(63, 500), seed=17)
    kv = gpu_cache(case)
    ham.ham_kv_set_attn_ctas(kv, 200)
    got, q_rot = _step(kv, case.q, case.k_new, case.v_new, case.ntok_new)
    t = torch()
    again = t.empty(case.q.shape, dtype=t.float32, device="cuda")
    ham.ham_decode_attn_ex(kv, 0, dev_bf16(q_rot), again)
    assert_parity(got, again.cpu().numpy().astype(np.float64), SAME_SPLIT_MAX, SAME_SPLIT_MEAN,
                  what="step vs attention after it")


def test_step_without_q_rot():
    """q_rot is optional; the cache and the output do not depend on it."""
    case = small_case(batch=2, hq=8, hkv=2, d=64, page=16, counts=(40, 70), seed=18)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    q_ref = case.q.copy()
    assert oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q_ref) == 0
    t = torch()
    out = t.full(case.q.shape, float("nan"), dtype=t.float32, device="cuda")
    ham.ham_decode_step(kv, 0, dev_bf16(case.q), dev_bf16(case.k_new), dev_bf16(case.v_new),
                        None, dev_i32(case.ntok_new), out)
    assert_parity(out.cpu().numpy().astype(np.float64), oc.decode_attn(q_ref), MAX_ABS,
                  MEAN_ABS, what="no q_rot")
    _assert_cache_equal(kv, oc)


@pytest.mark.parametrize("w", [wl.C1_LLAMA8B, wl.C2_RAGGED], ids=lambda w: w.name)
def test_step_full_size(w):
    """The bench's workloads and launch configuration (default CTAs, bf16 output)."""
    case = wl.make_case(w, extra_slots=4)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    q_ref = case.q.copy()
    assert oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q_ref) == 0
    ref = oc.decode_attn(q_ref)
    got, q_rot = _step(kv, case.q, case.k_new, case.v_new, case.ntok_new, f32=False)
    assert np.array_equal(q_rot, q_ref)
    assert_parity(got, ref, what=w.name)
    # the appended rows, bit for bit (the whole pool at this size is compared too)
    _assert_cache_equal(kv, oc)
