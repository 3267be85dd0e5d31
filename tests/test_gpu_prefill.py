"""GPU: chunked prefill (ham_prefill) against the fp64 oracle on the same seeded bits.

The stored slots (RoPE'd keys, values, positions, token counts, counters) and the rotated
queries are compared bit for bit; the attention output within the bf16 parity bar."""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import assert_parity, dev_bf16, dev_i32, gpu_cache, host_bits, torch

pytestmark = pytest.mark.gpu


def _w(batch, hq, hkv, d, page, seed, scale=1.0):
    return wl.Workload(f"prefill_s{seed}", batch=batch, n_q_heads=hq, n_kv_heads=hkv,
                       head_dim=d, page_slots=page, layers=1, value_scale=scale, seed=seed,
                       pool_factor=1.5)


def _gpu(case, pos_mode=ham.HAM_POS_SLOT, f32=False, pos=None, with_ntok=True, offsets=None):
    t = torch()
    kv = gpu_cache(case.base, pos_mode=pos_mode)
    q = dev_bf16(case.q)
    out = t.full(q.shape, float("nan"), dtype=t.float32 if f32 else t.bfloat16, device="cuda")
    ham.ham_prefill(kv, 0, q, dev_bf16(case.k_new), dev_bf16(case.v_new),
                    dev_i32(case.offsets if offsets is None else offsets), out,
                    pos=None if pos is None else dev_i32(pos),
                    ntok=dev_i32(case.ntok) if with_ntok else None)
    t.cuda.synchronize()
    return kv, q, out


def _oracle(case, pos_mode=ham.HAM_POS_SLOT, pos=None, want=None, offsets=None):
    oc = oracle.OracleCache.from_case(case.base)
    qq = case.q.copy()
    rc, out = oc.prefill(qq, case.k_new, case.v_new,
                         case.offsets if offsets is None else offsets, ntok=case.ntok,
                         pos=pos, pos_mode=pos_mode, want=want)
    return oc, qq, rc, out


def _check_state(kv, q, oc, q_ref):
    k, v, pos, ntok = ham.ham_kv_export(kv, 0)
    assert np.array_equal(host_bits(k), oc.k_pool), "stored keys"
    assert np.array_equal(host_bits(v), oc.v_pool), "stored values"
    assert np.array_equal(pos.cpu().numpy(), oc.slot_pos), "slot positions"
    assert np.array_equal(ntok.cpu().numpy(), oc.slot_ntok), "slot token counts"
    slots, tokens = ham.ham_kv_layer_lengths(kv, 0)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert np.array_equal(host_bits(q), q_ref), "rotated queries"


def _out(t):
    return t.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("hq,hkv,d,page,cached,rows", [
    (8, 2, 64, 16, (0, 37, 100), (50, 17, 130)),     # group 4: 32-row query blocks, ragged
    (32, 8, 128, 16, (0, 200), (300, 65)),           # the Llama-8B head shape
    (8, 8, 128, 32, (5,), (200,)),                   # group 1: 128-row query blocks
    (16, 2, 64, 16, (64, 0), (33, 16)),              # group 8: 16-row query blocks
    (8, 4, 128, 64, (0, 1, 2), (1, 0, 70)),          # group 2; an empty and a one-row chunk
])
def test_prefill_matches_oracle(hq, hkv, d, page, cached, rows):
    w = _w(len(rows), hq, hkv, d, page, seed=sum(rows))
    case = wl.make_prefill_case(w, rows, cached=np.array(cached, np.int32))
    kv, q, out = _gpu(case)
    oc, q_ref, rc, ref = _oracle(case)
    assert rc == 0
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    _check_state(kv, q, oc, q_ref)
    assert_parity(_out(out), ref, what="prefill output")


# Short chunks over long caches: the attention grid is split over the cached slots (each split at
# least 8 tiles of 64 cached slots) and a merge kernel combines the splits' partials; sequences
# with few cached slots in the same call stay whole.
@pytest.mark.parametrize("hq,hkv,d,page,cached,rows,f32", [
    (32, 8, 128, 16, (4096, 1500), (40, 9), False),      # 8 and 2 splits; Llama-8B heads
    (32, 8, 128, 16, (4096, 1500), (40, 9), True),       # the same, fp32 output
    (8, 2, 64, 16, (3000, 0, 700), (17, 5, 64), False),  # 5 splits, an empty cache, one split
    (16, 2, 64, 16, (2600,), (20,), False),              # group 8, 5 splits
    (8, 8, 128, 32, (5000,), (100,), False),             # group 1, 9 splits
    (8, 4, 128, 64, (2048, 4000), (1, 70), True),        # group 2; a one-row chunk
])
def test_prefill_split_over_slots_matches_oracle(hq, hkv, d, page, cached, rows, f32):
    w = _w(len(rows), hq, hkv, d, page, seed=sum(cached) % 97 + 5)
    case = wl.make_prefill_case(w, rows, cached=np.array(cached, np.int32))
    kv, q, out = _gpu(case, f32=f32)
    oc, q_ref, rc, ref = _oracle(case)
    assert rc == 0
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    _check_state(kv, q, oc, q_ref)
    assert_parity(_out(out), ref, what="split prefill output" + (" (f32)" if f32 else ""))


@pytest.mark.parametrize("mode", ["token", "explicit"])
def test_prefill_positions(mode):
    w = _w(2, 8, 2, 128, 16, seed=31)
    rng = wl.rng_for(31, 7)
    rows = (40, 75)
    ntok = rng.integers(1, 5, sum(rows)).astype(np.int32)
    case = wl.make_prefill_case(w, rows, cached=np.array([20, 3], np.int32), ntok=ntok)
    pos = None
    pos_mode = ham.HAM_POS_TOKEN if mode == "token" else ham.HAM_POS_SLOT
    if mode == "explicit":
        pos = rng.integers(0, 3000, sum(rows)).astype(np.int32)
    kv, q, out = _gpu(case, pos_mode=pos_mode, pos=pos)
    oc, q_ref, rc, ref = _oracle(case, pos_mode=pos_mode, pos=pos)
    assert rc == 0
    _check_state(kv, q, oc, q_ref)
    assert_parity(_out(out), ref, what=f"prefill output ({mode} positions)")


def test_prefill_f32_output_and_default_ntok():
    w = _w(2, 32, 8, 128, 16, seed=32)
    case = wl.make_prefill_case(w, (90, 130), cached=np.array([64, 10], np.int32))
    kv, q, out = _gpu(case, f32=True, with_ntok=False)   # NULL ntok: one token per row
    oc, q_ref, rc, ref = _oracle(case)
    assert rc == 0
    _check_state(kv, q, oc, q_ref)
    assert_parity(_out(out), ref, what="prefill output (f32)")


def test_prefill_then_decode_sees_the_new_slots():
    from gpu_helpers import gpu_decode
    w = _w(3, 8, 2, 64, 16, seed=33)
    case = wl.make_prefill_case(w, (70, 5, 0), cached=np.array([10, 99, 40], np.int32),
                                headroom=1)
    kv, _, _ = _gpu(case)
    oc, _, rc, _ = _oracle(case)
    assert rc == 0
    qd = wl.normal_bf16(wl.rng_for(33, 9), (3, 8, 64))
    assert_parity(gpu_decode(kv, qd), oc.decode_attn(qd), what="decode after prefill")


def test_prefill_rows_that_do_not_fit():
    w = _w(3, 8, 2, 64, 16, seed=34)
    rows = (6, 9, 4)
    case = wl.make_prefill_case(w, rows, cached=np.array([10, 20, 0], np.int32))
    # sequence 1 needs 29 slots: make the cache hold 25 per sequence
    case.base.max_slots = 25
    kv, q, out = _gpu(case)
    oc, q_ref, rc, ref = _oracle(case)
    assert rc == oracle.ECAPACITY
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_CAPACITY
    _check_state(kv, q, oc, q_ref)
    got = _out(out)
    assert np.all(got[6:15] == 0)
    assert_parity(got, ref, what="prefill output, one sequence rejected")


def test_prefill_bad_token_counts_and_offsets():
    w = _w(2, 8, 2, 64, 16, seed=35)
    ntok = np.ones(30, np.int32)
    ntok[25] = 0
    case = wl.make_prefill_case(w, (20, 10), cached=np.array([3, 4], np.int32), ntok=ntok)
    kv, q, out = _gpu(case)
    oc, q_ref, rc, ref = _oracle(case)
    assert rc == oracle.EINVAL
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NTOK
    _check_state(kv, q, oc, q_ref)
    assert np.all(_out(out)[20:] == 0)
    # offsets that do not describe the call's rows: nothing is stored, every output row is 0
    good = wl.make_prefill_case(w, (20, 10), cached=np.array([3, 4], np.int32))
    kv2, q2, out2 = _gpu(good, offsets=np.array([0, 25, 20], np.int32))
    assert ham.ham_kv_status(kv2) == ham.HAM_DEVERR_NTOK
    assert np.all(_out(out2) == 0)
    slots, _ = ham.ham_kv_layer_lengths(kv2, 0)
    assert list(slots) == [3, 4]
    assert np.array_equal(host_bits(q2), good.q)


def test_prefill_host_errors():
    t = torch()
    w = _w(2, 8, 2, 64, 16, seed=36)
    case = wl.make_prefill_case(w, (4, 4), cached=np.array([0, 0], np.int32))
    kv = gpu_cache(case.base)
    q, k, v = dev_bf16(case.q), dev_bf16(case.k_new), dev_bf16(case.v_new)
    offs = dev_i32(case.offsets)
    out = t.empty_like(q)
    with pytest.raises(ham.HamError):          # out overlapping q
        ham.ham_prefill(kv, 0, q, k, v, offs, q)
    with pytest.raises(ham.HamError):          # layer out of range
        ham.ham_prefill(kv, 1, q, k, v, offs, out)
    with pytest.raises(ValueError):            # offsets of the wrong length
        ham.ham_prefill(kv, 0, q, k, v, dev_i32(case.offsets[:-1]), out)
    with pytest.raises(ValueError):            # k rows differ from q rows
        ham.ham_prefill(kv, 0, q, k[:-1].contiguous(), v, offs, out)
    # zero rows: nothing to do
    z = t.empty((0, 8, 64), dtype=t.bfloat16, device="cuda")
    zk = t.empty((0, 2, 64), dtype=t.bfloat16, device="cuda")
    ham.ham_prefill(kv, 0, z, zk, zk, dev_i32(np.zeros(3, np.int32)), t.empty_like(z))
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


@pytest.mark.parametrize("pw", [wl.P1_PREFILL, wl.P2_CHUNK, wl.P3_SHORT], ids=lambda p: p.name)
def test_prefill_full_size_sampled(pw):
    """The bench workloads at full size: every stored bit, and the output rows of a sample
    (first, last and spread rows of every sequence) against the oracle."""
    B = pw.w.batch
    case = wl.make_prefill_case(pw.w, [pw.rows] * B,
                                cached=np.full(B, pw.cached, np.int32))
    kv, q, out = _gpu(case)
    want = np.zeros(int(case.offsets[-1]), bool)
    for b in range(B):
        a = int(case.offsets[b])
        idx = np.array([0, 1, 31, 32, 33, 63, 64, 127, pw.rows // 2, pw.rows - 2, pw.rows - 1])
        want[a + idx[idx < pw.rows]] = True
    oc, q_ref, rc, ref = _oracle(case, want=want)
    assert rc == 0
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    _check_state(kv, q, oc, q_ref)
    assert_parity(_out(out)[want], ref[want], what=f"{pw.name} sampled rows")
