"""GPU: the layer front (ham_qkv_append) against the oracle.

The projection accumulates in fp32 on the tensor cores while the oracle sums in fp64.  Each
stored bf16 value must lie within one bf16 ulp of the exact value plus the fp32 accumulation
slack 2^-14 * sum_k |W_ok x_k| (summed over both elements of a rotation pair), so a value that
cancels to near zero may differ by several of its own ulps; at most 1% of the values may differ
from the oracle's bits at all.  Everything else (slot placement, metadata, counters, rows the
call does not own) is exact, and attention over the result meets the decode parity bar.
"""
import numpy as np
import pytest

import oracle
from oracle import front as ofront
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import assert_parity, dev_bf16, dev_i32, gpu_cache, gpu_decode, host_bits, \
    small_case

pytestmark = pytest.mark.gpu

MAX_DIFF_SHARE = 0.01     # values whose bits differ from the oracle's (observed: well under 1%)
ACC_SLACK = 2.0 ** -14    # fp32 accumulation error bar, relative to sum_k |W_ok x_k|


def assert_front_close(got_bits, ref_bits, exact, mag, what):
    """got within one bf16 ulp of `exact` plus ACC_SLACK * mag; few bits differ from ref_bits."""
    g = ofront.bf16_bits_to_f64(got_bits)
    ulp = np.ldexp(1.0, np.frexp(np.abs(exact))[1] - 8)
    err = np.abs(g - exact)
    bound = ulp + ACC_SLACK * mag
    worst = float((err / bound).max()) if err.size else 0.0
    assert worst <= 1.0, f"{what}: error {worst:.2f} x the bound"
    share = float((np.asarray(got_bits) != np.asarray(ref_bits)).mean()) if err.size else 0.0
    assert share <= MAX_DIFF_SHARE, f"{what}: {share:.3%} of values differ from the oracle"
    return share


def _mag(x, W):
    """sum_k |W_ok x_k| for every (sequence, output row)."""
    return np.abs(ofront.bf16_bits_to_f64(x)) @ np.abs(ofront.bf16_bits_to_f64(W)).T


def _exact_heads(y, mag, p, d, rotate):
    """Exact fp64 head rows (rotated at p if asked) and their slack magnitudes; y, mag [n*d]."""
    y = y.reshape(-1, d)
    m = mag.reshape(-1, d)
    half = d // 2
    if not rotate:
        return y, m
    pair = m[:, :half] + m[:, half:]
    return ofront.rope_values(y, p), np.concatenate([pair, pair], axis=1)


def _export(kv, layer=0):
    k, v, pos, ntok = ham.ham_kv_export(kv, layer)
    return host_bits(k), host_bits(v), pos.cpu().numpy(), ntok.cpu().numpy()


def _step(oc, kv, x, W, ntok, hq, hkv, d, pos=None, pos_mode=ham.HAM_POS_SLOT):
    """One front call on both sides.  Returns the oracle status and the appended rows
    (page, row, exact k, k slack, exact v, v slack) per appended sequence; checks q_rot."""
    import torch
    B = x.shape[0]
    P = oc.shape["page_slots"]
    n0 = oc.num_slots.copy()
    st, q_ref, y = ofront.qkv_append(oc, x, W, ntok, pos=pos, pos_mode=pos_mode)
    mag = _mag(x, W)
    q_rot = torch.full((B, hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    ham.ham_qkv_append(kv, 0, dev_bf16(x), dev_bf16(W), dev_i32(ntok), q_rot,
                       pos=None if pos is None else dev_i32(pos))
    torch.cuda.synchronize()
    appended, q_exact, q_mag = [], [], []
    for b in range(B):
        ok = oc.num_slots[b] == n0[b] + 1
        n = int(n0[b])
        page, row = (int(oc.page_table[b, n // P]), n % P) if ok else (-1, -1)
        p = int(oc.slot_pos[page, row]) if ok else 0
        qe, qm = _exact_heads(y[b, : hq * d], mag[b, : hq * d], p, d, ok)
        q_exact.append(qe)
        q_mag.append(qm)
        if ok:
            ke, km = _exact_heads(y[b, hq * d: (hq + hkv) * d], mag[b, hq * d: (hq + hkv) * d],
                                  p, d, True)
            ve, vm = _exact_heads(y[b, (hq + hkv) * d:], mag[b, (hq + hkv) * d:], p, d, False)
            appended.append((page, row, ke, km, ve, vm))
    share = assert_front_close(host_bits(q_rot), q_ref, np.stack(q_exact), np.stack(q_mag),
                               "q_rot")
    return st, appended, q_rot, q_ref, share


def _check_pools(kv, oc, appended):
    """Rows the calls appended: within the bound; every other byte of the pools: exact."""
    k, v, p, n = _export(kv)
    mask = np.zeros(k.shape[:3], bool)            # [page][head][row]
    for page, row, ke, km, ve, vm in appended:
        mask[page, :, row] = True
        assert_front_close(k[page, :, row], oc.k_pool[page, :, row], ke, km, "K rows")
        assert_front_close(v[page, :, row], oc.v_pool[page, :, row], ve, vm, "V rows")
    assert np.array_equal(k[~mask], oc.k_pool[~mask]) and np.array_equal(v[~mask], oc.v_pool[~mask])
    assert np.array_equal(p, oc.slot_pos) and np.array_equal(n, oc.slot_ntok)


def _run(hq, hkv, d, H, counts, seed, pos_mode=ham.HAM_POS_SLOT, steps=2, explicit_pos=False):
    B = len(counts)
    case = small_case(batch=B, hq=hq, hkv=hkv, d=d, page=16, counts=counts, seed=seed,
                      extra_slots=steps + 2)
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case, pos_mode=pos_mode)
    fw = wl.front_workload(B, hidden=H, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, seed=seed)
    rng = wl.rng_for(seed, 77)
    appended = []
    for step in range(steps):
        x, W = wl.front_inputs(fw, stream=step)
        ntok = wl.ntok_capped_geometric(rng, (B,))
        pos = rng.integers(0, 200000, B).astype(np.int32) if explicit_pos else None
        st, rows, q_rot, q_ref, _ = _step(oc, kv, x, W, ntok, hq, hkv, d, pos=pos,
                                          pos_mode=pos_mode)
        assert st == 0
        appended += rows
    _check_pools(kv, oc, appended)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    return case, oc, kv, q_rot, q_ref


@pytest.mark.parametrize("hq,hkv,d,H,counts", [
    (8, 2, 64, 256, (37, 80, 15)),            # one 32-column step per warp
    (32, 8, 128, 4096, (5, 16, 100, 31, 0, 7, 64, 200)),   # Llama-3-8B shapes, batch 8
    (16, 4, 64, 768, tuple(range(1, 13))),    # 3 steps per warp (remainder loop), 2 n-tiles
    (8, 8, 128, 512, tuple((7 * i) % 50 for i in range(37))),  # 2 grid rows, 4 n-tiles
])
def test_front_matches_oracle(hq, hkv, d, H, counts):
    case, oc, kv, q_rot, q_ref = _run(hq, hkv, d, H, counts, seed=hq + H)
    # attention over the appended cache meets the decode parity bar
    got = gpu_decode(kv, host_bits(q_rot))
    ref = oc.decode_attn(q_ref)
    assert_parity(got, ref, what="attention after the front")


@pytest.mark.parametrize("pos_mode,explicit", [(ham.HAM_POS_TOKEN, False), (ham.HAM_POS_SLOT, True)])
def test_front_positions(pos_mode, explicit):
    _run(32, 8, 128, 1024, (3, 17, 40), seed=9, pos_mode=pos_mode, steps=3, explicit_pos=explicit)


def test_front_touches_only_the_new_rows():
    case = small_case(batch=2, hq=8, hkv=2, d=64, page=16, counts=(31, 64), seed=10)
    kv = gpu_cache(case)
    k0, v0, p0, n0 = _export(kv)
    fw = wl.front_workload(2, hidden=256, n_q_heads=8, n_kv_heads=2, head_dim=64, seed=10)
    x, W = wl.front_inputs(fw)
    import torch
    q_rot = torch.empty((2, 8, 64), dtype=torch.bfloat16, device="cuda")
    ham.ham_qkv_append(kv, 0, dev_bf16(x), dev_bf16(W), dev_i32(np.array([1, 2], np.int32)), q_rot)
    k1, v1, p1, n1 = _export(kv)
    changed = np.zeros(k0.shape[:3], bool)     # [page][head][row]
    for b, n in enumerate((31, 64)):
        page = case.page_table[b, n // 16]
        changed[page, :, n % 16] = True
    assert np.array_equal(k1[~changed], k0[~changed]) and np.array_equal(v1[~changed], v0[~changed])
    meta_changed = changed[:, 0, :]
    assert np.array_equal(p1[~meta_changed], p0[~meta_changed])
    assert np.array_equal(n1[~meta_changed], n0[~meta_changed])


def test_front_failed_sequences():
    """ntok < 1 and a full sequence: no slot, counters unchanged, device error set, q_rot is the
    unrotated projection; the other sequences are appended."""
    case = small_case(batch=3, hq=8, hkv=2, d=64, page=16, counts=(5, 10, 12), seed=11,
                      extra_slots=0)                           # capacity 12: sequence 2 is full
    oc = oracle.OracleCache.from_case(case)
    kv = gpu_cache(case)
    fw = wl.front_workload(3, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=64, seed=11)
    x, W = wl.front_inputs(fw)
    ntok = np.array([0, 2, 1], np.int32)
    st, appended, _, _, _ = _step(oc, kv, x, W, ntok, 8, 2, 64)
    assert st != 0 and len(appended) == 1
    assert ham.ham_kv_status(kv) in (ham.HAM_DEVERR_NTOK, ham.HAM_DEVERR_CAPACITY)
    _check_pools(kv, oc, appended)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert list(slots) == [5, 11, 12]
    assert np.array_equal(tokens, oc.num_tokens)


def test_front_rejects_bad_arguments():
    import torch
    case = small_case(batch=2, hq=8, hkv=2, d=64, page=16, counts=(3, 4), seed=12)
    kv = gpu_cache(case)
    x = torch.zeros((2, 200), dtype=torch.bfloat16, device="cuda")       # hidden not a multiple of 256
    W = torch.zeros((12 * 64, 200), dtype=torch.bfloat16, device="cuda")
    q_rot = torch.empty((2, 8, 64), dtype=torch.bfloat16, device="cuda")
    ntok = torch.ones(2, dtype=torch.int32, device="cuda")
    with pytest.raises(ham.HamError) as e:
        ham.ham_qkv_append(kv, 0, x, W, ntok, q_rot)
    assert e.value.status == ham.HAM_EINVAL
    x = torch.zeros((2, 256), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((12 * 64, 256), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ham.HamError):
        ham.ham_qkv_append(kv, 1, x, W, ntok, q_rot)                     # layer out of range
    slots, _ = ham.ham_slot_lengths(kv)
    assert list(slots) == [3, 4]                                          # nothing ran


@pytest.mark.parametrize("hq,hkv,H,counts", [
    (32, 8, 4096, (5, 16, 100, 31, 0, 7, 64, 200)),   # Llama-3-8B shapes, batch 8
    (8, 8, 512, tuple((7 * i) % 50 for i in range(37))),  # 2 grid rows (two last CTAs)
])
def test_front_over_fp8_pools(hq, hkv, H, counts):
    """FP8 (e4m3) pools: the row's last CTA encodes the new slot's rows.  Slot metadata and
    counters exactly as the oracle's; attention over the cache against the oracle's attention
    over its own front rows decoded through the FP8 format (the decode bar).  And, between two
    CUDA paths, the same call on a bf16 cache: the same q_rot bits, and its stored rows, encoded
    by the oracle's FP8 encoder, the FP8 cache's codes and exponents bit for bit."""
    import torch
    from oracle import fp8 as ofp8
    from test_gpu_fp8 import fp8_cache, _decoded_cache, _export as fp8_export
    d, B = 128, len(counts)
    case = small_case(batch=B, hq=hq, hkv=hkv, d=d, page=16, counts=counts, seed=hq + 7,
                      extra_slots=4)
    oc = oracle.OracleCache.from_case(case)
    kv8 = fp8_cache(case)
    kvb = gpu_cache(case)
    fw = wl.front_workload(B, hidden=H, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, seed=hq + 7)
    rng = wl.rng_for(hq + 7, 78)
    for step in range(2):
        x, W = wl.front_inputs(fw, stream=step)
        ntok = wl.ntok_capped_geometric(rng, (B,))
        st, q_ref, _ = ofront.qkv_append(oc, x, W, ntok)
        assert st == 0
        q8 = torch.full((B, hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        qb = torch.full_like(q8, float("nan"))
        ham.ham_qkv_append(kv8, 0, dev_bf16(x), dev_bf16(W), dev_i32(ntok), q8)
        ham.ham_qkv_append(kvb, 0, dev_bf16(x), dev_bf16(W), dev_i32(ntok), qb)
        torch.cuda.synchronize()
        assert np.array_equal(host_bits(q8), host_bits(qb)), "q_rot, FP8 against bf16 pools"
    assert ham.ham_kv_status(kv8) == ham.HAM_DEVERR_NONE
    slots, tokens = ham.ham_slot_lengths(kv8)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    k8, v8, e8, pos8, ntok8 = fp8_export(kv8)
    assert np.array_equal(pos8, oc.slot_pos) and np.array_equal(ntok8, oc.slot_ntok)
    # parity: attention over the FP8 cache against the oracle over its front rows, decoded
    got = gpu_decode(kv8, host_bits(q8))
    ref = _decoded_cache(case, oc).decode_attn(q_ref)
    assert_parity(got, ref, what="attention over FP8 pools after the front")
    # consistency with the bf16 pools' front (the oracle's encoder on its stored rows)
    kb, vb, _, _ = _export(kvb)
    kc, ke = ofp8.encode_rows(ofront.bf16_bits_to_f64(kb))
    vc, ve = ofp8.encode_rows(ofront.bf16_bits_to_f64(vb))
    pages, hk, P, _ = kc.shape
    assert np.array_equal(k8, kc), "K codes"
    perm = np.array([4 * ((s % 8) // 2) + 2 * (s // 8) + s % 2 for s in range(16)])
    vt = vc.transpose(0, 1, 3, 2).reshape(pages, hk, d, P // 16, 16)
    vp = np.empty_like(vt)
    vp[..., perm] = vt
    assert np.array_equal(v8, vp.reshape(pages, hk, d, P)), "V codes"
    e = np.stack([ke.reshape(pages, hk, P // 16, 16), ve.reshape(pages, hk, P // 16, 16)], axis=3)
    assert np.array_equal(e8, e.astype(np.int8)), "exponents"
