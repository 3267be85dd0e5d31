"""GPU: FP8 (e4m3) pools.  The stored codes and exponents match the oracle's encoder bit for
bit (after a fill and after appends), and decode attention over an FP8 pool matches the oracle
run on the decoded rows (every decoded value is an exact bf16 value) at the usual bar."""
import numpy as np
import pytest

import oracle
from oracle import fp8
from oracle.embedder import bf16_bits_to_f64
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import (assert_parity, dev_bf16, dev_i32, host_bits, small_case, torch)

pytestmark = pytest.mark.gpu

F32_MAX, F32_MEAN = 3e-3, 3e-4


def _bits_f64(bits):
    return bf16_bits_to_f64(bits)


def _to_bits(x):
    """Input rows: fp64 values to bf16 bits through the generators' own conversion."""
    return wl.f32_to_bf16_bits(np.asarray(x, np.float64).astype(np.float32))


def _decoded(bits):
    """bf16 bits of the rows an FP8 pool holds for these bf16 rows ([..., d] bits)."""
    codes, es = fp8.encode_rows(_bits_f64(bits))
    return fp8.decoded_bf16_bits(codes, es)


# byte of slot s of a chunk within the transposed value rows (ham.h): slots 0, 1, 8, 9, 2, 3, ...
V_SLOT_BYTE = np.array([4 * ((s % 8) // 2) + 2 * (s // 8) + s % 2 for s in range(16)])


def _expected_pools(k_pool_bits, v_pool_bits):
    """Expected FP8 export of an oracle layer's bf16 pools [pages][Hkv][P][d]: K codes, V codes
    transposed per page (a chunk's slots in the documented order), exponents
    [pages][Hkv][P/16][2][16]."""
    kc, ke = fp8.encode_rows(_bits_f64(k_pool_bits))
    vc, ve = fp8.encode_rows(_bits_f64(v_pool_bits))
    pages, hkv, P, d = kc.shape
    e = np.stack([ke.reshape(pages, hkv, P // 16, 16), ve.reshape(pages, hkv, P // 16, 16)], axis=3)
    vt = vc.transpose(0, 1, 3, 2).reshape(pages, hkv, d, P // 16, 16)
    vp = np.empty_like(vt)
    vp[..., V_SLOT_BYTE] = vt
    return kc, np.ascontiguousarray(vp.reshape(pages, hkv, d, P)), e.astype(np.int8)


def fp8_cache(case, layers=1, pos_mode=ham.HAM_POS_SLOT, fill=True):
    w = case.w
    kv = ham.ham_kv_alloc(layers, w.batch, w.n_q_heads, w.n_kv_heads, w.head_dim, w.page_slots,
                          case.max_slots, pos_mode=pos_mode, pool_pages=case.pool_pages,
                          kv_dtype=ham.HAM_KV_E4M3)
    ham.ham_kv_set_page_table(kv, case.page_table)
    if fill:
        for layer in range(layers):
            ham.ham_kv_fill(kv, layer, dev_bf16(case.k), dev_bf16(case.v),
                            dev_i32(case.num_slots), pos=dev_i32(case.slot_pos),
                            ntok=dev_i32(case.slot_ntok))
    return kv


def _export(kv, layer=0):
    k, v, pos, ntok = ham.ham_kv_export(kv, layer)
    e = ham.ham_kv_export_scales(kv, layer)
    return (k.cpu().numpy(), v.cpu().numpy(), e.cpu().numpy(), pos.cpu().numpy(),
            ntok.cpu().numpy())


def _decode(kv, q_bits, f32=False, layer=0):
    t = torch()
    q = dev_bf16(q_bits)
    out = t.full(q.shape, float("nan"), dtype=t.float32 if f32 else t.bfloat16, device="cuda")
    ham.ham_decode_attn_ex(kv, layer, q, out)
    t.cuda.synchronize()
    return out.float().cpu().numpy().astype(np.float64)


def _reference(case):
    """Oracle decode over the decoded rows of the case's cache."""
    oc = oracle.OracleCache.from_case(case, fill=False)
    oc.fill(_decoded(case.k), _decoded(case.v), case.slot_pos, case.slot_ntok, case.num_slots)
    return oc


@pytest.mark.parametrize("page,counts", [(16, (37, 80)), (32, (0, 100, 7)), (128, (255,))])
def test_fill_stores_the_oracle_encoding(page, counts):
    case = small_case(batch=len(counts), hq=32, hkv=8, d=128, page=page, counts=counts, seed=11)
    oc = oracle.OracleCache.from_case(case)
    kv = fp8_cache(case)
    k, v, e, pos, ntok = _export(kv)
    kc, vc, ee = _expected_pools(oc.k_pool, oc.v_pool)
    assert np.array_equal(k, kc), "K codes"
    assert np.array_equal(v, vc), "V codes (transposed)"
    assert np.array_equal(e, ee), "exponents"
    assert np.array_equal(pos, oc.slot_pos) and np.array_equal(ntok, oc.slot_ntok)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_fill_encodes_extreme_row_scales():
    """Rows whose largest magnitude ranges from bf16 subnormals to near the bf16 maximum: the
    exponent clamps at both ends, saturation and signed zeros, bit for bit."""
    case = small_case(batch=2, hq=8, hkv=2, d=128, page=16, counts=(40, 24), seed=12)
    k = _bits_f64(case.k)
    v = _bits_f64(case.v)
    tops = 2.0 ** np.array([-133, -130, -126, -124, -117, -116, -60, 0, 30, 90, 118, 126, 127])
    for i, top in enumerate(tops):
        b, j = i % 2, 3 * i
        k[b, j] *= top / np.abs(k[b, j]).max(axis=-1, keepdims=True)
        v[b, j + 1] *= top / np.abs(v[b, j + 1]).max(axis=-1, keepdims=True)
    k[0, 1, 0, :] = 0.0                       # a zero row
    v[1, 2, 1, :8] = -0.0                     # negative zeros
    k[1, 4, 0, :4] = -(2.0 ** -20) * k[1, 4, 0, :4] / np.abs(k[1, 4, 0, :4]).max()  # to -0 codes
    case.k[...] = _to_bits(k)
    case.v[...] = _to_bits(v)
    oc = oracle.OracleCache.from_case(case)
    kv = fp8_cache(case)
    kk, vv, e, _, _ = _export(kv)
    kc, vc, ee = _expected_pools(oc.k_pool, oc.v_pool)
    assert np.array_equal(e, ee), "exponents"
    assert np.array_equal(kk, kc), "K codes"
    assert np.array_equal(vv, vc), "V codes"


@pytest.mark.parametrize("pos_mode", [ham.HAM_POS_SLOT, ham.HAM_POS_TOKEN])
@pytest.mark.parametrize("hq,hkv", [(32, 8), (8, 8), (32, 16)])
def test_append_stores_the_oracle_encoding(pos_mode, hq, hkv):
    """The rotated bf16 key (as a bf16 cache stores it) and the value, encoded bit for bit; q
    turned in place as for a bf16 cache; several macro-steps crossing a page edge."""
    case = small_case(batch=3, hq=hq, hkv=hkv, d=128, page=16, counts=(15, 16, 200), seed=13,
                      extra_slots=8)
    oc = oracle.OracleCache.from_case(case)
    kv = fp8_cache(case, pos_mode=pos_mode)
    q_host = case.q.copy()
    q_dev = dev_bf16(case.q)
    rng = wl.rng_for(13, 50)
    for step in range(3):
        k_new = wl.normal_bf16(rng, case.k_new.shape)
        v_new = wl.normal_bf16(rng, case.v_new.shape)
        ntok = wl.ntok_capped_geometric(rng, (case.w.batch,))
        assert oc.append(k_new, v_new, ntok, q_inout=q_host, pos_mode=pos_mode) == 0
        ham.ham_kv_append(kv, 0, q_dev, dev_bf16(k_new), dev_bf16(v_new), None, dev_i32(ntok))
    k, v, e, pos, ntok_arr = _export(kv)
    kc, vc, ee = _expected_pools(oc.k_pool, oc.v_pool)
    assert np.array_equal(e, ee), "exponents"
    assert np.array_equal(k, kc), "K codes of the rotated keys"
    assert np.array_equal(v, vc), "V codes"
    assert np.array_equal(pos, oc.slot_pos) and np.array_equal(ntok_arr, oc.slot_ntok)
    assert np.array_equal(host_bits(q_dev), q_host)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


@pytest.mark.parametrize("hq,hkv,page,counts,scale", [
    (32, 8, 16, (37, 80), 1.0),                       # ragged tails inside a chunk
    (32, 8, 16, (1, 100, 1000), 1.0 / np.sqrt(128)),
    (32, 8, 16, (0, 17, 0, 4097), 1.0),               # empty sequences
    (32, 8, 32, (513, 2047), 1.0),
    (32, 8, 128, (256, 3), 1.0),
    (8, 8, 16, (300, 33), 1.0),                       # group 1
    (16, 8, 16, (300, 33), 1.0),                      # group 2
    (64, 8, 16, (300, 33), 1.0),                      # group 8 (32 product columns)
    (24, 8, 16, (129, 64), 1.0),                      # group 3
    (40, 8, 16, (1000, 129), 1.0),                    # group 5: every one of 16 columns in use
    (48, 8, 32, (700, 15), 1.0),                      # group 6: 32 columns, 18 in use
])
def test_decode_over_fp8_matches_oracle(hq, hkv, page, counts, scale):
    case = small_case(batch=len(counts), hq=hq, hkv=hkv, d=128, page=page, counts=counts,
                      scale=scale, seed=sum(counts) % 89 + 3)
    ref = _reference(case).decode_attn(case.q)
    kv = fp8_cache(case)
    out16 = _decode(kv, case.q)
    out32 = _decode(kv, case.q, f32=True)
    assert_parity(out16, ref, what="fp8 pool, bf16 out")
    assert_parity(out32, ref, max_abs=F32_MAX, mean_abs=F32_MEAN, what="fp8 pool, f32 out")
    for b, n in enumerate(counts):
        if n == 0:
            assert np.all(out16[b] == 0) and np.all(out32[b] == 0)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def test_decode_over_fp8_rows_of_very_different_scales():
    """Value rows whose scales differ by up to 2^40 across a sequence (the running value
    exponent is raised mid-segment and O rescaled), keys of mixed scales, and queries whose
    heads range from 2^-30 to 2^20."""
    case = small_case(batch=3, hq=32, hkv=8, d=128, page=16, counts=(700, 90, 1500), seed=31)
    rng = wl.rng_for(31, 7)
    k = _bits_f64(case.k)
    v = _bits_f64(case.v)
    L = k.shape[1]
    vs = 2.0 ** rng.integers(-20, 21, size=(k.shape[0], L, 1, 1))
    ks = 2.0 ** rng.integers(-6, 4, size=(k.shape[0], L, 1, 1))
    case.k[...] = _to_bits(k * ks * 0.25)
    case.v[...] = _to_bits(v * vs)
    q = _bits_f64(case.q)
    qs = 2.0 ** rng.integers(-30, 21, size=(q.shape[0], q.shape[1], 1))
    qs[:, ::5] = 1.0
    case.q[...] = _to_bits(np.clip(q * qs, -1e30, 1e30) * 2.0 ** -10)
    ref = _reference(case).decode_attn(case.q)
    kv = fp8_cache(case)
    out32 = _decode(kv, case.q, f32=True)
    # relative to each output row's size (the values span 2^40)
    scale = np.maximum(np.abs(ref).max(axis=-1, keepdims=True), 1e-30)
    err = np.abs(out32 - ref) / scale
    assert np.all(np.isfinite(out32))
    assert err.max() <= 3e-3, f"max relative {err.max():.3e}"
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


@pytest.mark.parametrize("ctas", [1, 7, 64, 600])
def test_fp8_split_count_invariance(ctas):
    case = small_case(batch=4, hq=32, hkv=8, d=128, page=16, counts=(1, 300, 2000, 45), seed=41)
    ref = _reference(case).decode_attn(case.q)
    kv = fp8_cache(case)
    ham.ham_kv_set_attn_ctas(kv, ctas)
    out = _decode(kv, case.q, f32=True)
    assert_parity(out, ref, max_abs=F32_MAX, mean_abs=F32_MEAN, what=f"{ctas} CTAs")


def test_fp8_append_then_decode():
    """Macro-steps through ham_kv_append then ham_decode_attn on an FP8 cache agree with the
    oracle's append followed by decoding over the decoded rows."""
    case = small_case(batch=3, hq=32, hkv=8, d=128, page=16, counts=(31, 200, 64), seed=51,
                      extra_slots=8)
    oc = oracle.OracleCache.from_case(case)
    kv = fp8_cache(case)
    q_host = case.q.copy()
    q_dev = dev_bf16(case.q)
    rng = wl.rng_for(51, 9)
    for step in range(4):
        k_new = wl.normal_bf16(rng, case.k_new.shape)
        v_new = wl.normal_bf16(rng, case.v_new.shape)
        ntok = wl.ntok_capped_geometric(rng, (case.w.batch,))
        assert oc.append(k_new, v_new, ntok, q_inout=q_host) == 0
        ham.ham_kv_append(kv, 0, q_dev, dev_bf16(k_new), dev_bf16(v_new), None, dev_i32(ntok))
    # the oracle's bf16 pools, decoded through the FP8 format, are the reference cache
    ref_cache = oracle.OracleCache.from_case(case, fill=False)
    ref_cache.k_pool[...] = _decoded(oc.k_pool)
    ref_cache.v_pool[...] = _decoded(oc.v_pool)
    ref_cache.slot_pos[...] = oc.slot_pos
    ref_cache.slot_ntok[...] = oc.slot_ntok
    ref_cache.num_slots[...] = oc.num_slots
    ref_cache.num_tokens[...] = oc.num_tokens
    ref = ref_cache.decode_attn(q_host)
    out = _decode(kv, q_host)
    assert_parity(out, ref, what="append then decode")
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


def _decoded_cache(case, oc):
    """An oracle cache holding the decoded rows of `oc`'s bf16 pools (the rows an FP8 cache
    holds after the same fills and appends)."""
    ref = oracle.OracleCache.from_case(case, fill=False)
    ref.k_pool[...] = _decoded(oc.k_pool)
    ref.v_pool[...] = _decoded(oc.v_pool)
    ref.slot_pos[...] = oc.slot_pos
    ref.slot_ntok[...] = oc.slot_ntok
    ref.num_slots[...] = oc.num_slots
    ref.num_tokens[...] = oc.num_tokens
    return ref


Q_ROT_UNWRITTEN = 0x7FC1  # a bf16 NaN pattern no rotation produces


@pytest.mark.parametrize("pos_mode", [ham.HAM_POS_SLOT, ham.HAM_POS_TOKEN])
@pytest.mark.parametrize("hq,hkv,page,counts", [
    (32, 8, 16, (15, 16, 0, 47)),          # new slot ends chunk 0 / opens chunk 1 / first
    (32, 8, 32, (31, 200, 5)),             # page edge
    (8, 8, 16, (1, 64)),                   # group 1
    (64, 8, 128, (127, 300)),              # group 8
    (40, 8, 16, (127, 128, 129)),          # group 5; one slot short of / exactly / past a tile
])
def test_fp8_step_matches_oracle(pos_mode, hq, hkv, page, counts):
    """ham_decode_step on an FP8 cache: the stored codes and exponents, the counters and q_rot
    bit for bit against the oracle's append (then encoded); the output against the oracle's
    attention over the decoded rows of all n + 1 slots.  q is never written."""
    case = small_case(batch=len(counts), hq=hq, hkv=hkv, d=128, page=page, counts=counts,
                      seed=71, extra_slots=8)
    oc = oracle.OracleCache.from_case(case)
    kv = fp8_cache(case, pos_mode=pos_mode)
    t = torch()
    q = case.q.copy()
    rng = wl.rng_for(71, 60)
    for step in range(3):
        k_new = wl.normal_bf16(rng, case.k_new.shape)
        v_new = wl.normal_bf16(rng, case.v_new.shape)
        ntok = wl.ntok_capped_geometric(rng, (case.w.batch,))
        q_ref = q.copy()
        assert oc.append(k_new, v_new, ntok, q_inout=q_ref, pos_mode=pos_mode) == 0
        ref = _decoded_cache(case, oc).decode_attn(q_ref)
        q_dev = dev_bf16(q)
        q_rot = dev_bf16(np.full(q.shape, Q_ROT_UNWRITTEN, np.uint16))
        out = t.full(q_dev.shape, float("nan"), dtype=t.float32, device="cuda")
        ham.ham_decode_step(kv, 0, q_dev, dev_bf16(k_new), dev_bf16(v_new), None, dev_i32(ntok),
                            out, q_rot=q_rot)
        t.cuda.synchronize()
        assert np.array_equal(host_bits(q_dev), q), "q was written"
        assert np.array_equal(host_bits(q_rot), q_ref), f"q_rot, step {step}"
        got = out.float().cpu().numpy().astype(np.float64)
        assert_parity(got, ref, what=f"fp8 step {step}")
    k, v, e, pos, ntok_arr = _export(kv)
    kc, vc, ee = _expected_pools(oc.k_pool, oc.v_pool)
    assert np.array_equal(e, ee), "exponents"
    assert np.array_equal(k, kc), "K codes"
    assert np.array_equal(v, vc), "V codes"
    assert np.array_equal(pos, oc.slot_pos) and np.array_equal(ntok_arr, oc.slot_ntok)
    slots, tokens = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, oc.num_slots) and np.array_equal(tokens, oc.num_tokens)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE


@pytest.mark.parametrize("batch", [3, 200])  # early and late combine modes
def test_fp8_step_equals_append_then_decode(batch):
    """The fused step and ham_kv_append + ham_decode_attn on two FP8 caches from the same fill:
    the same stored bits and counters, outputs within the bar of each other."""
    rng = np.random.default_rng(batch)
    counts = tuple(int(c) for c in rng.integers(0, 150, size=batch))
    case = small_case(batch=batch, hq=32, hkv=8, d=128, page=16, counts=counts, seed=81,
                      extra_slots=4)
    a, b = fp8_cache(case), fp8_cache(case)
    t = torch()
    k_new, v_new = dev_bf16(case.k_new), dev_bf16(case.v_new)
    ntok = dev_i32(case.ntok_new)
    q1 = dev_bf16(case.q)
    out1 = t.full(q1.shape, float("nan"), dtype=t.float32, device="cuda")
    ham.ham_decode_step(a, 0, q1, k_new, v_new, None, ntok, out1)
    q2 = dev_bf16(case.q)
    out2 = t.full(q2.shape, float("nan"), dtype=t.float32, device="cuda")
    ham.ham_kv_append(b, 0, q2, k_new, v_new, None, ntok)
    ham.ham_decode_attn_ex(b, 0, q2, out2)
    t.cuda.synchronize()
    ea, eb = _export(a), _export(b)
    for x, y, what in zip(ea, eb, ("K codes", "V codes", "exponents", "pos", "ntok")):
        assert np.array_equal(x, y), what
    o1 = out1.cpu().numpy().astype(np.float64)
    o2 = out2.cpu().numpy().astype(np.float64)
    assert_parity(o1, o2, what="step against append + decode")
    assert ham.ham_kv_status(a) == ham.HAM_DEVERR_NONE and ham.ham_kv_status(b) == ham.HAM_DEVERR_NONE


def test_fp8_unsupported_calls_are_refused():
    case = small_case(batch=2, hq=8, hkv=2, d=128, page=16, counts=(5, 6), seed=61)
    kv = fp8_cache(case)
    t = torch()
    q = dev_bf16(case.q)
    out = t.empty_like(q)
    with pytest.raises(ham.HamError) as e:
        ham.ham_prefill(kv, 0, q, dev_bf16(case.k_new), dev_bf16(case.v_new),
                        dev_i32(np.array([0, 1, 2], np.int32)), out)
    assert e.value.status == ham.HAM_EUNSUPPORTED
    with pytest.raises(ham.HamError) as e:
        ham.ham_kv_alloc(1, 2, 8, 2, 64, 16, 32, kv_dtype=ham.HAM_KV_E4M3)
    assert e.value.status == ham.HAM_EUNSUPPORTED
    slots, _ = ham.ham_slot_lengths(kv)
    assert list(slots) == [5, 6]


# ---------------------------------------------------------------------------------------
# full size, in the bench's launch configuration (default CTA count)
# ---------------------------------------------------------------------------------------

FULL_SIZE_PAGES = 16   # pages of the checked sequence whose codes are compared


def _full_size_reference(case, b):
    """Oracle attention with sequence b's rows decoded through the FP8 format (the other
    sequences' rows are left as bf16: their outputs are not compared, and the oracle's encoder
    is brute force, about 10 s per 4M elements)."""
    kd, vd = case.k.copy(), case.v.copy()
    kd[b], vd[b] = _decoded(case.k[b]), _decoded(case.v[b])
    ref = oracle.OracleCache.from_case(case, fill=False)
    ref.fill(kd, vd, case.slot_pos, case.slot_ntok, case.num_slots)
    return ref.decode_attn(case.q)


def _full_size_pages(case, b):
    """A spread of the pages sequence b uses."""
    used = -(-int(case.num_slots[b]) // case.w.page_slots)
    idx = np.unique(np.linspace(0, used - 1, FULL_SIZE_PAGES).round().astype(np.int64))
    return case.page_table[b, idx].astype(np.int64)


@pytest.mark.parametrize("w", [wl.C1_LLAMA8B, wl.C1_LLAMA8B_S8K], ids=lambda w: w.name)
def test_fp8_full_size_workloads(w):
    """The bench's Llama-8B layer at 4096 and 8192 slots over an FP8 pool: every output
    finite, the last sequence's attention (all 32 heads) against the oracle on its decoded rows
    at the usual bar, and the codes and exponents of a spread of its pages bit for bit."""
    case = wl.make_case(w, extra_slots=4)
    kv = fp8_cache(case)
    out = _decode(kv, case.q)
    assert np.all(np.isfinite(out))
    b = w.batch - 1
    ref = _full_size_reference(case, b)
    assert_parity(out[b], ref[b], what=f"{w.name}, sequence {b}")
    pages = _full_size_pages(case, b)
    raw = oracle.OracleCache.from_case(case)
    kc, vc, ee = _expected_pools(raw.k_pool[pages], raw.v_pool[pages])
    k, v, e, pos, ntok = _export(kv)
    assert np.array_equal(k[pages], kc), "K codes"
    assert np.array_equal(v[pages], vc), "V codes (transposed)"
    assert np.array_equal(e[pages], ee), "exponents"
    assert np.array_equal(pos, raw.slot_pos) and np.array_equal(ntok, raw.slot_ntok)
    slots, _ = ham.ham_slot_lengths(kv)
    assert np.array_equal(slots, case.num_slots)
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    ham.ham_kv_free(kv)
