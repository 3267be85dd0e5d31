"""Pins of the CPU oracle to things other than itself (no GPU needed).

Each test checks the oracle against a definition, a library routine, a closed form or an
invariant, chosen so that a dropped term, a wrong sign or index, or a transposed operand
in the oracle fails at least one of them.
"""
import math

import numpy as np
import pytest
import torch

from paper_2505_20438_gb300 import workload as wl

pytestmark = pytest.mark.usefixtures("oracle_lib")


def _oracle():
    import oracle
    return oracle


# ---------------------------------------------------------------------------
# bf16 rounding (the one place floating point decides stored bits)
# ---------------------------------------------------------------------------

def _bf16_value(bits):
    return float(wl.bf16_bits_to_f32(np.array([bits], np.uint16))[0])


@pytest.mark.parametrize("x,bits", [
    (1.0, 0x3F80),
    (1.0 + 2.0 ** -8, 0x3F80),                   # tie -> even (1.0)
    (1.0 + 3 * 2.0 ** -8, 0x3F82),               # tie -> even (1 + 2^-6)
    (1.0 + 2.0 ** -8 + 2.0 ** -40, 0x3F81),      # just above the tie: no double rounding
    (-(1.0 + 2.0 ** -8 + 2.0 ** -40), 0xBF81),
    (0.0, 0x0000), (-0.0, 0x8000),
    (2.0 ** -133, 0x0001),                       # smallest bf16 subnormal
    (2.0 ** -134, 0x0000),                       # half of it: tie -> even (0)
    (1.5 * 2.0 ** -133, 0x0002),                 # tie -> even (2 * 2^-133)
    (3.3895313892515355e38, 0x7F7F),             # largest finite bf16
    (2.0 ** 128 * (1 - 2.0 ** -9), 0x7F80),      # rounds past the largest: infinity
    (float("inf"), 0x7F80), (float("-inf"), 0xFF80),
])
def test_f64_to_bf16_exact_cases(x, bits):
    assert int(_oracle().f64_to_bf16(np.array([x]))[0]) == bits


def test_f64_to_bf16_is_nearest_ties_even():
    """Brute force: the result is one of the two neighbouring bf16 values, the nearer one,
    and the even one on an exact tie."""
    rng = np.random.default_rng(11)
    xs = np.concatenate([rng.standard_normal(3000) * 10.0 ** rng.integers(-30, 30, 3000),
                         # exact ties between bf16 neighbours
                         (rng.integers(1 << 7, 1 << 8, 500) + 0.5) * 2.0 ** -7])
    got = _oracle().f64_to_bf16(xs)
    for x, b in zip(xs, got):
        f = np.float32(x)
        u = int(np.array([f], np.float32).view(np.uint32)[0]) & 0xFFFF0000
        lo = np.array([u], np.uint32).view(np.float32)[0]          # toward zero
        hi_bits = (u + 0x10000) & 0xFFFFFFFF
        hi = np.array([hi_bits], np.uint32).view(np.float32)[0]    # away from zero
        cands = [(abs(x - float(lo)), u >> 16), (abs(x - float(hi)), hi_bits >> 16)]
        # float32(x) may itself have rounded across a bf16 neighbour; widen by one step
        lo2_bits = (u - 0x10000) & 0xFFFFFFFF
        lo2 = np.array([lo2_bits], np.uint32).view(np.float32)[0]
        cands.append((abs(x - float(lo2)), lo2_bits >> 16))
        best = min(c[0] for c in cands)
        winners = {c[1] for c in cands if c[0] == best}
        assert int(b) in winners, (x, hex(int(b)), [hex(w) for w in winners])
        if len(winners) == 2:
            assert int(b) % 2 == 0


def test_bf16_to_f64_matches_torch():
    bits = np.arange(0, 1 << 16, 7, dtype=np.uint16)
    bits = bits[(bits & 0x7F80) != 0x7F80]      # finite only
    ours = _oracle().bf16_to_f64(bits)
    ref = torch.from_numpy(bits.astype(np.int16)).view(torch.bfloat16).double().numpy()
    assert np.array_equal(ours, ref)


# ---------------------------------------------------------------------------
# RoPE
# ---------------------------------------------------------------------------

def _rope_complex(x_bits, pos, base):
    """RoPE written as complex rotation: z_i = x_i + i x_{i+d/2}, z_i * exp(i pos w_i)."""
    x = wl.bf16_bits_to_f32(x_bits).astype(np.float64)
    d = x.shape[-1]
    half = d // 2
    w = base ** (-(np.arange(half) * 2.0) / d)
    z = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * pos * w)
    return np.concatenate([z.real, z.imag], axis=-1)


@pytest.mark.parametrize("d", [2, 8, 64, 128])
@pytest.mark.parametrize("pos", [0, 1, 7, 255, 4096, 262143])
def test_rope_matches_complex_rotation(d, pos):
    rng = wl.rng_for(5, d)
    x = wl.normal_bf16(rng, (3, d))
    got = np.stack([_oracle().rope_f64(x[r], pos) for r in range(3)])
    ref = _rope_complex(x, pos, 10000.0)
    # different sin/cos implementations; arguments up to 2.6e5 rad
    assert np.allclose(got, ref, rtol=0, atol=1e-12 * max(1.0, pos) ** 0.5 + 1e-13)


def test_rope_hand_values():
    # d = 2: one pair with frequency 1, (1, 0) -> (cos p, sin p)
    one = wl.f32_to_bf16_bits(np.array([1.0, 0.0], np.float32))
    assert np.allclose(_oracle().rope_f64(one, 1), [math.cos(1.0), math.sin(1.0)], atol=1e-15)
    # d = 4, base 10000: second pair turns at 10000^(-1/2) = 0.01 rad per position
    x = wl.f32_to_bf16_bits(np.array([0.0, 1.0, 0.0, 0.0], np.float32))
    y = _oracle().rope_f64(x, 100, 10000.0)
    assert np.allclose(y, [0.0, math.cos(1.0), 0.0, math.sin(1.0)], atol=1e-14)


def test_rope_identity_at_zero_and_norm_preserved():
    rng = wl.rng_for(6)
    x = wl.normal_bf16(rng, (4, 128))
    assert np.array_equal(_oracle().rope_bf16(x, 0), x)          # bit-exact identity
    y = np.stack([_oracle().rope_f64(x[r], 12345) for r in range(4)])
    xf = wl.bf16_bits_to_f32(x).astype(np.float64)
    pair_in = xf[:, :64] ** 2 + xf[:, 64:] ** 2
    pair_out = y[:, :64] ** 2 + y[:, 64:] ** 2
    assert np.allclose(pair_in, pair_out, rtol=1e-13)


def test_rope_relative_position():
    """<R(p1) q, R(p2) k> depends on p1 - p2 only."""
    rng = wl.rng_for(7)
    q, k = wl.normal_bf16(rng, (2, 128))
    o = _oracle()
    a = np.dot(o.rope_f64(q, 9), o.rope_f64(k, 4))
    b = np.dot(o.rope_f64(q, 100009), o.rope_f64(k, 100004))
    c = np.dot(o.rope_f64(q, 9), o.rope_f64(k, 5))
    assert abs(a - b) < 1e-9
    assert abs(a - c) > 1e-6


# ---------------------------------------------------------------------------
# attention over the slot list
# ---------------------------------------------------------------------------

def _small_case(seed=0, batch=2, hq=8, hkv=2, d=64, page=16, counts=(37, 80), scale=1.0,
                scatter=True, pool_factor=1.5, extra_slots=1):
    w = wl.Workload("pin", batch=batch, n_q_heads=hq, n_kv_heads=hkv, head_dim=d,
                    page_slots=page, layers=1, value_scale=scale, seed=seed,
                    pool_factor=pool_factor, scatter_pages=scatter)
    return wl.make_case(w, num_slots=np.array(counts, np.int32), extra_slots=extra_slots)


def _dense_reference(case):
    """Dense softmax(q K^T / sqrt(d)) V in numpy fp64 from the LOGICAL arrays."""
    w = case.w
    G = w.group
    q = wl.bf16_bits_to_f32(case.q).astype(np.float64)
    k = wl.bf16_bits_to_f32(case.k).astype(np.float64)
    v = wl.bf16_bits_to_f32(case.v).astype(np.float64)
    out = np.zeros_like(q)
    for b in range(w.batch):
        L = int(case.num_slots[b])
        for h in range(w.n_q_heads):
            if L == 0:
                continue
            s = k[b, :L, h // G, :] @ q[b, h] / math.sqrt(w.head_dim)
            p = np.exp(s - s.max())
            out[b, h] = (p / p.sum()) @ v[b, :L, h // G, :]
    return out


def test_attention_matches_dense_brute_force():
    o = _oracle()
    for seed, counts in [(0, (37, 80)), (1, (1, 300)), (2, (16, 17))]:
        case = _small_case(seed=seed, counts=counts)
        oc = o.OracleCache.from_case(case)
        got = oc.decode_attn(case.q)
        ref = _dense_reference(case)
        assert np.allclose(got, ref, rtol=1e-12, atol=1e-13)


def test_attention_matches_torch_sdpa_gqa():
    """One token per slot (ntok = 1) is standard causal GQA decode (Sec. 3.4): the last
    row of torch's causal SDPA over the same keys equals the oracle's decode step."""
    o = _oracle()
    T, hq, hkv, d = 200, 8, 2, 64
    case = _small_case(seed=3, batch=1, hq=hq, hkv=hkv, d=d, counts=(T,))
    oc = o.OracleCache.from_case(case)
    got = oc.decode_attn(case.q)[0]
    # dense token sequence: keys/values of tokens 0..T-1; queries of earlier tokens are
    # arbitrary (causal mask), the last query is the decode query
    k = torch.from_numpy(wl.bf16_bits_to_f32(case.k[0]).astype(np.float64)).permute(1, 0, 2)
    v = torch.from_numpy(wl.bf16_bits_to_f32(case.v[0]).astype(np.float64)).permute(1, 0, 2)
    qs = torch.randn(hq, T, d, dtype=torch.float64, generator=torch.Generator().manual_seed(0))
    qs[:, -1, :] = torch.from_numpy(wl.bf16_bits_to_f32(case.q[0]).astype(np.float64))
    ref = torch.nn.functional.scaled_dot_product_attention(
        qs[None], k[None], v[None], is_causal=True, enable_gqa=True)[0, :, -1, :].numpy()
    assert np.allclose(got, ref, rtol=1e-10, atol=1e-12)


def test_weights_sum_to_one_and_reproduce_output():
    o = _oracle()
    case = _small_case(seed=4, counts=(129, 64))
    oc = o.OracleCache.from_case(case)
    out = oc.decode_attn(case.q)
    G = case.w.group
    for b in range(2):
        for h in range(8):
            w = oc.attn_weights(case.q, b, h)
            assert np.all(w >= 0)
            assert abs(w.sum() - 1.0) <= 1e-12
            _, v = oc.gather(b, h // G)
            assert np.allclose(w @ v, out[b, h], rtol=1e-12, atol=1e-14)


def test_output_independent_of_paging():
    """Same logical slots under different page tables and pool sizes: bit-identical."""
    o = _oracle()
    a = _small_case(seed=5, counts=(100, 33), page=16, scatter=False, pool_factor=1.0)
    b = _small_case(seed=5, counts=(100, 33), page=16, scatter=True, pool_factor=3.0)
    c = _small_case(seed=5, counts=(100, 33), page=32, scatter=True, pool_factor=2.0)
    assert np.array_equal(a.k, b.k) and not np.array_equal(a.page_table, b.page_table[:, :7])
    outs = [o.OracleCache.from_case(x).decode_attn(x.q) for x in (a, b, c)]
    assert np.array_equal(outs[0], outs[1]) and np.array_equal(outs[0], outs[2])


def test_special_cases():
    o = _oracle()
    # one slot: output is V_0 exactly
    case = _small_case(seed=6, counts=(1, 1))
    out = o.OracleCache.from_case(case).decode_attn(case.q)
    v0 = wl.bf16_bits_to_f32(case.v[:, 0]).astype(np.float64)
    for h in range(8):
        assert np.array_equal(out[:, h], v0[:, h // 4])
    # all keys equal: uniform weights, output is the mean of V
    case = _small_case(seed=7, counts=(50, 9))
    case.k[:] = case.k[0, 0, 0]
    out = o.OracleCache.from_case(case).decode_attn(case.q)
    v = wl.bf16_bits_to_f32(case.v).astype(np.float64)
    for b, L in enumerate((50, 9)):
        for h in range(8):
            assert np.allclose(out[b, h], v[b, :L, h // 4].mean(axis=0), rtol=1e-12,
                               atol=1e-14)
    # a planted key aligned with q wins: output is that slot's V
    case = _small_case(seed=8, batch=1, counts=(300,), scale=0.05)
    q = wl.bf16_bits_to_f32(case.q[0, 0]).astype(np.float64)
    planted = wl.f32_to_bf16_bits((q * (30.0 * 8.0 / (q @ q))).astype(np.float32))
    case.k[0, 123, 0] = planted
    out = o.OracleCache.from_case(case).decode_attn(case.q)
    v = wl.bf16_bits_to_f32(case.v[0, 123, 0]).astype(np.float64)
    assert np.allclose(out[0, 0], v, atol=1e-8)
    # empty sequence: output 0
    case = _small_case(seed=9, counts=(0, 5))
    out = o.OracleCache.from_case(case).decode_attn(case.q)
    assert np.array_equal(out[0], np.zeros_like(out[0])) and np.abs(out[1]).sum() > 0


def test_heads_map_to_groups_consecutively():
    """Query head h reads KV head h // G: changing KV head 1 moves only heads 4..7."""
    o = _oracle()
    case = _small_case(seed=10, batch=1, counts=(40,))
    before = o.OracleCache.from_case(case).decode_attn(case.q)
    case.v[0, :, 1] = case.v[0, ::-1, 1]
    after = o.OracleCache.from_case(case).decode_attn(case.q)
    assert np.array_equal(before[0, :4], after[0, :4])
    assert not np.allclose(before[0, 4:], after[0, 4:])


# ---------------------------------------------------------------------------
# append (one slot per macro-step, Sec. 3.1) and the ntok = 1 equivalence chain
# ---------------------------------------------------------------------------

def test_append_writes_only_its_slot_and_metadata():
    o = _oracle()
    case = _small_case(seed=11, counts=(31, 64), page=16)
    oc = o.OracleCache.from_case(case)
    k0, v0 = oc.k_pool.copy(), oc.v_pool.copy()
    pos0, nt0 = oc.slot_pos.copy(), oc.slot_ntok.copy()
    tokens0 = oc.num_tokens.copy()
    assert oc.append(case.k_new, case.v_new, case.ntok_new) == 0
    assert list(oc.num_slots) == [32, 65]
    assert list(oc.num_tokens) == list(tokens0 + case.ntok_new)
    changed = np.argwhere((oc.k_pool != k0).any(-1) | (oc.v_pool != v0).any(-1))
    for b, n in enumerate((31, 64)):
        page, row = case.page_table[b, n // 16], n % 16
        assert oc.slot_pos[page, row] == n and oc.slot_ntok[page, row] == case.ntok_new[b]
        assert np.array_equal(oc.v_pool[page, :, row], case.v_new[b])
        assert np.array_equal(oc.k_pool[page, :, row], o.rope_bf16(case.k_new[b], n))
    rows = {(int(p), int(r)) for p, _, r in changed}
    assert rows <= {(int(case.page_table[b, n // 16]), n % 16) for b, n in enumerate((31, 64))}
    meta = np.argwhere((oc.slot_pos != pos0) | (oc.slot_ntok != nt0))
    assert len(meta) <= 2


def test_append_positions_and_capacity():
    o = _oracle()
    case = _small_case(seed=12, batch=1, counts=(5,), extra_slots=2)
    oc = o.OracleCache.from_case(case)
    toks = int(oc.num_tokens[0])
    q = case.q.copy()
    assert oc.append(case.k_new, case.v_new, np.array([3], np.int32), q_inout=q,
                     pos_mode=o.POS_TOKEN) == 0
    page, row = case.page_table[0, 0], 5
    assert oc.slot_pos[page, row] == toks                       # first token of the group
    assert np.array_equal(q, o.rope_bf16(case.q, toks))         # q turned at the same position
    assert oc.append(case.k_new, case.v_new, np.array([1], np.int32), pos=np.array([77], np.int32)) == 0
    assert oc.slot_pos[page, 6] == 77
    oc.num_slots[0] = case.max_slots                           # full sequence
    assert oc.append(case.k_new, case.v_new, np.array([1], np.int32)) == o.ECAPACITY
    assert oc.append(case.k_new, case.v_new, np.array([0], np.int32)) == o.EINVAL


def test_token_by_token_appends_equal_causal_decode():
    """Appending T single-token slots at positions 0..T-1 through the oracle's own RoPE and
    then decoding equals causal SDPA over keys rotated by the complex-exponential RoPE
    (independent of the oracle's rotation code)."""
    o = _oracle()
    T, hq, hkv, d = 64, 8, 2, 64
    w = wl.Workload("chain", batch=1, n_q_heads=hq, n_kv_heads=hkv, head_dim=d,
                    page_slots=16, layers=1, seed=13, pool_factor=2.0)
    case = wl.make_case(w, num_slots=np.array([0], np.int32), extra_slots=T + 1)
    oc = o.OracleCache.from_case(case)
    rng = wl.rng_for(13, 99)
    ks = wl.normal_bf16(rng, (T, hkv, d))
    vs = wl.normal_bf16(rng, (T, hkv, d))
    for t in range(T):
        assert oc.append(ks[t][None], vs[t][None], np.array([1], np.int32)) == 0
    q = wl.normal_bf16(rng, (1, hq, d))
    q_rot = o.rope_bf16(q, T - 1)                 # query of the last token
    got = oc.decode_attn(q_rot)[0]
    k_ref = np.stack([_rope_complex(ks[t], t, 10000.0) for t in range(T)])   # [T][hkv][d]
    kt = torch.from_numpy(k_ref).permute(1, 0, 2)
    vt = torch.from_numpy(wl.bf16_bits_to_f32(vs).astype(np.float64)).permute(1, 0, 2)
    qs = torch.zeros(hq, T, d, dtype=torch.float64)
    qs[:, -1] = torch.from_numpy(wl.bf16_bits_to_f32(q_rot[0]).astype(np.float64))
    ref = torch.nn.functional.scaled_dot_product_attention(
        qs[None], kt[None], vt[None], is_causal=True, enable_gqa=True)[0, :, -1].numpy()
    # the stored keys are bf16-rounded rotations; the reference keeps them in fp64
    assert np.allclose(got, ref, atol=2e-2) and np.abs(got - ref).mean() < 2e-3


def test_large_logits_stay_finite():
    """Scores past exp()'s fp64 range (about 709.8): the softmax is shift-invariant, so the
    output is still the planted slot's V and the weights still sum to 1."""
    o = _oracle()
    case = _small_case(seed=14, batch=1, counts=(64,), scale=0.05)
    q = wl.bf16_bits_to_f32(case.q[0, 0]).astype(np.float64)
    for j, score in ((10, 900.0), (20, 880.0)):
        case.k[0, j, 0] = wl.f32_to_bf16_bits((q * (score * 8.0 / (q @ q))).astype(np.float32))
    oc = o.OracleCache.from_case(case)
    out = oc.decode_attn(case.q)
    w = oc.attn_weights(case.q, 0, 0)
    assert np.all(np.isfinite(out)) and abs(w.sum() - 1.0) < 1e-12
    v = wl.bf16_bits_to_f32(case.v[0, 10, 0]).astype(np.float64)
    assert np.allclose(out[0, 0], v, atol=1e-6)


def test_tiny_workload_regression_fixture():
    """The oracle still reproduces the stored fixture of the tiny workload's step (guards
    against unintended changes of the oracle or of the input generator)."""
    import os
    import sys
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    sys.path.insert(0, here)
    try:
        import make_golden
    finally:
        sys.path.remove(here)
    out, oc = make_golden.tiny_step()
    lines = open(os.path.join(here, "tiny_step_oracle.txt")).read().splitlines()
    meta = [l for l in lines if l.startswith("# num_slots")][0].split()
    assert int(oc.num_slots[0]) == int(meta[2]) == 256 and int(oc.num_tokens[0]) == int(meta[4])
    ref = np.array([float(l) for l in lines if not l.startswith("#")])
    assert np.array_equal(out.reshape(-1), ref)
