"""Pins of the FP8 (e4m3) row format of the oracle (oracle/fp8.py) to things other than itself.

Decoding is pinned by torch's float8_e4m3fn type (an independent implementation) on all 256
codes and by values the format's definition fixes; encoding by torch on the whole finite range
(every grid value, every midpoint between neighbours, zeros of both signs) and by brute force
against the grid (nearest, ties to the even code); the row scale by its defining inequalities;
the claim that decoded values are exact bf16 values by the C oracle's bf16 rounding.
"""
import numpy as np
import pytest

from paper_2505_20438_gb300 import workload as wl

pytestmark = pytest.mark.usefixtures("oracle_lib")


def _fp8():
    from oracle import fp8
    return fp8


def test_decode_matches_torch_on_every_code():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8_e4m3fn")
    codes = np.arange(256, dtype=np.uint8)
    mine = _fp8().e4m3_value(codes)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).float().numpy().astype(np.float64)
    both_nan = np.isnan(mine) & np.isnan(ref)
    assert np.all((mine == ref) | both_nan)
    assert set(np.nonzero(np.isnan(mine))[0]) == {0x7F, 0xFF}


@pytest.mark.parametrize("code,value", [
    (0x00, 0.0), (0x38, 1.0), (0xB8, -1.0), (0x7E, 448.0), (0xFE, -448.0), (0x08, 2.0 ** -6),
    (0x01, 2.0 ** -9), (0x07, 7 * 2.0 ** -9), (0x3C, 1.5), (0x40, 2.0), (0x77, 240.0),
])
def test_decode_closed_forms(code, value):
    assert float(_fp8().e4m3_value(np.array([code]))[0]) == value


def test_encode_matches_torch_on_the_finite_range():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8_e4m3fn")
    fp8 = _fp8()
    grid = fp8.e4m3_value(np.arange(0x7F))
    mids = (grid[1:] + grid[:-1]) / 2
    rng = np.random.default_rng(3)
    x = np.concatenate([grid, -grid, mids, -mids, rng.uniform(-448, 448, 20000),
                        rng.standard_normal(20000) * np.exp(rng.uniform(-14, 4, 20000)),
                        [0.0, -0.0, -1e-5, 2.0 ** -10, -(2.0 ** -10)]])
    x = np.clip(x, -448, 448).astype(np.float32).astype(np.float64)   # torch converts from fp32
    ref = torch.from_numpy(x.astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(fp8.e4m3_encode(x), ref)


def test_encode_is_nearest_ties_even_by_brute_force():
    fp8 = _fp8()
    grid = fp8.e4m3_value(np.arange(0x7F))
    rng = np.random.default_rng(4)
    x = np.concatenate([rng.uniform(0, 448, 3000), (grid[1:] + grid[:-1]) / 2])
    codes = fp8.e4m3_encode(x)
    for xi, c in zip(x, codes):
        d = np.abs(grid - xi)
        best = np.nonzero(d == d.min())[0]
        assert int(c) in best
        if len(best) == 2:                       # a tie: the even code
            assert int(c) % 2 == 0
    assert fp8.e4m3_encode(np.array([1000.0]))[0] == 0x7E      # saturation
    assert fp8.e4m3_encode(np.array([-1000.0]))[0] == 0xFE


def test_row_scale_and_round_trip():
    fp8 = _fp8()
    rng = wl.rng_for(5, 0)
    for scale in (1.0, 1.0 / 128, 300.0, 2.0 ** -30):
        rows = wl.bf16_bits_to_f32(wl.normal_bf16(rng, (64, 128), scale)).astype(np.float64)
        codes, es = fp8.encode_rows(rows)
        for row, c, e in zip(rows, codes, es):
            a = np.abs(row).max()
            assert 128.0 <= a * 2.0 ** -int(e) < 256.0           # the largest element's range
            back = fp8.decode_row(c, e)
            assert np.all(np.sign(back) * np.sign(row) >= 0)
            normal = np.abs(row) >= 2.0 ** (int(e) - 6)         # e4m3 normal range after scaling
            rel = np.abs(back - row)[normal] / np.abs(row)[normal]
            assert rel.max() <= 2.0 ** -4                          # half a unit of 3 mantissa bits
            assert np.all(np.abs(back - row)[~normal] <= 2.0 ** (int(e) - 10))
    z, ez = fp8.encode_row(np.zeros(64))
    assert ez == 0 and np.all(z == 0)
    # values already on a scaled grid come back exactly
    grid_row = fp8.e4m3_value(np.array([0x70, 0x41, 0x02, 0xC8, 0x38] * 4)) * 2.0 ** 5
    c, e = fp8.encode_row(grid_row)
    assert np.array_equal(fp8.decode_row(c, e), grid_row)


def test_decoded_values_are_exact_bf16():
    import oracle
    fp8 = _fp8()
    rng = wl.rng_for(6, 0)
    rows = wl.bf16_bits_to_f32(wl.normal_bf16(rng, (256, 64), 3.0)).astype(np.float64)
    codes, es = fp8.encode_rows(rows)
    back = fp8.decode_rows(codes, es)
    bits = oracle.f64_to_bf16(back.reshape(-1))
    assert np.array_equal(oracle.bf16_to_f64(bits), back.reshape(-1))


def test_fp8_cache_attention_is_attention_over_decoded_rows():
    """An FP8 pool's attention is the attention oracle on the decoded bf16 rows; against the
    bf16 pool it moves each output by the quantization of K and V only (values N(0, 1): a few
    units of 2^-4 relative at most, far smaller on average)."""
    import oracle
    fp8 = _fp8()
    w = wl.Workload("fp8_case", batch=2, n_q_heads=8, n_kv_heads=2, head_dim=64, page_slots=16,
                    layers=1, seed=7, pool_factor=1.5)
    case = wl.make_case(w, num_slots=np.array([40, 17], np.int32))
    kf = wl.bf16_bits_to_f32(case.k).astype(np.float64)
    vf = wl.bf16_bits_to_f32(case.v).astype(np.float64)
    k8, ek = fp8.encode_rows(kf)
    v8, ev = fp8.encode_rows(vf)
    kb, vb = fp8.decoded_bf16_bits(k8, ek), fp8.decoded_bf16_bits(v8, ev)
    assert np.array_equal(wl.bf16_bits_to_f32(kb).astype(np.float64), fp8.decode_rows(k8, ek))
    exact = oracle.OracleCache.from_case(case).decode_attn(case.q)
    q_case = wl.make_case(w, num_slots=np.array([40, 17], np.int32))
    q_case.k[...] = kb
    q_case.v[...] = vb
    got = oracle.OracleCache.from_case(q_case).decode_attn(case.q)
    # the same result computed directly from the decoded rows
    for b in range(2):
        L = int(case.num_slots[b])
        for h in range(8):
            g = h // 4
            kk = fp8.decode_rows(k8[b, :L, g], ek[b, :L, g])
            vv = fp8.decode_rows(v8[b, :L, g], ev[b, :L, g])
            s = kk @ wl.bf16_bits_to_f32(case.q[b, h]).astype(np.float64) / 8.0
            p = np.exp(s - s.max())
            assert np.allclose(got[b, h], (p / p.sum()) @ vv, atol=1e-12)
    err = np.abs(got - exact)
    assert err.max() < 0.1 and err.mean() < 0.02


@pytest.mark.parametrize("top", [2.0 ** -121, 2.0 ** -125, 2.0 ** -133, 2.0 ** -117,
                                 2.0 ** -116, 255.0 * 2.0 ** 120, 2.0 ** 127, 1.5 * 2.0 ** 126])
def test_row_scale_at_the_ends_of_the_bf16_range(top):
    """Rows whose largest magnitude sits near either end of bf16's range: the exponent stays in
    [-124, 119], every decoded value is finite and exactly representable in bf16 (checked through
    the C oracle's rounding, not this module's), and the largest element keeps its sign and
    lands within the e4m3 relative error of the input (or saturates at the top end)."""
    import oracle
    fp8 = _fp8()
    bf16_min_sub = 2.0 ** -133
    # a row of bf16 values: the top value, a few smaller ones, both signs, a zero
    row = np.array([top, -top / 2, top / 3, -top / 7, 0.0, top / 64, -top / 200, top / 1000])
    row = oracle.bf16_to_f64(oracle.f64_to_bf16(row))          # exact bf16 values
    assert np.abs(row).max() == top
    codes, e = fp8.encode_row(row)
    assert -124 <= e <= 119
    back = fp8.decode_row(codes, e)
    assert np.all(np.isfinite(back))
    assert np.array_equal(oracle.bf16_to_f64(oracle.f64_to_bf16(back)), back)  # exact bf16
    assert np.all(np.abs(back[back != 0]) >= bf16_min_sub)
    assert np.sign(back[0]) == 1.0
    _, E = np.frexp(top)
    assert e == min(max(int(E) - 8, -124), 119)        # the defining rule E - 8, clamped
    if int(E) - 8 <= 119:
        assert abs(back[0] - top) <= top * 2.0 ** -4
    else:                            # clamped at the top: the scaled maximum may saturate at 448
        assert back[0] <= 448.0 * 2.0 ** 119
        assert abs(back[0] - min(top, 448.0 * 2.0 ** 119)) <= top * 2.0 ** -4
    if top == 255.0 * 2.0 ** 120:
        assert back[0] == 448.0 * 2.0 ** 119           # 510 after scaling: saturated


def test_encode_rows_is_encode_row_on_every_row():
    """The vectorised encoding of many rows is the one-row encoding applied to each row, zero
    rows, clamped exponents and both signs included."""
    fp8 = _fp8()
    rng = wl.rng_for(8, 0)
    rows = wl.bf16_bits_to_f32(wl.normal_bf16(rng, (40, 32), 1.0)).astype(np.float64)
    rows *= 2.0 ** rng.integers(-140, 130, size=(40, 1))
    rows = np.clip(rows, -3.3e38, 3.3e38)
    rows[3] = 0.0
    rows[4, ::2] = -0.0
    codes, es = fp8.encode_rows(rows.reshape(4, 10, 32))
    assert codes.shape == (4, 10, 32) and es.shape == (4, 10)
    for i, row in enumerate(rows):
        c, e = fp8.encode_row(row)
        assert np.array_equal(codes.reshape(40, 32)[i], c) and int(es.reshape(40)[i]) == e
