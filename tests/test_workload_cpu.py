"""The seeded input recipe: what the generators draw is what the design states (token counts,
bf16 rounding, value scales, slot counts, page tables), reproducibly per seed."""
import numpy as np
import pytest

from paper_2505_20438_gb300 import workload as wl


def test_tokens_per_slot_follow_the_capped_geometric_law():
    t = wl.ntok_capped_geometric(wl.rng_for(5, 1), (400_000,))
    assert t.dtype == np.int32 and t.min() == 1 and t.max() == wl.MAX_TOKENS_PER_SLOT == 4
    freq = np.bincount(t, minlength=5)[1:] / t.size
    # P(1) = 1/2, P(2) = 1/4, P(3) = 1/8, P(4) = 1/8 (the tail folded into 4): mean 1.875
    expected = np.array([0.5, 0.25, 0.125, 0.125])
    sd = np.sqrt(expected * (1 - expected) / t.size)
    assert np.all(np.abs(freq - expected) < 5 * sd), freq
    assert abs(t.mean() - 1.875) < 0.01


def test_bf16_inputs_are_round_to_nearest_even():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(7)
    x = np.concatenate([
        rng.standard_normal(50_000).astype(np.float32),
        (rng.standard_normal(20_000) * 1e-30).astype(np.float32),
        (rng.standard_normal(20_000) * 1e30).astype(np.float32),
        # exact ties between two bf16 values, with even and odd lower neighbours
        (np.arange(1, 2001, dtype=np.uint32) << np.uint32(16) | np.uint32(0x8000)).view(np.float32),
        np.array([0.0, -0.0], np.float32)])
    bits = wl.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(bits, ref)
    assert np.array_equal(wl.f32_to_bf16_bits(wl.bf16_bits_to_f32(bits)), bits)


@pytest.mark.parametrize("scale", [1.0, 1.0 / np.sqrt(128.0)])
def test_values_are_normal_with_the_stated_scale(scale):
    b = wl.normal_bf16(wl.rng_for(3, 2), (300_000,), scale=scale, block=1 << 16)
    v = wl.bf16_bits_to_f32(b).astype(np.float64)
    assert abs(v.mean()) < 5 * scale / np.sqrt(v.size)
    assert abs(v.std() / scale - 1.0) < 0.01
    # the fraction within one standard deviation of a normal law: 68.27%
    assert abs(np.mean(np.abs(v) < scale) - 0.6827) < 0.005


def test_ragged_slot_counts_span_the_stated_range():
    w = wl.C2_RAGGED
    counts = np.concatenate([wl.slot_counts(w, wl.rng_for(s, 0)) for s in range(200)])
    assert counts.min() >= 512 and counts.max() <= 8192
    assert abs(counts.mean() - (512 + 8192) / 2) < 60
    assert np.array_equal(wl.slot_counts(wl.C1_LLAMA8B, wl.rng_for(0)), np.full(8, 4096))


def test_page_tables_are_distinct_pages_of_the_pool():
    B, max_pages = 8, 256
    pool = int(np.ceil(1.25 * B * max_pages))
    pt = wl.page_table(wl.rng_for(1, 3), B, max_pages, pool)
    assert pt.shape == (B, max_pages) and pt.dtype == np.int32
    assert len(np.unique(pt)) == B * max_pages and pt.min() >= 0 and pt.max() < pool
    # scattered: consecutive slots of a sequence do not sit in consecutive pages
    assert np.mean(np.diff(pt, axis=1) == 1) < 0.01
    seq = wl.page_table(wl.rng_for(1, 3), B, max_pages, pool, scatter=False)
    assert np.array_equal(seq.ravel(), np.arange(B * max_pages))
    with pytest.raises(ValueError):
        wl.page_table(wl.rng_for(1, 3), B, max_pages, B * max_pages - 1)


def test_cases_are_reproducible_per_seed():
    w = wl.scaled(wl.C1_LLAMA8B, batch=2, slots=40)
    a, b = wl.make_case(w), wl.make_case(w)
    for name in ("q", "k", "v", "k_new", "v_new", "slot_ntok", "page_table", "ntok_new"):
        assert np.array_equal(getattr(a, name), getattr(b, name)), name
    c = wl.make_case(wl.scaled(w, seed=w.seed + 1))
    assert not np.array_equal(a.q, c.q) and not np.array_equal(a.k, c.k)
    # the pool holds 1.25 x the pages the capacity needs, and the generator holds no arithmetic
    # of the method: keys are drawn as stored (already rotated), slot positions are indices
    assert a.pool_pages >= int(np.ceil(1.25 * w.batch * a.page_table.shape[1])) - 1
    assert np.array_equal(a.slot_pos[0, :40], np.arange(40))
