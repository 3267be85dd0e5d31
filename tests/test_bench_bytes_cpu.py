"""The algorithmic byte counts behind the bench's roofline numerators, against sizes worked out by
hand for the bench workloads (no GPU needed)."""
import math

from paper_2505_20438_gb300 import workload as wl


def _bench():
    import bench
    return bench


def test_attention_bytes_of_the_llama8b_layer():
    w = wl.C1_LLAMA8B
    b = _bench()
    # K and V of 8 x 4096 slots x 8 heads x 128 x 2 B, q and out 8 x 32 x 128 x 2 B each,
    # 256 page-table entries of 4 B per sequence
    kv = 8 * 4096 * 8 * 128 * 2 * 2
    assert b.attn_bytes(w, [4096] * 8) == kv + 2 * 8 * 32 * 128 * 2 + 8 * 256 * 4
    assert kv == 134_217_728                       # the 128 MiB of the workload's statement


def test_front_bytes_of_the_llama8b_layer():
    w = wl.front_workload(8)
    weights = (32 + 2 * 8) * 128 * 4096 * 2       # 6144 rows of 4096 bf16
    assert weights == 50_331_648
    expected = weights + 8 * 4096 * 2 + 8 * 32 * 128 * 2 + 8 * 2 * 8 * 128 * 2 + 8 * 40
    assert _bench().front_bytes(w) == expected == 50_495_808
    # ideal time at the measured copy bandwidth: about 7.4 us
    assert math.isclose(expected / 6784.5e9 * 1e6, 7.44, abs_tol=0.01)


def test_micro_call_bytes():
    w = wl.micro_workload(8)
    # 8 sequences x old slots x 8 KV heads x 64 x (K + V) x 2 B, q and out (32 heads), k/v new in
    # and the new rows out, 40 B of counters and metadata per sequence
    for old in (4, 5, 6):
        expected = (8 * old * 8 * 64 * 4 + 8 * 32 * 64 * 2 * 2 + 8 * 8 * 64 * 4 * 2 + 8 * 40)
        assert _bench().micro_call_bytes(w, old) == expected
    avg = sum(_bench().micro_call_bytes(w, 4 + i) for i in range(3)) / 3
    assert avg == 180_544


def test_workload_names_resolve():
    b = _bench()
    assert isinstance(b.workload("qkv_front_b8"), wl.FrontWorkload)
    assert b.workload("qkv_front_b8").out_rows == 6144
    m = b.workload("micro_b8")
    assert isinstance(m, wl.MicroWorkload) and (m.layers, m.context, m.micro_steps) == (4, 4, 3)
    c = wl.make_micro_case(m)
    assert c.max_slots == 8 and list(c.num_slots) == [4] * 8 and all(c.ntok_new == 1)


def test_fp8_attention_bytes_of_the_llama8b_layer():
    w = wl.C1_LLAMA8B
    b = _bench()
    # an e4m3 row is 128 codes and one exponent byte: 129 B against 256 B in bf16
    assert b.kv_row_bytes(w, "fp8") == 129 and b.kv_row_bytes(w) == 256
    kv8 = 8 * 4096 * 8 * 129 * 2
    assert b.attn_bytes(w, [4096] * 8, "fp8") == kv8 + 2 * 8 * 32 * 128 * 2 + 8 * 256 * 4
    # the appended rows shrink the same way; q, k_new and v_new stay bf16
    assert b.append_bytes(w) - b.append_bytes(w, "fp8") == 2 * 8 * 8 * (256 - 129)


def test_fp8_front_bytes_of_the_llama8b_layer():
    w = wl.front_workload(8)
    b = _bench()
    assert b.front_bytes(w) - b.front_bytes(w, "fp8") == 8 * 2 * 8 * (256 - 129)


def test_prefill_flops_count_every_attended_pair():
    b = _bench()
    # brute force on small chunks: every new row j of every sequence attends L + j + 1 slots
    for rows, cached in ((1, 0), (5, 3), (7, 64), (64, 1000)):
        pw = wl.PrefillWorkload("t", wl.C1_LLAMA8B, rows=rows, cached=cached)
        w = pw.w
        pairs = sum(cached + j + 1 for j in range(rows)) * w.batch
        assert b.prefill_flops(pw) == 4 * w.head_dim * w.n_q_heads * pairs
    # the bench workloads: 549.9 GFLOP for 4 fresh prompts of 4096 rows, 68.8 GFLOP for 64 rows
    # over 65,536 cached slots
    p1, p3 = wl.PREFILL_WORKLOADS["prefill_b4_s4096"], wl.PREFILL_WORKLOADS["prefill_b1_c64_s65536"]
    assert b.prefill_flops(p1) == 4 * 128 * 32 * 4 * (4096 * 4097 // 2) == 549_890_031_616
    assert b.prefill_flops(p3) == 4 * 128 * 32 * (64 * 65536 + 64 * 65 // 2)


def test_prefill_bytes_of_the_short_chunk():
    p3 = _bench().workload("prefill_b1_c64_s65536")
    # K and V of 65,536 + 64 slots x 8 heads x 128 x 2 B; q in and out (32 heads); k, v in
    kv = (65536 + 64) * 8 * 128 * 2 * 2
    q = 64 * 32 * 128 * 2 * 2
    new = 64 * 8 * 128 * 2 * 2
    assert _bench().prefill_bytes(p3) == kv + q + new == 270_008_320


def test_cost_model_follows_the_papers_speedup_formula():
    # Sec. 3.7: r = n C(S) / (C(S) + (n - 1) c); one token per slot gives no speed-up, a free
    # micro-step decoder gives n, and any c < C(S) with n > 1 gives r > 1
    cm = _bench().cost_model
    assert cm(1.0, 30.0)["r"] == 1.0
    assert cm(3.0, 30.0, c_ratio=0.0)["r"] == 3.0
    assert math.isclose(cm(2.0, 40.0, c_ratio=1 / 8)["r"], 16 / 9, abs_tol=1e-4)
    for n in (1.5, 1.875, 4.0):
        for ratio in (0.05, 0.125, 0.9):
            d = cm(n, 25.0, c_ratio=ratio)
            assert d["r"] > 1.0 and d["kind"] == "modelled"
            assert math.isclose(d["c_us"], ratio * 25.0, rel_tol=1e-3)
