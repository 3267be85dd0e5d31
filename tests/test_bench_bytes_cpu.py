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
