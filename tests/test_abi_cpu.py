"""The C ABI without a GPU: symbols, host-side argument checks and the split plan."""
import ctypes
import subprocess

import numpy as np
import pytest

from paper_2505_20438_gb300 import build as build_mod
from paper_2505_20438_gb300 import ham


@pytest.fixture(scope="module")
def libham():
    build_mod.build()
    return ham.lib()


def test_header_declares_the_four_calls():
    names = ham.header_functions()
    for required in ("ham_kv_alloc", "ham_decode_attn", "ham_kv_append", "ham_slot_lengths"):
        assert required in names
    assert len(names) >= 16


def test_library_exports_every_declared_symbol(libham):
    out = subprocess.run(["nm", "-D", "--defined-only", ham.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if line.strip()}
    for name in ham.header_functions():
        assert name in exported, name
        assert hasattr(libham, name)


def test_python_binding_covers_every_symbol():
    for name in ham.header_functions():
        assert hasattr(ham, name), name


def _cfg(**kw):
    base = dict(layers=1, batch=2, n_q_heads=8, n_kv_heads=2, head_dim=64, page_slots=16,
                max_slots_per_seq=64, pos_mode=0, pool_pages=0, rope_base=10000.0, page_seed=0,
                kv_dtype=0)
    base.update(kw)
    return ham.ham_config(**base)


@pytest.mark.parametrize("kw,status", [
    (dict(layers=0), ham.HAM_EINVAL),
    (dict(batch=0), ham.HAM_EINVAL),
    (dict(batch=5000), ham.HAM_EINVAL),
    (dict(n_q_heads=6, n_kv_heads=4), ham.HAM_EINVAL),
    (dict(page_slots=8), ham.HAM_EINVAL),
    (dict(page_slots=24), ham.HAM_EINVAL),
    (dict(max_slots_per_seq=0), ham.HAM_EINVAL),
    (dict(pos_mode=2), ham.HAM_EINVAL),
    (dict(rope_base=1.0), ham.HAM_EINVAL),
    (dict(head_dim=96), ham.HAM_EUNSUPPORTED),
    (dict(n_q_heads=32, n_kv_heads=2), ham.HAM_EUNSUPPORTED),
    (dict(pool_pages=3), ham.HAM_ECAPACITY),
    (dict(kv_dtype=7), ham.HAM_EINVAL),
    (dict(kv_dtype=ham.HAM_KV_E4M3), ham.HAM_EUNSUPPORTED),           # FP8 pools: head_dim 128
    (dict(kv_dtype=ham.HAM_KV_E4M3, head_dim=128, pool_pages=3), ham.HAM_ECAPACITY),
])
def test_alloc_rejects_bad_configs_on_the_host(libham, kw, status):
    out = ctypes.c_void_p(123)
    rc = libham.ham_kv_alloc(ctypes.byref(_cfg(**kw)), ctypes.byref(out))
    assert rc == status, ham.ham_last_error()
    assert out.value is None
    assert ham.ham_last_error()


def test_null_arguments_are_rejected(libham):
    assert libham.ham_kv_alloc(None, None) == ham.HAM_EINVAL
    out = ctypes.c_void_p()
    assert libham.ham_kv_alloc(None, ctypes.byref(out)) == ham.HAM_EINVAL
    assert libham.ham_kv_free(None) == ham.HAM_OK
    assert libham.ham_decode_attn(None, 0, None, None, None) == ham.HAM_EINVAL
    assert libham.ham_kv_export_scales(None, 0, None, None) == ham.HAM_EINVAL
    assert libham.ham_kv_append(None, 0, None, None, None, None, None, None) == ham.HAM_EINVAL
    assert libham.ham_prefill(None, 0, None, None, None, None, None, None, 0, None, 0,
                              None) == ham.HAM_EINVAL
    assert libham.ham_slot_lengths(None, None, None, None) == ham.HAM_EINVAL
    assert libham.ham_kv_status(None, None, None) == ham.HAM_EINVAL
    assert libham.ham_kv_get_info(None, None) == ham.HAM_EINVAL
    assert libham.ham_kv_set_wait_limit_ns(None, 1000) == ham.HAM_EINVAL


# ---------------------------------------------------------------------------------------
# split plan (the same inline arithmetic the kernel evaluates on the device)
# ---------------------------------------------------------------------------------------

def _chunks(n):
    return (n + 15) // 16


@pytest.mark.parametrize("counts,hkv,ctas", [
    ([4096] * 8, 8, 304),
    ([256], 2, 304),                                  # far fewer chunks than CTAs
    ([0, 17, 0, 1, 4096, 33], 8, 7),                  # empty and ragged sequences
    (list(np.random.default_rng(2).integers(512, 8193, 64)), 8, 304),
    ([65536] * 4, 8, 304),
    ([1], 1, 1),
    ([0, 0], 4, 10),                                  # nothing to do
])
def test_split_plan_partitions_every_chunk_once(libham, counts, hkv, ctas):
    counts = np.array(counts, np.int32)
    begin, first, last = ham.ham_split_plan(counts, hkv, ctas)
    W = hkv * int(sum(_chunks(int(n)) for n in counts))
    assert begin[0] == 0 and begin[-1] == W
    sizes = np.diff(begin)
    active = min(ctas, -(-W // 4))           # small problems: ranges of about 4 chunks
    assert np.all(sizes[:active] >= 1) and np.all(sizes[active:] == 0)
    if active:
        assert sizes[:active].max() - sizes[:active].min() <= 1       # balanced
    # chunk -> owner CTA, recomputed from the ranges
    owner = np.repeat(np.arange(ctas), sizes)
    assert len(owner) == W
    x = 0
    seen_partials = set()
    for b, n in enumerate(counts):
        for g in range(hkv):
            s = b * hkv + g
            nch = _chunks(int(n))
            if nch == 0:
                assert first[s] == -1 and last[s] == -1
                continue
            assert first[s] == owner[x] and last[s] == owner[x + nch - 1]
            # every CTA from first to last really holds chunks of this segment
            assert set(owner[x:x + nch]) == set(range(first[s], last[s] + 1))
            for c in range(first[s], last[s] + 1):
                idx = c + s                                  # partial slot of (CTA, segment)
                assert idx not in seen_partials
                assert 0 <= idx < ctas + len(counts) * hkv
                seen_partials.add(idx)
            x += nch
    assert x == W


def test_split_plan_rejects_bad_arguments(libham):
    with pytest.raises(ham.HamError):
        ham.ham_split_plan(np.array([-1], np.int32), 1, 4)
    with pytest.raises(ham.HamError):
        ham.ham_split_plan(np.array([5], np.int32), 1, 0)


@pytest.mark.parametrize("hidden,heads,batch,patch,status", [
    (100, 3, 4, 4, ham.HAM_EINVAL),          # not a multiple of the heads
    (256, 16, 4, 4, ham.HAM_EUNSUPPORTED),   # head_dim 16
    (256, 4, 0, 4, ham.HAM_EINVAL),          # no batch
    (256, 4, 4, 9, ham.HAM_EINVAL),          # patch above 8
])
def test_embedder_alloc_rejects_bad_configs_on_the_host(libham, hidden, heads, batch, patch,
                                                        status):
    cfg = ham.ham_embed_config(hidden, heads, batch, patch)
    out = ctypes.c_void_p()
    dummy = ctypes.c_void_p(16)   # never dereferenced: the config is checked first
    assert libham.ham_embedder_alloc(ctypes.byref(cfg), dummy, dummy, dummy, dummy, dummy,
                                     ctypes.byref(out)) == status
    assert out.value is None


def test_embedder_null_arguments_are_rejected(libham):
    cfg = ham.ham_embed_config(256, 4, 4, 4)
    out = ctypes.c_void_p()
    assert libham.ham_embedder_alloc(ctypes.byref(cfg), None, None, None, None, None,
                                     ctypes.byref(out)) == ham.HAM_EINVAL
    assert libham.ham_embed(None, None, None, 1, 1, None, None) == ham.HAM_EINVAL
    assert libham.ham_embedder_status(None, None, None) == ham.HAM_EINVAL
    assert libham.ham_embedder_set_vocab(None, None, 1) == ham.HAM_EINVAL
    assert libham.ham_embed_tokens(None, None, None, 1, 1, None, None) == ham.HAM_EINVAL
    assert libham.ham_embedder_free(None) == ham.HAM_OK


# ---------------------------------------------------------------------------------------
# the binding never hands a host pointer to a kernel: every tensor argument is checked for
# device, dtype, shape and layout before the library is called
# ---------------------------------------------------------------------------------------

def _fake_kv():
    import types
    return types.SimpleNamespace(batch=2, n_q_heads=8, n_kv_heads=2, head_dim=64, max_pages=4)


def _host_tensors():
    import torch
    B, Hq, Hkv, d = 2, 8, 2, 64
    return dict(q=torch.zeros(B, Hq, d, dtype=torch.bfloat16),
                kn=torch.zeros(B, Hkv, d, dtype=torch.bfloat16),
                vn=torch.zeros(B, Hkv, d, dtype=torch.bfloat16),
                ntok=torch.ones(B, dtype=torch.int32),
                out=torch.zeros(B, Hq, d, dtype=torch.bfloat16),
                x=torch.zeros(B, 256, dtype=torch.bfloat16),
                w=torch.zeros((Hq + 2 * Hkv) * d, 256, dtype=torch.bfloat16),
                off=torch.tensor([0, 1, 2], dtype=torch.int32),
                q1=torch.zeros(2, Hq, d, dtype=torch.bfloat16),
                k1=torch.zeros(2, Hkv, d, dtype=torch.bfloat16))


@pytest.mark.parametrize("call,first", [
    (lambda kv, t: ham.ham_kv_append(kv, 0, t["q"], t["kn"], t["vn"], None, t["ntok"]), "q_inout"),
    (lambda kv, t: ham.ham_decode_attn(kv, 0, t["q"], t["out"]), "q"),
    (lambda kv, t: ham.ham_decode_attn_ex(kv, 0, t["q"], t["out"]), "q"),
    (lambda kv, t: ham.ham_decode_step(kv, 0, t["q"], t["kn"], t["vn"], None, t["ntok"],
                                       t["out"]), "q"),
    (lambda kv, t: ham.ham_micro_step(kv, 0, t["q"], t["kn"], t["vn"], None, t["ntok"],
                                      t["out"]), "q"),
    (lambda kv, t: ham.ham_prefill(kv, 0, t["q1"], t["k1"], t["k1"], t["off"], t["q1"]), "q"),
    (lambda kv, t: ham.ham_qkv_append(kv, 0, t["x"], t["w"], t["ntok"], t["q"]), "x"),
    (lambda kv, t: ham.ham_kv_fill(kv, 0, t["kn"][:, None], t["vn"][:, None], t["ntok"]), "k"),
])
def test_binding_rejects_host_tensors_before_the_library(call, first):
    with pytest.raises(ValueError, match="must be a CUDA tensor") as e:
        call(_fake_kv(), _host_tensors())
    assert str(e.value).startswith(first)


def test_binding_rejects_host_tensors_without_a_handle():
    import torch
    t = _host_tensors()
    pool = torch.zeros(4, 2, 16, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="k_pool must be a CUDA tensor"):
        ham.ham_decode_attn_noalloc(pool, pool, torch.zeros(2, 4, dtype=torch.int32),
                                    t["ntok"], t["q"], t["out"], 64)
