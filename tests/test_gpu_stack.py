"""GPU: the 32-layer decode stack (Llama-3-8B layer shape, 2048 slots to start), batch 1, 8,
32 and 128, as repeated macro-steps of `ham_decode_step` over all layers captured in one CUDA
graph, the way a decoder runs it.  After three macro-steps, layers 0 and 31 are checked against
the oracle on sampled sequences: the attention output of the last macro-step, the rotated q,
every stored K/V row and the counters.  All other layers are checked for their counters.

Inputs are seeded torch draws on the device; the oracle reads the same bits back on the host.
"""
import numpy as np
import pytest

import oracle
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import MAX_ABS, MEAN_ABS, assert_parity, host_bits, torch

pytestmark = pytest.mark.gpu

STEPS = 3
CHECK_LAYERS = (0, 31)


def _sampled(batch):
    return list(range(batch)) if batch <= 8 else [0, batch // 2 + 1, batch - 1]


@pytest.mark.parametrize("batch", [1, 8, 32, 128])
def test_decode_stack_32_layers(batch):
    t = torch()
    w = wl.c4_sweep(batch)
    L, Hq, Hkv, d = w.slots, w.n_q_heads, w.n_kv_heads, w.head_dim
    max_slots = L + STEPS + 13
    kv = ham.ham_kv_alloc(w.layers, batch, Hq, Hkv, d, w.page_slots, max_slots,
                          page_seed=w.seed + 1)
    rng = wl.rng_for(w.seed, 20)
    counts = np.full(batch, L, np.int32)
    ntok_fill = wl.ntok_capped_geometric(rng, (batch, L))
    counts_dev = t.from_numpy(counts).cuda()
    ntok_fill_dev = t.from_numpy(ntok_fill).cuda()
    S = _sampled(batch)
    host_fill = {}
    for layer in range(w.layers):
        seed = w.seed * 1000 + 10 * layer
        k = wl.device_normal_bf16((batch, L, Hkv, d), w.value_scale, seed + 1)
        v = wl.device_normal_bf16((batch, L, Hkv, d), w.value_scale, seed + 2)
        ham.ham_kv_fill(kv, layer, k, v, counts_dev, ntok=ntok_fill_dev)
        if layer in CHECK_LAYERS:
            host_fill[layer] = (host_bits(k[S]), host_bits(v[S]))
        del k, v
    # per-layer step inputs, replayed by every macro-step
    q = [wl.device_normal_bf16((batch, Hq, d), w.value_scale, 7000 + l) for l in range(w.layers)]
    k_new = [wl.device_normal_bf16((batch, Hkv, d), w.value_scale, 8000 + l)
             for l in range(w.layers)]
    v_new = [wl.device_normal_bf16((batch, Hkv, d), w.value_scale, 9000 + l)
             for l in range(w.layers)]
    ntok_new = wl.ntok_capped_geometric(rng, (batch,))
    ntok_dev = t.from_numpy(ntok_new).cuda()
    out = [t.empty((batch, Hq, d), dtype=t.bfloat16, device="cuda") for _ in range(w.layers)]
    q_rot = [t.empty((batch, Hq, d), dtype=t.bfloat16, device="cuda") for _ in range(w.layers)]

    stream = t.cuda.Stream()

    def macro_step():
        for layer in range(w.layers):
            ham.ham_decode_step(kv, layer, q[layer], k_new[layer], v_new[layer], None, ntok_dev,
                                out[layer], q_rot=q_rot[layer])

    graph = t.cuda.CUDAGraph()
    with t.cuda.graph(graph, stream=stream):
        macro_step()
    with t.cuda.stream(stream):
        for _ in range(STEPS):
            graph.replay()
    t.cuda.synchronize()
    assert ham.ham_kv_status(kv) == ham.HAM_DEVERR_NONE
    for layer in range(w.layers):
        slots, tokens = ham.ham_kv_layer_lengths(kv, layer)
        assert np.all(slots == L + STEPS), layer
        assert np.array_equal(tokens, ntok_fill.sum(axis=1) + STEPS * ntok_new), layer

    # oracle on the sampled sequences of layers 0 and 31
    nS = len(S)
    max_pages = wl.pages_needed(max_slots, w.page_slots)
    pt = np.arange(nS * max_pages, dtype=np.int32).reshape(nS, max_pages)
    for layer in CHECK_LAYERS:
        oc = oracle.OracleCache(nS, Hq, Hkv, d, w.page_slots, pt, nS * max_pages, max_slots)
        kh, vh = host_fill[layer]
        pos = np.broadcast_to(np.arange(L, dtype=np.int32), (nS, L)).copy()
        oc.fill(kh, vh, pos, ntok_fill[S], counts[S])
        q_host = host_bits(q[layer])[S]
        kn, vn = host_bits(k_new[layer])[S], host_bits(v_new[layer])[S]
        for _ in range(STEPS):
            q_ref = q_host.copy()
            assert oc.append(kn, vn, ntok_new[S], q_inout=q_ref) == 0
        ref = oc.decode_attn(q_ref)
        got = out[layer].float().cpu().numpy().astype(np.float64)[S]
        assert_parity(got, ref, MAX_ABS, MEAN_ABS, what=f"layer {layer}")
        assert np.array_equal(host_bits(q_rot[layer])[S], q_ref), f"q_rot layer {layer}"
        # stored rows and slot metadata of the sampled sequences, through the page table
        n = L + STEPS
        pt_gpu = ham.ham_kv_get_page_table(kv)
        k_pool, v_pool, pos_pool, ntok_pool = ham.ham_kv_export(kv, layer)
        slots = np.arange(n)
        for j, b in enumerate(S):
            pages = t.from_numpy(pt_gpu[b, slots // w.page_slots].astype(np.int64)).cuda()
            rows = t.from_numpy((slots % w.page_slots).astype(np.int64)).cuda()
            k_rows = host_bits(k_pool[pages, :, rows])            # [n][Hkv][d]
            v_rows = host_bits(v_pool[pages, :, rows])
            assert np.array_equal(pos_pool[pages, rows].cpu().numpy(), np.arange(n)), (layer, b)
            assert np.array_equal(ntok_pool[pages, rows].cpu().numpy(),
                                  np.concatenate([ntok_fill[b], np.full(STEPS, ntok_new[b])]))
            for g in range(Hkv):
                ko, vo = oc.gather(j, g)
                assert np.array_equal(wl.f32_to_bf16_bits(ko.astype(np.float32)),
                                      k_rows[:, g]), (layer, b, g)
                assert np.array_equal(wl.f32_to_bf16_bits(vo.astype(np.float32)),
                                      v_rows[:, g]), (layer, b, g)
        del k_pool, v_pool, pos_pool, ntok_pool
    ham.ham_kv_free(kv)
