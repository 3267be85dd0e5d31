"""Shared set-up for the GPU tests: seeded host cases -> the CUDA cache and the CPU oracle."""
import numpy as np

from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

# Parity bar: bf16 inputs, fp32 accumulation (max-abs and mean-abs error vs the oracle).
MAX_ABS = 2e-2
MEAN_ABS = 2e-3


def torch():
    import torch as t
    return t


def dev_bf16(bits):
    t = torch()
    a = np.ascontiguousarray(bits, dtype=np.uint16).view(np.int16)
    return t.from_numpy(a).view(t.bfloat16).to("cuda")


def dev_i32(x):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).to("cuda")


def host_bits(tensor):
    t = torch()
    return tensor.detach().to("cpu").contiguous().view(t.int16).numpy().view(np.uint16)


def gpu_cache(case, layers=1, pos_mode=ham.HAM_POS_SLOT, fill=True, page_table=None):
    w = case.w
    kv = ham.ham_kv_alloc(layers, w.batch, w.n_q_heads, w.n_kv_heads, w.head_dim,
                          w.page_slots, case.max_slots, pos_mode=pos_mode,
                          pool_pages=case.pool_pages)
    ham.ham_kv_set_page_table(kv, case.page_table if page_table is None else page_table)
    if fill:
        for layer in range(layers):
            ham.ham_kv_fill(kv, layer, dev_bf16(case.k), dev_bf16(case.v),
                            dev_i32(case.num_slots), pos=dev_i32(case.slot_pos),
                            ntok=dev_i32(case.slot_ntok))
    return kv


def gpu_decode(kv, q_bits, layer=0, f32=False):
    t = torch()
    q = dev_bf16(q_bits)
    # NaN-filled so that an output the kernel never writes cannot pass as a stale value
    out = t.full(q.shape, float("nan"), dtype=t.float32 if f32 else t.bfloat16, device="cuda")
    ham.ham_decode_attn_ex(kv, layer, q, out)
    t.cuda.synchronize()
    return out.float().cpu().numpy().astype(np.float64)


def assert_parity(got, ref, max_abs=MAX_ABS, mean_abs=MEAN_ABS, what=""):
    assert got.shape == ref.shape
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - ref)
    assert err.max() <= max_abs, f"{what}: max-abs {err.max():.3e} > {max_abs}"
    assert err.mean() <= mean_abs, f"{what}: mean-abs {err.mean():.3e} > {mean_abs}"
    return float(err.max()), float(err.mean())


def small_case(batch=2, hq=8, hkv=2, d=64, page=16, counts=(37, 80), scale=1.0, seed=0,
               scatter=True, pool_factor=1.5, extra_slots=4):
    w = wl.Workload(f"case_s{seed}", batch=batch, n_q_heads=hq, n_kv_heads=hkv, head_dim=d,
                    page_slots=page, layers=1, value_scale=scale, seed=seed,
                    pool_factor=pool_factor, scatter_pages=scatter)
    return wl.make_case(w, num_slots=np.array(counts, np.int32), extra_slots=extra_slots)
