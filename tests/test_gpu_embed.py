"""GPU: the compositional embedder (Sec. 3.2, Sec. 3.4) against the fp64 oracle on the same
seeded bits.  Fused states within the bf16 bar; single-token sequences bit for bit."""
import numpy as np
import pytest

from oracle import embedder as oe
from paper_2505_20438_gb300 import ham
from paper_2505_20438_gb300 import workload as wl

from gpu_helpers import MEAN_ABS, dev_bf16, dev_i32, host_bits, torch

pytestmark = pytest.mark.gpu

# Tolerance from the arithmetic.  Projections and attention accumulate in fp32, o reaches the
# output linear as a hi + lo pair of bf16 values (about 16 bits) and the state is rounded to bf16
# once at the end.  Per element f of a fused state: at most one bf16 rounding of the state,
# 2^-8 |ref| (half a unit in the last place, where the GPU's fp32 sum may fall on the other side
# of a rounding boundary), plus the error of the fp32 sum itself, bounded by
# 2^-14 sum_k |W_o[f][k]| |o_k| (fp32 accumulation over the width and the 2^-17 representation
# of o, with the errors o inherits from the fp32 projections, all far below 2^-14).
ROUND = 2.0 ** -8
ACC = 2.0 ** -14


def assert_states(got, ref, wo_abs_o, what):
    """got, ref [n][H]; wo_abs_o [n][H] = sum_k |W_o[f][k]| |o_k| of each state."""
    assert np.all(np.isfinite(got)), what
    err = np.abs(got - ref)
    tol = ROUND * np.abs(ref) + ACC * wo_abs_o
    worst = np.unravel_index(np.argmax(err - tol), err.shape)
    assert np.all(err <= tol), (f"{what}: error {err[worst]:.3e} > bound {tol[worst]:.3e} at "
                                f"{worst} (ref {ref[worst]:.4f})")
    assert err.mean() <= MEAN_ABS, f"{what}: mean-abs {err.mean():.3e}"


def _run(c, offsets=None, max_batch=None):
    t = torch()
    w = c.w
    e = ham.ham_embedder_alloc(w.hidden, w.n_heads, max_batch or w.batch, w.max_patch,
                               dev_bf16(c.wq), dev_bf16(c.wk), dev_bf16(c.wv), dev_bf16(c.wo),
                               dev_bf16(c.pos))
    B = len(c.counts)
    out = t.full((B, w.hidden), float("nan"), dtype=t.bfloat16, device="cuda")
    ham.ham_embed(e, dev_bf16(c.x), dev_i32(c.offsets if offsets is None else offsets), out)
    t.cuda.synchronize()
    return e, out


def _reference(c, offsets=None):
    """The oracle's states and, per element, sum_k |W_o[f][k]| |o_k| (the accumulation term)."""
    ref, o = oe.embed(c.x, c.offsets if offsets is None else offsets, c.wq, c.wk, c.wv, c.wo,
                      c.pos, c.w.n_heads, return_o=True)
    wo = np.abs(oe.bf16_bits_to_f64(c.wo))
    return ref, np.abs(o) @ wo.T


def _check(c, out):
    ref, wo_abs_o = _reference(c)
    got = out.float().cpu().numpy().astype(np.float64)
    bits = host_bits(out)
    fused = c.counts > 1
    if fused.any():
        assert_states(got[fused], ref[fused], wo_abs_o[fused], "fused states")
    for b in np.nonzero(~fused)[0]:
        assert np.array_equal(bits[b], c.x[c.offsets[b]]), f"bypass row {b}"


@pytest.mark.parametrize("batch,hidden,heads", [
    (64, 2048, 32),    # the Llama-3.2-1B width; ~122 tokens: both projections streamed
    (8, 256, 8), (5, 512, 4), (12, 320, 10),   # head dims 32 / 128; one K split (5 chunks)
    (100, 512, 8),     # ~187 tokens: two 128-row tiles of the Q/K/V projection
    (160, 256, 8),     # 320 rows of o (hi and lo): three row tiles of the output projection
])
def test_embed_matches_oracle(batch, hidden, heads):
    c = wl.make_embed_case(wl.embed_workload(batch, hidden=hidden, n_heads=heads, seed=batch))
    e, out = _run(c)
    _check(c, out)
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NONE


@pytest.mark.parametrize("counts", [[1] * 9, [4] * 7, [2, 1, 4, 3, 1, 1, 2]])
def test_embed_patch_mixes(counts):
    c = wl.make_embed_case(wl.embed_workload(len(counts), hidden=1024, n_heads=16, seed=3),
                           counts=np.array(counts))
    e, out = _run(c, max_batch=16)
    _check(c, out)
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NONE


def test_bad_counts_give_zeros_and_the_error_word():
    c = wl.make_embed_case(wl.embed_workload(6, hidden=256, n_heads=8, seed=4),
                           counts=np.array([2, 1, 3, 2, 1, 3]))
    offsets = c.offsets.copy()
    offsets[2] = offsets[1]        # sequence 1: no token (sequence 2 now has 4)
    offsets[4] = offsets[5] + 1    # sequence 4: a negative count (sequence 3 now has 4)
    e, out = _run(c, offsets=offsets)
    bits = host_bits(out)
    counts = np.diff(offsets)
    ok = (counts >= 1) & (counts <= c.w.max_patch) & (offsets[:-1] >= 0) & \
        (offsets[1:] <= offsets[-1])
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NTOK
    for b in np.nonzero(~ok)[0]:
        assert np.all(bits[b] == 0), b
    ref, wo_abs_o = _reference(c)
    for b in np.nonzero(ok)[0]:    # untouched sequences keep their own tokens and result
        if offsets[b] == c.offsets[b] and offsets[b + 1] == c.offsets[b + 1]:
            got = out[b].float().cpu().numpy().astype(np.float64)
            if c.counts[b] > 1:
                assert_states(got[None], ref[b][None], wo_abs_o[b][None], f"sequence {b}")
            else:
                assert np.array_equal(bits[b], c.x[c.offsets[b]]), b


def test_host_errors():
    t = torch()
    c = wl.make_embed_case(wl.embed_workload(4, hidden=256, n_heads=8, seed=2))
    e, out = _run(c)
    x = dev_bf16(c.x)
    with pytest.raises(ham.HamError):          # batch above the handle's max_batch
        big = t.zeros((5, 256), dtype=t.bfloat16, device="cuda")
        ham.ham_embed(e, t.zeros((5, 256), dtype=t.bfloat16, device="cuda"),
                      dev_i32(np.arange(6)), big)
    with pytest.raises(ValueError):            # wrong offsets shape
        ham.ham_embed(e, x, dev_i32(c.offsets[:-1]), out)
    with pytest.raises(ham.HamError):          # head_dim 16 is not compiled
        ham.ham_embedder_alloc(256, 16, 4, 4, *(dev_bf16(w) for w in (c.wq, c.wk, c.wv, c.wo)),
                               dev_bf16(c.pos))


# ---- token ids through the tabulated vocabulary (ham_embedder_set_vocab / ham_embed_tokens) --

def _run_tokens(tc, ids=None, max_batch=None):
    t = torch()
    c = tc.case
    w = c.w
    e = ham.ham_embedder_alloc(w.hidden, w.n_heads, max_batch or len(c.counts), w.max_patch,
                               dev_bf16(c.wq), dev_bf16(c.wk), dev_bf16(c.wv), dev_bf16(c.wo),
                               dev_bf16(c.pos))
    ham.ham_embedder_set_vocab(e, dev_bf16(tc.table))
    out = t.full((len(c.counts), w.hidden), float("nan"), dtype=t.bfloat16, device="cuda")
    ham.ham_embed_tokens(e, dev_i32(tc.ids if ids is None else ids), dev_i32(c.offsets), out)
    t.cuda.synchronize()
    return e, out


@pytest.mark.parametrize("batch,hidden,heads,vocab", [
    (64, 2048, 32, wl.LLAMA3_VOCAB),   # the Llama-3.2-1B width and vocabulary
    (8, 256, 8, 1000), (12, 320, 10, 777), (160, 256, 8, 5000), (5, 512, 4, 3),
])
def test_embed_tokens_matches_oracle(batch, hidden, heads, vocab):
    tc = wl.make_embed_tokens_case(
        wl.embed_workload(batch, hidden=hidden, n_heads=heads, seed=batch + 1), vocab)
    e, out = _run_tokens(tc)
    _check(tc.case, out)     # case.x = table[ids]: fused states and bypass rows
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NONE


def test_embed_tokens_bad_ids_give_zeros_and_the_error_word():
    vocab = 300
    tc = wl.make_embed_tokens_case(wl.embed_workload(6, hidden=256, n_heads=8, seed=6), vocab,
                                   counts=np.array([2, 1, 3, 1, 4, 2]))
    c = tc.case
    ids = tc.ids.copy()
    ids[c.offsets[0] + 1] = vocab     # sequence 0: an id past the end
    ids[c.offsets[3]] = -1            # sequence 3: a single bad token
    e, out = _run_tokens(tc, ids=ids)
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NTOK
    bits = host_bits(out)
    for b in (0, 3):
        assert np.all(bits[b] == 0), b
    ref, wo_abs_o = _reference(c)
    got = out.float().cpu().numpy().astype(np.float64)
    for b in (2, 4, 5):
        if c.counts[b] > 1:
            assert_states(got[b][None], ref[b][None], wo_abs_o[b][None], f"sequence {b}")
        else:
            assert np.array_equal(bits[b], tc.table[ids[c.offsets[b]]]), b
    assert np.array_equal(bits[1], tc.table[ids[c.offsets[1]]])


def test_embed_tokens_host_errors():
    t = torch()
    tc = wl.make_embed_tokens_case(wl.embed_workload(4, hidden=256, n_heads=8, seed=2), 50)
    c = tc.case
    e = ham.ham_embedder_alloc(256, 8, 4, c.w.max_patch,
                               *(dev_bf16(w) for w in (c.wq, c.wk, c.wv, c.wo)), dev_bf16(c.pos))
    out = t.zeros((4, 256), dtype=t.bfloat16, device="cuda")
    with pytest.raises(ham.HamError):          # no vocabulary yet
        ham.ham_embed_tokens(e, dev_i32(tc.ids), dev_i32(c.offsets), out)
    with pytest.raises(ValueError):            # table of the wrong width
        ham.ham_embedder_set_vocab(e, t.zeros((50, 128), dtype=t.bfloat16, device="cuda"))
    ham.ham_embedder_set_vocab(e, dev_bf16(tc.table))
    ham.ham_embedder_set_vocab(e, dev_bf16(tc.table))   # replacing the table is allowed
    ham.ham_embed_tokens(e, dev_i32(tc.ids), dev_i32(c.offsets), out)
    t.cuda.synchronize()
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NONE
    # one id fewer than the offsets say: the last sequence's rows leave the call's tokens
    ham.ham_embed_tokens(e, dev_i32(tc.ids[:-1]), dev_i32(c.offsets), out)
    t.cuda.synchronize()
    assert ham.ham_embedder_status(e) == ham.HAM_DEVERR_NTOK
    assert np.all(host_bits(out)[-1] == 0)
