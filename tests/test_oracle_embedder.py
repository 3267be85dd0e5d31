"""Pins of the compositional-embedder oracle (Sec. 3.2, Sec. 3.4) against things other than
itself: torch's multi-head attention module, closed forms, symmetry and exact bypass."""
import numpy as np
import pytest

from oracle import embedder as oe
from paper_2505_20438_gb300 import workload as wl

H, NH = 64, 4   # small width: 4 heads of 16


def _case(counts, seed=1):
    w = wl.embed_workload(len(counts), hidden=H, n_heads=NH, seed=seed)
    return wl.make_embed_case(w, counts=np.array(counts))


def _embed(c, pos=None, x=None):
    return oe.embed(c.x if x is None else x, c.offsets, c.wq, c.wk, c.wv, c.wo,
                    c.pos if pos is None else pos, NH)


def test_single_token_bypasses_exactly():
    c = _case([1, 3, 1, 2, 1])
    out = _embed(c)
    x = oe.bf16_bits_to_f64(c.x)
    for b, n in enumerate(c.counts):
        if n == 1:
            assert np.array_equal(out[b], x[c.offsets[b]])


def test_matches_torch_multihead_attention():
    """The library's multi-head attention with the same projections: query = mean of the
    tokens, key = value = token + position embedding, one query per sequence."""
    torch = pytest.importorskip("torch")
    c = _case([2, 3, 4, 2, 4], seed=3)
    out = _embed(c)
    mha = torch.nn.MultiheadAttention(H, NH, bias=False, batch_first=True, dtype=torch.float64)
    with torch.no_grad():
        mha.in_proj_weight.copy_(torch.from_numpy(np.concatenate(
            [oe.bf16_bits_to_f64(w) for w in (c.wq, c.wk, c.wv)])))
        mha.out_proj.weight.copy_(torch.from_numpy(oe.bf16_bits_to_f64(c.wo)))
    x = oe.bf16_bits_to_f64(c.x)
    pos = oe.bf16_bits_to_f64(c.pos)
    for b, n in enumerate(c.counts):
        xs = x[c.offsets[b]:c.offsets[b + 1]]
        q = torch.from_numpy(xs.mean(axis=0))[None, None, :]
        kv = torch.from_numpy(xs + pos[:n])[None]
        with torch.no_grad():
            ref, _ = mha(q, kv, kv, need_weights=False)
        np.testing.assert_allclose(out[b], ref[0, 0].numpy(), rtol=1e-10, atol=1e-12)


def test_order_matters_only_through_the_position_embeddings():
    c = _case([4, 3], seed=5)
    x = c.x.copy()
    perm = np.array([2, 0, 3, 1])
    xp = x.copy()
    xp[0:4] = x[0:4][perm]
    zero = np.zeros_like(c.pos)
    # without position embeddings the mean query and the weighted sum are symmetric
    np.testing.assert_allclose(_embed(c, pos=zero, x=xp)[0], _embed(c, pos=zero, x=x)[0],
                               rtol=1e-12, atol=1e-12)
    # with them, the fused state depends on the order (the module is permutation-variant)
    assert np.max(np.abs(_embed(c, x=xp)[0] - _embed(c, x=x)[0])) > 1e-3


@pytest.mark.parametrize("n", [2, 3, 4])
def test_identical_tokens_give_the_projected_value(n):
    """n copies of one embedding, no position embeddings: every key is equal, so whatever the
    weights, the output is W_o W_v x."""
    c = _case([n], seed=7)
    x = c.x.copy()
    x[:] = x[0]
    out = _embed(c, pos=np.zeros_like(c.pos), x=x)[0]
    x0 = oe.bf16_bits_to_f64(x[0])
    want = oe.bf16_bits_to_f64(c.wo) @ (oe.bf16_bits_to_f64(c.wv) @ x0)
    np.testing.assert_allclose(out, want, rtol=1e-12, atol=1e-12)


def test_softmax_weights_sum_to_one():
    c = _case([4, 2], seed=9)
    a = oe.attention_weights(c.x, 4, c.wq, c.wk, c.pos, NH)
    assert a.shape == (NH, 4)
    assert np.all(a > 0)
    np.testing.assert_allclose(a.sum(axis=1), 1.0, rtol=0, atol=1e-14)


@pytest.mark.parametrize("counts", [[0, 2], [5, 1]])
def test_token_count_outside_one_to_four_is_an_error(counts):
    c = _case([1, 1])
    offsets = np.concatenate([[0], np.cumsum(counts)])
    x = np.zeros((int(offsets[-1]), H), np.uint16)
    with pytest.raises(ValueError):
        oe.embed(x, offsets, c.wq, c.wk, c.wv, c.wo, c.pos, NH)
