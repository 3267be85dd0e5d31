"""Compositional embedder of HAMburger, plain fp64 numpy (TEST INFRASTRUCTURE ONLY: the
tests, `__graft_entry__.smoke()` and the CPU-baseline leg of `bench.py` use it; the product
path never imports this package).

What it computes (Sec. 3.2 "Compositional Embedder", Sec. 3.4, Sec. 4.1): the tokens a
macro-step produced (1..4 of them) are fused into one hidden state of the model width H
before the base model's next forward.  A cross-attention with the mean of the inputs as the
query reads keys and values computed from the token embeddings, to which a learned position
embedding of the token's place inside the patch is added; a linear layer follows.  A list of
one token skips the module: the hidden state is that token's embedding.

Readings where the paper leaves details open, taken here:
  E1  the query comes from the mean of the raw token embeddings x_i;
  E2  keys and values come from u_i = x_i + P[i], P[i] the learned embedding of place i;
  E3  multi-head attention of the base model's head layout (H = n_heads * head_dim), scale
      1/sqrt(head_dim), no biases; the output linear is one H x H matrix W_o (a second linear
      without a non-linearity in between would compose into it);
  E4  one token: the output is that token's embedding, bit for bit.

For sequence b with tokens x_0..x_{n-1} (rows offsets[b]..offsets[b+1]-1 of X), n >= 2:
    m   = (1/n) sum_i x_i
    q   = W_q m,   k_i = W_k u_i,   v_i = W_v u_i,   u_i = x_i + P[i]
    per head h (slices of head_dim):  a = softmax_i(q_h . k_{i,h} / sqrt(head_dim)),
                                      o_h = sum_i a_i v_{i,h}
    e_b = W_o o
Weights are stored [out][in] (y = W x), as bf16 bit patterns like every input here.
"""
from __future__ import annotations

import numpy as np


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact value of bf16 bit patterns (the upper half of an fp32)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def softmax(s: np.ndarray) -> np.ndarray:
    """exp(s - max) / sum, fp64."""
    e = np.exp(s - np.max(s))
    return e / np.sum(e)


def embed(x_bits, offsets, wq_bits, wk_bits, wv_bits, wo_bits, pos_bits, n_heads,
          return_o=False):
    """Fused hidden state of every sequence, fp64 [B][H] (Sec. 3.2 "Compositional Embedder":
    the mean of a sequence's token embeddings queries the embeddings plus their in-patch position
    embeddings, multi-head, then a linear layer; Sec. 3.4: a single token bypasses it); with
    return_o also the attention output o [B][H] that enters the output linear (zeros for
    single-token sequences)."""
    x = bf16_bits_to_f64(x_bits)
    wq, wk, wv, wo = (bf16_bits_to_f64(w) for w in (wq_bits, wk_bits, wv_bits, wo_bits))
    pos = bf16_bits_to_f64(pos_bits)
    offsets = np.asarray(offsets, dtype=np.int64)
    B, H = len(offsets) - 1, x.shape[1]
    hd = H // n_heads
    out = np.zeros((B, H))
    o_rows = np.zeros((B, H))
    for b in range(B):
        xs = x[offsets[b]:offsets[b + 1]]
        n = len(xs)
        if n < 1 or n > len(pos):
            raise ValueError(f"sequence {b} has {n} tokens")
        if n == 1:                      # E4: the single token passes through
            out[b] = xs[0]
            continue
        m = xs.mean(axis=0)             # E1
        u = xs + pos[:n]                # E2
        q = wq @ m
        k = u @ wk.T
        v = u @ wv.T
        o = np.zeros(H)
        for h in range(n_heads):        # E3
            sl = slice(h * hd, (h + 1) * hd)
            a = softmax(k[:, sl] @ q[sl] / np.sqrt(hd))
            o[sl] = a @ v[:, sl]
        out[b] = wo @ o
        o_rows[b] = o
    return (out, o_rows) if return_o else out


def attention_weights(x_bits, n_tokens_first, wq_bits, wk_bits, pos_bits, n_heads):
    """Softmax weights [n_heads][n] of the first sequence (for the sum-to-one pin): the
    cross-attention of `embed` (Sec. 3.2), weights only."""
    x = bf16_bits_to_f64(x_bits)[:n_tokens_first]
    wq, wk = bf16_bits_to_f64(wq_bits), bf16_bits_to_f64(wk_bits)
    pos = bf16_bits_to_f64(pos_bits)
    H = x.shape[1]
    hd = H // n_heads
    q = wq @ x.mean(axis=0)
    k = (x + pos[:n_tokens_first]) @ wk.T
    return np.stack([softmax(k[:, h * hd:(h + 1) * hd] @ q[h * hd:(h + 1) * hd] / np.sqrt(hd))
                     for h in range(n_heads)])
