"""Seeded synthetic inputs for smashed-KV decode attention.

This module only draws inputs: bf16 query/key/value bits, per-slot token
counts, slot counts and page tables.  It holds none of the attention, RoPE or
append arithmetic, so both the CUDA path and the CPU oracle can be fed from it
without sharing any of the method's code.

Workloads stand in for the paper's decode workloads (short-context GSM8K /
HumanEval / MGSM and long-context MultiNews / LongBench decoding, Sec. 4.3 and
Fig. 5); the datasets and trained weights are not used.  A slot is one
"smashed" KV entry that stands for 1..4 tokens (Sec. 3.1 and Sec. 3.7, token
fusion), with at most 4 tokens per macro-step (Sec. 4.1).

Token counts per slot follow a geometric law with p = 0.5 whose tail is folded
into 4: P(1)=1/2, P(2)=1/4, P(3)=1/8, P(4)=1/8 (mean 1.875).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Sequence

import numpy as np

# Maximum micro-step size: a macro-step emits (so a slot fuses) at most 4 tokens (Sec. 4.1).
MAX_TOKENS_PER_SLOT = 4


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and value distribution of one decode-attention workload."""

    name: str
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    page_slots: int
    layers: int
    slots: int = 0                       # slots per sequence (uniform batches)
    slot_range: Optional[tuple] = None   # inclusive (lo, hi) for ragged batches
    value_scale: float = 1.0             # std of q, K, V
    seed: int = 0
    pool_factor: float = 1.25            # pool pages / pages needed
    scatter_pages: bool = True           # random page table vs sequential
    attend_then_append: bool = False     # step order stated by the workload

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads


# Tiny CPU-checkable case: 1 sequence, 8/2 heads, d=64, 2 pages of 128 slots.  The cache
# is built by 255 appends at slot positions 0..254; the decode step appends slot 255 (so
# positions run 0..255 and the 256 slots fill both pages) and attends over all 256.
C0_TINY = Workload("tiny_b1_h8x2_d64_s256_p128", batch=1, n_q_heads=8, n_kv_heads=2,
                   head_dim=64, page_slots=128, layers=1, slots=255, value_scale=1.0,
                   seed=0, pool_factor=1.0, scatter_pages=False)
# Llama-3-8B-shaped layer: batch 8, 32/8 heads, d=128, 4096 slots, 16-slot scattered pages.
C1_LLAMA8B = Workload("llama8b_layer_b8_s4096", batch=8, n_q_heads=32, n_kv_heads=8,
                      head_dim=128, page_slots=16, layers=1, slots=4096,
                      value_scale=1.0 / math.sqrt(128.0), seed=1)
# The same layer at 8192 slots per sequence: the smallest batch-8 case with 8k slots.
C1_LLAMA8B_S8K = dataclasses.replace(C1_LLAMA8B, name="llama8b_layer_b8_s8192", slots=8192)
# Ragged serving batch: 64 sequences, slots uniform in [512, 8192], attend then append.
C2_RAGGED = Workload("ragged_b64_s512to8192", batch=64, n_q_heads=32, n_kv_heads=8,
                     head_dim=128, page_slots=16, layers=1, slot_range=(512, 8192),
                     value_scale=1.0, seed=2, attend_then_append=True)
# Long context: batch 4, 65536 slots (~123k tokens at 1.875 tokens per slot).
C3_LONG = Workload("long_b4_s65536", batch=4, n_q_heads=32, n_kv_heads=8, head_dim=128,
                   page_slots=16, layers=1, slots=65536, value_scale=1.0, seed=3)


def c4_sweep(batch: int, slots: int = 2048, layers: int = 32) -> Workload:
    """32-layer decode stack of the Llama-8B layer shape, starting from 2048 slots."""
    return Workload(f"stack_l{layers}_b{batch}_s{slots}", batch=batch, n_q_heads=32,
                    n_kv_heads=8, head_dim=128, page_slots=16, layers=layers, slots=slots,
                    value_scale=1.0 / math.sqrt(128.0), seed=4)


WORKLOADS = {w.name: w for w in (C0_TINY, C1_LLAMA8B, C1_LLAMA8B_S8K, C2_RAGGED, C3_LONG)}


def scaled(w: Workload, **changes) -> Workload:
    """Same workload with some fields replaced (smaller parity cases)."""
    return dataclasses.replace(w, **changes)


# ----------------------------------------------------------------------------
# draws
# ----------------------------------------------------------------------------

def rng_for(seed: int, stream: int = 0) -> np.random.Generator:
    """Independent PCG64 stream per (seed, purpose)."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream])))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even) and return the raw uint16 bits.

    Used only to turn drawn normals into bf16 inputs; finite inputs only.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16(rng: np.random.Generator, shape: Sequence[int], scale: float = 1.0,
                block: int = 1 << 24) -> np.ndarray:
    """bf16 bits of N(0, scale^2) draws, generated in blocks to bound host memory."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint16)
    for s in range(0, n, block):
        e = min(n, s + block)
        x = rng.standard_normal(e - s, dtype=np.float32)
        if scale != 1.0:
            x *= np.float32(scale)
        out[s:e] = f32_to_bf16_bits(x)
    return out.reshape(shape)


def ntok_capped_geometric(rng: np.random.Generator, shape, p: float = 0.5,
                          cap: int = MAX_TOKENS_PER_SLOT) -> np.ndarray:
    """Tokens fused into each slot: geometric(p) on {1, 2, ...}, tail folded into `cap`."""
    return np.minimum(rng.geometric(p, size=shape), cap).astype(np.int32)


def slot_counts(w: Workload, rng: np.random.Generator) -> np.ndarray:
    if w.slot_range is not None:
        lo, hi = w.slot_range
        return rng.integers(lo, hi + 1, size=w.batch).astype(np.int32)
    return np.full(w.batch, w.slots, dtype=np.int32)


def pages_needed(max_slots: int, page_slots: int) -> int:
    return -(-max_slots // page_slots)


def page_table(rng: np.random.Generator, batch: int, max_pages: int, pool_pages: int,
               scatter: bool = True) -> np.ndarray:
    """[batch][max_pages] distinct page ids drawn from a pool of `pool_pages`."""
    need = batch * max_pages
    if need > pool_pages:
        raise ValueError(f"pool of {pool_pages} pages cannot hold {need}")
    ids = rng.permutation(pool_pages)[:need] if scatter else np.arange(need)
    return ids.astype(np.int32).reshape(batch, max_pages)


@dataclasses.dataclass
class HostCase:
    """A whole decode-attention case on the host (bf16 as uint16 bits)."""

    w: Workload
    num_slots: np.ndarray        # [B] int32: slots already in the cache
    max_slots: int               # capacity per sequence (slots)
    pool_pages: int
    page_table: np.ndarray       # [B][max_pages] int32
    k: np.ndarray                # [B][Lmax][Hkv][d] uint16 (already rotated keys)
    v: np.ndarray                # [B][Lmax][Hkv][d] uint16
    slot_ntok: np.ndarray        # [B][Lmax] int32
    slot_pos: np.ndarray         # [B][Lmax] int32 (slot index)
    q: np.ndarray                # [B][Hq][d] uint16 (already rotated query)
    k_new: np.ndarray            # [B][Hkv][d] uint16 (unrotated key of the new slot)
    v_new: np.ndarray            # [B][Hkv][d] uint16
    ntok_new: np.ndarray         # [B] int32

    @property
    def lmax(self) -> int:
        return self.k.shape[1]


def make_case(w: Workload, extra_slots: int = 1, num_slots: Optional[np.ndarray] = None,
              pool_pages: Optional[int] = None) -> HostCase:
    """Draw every input of workload `w` on the host from its seed.

    `extra_slots` is the headroom per sequence for appends after the cache is filled.
    """
    counts = slot_counts(w, rng_for(w.seed, 1)) if num_slots is None else \
        np.asarray(num_slots, dtype=np.int32)
    lmax = int(counts.max()) if counts.size else 0
    max_slots = lmax + extra_slots
    max_pages = pages_needed(max(max_slots, 1), w.page_slots)
    if pool_pages is None:
        pool_pages = int(math.ceil(w.batch * max_pages * w.pool_factor))
    pt = page_table(rng_for(w.seed, 2), w.batch, max_pages, pool_pages, w.scatter_pages)
    shape = (w.batch, lmax, w.n_kv_heads, w.head_dim)
    k = normal_bf16(rng_for(w.seed, 3), shape, w.value_scale)
    v = normal_bf16(rng_for(w.seed, 4), shape, w.value_scale)
    ntok = ntok_capped_geometric(rng_for(w.seed, 5), (w.batch, lmax))
    pos = np.broadcast_to(np.arange(lmax, dtype=np.int32), (w.batch, lmax)).copy()
    for b in range(w.batch):           # slots past a sequence's length are unused
        ntok[b, counts[b]:] = 0
        pos[b, counts[b]:] = 0
    q = normal_bf16(rng_for(w.seed, 6), (w.batch, w.n_q_heads, w.head_dim), w.value_scale)
    k_new = normal_bf16(rng_for(w.seed, 7), (w.batch, w.n_kv_heads, w.head_dim), w.value_scale)
    v_new = normal_bf16(rng_for(w.seed, 8), (w.batch, w.n_kv_heads, w.head_dim), w.value_scale)
    ntok_new = ntok_capped_geometric(rng_for(w.seed, 9), (w.batch,))
    return HostCase(w, counts, max_slots, pool_pages, pt, k, v, ntok, pos, q, k_new, v_new,
                    ntok_new)


# ---------------------------------------------------------------------------------------
# Chunked prefill (prompt ingestion): prompt tokens are not fused (Figure 2, training), so each
# becomes one slot with one token; the chunk's rows attend causally over the cache.
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass
class PrefillCase:
    base: HostCase               # the cache before the chunk (base.num_slots slots each)
    rows: np.ndarray             # [B] int32: new rows per sequence (0 allowed)
    offsets: np.ndarray          # [B+1] int32: sequence b owns rows offsets[b] .. offsets[b+1]-1
    q: np.ndarray                # [T][Hq][d] uint16: unrotated queries
    k_new: np.ndarray            # [T][Hkv][d] uint16: unrotated keys
    v_new: np.ndarray            # [T][Hkv][d] uint16
    ntok: np.ndarray             # [T] int32: tokens per new slot (1 for prompt tokens)

    @property
    def w(self) -> Workload:
        return self.base.w


def make_prefill_case(w: Workload, rows, cached=None, ntok=None,
                      headroom: int = 0) -> PrefillCase:
    """A chunk of rows[b] new rows per sequence over a cache holding cached[b] slots (the
    workload's own slot counts if None), with room for `headroom` more slots."""
    rows = np.asarray(rows, dtype=np.int32)
    base = make_case(w, extra_slots=int(rows.max(initial=0)) + headroom, num_slots=cached)
    offsets = np.concatenate([[0], np.cumsum(rows)]).astype(np.int32)
    T = int(offsets[-1])
    q = normal_bf16(rng_for(w.seed, 20), (T, w.n_q_heads, w.head_dim), w.value_scale)
    k_new = normal_bf16(rng_for(w.seed, 21), (T, w.n_kv_heads, w.head_dim), w.value_scale)
    v_new = normal_bf16(rng_for(w.seed, 22), (T, w.n_kv_heads, w.head_dim), w.value_scale)
    ntok = np.ones(T, np.int32) if ntok is None else np.asarray(ntok, np.int32)
    return PrefillCase(base, rows, offsets, q, k_new, v_new, ntok)


@dataclasses.dataclass(frozen=True)
class PrefillWorkload:
    name: str
    w: Workload                  # head shape, page size, value scale, seed
    rows: int                    # new rows per sequence
    cached: int                  # slots per sequence before the chunk


# Fresh 4096-token prompts of a Llama-3-8B layer, batch 4.
P1_PREFILL = PrefillWorkload("prefill_b4_s4096", dataclasses.replace(
    C1_LLAMA8B, name="prefill_b4_s4096", batch=4, slots=0, seed=11), rows=4096, cached=0)
# A 1024-row chunk over 3072 cached slots (the last chunk of a 4096-token prompt), batch 4.
P2_CHUNK = PrefillWorkload("prefill_b4_c1024_s3072", dataclasses.replace(
    C1_LLAMA8B, name="prefill_b4_c1024_s3072", batch=4, slots=3072, seed=12), rows=1024,
    cached=3072)
# A 64-row chunk over 65,536 cached slots, batch 1: few query blocks over a long cache (the
# attention splits over the cached slots).
P3_SHORT = PrefillWorkload("prefill_b1_c64_s65536", dataclasses.replace(
    C1_LLAMA8B, name="prefill_b1_c64_s65536", batch=1, slots=65536, seed=13), rows=64,
    cached=65536)
PREFILL_WORKLOADS = {p.name: p for p in (P1_PREFILL, P2_CHUNK, P3_SHORT)}


def device_normal_bf16(shape, scale: float, seed: int, device="cuda"):
    """bf16 N(0, scale^2) tensor drawn on the device from a seeded torch generator.

    Used where host generation would dominate start-up time (full-size bench workloads).
    """
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if scale != 1.0:
        x.mul_(scale)
    return x.to(torch.bfloat16)


# ---------------------------------------------------------------------------------------
# Compositional embedder inputs (Sec. 3.2): the tokens each sequence produced in the last
# macro-step (1..4, capped-geometric like the slots they become), their embeddings, and
# synthetic module weights (the trained ones are not used).  Llama-3.2-1B width: H = 2048,
# 32 heads of 64 (Sec. 4.1).
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class EmbedWorkload:
    name: str
    batch: int
    hidden: int = 2048
    n_heads: int = 32
    max_patch: int = MAX_TOKENS_PER_SLOT
    seed: int = 5
    vocab: int = 0          # > 0: tokens arrive as ids into a table of this many entries


@dataclasses.dataclass
class EmbedCase:
    w: EmbedWorkload
    counts: np.ndarray      # [B] tokens per sequence, 1..max_patch
    offsets: np.ndarray     # [B+1] prefix of counts: sequence b owns rows offsets[b].. of x
    x: np.ndarray           # bf16 bits [T][H]: token embeddings, N(0, 1)
    wq: np.ndarray          # bf16 bits [H][H] ([out][in]), N(0, 1/H)
    wk: np.ndarray
    wv: np.ndarray
    wo: np.ndarray
    pos: np.ndarray         # bf16 bits [max_patch][H]: position embeddings, N(0, 1)


def embed_workload(batch: int, **kw) -> EmbedWorkload:
    return EmbedWorkload(f"embed_b{batch}", batch=batch, **kw)


def embed_tokens_workload(batch: int, **kw) -> EmbedWorkload:
    """The embedder fed token ids of the Llama-3 vocabulary (width 2048, as Llama-3.2-1B)."""
    kw.setdefault("vocab", LLAMA3_VOCAB)
    return EmbedWorkload(f"embedtok_b{batch}", batch=batch, **kw)


def make_embed_case(w: EmbedWorkload, counts: Optional[np.ndarray] = None) -> EmbedCase:
    rng = rng_for(w.seed, 40)
    if counts is None:
        counts = ntok_capped_geometric(rng, (w.batch,), cap=w.max_patch)
    counts = np.asarray(counts, dtype=np.int32)
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    H = w.hidden
    ws = 1.0 / math.sqrt(H)
    return EmbedCase(w, counts, offsets, normal_bf16(rng, (int(offsets[-1]), H)),
                     normal_bf16(rng, (H, H), ws), normal_bf16(rng, (H, H), ws),
                     normal_bf16(rng, (H, H), ws), normal_bf16(rng, (H, H), ws),
                     normal_bf16(rng, (w.max_patch, H)))


LLAMA3_VOCAB = 128256   # entries of the Llama-3 token-embedding table (width 2048 at 1B)


@dataclasses.dataclass
class EmbedTokensCase:
    case: EmbedCase         # the same weights and counts; case.x = table[ids]
    table: np.ndarray       # bf16 bits [vocab][H]: the token-embedding table, N(0, 1)
    ids: np.ndarray         # int32 [T]: token ids, uniform over the vocabulary


def make_embed_tokens_case(w: EmbedWorkload, vocab: int,
                           counts: Optional[np.ndarray] = None) -> EmbedTokensCase:
    """An embedder case whose tokens are ids into a seeded embedding table: the weights and
    counts of make_embed_case(w, counts), the embeddings gathered from the table."""
    c = make_embed_case(w, counts)
    rng = rng_for(w.seed, 41)
    table = normal_bf16(rng, (vocab, w.hidden))
    ids = rng.integers(0, vocab, int(c.offsets[-1]), dtype=np.int32)
    c.x = table[ids]
    return EmbedTokensCase(c, table, ids)


# ---------------------------------------------------------------------------------------
# Macro-step layer front: the layer input x of width H is projected to q, k, v by one fused
# bias-free weight [W_q; W_k; W_v] ([out][in]), as in the Llama base model (Sec. 4.1).  The
# weights are drawn N(0, 1/H) (so q, k, v are about N(0, 1) for x ~ N(0, 1)), the inputs
# N(0, 1), as a normalised hidden state is.
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class FrontWorkload:
    name: str
    batch: int
    hidden: int
    n_q_heads: int = 32
    n_kv_heads: int = 8
    head_dim: int = 128
    seed: int = 0

    @property
    def out_rows(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim


def front_workload(batch: int, hidden: int = 4096, **kw) -> FrontWorkload:
    """Llama-3-8B-shaped layer front (H 4096, 32/8 heads of 128) unless overridden."""
    return FrontWorkload(f"qkv_front_b{batch}_h{hidden}", batch=batch, hidden=hidden, **kw)


def front_inputs(w: FrontWorkload, stream: int = 0):
    """(x bits [B][H], weight bits [(Hq + 2 Hkv) d][H]) of one layer, seeded by (seed, stream)."""
    x = normal_bf16(rng_for(w.seed, 40 + 2 * stream), (w.batch, w.hidden), 1.0)
    wt = normal_bf16(rng_for(w.seed, 41 + 2 * stream), (w.out_rows, w.hidden),
                     1.0 / math.sqrt(w.hidden))
    return x, wt


# ---------------------------------------------------------------------------------------
# Micro-step decoder attention (Sec. 3.3, Sec. 4.1): four layers with the base model's
# configuration (Llama-3.2-1B: 32 query / 8 KV heads of 64) over a local cache holding
# `context` entries (hidden states of middle layers of the base model, already projected) and
# the micro-tokens of the current macro-step; a macro-step emits at most 4 tokens, the first
# from the base model itself (Sec. 3.4), so the decoder runs at most 3 micro-steps.
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class MicroWorkload:
    name: str
    batch: int
    layers: int = 4
    n_q_heads: int = 32
    n_kv_heads: int = 8
    head_dim: int = 64
    context: int = 4
    micro_steps: int = MAX_TOKENS_PER_SLOT - 1
    seed: int = 5


def micro_workload(batch: int, **kw) -> MicroWorkload:
    return MicroWorkload(f"micro_b{batch}", batch=batch, **kw)


def make_micro_case(w: MicroWorkload) -> HostCase:
    """One layer's local cache (w.context entries per sequence, one 16-slot page each) and the
    inputs of one micro-step, values N(0, 1)."""
    base = Workload(w.name, batch=w.batch, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                    head_dim=w.head_dim, page_slots=16, layers=1, value_scale=1.0, seed=w.seed,
                    pool_factor=1.0, scatter_pages=True)
    case = make_case(base, num_slots=np.full(w.batch, w.context, np.int32),
                     extra_slots=w.micro_steps + 1)
    case.ntok_new[:] = 1
    return case
