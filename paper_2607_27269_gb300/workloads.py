"""Seeded synthetic inputs for the MLA decode step.

This module only draws numbers and lays them out; it holds none of the
attention arithmetic, so both the CUDA path and the CPU oracle can consume it.

Five workloads mirror the draft-model shapes the method is evaluated on: a
tiny single layer, a Qwen2.5-0.5B-shaped layer, a Llama-3.2-1B-shaped layer in
a gamma+1 = 5 token speculative chunk (gamma = 4, Sec. 5.2), a Llama-3.2-3B-
shaped long-context layer, and a paged ragged batch of the Llama-3.2-1B shape
with 5 appended entries per sequence.  The paper evaluates on natural-language
prompt sets; these synthetic tensors stand in for the caches and queries those
prompts would produce.

Recipe (one ``torch.Generator('cpu')`` seeded with ``seed``, drawn in this order):
  1. per-sequence lengths (uniform integers in the stated range);
  2. for paged caches, a random permutation of the physical page ids;
  3. W_UK [G, d_nope, r], W_UV [G, d_v, r] ~ N(0, 1/sqrt(r));
     W_O [D, H*d_v] ~ N(0, 1/sqrt(H*d_v));
  4. latent cache c_kv and positional-key cache k_rope ~ N(0, 1) (the stored
     k_rope values are taken as already rotated);
  5. q_nope [B, q, H, d_nope], q_pe [B, q, H, d_rope] ~ N(0, 1);
  6. the entries appended this step, c_new [B, q, r], kr_new [B, q, d_rope]
     ~ N(0, 1) (kr_new not yet rotated).
Every tensor is drawn in fp32 and rounded to bf16.

Draft and target logits for the acceptance statistics (``logits``) come from a
third generator seeded with ``seed + 104729``: target rows ~ N(0, 3^2) over the
vocabulary of the model the shape follows (a peaked distribution: the largest
of ~10^5 draws sits ~4.5 sigma out), draft = target + N(0, 1) (a draft that
mostly agrees), both rounded to bf16; one row per (sequence, query position).

The original GQA layer at the same shape (``gqa``: the draft before conversion,
head width d = d_v of the shape for keys and values alike, one key and value
cache per KV group) keeps the MLA workload's lengths, positions and page
counts and draws from a fourth generator seeded with ``seed + 15485863``: the
page permutation (paged), key and value caches ~ N(0, 1) (keys taken as
already rotated), queries q [B, q_len, H, d] and this step's new keys and
values [B, q_len, G, d] ~ N(0, 1).

Inputs of the projection that precedes the step (``projection``) come from a
second generator seeded with ``seed + 7919``, drawn in this order: hidden
states h [B, q, D] ~ N(0, 1); W^DKV [r, D], W^KR [d_rope, D] and
W^Q [H (d_nope + d_rope), D] ~ N(0, 1/sqrt(D)), so that the projected latents
and keys have unit variance like the cache above.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional

import torch

PAGE = 64


@dataclass(frozen=True)
class Shape:
    name: str
    batch: int
    num_heads: int
    num_kv_groups: int
    d_nope: int
    d_rope: int
    d_v: int
    rank: int
    hidden: int            # 0: no output projection W_O
    q_len: int
    kv_lo: int             # kv_len range at attention time (inclusive), after the append
    kv_hi: int
    paged: bool = False
    page_size: int = PAGE
    rope_base: float = 10000.0
    rope_style: int = 0

    @property
    def sm_scale(self) -> float:
        # 1/sqrt(d_k) with d_k the converted head's query-key width (Sec. 3.1, 3.3).
        return 1.0 / math.sqrt(self.d_nope + self.d_rope)

    @property
    def rows(self) -> int:
        return self.q_len * self.num_heads


# The five workloads (name: what it is, with its sizes).
SHAPES = {
    "tiny_b1_h8_r128_t256": Shape("tiny_b1_h8_r128_t256", 1, 8, 8, 64, 32, 64, 128, 0, 1, 256, 256),
    "qwen05b_b16_h14_r256_t2048": Shape("qwen05b_b16_h14_r256_t2048", 16, 14, 2, 64, 64, 64, 256, 896, 1,
                                        2048, 2048),
    "llama1b_chunk5_b32_h32_r512_t4096": Shape("llama1b_chunk5_b32_h32_r512_t4096", 32, 32, 8, 64, 64, 64,
                                               512, 2048, 5, 4096, 4096),
    "llama3b_long_b8_h24_r512_t16k_32k": Shape("llama3b_long_b8_h24_r512_t16k_32k", 8, 24, 8, 128, 64, 128,
                                               512, 3072, 1, 16384, 32768),
    # pre-append lengths U[128, 8192] plus the 5 appended entries
    "llama1b_paged_b128_h32_r512_t128_8192": Shape("llama1b_paged_b128_h32_r512_t128_8192", 128, 32, 8, 64,
                                                   64, 64, 512, 2048, 5, 128 + 5, 8192 + 5, paged=True),
}
ORDER = list(SHAPES)


@dataclass
class Workload:
    shape: Shape
    kv_len: torch.Tensor          # int32 [B], cache length at attention time (after the append)
    start_pos: torch.Tensor       # int32 [B], position of the first appended entry = kv_len - q_len
    capacity: int                 # tokens a sequence may hold
    c_kv: torch.Tensor            # bf16 [blocks, block_tokens, r]
    k_rope: torch.Tensor          # bf16 [blocks, block_tokens, d_rope]
    block_table: Optional[torch.Tensor]  # int32 [B, max_pages] (paged) or None
    num_pages: int
    w_uk: torch.Tensor            # bf16 [G, d_nope, r]
    w_uv: torch.Tensor            # bf16 [G, d_v, r]
    w_o: Optional[torch.Tensor]   # bf16 [D, H*d_v] or None
    q_nope: torch.Tensor          # bf16 [B, q, H, d_nope]
    q_pe: torch.Tensor            # bf16 [B, q, H, d_rope]
    c_new: torch.Tensor           # bf16 [B, q, r]
    kr_new: torch.Tensor          # bf16 [B, q, d_rope]
    extra: dict = field(default_factory=dict)

    @property
    def cache_tokens(self) -> int:
        return int(self.kv_len.sum())

    @property
    def cache_bytes(self) -> int:
        """Bytes of latent + positional cache one attention step must read."""
        s = self.shape
        return self.cache_tokens * (s.rank + s.d_rope) * 2


def _randn(gen: torch.Generator, shape, std: float = 1.0) -> torch.Tensor:
    t = torch.randn(*shape, generator=gen, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(torch.bfloat16)


def make(shape: Shape | str, seed: int = 0, batch: Optional[int] = None, kv_range=None,
         q_len: Optional[int] = None, capacity: Optional[int] = None, shuffle_pages: bool = True,
         spare_pages: int = 0) -> Workload:
    """Draw one workload.  ``batch``, ``kv_range``, ``q_len`` and ``capacity``
    override the shape's sizes (used for small test cases of the same shape)."""
    if isinstance(shape, str):
        shape = SHAPES[shape]
    B = shape.batch if batch is None else batch
    q = shape.q_len if q_len is None else q_len
    lo, hi = (shape.kv_lo, shape.kv_hi) if kv_range is None else kv_range
    lo = max(lo, q)
    hi = max(hi, lo)
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed)

    if lo == hi:
        kv = torch.full((B,), lo, dtype=torch.int32)
    else:
        kv = torch.randint(lo, hi + 1, (B,), generator=gen, dtype=torch.int64).to(torch.int32)
    H, G, r, dr = shape.num_heads, shape.num_kv_groups, shape.rank, shape.d_rope

    if shape.paged:
        ps = shape.page_size
        pages_per_seq = [(int(k) + ps - 1) // ps for k in kv]
        max_pages = max(pages_per_seq) if B else 1
        num_pages = sum(pages_per_seq) + spare_pages
        perm = torch.randperm(num_pages, generator=gen) if shuffle_pages else torch.arange(num_pages)
        bt = torch.full((B, max(max_pages, 1)), -1, dtype=torch.int32)
        nxt = 0
        for b, npg in enumerate(pages_per_seq):
            bt[b, :npg] = perm[nxt:nxt + npg].to(torch.int32)
            nxt += npg
        cap = max_pages * ps if capacity is None else capacity
        blocks, block_tokens = num_pages, ps
    else:
        bt = None
        num_pages = 0
        cap = int(kv.max()) if capacity is None else capacity
        if B == 0:
            cap = max(cap, 1) if capacity is None else capacity
        blocks, block_tokens = B, cap

    w_uk = _randn(gen, (G, shape.d_nope, r), 1.0 / math.sqrt(r))
    w_uv = _randn(gen, (G, shape.d_v, r), 1.0 / math.sqrt(r))
    w_o = _randn(gen, (shape.hidden, H * shape.d_v), 1.0 / math.sqrt(H * shape.d_v)) if shape.hidden else None
    c_kv = _randn(gen, (blocks, block_tokens, r))
    k_rope = _randn(gen, (blocks, block_tokens, dr))
    q_nope = _randn(gen, (B, q, H, shape.d_nope))
    q_pe = _randn(gen, (B, q, H, dr))
    c_new = _randn(gen, (B, q, r))
    kr_new = _randn(gen, (B, q, dr))
    return Workload(shape=shape, kv_len=kv, start_pos=(kv - q).to(torch.int32), capacity=cap, c_kv=c_kv,
                    k_rope=k_rope, block_table=bt, num_pages=num_pages, w_uk=w_uk, w_uv=w_uv, w_o=w_o,
                    q_nope=q_nope, q_pe=q_pe, c_new=c_new, kr_new=kr_new)


def small(name: str, seed: int = 0) -> Workload:
    """A reduced case of a shape that the oracle finishes in seconds but that
    still spans several 128-token tiles and ends on a ragged tail."""
    s = SHAPES[name]
    if name.startswith("tiny"):
        return make(s, seed)
    if s.paged:
        return make(s, seed, batch=6, kv_range=(s.q_len + 1, 700))
    if s.kv_lo != s.kv_hi:
        return make(s, seed, batch=3, kv_range=(300, 1100))
    return make(s, seed, batch=3, kv_range=(517, 517))


@dataclass
class Projection:
    """Hidden states and stacked projection weights of the step's new tokens."""
    hidden: int                   # D
    h: torch.Tensor               # bf16 [B, q, D]
    w_dkv: torch.Tensor           # bf16 [r, D]
    w_kr: torch.Tensor            # bf16 [d_rope, D]
    w_q: torch.Tensor             # bf16 [H (d_nope + d_rope), D]


def projection(w: Workload, seed: int = 0, hidden: Optional[int] = None) -> Projection:
    """Projection inputs for workload ``w``'s new tokens; D = the shape's
    hidden width (256 for a shape without one) unless ``hidden`` is given."""
    s = w.shape
    D = hidden if hidden is not None else (s.hidden if s.hidden > 0 else 256)
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 7919)
    B, q = w.c_new.shape[0], w.c_new.shape[1]
    std = 1.0 / math.sqrt(D)
    h = _randn(gen, (B, q, D))
    w_dkv = _randn(gen, (s.rank, D), std)
    w_kr = _randn(gen, (s.d_rope, D), std)
    w_q = _randn(gen, (s.num_heads * (s.d_nope + s.d_rope), D), std)
    return Projection(D, h, w_dkv, w_kr, w_q)


# Vocabulary of the model each shape follows (Qwen2.5, Llama-3.2; the tiny
# layer gets a small one).
VOCAB = {
    "tiny_b1_h8_r128_t256": 32000,
    "qwen05b_b16_h14_r256_t2048": 151936,
    "llama1b_chunk5_b32_h32_r512_t4096": 128256,
    "llama3b_long_b8_h24_r512_t16k_32k": 128256,
    "llama1b_paged_b128_h32_r512_t128_8192": 128256,
}


@dataclass
class Logits:
    draft: torch.Tensor           # bf16 [rows, vocab]
    target: torch.Tensor          # bf16 [rows, vocab]


def logits(name: str, seed: int = 0, rows: Optional[int] = None, vocab: Optional[int] = None) -> Logits:
    """Draft / target logits for shape ``name``: rows = batch * q_len unless given."""
    s = SHAPES[name]
    R = s.batch * s.q_len if rows is None else rows
    V = VOCAB[name] if vocab is None else vocab
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 104729)
    t = torch.randn(R, V, generator=gen, dtype=torch.float32) * 3.0
    d = t + torch.randn(R, V, generator=gen, dtype=torch.float32)
    return Logits(d.to(torch.bfloat16), t.to(torch.bfloat16))


@dataclass
class GqaWorkload:
    """The original GQA layer at a shape: caches, queries and new entries."""
    shape: Shape
    num_heads: int
    num_kv_groups: int
    d: int                        # key and value width per head
    kv_len: torch.Tensor          # int32 [B]
    start_pos: torch.Tensor       # int32 [B]
    capacity: int
    k_cache: torch.Tensor         # bf16 [blocks, block_tokens, d] (rotated keys)
    v_cache: torch.Tensor         # bf16 [blocks, block_tokens, d]
    block_table: Optional[torch.Tensor]  # int32 [B * G, pages] (paged) or None
    num_pages: int
    q: torch.Tensor               # bf16 [B, q_len, H, d]
    k_new: torch.Tensor           # bf16 [B, q_len, G, d] (not rotated)
    v_new: torch.Tensor           # bf16 [B, q_len, G, d]

    @property
    def sm_scale(self) -> float:
        return 1.0 / math.sqrt(self.d)

    @property
    def cache_bytes(self) -> int:
        """Key and value bytes one attention step reads (every group's cache)."""
        return int(self.kv_len.sum()) * self.num_kv_groups * 2 * self.d * 2


def gqa(w: Workload, seed: int = 0) -> GqaWorkload:
    """The original GQA layer for workload ``w`` (its lengths and layout)."""
    s = w.shape
    B, q = w.kv_len.numel(), w.q_nope.shape[1]
    G, H, d = s.num_kv_groups, s.num_heads, s.d_v
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 15485863)
    if s.paged:
        ps = s.page_size
        pages_per_seq = [(int(k) + ps - 1) // ps for k in w.kv_len]
        max_pages = max(pages_per_seq) if B else 1
        num_pages = G * sum(pages_per_seq)
        perm = torch.randperm(num_pages, generator=gen)
        bt = torch.full((B * G, max(max_pages, 1)), -1, dtype=torch.int32)
        nxt = 0
        for b, npg in enumerate(pages_per_seq):
            for g in range(G):
                bt[b * G + g, :npg] = perm[nxt:nxt + npg].to(torch.int32)
                nxt += npg
        blocks, block_tokens, cap = num_pages, ps, max_pages * ps
    else:
        bt, num_pages = None, 0
        blocks, block_tokens, cap = B * G, w.capacity, w.capacity
    k_cache = _randn(gen, (blocks, block_tokens, d))
    v_cache = _randn(gen, (blocks, block_tokens, d))
    qq = _randn(gen, (B, q, H, d))
    k_new = _randn(gen, (B, q, G, d))
    v_new = _randn(gen, (B, q, G, d))
    return GqaWorkload(s, H, G, d, w.kv_len.clone(), w.start_pos.clone(), cap, k_cache, v_cache, bt, num_pages, qq,
                       k_new, v_new)


@dataclass
class GqaProjection:
    """Projection weights of the original GQA layer (its W_O is the shared one)."""
    w_q: torch.Tensor             # bf16 [H d, D]
    w_k: torch.Tensor             # bf16 [G d, D]
    w_v: torch.Tensor             # bf16 [G d, D]


def gqa_projection(w: Workload, seed: int = 0, hidden: Optional[int] = None) -> GqaProjection:
    """W_Q, W_K, W_V ~ N(0, 1/sqrt(D)) of the original layer at ``w``'s shape
    (a fifth generator, seed + 32452843); D as in ``projection``."""
    s = w.shape
    D = hidden if hidden is not None else (s.hidden if s.hidden > 0 else 256)
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed + 32452843)
    std = 1.0 / math.sqrt(D)
    d = s.d_v
    return GqaProjection(_randn(gen, (s.num_heads * d, D), std), _randn(gen, (s.num_kv_groups * d, D), std),
                         _randn(gen, (s.num_kv_groups * d, D), std))
