"""Shared test helpers: bf16 bit views and oracle views of a workload."""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300.workloads import Workload


def bits(t: torch.Tensor) -> np.ndarray:
    """uint16 bit patterns of a bf16 tensor (a copy)."""
    assert t.dtype == torch.bfloat16
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16).copy()


def from_bits(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)


def bf16_to_f64(a: np.ndarray) -> np.ndarray:
    """Exact values of bf16 bit patterns."""
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def dims_of(w: Workload) -> orc.Dims:
    s = w.shape
    return orc.Dims(s.num_heads, s.num_kv_groups, s.d_nope, s.d_rope, s.d_v, s.rank, s.hidden, s.sm_scale,
                    s.rope_style, s.rope_base)


def oracle_cache(w: Workload, c_kv: np.ndarray | None = None, k_rope: np.ndarray | None = None) -> orc.Cache:
    """Oracle view of the workload's cache (copies of the bit patterns unless given)."""
    s = w.shape
    c = bits(w.c_kv) if c_kv is None else c_kv
    k = bits(w.k_rope) if k_rope is None else k_rope
    blk_tokens = c.shape[1]
    bt = None if w.block_table is None else w.block_table.numpy().astype(np.int32).copy()
    return orc.Cache(c_kv=c, k_rope=k, c_tok_stride=s.rank, r_tok_stride=s.d_rope,
                     c_blk_stride=blk_tokens * s.rank, r_blk_stride=blk_tokens * s.d_rope,
                     capacity=w.capacity, block_table=bt, page_size=s.page_size if s.paged else 0,
                     num_pages=w.num_pages)


def oracle_step(w: Workload, seqs=None, with_append: bool = True) -> dict:
    """Append this step's entries, then run the decode step, all in the oracle."""
    dims = dims_of(w)
    cache = oracle_cache(w)
    if with_append:
        orc.cache_append(dims, cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    res = orc.mla_decode(dims, cache, bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk),
                         bits(w.w_uv), None if w.w_o is None else bits(w.w_o), seqs=seqs)
    res["cache"] = cache
    return res


def rope_complex(x: np.ndarray, pos, base: float = 10000.0, style: int = 0) -> np.ndarray:
    """RoPE written as complex multiplication z_k * exp(i * pos * theta_k),
    theta_k = base^(-2k/d) (the RoFormer form the paper cites in Sec. 3.1).
    Independent of the oracle's real cos/sin form; ``pos`` broadcasts over the
    leading axes of ``x``."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    theta = base ** (-np.arange(half, dtype=np.float64) * 2.0 / d)
    if style == 0:
        z = x[..., :half] + 1j * x[..., half:]
    else:
        z = x[..., 0::2] + 1j * x[..., 1::2]
    ang = np.asarray(pos, dtype=np.float64)[..., None] * theta
    z = z * np.exp(1j * ang)
    y = np.empty_like(x)
    if style == 0:
        y[..., :half], y[..., half:] = z.real, z.imag
    else:
        y[..., 0::2], y[..., 1::2] = z.real, z.imag
    return y


def rel_errors(got: np.ndarray, ref: np.ndarray):
    """(max|d| / max|ref|, sum|d| / sum|ref|): the two parity measures."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    d = np.abs(got - ref)
    return float(d.max() / max(np.abs(ref).max(), 1e-300)), float(d.sum() / max(np.abs(ref).sum(), 1e-300))
