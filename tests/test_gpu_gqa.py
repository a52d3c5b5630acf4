"""GPU parity of the original-GQA decode path (mla_gqa_append,
mla_gqa_decode_attn; Sec. 3.1 Eqs. 1-4) against the fp64 oracle on the same
seeded inputs, at every workload's shape.

Bars: appended values bit-exact and keys within one bf16 rounding of the
exact rotation (as for the MLA append); attention outputs within
max|d| <= 2e-2 max|ref| and mean relative error <= 5e-3 (the softmax weights
are rounded to bf16 before they multiply the bf16 values, as in the MLA path).
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, rel_errors

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 5e-3


def assert_close(got, ref, what):
    mx, mean = rel_errors(got, ref)
    assert mx <= MAX_TOL and mean <= MEAN_TOL, f"{what}: max {mx:.3e} mean {mean:.3e}"


def devices(gw, splits=0):
    s = gw.shape
    dims = abi.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
    bt = None if gw.block_table is None else gw.block_table.cuda()
    cache = abi.Cache(gw.v_cache.cuda(), gw.k_cache.cuda(), gw.capacity, bt, s.page_size if s.paged else 0,
                      gw.num_pages)
    step = abi.GqaStep(dims, cache, gw.kv_len.numel(), gw.q.shape[1], int(gw.kv_len.max()), splits)
    return dims, cache, step


def oracle_run(gw):
    s = gw.shape
    dims = orc.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
    bt = None if gw.block_table is None else gw.block_table.numpy().astype(np.int32).copy()
    cache = orc.Cache(c_kv=bits(gw.v_cache), k_rope=bits(gw.k_cache), c_tok_stride=gw.d, r_tok_stride=gw.d,
                      c_blk_stride=gw.k_cache.shape[1] * gw.d, r_blk_stride=gw.k_cache.shape[1] * gw.d,
                      capacity=gw.capacity, block_table=bt, page_size=s.page_size if s.paged else 0,
                      num_pages=gw.num_pages)
    orc.gqa_append(dims, cache, bits(gw.k_new), bits(gw.v_new), gw.start_pos.numpy())
    res = orc.gqa_decode(dims, cache, bits(gw.q), gw.kv_len.numpy())
    return cache, res


def run(gw, splits=0):
    dims, cache, step = devices(gw, splits)
    abi.gqa_append(dims, cache, gw.k_new.cuda(), gw.v_new.cuda(), gw.start_pos.cuda())
    o = step(gw.q.cuda(), gw.kv_len.cuda())
    code = abi.check_status()
    assert code == abi.MLA_OK, abi.status_name(code)
    return cache, step


@pytest.mark.parametrize("name", wl.ORDER)
def test_gqa_decode_matches_oracle(name):
    w = wl.small(name, seed=61)
    gw = wl.gqa(w, seed=61)
    cache, step = run(gw)
    ocache, ref = oracle_run(gw)
    # the append: values bit-exact, keys within one rounding, nothing else touched
    assert np.array_equal(bits(cache.c_kv.cpu()), ocache.c_kv)
    got_k = bits(cache.k_rope.cpu()).astype(np.int32)
    d = np.abs(got_k - ocache.k_rope.astype(np.int32))
    assert d.max() <= 1 and (d > 0).mean() < 0.01
    assert_close(step.o.cpu().numpy(), ref["o"], "o")
    assert_close(step.lse.cpu().numpy(), ref["lse"], "lse")


@pytest.mark.parametrize("splits", [1, 3, 7])
def test_gqa_split_counts_and_paged(splits):
    """Several units per CTA and ragged tails in both layouts; the paged and
    contiguous runs of the same logical cache agree bit for bit."""
    shape = wl.SHAPES["llama1b_paged_b128_h32_r512_t128_8192"]
    wp = wl.make(shape, seed=62, batch=4, kv_range=(70, 650))
    gp = wl.gqa(wp, seed=62)
    cache_p, step_p = run(gp, splits)
    ocache, ref = oracle_run(gp)
    G = gp.num_kv_groups
    assert_close(step_p.o.cpu().numpy(), ref["o"], "o")
    # the same logical cache laid out contiguously
    cap = int(gp.kv_len.max())
    B, d = 4, gp.d
    kc = torch.zeros(B * G, cap, d, dtype=torch.bfloat16)
    vc = torch.zeros(B * G, cap, d, dtype=torch.bfloat16)
    for u in range(B * G):
        for t in range(int(gp.kv_len[u // G]) - shape.q_len):     # the rows before this step's append
            pg = int(gp.block_table[u, t // 64])
            kc[u, t], vc[u, t] = gp.k_cache[pg, t % 64], gp.v_cache[pg, t % 64]
    gc = dataclasses.replace(gp, shape=dataclasses.replace(shape, paged=False), k_cache=kc, v_cache=vc,
                             block_table=None, num_pages=0, capacity=cap)
    _, step_c = run(gc, splits)
    assert torch.equal(step_p.o.cpu(), step_c.o.cpu())
