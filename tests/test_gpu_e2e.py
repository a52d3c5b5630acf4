"""GPU parity of the E2E functional-reconstruction loss forward (Sec. 4.1):
the loss kernel alone, and the whole forward (the converted MLA layer and the
original GQA layer on the same hidden states, sharing W_O) against the fp64
oracle doing the same, its stored intermediates (queries, new keys and
values) rounded to bf16 as the GPU path stores them.

Bars: the loss kernel alone within 1e-5 relative (fp32 products of bf16
inputs, fp64 sums); the whole forward within 2e-2 relative (the blocks'
outputs are bf16 and their intermediates carry the step's own roundings).
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, dims_of, oracle_cache

pytestmark = pytest.mark.gpu


def test_e2e_loss_kernel_matches_oracle():
    g = torch.Generator().manual_seed(71)
    for rows, hidden in ((1, 8), (37, 896), (640, 2048)):
        a = torch.randn(rows, hidden, generator=g).to(torch.bfloat16)
        b = (a.float() + 0.3 * torch.randn(rows, hidden, generator=g)).to(torch.bfloat16)
        mask = (torch.rand(rows, generator=g) < 0.7).to(torch.uint8)
        mask[0] = 1
        for m in (mask, None):
            got = abi.e2e_loss(a.cuda(), b.cuda(), None if m is None else m.cuda()).item()
            ref = orc.e2e_loss(bf16_to_f64(bits(a)), bf16_to_f64(bits(b)), None if m is None else m.numpy())
            assert abs(got - ref) <= 1e-5 * ref, (rows, hidden, got, ref)
    z = torch.zeros(4, 16, dtype=torch.bfloat16, device="cuda")
    assert abi.e2e_loss(z, z, torch.zeros(4, dtype=torch.uint8, device="cuda")).item() == 0.0


def _round(x: np.ndarray) -> np.ndarray:
    return np.vectorize(orc.bf16_round, otypes=[np.uint16])(x)


@pytest.mark.parametrize("name", ["qwen05b_b16_h14_r256_t2048", "llama1b_chunk5_b32_h32_r512_t4096"])
def test_e2e_forward_matches_oracle(name):
    w = wl.small(name, seed=72)
    p = wl.projection(w, seed=72)
    gw = wl.gqa(w, seed=72)
    gp = wl.gqa_projection(w, seed=72)
    s = w.shape
    B, q, D = w.kv_len.numel(), s.q_len, p.hidden
    mask = (torch.arange(B * q) % 3 != 1).to(torch.uint8).reshape(B, q)
    # ---- GPU
    dw = abi.to_device(w)
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    gdims = abi.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
    gcache = abi.Cache(gw.v_cache.cuda(), gw.k_cache.cuda(), gw.capacity, None, 0, 0)
    fwd = abi.E2EForward(step, gdims, gcache, D)
    cu = lambda t: t.cuda()
    loss = fwd(cu(p.h), tuple(map(cu, (p.w_dkv, p.w_kr, p.w_q, w.w_uk, w.w_uv))), tuple(map(cu, (gp.w_q, gp.w_k, gp.w_v))),
               cu(w.w_o), dw.start_pos, dw.kv_len, mask.cuda()).item()
    assert abi.check_status() == abi.MLA_OK
    # ---- oracle: the converted layer ...
    mdims = dataclasses.replace(dims_of(w), hidden=D)
    mcache = oracle_cache(w)
    qn, qp = orc.project_append(mdims, mcache, bits(p.h), bits(p.w_dkv), bits(p.w_kr), bits(p.w_q),
                                w.start_pos.numpy())
    a_mla = orc.mla_decode(mdims, mcache, _round(qn), _round(qp), w.kv_len.numpy(), bits(w.w_uk), bits(w.w_uv),
                           bits(w.w_o))["out"]
    # ... and the original one, on the same hidden states, with the same W_O
    h = bf16_to_f64(bits(p.h)).reshape(B * q, D)
    qg = _round(h @ bf16_to_f64(bits(gp.w_q)).T).reshape(B, q, gw.num_heads, gw.d)
    kg = _round(h @ bf16_to_f64(bits(gp.w_k)).T).reshape(B, q, gw.num_kv_groups, gw.d)
    vg = _round(h @ bf16_to_f64(bits(gp.w_v)).T).reshape(B, q, gw.num_kv_groups, gw.d)
    odims = orc.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
    ocache = orc.Cache(c_kv=bits(gw.v_cache), k_rope=bits(gw.k_cache), c_tok_stride=gw.d, r_tok_stride=gw.d,
                       c_blk_stride=gw.k_cache.shape[1] * gw.d, r_blk_stride=gw.k_cache.shape[1] * gw.d,
                       capacity=gw.capacity)
    orc.gqa_append(odims, ocache, kg, vg, w.start_pos.numpy())
    og = orc.gqa_decode(odims, ocache, qg, w.kv_len.numpy())["o"]
    a_orig = og.reshape(B, q, -1) @ bf16_to_f64(bits(w.w_o)).T
    ref = orc.e2e_loss(a_mla.reshape(B * q, D), a_orig.reshape(B * q, D), mask.numpy().reshape(-1))
    assert abs(loss - ref) <= 2e-2 * ref, (loss, ref)
