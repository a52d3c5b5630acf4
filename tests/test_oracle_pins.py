"""Pins of the fp64 oracle against the paper and against mathematics.

None of these compares the oracle with itself: each checks it against a
library routine (torch SDPA, numpy matmul, scipy logsumexp), a closed form, an
exact identity stated by the paper, an invariant, or brute force on tiny
inputs.  Together they are chosen so that a dropped term, a wrong sign or
index, a wrong group map or a transposed operand in the oracle fails one.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

from oracle import oracle as orc
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, dims_of, oracle_cache, rope_complex

RNG = np.random.default_rng(1234)


def rand_bf16(shape, std=1.0) -> np.ndarray:
    return bits((torch.from_numpy(RNG.standard_normal(shape) * std)).to(torch.bfloat16))


# ---------------------------------------------------------------- bf16 helpers

def test_bf16_value_exact_patterns():
    assert orc.bf16_value(0x3F80) == 1.0
    assert orc.bf16_value(0xC000) == -2.0
    assert orc.bf16_value(0x7F7F) == (2 - 2 ** -7) * 2.0 ** 127  # largest finite bf16
    assert orc.bf16_value(0x0001) == 2.0 ** -133                  # smallest subnormal
    assert math.isinf(orc.bf16_value(0x7F80))


def test_bf16_round_ties_to_even_and_single_rounding():
    assert orc.bf16_round(1.0 + 2 ** -8) == 0x3F80          # tie -> even mantissa 0
    assert orc.bf16_round(1.0 + 3 * 2 ** -8) == 0x3F82      # tie -> even mantissa 2
    assert orc.bf16_round(1.0 + 2 ** -8 + 2 ** -40) == 0x3F81  # above the tie: one rounding, up
    assert orc.bf16_round(-(1.0 + 2 ** -8 + 2 ** -40)) == 0xBF81
    assert orc.bf16_round(3.0e38 * 10) == 0x7F80            # overflow -> inf
    assert orc.bf16_round(2.0 ** -134) == 0x0000            # tie below the smallest subnormal -> 0
    assert orc.bf16_round(1.5 * 2.0 ** -133) == 0x0002      # tie -> even


def test_bf16_round_within_half_ulp_and_matches_fp32_rounding():
    x = RNG.standard_normal(2000) * np.exp(RNG.uniform(-20, 20, 2000))
    got = np.array([orc.bf16_round(v) for v in x], dtype=np.uint16)
    val = bf16_to_f64(got)
    # nearest: error at most half a unit in the last place (8 significant bits)
    ulp = 2.0 ** (np.floor(np.log2(np.abs(x))) - 7)
    assert np.all(np.abs(val - x) <= ulp / 2)
    # on fp32-representable inputs it agrees with torch's fp32 -> bf16 rounding
    x32 = x.astype(np.float32)
    got32 = np.array([orc.bf16_round(float(v)) for v in x32], dtype=np.uint16)
    ref32 = bits(torch.from_numpy(x32).to(torch.bfloat16))
    assert np.array_equal(got32, ref32)


# ---------------------------------------------------------------- RoPE (Sec. 3.1)

@pytest.mark.parametrize("style", [0, 1])
def test_rope_matches_complex_form(style):
    for d in (8, 32, 64):
        x = RNG.standard_normal(d)
        for pos in (0, 1, 7, 4099, 32767):
            # a 1-ulp difference in theta_k moves the angle pos * theta_k by ~pos * 2^-52
            tol = 1e-14 + 4 * max(pos, 1) * 2.0 ** -52 * np.abs(x).max()
            assert np.allclose(orc.rope(x, pos, 10000.0, style), rope_complex(x, pos, 10000.0, style),
                               rtol=0, atol=tol)


def test_rope_closed_form_unit_vectors():
    # d=8 rotate-half: pair k=(k, k+4), theta = 10000^(-k/4) = 1, 0.1, 0.01, 0.001
    x = np.zeros(8)
    x[0], x[5] = 1.0, 2.0
    y = orc.rope(x, 3, 10000.0, 0)
    ref = [math.cos(3), -2 * math.sin(0.3), 0, 0, math.sin(3), 2 * math.cos(0.3), 0, 0]
    assert np.allclose(y, ref, atol=1e-15)
    # interleaved: pair k=(2k, 2k+1)
    x = np.zeros(8)
    x[2] = 1.0
    y = orc.rope(x, 5, 10000.0, 1)
    ref = [0, 0, math.cos(0.5), math.sin(0.5), 0, 0, 0, 0]
    assert np.allclose(y, ref, atol=1e-15)


def test_rope_group_properties():
    d = 64
    q, k = RNG.standard_normal(d), RNG.standard_normal(d)
    assert np.array_equal(orc.rope(q, 0), q)                                    # R_0 = I
    assert abs(np.linalg.norm(orc.rope(q, 12345)) - np.linalg.norm(q)) < 1e-12  # orthogonal
    assert np.allclose(orc.rope(orc.rope(q, 100), 23), orc.rope(q, 123), atol=1e-12)  # R_a R_b = R_{a+b}
    # R_tj = R_t^T R_j: the score depends on positions only through t - j
    base = np.dot(orc.rope(q, 40), orc.rope(k, 17))
    for shift in (1, 1000, 20000):
        assert abs(np.dot(orc.rope(q, 40 + shift), orc.rope(k, 17 + shift)) - base) < 1e-10


def test_logit_error_identity():
    """Eq. (logit-error), Sec. 3.3, holds exactly with R_tj realised as
    q^T R_tj k = (R_t q) . (R_j k)."""
    d = 64
    t, j = 300, 120
    q, dq = RNG.standard_normal(d), RNG.standard_normal(d) * 0.1
    k_keep, k_drop, dk = RNG.standard_normal(d), RNG.standard_normal(d), RNG.standard_normal(d) * 0.1

    def bil(a, b):  # a^T R_tj b
        return float(np.dot(orc.rope(a, t), orc.rope(b, j)))

    s = (bil(q, k_keep) + bil(q, k_drop)) / math.sqrt(d)
    s_hat = (bil(q + dq, k_keep + dk) + np.dot(q + dq, k_drop)) / math.sqrt(d)
    rhs = (bil(q, dk) + (np.dot(q, k_drop) - bil(q, k_drop)) + bil(dq, k_keep + dk)
           + np.dot(dq, k_drop)) / math.sqrt(d)
    assert abs((s_hat - s) - rhs) < 1e-12


# ---------------------------------------------------------------- attention (Eqs. 2-5)

def _tiny(batch=2, H=4, G=2, dn=8, dr=8, dv=6, r=12, q_len=3, kv=(5, 9), D=0, paged=False, seed=3):
    s = wl.Shape("tiny_test", batch, H, G, dn, dr, dv, r, D, q_len, kv[0], kv[1], paged=paged, page_size=4)
    return wl.make(s, seed)


def _explicit_reference(w, cache):
    """Brute-force attention with explicit keys/values through torch SDPA (fp64)."""
    s = w.shape
    H, G = s.num_heads, s.num_kv_groups
    hpg = H // G
    outs, lses = {}, {}
    for b in range(s.batch):
        kv = int(w.kv_len[b])
        C = np.stack([_read_row(cache, b, j, "c") for j in range(kv)])
        KR = np.stack([_read_row(cache, b, j, "r") for j in range(kv)])
        wuk, wuv = bf16_to_f64(bits(w.w_uk)), bf16_to_f64(bits(w.w_uv))
        qn, qp = bf16_to_f64(bits(w.q_nope))[b], bf16_to_f64(bits(w.q_pe))[b]
        for h in range(H):
            g = h // hpg
            K = np.concatenate([C @ wuk[g].T, KR], axis=1)     # [kv, dn+dr]
            V = C @ wuv[g].T                                   # [kv, dv]
            pos = np.arange(kv - s.q_len, kv)
            Q = np.concatenate([qn[:, h], rope_complex(qp[:, h], pos, s.rope_base, s.rope_style)], axis=1)
            mask = np.arange(kv)[None, :] <= pos[:, None]
            o = F.scaled_dot_product_attention(torch.from_numpy(Q)[None], torch.from_numpy(K)[None],
                                               torch.from_numpy(V)[None], attn_mask=torch.from_numpy(mask)[None],
                                               scale=s.sm_scale)[0].numpy()
            scores = s.sm_scale * (Q @ K.T)
            scores[~mask] = -np.inf
            outs[(b, h)] = o
            lses[(b, h)] = scipy.special.logsumexp(scores, axis=1)
    return outs, lses


def _read_row(cache, b, j, which):
    if cache.block_table is not None:
        blk, slot = cache.block_table[b, j // cache.page_size], j % cache.page_size
    else:
        blk, slot = b, j
    if which == "c":
        off = blk * cache.c_blk_stride + slot * cache.c_tok_stride
        return bf16_to_f64(cache.c_kv.reshape(-1)[off:off + cache.c_tok_stride])
    off = blk * cache.r_blk_stride + slot * cache.r_tok_stride
    return bf16_to_f64(cache.k_rope.reshape(-1)[off:off + cache.r_tok_stride])


@pytest.mark.parametrize("G", [1, 2, 4])   # MQA, GQA and MHA (G = H, Sec. 3.1)
@pytest.mark.parametrize("paged", [False, True])
def test_attention_matches_sdpa_bruteforce(G, paged):
    w = _tiny(G=G, paged=paged)
    cache = oracle_cache(w)
    res = orc.mla_decode(dims_of(w), cache, bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk),
                         bits(w.w_uv))
    outs, lses = _explicit_reference(w, cache)
    for (b, h), o in outs.items():
        assert np.allclose(res["o"][b, :, h], o, rtol=1e-12, atol=1e-13)
        assert np.allclose(res["lse"][b, :, h], lses[(b, h)], rtol=1e-12, atol=1e-12)


def test_absorbed_form_equals_non_absorbed():
    """Associativity behind absorption (Sec. 1, Eq. 5): q_nope.(W_UK c) =
    (W_UK^T q_nope).c and W_UV sum a c = sum a W_UV c."""
    w = _tiny(batch=3, H=6, G=3, dn=16, dr=8, dv=8, r=40, q_len=2, kv=(7, 19))
    s = w.shape
    cache = oracle_cache(w)
    dims = dims_of(w)
    res = orc.mla_decode(dims, cache, bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk), bits(w.w_uv))
    q_lat, q_rot = orc.absorb_q(dims, bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk))
    wuk, wuv = bf16_to_f64(bits(w.w_uk)), bf16_to_f64(bits(w.w_uv))
    qn, qp = bf16_to_f64(bits(w.q_nope)), bf16_to_f64(bits(w.q_pe))
    hpg = s.num_heads // s.num_kv_groups
    for b in range(s.batch):
        kv = int(w.kv_len[b])
        C = np.stack([_read_row(cache, b, j, "c") for j in range(kv)])
        KR = np.stack([_read_row(cache, b, j, "r") for j in range(kv)])
        for i in range(s.q_len):
            p = kv - s.q_len + i
            for h in range(s.num_heads):
                g = h // hpg
                ql = wuk[g].T @ qn[b, i, h]                     # absorbed latent query
                assert np.allclose(q_lat[b, i, h], ql, rtol=1e-13, atol=1e-13)
                qr = rope_complex(qp[b, i, h], p)
                assert np.allclose(q_rot[b, i, h], qr, atol=1e-13)
                sc = s.sm_scale * (C[:p + 1] @ ql + KR[:p + 1] @ qr)
                a = np.exp(sc - sc.max())
                a /= a.sum()
                assert np.allclose(res["o_lat"][b, i, h], a @ C[:p + 1], rtol=1e-11, atol=1e-12)
                assert np.allclose(res["o"][b, i, h], wuv[g] @ (a @ C[:p + 1]), rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("G,dr", [(2, 8), (4, 8), (2, 0)])
def test_full_rank_identity_mla_equals_gqa(G, dr):
    """Rank condition (Sec. 3.2, Eq. rank-condition / rank-bound): with
    r = G (d_nope + d_v) the stacked K/V map factorises exactly
    (W^DKV = the stacked original projections, W^UKV = I), so MLA must
    reproduce GQA attention with a shared decoupled RoPE key exactly."""
    H, dn, dv, q_len, B = 4, 8, 6, 2, 2
    r = G * (dn + dv)
    kv = np.array([6, 11], dtype=np.int32)
    cap = int(kv.max())
    # original GQA keys/values per group and a shared positional key
    k_nope = rand_bf16((B, cap, G, dn))
    v = rand_bf16((B, cap, G, dv))
    k_pe_rot = rand_bf16((B, cap, dr))                  # stored already rotated
    qn, qp = rand_bf16((B, q_len, H, dn)), rand_bf16((B, q_len, H, dr))
    # MLA factorisation: c_j = concat_g [k_nope_g ; v_g], W_UK / W_UV select blocks
    c = np.concatenate([k_nope, v], axis=3).reshape(B, cap, r)
    one, zero = 0x3F80, 0
    w_uk = np.full((G, dn, r), zero, dtype=np.uint16)
    w_uv = np.full((G, dv, r), zero, dtype=np.uint16)
    for g in range(G):
        for d in range(dn):
            w_uk[g, d, g * (dn + dv) + d] = one
        for e in range(dv):
            w_uv[g, e, g * (dn + dv) + dn + e] = one
    scale = 1 / math.sqrt(dn + dr)
    dims = orc.Dims(H, G, dn, dr, dv, r, 0, scale)
    cache = orc.Cache(c_kv=np.ascontiguousarray(c), k_rope=np.ascontiguousarray(k_pe_rot), c_tok_stride=r,
                      r_tok_stride=dr, c_blk_stride=cap * r, r_blk_stride=cap * dr, capacity=cap)
    res = orc.mla_decode(dims, cache, qn, qp, kv, w_uk, w_uv)
    # GQA through torch SDPA with enable_gqa: head h reads group h // (H/G)
    for b in range(B):
        n = int(kv[b])
        pos = np.arange(n - q_len, n)
        Qh = np.concatenate([bf16_to_f64(qn[b]), rope_complex(bf16_to_f64(qp[b]), pos[:, None])], axis=2)
        Kg = np.concatenate([bf16_to_f64(k_nope[b, :n]),
                             np.broadcast_to(bf16_to_f64(k_pe_rot[b, :n])[:, None, :], (n, G, dr))], axis=2)
        Vg = bf16_to_f64(v[b, :n])
        mask = np.arange(n)[None, :] <= pos[:, None]
        o = F.scaled_dot_product_attention(torch.from_numpy(Qh.transpose(1, 0, 2)),
                                           torch.from_numpy(np.ascontiguousarray(Kg.transpose(1, 0, 2))),
                                           torch.from_numpy(np.ascontiguousarray(Vg.transpose(1, 0, 2))),
                                           attn_mask=torch.from_numpy(mask), scale=scale,
                                           enable_gqa=True).numpy().transpose(1, 0, 2)
        assert np.allclose(res["o"][b], o, rtol=1e-12, atol=1e-13)


def test_single_key_closed_form():
    """kv = 1: the softmax has one term, so a = 1, o_lat = c_0, o = W_UV c_0
    and lse = s_0."""
    w = _tiny(batch=2, q_len=1, kv=(1, 1))
    s = w.shape
    cache = oracle_cache(w)
    res = orc.mla_decode(dims_of(w), cache, bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk),
                         bits(w.w_uv))
    wuk, wuv = bf16_to_f64(bits(w.w_uk)), bf16_to_f64(bits(w.w_uv))
    hpg = s.num_heads // s.num_kv_groups
    for b in range(2):
        c0, kr0 = _read_row(cache, b, 0, "c"), _read_row(cache, b, 0, "r")
        for h in range(s.num_heads):
            assert np.array_equal(res["o_lat"][b, 0, h], c0)
            assert np.allclose(res["o"][b, 0, h], wuv[h // hpg] @ c0, rtol=1e-14, atol=1e-14)
            qn = bf16_to_f64(bits(w.q_nope))[b, 0, h]
            qp = bf16_to_f64(bits(w.q_pe))[b, 0, h]        # position 0: no rotation
            s0 = s.sm_scale * (qn @ (wuk[h // hpg] @ c0) + qp @ kr0)
            assert abs(res["lse"][b, 0, h] - s0) < 1e-12


def test_zero_query_gives_uniform_average():
    """All scores equal: a_j = 1/(p+1), o_lat = mean of c_0..c_p, lse = ln(p+1)."""
    w = _tiny(batch=2, q_len=3, kv=(9, 14))
    w.q_nope.zero_()
    w.q_pe.zero_()
    cache = oracle_cache(w)
    res = orc.mla_decode(dims_of(w), cache, bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk),
                         bits(w.w_uv))
    for b in range(2):
        kv = int(w.kv_len[b])
        C = np.stack([_read_row(cache, b, j, "c") for j in range(kv)])
        for i in range(3):
            p = kv - 3 + i
            for h in range(w.shape.num_heads):
                assert np.allclose(res["o_lat"][b, i, h], C[:p + 1].mean(axis=0), rtol=1e-13, atol=1e-14)
                assert abs(res["lse"][b, i, h] - math.log(p + 1)) < 1e-13


def test_causal_mask_and_rows_past_kv_len_are_not_read():
    """A query at position p sees keys 0..p only (Eq. 3): a huge planted key
    at position kv-1 changes only the last query of the chunk; NaN rows past
    kv_len change nothing."""
    w = _tiny(batch=2, q_len=3, kv=(8, 8), seed=5)
    w2 = _tiny(batch=2, q_len=3, kv=(8, 8), seed=5)
    w.c_kv[:, 7, :] = 1.0e4
    w.k_rope[:, 7, :] = 1.0e4
    nan_c = torch.full((2, 12, 12), float("nan"), dtype=torch.bfloat16)
    nan_r = torch.full((2, 12, 8), float("nan"), dtype=torch.bfloat16)
    nan_c[:, :8], nan_r[:, :8] = w2.c_kv, w2.k_rope
    cap_w = dataclasses.replace(w2, c_kv=nan_c, k_rope=nan_r, capacity=12)
    run = lambda x: orc.mla_decode(dims_of(x), oracle_cache(x), bits(x.q_nope), bits(x.q_pe), x.kv_len.numpy(),
                                   bits(x.w_uk), bits(x.w_uv))
    a, b2, c = run(w), run(w2), run(cap_w)
    assert np.array_equal(a["o"][:, :2], b2["o"][:, :2])
    assert not np.allclose(a["o"][:, 2], b2["o"][:, 2])
    assert np.array_equal(c["o"], b2["o"]) and np.array_equal(c["lse"], b2["lse"])


def test_output_projection_identity_and_matmul():
    """out = W_O concat_h o_h (Sec. 4.1): with W_O = I (D = H d_v) out is the
    concatenation itself; a random W_O matches a numpy matmul."""
    w = _tiny(batch=2, H=4, G=2, dv=6, D=24, q_len=2, kv=(5, 9))
    eye = np.zeros((24, 24), dtype=np.uint16)
    eye[np.arange(24), np.arange(24)] = 0x3F80
    res = orc.mla_decode(dims_of(w), oracle_cache(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(),
                         bits(w.w_uk), bits(w.w_uv), eye)
    assert np.array_equal(res["out"], res["o"].reshape(2, 2, 24))
    res = orc.mla_decode(dims_of(w), oracle_cache(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(),
                         bits(w.w_uk), bits(w.w_uv), bits(w.w_o))
    ref = res["o"].reshape(2, 2, 24) @ bf16_to_f64(bits(w.w_o)).T
    assert np.allclose(res["out"], ref, rtol=1e-13, atol=1e-14)


def test_subset_of_sequences():
    w = _tiny(batch=4, kv=(5, 13))
    full = orc.mla_decode(dims_of(w), oracle_cache(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(),
                          bits(w.w_uk), bits(w.w_uv))
    part = orc.mla_decode(dims_of(w), oracle_cache(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(),
                          bits(w.w_uk), bits(w.w_uv), seqs=[2, 0])
    for b in (0, 2):
        assert np.array_equal(part["o"][b], full["o"][b])
    assert np.isnan(part["o"][1]).all() and np.isnan(part["o"][3]).all()


# ---------------------------------------------------------------- cache append (Sec. 3.2)

def test_append_contiguous_positions_and_rounding():
    w = _tiny(batch=3, q_len=3, kv=(4, 9), D=0)
    s = w.shape
    before_c, before_r = bits(w.c_kv), bits(w.k_rope)
    cache = oracle_cache(w)
    orc.cache_append(dims_of(w), cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    krn = bf16_to_f64(bits(w.kr_new))
    for b in range(3):
        sp = int(w.start_pos[b])
        for t in range(w.capacity):
            if sp <= t < sp + 3:
                assert np.array_equal(cache.c_kv[b, t], bits(w.c_new)[b, t - sp])      # bit copy
                exact = rope_complex(krn[b, t - sp], t, s.rope_base, s.rope_style)
                got = bf16_to_f64(cache.k_rope[b, t])
                ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(exact), 1e-30))) - 7)
                assert np.all(np.abs(got - exact) <= ulp / 2 + 1e-15)                  # one RNE rounding
            else:
                assert np.array_equal(cache.c_kv[b, t], before_c[b, t])
                assert np.array_equal(cache.k_rope[b, t], before_r[b, t])


def test_append_paged_equals_contiguous_logically():
    """Paged addressing (page block_table[b][t // P], slot t % P) stores the
    same logical sequence as the contiguous layout."""
    shape_p = wl.Shape("p", 3, 4, 2, 8, 8, 6, 12, 0, 3, 5, 14, paged=True, page_size=4)
    wp = wl.make(shape_p, seed=9)
    cp = oracle_cache(wp)
    orc.cache_append(dims_of(wp), cp, bits(wp.c_new), bits(wp.kr_new), wp.start_pos.numpy())
    # rebuild a contiguous cache holding the same pre-append logical content
    cap = int(wp.kv_len.max())
    cc = np.zeros((3, cap, 12), dtype=np.uint16)
    rc = np.zeros((3, cap, 8), dtype=np.uint16)
    pre = oracle_cache(wp)
    for b in range(3):
        for t in range(int(wp.kv_len[b])):
            blk, slot = pre.block_table[b, t // 4], t % 4
            cc[b, t], rc[b, t] = pre.c_kv[blk, slot], pre.k_rope[blk, slot]
    ccache = orc.Cache(c_kv=cc, k_rope=rc, c_tok_stride=12, r_tok_stride=8, c_blk_stride=cap * 12,
                       r_blk_stride=cap * 8, capacity=cap)
    orc.cache_append(dims_of(wp), ccache, bits(wp.c_new), bits(wp.kr_new), wp.start_pos.numpy())
    for b in range(3):
        for t in range(int(wp.kv_len[b])):
            blk, slot = cp.block_table[b, t // 4], t % 4
            assert np.array_equal(cp.c_kv[blk, slot], cc[b, t])
            assert np.array_equal(cp.k_rope[blk, slot], rc[b, t])
    dims = dims_of(wp)
    a = orc.mla_decode(dims, cp, bits(wp.q_nope), bits(wp.q_pe), wp.kv_len.numpy(), bits(wp.w_uk), bits(wp.w_uv))
    c = orc.mla_decode(dims, ccache, bits(wp.q_nope), bits(wp.q_pe), wp.kv_len.numpy(), bits(wp.w_uk),
                       bits(wp.w_uv))
    assert np.array_equal(a["o"], c["o"]) and np.array_equal(a["o_lat"], c["o_lat"])


def test_append_position_zero_is_a_copy_and_errors():
    w = _tiny(batch=1, q_len=1, kv=(1, 1))
    cache = oracle_cache(w)
    orc.cache_append(dims_of(w), cache, bits(w.c_new), bits(w.kr_new), [0])
    assert np.array_equal(cache.k_rope[0, 0], bits(w.kr_new)[0, 0])   # R_0 = I, exact
    with pytest.raises(orc.OracleError, match="bad position"):
        orc.cache_append(dims_of(w), oracle_cache(w), bits(w.c_new), bits(w.kr_new), [1])
    shape_p = wl.Shape("p", 1, 4, 2, 8, 8, 6, 12, 0, 1, 6, 6, paged=True, page_size=4)
    wp = wl.make(shape_p, seed=1)
    cp = oracle_cache(wp)
    cp.block_table[0, 1] = -1
    with pytest.raises(orc.OracleError, match="bad page"):
        orc.cache_append(dims_of(wp), cp, bits(wp.c_new), bits(wp.kr_new), wp.start_pos.numpy())


# ---------------------------------------------------------------- projection + append (Sec. 3.2, Eq. 1)

def _proj_case(paged=False, batch=3, q_len=2, kv=(3, 9), D=24, seed=5):
    w = _tiny(batch=batch, q_len=q_len, kv=kv, paged=paged, seed=seed)
    p = wl.projection(w, seed=seed, hidden=D)
    dims = dataclasses.replace(dims_of(w), hidden=D)
    return w, p, dims


def _within_half_ulp(got_bits, exact):
    got = bf16_to_f64(got_bits)
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(exact), 1e-30))) - 7)
    return np.all(np.abs(got - exact) <= ulp / 2 + 1e-15)


def test_projection_of_unit_vectors_selects_weight_columns():
    """h = e_k gives column k of every weight: the latent and the queries
    exactly, the positional key exactly at position 0 and rotated elsewhere."""
    w, p, dims = _proj_case(batch=2, q_len=3, kv=(3, 6))
    s = w.shape
    D = p.hidden
    ks = [[0, 5, D - 1], [7, 11, 2]]
    h = np.zeros((2, 3, D), dtype=np.uint16)
    for b in range(2):
        for i in range(3):
            h[b, i, ks[b][i]] = 0x3F80                                   # bf16 1.0
    start = np.array([0, int(w.start_pos[1])], dtype=np.int32)
    cache = oracle_cache(w)
    q_nope, q_pe = orc.project_append(dims, cache, h, bits(p.w_dkv), bits(p.w_kr), bits(p.w_q), start)
    wd, wk, wq = bits(p.w_dkv), bits(p.w_kr), bf16_to_f64(bits(p.w_q))
    dq = s.d_nope + s.d_rope
    for b in range(2):
        for i in range(3):
            k, pos = ks[b][i], int(start[b]) + i
            assert np.array_equal(cache.c_kv[b, pos], wd[:, k])
            if pos == 0:
                assert np.array_equal(cache.k_rope[b, pos], wk[:, k])   # R_0 = I
            exact = rope_complex(bf16_to_f64(wk[:, k]), pos, s.rope_base, s.rope_style)
            assert _within_half_ulp(cache.k_rope[b, pos], exact)
            col = wq[:, k].reshape(s.num_heads, dq)
            assert np.array_equal(q_nope[b, i], col[:, :s.d_nope])
            assert np.array_equal(q_pe[b, i], col[:, s.d_nope:])


@pytest.mark.parametrize("style", [0, 1])
def test_projection_matches_matmul_and_rounds_once(style):
    """Random inputs: the cache rows are the numpy fp64 products rounded once
    (the positional key rotated first, by the complex form), the queries are
    the products themselves."""
    w, p, dims = _proj_case(seed=6)
    w = dataclasses.replace(w, shape=dataclasses.replace(w.shape, rope_style=style))
    dims = dataclasses.replace(dims, rope_style=style)
    s = w.shape
    before_c, before_r = bits(w.c_kv), bits(w.k_rope)
    cache = oracle_cache(w)
    q_nope, q_pe = orc.project_append(dims, cache, bits(p.h), bits(p.w_dkv), bits(p.w_kr), bits(p.w_q),
                                      w.start_pos.numpy())
    h = bf16_to_f64(bits(p.h))
    c = h @ bf16_to_f64(bits(p.w_dkv)).T
    kr = h @ bf16_to_f64(bits(p.w_kr)).T
    q = (h @ bf16_to_f64(bits(p.w_q)).T).reshape(*h.shape[:2], s.num_heads, s.d_nope + s.d_rope)
    np.testing.assert_allclose(q_nope, q[..., :s.d_nope], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(q_pe, q[..., s.d_nope:], rtol=1e-12, atol=1e-12)
    for b in range(s.batch):
        sp = int(w.start_pos[b])
        for t in range(w.capacity):
            if sp <= t < sp + s.q_len:
                assert _within_half_ulp(cache.c_kv[b, t], c[b, t - sp])
                assert _within_half_ulp(cache.k_rope[b, t],
                                        rope_complex(kr[b, t - sp], t, s.rope_base, style))
            else:
                assert np.array_equal(cache.c_kv[b, t], before_c[b, t])
                assert np.array_equal(cache.k_rope[b, t], before_r[b, t])


def test_projection_paged_equals_contiguous_and_errors():
    """The paged cache receives the same rows at block_table[b][t // P],
    slot t % P; a position past the capacity or a bad page is an error that
    leaves the cache untouched."""
    wp, p, dims = _proj_case(paged=True, seed=8)
    cp = oracle_cache(wp)
    orc.project_append(dims, cp, bits(p.h), bits(p.w_dkv), bits(p.w_kr), None, wp.start_pos.numpy())
    s = wp.shape
    cap = int(wp.kv_len.max())
    cc = np.zeros((s.batch, cap, s.rank), dtype=np.uint16)
    rc = np.zeros((s.batch, cap, s.d_rope), dtype=np.uint16)
    ccache = orc.Cache(c_kv=cc, k_rope=rc, c_tok_stride=s.rank, r_tok_stride=s.d_rope,
                       c_blk_stride=cap * s.rank, r_blk_stride=cap * s.d_rope, capacity=cap)
    orc.project_append(dims, ccache, bits(p.h), bits(p.w_dkv), bits(p.w_kr), None, wp.start_pos.numpy())
    for b in range(s.batch):
        for t in range(int(wp.start_pos[b]), int(wp.kv_len[b])):
            blk, slot = cp.block_table[b, t // s.page_size], t % s.page_size
            assert np.array_equal(cp.c_kv[blk, slot], cc[b, t])
            assert np.array_equal(cp.k_rope[blk, slot], rc[b, t])
    bad = oracle_cache(wp)
    snapshot = bad.c_kv.copy()
    bad.block_table[s.batch - 1, (int(wp.kv_len[-1]) - 1) // s.page_size] = -1
    with pytest.raises(orc.OracleError, match="bad page"):
        orc.project_append(dims, bad, bits(p.h), bits(p.w_dkv), bits(p.w_kr), None, wp.start_pos.numpy())
    assert np.array_equal(bad.c_kv, snapshot)
    with pytest.raises(orc.OracleError, match="bad position"):
        orc.project_append(dims, oracle_cache(wp), bits(p.h), bits(p.w_dkv), bits(p.w_kr), None,
                           np.full(s.batch, wp.capacity, dtype=np.int32))


# ---------------------------------------------------------------- acceptance statistics (Sec. 3.3, Eqs. 9-10)

def _logits(rows, vocab, scale=3.0, seed=0):
    g = np.random.default_rng(seed)
    return g.standard_normal((rows, vocab)) * scale


def test_acceptance_identical_rows():
    d = _logits(4, 500)
    res = orc.acceptance(d, d)
    np.testing.assert_allclose(res["alpha_sample"], 1.0, rtol=0, atol=1e-12)
    assert np.array_equal(res["argmax_draft"], np.argmax(d, axis=1))
    assert np.all(res["greedy"] == 1)


def test_acceptance_is_one_minus_total_variation():
    """Eq. 9 states both forms: sum_y min(p_D, p_T) = 1 - TV(p_D, p_T)."""
    d = _logits(6, 3000, seed=1)
    t = d + 0.7 * _logits(6, 3000, scale=1.0, seed=2)
    res = orc.acceptance(d, t)
    pd, pt = scipy.special.softmax(d, axis=1), scipy.special.softmax(t, axis=1)
    tv = 0.5 * np.abs(pd - pt).sum(axis=1)
    np.testing.assert_allclose(res["alpha_sample"], 1.0 - tv, rtol=0, atol=1e-12)
    assert np.array_equal(res["argmax_draft"], np.argmax(d, axis=1))    # numpy: first maximum
    assert np.array_equal(res["argmax_target"], np.argmax(t, axis=1))
    assert np.array_equal(res["greedy"], (np.argmax(d, axis=1) == np.argmax(t, axis=1)).astype(np.int32))
    assert np.all((res["alpha_sample"] > 0) & (res["alpha_sample"] < 1))


def test_acceptance_two_token_closed_form():
    """Two tokens: alpha = 1 - |sigmoid(a - b) - sigmoid(c - e)|."""
    d = np.array([[0.3, -1.2], [2.0, 2.0], [5.0, -5.0]])
    t = np.array([[-0.4, 0.1], [2.0, 1.0], [-5.0, 5.0]])
    res = orc.acceptance(d, t)
    sig = lambda x: 1.0 / (1.0 + np.exp(-x))
    ref = 1.0 - np.abs(sig(d[:, 0] - d[:, 1]) - sig(t[:, 0] - t[:, 1]))
    np.testing.assert_allclose(res["alpha_sample"], ref, rtol=0, atol=1e-14)
    assert list(res["argmax_draft"]) == [0, 0, 0] and list(res["argmax_target"]) == [1, 0, 1]
    assert list(res["greedy"]) == [0, 1, 0]


def test_acceptance_invariances_and_ties():
    """Shifting a row's logits changes nothing; alpha is symmetric in the two
    distributions; equal maxima resolve to the lowest index."""
    d = _logits(5, 777, seed=3)
    t = d + _logits(5, 777, scale=0.5, seed=4)
    base = orc.acceptance(d, t)
    shifted = orc.acceptance(d + 11.0, t - 3.5)
    np.testing.assert_allclose(shifted["alpha_sample"], base["alpha_sample"], rtol=0, atol=1e-12)
    assert np.array_equal(shifted["argmax_draft"], base["argmax_draft"])
    swapped = orc.acceptance(t, d)
    np.testing.assert_allclose(swapped["alpha_sample"], base["alpha_sample"], rtol=0, atol=1e-12)
    tie = np.zeros((2, 10))
    tie[0, [3, 7]] = 4.0
    tie[1, [9, 2, 5]] = 1.0
    res = orc.acceptance(tie, tie[::-1])
    assert list(res["argmax_draft"]) == [3, 2] and list(res["argmax_target"]) == [2, 3]


# ---------------------------------------------------------------- original GQA (Sec. 3.1, Eqs. 1-4)

def _gqa_case(paged, q_len=3, seed=21):
    s = wl.Shape("gqa_test", 3, 6, 2, 8, 8, 8, 16, 0, q_len, 5, 14, paged=paged, page_size=4)
    w = wl.make(s, seed=seed)
    gw = wl.gqa(w, seed=seed)
    dims = orc.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.d, gw.sm_scale)
    bt = None if gw.block_table is None else gw.block_table.numpy().astype(np.int32).copy()
    cache = orc.Cache(c_kv=bits(gw.v_cache), k_rope=bits(gw.k_cache), c_tok_stride=gw.d, r_tok_stride=gw.d,
                      c_blk_stride=gw.k_cache.shape[1] * gw.d, r_blk_stride=gw.k_cache.shape[1] * gw.d,
                      capacity=gw.capacity, block_table=bt, page_size=s.page_size if paged else 0,
                      num_pages=gw.num_pages)
    return s, gw, dims, cache


def _gqa_logical(gw, cache, b, g, t):
    """(rotated key, value) of token t of sequence b, group g, read through the block table."""
    if cache.block_table is not None:
        blk, slot = cache.block_table[b * gw.num_kv_groups + g, t // 4], t % 4
    else:
        blk, slot = b * gw.num_kv_groups + g, t
    return bf16_to_f64(cache.k_rope[blk, slot]), bf16_to_f64(cache.c_kv[blk, slot])


@pytest.mark.parametrize("paged", [False, True])
def test_gqa_oracle_matches_sdpa(paged):
    """Append then decode, against torch SDPA over keys rotated by the complex
    form and a causal chunk mask."""
    s, gw, dims, cache = _gqa_case(paged)
    orc.gqa_append(dims, cache, bits(gw.k_new), bits(gw.v_new), gw.start_pos.numpy())
    res = orc.gqa_decode(dims, cache, bits(gw.q), gw.kv_len.numpy())
    H, G, d, q_len = gw.num_heads, gw.num_kv_groups, gw.d, s.q_len
    for b in range(s.batch):
        kv = int(gw.kv_len[b])
        for t in range(int(gw.start_pos[b]), kv):          # appended keys: one rounding of the exact rotation
            for g in range(G):
                k, _ = _gqa_logical(gw, cache, b, g, t)
                exact = rope_complex(bf16_to_f64(bits(gw.k_new))[b, t - int(gw.start_pos[b]), g], t)
                ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(exact), 1e-30))) - 7)
                assert np.all(np.abs(k - exact) <= ulp / 2 + 1e-15)
        K = np.stack([np.stack([_gqa_logical(gw, cache, b, g, t)[0] for t in range(kv)]) for g in range(G)])
        V = np.stack([np.stack([_gqa_logical(gw, cache, b, g, t)[1] for t in range(kv)]) for g in range(G)])
        pos = kv - q_len + np.arange(q_len)
        Q = np.stack([rope_complex(bf16_to_f64(bits(gw.q))[b, i], pos[i]) for i in range(q_len)])  # [q, H, d]
        mask = np.arange(kv)[None, :] <= pos[:, None]                                              # [q, kv]
        qt = torch.from_numpy(Q.transpose(1, 0, 2))[None]                                         # [1, H, q, d]
        kt = torch.from_numpy(K)[None].repeat_interleave(H // G, dim=1)
        vt = torch.from_numpy(V)[None].repeat_interleave(H // G, dim=1)
        ref = F.scaled_dot_product_attention(qt, kt, vt, attn_mask=torch.from_numpy(mask), scale=gw.sm_scale)
        np.testing.assert_allclose(res["o"][b].transpose(1, 0, 2), ref[0].numpy(), rtol=1e-12, atol=1e-12)
        logits = np.einsum("qhd,htd->hqt", Q, np.repeat(K, H // G, axis=0)) * gw.sm_scale
        logits = np.where(mask[None], logits, -np.inf)
        np.testing.assert_allclose(res["lse"][b].T, scipy.special.logsumexp(logits, axis=2), rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- E2E loss forward (Sec. 4.1)

def test_e2e_loss_closed_forms_and_invariances():
    g = np.random.default_rng(7)
    a = g.standard_normal((9, 40))
    b = g.standard_normal((9, 40))
    mask = (g.random(9) < 0.6).astype(np.uint8)
    mask[0] = 1
    assert orc.e2e_loss(a, a, mask) == 0.0                                     # identical blocks
    np.testing.assert_allclose(orc.e2e_loss(a + 0.3, a, mask), 0.09, rtol=1e-13)  # constant offset c: c^2
    base = orc.e2e_loss(a, b, mask)
    np.testing.assert_allclose(orc.e2e_loss(2.5 * a, 2.5 * b, mask), 6.25 * base, rtol=1e-13)  # scaling
    b2 = b.copy()
    b2[mask == 0] += 100.0                                                     # masked-out rows do not count
    assert orc.e2e_loss(a, b2, mask) == base
    one = np.zeros(9, dtype=np.uint8)
    one[3] = 1                                                                 # one row: its mean square
    np.testing.assert_allclose(orc.e2e_loss(a, b, one), np.mean((a[3] - b[3]) ** 2), rtol=1e-13)
    np.testing.assert_allclose(orc.e2e_loss(a, b), np.mean((a - b) ** 2), rtol=1e-13)  # no mask: every row
    assert orc.e2e_loss(a, b, np.zeros(9, dtype=np.uint8)) == 0.0             # no counted row
