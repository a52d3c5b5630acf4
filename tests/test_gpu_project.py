"""GPU parity of mla_project_append (Sec. 3.2 latent and positional key,
Eq. 1 queries) against the fp64 oracle on the same seeded inputs.

Bars: the cache rows and the queries are one bf16 rounding of an fp32 sum on
the GPU and of the exact fp64 value in the oracle, so every element agrees
within one bf16 unit in the last place plus the fp32 accumulation error (a
bound proportional to the sum of the products' magnitudes, which matters only
for values near zero), and almost all agree bit for bit; rows the call does
not own are untouched, bit for bit.  The whole step fed by
the projection meets the step's tolerance (max|d| <= 2e-2 max|ref|, mean
relative error <= 5e-3).
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, dims_of, oracle_cache, rel_errors

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 5e-3


def _ulp(x):
    return 2.0 ** (np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** -126))) - 7)


# fp32 accumulation of K products (tensor-core adds, any order) stays far
# inside 2^-18 of the sum of the products' magnitudes for these K (<= 3072)
ACC = 2.0 ** -18


def assert_one_rounding(got_bits, exact, mag, what, min_exact=0.98):
    """got (bf16 bits) is the rounding of an fp32 value within ACC * mag of
    exact (fp64): within half an ulp plus that, and identical to the
    nearest-even rounding of exact nearly everywhere."""
    got = bf16_to_f64(got_bits)
    err = np.abs(got - exact)
    bound = _ulp(np.maximum(np.abs(got), np.abs(exact))) / 2 + ACC * mag
    assert np.all(err <= bound), f"{what}: worst excess {np.max(err - bound):.3e}"
    near = err <= _ulp(exact) / 2 + 1e-30
    assert near.mean() >= min_exact, f"{what}: only {near.mean():.4f} rounded to nearest"


def assert_same_rounding(got_bits, ref_bits, mag, what, min_exact=0.98):
    """Two roundings to bf16 (fp32 sum on the GPU, exact in the oracle) of one
    value: within one ulp plus the accumulation bound, mostly bit-identical."""
    got, ref = bf16_to_f64(got_bits), bf16_to_f64(ref_bits)
    bound = _ulp(np.maximum(np.abs(got), np.abs(ref))) + ACC * mag
    assert np.all(np.abs(got - ref) <= bound), f"{what}: worst excess {np.max(np.abs(got - ref) - bound):.3e}"
    same = got_bits == ref_bits
    assert same.mean() >= min_exact, f"{what}: only {same.mean():.4f} identical"


def magnitudes(w, p):
    """Per output element, the sum over k of |W[e, k] h[k]| (fp64)."""
    h = np.abs(bf16_to_f64(bits(p.h)))
    B, n = h.shape[:2]
    s = w.shape
    c = h @ np.abs(bf16_to_f64(bits(p.w_dkv))).T
    kr = h @ np.abs(bf16_to_f64(bits(p.w_kr))).T
    if s.rope_style == 0:                                   # a rotated element mixes its pair
        half = s.d_rope // 2
        kr = np.concatenate([kr[..., :half] + kr[..., half:]] * 2, axis=-1)
    else:
        pair = kr[..., 0::2] + kr[..., 1::2]
        kr = np.repeat(pair, 2, axis=-1)
    q = (h @ np.abs(bf16_to_f64(bits(p.w_q))).T).reshape(B, n, s.num_heads, s.d_nope + s.d_rope)
    return c, kr, q[..., :s.d_nope], q[..., s.d_nope:]


def dims_with_hidden(w, D):
    return dataclasses.replace(dims_of(w), hidden=D)


def gpu_dims(w, D):
    s = w.shape
    return abi.Dims(s.num_heads, s.num_kv_groups, s.d_nope, s.d_rope, s.d_v, s.rank, D, s.sm_scale, s.rope_style,
                    s.rope_base)


def run_projection(w, p, with_q=True):
    dw = abi.to_device(w)
    s = w.shape
    d = gpu_dims(w, p.hidden)
    B, n = w.c_new.shape[0], w.c_new.shape[1]
    q_nope = torch.empty(B, n, s.num_heads, s.d_nope, dtype=torch.bfloat16, device="cuda") if with_q else None
    q_pe = torch.empty(B, n, s.num_heads, s.d_rope, dtype=torch.bfloat16, device="cuda") if with_q else None
    abi.project_append(d, dw.cache, p.h.cuda(), p.w_dkv.cuda(), p.w_kr.cuda(), p.w_q.cuda() if with_q else None,
                       dw.start_pos, q_nope, q_pe)
    return dw, q_nope, q_pe


def oracle_projection(w, p, with_q=True):
    cache = oracle_cache(w)
    qn, qp = orc.project_append(dims_with_hidden(w, p.hidden), cache, bits(p.h), bits(p.w_dkv), bits(p.w_kr),
                                bits(p.w_q) if with_q else None, w.start_pos.numpy())
    return cache, qn, qp


def check_projection(w, p, dw, q_nope, q_pe, with_q=True):
    code = abi.check_status()
    assert code == abi.MLA_OK, abi.status_name(code)
    cache, qn, qp = oracle_projection(w, p, with_q)
    got_c, got_r = bits(dw.cache.c_kv.cpu()), bits(dw.cache.k_rope.cpu())
    mc, mr, mqn, mqp = magnitudes(w, p)
    owned = np.zeros(got_c.shape[:2], bool)
    s = w.shape
    rows = []                                          # (block, slot, b, k) of every written row
    for b in range(w.kv_len.numel()):
        for t in range(int(w.start_pos[b]), int(w.kv_len[b])):
            blk, slot = (int(w.block_table[b, t // s.page_size]), t % s.page_size) if s.paged else (b, t)
            owned[blk, slot] = True
            rows.append((blk, slot, b, t - int(w.start_pos[b])))
    assert np.array_equal(got_c[~owned], cache.c_kv[~owned])
    assert np.array_equal(got_r[~owned], cache.k_rope[~owned])
    idx = tuple(np.array(x) for x in zip(*rows))
    assert_same_rounding(got_c[idx[0], idx[1]], cache.c_kv[idx[0], idx[1]], mc[idx[2], idx[3]], "latent rows")
    assert_same_rounding(got_r[idx[0], idx[1]], cache.k_rope[idx[0], idx[1]], mr[idx[2], idx[3]], "positional keys")
    if with_q:
        assert_one_rounding(bits(q_nope.cpu()), qn, mqn, "q_nope")
        assert_one_rounding(bits(q_pe.cpu()), qp, mqp, "q_pe")


@pytest.mark.parametrize("name", wl.ORDER)
def test_projection_matches_oracle(name):
    w = wl.small(name, seed=41)
    p = wl.projection(w, seed=41)
    dw, qn, qp = run_projection(w, p)
    check_projection(w, p, dw, qn, qp)


@pytest.mark.parametrize("name,batch", [
    ("qwen05b_b16_h14_r256_t2048", 129),          # 129 rows: 128-column tiles, a one-row tail tile
    ("llama1b_paged_b128_h32_r512_t128_8192", 40),  # 200 rows of 5-token chunks, paged
    ("llama3b_long_b8_h24_r512_t16k_32k", 33),    # 33 rows, 192-wide query heads
    ("llama1b_paged_b128_h32_r512_t128_8192", 128),  # 640 rows: 256-column tiles (one wave of 95 CTAs)
    ("llama1b_paged_b128_h32_r512_t128_8192", 127),  # 635 rows: 256-column tiles, a 123-row tail tile
])
def test_projection_row_tiles(name, batch):
    s = wl.SHAPES[name]
    w = wl.make(s, seed=42, batch=batch, kv_range=(s.q_len + 1, 300))
    p = wl.projection(w, seed=42)
    dw, qn, qp = run_projection(w, p)
    check_projection(w, p, dw, qn, qp)


def test_projection_without_queries_and_other_rotation():
    s = dataclasses.replace(wl.SHAPES["llama1b_chunk5_b32_h32_r512_t4096"], rope_style=1, rope_base=500000.0)
    w = wl.make(s, seed=43, batch=4, kv_range=(6, 700))
    p = wl.projection(w, seed=43)
    dw, _, _ = run_projection(w, p, with_q=False)
    check_projection(w, p, dw, None, None, with_q=False)


def test_projection_paged_equals_contiguous_bitwise():
    shape = wl.SHAPES["llama1b_paged_b128_h32_r512_t128_8192"]
    wp = wl.make(shape, seed=44, batch=5, kv_range=(70, 650))
    p = wl.projection(wp, seed=44)
    cap = int(wp.kv_len.max())
    c = torch.zeros(5, cap, shape.rank, dtype=torch.bfloat16)
    r = torch.zeros(5, cap, shape.d_rope, dtype=torch.bfloat16)
    wc = dataclasses.replace(wp, shape=dataclasses.replace(shape, paged=False), c_kv=c, k_rope=r, block_table=None,
                             num_pages=0, capacity=cap)
    dp, qn_p, qp_p = run_projection(wp, p)
    dc, qn_c, qp_c = run_projection(wc, p)
    assert abi.check_status() == abi.MLA_OK
    assert torch.equal(qn_p, qn_c) and torch.equal(qp_p, qp_c)
    for b in range(5):
        for t in range(int(wp.start_pos[b]), int(wp.kv_len[b])):
            pg, sl = int(wp.block_table[b, t // 64]), t % 64
            assert torch.equal(dp.cache.c_kv[pg, sl], dc.cache.c_kv[b, t])
            assert torch.equal(dp.cache.k_rope[pg, sl], dc.cache.k_rope[b, t])


def test_projection_bad_position_is_reported_and_queries_still_written():
    w = wl.small("qwen05b_b16_h14_r256_t2048", seed=45)
    p = wl.projection(w, seed=45)
    w.start_pos[1] = w.capacity                   # past the end: that entry's cache rows are skipped
    dw, qn, qp = run_projection(w, p)
    assert abi.check_status() == abi.MLA_ERR_DEVICE_BOUNDS
    w_ok = dataclasses.replace(w, start_pos=w.start_pos.clone())
    w_ok.start_pos[1] = 0
    _, qn_ref, qp_ref = oracle_projection(w_ok, p)
    _, _, mqn, mqp = magnitudes(w, p)
    assert_one_rounding(bits(qn.cpu()), qn_ref, mqn, "q_nope")
    assert_one_rounding(bits(qp.cpu()), qp_ref, mqp, "q_pe")


def _round_bf16(x: np.ndarray) -> np.ndarray:
    """The oracle's own single rounding of fp64 values to bf16 bits."""
    return np.vectorize(orc.bf16_round, otypes=[np.uint16])(x)


@pytest.mark.parametrize("name", ["qwen05b_b16_h14_r256_t2048", "llama1b_paged_b128_h32_r512_t128_8192"])
def test_step_from_hidden_states_matches_oracle(name):
    """Projection, absorption, attention, combine and output projection from
    the hidden states, against the oracle doing the same (its queries rounded
    to bf16 like the ones the step stores)."""
    w = wl.small(name, seed=46)
    p = wl.projection(w, seed=46)
    dw = abi.to_device(w)
    d = gpu_dims(w, p.hidden) if w.shape.hidden == 0 else dw.dims
    step = abi.DecodeStep(d, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    step.from_hidden(p.h.cuda(), p.w_dkv.cuda(), p.w_kr.cuda(), p.w_q.cuda(), dw.start_pos, dw.kv_len, dw.w_uk,
                     dw.w_uv, dw.w_o)
    assert abi.check_status() == abi.MLA_OK
    cache, qn, qp = oracle_projection(w, p)
    ref = orc.mla_decode(dims_with_hidden(w, p.hidden), cache, _round_bf16(qn), _round_bf16(qp), w.kv_len.numpy(),
                         bits(w.w_uk), bits(w.w_uv), None if w.w_o is None else bits(w.w_o))
    for key, got in (("o_lat", step.o_lat.cpu().numpy()), ("o", bf16_to_f64(bits(step.o.cpu())))):
        mx, mean = rel_errors(got, ref[key])
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"{key}: max {mx:.3e} mean {mean:.3e}"
    if w.w_o is not None:
        mx, mean = rel_errors(bf16_to_f64(bits(step.out.cpu())), ref["out"])
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"out: max {mx:.3e} mean {mean:.3e}"
