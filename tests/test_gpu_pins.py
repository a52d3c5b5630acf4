"""GPU pins that hold by the mathematics of the method rather than by
comparison with the oracle's numbers: relative-position invariance of the
rotary scores (Sec. 2, the rotation R_t), identity rotation at position 0,
masked rows that are never read, the causal mask inside a query chunk, the
single-key closed form o = W_UV c_0 (Eq. 3 with one key), the interleaved
pairing and other bases of the rotation, and projection shapes whose row
counts end on ragged tiles for every heads-per-group count of the workloads.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, dims_of, oracle_step, rel_errors, rope_complex

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 5e-3


def assert_close(got, ref, what):
    mx, mean = rel_errors(got, ref)
    assert mx <= MAX_TOL and mean <= MEAN_TOL, f"{what}: max {mx:.3e} mean {mean:.3e}"


def run_step(dw: abi.DeviceWorkload, num_splits=0):
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len, num_splits)
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, c_new=dw.c_new, kr_new=dw.kr_new,
         start_pos=dw.start_pos)
    code = abi.check_status()
    assert code == abi.MLA_OK, abi.status_name(code)
    return step


def outputs(step):
    return [step.o_lat.cpu(), step.lse.cpu(), step.o.cpu()] + ([step.out.cpu()] if step.out is not None else [])


@pytest.mark.parametrize("style", [0, 1])
def test_rotary_scores_depend_only_on_relative_position(style):
    """Rotating the query at p + d and the key at j + d gives the score of
    (p, j) for every shift d (R_p^T R_j = R_{j-p}); a key appended at position
    0 and a query at position 0 are not rotated at all (bit-exact copies)."""
    shape = dataclasses.replace(wl.SHAPES["tiny_b1_h8_r128_t256"], rope_style=style)
    shifts = [0, 1, 1000, 30000]
    p0, j0 = 37, 0
    B = len(shifts)
    w = wl.make(shape, seed=31, batch=B, kv_range=(1, 1), capacity=j0 + max(shifts) + 1)
    # the same query and key vectors in every sequence
    q_pe = w.q_pe[:1].expand(B, -1, -1, -1).contiguous()
    kr_new = w.kr_new[:1].expand(B, -1, -1).contiguous()
    w = dataclasses.replace(w, q_pe=q_pe, kr_new=kr_new)
    dw = abi.to_device(w)
    key_pos = torch.tensor([j0 + d for d in shifts], dtype=torch.int32, device="cuda")
    abi.cache_append(dw.dims, dw.cache, dw.c_new, dw.kr_new, key_pos)
    assert abi.check_status() == abi.MLA_OK
    s = shape
    q_abs = torch.empty(B, 1, s.num_heads, s.rank + s.d_rope, dtype=torch.bfloat16, device="cuda")
    qry_len = torch.tensor([p0 + d + 1 for d in shifts], dtype=torch.int32, device="cuda")
    abi.absorb_q(dw.dims, dw.q_nope, dw.q_pe, qry_len, dw.w_uk, q_abs)
    assert abi.check_status() == abi.MLA_OK
    qr = bf16_to_f64(bits(q_abs[..., s.rank:].cpu()))                        # [B, 1, H, dr]
    kr_rows = bits(dw.cache.k_rope.cpu())
    kr = np.stack([bf16_to_f64(kr_rows[b, j0 + shifts[b]]) for b in range(B)])  # [B, dr]
    qv, kv = bf16_to_f64(bits(q_pe[0, 0])), bf16_to_f64(bits(kr_new[0, 0]))
    kx = rope_complex(kv, j0, s.rope_base, style)
    for h in range(s.num_heads):
        qx = rope_complex(qv[h], p0, s.rope_base, style)
        exact = float(qx @ kx)
        # each rotated element carries one bf16 rounding (2^-9 relative) and
        # an fp32 rotation error far below it
        tol = 2.0 ** -8 * float(np.abs(qx) @ np.abs(kx)) * 1.05 + 1e-5 * np.linalg.norm(qx) * np.linalg.norm(kx)
        for b in range(B):
            got = float(qr[b, 0, h] @ kr[b])
            assert abs(got - exact) <= tol, (style, shifts[b], h, got, exact, tol)
    # position 0: the stored key is the appended key, bit for bit
    assert np.array_equal(kr_rows[0, 0], bits(kr_new[0, 0]))
    # a query at position 0 keeps its positional part unchanged
    abi.absorb_q(dw.dims, dw.q_nope, dw.q_pe, torch.ones(B, dtype=torch.int32, device="cuda"), dw.w_uk, q_abs)
    assert abi.check_status() == abi.MLA_OK
    assert np.array_equal(bits(q_abs[..., s.rank:].cpu()), bits(q_pe))


def _plant(t: torch.Tensor, mask: torch.Tensor, gen: torch.Generator):
    """Write +-1e4 into the rows of ``t`` [blocks, tokens, d] that ``mask`` marks."""
    sign = torch.randint(0, 2, t.shape, generator=gen).to(torch.float32) * 2 - 1
    big = (sign * 1e4).to(torch.bfloat16)
    return torch.where(mask[..., None], big, t)


@pytest.mark.parametrize("kernel", ["simt", "tc"])
@pytest.mark.parametrize("name", ["qwen05b_b16_h14_r256_t2048", "llama1b_paged_b128_h32_r512_t128_8192"])
def test_rows_past_kv_len_are_never_read(name, kernel, tuning):
    """Rows at or past a sequence's length (inside its capacity, in the tail of
    its last page, or in pages no sequence owns) hold +-1e4: every output is
    bit-identical to the run with ordinary values there."""
    tuning(GBMLA_ATTN_KERNEL=kernel)
    s = wl.SHAPES[name]
    if s.paged:
        w = wl.make(s, seed=32, batch=6, kv_range=(s.q_len + 1, 700), spare_pages=3)
        live = torch.zeros(w.c_kv.shape[:2], dtype=torch.bool)
        for b in range(6):
            for t in range(int(w.kv_len[b])):
                live[int(w.block_table[b, t // s.page_size]), t % s.page_size] = True
    else:
        w = wl.make(s, seed=32, batch=3, kv_range=(300, 700), capacity=900)
        live = torch.arange(w.capacity)[None, :] < w.kv_len[:, None]
    clean = outputs(run_step(abi.to_device(w)))
    g = torch.Generator().manual_seed(33)
    wp = dataclasses.replace(w, c_kv=_plant(w.c_kv, ~live, g), k_rope=_plant(w.k_rope, ~live, g))
    assert not torch.equal(wp.c_kv, w.c_kv)
    planted = outputs(run_step(abi.to_device(wp)))
    for a, b in zip(clean, planted):
        assert torch.equal(a, b)


@pytest.mark.parametrize("kernel", ["simt", "tc"])
def test_causal_mask_inside_the_chunk(kernel, tuning):
    """Query i of a chunk sees chunk tokens up to i only: replacing the last
    chunk token by +-1e4 leaves the outputs of every earlier query bit-identical
    and changes those of the last query."""
    tuning(GBMLA_ATTN_KERNEL=kernel)
    s = wl.SHAPES["llama1b_chunk5_b32_h32_r512_t4096"]
    w = wl.make(s, seed=34, batch=3, kv_range=(300, 1100))
    clean = outputs(run_step(abi.to_device(w)))
    g = torch.Generator().manual_seed(35)
    last = torch.zeros(3, s.q_len, dtype=torch.bool)
    last[:, -1] = True
    wp = dataclasses.replace(w, c_new=_plant(w.c_new, last, g), kr_new=_plant(w.kr_new, last, g))
    planted = outputs(run_step(abi.to_device(wp)))
    for a, b in zip(clean, planted):
        assert torch.equal(a[:, :-1], b[:, :-1])
        assert not torch.equal(a[:, -1], b[:, -1])


def test_single_key_gives_value_of_that_key():
    """With one key the softmax weight is exactly 1: o_lat = c_0 bit for bit,
    lse = the key's score, o[h] = W_UV[g(h)] c_0 and out = W_O concat_h o[h]."""
    s = wl.SHAPES["llama1b_paged_b128_h32_r512_t128_8192"]
    w = wl.make(s, seed=36, batch=4, kv_range=(1, 1))
    step = run_step(abi.to_device(w))
    c0 = bf16_to_f64(bits(w.c_new[:, 0]))                              # [B, r]
    hpg = s.num_heads // s.num_kv_groups
    for b in range(4):
        for h in range(s.num_heads):
            assert torch.equal(step.o_lat[b, 0, h].cpu(), w.c_new[b, 0].float())
    w_uv = bf16_to_f64(bits(w.w_uv))                                   # [G, dv, r]
    o_ref = np.stack([np.stack([w_uv[h // hpg] @ c0[b] for h in range(s.num_heads)]) for b in range(4)])
    o = bf16_to_f64(bits(step.o.cpu()))[:, 0]
    assert_close(o, o_ref, "o")
    # the output projection sees the bf16-rounded o, as the step computes it
    out_ref = o.reshape(4, -1) @ bf16_to_f64(bits(w.w_o)).T
    assert_close(bf16_to_f64(bits(step.out.cpu()))[:, 0], out_ref, "out")
    # lse of a single key is its scaled score
    ref = oracle_step(w)
    assert np.abs(step.lse.cpu().numpy() - ref["lse"]).max() < 1e-2


@pytest.mark.parametrize("style,base", [(1, 10000.0), (0, 500000.0), (1, 1e6)])
def test_rotation_pairing_and_base(style, base):
    """The interleaved pairing and other rotation bases through the whole step
    (cache append, absorption, attention, combine and projections)."""
    s = dataclasses.replace(wl.SHAPES["llama3b_long_b8_h24_r512_t16k_32k"], rope_style=style, rope_base=base)
    w = wl.make(s, seed=37, batch=3, kv_range=(300, 1100))
    step = run_step(abi.to_device(w))
    ref = oracle_step(w)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(bf16_to_f64(bits(step.out.cpu())), ref["out"], "out")


@pytest.mark.parametrize("name,batch", [
    ("tiny_b1_h8_r128_t256", 37),                 # 1 head per group, 37 rows
    ("qwen05b_b16_h14_r256_t2048", 1),            # 7 heads per group, 7 rows
    ("qwen05b_b16_h14_r256_t2048", 19),           # 133 rows: one full tile and a 5-row tail
    ("qwen05b_b16_h14_r256_t2048", 37),           # 259 rows
    ("llama3b_long_b8_h24_r512_t16k_32k", 5),     # 3 heads per group
    ("llama3b_long_b8_h24_r512_t16k_32k", 70),    # 210 rows
    ("llama1b_chunk5_b32_h32_r512_t4096", 7),     # 4 heads x 5 queries per sequence
])
def test_projection_ragged_rows(name, batch):
    """Absorption and output projections for row counts that end inside a
    tile, for every heads-per-group count of the workloads."""
    s = wl.SHAPES[name]
    w = wl.make(s, seed=38, batch=batch, kv_range=(s.q_len, 40))
    dw = abi.to_device(w)
    q_abs = torch.empty(batch, s.q_len, s.num_heads, s.rank + s.d_rope, dtype=torch.bfloat16, device="cuda")
    abi.absorb_q(dw.dims, dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, q_abs)
    assert abi.check_status() == abi.MLA_OK
    ref = oracle_step(w)
    q_lat = bf16_to_f64(bits(q_abs[..., :s.rank].cpu()))
    ref_lat, _ = orc.absorb_q(dims_of(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk))
    assert_close(q_lat, ref_lat, "q_lat")
    step = run_step(dw)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(bf16_to_f64(bits(step.o.cpu())), ref["o"], "o")
    if w.w_o is not None:
        assert_close(bf16_to_f64(bits(step.out.cpu())), ref["out"], "out")


def test_rank_that_is_not_a_multiple_of_128():
    """A latent rank of 192 (a multiple of 64 only) runs the CUDA-core
    attention kernel and a combine whose rows do not fill its blocks."""
    s = wl.Shape("rank192", 5, 8, 2, 64, 32, 64, 192, 256, 2, 100, 400)
    w = wl.make(s, seed=39)
    step = run_step(abi.to_device(w), num_splits=6)
    ref = oracle_step(w)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(step.lse.cpu().numpy(), ref["lse"], "lse")
    assert_close(bf16_to_f64(bits(step.out.cpu())), ref["out"], "out")
