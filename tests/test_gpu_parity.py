"""GPU parity: every entry point of the C ABI against the fp64 oracle on the
same seeded inputs.

Bars: cache append and paged addressing bit-exact (latent rows are copies;
rotated keys within one bf16 rounding of the exact fp64 rotation); every
floating-point output within max|d| <= 2e-2 max|ref| and mean relative error
sum|d| / sum|ref| <= 5e-3.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, dims_of, oracle_cache, oracle_step, rel_errors

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 5e-3


def assert_close(got, ref, what):
    mx, mean = rel_errors(got, ref)
    assert mx <= MAX_TOL and mean <= MEAN_TOL, f"{what}: max {mx:.3e} mean {mean:.3e}"
    return mx, mean


def run_step(dw: abi.DeviceWorkload, num_splits=0, append=True):
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len, num_splits)
    kw = dict(c_new=dw.c_new, kr_new=dw.kr_new, start_pos=dw.start_pos) if append else {}
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, **kw)
    code = abi.check_status()
    assert code == abi.MLA_OK, abi.status_name(code)
    return step


def test_bounded_wait_times_out_and_reports():
    abi.check_status()
    abi.selftest_wait_timeout(2_000_000)                 # 2 ms, nothing ever signals the barrier
    assert abi.check_status() == abi.MLA_ERR_DEVICE_TIMEOUT
    assert abi.check_status() == abi.MLA_OK              # the word is cleared by the read


@pytest.mark.parametrize("name", wl.ORDER)
def test_cache_append_bit_exact(name):
    w = wl.small(name, seed=11)
    dw = abi.to_device(w)
    abi.cache_append(dw.dims, dw.cache, dw.c_new, dw.kr_new, dw.start_pos)
    assert abi.check_status() == abi.MLA_OK
    cache = oracle_cache(w)
    orc.cache_append(dims_of(w), cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    got_c, got_r = bits(dw.cache.c_kv.cpu()), bits(dw.cache.k_rope.cpu())
    # latent rows and every untouched row: identical bits
    assert np.array_equal(got_c, cache.c_kv)
    diff = got_r != cache.k_rope
    # rotated keys: the GPU rotates in fp32, the oracle in fp64; both round once
    # to bf16, so they may differ by one unit in the last place, nowhere else
    if diff.any():
        a = got_r[diff].astype(np.int32)
        b = cache.k_rope[diff].astype(np.int32)
        assert np.all(np.abs(a - b) <= 1), "rotated key off by more than one bf16 ulp"
        assert diff.mean() < 0.01
    untouched = np.ones(got_r.shape[:2], bool)
    s = w.shape
    for bi in range(w.kv_len.numel()):
        for t in range(int(w.start_pos[bi]), int(w.kv_len[bi])):
            if s.paged:
                untouched[int(w.block_table[bi, t // s.page_size]), t % s.page_size] = False
            else:
                untouched[bi, t] = False
    assert not diff[untouched].any()


@pytest.mark.parametrize("name", wl.ORDER)
def test_absorb_q(name):
    w = wl.small(name, seed=12)
    dw = abi.to_device(w)
    s = w.shape
    q_abs = torch.empty(dw.batch, dw.q_len, s.num_heads, s.rank + s.d_rope, dtype=torch.bfloat16, device="cuda")
    abi.absorb_q(dw.dims, dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, q_abs)
    assert abi.check_status() == abi.MLA_OK
    q_lat, q_rot = orc.absorb_q(dims_of(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk))
    got = bf16_to_f64(bits(q_abs.cpu()))
    assert_close(got[..., :s.rank], q_lat, "q_lat")
    # the rotated positional query: one fp32 rotation rounded to bf16
    ref = q_rot
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(ref), 1e-30))) - 7)
    assert np.all(np.abs(got[..., s.rank:] - ref) <= ulp + 1e-6)


@pytest.mark.parametrize("path", ["persistent", "gemm"])
@pytest.mark.parametrize("shape,batch", [
    ("llama1b_paged_b128_h32_r512_t128_8192", 128),  # 4 heads per group: 20 whole 128-row tiles per group
    ("llama1b_paged_b128_h32_r512_t128_8192", 127),  # a 108-row tail tile
    ("llama3b_long_b8_h24_r512_t16k_32k", 700),      # 3 heads per group (126-row tiles), d_nope 128: two K chunks
    ("llama1b_chunk5_b32_h32_r512_t4096", 16),       # 128-column slices, a 64-row tail tile
    ("qwen05b_b16_h14_r256_t2048", 19),              # 7 heads per group, 133 rows: a 7-row tail tile
    ("tiny_b1_h8_r128_t256", 3),                     # one head per group
    (wl.Shape("rank192", 5, 8, 2, 64, 32, 64, 192, 256, 2, 100, 400), 40),  # rank 192: 64-column slices
])
def test_absorb_q_both_kernels(shape, batch, path, tuning):
    """The persistent absorption kernel and the grouped GEMM, each forced,
    against the oracle: whole and ragged row tiles, every heads-per-group
    count, one and two K chunks, 64-, 128- and 256-column slices of the
    latent (narrower for fewer rows), and several items per CTA (the paged
    rows)."""
    tuning(GBMLA_ABSORB=path)
    s = wl.SHAPES[shape] if isinstance(shape, str) else shape
    w = wl.make(s, seed=40, batch=batch, kv_range=(s.q_len, 64))
    dw = abi.to_device(w)
    q_abs = torch.empty(batch, s.q_len, s.num_heads, s.rank + s.d_rope, dtype=torch.bfloat16, device="cuda")
    abi.absorb_q(dw.dims, dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, q_abs)
    assert abi.check_status() == abi.MLA_OK
    q_lat, q_rot = orc.absorb_q(dims_of(w), bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk))
    got = bf16_to_f64(bits(q_abs.cpu()))
    assert_close(got[..., :s.rank], q_lat, "q_lat")
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(q_rot), 1e-30))) - 7)
    assert np.all(np.abs(got[..., s.rank:] - q_rot) <= ulp + 1e-6)


@pytest.mark.parametrize("name", wl.ORDER)
def test_decode_step_matches_oracle(name):
    w = wl.small(name, seed=13)
    dw = abi.to_device(w)
    step = run_step(dw)
    ref = oracle_step(w)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(step.lse.cpu().numpy(), ref["lse"], "lse")
    assert_close(bf16_to_f64(bits(step.o.cpu())), ref["o"], "o")
    if w.w_o is not None:
        assert_close(bf16_to_f64(bits(step.out.cpu())), ref["out"], "out")


@pytest.mark.parametrize("kernel", ["simt", "tc"])
@pytest.mark.parametrize("name", ["qwen05b_b16_h14_r256_t2048", "llama1b_paged_b128_h32_r512_t128_8192"])
def test_split_count_invariance(name, kernel, tuning):
    """The split count changes only how the softmax sum is grouped.  The
    CUDA-core kernel keeps the weights in fp32 (agreement to fp32 noise); the
    tensor-core kernel rounds each weight to bf16 relative to the running
    maximum, which depends on where a split starts, so its bound is the bf16
    rounding of the weights (2^-9 relative each)."""
    tuning(GBMLA_ATTN_KERNEL=kernel)
    o_tol, l_tol = (1e-5, 1e-5) if kernel == "simt" else (4e-3, 1e-3)
    w = wl.small(name, seed=14)
    outs = []
    for S in (1, 2, 7, 0):
        dw = abi.to_device(w)
        step = run_step(dw, num_splits=S)
        outs.append((step.o_lat.cpu().numpy().astype(np.float64), step.lse.cpu().numpy().astype(np.float64)))
    for o, l in outs[1:]:
        assert rel_errors(o, outs[0][0])[0] < o_tol
        assert np.abs(l - outs[0][1]).max() < l_tol


@pytest.mark.parametrize("kernel", ["simt", "tc"])
@pytest.mark.parametrize("shape,many", [
    ("llama3b_long_b8_h24_r512_t16k_32k", 24),   # rank 512: four slot groups of 64 threads
    ("llama3b_long_b8_h24_r512_t16k_32k", 64),   # more partitions than tiles: empty ones in every group
    ("qwen05b_b16_h14_r256_t2048", 16),          # rank 256: eight groups of 32 threads
    ("tiny_b1_h8_r128_t256", 9),                 # rank 128: eight groups, two rows side by side
    (wl.Shape("rank192", 5, 8, 2, 64, 32, 64, 192, 256, 2, 100, 400), 12),  # 24 threads of each 32 hold the row
])
def test_combine_slot_groups(shape, many, kernel, tuning):
    """Many partitions per sequence (at least four) take the combine whose
    slot groups merge a row's partitions in parallel and meet in shared
    memory; one partition takes the plain merge.  The two agree to the
    attention kernel's split invariance, and the split run matches the
    oracle."""
    s = wl.SHAPES[shape] if isinstance(shape, str) else shape
    if kernel == "tc" and s.rank % 128:
        pytest.skip("the tensor-core kernel serves rank % 128 == 0")
    tuning(GBMLA_ATTN_KERNEL=kernel)
    o_tol, l_tol = (1e-5, 1e-5) if kernel == "simt" else (4e-3, 1e-3)
    w = wl.make(s, seed=41, batch=2, kv_range=(max(s.q_len, 300), 3000))
    ref = oracle_step(w)
    outs = []
    for S in (1, many):
        step = run_step(abi.to_device(w), num_splits=S)
        assert step.num_splits == S
        outs.append((step.o_lat.cpu().numpy().astype(np.float64), step.lse.cpu().numpy().astype(np.float64)))
    assert rel_errors(outs[1][0], outs[0][0])[0] < o_tol
    assert np.abs(outs[1][1] - outs[0][1]).max() < l_tol
    assert_close(outs[1][0], ref["o_lat"], "o_lat")
    assert_close(outs[1][1], ref["lse"], "lse")


@pytest.mark.parametrize("name", ["llama1b_paged_b128_h32_r512_t128_8192", "llama3b_long_b8_h24_r512_t16k_32k",
                                  "tiny_b1_h8_r128_t256"])
def test_decode_step_call_equals_the_five_calls(name):
    """mla_decode_step (the step in one call, as DecodeStep makes it) and
    the five entry points called one after another give the same bits."""
    w = wl.small(name, seed=42)
    dw1, dw2 = abi.to_device(w), abi.to_device(w)
    st1 = run_step(dw1)
    st2 = abi.DecodeStep(dw2.dims, dw2.cache, dw2.batch, dw2.q_len, dw2.max_kv_len)
    abi.cache_append(dw2.dims, dw2.cache, dw2.c_new, dw2.kr_new, dw2.start_pos)
    abi.absorb_q(dw2.dims, dw2.q_nope, dw2.q_pe, dw2.kv_len, dw2.w_uk, st2.q_abs)
    abi.decode_attn(dw2.dims, dw2.cache, dw2.kv_len, dw2.max_kv_len, st2.q_abs, st2.o_part, st2.lse_part,
                    st2.num_splits)
    abi.combine(dw2.dims, dw2.batch, dw2.q_len, dw2.kv_len, dw2.max_kv_len, st2.o_part, st2.lse_part, st2.o_lat,
                st2.lse, st2.num_splits)
    abi.out_proj(dw2.dims, st2.o_lat, dw2.w_uv, dw2.w_o, st2.o, st2.out)
    assert abi.check_status() == abi.MLA_OK
    for a, b in ((dw1.cache.c_kv, dw2.cache.c_kv), (dw1.cache.k_rope, dw2.cache.k_rope), (st1.q_abs, st2.q_abs),
                 (st1.o_lat, st2.o_lat), (st1.lse, st2.lse), (st1.o, st2.o)):
        assert torch.equal(a, b)
    if st1.out is not None:
        assert torch.equal(st1.out, st2.out)


def test_decode_step_graph_mode_replays_the_same_bits():
    """DecodeStep(graph=True) captures the step per set of input tensors and
    replays it: each replay gives the eager step's bits, and new inputs in the
    same buffers are picked up by the replay."""
    w = wl.small("llama1b_paged_b128_h32_r512_t128_8192", seed=44)
    dw1, dw2 = abi.to_device(w), abi.to_device(w)
    eager = run_step(dw1)
    ref_out = eager.out.clone()
    st = abi.DecodeStep(dw2.dims, dw2.cache, dw2.batch, dw2.q_len, dw2.max_kv_len, graph=True)
    for _ in range(3):
        out = st(dw2.q_nope, dw2.q_pe, dw2.kv_len, dw2.w_uk, dw2.w_uv, dw2.w_o, c_new=dw2.c_new, kr_new=dw2.kr_new,
                 start_pos=dw2.start_pos)
        torch.cuda.synchronize()
        assert torch.equal(out, ref_out)
        assert torch.equal(st.o_lat, eager.o_lat)
    assert len(st._graphs) == 1
    # new queries written into the captured buffers: the replay computes with them
    q2 = torch.randn(dw2.q_nope.shape, generator=torch.Generator().manual_seed(5)).to(torch.bfloat16)
    dw1.q_nope.copy_(q2)
    dw2.q_nope.copy_(q2)
    eager = run_step(dw1)
    out = st(dw2.q_nope, dw2.q_pe, dw2.kv_len, dw2.w_uk, dw2.w_uv, dw2.w_o, c_new=dw2.c_new, kr_new=dw2.kr_new,
             start_pos=dw2.start_pos)
    torch.cuda.synchronize()
    assert torch.equal(out, eager.out)
    assert abi.check_status() == abi.MLA_OK


def test_decode_step_checks_every_stage_before_launching():
    """An argument only a late stage rejects (a misaligned o_lat) fails the
    call before anything runs: the cache keeps its rows (the append, the
    first stage, did not run)."""
    w = wl.small("qwen05b_b16_h14_r256_t2048", seed=43)
    dw = abi.to_device(w)
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    before = dw.cache.c_kv.clone()
    step.o_lat = torch.empty(step.o_lat.numel() + 1, dtype=torch.float32, device="cuda")[1:].view(step.o_lat.shape)
    with pytest.raises(abi.MlaError):
        step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, c_new=dw.c_new, kr_new=dw.kr_new,
             start_pos=dw.start_pos)
    torch.cuda.synchronize()
    assert torch.equal(dw.cache.c_kv, before)


def test_paged_equals_contiguous_bitwise():
    """The same logical cache, paged through a shuffled block table or laid out
    contiguously, gives bit-identical attention outputs."""
    shape = wl.SHAPES["llama1b_paged_b128_h32_r512_t128_8192"]
    wp = wl.make(shape, seed=15, batch=5, kv_range=(70, 650))
    s = shape
    cap = int(wp.kv_len.max())
    c = torch.zeros(5, cap, s.rank, dtype=torch.bfloat16)
    r = torch.zeros(5, cap, s.d_rope, dtype=torch.bfloat16)
    for b in range(5):
        for t in range(int(wp.kv_len[b])):
            pg = int(wp.block_table[b, t // s.page_size])
            c[b, t], r[b, t] = wp.c_kv[pg, t % s.page_size], wp.k_rope[pg, t % s.page_size]
    wc = dataclasses.replace(wp, shape=dataclasses.replace(s, paged=False), c_kv=c, k_rope=r, block_table=None,
                             num_pages=0, capacity=cap)
    res = []
    for w in (wp, wc):
        dw = abi.to_device(w)
        step = run_step(dw, num_splits=3)
        res.append((step.o_lat.cpu(), step.lse.cpu(), step.o.cpu(), step.out.cpu()))
    for a, b in zip(*res):
        assert torch.equal(a, b)


def test_edge_lengths():
    """kv_len == q_len (the chunk alone), kv_len == 1, lengths ending exactly
    on a tile boundary and one past it, and kv_len == capacity."""
    shape = wl.SHAPES["llama1b_chunk5_b32_h32_r512_t4096"]
    base = wl.make(shape, seed=16, batch=6, kv_range=(5, 5))
    kv = torch.tensor([5, 6, 128, 129, 256, 300], dtype=torch.int32)
    w = dataclasses.replace(base, kv_len=kv, start_pos=kv - 5, capacity=300,
                            c_kv=wl._randn(torch.Generator().manual_seed(1), (6, 300, shape.rank)),
                            k_rope=wl._randn(torch.Generator().manual_seed(2), (6, 300, shape.d_rope)))
    dw = abi.to_device(w)
    step = run_step(dw)
    ref = oracle_step(w)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(bf16_to_f64(bits(step.out.cpu())), ref["out"], "out")
    # kv_len == 1 with q_len == 1: o_lat is exactly the single appended latent row
    s1 = wl.SHAPES["tiny_b1_h8_r128_t256"]
    w1 = wl.make(s1, seed=17, kv_range=(1, 1))
    dw1 = abi.to_device(w1)
    st1 = run_step(dw1)
    c0 = w1.c_new[0, 0].float()
    for h in range(s1.num_heads):
        assert torch.equal(st1.o_lat[0, 0, h].cpu(), c0)


@pytest.mark.parametrize("kernel", ["tc", "simt"])
@pytest.mark.parametrize("name", ["llama1b_chunk5_b32_h32_r512_t4096", "llama3b_long_b8_h24_r512_t16k_32k"])
def test_longest_query_chunk(name, kernel, tuning):
    """q_len = 16, the most the entry points take (a catch-up chunk of
    gamma = 15): 512 or 384 query rows per sequence (seven or five row groups
    of the tensor-core kernel), causal inside the chunk, the absorption on its
    persistent kernel (d_nope 64) or its grouped GEMM (d_nope 128) -- the
    step against the oracle."""
    tuning(GBMLA_ATTN_KERNEL=kernel)
    s = wl.SHAPES[name]
    w = wl.make(s, seed=45, batch=3, kv_range=(16, 700), q_len=16)
    step = run_step(abi.to_device(w))
    ref = oracle_step(w)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(step.lse.cpu().numpy(), ref["lse"], "lse")
    assert_close(bf16_to_f64(bits(step.out.cpu())), ref["out"], "out")


def test_empty_batch_is_a_noop():
    w = wl.small("tiny_b1_h8_r128_t256")
    dw = abi.to_device(w)
    empty = torch.empty(0, 1, 8, 64, dtype=torch.bfloat16, device="cuda")
    q_abs = torch.empty(0, 1, 8, 160, dtype=torch.bfloat16, device="cuda")
    abi.absorb_q(dw.dims, empty, empty[..., :32], dw.kv_len[:0], dw.w_uk, q_abs)
    assert abi.check_status() == abi.MLA_OK


def test_device_faults_are_reported_not_trapped():
    # a block-table entry outside the page pool
    w = wl.small("llama1b_paged_b128_h32_r512_t128_8192", seed=18)
    w.block_table[1, 0] = w.num_pages + 7
    dw = abi.to_device(w)
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, c_new=dw.c_new, kr_new=dw.kr_new,
         start_pos=dw.start_pos)
    assert abi.check_status() == abi.MLA_ERR_DEVICE_BOUNDS
    # a length above the stated maximum
    w = wl.small("qwen05b_b16_h14_r256_t2048", seed=19)
    dw = abi.to_device(w)
    dw.kv_len[0] = dw.max_kv_len + 1
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o)
    assert abi.check_status() == abi.MLA_ERR_DEVICE_BOUNDS
    # an append position past the capacity
    dw.start_pos[0] = dw.cache.capacity
    abi.cache_append(dw.dims, dw.cache, dw.c_new, dw.kr_new, dw.start_pos)
    assert abi.check_status() == abi.MLA_ERR_DEVICE_BOUNDS
    # the context is still usable afterwards
    dw = abi.to_device(wl.small("tiny_b1_h8_r128_t256"))
    run_step(dw)


def test_deterministic():
    w = wl.small("llama3b_long_b8_h24_r512_t16k_32k", seed=20)
    a = run_step(abi.to_device(w)).o_lat.cpu()
    b = run_step(abi.to_device(w)).o_lat.cpu()
    assert torch.equal(a, b)


@pytest.mark.parametrize("name", wl.ORDER)
def test_tensor_core_kernel_matches_cuda_core_kernel(name, tuning):
    """The two attention kernels of the library agree on the same inputs (they
    differ only in rounding: the tensor-core kernel multiplies bf16 weights)."""
    w = wl.small(name, seed=21)
    res = {}
    for kern in ("simt", "tc"):
        tuning(GBMLA_ATTN_KERNEL=kern)
        step = run_step(abi.to_device(w))
        res[kern] = (step.o_lat.cpu().numpy().astype(np.float64), step.lse.cpu().numpy().astype(np.float64))
    mx, mean = rel_errors(res["tc"][0], res["simt"][0])
    assert mx <= MAX_TOL and mean <= MEAN_TOL, (mx, mean)
    assert np.abs(res["tc"][1] - res["simt"][1]).max() < 1e-2


@pytest.mark.parametrize("env", [
    {},                                                   # 2 x 80 rows, independent CTAs, streamed queries
    {"GBMLA_TC_MAX_SLOTS": "4"},                          # the smallest ring: every slot reused within a tile
    {"GBMLA_TC_MAX_N": "32", "GBMLA_TC_MAX_SLOTS": "4"},  # 5 x 32 rows
    {"GBMLA_TC_MAX_N": "48"},
    {"GBMLA_TC_MAX_N": "64"},
    {"GBMLA_TC_PV_SLOTS": "4"},                           # five streamed-query QK slots
    {"GBMLA_TC_QUERY": "resident"},                       # queries resident in shared memory
    {"GBMLA_TC_QUERY": "resident", "GBMLA_TC_MAX_SLOTS": "4"},
    {"GBMLA_TC_QUERY": "resident", "GBMLA_TC_MAX_N": "32"},
], ids=["rows80", "ring4", "n32_ring4", "n48", "n64", "pv4", "resident", "resident_ring4", "resident_n32"])
@pytest.mark.parametrize("splits", [1, 3, 7])
def test_tensor_core_kernel_shapes_and_rings(env, splits, tuning):
    """Several sequences per CTA, tail tiles of one or two pages, and rings
    smaller than a tile's chunk count (the regime where a look-ahead barrier
    wait once cleared the next sequence's rows): every query-group size and
    ring size matches the oracle, with the queries streamed through the
    ring beside each cache chunk (the default) or resident in shared
    memory.  With 32 and 48 rows the
    kernel alternates two O^T buffers between sequences and drains each after
    the next one's first tile; one split puts all five sequences in one CTA,
    so both buffers are reused and every deferred drain runs."""
    tuning(**env)
    shape = wl.SHAPES["llama1b_paged_b128_h32_r512_t128_8192"]
    w = wl.make(shape, seed=15, batch=5, kv_range=(70, 650))
    step = run_step(abi.to_device(w), num_splits=splits)
    ref = oracle_step(w)
    assert_close(step.o_lat.cpu().numpy(), ref["o_lat"], "o_lat")
    assert_close(step.lse.cpu().numpy(), ref["lse"], "lse")


@pytest.mark.parametrize("name,groups", [("tiny_b1_h8_r128_t256", 1), ("qwen05b_b16_h14_r256_t2048", 1),
                                         ("llama3b_long_b8_h24_r512_t16k_32k", 1),
                                         ("llama1b_chunk5_b32_h32_r512_t4096", 2)])
def test_automatic_split_count(name, groups):
    """num_splits = 0 resolves by the rule mla_workspace_size documents: one
    partition per SM (per pair of SMs for two query groups), capped by the
    tile count T = batch ceil(max_kv_len / 128); when that leaves at most four
    tiles per partition, the fewest partitions with the same most tiles."""
    s = wl.SHAPES[name]
    dims = abi.Dims(s.num_heads, s.num_kv_groups, s.d_nope, s.d_rope, s.d_v, s.rank, s.hidden, s.sm_scale,
                    s.rope_style, s.rope_base)
    max_kv = s.kv_hi
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    tiles = s.batch * -(-max_kv // abi.SPLIT_TILE)
    want = max(1, min(sms // groups, tiles))
    per = -(-tiles // want)
    if per <= 4:
        want = -(-tiles // per)
    assert abi.workspace_size(dims, s.batch, s.q_len, max_kv)[2] == want
    # a requested count is taken as given
    assert abi.workspace_size(dims, s.batch, s.q_len, max_kv, 7)[2] == 7
