"""mla_decode_attn_noalloc: the attention core and split combine for callers
that cannot allocate device memory (runtimes that own every device byte
through their own pool, inference paths with a memory budget fixed up front,
plugins handed only their inputs and outputs).  Its split partials live in an
array the library reserves statically, so the call takes no partial buffers.

Checked through the C ABI against mla_decode_attn + mla_combine (the entry
points that take caller-allocated partials), on two calls in a row, so that
the second call runs on whatever the first left in the shared array.  This
file sorts last so that a run stopping at its first failure has already run
every other test; it passes alone and after the others."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import rel_errors

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 5e-3


def _reference(dw: abi.DeviceWorkload):
    """q_abs, and o_lat / lse through the caller-buffer entry points."""
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, c_new=dw.c_new, kr_new=dw.kr_new,
         start_pos=dw.start_pos)
    assert abi.check_status() == abi.MLA_OK
    return step


@pytest.mark.parametrize("case", ["qwen05b_full", "llama3b_long_full", "paged_small"])
def test_noalloc_matches_caller_buffer_path_twice(case):
    if case == "qwen05b_full":
        w = wl.make("qwen05b_b16_h14_r256_t2048", seed=3)
    elif case == "llama3b_long_full":
        w = wl.make("llama3b_long_b8_h24_r512_t16k_32k", seed=3)
    else:
        w = wl.small("llama1b_paged_b128_h32_r512_t128_8192", seed=3)
    dw = abi.to_device(w)
    ref = _reference(dw)
    s = w.shape
    for call in range(2):
        o_lat = torch.full((dw.batch, dw.q_len, s.num_heads, s.rank), float("nan"), device="cuda")
        lse = torch.full((dw.batch, dw.q_len, s.num_heads), float("nan"), device="cuda")
        abi.decode_attn_noalloc(dw.dims, dw.cache, dw.kv_len, dw.max_kv_len, ref.q_abs, o_lat, lse,
                                num_splits=ref.num_splits)
        assert abi.check_status() == abi.MLA_OK
        got, want = o_lat.cpu().numpy().astype(np.float64), ref.o_lat.cpu().numpy().astype(np.float64)
        mx, mean = rel_errors(got, want)
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"call {call}: max {mx:.3e} mean {mean:.3e}"
        # the same kernels over the same partition: identical bits
        assert torch.equal(o_lat.cpu(), ref.o_lat.cpu()), f"call {call}: o_lat differs"
        assert torch.equal(lse.cpu(), ref.lse.cpu()), f"call {call}: lse differs"
    # the automatic split count gives the same result within tolerance
    o_auto = torch.empty_like(ref.o_lat)
    abi.decode_attn_noalloc(dw.dims, dw.cache, dw.kv_len, dw.max_kv_len, ref.q_abs, o_auto, None)
    assert abi.check_status() == abi.MLA_OK
    mx, mean = rel_errors(o_auto.cpu().numpy(), ref.o_lat.cpu().numpy())
    assert mx <= MAX_TOL and mean <= MEAN_TOL


SCRATCH_FLOATS = (32 << 20) // 4  # the library's static array of partials


def _fitting_splits(batch: int, rows: int, rank: int, s_auto: int) -> int:
    """The automatic split count lowered until (batch + S - 1) partial slots
    of rows x rank floats (plus the lse slots, rounded up to 64 floats) fit."""
    def need(S):
        slots = batch + S - 1
        return slots * rows * rank + ((slots * rows + 63) // 64) * 64
    S = s_auto
    while S >= 1 and need(S) > SCRATCH_FLOATS:
        S -= 1
    return S


def test_noalloc_lowers_the_automatic_split_count_to_fit():
    """The full chunk workload (32 sequences of 4096 tokens, 160 query rows,
    rank 512) needs more partial slots at the automatic split count than the
    array holds; with num_splits = 0 the call lowers S until they fit.  Its
    output equals, bit for bit, mla_decode_attn + mla_combine run at that lowered
    S with caller buffers, and the automatic-S caller-buffer result within
    tolerance -- on two calls in a row."""
    w = wl.make("llama1b_chunk5_b32_h32_r512_t4096", seed=5)
    dw = abi.to_device(w)
    s = w.shape
    ref = _reference(dw)  # automatic S, caller buffers
    s_auto = ref.num_splits
    s_fit = _fitting_splits(dw.batch, dw.q_len * s.num_heads, s.rank, s_auto)
    assert 1 <= s_fit < s_auto, (s_fit, s_auto)  # the lowering branch is the one under test
    low = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len, s_fit)
    assert low.num_splits == s_fit
    abi.decode_attn(dw.dims, dw.cache, dw.kv_len, dw.max_kv_len, ref.q_abs, low.o_part, low.lse_part, s_fit)
    abi.combine(dw.dims, dw.batch, dw.q_len, dw.kv_len, dw.max_kv_len, low.o_part, low.lse_part, low.o_lat, low.lse,
                s_fit)
    assert abi.check_status() == abi.MLA_OK
    for call in range(2):
        o_lat = torch.full_like(ref.o_lat, float("nan"))
        lse = torch.full_like(ref.lse, float("nan"))
        abi.decode_attn_noalloc(dw.dims, dw.cache, dw.kv_len, dw.max_kv_len, ref.q_abs, o_lat, lse, num_splits=0)
        assert abi.check_status() == abi.MLA_OK
        assert torch.equal(o_lat.cpu(), low.o_lat.cpu()), f"call {call}: o_lat differs from the lowered-S path"
        assert torch.equal(lse.cpu(), low.lse.cpu()), f"call {call}: lse differs from the lowered-S path"
        mx, mean = rel_errors(o_lat.cpu().numpy(), ref.o_lat.cpu().numpy())
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"call {call}: max {mx:.3e} mean {mean:.3e}"


def test_noalloc_refuses_sizes_beyond_its_array():
    """The full paged workload needs more partial slots than the 32 MiB array
    holds even with one split per sequence: refused before any launch."""
    w = wl.make("llama1b_paged_b128_h32_r512_t128_8192", seed=3)
    dw = abi.to_device(w)
    s = w.shape
    q_abs = torch.zeros(dw.batch, dw.q_len, s.num_heads, s.rank + s.d_rope, dtype=torch.bfloat16, device="cuda")
    o_lat = torch.empty(dw.batch, dw.q_len, s.num_heads, s.rank, device="cuda")
    for splits in (0, 76):
        with pytest.raises(abi.MlaError) as exc:
            abi.decode_attn_noalloc(dw.dims, dw.cache, dw.kv_len, dw.max_kv_len, q_abs, o_lat, None,
                                    num_splits=splits)
        assert exc.value.code == abi.MLA_ERR_UNSUPPORTED
    assert abi.check_status() == abi.MLA_OK
