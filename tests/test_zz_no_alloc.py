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
