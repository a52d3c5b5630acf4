"""Output projection through the C ABI at row counts that take every tiling
of the tensor-core GEMM behind it: W_UV per KV group on o_lat (Sec. 3.2, the
value up-projection read through absorption) and the fixed W_O over the
concatenated heads (Sec. 4.1).

The row count B q picks the GEMM's layout: a few rows against a deep W_O split
K over a cluster with ring stages of only those rows (8 and 13 rows of the
long-context model, 16 and 3 of the Qwen one); a mid-size batch against the
2048-wide W_O splits full 128-row tiles over a cluster (160 rows); a large
batch runs several waves of unsplit tiles (640 rows); W_UV's short K shrinks
its row tiles when they would leave the SMs idle.  The fp64 oracle's o_lat is
handed to the GPU in fp32 and both outputs are compared with the oracle's."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, oracle_step, rel_errors

pytestmark = pytest.mark.gpu

MAX_TOL, MEAN_TOL = 2e-2, 5e-3

CASES = [
    ("llama3b_long_b8_h24_r512_t16k_32k", 8),
    ("llama3b_long_b8_h24_r512_t16k_32k", 13),
    ("llama3b_long_b8_h24_r512_t16k_32k", 1),
    ("qwen05b_b16_h14_r256_t2048", 16),
    ("qwen05b_b16_h14_r256_t2048", 3),
    ("llama1b_chunk5_b32_h32_r512_t4096", 32),
    ("llama1b_chunk5_b32_h32_r512_t4096", 7),
    ("llama1b_chunk5_b32_h32_r512_t4096", 128),
]


@pytest.mark.parametrize("name,batch", CASES)
def test_out_proj_row_counts(name, batch):
    s = wl.SHAPES[name]
    # short caches: the oracle's attention is cheap, the projection keeps its full width
    w = wl.make(s, seed=29, batch=batch, kv_range=(s.q_len + 3, s.q_len + 40))
    ref = oracle_step(w)
    dw = abi.to_device(w)
    o_lat = torch.from_numpy(ref["o_lat"].astype(np.float32)).cuda()
    o = torch.empty(batch, s.q_len, s.num_heads, s.d_v, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(batch, s.q_len, s.hidden, dtype=torch.bfloat16, device="cuda") if s.hidden else None
    abi.out_proj(dw.dims, o_lat, dw.w_uv, dw.w_o, o, out)
    assert abi.check_status() == abi.MLA_OK
    mx, mean = rel_errors(bf16_to_f64(bits(o.cpu())), ref["o"])
    assert mx <= MAX_TOL and mean <= MEAN_TOL, f"o: max {mx:.3e} mean {mean:.3e}"
    if out is not None:
        mx, mean = rel_errors(bf16_to_f64(bits(out.cpu())), ref["out"])
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"out: max {mx:.3e} mean {mean:.3e}"
