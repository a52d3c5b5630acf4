"""The interleaved cache layout: one [r + d_rope] row per token, the latent
part first, with c_kv and k_rope pointing into the same buffer and both token
strides r + d_rope (the layout include/gbmla.h allows through the strides).
The step through the C ABI (append into the fused rows, absorption,
attention, combine, output projection) is checked against the fp64 oracle,
and against the same step on separate buffers: the kernels read the same
values over the same partition, so the outputs are bit-identical.  The fused
rows after the append equal the oracle's two caches side by side, bit for bit
(latent rows copied, rotated keys within one bf16 rounding)."""
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


def fused(dw: abi.DeviceWorkload) -> abi.DeviceWorkload:
    """The same workload with its two caches copied into one interleaved buffer."""
    c, k = dw.cache.c_kv, dw.cache.k_rope
    r = c.shape[2]
    buf = torch.empty(c.shape[0], c.shape[1], r + k.shape[2], dtype=torch.bfloat16, device=c.device)
    buf[..., :r] = c
    buf[..., r:] = k
    cache = dataclasses.replace(dw.cache, c_kv=buf[..., :r], k_rope=buf[..., r:])
    assert cache.c_kv.stride(1) == r + k.shape[2] and cache.k_rope.stride(1) == r + k.shape[2]
    return dataclasses.replace(dw, cache=cache)


def run_step(dw: abi.DeviceWorkload):
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, c_new=dw.c_new, kr_new=dw.kr_new,
         start_pos=dw.start_pos)
    code = abi.check_status()
    assert code == abi.MLA_OK, abi.status_name(code)
    return step


@pytest.mark.parametrize("case", ["qwen_small", "qwen_full", "paged_small", "long_small"])
def test_interleaved_rows_match_oracle_and_separate_buffers(case):
    if case == "qwen_full":
        w = wl.make("qwen05b_b16_h14_r256_t2048", seed=41)
        seqs = [0, 7, 15]  # the oracle checks sampled sequences at full size
    else:
        name = {"qwen_small": "qwen05b_b16_h14_r256_t2048", "paged_small": "llama1b_paged_b128_h32_r512_t128_8192",
                "long_small": "llama3b_long_b8_h24_r512_t16k_32k"}[case]
        w = wl.small(name, seed=41)
        seqs = None
    s = w.shape
    sep = run_step(abi.to_device(w))
    dwf = fused(abi.to_device(w))
    fus = run_step(dwf)

    # identical bits to the separate-buffer step
    for a, b, what in ((fus.o_lat, sep.o_lat, "o_lat"), (fus.lse, sep.lse, "lse"), (fus.o, sep.o, "o")):
        assert torch.equal(a.cpu(), b.cpu()), what
    if sep.out is not None:
        assert torch.equal(fus.out.cpu(), sep.out.cpu()), "out"

    # the fused rows after the append hold the oracle's caches side by side
    cache = oracle_cache(w)
    orc.cache_append(dims_of(w), cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    buf = dwf.cache.c_kv.as_strided((dwf.cache.c_kv.shape[0], dwf.cache.c_kv.shape[1], s.rank + s.d_rope),
                                    (dwf.cache.c_kv.stride(0), dwf.cache.c_kv.stride(1), 1)).cpu()
    assert np.array_equal(bits(buf[..., :s.rank]), cache.c_kv)
    got_r = bf16_to_f64(bits(buf[..., s.rank:]))
    want_r = bf16_to_f64(cache.k_rope)
    ulp = np.abs(want_r) * 2.0 ** -7 + 1e-30
    assert (np.abs(got_r - want_r) <= ulp).all()

    # and the oracle's attention and output projection
    ref = oracle_step(w, seqs=seqs)
    idx = slice(None) if seqs is None else seqs
    for got, key in ((fus.o_lat, "o_lat"), (fus.out if fus.out is not None else fus.o, "out" if s.hidden else "o")):
        g = got.cpu()
        g = bf16_to_f64(bits(g)) if g.dtype == torch.bfloat16 else g.numpy().astype(np.float64)
        mx, mean = rel_errors(g[idx], ref[key][idx])
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"{key}: max {mx:.3e} mean {mean:.3e}"
