"""Parity at the five workloads' full sizes, in the launch configuration the
benchmark times (automatic split count): the whole batch runs on the GPU, and
the fp64 oracle recomputes a sample of sequences (the longest, the shortest
and one in between) which must match within the tolerances."""
from __future__ import annotations

import numpy as np
import pytest

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits, dims_of, oracle_cache, rel_errors

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

MAX_TOL, MEAN_TOL = 2e-2, 5e-3


@pytest.mark.parametrize("name", wl.ORDER)
def test_full_size_sampled(name):
    w = wl.make(name, seed=0)
    dw = abi.to_device(w)
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    step(dw.q_nope, dw.q_pe, dw.kv_len, dw.w_uk, dw.w_uv, dw.w_o, c_new=dw.c_new, kr_new=dw.kr_new,
         start_pos=dw.start_pos)
    assert abi.check_status() == abi.MLA_OK
    kv = w.kv_len.numpy()
    order = np.argsort(kv)
    seqs = sorted({int(order[-1]), int(order[0]), int(order[len(order) // 2])})
    dims = dims_of(w)
    cache = oracle_cache(w)
    orc.cache_append(dims, cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    ref = orc.mla_decode(dims, cache, bits(w.q_nope), bits(w.q_pe), kv, bits(w.w_uk), bits(w.w_uv),
                         None if w.w_o is None else bits(w.w_o), seqs=seqs)
    got = {"o_lat": step.o_lat.cpu().numpy(), "lse": step.lse.cpu().numpy(), "o": bf16_to_f64(bits(step.o.cpu()))}
    if w.w_o is not None:
        got["out"] = bf16_to_f64(bits(step.out.cpu()))
    for key, g in got.items():
        mx, mean = rel_errors(g[seqs], ref[key][seqs])
        assert mx <= MAX_TOL and mean <= MEAN_TOL, f"{name} {key}: max {mx:.3e} mean {mean:.3e}"
    # and the appended cache rows themselves are bit-exact copies on the GPU too
    got_c = bits(dw.cache.c_kv.cpu())
    assert np.array_equal(got_c, cache.c_kv)
