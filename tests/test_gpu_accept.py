"""GPU parity of mla_acceptance_stats (Sec. 3.3, Eqs. 9-10) against the fp64
oracle on the same seeded logits.

Bars: the argmaxes and the greedy decision are integers decided on the
logits themselves, so they must match exactly (lowest index on ties);
alpha_sample is an fp32 sum of ~10^5 probabilities formed with fp32
exponentials (each within a few ulp) and summed hierarchically (at most a few
hundred serial additions per thread, then trees), so its error is ~1e-5 at
most: the bar is 1e-4 absolute.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_27269_gb300 import abi
from paper_2607_27269_gb300 import workloads as wl
from tests.helpers import bf16_to_f64, bits

pytestmark = pytest.mark.gpu

ALPHA_TOL = 1e-4


def values(t: torch.Tensor) -> np.ndarray:
    return bf16_to_f64(bits(t)) if t.dtype == torch.bfloat16 else t.double().numpy()


def padded(x: torch.Tensor) -> torch.Tensor:
    """x on the GPU in rows padded to a 16-byte multiple (a view of the first vocab entries)."""
    per = 16 // x.element_size()
    stride = (x.shape[1] + per - 1) // per * per
    buf = torch.zeros(x.shape[0], stride, dtype=x.dtype, device="cuda")
    buf[:, :x.shape[1]] = x.cuda()
    return buf[:, :x.shape[1]]


def check(draft: torch.Tensor, target: torch.Tensor):
    alpha, ad, at, gr = abi.acceptance_stats(padded(draft), padded(target))
    torch.cuda.synchronize()
    ref = orc.acceptance(values(draft), values(target))
    assert np.array_equal(ad.cpu().numpy(), ref["argmax_draft"])
    assert np.array_equal(at.cpu().numpy(), ref["argmax_target"])
    assert np.array_equal(gr.cpu().numpy(), ref["greedy"])
    err = np.abs(alpha.cpu().numpy().astype(np.float64) - ref["alpha_sample"])
    assert err.max() <= ALPHA_TOL, err.max()
    return ref


@pytest.mark.parametrize("name", wl.ORDER)
def test_acceptance_matches_oracle(name):
    lg = wl.logits(name, seed=51, rows=6)
    ref = check(lg.draft, lg.target)
    assert 0.05 < ref["alpha_sample"].mean() < 0.99      # the inputs exercise the overlap, not an edge


def test_acceptance_fp32_logits_and_identical_rows():
    lg = wl.logits("qwen05b_b16_h14_r256_t2048", seed=52, rows=5)
    check(lg.draft.float(), lg.target.float())
    ref = check(lg.target, lg.target)
    assert np.all(ref["greedy"] == 1)


def test_acceptance_ties_ragged_and_tiny_vocabularies():
    g = torch.Generator().manual_seed(53)
    for vocab in (13, 1003, 40961):
        d = (torch.randn(4, vocab, generator=g) * 2).to(torch.bfloat16)
        t = (torch.randn(4, vocab, generator=g) * 2).to(torch.bfloat16)
        # equal maxima far apart (different slices of the cluster): the lowest index wins
        d[0, vocab - 1] = d[0, 0] = 30.0
        t[1, vocab // 2] = t[1, 1] = 30.0
        check(d, t)


def test_acceptance_row_stride_and_empty():
    g = torch.Generator().manual_seed(54)
    full = (torch.randn(3, 1008, generator=g) * 3).to(torch.bfloat16).cuda()
    full2 = (torch.randn(3, 1008, generator=g) * 3).to(torch.bfloat16).cuda()
    d, t = full[:, :1001], full2[:, :1001]          # rows 1008 apart, 1001 tokens used
    alpha, ad, at, gr = abi.acceptance_stats(d, t)
    ref = orc.acceptance(values(d.cpu()), values(t.cpu()))
    assert np.array_equal(ad.cpu().numpy(), ref["argmax_draft"])
    assert np.abs(alpha.cpu().numpy() - ref["alpha_sample"]).max() <= ALPHA_TOL
    e = torch.empty(0, 100, dtype=torch.bfloat16, device="cuda")
    abi.acceptance_stats(e, e)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_acceptance_many_rows_ties_ragged_and_strided(dtype):
    """160 rows take the one-CTA-per-row kernel (more than one row per CTA
    on the grid of two CTAs per SM): ragged vocabularies (a tail past the last
    whole vector; a vocabulary shorter than one vector), equal maxima far
    apart (the lowest index wins), identical rows (greedy agreement, alpha =
    1) and rows padded to a longer stride -- every row against the oracle."""
    g = torch.Generator().manual_seed(56)
    rows = 160
    for vocab in (7, 1003, 40961):
        d = (torch.randn(rows, vocab, generator=g) * 2).to(dtype)
        t = (torch.randn(rows, vocab, generator=g) * 2).to(dtype)
        d[0, vocab - 1] = d[0, 0] = 30.0
        t[1, vocab // 2] = t[1, 1] = 30.0
        d[rows - 1, vocab - 1] = 40.0  # the maximum in the tail
        t[7] = d[7]
        ref = check(d, t)
        assert ref["greedy"][7] == 1 and abs(ref["alpha_sample"][7] - 1.0) < 1e-12
    # rows 1040 entries apart, 1001 used
    full = (torch.randn(rows, 1040, generator=g) * 3).to(dtype).cuda()
    full2 = (torch.randn(rows, 1040, generator=g) * 3).to(dtype).cuda()
    dd, tt = full[:, :1001], full2[:, :1001]
    alpha, ad, at, gr = abi.acceptance_stats(dd, tt)
    ref = orc.acceptance(values(dd.cpu()), values(tt.cpu()))
    assert np.array_equal(ad.cpu().numpy(), ref["argmax_draft"])
    assert np.array_equal(at.cpu().numpy(), ref["argmax_target"])
    assert np.abs(alpha.cpu().numpy().astype(np.float64) - ref["alpha_sample"]).max() <= ALPHA_TOL


@pytest.mark.parametrize("name", ["qwen05b_b16_h14_r256_t2048", "llama1b_paged_b128_h32_r512_t128_8192"])
def test_acceptance_full_rows_sampled(name):
    """Every row of the workload on the GPU (the size bench.py times); the
    oracle checks a sample of rows."""
    lg = wl.logits(name, seed=55)
    alpha, ad, at, gr = abi.acceptance_stats(lg.draft.cuda(), lg.target.cuda())
    rows = lg.draft.shape[0]
    pick = np.unique(np.linspace(0, rows - 1, 8).astype(int))
    ref = orc.acceptance(values(lg.draft[pick]), values(lg.target[pick]))
    assert np.array_equal(ad.cpu().numpy()[pick], ref["argmax_draft"])
    assert np.array_equal(gr.cpu().numpy()[pick], ref["greedy"])
    assert np.abs(alpha.cpu().numpy()[pick] - ref["alpha_sample"]).max() <= ALPHA_TOL
