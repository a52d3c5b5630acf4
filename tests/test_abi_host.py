"""CPU-only checks of the C ABI: the library builds, loads without a GPU and
exports every entry point include/gbmla.h declares; host-side argument checks
return their error codes before anything touches the device."""
from __future__ import annotations

import ctypes
import os
import re

import pytest

from paper_2607_27269_gb300 import abi

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "gbmla.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[a-z_]+\s*\*?\s*(mla_[a-z_0-9]+)\s*\(", src, flags=re.M)))


def test_header_declares_the_five_steps():
    names = declared_functions()
    for n in ("mla_cache_append", "mla_absorb_q", "mla_decode_attn", "mla_combine", "mla_out_proj",
              "mla_workspace_size", "mla_check_status", "mla_status_str"):
        assert n in names


def test_library_exports_every_declared_symbol():
    lib = abi.lib()
    for n in declared_functions():
        assert hasattr(lib, n), n
    assert set(abi.EXPORTS) <= set(declared_functions())


def test_status_strings():
    assert abi.status_name(0) == "MLA_OK"
    assert abi.status_name(4) == "MLA_ERR_DEVICE_BOUNDS"
    assert abi.status_name(5) == "MLA_ERR_DEVICE_TIMEOUT"
    assert abi.status_name(99) == "MLA_ERR_UNKNOWN"


def _dims(**kw):
    base = dict(num_heads=8, num_kv_groups=2, d_nope=64, d_rope=64, d_v=64, rank=512, hidden=0, sm_scale=0.1,
                rope_style=0, rope_base=10000.0)
    base.update(kw)
    return abi.Dims(**base)


@pytest.mark.parametrize("kw,code", [
    (dict(num_heads=6, num_kv_groups=4), abi.MLA_ERR_INVALID_ARG),   # H % G != 0
    (dict(sm_scale=0.0), abi.MLA_ERR_INVALID_ARG),
    (dict(rope_style=2), abi.MLA_ERR_INVALID_ARG),
    (dict(rope_base=1.0), abi.MLA_ERR_INVALID_ARG),
    (dict(d_rope=48), abi.MLA_ERR_UNSUPPORTED),
    (dict(rank=96), abi.MLA_ERR_UNSUPPORTED),
    (dict(rank=1024), abi.MLA_ERR_UNSUPPORTED),
    (dict(d_nope=12), abi.MLA_ERR_UNSUPPORTED),
])
def test_dims_are_checked_on_the_host(kw, code):
    L = abi.lib()
    d = _dims(**kw).c()
    ob = ctypes.c_size_t()
    assert L.mla_workspace_size(ctypes.byref(d), 4, 1, 128, 0, ctypes.byref(ob), None, None) == code
    assert L.mla_absorb_q(ctypes.byref(d), 4, 1, None, None, None, None, None, None) == code


def test_other_arguments_are_checked_on_the_host():
    L = abi.lib()
    d = _dims().c()
    # q_len out of range, max_kv_len < q_len, negative splits
    assert L.mla_workspace_size(ctypes.byref(d), 4, 0, 128, 0, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_workspace_size(ctypes.byref(d), 4, 17, 128, 0, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_workspace_size(ctypes.byref(d), 4, 5, 4, 0, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_workspace_size(ctypes.byref(d), 4, 1, 128, -1, None, None, None) == abi.MLA_ERR_INVALID_ARG
    # caches: NULL / misaligned pointers, bad strides, paged page size
    c = abi.MlaCache(None, None, 512, 64, 512 * 64, 64 * 64, None, 0, 0, 0, 64)
    assert L.mla_cache_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 16, 16, 16, None) == abi.MLA_ERR_INVALID_ARG
    c = abi.MlaCache(0x1008, 0x2000, 512, 64, 512 * 64, 64 * 64, None, 0, 0, 0, 64)
    assert L.mla_cache_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 16, 16, 16, None) == abi.MLA_ERR_INVALID_ARG
    c = abi.MlaCache(0x1000, 0x2000, 500, 64, 512 * 64, 64 * 64, None, 0, 0, 0, 64)
    assert L.mla_cache_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 16, 16, 16, None) == abi.MLA_ERR_INVALID_ARG
    c = abi.MlaCache(0x1000, 0x2000, 512, 64, 512 * 64, 64 * 64, 0x3000, 4, 32, 10, 128)
    assert L.mla_cache_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 16, 16, 16, None) == abi.MLA_ERR_UNSUPPORTED
    c = abi.MlaCache(0x1000, 0x2000, 512, 64, 512 * 64, 64 * 64, 0x3000, 1, 64, 10, 128)  # table too short
    assert L.mla_cache_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 16, 16, 16, None) == abi.MLA_ERR_INVALID_ARG
    # an empty batch is a valid no-op that never touches the device
    c = abi.MlaCache(0x1000, 0x2000, 512, 64, 512 * 64, 64 * 64, None, 0, 0, 0, 64)
    assert L.mla_cache_append(ctypes.byref(d), ctypes.byref(c), 0, 1, None, None, None, None) == abi.MLA_OK
    assert L.mla_absorb_q(ctypes.byref(d), 0, 1, None, None, None, None, None, None) == abi.MLA_OK
    assert L.mla_out_proj(ctypes.byref(d), 0, 1, None, None, None, None, None, None) == abi.MLA_OK
    # out_proj with W_O needs `out`
    dd = _dims(hidden=256).c()
    assert L.mla_out_proj(ctypes.byref(dd), 1, 1, 16, 16, 16, 16, None, None) == abi.MLA_ERR_INVALID_ARG


def test_projection_arguments_are_checked_on_the_host():
    L = abi.lib()
    c = abi.MlaCache(0x1000, 0x2000, 512, 64, 512 * 64, 64 * 64, None, 0, 0, 0, 64)
    # the projection needs the model width
    d0 = _dims(hidden=0).c()
    assert L.mla_project_append(ctypes.byref(d0), ctypes.byref(c), 1, 1, 16, 16, 16, None, 16, None, None,
                                None) == abi.MLA_ERR_INVALID_ARG
    d = _dims(hidden=256).c()
    dodd = _dims(hidden=252).c()                                    # row stride not a multiple of 16 bytes
    assert L.mla_project_append(ctypes.byref(dodd), ctypes.byref(c), 1, 1, 16, 16, 16, None, 16, None, None,
                                None) == abi.MLA_ERR_INVALID_ARG
    # missing or misaligned inputs; W_Q without query outputs
    assert L.mla_project_append(ctypes.byref(d), ctypes.byref(c), 1, 1, None, 16, 16, None, 16, None, None,
                                None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_project_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 24, 16, 16, None, 16, None, None,
                                None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_project_append(ctypes.byref(d), ctypes.byref(c), 1, 1, 16, 16, 16, 16, 16, None, None,
                                None) == abi.MLA_ERR_INVALID_ARG
    # an empty batch is a no-op
    assert L.mla_project_append(ctypes.byref(d), ctypes.byref(c), 0, 1, None, None, None, None, None, None, None,
                                None) == abi.MLA_OK


def test_acceptance_arguments_are_checked_on_the_host():
    L = abi.lib()
    assert L.mla_acceptance_stats(4, 0, 1, 16, 16, 16, None, None, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_acceptance_stats(4, 100, 2, 16, 16, 104, None, None, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_acceptance_stats(4, 100, 1, 16, 16, 99, None, None, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_acceptance_stats(4, 100, 1, 16, 16, 100, None, None, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_acceptance_stats(4, 100, 1, 24, 16, 104, None, None, None, None, None) == abi.MLA_ERR_INVALID_ARG
    assert L.mla_acceptance_stats(0, 100, 1, None, None, 104, None, None, None, None, None) == abi.MLA_OK


def test_decode_step_validates_every_stage_before_the_device():
    """mla_decode_step checks the arguments of all five stages before its
    first launch.  With no GPU present, a bad argument of any stage -- the
    last one's included (W_O given without `out`) -- comes back as
    MLA_ERR_INVALID_ARG, while a call whose arguments are all valid gets as
    far as the device and fails there; an empty batch is a no-op."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present: the all-valid call would launch on stand-in pointers")
    L = abi.lib()
    d = _dims(hidden=256).c()
    c = abi.MlaCache(0x1000, 0x2000, 512, 64, 512 * 64, 64 * 64, None, 0, 0, 0, 64)
    A = 0x10000  # 16-byte aligned stand-in for every buffer (never dereferenced: no device)

    def step(batch=2, q_len=1, c_new=A, kr_new=A, start_pos=A, max_kv=64, splits=4, q_abs=A, o_lat=A, out=A):
        return L.mla_decode_step(ctypes.byref(d), ctypes.byref(c), batch, q_len, c_new, kr_new, start_pos, A, A, A,
                                 max_kv, A, A, A, splits, q_abs, A, A, o_lat, A, A, out, None)

    assert step() == abi.MLA_ERR_CUDA
    assert step(batch=0) == abi.MLA_OK
    assert step(out=None) == abi.MLA_ERR_INVALID_ARG        # out_proj, the fifth stage
    assert step(o_lat=A + 4) == abi.MLA_ERR_INVALID_ARG     # combine / out_proj
    assert step(q_abs=None) == abi.MLA_ERR_INVALID_ARG      # absorption / attention
    assert step(splits=-1) == abi.MLA_ERR_INVALID_ARG       # attention
    assert step(c_new=A + 2) == abi.MLA_ERR_INVALID_ARG     # append, the first stage
    assert step(q_len=4, max_kv=2) == abi.MLA_ERR_INVALID_ARG
