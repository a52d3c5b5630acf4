"""ctypes front end of the fp64 MLA oracle (``mla_oracle.c``).

TEST INFRASTRUCTURE ONLY.  The tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference arm of ``bench.py`` may import this module; the
product package never does.  Inputs are numpy arrays: bf16 tensors are passed
as their ``uint16`` bit patterns and read exactly, outputs are float64.

Every function cites the passage of the paper it follows; the C file holds the
arithmetic and the readings of points the paper leaves open.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mla_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

ERRORS = {0: "ok", 1: "bad argument", 2: "bad position", 3: "bad page", 4: "no memory"}


class OracleError(RuntimeError):
    pass


class _Dims(ctypes.Structure):
    _fields_ = [
        ("num_heads", ctypes.c_int32),
        ("num_kv_groups", ctypes.c_int32),
        ("d_nope", ctypes.c_int32),
        ("d_rope", ctypes.c_int32),
        ("d_v", ctypes.c_int32),
        ("rank", ctypes.c_int32),
        ("hidden", ctypes.c_int32),
        ("sm_scale", ctypes.c_double),
        ("rope_style", ctypes.c_int32),
        ("rope_base", ctypes.c_double),
    ]


class _Cache(ctypes.Structure):
    _fields_ = [
        ("c_kv", ctypes.c_void_p),
        ("k_rope", ctypes.c_void_p),
        ("c_tok_stride", ctypes.c_int64),
        ("r_tok_stride", ctypes.c_int64),
        ("c_blk_stride", ctypes.c_int64),
        ("r_blk_stride", ctypes.c_int64),
        ("block_table", ctypes.c_void_p),
        ("bt_stride", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("capacity", ctypes.c_int32),
    ]


class _GqaDims(ctypes.Structure):
    _fields_ = [
        ("num_heads", ctypes.c_int32),
        ("num_kv_groups", ctypes.c_int32),
        ("d_k", ctypes.c_int32),
        ("d_v", ctypes.c_int32),
        ("sm_scale", ctypes.c_double),
        ("rope_style", ctypes.c_int32),
        ("rope_base", ctypes.c_double),
    ]


@dataclass
class GqaDims:
    """Shape of an original GQA layer (Sec. 3.1)."""
    num_heads: int
    num_kv_groups: int
    d_k: int
    d_v: int
    sm_scale: float
    rope_style: int = 0
    rope_base: float = 10000.0

    def _c(self) -> _GqaDims:
        return _GqaDims(self.num_heads, self.num_kv_groups, self.d_k, self.d_v, self.sm_scale, self.rope_style,
                        self.rope_base)


def build(force: bool = False) -> str:
    """Compile ``mla_oracle.c`` with gcc (fp64, OpenMP, no fast-math)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    tmp = _SO + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-Wall", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = configure(ctypes.CDLL(build()))
        return _lib


def compile_variant(src: str, out_so: str) -> str:
    """Compile an edited copy of the oracle source (used by the tests that
    plant mistakes in the oracle to show that the pins catch them)."""
    c_path = out_so[:-3] + ".c"
    with open(c_path, "w") as f:
        f.write(src)
    subprocess.run(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-o", out_so, c_path, "-lm"], check=True)
    return out_so


def source() -> str:
    with open(_SRC) as f:
        return f.read()


def configure(lib):
    """Declare the C signatures on a loaded oracle library."""
    vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    lib.orc_num_threads.restype = ctypes.c_int
    lib.orc_bf16_round.restype = ctypes.c_uint16
    lib.orc_bf16_round.argtypes = [dbl]
    lib.orc_bf16_value.restype = dbl
    lib.orc_bf16_value.argtypes = [ctypes.c_uint16]
    lib.orc_rope.restype = None
    lib.orc_rope.argtypes = [vp, vp, ctypes.c_int, i64, dbl, ctypes.c_int]
    lib.orc_cache_append.restype = ctypes.c_int
    lib.orc_cache_append.argtypes = [ctypes.POINTER(_Dims), ctypes.POINTER(_Cache), ctypes.c_int,
                                     ctypes.c_int, vp, vp, vp]
    lib.orc_absorb_q.restype = ctypes.c_int
    lib.orc_absorb_q.argtypes = [ctypes.POINTER(_Dims), ctypes.c_int, ctypes.c_int, vp, vp, vp, vp,
                                 vp, vp]
    lib.orc_project_append.restype = ctypes.c_int
    lib.orc_project_append.argtypes = [ctypes.POINTER(_Dims), ctypes.POINTER(_Cache), ctypes.c_int, ctypes.c_int,
                                       vp, vp, vp, vp, vp, vp, vp]
    lib.orc_acceptance.restype = ctypes.c_int
    lib.orc_acceptance.argtypes = [ctypes.c_int, ctypes.c_int, vp, vp, vp, vp, vp, vp]
    lib.orc_gqa_append.restype = ctypes.c_int
    lib.orc_gqa_append.argtypes = [ctypes.POINTER(_GqaDims), ctypes.POINTER(_Cache), ctypes.c_int, ctypes.c_int,
                                   vp, vp, vp]
    lib.orc_gqa_decode.restype = ctypes.c_int
    lib.orc_gqa_decode.argtypes = [ctypes.POINTER(_GqaDims), ctypes.POINTER(_Cache), ctypes.c_int, ctypes.c_int,
                                   vp, vp, vp, vp]
    lib.orc_e2e_loss.restype = ctypes.c_int
    lib.orc_e2e_loss.argtypes = [ctypes.c_int, ctypes.c_int, vp, vp, vp, vp]
    lib.orc_mla_decode.restype = ctypes.c_int
    lib.orc_mla_decode.argtypes = [ctypes.POINTER(_Dims), ctypes.POINTER(_Cache), ctypes.c_int,
                                   ctypes.c_int, vp, vp, vp, vp, vp, vp, vp, ctypes.c_int,
                                   vp, vp, vp, vp]
    return lib


@dataclass
class Dims:
    """MLA layer shape (Sec. 3.1-3.2 notation): H query heads in G KV groups,
    per-head widths d_nope / d_rope / d_v, latent rank r, model width D."""
    num_heads: int
    num_kv_groups: int
    d_nope: int
    d_rope: int
    d_v: int
    rank: int
    hidden: int = 0
    sm_scale: float = 1.0
    rope_style: int = 0
    rope_base: float = 10000.0

    def _c(self) -> _Dims:
        return _Dims(self.num_heads, self.num_kv_groups, self.d_nope, self.d_rope, self.d_v, self.rank,
                     self.hidden, float(self.sm_scale), self.rope_style, float(self.rope_base))


@dataclass
class Cache:
    """Latent cache c and rotated positional-key cache k_rope (Sec. 3.2), as
    bf16 bit patterns.  ``block_table`` None means one block per sequence."""
    c_kv: np.ndarray
    k_rope: np.ndarray
    c_tok_stride: int
    r_tok_stride: int
    c_blk_stride: int
    r_blk_stride: int
    capacity: int
    block_table: Optional[np.ndarray] = None
    page_size: int = 0
    num_pages: int = 0

    def _c(self) -> _Cache:
        assert self.c_kv.dtype == np.uint16 and self.k_rope.dtype == np.uint16
        assert self.c_kv.flags.c_contiguous and self.k_rope.flags.c_contiguous
        bt = None
        bt_stride = 0
        if self.block_table is not None:
            assert self.block_table.dtype == np.int32 and self.block_table.flags.c_contiguous
            bt = self.block_table.ctypes.data
            bt_stride = self.block_table.shape[-1]
        return _Cache(self.c_kv.ctypes.data, self.k_rope.ctypes.data, self.c_tok_stride,
                      self.r_tok_stride, self.c_blk_stride, self.r_blk_stride, bt, bt_stride,
                      self.page_size, self.num_pages, self.capacity)


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _u16(a: np.ndarray) -> np.ndarray:
    a = np.ascontiguousarray(a)
    assert a.dtype == np.uint16, a.dtype
    return a


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _check(code: int, what: str):
    if code != 0:
        raise OracleError(f"{what}: {ERRORS.get(code, code)}")


def num_threads() -> int:
    return _load().orc_num_threads()


def bf16_value(bits: int) -> float:
    return _load().orc_bf16_value(int(bits))


def bf16_round(x: float) -> int:
    """fp64 -> bf16 bit pattern, one rounding to nearest-even."""
    return int(_load().orc_bf16_round(float(x)))


def rope(x: np.ndarray, pos: int, base: float = 10000.0, style: int = 0) -> np.ndarray:
    """RoPE rotation R_pos (Sec. 3.1) of one vector, fp64."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty_like(x)
    _load().orc_rope(x.ctypes.data, y.ctypes.data, x.shape[-1], int(pos), float(base), int(style))
    return y


def cache_append(dims: Dims, cache: Cache, c_new: np.ndarray, kr_new: np.ndarray, start_pos) -> None:
    """Write n_new latent rows and rotated positional keys per sequence into
    ``cache`` in place (Sec. 3.2 latent cache; Sec. 3.1 rotation)."""
    c_new, kr_new, start_pos = _u16(c_new), _u16(kr_new), _i32(start_pos)
    batch, n_new = c_new.shape[0], c_new.shape[1]
    d, c = dims._c(), cache._c()
    _check(_load().orc_cache_append(ctypes.byref(d), ctypes.byref(c), batch, n_new, c_new.ctypes.data,
                                    kr_new.ctypes.data, start_pos.ctypes.data), "cache_append")


def project_append(dims: Dims, cache: Cache, h: np.ndarray, w_dkv: np.ndarray, w_kr: np.ndarray,
                   w_q: Optional[np.ndarray], start_pos):
    """Project hidden states h [B, n, D] into the cache and the queries
    (Sec. 3.2 latent c = W^DKV h with the rotated positional key R_pos W^KR h;
    Sec. 3.1 Eq. 1 q_i = W^Q_i h).  Writes the cache in place; returns
    (q_nope, q_pe) fp64 (None without ``w_q``)."""
    h, w_dkv, w_kr, start_pos = _u16(h), _u16(w_dkv), _u16(w_kr), _i32(start_pos)
    w_q = None if w_q is None else _u16(w_q)
    batch, n_new = h.shape[0], h.shape[1]
    q_nope = np.zeros((batch, n_new, dims.num_heads, dims.d_nope)) if w_q is not None else None
    q_pe = np.zeros((batch, n_new, dims.num_heads, dims.d_rope)) if w_q is not None else None
    d, c = dims._c(), cache._c()
    _check(_load().orc_project_append(ctypes.byref(d), ctypes.byref(c), batch, n_new, h.ctypes.data,
                                      w_dkv.ctypes.data, w_kr.ctypes.data, _ptr(w_q), start_pos.ctypes.data,
                                      _ptr(q_nope), _ptr(q_pe)), "project_append")
    return q_nope, q_pe


def absorb_q(dims: Dims, q_nope: np.ndarray, q_pe: np.ndarray, kv_len, w_uk: np.ndarray):
    """Latent query q_lat = W_UK[g]^T q_nope and rotated positional query
    (Sec. 1 absorbed projections; Sec. 3.2 Eq. 5).  Returns (q_lat, q_pe_rot)."""
    q_nope, q_pe, w_uk, kv_len = _u16(q_nope), _u16(q_pe), _u16(w_uk), _i32(kv_len)
    batch, q_len, H = q_nope.shape[:3]
    q_lat = np.zeros((batch, q_len, H, dims.rank))
    q_pe_rot = np.zeros((batch, q_len, H, dims.d_rope))
    d = dims._c()
    _check(_load().orc_absorb_q(ctypes.byref(d), batch, q_len, q_nope.ctypes.data, q_pe.ctypes.data,
                                kv_len.ctypes.data, w_uk.ctypes.data, q_lat.ctypes.data,
                                q_pe_rot.ctypes.data), "absorb_q")
    return q_lat, q_pe_rot


def mla_decode(dims: Dims, cache: Cache, q_nope: np.ndarray, q_pe: np.ndarray, kv_len,
               w_uk: np.ndarray, w_uv: np.ndarray, w_o: Optional[np.ndarray] = None,
               seqs=None) -> dict:
    """One MLA decode step in the plain non-absorbed form (Sec. 3.1 Eqs. 2-4,
    Sec. 3.2 Eq. 5, Sec. 3.3 score routing, Sec. 4.1 output projection).

    Returns float64 arrays ``o_lat`` [B,q,H,r], ``lse`` [B,q,H], ``o`` [B,q,H,d_v]
    and, with ``w_o``, ``out`` [B,q,D].  With ``seqs`` only those sequences are
    computed; the rows of the others are NaN."""
    q_nope, q_pe, kv_len = _u16(q_nope), _u16(q_pe), _i32(kv_len)
    w_uk, w_uv = _u16(w_uk), _u16(w_uv)
    w_o = None if w_o is None else _u16(w_o)
    batch, q_len, H = q_nope.shape[:3]
    o_lat = np.full((batch, q_len, H, dims.rank), np.nan)
    lse = np.full((batch, q_len, H), np.nan)
    o = np.full((batch, q_len, H, dims.d_v), np.nan)
    out = np.full((batch, q_len, dims.hidden), np.nan) if (w_o is not None and dims.hidden) else None
    seq_arr = None if seqs is None else _i32(seqs)
    d, c = dims._c(), cache._c()
    code = _load().orc_mla_decode(
        ctypes.byref(d), ctypes.byref(c), batch, q_len, kv_len.ctypes.data, q_nope.ctypes.data,
        q_pe.ctypes.data, w_uk.ctypes.data, w_uv.ctypes.data, _ptr(w_o), _ptr(seq_arr),
        0 if seq_arr is None else len(seq_arr), o_lat.ctypes.data, lse.ctypes.data, o.ctypes.data,
        _ptr(out))
    _check(code, "mla_decode")
    res = {"o_lat": o_lat, "lse": lse, "o": o}
    if out is not None:
        res["out"] = out
    return res


def acceptance(draft: np.ndarray, target: np.ndarray) -> dict:
    """Acceptance statistics of draft against target logits [rows, vocab]
    (Sec. 3.3: Eq. 9 alpha_sample = sum_y min(p_D, p_T), Eq. 10 greedy
    agreement of the argmaxes, lowest index on ties).  Logits are taken as
    given (fp64)."""
    draft = np.ascontiguousarray(draft, dtype=np.float64)
    target = np.ascontiguousarray(target, dtype=np.float64)
    rows, vocab = draft.shape
    alpha = np.zeros(rows)
    ad = np.zeros(rows, dtype=np.int32)
    at = np.zeros(rows, dtype=np.int32)
    gr = np.zeros(rows, dtype=np.int32)
    _check(_load().orc_acceptance(rows, vocab, draft.ctypes.data, target.ctypes.data, alpha.ctypes.data,
                                  ad.ctypes.data, at.ctypes.data, gr.ctypes.data), "acceptance")
    return {"alpha_sample": alpha, "argmax_draft": ad, "argmax_target": at, "greedy": gr}


def gqa_append(dims: GqaDims, cache: Cache, k_new: np.ndarray, v_new: np.ndarray, start_pos) -> None:
    """Original GQA cache append (Sec. 3.1): keys [B, n, G, d_k] rotated to
    their positions (one bf16 rounding), values [B, n, G, d_v] copied; the
    cache's c_kv holds values, k_rope keys, block (or table row) b * G + g."""
    k_new, v_new, start_pos = _u16(k_new), _u16(v_new), _i32(start_pos)
    batch, n_new = k_new.shape[0], k_new.shape[1]
    _check(_load().orc_gqa_append(ctypes.byref(dims._c()), ctypes.byref(cache._c()), batch, n_new,
                                  k_new.ctypes.data, v_new.ctypes.data, start_pos.ctypes.data), "gqa_append")


def gqa_decode(dims: GqaDims, cache: Cache, q: np.ndarray, kv_len) -> dict:
    """One decode step of the original GQA attention (Sec. 3.1 Eqs. 1-4):
    q [B, q_len, H, d_k] (not rotated) -> o [B, q_len, H, d_v], lse [B, q_len, H]."""
    q, kv_len = _u16(q), _i32(kv_len)
    batch, q_len = q.shape[:2]
    o = np.zeros((batch, q_len, dims.num_heads, dims.d_v))
    lse = np.zeros((batch, q_len, dims.num_heads))
    _check(_load().orc_gqa_decode(ctypes.byref(dims._c()), ctypes.byref(cache._c()), batch, q_len, kv_len.ctypes.data,
                                  q.ctypes.data, o.ctypes.data, lse.ctypes.data), "gqa_decode")
    return {"o": o, "lse": lse}


def e2e_loss(a_mla: np.ndarray, a_orig: np.ndarray, mask: Optional[np.ndarray] = None) -> float:
    """E2E functional-reconstruction loss forward (Sec. 4.1): masked MSE of the
    two blocks' post-W_O outputs [rows, D] (fp64), mask [rows] in {0, 1}."""
    a = np.ascontiguousarray(a_mla, dtype=np.float64).reshape(-1, a_mla.shape[-1])
    b = np.ascontiguousarray(a_orig, dtype=np.float64).reshape(-1, a_orig.shape[-1])
    m = None if mask is None else np.ascontiguousarray(mask, dtype=np.uint8).reshape(-1)
    out = np.zeros(1)
    _check(_load().orc_e2e_loss(a.shape[0], a.shape[1], a.ctypes.data, b.ctypes.data, _ptr(m), out.ctypes.data),
           "e2e_loss")
    return float(out[0])
