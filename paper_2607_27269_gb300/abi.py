"""ctypes binding of libgbmla.so (``include/gbmla.h``).

Argument marshalling only: every function here forwards torch tensors' device
pointers, sizes and the current CUDA stream to the C entry point of the same
name and raises ``MlaError`` on a non-OK status.  All compute happens in the
library's kernels.  PyTorch supplies device memory and streams.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass
from typing import Optional

import torch

from . import build as _build

MLA_OK, MLA_ERR_INVALID_ARG, MLA_ERR_UNSUPPORTED, MLA_ERR_CUDA, MLA_ERR_DEVICE_BOUNDS, MLA_ERR_DEVICE_TIMEOUT = range(6)
SPLIT_TILE = 128
EXPORTS = ("mla_workspace_size", "mla_cache_append", "mla_project_append", "mla_acceptance_stats",
           "mla_gqa_append", "mla_gqa_workspace_size", "mla_gqa_decode_attn", "mla_gqa_project", "mla_gqa_out_proj",
           "mla_e2e_loss", "mla_absorb_q", "mla_decode_attn", "mla_combine",
           "mla_out_proj", "mla_decode_step", "mla_check_status", "mla_selftest_wait_timeout",
           "mla_decode_attn_noalloc", "mla_reload_tuning", "mla_status_str", "mla_last_error")


class MlaError(RuntimeError):
    def __init__(self, where: str, code: int, name: str):
        super().__init__(f"{where}: {name}")
        self.code = code
        self.name = name


class MlaDims(ctypes.Structure):
    _fields_ = [("num_heads", ctypes.c_int32), ("num_kv_groups", ctypes.c_int32), ("d_nope", ctypes.c_int32),
                ("d_rope", ctypes.c_int32), ("d_v", ctypes.c_int32), ("rank", ctypes.c_int32),
                ("hidden", ctypes.c_int32), ("sm_scale", ctypes.c_float), ("rope_style", ctypes.c_int32),
                ("rope_base", ctypes.c_float)]


class MlaGqaDims(ctypes.Structure):
    _fields_ = [("num_heads", ctypes.c_int32), ("num_kv_groups", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("sm_scale", ctypes.c_float), ("rope_style", ctypes.c_int32), ("rope_base", ctypes.c_float)]


class MlaCache(ctypes.Structure):
    _fields_ = [("c_kv", ctypes.c_void_p), ("k_rope", ctypes.c_void_p), ("c_tok_stride", ctypes.c_int64),
                ("r_tok_stride", ctypes.c_int64), ("c_blk_stride", ctypes.c_int64), ("r_blk_stride", ctypes.c_int64),
                ("block_table", ctypes.c_void_p), ("bt_stride", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("num_pages", ctypes.c_int32), ("capacity", ctypes.c_int32)]


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def lib(auto_build: bool = True):
    """The loaded library (built first if missing or stale and ``auto_build``)."""
    global _lib
    with _lock:
        if _lib is None:
            # GBMLA_LIBRARY selects another build of the library
            path = os.environ.get("GBMLA_LIBRARY") or (_build.build() if auto_build else _build.LIB)
            if not os.path.exists(path):
                raise RuntimeError(f"libgbmla.so is missing at {path}; run paper_2607_27269_gb300.build.build()")
            L = ctypes.CDLL(path)
            vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
            P = ctypes.POINTER
            L.mla_status_str.restype = ctypes.c_char_p
            L.mla_status_str.argtypes = [ctypes.c_int]
            L.mla_workspace_size.argtypes = [P(MlaDims), i32, i32, i32, i32, P(sz), P(sz), P(i32)]
            L.mla_cache_append.argtypes = [P(MlaDims), P(MlaCache), i32, i32, vp, vp, vp, vp]
            L.mla_project_append.argtypes = [P(MlaDims), P(MlaCache), i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]
            L.mla_absorb_q.argtypes = [P(MlaDims), i32, i32, vp, vp, vp, vp, vp, vp]
            L.mla_acceptance_stats.argtypes = [i32, i32, i32, vp, vp, i64, vp, vp, vp, vp, vp]
            L.mla_gqa_append.argtypes = [P(MlaGqaDims), P(MlaCache), i32, i32, vp, vp, vp, vp]
            L.mla_gqa_project.argtypes = [P(MlaGqaDims), i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp]
            L.mla_gqa_out_proj.argtypes = [P(MlaGqaDims), i32, i32, i32, vp, vp, vp, vp]
            L.mla_e2e_loss.argtypes = [i32, i32, vp, vp, vp, vp, vp]
            L.mla_gqa_workspace_size.argtypes = [P(MlaGqaDims), i32, i32, i32, i32, P(sz), P(sz), P(i32)]
            L.mla_gqa_decode_attn.argtypes = [P(MlaGqaDims), P(MlaCache), i32, i32, vp, i32, vp, i32, vp, vp, vp, vp,
                                              vp]
            L.mla_decode_attn.argtypes = [P(MlaDims), P(MlaCache), i32, i32, vp, i32, vp, i32, vp, vp, vp]
            L.mla_combine.argtypes = [P(MlaDims), i32, i32, i32, vp, i32, vp, vp, vp, vp, vp]
            L.mla_out_proj.argtypes = [P(MlaDims), i32, i32, vp, vp, vp, vp, vp, vp]
            L.mla_decode_step.argtypes = [P(MlaDims), P(MlaCache), i32, i32, vp, vp, vp, vp, vp, vp, i32, vp, vp, vp,
                                          i32, vp, vp, vp, vp, vp, vp, vp, vp]
            L.mla_check_status.argtypes = [vp]
            L.mla_selftest_wait_timeout.argtypes = [i64, vp]
            L.mla_decode_attn_noalloc.argtypes = [P(MlaDims), P(MlaCache), i32, i32, vp, i32, vp, i32, vp, vp, vp]
            L.mla_last_error.restype = ctypes.c_char_p
            L.mla_last_error.argtypes = []
            for name in EXPORTS[:-3]:
                getattr(L, name).restype = ctypes.c_int
            L.mla_reload_tuning.restype = None
            L.mla_reload_tuning.argtypes = []
            _lib = L
        return _lib


def reload_tuning() -> None:
    """Re-read the GBMLA_* testing variables (mla_reload_tuning)."""
    lib().mla_reload_tuning()


def status_name(code: int) -> str:
    return lib().mla_status_str(code).decode()


def _check(where: str, code: int):
    if code != MLA_OK:
        name = status_name(code)
        if code == MLA_ERR_CUDA:
            name += f" ({lib().mla_last_error().decode()})"
        raise MlaError(where, code, name)


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _p(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("tensor must live on the GPU")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


@dataclass
class Dims:
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

    def c(self) -> MlaDims:
        return MlaDims(self.num_heads, self.num_kv_groups, self.d_nope, self.d_rope, self.d_v, self.rank,
                       self.hidden, self.sm_scale, self.rope_style, self.rope_base)


@dataclass
class Cache:
    """Device cache: ``c_kv`` [blocks, block_tokens, r] and ``k_rope``
    [blocks, block_tokens, d_rope] bf16 (or strided views of one fused
    buffer), blocks = sequences (contiguous) or pages (paged)."""
    c_kv: torch.Tensor
    k_rope: torch.Tensor
    capacity: int
    block_table: Optional[torch.Tensor] = None
    page_size: int = 0
    num_pages: int = 0

    def c(self) -> MlaCache:
        c, k = self.c_kv, self.k_rope
        for t in (c, k):
            if not t.is_cuda or t.dtype != torch.bfloat16 or t.dim() != 3 or t.stride(2) != 1:
                raise ValueError("cache tensors must be 3-d bf16 CUDA tensors with unit inner stride")
        bt = self.block_table
        return MlaCache(c.data_ptr(), k.data_ptr(), c.stride(1), k.stride(1), c.stride(0), k.stride(0),
                        _p(bt), 0 if bt is None else bt.shape[1], self.page_size, self.num_pages, self.capacity)


def workspace_size(dims: Dims, batch: int, q_len: int, max_kv_len: int, num_splits: int = 0):
    """(o_part_bytes, lse_part_bytes, num_splits_used)."""
    ob, lb, s = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_int32()
    _check("mla_workspace_size", lib().mla_workspace_size(ctypes.byref(dims.c()), batch, q_len, max_kv_len,
                                                          num_splits, ctypes.byref(ob), ctypes.byref(lb),
                                                          ctypes.byref(s)))
    return ob.value, lb.value, s.value


def cache_append(dims: Dims, cache: Cache, c_new: torch.Tensor, kr_new: torch.Tensor, start_pos: torch.Tensor,
                 stream=None):
    batch, n_new = c_new.shape[0], c_new.shape[1]
    _check("mla_cache_append", lib().mla_cache_append(ctypes.byref(dims.c()), ctypes.byref(cache.c()), batch, n_new,
                                                      _p(c_new), _p(kr_new), _p(start_pos), _stream(stream)))


def project_append(dims: Dims, cache: Cache, h: torch.Tensor, w_dkv: torch.Tensor, w_kr: torch.Tensor,
                   w_q: Optional[torch.Tensor], start_pos: torch.Tensor, q_nope: Optional[torch.Tensor] = None,
                   q_pe: Optional[torch.Tensor] = None, stream=None):
    """h [B, n, hidden] -> cache rows at start_pos + k and, with ``w_q``, the
    query parts q_nope [B, n, H, d_nope] / q_pe [B, n, H, d_rope]."""
    batch, n_new = h.shape[0], h.shape[1]
    _check("mla_project_append", lib().mla_project_append(ctypes.byref(dims.c()), ctypes.byref(cache.c()), batch,
                                                          n_new, _p(h), _p(w_dkv), _p(w_kr), _p(w_q),
                                                          _p(start_pos), _p(q_nope), _p(q_pe), _stream(stream)))


@dataclass
class GqaDims:
    """Shape of an original GQA layer (key and value width head_dim)."""
    num_heads: int
    num_kv_groups: int
    head_dim: int
    sm_scale: float
    rope_style: int = 0
    rope_base: float = 10000.0

    def c(self) -> MlaGqaDims:
        return MlaGqaDims(self.num_heads, self.num_kv_groups, self.head_dim, self.sm_scale, self.rope_style,
                          self.rope_base)


def gqa_append(dims: GqaDims, cache: Cache, k_new: torch.Tensor, v_new: torch.Tensor, start_pos: torch.Tensor,
               stream=None):
    """k_new / v_new [B, n, G, head_dim] into the GQA cache (keys in cache.k_rope, values in cache.c_kv)."""
    batch, n_new = k_new.shape[0], k_new.shape[1]
    _check("mla_gqa_append", lib().mla_gqa_append(ctypes.byref(dims.c()), ctypes.byref(cache.c()), batch, n_new,
                                                  _p(k_new), _p(v_new), _p(start_pos), _stream(stream)))


def gqa_workspace_size(dims: GqaDims, batch: int, q_len: int, max_kv_len: int, num_splits: int = 0):
    ob, lb, s = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_int32()
    _check("mla_gqa_workspace_size", lib().mla_gqa_workspace_size(ctypes.byref(dims.c()), batch, q_len, max_kv_len,
                                                                  num_splits, ctypes.byref(ob), ctypes.byref(lb),
                                                                  ctypes.byref(s)))
    return ob.value, lb.value, s.value


class GqaStep:
    """GQA decode attention with its partial buffers allocated once:
    o [B, q_len, H, head_dim] fp32, lse [B, q_len, H]."""

    def __init__(self, dims: GqaDims, cache: Cache, batch: int, q_len: int, max_kv_len: int, num_splits: int = 0):
        self.dims, self.cache, self.batch, self.q_len, self.max_kv_len = dims, cache, batch, q_len, max_kv_len
        dev = cache.c_kv.device
        ob, lb, self.num_splits = gqa_workspace_size(dims, batch, q_len, max_kv_len, num_splits)
        G, hpg, d = dims.num_kv_groups, dims.num_heads // dims.num_kv_groups, dims.head_dim
        self.o_part = torch.empty(max(ob // 4, 1), dtype=torch.float32, device=dev)
        self.lse_part = torch.empty(max(lb // 4, 1), dtype=torch.float32, device=dev)
        self.o = torch.empty(batch, q_len, dims.num_heads, d, dtype=torch.float32, device=dev)
        self.lse = torch.empty(batch, q_len, dims.num_heads, dtype=torch.float32, device=dev)

    def __call__(self, q: torch.Tensor, kv_len: torch.Tensor, stream=None):
        _check("mla_gqa_decode_attn", lib().mla_gqa_decode_attn(
            ctypes.byref(self.dims.c()), ctypes.byref(self.cache.c()), self.batch, self.q_len, _p(kv_len),
            self.max_kv_len, _p(q), self.num_splits, _p(self.o_part), _p(self.lse_part), _p(self.o), _p(self.lse),
            _stream(stream)))
        return self.o


def gqa_project(dims: GqaDims, h: torch.Tensor, w_q, w_k, w_v, q, k_new, v_new, stream=None):
    """q [B, n, H, d], k_new / v_new [B, n, G, d] = h [B, n, D] times W_Q^T, W_K^T, W_V^T (bf16)."""
    batch, n_new, hidden = h.shape
    _check("mla_gqa_project", lib().mla_gqa_project(ctypes.byref(dims.c()), batch, n_new, hidden, _p(h), _p(w_q),
                                                    _p(w_k), _p(w_v), _p(q), _p(k_new), _p(v_new), _stream(stream)))


def gqa_out_proj(dims: GqaDims, o: torch.Tensor, w_o: torch.Tensor, out: torch.Tensor, stream=None):
    """out [B, q, D] = W_O concat_h o (o fp32 [B, q, H, d])."""
    batch, q_len = o.shape[:2]
    _check("mla_gqa_out_proj", lib().mla_gqa_out_proj(ctypes.byref(dims.c()), batch, q_len, w_o.shape[0], _p(o),
                                                      _p(w_o), _p(out), _stream(stream)))


def e2e_loss(a_mla: torch.Tensor, a_orig: torch.Tensor, mask: Optional[torch.Tensor] = None,
             loss: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """E2E functional-reconstruction loss forward (masked MSE of the two blocks'
    post-W_O outputs, bf16 [.., D]); returns a one-element fp32 device tensor."""
    hidden = a_mla.shape[-1]
    rows = a_mla.numel() // hidden
    loss = torch.empty(1, dtype=torch.float32, device=a_mla.device) if loss is None else loss
    _check("mla_e2e_loss", lib().mla_e2e_loss(rows, hidden, _p(a_mla), _p(a_orig), _p(mask), _p(loss),
                                              _stream(stream)))
    return loss


class E2EForward:
    """Forward of the E2E functional-reconstruction loss (Sec. 4.1) on one
    chunk of calibration hidden states: the converted MLA layer (projection
    into its latent cache, absorbed attention, W_UV, W_O) and the original GQA
    layer (its projections, cache append, attention, the same frozen W_O) run
    on the same h, and their post-W_O outputs meet in the masked MSE.  Every
    buffer is allocated once here."""

    def __init__(self, mla_step: "DecodeStep", gqa_dims: GqaDims, gqa_cache: Cache, hidden: int):
        self.mla = mla_step
        b, q = mla_step.batch, mla_step.q_len
        dev = mla_step.q_abs.device
        self.gqa_dims = gqa_dims
        self.gqa = GqaStep(gqa_dims, gqa_cache, b, q, mla_step.max_kv_len)
        d, H, G = gqa_dims.head_dim, gqa_dims.num_heads, gqa_dims.num_kv_groups
        self.q = torch.empty(b, q, H, d, dtype=torch.bfloat16, device=dev)
        self.k_new = torch.empty(b, q, G, d, dtype=torch.bfloat16, device=dev)
        self.v_new = torch.empty(b, q, G, d, dtype=torch.bfloat16, device=dev)
        self.out_orig = torch.empty(b, q, hidden, dtype=torch.bfloat16, device=dev)
        self.loss = torch.empty(1, dtype=torch.float32, device=dev)

    def __call__(self, h, mla_w, gqa_w, w_o, start_pos, kv_len, mask=None, stream=None):
        """mla_w = (w_dkv, w_kr, w_q, w_uk, w_uv), gqa_w = (w_q, w_k, w_v); returns the loss tensor."""
        w_dkv, w_kr, w_qm, w_uk, w_uv = mla_w
        out_mla = self.mla.from_hidden(h, w_dkv, w_kr, w_qm, start_pos, kv_len, w_uk, w_uv, w_o, stream=stream)
        gqa_project(self.gqa_dims, h, *gqa_w, self.q, self.k_new, self.v_new, stream)
        gqa_append(self.gqa_dims, self.gqa.cache, self.k_new, self.v_new, start_pos, stream)
        o = self.gqa(self.q, kv_len, stream)
        gqa_out_proj(self.gqa_dims, o, w_o, self.out_orig, stream)
        return e2e_loss(out_mla, self.out_orig, mask, self.loss, stream)


def acceptance_stats(draft: torch.Tensor, target: torch.Tensor, alpha: Optional[torch.Tensor] = None,
                     argmax_draft: Optional[torch.Tensor] = None, argmax_target: Optional[torch.Tensor] = None,
                     greedy: Optional[torch.Tensor] = None, stream=None):
    """draft / target logits [rows, vocab] (fp32 or bf16, same dtype) -> the
    per-row overlap alpha_sample (fp32), the two argmaxes and greedy agreement
    (int32), written into the given device tensors (allocated if None)."""
    if draft.dtype != target.dtype or draft.dtype not in (torch.float32, torch.bfloat16) or draft.shape != target.shape:
        raise ValueError("draft and target logits must share a shape and be fp32 or bf16")
    rows, vocab = draft.shape
    if draft.stride() != target.stride() or draft.stride(1) != 1 or not draft.is_cuda or not target.is_cuda:
        raise ValueError("logits must be CUDA tensors with unit inner stride and equal row strides")
    row_stride = draft.stride(0) if rows > 1 else vocab
    dev = draft.device
    alpha = torch.empty(rows, dtype=torch.float32, device=dev) if alpha is None else alpha
    argmax_draft = torch.empty(rows, dtype=torch.int32, device=dev) if argmax_draft is None else argmax_draft
    argmax_target = torch.empty(rows, dtype=torch.int32, device=dev) if argmax_target is None else argmax_target
    greedy = torch.empty(rows, dtype=torch.int32, device=dev) if greedy is None else greedy
    _check("mla_acceptance_stats", lib().mla_acceptance_stats(rows, vocab, 0 if draft.dtype == torch.float32 else 1,
                                                              draft.data_ptr(), target.data_ptr(), row_stride,
                                                              _p(alpha),
                                                              _p(argmax_draft), _p(argmax_target), _p(greedy),
                                                              _stream(stream)))
    return alpha, argmax_draft, argmax_target, greedy


def absorb_q(dims: Dims, q_nope: torch.Tensor, q_pe: torch.Tensor, kv_len: torch.Tensor, w_uk: torch.Tensor,
             q_abs: torch.Tensor, stream=None):
    batch, q_len = q_nope.shape[0], q_nope.shape[1]
    _check("mla_absorb_q", lib().mla_absorb_q(ctypes.byref(dims.c()), batch, q_len, _p(q_nope), _p(q_pe),
                                              _p(kv_len), _p(w_uk), _p(q_abs), _stream(stream)))


def decode_attn(dims: Dims, cache: Cache, kv_len: torch.Tensor, max_kv_len: int, q_abs: torch.Tensor,
                o_part: torch.Tensor, lse_part: torch.Tensor, num_splits: int = 0, stream=None):
    batch, q_len = q_abs.shape[0], q_abs.shape[1]
    _check("mla_decode_attn", lib().mla_decode_attn(ctypes.byref(dims.c()), ctypes.byref(cache.c()), batch, q_len,
                                                    _p(kv_len), max_kv_len, _p(q_abs), num_splits, _p(o_part),
                                                    _p(lse_part), _stream(stream)))


def combine(dims: Dims, batch: int, q_len: int, kv_len: torch.Tensor, max_kv_len: int, o_part: torch.Tensor,
            lse_part: torch.Tensor, o_lat: torch.Tensor, lse: Optional[torch.Tensor] = None, num_splits: int = 0,
            stream=None):
    _check("mla_combine", lib().mla_combine(ctypes.byref(dims.c()), batch, q_len, num_splits, _p(kv_len), max_kv_len,
                                            _p(o_part), _p(lse_part), _p(o_lat), _p(lse), _stream(stream)))


def out_proj(dims: Dims, o_lat: torch.Tensor, w_uv: torch.Tensor, w_o: Optional[torch.Tensor], o: torch.Tensor,
             out: Optional[torch.Tensor], stream=None):
    batch, q_len = o_lat.shape[0], o_lat.shape[1]
    _check("mla_out_proj", lib().mla_out_proj(ctypes.byref(dims.c()), batch, q_len, _p(o_lat), _p(w_uv), _p(w_o),
                                              _p(o), _p(out), _stream(stream)))


def decode_attn_noalloc(dims: Dims, cache: Cache, kv_len: torch.Tensor, max_kv_len: int, q_abs: torch.Tensor,
                        o_lat: torch.Tensor, lse: Optional[torch.Tensor] = None, num_splits: int = 0, stream=None):
    """Attention core and combine with the library's static scratch (for callers
    that cannot allocate device memory): writes o_lat and lse directly."""
    batch, q_len = q_abs.shape[0], q_abs.shape[1]
    _check("mla_decode_attn_noalloc",
           lib().mla_decode_attn_noalloc(ctypes.byref(dims.c()), ctypes.byref(cache.c()), batch, q_len, _p(kv_len),
                                         max_kv_len, _p(q_abs), num_splits, _p(o_lat), _p(lse), _stream(stream)))


def check_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device status code."""
    return lib().mla_check_status(_stream(stream))


def selftest_wait_timeout(limit_ns: int, stream=None):
    _check("mla_selftest_wait_timeout", lib().mla_selftest_wait_timeout(int(limit_ns), _stream(stream)))


class DecodeStep:
    """One decode step of an MLA layer (mla_decode_step: the five entry points
    in one call), with every intermediate buffer allocated once (by PyTorch)
    up front: append -> absorb -> split-KV attention -> combine -> up/out
    projection (or, through ``from_hidden``, projection -> absorb -> ...).

    ``graph=True`` replays the step as a CUDA graph: the first call with a
    given set of input tensors (their addresses) runs the step once and
    captures it, later calls with the same tensors replay the capture, on the
    current stream (or ``stream``, a ``torch.cuda.Stream``).  A serving loop
    that refills fixed input buffers pays one graph launch per step instead of
    the launches of every kernel."""

    def __init__(self, dims: Dims, cache: Cache, batch: int, q_len: int, max_kv_len: int, num_splits: int = 0,
                 device=None, graph: bool = False):
        self.graph = graph
        self._graphs = {}
        self.dims, self.cache = dims, cache
        self.batch, self.q_len, self.max_kv_len = batch, q_len, max_kv_len
        dev = device or cache.c_kv.device
        ob, lb, s = workspace_size(dims, batch, q_len, max_kv_len, num_splits)
        self.num_splits = s
        H, r, dr = dims.num_heads, dims.rank, dims.d_rope
        slots = max(ob // 4 // max(q_len * H * r, 1), 1)
        self.q_abs = torch.empty(batch, q_len, H, r + dr, dtype=torch.bfloat16, device=dev)
        self.o_part = torch.empty(slots, q_len, H, r, dtype=torch.float32, device=dev)
        self.lse_part = torch.empty(slots, q_len, H, dtype=torch.float32, device=dev)
        self.o_lat = torch.empty(batch, q_len, H, r, dtype=torch.float32, device=dev)
        self.lse = torch.empty(batch, q_len, H, dtype=torch.float32, device=dev)
        self.o = torch.empty(batch, q_len, H, dims.d_v, dtype=torch.bfloat16, device=dev)
        self.out = (torch.empty(batch, q_len, dims.hidden, dtype=torch.bfloat16, device=dev)
                    if dims.hidden else None)

    def __call__(self, q_nope, q_pe, kv_len, w_uk, w_uv, w_o=None, c_new=None, kr_new=None, start_pos=None,
                 stream=None):
        args = (q_nope, q_pe, kv_len, w_uk, w_uv, w_o, c_new, kr_new, start_pos)
        if not self.graph:
            return self._launch(*args, stream=stream)
        if stream is not None and not isinstance(stream, torch.cuda.Stream):
            raise ValueError("graph mode takes a torch.cuda.Stream (or None)")
        key = tuple(0 if t is None else t.data_ptr() for t in args)
        entry = self._graphs.get(key)
        if entry is None:
            self._launch(*args, stream=stream)  # the library's per-device set-up runs outside the capture
            g = torch.cuda.CUDAGraph()
            side = torch.cuda.Stream()
            side.wait_stream(stream or torch.cuda.current_stream())
            with torch.cuda.graph(g, stream=side):
                self._launch(*args)
            (stream or torch.cuda.current_stream()).wait_stream(side)
            entry = self._graphs[key] = (g, args)  # the tensors stay referenced while the graph lives
        if stream is None:
            entry[0].replay()
        else:
            with torch.cuda.stream(stream):
                entry[0].replay()
        return self.out if (self.dims.hidden and w_o is not None) else self.o

    def _launch(self, q_nope, q_pe, kv_len, w_uk, w_uv, w_o=None, c_new=None, kr_new=None, start_pos=None,
                stream=None):
        # the layer's descriptors and the step's own buffers are fixed: marshal
        # them once, so that a step costs the five library calls and little else
        if getattr(self, "_fixed", None) is None:
            self._structs = (self.dims.c(), self.cache.c())  # kept alive for the references below
            self._fixed = (ctypes.byref(self._structs[0]), ctypes.byref(self._structs[1]), self.q_abs.data_ptr(),
                           self.o_part.data_ptr(), self.lse_part.data_ptr(), self.o_lat.data_ptr(),
                           self.lse.data_ptr(), self.o.data_ptr(),
                           self.out.data_ptr() if self.out is not None else None)
        dims, cache, qa, op, lp, ol, ls, o, out = self._fixed
        d, L, sp = self.dims, lib(), _stream(stream)
        if c_new is not None and c_new.shape[1] != self.q_len:
            raise ValueError("c_new must hold q_len new entries per sequence")
        with_o = d.hidden and w_o is not None
        # the whole step in one library call (append, absorption, attention, combine, projections)
        _check("mla_decode_step", L.mla_decode_step(dims, cache, self.batch, self.q_len, _p(c_new), _p(kr_new),
                                                    _p(start_pos), _p(q_nope), _p(q_pe), _p(kv_len), self.max_kv_len,
                                                    _p(w_uk), _p(w_uv), _p(w_o) if with_o else None,
                                                    self.num_splits, qa, op, lp, ol, ls, o,
                                                    out if with_o else None, sp))
        return self.out if with_o else self.o

    def from_hidden(self, h, w_dkv, w_kr, w_q, start_pos, kv_len, w_uk, w_uv, w_o=None, stream=None):
        """The step fed by hidden states h [B, q_len, hidden]: the projection
        writes the cache rows and the queries (kept in ``self.q_nope`` /
        ``self.q_pe``), then absorption, attention, combine and projections."""
        d = self.dims
        if getattr(self, "q_nope", None) is None:
            dev = h.device
            self.q_nope = torch.empty(self.batch, self.q_len, d.num_heads, d.d_nope, dtype=torch.bfloat16, device=dev)
            self.q_pe = torch.empty(self.batch, self.q_len, d.num_heads, d.d_rope, dtype=torch.bfloat16, device=dev)
        project_append(d, self.cache, h, w_dkv, w_kr, w_q, start_pos, self.q_nope, self.q_pe, stream)
        return self(self.q_nope, self.q_pe, kv_len, w_uk, w_uv, w_o, stream=stream)


@dataclass
class DeviceWorkload:
    """A workload's tensors on the GPU plus its Dims and Cache descriptors."""
    dims: Dims
    cache: Cache
    batch: int
    q_len: int
    max_kv_len: int
    kv_len: torch.Tensor
    start_pos: torch.Tensor
    w_uk: torch.Tensor
    w_uv: torch.Tensor
    w_o: Optional[torch.Tensor]
    q_nope: torch.Tensor
    q_pe: torch.Tensor
    c_new: torch.Tensor
    kr_new: torch.Tensor


def to_device(w, device="cuda") -> DeviceWorkload:
    """Copy a ``workloads.Workload`` to the GPU (plain host-to-device copies)."""
    s = w.shape
    dims = Dims(s.num_heads, s.num_kv_groups, s.d_nope, s.d_rope, s.d_v, s.rank, s.hidden, s.sm_scale,
                s.rope_style, s.rope_base)
    put = lambda t: None if t is None else t.to(device)
    bt = put(w.block_table)
    cache = Cache(put(w.c_kv), put(w.k_rope), w.capacity, bt, s.page_size if s.paged else 0, w.num_pages)
    batch, q_len = w.kv_len.numel(), w.q_nope.shape[1]
    return DeviceWorkload(dims, cache, batch, q_len, int(w.kv_len.max()) if batch else q_len, put(w.kv_len),
                          put(w.start_pos), put(w.w_uk), put(w.w_uv), put(w.w_o), put(w.q_nope), put(w.q_pe),
                          put(w.c_new), put(w.kr_new))
