"""Python binding of libism (ctypes).  Argument marshalling only: every step
of the attention path runs in the library's CUDA kernels.  PyTorch supplies
device memory (outputs and workspaces) and the current CUDA stream.

There is no fallback: if libism.so is missing or a call fails, an exception
is raised.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass
from typing import Optional

import numpy as np
import torch

from . import build as _build

ISM_BF16, ISM_FP32, ISM_E4M3 = 0, 1, 2
QUERY, ANSWER = 0, 1
TILE_EMPTY, TILE_FULL, TILE_PARTIAL = 0, 1, 2

_STATUS = {0: "ISM_OK", 1: "ISM_ERR_INVALID_ARG", 2: "ISM_ERR_UNSUPPORTED", 3: "ISM_ERR_CUDA",
           4: "ISM_ERR_TIMEOUT", 5: "ISM_ERR_WORKSPACE"}


class IsmError(RuntimeError):
    def __init__(self, code: int, where: str, detail: str):
        super().__init__(f"{where}: {_STATUS.get(code, code)}: {detail}")
        self.code = code


class _Segments(C.Structure):
    _fields_ = [("num_seqs", C.c_int32), ("num_segs", C.c_int32),
                ("cu_seqlens", C.c_void_p), ("cu_seqlens_host", C.c_void_p),
                ("cu_segs", C.c_void_p), ("cu_segs_host", C.c_void_p),
                ("seg_end", C.c_void_p), ("seg_end_host", C.c_void_p),
                ("seg_type", C.c_void_p), ("seg_type_host", C.c_void_p)]


class _Rope(C.Structure):
    _fields_ = [("cos", C.c_void_p), ("sin", C.c_void_p), ("rows", C.c_int32)]


class _Shape(C.Structure):
    _fields_ = [("num_heads_q", C.c_int32), ("num_heads_kv", C.c_int32), ("head_dim", C.c_int32),
                ("dtype", C.c_int32), ("softmax_scale", C.c_float)]


class _PlanInfo(C.Structure):
    _fields_ = [("fingerprint", C.c_uint64), ("bytes", C.c_size_t)]


EXPORTS = {
    "ism_tile_map_size": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p]),
    "ism_build_tile_map": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32] + [C.c_void_p] * 6),
    "ism_attn_fwd_workspace_size": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "ism_attn_fwd": (C.c_int, [C.c_void_p] * 8 + [C.c_size_t, C.c_void_p]),
    "ism_attn_fwd_e4m3": (C.c_int, [C.c_void_p] * 5 + [C.c_float] * 3 + [C.c_void_p] * 3 + [C.c_size_t, C.c_void_p]),
    "ism_attn_bwd_workspace_size": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "ism_attn_bwd_workspace_size_min": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "ism_attn_bwd": (C.c_int, [C.c_void_p] * 12 + [C.c_size_t, C.c_void_p]),
    "ism_attn_fwd_rope": (C.c_int, [C.c_void_p] * 11 + [C.c_size_t, C.c_void_p]),
    "ism_attn_bwd_rope": (C.c_int, [C.c_void_p] * 13 + [C.c_size_t, C.c_void_p]),
    "ism_attn_prefill_append_workspace_size": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_void_p]),
    "ism_attn_prefill_append": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                          C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_int64,
                                          C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                          C.c_size_t, C.c_void_p]),
    "ism_attn_prefill_append_e4m3": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                               C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_int64,
                                               C.c_void_p, C.c_void_p, C.c_float, C.c_float, C.c_float, C.c_void_p,
                                               C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "ism_attn_prefill_append_paged": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                                C.c_int32, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p,
                                                C.c_int32, C.c_int32, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                                C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t,
                                                C.c_void_p]),
    "ism_attn_prefill_append_rope_workspace_size": (C.c_int, [C.c_void_p, C.c_int32, C.c_int32, C.c_void_p]),
    "ism_attn_prefill_append_rope": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                               C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_int64,
                                               C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                               C.c_void_p, C.c_size_t, C.c_void_p]),
    "ism_attn_prefill_append_paged_rope": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                                     C.c_int32, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                                     C.c_void_p, C.c_int32, C.c_int32, C.c_void_p, C.c_void_p,
                                                     C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                                     C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]),
    "ism_attn_prefill_append_e4m3_rope": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                                    C.c_int32, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p,
                                                    C.c_void_p, C.c_int64, C.c_void_p, C.c_void_p, C.c_float,
                                                    C.c_float, C.c_float, C.c_void_p, C.c_void_p, C.c_void_p,
                                                    C.c_void_p, C.c_size_t, C.c_void_p]),
    "ism_check_status": (C.c_int, [C.c_void_p]),
    "ism_debug_timeout_probe": (C.c_int, [C.c_uint32, C.c_void_p]),
    "ism_status_string": (C.c_char_p, [C.c_int]),
    "ism_last_error": (C.c_char_p, []),
    "ism_has_tensor_cores": (C.c_int32, []),
    "ism_set_kernel_timer": (C.c_int, [C.c_int32, C.c_void_p, C.c_void_p]),
    "ism_kernel_launches": (C.c_uint64, []),
    "ism_debug_reload_env": (None, []),
    "ism_debug_mma_tile": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p]),
    "ism_debug_mma_tile_e4m3": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32, C.c_void_p]),
    "ism_attn_fwd_noalloc_max_workspace": (C.c_size_t, []),
    "ism_attn_fwd_noalloc": (C.c_int, [C.c_void_p] * 8),
    "ism_attn_plan_size": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "ism_attn_plan_build": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p, C.c_void_p]),
    "ism_attn_fwd_planned": (C.c_int, [C.c_void_p] * 10),
    "ism_attn_bwd_planned": (C.c_int, [C.c_void_p] * 14 + [C.c_size_t, C.c_void_p]),
    "ism_attn_fwd_rope_planned": (C.c_int, [C.c_void_p] * 13),
    "ism_attn_bwd_rope_planned": (C.c_int, [C.c_void_p] * 15 + [C.c_size_t, C.c_void_p]),
}

KERNEL_FWD, KERNEL_BWD_DKDV, KERNEL_BWD_DQ, KERNEL_BWD_PRE, KERNEL_DECODE, KERNEL_META, KERNEL_ROPE = 1, 2, 3, 4, 5, 6, 7

_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False):
    """Load libism.so (building it first when asked)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise RuntimeError(f"libism.so not built ({path}); run __graft_entry__.build()")
        _build.build()
    lib = C.CDLL(path)
    for name, (res, args) in EXPORTS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(code: int, where: str):
    if code != 0:
        raise IsmError(code, where, load().ism_last_error().decode())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(device=None):
    return C.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return ISM_BF16
    if t.dtype == torch.float32:
        return ISM_FP32
    if t.dtype == torch.float8_e4m3fn:
        return ISM_E4M3
    raise TypeError(f"unsupported dtype {t.dtype}")


def _workspace(nbytes: int, device) -> torch.Tensor:
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
    off = (-ws.data_ptr()) % 256
    return ws[off:off + nbytes] if nbytes else ws[off:off]


@dataclass
class Segments:
    """Varlen turn boundaries in both device and host form (the host mirrors
    are used for validation and sizing without a device synchronisation)."""
    cu_seqlens: torch.Tensor
    cu_segs: torch.Tensor
    seg_end: torch.Tensor
    seg_type: torch.Tensor
    cu_seqlens_host: np.ndarray
    cu_segs_host: np.ndarray
    seg_end_host: np.ndarray
    seg_type_host: np.ndarray

    @staticmethod
    def from_numpy(cu_seqlens, cu_segs, seg_end, seg_type, device="cuda") -> "Segments":
        h = [np.ascontiguousarray(cu_seqlens, dtype=np.int32), np.ascontiguousarray(cu_segs, dtype=np.int32),
             np.ascontiguousarray(seg_end, dtype=np.int32), np.ascontiguousarray(seg_type, dtype=np.uint8)]
        d = [torch.from_numpy(x.copy()).to(device) for x in h]
        return Segments(*d, *h)

    @staticmethod
    def from_workload(segs, device="cuda") -> "Segments":
        return Segments.from_numpy(segs.cu_seqlens, segs.cu_segs, segs.seg_end, segs.seg_type, device)

    @property
    def total_tokens(self) -> int:
        return int(self.cu_seqlens_host[-1])

    def struct(self) -> _Segments:
        s = _Segments()
        s.num_seqs = self.cu_seqlens_host.shape[0] - 1
        s.num_segs = self.seg_end_host.shape[0]
        s.cu_seqlens, s.cu_seqlens_host = self.cu_seqlens.data_ptr(), self.cu_seqlens_host.ctypes.data
        s.cu_segs, s.cu_segs_host = self.cu_segs.data_ptr(), self.cu_segs_host.ctypes.data
        s.seg_end, s.seg_end_host = self.seg_end.data_ptr(), self.seg_end_host.ctypes.data
        s.seg_type, s.seg_type_host = self.seg_type.data_ptr(), self.seg_type_host.ctypes.data
        return s


def _shape(q: torch.Tensor, k: torch.Tensor, scale: float) -> _Shape:
    sh = _Shape()
    sh.num_heads_q, sh.head_dim = q.shape[-2], q.shape[-1]
    sh.num_heads_kv = k.shape[-2]
    sh.dtype = _dtype_code(q)
    sh.softmax_scale = float(scale)
    return sh


def _contig(*ts):
    for t in ts:
        if t is not None and not t.is_contiguous():
            raise ValueError("tensors must be contiguous")


def tile_map(segs: Segments, bm: int = 128, bn: int = 128):
    """Tile map of the segments (device tensors): tile_class, kt_full_end,
    kt_end, qt_begin, kv_end."""
    lib = load()
    s = segs.struct()
    nt, nq, nk = C.c_int64(), C.c_int64(), C.c_int64()
    _check(lib.ism_tile_map_size(C.byref(s), bm, bn, C.byref(nt), C.byref(nq), C.byref(nk)), "ism_tile_map_size")
    dev = segs.cu_seqlens.device
    out = {
        "tile_class": torch.empty(nt.value, dtype=torch.uint8, device=dev),
        "kt_full_end": torch.empty(nq.value, dtype=torch.int32, device=dev),
        "kt_end": torch.empty(nq.value, dtype=torch.int32, device=dev),
        "qt_begin": torch.empty(nk.value, dtype=torch.int32, device=dev),
        "kv_end": torch.empty(segs.total_tokens, dtype=torch.int32, device=dev),
    }
    _check(lib.ism_build_tile_map(C.byref(s), bm, bn, _ptr(out["tile_class"]), _ptr(out["kt_full_end"]),
                                  _ptr(out["kt_end"]), _ptr(out["qt_begin"]), _ptr(out["kv_end"]), _stream(dev)),
           "ism_build_tile_map")
    return out


class Plan:
    """The metadata of one batch of segments (ism_attn_plan_build) for the
    forward and backward of every layer over those segments and head counts:
    built once, passed to fwd / bwd as plan=.  Holds its device buffer."""

    def __init__(self, segs: Segments, num_heads_q: int, num_heads_kv: int, head_dim: int = 128,
                 dtype: torch.dtype = torch.bfloat16, device="cuda"):
        lib = load()
        self.segs = segs
        probe = torch.empty((0, num_heads_q, head_dim), dtype=dtype)
        self._shape = _shape(probe, torch.empty((0, num_heads_kv, head_dim), dtype=dtype), 1.0)
        n = C.c_size_t()
        _check(lib.ism_attn_plan_size(C.byref(segs.struct()), C.byref(self._shape), C.byref(n)), "ism_attn_plan_size")
        self.buffer = _workspace(n.value, device)
        self.info = _PlanInfo()
        self.build()

    def build(self):
        """Run the metadata pass into the plan (on the current stream)."""
        lib = load()
        _check(lib.ism_attn_plan_build(C.byref(self.segs.struct()), C.byref(self._shape), _ptr(self.buffer),
                                       self.buffer.numel(), C.byref(self.info), _stream(self.buffer.device)),
               "ism_attn_plan_build")
        return self


def fwd(segs: Segments, q, k, v, softmax_scale: float, out=None, lse=None, workspace=None, plan: Plan = None):
    """Forward over packed dialogues.  q [T,Hq,D], k/v [T,Hkv,D] -> (o, lse [Hq,T]).
    With a plan of these segments the metadata pass is not run again (and no
    workspace is needed)."""
    lib = load()
    _contig(q, k, v)
    T, hq, D = q.shape
    s, sh = segs.struct(), _shape(q, k, softmax_scale)
    if plan is not None:
        if out is None:
            out = torch.empty_like(q)
        if lse is None:
            lse = torch.empty((hq, T), dtype=torch.float32, device=q.device)
        _check(lib.ism_attn_fwd_planned(C.byref(s), C.byref(sh), _ptr(plan.buffer), C.byref(plan.info), _ptr(q),
                                        _ptr(k), _ptr(v), _ptr(out), _ptr(lse), _stream(q.device)),
               "ism_attn_fwd_planned")
        return out, lse
    nbytes = C.c_size_t()
    _check(lib.ism_attn_fwd_workspace_size(C.byref(s), C.byref(sh), C.byref(nbytes)), "ism_attn_fwd_workspace_size")
    if out is None:
        out = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((hq, T), dtype=torch.float32, device=q.device)
    if workspace is None or workspace.numel() < nbytes.value:
        workspace = _workspace(nbytes.value, q.device)
    _check(lib.ism_attn_fwd(C.byref(s), C.byref(sh), _ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(lse),
                            _ptr(workspace), workspace.numel(), _stream(q.device)), "ism_attn_fwd")
    return out, lse


def fwd_e4m3(segs: Segments, q, k, v, q_descale: float, k_descale: float, v_descale: float, softmax_scale: float,
             out=None, lse=None, workspace=None):
    """Forward with e4m3 inputs (torch.float8_e4m3fn; head_dim 128): the
    attention of q * q_descale, k * k_descale, v * v_descale.  Returns
    (o bf16 [T,Hq,D], lse [Hq,T])."""
    lib = load()
    _contig(q, k, v)
    T, hq, D = q.shape
    s, sh = segs.struct(), _shape(q, k, softmax_scale)
    nbytes = C.c_size_t()
    _check(lib.ism_attn_fwd_workspace_size(C.byref(s), C.byref(sh), C.byref(nbytes)), "ism_attn_fwd_workspace_size")
    if out is None:
        out = torch.empty(q.shape, dtype=torch.bfloat16, device=q.device)
    if lse is None:
        lse = torch.empty((hq, T), dtype=torch.float32, device=q.device)
    if workspace is None or workspace.numel() < nbytes.value:
        workspace = _workspace(nbytes.value, q.device)
    _check(lib.ism_attn_fwd_e4m3(C.byref(s), C.byref(sh), _ptr(q), _ptr(k), _ptr(v), q_descale, k_descale, v_descale,
                                 _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(), _stream(q.device)),
           "ism_attn_fwd_e4m3")
    return out, lse


def fwd_rope(segs: Segments, q, k, v, rope_cos, rope_sin, softmax_scale: float, q_rot=None, k_rot=None, out=None,
             lse=None, workspace=None, plan: "Plan" = None):
    """Forward with rotary encoding: q [T,Hq,D] and k [T,Hkv,D] (unrotated)
    are rotated at their positions inside their sequences (tables rope_cos /
    rope_sin float32 [rows, D/2]) into q_rot / k_rot, then attended.
    Returns (o, lse, q_rot, k_rot); the backward takes q_rot and k_rot."""
    lib = load()
    _contig(q, k, v)
    T, hq, D = q.shape
    s, sh = segs.struct(), _shape(q, k, softmax_scale)
    rope = _rope_struct(rope_cos, rope_sin)
    nbytes = C.c_size_t()
    _check(lib.ism_attn_fwd_workspace_size(C.byref(s), C.byref(sh), C.byref(nbytes)), "ism_attn_fwd_workspace_size")
    q_rot = torch.empty_like(q) if q_rot is None else q_rot
    k_rot = torch.empty_like(k) if k_rot is None else k_rot
    out = torch.empty_like(q) if out is None else out
    lse = torch.empty((hq, T), dtype=torch.float32, device=q.device) if lse is None else lse
    if plan is not None:  # the plan's metadata instead of a metadata pass
        _check(lib.ism_attn_fwd_rope_planned(C.byref(s), C.byref(sh), _ptr(plan.buffer), C.byref(plan.info),
                                             _ptr(q), _ptr(k), _ptr(v), C.byref(rope), _ptr(q_rot), _ptr(k_rot),
                                             _ptr(out), _ptr(lse), _stream(q.device)), "ism_attn_fwd_rope_planned")
        return out, lse, q_rot, k_rot
    if workspace is None or workspace.numel() < nbytes.value:
        workspace = _workspace(nbytes.value, q.device)
    _check(lib.ism_attn_fwd_rope(C.byref(s), C.byref(sh), _ptr(q), _ptr(k), _ptr(v), C.byref(rope), _ptr(q_rot),
                                 _ptr(k_rot), _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(),
                                 _stream(q.device)), "ism_attn_fwd_rope")
    return out, lse, q_rot, k_rot


def bwd_rope(segs: Segments, q_rot, k_rot, v, o, lse, dout, rope_cos, rope_sin, softmax_scale: float, dq=None,
             dk=None, dv=None, workspace=None, minimal_workspace: bool = False, plan: "Plan" = None):
    """Backward of ``fwd_rope``: takes the rotated q_rot / k_rot the forward
    wrote and returns (dq, dk, dv) with dq, dk the gradients of the UNROTATED
    queries and keys.  Workspace as for ``bwd``."""
    lib = load()
    _contig(q_rot, k_rot, v, o, lse, dout)
    s, sh = segs.struct(), _shape(q_rot, k_rot, softmax_scale)
    rope = _rope_struct(rope_cos, rope_sin)
    full, low = C.c_size_t(), C.c_size_t()
    _check(lib.ism_attn_bwd_workspace_size(C.byref(s), C.byref(sh), C.byref(full)), "ism_attn_bwd_workspace_size")
    _check(lib.ism_attn_bwd_workspace_size_min(C.byref(s), C.byref(sh), C.byref(low)),
           "ism_attn_bwd_workspace_size_min")
    dq = torch.empty_like(q_rot) if dq is None else dq
    dk = torch.empty_like(k_rot) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    if workspace is None or workspace.numel() < low.value:
        workspace = _workspace(low.value if minimal_workspace else full.value, q_rot.device)
    if plan is not None:  # the plan's metadata instead of a metadata pass
        _check(lib.ism_attn_bwd_rope_planned(C.byref(s), C.byref(sh), _ptr(plan.buffer), C.byref(plan.info),
                                             _ptr(q_rot), _ptr(k_rot), _ptr(v), _ptr(o), _ptr(lse), _ptr(dout),
                                             C.byref(rope), _ptr(dq), _ptr(dk), _ptr(dv), _ptr(workspace),
                                             workspace.numel(), _stream(q_rot.device)), "ism_attn_bwd_rope_planned")
        return dq, dk, dv
    _check(lib.ism_attn_bwd_rope(C.byref(s), C.byref(sh), _ptr(q_rot), _ptr(k_rot), _ptr(v), _ptr(o), _ptr(lse),
                                 _ptr(dout), C.byref(rope), _ptr(dq), _ptr(dk), _ptr(dv), _ptr(workspace),
                                 workspace.numel(), _stream(q_rot.device)), "ism_attn_bwd_rope")
    return dq, dk, dv


def bwd_workspace_size(segs: Segments, q, k, softmax_scale: float, minimal: bool = False) -> int:
    """Workspace bytes of the backward: the stored-dS schedule's size where
    it applies (else the minimum), or the minimum with minimal=True."""
    lib = load()
    s, sh = segs.struct(), _shape(q, k, softmax_scale)
    nbytes = C.c_size_t()
    fn = "ism_attn_bwd_workspace_size_min" if minimal else "ism_attn_bwd_workspace_size"
    _check(getattr(lib, fn)(C.byref(s), C.byref(sh), C.byref(nbytes)), fn)
    return nbytes.value


def bwd(segs: Segments, q, k, v, o, lse, dout, softmax_scale: float, dq=None, dk=None, dv=None, workspace=None,
        minimal_workspace: bool = False, plan: Plan = None):
    """Backward: (dq, dk, dv) of sum(O * dout).  The library takes the
    stored-dS schedule when the workspace is large enough for it, else the
    recompute schedule.  A given workspace is used as it is (it must hold at
    least the minimum); without one, a workspace of the stored-dS size is
    allocated (the minimum with minimal_workspace=True, or when the larger
    one does not fit in device memory)."""
    lib = load()
    _contig(q, k, v, o, lse, dout)
    s, sh = segs.struct(), _shape(q, k, softmax_scale)
    full, low = C.c_size_t(), C.c_size_t()
    _check(lib.ism_attn_bwd_workspace_size(C.byref(s), C.byref(sh), C.byref(full)), "ism_attn_bwd_workspace_size")
    _check(lib.ism_attn_bwd_workspace_size_min(C.byref(s), C.byref(sh), C.byref(low)),
           "ism_attn_bwd_workspace_size_min")
    dq = torch.empty_like(q) if dq is None else dq
    dk = torch.empty_like(k) if dk is None else dk
    dv = torch.empty_like(v) if dv is None else dv
    if workspace is None or workspace.numel() < low.value:
        if minimal_workspace:
            workspace = _workspace(low.value, q.device)
        else:
            try:
                workspace = _workspace(full.value, q.device)
            except torch.cuda.OutOfMemoryError:
                workspace = _workspace(low.value, q.device)
    if plan is not None:  # the plan's metadata instead of a metadata pass
        _check(lib.ism_attn_bwd_planned(C.byref(s), C.byref(sh), _ptr(plan.buffer), C.byref(plan.info), _ptr(q),
                                        _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(dout), _ptr(dq), _ptr(dk),
                                        _ptr(dv), _ptr(workspace), workspace.numel(), _stream(q.device)),
               "ism_attn_bwd_planned")
        return dq, dk, dv
    _check(lib.ism_attn_bwd(C.byref(s), C.byref(sh), _ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(dout),
                            _ptr(dq), _ptr(dk), _ptr(dv), _ptr(workspace), workspace.numel(), _stream(q.device)),
           "ism_attn_bwd")
    return dq, dk, dv


def append_workspace_size(q_new, k_new, softmax_scale: float, rope: bool = False) -> int:
    """Workspace bytes ``prefill_append`` (``prefill_append_rope`` when rope is
    set) needs for this batch and chunk length."""
    lib = load()
    B, Ln = q_new.shape[0], q_new.shape[1]
    sh = _shape(q_new, k_new, softmax_scale)
    nbytes = C.c_size_t()
    name = "ism_attn_prefill_append_rope_workspace_size" if rope else "ism_attn_prefill_append_workspace_size"
    _check(getattr(lib, name)(C.byref(sh), B, Ln, C.byref(nbytes)), name)
    return nbytes.value


def _rope_struct(cos, sin) -> _Rope:
    _contig(cos, sin)
    if cos.dtype != torch.float32 or sin.dtype != torch.float32 or cos.shape != sin.shape or cos.dim() != 2:
        raise ValueError("rope tables must be float32 [rows, head_dim/2] tensors of one shape")
    return _Rope(_ptr(cos), _ptr(sin), cos.shape[0])


def prefill_append_rope(q_new, k_new, v_new, k_cache, v_cache, cache_len, cache_len_host, new_seg_end, new_seg_type,
                        rope_cos, rope_sin, softmax_scale: float, out=None, lse=None, workspace=None):
    """``prefill_append`` with rotary encoding of the new queries and keys at
    positions cache_len[b] + j (rotate-half pairs, angles given by the fp32
    tables rope_cos / rope_sin [rows, D/2]); the caches receive the rotated
    keys.  Returns (o_new, lse [Hq,B,Ln])."""
    lib = load()
    _contig(q_new, k_new, v_new, k_cache, v_cache, cache_len)
    B, Ln, hq, D = q_new.shape
    sh = _shape(q_new, k_new, softmax_scale)
    se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
    st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
    ch = np.ascontiguousarray(cache_len_host, dtype=np.int32)
    rope = _rope_struct(rope_cos, rope_sin)
    nbytes = append_workspace_size(q_new, k_new, softmax_scale, rope=True)
    if out is None:
        out = torch.empty_like(q_new)
    if lse is None:
        lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device)
    if workspace is None or workspace.numel() < nbytes:
        workspace = _workspace(nbytes, q_new.device)
    _check(lib.ism_attn_prefill_append_rope(C.byref(sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                                            C.c_void_p(se.ctypes.data), C.c_void_p(st.ctypes.data), se.shape[0],
                                            _ptr(k_cache), _ptr(v_cache), k_cache.shape[1], _ptr(cache_len),
                                            C.c_void_p(ch.ctypes.data), C.byref(rope), _ptr(out), _ptr(lse),
                                            _ptr(workspace), workspace.numel(), _stream(q_new.device)),
           "ism_attn_prefill_append_rope")
    return out, lse


def prefill_append(q_new, k_new, v_new, k_cache, v_cache, cache_len, cache_len_host, new_seg_end, new_seg_type,
                   softmax_scale: float, out=None, lse=None, workspace=None):
    """Append a new turn to the KV caches and attend (Section 2.3).
    q_new [B,Ln,Hq,D], k_new/v_new [B,Ln,Hkv,D], caches [B,cap,Hkv,D],
    cache_len int32 [B] on the device (advanced by Ln), cache_len_host its
    host mirror (the caller advances it).  Returns (o_new, lse [Hq,B,Ln])."""
    lib = load()
    _contig(q_new, k_new, v_new, k_cache, v_cache, cache_len)
    B, Ln, hq, D = q_new.shape
    cap = k_cache.shape[1]
    sh = _shape(q_new, k_new, softmax_scale)
    se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
    st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
    ch = np.ascontiguousarray(cache_len_host, dtype=np.int32)
    nbytes = C.c_size_t()
    _check(lib.ism_attn_prefill_append_workspace_size(C.byref(sh), B, Ln, C.byref(nbytes)),
           "ism_attn_prefill_append_workspace_size")
    if out is None:
        out = torch.empty_like(q_new)
    if lse is None:
        lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device)
    if workspace is None or workspace.numel() < nbytes.value:
        workspace = _workspace(nbytes.value, q_new.device)
    _check(lib.ism_attn_prefill_append(C.byref(sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                                       C.c_void_p(se.ctypes.data), C.c_void_p(st.ctypes.data), se.shape[0],
                                       _ptr(k_cache), _ptr(v_cache), cap, _ptr(cache_len), C.c_void_p(ch.ctypes.data),
                                       _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(),
                                       _stream(q_new.device)),
           "ism_attn_prefill_append")
    return out, lse


class AppendStep:
    """A prepared ``prefill_append`` call for a generation loop: the arguments
    are marshalled once, so each step is one C call.  The caller keeps the new
    token buffers (q_new, k_new, v_new) and the int32 numpy ``cache_len_host``
    array, refills the buffers before each call and advances the host array in
    place after it (the device ``cache_len`` advances itself)."""

    def __init__(self, q_new, k_new, v_new, k_cache, v_cache, cache_len, cache_len_host: np.ndarray, new_seg_end,
                 new_seg_type, softmax_scale: float, out=None, lse=None, workspace=None, rope=None):
        lib = load()
        _contig(q_new, k_new, v_new, k_cache, v_cache, cache_len)
        if not (isinstance(cache_len_host, np.ndarray) and cache_len_host.dtype == np.int32 and
                cache_len_host.flags["C_CONTIGUOUS"]):
            raise TypeError("cache_len_host must be a contiguous int32 numpy array (advanced in place)")
        B, Ln, hq, D = q_new.shape
        self._sh = _shape(q_new, k_new, softmax_scale)
        self._se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
        self._st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
        self._host = cache_len_host
        self.out = torch.empty_like(q_new) if out is None else out
        self.lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device) if lse is None else lse
        if workspace is None:
            workspace = _workspace(append_workspace_size(q_new, k_new, softmax_scale, rope=rope is not None),
                                   q_new.device)
        self._keep = (q_new, k_new, v_new, k_cache, v_cache, cache_len, workspace, rope)
        head = (C.byref(self._sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                C.c_void_p(self._se.ctypes.data), C.c_void_p(self._st.ctypes.data), self._se.shape[0],
                _ptr(k_cache), _ptr(v_cache), k_cache.shape[1], _ptr(cache_len),
                C.c_void_p(cache_len_host.ctypes.data))
        tail = (_ptr(self.out), _ptr(self.lse), _ptr(workspace), workspace.numel(), _stream(q_new.device))
        if rope is None:
            self._name = "ism_attn_prefill_append"
            self._args = head + tail
        else:
            self._rope = _rope_struct(*rope)
            self._name = "ism_attn_prefill_append_rope"
            self._args = head + (C.byref(self._rope),) + tail
        self._fn = getattr(lib, self._name)

    def __call__(self):
        _check(self._fn(*self._args), self._name)
        return self.out, self.lse


def prefill_append_e4m3(q_new, k_new, v_new, k_cache, v_cache, cache_len, cache_len_host, new_seg_end, new_seg_type,
                        q_descale: float, k_descale: float, v_descale: float, softmax_scale: float, out=None, lse=None,
                        workspace=None):
    """``prefill_append`` with e4m3 (torch.float8_e4m3fn) q_new, k_new, v_new and
    caches, dequantised by the per-tensor factors; returns (o bf16, lse)."""
    lib = load()
    _contig(q_new, k_new, v_new, k_cache, v_cache, cache_len)
    B, Ln, hq, D = q_new.shape
    cap = k_cache.shape[1]
    sh = _shape(q_new, k_new, softmax_scale)
    se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
    st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
    ch = np.ascontiguousarray(cache_len_host, dtype=np.int32)
    if out is None:
        out = torch.empty(q_new.shape, dtype=torch.bfloat16, device=q_new.device)
    if lse is None:
        lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device)
    if workspace is None:
        workspace = _workspace(append_workspace_size(q_new, k_new, softmax_scale), q_new.device)
    _check(lib.ism_attn_prefill_append_e4m3(C.byref(sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                                            C.c_void_p(se.ctypes.data), C.c_void_p(st.ctypes.data), se.shape[0],
                                            _ptr(k_cache), _ptr(v_cache), cap, _ptr(cache_len),
                                            C.c_void_p(ch.ctypes.data), q_descale, k_descale, v_descale, _ptr(out),
                                            _ptr(lse), _ptr(workspace), workspace.numel(), _stream(q_new.device)),
           "ism_attn_prefill_append_e4m3")
    return out, lse


def prefill_append_paged(q_new, k_new, v_new, k_pool, v_pool, page_size: int, block_table, block_table_host,
                         cache_len, cache_len_host, new_seg_end, new_seg_type, softmax_scale: float, out=None,
                         lse=None, workspace=None):
    """``prefill_append`` against a paged cache (Section 2.3): k_pool/v_pool
    [num_pages * page_size, Hkv, D]; key p of sequence b is pool row
    block_table[b, p // page_size] * page_size + p % page_size.  block_table
    int32 [B, max_pages] on the device, block_table_host its host mirror
    (numpy); cache_len / cache_len_host as for ``prefill_append``."""
    lib = load()
    _contig(q_new, k_new, v_new, k_pool, v_pool, cache_len, block_table)
    B, Ln, hq, D = q_new.shape
    rows = k_pool.shape[0]
    if rows % page_size:
        raise ValueError("pool rows must be a whole number of pages")
    sh = _shape(q_new, k_new, softmax_scale)
    se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
    st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
    ch = np.ascontiguousarray(cache_len_host, dtype=np.int32)
    bt = np.ascontiguousarray(block_table_host, dtype=np.int32)
    if out is None:
        out = torch.empty_like(q_new)
    if lse is None:
        lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device)
    if workspace is None:
        workspace = _workspace(append_workspace_size(q_new, k_new, softmax_scale), q_new.device)
    _check(lib.ism_attn_prefill_append_paged(C.byref(sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                                             C.c_void_p(se.ctypes.data), C.c_void_p(st.ctypes.data), se.shape[0],
                                             _ptr(k_pool), _ptr(v_pool), rows // page_size, page_size,
                                             _ptr(block_table), C.c_void_p(bt.ctypes.data), block_table.shape[1],
                                             _ptr(cache_len), C.c_void_p(ch.ctypes.data), _ptr(out), _ptr(lse),
                                             _ptr(workspace), workspace.numel(), _stream(q_new.device)),
           "ism_attn_prefill_append_paged")
    return out, lse


def prefill_append_paged_rope(q_new, k_new, v_new, k_pool, v_pool, page_size: int, block_table, block_table_host,
                              cache_len, cache_len_host, new_seg_end, new_seg_type, rope_cos, rope_sin,
                              softmax_scale: float, out=None, lse=None, workspace=None):
    """``prefill_append_paged`` with rotary encoding of the new queries and
    keys at positions cache_len[b] + j (as ``prefill_append_rope``)."""
    lib = load()
    _contig(q_new, k_new, v_new, k_pool, v_pool, cache_len, block_table)
    B, Ln, hq, D = q_new.shape
    rows = k_pool.shape[0]
    if rows % page_size:
        raise ValueError("pool rows must be a whole number of pages")
    sh = _shape(q_new, k_new, softmax_scale)
    se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
    st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
    ch = np.ascontiguousarray(cache_len_host, dtype=np.int32)
    bt = np.ascontiguousarray(block_table_host, dtype=np.int32)
    rope = _rope_struct(rope_cos, rope_sin)
    out = torch.empty_like(q_new) if out is None else out
    lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device) if lse is None else lse
    if workspace is None:
        workspace = _workspace(append_workspace_size(q_new, k_new, softmax_scale, rope=True), q_new.device)
    _check(lib.ism_attn_prefill_append_paged_rope(C.byref(sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                                                  C.c_void_p(se.ctypes.data), C.c_void_p(st.ctypes.data),
                                                  se.shape[0], _ptr(k_pool), _ptr(v_pool), rows // page_size,
                                                  page_size, _ptr(block_table), C.c_void_p(bt.ctypes.data),
                                                  block_table.shape[1], _ptr(cache_len), C.c_void_p(ch.ctypes.data),
                                                  C.byref(rope), _ptr(out), _ptr(lse), _ptr(workspace),
                                                  workspace.numel(), _stream(q_new.device)),
           "ism_attn_prefill_append_paged_rope")
    return out, lse


def prefill_append_e4m3_rope(q_new, k_new, v_new, k_cache, v_cache, cache_len, cache_len_host, new_seg_end,
                             new_seg_type, q_descale: float, k_descale: float, v_descale: float, rope_cos, rope_sin,
                             softmax_scale: float, out=None, lse=None, workspace=None):
    """Rotary append against e4m3 caches: q_new, k_new, v_new are bf16 and
    unrotated; queries and keys are rotated at positions cache_len[b] + j,
    then quantised with the factors (keys and values into the caches).
    Returns (o bf16, lse [Hq,B,Ln])."""
    lib = load()
    _contig(q_new, k_new, v_new, k_cache, v_cache, cache_len)
    B, Ln, hq, D = q_new.shape
    sh = _Shape()
    sh.num_heads_q, sh.num_heads_kv, sh.head_dim = hq, k_new.shape[2], D
    sh.dtype, sh.softmax_scale = ISM_E4M3, float(softmax_scale)
    se = np.ascontiguousarray(new_seg_end, dtype=np.int32)
    st = np.ascontiguousarray(new_seg_type, dtype=np.uint8)
    ch = np.ascontiguousarray(cache_len_host, dtype=np.int32)
    rope = _rope_struct(rope_cos, rope_sin)
    out = torch.empty(q_new.shape, dtype=torch.bfloat16, device=q_new.device) if out is None else out
    lse = torch.empty((hq, B, Ln), dtype=torch.float32, device=q_new.device) if lse is None else lse
    if workspace is None:
        nbytes = C.c_size_t()
        _check(lib.ism_attn_prefill_append_rope_workspace_size(C.byref(sh), B, Ln, C.byref(nbytes)),
               "ism_attn_prefill_append_rope_workspace_size")
        workspace = _workspace(nbytes.value, q_new.device)
    _check(lib.ism_attn_prefill_append_e4m3_rope(C.byref(sh), B, _ptr(q_new), _ptr(k_new), _ptr(v_new), Ln,
                                                 C.c_void_p(se.ctypes.data), C.c_void_p(st.ctypes.data), se.shape[0],
                                                 _ptr(k_cache), _ptr(v_cache), k_cache.shape[1], _ptr(cache_len),
                                                 C.c_void_p(ch.ctypes.data), q_descale, k_descale, v_descale,
                                                 C.byref(rope), _ptr(out), _ptr(lse), _ptr(workspace),
                                                 workspace.numel(), _stream(q_new.device)),
           "ism_attn_prefill_append_e4m3_rope")
    return out, lse


def debug_mma_tile_e4m3(a: torch.Tensor, b: torch.Tensor, mode: int) -> torch.Tensor:
    """One 128x128x128 e4m3 tcgen05 tile product (diagnostic): mode 0 a @ b.T,
    mode 1 a @ b, mode 2 a @ b with a in tensor memory; a, b float8_e4m3fn."""
    c = torch.empty((128, 128), dtype=torch.float32, device=a.device)
    _check(load().ism_debug_mma_tile_e4m3(_ptr(a), _ptr(b), _ptr(c), mode, _stream(a.device)),
           "ism_debug_mma_tile_e4m3")
    return c


def check_status(device=None):
    """Synchronise the current stream and raise if a kernel gave up a wait."""
    _check(load().ism_check_status(_stream(device)), "ism_check_status")


def debug_timeout_probe(spin_limit: int = 64, device=None) -> int:
    """Run the bounded-wait probe; returns the status code ism_check_status
    reports afterwards (expected ISM_ERR_TIMEOUT = 4)."""
    lib = load()
    _check(lib.ism_debug_timeout_probe(spin_limit, _stream(device)), "ism_debug_timeout_probe")
    return lib.ism_check_status(_stream(device))


def has_tensor_cores() -> bool:
    return bool(load().ism_has_tensor_cores())


def set_kernel_timer(kernel_id: int, start: "torch.cuda.Event" = None, stop: "torch.cuda.Event" = None):
    """Bracket every launch of one kernel kind (on this thread) with the
    given CUDA events; call with no events to clear."""
    sp = None if start is None else C.c_void_p(start.cuda_event)
    ep = None if stop is None else C.c_void_p(stop.cuda_event)
    _check(load().ism_set_kernel_timer(kernel_id, sp, ep), "ism_set_kernel_timer")


def kernel_launches() -> int:
    return int(load().ism_kernel_launches())


def debug_mma_tile(a: torch.Tensor, b: torch.Tensor, mode: int) -> torch.Tensor:
    """One 128x128x128 tcgen05 tile product (diagnostic): mode 0/2/4 a @ b.T,
    mode 1/3/5 a @ b, mode 6/7 a.T @ b; modes 2/3 stage operands with TMA,
    4/5 put a in tensor memory, 7 stages a 8-interleaved; mode + 8 issues the
    k-steps through the batched one-election form."""
    c = torch.empty((128, 128), dtype=torch.float32, device=a.device)
    _check(load().ism_debug_mma_tile(_ptr(a), _ptr(b), _ptr(c), mode, _stream(a.device)), "ism_debug_mma_tile")
    return c
